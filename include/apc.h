/*
 * apc: the committed optimizer step of zero-I/O fault recovery, as a C ABI.
 *
 * arxiv 2609.18178 recovers sharded training in place when a collective
 * fails at a committed optimizer boundary: the point where the parameter
 * and moment updates of the step have landed, flat-parameter gradients are
 * zeroed and device streams are synchronized (Section I; Section III-C,
 * phase 2).  The device state it keeps is S_app = {W, M, V, ..., tau_opt}
 * (Section III-A, Eq. 2), and it relies on every rank holding bit-identical
 * parameter and optimizer state after repair (Abstract; Sections IV-F and
 * IV-G, "rank state checks passing bitwise").
 *
 * This library computes, on one GPU, the step that reaches that boundary for
 * one rank's flat parameter shard, and a 64-bit digest per state buffer that
 * lets peers prove bit-identity by exchanging 32 bytes instead of
 * checkpoints:
 *
 *   apc_commit_step  AdamW update of fp32 master params p and moments m, v
 *                    from a bf16 gradient g, a bf16 copy w of p', and the
 *                    digests of p', m', v', w, in one pass over HBM.
 *   apc_digest       the same digests of arbitrary buffers, read-only (the
 *                    post-recovery verification).
 *
 * Numeric contract (identical bits on every run, grid size and table split):
 *   scalars  b1, 1-b1, b2, 1-b2, eps, 1-lr*wd, lr/(1-b1^t), 1/sqrt(1-b2^t),
 *            each formed in double from the hyper-parameters and rounded once
 *            to binary32 on the host (apc_resolve_hparams);
 *   update   per element, binary32, one rounding per operation, no fusion:
 *              g  = bf16 -> f32 (exact)
 *              m' = b1*m + (1-b1)*g
 *              v' = b2*v + (1-b2)*(g*g)
 *              den = sqrt(v') * rsb2 + eps          (IEEE sqrt)
 *              p' = p*(1-lr*wd) - step*(m'/den)     (IEEE divide)
 *              w  = bf16 round-to-nearest-even of p'
 *            Infinities and NaNs in p, m, v or g follow IEEE 754 through
 *            each operation.  A NaN result is written as a NaN whose payload
 *            is left open (IEEE 754 does not fix it), and the bf16 copy of a
 *            NaN is a bf16 NaN; every other result is the exact bits above.
 *   digest   D_B = sum over elements of
 *              splitmix64(((G mod 2^32) << 32) | bits_B)   (mod 2^64)
 *            G the element's index in the flat model (global_offset + i),
 *            bits_B its binary32 bits or zero-extended bf16 bits, and
 *            splitmix64(x) the first output of SplitMix64 seeded with x.
 *            Only G mod 2^32 enters the key: equal words exactly k*2^32
 *            elements apart have equal keys.
 *
 * Conventions for every call:
 *   - Device pointers belong to the calling thread's current CUDA device:
 *     every buffer a kernel reads or writes, and every output, must be
 *     device memory of that device (or managed memory).  Each call checks
 *     this with one cudaPointerGetAttributes query per distinct address and
 *     returns APC_EINVAL for host memory or another device's memory.
 *     The caller owns all memory and the library allocates nothing.  Between
 *     calls it keeps only each device's SM count and kernel residency
 *     (queried once), the kernels' device status word (apc_device_status)
 *     and the number of SMs to leave free (apc_set_reserved_sms).
 *   - Work is enqueued on `stream` (NULL = the legacy default stream); the
 *     call never synchronizes.  Results, including the digests, are valid
 *     once the stream reaches that point.
 *   - Tables and buffer lists are read before the call returns; the caller
 *     may reuse them at once.
 *   - Errors are returned, never raised: no call aborts the process.  On an
 *     error before launch nothing is enqueued.  apc_last_error() gives a
 *     human-readable detail of the calling thread's last failure.
 *   - Every kernel runs a persistent grid of (SM count x residency) CTAs, or
 *     fewer when there is less work.  The environment variable
 *     APC_GRID_LIMIT, if set to a positive integer when a call is made, caps
 *     that grid (for tests of grid independence and for sharing the GPU);
 *     results do not depend on it.
 */
#ifndef APC_H
#define APC_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* The same type as cudaStream_t. */
typedef struct CUstream_st *apc_stream_t;

typedef enum apc_status {
  APC_OK = 0,
  APC_EINVAL = 1, /* null pointer, bad count, out-of-range hyper-parameter or step,
                     overlapping outputs, memory that is not the current device's */
  APC_EALIGN = 2, /* pointer not aligned to its element size                       */
  APC_ERANGE = 3, /* global_offset + n overflows 64 bits                           */
  APC_ECUDA = 4,  /* the CUDA runtime reported an error (launch or attribute query) */
  APC_ETIMEOUT = 5 /* a bounded wait inside a kernel gave up (see apc_device_status) */
} apc_status;

/* Decimal AdamW hyper-parameters (double).  Valid: lr >= 0, 0 <= beta < 1,
 * eps > 0, weight_decay >= 0, all finite. */
typedef struct apc_adamw_hparams {
  double lr, beta1, beta2, eps, weight_decay;
} apc_adamw_hparams;

/* One entry of the chunk table: a tensor of the flat shard, or a slice of it.
 *   p, m, v  fp32, device, n elements each, read and updated in place
 *   g        bf16 bits, device, n elements, read only
 *   w        bf16 bits, device, n elements, written (p' rounded to bf16)
 *   global_offset  index of element 0 in the flat model (the digest key)
 * p, m, v need 4-byte and g, w 2-byte alignment; the kernel runs 16-byte
 * vectors wherever the five buffers are mutually aligned and scalar code
 * elsewhere.  n == 0 entries are skipped and their pointers may be NULL.
 * The written ranges of all entries (p, m, v, w) must not overlap each other
 * or any gradient range. */
typedef struct apc_tensor {
  float *p, *m, *v;
  const uint16_t *g;
  uint16_t *w;
  uint64_t n;
  uint64_t global_offset;
} apc_tensor;

typedef enum apc_dtype { APC_F32 = 0, APC_BF16 = 1 } apc_dtype;

/* One buffer for apc_digest: n elements of `dtype` at `data` (device), whose
 * element 0 has index global_offset in the flat model, summed into digest
 * slot `slot`. */
typedef struct apc_buffer {
  const void *data;
  uint64_t n;
  uint64_t global_offset;
  uint32_t dtype; /* apc_dtype */
  uint32_t slot;
} apc_buffer;

#define APC_MAX_SLOTS 8

/* The committed AdamW step plus state digest over a chunk table.
 *
 * Defines the step that reaches the committed optimizer boundary (arxiv
 * 2609.18178 Section I; Section III-C, phase 2): it updates the preserved
 * state W, M, V of S_app for optimizer step tau_opt (Section III-A, Eq. 2)
 * and emits the digests that the bitwise rank-state checks compare
 * (Sections IV-F, IV-G).
 *
 * table[0..num_tensors): the tensors of one rank's shard (any number; tables
 *   larger than one launch's capacity are split into several launches on
 *   `stream`, with identical results).  num_tensors == 0 is valid.
 * hp, step: hyper-parameters and the 1-based optimizer step t (tau_opt).
 * out_digests: device, 4 x uint64, written as {D_p', D_m', D_v', D_w}; it is
 *   zeroed on `stream` first, so it need not be initialised.  It must not
 *   overlap any buffer of the table.
 * Returns APC_EINVAL (null table with num_tensors > 0, null hp or
 * out_digests, num_tensors < 0, step < 1, hyper-parameters out of range,
 * overlapping outputs, a buffer or out_digests that is not memory of the
 * current device), APC_EALIGN, APC_ERANGE, APC_ECUDA, or APC_OK. */
apc_status apc_commit_step(const apc_tensor *table, int32_t num_tensors, const apc_adamw_hparams *hp,
                           int64_t step, apc_stream_t stream, uint64_t *out_digests);

/* Flags of apc_commit_step_ex. */
#define APC_COMMIT_ZERO_GRAD 1u /* also write g := +0 in the same pass (the gradient buffers are written) */

/* apc_commit_step with options.  flags = 0 is apc_commit_step.  With
 * APC_COMMIT_ZERO_GRAD the pass also zeroes every gradient element after
 * reading it, so that on return the shard sits at a committed boundary:
 * updates landed and flat-parameter gradients zeroed (arxiv 2609.18178,
 * Section I).  The `g` pointers are then written despite their const type,
 * and gradient ranges count as written ranges for the overlap check.
 * Results (p', m', v', w, digests) are identical with and without the flag.
 * Returns APC_EINVAL for unknown flag bits, otherwise as apc_commit_step. */
apc_status apc_commit_step_ex(const apc_tensor *table, int32_t num_tensors, const apc_adamw_hparams *hp,
                              int64_t step, uint32_t flags, apc_stream_t stream, uint64_t *out_digests);

/* One entry of a bf16-state chunk table: p, m, v bf16 bits (device, n
 * elements, read and updated in place), g bf16 bits (read; written with
 * APC_COMMIT_ZERO_GRAD).  2-byte alignment; same skipping and overlap rules
 * as apc_tensor. */
typedef struct apc_tensor_bf16 {
  uint16_t *p, *m, *v;
  const uint16_t *g;
  uint64_t n;
  uint64_t global_offset;
} apc_tensor_bf16;

/* The committed step with parameters and moments kept in bf16 (the paper's
 * own setting: "Model parameters and AdamW moments use BF16", arxiv
 * 2609.18178 Section IV-A).  Per element: p, m, v and g are widened exactly
 * to binary32, the update runs in the same fixed order as apc_commit_step,
 * and p', m', v' are each rounded once to bf16 (nearest even) when stored;
 * there is no separate working copy.  out_digests: device, 3 x uint64,
 * written as {D_p', D_m', D_v'} over the bf16 words (zero-extended).  flags
 * as apc_commit_step_ex.  Errors as apc_commit_step. */
apc_status apc_commit_step_bf16(const apc_tensor_bf16 *table, int32_t num_tensors, const apc_adamw_hparams *hp,
                                int64_t step, uint32_t flags, apc_stream_t stream, uint64_t *out_digests);

/* The state digest of a list of buffers, read only.
 *
 * The post-recovery verification: peers compare these digests to prove
 * that device state is bit-identical without checkpoint I/O (the bitwise
 * rank-state checks of arxiv 2609.18178, Abstract and Sections IV-F, IV-G,
 * over the preserved W, M, V of Section III-A, Eq. 2).
 *
 * bufs[0..num_bufs): buffers; each adds its elements into out_digests[slot].
 * num_slots: 1..APC_MAX_SLOTS; out_digests (device, num_slots x uint64) is
 *   zeroed on `stream` first; it must not overlap any buffer of the list.
 * The digest of the four buffers that apc_commit_step wrote, given as slots
 * 0..3 with the table's offsets, equals that call's out_digests.
 * Returns APC_EINVAL (null pointers, bad counts, bad dtype, slot >=
 * num_slots, an output that overlaps a buffer, a pointer that is not memory
 * of the current device), APC_EALIGN, APC_ERANGE, APC_ECUDA, or APC_OK. */
apc_status apc_digest(const apc_buffer *bufs, int32_t num_bufs, int32_t num_slots, apc_stream_t stream,
                      uint64_t *out_digests);

/* The quiescence guard: per-slot counts of buffer words whose bit pattern
 * is nonzero, read only (the "zero outstanding gradients" check of the
 * recovery protocol's guard, arxiv 2609.18178 Section III-C, phase 2).
 * Same buffer list, slots and error behaviour as apc_digest (global_offset
 * is ignored); out_counts: device, num_slots x uint64, zeroed on `stream`
 * first.  A -0.0 word counts as nonzero. */
apc_status apc_count_nonzero(const apc_buffer *bufs, int32_t num_bufs, int32_t num_slots, apc_stream_t stream,
                             uint64_t *out_counts);

/* The eight binary32 scalars that apc_commit_step passes to the device for
 * step t, in the order b1, 1-b1, b2, 1-b2, eps, 1-lr*wd, lr/(1-b1^t),
 * 1/sqrt(1-b2^t).  t is the optimizer step tau_opt of the preserved state
 * (arxiv 2609.18178 Section III-A, Eq. 2), on which the bias corrections
 * depend.  Host only; no CUDA call.  out: host, 8 floats. */
apc_status apc_resolve_hparams(const apc_adamw_hparams *hp, int64_t step, float out[8]);

/* One segment of apc_upload: `bytes` bytes from `src` to `dst`.
 *   dst  device memory of the current device (or managed memory), written
 *   src  memory the current device can read: page-locked host memory mapped
 *        for the device (cudaHostAlloc, cudaHostRegister), pageable host
 *        memory on devices that read it through the host's page tables
 *        (cudaDevAttrPageableMemoryAccess), managed memory, or the current
 *        device's own memory */
typedef struct apc_segment {
  void *dst;
  const void *src;
  uint64_t bytes;
} apc_segment;

/* Host-to-device upload executed by the SMs: the CTAs of one kernel load the
 * sources in 16-byte words (bytes outside mutually 16-byte-aligned runs one
 * by one) and store them to device memory.  On Grace-Blackwell the loads
 * cross NVLink-C2C at the link's rate and need no DMA copy engine.  The
 * kernel runs on at most max_ctas CTAs (0 = one per SM; 1 .. 4096), so that
 * it can run on another stream beside this library's persistent kernels when
 * those leave SMs free (apc_set_reserved_sms): for example, the next
 * gradients' upload beside the current step.  A segment's destination must
 * not overlap another destination or any source.  bytes == 0 segments are
 * skipped.  Ordered on `stream` like
 * a kernel; the call never synchronizes.
 * Returns APC_EINVAL (null pointers, num_segments < 0, max_ctas out of
 * range, a source the current device cannot read, a destination outside the
 * current device's memory, overlapping ranges), APC_ERANGE (address + bytes
 * overflows), APC_ECUDA, or APC_OK. */
apc_status apc_upload(const apc_segment *segs, int32_t num_segments, int32_t max_ctas, apc_stream_t stream);

/* Leave n SMs free of this library's persistent kernels: later launches of
 * the step, digest and guard kernels run at most (SM count - n) x residency
 * CTAs (at least one SM's worth), so that kernels of other streams, such as
 * apc_upload, run beside them.  Results do not depend on it.  Process-wide,
 * for every device; n: 0 (the default) .. 1024.  Returns APC_EINVAL for n
 * out of range. */
apc_status apc_set_reserved_sms(int32_t n);

/* Device-side status of this library's kernels on the current device since
 * the previous call: APC_OK, or APC_ETIMEOUT if a bounded wait inside a
 * kernel gave up.  A kernel that gives up stops, drains its own copies and
 * exits, leaving the context usable, but its work is incomplete:
 *   - after apc_commit_step(_ex, _bf16), the shard is torn: some tiles hold
 *     step t and others step t-1, in place, and the launch's digests are
 *     dropped.  Nothing in the library can roll it back.  The shard must be
 *     restored from a replica (or checkpoint) before training continues:
 *     the fail-stop rule of the recovery protocol (arxiv 2609.18178 Section
 *     III-C, safety invariant).
 *   - after apc_digest or apc_count_nonzero, only the outputs are wrong; the
 *     call can be repeated.
 * A wait gives up after at least 2^20 polls and 1 s of the GPU's global
 * timer; a kernel that is descheduled does not poll, so time slicing alone
 * does not make it give up, but a GPU shared with other contexts can in
 * principle delay a healthy wait past the limit.
 * Synchronizes the device, reads the status word and clears it.  Returns
 * APC_ECUDA if the CUDA runtime reports an error. */
apc_status apc_device_status(void);

/* Self-test of the bounded-wait path: launch one thread on `stream` that
 * waits on a shared-memory barrier that nothing completes; it gives up after
 * limit_ns nanoseconds (and at least 2^20 polls) and records APC_ETIMEOUT,
 * which the next apc_device_status() returns.  limit_ns: 1 .. 10^10. */
apc_status apc_selftest_wait_timeout(uint64_t limit_ns, apc_stream_t stream);

/* Static description of a status code. */
const char *apc_status_string(apc_status s);

/* Detail of the calling thread's last failing call ("" if none).  The
 * pointer stays valid until that thread's next apc_* call. */
const char *apc_last_error(void);

/* ABI version of this header: 3. */
int32_t apc_version(void);

#ifdef __cplusplus
}
#endif

#endif /* APC_H */
