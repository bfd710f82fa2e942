// Launch plans shared by the host side of the C ABI and the kernels.
//
// A plan is a kernel parameter block (__grid_constant__, at most 32,764
// bytes): the chunk table is copied by the driver at launch, so nothing is
// staged in device memory and no allocation is needed.  Tables larger than
// one block are split over several launches that add into the same digests.
#pragma once

#include <stdint.h>

namespace apc {

constexpr int kVec = 8;                    // vector granularity: 16 bytes of bf16, 32 bytes of fp32
constexpr uint32_t kScalarMode = 0xFFFFFFFFu;  // `head` value of an entry run without vectors

// Commit kernel: warp-specialized pipeline.  One producer warp streams each
// tile of p, m, v and g into a ring of shared-memory stages with bulk
// asynchronous copies; the consumer warps compute from shared memory and
// store straight to global memory.
//
// Pipeline shape (compile-time, per state layout; the defaults are the
// measured best on GB300).
//  * fp32 state: 19 consumer warps + 1 producer = 20 warps, 5 per SM
//    sub-partition: each sub-partition's 16,384 registers then give 96 per
//    thread with no spills, the same budget as 16 + 1 warps (whose fifth
//    warp on one sub-partition sets the cap), with three more warps issuing.
//    Each consumer thread takes 2 groups of 4 elements per tile (3 ran 6%
//    slower).
//  * bf16 state stages 8 bytes per element instead of 14 and needs fewer
//    registers: 27 consumer warps + 1 producer = 28 warps at 72 registers
//    with no spills, 3 groups per thread per tile.  That is 3.2% faster than
//    the fp32 layout's shape there (19 warps and 4 groups were 1.8% faster
//    than 19 and 2; 23 warps with 3 groups and 31 with 2 were in between).
#ifndef APC_COMMIT_CONSUMER_WARPS
#define APC_COMMIT_CONSUMER_WARPS 19
#endif
#ifndef APC_COMMIT_CONSUMER_WARPS_BF16
#define APC_COMMIT_CONSUMER_WARPS_BF16 27
#endif
#ifndef APC_COMMIT_GROUPS
#define APC_COMMIT_GROUPS 2
#endif
#ifndef APC_COMMIT_GROUPS_BF16
#define APC_COMMIT_GROUPS_BF16 3
#endif
// Ring stages per CTA: three for fp32 state (0.3% faster than two), two for
// bf16 state (three of its larger tiles exceed a CTA's shared memory).
#ifndef APC_COMMIT_STAGES
#define APC_COMMIT_STAGES 3
#endif
#ifndef APC_COMMIT_BLOCKS_PER_SM
#define APC_COMMIT_BLOCKS_PER_SM 1
#endif
constexpr int kCommitConsumerWarps = APC_COMMIT_CONSUMER_WARPS;
constexpr int kCommitConsumerWarpsBF16 = APC_COMMIT_CONSUMER_WARPS_BF16;
constexpr int kCommitGroups = APC_COMMIT_GROUPS;
constexpr int kCommitGroupsBF16 = APC_COMMIT_GROUPS_BF16;
constexpr uint64_t kCommitTile = (uint64_t)kCommitConsumerWarps * 32 * 4 * kCommitGroups;              // 4,864 elements
constexpr uint64_t kCommitTileBF16 = (uint64_t)kCommitConsumerWarpsBF16 * 32 * 4 * kCommitGroupsBF16;  // 10,368 elements
constexpr int kCommitStages = APC_COMMIT_STAGES;
#ifndef APC_COMMIT_STAGES_BF16
#define APC_COMMIT_STAGES_BF16 2
#endif
constexpr int kCommitStagesBF16 = APC_COMMIT_STAGES_BF16;
constexpr int kCommitBlocksPerSm = APC_COMMIT_BLOCKS_PER_SM;
// Register budget of the fp32-state commit kernel: its launch bound is
// max(block size, APC_COMMIT_BOUND_THREADS) threads, so a build with fewer
// consumer warps can keep the default 96 registers per thread (and leave the
// rest of the SM to a co-resident kernel) instead of growing into them.
#ifndef APC_COMMIT_BOUND_THREADS
#define APC_COMMIT_BOUND_THREADS 0
#endif
// Shared-memory carveout preference (percent of the unified L1/shared
// capacity) given to the commit and digest kernels; -1 leaves the driver's
// default.  100 lets two different kernels' CTAs share an SM.
#ifndef APC_SMEM_CARVEOUT
#define APC_SMEM_CARVEOUT -1
#endif
// Tile order of the commit kernel: 1 = CTA b takes one contiguous run of
// tiles (the runs differ by at most one tile), 0.3-0.7% faster than 0 = CTA b
// takes tiles b, b + grid, ... (the grid sweeping the table together).
#ifndef APC_COMMIT_CONTIGUOUS
#define APC_COMMIT_CONTIGUOUS 1
#endif
// AdamW's multiplies as packed two-lane binary32 instructions over pairs of
// elements (1), or one element at a time (0); the bits are the same.
#ifndef APC_PAIRED_ADAMW
#define APC_PAIRED_ADAMW 1
#endif
// A stage holds one tile of p, m, v and g: 14 bytes per element for fp32
// state (66.5 KB, 200 KB per CTA at the defaults), 8 for bf16 state (81 KB,
// 162 KB per CTA).

// State layouts of the commit kernel.
constexpr int kLayoutF32 = 0;   // fp32 p, m, v; bf16 g; bf16 copy w
constexpr int kLayoutBF16 = 1;  // bf16 p, m, v; bf16 g; no copy

constexpr uint64_t commit_tile(int layout) { return layout == kLayoutBF16 ? kCommitTileBF16 : kCommitTile; }
constexpr int commit_consumers(int layout) {
  return 32 * (layout == kLayoutBF16 ? kCommitConsumerWarpsBF16 : kCommitConsumerWarps);
}

// One chunk-table entry of the commit kernel (72 bytes).
//   p, m, v: fp32 or bf16 state (by the launch's layout); w: the bf16 copy
//         (fp32 layout only).
//   head: elements [0, head) are scalar items, then 16-byte aligned vectors
//         up to vec_end = head + 8 * floor((n - head) / 8) in tiles of
//         commit_tile(layout), then scalar items up to n; kScalarMode when the
//         buffers are not mutually 16-byte aligned (all n elements scalar).
//   tile_begin: the entry's first tile in the launch's tile space.
//   scalar_begin: the entry's first item in the launch's scalar-item space.
//   key_base: global_offset mod 2^32 (the digest key of element 0).
struct CommitEntry {
  void *p, *m, *v;
  const uint16_t *g;
  uint16_t *w;
  uint64_t n;
  uint64_t tile_begin;
  uint64_t scalar_begin;
  uint32_t key_base;
  uint32_t head;
};

template <int MAXE>
struct CommitPlan {
  float h[8];            // b1, 1-b1, b2, 1-b2, eps, 1-lr*wd, lr/bc1, 1/sqrt(bc2)
  uint64_t total_tiles;
  uint64_t total_scalar;
  uint32_t count;
  uint32_t one;          // 1: the FMA-pipe carry-add multiplier of the digest
  CommitEntry e[MAXE];
};

constexpr int kCommitSmall = 16;
constexpr int kCommitLarge = 440;
static_assert(sizeof(CommitEntry) == 72, "entry layout");
static_assert(sizeof(CommitPlan<kCommitLarge>) <= 32764, "kernel parameter limit");

// Digest kernel: the loads are issued by the compute warps themselves (the
// pass is bound by integer issue): a thread handles kDigestUnroll 8-element
// vectors per tile.  One CTA of 1024 threads per SM puts 8 warps on each of
// its four schedulers and gives each SM one contiguous run of tiles; two
// CTAs of the same warps per SM run 2-3% slower, and shapes that load the
// schedulers unevenly (11 or 13 warps per CTA) about 8% slower.
#ifndef APC_DIGEST_THREADS
#define APC_DIGEST_THREADS 1024
#endif
#ifndef APC_DIGEST_UNROLL
#define APC_DIGEST_UNROLL 2
#endif
constexpr int kThreads = APC_DIGEST_THREADS;     // threads per CTA of the digest kernel
constexpr int kDigestUnroll = APC_DIGEST_UNROLL; // thread-vectors per thread per tile
constexpr uint64_t kDigestTile = (uint64_t)kThreads * kVec * kDigestUnroll;  // 16,384 elements

// Guard (count) kernel: the same plans and tiling scheme with its own shape;
// one compare per word leaves it bound by HBM, so its shape is set by the
// bytes each SM keeps in flight: one CTA of 1024 threads per SM with 4
// vectors each (64 KB of bf16 words) reaches 99% of the copy rate, where
// three CTAs of 384 x 3 reached 96%.
#ifndef APC_COUNT_THREADS
#define APC_COUNT_THREADS 1024
#endif
#ifndef APC_COUNT_UNROLL
#define APC_COUNT_UNROLL 4
#endif
constexpr int kCountThreads = APC_COUNT_THREADS;
constexpr int kCountUnroll = APC_COUNT_UNROLL;
constexpr uint64_t kCountTile = (uint64_t)kCountThreads * kVec * kCountUnroll;  // 32,768 elements
// Minimum resident CTAs per SM the digest kernel is compiled for (its
// register cap: 65,536 / (threads x this)), and extra dynamic shared memory
// per CTA beyond its stages (0 by default; a larger CTA footprint keeps two
// digest CTAs off one SM when another kernel is to share it).
#ifndef APC_DIGEST_MIN_BLOCKS
#define APC_DIGEST_MIN_BLOCKS 1
#endif
#ifndef APC_DIGEST_EXTRA_SMEM
#define APC_DIGEST_EXTRA_SMEM 0
#endif

// One buffer of the digest kernel (32 bytes).
//   head: scalar elements before the first 16-byte boundary (<= 7); then
//         8-element vectors in tiles of kDigestTile (kCountTile for the
//         count kernel); then a scalar tail, done
//         by the CTA that owns the buffer's first tile.
struct DigestEntry {
  const void *data;
  uint64_t n;
  uint64_t tile_begin;
  uint32_t key_base;
  uint8_t head;
  uint8_t dtype;        // 0 fp32, 1 bf16
  uint8_t slot;
  uint8_t pad_;
};

template <int MAXE>
struct DigestPlan {
  uint64_t total_tiles;
  uint32_t count;
  uint32_t one;          // 1: the FMA-pipe carry-add multiplier of the digest
  DigestEntry e[MAXE];
};

constexpr int kDigestSmall = 16;
constexpr int kDigestLarge = 1000;
static_assert(sizeof(DigestEntry) == 32, "entry layout");
static_assert(sizeof(DigestPlan<kDigestLarge>) <= 32764, "kernel parameter limit");

// One segment of the upload kernel (48 bytes).  Where dst and src are
// mutually 16-byte aligned, the `body` bytes from dst + head on are copied
// in 16-byte words, in tiles of kUploadTile bytes; the head (fewer than 16
// bytes before dst's 16-byte boundary) and the tail (body end to `bytes`)
// are "scalar items", copied byte by byte after the tiles.  Mutually
// misaligned segments have body = 0 and head = bytes.
struct UploadEntry {
  uint8_t *dst;
  const uint8_t *src;   // device-side address of the source
  uint64_t bytes;
  uint64_t body;
  uint64_t tile_begin;   // first tile of the segment (prefix over the launch)
  uint64_t scalar_begin;  // first scalar item of the segment
};
// head = bytes before dst's 16-byte boundary, derived on the device:
// (16 - dst % 16) % 16 when body > 0.

template <int MAXE>
struct UploadPlan {
  uint64_t total_tiles;
  uint64_t total_scalar;
  uint32_t count;
  uint32_t pad_;
  UploadEntry e[MAXE];
};

#ifndef APC_UPLOAD_THREADS
#define APC_UPLOAD_THREADS 512
#endif
#ifndef APC_UPLOAD_UNROLL
#define APC_UPLOAD_UNROLL 8
#endif
constexpr int kUploadThreads = APC_UPLOAD_THREADS;
constexpr int kUploadUnroll = APC_UPLOAD_UNROLL;                                       // 16-byte words per thread per tile
constexpr uint64_t kUploadTile = (uint64_t)kUploadThreads * kUploadUnroll * 16;      // 64 KB
constexpr int kUploadMax = 600;
static_assert(sizeof(UploadEntry) == 48, "entry layout");
static_assert(sizeof(UploadPlan<kUploadMax>) <= 32764, "kernel parameter limit");

// Upload kernel (apc_upload.cu): the plan's segments, on `grid` CTAs.
int launch_upload(const UploadPlan<kUploadMax> &plan, unsigned grid, void *stream);

// Launch wrappers (apc_commit.cu, apc_digest.cu).  They return a cudaError_t
// value and launch on `stream` with `grid` CTAs.
int launch_commit_small(const CommitPlan<kCommitSmall> &plan, int layout, bool zero_grad, unsigned grid,
                        void *stream, unsigned long long *out);
int launch_commit_large(const CommitPlan<kCommitLarge> &plan, int layout, bool zero_grad, unsigned grid,
                        void *stream, unsigned long long *out);
int launch_digest_small(const DigestPlan<kDigestSmall> &plan, unsigned grid, void *stream,
                        unsigned long long *out);
int launch_digest_large(const DigestPlan<kDigestLarge> &plan, unsigned grid, void *stream,
                        unsigned long long *out);

// Resident CTAs per SM of each kernel (cudaOccupancyMaxActiveBlocksPerMultiprocessor).
int commit_blocks_per_sm(bool large, int *out);
int digest_blocks_per_sm(bool large, int *out);

// Count kernel (apc_guard.cu): per-slot counts of nonzero words over the
// same buffer plans as the digest.
int launch_count_small(const DigestPlan<kDigestSmall> &plan, unsigned grid, void *stream, unsigned long long *out);
int launch_count_large(const DigestPlan<kDigestLarge> &plan, unsigned grid, void *stream, unsigned long long *out);
int count_blocks_per_sm(bool large, int *out);

// Device status word of the kernels of one translation unit on the current
// device: nonzero after a bounded wait gave up.  read_* copies it to the host
// (synchronously) and clears it.
int read_commit_status(unsigned *out);
// Self-test of the bounded wait: one thread waits on an mbarrier that nothing
// completes, gives up after limit_ns and records APC_ETIMEOUT.
int launch_wait_timeout(uint64_t limit_ns, void *stream);

}  // namespace apc
