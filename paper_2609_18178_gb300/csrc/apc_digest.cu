// The read-only state digest over a list of buffers (the verification pass
// after recovery): 4 (fp32) or 2 (bf16) bytes read per element and one
// splitmix64 term per element, so the pass is bound by integer issue, not by
// HBM.
//
// Work split: each buffer's 16-byte aligned body is cut into tiles of
// kDigestTile elements, and each CTA of a persistent grid takes one
// contiguous run of the launch's tile space (the runs differ by at most one
// tile).  Inside its run a CTA finds the buffer of its first tile once, then
// moves to the next buffer only when it crosses one, carrying the element
// offset and key forward by a tile per step; this costs measurably fewer
// integer instructions per tile than striding over the tile space with a
// grid-wide step, which looks the buffer up and rebuilds the offsets for
// every tile.
//
// Loads: a thread's part of a tile is kDigestUnroll vectors of 8 words.  All
// tiles of a buffer but its last are full; they run without per-vector bounds
// checks, and each thread keeps its next full tile in flight with cp.async
// into shared-memory slots that only it reads (two stages, no barrier), then
// folds the current one from there.  A buffer's last tile is loaded straight
// into registers with per-vector checks, and its scalar head and tail go to
// the CTA that owns its first tile.  (A CTA-wide bulk-copy pipeline like the
// commit kernel's measured slower here: its per-tile synchronisation costs
// issue slots, the one resource this pass is short of.)
//
// A thread keeps one running 64-bit sum for the slot of the buffer it is in;
// all threads of a CTA visit the same tiles, so slot changes are CTA-uniform
// and the running sum is flushed (warp shuffle reduce, then a shared-memory
// atomic) only when the CTA moves to a buffer of another slot and at exit.
#include <cuda_runtime.h>

#include <atomic>

#include "../../include/apc.h"
#include "apc_device.cuh"
#include "apc_internal.h"

namespace apc {
namespace {

// One digest term of this pass.  The pass is bound by the integer ALU, not
// by issue, and runs faster with the compiler's own 64-bit multiply.
template <uint32_t K>
__device__ __forceinline__ uint64_t term(uint32_t gidx, uint32_t bits, uint32_t one) {
  return digest_term<K, MulCompiler>(gidx, bits, one);
}

// The same with SHARED: the caller has checked that all of a thread's terms
// in the tile share the top two bits of the incremented key high word
// (top_bits_shared over the keys G0 .. G0 + (kDigestUnroll - 1) * kThreads *
// kVec + 7) and passes them as `top`, so no term computes hi >> 30 itself.
template <uint32_t K, bool SHARED>
__device__ __forceinline__ uint64_t vterm(uint32_t gidx, uint32_t bits, uint32_t one, uint32_t top) {
  if constexpr (SHARED) return digest_term<K, MulCompiler>(gidx, bits, one, top);
  else return digest_term<K, MulCompiler>(gidx, bits, one);
}

// A thread's terms of one fp32 tile (kDigestUnroll vectors of 8 words).
template <bool SHARED>
__device__ __forceinline__ void fold32(const uint4 (&x)[kDigestUnroll][2], const bool (&ok)[kDigestUnroll], uint32_t G0,
                                       uint32_t one, uint32_t top, uint64_t &t0, uint64_t &t1) {
#pragma unroll
  for (int u = 0; u < kDigestUnroll; ++u) {
    if (!ok[u]) continue;
    const uint32_t G = G0 + (uint32_t)(u * kThreads * kVec);
    t0 += vterm<0, SHARED>(G, x[u][0].x, one, top) + vterm<1, SHARED>(G, x[u][0].y, one, top);
    t1 += vterm<2, SHARED>(G, x[u][0].z, one, top) + vterm<3, SHARED>(G, x[u][0].w, one, top);
    t0 += vterm<4, SHARED>(G, x[u][1].x, one, top) + vterm<5, SHARED>(G, x[u][1].y, one, top);
    t1 += vterm<6, SHARED>(G, x[u][1].z, one, top) + vterm<7, SHARED>(G, x[u][1].w, one, top);
  }
}

// A bf16 word's term: with the shared top bits, the 16-bit form of
// digest_term_u16 (its increment and first xor-shift take two ALU
// instructions instead of four).
template <uint32_t K, bool SHARED>
__device__ __forceinline__ uint64_t hterm(uint32_t gidx, uint32_t bits, uint32_t one, uint32_t top) {
  if constexpr (SHARED) return digest_term_u16<K, MulCompiler>(gidx, bits, one, top);
  else return digest_term<K, MulCompiler>(gidx, bits, one);
}

// A thread's terms of one bf16 tile (kDigestUnroll vectors of 8 words).
template <bool SHARED>
__device__ __forceinline__ void fold16(const uint4 (&x)[kDigestUnroll], const bool (&ok)[kDigestUnroll], uint32_t G0,
                                       uint32_t one, uint32_t top, uint64_t &t0, uint64_t &t1) {
#pragma unroll
  for (int u = 0; u < kDigestUnroll; ++u) {
    if (!ok[u]) continue;
    const uint32_t G = G0 + (uint32_t)(u * kThreads * kVec);
    t0 += hterm<0, SHARED>(G, x[u].x & 0xFFFFu, one, top) + hterm<1, SHARED>(G, x[u].x >> 16, one, top);
    t1 += hterm<2, SHARED>(G, x[u].y & 0xFFFFu, one, top) + hterm<3, SHARED>(G, x[u].y >> 16, one, top);
    t0 += hterm<4, SHARED>(G, x[u].z & 0xFFFFu, one, top) + hterm<5, SHARED>(G, x[u].z >> 16, one, top);
    t1 += hterm<6, SHARED>(G, x[u].w & 0xFFFFu, one, top) + hterm<7, SHARED>(G, x[u].w >> 16, one, top);
  }
}

// The keys of a thread's terms in a tile lie in [G0, G0 + kTileKeySpan - 1];
// with the increment's carry their high words lie in [B, B + kTileKeySpan].
constexpr uint32_t kTileKeySpan = (kDigestUnroll - 1) * kThreads * kVec + kVec;

// One tile of a thread's words: kDigestUnroll vectors of 8, the first at q
// (element `base` of the buffer), the others kThreads vectors apart.  Only
// the vectors with ok[u] are loaded and folded.
__device__ __forceinline__ void tile32(const uint4 *q, const bool (&ok)[kDigestUnroll], uint32_t G0, uint32_t one,
                                       uint64_t &t0, uint64_t &t1) {
  uint4 x[kDigestUnroll][2];
#pragma unroll
  for (int u = 0; u < kDigestUnroll; ++u) {
    if (ok[u]) {
      x[u][0] = __ldcs(q + 2 * u * kThreads);
      x[u][1] = __ldcs(q + 2 * u * kThreads + 1);
    }
  }
  const uint32_t B = G0 + 0x9E3779B9u;
  if (top_bits_shared(B, kTileKeySpan)) fold32<true>(x, ok, G0, one, B >> 30, t0, t1);
  else fold32<false>(x, ok, G0, one, 0, t0, t1);
}

__device__ __forceinline__ void tile16(const uint4 *q, const bool (&ok)[kDigestUnroll], uint32_t G0, uint32_t one,
                                       uint64_t &t0, uint64_t &t1) {
  uint4 x[kDigestUnroll];
#pragma unroll
  for (int u = 0; u < kDigestUnroll; ++u) {
    if (ok[u]) x[u] = __ldcs(q + u * kThreads);
  }
  const uint32_t B = G0 + 0x9E3779B9u;
  if (top_bits_shared(B, kTileKeySpan)) fold16<true>(x, ok, G0, one, B >> 30, t0, t1);
  else fold16<false>(x, ok, G0, one, 0, t0, t1);
}

// Which of a thread's vectors in an entry's last tile lie in its body.
__device__ __forceinline__ void last_tile_ok(uint64_t base, uint64_t vec_end, bool (&ok)[kDigestUnroll]) {
#pragma unroll
  for (int u = 0; u < kDigestUnroll; ++u) ok[u] = base + (uint64_t)(u * kThreads) * kVec < vec_end;
}

// Per-thread double buffering of full tiles in shared memory: while a thread
// folds one tile it has the next one in flight with cp.async, into slots that
// only it reads, so no barrier is needed; cp.async.wait_group orders each
// thread's own copies.  Slot k of stage b of thread t is
// stg[(b * kStageSlots + k) * kThreads + t]: a warp's 16-byte reads of one
// slot are contiguous.
constexpr int kStageSlots = 2 * kDigestUnroll;                       // 16-byte words per thread per stage
constexpr uint32_t kStageBytes = 2u * kStageSlots * kThreads * 16u;  // two stages: 131,072 bytes
constexpr uint32_t kLaunchSmem = kStageBytes + APC_DIGEST_EXTRA_SMEM;

__device__ __forceinline__ void cp16(uint32_t dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_wait_all_but_newest() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }

__device__ __forceinline__ void flush(uint64_t &acc, int slot, unsigned long long *s_acc) {
  uint64_t x = acc;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
  if ((threadIdx.x & 31) == 0 && slot >= 0 && x) atomicAdd(&s_acc[slot], (unsigned long long)x);
  acc = 0;
}

__device__ __forceinline__ uint32_t word_at(const DigestEntry &E, uint64_t i) {
  return E.dtype == 0 ? reinterpret_cast<const uint32_t *>(E.data)[i]
                      : (uint32_t) reinterpret_cast<const uint16_t *>(E.data)[i];
}

// One CTA per SM (32 warps, 128 KB of stages), which caps the kernel at 64
// registers: a full tile's 16 terms per thread, without per-vector checks,
// form one block that the compiler schedules within them.
template <int MAXE>
__global__ void __launch_bounds__(kThreads, APC_DIGEST_MIN_BLOCKS) digest_kernel(const __grid_constant__ DigestPlan<MAXE> plan,
                                                          unsigned long long *out) {
  __shared__ unsigned long long s_acc[APC_MAX_SLOTS];
  extern __shared__ __align__(16) uint4 stg[];
  const uint32_t stg_t = (uint32_t)__cvta_generic_to_shared(stg + threadIdx.x);  // this thread's slot 0, stage 0
  if (threadIdx.x < APC_MAX_SLOTS) s_acc[threadIdx.x] = 0;
  __syncthreads();
  const uint32_t one = plan.one;
  int slot = -1;
  uint64_t acc = 0;
  // this CTA's contiguous run of the launch's tiles: [tile, t_end)
  const uint64_t per = plan.total_tiles / gridDim.x, rem = plan.total_tiles % gridDim.x;
  uint64_t tile = blockIdx.x * per + (blockIdx.x < rem ? blockIdx.x : rem);
  const uint64_t t_end = tile + per + (blockIdx.x < rem ? 1 : 0);
  uint32_t cur = 0;
  while (cur + 1 < plan.count && tile >= plan.e[cur + 1].tile_begin) ++cur;
  const uint64_t t8 = (uint64_t)threadIdx.x * kVec;
  for (; tile < t_end; ++cur) {
    const DigestEntry &E = plan.e[cur];
    const uint64_t stop_e = cur + 1 < plan.count ? plan.e[cur + 1].tile_begin : plan.total_tiles;
    const uint64_t stop = stop_e < t_end ? stop_e : t_end;
    if (tile >= stop) continue;
    if ((int)E.slot != slot) {
      flush(acc, slot, s_acc);
      slot = E.slot;
    }
    const uint64_t head = E.head;
    const uint64_t vec_end = head + ((E.n - head) & ~(uint64_t)(kVec - 1));
    uint64_t base = head + (tile - E.tile_begin) * kDigestTile + t8;   // this thread's first element
    uint32_t G0 = E.key_base + (uint32_t)base;
    const bool first = tile == E.tile_begin;
    uint64_t t0 = 0, t1 = 0;
    // Every tile of an entry but its last is full (all vectors of all threads
    // lie in the body) and runs without per-vector checks.
    const uint64_t full_end = stop_e - 1 < stop ? stop_e - 1 : stop;
    bool all[kDigestUnroll], ok[kDigestUnroll];
#pragma unroll
    for (int u = 0; u < kDigestUnroll; ++u) all[u] = true;
    if (E.dtype == 0) {
      const uint32_t *d = reinterpret_cast<const uint32_t *>(E.data);
      const uint4 *q = reinterpret_cast<const uint4 *>(d + base);
      if (tile < full_end) {
        uint32_t b = 0;
#pragma unroll
        for (int k = 0; k < kStageSlots; ++k) cp16(stg_t + k * kThreads * 16u, q + (k >> 1) * 2 * kThreads + (k & 1));
        cp_commit();
        for (; tile < full_end; ++tile, q += kDigestTile / 4, G0 += (uint32_t)kDigestTile) {
          if (tile + 1 < full_end) {
            const uint4 *n = q + kDigestTile / 4;
            const uint32_t dst = stg_t + (b ^ 1) * kStageSlots * kThreads * 16u;
#pragma unroll
            for (int k = 0; k < kStageSlots; ++k) cp16(dst + k * kThreads * 16u, n + (k >> 1) * 2 * kThreads + (k & 1));
          }
          cp_commit();
          cp_wait_all_but_newest();
          const uint4 *src = stg + b * kStageSlots * kThreads + threadIdx.x;
          uint4 x[kDigestUnroll][2];
#pragma unroll
          for (int u = 0; u < kDigestUnroll; ++u) {
            x[u][0] = src[(2 * u) * kThreads];
            x[u][1] = src[(2 * u + 1) * kThreads];
          }
          const uint32_t B = G0 + 0x9E3779B9u;
          if (top_bits_shared(B, kTileKeySpan)) fold32<true>(x, all, G0, one, B >> 30, t0, t1);
          else fold32<false>(x, all, G0, one, 0, t0, t1);
          b ^= 1;
        }
      }
      if (tile < stop) {  // the entry's last tile
        last_tile_ok((uint64_t)(reinterpret_cast<const uint32_t *>(q) - d), vec_end, ok);
        tile32(q, ok, G0, one, t0, t1);
        ++tile;
      }
    } else {
      const uint16_t *d = reinterpret_cast<const uint16_t *>(E.data);
      const uint4 *q = reinterpret_cast<const uint4 *>(d + base);
      if (tile < full_end) {
        uint32_t b = 0;
#pragma unroll
        for (int u = 0; u < kDigestUnroll; ++u) cp16(stg_t + u * kThreads * 16u, q + u * kThreads);
        cp_commit();
        for (; tile < full_end; ++tile, q += kDigestTile / 8, G0 += (uint32_t)kDigestTile) {
          if (tile + 1 < full_end) {
            const uint4 *n = q + kDigestTile / 8;
            const uint32_t dst = stg_t + (b ^ 1) * kStageSlots * kThreads * 16u;
#pragma unroll
            for (int u = 0; u < kDigestUnroll; ++u) cp16(dst + u * kThreads * 16u, n + u * kThreads);
          }
          cp_commit();
          cp_wait_all_but_newest();
          const uint4 *src = stg + b * kStageSlots * kThreads + threadIdx.x;
          uint4 x[kDigestUnroll];
#pragma unroll
          for (int u = 0; u < kDigestUnroll; ++u) x[u] = src[u * kThreads];
          const uint32_t B = G0 + 0x9E3779B9u;
          if (top_bits_shared(B, kTileKeySpan)) fold16<true>(x, all, G0, one, B >> 30, t0, t1);
          else fold16<false>(x, all, G0, one, 0, t0, t1);
          b ^= 1;
        }
      }
      if (tile < stop) {  // the entry's last tile
        last_tile_ok((uint64_t)(reinterpret_cast<const uint16_t *>(q) - d), vec_end, ok);
        tile16(q, ok, G0, one, t0, t1);
        ++tile;
      }
    }
    if (first) {   // the CTA that owns an entry's first tile also does its scalar head and tail
      const uint32_t t = threadIdx.x;
      if (t < head) { acc_add(t0, term<0>(E.key_base + t, word_at(E, t), one), one); }
      if (t >= 32 && t - 32 < E.n - vec_end) {
        const uint64_t i = vec_end + (t - 32);
        acc_add(t0, term<0>(E.key_base + (uint32_t)i, word_at(E, i), one), one);
      }
    }
    acc_add(acc, t0, one);
    acc_add(acc, t1, one);
  }
  flush(acc, slot, s_acc);
  __syncthreads();
  if (threadIdx.x < APC_MAX_SLOTS && s_acc[threadIdx.x]) atomicAdd(&out[threadIdx.x], s_acc[threadIdx.x]);
}

// The dynamic shared-memory limit of one instantiation, raised once per
// device (later launches, for example inside a stream capture, only enqueue).
template <int MAXE>
int ensure_stage_attribute() {
  static std::atomic<uint64_t> done_mask{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return (int)e;
  const uint64_t bit = dev < 64 ? (1ull << dev) : 0;
  if (bit && (done_mask.load(std::memory_order_acquire) & bit)) return 0;
  e = cudaFuncSetAttribute(digest_kernel<MAXE>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kLaunchSmem);
  if (e != cudaSuccess) return (int)e;
  if (APC_SMEM_CARVEOUT >= 0) {
    e = cudaFuncSetAttribute(digest_kernel<MAXE>, cudaFuncAttributePreferredSharedMemoryCarveout, APC_SMEM_CARVEOUT);
    if (e != cudaSuccess) return (int)e;
  }
  if (bit) done_mask.fetch_or(bit, std::memory_order_acq_rel);
  return 0;
}

template <int MAXE>
int launch_t(const DigestPlan<MAXE> &plan, unsigned grid, void *stream, unsigned long long *out) {
  int e = ensure_stage_attribute<MAXE>();
  if (e) return e;
  digest_kernel<MAXE><<<grid, kThreads, kLaunchSmem, (cudaStream_t)stream>>>(plan, out);
  return (int)cudaGetLastError();
}

template <int MAXE>
int blocks_t(int *out) {
  int e = ensure_stage_attribute<MAXE>();
  if (e) return e;
  return (int)cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, digest_kernel<MAXE>, kThreads, kLaunchSmem);
}

}  // namespace

int launch_digest_small(const DigestPlan<kDigestSmall> &plan, unsigned grid, void *stream,
                        unsigned long long *out) {
  return launch_t<kDigestSmall>(plan, grid, stream, out);
}

int launch_digest_large(const DigestPlan<kDigestLarge> &plan, unsigned grid, void *stream,
                        unsigned long long *out) {
  return launch_t<kDigestLarge>(plan, grid, stream, out);
}

int digest_blocks_per_sm(bool large, int *out) { return large ? blocks_t<kDigestLarge>(out) : blocks_t<kDigestSmall>(out); }

}  // namespace apc
