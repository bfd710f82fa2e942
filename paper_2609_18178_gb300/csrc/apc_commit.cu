// The fused committed-step kernel: AdamW over a chunk table of ragged
// tensors, the bf16 working copy, and the four state digests, in one pass
// over HBM (28 bytes per element: p, m, v read and written, g read, w written).
//
// Warp-specialized pipeline (one persistent CTA per SM by default):
//  * The producer warp walks the launch's tiles (kCommitTile = 4864 elements
//    of one entry's 16-byte aligned body) and, for each, waits until a ring
//    stage is free and issues four bulk asynchronous copies -- p, m, v (19 KB
//    each) and g (9.5 KB) -- that complete on the stage's "full" mbarrier.
//    Loads never occupy consumer registers, and up to kCommitStages tiles
//    per CTA are in flight.
//  * The consumer warps (19 by default) wait for a stage, read their
//    elements from shared memory (thread t of C takes elements 4t..4t+3 and
//    4C+4t..4C+4t+3, so both the shared-memory reads and the global stores
//    are contiguous across the warp), release the stage to the producer, then
//    apply AdamW, store
//    p', m', v' and the bf16 copy with 16- and 8-byte streaming stores, and
//    fold the four digest terms into 64-bit registers.
//  * Elements outside the aligned bodies (entry heads and tails under 8
//    elements, and entries whose five buffers are not mutually 16-byte
//    aligned) are "scalar items", done afterwards by the consumers with a
//    grid-stride loop straight from global memory.
//  * At exit the CTA sums each digest (warp shuffles, shared memory) and adds
//    it into the caller's output with one 64-bit atomic; addition mod 2^64 is
//    order-free, so digests do not depend on grid size or table split.
//
// Every mbarrier wait is bounded (apc_tma.cuh).  A wait that gives up sets
// the translation unit's device status word, makes the CTA stop issuing and
// consuming, drains the copies already issued (bounded again) and returns.
#include <cuda_runtime.h>

#include "../../include/apc.h"
#include "apc_device.cuh"
#include "apc_internal.h"
#include "apc_tma.cuh"

namespace apc {
namespace {

__device__ unsigned int g_commit_status;

struct Acc {
  uint64_t p, m, v, w;
};

__device__ __forceinline__ uint64_t umin64(uint64_t a, uint64_t b) { return a < b ? a : b; }

__device__ __forceinline__ void fail_wait(int *abort_flag) {
  atomicOr(&g_commit_status, (unsigned)APC_ETIMEOUT);
  *(volatile int *)abort_flag = 1;
}

template <bool ZERO>
__device__ __forceinline__ void commit_one(const CommitEntry &E, uint64_t i, const Scalars &s, Acc &a) {
  float p = E.p[i], m = E.m[i], v = E.v[i];
  const uint32_t w = adamw_element(p, m, v, (uint32_t)E.g[i], s);
  if (ZERO) const_cast<uint16_t *>(E.g)[i] = 0;
  E.p[i] = p;
  E.m[i] = m;
  E.v[i] = v;
  E.w[i] = (uint16_t)w;
  const uint32_t G = E.key_base + (uint32_t)i;
  a.p += digest_term(G, __float_as_uint(p));
  a.m += digest_term(G, __float_as_uint(m));
  a.v += digest_term(G, __float_as_uint(v));
  a.w += digest_term(G, w);
}

// Four consecutive elements from shared memory, updated and stored at p, m,
// v, w (the element's addresses in the entry); G is its digest index.
__device__ __forceinline__ void commit_group(float *pp, float *mp, float *vp, uint16_t *wp, uint32_t G, float4 P,
                                             float4 M, float4 V, uint2 g2, const Scalars &s, Acc &a) {
  float p[4] = {P.x, P.y, P.z, P.w};
  float m[4] = {M.x, M.y, M.z, M.w};
  float v[4] = {V.x, V.y, V.z, V.w};
  const uint32_t gw[4] = {g2.x & 0xFFFFu, g2.x >> 16, g2.y & 0xFFFFu, g2.y >> 16};
  uint32_t w[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) w[j] = adamw_element(p[j], m[j], v[j], gw[j], s);
  __stcs(reinterpret_cast<float4 *>(pp), make_float4(p[0], p[1], p[2], p[3]));
  __stcs(reinterpret_cast<float4 *>(mp), make_float4(m[0], m[1], m[2], m[3]));
  __stcs(reinterpret_cast<float4 *>(vp), make_float4(v[0], v[1], v[2], v[3]));
  __stcs(reinterpret_cast<uint2 *>(wp), make_uint2(w[0] | (w[1] << 16), w[2] | (w[3] << 16)));
  a.p += digest_term(G, __float_as_uint(p[0])) + digest_term(G + 1, __float_as_uint(p[1]));
  a.p += digest_term(G + 2, __float_as_uint(p[2])) + digest_term(G + 3, __float_as_uint(p[3]));
  a.m += digest_term(G, __float_as_uint(m[0])) + digest_term(G + 1, __float_as_uint(m[1]));
  a.m += digest_term(G + 2, __float_as_uint(m[2])) + digest_term(G + 3, __float_as_uint(m[3]));
  a.v += digest_term(G, __float_as_uint(v[0])) + digest_term(G + 1, __float_as_uint(v[1]));
  a.v += digest_term(G + 2, __float_as_uint(v[2])) + digest_term(G + 3, __float_as_uint(v[3]));
  a.w += digest_term(G, w[0]) + digest_term(G + 1, w[1]);
  a.w += digest_term(G + 2, w[2]) + digest_term(G + 3, w[3]);
}

struct Stage {
  float *p, *m, *v;
  uint16_t *g;
};

__device__ __forceinline__ Stage stage_at(uint8_t *smem, int s) {
  uint8_t *b = smem + (size_t)s * kCommitStageBytes;
  Stage st;
  st.p = reinterpret_cast<float *>(b);
  st.m = reinterpret_cast<float *>(b + 4 * kCommitTile);
  st.v = reinterpret_cast<float *>(b + 8 * kCommitTile);
  st.g = reinterpret_cast<uint16_t *>(b + 12 * kCommitTile);
  return st;
}

template <int MAXE>
__device__ __forceinline__ uint32_t find_tile(const CommitPlan<MAXE> &plan, uint32_t cur, uint64_t tile) {
  while (cur + 1 < plan.count && tile >= plan.e[cur + 1].tile_begin) ++cur;
  return cur;
}

template <int MAXE, bool ZERO>
__global__ void __launch_bounds__(kCommitThreads, kCommitBlocksPerSm)
    commit_kernel(const __grid_constant__ CommitPlan<MAXE> plan, unsigned long long *out) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ __align__(8) uint64_t full[kCommitStages];
  __shared__ __align__(8) uint64_t empty[kCommitStages];
  __shared__ uint64_t red[kCommitThreads / 32];
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kCommitStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kCommitConsumerWarps);
    }
    abort_flag = 0;
    mbar_init_fence();
  }
  __syncthreads();

  Acc a{0, 0, 0, 0};
  if (warp == kCommitConsumerWarps) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t policy = l2_evict_first();
      uint32_t cur = 0, phase = 0;
      int stage = 0;
      uint64_t issued = 0;
      for (uint64_t tile = blockIdx.x; tile < plan.total_tiles; tile += gridDim.x) {
        if (*(volatile int *)&abort_flag) break;
        cur = find_tile(plan, cur, tile);
        const CommitEntry &E = plan.e[cur];
        const uint64_t start = E.head + (tile - E.tile_begin) * kCommitTile;
        const uint64_t vec_end = E.head + ((E.n - E.head) & ~(uint64_t)7);
        const uint32_t cnt = (uint32_t)umin64(kCommitTile, vec_end - start);
        if (!mbar_wait(&empty[stage], phase ^ 1)) {
          fail_wait(&abort_flag);
          break;
        }
        const Stage st = stage_at(smem, stage);
        mbar_arrive_expect_tx(&full[stage], cnt * 14);
        bulk_g2s(st.p, E.p + start, cnt * 4, &full[stage], policy);
        bulk_g2s(st.m, E.m + start, cnt * 4, &full[stage], policy);
        bulk_g2s(st.v, E.v + start, cnt * 4, &full[stage], policy);
        bulk_g2s(st.g, E.g + start, cnt * 2, &full[stage], policy);
        ++issued;
        if (++stage == kCommitStages) {
          stage = 0;
          phase ^= 1;
        }
      }
      // Drain: the last min(issued, stages) copies must have landed before
      // the CTA may exit (normally the consumers already waited for them).
      const int n_drain = (int)umin64(issued, (uint64_t)kCommitStages);
      for (int k = 0; k < n_drain; ++k) {
        if (--stage < 0) {
          stage = kCommitStages - 1;
          phase ^= 1;
        }
        if (!mbar_wait(&full[stage], phase)) atomicOr(&g_commit_status, (unsigned)APC_ETIMEOUT);
      }
    }
    __syncwarp();
  } else {
    // ----------------------------------------------------------- consumers
    const Scalars s{plan.h};
    const int ct = threadIdx.x;  // 0..255
    uint32_t cur = 0, phase = 0;
    int stage = 0;
    for (uint64_t tile = blockIdx.x; tile < plan.total_tiles; tile += gridDim.x) {
      cur = find_tile(plan, cur, tile);
      const CommitEntry &E = plan.e[cur];
      const uint64_t start = E.head + (tile - E.tile_begin) * kCommitTile;
      const uint64_t vec_end = E.head + ((E.n - E.head) & ~(uint64_t)7);
      const uint32_t cnt = (uint32_t)umin64(kCommitTile, vec_end - start);
      if (!mbar_wait(&full[stage], phase)) {
        fail_wait(&abort_flag);
        break;
      }
      if (*(volatile int *)&abort_flag) break;
      const Stage st = stage_at(smem, stage);
      float4 P[kCommitGroups], M[kCommitGroups], V[kCommitGroups];
      uint2 G[kCommitGroups];
      bool ok[kCommitGroups];
#pragma unroll
      for (int k = 0; k < kCommitGroups; ++k) {
        const uint32_t e = (uint32_t)(k * kCommitConsumers + ct) * 4;
        ok[k] = e < cnt;
        if (ok[k]) {
          P[k] = *reinterpret_cast<const float4 *>(st.p + e);
          M[k] = *reinterpret_cast<const float4 *>(st.m + e);
          V[k] = *reinterpret_cast<const float4 *>(st.v + e);
          G[k] = *reinterpret_cast<const uint2 *>(st.g + e);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[stage]);
      // the entry's fields once per tile, in registers
      float *const pp = E.p + start, *const mp = E.m + start, *const vp = E.v + start;
      uint16_t *const wp = E.w + start;
      const uint32_t G0 = E.key_base + (uint32_t)start;
#pragma unroll
      for (int k = 0; k < kCommitGroups; ++k) {
        const uint32_t e = (uint32_t)(k * kCommitConsumers + ct) * 4;
        if (ok[k]) {
          if (ZERO) __stcs(reinterpret_cast<uint2 *>(const_cast<uint16_t *>(E.g) + start + e), make_uint2(0u, 0u));
          commit_group(pp + e, mp + e, vp + e, wp + e, G0 + e, P[k], M[k], V[k], G[k], s, a);
        }
      }
      if (++stage == kCommitStages) {
        stage = 0;
        phase ^= 1;
      }
    }
    // scalar items: entry heads and tails, and entries without vectors
    if (!*(volatile int *)&abort_flag) {
      cur = 0;
      for (uint64_t it = (uint64_t)blockIdx.x * kCommitConsumers + ct; it < plan.total_scalar;
           it += (uint64_t)gridDim.x * kCommitConsumers) {
        while (cur + 1 < plan.count && it >= plan.e[cur + 1].scalar_begin) ++cur;
        const CommitEntry &E = plan.e[cur];
        const uint64_t k = it - E.scalar_begin;
        uint64_t i;
        if (E.head == kScalarMode) {
          i = k;
        } else {
          const uint64_t vec_end = E.head + ((E.n - E.head) & ~(uint64_t)7);
          i = k < E.head ? k : vec_end + (k - E.head);
        }
        commit_one<ZERO>(E, i, s, a);
      }
    }
  }

  const bool ok = !*(volatile int *)&abort_flag;
  uint64_t r;
  r = cta_sum<kCommitThreads>(a.p, red);
  if (threadIdx.x == 0 && ok && r) atomicAdd(&out[0], (unsigned long long)r);
  r = cta_sum<kCommitThreads>(a.m, red);
  if (threadIdx.x == 0 && ok && r) atomicAdd(&out[1], (unsigned long long)r);
  r = cta_sum<kCommitThreads>(a.v, red);
  if (threadIdx.x == 0 && ok && r) atomicAdd(&out[2], (unsigned long long)r);
  r = cta_sum<kCommitThreads>(a.w, red);
  if (threadIdx.x == 0 && ok && r) atomicAdd(&out[3], (unsigned long long)r);
}

// One thread waits on an mbarrier that nothing completes: the bounded wait
// must give up after `limit_ns` and record APC_ETIMEOUT.
__global__ void wait_timeout_kernel(uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  mbar_init(&bar, 1);
  mbar_init_fence();
  if (!mbar_wait(&bar, 0, limit_ns)) atomicOr(&g_commit_status, (unsigned)APC_ETIMEOUT);
}

template <int MAXE, bool ZERO>
int launch_t(const CommitPlan<MAXE> &plan, unsigned grid, void *stream, unsigned long long *out) {
  cudaError_t e = cudaFuncSetAttribute(commit_kernel<MAXE, ZERO>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kCommitSmemBytes);
  if (e != cudaSuccess) return (int)e;
  commit_kernel<MAXE, ZERO><<<grid, kCommitThreads, kCommitSmemBytes, (cudaStream_t)stream>>>(plan, out);
  return (int)cudaGetLastError();
}

template <int MAXE>
int launch(const CommitPlan<MAXE> &plan, bool zero_grad, unsigned grid, void *stream, unsigned long long *out) {
  return zero_grad ? launch_t<MAXE, true>(plan, grid, stream, out) : launch_t<MAXE, false>(plan, grid, stream, out);
}

template <int MAXE>
int blocks_per_sm(int *out) {
  cudaError_t e = cudaFuncSetAttribute(commit_kernel<MAXE, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kCommitSmemBytes);
  if (e != cudaSuccess) return (int)e;
  return (int)cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, commit_kernel<MAXE, false>, kCommitThreads,
                                                            kCommitSmemBytes);
}

}  // namespace

int launch_commit_small(const CommitPlan<kCommitSmall> &plan, bool zero_grad, unsigned grid, void *stream,
                        unsigned long long *out) {
  return launch(plan, zero_grad, grid, stream, out);
}

int launch_commit_large(const CommitPlan<kCommitLarge> &plan, bool zero_grad, unsigned grid, void *stream,
                        unsigned long long *out) {
  return launch(plan, zero_grad, grid, stream, out);
}

int commit_blocks_per_sm(bool large, int *out) {
  return large ? blocks_per_sm<kCommitLarge>(out) : blocks_per_sm<kCommitSmall>(out);
}

int launch_wait_timeout(uint64_t limit_ns, void *stream) {
  wait_timeout_kernel<<<1, 1, 0, (cudaStream_t)stream>>>(limit_ns);
  return (int)cudaGetLastError();
}

int read_commit_status(unsigned *out) {
  cudaError_t e = cudaMemcpyFromSymbol(out, g_commit_status, sizeof(unsigned));
  if (e != cudaSuccess) return (int)e;
  const unsigned zero = 0;
  return (int)cudaMemcpyToSymbol(g_commit_status, &zero, sizeof(unsigned));
}

}  // namespace apc
