// The fused committed-step kernel: AdamW over a chunk table of ragged
// tensors, the bf16 working copy, and the four state digests, in one pass.
//
// Work decomposition.  Each table entry's vector body is cut into tiles of
// kCommitTile = 4096 elements; a persistent grid (a multiple of the SM count)
// walks the launch's tile space with a grid stride, so every CTA streams
// through many tiles and the table is read from the kernel's parameter block.
// A thread handles kCommitUnroll 8-element vectors per tile: two 16-byte
// loads per fp32 buffer and one 16-byte bf16 load of the gradient, issued
// for all vectors before any arithmetic so that the loads overlap.  The
// scalar head and tail of an entry (fewer than 8 elements each) are done by
// the CTA that owns the entry's first tile; entries whose buffers are not
// mutually 16-byte aligned run element-wise.
//
// Digest reduction.  Each thread folds its elements into four 64-bit
// wrapping sums in registers; at exit the CTA reduces them with warp
// shuffles and shared memory and adds one value per digest into the
// caller's output with a 64-bit atomic.  Addition mod 2^64 is associative
// and commutative, so the digests do not depend on the grid, the tile
// order or the table split.
#include <cuda_runtime.h>

#include "apc_device.cuh"
#include "apc_internal.h"

namespace apc {
namespace {

struct Acc {
  uint64_t p, m, v, w;
};

struct Vec8 {
  float4 p0, p1, m0, m1, v0, v1;
  uint4 g;
};

__device__ __forceinline__ void commit_one(const CommitEntry &E, uint64_t i, const Scalars &s, Acc &a) {
  float p = E.p[i], m = E.m[i], v = E.v[i];
  const uint32_t w = adamw_element(p, m, v, (uint32_t)E.g[i], s);
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

__device__ __forceinline__ void load8(const CommitEntry &E, uint64_t i, Vec8 &x) {
  const float4 *p = reinterpret_cast<const float4 *>(E.p + i);
  const float4 *m = reinterpret_cast<const float4 *>(E.m + i);
  const float4 *v = reinterpret_cast<const float4 *>(E.v + i);
  x.p0 = __ldcs(p);
  x.p1 = __ldcs(p + 1);
  x.m0 = __ldcs(m);
  x.m1 = __ldcs(m + 1);
  x.v0 = __ldcs(v);
  x.v1 = __ldcs(v + 1);
  x.g = __ldcs(reinterpret_cast<const uint4 *>(E.g + i));
}

__device__ __forceinline__ void compute_store8(const CommitEntry &E, uint64_t i, const Vec8 &x, const Scalars &s,
                                               Acc &a) {
  float p[8] = {x.p0.x, x.p0.y, x.p0.z, x.p0.w, x.p1.x, x.p1.y, x.p1.z, x.p1.w};
  float m[8] = {x.m0.x, x.m0.y, x.m0.z, x.m0.w, x.m1.x, x.m1.y, x.m1.z, x.m1.w};
  float v[8] = {x.v0.x, x.v0.y, x.v0.z, x.v0.w, x.v1.x, x.v1.y, x.v1.z, x.v1.w};
  const uint32_t gw[4] = {x.g.x, x.g.y, x.g.z, x.g.w};
  uint32_t w[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const uint32_t g16 = (j & 1) ? (gw[j >> 1] >> 16) : (gw[j >> 1] & 0xFFFFu);
    w[j] = adamw_element(p[j], m[j], v[j], g16, s);
  }
  float4 *pp = reinterpret_cast<float4 *>(E.p + i);
  float4 *mp = reinterpret_cast<float4 *>(E.m + i);
  float4 *vp = reinterpret_cast<float4 *>(E.v + i);
  __stcs(pp, make_float4(p[0], p[1], p[2], p[3]));
  __stcs(pp + 1, make_float4(p[4], p[5], p[6], p[7]));
  __stcs(mp, make_float4(m[0], m[1], m[2], m[3]));
  __stcs(mp + 1, make_float4(m[4], m[5], m[6], m[7]));
  __stcs(vp, make_float4(v[0], v[1], v[2], v[3]));
  __stcs(vp + 1, make_float4(v[4], v[5], v[6], v[7]));
  __stcs(reinterpret_cast<uint4 *>(E.w + i),
         make_uint4(w[0] | (w[1] << 16), w[2] | (w[3] << 16), w[4] | (w[5] << 16), w[6] | (w[7] << 16)));
  const uint32_t G = E.key_base + (uint32_t)i;
#pragma unroll
  for (int j = 0; j < 8; j += 2) {
    a.p += digest_term(G + j, __float_as_uint(p[j])) + digest_term(G + j + 1, __float_as_uint(p[j + 1]));
    a.m += digest_term(G + j, __float_as_uint(m[j])) + digest_term(G + j + 1, __float_as_uint(m[j + 1]));
    a.v += digest_term(G + j, __float_as_uint(v[j])) + digest_term(G + j + 1, __float_as_uint(v[j + 1]));
    a.w += digest_term(G + j, w[j]) + digest_term(G + j + 1, w[j + 1]);
  }
}

template <int MAXE>
__global__ void __launch_bounds__(kThreads) commit_kernel(const __grid_constant__ CommitPlan<MAXE> plan,
                                                          unsigned long long *out) {
  __shared__ uint64_t red[kThreads / 32];
  const Scalars s = load_scalars(plan.h);
  Acc a{0, 0, 0, 0};
  uint32_t cur = 0;
  for (uint64_t tile = blockIdx.x; tile < plan.total_tiles; tile += gridDim.x) {
    while (cur + 1 < plan.count && tile >= plan.e[cur + 1].tile_begin) ++cur;
    const CommitEntry &E = plan.e[cur];
    const uint64_t local = tile - E.tile_begin;
    if (E.head != kScalarMode) {
      const uint64_t head = E.head;
      const uint64_t vec_end = head + ((E.n - head) & ~(uint64_t)(kVec - 1));
      const uint64_t base = head + local * kCommitTile;
      Vec8 x[kCommitUnroll];
      bool ok[kCommitUnroll];
#pragma unroll
      for (int u = 0; u < kCommitUnroll; ++u) {
        const uint64_t i = base + (uint64_t)(u * kThreads + threadIdx.x) * kVec;
        ok[u] = i < vec_end;
        if (ok[u]) load8(E, i, x[u]);
      }
#pragma unroll
      for (int u = 0; u < kCommitUnroll; ++u) {
        const uint64_t i = base + (uint64_t)(u * kThreads + threadIdx.x) * kVec;
        if (ok[u]) compute_store8(E, i, x[u], s, a);
      }
      if (local == 0) {
        const uint32_t t = threadIdx.x;
        if (t < head) commit_one(E, t, s, a);
        if (t >= 32 && t - 32 < E.n - vec_end) commit_one(E, vec_end + (t - 32), s, a);
      }
    } else {
      const uint64_t base = local * kCommitTile;
#pragma unroll 4
      for (int k = 0; k < kVec * kCommitUnroll; ++k) {
        const uint64_t i = base + (uint64_t)k * kThreads + threadIdx.x;
        if (i < E.n) commit_one(E, i, s, a);
      }
    }
  }
  uint64_t r;
  r = cta_sum<kThreads>(a.p, red);
  if (threadIdx.x == 0 && r) atomicAdd(&out[0], (unsigned long long)r);
  r = cta_sum<kThreads>(a.m, red);
  if (threadIdx.x == 0 && r) atomicAdd(&out[1], (unsigned long long)r);
  r = cta_sum<kThreads>(a.v, red);
  if (threadIdx.x == 0 && r) atomicAdd(&out[2], (unsigned long long)r);
  r = cta_sum<kThreads>(a.w, red);
  if (threadIdx.x == 0 && r) atomicAdd(&out[3], (unsigned long long)r);
}

}  // namespace

int launch_commit_small(const CommitPlan<kCommitSmall> &plan, unsigned grid, void *stream,
                        unsigned long long *out) {
  commit_kernel<kCommitSmall><<<grid, kThreads, 0, (cudaStream_t)stream>>>(plan, out);
  return (int)cudaGetLastError();
}

int launch_commit_large(const CommitPlan<kCommitLarge> &plan, unsigned grid, void *stream,
                        unsigned long long *out) {
  commit_kernel<kCommitLarge><<<grid, kThreads, 0, (cudaStream_t)stream>>>(plan, out);
  return (int)cudaGetLastError();
}

int commit_blocks_per_sm(bool large, int *out) {
  cudaError_t e = large ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, commit_kernel<kCommitLarge>, kThreads, 0)
                        : cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, commit_kernel<kCommitSmall>, kThreads, 0);
  return (int)e;
}

}  // namespace apc
