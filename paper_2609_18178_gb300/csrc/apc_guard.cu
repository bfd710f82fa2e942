// The quiescence guard: per-slot counts of nonzero words over a list of
// buffers, read only.  At a committed optimizer boundary the flat-parameter
// gradients have been zeroed (arxiv 2609.18178, Section I), and the recovery
// protocol's guard admits a repair only with zero outstanding gradients
// (Section III-C, phase 2); this kernel is that check on the device.
//
// A word counts when its bit pattern is nonzero (so a -0.0 gradient counts).
// The pass reads 4 (fp32) or 2 (bf16) bytes per element and does one compare
// per element, so it is bound by HBM.  Same buffer plans and tiling scheme as
// the digest kernel (apc_digest.cu), with its own shape: 16-byte aligned
// bodies in tiles of kCountTile elements over a persistent grid, loads
// issued for the whole tile before counting, scalar head and tail by the CTA
// that owns the first tile, per-slot running counts flushed on CTA-uniform
// slot changes.
#include <cuda_runtime.h>

#include "../../include/apc.h"
#include "apc_internal.h"

namespace apc {
namespace {

__device__ __forceinline__ void flush(uint64_t &acc, int slot, unsigned long long *s_acc) {
  uint64_t x = acc;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
  if ((threadIdx.x & 31) == 0 && slot >= 0 && x) atomicAdd(&s_acc[slot], (unsigned long long)x);
  acc = 0;
}

__device__ __forceinline__ uint32_t nz32(uint4 x) {
  return (uint32_t)(x.x != 0) + (uint32_t)(x.y != 0) + (uint32_t)(x.z != 0) + (uint32_t)(x.w != 0);
}

__device__ __forceinline__ uint32_t nz16(uint32_t w) {
  return (uint32_t)((w & 0xFFFFu) != 0) + (uint32_t)((w >> 16) != 0);
}

template <int MAXE>
__global__ void __launch_bounds__(kCountThreads) count_kernel(const __grid_constant__ DigestPlan<MAXE> plan,
                                                         unsigned long long *out) {
  __shared__ unsigned long long s_acc[APC_MAX_SLOTS];
  if (threadIdx.x < APC_MAX_SLOTS) s_acc[threadIdx.x] = 0;
  __syncthreads();
  uint32_t cur = 0;
  int slot = -1;
  uint64_t acc = 0;
  for (uint64_t tile = blockIdx.x; tile < plan.total_tiles; tile += gridDim.x) {
    while (cur + 1 < plan.count && tile >= plan.e[cur + 1].tile_begin) ++cur;
    const DigestEntry &E = plan.e[cur];
    if ((int)E.slot != slot) {
      flush(acc, slot, s_acc);
      slot = E.slot;
    }
    const uint64_t local = tile - E.tile_begin;
    const uint64_t head = E.head;
    const uint64_t vec_end = head + ((E.n - head) & ~(uint64_t)(kVec - 1));
    const uint64_t base = head + local * kCountTile;
    uint32_t c = 0;
    if (E.dtype == 0) {
      const uint32_t *d = reinterpret_cast<const uint32_t *>(E.data);
      uint4 x[kCountUnroll][2];
      bool ok[kCountUnroll];
#pragma unroll
      for (int u = 0; u < kCountUnroll; ++u) {
        const uint64_t i = base + (uint64_t)(u * kCountThreads + threadIdx.x) * kVec;
        ok[u] = i < vec_end;
        if (ok[u]) {
          x[u][0] = __ldcs(reinterpret_cast<const uint4 *>(d + i));
          x[u][1] = __ldcs(reinterpret_cast<const uint4 *>(d + i) + 1);
        }
      }
#pragma unroll
      for (int u = 0; u < kCountUnroll; ++u)
        if (ok[u]) c += nz32(x[u][0]) + nz32(x[u][1]);
    } else {
      const uint16_t *d = reinterpret_cast<const uint16_t *>(E.data);
      uint4 x[kCountUnroll];
      bool ok[kCountUnroll];
#pragma unroll
      for (int u = 0; u < kCountUnroll; ++u) {
        const uint64_t i = base + (uint64_t)(u * kCountThreads + threadIdx.x) * kVec;
        ok[u] = i < vec_end;
        if (ok[u]) x[u] = __ldcs(reinterpret_cast<const uint4 *>(d + i));
      }
#pragma unroll
      for (int u = 0; u < kCountUnroll; ++u)
        if (ok[u]) c += nz16(x[u].x) + nz16(x[u].y) + nz16(x[u].z) + nz16(x[u].w);
    }
    if (local == 0) {
      const uint32_t t = threadIdx.x;
      if (t < head) {
        c += E.dtype == 0 ? (reinterpret_cast<const uint32_t *>(E.data)[t] != 0)
                          : (reinterpret_cast<const uint16_t *>(E.data)[t] != 0);
      }
      if (t >= 32 && t - 32 < E.n - vec_end) {
        const uint64_t i = vec_end + (t - 32);
        c += E.dtype == 0 ? (reinterpret_cast<const uint32_t *>(E.data)[i] != 0)
                          : (reinterpret_cast<const uint16_t *>(E.data)[i] != 0);
      }
    }
    acc += c;
  }
  flush(acc, slot, s_acc);
  __syncthreads();
  if (threadIdx.x < APC_MAX_SLOTS && s_acc[threadIdx.x]) atomicAdd(&out[threadIdx.x], s_acc[threadIdx.x]);
}

}  // namespace

int launch_count_small(const DigestPlan<kDigestSmall> &plan, unsigned grid, void *stream, unsigned long long *out) {
  count_kernel<kDigestSmall><<<grid, kCountThreads, 0, (cudaStream_t)stream>>>(plan, out);
  return (int)cudaGetLastError();
}

int launch_count_large(const DigestPlan<kDigestLarge> &plan, unsigned grid, void *stream, unsigned long long *out) {
  count_kernel<kDigestLarge><<<grid, kCountThreads, 0, (cudaStream_t)stream>>>(plan, out);
  return (int)cudaGetLastError();
}

int count_blocks_per_sm(bool large, int *out) {
  cudaError_t e = large ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, count_kernel<kDigestLarge>, kCountThreads, 0)
                        : cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, count_kernel<kDigestSmall>, kCountThreads, 0);
  return (int)e;
}

}  // namespace apc
