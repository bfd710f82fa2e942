// Host-to-device upload by the SMs (apc_upload).  On a Grace-Blackwell node
// the GPU reads page-locked (and, where supported, pageable) host memory
// coherently over NVLink-C2C, so plain 16-byte loads of the source, issued
// by a few CTAs, stream it into device memory at the link's rate without a
// DMA copy engine.  The launch is sized by the caller (max_ctas) so that it
// can run beside the step's persistent kernels on SMs they leave free.
//
// Each thread issues all of its kUploadUnroll loads of a tile before any
// store, which keeps enough bytes in flight to cover the link's latency.
#include <cuda_runtime.h>

#include "../../include/apc.h"
#include "apc_internal.h"

namespace apc {
namespace {

__global__ void __launch_bounds__(kUploadThreads) upload_kernel(const __grid_constant__ UploadPlan<kUploadMax> plan) {
  uint32_t cur = 0;
  for (uint64_t tile = blockIdx.x; tile < plan.total_tiles; tile += gridDim.x) {
    while (cur + 1 < plan.count && tile >= plan.e[cur + 1].tile_begin) ++cur;
    const UploadEntry &E = plan.e[cur];
    const uint64_t head = (16 - ((uintptr_t)E.dst & 15)) & 15;
    const uint64_t base = (tile - E.tile_begin) * kUploadTile;  // byte offset in the body
    const uint4 *src = reinterpret_cast<const uint4 *>(E.src + head);
    uint4 *dst = reinterpret_cast<uint4 *>(E.dst + head);
    uint4 x[kUploadUnroll];
    bool ok[kUploadUnroll];
#pragma unroll
    for (int u = 0; u < kUploadUnroll; ++u) {
      const uint64_t off = base + (uint64_t)(u * kUploadThreads + threadIdx.x) * 16;
      ok[u] = off < E.body;
      if (ok[u]) x[u] = __ldcs(src + off / 16);
    }
#pragma unroll
    for (int u = 0; u < kUploadUnroll; ++u) {
      const uint64_t off = base + (uint64_t)(u * kUploadThreads + threadIdx.x) * 16;
      if (ok[u]) dst[off / 16] = x[u];
    }
  }
  // scalar items: segment heads and tails, and mutually misaligned segments
  cur = 0;
  for (uint64_t it = (uint64_t)blockIdx.x * kUploadThreads + threadIdx.x; it < plan.total_scalar;
       it += (uint64_t)gridDim.x * kUploadThreads) {
    while (cur + 1 < plan.count && it >= plan.e[cur + 1].scalar_begin) ++cur;
    const UploadEntry &E = plan.e[cur];
    const uint64_t k = it - E.scalar_begin;
    uint64_t i;
    if (E.body == 0) {
      i = k;
    } else {
      const uint64_t head = (16 - ((uintptr_t)E.dst & 15)) & 15;
      i = k < head ? k : head + E.body + (k - head);
    }
    E.dst[i] = E.src[i];
  }
}

}  // namespace

int launch_upload(const UploadPlan<kUploadMax> &plan, unsigned grid, void *stream) {
  upload_kernel<<<grid, kUploadThreads, 0, (cudaStream_t)stream>>>(plan);
  return (int)cudaGetLastError();
}

}  // namespace apc
