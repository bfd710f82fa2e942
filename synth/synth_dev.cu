/*
 * Device fill routines for the seeded synthetic inputs (values defined in
 * philox.h, bit-identical to synth_host.c).  Used to place full-size
 * workloads directly in HBM without a host round trip.  Compiled with
 * -fmad=false so that no multiply is fused with a neighbouring add.
 */
#include <cuda_runtime.h>
#include <stdint.h>

#include "philox.h"

#define SYNTH_EXPORT extern "C" __attribute__((visibility("default")))

__global__ void synth_fill_kernel(int kind, uint64_t seed, uint64_t goff, uint64_t n, int64_t step,
                                  void *out) {
  uint64_t j = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  float *f = (float *)out;
  uint16_t *h = (uint16_t *)out;
  for (; j < n; j += stride) {
    const uint64_t i = goff + j;
    switch (kind) {
      case SYNTH_P: f[j] = synth_p(seed, i); break;
      case SYNTH_M: f[j] = synth_m(seed, i); break;
      case SYNTH_V: f[j] = synth_v(seed, i); break;
      case SYNTH_G: h[j] = synth_g(seed, i, step); break;
      case SYNTH_P16: h[j] = synth_p16(seed, i); break;
      case SYNTH_M16: h[j] = synth_m16(seed, i); break;
      case SYNTH_V16: h[j] = synth_v16(seed, i); break;
      default: break;
    }
  }
}

/* Fill a device buffer out[0..n) with the values of global indices
 * goff..goff+n-1 on `stream` (a cudaStream_t, may be null).
 * Returns a cudaError_t value (0 on success); -1 on a bad kind. */
SYNTH_EXPORT int synth_fill_dev(int kind, uint64_t seed, uint64_t goff, uint64_t n, int64_t step,
                                void *out, void *stream) {
  if (kind < SYNTH_P || kind > SYNTH_V16 || kind == SYNTH_GZERO) return -1;
  if (n == 0) return 0;
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return (int)e;
  e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return (int)e;
  uint64_t blocks = (n + 255) / 256;
  const uint64_t cap = (uint64_t)sms * 16;
  if (blocks > cap) blocks = cap;
  synth_fill_kernel<<<(unsigned)blocks, 256, 0, (cudaStream_t)stream>>>(kind, seed, goff, n, step, out);
  return (int)cudaGetLastError();
}
