// Device arithmetic of the committed step: the AdamW element update in its
// fixed binary32 order and the splitmix64 digest term.
//
// Every floating-point operation is an explicit round-to-nearest intrinsic
// (__fmul_rn, __fadd_rn, __fsub_rn, __fsqrt_rn, __fdiv_rn), which the
// compiler never fuses into FMA; the library is also built with -fmad=false
// and without flush-to-zero.  The update is decoupled-weight-decay AdamW
// (the optimizer whose committed W, M, V the paper preserves, arxiv
// 2609.18178 Section III-A, Eq. 2) and the digest realises its bitwise rank
// state checks (Sections IV-F, IV-G).
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

namespace apc {

// The step's eight binary32 scalars, read where they are used.  In the
// kernels they point into the launch's __grid_constant__ parameter block, so
// every use is a constant-bank operand and holds no register.
struct Scalars {
  const float *h;  // b1, 1-b1, b2, 1-b2, eps, 1-lr*wd, lr/(1-b1^t), 1/sqrt(1-b2^t)
};

// One element: p, m, v updated in place, returns the bf16 bits of p'.
__device__ __forceinline__ uint32_t adamw_element(float &p, float &m, float &v, uint32_t g16, const Scalars &s) {
  const float g = __uint_as_float(g16 << 16);
  const float t1 = __fmul_rn(s.h[0], m);
  const float t2 = __fmul_rn(s.h[1], g);
  const float mn = __fadd_rn(t1, t2);
  const float gg = __fmul_rn(g, g);
  const float t3 = __fmul_rn(s.h[2], v);
  const float t4 = __fmul_rn(s.h[3], gg);
  const float vn = __fadd_rn(t3, t4);
  const float sq = __fsqrt_rn(vn);
  const float t5 = __fmul_rn(sq, s.h[7]);
  const float den = __fadd_rn(t5, s.h[4]);
  const float u = __fdiv_rn(mn, den);
  const float t6 = __fmul_rn(p, s.h[5]);
  const float t7 = __fmul_rn(s.h[6], u);
  const float pn = __fsub_rn(t6, t7);
  p = pn;
  m = mn;
  v = vn;
  return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(pn));
}

// splitmix64 of the digest key ((G mod 2^32) << 32) | bits: the first output
// of Vigna's SplitMix64 seeded with the key (golden-ratio increment, then the
// 30/27/31 xor-shift multiply finaliser).
__device__ __forceinline__ uint64_t digest_term(uint32_t gidx, uint32_t bits) {
  uint64_t z = (((uint64_t)gidx << 32) | bits) + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Sum of a CTA's per-thread values; the result is valid in thread 0.
// `scratch` holds THREADS/32 words.
template <int THREADS>
__device__ __forceinline__ uint64_t cta_sum(uint64_t x, uint64_t *scratch) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) scratch[warp] = x;
  __syncthreads();
  uint64_t r = 0;
  if (threadIdx.x == 0) {
#pragma unroll
    for (int i = 0; i < THREADS / 32; ++i) r += scratch[i];
  }
  __syncthreads();
  return r;
}

}  // namespace apc
