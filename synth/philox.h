/*
 * Seeded synthetic input generator for the committed-step workloads.
 *
 * This header is the one piece of arithmetic that both the CUDA path's
 * callers (tests, bench) and the CPU oracle's callers use: it only makes
 * INPUTS.  It holds none of the committed step's own arithmetic (no AdamW,
 * no digest mixing, no round-to-nearest bf16 conversion).
 *
 * Random bits: Philox4x32-10, the counter-based generator of Salmon, Moraes,
 * Dror and Shaw, "Parallel random numbers: as easy as 1, 2, 3" (SC'11):
 * a 128-bit counter and a 64-bit key go through ten rounds of two 32x32->64
 * multiplies (multipliers 0xD2511F53, 0xCD9E8D57), each round xoring the
 * high halves with the other counter words and the key, with the key bumped
 * by the Weyl constants (0x9E3779B9, 0xBB67AE85) between rounds.
 *
 * Values (every value is a pure function of (seed, kind, global index, step),
 * so any index range of any buffer can be regenerated independently):
 *   counter = (i mod 2^32, i >> 32, kind << 16 | call, step), key = seed
 *   z  = (sum of the 12 32-bit words of calls 0,1,2) * 2^-32 - 6
 *        (Irwin-Hall sum of 12 uniforms: mean 0, variance 1, |z| <= 6;
 *         exact in double because the integer sum is below 2^36)
 *   p  = fp32(0.02 * z)                  params      ~ N(0, 0.02)
 *   m  = fp32(1e-4 * z)                  first moment ~ N(0, 1e-4)
 *   v  = x * x (fp32), x = fp32(1e-3 * z)   second moment = N(0,1e-3)^2
 *   g  = top 16 bits of fp32(1e-3 * z)   bf16 gradient ~ N(0, 1e-3), made by
 *        truncation; exactly +0 when word 0 of call 0 of kind GZERO is a
 *        multiple of 100 (1% exact zeros).  The gradient depends on the step.
 *   p16, m16, v16 = top 16 bits of p, m, v  (bf16 state, by truncation)
 * Only integer operations and single IEEE-rounded double/float operations are
 * used, so host and device produce the same bits.
 */
#ifndef SYNTH_PHILOX_H
#define SYNTH_PHILOX_H

#include <stdint.h>

#if defined(__CUDACC__)
#define SYNTH_HD __host__ __device__ __forceinline__
#else
#define SYNTH_HD static inline
#endif

enum {
  SYNTH_P = 1,      /* fp32 master parameters            */
  SYNTH_M = 2,      /* fp32 first moment                 */
  SYNTH_V = 3,      /* fp32 second moment                */
  SYNTH_G = 4,      /* bf16 gradient (depends on step)   */
  SYNTH_GZERO = 5,  /* zero mask of the gradient         */
  SYNTH_P16 = 6,    /* bf16 parameters: top half of SYNTH_P's value */
  SYNTH_M16 = 7,    /* bf16 first moment: top half of SYNTH_M's     */
  SYNTH_V16 = 8     /* bf16 second moment: top half of SYNTH_V's    */
};

SYNTH_HD void synth_mulhilo(uint32_t a, uint32_t b, uint32_t *hi, uint32_t *lo) {
  uint64_t r = (uint64_t)a * (uint64_t)b;
  *hi = (uint32_t)(r >> 32);
  *lo = (uint32_t)r;
}

/* Philox4x32 with 10 rounds; ctr[4] in, out[4] out. */
SYNTH_HD void synth_philox4x32_10(const uint32_t ctr[4], uint32_t k0, uint32_t k1, uint32_t out[4]) {
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  for (int r = 0; r < 10; ++r) {
    if (r > 0) { k0 += 0x9E3779B9u; k1 += 0xBB67AE85u; }
    uint32_t hi0, lo0, hi1, lo1;
    synth_mulhilo(0xD2511F53u, c0, &hi0, &lo0);
    synth_mulhilo(0xCD9E8D57u, c2, &hi1, &lo1);
    uint32_t n0 = hi1 ^ c1 ^ k0;
    uint32_t n2 = hi0 ^ c3 ^ k1;
    c0 = n0; c1 = lo1; c2 = n2; c3 = lo0;
  }
  out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

SYNTH_HD void synth_draw(uint64_t seed, int kind, uint32_t call, uint64_t i, int64_t step, uint32_t out[4]) {
  uint32_t ctr[4];
  ctr[0] = (uint32_t)i;
  ctr[1] = (uint32_t)(i >> 32);
  ctr[2] = ((uint32_t)kind << 16) | call;
  ctr[3] = (uint32_t)(uint64_t)step;
  synth_philox4x32_10(ctr, (uint32_t)seed, (uint32_t)(seed >> 32), out);
}

/* Irwin-Hall(12) standard normal approximation, exact in double. */
SYNTH_HD double synth_normal(uint64_t seed, int kind, uint64_t i, int64_t step) {
  uint64_t s = 0;
  for (uint32_t call = 0; call < 3; ++call) {
    uint32_t w[4];
    synth_draw(seed, kind, call, i, step, w);
    s += (uint64_t)w[0] + (uint64_t)w[1] + (uint64_t)w[2] + (uint64_t)w[3];
  }
  int64_t c = (int64_t)s - ((int64_t)6 << 32);
  return (double)c * (1.0 / 4294967296.0);
}

SYNTH_HD uint32_t synth_f32_bits(float f) {
  union { float f; uint32_t u; } x;
  x.f = f;
  return x.u;
}

SYNTH_HD float synth_p(uint64_t seed, uint64_t i) {
  return (float)(0.02 * synth_normal(seed, SYNTH_P, i, 0));
}

SYNTH_HD float synth_m(uint64_t seed, uint64_t i) {
  return (float)(1e-4 * synth_normal(seed, SYNTH_M, i, 0));
}

SYNTH_HD float synth_v(uint64_t seed, uint64_t i) {
  float x = (float)(1e-3 * synth_normal(seed, SYNTH_V, i, 0));
#if defined(__CUDA_ARCH__)
  return __fmul_rn(x, x);
#else
  return x * x;
#endif
}

SYNTH_HD uint16_t synth_g(uint64_t seed, uint64_t i, int64_t step) {
  uint32_t w[4];
  synth_draw(seed, SYNTH_GZERO, 0, i, step, w);
  if (w[0] % 100u == 0u) return 0;
  float x = (float)(1e-3 * synth_normal(seed, SYNTH_G, i, step));
  return (uint16_t)(synth_f32_bits(x) >> 16);
}

SYNTH_HD uint16_t synth_p16(uint64_t seed, uint64_t i) { return (uint16_t)(synth_f32_bits(synth_p(seed, i)) >> 16); }
SYNTH_HD uint16_t synth_m16(uint64_t seed, uint64_t i) { return (uint16_t)(synth_f32_bits(synth_m(seed, i)) >> 16); }
SYNTH_HD uint16_t synth_v16(uint64_t seed, uint64_t i) { return (uint16_t)(synth_f32_bits(synth_v(seed, i)) >> 16); }

#endif /* SYNTH_PHILOX_H */
