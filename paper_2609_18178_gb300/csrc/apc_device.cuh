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
  uint32_t one;    // 1, from the launch parameters (see digest_term)
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

// Two binary32 values in one 64-bit register pair, lane 0 in the low half,
// for the packed two-lane multiply (mul.rn.f32x2): each lane is an IEEE
// binary32 multiply rounded to nearest even, subnormals kept, so it gives
// each lane the bits of the scalar multiply.
__device__ __forceinline__ uint64_t pack2(float a, float b) {
  return ((uint64_t)__float_as_uint(b) << 32) | __float_as_uint(a);
}
__device__ __forceinline__ float lane0(uint64_t x) { return __uint_as_float((uint32_t)x); }
__device__ __forceinline__ float lane1(uint64_t x) { return __uint_as_float((uint32_t)(x >> 32)); }
__device__ __forceinline__ uint64_t mul2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

// adamw_element for two elements at once: the same binary32 operations in
// the same order, each multiply issued as one packed two-lane instruction.
// The adds and the subtract stay scalar __fadd_rn / __fsub_rn: a packed
// product feeding a packed add was found contracted into a fused
// multiply-add by the assembler (a 1-ulp change in a quarter of the
// elements), while the scalar round-to-nearest adds are never fused.  The
// square root and the divide run per lane.  w0, w1: the bf16 bits of p'.
__device__ __forceinline__ void adamw_pair(float &p0, float &p1, float &m0, float &m1, float &v0, float &v1,
                                           uint32_t g16a, uint32_t g16b, const Scalars &s, uint32_t &w0,
                                           uint32_t &w1) {
  const uint64_t g = pack2(__uint_as_float(g16a << 16), __uint_as_float(g16b << 16));
  const uint64_t t1 = mul2(pack2(s.h[0], s.h[0]), pack2(m0, m1));
  const uint64_t t2 = mul2(pack2(s.h[1], s.h[1]), g);
  const uint64_t gg = mul2(g, g);
  const uint64_t t3 = mul2(pack2(s.h[2], s.h[2]), pack2(v0, v1));
  const uint64_t t4 = mul2(pack2(s.h[3], s.h[3]), gg);
  const float mn0 = __fadd_rn(lane0(t1), lane0(t2)), mn1 = __fadd_rn(lane1(t1), lane1(t2));
  const float vn0 = __fadd_rn(lane0(t3), lane0(t4)), vn1 = __fadd_rn(lane1(t3), lane1(t4));
  const uint64_t t5 = mul2(pack2(__fsqrt_rn(vn0), __fsqrt_rn(vn1)), pack2(s.h[7], s.h[7]));
  const float den0 = __fadd_rn(lane0(t5), s.h[4]), den1 = __fadd_rn(lane1(t5), s.h[4]);
  const uint64_t t6 = mul2(pack2(p0, p1), pack2(s.h[5], s.h[5]));
  const uint64_t t7 = mul2(pack2(s.h[6], s.h[6]), pack2(__fdiv_rn(mn0, den0), __fdiv_rn(mn1, den1)));
  p0 = __fsub_rn(lane0(t6), lane0(t7));
  p1 = __fsub_rn(lane1(t6), lane1(t7));
  m0 = mn0;
  m1 = mn1;
  v0 = vn0;
  v1 = vn1;
  w0 = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(p0));
  w1 = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(p1));
}

// The two 64-bit multiplies of the splitmix64 finaliser, z * C mod 2^64 for
// a constant C = (chi : clo), in one of two instruction forms.  Which one is
// faster depends on the kernel around it (both give the same bits):
//  * MulWide: three multiply-adds, lo*clo widened, then lo*chi and hi*clo
//    added into the high word.  Fewest instructions; the commit kernel,
//    which is bound by instruction issue, runs 2.7% faster with it.
//  * MulCompiler: the compiler's own 64-bit multiply.  The verification
//    pass, which is bound by the integer ALU rather than by issue, runs 3.3%
//    faster with it.
struct MulWide {
  template <uint32_t CLO, uint32_t CHI>
  __device__ __forceinline__ static uint64_t mul(uint64_t z) {
    uint64_t r;
    asm("{\n\t.reg .u32 l, h, rl, rh;\n\t"
        "mov.b64 {l, h}, %1;\n\t"
        "mul.wide.u32 %0, l, %2;\n\t"
        "mov.b64 {rl, rh}, %0;\n\t"
        "mad.lo.u32 rh, l, %3, rh;\n\t"
        "mad.lo.u32 rh, h, %2, rh;\n\t"
        "mov.b64 %0, {rl, rh};\n\t}"
        : "=l"(r)
        : "l"(z), "n"(CLO), "n"(CHI));
    return r;
  }
};

struct MulCompiler {
  template <uint32_t CLO, uint32_t CHI>
  __device__ __forceinline__ static uint64_t mul(uint64_t z) {
    return z * (((uint64_t)CHI << 32) | CLO);
  }
};

// splitmix64 of the digest key (((G + K) mod 2^32) << 32) | bits: the first
// output of Vigna's SplitMix64 seeded with the key (golden-ratio increment,
// then the 30/27/31 xor-shift multiply finaliser).  K is a compile-time
// element offset from G.
//
// Instruction mix: the kernels are short of integer-ALU issue, so the 64-bit
// increment puts its high half on the FMA pipe as an extended-precision
// multiply-add: lo = bits + 0x7F4A7C15 sets the carry, then
// hi = one * (0x9E3779B9 + K) + G + carry, with `one` a launch parameter
// equal to 1 (so the assembler cannot turn it back into an ALU add) and the
// offset K folded into the immediate: (G + K) + 0x9E3779B9 and
// G + (0x9E3779B9 + K) are equal mod 2^32, and no add of K is issued.
//
// The first xor-shift needs hi >> 30, the top two bits of the incremented
// high word.  Callers that know them for a whole run of terms pass them as
// `hi_top` (see digest_term's four-argument form); otherwise they are
// computed here.
template <uint32_t K, class Mul>
__device__ __forceinline__ uint64_t digest_term_core(uint32_t gidx, uint32_t bits, uint32_t one, bool have_top,
                                                     uint32_t hi_top) {
  uint32_t lo, hi;
  asm("add.cc.u32 %0, %2, 0x7F4A7C15;\n\t"
      "madc.lo.u32 %1, %4, %5, %3;"
      : "=r"(lo), "=r"(hi)
      : "r"(bits), "r"(gidx), "r"(one), "n"(0x9E3779B9u + K));
  const uint32_t l1 = lo ^ __funnelshift_r(lo, hi, 30);
  const uint32_t h1 = hi ^ (have_top ? hi_top : hi >> 30);
  uint64_t z = ((uint64_t)h1 << 32) | l1;
  z = Mul::template mul<0x1CE4E5B9u, 0xBF58476Du>(z);
  z = Mul::template mul<0x133111EBu, 0x94D049BBu>(z ^ (z >> 27));
  return z ^ (z >> 31);
}

template <uint32_t K = 0, class Mul = MulWide>
__device__ __forceinline__ uint64_t digest_term(uint32_t gidx, uint32_t bits, uint32_t one) {
  return digest_term_core<K, Mul>(gidx, bits, one, false, 0);
}

// The same term with hi >> 30 supplied: hi_top must equal the top two bits
// of gidx + 0x9E3779B9 + K + carry.  For terms whose keys G + K lie in
// [G0, G0 + R), every incremented high word lies in [B, B + R] with
// B = G0 + 0x9E3779B9 (the carry adds at most 1); when B and B + R have the
// same top two bits (top_bits_shared), those bits are B >> 30 for all of them.
template <uint32_t K = 0, class Mul = MulWide>
__device__ __forceinline__ uint64_t digest_term(uint32_t gidx, uint32_t bits, uint32_t one, uint32_t hi_top) {
  return digest_term_core<K, Mul>(gidx, bits, one, true, hi_top);
}

// splitmix64 term of a 16-bit word (bits < 2^16).  Its low key half plus
// 0x7F4A7C15 never carries and always has top bits 01, so after the
// increment lo = bits + 0x7F4A7C15, hi = gidx + 0x9E3779B9 + K, and the
// first xor-shift's low word is lo ^ ((hi << 2) | 1) = lo ^ (4 * hi + 1).
// All three are multiply-adds by `one` (the FMA pipe); `top` is hi >> 30,
// shared by the caller (digest_term's hi_top rule).
template <uint32_t K = 0, class Mul = MulWide>
__device__ __forceinline__ uint64_t digest_term_u16(uint32_t gidx, uint32_t bits, uint32_t one, uint32_t top) {
  uint32_t lo, hi, m4;
  asm("mad.lo.u32 %0, %3, %4, 0x7F4A7C15;\n\t"
      "mad.lo.u32 %1, %4, %6, %5;\n\t"
      "mad.lo.u32 %2, %1, 4, %4;"
      : "=r"(lo), "=r"(hi), "=r"(m4)
      : "r"(bits), "r"(one), "r"(gidx), "n"(0x9E3779B9u + K));
  const uint32_t l1 = lo ^ m4, h1 = hi ^ top;
  uint64_t z = ((uint64_t)h1 << 32) | l1;
  z = Mul::template mul<0x1CE4E5B9u, 0xBF58476Du>(z);
  z = Mul::template mul<0x133111EBu, 0x94D049BBu>(z ^ (z >> 27));
  return z ^ (z >> 31);
}

__device__ __forceinline__ bool top_bits_shared(uint32_t B, uint32_t R) { return ((B ^ (B + R)) >> 30) == 0; }

// acc += z (mod 2^64), with the high half's carry-add on the FMA pipe.  Used
// for single terms; pairs of terms are summed as acc += a + b, which the
// compiler folds into one three-input add per 32-bit half.
__device__ __forceinline__ void acc_add(uint64_t &acc, uint64_t z, uint32_t one) {
  uint32_t alo = (uint32_t)acc, ahi = (uint32_t)(acc >> 32);
  asm("add.cc.u32 %0, %0, %2;\n\t"
      "madc.lo.u32 %1, %3, %4, %1;"
      : "+r"(alo), "+r"(ahi)
      : "r"((uint32_t)z), "r"((uint32_t)(z >> 32)), "r"(one));
  acc = ((uint64_t)ahi << 32) | alo;
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
