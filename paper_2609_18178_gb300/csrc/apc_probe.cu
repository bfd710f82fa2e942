// Register-only throughput probes of the SM's integer pipes, the measured
// denominators of the verification pass's roofline.  Not part of the hot
// path: libapc_probe.so is a separate library that the benchmark loads.
//
// Every thread runs `iters` steps over kChains independent chains held in
// registers; no memory is touched between the two clock reads.  A step is:
//   kind 0 (ALU pipe): a 32-bit funnel shift and an xor       2 lane-ops
//   kind 1 (multiply-add pipe): two 32-bit multiply-adds      2 lane-ops
//   kind 2 (both): the two ALU operations and the two
//          multiply-adds of kinds 0 and 1, interleaved          4 lane-ops
//   kind 3 (high multiply): two 32-bit high multiply-adds     2 lane-ops
//   kind 4 (wide multiply, low half): two 32 x 32 -> 64-bit
//          multiply-adds of which only the low half is used
//          (so the assembler may issue a plain multiply-add)   2 lane-ops
//   kind 5 (64-bit multiply): two 64 x 64 -> 64-bit multiplies,
//          each counted as the three 32-bit multiply-adds that
//          define it (the low halves' widening product, then the
//          two cross products into the high word)             6 lane-ops
//   kind 6 (64-bit multiply, explicit form): the same multiplies
//          written as one widening and two 32-bit multiply-adds
//          in the probe's own PTX                              6 lane-ops
// The operands of each operation come from the previous step, so the
// compiler can neither fold nor hoist them.  Thread 0 of every CTA records
// its SM's id and the SM clock counter when the CTA's loop starts and ends;
// per SM, the lane-ops of all CTAs it ran over the span from the first start
// to the last end is the SM's rate per clock, independent of the clock
// frequency and of how the CTAs were placed.
#include <cuda_runtime.h>
#include <stdint.h>

#define APC_PROBE_EXPORT extern "C" __attribute__((visibility("default")))

namespace {

constexpr int kChains = 8;
constexpr int kProbeThreads = 1024;

template <int KIND>
__global__ void __launch_bounds__(kProbeThreads)
    int_rate_kernel(uint32_t iters, uint32_t seed, uint32_t marker, unsigned long long *clocks) {
  uint32_t a[kChains], b[kChains];
  uint64_t w[kChains], v[kChains];
#pragma unroll
  for (int k = 0; k < kChains; ++k) {
    a[k] = seed ^ (threadIdx.x * kChains + k);
    b[k] = a[k] * 0x9E3779B9u + 0x7F4A7C15u;
    w[k] = ((uint64_t)b[k] << 32) | a[k] | 1u;
    v[k] = ((uint64_t)a[k] << 32) | b[k] | 1u;
  }
  __syncthreads();
  const long long t0 = clock64();
  for (uint32_t i = 0; i < iters; ++i) {
#pragma unroll
    for (int k = 0; k < kChains; ++k) {
      if (KIND == 0 || KIND == 2) {
        uint32_t t;
        asm volatile("shf.r.wrap.b32 %0, %1, %2, 7;" : "=r"(t) : "r"(a[k]), "r"(b[k]));
        asm volatile("xor.b32 %0, %0, %1;" : "+r"(a[k]) : "r"(t));
      }
      if (KIND == 1 || KIND == 2) {
        asm volatile("mad.lo.u32 %0, %0, %1, 0x7F4A7C15;" : "+r"(b[k]) : "r"(a[k]));
        asm volatile("mad.lo.u32 %0, %0, %1, 0x1CE4E5B9;" : "+r"(a[k]) : "r"(b[k]));
      }
      if (KIND == 3) {
        asm volatile("mad.hi.u32 %0, %0, %1, 0x7F4A7C15;" : "+r"(b[k]) : "r"(a[k]));
        asm volatile("mad.hi.u32 %0, %0, %1, 0x1CE4E5B9;" : "+r"(a[k]) : "r"(b[k]));
      }
      if (KIND == 5) {
        asm volatile("mul.lo.u64 %0, %0, %1;" : "+l"(w[k]) : "l"(v[k]));
        asm volatile("mul.lo.u64 %0, %0, %1;" : "+l"(v[k]) : "l"(w[k]));
      }
      if (KIND == 6) {
        asm volatile("{\n\t.reg .u32 al, ah, bl, bh, rl, rh;\n\t"
                     "mov.b64 {al, ah}, %0;\n\tmov.b64 {bl, bh}, %1;\n\t"
                     "mul.wide.u32 %0, al, bl;\n\tmov.b64 {rl, rh}, %0;\n\t"
                     "mad.lo.u32 rh, al, bh, rh;\n\tmad.lo.u32 rh, ah, bl, rh;\n\t"
                     "mov.b64 %0, {rl, rh};\n\t}"
                     : "+l"(w[k]) : "l"(v[k]));
        asm volatile("{\n\t.reg .u32 al, ah, bl, bh, rl, rh;\n\t"
                     "mov.b64 {al, ah}, %0;\n\tmov.b64 {bl, bh}, %1;\n\t"
                     "mul.wide.u32 %0, al, bl;\n\tmov.b64 {rl, rh}, %0;\n\t"
                     "mad.lo.u32 rh, al, bh, rh;\n\tmad.lo.u32 rh, ah, bl, rh;\n\t"
                     "mov.b64 %0, {rl, rh};\n\t}"
                     : "+l"(v[k]) : "l"(w[k]));
      }
      if (KIND == 4) {
        asm volatile("{\n\t.reg .u64 w;\n\tmad.wide.u32 w, %0, %1, %2;\n\tcvt.u32.u64 %0, w;\n\t}"
                     : "+r"(b[k]) : "r"(a[k]), "l"((uint64_t)a[k]));
        asm volatile("{\n\t.reg .u64 w;\n\tmad.wide.u32 w, %0, %1, %2;\n\tcvt.u32.u64 %0, w;\n\t}"
                     : "+r"(a[k]) : "r"(b[k]), "l"((uint64_t)b[k]));
      }
    }
  }
  __syncthreads();
  const long long t1 = clock64();
  // Every thread's chains stay live through a store that only a result
  // equal to the caller's marker makes (the compiler cannot rule it out).
  uint32_t x = 0;
#pragma unroll
  for (int k = 0; k < kChains; ++k) x ^= a[k] + b[k] + (uint32_t)(w[k] >> 32) + (uint32_t)(v[k] >> 32);
  if (x == marker) clocks[3 * gridDim.x] = x;
  if (threadIdx.x == 0) {
    uint32_t sm;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(sm));
    clocks[3 * blockIdx.x] = sm;
    clocks[3 * blockIdx.x + 1] = (unsigned long long)t0;
    clocks[3 * blockIdx.x + 2] = (unsigned long long)t1;
  }
}

}  // namespace

// Launch one probe on `stream`: kind 0 .. 6 (see above), `iters` steps,
// `grid` CTAs of 1024 threads.  clocks: device, 3 x grid + 1 uint64 (written:
// per CTA its SM id and the SM clock counter at the start and the end of its
// loop; the last word only if some thread's result equals `marker`, which
// keeps the chains from being optimised away).  Returns 0 or a cudaError_t
// value.  Lane-ops per CTA: 1024 x iters x 8 x (4 for kind 2, else 2).
APC_PROBE_EXPORT int apc_probe_int_rate(int kind, uint32_t iters, uint32_t grid, uint32_t marker,
                                        unsigned long long *clocks, void *stream) {
  if (kind < 0 || kind > 6 || grid == 0 || !clocks) return (int)cudaErrorInvalidValue;
  cudaStream_t s = (cudaStream_t)stream;
  if (kind == 0) int_rate_kernel<0><<<grid, kProbeThreads, 0, s>>>(iters, 12345u, marker, clocks);
  else if (kind == 1) int_rate_kernel<1><<<grid, kProbeThreads, 0, s>>>(iters, 12345u, marker, clocks);
  else if (kind == 2) int_rate_kernel<2><<<grid, kProbeThreads, 0, s>>>(iters, 12345u, marker, clocks);
  else if (kind == 3) int_rate_kernel<3><<<grid, kProbeThreads, 0, s>>>(iters, 12345u, marker, clocks);
  else if (kind == 4) int_rate_kernel<4><<<grid, kProbeThreads, 0, s>>>(iters, 12345u, marker, clocks);
  else if (kind == 5) int_rate_kernel<5><<<grid, kProbeThreads, 0, s>>>(iters, 12345u, marker, clocks);
  else int_rate_kernel<6><<<grid, kProbeThreads, 0, s>>>(iters, 12345u, marker, clocks);
  return (int)cudaGetLastError();
}

APC_PROBE_EXPORT int apc_probe_threads(void) { return kProbeThreads; }
APC_PROBE_EXPORT int apc_probe_chains(void) { return kChains; }
