/*
 * CPU oracle for the committed optimizer step and its state digest.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the package smoke check and the
 * benchmark's CPU-baseline leg may load this library.  It shares no source
 * with the CUDA path (kernels, host library or headers).
 *
 * What it computes (arxiv 2609.18178):
 *  - The committed boundary (Section I; Section III-C, phase 2) is the point
 *    where the parameter and moment updates of the optimizer step have landed.
 *    The state the paper preserves across a communicator fault is
 *    S_app = {W, M, V, ..., tau_opt} (Section III-A, Eq. 2): the sharded
 *    weights, the AdamW first/second moments and the step counter.  The step
 *    that produces W, M, V at that boundary is AdamW.  The paper prints no
 *    formula for it, so this file takes decoupled-weight-decay AdamW
 *    (Loshchilov & Hutter) with the bias corrections folded into two scalars,
 *    in one fixed binary32 operation order (one rounding per operation, no
 *    fused multiply-add):
 *        m' = b1*m + (1-b1)*g
 *        v' = b2*v + (1-b2)*(g*g)
 *        den = sqrt(v') * (1/sqrt(1-b2^t)) + eps
 *        p' = p*(1 - lr*wd) - (lr/(1-b1^t)) * (m'/den)
 *        w  = bf16 round-to-nearest-even of p'
 *    with the eight scalars computed in double from the decimal
 *    hyper-parameters and rounded once to binary32.
 *  - The paper checks that ranks hold bit-identical parameter and optimizer
 *    state after recovery (Abstract; Section IV-F, IV-G) without saying how.
 *    The digest here is the order-independent wrapping sum
 *        D_B = sum_i splitmix64(((G_i mod 2^32) << 32) | bits_B(i))  mod 2^64
 *    over the post-update buffers B in {p', m', v', w}, G_i the element's
 *    index in the flat model, bf16 bits zero-extended, where splitmix64(x)
 *    is the first output of Vigna's SplitMix64 generator seeded with x.
 *
 * Build: gcc -O2 -std=c11 -ffp-contract=off -fno-fast-math (no FTZ), so that
 * every float operation below rounds once, to nearest even.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <string.h>

#define ORACLE_EXPORT __attribute__((visibility("default")))

/* ---------------------------------------------------------------- hparams */

/* The eight binary32 scalars of one step, in this order. */
enum { HB1 = 0, HOMB1, HB2, HOMB2, HEPS, HDECAY, HSTEP, HRSB2, HNUM };

/* Resolve the step's scalars: every quantity is formed in double from the
 * decimal hyper-parameters and rounded once to binary32.
 *   bc1 = 1 - b1^t, bc2 = 1 - b2^t (double, pow)
 *   b1, 1-b1, b2, 1-b2, eps, 1-lr*wd, lr/bc1, 1/sqrt(bc2).
 * Returns 0, or -1 when the inputs are out of range (t < 1, beta outside
 * [0,1), eps <= 0, a non-finite value, lr or wd negative). */
ORACLE_EXPORT int oracle_resolve_hparams(double lr, double b1, double b2, double eps, double wd,
                                         int64_t t, float out[HNUM]) {
  if (t < 1) return -1;
  if (!isfinite(lr) || !isfinite(b1) || !isfinite(b2) || !isfinite(eps) || !isfinite(wd)) return -1;
  if (!(b1 >= 0.0 && b1 < 1.0) || !(b2 >= 0.0 && b2 < 1.0)) return -1;
  if (!(eps > 0.0) || lr < 0.0 || wd < 0.0) return -1;
  double bc1 = 1.0 - pow(b1, (double)t);
  double bc2 = 1.0 - pow(b2, (double)t);
  out[HB1] = (float)b1;
  out[HOMB1] = (float)(1.0 - b1);
  out[HB2] = (float)b2;
  out[HOMB2] = (float)(1.0 - b2);
  out[HEPS] = (float)eps;
  out[HDECAY] = (float)(1.0 - lr * wd);
  out[HSTEP] = (float)(lr / bc1);
  out[HRSB2] = (float)(1.0 / sqrt(bc2));
  return 0;
}

/* ------------------------------------------------------------------- bf16 */

static uint32_t f2u(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  return u;
}

static float u2f(uint32_t u) {
  float f;
  memcpy(&f, &u, 4);
  return f;
}

/* bf16 value of a gradient word: the 16 bits are the top half of a binary32. */
ORACLE_EXPORT float oracle_bf16_to_f32(uint16_t h) { return u2f((uint32_t)h << 16); }

/* Round a binary32 to bf16, nearest, ties to even (non-NaN inputs). */
ORACLE_EXPORT uint16_t oracle_bf16_rne(float x) {
  uint32_t u = f2u(x);
  uint32_t lsb = (u >> 16) & 1u;
  return (uint16_t)((u + 0x7FFFu + lsb) >> 16);
}

/* ------------------------------------------------------------------ AdamW */

/* One element of the step in the fixed operation order, in binary32:
 * (p, m, v, g) -> (p', m', v'). */
static void adamw_core(float p, float m, float v, float g, const float h[HNUM], float *pn_out, float *mn_out,
                       float *vn_out) {
  float t1 = h[HB1] * m;
  float t2 = h[HOMB1] * g;
  float mn = t1 + t2;
  float gg = g * g;
  float t3 = h[HB2] * v;
  float t4 = h[HOMB2] * gg;
  float vn = t3 + t4;
  float s = sqrtf(vn);
  float t5 = s * h[HRSB2];
  float den = t5 + h[HEPS];
  float u = mn / den;
  float t6 = p * h[HDECAY];
  float t7 = h[HSTEP] * u;
  *pn_out = t6 - t7;
  *mn_out = mn;
  *vn_out = vn;
}

/* One element of the fp32-state step; w receives the bf16 copy of p'. */
static void adamw_one(float *p, float *m, float *v, uint16_t g16, uint16_t *w, const float h[HNUM]) {
  float pn, mn, vn;
  adamw_core(*p, *m, *v, oracle_bf16_to_f32(g16), h, &pn, &mn, &vn);
  *p = pn;
  *m = mn;
  *v = vn;
  *w = oracle_bf16_rne(pn);
}

/* In-place AdamW over n elements; w receives the bf16 copy of p'. */
ORACLE_EXPORT void oracle_adamw(float *p, float *m, float *v, const uint16_t *g, uint16_t *w, uint64_t n,
                                const float h[HNUM]) {
  for (uint64_t i = 0; i < n; ++i) adamw_one(&p[i], &m[i], &v[i], g[i], &w[i], h);
}

/* ----------------------------------------------------------------- digest */

/* First output of SplitMix64 (Vigna, splitmix64.c) seeded with x. */
ORACLE_EXPORT uint64_t oracle_splitmix64(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

static uint64_t key_of(uint64_t gidx, uint32_t bits) { return (gidx << 32) | (uint64_t)bits; }

/* Digest of n binary32 words (given as their bits) at global indices goff.. */
ORACLE_EXPORT uint64_t oracle_digest_u32(const uint32_t *bits, uint64_t n, uint64_t goff) {
  uint64_t d = 0;
  for (uint64_t i = 0; i < n; ++i) d += oracle_splitmix64(key_of(goff + i, bits[i]));
  return d;
}

/* Digest of n bf16 words (zero-extended) at global indices goff.. */
ORACLE_EXPORT uint64_t oracle_digest_u16(const uint16_t *bits, uint64_t n, uint64_t goff) {
  uint64_t d = 0;
  for (uint64_t i = 0; i < n; ++i) d += oracle_splitmix64(key_of(goff + i, (uint32_t)bits[i]));
  return d;
}

/* Elementwise bf16 rounding of an array (test helper). */
ORACLE_EXPORT void oracle_bf16_rne_array(const float *x, uint16_t *out, uint64_t n) {
  for (uint64_t i = 0; i < n; ++i) out[i] = oracle_bf16_rne(x[i]);
}

/* ------------------------------------------------------ quiescence guard */

/* Number of words whose bit pattern is nonzero (the "zero outstanding
 * gradients" guard of the recovery protocol, Section III-C, phase 2). */
ORACLE_EXPORT uint64_t oracle_count_nonzero_u16(const uint16_t *x, uint64_t n) {
  uint64_t c = 0;
  for (uint64_t i = 0; i < n; ++i) c += x[i] != 0;
  return c;
}

ORACLE_EXPORT uint64_t oracle_count_nonzero_u32(const uint32_t *x, uint64_t n) {
  uint64_t c = 0;
  for (uint64_t i = 0; i < n; ++i) c += x[i] != 0;
  return c;
}

/* --------------------------------------------------------- bf16 state */

/* The step with p, m, v stored in bf16 (the paper keeps parameters and AdamW
 * moments in BF16, Section IV-A): widen exactly, run the same binary32
 * order, round each of p', m', v' once to bf16 when storing. */
ORACLE_EXPORT void oracle_adamw_bf16(uint16_t *p, uint16_t *m, uint16_t *v, const uint16_t *g, uint64_t n,
                                     const float h[HNUM]) {
  for (uint64_t i = 0; i < n; ++i) {
    float pn, mn, vn;
    adamw_core(oracle_bf16_to_f32(p[i]), oracle_bf16_to_f32(m[i]), oracle_bf16_to_f32(v[i]),
               oracle_bf16_to_f32(g[i]), h, &pn, &mn, &vn);
    p[i] = oracle_bf16_rne(pn);
    m[i] = oracle_bf16_rne(mn);
    v[i] = oracle_bf16_rne(vn);
  }
}

/* bf16-state step over one tensor, then the three digests of the written
 * words (p', m', v'), added into out[0..2] mod 2^64. */
ORACLE_EXPORT void oracle_commit_bf16(uint16_t *p, uint16_t *m, uint16_t *v, const uint16_t *g, uint64_t n,
                                      uint64_t goff, const float h[HNUM], uint64_t out[3]) {
  oracle_adamw_bf16(p, m, v, g, n, h);
  out[0] += oracle_digest_u16(p, n, goff);
  out[1] += oracle_digest_u16(m, n, goff);
  out[2] += oracle_digest_u16(v, n, goff);
}

/* ---------------------------------------------------------- whole commit */

/* The committed step over one tensor: AdamW in place, then the four digests
 * of the written buffers (p', m', v', w) added into out[0..3] mod 2^64. */
ORACLE_EXPORT void oracle_commit(float *p, float *m, float *v, const uint16_t *g, uint16_t *w, uint64_t n,
                                 uint64_t goff, const float h[HNUM], uint64_t out[4]) {
  oracle_adamw(p, m, v, g, w, n, h);
  out[0] += oracle_digest_u32((const uint32_t *)p, n, goff);
  out[1] += oracle_digest_u32((const uint32_t *)m, n, goff);
  out[2] += oracle_digest_u32((const uint32_t *)v, n, goff);
  out[3] += oracle_digest_u16(w, n, goff);
}

typedef struct {
  float *p, *m, *v;
  const uint16_t *g;
  uint16_t *w;
  uint64_t n, goff;
  const float *h;
  uint64_t d[4];
} commit_job;

static void *commit_worker(void *arg) {
  commit_job *j = (commit_job *)arg;
  j->d[0] = j->d[1] = j->d[2] = j->d[3] = 0;
  oracle_commit(j->p, j->m, j->v, j->g, j->w, j->n, j->goff, j->h, j->d);
  return NULL;
}

/* The same step split into nthreads contiguous pieces run on POSIX threads;
 * the per-piece digests are combined by the same wrapping sum. */
ORACLE_EXPORT void oracle_commit_mt(float *p, float *m, float *v, const uint16_t *g, uint16_t *w, uint64_t n,
                                    uint64_t goff, const float h[HNUM], uint64_t out[4], int nthreads) {
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  pthread_t th[256];
  commit_job jobs[256];
  int started[256];
  for (int t = 0; t < nthreads; ++t) {
    uint64_t lo = n * (uint64_t)t / (uint64_t)nthreads, hi = n * (uint64_t)(t + 1) / (uint64_t)nthreads;
    commit_job *j = &jobs[t];
    j->p = p + lo; j->m = m + lo; j->v = v + lo; j->g = g + lo; j->w = w + lo;
    j->n = hi - lo; j->goff = goff + lo; j->h = h;
    started[t] = pthread_create(&th[t], NULL, commit_worker, j) == 0;
    if (!started[t]) commit_worker(j);
  }
  for (int t = 0; t < nthreads; ++t) {
    if (started[t]) pthread_join(th[t], NULL);
    for (int k = 0; k < 4; ++k) out[k] += jobs[t].d[k];
  }
}
