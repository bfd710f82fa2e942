/*
 * Host fill routines for the seeded synthetic inputs (values defined in
 * philox.h).  Plain C with POSIX threads; shared by the tests, the bench
 * and the oracle's callers.  Compiled with -ffp-contract=off so that the
 * single double multiply and the conversion to float round exactly like
 * the device fill.
 */
#include <pthread.h>
#include <stdint.h>
#include <string.h>

#include "philox.h"

#define SYNTH_EXPORT __attribute__((visibility("default")))

/* Lane blocks: the host fills kLanes consecutive indices at a time, with
 * every Philox round applied to all lanes before the next, so that the
 * compiler can keep the lanes in vector registers (SSE2 on x86-64, NEON on
 * aarch64).  Each lane performs exactly the operations of philox.h's scalar
 * functions in the same order, so the values are bit-identical to theirs
 * (and to the device fill); synth_fill_at keeps the scalar path. */
enum { kLanes = 16 };

static void philox_lanes(uint32_t *restrict c0, uint32_t *restrict c1, uint32_t *restrict c2, uint32_t *restrict c3,
                         uint32_t k0, uint32_t k1) {
  for (int r = 0; r < 10; ++r) {
    if (r > 0) { k0 += 0x9E3779B9u; k1 += 0xBB67AE85u; }
    for (int l = 0; l < kLanes; ++l) {
      const uint64_t a = (uint64_t)0xD2511F53u * (uint64_t)c0[l];
      const uint64_t b = (uint64_t)0xCD9E8D57u * (uint64_t)c2[l];
      const uint32_t n0 = (uint32_t)(b >> 32) ^ c1[l] ^ k0;
      const uint32_t n2 = (uint32_t)(a >> 32) ^ c3[l] ^ k1;
      c0[l] = n0;
      c1[l] = (uint32_t)b;
      c2[l] = n2;
      c3[l] = (uint32_t)a;
    }
  }
}

/* Philox blocks of (kind, call) at indices i0 .. i0 + kLanes - 1. */
static void draw_lanes(uint64_t seed, int kind, uint32_t call, uint64_t i0, int64_t step, uint32_t *restrict w0,
                       uint32_t *restrict w1, uint32_t *restrict w2, uint32_t *restrict w3) {
  for (int l = 0; l < kLanes; ++l) {
    const uint64_t i = i0 + (uint64_t)l;
    w0[l] = (uint32_t)i;
    w1[l] = (uint32_t)(i >> 32);
    w2[l] = ((uint32_t)kind << 16) | call;
    w3[l] = (uint32_t)(uint64_t)step;
  }
  philox_lanes(w0, w1, w2, w3, (uint32_t)seed, (uint32_t)(seed >> 32));
}

/* synth_normal for kLanes consecutive indices. */
static void normal_lanes(uint64_t seed, int kind, uint64_t i0, int64_t step, double z[kLanes]) {
  uint64_t s[kLanes];
  uint32_t w0[kLanes], w1[kLanes], w2[kLanes], w3[kLanes];
  for (int l = 0; l < kLanes; ++l) s[l] = 0;
  for (uint32_t call = 0; call < 3; ++call) {
    draw_lanes(seed, kind, call, i0, step, w0, w1, w2, w3);
    for (int l = 0; l < kLanes; ++l)
      s[l] += (uint64_t)w0[l] + (uint64_t)w1[l] + (uint64_t)w2[l] + (uint64_t)w3[l];
  }
  for (int l = 0; l < kLanes; ++l) {
    const int64_t c = (int64_t)s[l] - ((int64_t)6 << 32);
    z[l] = (double)c * (1.0 / 4294967296.0);
  }
}

/* One block of kLanes values of `kind` at global indices i0.., into f or h. */
static void fill_block(int kind, uint64_t seed, uint64_t i0, int64_t step, float *f, uint16_t *h) {
  double z[kLanes];
  switch (kind) {
    case SYNTH_P:
    case SYNTH_P16:
      normal_lanes(seed, SYNTH_P, i0, 0, z);
      for (int l = 0; l < kLanes; ++l) {
        const float x = (float)(0.02 * z[l]);
        if (kind == SYNTH_P) f[l] = x; else h[l] = (uint16_t)(synth_f32_bits(x) >> 16);
      }
      break;
    case SYNTH_M:
    case SYNTH_M16:
      normal_lanes(seed, SYNTH_M, i0, 0, z);
      for (int l = 0; l < kLanes; ++l) {
        const float x = (float)(1e-4 * z[l]);
        if (kind == SYNTH_M) f[l] = x; else h[l] = (uint16_t)(synth_f32_bits(x) >> 16);
      }
      break;
    case SYNTH_V:
    case SYNTH_V16:
      normal_lanes(seed, SYNTH_V, i0, 0, z);
      for (int l = 0; l < kLanes; ++l) {
        const float x = (float)(1e-3 * z[l]);
        const float y = x * x;
        if (kind == SYNTH_V) f[l] = y; else h[l] = (uint16_t)(synth_f32_bits(y) >> 16);
      }
      break;
    case SYNTH_G: {
      uint32_t w0[kLanes], w1[kLanes], w2[kLanes], w3[kLanes];
      draw_lanes(seed, SYNTH_GZERO, 0, i0, step, w0, w1, w2, w3);
      normal_lanes(seed, SYNTH_G, i0, step, z);
      for (int l = 0; l < kLanes; ++l) {
        const float x = (float)(1e-3 * z[l]);
        h[l] = w0[l] % 100u == 0u ? (uint16_t)0 : (uint16_t)(synth_f32_bits(x) >> 16);
      }
      break;
    }
    default:
      break;
  }
}

static void fill_one(int kind, uint64_t seed, uint64_t i, int64_t step, float *f, uint16_t *h) {
  switch (kind) {
    case SYNTH_P: *f = synth_p(seed, i); break;
    case SYNTH_M: *f = synth_m(seed, i); break;
    case SYNTH_V: *f = synth_v(seed, i); break;
    case SYNTH_G: *h = synth_g(seed, i, step); break;
    case SYNTH_P16: *h = synth_p16(seed, i); break;
    case SYNTH_M16: *h = synth_m16(seed, i); break;
    case SYNTH_V16: *h = synth_v16(seed, i); break;
    default: break;
  }
}

static void fill_range(int kind, uint64_t seed, uint64_t goff, uint64_t lo, uint64_t hi,
                       int64_t step, void *out) {
  float *f = (float *)out;
  uint16_t *h = (uint16_t *)out;
  uint64_t j = lo;
  for (; j + kLanes <= hi; j += kLanes) fill_block(kind, seed, goff + j, step, f + j, h + j);
  for (; j < hi; ++j) fill_one(kind, seed, goff + j, step, f + j, h + j);
}

typedef struct {
  int kind;
  uint64_t seed, goff, lo, hi;
  int64_t step;
  void *out;
} fill_job;

static void *fill_worker(void *arg) {
  fill_job *j = (fill_job *)arg;
  fill_range(j->kind, j->seed, j->goff, j->lo, j->hi, j->step, j->out);
  return NULL;
}

/* Fill out[0..n) with the values of global indices goff..goff+n-1.
 * kind: SYNTH_P/M/V (float out) or SYNTH_G/P16/M16/V16 (uint16 bf16 bits out).
 * Returns 0 on success, -1 on a bad kind. */
SYNTH_EXPORT int synth_fill(int kind, uint64_t seed, uint64_t goff, uint64_t n, int64_t step,
                            void *out, int nthreads) {
  if (kind < SYNTH_P || kind > SYNTH_V16 || kind == SYNTH_GZERO) return -1;
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  if ((uint64_t)nthreads > n / 65536 + 1) nthreads = (int)(n / 65536 + 1);
  if (nthreads == 1) {
    fill_range(kind, seed, goff, 0, n, step, out);
    return 0;
  }
  pthread_t th[256];
  fill_job jobs[256];
  int started[256];
  for (int t = 0; t < nthreads; ++t) {
    jobs[t].kind = kind; jobs[t].seed = seed; jobs[t].goff = goff; jobs[t].step = step;
    jobs[t].out = out;
    jobs[t].lo = n * (uint64_t)t / (uint64_t)nthreads;
    jobs[t].hi = n * (uint64_t)(t + 1) / (uint64_t)nthreads;
    started[t] = pthread_create(&th[t], NULL, fill_worker, &jobs[t]) == 0;
    if (!started[t]) fill_worker(&jobs[t]);
  }
  for (int t = 0; t < nthreads; ++t)
    if (started[t]) pthread_join(th[t], NULL);
  return 0;
}

/* Values at arbitrary global indices idx[0..n). */
SYNTH_EXPORT int synth_fill_at(int kind, uint64_t seed, const uint64_t *idx, uint64_t n, int64_t step,
                               void *out) {
  if (kind < SYNTH_P || kind > SYNTH_V16 || kind == SYNTH_GZERO) return -1;
  float *f = (float *)out;
  uint16_t *h = (uint16_t *)out;
  for (uint64_t j = 0; j < n; ++j) {
    switch (kind) {
      case SYNTH_P: f[j] = synth_p(seed, idx[j]); break;
      case SYNTH_M: f[j] = synth_m(seed, idx[j]); break;
      case SYNTH_V: f[j] = synth_v(seed, idx[j]); break;
      case SYNTH_G: h[j] = synth_g(seed, idx[j], step); break;
      case SYNTH_P16: h[j] = synth_p16(seed, idx[j]); break;
      case SYNTH_M16: h[j] = synth_m16(seed, idx[j]); break;
      case SYNTH_V16: h[j] = synth_v16(seed, idx[j]); break;
      default: break;
    }
  }
  return 0;
}

/* Raw Philox4x32-10 block, exported for known-answer tests. */
SYNTH_EXPORT void synth_philox(const uint32_t ctr[4], uint32_t k0, uint32_t k1, uint32_t out[4]) {
  synth_philox4x32_10(ctr, k0, k1, out);
}

/* Raw Irwin-Hall normal (double), exported for distribution tests. */
SYNTH_EXPORT double synth_normal_at(uint64_t seed, int kind, uint64_t i, int64_t step) {
  return synth_normal(seed, kind, i, step);
}
