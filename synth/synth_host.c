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

static void fill_range(int kind, uint64_t seed, uint64_t goff, uint64_t lo, uint64_t hi,
                       int64_t step, void *out) {
  float *f = (float *)out;
  uint16_t *h = (uint16_t *)out;
  for (uint64_t j = lo; j < hi; ++j) {
    uint64_t i = goff + j;
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
