/* Seeded synthetic inputs for the embed-and-retrieve hot path.
 *
 * This module only draws random numbers and lays them out; it holds none of
 * the method's arithmetic (no hashing, merging, scoring or selection).  The
 * oracle and the GPU library both consume what it writes.
 *
 * Random numbers come from one counter-based generator: the SplitMix64 output
 * function (Steele, Lea and Flood, "Fast splittable pseudorandom number
 * generators", OOPSLA 2014) applied to key + (counter + 1) * golden gamma.
 * Every value depends only on (seed, stream, counter), so any slice of any
 * array can be produced independently, in any order and on any thread.
 *
 * Gaussian values use the Box-Muller transform on two uniforms from adjacent
 * counters; vectors are normalised in fp64, rounded to fp32 and then to bf16
 * (round to nearest even at each step).  libm's log/cos make the Gaussian
 * draws platform-dependent in the last ulp, which is harmless: both sides of
 * every comparison read the same generated buffer.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define GOLDEN_GAMMA 0x9e3779b97f4a7c15ULL

static inline uint64_t sm64_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
  z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
  return z ^ (z >> 31);
}

/* Key of one independent stream of a seed. */
static inline uint64_t stream_key(uint64_t seed, uint64_t stream) {
  return sm64_mix(sm64_mix(seed + GOLDEN_GAMMA) ^ (stream * 0xd1b54a32d192ed03ULL + 1));
}

static inline uint64_t ctr_u64(uint64_t key, uint64_t i) {
  return sm64_mix(key + (i + 1) * GOLDEN_GAMMA);
}

/* Uniform in (0, 1]. */
static inline double ctr_unit(uint64_t key, uint64_t i) {
  return ((double)(ctr_u64(key, i) >> 11) + 1.0) * (1.0 / 9007199254740992.0);
}

/* Uniform integer in [0, m), m >= 1 (Lemire's multiply-shift on 32 bits when
 * m fits, otherwise a 64-bit modulo; the bias is irrelevant here). */
static inline uint64_t ctr_below(uint64_t key, uint64_t i, uint64_t m) {
  uint64_t u = ctr_u64(key, i);
  if (m <= 0xffffffffULL) return ((u >> 32) * m) >> 32;
  return u % m;
}

static inline double ctr_normal(uint64_t key, uint64_t i) {
  double u1 = ctr_unit(key, 2 * i);
  double u2 = ctr_unit(key, 2 * i + 1);
  return sqrt(-2.0 * log(u1)) * cos(6.283185307179586476925286766559 * u2);
}

static inline uint16_t f32_to_bf16_rne(float f) {
  uint32_t b;
  memcpy(&b, &f, 4);
  if ((b & 0x7f800000u) == 0x7f800000u) return (uint16_t)(b >> 16); /* inf/nan */
  b += 0x7fffu + ((b >> 16) & 1u);
  return (uint16_t)(b >> 16);
}

uint64_t synth_u64(uint64_t seed, uint64_t stream, uint64_t i) {
  return ctr_u64(stream_key(seed, stream), i);
}

double synth_normal(uint64_t seed, uint64_t stream, uint64_t i) {
  return ctr_normal(stream_key(seed, stream), i);
}

/* ---- threading helper ---------------------------------------------------- */

typedef void (*range_fn)(void* ctx, int64_t lo, int64_t hi);
typedef struct { range_fn fn; void* ctx; int64_t lo, hi; } range_job;

static void* run_range(void* p) {
  range_job* j = (range_job*)p;
  j->fn(j->ctx, j->lo, j->hi);
  return NULL;
}

static void parallel_rows(range_fn fn, void* ctx, int64_t n, int nthreads) {
  if (nthreads <= 1 || n < 4096) { fn(ctx, 0, n); return; }
  if (nthreads > 256) nthreads = 256;
  pthread_t th[256];
  range_job jobs[256];
  int started = 0;
  for (int t = 0; t < nthreads; ++t) {
    jobs[t].fn = fn; jobs[t].ctx = ctx;
    jobs[t].lo = n * t / nthreads; jobs[t].hi = n * (t + 1) / nthreads;
    if (pthread_create(&th[t], NULL, run_range, &jobs[t]) != 0) {
      fn(ctx, jobs[t].lo, jobs[t].hi);  /* could not start a thread: do it here */
      th[t] = 0;
    } else {
      ++started;
    }
  }
  for (int t = 0; t < nthreads; ++t) if (th[t]) pthread_join(th[t], NULL);
  (void)started;
}

/* ---- token rows ------------------------------------------------------------ */

typedef struct {
  int32_t* out; int32_t stride; const int32_t* lens; int32_t vocab;
  uint64_t key; int64_t ordinal0;
} tok_ctx;

static void tok_range(void* p, int64_t lo, int64_t hi) {
  tok_ctx* c = (tok_ctx*)p;
  for (int64_t r = lo; r < hi; ++r) {
    int32_t* row = c->out + r * (int64_t)c->stride;
    int32_t len = c->lens ? c->lens[r] : c->stride;
    int64_t ord = c->ordinal0 + r;
    for (int32_t t = 0; t < c->stride; ++t) {
      int32_t v;
      if (t >= len) v = 0;                                  /* zero padding */
      else if (t == 0) v = (int32_t)(ord % c->vocab);       /* ordinal stamp: */
      else if (t == 1) v = (int32_t)((ord / c->vocab) % c->vocab); /* rows distinct */
      else v = (int32_t)ctr_below(c->key, (uint64_t)(r * (int64_t)c->stride + t), (uint64_t)c->vocab);
      row[t] = v;
    }
  }
}

/* Distinct token rows: row r gets tokens uniform in [0, vocab) except that its
 * first two tokens spell the ordinal (ordinal0 + r) in base vocab, so rows of
 * length >= 2 are pairwise distinct by construction.  Tokens at t >= lens[r]
 * are 0 (lens may be NULL: full rows). */
void synth_token_rows(int32_t* out, int64_t n, int32_t stride, const int32_t* lens,
                      int32_t vocab, uint64_t seed, uint64_t stream, int64_t ordinal0,
                      int nthreads) {
  tok_ctx c = {out, stride, lens, vocab, stream_key(seed, stream), ordinal0};
  parallel_rows(tok_range, &c, n, nthreads);
}

/* Uniform integers in [lo, hi] inclusive. */
void synth_uniform_ints(int32_t* out, int64_t n, int32_t lo, int32_t hi, uint64_t seed,
                        uint64_t stream) {
  uint64_t key = stream_key(seed, stream);
  uint64_t span = (uint64_t)((int64_t)hi - lo + 1);
  for (int64_t i = 0; i < n; ++i) out[i] = lo + (int32_t)ctr_below(key, (uint64_t)i, span);
}

/* ---- bf16 vectors ------------------------------------------------------------ */

typedef struct {
  uint16_t* out; int32_t d; uint64_t key; int64_t counter0;
  const double* centres; const int64_t* centre_of_row; double noise;
} vec_ctx;

static void write_normalised(uint16_t* dst, double* v, int32_t d) {
  double ss = 0.0;
  for (int32_t t = 0; t < d; ++t) ss += v[t] * v[t];
  double inv = ss > 0.0 ? 1.0 / sqrt(ss) : 0.0;
  for (int32_t t = 0; t < d; ++t) dst[t] = f32_to_bf16_rne((float)(v[t] * inv));
}

static void vec_range(void* p, int64_t lo, int64_t hi) {
  vec_ctx* c = (vec_ctx*)p;
  double* v = (double*)malloc(sizeof(double) * (size_t)c->d);
  if (!v) return;
  for (int64_t r = lo; r < hi; ++r) {
    int64_t base = (c->counter0 + r) * (int64_t)c->d;
    const double* ctr = NULL;
    if (c->centres && c->centre_of_row) {
      int64_t ci = c->centre_of_row[r];
      if (ci >= 0) ctr = c->centres + ci * (int64_t)c->d;
    }
    for (int32_t t = 0; t < c->d; ++t) {
      double z = ctr_normal(c->key, (uint64_t)(base + t));
      v[t] = ctr ? ctr[t] + c->noise * z : z;
    }
    write_normalised(c->out + r * (int64_t)c->d, v, c->d);
  }
  free(v);
}

/* n unit-norm rows: Gaussian N(0,1) components, normalised.  Row r uses the
 * counters of row (counter0 + r), so slices of one big array can be drawn
 * separately and agree with drawing it whole. */
void synth_unit_rows_bf16(uint16_t* out, int64_t n, int32_t d, uint64_t seed,
                          uint64_t stream, int64_t counter0, int nthreads) {
  vec_ctx c = {out, d, stream_key(seed, stream), counter0, NULL, NULL, 0.0};
  parallel_rows(vec_range, &c, n, nthreads);
}

/* Rows near given centres: row r = normalise(centres[centre_of_row[r]] +
 * noise * z) with z ~ N(0, I); rows whose centre index is negative are plain
 * Gaussian rows.  centres is fp64 [n_centres, d]. */
void synth_rows_near_bf16(uint16_t* out, int64_t n, int32_t d, const double* centres,
                          const int64_t* centre_of_row, double noise, uint64_t seed,
                          uint64_t stream, int64_t counter0, int nthreads) {
  vec_ctx c = {out, d, stream_key(seed, stream), counter0, centres, centre_of_row, noise};
  parallel_rows(vec_range, &c, n, nthreads);
}

/* Unit-norm fp64 centres (Gaussian, normalised, no rounding). */
void synth_unit_centres_f64(double* out, int64_t n, int32_t d, uint64_t seed,
                            uint64_t stream) {
  uint64_t key = stream_key(seed, stream);
  for (int64_t r = 0; r < n; ++r) {
    double ss = 0.0;
    for (int32_t t = 0; t < d; ++t) {
      double z = ctr_normal(key, (uint64_t)(r * (int64_t)d + t));
      out[r * (int64_t)d + t] = z;
      ss += z * z;
    }
    double inv = 1.0 / sqrt(ss);
    for (int32_t t = 0; t < d; ++t) out[r * (int64_t)d + t] *= inv;
  }
}

/* ---- index draws --------------------------------------------------------------- */

/* First m entries of a seeded Fisher-Yates shuffle of [0, n): distinct
 * positions, written to out[0:m].  Needs an n-entry scratch array. */
int synth_choose_distinct(int64_t* out, int64_t n, int64_t m, uint64_t seed,
                          uint64_t stream) {
  if (m < 0 || m > n) return 1;
  int64_t* a = (int64_t*)malloc(sizeof(int64_t) * (size_t)(n > 0 ? n : 1));
  if (!a) return 2;
  for (int64_t i = 0; i < n; ++i) a[i] = i;
  uint64_t key = stream_key(seed, stream);
  for (int64_t i = 0; i < m; ++i) {
    int64_t j = i + (int64_t)ctr_below(key, (uint64_t)i, (uint64_t)(n - i));
    int64_t t = a[i]; a[i] = a[j]; a[j] = t;
    out[i] = a[i];
  }
  free(a);
  return 0;
}

/* Zipf draws: n i.i.d. ranks r in [0, pool) with P(r) proportional to
 * (r + 1)^(-s), by inverse CDF (binary search on the cumulative weights). */
int synth_zipf_ranks(int64_t* out, int64_t n, int64_t pool, double s, uint64_t seed,
                     uint64_t stream) {
  double* cdf = (double*)malloc(sizeof(double) * (size_t)pool);
  if (!cdf) return 2;
  double acc = 0.0;
  for (int64_t r = 0; r < pool; ++r) { acc += pow((double)(r + 1), -s); cdf[r] = acc; }
  uint64_t key = stream_key(seed, stream);
  for (int64_t i = 0; i < n; ++i) {
    double u = ctr_unit(key, (uint64_t)i) * acc;   /* (0, acc] */
    int64_t lo = 0, hi = pool - 1;
    while (lo < hi) {                              /* first r with cdf[r] >= u */
      int64_t mid = lo + (hi - lo) / 2;
      if (cdf[mid] >= u) hi = mid; else lo = mid + 1;
    }
    out[i] = lo;
  }
  free(cdf);
  return 0;
}

/* Uniform integers below per-element bounds: out[i] in [0, bound[i]). */
void synth_below(int64_t* out, const int64_t* bound, int64_t n, uint64_t seed,
                 uint64_t stream) {
  uint64_t key = stream_key(seed, stream);
  for (int64_t i = 0; i < n; ++i)
    out[i] = bound[i] > 0 ? (int64_t)ctr_below(key, (uint64_t)i, (uint64_t)bound[i]) : 0;
}
