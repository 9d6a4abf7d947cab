/*
 * rng.c — seeded synthetic inputs (weights, activations, token ids).
 *
 * This file draws random numbers and nothing else: it holds none of the
 * decode step's arithmetic and is shared, as an input generator only, by the
 * CPU oracle's tests and by the CUDA path's tests and benchmark.
 *
 * Generator (counter-based, so any element can be drawn independently and
 * the fill runs on many threads with identical results):
 *   mix(z)        the splitmix64 output function (Steele, Lea & Flood,
 *                 "Fast splittable pseudorandom number generators", 2014);
 *   key(seed,s)   mix(mix(seed + G) + (s + 1) * G), G = 0x9E3779B97F4A7C15,
 *                 one independent stream s per tensor;
 *   draw(key,i)   mix(key + (i + 1) * G), the (i+1)-th splitmix64 output;
 *   u53(z)        (z >> 11) * 2^-53, uniform in [0, 1).
 * Normals use the Box-Muller transform (Box & Muller, 1958) in double:
 * pair j takes u1 = 1 - u53(draw(2j)) in (0, 1] and u2 = u53(draw(2j+1));
 * element 2j is r*cos(2*pi*u2) and element 2j+1 is r*sin(2*pi*u2), with
 * r = sqrt(-2 ln u1). The value mean + std * z is rounded once to float.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>

#define GOLDEN 0x9E3779B97F4A7C15ULL

static inline uint64_t mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

uint64_t tvl_synth_key(uint64_t seed, uint64_t stream) {
  return mix(mix(seed + GOLDEN) + (stream + 1) * GOLDEN);
}

static inline uint64_t draw(uint64_t key, uint64_t i) { return mix(key + (i + 1) * GOLDEN); }
static inline double u53(uint64_t z) { return (double)(z >> 11) * (1.0 / 9007199254740992.0); }

static const double TWO_PI = 6.283185307179586476925286766559;

static double normal_at(uint64_t key, uint64_t i) {
  const uint64_t j = i >> 1;
  const double u1 = 1.0 - u53(draw(key, 2 * j));
  const double u2 = u53(draw(key, 2 * j + 1));
  const double r = sqrt(-2.0 * log(u1));
  return (i & 1) ? r * sin(TWO_PI * u2) : r * cos(TWO_PI * u2);
}

typedef struct {
  float* dst;
  uint64_t begin, end, key;
  double mean, std;
} job_t;

static void* fill_job(void* p) {
  job_t* j = (job_t*)p;
  uint64_t i = j->begin;
  /* an odd start takes the sine half of its pair */
  if (i < j->end && (i & 1)) {
    j->dst[i] = (float)(j->mean + j->std * normal_at(j->key, i));
    ++i;
  }
  for (; i + 1 < j->end; i += 2) {
    const uint64_t p2 = i >> 1;
    const double u1 = 1.0 - u53(draw(j->key, 2 * p2));
    const double u2 = u53(draw(j->key, 2 * p2 + 1));
    const double r = sqrt(-2.0 * log(u1));
    j->dst[i] = (float)(j->mean + j->std * (r * cos(TWO_PI * u2)));
    j->dst[i + 1] = (float)(j->mean + j->std * (r * sin(TWO_PI * u2)));
  }
  if (i < j->end) j->dst[i] = (float)(j->mean + j->std * normal_at(j->key, i));
  return NULL;
}

/* dst[i] = mean + std * N_i for i in [0, n), stream (seed, stream). */
void tvl_synth_fill_normal(float* dst, int64_t n, uint64_t seed, uint64_t stream, double mean,
                           double std, int nthreads) {
  if (n <= 0) return;
  const uint64_t key = tvl_synth_key(seed, stream);
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  if ((uint64_t)n < (uint64_t)nthreads * 65536u) nthreads = 1;
  job_t jobs[256];
  pthread_t th[256];
  for (int t = 0; t < nthreads; ++t) {
    jobs[t].dst = dst;
    jobs[t].begin = (uint64_t)n * t / nthreads;
    jobs[t].end = (uint64_t)n * (t + 1) / nthreads;
    jobs[t].key = key;
    jobs[t].mean = mean;
    jobs[t].std = std;
  }
  int started = 0;
  for (int t = 1; t < nthreads; ++t) {
    if (pthread_create(&th[t], NULL, fill_job, &jobs[t]) != 0) break;
    started = t;
  }
  fill_job(&jobs[0]);
  for (int t = 1; t <= started; ++t) pthread_join(th[t], NULL);
  for (int t = started + 1; t < nthreads; ++t) fill_job(&jobs[t]); /* threads that failed to start */
}

/* dst[i] uniform integers in [lo, hi] (inclusive): lo + floor(u53 * (hi - lo + 1)). */
void tvl_synth_uniform_ints(int32_t* dst, int64_t n, uint64_t seed, uint64_t stream, int32_t lo,
                            int32_t hi) {
  const uint64_t key = tvl_synth_key(seed, stream);
  const double span = (double)hi - (double)lo + 1.0;
  for (int64_t i = 0; i < n; ++i) {
    int64_t v = (int64_t)lo + (int64_t)floor(u53(draw(key, (uint64_t)i)) * span);
    if (v > hi) v = hi;
    dst[i] = (int32_t)v;
  }
}

/* Raw access for tests of the generator itself: the i-th output (from 0)
 * of a splitmix64 generator whose state starts at `state`. */
uint64_t tvl_synth_splitmix64(uint64_t state, uint64_t i) { return draw(state, i); }

uint64_t tvl_synth_draw(uint64_t seed, uint64_t stream, uint64_t i) {
  return draw(tvl_synth_key(seed, stream), i);
}
double tvl_synth_normal_at(uint64_t seed, uint64_t stream, uint64_t i) {
  return normal_at(tvl_synth_key(seed, stream), i);
}
