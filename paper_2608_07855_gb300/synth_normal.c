/*
 * Counter-based N(0,1) generator for the synthetic agent-shaped KV caches.
 *
 * This file holds no arithmetic of the scoring method: it only turns
 * (seed, stream, element index) into a standard-normal sample, so that the
 * CPU oracle's inputs and the GPU library's inputs are the same numbers.
 *
 *   key      = splitmix64(seed * 0x9E3779B97F4A7C15 + stream)
 *   u1, u2   = two 53-bit uniforms in (0, 1) from splitmix64(key + 2j),
 *              splitmix64(key + 2j + 1)
 *   z0, z1   = Box-Muller pair: sqrt(-2 ln u1) * (cos, sin)(2 pi u2)
 *   element 2j = z0, element 2j+1 = z1, times an optional per-channel
 *   scale (channel = element index mod channels).
 *
 * splitmix64 is the published mixing function of Steele, Lea and Flood
 * ("Fast splittable pseudorandom number generators", OOPSLA 2014).
 * Output is fp32 or bf16 (round to nearest even).  Threads split the index
 * range; the values do not depend on the thread count.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <string.h>

static inline uint64_t mix64(uint64_t x) {
  x += 0x9E3779B97F4A7C15ull;
  x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
  x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
  return x ^ (x >> 31);
}

static inline uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) return (uint16_t)((u >> 16) | 0x40u);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

typedef struct {
  uint64_t key;
  int64_t begin, end; /* element range [begin, end) */
  int dtype;          /* 0 = fp32, 1 = bf16 */
  void *out;
  const float *chan_scale; /* NULL or [channels] */
  int64_t channels;
} fill_job;

static inline void put(const fill_job *j, int64_t i, double z) {
  float f = (float)z;
  if (j->chan_scale) f *= j->chan_scale[i % j->channels];
  if (j->dtype == 0)
    ((float *)j->out)[i - j->begin] = f;
  else
    ((uint16_t *)j->out)[i - j->begin] = f32_to_bf16_rne(f);
}

static void *fill_worker(void *arg) {
  fill_job *j = (fill_job *)arg;
  const double two_pi = 6.283185307179586476925286766559;
  const double inv53 = 1.0 / 9007199254740992.0; /* 2^-53 */
  for (int64_t p = j->begin >> 1; 2 * p < j->end; ++p) {
    uint64_t r1 = mix64(j->key + 2 * (uint64_t)p);
    uint64_t r2 = mix64(j->key + 2 * (uint64_t)p + 1);
    double u1 = ((double)(r1 >> 11) + 0.5) * inv53;
    double u2 = ((double)(r2 >> 11) + 0.5) * inv53;
    double rad = sqrt(-2.0 * log(u1));
    double ang = two_pi * u2;
    int64_t i0 = 2 * p, i1 = 2 * p + 1;
    if (i0 >= j->begin) put(j, i0, rad * cos(ang));
    if (i1 < j->end) put(j, i1, rad * sin(ang));
  }
  return NULL;
}

/* Fill out[0..n) with elements [offset, offset + n) of stream (seed, stream).
 * dtype 0 writes float, 1 writes bf16 bits.  chan_scale may be NULL.
 * Returns 0 on success, -1 on bad arguments. */
int synth_normal_fill(uint64_t seed, uint64_t stream, int64_t offset, int64_t n, int dtype,
                      void *out, const float *chan_scale, int64_t channels, int nthreads) {
  if (n < 0 || offset < 0 || (dtype != 0 && dtype != 1) || (!out && n > 0)) return -1;
  if (chan_scale && channels <= 0) return -1;
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 64) nthreads = 64;
  if (n < 65536) nthreads = 1;
  uint64_t key = mix64(seed * 0x9E3779B97F4A7C15ull + stream);
  pthread_t th[64];
  int created[64];
  fill_job jobs[64];
  int64_t per = (n + nthreads - 1) / nthreads;
  size_t esz = dtype == 0 ? 4 : 2;
  for (int t = 0; t < nthreads; ++t) {
    created[t] = 0;
    int64_t b = (int64_t)t * per, e = b + per;
    if (e > n) e = n;
    if (b >= e) continue;
    jobs[t].key = key;
    jobs[t].begin = offset + b;
    jobs[t].end = offset + e;
    jobs[t].dtype = dtype;
    jobs[t].out = (char *)out + (size_t)b * esz;
    jobs[t].chan_scale = chan_scale;
    jobs[t].channels = channels;
    if (nthreads > 1 && pthread_create(&th[t], NULL, fill_worker, &jobs[t]) == 0)
      created[t] = 1;
    else
      fill_worker(&jobs[t]);
  }
  for (int t = 0; t < nthreads; ++t)
    if (created[t]) pthread_join(th[t], NULL);
  return 0;
}
