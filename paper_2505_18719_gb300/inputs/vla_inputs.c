/*
 * Seeded, counter-based input generator for the synthetic rollout workloads.
 *
 * This file holds no arithmetic of the method (no decoder, no sampler): it only
 * turns (seed, stream, index) into bytes.  Both the fp64 oracle and the CUDA path
 * consume the bytes it writes, so the two sides see identical inputs.
 *
 * Generator: SplitMix64 (G. Steele, D. Lea, C. Flood, "Fast splittable pseudorandom
 * number generators", OOPSLA 2014; constants as published by S. Vigna).  Element i of
 * stream s is the (i+1)-th SplitMix64 output of the state
 *     key(seed, s) = mix64(mix64(seed) ^ (s * GAMMA)),
 * i.e. mix64(key + (i+1) * GAMMA).  Being counter-based, any element can be produced
 * independently, so the result does not depend on the thread count.
 *
 * Normals: Box-Muller (G. Box, M. Muller, 1958) in fp64 on a pair of 53-bit uniforms,
 * element 2j from the cosine branch and 2j+1 from the sine branch; scaled by `std`,
 * rounded to fp32 (round-to-nearest) and then to bf16 (round-to-nearest-even).
 *
 * Pure C99 + pthreads; no architecture-specific code, so x86_64 and aarch64 agree.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <string.h>
#include <unistd.h>

#define GAMMA 0x9E3779B97F4A7C15ULL

static inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

static inline uint64_t stream_key(uint64_t seed, uint64_t stream) {
  return mix64(mix64(seed) ^ (stream * GAMMA));
}

static inline uint64_t draw(uint64_t key, uint64_t i) { return mix64(key + (i + 1) * GAMMA); }

/* fp32 -> bf16 bits, round to nearest even (inputs here are finite). */
static inline uint16_t f32_to_bf16(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  uint32_t lsb = (u >> 16) & 1u;
  u += 0x7FFFu + lsb;
  return (uint16_t)(u >> 16);
}

/* ---- work splitting ---------------------------------------------------- */
typedef struct {
  int kind;
  void* out;
  int64_t begin, end;
  uint64_t key;
  double a, b;
  int32_t lo, hi;
} job_t;

enum { K_NORMAL_BF16 = 0, K_UNIFORM_F32 = 1, K_RANDINT_I32 = 2 };

static void run_range(const job_t* j) {
  if (j->kind == K_NORMAL_BF16) {
    uint16_t* o = (uint16_t*)j->out;
    const double two_pi = 6.283185307179586476925286766559;
    /* element e uses pair p = e/2 (draws 2p and 2p+1) */
    for (int64_t e = j->begin; e < j->end; ++e) {
      uint64_t p = (uint64_t)e >> 1;
      double u1 = ((double)(draw(j->key, 2 * p) >> 11) + 0.5) * 0x1p-53;
      double u2 = ((double)(draw(j->key, 2 * p + 1) >> 11) + 0.5) * 0x1p-53;
      double r = sqrt(-2.0 * log(u1));
      double z = (e & 1) ? r * sin(two_pi * u2) : r * cos(two_pi * u2);
      o[e] = f32_to_bf16((float)(z * j->a + j->b));
    }
  } else if (j->kind == K_UNIFORM_F32) {
    float* o = (float*)j->out;
    for (int64_t e = j->begin; e < j->end; ++e) {
      uint64_t m = draw(j->key, (uint64_t)e) >> 41; /* 23 bits */
      o[e] = (float)(((double)m + 0.5) * 0x1p-23);  /* (2m+1) 2^-24: exact in fp32, in (0,1) */
    }
  } else {
    int32_t* o = (int32_t*)j->out;
    uint64_t span = (uint64_t)((int64_t)j->hi - (int64_t)j->lo + 1);
    for (int64_t e = j->begin; e < j->end; ++e) {
      uint64_t m = draw(j->key, (uint64_t)e) >> 32; /* 32 bits, multiply-shift range map */
      o[e] = (int32_t)((int64_t)j->lo + (int64_t)((m * span) >> 32));
    }
  }
}

static void* thread_main(void* arg) {
  run_range((const job_t*)arg);
  return 0;
}

static int n_threads_for(int64_t n) {
  long hw = sysconf(_SC_NPROCESSORS_ONLN);
  if (hw < 1) hw = 1;
  if (hw > 64) hw = 64;
  int64_t by_size = n / (1 << 16) + 1;
  return (int)(by_size < hw ? by_size : hw);
}

static void run_parallel(job_t proto, int64_t n) {
  int nt = n_threads_for(n);
  if (nt <= 1) {
    proto.begin = 0;
    proto.end = n;
    run_range(&proto);
    return;
  }
  pthread_t th[64];
  job_t jobs[64];
  int64_t chunk = (n + nt - 1) / nt;
  chunk = (chunk + 1) & ~(int64_t)1; /* keep Box-Muller pairs inside one chunk (not required) */
  int started = 0;
  for (int t = 0; t < nt; ++t) {
    jobs[t] = proto;
    jobs[t].begin = (int64_t)t * chunk;
    jobs[t].end = jobs[t].begin + chunk < n ? jobs[t].begin + chunk : n;
    if (jobs[t].begin >= jobs[t].end) break;
    if (pthread_create(&th[t], 0, thread_main, &jobs[t]) != 0) {
      run_range(&jobs[t]);
      jobs[t].kind = -1;
    }
    started = t + 1;
  }
  for (int t = 0; t < started; ++t)
    if (jobs[t].kind != -1) pthread_join(th[t], 0);
}

/* ---- exported --------------------------------------------------------- */

/* out[i] = bf16(std * N(0,1) + mean), i in [0, n). */
void vla_gen_normal_bf16(uint16_t* out, int64_t n, uint64_t seed, uint64_t stream, double std,
                         double mean) {
  job_t j = {K_NORMAL_BF16, out, 0, 0, stream_key(seed, stream), std, mean, 0, 0};
  run_parallel(j, n);
}

/* out[i] = (m + 0.5) * 2^-23, m uniform in [0, 2^23): exact in fp32, in [2^-24, 1 - 2^-24]. */
void vla_gen_uniform_f32(float* out, int64_t n, uint64_t seed, uint64_t stream) {
  job_t j = {K_UNIFORM_F32, out, 0, 0, stream_key(seed, stream), 0, 0, 0, 0};
  run_parallel(j, n);
}

/* out[i] uniform integer in [lo, hi] inclusive. */
void vla_gen_randint_i32(int32_t* out, int64_t n, uint64_t seed, uint64_t stream, int32_t lo,
                         int32_t hi) {
  job_t j = {K_RANDINT_I32, out, 0, 0, stream_key(seed, stream), 0, 0, lo, hi};
  run_parallel(j, n);
}

/* Raw SplitMix64 outputs, for the generator's own tests. */
void vla_gen_raw_u64(uint64_t* out, int64_t n, uint64_t seed, uint64_t stream) {
  uint64_t key = stream_key(seed, stream);
  for (int64_t e = 0; e < n; ++e) out[e] = draw(key, (uint64_t)e);
}

/* Plain SplitMix64 sequence from `state` (outputs 1..n), for checking mix64 against the
 * published reference outputs. */
void vla_gen_splitmix64(uint64_t* out, int64_t n, uint64_t state) {
  for (int64_t e = 0; e < n; ++e) {
    state += GAMMA;
    out[e] = mix64(state);
  }
}
