/*
 * Seeded synthetic inputs: Gaussian-mixture base/query vectors and N(0, s^2)
 * encoder weights, all drawn from the Philox4x32-10 counter-based generator
 * (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy as 1, 2, 3",
 * SC'11), written here from its published definition.
 *
 * This module holds none of the search method's arithmetic. It only produces
 * inputs; both the oracle and the CUDA path are fed from it. Every value is a
 * pure function of (seed, stream, row, column), so any row can be regenerated
 * on its own and the output does not depend on the thread count.
 *
 * Workloads (stand-ins for the paper's BigANN / Deep1B data, which are not
 * available here; paper Sec. 4.1, Table "datasets_all"):
 *   u8  : x = clip(rint(c_m + sigma * z), 0, 255), c_m uniform in [20, 235]^D
 *   f32 : x = normalize(c_m + sigma * z),          c_m ~ N(0, I_D)
 * with m uniform over M components and z ~ N(0, I_D).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define PHILOX_M0 0xD2511F53u
#define PHILOX_M1 0xCD9E8D57u
#define PHILOX_W0 0x9E3779B9u
#define PHILOX_W1 0xBB67AE85u

/* streams: the Philox key is (seed, stream) */
#define STREAM_ROWS 0x524F5753u    /* component choice + noise of each row */
#define STREAM_CENTRES 0x43454E54u /* mixture centres */
#define STREAM_NORMAL 0x4E524D4Cu  /* plain normal arrays (encoder weights) */

static inline void mulhilo32(uint32_t a, uint32_t b, uint32_t *hi, uint32_t *lo) {
  uint64_t p = (uint64_t)a * (uint64_t)b;
  *hi = (uint32_t)(p >> 32);
  *lo = (uint32_t)p;
}

/* Philox4x32 with 10 rounds: 10 S-box rounds, key bumped by the Weyl
 * constants between rounds. */
void synth_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int r = 0; r < 10; ++r) {
    uint32_t hi0, lo0, hi1, lo1;
    mulhilo32(PHILOX_M0, c0, &hi0, &lo0);
    mulhilo32(PHILOX_M1, c2, &hi1, &lo1);
    uint32_t n0 = hi1 ^ c1 ^ k0;
    uint32_t n1 = lo1;
    uint32_t n2 = hi0 ^ c3 ^ k1;
    uint32_t n3 = lo0;
    c0 = n0; c1 = n1; c2 = n2; c3 = n3;
    k0 += PHILOX_W0;
    k1 += PHILOX_W1;
  }
  out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

static inline void philox(uint32_t a, uint32_t b, uint32_t c, uint32_t d, uint64_t seed,
                          uint32_t stream, uint32_t out[4]) {
  uint32_t ctr[4] = {a, b, c, d};
  uint32_t key[2] = {(uint32_t)seed ^ (uint32_t)(seed >> 32), stream};
  synth_philox4x32_10(ctr, key, out);
}

/* 53-bit uniform in [0, 1) from two 32-bit words */
static inline double u53(uint32_t hi, uint32_t lo) {
  uint64_t v = (((uint64_t)hi << 32) | lo) >> 11;
  return (double)v * (1.0 / 9007199254740992.0);
}

/* Box-Muller: one Philox block -> two independent N(0,1) draws */
static inline void box_muller(const uint32_t w[4], double *z0, double *z1) {
  double u1 = 1.0 - u53(w[0], w[1]); /* (0, 1] */
  double u2 = u53(w[2], w[3]);
  double r = sqrt(-2.0 * log(u1));
  double a = 6.283185307179586476925 * u2;
  *z0 = r * cos(a);
  *z1 = r * sin(a);
}

/* centre coordinate (m, j) */
static double centre_u8(uint64_t seed, int64_t m, int j) {
  uint32_t w[4];
  philox((uint32_t)m, (uint32_t)(j >> 1), 0u, 2u, seed, STREAM_CENTRES, w);
  double u = (j & 1) ? u53(w[2], w[3]) : u53(w[0], w[1]);
  return 20.0 + 215.0 * u;
}

static double centre_f32(uint64_t seed, int64_t m, int j) {
  uint32_t w[4];
  double z0, z1;
  philox((uint32_t)m, (uint32_t)(j >> 1), 0u, 3u, seed, STREAM_CENTRES, w);
  box_muller(w, &z0, &z1);
  return (j & 1) ? z1 : z0;
}

static int64_t row_component(uint64_t seed, int64_t i, int M) {
  uint32_t w[4];
  philox((uint32_t)i, (uint32_t)((uint64_t)i >> 32), 0xFFFFFFFFu, 1u, seed, STREAM_ROWS, w);
  int64_t m = (int64_t)(u53(w[0], w[1]) * (double)M);
  return m < M ? m : M - 1;
}

/* z_{i, 2p}, z_{i, 2p+1} */
static void row_noise_pair(uint64_t seed, int64_t i, int p, double *z0, double *z1) {
  uint32_t w[4];
  philox((uint32_t)i, (uint32_t)((uint64_t)i >> 32), (uint32_t)p, 0u, seed, STREAM_ROWS, w);
  box_muller(w, z0, z1);
}

typedef struct {
  int kind; /* 0 = u8 mixture, 1 = f32 mixture, 2 = normal array */
  uint64_t seed_rows, seed_centres;
  int M, D;
  double sigma;
  int64_t row0, n;
  void *out;
  const double *centres; /* [M x D] precomputed */
  int64_t lo, hi;
} job_t;

static void *run_rows(void *arg) {
  job_t *jb = (job_t *)arg;
  int D = jb->D;
  double *v = (double *)malloc(sizeof(double) * (size_t)(D + 1));
  for (int64_t r = jb->lo; r < jb->hi; ++r) {
    int64_t i = jb->row0 + r;
    int64_t m = row_component(jb->seed_rows, i, jb->M);
    const double *c = jb->centres + (size_t)m * D;
    for (int p = 0; 2 * p < D; ++p) {
      double z0, z1;
      row_noise_pair(jb->seed_rows, i, p, &z0, &z1);
      v[2 * p] = c[2 * p] + jb->sigma * z0;
      if (2 * p + 1 < D) v[2 * p + 1] = c[2 * p + 1] + jb->sigma * z1;
    }
    if (jb->kind == 0) {
      uint8_t *o = (uint8_t *)jb->out + (size_t)r * D;
      for (int j = 0; j < D; ++j) {
        double t = nearbyint(v[j]);
        if (t < 0.0) t = 0.0;
        if (t > 255.0) t = 255.0;
        o[j] = (uint8_t)t;
      }
    } else {
      float *o = (float *)jb->out + (size_t)r * D;
      double s = 0.0;
      for (int j = 0; j < D; ++j) s += v[j] * v[j];
      double inv = s > 0.0 ? 1.0 / sqrt(s) : 0.0;
      for (int j = 0; j < D; ++j) o[j] = (float)(v[j] * inv);
    }
  }
  free(v);
  return NULL;
}

static int run_parallel(job_t *proto, int nthreads) {
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  if (proto->n < 4096) nthreads = 1;
  pthread_t th[256];
  job_t jobs[256];
  int64_t per = (proto->n + nthreads - 1) / nthreads;
  int started = 0;
  for (int t = 0; t < nthreads; ++t) {
    jobs[t] = *proto;
    jobs[t].lo = (int64_t)t * per;
    jobs[t].hi = jobs[t].lo + per < proto->n ? jobs[t].lo + per : proto->n;
    if (jobs[t].lo >= jobs[t].hi) break;
    if (pthread_create(&th[t], NULL, run_rows, &jobs[t]) != 0) {
      run_rows(&jobs[t]);
      th[t] = 0;
    }
    started = t + 1;
  }
  for (int t = 0; t < started; ++t)
    if (th[t]) pthread_join(th[t], NULL);
  return 0;
}

/* Rows [row0, row0 + n) of the mixture. kind 0 = u8, 1 = f32 (normalised).
 * Returns 0, or -1 on bad arguments / allocation failure. */
int synth_mixture(int kind, uint64_t seed_rows, uint64_t seed_centres, int M, int D,
                  double sigma, int64_t row0, int64_t n, void *out, int nthreads) {
  if ((kind != 0 && kind != 1) || M < 1 || D < 1 || n < 0 || row0 < 0 || !out) return -1;
  if (n == 0) return 0;
  double *cent = (double *)malloc(sizeof(double) * (size_t)M * (size_t)D);
  if (!cent) return -1;
  for (int64_t m = 0; m < M; ++m)
    for (int j = 0; j < D; ++j)
      cent[(size_t)m * D + j] = kind == 0 ? centre_u8(seed_centres, m, j) : centre_f32(seed_centres, m, j);
  job_t jb;
  memset(&jb, 0, sizeof(jb));
  jb.kind = kind;
  jb.seed_rows = seed_rows;
  jb.seed_centres = seed_centres;
  jb.M = M;
  jb.D = D;
  jb.sigma = sigma;
  jb.row0 = row0;
  jb.n = n;
  jb.out = out;
  jb.centres = cent;
  run_parallel(&jb, nthreads);
  free(cent);
  return 0;
}

/* Component index of rows [row0, row0 + n) (for test diagnostics). */
int synth_components(uint64_t seed_rows, int M, int64_t row0, int64_t n, int32_t *out) {
  if (M < 1 || n < 0 || !out) return -1;
  for (int64_t r = 0; r < n; ++r) out[r] = (int32_t)row_component(seed_rows, row0 + r, M);
  return 0;
}

/* n draws of N(0, scale^2) as fp32: element e uses block e/2 of (seed, stream). */
int synth_normal(uint64_t seed, uint32_t stream, int64_t n, double scale, float *out) {
  if (n < 0 || !out) return -1;
  for (int64_t e = 0; e < n; e += 2) {
    uint32_t w[4];
    double z0, z1;
    int64_t p = e >> 1;
    philox((uint32_t)p, (uint32_t)((uint64_t)p >> 32), stream, 4u, seed, STREAM_NORMAL, w);
    box_muller(w, &z0, &z1);
    out[e] = (float)(scale * z0);
    if (e + 1 < n) out[e + 1] = (float)(scale * z1);
  }
  return 0;
}

/* Mixture centres [M x D] as doubles (kind 0 = u8, 1 = f32), the values every
 * row generator adds its noise to. */
int synth_centres(int kind, uint64_t seed_centres, int M, int D, double *out) {
  if ((kind != 0 && kind != 1) || M < 1 || D < 1 || !out) return -1;
  for (int64_t m = 0; m < M; ++m)
    for (int j = 0; j < D; ++j)
      out[(size_t)m * D + j] = kind == 0 ? centre_u8(seed_centres, m, j) : centre_f32(seed_centres, m, j);
  return 0;
}
