/*
 * Seeded synthetic mixture rows generated on the GPU: the same definition as
 * synth.c (Philox4x32-10 counters, double-precision Box-Muller, rint and clip
 * for uint8 rows, normalisation for fp32 rows), for workloads whose base is
 * too large to generate on the host. The mixture centres come from synth.c
 * (synth_centres) and are passed in.
 *
 * log, sqrt, sin and cos are CUDA's double-precision functions; where they
 * differ from the host C library in the last bit, a uint8 value can differ
 * only when c + sigma z falls within that bit of a half-integer, and an fp32
 * value by one rounding step.
 *
 * Holds none of the search method's arithmetic.
 */
#include <cuda_runtime.h>
#include <stdint.h>

#define PHILOX_M0 0xD2511F53u
#define PHILOX_M1 0xCD9E8D57u
#define PHILOX_W0 0x9E3779B9u
#define PHILOX_W1 0xBB67AE85u
#define STREAM_ROWS 0x524F5753u

namespace {

__device__ __forceinline__ void philox(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                       uint64_t seed, uint32_t stream, uint32_t out[4]) {
  uint32_t k0 = (uint32_t)seed ^ (uint32_t)(seed >> 32), k1 = stream;
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t hi0 = __umulhi(PHILOX_M0, c0), lo0 = PHILOX_M0 * c0;
    const uint32_t hi1 = __umulhi(PHILOX_M1, c2), lo1 = PHILOX_M1 * c2;
    const uint32_t n0 = hi1 ^ c1 ^ k0, n1 = lo1, n2 = hi0 ^ c3 ^ k1, n3 = lo0;
    c0 = n0;
    c1 = n1;
    c2 = n2;
    c3 = n3;
    k0 += PHILOX_W0;
    k1 += PHILOX_W1;
  }
  out[0] = c0;
  out[1] = c1;
  out[2] = c2;
  out[3] = c3;
}

__device__ __forceinline__ double u53(uint32_t hi, uint32_t lo) {
  const uint64_t v = (((uint64_t)hi << 32) | lo) >> 11;
  return __dmul_rn((double)v, 1.0 / 9007199254740992.0);
}

__device__ __forceinline__ void box_muller(const uint32_t w[4], double *z0, double *z1) {
  const double u1 = __dsub_rn(1.0, u53(w[0], w[1]));
  const double u2 = u53(w[2], w[3]);
  const double r = sqrt(__dmul_rn(-2.0, log(u1)));
  const double a = __dmul_rn(6.283185307179586476925, u2);
  *z0 = __dmul_rn(r, cos(a));
  *z1 = __dmul_rn(r, sin(a));
}

__device__ __forceinline__ int64_t row_component(uint64_t seed, int64_t i, int M) {
  uint32_t w[4];
  philox((uint32_t)i, (uint32_t)((uint64_t)i >> 32), 0xFFFFFFFFu, 1u, seed, STREAM_ROWS, w);
  const int64_t m = (int64_t)__dmul_rn(u53(w[0], w[1]), (double)M);
  return m < M ? m : M - 1;
}

// uint8 rows: one thread per (row, coordinate pair)
__global__ void mixture_u8_kernel(uint64_t seed, int M, int D, double sigma, int64_t row0, int64_t n,
                                  const double *__restrict__ cent, uint8_t *out) {
  const int pairs = (D + 1) / 2;
  const int64_t total = n * pairs;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = t / pairs;
    const int p = (int)(t - r * pairs);
    const int64_t i = row0 + r;
    const double *c = cent + (size_t)row_component(seed, i, M) * D;
    uint32_t w[4];
    philox((uint32_t)i, (uint32_t)((uint64_t)i >> 32), (uint32_t)p, 0u, seed, STREAM_ROWS, w);
    double z[2];
    box_muller(w, &z[0], &z[1]);
    for (int h = 0; h < 2; ++h) {
      const int j = 2 * p + h;
      if (j >= D) break;
      double v = rint(__dadd_rn(c[j], __dmul_rn(sigma, z[h])));
      v = v < 0.0 ? 0.0 : (v > 255.0 ? 255.0 : v);
      out[(size_t)r * D + j] = (uint8_t)v;
    }
  }
}

// fp32 rows: one warp per row; lane 0 sums the squares in coordinate order
__global__ void mixture_f32_kernel(uint64_t seed, int M, int D, double sigma, int64_t row0, int64_t n,
                                   const double *__restrict__ cent, float *out) {
  extern __shared__ double sv[];  // [warps per block][D]
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  double *v = sv + (size_t)wib * D;
  const int64_t nw = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t r = (int64_t)blockIdx.x * (blockDim.x >> 5) + wib; r < n; r += nw) {
    const int64_t i = row0 + r;
    const double *c = cent + (size_t)row_component(seed, i, M) * D;
    for (int p = lane; 2 * p < D; p += 32) {
      uint32_t w[4];
      philox((uint32_t)i, (uint32_t)((uint64_t)i >> 32), (uint32_t)p, 0u, seed, STREAM_ROWS, w);
      double z0, z1;
      box_muller(w, &z0, &z1);
      v[2 * p] = __dadd_rn(c[2 * p], __dmul_rn(sigma, z0));
      if (2 * p + 1 < D) v[2 * p + 1] = __dadd_rn(c[2 * p + 1], __dmul_rn(sigma, z1));
    }
    __syncwarp();
    double inv = 0.0;
    if (lane == 0) {
      double s = 0.0;
      for (int j = 0; j < D; ++j) s = __dadd_rn(s, __dmul_rn(v[j], v[j]));
      inv = s > 0.0 ? __ddiv_rn(1.0, sqrt(s)) : 0.0;
    }
    inv = __shfl_sync(0xffffffffu, inv, 0);
    for (int j = lane; j < D; j += 32) out[(size_t)r * D + j] = __double2float_rn(__dmul_rn(v[j], inv));
    __syncwarp();
  }
}

}  // namespace

extern "C" {

/* Rows [row0, row0 + n) of the mixture into d_out ([n x D] uint8 for kind 0,
 * fp32 for kind 1), with d_centres [M x D] doubles from synth_centres.
 * Enqueued on `stream`. Returns 0, or -1 on bad arguments or a launch error. */
int synth_mixture_cuda(int kind, uint64_t seed_rows, int M, int D, double sigma, int64_t row0,
                       int64_t n, const double *d_centres, void *d_out, void *stream) {
  if ((kind != 0 && kind != 1) || M < 1 || D < 1 || D > 4096 || n < 0 || row0 < 0 || !d_centres ||
      !d_out)
    return -1;
  if (n == 0) return 0;
  cudaStream_t s = (cudaStream_t)stream;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (sms < 1) sms = 1;
  if (kind == 0) {
    mixture_u8_kernel<<<sms * 16, 256, 0, s>>>(seed_rows, M, D, sigma, row0, n, d_centres,
                                               static_cast<uint8_t *>(d_out));
  } else {
    // warps per block: as many (up to 8) as the default 48 KB of shared memory
    // holds rows of D doubles; the values do not depend on it
    int wpb = (int)((48 * 1024) / ((size_t)D * sizeof(double)));
    wpb = wpb < 1 ? 1 : (wpb > 8 ? 8 : wpb);
    const size_t smem = (size_t)wpb * D * sizeof(double);
    mixture_f32_kernel<<<sms * 8, 32 * wpb, smem, s>>>(seed_rows, M, D, sigma, row0, n, d_centres,
                                                       static_cast<float *>(d_out));
  }
  return cudaGetLastError() == cudaSuccess ? 0 : -1;
}

}  // extern "C"
