// K1 encode: l = E(x), one hidden layer (Sec. 3.2.1):
//   h = ReLU(W1 (s x) + b1),  l = W2 h + b2,  fp32 accumulation.
// CUDA-core version: QB queries per CTA share every weight load.
#include <cuda_runtime.h>
#include <stdint.h>

#include "nr_internal.cuh"

namespace {

constexpr int kQB = 8;
constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads)
    encode_simt_kernel(const void *__restrict__ x, int dtype, int D, int H, int b, float s,
                       const float *__restrict__ W1T, const float *__restrict__ b1,
                       const float *__restrict__ W2, const float *__restrict__ b2, int64_t nq,
                       float *__restrict__ out) {
  extern __shared__ float sm[];
  float *xs = sm;                  // [kQB][D]
  float *hs = sm + (size_t)kQB * D;  // [kQB][H]
  const int tid = threadIdx.x;
  const int64_t q0 = (int64_t)blockIdx.x * kQB;
  for (int i = tid; i < kQB * D; i += kThreads) {
    const int qi = i / D, j = i - qi * D;
    const int64_t qq = q0 + qi;
    float v = 0.0f;
    if (qq < nq)
      v = dtype == 0 ? (float)static_cast<const uint8_t *>(x)[qq * D + j]
                     : static_cast<const float *>(x)[qq * D + j];
    xs[i] = __fmul_rn(v, s);
  }
  __syncthreads();
  for (int u = tid; u < H; u += kThreads) {
    float acc[kQB];
#pragma unroll
    for (int qi = 0; qi < kQB; ++qi) acc[qi] = b1[u];
    for (int j = 0; j < D; ++j) {
      const float w = W1T[(size_t)j * H + u];
#pragma unroll
      for (int qi = 0; qi < kQB; ++qi) acc[qi] = __fmaf_rn(w, xs[qi * D + j], acc[qi]);
    }
#pragma unroll
    for (int qi = 0; qi < kQB; ++qi) hs[qi * H + u] = acc[qi] > 0.0f ? acc[qi] : 0.0f;
  }
  __syncthreads();
  for (int o = tid; o < kQB * b; o += kThreads) {
    const int qi = o / b, j = o - qi * b;
    const int64_t qq = q0 + qi;
    if (qq >= nq) continue;
    float acc = b2[j];
    const float *w = W2 + (size_t)j * H;
    for (int u = 0; u < H; ++u) acc = __fmaf_rn(w[u], hs[qi * H + u], acc);
    out[qq * b + j] = acc;
  }
}

}  // namespace

cudaError_t nr_launch_encode(nr_index *ix, const void *d_x, int64_t nq, float *d_logits,
                             cudaStream_t s) {
  if (nq <= 0) return cudaSuccess;
  const size_t smem = (size_t)kQB * (ix->D + ix->H) * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(encode_simt_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int64_t grid = (nq + kQB - 1) / kQB;
  encode_simt_kernel<<<(unsigned)grid, kThreads, smem, s>>>(d_x, ix->dtype, ix->D, ix->H, ix->b,
                                                             ix->in_scale, ix->W1T, ix->b1, ix->W2,
                                                             ix->b2, nq, d_logits);
  ix->launches += 1;
  return cudaGetLastError();
}
