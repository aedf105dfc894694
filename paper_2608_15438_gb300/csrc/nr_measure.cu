// nr_measure_gather: the rate at which this GPU reads rows at random, the
// bound of a kernel whose bytes are random row gathers (the centroid stage
// reads one centroid row per scored cluster from anywhere in a multi-GB
// array), as the copy bandwidth bounds a stream. nr_measure_read: the rate
// of a pure sequential read (no writes), the bound of a kernel whose bytes
// are reads of long runs (the refinement). Neither is part of the search path.
#include <cuda_runtime.h>
#include <stdint.h>

#include "neuroute.h"
#include "nr_internal.cuh"

namespace {

// splitmix64 finaliser: a well-mixed 64-bit value for each gather number
__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ull;
  z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;
  return z ^ (z >> 31);
}

// One row per thread at a random index below `rows`; each 16-byte piece of
// the row is read once; out[i] keeps the reads live.
__global__ void gather_kernel(const uint4 *__restrict__ a, int64_t rows, int q16, int64_t n,
                              uint64_t seed, uint32_t *__restrict__ out) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const uint64_t r = mix64(seed + (uint64_t)i) % (uint64_t)rows;
  const uint4 *p = a + r * (uint64_t)q16;
  uint32_t s = 0;
  for (int q = 0; q < q16; ++q) {
    const uint4 v = __ldg(p + q);
    s += v.x ^ v.y ^ v.z ^ v.w;
  }
  out[i] = s;
}

// Sequential read of n16 16-byte words, grid-stride with four loads in flight
// a thread (each vector folded on its own: an expression mixing the four
// vectors measured 30% slower); one word a thread out keeps the reads live.
__global__ void read_kernel(const uint4 *__restrict__ a, int64_t n16, uint32_t *__restrict__ out) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  uint32_t s = 0;
  for (; i + 3 * stride < n16; i += 4 * stride) {
    uint4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) v[u] = __ldg(a + i + u * stride);
#pragma unroll
    for (int u = 0; u < 4; ++u) s += v[u].x ^ v[u].y ^ v[u].z ^ v[u].w;
  }
  for (; i < n16; i += stride) {
    const uint4 v = __ldg(a + i);
    s += v.x ^ v.y ^ v.z ^ v.w;
  }
  out[(int64_t)blockIdx.x * blockDim.x + threadIdx.x] = s;
}

}  // namespace

extern "C" nr_status nr_measure_read(int device, int64_t bytes, int reps, double *h_gbs) {
  if (!h_gbs || bytes < ((int64_t)1 << 20) || bytes % 16 != 0 || reps < 1) return NR_ERR_INVALID_ARG;
  DeviceGuard g(device);
  if (!g.ok) return NR_ERR_CUDA;
  int sms = 0;
  cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
  const int threads = 512, blocks = (sms > 0 ? sms : 1) * 4;
  const size_t flush_bytes = (size_t)512 << 20;
  void *a = nullptr, *out = nullptr, *flush = nullptr;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  if (e == cudaSuccess) e = cudaMalloc(&a, (size_t)bytes);
  if (e == cudaSuccess) e = cudaMalloc(&out, (size_t)blocks * threads * 4);
  if (e == cudaSuccess) e = cudaMalloc(&flush, flush_bytes);
  if (e == cudaSuccess) e = cudaMemset(a, 1, (size_t)bytes);
  if (e == cudaSuccess) e = cudaEventCreate(&e0);
  if (e == cudaSuccess) e = cudaEventCreate(&e1);
  float best = -1.0f;
  for (int it = 0; it < reps && e == cudaSuccess; ++it) {
    e = cudaMemsetAsync(flush, it & 0xff, flush_bytes, 0);  // evict L2
    if (e == cudaSuccess) e = cudaEventRecord(e0, 0);
    if (e == cudaSuccess) {
      read_kernel<<<blocks, threads>>>(static_cast<const uint4 *>(a), bytes / 16, static_cast<uint32_t *>(out));
      e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaEventRecord(e1, 0);
    if (e == cudaSuccess) e = cudaEventSynchronize(e1);
    float ms = 0.0f;
    if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, e0, e1);
    if (e == cudaSuccess && (best < 0.0f || ms < best)) best = ms;
  }
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  if (a) cudaFree(a);
  if (out) cudaFree(out);
  if (flush) cudaFree(flush);
  if (e != cudaSuccess) return cuda_status(e);
  *h_gbs = (double)bytes / (best / 1e3) / 1e9;
  return NR_OK;
}

extern "C" nr_status nr_measure_gather(int device, int64_t rows, int row_bytes, int64_t n, int reps,
                                       double *h_gbs) {
  if (!h_gbs || rows < 1 || n < 1 || reps < 1 || row_bytes < 16 || row_bytes > 1024 ||
      row_bytes % 16 != 0 || n > ((int64_t)1 << 31) * 256)
    return NR_ERR_INVALID_ARG;
  DeviceGuard g(device);
  if (!g.ok) return NR_ERR_CUDA;
  const size_t arr = (size_t)rows * row_bytes, flush_bytes = (size_t)512 << 20;
  void *a = nullptr, *out = nullptr, *flush = nullptr;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  cudaError_t e = cudaMalloc(&a, arr);
  if (e == cudaSuccess) e = cudaMalloc(&out, (size_t)n * 4);
  if (e == cudaSuccess) e = cudaMalloc(&flush, flush_bytes);
  if (e == cudaSuccess) e = cudaMemset(a, 0, arr);
  if (e == cudaSuccess) e = cudaEventCreate(&e0);
  if (e == cudaSuccess) e = cudaEventCreate(&e1);
  float best = -1.0f;
  const int threads = 256;
  const int64_t blocks = (n + threads - 1) / threads;
  for (int it = 0; it < reps && e == cudaSuccess; ++it) {
    e = cudaMemsetAsync(flush, it & 0xff, flush_bytes, 0);  // evict L2
    if (e == cudaSuccess) e = cudaEventRecord(e0, 0);
    if (e == cudaSuccess) {
      gather_kernel<<<(unsigned)blocks, threads>>>(static_cast<const uint4 *>(a), rows, row_bytes / 16,
                                                    n, 0x9e3779b97f4a7c15ull * (uint64_t)(it + 1),
                                                    static_cast<uint32_t *>(out));
      e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaEventRecord(e1, 0);
    if (e == cudaSuccess) e = cudaEventSynchronize(e1);
    float ms = 0.0f;
    if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, e0, e1);
    if (e == cudaSuccess && (best < 0.0f || ms < best)) best = ms;
  }
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  if (a) cudaFree(a);
  if (out) cudaFree(out);
  if (flush) cudaFree(flush);
  if (e != cudaSuccess) return cuda_status(e);
  *h_gbs = (double)n * row_bytes / (best / 1e3) / 1e9;
  return NR_OK;
}
