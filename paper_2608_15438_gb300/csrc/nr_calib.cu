// Helpers for calibrating the centroid gate and the score cutoff (Sec. 3.4):
// where given ids are stored (their cluster and bucket), and centroid
// distances of queries to given clusters. Off the query path.
#include <cuda_runtime.h>
#include <stdint.h>

#include <cub/device/device_radix_sort.cuh>

#include "neuroute.h"
#include "nr_internal.cuh"

namespace {

__global__ void iota_kernel(uint32_t *v, int64_t n) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    v[i] = (uint32_t)i;
}

__global__ void key_kernel(const int64_t *__restrict__ ids, int64_t n, uint32_t *keys) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t v = ids[i];
    keys[i] = (v < 0 || v >= 0xFFFFFFFFll) ? 0xFFFFFFFFu : (uint32_t)v;  // never stored
  }
}

__global__ void fill_kernel(int32_t *out, int64_t n) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    out[i * 4 + 0] = -1;
    out[i * 4 + 1] = -1;
    out[i * 4 + 2] = -1;
    out[i * 4 + 3] = 0;
  }
}

// every stored row p: if its id is requested, record its cluster and bucket
// for each request of that id
__global__ void locate_kernel(const uint32_t *__restrict__ ids, int64_t N,
                              const uint32_t *__restrict__ cl_off, int64_t n_cl,
                              const uint32_t *__restrict__ bkt_off, int b,
                              const uint32_t *__restrict__ skeys, const uint32_t *__restrict__ sidx,
                              int64_t n, int32_t *out) {
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < N;
       p += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t id = ids[p];
    int64_t lo = 0, hi = n;  // first requested key >= id
    while (lo < hi) {
      const int64_t mid = (lo + hi) >> 1;
      if (skeys[mid] < id) lo = mid + 1;
      else hi = mid;
    }
    if (lo >= n || skeys[lo] != id) continue;
    int64_t a = 0, z = n_cl - 1;  // cluster: last c with cl_off[c] <= p
    while (a < z) {
      const int64_t mid = (a + z + 1) >> 1;
      if ((int64_t)cl_off[mid] <= p) a = mid;
      else z = mid - 1;
    }
    const int64_t nb = (int64_t)1 << b;
    int64_t u = 0, w = nb - 1;  // bucket: last u with bkt_off[u] <= c
    while (u < w) {
      const int64_t mid = (u + w + 1) >> 1;
      if ((int64_t)bkt_off[mid] <= a) u = mid;
      else w = mid - 1;
    }
    const uint32_t f = bkt_off[u], e = bkt_off[u + 1];
    for (int64_t t = lo; t < n && skeys[t] == id; ++t) {
      int32_t *o = out + (size_t)sidx[t] * 4;
      o[0] = (int32_t)a;
      o[1] = (int32_t)u;
      o[2] = (int32_t)f;
      o[3] = (int32_t)(e - f);
    }
  }
}

// d_c = sum_j (l_j - mu_cj)^2 as a sequential fmaf chain (the select kernel's)
__global__ void cent_dist_kernel(const float *__restrict__ logits, int64_t nq, int b,
                                 const int32_t *__restrict__ clusters, int m,
                                 const float *__restrict__ cent, int64_t n_cl, float *out) {
  const int64_t total = nq * (int64_t)m;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int64_t q = t / m;
    const int32_t c = clusters[t];
    float acc = __int_as_float(0x7f800000);
    if (c >= 0 && c < n_cl) {
      acc = 0.0f;
      const float *mu = cent + (size_t)c * b;
      const float *l = logits + (size_t)q * b;
      for (int j = 0; j < b; ++j) {
        const float d = __fsub_rn(l[j], mu[j]);
        acc = __fmaf_rn(d, d, acc);
      }
    }
    out[t] = acc;
  }
}

int grid_for(int64_t work, int sms) {
  int64_t g = (work + 255) / 256;
  if (g > (int64_t)sms * 16) g = (int64_t)sms * 16;
  return g < 1 ? 1 : (int)g;
}

}  // namespace

extern "C" {

nr_status nr_index_locate(nr_index *ix, const int64_t *d_ids, int64_t n, int32_t *d_out,
                          void *stream) {
  if (!ix || n < 0 || n > ((int64_t)1 << 31) - 1) return NR_ERR_INVALID_ARG;
  if (n == 0) return NR_OK;
  if (!d_ids || !d_out) return NR_ERR_INVALID_ARG;
  DeviceGuard g(ix->device);
  cudaStream_t s = (cudaStream_t)stream;
  uint32_t *keys = nullptr, *idx = nullptr, *skeys = nullptr, *sidx = nullptr;
  void *tmp = nullptr;
  size_t tb = 0;
  nr_status st = NR_OK;
  auto fail = [&](cudaError_t e) {
    if (st == NR_OK && e != cudaSuccess) st = cuda_status(e);
    return st != NR_OK;
  };
  if (!fail(cudaMalloc((void **)&keys, (size_t)n * 4)) && !fail(cudaMalloc((void **)&idx, (size_t)n * 4)) &&
      !fail(cudaMalloc((void **)&skeys, (size_t)n * 4)) && !fail(cudaMalloc((void **)&sidx, (size_t)n * 4))) {
    const int sms = ix->num_sms > 0 ? ix->num_sms : 1;
    key_kernel<<<grid_for(n, sms), 256, 0, s>>>(d_ids, n, keys);
    iota_kernel<<<grid_for(n, sms), 256, 0, s>>>(idx, n);
    fill_kernel<<<grid_for(n, sms), 256, 0, s>>>(d_out, n);
    if (!fail(cudaGetLastError()) &&
        !fail(cub::DeviceRadixSort::SortPairs(nullptr, tb, keys, skeys, idx, sidx, n, 0, 32, s)) &&
        !fail(cudaMalloc(&tmp, tb > 0 ? tb : 16)) &&
        !fail(cub::DeviceRadixSort::SortPairs(tmp, tb, keys, skeys, idx, sidx, n, 0, 32, s))) {
      locate_kernel<<<grid_for(ix->N, sms), 256, 0, s>>>(ix->ids, ix->N, ix->cl_off, ix->n_cl,
                                                         ix->bkt_off, ix->b, skeys, sidx, n, d_out);
      fail(cudaGetLastError());
      fail(cudaStreamSynchronize(s));
    }
  }
  for (void *p : {(void *)keys, (void *)idx, (void *)skeys, (void *)sidx, tmp})
    if (p) cudaFree(p);
  return st;
}

nr_status nr_centroid_dists(nr_index *ix, const float *d_logits, int64_t nq,
                            const int32_t *d_clusters, int m, float *d_out, void *stream) {
  if (!ix || nq < 0 || m < 0) return NR_ERR_INVALID_ARG;
  if (nq == 0 || m == 0) return NR_OK;
  if (!d_logits || !d_clusters || !d_out) return NR_ERR_INVALID_ARG;
  DeviceGuard g(ix->device);
  const int sms = ix->num_sms > 0 ? ix->num_sms : 1;
  cent_dist_kernel<<<grid_for(nq * (int64_t)m, sms), 256, 0, (cudaStream_t)stream>>>(
      d_logits, nq, ix->b, d_clusters, m, ix->cent, ix->n_cl, d_out);
  return cuda_status(cudaGetLastError());
}

}  // extern "C"
