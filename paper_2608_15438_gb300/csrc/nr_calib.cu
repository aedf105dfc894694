// Calibration of the centroid gate M(x) and the bucket-score cutoff S_max
// (Sec. 3.4), off the query path: where given ids are stored (their cluster
// and bucket), centroid distances of queries to given clusters, the
// observations (each target's bucket score; per query x and y) on the GPU,
// and the two fits on the host.
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <cmath>
#include <limits>
#include <utility>
#include <vector>

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

// The bucket enumeration's cost of bucket codes[q k + t] for query q
// (Algorithm 1): deviations delta_j = |l_j - tau_j|, ranks by (delta_j, j),
// the fp32 sum of delta over the ranks whose bit differs from the base code,
// in ascending rank; NaN for a negative code. One warp per query.
__device__ __forceinline__ void warp_ranks(const float *l, const float *tau, int b, float *sdel,
                                           int *sbit, uint32_t *u0) {
  const int lane = threadIdx.x & 31;
  float dj = __int_as_float(0x7f800000);
  bool bit = false;
  if (lane < b) {
    bit = l[lane] >= tau[lane];
    dj = fabsf(__fsub_rn(l[lane], tau[lane]));
  }
  *u0 = __ballot_sync(0xffffffffu, bit);
  int rank = 0;
  for (int i = 0; i < b; ++i) {
    const float di = __shfl_sync(0xffffffffu, dj, i);
    if (di < dj || (di == dj && i < lane)) ++rank;
  }
  if (lane < b) {
    sdel[rank] = dj;
    sbit[rank] = lane;
  }
  __syncwarp();
}

__device__ __forceinline__ float code_cost(uint32_t diff, const float *sdel, const int *sbit, int b) {
  float s = 0.0f;
  for (int r = 0; r < b; ++r)
    if ((diff >> sbit[r]) & 1u) s = __fadd_rn(s, sdel[r]);
  return s;
}

constexpr int kObsWarps = 4;

__global__ void bucket_scores_kernel(const float *__restrict__ logits, const float *__restrict__ tau,
                                     int b, const int32_t *__restrict__ codes, int64_t nq, int k,
                                     float *__restrict__ scores) {
  __shared__ float sdel[kObsWarps][32];
  __shared__ int sbit[kObsWarps][32];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t q = (int64_t)blockIdx.x * kObsWarps + w;
  if (q >= nq) return;  // uniform per warp
  uint32_t u0;
  warp_ranks(logits + q * b, tau, b, sdel[w], sbit[w], &u0);
  for (int t = lane; t < k; t += 32) {
    const int32_t c = codes[q * k + t];
    scores[q * k + t] = c < 0 ? __int_as_float(0x7fc00000)
                              : code_cost((uint32_t)c ^ u0, sdel[w], sbit[w], b);
  }
}

// Observations of the calibration from the targets' locations loc [nq k][4]
// (cluster, bucket code, first cluster of the bucket, clusters in it; -1 when
// the id is not stored): scores[q k + t] the bucket score of target t (NaN
// when not stored); over the targets whose bucket holds two or more clusters,
// x[q] = the smallest centroid distance of every cluster of those buckets and
// y[q] = the largest distance of such a target's own cluster minus x[q]
// (NaN, NaN without one). Distances are the select kernel's fmaf chain.
__global__ void observe_kernel(const float *__restrict__ logits, const float *__restrict__ tau,
                               int b, const int32_t *__restrict__ loc, int64_t nq, int k,
                               const float *__restrict__ cent, int64_t n_cl,
                               float *__restrict__ scores, float *__restrict__ xo,
                               float *__restrict__ yo) {
  __shared__ float sdel[kObsWarps][32];
  __shared__ int sbit[kObsWarps][32];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t q = (int64_t)blockIdx.x * kObsWarps + w;
  if (q >= nq) return;  // uniform per warp
  const float *l = logits + q * b;
  uint32_t u0;
  warp_ranks(l, tau, b, sdel[w], sbit[w], &u0);
  const float inf = __int_as_float(0x7f800000);
  float best = inf, far = -inf;
  for (int t = lane; t < k; t += 32) {
    const int32_t *o = loc + (q * k + t) * 4;
    const int32_t c = o[0], u = o[1], first = o[2], count = o[3];
    scores[q * k + t] = c < 0 ? __int_as_float(0x7fc00000)
                              : code_cost((uint32_t)u ^ u0, sdel[w], sbit[w], b);
    if (c < 0 || count < 2) continue;
    for (int32_t cc = first; cc < first + count; ++cc) {
      float d = inf;
      if (cc >= 0 && cc < n_cl) {
        d = 0.0f;
        const float *mu = cent + (size_t)cc * b;
        for (int j = 0; j < b; ++j) {
          const float e = __fsub_rn(l[j], mu[j]);
          d = __fmaf_rn(e, e, d);
        }
      }
      best = fminf(best, d);
      if (cc == c) far = fmaxf(far, d);
    }
  }
  for (int o = 16; o > 0; o >>= 1) {
    best = fminf(best, __shfl_xor_sync(0xffffffffu, best, o));
    far = fmaxf(far, __shfl_xor_sync(0xffffffffu, far, o));
  }
  if (lane == 0) {
    const bool has = far > -inf;
    xo[q] = has ? best : __int_as_float(0x7fc00000);
    yo[q] = has ? __fsub_rn(far, best) : __int_as_float(0x7fc00000);
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

nr_status nr_bucket_scores(const float *d_logits, const float *d_tau, int b, const int32_t *d_codes,
                           int64_t nq, int k, float *d_scores, void *stream) {
  if (b < 1 || b > 31 || nq < 0 || k < 1 || nq > ((int64_t)1 << 31) - 1) return NR_ERR_INVALID_ARG;
  if (nq == 0) return NR_OK;
  if (!d_logits || !d_tau || !d_codes || !d_scores) return NR_ERR_INVALID_ARG;
  const int64_t grid = (nq + kObsWarps - 1) / kObsWarps;
  bucket_scores_kernel<<<(unsigned)grid, 32 * kObsWarps, 0, (cudaStream_t)stream>>>(
      d_logits, d_tau, b, d_codes, nq, k, d_scores);
  return cuda_status(cudaGetLastError());
}

nr_status nr_calib_observe(nr_index *ix, const float *d_logits, const int64_t *d_targets, int64_t nq,
                           int k, float *d_scores, float *d_x, float *d_y, void *stream) {
  if (!ix || nq < 0 || k < 1 || nq * (int64_t)k > ((int64_t)1 << 31) - 1) return NR_ERR_INVALID_ARG;
  if (nq == 0) return NR_OK;
  if (!d_logits || !d_targets || !d_scores || !d_x || !d_y) return NR_ERR_INVALID_ARG;
  DeviceGuard g(ix->device);
  cudaStream_t s = (cudaStream_t)stream;
  int32_t *loc = nullptr;
  if (cudaMalloc((void **)&loc, (size_t)nq * k * 4 * sizeof(int32_t)) != cudaSuccess) {
    cudaGetLastError();
    return NR_ERR_OOM;
  }
  nr_status st = nr_index_locate(ix, d_targets, nq * k, loc, stream);
  if (st == NR_OK) {
    const int64_t grid = (nq + kObsWarps - 1) / kObsWarps;
    observe_kernel<<<(unsigned)grid, 32 * kObsWarps, 0, s>>>(d_logits, ix->tau, ix->b, loc, nq, k,
                                                             ix->cent, ix->n_cl, d_scores, d_x, d_y);
    st = cuda_status(cudaGetLastError());
    if (st == NR_OK) st = cuda_status(cudaStreamSynchronize(s));
  }
  cudaFree(loc);
  return st;
}

// S_max: the pair scores (NaN skipped) sorted, the entry at position
// ceil(coverage m) - 1 (clamped to [0, m - 1]); the fraction of pairs at or
// below it, and of queries with a score all of whose scores are.
nr_status nr_calib_fit_s_max(const float *h_scores, int64_t nq, int k, double coverage,
                             float *s_max, double *pair_coverage, double *query_coverage) {
  if (!h_scores || nq < 0 || k < 1 || !s_max || !pair_coverage || !query_coverage)
    return NR_ERR_INVALID_ARG;
  std::vector<float> flat;
  flat.reserve((size_t)nq * k);
  for (int64_t i = 0; i < nq * (int64_t)k; ++i)
    if (!std::isnan(h_scores[i])) flat.push_back(h_scores[i]);
  const int64_t m = (int64_t)flat.size();
  *s_max = std::numeric_limits<float>::quiet_NaN();
  *pair_coverage = 0.0;
  *query_coverage = 0.0;
  if (m == 0) return NR_OK;
  std::sort(flat.begin(), flat.end());
  int64_t pos = (int64_t)std::ceil(coverage * (double)m) - 1;
  pos = std::min<int64_t>(m - 1, std::max<int64_t>(0, pos));
  const float t = flat[(size_t)pos];
  int64_t within = 0;
  for (float v : flat) within += v <= t ? 1 : 0;
  int64_t with = 0, covered = 0;
  for (int64_t q = 0; q < nq; ++q) {
    bool any = false, all = true;
    for (int j = 0; j < k; ++j) {
      const float v = h_scores[q * k + j];
      if (std::isnan(v)) continue;
      any = true;
      all = all && v <= t;
    }
    if (any) {
      ++with;
      covered += all ? 1 : 0;
    }
  }
  *s_max = t;
  *pair_coverage = (double)within / (double)m;
  *query_coverage = (double)covered / (double)with;
  return NR_OK;
}

// M(x): the queries with an x sorted by (x, y) into B = min(n_bins, n)
// equal-frequency bins [floor(i n / B), floor((i + 1) n / B)); a bin's point is
// (x at its lower-median position, its y's order statistic ceil(q m) - 1);
// equal x merge (larger y); the ys' running maximum; one point becomes the
// flat curve through (x0, y0) and (the next float above x0, y0).
nr_status nr_calib_fit_gate(const float *h_x, const float *h_y, int64_t n, int n_bins, double q,
                            int *gate_n, float *gate_x, float *gate_y) {
  if (!h_x || !h_y || n < 0 || n_bins < 1 || n_bins > 16 || !gate_n || !gate_x || !gate_y)
    return NR_ERR_INVALID_ARG;
  std::vector<std::pair<float, float>> obs;
  for (int64_t i = 0; i < n; ++i)
    if (!std::isnan(h_x[i])) obs.push_back({h_x[i], h_y[i]});
  *gate_n = 0;
  const int64_t m0 = (int64_t)obs.size();
  if (m0 == 0) return NR_OK;
  std::sort(obs.begin(), obs.end());
  const int64_t B = std::min<int64_t>(n_bins, m0);
  std::vector<float> px, py;
  for (int64_t i = 0; i < B; ++i) {
    const int64_t lo = i * m0 / B, hi = (i + 1) * m0 / B, m = hi - lo;
    const float xm = obs[(size_t)(lo + (m - 1) / 2)].first;
    std::vector<float> ys;
    for (int64_t t = lo; t < hi; ++t) ys.push_back(obs[(size_t)t].second);
    std::sort(ys.begin(), ys.end());
    int64_t pos = (int64_t)std::ceil(q * (double)m) - 1;
    pos = std::min<int64_t>(m - 1, std::max<int64_t>(0, pos));
    const float yq = ys[(size_t)pos];
    if (!px.empty() && px.back() == xm) {
      py.back() = std::max(py.back(), yq);
    } else {
      px.push_back(xm);
      py.push_back(yq);
    }
  }
  for (size_t i = 1; i < py.size(); ++i) py[i] = std::max(py[i], py[i - 1]);
  if (px.size() == 1) {
    px.push_back(std::nextafter(px[0], std::numeric_limits<float>::infinity()));
    py.push_back(py[0]);
  }
  *gate_n = (int)px.size();
  for (size_t i = 0; i < px.size(); ++i) {
    gate_x[i] = px[i];
    gate_y[i] = py[i];
  }
  return NR_OK;
}

nr_status nr_calibrate(nr_index *ix, const float *d_logits, const int64_t *d_targets, int64_t nq,
                       int k, int n_bins, double quantile, double coverage, nr_params *p,
                       double *info, void *stream) {
  if (!ix || !p || nq < 1 || k < 1 || n_bins < 1 || n_bins > 16) return NR_ERR_INVALID_ARG;
  if (nq * (int64_t)k > ((int64_t)1 << 31) - 1) return NR_ERR_INVALID_ARG;
  DeviceGuard g(ix->device);
  float *d = nullptr;
  const size_t nsc = (size_t)nq * k;
  if (cudaMalloc((void **)&d, (nsc + 2 * (size_t)nq) * sizeof(float)) != cudaSuccess) {
    cudaGetLastError();
    return NR_ERR_OOM;
  }
  nr_status st = nr_calib_observe(ix, d_logits, d_targets, nq, k, d, d + nsc, d + nsc + nq, stream);
  std::vector<float> h(nsc + 2 * (size_t)nq);
  if (st == NR_OK)
    st = cuda_status(cudaMemcpy(h.data(), d, h.size() * sizeof(float), cudaMemcpyDeviceToHost));
  cudaFree(d);
  if (st != NR_OK) return st;
  float smax;
  double pc, qc;
  int gn;
  float gx[16], gy[16];
  st = nr_calib_fit_s_max(h.data(), nq, k, coverage, &smax, &pc, &qc);
  if (st == NR_OK) st = nr_calib_fit_gate(h.data() + nsc, h.data() + nsc + nq, nq, n_bins, quantile, &gn, gx, gy);
  if (st != NR_OK) return st;
  if (!std::isnan(smax)) p->s_max = smax;
  if (gn >= 2) {
    p->gate_n = gn;
    for (int i = 0; i < 16; ++i) {
      p->gate_x[i] = i < gn ? gx[i] : 0.0f;
      p->gate_y[i] = i < gn ? gy[i] : 0.0f;
    }
  }
  if (info) {
    int64_t gated = 0;
    for (int64_t i = 0; i < nq; ++i) gated += std::isnan(h[nsc + (size_t)i]) ? 0 : 1;
    info[0] = pc;
    info[1] = qc;
    info[2] = (double)gated;
  }
  return NR_OK;
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
