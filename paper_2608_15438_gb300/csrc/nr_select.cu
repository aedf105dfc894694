// K3 select: bucket lookup through the CSR directory (Sec. 3.3) and the
// centroid stage of Sec. 3.4.2 / Algorithm 2, one 128-thread CTA per query
// (nrq::select_block):
//   1. probe i -> cluster range [bkt_off[u_i], bkt_off[u_i + 1]) (range-checked);
//   2. every cluster c of every probed bucket gets its centroid distance
//      d_c = sum_j (l_j - mu_cj)^2 as a sequential fp32 fmaf chain over j;
//   3. buckets holding exactly one cluster go to C^dir; over the other clusters
//      d_min, the gate theta = d_min + fmaf(m1, d_min, m0), survivors d_c <= theta
//      (keys of C^dir and the survivors collected in shared memory by two
//      passes over the candidates, or, when they do not fit, all candidate
//      keys sorted in the query's global slab);
//   4. a bitonic sort of the 64-bit keys (d_c bits, c) of C^dir and the
//      survivors, the first C survivors kept (top-C by (d_c, c)), and the kept
//      list written in key order together with its refinement segments.
// Sorting by exact keys makes the result independent of thread scheduling.
#include <cuda_runtime.h>
#include <stdint.h>

#include <cmath>

#include "nr_internal.cuh"
#include "nrq_select.cuh"

namespace {

constexpr int kThreads = 128;

// MODE 0: the order-independent stage; MODE 1: the sequential stage
template <int MODE>
__global__ void __launch_bounds__(kThreads, MODE == 0 ? 6 : 1)
    select_kernel(nrq::SelectParams sp, const float *__restrict__ logits,
                  const uint32_t *__restrict__ codes, const int32_t *__restrict__ nprobe,
                  int32_t *L, int32_t *nL, nr_seg *seg, uint32_t *slen, int64_t *stats,
                  unsigned char *slab, size_t slab_bytes, unsigned *ovf) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int q = blockIdx.x, tid = threadIdx.x;
  const int Lmax = sp.P + sp.C;
  unsigned char *scratch = smem;
  const size_t sbytes = MODE == 1 ? nrq::select_seq_bytes(sp.P, sp.C, sp.b_batch)
                                   : nrq::select_scratch_bytes(sp.P, sp.K_max);
  float *slog = reinterpret_cast<float *>(smem + sbytes);
  int *warp_sums = reinterpret_cast<int *>(slog + 32);
  unsigned *sred = reinterpret_cast<unsigned *>(warp_sums + 32);
  const int np = nprobe[q];
  if (tid < sp.b) slog[tid] = logits[(size_t)q * sp.b + tid];
  __syncthreads();
  uint32_t total = 0;
  int scored = 0;
  unsigned char *qslab = slab ? slab + (size_t)q * slab_bytes : nullptr;
  const int nl =
      MODE == 1
          ? nrq::select_block_seq(sp, slog, codes + (size_t)q * sp.P, np, scratch, warp_sums, sred,
                                  seg + (size_t)q * Lmax, L ? L + (size_t)q * Lmax : nullptr, Lmax,
                                  &total, &scored)
          : nrq::select_block(sp, slog, codes + (size_t)q * sp.P, np, scratch, qslab, warp_sums,
                              sred, seg + (size_t)q * Lmax, L ? L + (size_t)q * Lmax : nullptr,
                              Lmax, &total, &scored);
  if (tid == 0) {
    if (nl < 0) {  // deferred: the overflow kernel writes its list
      const unsigned i = atomicAdd(&ovf[0], 1u);
      ovf[4 + 2 * (size_t)i] = (unsigned)q;
      ovf[4 + 2 * (size_t)i + 1] = (unsigned)scored;
    } else {
      nL[q] = nl;
      slen[q] = total;
    }
    if (stats) {
      if (nl >= 0) stats[(size_t)q * NR_QSTATS + 2] = nl;
      stats[(size_t)q * NR_QSTATS + 3] = np;
      stats[(size_t)q * NR_QSTATS + 4] = scored;
    }
  }
}

// The queries select deferred (more kept keys than its shared memory holds):
// persistent blocks of kSelOvfThreads take them from the list one at a time
// and finish their lists (nrq::select_overflow_block). ovf: [0] deferred
// queries, [1] queries taken, then (query, clusters in its slab) pairs.
__global__ void __launch_bounds__(nrq::kSelOvfThreads, 2)
    select_overflow_kernel(nrq::SelectParams sp, unsigned *ovf, unsigned char *slab,
                           size_t slab_bytes, int32_t *L, int32_t *nL, nr_seg *seg, uint32_t *slen,
                           int64_t *stats) {
  extern __shared__ __align__(16) unsigned char smem[];
  uint64_t *skeys = reinterpret_cast<uint64_t *>(smem);
  uint32_t *hist = reinterpret_cast<uint32_t *>(smem + (size_t)nrq::select_smem_keys(nrq::kSelOvfKeys) * 8);
  int *warp_sums = reinterpret_cast<int *>(hist + nrq::kSelOvfBuckets);
  unsigned *sctl = reinterpret_cast<unsigned *>(warp_sums + 32);
  unsigned *item = sctl + 4;  // the query a block works on; sctl[0..3] are select_overflow_block's
  const int Lmax = sp.P + sp.C;
  for (;;) {
    if (threadIdx.x == 0) {
      const unsigned i = atomicAdd(&ovf[1], 1u);
      *item = i < ovf[0] ? i : 0xffffffffu;
    }
    __syncthreads();
    const unsigned i = *item;
    if (i == 0xffffffffu) break;
    const int q = (int)ovf[4 + 2 * (size_t)i], M = (int)ovf[4 + 2 * (size_t)i + 1];
    uint32_t total = 0;
    const int nl = nrq::select_overflow_block(sp, slab + (size_t)q * slab_bytes, M, skeys, hist, sctl,
                                              warp_sums, seg + (size_t)q * Lmax,
                                              L ? L + (size_t)q * Lmax : nullptr, Lmax, &total);
    if (threadIdx.x == 0) {
      nL[q] = nl;
      slen[q] = total;
      if (stats) stats[(size_t)q * NR_QSTATS + 2] = nl;
    }
    __syncthreads();  // item and sctl are reused by the next query
  }
}

}  // namespace


nrq::SelectParams nr_select_params(nr_index *ix, int P, int C) {
  nrq::SelectParams sp;
  sp.b = ix->b;
  sp.K_max = ix->K_max;
  sp.P = P;
  sp.C = C;
  sp.n_cl = ix->n_cl;
  sp.N = ix->N;
  sp.bkt_off = ix->bkt_off;
  sp.cl_off = ix->cl_off;
  sp.cent = ix->cent;
  const float m0 = ix->params.gate_m0;
  sp.gate_n = ix->params.gate_n;
  for (int i = 0; i < 16; ++i) {
    sp.gate_x[i] = ix->params.gate_x[i];
    sp.gate_y[i] = ix->params.gate_y[i];
  }
  sp.gate_off = sp.gate_n < 2 && std::isinf(m0) && m0 > 0.0f;
  sp.m0 = m0;
  sp.m1 = ix->params.gate_m1;
  sp.err = ix->d_err;
  sp.mode = ix->params.cent_mode;
  sp.n_bins = ix->params.n_bins;
  sp.b_batch = ix->params.b_batch;
  sp.b_min = ix->params.b_min;
  sp.c_t_low = ix->params.c_t_low;
  sp.c_u_min = ix->params.c_u_min;
  sp.c_f_min = ix->params.c_f_min;
  sp.s_max = ix->params.s_max;
  sp.c_alpha_front = ix->params.c_alpha_front;
  sp.tau = ix->tau;
  return sp;
}

size_t nr_select_slab_bytes(int P, int K_max) { return nrq::select_slab_bytes(P, K_max); }

size_t nr_select_slab_total(int64_t nq, int P, int K_max) {
  const size_t per = nrq::select_slab_bytes(P, K_max);
  if (per == 0) return 0;
  // the slabs, then the deferred-query list: two counters, two spare words,
  // a (query, clusters) pair per query
  return (((size_t)nq * per + 255) & ~(size_t)255) + 16 + (size_t)nq * 8;
}

size_t nr_select_smem_bytes(const nr_index *ix, int P, int C) {
  const nr_params &p = ix->params;
  const size_t s = p.cent_mode == 1 ? nrq::select_seq_bytes(P, C, p.b_batch)
                                    : nrq::select_scratch_bytes(P, ix->K_max);
  return s + 32 * 4 + 32 * 4 + 16;
}

cudaError_t nr_launch_select(nr_index *ix, const float *d_logits, const uint32_t *d_codes,
                             const int32_t *d_nprobe, int64_t nq, int P, int C, int32_t *d_L,
                             int32_t *d_nL, nr_seg *d_seg, uint32_t *d_slen, int64_t *d_stats,
                             void *d_slab, cudaStream_t s) {
  if (nq <= 0) return cudaSuccess;
  const size_t smem = nr_select_smem_bytes(ix, P, C);
  const nrq::SelectParams sp = nr_select_params(ix, P, C);  // before the launch configuration
  const size_t slab_bytes = nrq::select_slab_bytes(P, ix->K_max);
  unsigned char *slab = static_cast<unsigned char *>(d_slab);
  unsigned *ovf = nullptr;  // the deferred-query list after the slabs
  cudaError_t e;
  if (slab && slab_bytes && sp.mode == 0) {
    ovf = reinterpret_cast<unsigned *>(slab + (((size_t)nq * slab_bytes + 255) & ~(size_t)255));
    e = cudaMemsetAsync(ovf, 0, 16, s);
    if (e != cudaSuccess) return e;
  }
  if (sp.mode == 1) {
    e = cudaFuncSetAttribute(select_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    select_kernel<1><<<(unsigned)nq, kThreads, smem, s>>>(sp, d_logits, d_codes, d_nprobe, d_L, d_nL,
                                                          d_seg, d_slen, d_stats, slab, slab_bytes,
                                                          nullptr);
  } else {
    e = cudaFuncSetAttribute(select_kernel<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    select_kernel<0><<<(unsigned)nq, kThreads, smem, s>>>(sp, d_logits, d_codes, d_nprobe, d_L, d_nL,
                                                          d_seg, d_slen, d_stats, slab, slab_bytes,
                                                          ovf);
    ix->launches += 1;
    e = cudaGetLastError();
    if (e != cudaSuccess || !ovf) return e;
    // the deferred queries (none at most budgets: its blocks exit at once)
    const size_t osm = nrq::select_overflow_smem_bytes();
    e = cudaFuncSetAttribute(select_overflow_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)osm);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, select_overflow_kernel,
                                                      nrq::kSelOvfThreads, osm);
    if (e != cudaSuccess) return e;
    int64_t grid = (int64_t)(per_sm > 0 ? per_sm : 1) * ix->num_sms;
    if (grid > nq) grid = nq;
    select_overflow_kernel<<<(unsigned)grid, nrq::kSelOvfThreads, osm, s>>>(sp, ovf, slab, slab_bytes,
                                                                          d_L, d_nL, d_seg, d_slen,
                                                                          d_stats);
  }
  ix->launches += 1;
  return cudaGetLastError();
}
