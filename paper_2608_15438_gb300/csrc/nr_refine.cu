// K4 refine (Sec. 3.4, Algorithm 2's T_low rule; uint8 distances kept as
// integers, Sec. 4.1.1): persistent CTAs pull queries from an atomic counter
// and run nrq::refine_block on the segments K3 wrote to global memory.
//
// Launch shapes measured on GB300 (u8-10m / f32-10m operating points): the
// scan is limited by how many queries stream concurrently per SM, so tiles are
// small (128 uint8 rows, 32-64 fp32 rows), two stages deep, and registers are
// capped for many CTAs per SM.
#include <cuda_runtime.h>
#include <stdint.h>

#include "nr_internal.cuh"
#include "nrq_refine.cuh"

namespace {

// Longest streams first: one CTA buckets the queries by stream length
// (1024 buckets scaled to the longest stream) and writes them in decreasing
// bucket order, so the persistent refinement CTAs finish together instead of
// waiting on a long query picked up last. Order inside a bucket is arbitrary;
// it does not affect any result.
constexpr int kOrderBins = 1024;

__global__ void __launch_bounds__(1024) order_kernel(const uint32_t *__restrict__ slen, int64_t nq,
                                                     int32_t *__restrict__ perm) {
  __shared__ unsigned int hist[kOrderBins];
  __shared__ unsigned int smax;
  const int tid = threadIdx.x;
  if (tid == 0) smax = 1;
  for (int i = tid; i < kOrderBins; i += blockDim.x) hist[i] = 0;
  __syncthreads();
  unsigned int m = 1;
  for (int64_t q = tid; q < nq; q += blockDim.x) m = max(m, slen[q]);
  atomicMax(&smax, m);
  __syncthreads();
  const uint64_t top = (uint64_t)smax + 1;
  for (int64_t q = tid; q < nq; q += blockDim.x)
    atomicAdd(&hist[kOrderBins - 1 - (int)((uint64_t)slen[q] * kOrderBins / top)], 1u);
  __syncthreads();
  if (tid == 0) {  // exclusive scan (1024 entries)
    unsigned int run = 0;
    for (int i = 0; i < kOrderBins; ++i) {
      const unsigned int v = hist[i];
      hist[i] = run;
      run += v;
    }
  }
  __syncthreads();
  for (int64_t q = tid; q < nq; q += blockDim.x) {
    const int bin = kOrderBins - 1 - (int)((uint64_t)slen[q] * kOrderBins / top);
    perm[atomicAdd(&hist[bin], 1u)] = (int32_t)q;
  }
}

struct RefineArgs {
  nrq::RefineParams rf;
  const uint8_t *q;  // [nq x row_bytes]
  int64_t nq;
  int64_t row_bytes;
  int Lmax;
  const nr_seg *seg;
  const int32_t *nL;
  const uint32_t *slen;
  int64_t *out_ids;
  float *out_d;
  int64_t *stats;
  unsigned int *counter;
  const int32_t *perm;  // processing order (null: index order)
};

template <int DT, int TR, int STAGES, int CPR, int MINB>
__global__ void __launch_bounds__(TR, MINB) refine_kernel(RefineArgs a) {
  extern __shared__ __align__(128) unsigned char smem[];
  const int tid = threadIdx.x;
  const int k = a.rf.k;
  const nrq::RefineSmem m = nrq::refine_carve<TR, STAGES>(smem, a.row_bytes, k);
  int *qslot = m.sctl + 4;
  for (;;) {
    if (tid == 0) {
      const unsigned int slot = atomicAdd(a.counter, 1u);
      *qslot = slot < a.nq ? (a.perm ? a.perm[slot] : (int)slot) : -1;
    }
    __syncthreads();
    const int64_t q = *qslot;
    if (q < 0) break;
    for (int c = tid; c * 16 < a.row_bytes; c += TR)
      reinterpret_cast<uint4 *>(m.sq)[c] = reinterpret_cast<const uint4 *>(a.q + q * a.row_bytes)[c];
    nrq::refine_block<DT, TR, STAGES, CPR>(a.rf, m, a.slen[q], a.nL[q], a.seg + (size_t)q * a.Lmax,
                                           a.out_ids + q * k, a.out_d + q * k,
                                           a.stats ? a.stats + q * NR_QSTATS : nullptr);
  }
}

// fp32 rows longer than 1 KB: tiles staged in pieces (refine_block_split)
template <int TR, int STAGES, int KCC, int MINB>
__global__ void __launch_bounds__(TR, MINB) refine_split_kernel(RefineArgs a) {
  extern __shared__ __align__(128) unsigned char smem[];
  const int tid = threadIdx.x;
  const int k = a.rf.k;
  const nrq::RefineSmem m = nrq::refine_split_carve<TR, STAGES, KCC>(smem, a.row_bytes, k);
  int *qslot = m.sctl + 4;
  for (;;) {
    if (tid == 0) {
      const unsigned int slot = atomicAdd(a.counter, 1u);
      *qslot = slot < a.nq ? (a.perm ? a.perm[slot] : (int)slot) : -1;
    }
    __syncthreads();
    const int64_t q = *qslot;
    if (q < 0) break;
    for (int c = tid; c * 16 < a.row_bytes; c += TR)
      reinterpret_cast<uint4 *>(m.sq)[c] = reinterpret_cast<const uint4 *>(a.q + q * a.row_bytes)[c];
    nrq::refine_block_split<TR, STAGES, KCC>(a.rf, m, a.slen[q], a.nL[q],
                                             a.seg + (size_t)q * a.Lmax, a.out_ids + q * k,
                                             a.out_d + q * k, a.stats ? a.stats + q * NR_QSTATS : nullptr);
  }
}

template <typename K>
cudaError_t persistent_launch(nr_index *ix, K kern, int threads, size_t smem, int64_t nq,
                              const void *args, cudaStream_t s, void (*go)(K, int, int, size_t,
                                                                           cudaStream_t, const void *)) {
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, threads, smem);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  if (ix->params.refine_ctas > 0 && per_sm > ix->params.refine_ctas) per_sm = ix->params.refine_ctas;
  int64_t grid = (int64_t)per_sm * ix->num_sms;
  if (grid > nq) grid = nq;
  go(kern, (int)grid, threads, smem, s, args);
  ix->launches += 1;
  return cudaGetLastError();
}

template <int DT, int TR, int STAGES, int CPR, int MINB = 1>
cudaError_t launch_refine(nr_index *ix, const RefineArgs &a, cudaStream_t s) {
  const size_t smem = nrq::refine_smem_bytes<DT, TR, STAGES>(a.row_bytes, a.rf.k) + 16;
  auto kern = refine_kernel<DT, TR, STAGES, CPR, MINB>;
  return persistent_launch(ix, kern, TR, smem, a.nq, &a, s,
                           +[](decltype(kern) kk, int g, int t, size_t sm, cudaStream_t st,
                               const void *p) {
                             kk<<<g, t, sm, st>>>(*static_cast<const RefineArgs *>(p));
                           });
}

template <int TR, int STAGES, int KCC, int MINB>
cudaError_t launch_refine_split(nr_index *ix, const RefineArgs &a, cudaStream_t s) {
  const size_t smem = nrq::refine_split_smem_bytes<TR, STAGES, KCC>(a.row_bytes, a.rf.k) + 16;
  auto kern = refine_split_kernel<TR, STAGES, KCC, MINB>;
  return persistent_launch(ix, kern, TR, smem, a.nq, &a, s,
                           +[](decltype(kern) kk, int g, int t, size_t sm, cudaStream_t st,
                               const void *p) {
                             kk<<<g, t, sm, st>>>(*static_cast<const RefineArgs *>(p));
                           });
}

nrq::RefineParams refine_params(const nr_index *ix, int k) {
  const nr_params &p = ix->params;
  nrq::RefineParams rf;
  rf.vec = static_cast<const uint8_t *>(ix->vec);
  rf.ids = ix->ids;
  rf.cpr = (int)(ix->row_bytes / 16);
  rf.swz_mask = (rf.cpr % 8 == 0) ? 7 : (rf.cpr % 4 == 0) ? 3 : (rf.cpr % 2 == 0) ? 1 : 0;
  rf.k = k;
  rf.R = p.round_size;
  rf.t_low = p.t_low;
  rf.u_min = p.u_min;
  rf.f_min = p.f_min;
  rf.r_min = p.r_min;
  const double f = (double)p.alpha_front * (double)k;
  int nf = (int)f;
  if ((double)nf < f) nf += 1;  // ceil
  if (nf < 0) nf = 0;
  if (nf > k) nf = k;
  rf.nfront = nf;
  return rf;
}

}  // namespace

cudaError_t nr_launch_refine(nr_index *ix, const void *d_q, int64_t nq, int k, int Lmax,
                             const nr_seg *d_seg, const int32_t *d_nL, const uint32_t *d_slen,
                             int64_t *d_ids, float *d_dists, int64_t *d_stats,
                             unsigned int *d_counter, int32_t *d_perm, cudaStream_t s) {
  if (nq <= 0) return cudaSuccess;
  if (d_perm) {
    order_kernel<<<1, 1024, 0, s>>>(d_slen, nq, d_perm);
    ix->launches += 1;
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  RefineArgs a;
  a.rf = refine_params(ix, k);
  a.q = static_cast<const uint8_t *>(d_q);
  a.nq = nq;
  a.row_bytes = ix->row_bytes;
  a.Lmax = Lmax;
  a.seg = d_seg;
  a.nL = d_nL;
  a.slen = d_slen;
  a.out_ids = d_ids;
  a.out_d = d_dists;
  a.stats = d_stats;
  a.counter = d_counter;
  a.perm = d_perm;
  cudaError_t e = cudaMemsetAsync(d_counter, 0, sizeof(unsigned int), s);
  if (e != cudaSuccess) return e;
  if (ix->dtype == 0) {
    if (a.rf.cpr == 8) return launch_refine<0, 128, 2, 8, 6>(ix, a, s);  // uint8, D = 128
    if (ix->row_bytes <= 512) return launch_refine<0, 128, 2, 0, 4>(ix, a, s);
    return launch_refine<0, 64, 2, 0, 4>(ix, a, s);
  }
  if (ix->row_bytes > 1024) {  // fp32, D above 256: rows staged in pieces
    if (ix->row_bytes % 256 == 0) return launch_refine_split<128, 2, 16, 3>(ix, a, s);
    if (ix->row_bytes % 128 == 0) return launch_refine_split<128, 2, 8, 3>(ix, a, s);
    return launch_refine_split<128, 2, 4, 3>(ix, a, s);  // row_bytes % 64 == 0 (load check)
  }
  if (a.rf.cpr == 24) return launch_refine<1, 32, 2, 24, 12>(ix, a, s);  // fp32, D = 96
  if (ix->row_bytes <= 512) return launch_refine<1, 64, 2, 0, 4>(ix, a, s);
  return launch_refine<1, 32, 2, 0, 4>(ix, a, s);
}
