// K4 refine: exact squared-L2 refinement of the candidate stream into a
// per-query top-k with heap-quality early stopping in fixed-size rounds
// (Sec. 3.4 and Algorithm 2's T_low rule; uint8 distances kept as integers,
// Sec. 4.1.1).
//
// Persistent CTAs pull queries from an atomic counter. For one query the
// candidate stream is the concatenation of the rows of the ordered cluster
// list; each stored cluster is a contiguous run of rows, so the stream is a
// list of contiguous segments (K3 writes their first row and stream position).
//
// Data movement: the stream is consumed in tiles of TR rows (one row per
// thread). Each warp gathers its own 32 rows of a tile with 16-byte cp.async
// copies issued across lanes so that a warp-wide copy covers whole 128-byte
// lines, into a shared-memory stage whose 16-byte chunks are XOR-swizzled by
// row so that one-row-per-thread reads are bank-conflict free. STAGES tiles
// are in flight per CTA.
//
// Distances: uint8 rows use per-byte |x - q| (__vabsdiffu4) squared and summed
// with __dp4a in int32 (exact); fp32 rows use the sequential fmaf chain over
// j = 0..D-1, so a distance is bit-identical to a sequential CPU evaluation.
//
// Top-k: keys (distance bits << 32 | id) are unique. Rows at or below the
// current k-th key are collected and merged by rank (each element's rank is
// its position in the merged order), keeping for every member the round in
// which it entered. After round t: updates = members entered in round t,
// front updates = those within the first ceil(alpha * k) slots.
#include <cuda_runtime.h>
#include <stdint.h>

#include "nr_internal.cuh"

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr uint64_t kMaxKey = ~0ull;
constexpr int kMaxK = 256;

struct RefineArgs {
  const uint8_t *q;  // [nq x row_bytes]
  int64_t nq;
  int k, Lmax;
  const nr_seg *seg;
  const int32_t *nL;
  const uint32_t *slen;
  const uint8_t *vec;
  const uint32_t *ids;
  int64_t row_bytes;
  int cpr;       // 16-byte chunks per row
  int swz_mask;  // XOR mask applied to the chunk index (by row)
  int R;         // round size (power of two)
  int t_low, u_min, f_min, r_min, nfront;
  int64_t *out_ids;
  float *out_d;
  int64_t *stats;
  unsigned int *counter;
};

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

template <int DT, int TR, int STAGES>
__global__ void __launch_bounds__(TR) refine_kernel(RefineArgs a) {
  extern __shared__ __align__(128) unsigned char smem[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t RB = a.row_bytes;
  unsigned char *stage_base = smem;                                        // STAGES x TR x RB
  unsigned char *sq = smem + (size_t)STAGES * TR * RB;                     // RB (query)
  uint32_t *srow = reinterpret_cast<uint32_t *>(sq + ((RB + 15) & ~15));   // STAGES x TR
  uint64_t *hkey = reinterpret_cast<uint64_t *>(srow + STAGES * TR);       // 2 x kMaxK
  int *htag = reinterpret_cast<int *>(hkey + 2 * kMaxK);                   // 2 x kMaxK
  uint64_t *skey = reinterpret_cast<uint64_t *>(htag + 2 * kMaxK);         // TR survivors
  int *sctl = reinterpret_cast<int *>(skey + TR);                          // control words
  // sctl: 0 query, 1 survivors, 2 stop
  const uint32_t stage_s = (uint32_t)__cvta_generic_to_shared(stage_base);
  const int k = a.k;
  const int chunk = a.R < TR ? a.R : TR;

  for (;;) {
    if (tid == 0) sctl[0] = (int)atomicAdd(a.counter, 1u);
    __syncthreads();
    const int64_t q = sctl[0];
    if (q >= a.nq) break;
    // query row to shared memory
    for (int c = tid; c < a.cpr; c += TR)
      reinterpret_cast<uint4 *>(sq)[c] = reinterpret_cast<const uint4 *>(a.q + q * RB)[c];
    const int64_t n = a.slen[q];
    const int nl = a.nL[q];
    const nr_seg *segs = a.seg + (size_t)q * a.Lmax;
    const int64_t ntiles = (n + TR - 1) / TR;
    if (tid == 0) {
      sctl[1] = 0;
      sctl[2] = 0;
    }
    __syncthreads();

    // gather the rows of tile t into stage t % STAGES (each warp its own 32 rows)
    auto issue = [&](int64_t t) {
      if (t < ntiles) {
        const int st = (int)(t % STAGES);
        const int64_t p = t * TR + tid;
        uint32_t grow = 0;
        if (p < n) {
          int lo = 0, hi = nl - 1;  // last segment starting at or before p
          while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if ((int64_t)__ldg(&segs[mid].pos) <= p) lo = mid; else hi = mid - 1;
          }
          grow = __ldg(&segs[lo].row0) + (uint32_t)(p - (int64_t)__ldg(&segs[lo].pos));
          srow[st * TR + tid] = grow;
        }
        const int64_t wbase = t * TR + warp * 32;
        const uint32_t sbase = stage_s + (uint32_t)((size_t)st * TR * RB);
        for (int f = lane; f < 32 * a.cpr; f += 32) {
          const int rr = f / a.cpr;
          const int c = f - rr * a.cpr;
          const uint32_t gr = __shfl_sync(kFull, grow, rr);
          if (wbase + rr < n) {
            const int r = warp * 32 + rr;
            const uint32_t dst = sbase + (uint32_t)(r * RB) + (uint32_t)(((c ^ (r & a.swz_mask))) << 4);
            cp_async16(dst, a.vec + (size_t)gr * RB + ((size_t)c << 4));
          }
        }
      }
      cp_async_commit();
    };

    for (int s = 0; s < STAGES - 1; ++s) issue(s);
    int cur = 0, hn = 0, rounds = 0, low = 0;
    bool stop = false;
    int64_t done = 0;  // stream positions consumed in completed rounds
    for (int64_t t = 0; t < ntiles && !stop; ++t) {
      issue(t + STAGES - 1);
      cp_async_wait<STAGES - 1>();
      __syncwarp();
      const int st = (int)(t % STAGES);
      const int64_t p = t * TR + tid;
      uint32_t dkey = 0xffffffffu;
      if (p < n) {
        const unsigned char *row = stage_base + (size_t)st * TR * RB + (size_t)tid * RB;
        if (DT == 0) {
          unsigned acc = 0;
#pragma unroll 8
          for (int c = 0; c < a.cpr; ++c) {
            const uint4 v = *reinterpret_cast<const uint4 *>(row + ((c ^ (tid & a.swz_mask)) << 4));
            const uint4 w = reinterpret_cast<const uint4 *>(sq)[c];
            unsigned d;
            d = __vabsdiffu4(v.x, w.x); acc = __dp4a(d, d, acc);
            d = __vabsdiffu4(v.y, w.y); acc = __dp4a(d, d, acc);
            d = __vabsdiffu4(v.z, w.z); acc = __dp4a(d, d, acc);
            d = __vabsdiffu4(v.w, w.w); acc = __dp4a(d, d, acc);
          }
          dkey = acc;
        } else {
          float acc = 0.0f;
#pragma unroll 4
          for (int c = 0; c < a.cpr; ++c) {
            const float4 v = *reinterpret_cast<const float4 *>(row + ((c ^ (tid & a.swz_mask)) << 4));
            const float4 w = reinterpret_cast<const float4 *>(sq)[c];
            float d;
            d = __fsub_rn(v.x, w.x); acc = __fmaf_rn(d, d, acc);
            d = __fsub_rn(v.y, w.y); acc = __fmaf_rn(d, d, acc);
            d = __fsub_rn(v.z, w.z); acc = __fmaf_rn(d, d, acc);
            d = __fsub_rn(v.w, w.w); acc = __fmaf_rn(d, d, acc);
          }
          dkey = __float_as_uint(acc);
        }
      }
      // merge chunk by chunk; a round ends every R stream positions
      for (int cs = 0; cs < TR && !stop; cs += chunk) {
        const int64_t cstart = t * TR + cs;
        if (cstart >= n) break;
        const uint64_t thr = hn == k ? hkey[cur * kMaxK + k - 1] : kMaxKey;
        const uint32_t thr_hi = (uint32_t)(thr >> 32);
        if (tid >= cs && tid < cs + chunk && p < n && dkey <= thr_hi) {
          const uint32_t id = __ldg(&a.ids[srow[st * TR + tid]]);
          const uint64_t key = ((uint64_t)dkey << 32) | id;
          if (key < thr) skey[atomicAdd(&sctl[1], 1)] = key;
        }
        __syncthreads();
        const int ns = sctl[1];
        const int roundno = rounds + 1;
        if (ns > 0) {
          const int nxt = cur ^ 1;
          const uint64_t *H = hkey + cur * kMaxK;
          // merged order: by key; on equal keys (possible only when an index
          // stores a row twice) H before S, and S by slot, so ranks are unique
          for (int i = tid; i < ns; i += TR) {
            const uint64_t sk = skey[i];
            int lo = 0, hi = hn;  // # of H at or below sk
            while (lo < hi) {
              const int mid = (lo + hi) >> 1;
              if (H[mid] <= sk) lo = mid + 1; else hi = mid;
            }
            int r = lo;
            for (int j = 0; j < ns; ++j) r += (skey[j] < sk || (skey[j] == sk && j < i)) ? 1 : 0;
            if (r < k) {
              hkey[nxt * kMaxK + r] = sk;
              htag[nxt * kMaxK + r] = roundno;
            }
          }
          for (int j = tid; j < hn; j += TR) {
            const uint64_t hk = H[j];
            int r = j;
            for (int i = 0; i < ns; ++i) r += skey[i] < hk ? 1 : 0;
            if (r < k) {
              hkey[nxt * kMaxK + r] = hk;
              htag[nxt * kMaxK + r] = htag[cur * kMaxK + j];
            }
          }
          __syncthreads();
          cur = nxt;
          hn = hn + ns < k ? hn + ns : k;
          if (tid == 0) sctl[1] = 0;
        }
        const int64_t cend = cstart + chunk < n ? cstart + chunk : n;
        if ((cend % a.R) == 0 || cend >= n) {  // round complete
          rounds = roundno;
          done = cend;
          if (warp == 0) {
            int newc = 0, frontc = 0;
            for (int i = lane; i < hn; i += 32) {
              const bool nw = htag[cur * kMaxK + i] == roundno;
              newc += nw ? 1 : 0;
              frontc += (nw && i < a.nfront) ? 1 : 0;
            }
            for (int o = 16; o > 0; o >>= 1) {
              newc += __shfl_xor_sync(kFull, newc, o);
              frontc += __shfl_xor_sync(kFull, frontc, o);
            }
            const bool lowq = newc < a.u_min && frontc < a.f_min;
            const int nlow = lowq ? low + 1 : 0;
            if (lane == 0)
              sctl[2] = (a.t_low > 0 && hn == k && roundno >= a.r_min && nlow >= a.t_low) ? 1 : 0;
            low = nlow;
          }
          __syncthreads();  // only warp 0 tracks `low`; everyone reads the decision
          stop = sctl[2] != 0;
        }
        __syncthreads();
      }
    }
    cp_async_wait<0>();
    __syncthreads();
    // output, sorted by (distance, id), padded
    const uint64_t *H = hkey + cur * kMaxK;
    for (int i = tid; i < k; i += TR) {
      int64_t id = -1;
      float d = __int_as_float(0x7f800000);
      if (i < hn) {
        const uint64_t kk = H[i];
        id = (int64_t)(uint32_t)kk;
        const uint32_t db = (uint32_t)(kk >> 32);
        d = DT == 0 ? (float)db : __uint_as_float(db);
      }
      a.out_ids[q * k + i] = id;
      a.out_d[q * k + i] = d;
    }
    if (tid == 0 && a.stats) {
      a.stats[q * 4 + 0] = done;
      a.stats[q * 4 + 1] = rounds;
    }
    __syncthreads();
  }
}

template <int DT, int TR, int STAGES>
cudaError_t launch(nr_index *ix, const RefineArgs &a, cudaStream_t s) {
  const size_t smem = (size_t)STAGES * TR * a.row_bytes + ((a.row_bytes + 15) & ~15) +
                      (size_t)STAGES * TR * 4 + 2 * kMaxK * 8 + 2 * kMaxK * 4 + (size_t)TR * 8 + 16;
  auto kern = refine_kernel<DT, TR, STAGES>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, TR, smem);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  int64_t grid = (int64_t)per_sm * ix->num_sms;
  if (grid > a.nq) grid = a.nq;
  kern<<<(unsigned)grid, TR, smem, s>>>(a);
  ix->launches += 1;
  return cudaGetLastError();
}

}  // namespace

cudaError_t nr_launch_refine(nr_index *ix, const void *d_q, int64_t nq, int k, int Lmax,
                             const nr_seg *d_seg, const int32_t *d_nL, const uint32_t *d_slen,
                             int64_t *d_ids, float *d_dists, int64_t *d_stats,
                             unsigned int *d_counter, cudaStream_t s) {
  if (nq <= 0) return cudaSuccess;
  const nr_params &p = ix->params;
  RefineArgs a;
  a.q = static_cast<const uint8_t *>(d_q);
  a.nq = nq;
  a.k = k;
  a.Lmax = Lmax;
  a.seg = d_seg;
  a.nL = d_nL;
  a.slen = d_slen;
  a.vec = static_cast<const uint8_t *>(ix->vec);
  a.ids = ix->ids;
  a.row_bytes = ix->row_bytes;
  a.cpr = (int)(ix->row_bytes / 16);
  a.swz_mask = (a.cpr % 8 == 0) ? 7 : (a.cpr % 4 == 0) ? 3 : (a.cpr % 2 == 0) ? 1 : 0;
  a.R = p.round_size;
  a.t_low = p.t_low;
  a.u_min = p.u_min;
  a.f_min = p.f_min;
  a.r_min = p.r_min;
  double f = (double)p.alpha_front * (double)k;
  int nf = (int)f;
  if ((double)nf < f) nf += 1;  // ceil
  if (nf < 0) nf = 0;
  if (nf > k) nf = k;
  a.nfront = nf;
  a.out_ids = d_ids;
  a.out_d = d_dists;
  a.stats = d_stats;
  a.counter = d_counter;
  cudaError_t e = cudaMemsetAsync(d_counter, 0, sizeof(unsigned int), s);
  if (e != cudaSuccess) return e;
  if (ix->dtype == 0) {
    if (ix->row_bytes <= 256) return launch<0, 256, 3>(ix, a, s);
    if (ix->row_bytes <= 512) return launch<0, 128, 3>(ix, a, s);
    return launch<0, 64, 3>(ix, a, s);
  }
  if (ix->row_bytes <= 384) return launch<1, 256, 2>(ix, a, s);
  if (ix->row_bytes <= 768) return launch<1, 128, 2>(ix, a, s);
  return launch<1, 64, 2>(ix, a, s);
}
