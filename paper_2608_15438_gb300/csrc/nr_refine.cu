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
// row so that one-row-per-thread reads are bank-conflict free. Tiles are small
// (128 uint8 rows, 32 fp32 rows) and two stages deep, so that many queries
// stream concurrently on every SM.
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

// CPR = 16-byte chunks per row when known at compile time (0: a.cpr)
template <int DT, int TR, int STAGES, int CPR, int MINB>
__global__ void __launch_bounds__(TR, MINB) refine_kernel(RefineArgs a) {
  extern __shared__ __align__(128) unsigned char smem[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int cpr = CPR > 0 ? CPR : a.cpr;
  const int swz = CPR > 0 ? ((CPR % 8 == 0) ? 7 : (CPR % 4 == 0) ? 3 : (CPR % 2 == 0) ? 1 : 0)
                          : a.swz_mask;
  const int64_t RB = (int64_t)cpr * 16;
  unsigned char *stage_base = smem;                                       // STAGES x TR x RB
  unsigned char *sq = smem + (size_t)STAGES * TR * RB;                    // RB (query)
  uint32_t *srow = reinterpret_cast<uint32_t *>(sq + RB);                 // STAGES x TR
  const int kMaxK = a.k;                                                  // top-k buffers sized by k
  uint64_t *hkey = reinterpret_cast<uint64_t *>(srow + STAGES * TR);      // 2 x k
  uint64_t *skey = hkey + 2 * kMaxK;                                      // 2 x TR survivors
  int *htag = reinterpret_cast<int *>(skey + 2 * TR);                     // 2 x k
  int *sctl = htag + 2 * kMaxK;                                           // [0] query, [1..3] counters
  const uint32_t stage_s = (uint32_t)__cvta_generic_to_shared(stage_base);
  const int k = a.k;
  const int chunk = a.R < TR ? a.R : TR;

  for (;;) {
    if (tid == 0) {
      sctl[0] = (int)atomicAdd(a.counter, 1u);
      sctl[1] = sctl[2] = sctl[3] = 0;
    }
    __syncthreads();
    const int64_t q = sctl[0];
    if (q >= a.nq) break;
    for (int c = tid; c < cpr; c += TR)
      reinterpret_cast<uint4 *>(sq)[c] = reinterpret_cast<const uint4 *>(a.q + q * RB)[c];
    const uint32_t n = a.slen[q];  // stream positions fit 32 bits (N < 2^32)
    const int nl = a.nL[q];
    const nr_seg *segs = a.seg + (size_t)q * a.Lmax;
    const uint32_t ntiles = (uint32_t)(((uint64_t)n + TR - 1) / TR);
    __syncthreads();
    uint4 qreg[DT == 0 && CPR > 0 && CPR <= 8 ? CPR : 1];
    if (DT == 0 && CPR > 0 && CPR <= 8) {
#pragma unroll
      for (int c = 0; c < (CPR > 0 && CPR <= 8 ? CPR : 1); ++c) qreg[c] = reinterpret_cast<const uint4 *>(sq)[c];
    }

    // Gather the rows of tile t into stage t % STAGES. A warp copies and later
    // reads only its own 32 rows, so stage reuse needs no block barrier.
    int seg_i = 0;  // this thread's segment cursor (positions only grow)
    auto issue = [&](uint32_t t, int st) {
      if (t < ntiles) {
        const uint32_t p = t * TR + tid;
        uint32_t grow = 0;
        if (p < n) {
          // last segment starting at or before p: exponential search from the cursor
          int step = 1;
          while (seg_i + step < nl && __ldg(&segs[seg_i + step].pos) <= p) {
            seg_i += step;
            step <<= 1;
          }
          for (step >>= 1; step > 0; step >>= 1)
            if (seg_i + step < nl && __ldg(&segs[seg_i + step].pos) <= p) seg_i += step;
          grow = __ldg(&segs[seg_i].row0) + (p - __ldg(&segs[seg_i].pos));
          srow[st * TR + tid] = grow;
        }
        const uint32_t wbase = t * TR + warp * 32;
        const uint32_t sbase = stage_s + (uint32_t)((size_t)st * TR * RB);
#pragma unroll 4
        for (int f = lane; f < 32 * cpr; f += 32) {
          const int rr = f / cpr;
          const int c = f - rr * cpr;
          const uint32_t gr = __shfl_sync(kFull, grow, rr);
          if (wbase + rr < n) {
            const int r = warp * 32 + rr;
            const uint32_t dst = sbase + (uint32_t)(r * RB) + (uint32_t)((c ^ (r & swz)) << 4);
            cp_async16(dst, a.vec + (size_t)gr * RB + ((size_t)c << 4));
          }
        }
      }
      cp_async_commit();
    };

    for (int s = 0; s < STAGES - 1; ++s) issue((uint32_t)s, s);
    int cur = 0, hn = 0, rounds = 0, low = 0, ci = 0;
    bool stop = false;
    uint32_t done = 0;  // stream positions consumed in completed rounds
    const uint32_t rmask_round = (uint32_t)a.R - 1u;  // R is a power of two
    int st = 0;                                        // stage of tile t
    for (uint32_t t = 0; t < ntiles && !stop; ++t) {
      issue(t + STAGES - 1, st == 0 ? STAGES - 1 : st - 1);
      cp_async_wait<STAGES - 1>();
      __syncwarp();
      const uint32_t p = t * TR + tid;
      uint32_t dkey = 0xffffffffu;
      if (p < n) {
        const unsigned char *row = stage_base + (size_t)st * TR * RB + (size_t)tid * RB;
        if (DT == 0) {
          unsigned a0 = 0, a1 = 0, a2 = 0, a3 = 0;  // integer sums: any order is exact
#pragma unroll 8
          for (int c = 0; c < cpr; ++c) {
            const uint4 v = *reinterpret_cast<const uint4 *>(row + ((c ^ (tid & swz)) << 4));
            uint4 w;
            if (CPR > 0 && CPR <= 8) w = qreg[c < (CPR > 0 && CPR <= 8 ? CPR : 1) ? c : 0];
            else w = reinterpret_cast<const uint4 *>(sq)[c];
            unsigned d;
            d = __vabsdiffu4(v.x, w.x); a0 = __dp4a(d, d, a0);
            d = __vabsdiffu4(v.y, w.y); a1 = __dp4a(d, d, a1);
            d = __vabsdiffu4(v.z, w.z); a2 = __dp4a(d, d, a2);
            d = __vabsdiffu4(v.w, w.w); a3 = __dp4a(d, d, a3);
          }
          dkey = (a0 + a1) + (a2 + a3);
        } else {
          float acc = 0.0f;  // sequential over j: the order fixes the rounding
#pragma unroll 4
          for (int c = 0; c < cpr; ++c) {
            const float4 v = *reinterpret_cast<const float4 *>(row + ((c ^ (tid & swz)) << 4));
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
      // Merge chunk by chunk; a round ends every R stream positions. One block
      // barrier per chunk (two when the top-k changes): survivor counters
      // rotate over three slots and survivor buffers over two, and every warp
      // evaluates the stop rule itself from the shared top-k.
      for (int cs = 0; cs < TR && !stop; cs += chunk, ++ci) {
        const uint32_t cstart = t * TR + cs;
        if (cstart >= n) break;
        int *cnt = &sctl[1 + ci % 3];
        uint64_t *sk_buf = skey + (ci & 1) * TR;
        const uint64_t thr = hn == k ? hkey[cur * kMaxK + k - 1] : kMaxKey;
        const uint32_t thr_hi = (uint32_t)(thr >> 32);
        if (tid >= cs && tid < cs + chunk && p < n && dkey <= thr_hi) {
          const uint32_t id = __ldg(&a.ids[srow[st * TR + tid]]);
          const uint64_t key = ((uint64_t)dkey << 32) | id;
          if (key < thr) sk_buf[atomicAdd(cnt, 1)] = key;
        }
        if (tid == 0) sctl[1 + (ci + 1) % 3] = 0;  // counter of the next chunk
        __syncthreads();
        const int ns = *cnt;
        const int roundno = rounds + 1;
        if (ns > 0) {
          const int nxt = cur ^ 1;
          const uint64_t *H = hkey + cur * kMaxK;
          // merged order: by key; on equal keys (possible only when an index
          // stores a row twice) H before S, and S by slot, so ranks are unique
          for (int i = tid; i < ns; i += TR) {
            const uint64_t sk = sk_buf[i];
            int lo = 0, hi = hn;  // # of H at or below sk
            while (lo < hi) {
              const int mid = (lo + hi) >> 1;
              if (H[mid] <= sk) lo = mid + 1; else hi = mid;
            }
            int r = lo;
            for (int j = 0; j < ns; ++j) r += (sk_buf[j] < sk || (sk_buf[j] == sk && j < i)) ? 1 : 0;
            if (r < k) {
              hkey[nxt * kMaxK + r] = sk;
              htag[nxt * kMaxK + r] = roundno;
            }
          }
          for (int j = tid; j < hn; j += TR) {
            const uint64_t hk = H[j];
            int r = j;
            for (int i = 0; i < ns; ++i) r += sk_buf[i] < hk ? 1 : 0;
            if (r < k) {
              hkey[nxt * kMaxK + r] = hk;
              htag[nxt * kMaxK + r] = htag[cur * kMaxK + j];
            }
          }
          __syncthreads();
          cur = nxt;
          hn = hn + ns < k ? hn + ns : k;
        }
        const uint32_t cend = n - cstart > (uint32_t)chunk ? cstart + chunk : n;
        if ((cend & rmask_round) == 0 || cend >= n) {  // round complete
          rounds = roundno;
          done = cend;
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
          low = lowq ? low + 1 : 0;
          stop = a.t_low > 0 && hn == k && roundno >= a.r_min && low >= a.t_low;
        }
      }
      st = st + 1 == STAGES ? 0 : st + 1;
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
      a.stats[q * 4 + 0] = (int64_t)done;
      a.stats[q * 4 + 1] = rounds;
    }
    __syncthreads();
  }
}

template <int DT, int TR, int STAGES, int CPR, int MINB = 1>
cudaError_t launch(nr_index *ix, const RefineArgs &a, cudaStream_t s) {
  const size_t smem = (size_t)STAGES * TR * a.row_bytes + (size_t)a.row_bytes +
                      (size_t)STAGES * TR * 4 + (size_t)2 * a.k * 12 + (size_t)2 * TR * 8 + 32;
  auto kern = refine_kernel<DT, TR, STAGES, CPR, MINB>;
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
  // Launch shapes measured on GB300 (u8-10m / f32-10m operating points): the
  // scan is limited by how many queries stream concurrently per SM, so tiles
  // are small, two stages deep, and registers are capped for many CTAs per SM.
  if (ix->dtype == 0) {
    if (a.cpr == 8) return launch<0, 128, 2, 8, 6>(ix, a, s);  // uint8, D = 128
    if (ix->row_bytes <= 512) return launch<0, 128, 2, 0, 4>(ix, a, s);
    return launch<0, 64, 2, 0, 4>(ix, a, s);
  }
  if (a.cpr == 24) return launch<1, 32, 2, 24, 12>(ix, a, s);  // fp32, D = 96
  if (ix->row_bytes <= 512) return launch<1, 64, 2, 0, 4>(ix, a, s);
  return launch<1, 32, 2, 0, 4>(ix, a, s);
}
