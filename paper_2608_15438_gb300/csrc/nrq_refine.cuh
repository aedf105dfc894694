// refine_block: one block per query refines the candidate stream exactly
// with round-based early stop (Sec. 3.4, Algorithm 2's T_low rule).
#pragma once

#include "nrq_common.cuh"

namespace nrq {

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;\n" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

// ============================================================== refine
// Candidate stream = rows of the kept clusters in list order, a list of
// contiguous segments. Tiles of TR rows (one row per thread) are gathered by
// 16-byte cp.async copies (each warp copies and later reads only its own 32
// rows, so stage reuse needs no block barrier) into STAGES shared-memory
// stages whose 16-byte chunks are XOR-swizzled by row, so one-row-per-thread
// reads are bank-conflict free.
// Distances: uint8 rows: per-byte |x - q| (__vabsdiffu4) squared and summed by
// __dp4a in int32 (exact); fp32 rows: the sequential fmaf chain over j, so a
// distance is bit-identical to a sequential CPU evaluation.
// Top-k: keys (distance bits << 32 | id) are unique; rows at or below the
// current k-th key are merged by rank, each member tagged with the round it
// entered. After round t: updates = members entered in round t, front
// updates = those within the first nfront slots.
struct RefineParams {
  const uint8_t *vec;
  const uint32_t *ids;
  int cpr;       // 16-byte chunks per row (runtime value when CPR = 0)
  int swz_mask;  // XOR mask of the chunk index (runtime value when CPR = 0)
  int k, R;      // top-k size; round size (power of two)
  int t_low, u_min, f_min, r_min, nfront;
};

// Shared memory of refine_block beyond the stages.
struct RefineSmem {
  unsigned char *stage;  // STAGES x TR x row_bytes (16-byte aligned)
  unsigned char *sq;     // the query row (row_bytes)
  uint32_t *srow;        // STAGES x TR
  uint64_t *hkey;        // 2 x k
  uint64_t *skey;        // 2 x TR
  int *htag;             // 2 x k
  int *sctl;             // 4 ints: survivor counters [1..3]
};

template <int DT, int TR, int STAGES>
__host__ __device__ inline size_t refine_smem_bytes(int64_t row_bytes, int k) {
  return (size_t)STAGES * TR * row_bytes + (size_t)row_bytes + (size_t)STAGES * TR * 4 +
         (size_t)2 * k * 8 + (size_t)2 * TR * 8 + (size_t)2 * k * 4 + 16;
}

// Carve RefineSmem from base (16-byte aligned).
template <int TR, int STAGES>
__device__ __forceinline__ RefineSmem refine_carve(unsigned char *base, int64_t row_bytes, int k) {
  RefineSmem m;
  m.stage = base;
  m.sq = base + (size_t)STAGES * TR * row_bytes;
  m.srow = reinterpret_cast<uint32_t *>(m.sq + row_bytes);
  m.hkey = reinterpret_cast<uint64_t *>(m.srow + STAGES * TR);
  m.skey = m.hkey + 2 * k;
  m.htag = reinterpret_cast<int *>(m.skey + 2 * TR);
  m.sctl = m.htag + 2 * k;
  return m;
}

// One query. The caller has written the query row into m.sq (block-visible
// after this function's first barrier).
// segs: nl segments (any address space) of a stream of n positions. Writes
// out_ids/out_d [k] and stats[0..1]. Whole block (TR threads) calls.
template <int DT, int TR, int STAGES, int CPR>
__device__ __forceinline__ void refine_block(const RefineParams &a, const RefineSmem &m, uint32_t n,
                                             int nl, const nr_seg *segs, int64_t *out_ids,
                                             float *out_d, int64_t *stats) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int cpr = CPR > 0 ? CPR : a.cpr;
  const int swz = CPR > 0 ? ((CPR % 8 == 0) ? 7 : (CPR % 4 == 0) ? 3 : (CPR % 2 == 0) ? 1 : 0)
                          : a.swz_mask;
  const int64_t RB = (int64_t)cpr * 16;
  const uint32_t stage_s = (uint32_t)__cvta_generic_to_shared(m.stage);
  const int k = a.k;
  const int chunk = a.R < TR ? a.R : TR;
  const uint32_t ntiles = (uint32_t)(((uint64_t)n + TR - 1) / TR);
  if (tid == 0) m.sctl[1] = m.sctl[2] = m.sctl[3] = 0;
  __syncthreads();  // the caller's copy of the query row into m.sq is visible after this
  uint4 qreg[DT == 0 && CPR > 0 && CPR <= 8 ? CPR : 1];
  if (DT == 0 && CPR > 0 && CPR <= 8) {
#pragma unroll
    for (int c = 0; c < (CPR > 0 && CPR <= 8 ? CPR : 1); ++c) qreg[c] = reinterpret_cast<const uint4 *>(m.sq)[c];
  }

  int seg_i = 0;  // this thread's segment cursor (positions only grow)
  auto issue = [&](uint32_t t, int st) {
    if (t < ntiles) {
      const uint32_t p = t * TR + tid;
      uint32_t grow = 0;
      if (p < n) {
        // last segment starting at or before p: exponential search from the cursor
        int step = 1;
        while (seg_i + step < nl && segs[seg_i + step].pos <= p) {
          seg_i += step;
          step <<= 1;
        }
        for (step >>= 1; step > 0; step >>= 1)
          if (seg_i + step < nl && segs[seg_i + step].pos <= p) seg_i += step;
        grow = segs[seg_i].row0 + (p - segs[seg_i].pos);
        m.srow[st * TR + tid] = grow;
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
  uint32_t done = 0;                                 // positions in completed rounds
  const uint32_t rmask_round = (uint32_t)a.R - 1u;  // R is a power of two
  int st = 0;                                        // stage of tile t
  for (uint32_t t = 0; t < ntiles && !stop; ++t) {
    issue(t + STAGES - 1, st == 0 ? STAGES - 1 : st - 1);
    cp_async_wait<STAGES - 1>();
    __syncwarp();
    const uint32_t p = t * TR + tid;
    uint32_t dkey = 0xffffffffu;
    if (p < n) {
      const unsigned char *row = m.stage + (size_t)st * TR * RB + (size_t)tid * RB;
      if (DT == 0) {
        unsigned a0 = 0, a1 = 0, a2 = 0, a3 = 0;  // integer sums: any order is exact
#pragma unroll 8
        for (int c = 0; c < cpr; ++c) {
          const uint4 v = *reinterpret_cast<const uint4 *>(row + ((c ^ (tid & swz)) << 4));
          uint4 w;
          if (CPR > 0 && CPR <= 8) w = qreg[c < (CPR > 0 && CPR <= 8 ? CPR : 1) ? c : 0];
          else w = reinterpret_cast<const uint4 *>(m.sq)[c];
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
          const float4 w = reinterpret_cast<const float4 *>(m.sq)[c];
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
      int *cnt = &m.sctl[1 + ci % 3];
      uint64_t *sk_buf = m.skey + (ci & 1) * TR;
      const uint64_t thr = hn == k ? m.hkey[cur * k + k - 1] : kEmpty;
      const uint32_t thr_hi = (uint32_t)(thr >> 32);
      if (tid >= cs && tid < cs + chunk && p < n && dkey <= thr_hi) {
        const uint32_t id = __ldg(&a.ids[m.srow[st * TR + tid]]);
        const uint64_t key = ((uint64_t)dkey << 32) | id;
        if (key < thr) sk_buf[atomicAdd(cnt, 1)] = key;
      }
      if (tid == 0) m.sctl[1 + (ci + 1) % 3] = 0;  // counter of the next chunk
      __syncthreads();
      const int ns = *cnt;
      const int roundno = rounds + 1;
      if (ns > 0) {
        const int nxt = cur ^ 1;
        const uint64_t *H = m.hkey + cur * k;
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
            m.hkey[nxt * k + r] = sk;
            m.htag[nxt * k + r] = roundno;
          }
        }
        for (int j = tid; j < hn; j += TR) {
          const uint64_t hk = H[j];
          int r = j;
          for (int i = 0; i < ns; ++i) r += sk_buf[i] < hk ? 1 : 0;
          if (r < k) {
            m.hkey[nxt * k + r] = hk;
            m.htag[nxt * k + r] = m.htag[cur * k + j];
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
          const bool nw = m.htag[cur * k + i] == roundno;
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
  const uint64_t *H = m.hkey + cur * k;
  for (int i = tid; i < k; i += TR) {
    int64_t id = -1;
    float d = __int_as_float(0x7f800000);
    if (i < hn) {
      const uint64_t kk = H[i];
      id = (int64_t)(uint32_t)kk;
      const uint32_t db = (uint32_t)(kk >> 32);
      d = DT == 0 ? (float)db : __uint_as_float(db);
    }
    out_ids[i] = id;
    out_d[i] = d;
  }
  if (tid == 0 && stats) {
    stats[0] = (int64_t)done;
    stats[1] = rounds;
  }
  __syncthreads();
}

// ============================================================== refine, long rows
// fp32 rows too long for whole-row stages (D above 256): each tile of TR rows
// is staged in pieces of KCC 16-byte chunks of every row (TR x 16 KCC bytes a
// stage), and each thread carries its row's distance from piece to piece, so
// the sum over j stays the sequential fmaf chain of refine_block; the merge,
// rounds and stop rule are refine_block's. row_bytes is a multiple of 16 KCC.
template <int TR, int STAGES, int KCC>
__host__ __device__ inline size_t refine_split_smem_bytes(int64_t row_bytes, int k) {
  return (size_t)STAGES * TR * KCC * 16 + (size_t)row_bytes + (size_t)2 * TR * 4 +
         (size_t)2 * k * 8 + (size_t)2 * TR * 8 + (size_t)2 * k * 4 + 16;
}

template <int TR, int STAGES, int KCC>
__device__ __forceinline__ RefineSmem refine_split_carve(unsigned char *base, int64_t row_bytes,
                                                         int k) {
  RefineSmem m;
  m.stage = base;
  m.sq = base + (size_t)STAGES * TR * KCC * 16;
  m.srow = reinterpret_cast<uint32_t *>(m.sq + row_bytes);  // 2 x TR: rows of the open tiles
  m.hkey = reinterpret_cast<uint64_t *>(m.srow + 2 * TR);
  m.skey = m.hkey + 2 * k;
  m.htag = reinterpret_cast<int *>(m.skey + 2 * TR);
  m.sctl = m.htag + 2 * k;
  return m;
}

template <int TR, int STAGES, int KCC>
__device__ __forceinline__ void refine_block_split(const RefineParams &a, const RefineSmem &m,
                                                   uint32_t n, int nl, const nr_seg *segs,
                                                   int64_t *out_ids, float *out_d, int64_t *stats) {
  constexpr int swz = KCC % 8 == 0 ? 7 : KCC % 4 == 0 ? 3 : KCC % 2 == 0 ? 1 : 0;
  constexpr uint32_t PB = KCC * 16;  // bytes of one row in one stage
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t RB = (int64_t)a.cpr * 16;
  const int nk = a.cpr / KCC;  // pieces per row
  const uint32_t stage_s = (uint32_t)__cvta_generic_to_shared(m.stage);
  const int k = a.k;
  const int chunk = a.R < TR ? a.R : TR;
  const uint32_t ntiles = (uint32_t)(((uint64_t)n + TR - 1) / TR);
  const uint32_t nitems = ntiles * (uint32_t)nk;
  if (tid == 0) m.sctl[1] = m.sctl[2] = m.sctl[3] = 0;
  __syncthreads();  // the caller's copy of the query row into m.sq is visible after this

  int seg_i = 0;       // this thread's segment cursor (positions only grow)
  uint32_t grow = 0;   // this thread's row in the tile being issued
  auto issue = [&](uint32_t it, int st) {
    if (it < nitems) {
      const uint32_t t = it / (uint32_t)nk;
      const int kk = (int)(it - t * (uint32_t)nk);
      if (kk == 0) {  // a new tile: find this thread's row
        const uint32_t p = t * TR + tid;
        grow = 0;
        if (p < n) {
          int step = 1;
          while (seg_i + step < nl && segs[seg_i + step].pos <= p) {
            seg_i += step;
            step <<= 1;
          }
          for (step >>= 1; step > 0; step >>= 1)
            if (seg_i + step < nl && segs[seg_i + step].pos <= p) seg_i += step;
          grow = segs[seg_i].row0 + (p - segs[seg_i].pos);
          m.srow[(t & 1) * TR + tid] = grow;
        }
      }
      const uint32_t wbase = t * TR + warp * 32;
      const uint32_t sbase = stage_s + (uint32_t)((size_t)st * TR * PB);
#pragma unroll 4
      for (int f = lane; f < 32 * KCC; f += 32) {
        const int rr = f / KCC;
        const int c = f - rr * KCC;
        const uint32_t gr = __shfl_sync(kFull, grow, rr);
        if (wbase + rr < n) {
          const int r = warp * 32 + rr;
          const uint32_t dst = sbase + (uint32_t)(r * PB) + (uint32_t)((c ^ (r & swz)) << 4);
          cp_async16(dst, a.vec + (size_t)gr * RB + (size_t)kk * PB + ((size_t)c << 4));
        }
      }
    }
    cp_async_commit();
  };

  for (int s = 0; s < STAGES - 1; ++s) issue((uint32_t)s, s);
  int cur = 0, hn = 0, rounds = 0, low = 0, ci = 0;
  bool stop = false;
  uint32_t done = 0;
  const uint32_t rmask_round = (uint32_t)a.R - 1u;
  int st = 0;
  float acc = 0.0f;  // sequential over j across the pieces of a row
  for (uint32_t it = 0; it < nitems && !stop; ++it) {
    issue(it + STAGES - 1, st == 0 ? STAGES - 1 : st - 1);
    cp_async_wait<STAGES - 1>();
    __syncwarp();
    const uint32_t t = it / (uint32_t)nk;
    const int kk = (int)(it - t * (uint32_t)nk);
    const uint32_t p = t * TR + tid;
    if (p < n) {
      const unsigned char *row = m.stage + (size_t)st * TR * PB + (size_t)tid * PB;
      const float4 *q4 = reinterpret_cast<const float4 *>(m.sq + (size_t)kk * PB);
#pragma unroll 4
      for (int c = 0; c < KCC; ++c) {
        const float4 v = *reinterpret_cast<const float4 *>(row + ((c ^ (tid & swz)) << 4));
        const float4 w = q4[c];
        float d;
        d = __fsub_rn(v.x, w.x); acc = __fmaf_rn(d, d, acc);
        d = __fsub_rn(v.y, w.y); acc = __fmaf_rn(d, d, acc);
        d = __fsub_rn(v.z, w.z); acc = __fmaf_rn(d, d, acc);
        d = __fsub_rn(v.w, w.w); acc = __fmaf_rn(d, d, acc);
      }
    }
    st = st + 1 == STAGES ? 0 : st + 1;
    if (kk + 1 < nk) continue;  // the row is not complete yet
    const uint32_t dkey = p < n ? __float_as_uint(acc) : 0xffffffffu;
    acc = 0.0f;
    for (int cs = 0; cs < TR && !stop; cs += chunk, ++ci) {
      const uint32_t cstart = t * TR + cs;
      if (cstart >= n) break;
      int *cnt = &m.sctl[1 + ci % 3];
      uint64_t *sk_buf = m.skey + (ci & 1) * TR;
      const uint64_t thr = hn == k ? m.hkey[cur * k + k - 1] : kEmpty;
      const uint32_t thr_hi = (uint32_t)(thr >> 32);
      if (tid >= cs && tid < cs + chunk && p < n && dkey <= thr_hi) {
        const uint32_t id = __ldg(&a.ids[m.srow[(t & 1) * TR + tid]]);
        const uint64_t key = ((uint64_t)dkey << 32) | id;
        if (key < thr) sk_buf[atomicAdd(cnt, 1)] = key;
      }
      if (tid == 0) m.sctl[1 + (ci + 1) % 3] = 0;
      __syncthreads();
      const int ns = *cnt;
      const int roundno = rounds + 1;
      if (ns > 0) {
        const int nxt = cur ^ 1;
        const uint64_t *H = m.hkey + cur * k;
        for (int i = tid; i < ns; i += TR) {
          const uint64_t sk = sk_buf[i];
          int lo = 0, hi = hn;
          while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (H[mid] <= sk) lo = mid + 1; else hi = mid;
          }
          int r = lo;
          for (int j = 0; j < ns; ++j) r += (sk_buf[j] < sk || (sk_buf[j] == sk && j < i)) ? 1 : 0;
          if (r < k) {
            m.hkey[nxt * k + r] = sk;
            m.htag[nxt * k + r] = roundno;
          }
        }
        for (int j = tid; j < hn; j += TR) {
          const uint64_t hk = H[j];
          int r = j;
          for (int i = 0; i < ns; ++i) r += sk_buf[i] < hk ? 1 : 0;
          if (r < k) {
            m.hkey[nxt * k + r] = hk;
            m.htag[nxt * k + r] = m.htag[cur * k + j];
          }
        }
        __syncthreads();
        cur = nxt;
        hn = hn + ns < k ? hn + ns : k;
      }
      const uint32_t cend = n - cstart > (uint32_t)chunk ? cstart + chunk : n;
      if ((cend & rmask_round) == 0 || cend >= n) {
        rounds = roundno;
        done = cend;
        int newc = 0, frontc = 0;
        for (int i = lane; i < hn; i += 32) {
          const bool nw = m.htag[cur * k + i] == roundno;
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
  }
  cp_async_wait<0>();
  __syncthreads();
  const uint64_t *H = m.hkey + cur * k;
  for (int i = tid; i < k; i += TR) {
    int64_t id = -1;
    float d = __int_as_float(0x7f800000);
    if (i < hn) {
      const uint64_t kk2 = H[i];
      id = (int64_t)(uint32_t)kk2;
      d = __uint_as_float((uint32_t)(kk2 >> 32));
    }
    out_ids[i] = id;
    out_d[i] = d;
  }
  if (tid == 0 && stats) {
    stats[0] = (int64_t)done;
    stats[1] = rounds;
  }
  __syncthreads();
}

}  // namespace nrq
