// Per-query building blocks of the query path, used by the route, select and
// refine kernels:
//   route_warp     one warp: binarise, rank bits, probe codes (Eq. 10, Algorithm 1)
//   select_block   one block: CSR lookup, centroid distances, gate, top-C and the
//                  refinement segments of the kept clusters (Sec. 3.3, 3.4.2, Algorithm 2)
//   refine_block   one block: exact refinement with round-based early stop
//                  (Sec. 3.4, Algorithm 2's T_low rule)
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "nr_internal.cuh"

namespace nrq {

constexpr unsigned kFull = 0xffffffffu;
constexpr uint64_t kEmpty = ~0ull;

__device__ __forceinline__ void set_err(int *err, int code) { atomicCAS(err, 0, code); }

__device__ __forceinline__ uint64_t pack_key(float cost, uint32_t size, uint32_t mask) {
  return ((uint64_t)__float_as_uint(cost) << 32) | ((uint64_t)size << 24) | (uint64_t)mask;
}

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

// ============================================================== route
// Ranks order the bits by (delta_j, j); a flip set F is a set of ranks with key
//   (cost(F), |F|, rank mask),  cost = fp32 sum of delta over F, ascending rank.
// Flip sets form a tree rooted at {0}: a set whose largest rank is m has the
// children "shift" (m -> m+1) and "expand" (add m+1). Every child's key is
// larger than its parent's (delta sorted ascending, fp32 round-to-nearest is
// monotone), so popping the smallest key of the frontier P-1 times yields the
// first P sets in key order, the empty set (the base bucket) first. Costs are
// carried as (cost, cost without the largest rank), so each child's cost is
// one addition in the same left-to-right order a sequential sum would use.
//
// The frontier is a 32-ary min-heap of keys in shared memory (capacity P + 2,
// 8 bytes an entry): a sift-down level is one load per lane and two warp
// min-reductions; the frontier never holds more than P + 1 entries. The cost
// without the largest rank, needed for the shift child, is recomputed from
// the popped rank mask in the same left-to-right fp32 order. Lane j holds bit j.
struct RouteParams {
  const float *tau;
  int b, bsel, rmax;
  float smax;
  int P;
};

// Bytes of shared memory route_warp needs for probe budget P.
__host__ __device__ inline size_t route_heap_bytes(int P) { return (size_t)(P + 2) * 8 + 128; }

// Writes codes[0..n) (any address space) and returns n, uniform in the warp.
// Must be called by a whole warp. heap: route_heap_bytes(P) bytes of shared
// memory (8-byte aligned).
__device__ __forceinline__ int route_warp(const RouteParams &rp, const float *__restrict__ logit,
                                          unsigned char *heap, uint32_t *codes) {
  const int lane = threadIdx.x & 31;
  const int b = rp.b;
  uint64_t *hkey = reinterpret_cast<uint64_t *>(heap);
  float *ssd = reinterpret_cast<float *>(heap + (size_t)(rp.P + 2) * 8);
  float dj = __int_as_float(0x7f800000);
  bool bit = false;
  if (lane < b) {
    const float l = logit[lane];
    const float tj = rp.tau[lane];
    bit = l >= tj;                   // Eq. 10
    dj = fabsf(__fsub_rn(l, tj));    // deviation
  }
  const uint32_t u0 = __ballot_sync(kFull, bit);
  int rank = 0;
  for (int i = 0; i < b; ++i) {
    const float di = __shfl_sync(kFull, dj, i);
    if (di < dj || (di == dj && i < lane)) ++rank;
  }
  uint32_t rbit = 0;  // lane r: 1 << (bit index of rank r)
  for (int j = 0; j < b; ++j) {
    const int rj = __shfl_sync(kFull, rank, j);
    if (rj == lane) rbit = 1u << j;
  }
  if (lane < b) ssd[rank] = dj;
  __syncwarp();
  if (lane == 0) codes[0] = u0;
  int n = 1, hs = 0;
  if (rp.P > 1 && rp.bsel >= 1 && ssd[0] <= rp.smax) {
    if (lane == 0) hkey[0] = pack_key(ssd[0], 1u, 1u);
    hs = 1;
  }
  __syncwarp();
  while (n < rp.P && hs > 0) {
    const uint64_t top = hkey[0];
    const uint32_t rmask = (uint32_t)top & 0xffffffu;
    const uint32_t size = ((uint32_t)top >> 24) & 0xffu;
    const float cost = __uint_as_float((uint32_t)(top >> 32));
    // ApplyFlips: code = u0 XOR (bits of the ranks in F)
    const uint32_t flips = __reduce_or_sync(kFull, ((rmask >> lane) & 1u) ? rbit : 0u);
    if (lane == 0) codes[n] = u0 ^ flips;
    ++n;
    const int m = 31 - __clz((int)rmask);
    bool v1 = false, v2 = false;
    uint64_t k1 = kEmpty, k2 = kEmpty;
    if (m + 1 < rp.bsel) {
      const float sdn = ssd[m + 1];
      // cost without rank m: fp32 sum from 0 over the other ranks, ascending
      float costp = 0.0f;
      for (uint32_t mm = rmask & ~(1u << m); mm; mm &= mm - 1) costp = __fadd_rn(costp, ssd[__ffs(mm) - 1]);
      const float c1 = __fadd_rn(costp, sdn);  // shift: rank m -> m + 1
      if (c1 <= rp.smax) {
        v1 = true;
        k1 = pack_key(c1, size, rmask + (1u << m));
      }
      if (rp.rmax <= 0 || (int)size < rp.rmax) {  // expand: add rank m + 1
        const float c2 = __fadd_rn(cost, sdn);
        if (c2 <= rp.smax) {
          v2 = true;
          k2 = pack_key(c2, size + 1, rmask | (1u << (m + 1)));
        }
      }
    }
    uint64_t x = kEmpty;
    if (v1) {
      x = k1;
    } else if (v2) {
      x = k2;
    } else {
      hs -= 1;
      if (hs > 0) x = hkey[hs];
    }
    if (x != kEmpty) {  // sift-down of x from the root
      int i = 0;
      for (;;) {
        const int c = 32 * i + 1 + lane;
        const uint64_t ck = c < hs ? hkey[c] : kEmpty;
        const uint32_t chi = (uint32_t)(ck >> 32), clo = (uint32_t)ck;
        const uint32_t mhi = __reduce_min_sync(kFull, chi);
        const uint32_t mlo = __reduce_min_sync(kFull, chi == mhi ? clo : 0xffffffffu);
        const uint64_t mk = ((uint64_t)mhi << 32) | mlo;
        if (mk < x) {
          const int src = __ffs(__ballot_sync(kFull, ck == mk)) - 1;
          if (lane == src) hkey[i] = mk;
          i = 32 * i + 1 + src;
          __syncwarp();
        } else {
          if (lane == 0) hkey[i] = x;
          break;
        }
      }
    }
    __syncwarp();
    if (v1 && v2) {  // sift-up of the expand child
      if (lane == 0) {
        int j = hs;
        while (j > 0) {
          const int pj = (j - 1) >> 5;
          const uint64_t pk = hkey[pj];
          if (pk < k2) break;
          hkey[j] = pk;
          j = pj;
        }
        hkey[j] = k2;
      }
      hs += 1;
    }
    __syncwarp();
  }
  return n;
}

// ============================================================== select
// Exclusive scan of a[0..n) in shared memory by the whole block (blockDim a
// multiple of 32, at most 1024); returns the total.
__device__ __forceinline__ int block_exclusive_scan(int *a, int n, int *warp_sums) {
  const int nt = blockDim.x, tid = threadIdx.x, lane = tid & 31, wid = tid >> 5, nw = nt >> 5;
  const int per = (n + nt - 1) / nt;
  const int lo = tid * per, hi = min(n, lo + per);
  int local = 0;
  for (int i = lo; i < hi; ++i) local += a[i];
  int incl = local;
  for (int o = 1; o < 32; o <<= 1) {
    const int v = __shfl_up_sync(kFull, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) warp_sums[wid] = incl;
  __syncthreads();
  if (wid == 0) {
    int ws = lane < nw ? warp_sums[lane] : 0;
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(kFull, ws, o);
      if (lane >= o) ws += v;
    }
    if (lane < nw) warp_sums[lane] = ws;  // inclusive
  }
  __syncthreads();
  int run = (wid > 0 ? warp_sums[wid - 1] : 0) + incl - local;
  for (int i = lo; i < hi; ++i) {
    const int v = a[i];
    a[i] = run;
    run += v;
  }
  const int total = warp_sums[nw - 1];
  __syncthreads();
  return total;
}

// Bitonic sort of k[0..n), n a power of two, by the whole block. Thread i
// owns the pairs (lo, lo + stride) with lo = 2i - (i mod stride); for strides
// up to 32 the pairs of one warp stay inside its own 64-element blocks, so
// consecutive such stages need only a warp barrier.
__device__ __forceinline__ void bitonic_sort(uint64_t *k, int n) {
  const int nt = blockDim.x;
  for (int size = 2; size <= n; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < n / 2; i += nt) {
        const int lo = 2 * i - (i & (stride - 1));
        const int hi = lo + stride;
        const bool up = (lo & size) == 0;
        const uint64_t a = k[lo], c = k[hi];
        if ((a > c) == up) {
          k[lo] = c;
          k[hi] = a;
        }
      }
      const int next = stride > 1 ? stride >> 1 : size;
      if (stride > 32 || next > 32 || nt <= 32) __syncthreads();
      else __syncwarp();
    }
  }
  __syncthreads();
}

// Block merge sort of k[0..n) ascending, for keys that are distinct apart
// from kEmpty padding; n <= 16 * blockDim.x, blockDim.x a power of two.
// Each thread sorts a run of E keys in registers (a bitonic network with
// compile-time indices), then runs are merged pairwise through shared memory:
// every thread finds where its E outputs start on the merge path of its pair
// of runs by binary search and merges E keys. Leaves k[n..E*blockDim.x)
// holding kEmpty.
template <int E>
__device__ __forceinline__ void merge_sort_e(uint64_t *k, int n) {
  const int tid = threadIdx.x;
  const int N = E * (int)blockDim.x;
  uint64_t r[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int i = tid * E + e;
    r[e] = i < n ? k[i] : kEmpty;
  }
#pragma unroll
  for (int size = 2; size <= E; size <<= 1)
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1)
#pragma unroll
      for (int i = 0; i < E; ++i) {
        const int j = i ^ stride;
        if (j > i) {
          const bool up = (i & size) == 0;
          const uint64_t a = r[i], c = r[j];
          if ((a > c) == up) {
            r[i] = c;
            r[j] = a;
          }
        }
      }
  __syncthreads();
#pragma unroll
  for (int e = 0; e < E; ++e) k[tid * E + e] = r[e];
  __syncthreads();
  for (int w = E; w < N; w <<= 1) {
    const int lo = (tid * E) & ~(2 * w - 1);  // first key of my pair of runs
    const int d = tid * E - lo;               // my first output on its merge path
    const uint64_t *A = k + lo, *B = k + lo + w;
    int a = d > w ? d - w : 0, hi = d < w ? d : w;
    while (a < hi) {
      const int mid = (a + hi) >> 1;
      if (A[mid] > B[d - 1 - mid]) hi = mid;
      else a = mid + 1;
    }
    int i = a, j = d - a;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      const uint64_t x = i < w ? A[i] : kEmpty, y = j < w ? B[j] : kEmpty;
      const bool takeA = j >= w || (i < w && x <= y);
      r[e] = takeA ? x : y;
      i += takeA ? 1 : 0;
      j += takeA ? 0 : 1;
    }
    __syncthreads();
#pragma unroll
    for (int e = 0; e < E; ++e) k[tid * E + e] = r[e];
    __syncthreads();
  }
}

// merge_sort_e with the smallest run length E (a power of two) that covers n;
// returns the padded length E * blockDim.x.
__device__ __forceinline__ int merge_sort(uint64_t *k, int n) {
  const int nt = blockDim.x;
  if (n <= nt) return merge_sort_e<1>(k, n), nt;
  if (n <= 2 * nt) return merge_sort_e<2>(k, n), 2 * nt;
  if (n <= 4 * nt) return merge_sort_e<4>(k, n), 4 * nt;
  if (n <= 8 * nt) return merge_sort_e<8>(k, n), 8 * nt;
  return merge_sort_e<16>(k, n), 16 * nt;
}

struct SelectParams {
  int b, K_max, P, C;
  int64_t n_cl, N;
  const uint32_t *bkt_off, *cl_off;
  const float *cent;
  const uint8_t *single;  // [n_cl] 1 if the cluster's bucket holds one cluster
  bool gate_off;
  float m0, m1;
  int *err;
};

// Sort capacity for probe budget P: all clusters of P buckets. Shared memory
// holds at most kSelectSmemKeys keys; a query with more candidate clusters
// sorts in its slab of global memory (select_slab_bytes, 0 when unneeded).
constexpr int kSelectSmemKeys = 2048;
__host__ __device__ inline int select_sort_cap(int P, int K_max) {
  int s = 1;
  while (s < P * K_max) s <<= 1;
  return s;
}
// at least one key per thread of the 128-thread select block (the merge
// sort's shortest padded length), at most kSelectSmemKeys
constexpr int kSelectMinKeys = 128;
__host__ __device__ inline int select_smem_cap(int P, int K_max) {
  const int s = select_sort_cap(P, K_max);
  return s < kSelectMinKeys ? kSelectMinKeys : (s < kSelectSmemKeys ? s : kSelectSmemKeys);
}
__host__ __device__ inline size_t select_scratch_bytes(int P, int K_max) {
  const int S = select_smem_cap(P, K_max);
  const int ib = S > 2 * P + 1 ? S : 2 * P + 1;
  return (size_t)S * 8 + (size_t)ib * 4;
}
__host__ __device__ inline size_t select_slab_bytes(int P, int K_max) {
  const int full = select_sort_cap(P, K_max);
  return full > select_smem_cap(P, K_max) ? (size_t)full * 12 : 0;
}

// Centroid distance d_c = sum_j (l_j - mu_cj)^2 as a sequential fmaf chain.
// When b is a multiple of 4 (rows 16-byte aligned) the row is loaded as
// float4s up front; the arithmetic is the same chain either way.
__device__ __forceinline__ float centroid_dist(const float *__restrict__ mu, const float *slog, int b) {
  float acc = 0.0f;
  if ((b & 3) == 0 && b <= 32) {
#pragma unroll
    for (int g = 0; g < 2; ++g) {
      float4 v[4];
#pragma unroll
      for (int q = 0; q < 4; ++q)
        if (16 * g + 4 * q < b) v[q] = __ldg(reinterpret_cast<const float4 *>(mu) + 4 * g + q);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        if (16 * g + 4 * q < b) {
          const float m[4] = {v[q].x, v[q].y, v[q].z, v[q].w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float t = __fsub_rn(slog[16 * g + 4 * q + e], m[e]);
            acc = __fmaf_rn(t, t, acc);
          }
        }
    }
    return acc;
  }
  for (int j = 0; j < b; ++j) {
    const float t = __fsub_rn(slog[j], __ldg(&mu[j]));
    acc = __fmaf_rn(t, t, acc);
  }
  return acc;
}

// Cluster of candidate slot s: slots are numbered probe by probe, off[i] the
// first slot of probe i (nondecreasing), c0[i] the first cluster of probe i.
__device__ __forceinline__ uint32_t slot_cluster(const int *off, const int *c0, int np, int s) {
  int lo = 0, hi = np - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (off[mid] <= s) lo = mid;
    else hi = mid - 1;
  }
  return (uint32_t)(c0[lo] + (s - off[lo]));
}

// One query: codes[0..np) -> the kept clusters C^dir U C^cent in (d, cluster)
// order and their refinement segments. Writes seg[i] = (first row, stream
// position) for i < nl, and L[i] (cluster index, -1 padded to Lmax) when L is
// not null. slog: the query's b logits in shared memory; scratch:
// select_scratch_bytes(P, K_max) bytes of shared memory; slab: this query's
// select_slab_bytes(P, K_max) bytes of global memory (null when that is 0);
// warp_sums: 32 ints; sred: 2 unsigned. Returns nl; *total = stream length.
// Whole block calls.
//
// The keys to sort (C^dir and the gate's survivors) are collected straight
// into shared memory: one pass over the candidate clusters computes their
// distances, keeps the single-cluster buckets' and takes d_min over the rest;
// a second pass recomputes the others' distances and keeps those within the
// gate. Only when they do not fit does the query fall back to sorting all its
// candidate keys in the global slab. Both give the same keys, and the sort
// orders them by exact value.
__device__ __forceinline__ int select_block(const SelectParams &sp, const float *slog,
                                            const uint32_t *codes, int np, unsigned char *scratch,
                                            unsigned char *slab, int *warp_sums, unsigned *sred,
                                            nr_seg *seg, int32_t *L, int Lmax, uint32_t *total) {
  const int tid = threadIdx.x, nt = blockDim.x;
  const int S_smem = select_smem_cap(sp.P, sp.K_max);
  const int S_full = select_sort_cap(sp.P, sp.K_max);
  uint64_t *keys = reinterpret_cast<uint64_t *>(scratch);
  int *ibuf = reinterpret_cast<int *>(scratch + (size_t)S_smem * 8);
  if (tid == 0) {
    sred[0] = 0xffffffffu;  // d_min bits over non-singleton candidates
    sred[1] = 0u;           // keys collected
  }
  int *cnt = ibuf;        // [P] clusters per probe -> exclusive offsets
  int *c0s = ibuf + sp.P;  // [P] first cluster per probe
  const uint32_t nb = 1u << sp.b;
  for (int i = tid; i < np; i += nt) {
    const uint32_t u = codes[i];
    int n = 0, c0 = 0;
    if (u >= nb) {
      set_err(sp.err, NR_DEV_BAD_CODE);
    } else {
      const uint32_t lo = __ldg(&sp.bkt_off[u]), hi = __ldg(&sp.bkt_off[u + 1]);
      if (hi < lo || (int64_t)hi > sp.n_cl) {
        set_err(sp.err, NR_DEV_BAD_BUCKET);
      } else {
        n = (int)(hi - lo);
        c0 = (int)lo;
        if (n > sp.K_max) {
          set_err(sp.err, NR_DEV_TOO_MANY);
          n = sp.K_max;
        }
      }
    }
    cnt[i] = n;
    c0s[i] = c0;
  }
  __syncthreads();
  int M = block_exclusive_scan(cnt, np, warp_sums);
  // One pass over the candidates. C^dir keys are collected from the back of
  // the key array; the other clusters from the front when they are within the
  // gate of the running d_min (for m1 >= 0 that gate is never tighter than the
  // final one: x + fmaf(m1, x, m0) does not decrease with x).
  if (tid == 0) sred[2] = 0u;  // keys collected from the front
  __syncthreads();
  const float m0 = sp.m0, m1 = sp.m1;
  const bool prefilter = !sp.gate_off && m1 >= 0.0f;
  for (int s = tid; s < M; s += nt) {
    const uint32_t c = slot_cluster(cnt, c0s, np, s);
    const float d = centroid_dist(sp.cent + (size_t)c * sp.b, slog, sp.b);
    const uint64_t key = ((uint64_t)__float_as_uint(d) << 32) | c;
    if (__ldg(&sp.single[c])) {
      const unsigned pos = atomicAdd(&sred[1], 1u);
      if (pos < (unsigned)S_smem) keys[S_smem - 1 - pos] = key;
    } else {
      const uint32_t db = __float_as_uint(d);
      const uint32_t prev = atomicMin(&sred[0], db);  // d >= 0: bits order as values
      bool maybe = true;
      if (prefilter) {
        const float dm = __uint_as_float(prev < db ? prev : db);
        maybe = d <= __fadd_rn(dm, __fmaf_rn(m1, dm, m0));
      }
      if (maybe) {
        const unsigned pos = atomicAdd(&sred[2], 1u);
        if (pos < (unsigned)S_smem) keys[pos] = key;
      }
    }
  }
  __syncthreads();
  const uint32_t dmin_bits = sred[0];
  float theta = __int_as_float(0x7f800000);
  if (!sp.gate_off && dmin_bits != 0xffffffffu) {
    const float dmin = __uint_as_float(dmin_bits);
    theta = __fadd_rn(dmin, __fmaf_rn(m1, dmin, m0));  // theta = d_min + M(d_min)
  }
  const int nA = (int)sred[1], nB = (int)sred[2];
  int Mk = nA + nB;
  if (Mk <= S_smem) {
    // keep the front keys within the final gate, compacted toward the front
    // (a key never moves up, and each chunk reads before it writes), then move
    // the C^dir keys down behind them
    int *flag = ibuf;  // the probe offsets are no longer needed
    __syncthreads();
    for (int i = tid; i < nB; i += nt)
      flag[i] = __uint_as_float((uint32_t)(keys[i] >> 32)) <= theta ? 1 : 0;
    __syncthreads();
    const int nS = block_exclusive_scan(flag, nB, warp_sums);
    for (int i0 = 0; i0 < nB; i0 += 4 * nt) {
      uint64_t kb[4];
      int rk[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int i = i0 + e * nt + tid;
        rk[e] = -1;
        kb[e] = 0;
        if (i < nB && (i + 1 < nB ? flag[i + 1] : nS) > flag[i]) {
          rk[e] = flag[i];
          kb[e] = keys[i];
        }
      }
      __syncthreads();
#pragma unroll
      for (int e = 0; e < 4; ++e)
        if (rk[e] >= 0) keys[rk[e]] = kb[e];
      __syncthreads();
    }
    for (int t0 = 0; t0 < nA; t0 += 4 * nt) {
      uint64_t kb[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int t = t0 + e * nt + tid;
        kb[e] = t < nA ? keys[S_smem - nA + t] : 0;
      }
      __syncthreads();
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int t = t0 + e * nt + tid;
        if (t < nA) keys[nS + t] = kb[e];
      }
      __syncthreads();
    }
    Mk = nS + nA;
  } else {
    Mk = S_smem + 1;  // does not fit: the slab path below
  }
  int Sn = 1;
  int *ints = ibuf;
  if (Mk <= S_smem) {
    M = Mk;
    Sn = merge_sort(keys, M);  // keys[M..Sn) = kEmpty
  } else {
    // more keys than shared memory holds: all candidate keys in the global slab
    // (slab is present: without it M <= S_full = S_smem)
    while (Sn < M) Sn <<= 1;
    if (slab == nullptr || Sn > S_full) {
      if (tid == 0) set_err(sp.err, NR_DEV_TOO_MANY);
      *total = 0;
      return 0;
    }
    keys = reinterpret_cast<uint64_t *>(slab);
    ints = reinterpret_cast<int *>(slab + (size_t)S_full * 8);
    for (int i = tid; i < np; i += nt) {  // each probe fills its clusters' slots
      const int o = cnt[i], n = (i + 1 < np ? cnt[i + 1] : M) - o;
      for (int j = 0; j < n; ++j) keys[o + j] = (uint64_t)(uint32_t)(c0s[i] + j);
    }
    __syncthreads();
    for (int s = tid; s < M; s += nt) {
      const uint32_t c = (uint32_t)keys[s];
      const float d = centroid_dist(sp.cent + (size_t)c * sp.b, slog, sp.b);
      const bool keep = __ldg(&sp.single[c]) || d <= theta;
      keys[s] = keep ? (((uint64_t)__float_as_uint(d) << 32) | c) : kEmpty;
    }
    for (int s = M + tid; s < Sn; s += nt) keys[s] = kEmpty;
    __syncthreads();
    bitonic_sort(keys, Sn);
  }
  // keep C^dir and the first C survivors in key order
  int *keep = ints;  // [Sn]
  for (int s = tid; s < Sn; s += nt) {
    const uint64_t kk = keys[s];
    keep[s] = (s < M && kk != kEmpty && !__ldg(&sp.single[(uint32_t)kk])) ? 1 : 0;
  }
  __syncthreads();
  block_exclusive_scan(keep, Sn, warp_sums);  // survivor rank in key order
  for (int s = tid; s < Sn; s += nt) {
    const uint64_t kk = keys[s];
    int kp = 0;
    if (s < M && kk != kEmpty) kp = __ldg(&sp.single[(uint32_t)kk]) ? 1 : (keep[s] < sp.C ? 1 : 0);
    keep[s] = kp;
  }
  __syncthreads();
  const int nl = block_exclusive_scan(keep, Sn, warp_sums);  // output positions
  for (int s = tid; s < Sn; s += nt) {
    const uint64_t kk = keys[s];
    if (s < M && kk != kEmpty) {
      const int pos = keep[s];
      const bool kept = (s + 1 < Sn ? keep[s + 1] : nl) > pos;
      if (kept) seg[pos].row0 = (uint32_t)kk;  // cluster index for now
    }
  }
  __syncthreads();
  int *len = ints;  // [nl]
  for (int i = tid; i < nl; i += nt) {
    const uint32_t c = seg[i].row0;
    if (L) L[i] = (int32_t)c;
    const uint32_t r0 = __ldg(&sp.cl_off[c]), r1 = __ldg(&sp.cl_off[c + 1]);
    int ln = 0;
    if (r1 < r0 || (int64_t)r1 > sp.N) set_err(sp.err, NR_DEV_BAD_CLUSTER);
    else ln = (int)(r1 - r0);
    len[i] = ln;
    seg[i].row0 = r0;
  }
  if (L)
    for (int i = nl + tid; i < Lmax; i += nt) L[i] = -1;
  __syncthreads();
  const int tot = block_exclusive_scan(len, nl, warp_sums);
  for (int i = tid; i < nl; i += nt) seg[i].pos = (uint32_t)len[i];
  __syncthreads();
  *total = (uint32_t)tot;
  return nl;
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

}  // namespace nrq
