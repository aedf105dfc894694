// route_warp: one warp per query binarises the logits, ranks the bits and
// lists the probe codes (Eq. 10, Algorithm 1).
#pragma once

#include "nrq_block.cuh"

namespace nrq {

__device__ __forceinline__ uint64_t pack_key(float cost, uint32_t size, uint32_t mask) {
  return ((uint64_t)__float_as_uint(cost) << 32) | ((uint64_t)size << 24) | (uint64_t)mask;
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
  // non-empty budget: bucket directory, and Q = the most flip sets examined
  // (NR_NONEMPTY_SCAN P); without it Q = P and bkt_off is unused
  const uint32_t *bkt_off;
  int nonempty, Q;
};

// Bytes of shared memory route_warp needs to examine at most Q flip sets:
// heap keys [(Q + 2) x 8 B], deviations by rank [32 x 4 B], and the table of
// left-to-right sums over subsets of ranks 0..7 [256 x 4 B]
__host__ __device__ inline size_t route_heap_bytes(int Q) { return (size_t)(Q + 2) * 8 + 128 + 1024; }

// Writes codes[0..n) (any address space) and returns n, uniform in the warp.
// Must be called by a whole warp. heap: route_heap_bytes(P) bytes of shared
// memory (8-byte aligned).
__device__ __forceinline__ int route_warp(const RouteParams &rp, const float *__restrict__ logit,
                                          unsigned char *heap, uint32_t *codes) {
  const int lane = threadIdx.x & 31;
  const int b = rp.b;
  uint64_t *hkey = reinterpret_cast<uint64_t *>(heap);
  float *ssd = reinterpret_cast<float *>(heap + (size_t)(rp.Q + 2) * 8);
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
  // psum[s] = left-to-right fp32 sum of ssd over the ranks in s (s over ranks
  // 0..7), built by adding each s's highest rank to psum of the rest: the
  // same order as summing the ranks one by one from 0.0f
  float *psum = ssd + 32;
  const int lo_ranks = b < 8 ? b : 8;
  if (lane == 0) psum[0] = 0.0f;
  __syncwarp();
  for (int j = 0; j < lo_ranks; ++j) {
    const float sj = ssd[j];
    for (int t = lane; t < (1 << j); t += 32) psum[(1 << j) + t] = __fadd_rn(psum[t], sj);
    __syncwarp();
  }
  // with the non-empty budget a code is listed only when its bucket holds a
  // cluster; every examined flip set counts toward Q
  auto listed = [&](uint32_t code) {
    if (!rp.nonempty) return true;
    uint32_t occ = 0;
    if (lane == 0) occ = __ldg(&rp.bkt_off[code + 1]) - __ldg(&rp.bkt_off[code]);
    return __shfl_sync(kFull, occ, 0) != 0u;
  };
  int n = 0, seen = 1, hs = 0;
  if (listed(u0)) {
    if (lane == 0) codes[0] = u0;
    n = 1;
  }
  if (rp.Q > 1 && rp.bsel >= 1 && ssd[0] <= rp.smax) {  // Q > 1: a flip set may be examined
    if (lane == 0) hkey[0] = pack_key(ssd[0], 1u, 1u);
    hs = 1;
  }
  __syncwarp();
  while (n < rp.P && hs > 0 && seen < rp.Q) {
    const uint64_t top = hkey[0];
    const uint32_t rmask = (uint32_t)top & 0xffffffu;
    const uint32_t size = ((uint32_t)top >> 24) & 0xffu;
    const float cost = __uint_as_float((uint32_t)(top >> 32));
    // ApplyFlips: code = u0 XOR (bits of the ranks in F)
    const uint32_t flips = __reduce_or_sync(kFull, ((rmask >> lane) & 1u) ? rbit : 0u);
    ++seen;
    if (listed(u0 ^ flips)) {
      if (lane == 0) codes[n] = u0 ^ flips;
      ++n;
    }
    const int m = 31 - __clz((int)rmask);
    bool v1 = false, v2 = false;
    uint64_t k1 = kEmpty, k2 = kEmpty;
    if (m + 1 < rp.bsel) {
      const float sdn = ssd[m + 1];
      // cost without rank m: fp32 sum from 0 over the other ranks, ascending
      // (ranks below 8 from the table, the rest one by one)
      const uint32_t rest = rmask & ~(1u << m);
      float costp = psum[rest & 0xffu];
      for (uint32_t mm = rest >> 8; mm; mm &= mm - 1) costp = __fadd_rn(costp, ssd[7 + __ffs(mm)]);
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
        if (32 * i + 1 >= hs) {  // a leaf (warp-uniform)
          if (lane == 0) hkey[i] = x;
          break;
        }
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

// ============================================================== route_block
// The same probe list by a threshold enumeration, one 128-thread block per
// query. The flip sets with cost <= T form a subtree of the tree above (costs
// never decrease along an edge), so for any T with at least N - 1 of them, the
// first N - 1 sets in key order are the N - 1 smallest keys of that subtree:
// enumerate it breadth first, order it, keep the front. T comes from counting
// subsets by cost on a grid of kRouteBins steps D over [0, T_range], T_range
// the cost of ranks {0..m-1} with 2^m >= N (its 2^m - 1 subsets cost no more,
// so the N - 1-th set does not either): each deviation rounded up to
// s_r = floor(delta_r / D) + 1 steps, the number of subsets with sum of steps
// <= c is a dynamic program over the ranks, and every such subset costs at most
// c D in exact arithmetic, below c D (1 + 2^-16) after fp32 rounding. The
// smallest c whose count reaches N (the empty set included) gives T.
//
// The subtree's keys are ordered by a bucket sort: kRouteBuckets buckets over
// [0, largest cost] by a monotone map of the cost (a key in a lower bucket
// costs less, so buckets keep key order), a histogram and scan give each
// bucket's range, and a key's rank is its bucket's start plus the number of
// smaller keys in its bucket. Keys are distinct (distinct rank masks), so the
// ranks are a permutation.
//
// Plain budget: N = P, and the first P - 1 ranks become the codes after the
// base code. Non-empty budget: N = min(Q, 2P, 4096) flip sets (the base code
// included) are enumerated; the bucket occupancy of each of the first
// min(N, Q) in key order is looked up (all lookups in flight at once), and a
// scan over them in rank order lists the first P non-empty codes. When that
// prefix holds fewer than P non-empty codes while more flip sets may be
// examined (fewer than Q examined, and sets above T remain), the block takes
// route_warp instead. Keys, ties and codes are those of route_warp; the R_max
// filter, a subtree beyond its capacity of 2N keys, or a bucket above
// kRouteBucketMax keys take route_warp too (warp 0 of the block).
constexpr int kRouteThreads = 128;
constexpr int kRouteBins = 480;
constexpr int kRouteSeedRanks = 7;          // the walk starts from all subsets of ranks 0..6
constexpr int kRouteDp = kRouteBins + 32;  // sums of rounded-up steps overshoot by < 1 per rank
constexpr int kRouteBuckets = 1024;        // <= 2 kRouteDp: the histogram reuses the count arrays
static_assert(kRouteBuckets <= 2 * kRouteDp, "the bucket histogram must fit the count arrays");
static_assert(kRouteDp % 32 == 0, "the count scan gives each lane kRouteDp / 32 bins");
constexpr int kRouteBucketMax = 64;
constexpr int kRouteNonemptyMax = 4096;    // flip sets a block enumerates for the non-empty budget

// Flip sets (the base code included) the block enumerates.
__host__ __device__ inline int route_enum_target(int P, int nonempty, int Q) {
  if (!nonempty) return P;
  int n = 2 * P < Q ? 2 * P : Q;
  return n < kRouteNonemptyMax ? n : kRouteNonemptyMax;
}
// Subtree capacity for an enumeration of N: 2N keys, a whole number of block strides.
__host__ __device__ inline int route_cap(int N) {
  const int c = 2 * N;
  return c <= kRouteThreads ? kRouteThreads : (c + kRouteThreads - 1) / kRouteThreads * kRouteThreads;
}

struct RouteSmem {
  uint64_t *keys;   // subtree keys; or route_warp's heap
  float *costp;     // per subtree key: its cost without the largest rank; then the bucket order
  uint32_t *rc;     // non-empty budget: code of rank r | occupied << 31
  uint32_t *dp;     // two count arrays of kRouteDp; then the bucket histogram
  uint32_t *flip;   // [3][256]: bit mask of the ranks in each byte of a rank mask
  float *ssd;       // deviation of rank r
  int *bitidx;      // bit index of rank r
  int *ctl;         // [0] tail, [1] chosen bin, [2] u0, [3] route_warp's count, [4] largest
                    // cost bits, [5] largest bucket, [6] base code occupied, [8..11] warp totals
};

__host__ __device__ inline size_t route_region_bytes(int N, int Q) {
  const size_t keys = (size_t)route_cap(N) * 8;
  const size_t heap = route_heap_bytes(Q);
  return ((keys > heap ? keys : heap) + 15) & ~(size_t)15;
}

// Shared memory of route_block for probe budget P (Q: route_warp's limit).
__host__ __device__ inline size_t route_block_bytes(int P, int nonempty, int Q) {
  const int N = route_enum_target(P, nonempty, Q);
  return route_region_bytes(N, Q) + (size_t)route_cap(N) * 4 * (nonempty ? 2 : 1) +
         (size_t)2 * kRouteDp * 4 + (size_t)3 * 256 * 4 + 32 * 4 + 32 * 4 + 16 * 4;
}

__device__ __forceinline__ RouteSmem route_carve(unsigned char *base, int N, int Q, int nonempty) {
  RouteSmem m;
  m.keys = reinterpret_cast<uint64_t *>(base);
  m.costp = reinterpret_cast<float *>(base + route_region_bytes(N, Q));
  m.rc = reinterpret_cast<uint32_t *>(m.costp + route_cap(N));
  m.dp = m.rc + (nonempty ? route_cap(N) : 0);
  m.flip = m.dp + 2 * kRouteDp;
  m.ssd = reinterpret_cast<float *>(m.flip + 3 * 256);
  m.bitidx = reinterpret_cast<int *>(m.ssd + 32);
  m.ctl = m.bitidx + 32;
  return m;
}

// Whether bucket `code` holds a cluster.
__device__ __forceinline__ bool route_occupied(const RouteParams &rp, uint32_t code) {
  return __ldg(&rp.bkt_off[code + 1]) != __ldg(&rp.bkt_off[code]);
}

// Writes codes[0..n) (any address space) and returns n, uniform in the block.
// Called by the whole 128-thread block; smem: route_block_bytes(P, nonempty, Q) bytes.
__device__ __forceinline__ int route_block(const RouteParams &rp, const float *__restrict__ logit,
                                           unsigned char *smem, uint32_t *codes) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int b = rp.b, bsel = rp.bsel, P = rp.P;
  const int N = route_enum_target(P, rp.nonempty, rp.Q);
  const int cap = route_cap(N);
  const RouteSmem m = route_carve(smem, N, rp.Q, rp.nonempty);
  if (warp == 0) {  // deviations, base code and ranks (Eq. 10, Sec. 3.2.3)
    float dj = __int_as_float(0x7f800000);
    bool bit = false;
    if (lane < b) {
      const float l = logit[lane];
      const float tj = rp.tau[lane];
      bit = l >= tj;
      dj = fabsf(__fsub_rn(l, tj));
    }
    const uint32_t u0 = __ballot_sync(kFull, bit);
    int rank = 0;
    for (int i = 0; i < b; ++i) {
      const float di = __shfl_sync(kFull, dj, i);
      if (di < dj || (di == dj && i < lane)) ++rank;
    }
    if (lane < b) {
      m.ssd[rank] = dj;
      m.bitidx[rank] = lane;
    }
    if (lane == 0) {
      m.ctl[0] = 0;
      m.ctl[1] = -1;
      m.ctl[2] = (int)u0;
      m.ctl[4] = 0;
      m.ctl[5] = 0;
      m.ctl[6] = rp.nonempty ? (route_occupied(rp, u0) ? 1 : 0) : 1;
    }
  }
  __syncthreads();
  const uint32_t u0 = (uint32_t)m.ctl[2];
  // flip[t][v] = the bits of the ranks 8t + i, i in v (ApplyFlips by bytes)
  for (int e = tid; e < 3 * 256; e += kRouteThreads) {
    const int t = e >> 8, v = e & 255;
    uint32_t f = 0;
    for (int i = 0; i < 8; ++i)
      if (((v >> i) & 1) && 8 * t + i < b) f |= 1u << m.bitidx[8 * t + i];
    m.flip[e] = f;
  }
  bool use_heap = rp.rmax > 0;
  float T = __int_as_float(0x7f800000);  // the whole tree
  const bool none = N <= 1 || bsel < 1;
  if (!use_heap && !none && N - 1 < (1 << bsel) - 1) {
    int mr = 0;
    while ((1 << mr) < N) ++mr;  // mr <= bsel here
    float thi = 0.0f;
    for (int r = 0; r < mr; ++r) thi = __fadd_rn(thi, m.ssd[r]);
    const float trange = fminf(thi, rp.smax);
    if (!(trange > 0.0f)) {
      T = trange;
    } else {
      // step D = T_range / kRouteBins (rounded); s_r = floor(q + 0.001) + 1
      // with q = delta_r / D rounded, whose error (< 1e-4 for q below
      // kRouteDp) the 0.001 covers, so s_r D >= delta_r exactly
      const float step = __fdiv_rn(trange, (float)kRouteBins);
      uint32_t *d0 = m.dp, *d1 = m.dp + kRouteDp;
      for (int c = tid; c < kRouteDp; c += kRouteThreads) d0[c] = 0u;
      // the counts over the first ranks in one step: each subset of ranks
      // 0 .. r0 - 1 (those that fit a bin, at most kRouteSeedRanks) adds one
      // to the bin of its sum of steps, as the passes below would
      const int rs = bsel < kRouteSeedRanks ? bsel : kRouteSeedRanks;
      int r0 = 0, sr_seed[kRouteSeedRanks];
#pragma unroll
      for (int r = 0; r < kRouteSeedRanks; ++r) {
        sr_seed[r] = 0;
        if (r < rs && r0 == r) {
          const float qv = __fdiv_rn(m.ssd[r], step);
          if (qv < (float)(kRouteDp - 2)) {
            sr_seed[r] = (int)__fadd_rn(qv, 0.001f) + 1;
            r0 = r + 1;
          }
        }
      }
      __syncthreads();
      if (tid < (1 << r0)) {
        int sum = 0;
#pragma unroll
        for (int r = 0; r < kRouteSeedRanks; ++r)
          if ((tid >> r) & 1) sum += sr_seed[r];
        if (sum < kRouteDp) atomicAdd(&d0[sum], 1u);
      }
      __syncthreads();
      for (int r = r0; r < bsel; ++r) {
        const float qv = __fdiv_rn(m.ssd[r], step);
        if (!(qv < (float)(kRouteDp - 2))) break;  // this rank and all later ones fit no bin
        const int sr = (int)__fadd_rn(qv, 0.001f) + 1;
        for (int c = tid; c < kRouteDp; c += kRouteThreads) d1[c] = d0[c] + (c >= sr ? d0[c - sr] : 0u);
        __syncthreads();
        uint32_t *t = d0;
        d0 = d1;
        d1 = t;
      }
      if (warp == 0) {  // smallest c with count(sum of steps <= c) >= N
        constexpr int per = kRouteDp / 32;
        uint32_t loc = 0;
        for (int i = 0; i < per; ++i) loc += d0[lane * per + i];
        uint32_t incl = loc;
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t v = __shfl_up_sync(kFull, incl, o);
          if (lane >= o) incl += v;
        }
        const unsigned hit = __ballot_sync(kFull, incl >= (uint32_t)N);
        if (hit) {
          const int src = __ffs(hit) - 1;
          if (lane == src) {
            uint32_t run = incl - loc;
            int c = lane * per;
            for (;; ++c) {
              run += d0[c];
              if (run >= (uint32_t)N) break;
            }
            m.ctl[1] = c;
          }
        }
      }
      __syncthreads();
      const int c = m.ctl[1];
      // T >= c D (1 + 2^-16): products rounded up
      T = c < 0 ? rp.smax : __fmul_ru(__fmul_ru((float)c, step), 1.0f + 1.0f / 65536.0f);
    }
  }
  const float teff = fminf(T, rp.smax);
  // breadth-first enumeration of the subtree with cost <= teff
  int tail = 0;
  // The walk starts from every non-empty subset of ranks 0 .. s7 - 1 within
  // the threshold, one a thread (the subtree's sets of those ranks: costs
  // never fall along an edge, so their ancestors are within it too), each
  // cost the left-to-right sum over its ranks as the tree's additions give
  // it; only seeds whose largest rank is s7 - 1 have children outside them.
  const int s7 = bsel < kRouteSeedRanks ? bsel : kRouteSeedRanks;
  if (!use_heap && !none) {
    {
      uint64_t key = kEmpty;
      float cp = 0.0f;
      if (tid >= 1 && tid < (1 << s7)) {
        const int mx = 31 - __clz(tid);
        float c = 0.0f;
        for (int r = 0; r <= mx; ++r)
          if ((tid >> r) & 1) {
            cp = c;
            c = __fadd_rn(c, m.ssd[r]);
          }
        if (c <= teff) key = pack_key(c, (uint32_t)__popc(tid), (uint32_t)tid);
      }
      const unsigned bal = __ballot_sync(kFull, key != kEmpty);
      int base = 0;
      if (lane == 0 && bal) base = atomicAdd(&m.ctl[0], __popc(bal));
      base = __shfl_sync(kFull, base, 0);
      if (key != kEmpty) {
        const int pos = base + __popc(bal & ((1u << lane) - 1u));
        m.keys[pos] = key;  // at most 127 seeds, within the capacity
        m.costp[pos] = cp;
      }
    }
    __syncthreads();
    int head = 0;
    tail = m.ctl[0];
    __syncthreads();  // every thread has read the tail before the first appends
    while (head < tail && tail <= cap) {
      const int nb = min(tail - head, kRouteThreads);
      uint64_t k1 = kEmpty, k2 = kEmpty;
      float p1 = 0.0f, p2 = 0.0f;
      if (tid < nb) {
        const uint64_t key = m.keys[head + tid];
        const float cp = m.costp[head + tid];
        const uint32_t mask = (uint32_t)key & 0xffffffu;
        const uint32_t size = ((uint32_t)key >> 24) & 0xffu;
        const float cost = __uint_as_float((uint32_t)(key >> 32));
        const int mx = 31 - __clz((int)mask);
        if (mx + 1 < bsel && mx + 1 >= s7) {  // children of smaller seeds are seeds
          const float sdn = m.ssd[mx + 1];
          const float c1 = __fadd_rn(cp, sdn);  // shift: rank mx -> mx + 1
          if (c1 <= teff) {
            k1 = pack_key(c1, size, mask + (1u << mx));
            p1 = cp;
          }
          const float c2 = __fadd_rn(cost, sdn);  // expand: add rank mx + 1
          if (c2 <= teff) {
            k2 = pack_key(c2, size + 1, mask | (1u << (mx + 1)));
            p2 = cost;
          }
        }
      }
      const int cnt = (k1 != kEmpty ? 1 : 0) + (k2 != kEmpty ? 1 : 0);
      int incl = cnt;
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += v;
      }
      int base = 0;
      if (lane == 31 && incl > 0) base = atomicAdd(&m.ctl[0], incl);
      base = __shfl_sync(kFull, base, 31);
      int pos = base + incl - cnt;
      if (k1 != kEmpty) {
        if (pos < cap) {
          m.keys[pos] = k1;
          m.costp[pos] = p1;
        }
        ++pos;
      }
      if (k2 != kEmpty && pos < cap) {
        m.keys[pos] = k2;
        m.costp[pos] = p2;
      }
      __syncthreads();
      head += nb;
      tail = m.ctl[0];
      __syncthreads();  // every thread has read the tail before the next appends
    }
    if (tail > cap) use_heap = true;  // uniform: every thread read the same tail
  }
  int *order = reinterpret_cast<int *>(m.costp);  // bucket order of the keys
  uint32_t *hist = m.dp;                           // kRouteBuckets counts, then bucket ends
  float scale = 0.0f;
  if (!use_heap && tail > 0) {
    // bucket histogram over [0, largest cost]; costs are non-negative, so
    // their bits order as their values
    for (int i = tid; i < kRouteBuckets; i += kRouteThreads) hist[i] = 0u;
    uint32_t cmax = 0u;
    for (int i = tid; i < tail; i += kRouteThreads) cmax = max(cmax, (uint32_t)(m.keys[i] >> 32));
    cmax = __reduce_max_sync(kFull, cmax);
    if (lane == 0) atomicMax(reinterpret_cast<unsigned *>(&m.ctl[4]), cmax);
    __syncthreads();
    const float top = __uint_as_float((uint32_t)m.ctl[4]);
    if (top > 0.0f && top < __int_as_float(0x7f800000))
      scale = __fdiv_rn((float)kRouteBuckets, top);
    for (int i = tid; i < tail; i += kRouteThreads) {
      const float cost = __uint_as_float((uint32_t)(m.keys[i] >> 32));
      atomicAdd(&hist[min(kRouteBuckets - 1, (int)__fmul_rn(cost, scale))], 1u);
    }
    __syncthreads();
    uint32_t bmax = 0u;
    for (int i = tid; i < kRouteBuckets; i += kRouteThreads) bmax = max(bmax, hist[i]);
    bmax = __reduce_max_sync(kFull, bmax);
    if (lane == 0) atomicMax(reinterpret_cast<unsigned *>(&m.ctl[5]), bmax);
    __syncthreads();
    if (m.ctl[5] > kRouteBucketMax) use_heap = true;  // uniform
  }
  int nlist = 0;  // codes listed (uniform)
  if (!use_heap) {
    if (tail > 0) {
      // bucket ranges: an exclusive scan of the histogram (kRouteBuckets /
      // 128 buckets a thread), then a scatter in which each key takes the
      // next slot of its bucket, leaving hist[z] = the end of bucket z
      constexpr int per = kRouteBuckets / kRouteThreads;
      uint32_t loc[per], sum = 0;
#pragma unroll
      for (int e = 0; e < per; ++e) {
        loc[e] = hist[tid * per + e];
        sum += loc[e];
      }
      uint32_t incl = sum;
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t v = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += v;
      }
      uint32_t *wsum = reinterpret_cast<uint32_t *>(m.ctl + 8);  // 4 warp totals
      if (lane == 31) wsum[warp] = incl;
      __syncthreads();
      uint32_t run = incl - sum;
      for (int w = 0; w < warp; ++w) run += wsum[w];
#pragma unroll
      for (int e = 0; e < per; ++e) {
        hist[tid * per + e] = run;
        run += loc[e];
      }
      __syncthreads();
      for (int i = tid; i < tail; i += kRouteThreads) {
        const float cost = __uint_as_float((uint32_t)(m.keys[i] >> 32));
        const int z = min(kRouteBuckets - 1, (int)__fmul_rn(cost, scale));
        order[atomicAdd(&hist[z], 1u)] = i;
      }
      __syncthreads();
    }
    // rank of each key = its bucket's start + the smaller keys of its bucket;
    // its code is u0 XOR the flips of its rank mask
    const int nexam = rp.nonempty ? min(tail, rp.Q - 1) : min(tail, P - 1);
    for (int i = tid; i < tail; i += kRouteThreads) {
      const uint64_t key = m.keys[i];
      const float cost = __uint_as_float((uint32_t)(key >> 32));
      const int z = min(kRouteBuckets - 1, (int)__fmul_rn(cost, scale));
      const int lo = z > 0 ? (int)hist[z - 1] : 0, hi = (int)hist[z];
      int r = lo;
      for (int j = lo; j < hi; ++j) r += m.keys[order[j]] < key ? 1 : 0;
      if (r < nexam) {
        const uint32_t mk = (uint32_t)key & 0xffffffu;
        const uint32_t code =
            u0 ^ (m.flip[mk & 255] | m.flip[256 + ((mk >> 8) & 255)] | m.flip[512 + (mk >> 16)]);
        if (rp.nonempty) m.rc[r] = code | (route_occupied(rp, code) ? 0x80000000u : 0u);
        else codes[1 + r] = code;
      }
    }
    if (!rp.nonempty) {
      if (tid == 0) codes[0] = u0;
      return 1 + nexam;
    }
    // non-empty budget: the non-empty codes of ranks [0, nexam) in rank
    // order, after the base code when it is non-empty
    __syncthreads();
    const int base_ne = m.ctl[6];
    const int per = (nexam + kRouteThreads - 1) / kRouteThreads;
    const int r0 = min(nexam, tid * per), r1 = min(nexam, r0 + per);
    int cnt = 0;
    for (int r = r0; r < r1; ++r) cnt += (int)(m.rc[r] >> 31);
    int incl = cnt;
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += v;
    }
    int *wsum = m.ctl + 8;
    __syncthreads();  // the warp totals of the scan above are read
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    int before = incl - cnt, total = 0;
    for (int w = 0; w < 4; ++w) {
      before += w < warp ? wsum[w] : 0;
      total += wsum[w];
    }
    // fewer than P non-empty codes, fewer than Q flip sets examined and sets
    // above the enumerated cost left: the heap continues where this stopped
    const bool complete = tail >= rp.Q - 1 || !(T < rp.smax);
    if (base_ne + total >= P || complete) {
      if (tid == 0 && base_ne) codes[0] = u0;
      int pos = base_ne + before;
      for (int r = r0; r < r1 && pos < P; ++r)
        if (m.rc[r] >> 31) codes[pos++] = m.rc[r] & 0x7fffffffu;
      return min(P, base_ne + total);
    }
    use_heap = true;  // uniform
  }
  __syncthreads();
  if (warp == 0) {
    const int n = route_warp(rp, logit, reinterpret_cast<unsigned char *>(m.keys), codes);
    if (lane == 0) m.ctl[3] = n;
  }
  __syncthreads();
  nlist = m.ctl[3];
  return nlist;
}

}  // namespace nrq
