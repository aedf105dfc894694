// route_warp: one warp per query binarises the logits, ranks the bits and
// lists the probe codes (Eq. 10, Algorithm 1).
#pragma once

#include "nrq_common.cuh"

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
};

// Bytes of shared memory route_warp needs for probe budget P.
// heap keys [(P + 2) x 8 B], deviations by rank [32 x 4 B], and the table of
// left-to-right sums over subsets of ranks 0..7 [256 x 4 B]
__host__ __device__ inline size_t route_heap_bytes(int P) { return (size_t)(P + 2) * 8 + 128 + 1024; }

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

}  // namespace nrq
