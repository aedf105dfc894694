// K2 route: binarisation (Eq. 10), deviation scores (Sec. 3.2.3) and the
// probe list of Algorithm 1 as an exact best-first enumeration of flip sets.
//
// Ranks order the bits by (delta_j, j); a flip set F is a set of ranks with key
//   (cost(F), |F|, rank mask),  cost = fp32 sum of delta over F, ascending rank.
// Flip sets form a tree rooted at {0}: a set whose largest rank is m has the
// children "shift" (m -> m+1) and "expand" (add m+1). Every child's key is
// larger than its parent's (delta sorted ascending, fp32 round-to-nearest is
// monotone), so popping the smallest key of the frontier P-1 times yields the
// first P sets in key order, the empty set (the base bucket) first. Costs are
// carried as (cost, cost without the largest rank), so each child's cost is
// one addition in the same left-to-right order a sequential sum would use.
#include <cuda_runtime.h>
#include <stdint.h>

#include "nr_internal.cuh"

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr uint64_t kEmpty = ~0ull;
constexpr int kGroup = 8;             // lanes per query
constexpr int kQPW = 32 / kGroup;     // queries per warp

__device__ __forceinline__ uint64_t pack_key(float cost, uint32_t size, uint32_t mask) {
  return ((uint64_t)__float_as_uint(cost) << 32) | ((uint64_t)size << 24) | (uint64_t)mask;
}

__device__ __forceinline__ uint64_t shfl_xor64(uint64_t v, int o) {
  const uint32_t lo = __shfl_xor_sync(kFull, (uint32_t)v, o, kGroup);
  const uint32_t hi = __shfl_xor_sync(kFull, (uint32_t)(v >> 32), o, kGroup);
  return ((uint64_t)hi << 32) | lo;
}

// One 8-lane group per query, four queries per warp. Lane gl of a group holds
// bits gl, gl + 8, gl + 16. The frontier is an 8-ary min-heap of
// (key, prefix cost) in shared memory: a pop that also inserts the shift child
// is one sift-down (the 8 lanes compare the 8 children of a node at once); the
// expand child is a sift-up by the group leader. The frontier never holds more
// than P + 1 entries.
__global__ void route_heap_kernel(const float *__restrict__ logits, const float *__restrict__ tau,
                                  int b, int bsel, int rmax, float smax, int64_t nq, int P, int cap,
                                  uint32_t *__restrict__ codes, int32_t *__restrict__ nprobe) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, wpb = blockDim.x >> 5;
  const int g = lane / kGroup, gl = lane % kGroup;
  const int slot = warp * kQPW + g;                 // group slot within the block
  const int nslot = wpb * kQPW;
  const int64_t q = ((int64_t)blockIdx.x * wpb + warp) * kQPW + g;
  const bool live = q < nq;
  uint64_t *hkey = reinterpret_cast<uint64_t *>(smem) + (size_t)slot * cap;
  float *hcp = reinterpret_cast<float *>(smem + (size_t)nslot * cap * 8) + (size_t)slot * cap;
  float *ssd = reinterpret_cast<float *>(smem + (size_t)nslot * cap * 12) + slot * 32;
  int *spi = reinterpret_cast<int *>(smem + (size_t)nslot * cap * 12 + (size_t)nslot * 128) + slot * 32;

  // Eq. 10 and the deviations of this lane's three bits
  float dj[3];
  uint32_t mybits = 0;
#pragma unroll
  for (int t = 0; t < 3; ++t) {
    const int j = gl + kGroup * t;
    dj[t] = __int_as_float(0x7f800000);
    if (live && j < b) {
      const float l = logits[q * b + j];
      const float tj = tau[j];
      if (l >= tj) mybits |= 1u << j;
      dj[t] = fabsf(__fsub_rn(l, tj));
    }
  }
  uint32_t u0 = mybits;
#pragma unroll
  for (int o = 1; o < kGroup; o <<= 1) u0 |= __shfl_xor_sync(kFull, u0, o, kGroup);
  // ranks by (delta, bit index)
  int rank[3] = {0, 0, 0};
  for (int i = 0; i < b; ++i) {
    const float di = __shfl_sync(kFull, dj[i / kGroup], i % kGroup, kGroup);
#pragma unroll
    for (int t = 0; t < 3; ++t) {
      const int j = gl + kGroup * t;
      if (di < dj[t] || (di == dj[t] && i < j)) ++rank[t];
    }
  }
#pragma unroll
  for (int t = 0; t < 3; ++t) {
    const int j = gl + kGroup * t;
    if (live && j < b) {
      ssd[rank[t]] = dj[t];
      spi[rank[t]] = j;
    }
  }
  __syncwarp();

  uint32_t *out = codes + (size_t)(live ? q : 0) * P;
  if (live && gl == 0) out[0] = u0;
  int n = 1, hs = 0;
  if (live && P > 1 && bsel >= 1 && ssd[0] <= smax) {
    if (gl == 0) {
      hkey[0] = pack_key(ssd[0], 1u, 1u);
      hcp[0] = 0.0f;
    }
    hs = 1;
  }
  __syncwarp();
  bool active = live && n < P && hs > 0;
  while (__any_sync(kFull, active)) {
    uint64_t top = kEmpty, x = kEmpty, c2key = kEmpty;
    float topcp = 0.0f, xcp = 0.0f, c2cp = 0.0f;
    bool push2 = false;
    if (active) {
      top = hkey[0];
      topcp = hcp[0];
      const uint32_t rmask = (uint32_t)top & 0xffffffu;
      const uint32_t size = ((uint32_t)top >> 24) & 0xffu;
      const float cost = __uint_as_float((uint32_t)(top >> 32));
      if (gl == 0) {  // ApplyFlips
        uint32_t f = 0, mm = rmask;
        while (mm) {
          const int r = __ffs(mm) - 1;
          f |= 1u << spi[r];
          mm &= mm - 1;
        }
        out[n] = u0 ^ f;
      }
      ++n;
      const int m = 31 - __clz((int)rmask);
      bool v1 = false, v2 = false;
      uint64_t k1 = kEmpty, k2 = kEmpty;
      float cp1 = 0.0f, cp2 = 0.0f;
      if (m + 1 < bsel) {
        const float sdn = ssd[m + 1];
        const float c1 = __fadd_rn(topcp, sdn);  // shift: rank m -> m + 1
        if (c1 <= smax) {
          v1 = true;
          k1 = pack_key(c1, size, rmask + (1u << m));
          cp1 = topcp;
        }
        if (rmax <= 0 || (int)size < rmax) {  // expand: add rank m + 1
          const float c2 = __fadd_rn(cost, sdn);
          if (c2 <= smax) {
            v2 = true;
            k2 = pack_key(c2, size + 1, rmask | (1u << (m + 1)));
            cp2 = cost;
          }
        }
      }
      // the root is replaced by a child, or by the last entry
      if (v1) {
        x = k1; xcp = cp1;
        if (v2) { push2 = true; c2key = k2; c2cp = cp2; }
      } else if (v2) {
        x = k2; xcp = cp2;
      } else {
        hs -= 1;
        if (hs > 0) { x = hkey[hs]; xcp = hcp[hs]; }
      }
    }
    __syncwarp();
    // sift-down of x from the root (groups with nothing to place idle along)
    int i = 0;
    bool sifting = active && x != kEmpty;
    while (__any_sync(kFull, sifting)) {
      uint64_t ck = kEmpty;
      int ci = -1;
      if (sifting) {
        const int c = kGroup * i + 1 + gl;
        if (c < hs) { ck = hkey[c]; ci = c; }
      }
      // group minimum over the 8 children (keys are unique)
      uint64_t mk = ck;
#pragma unroll
      for (int o = 1; o < kGroup; o <<= 1) {
        const uint64_t ok = shfl_xor64(mk, o);
        mk = ok < mk ? ok : mk;
      }
      const unsigned who = __ballot_sync(kFull, sifting && ck == mk && ci >= 0);
      const int src = __ffs((who >> (g * kGroup)) & 0xffu) - 1;  // lane in group holding the min
      const int mci = __shfl_sync(kFull, ci, src < 0 ? 0 : src, kGroup);
      if (sifting) {
        if (src >= 0 && mk < x) {
          if (gl == 0) {
            hkey[i] = mk;
            hcp[i] = hcp[mci];
          }
          i = mci;
        } else {
          if (gl == 0) {
            hkey[i] = x;
            hcp[i] = xcp;
          }
          sifting = false;
        }
      }
      __syncwarp();
    }
    // sift-up of the expand child
    if (push2 && gl == 0) {
      int j = hs;
      while (j > 0) {
        const int pj = (j - 1) / kGroup;
        const uint64_t pk = hkey[pj];
        if (pk < c2key) break;
        hkey[j] = pk;
        hcp[j] = hcp[pj];
        j = pj;
      }
      hkey[j] = c2key;
      hcp[j] = c2cp;
    }
    if (push2) hs += 1;
    __syncwarp();
    active = active && n < P && hs > 0;
  }
  if (live) {
    for (int t = n + gl; t < P; t += kGroup) out[t] = 0xffffffffu;
    if (gl == 0) nprobe[q] = n;
  }
}


// Warp-per-query variant: the frontier is a 32-ary min-heap in shared memory,
// so a sift-down level is one load per lane and two warp min-reductions
// (redux.sync) over the 32 children of a node; a 512-entry frontier is two
// levels deep. Lane j holds bit j.
__global__ void route_warp_kernel(const float *__restrict__ logits, const float *__restrict__ tau,
                                  int b, int bsel, int rmax, float smax, int64_t nq, int P, int cap,
                                  uint32_t *__restrict__ codes, int32_t *__restrict__ nprobe) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, wpb = blockDim.x >> 5;
  const int64_t q = (int64_t)blockIdx.x * wpb + warp;
  if (q >= nq) return;  // uniform per warp
  uint64_t *hkey = reinterpret_cast<uint64_t *>(smem) + (size_t)warp * cap;
  float *hcp = reinterpret_cast<float *>(smem + (size_t)wpb * cap * 8) + (size_t)warp * cap;
  float *ssd = reinterpret_cast<float *>(smem + (size_t)wpb * cap * 12) + warp * 32;

  float dj = __int_as_float(0x7f800000);
  bool bit = false;
  if (lane < b) {
    const float l = logits[q * b + lane];
    const float tj = tau[lane];
    bit = l >= tj;
    dj = fabsf(__fsub_rn(l, tj));
  }
  const uint32_t u0 = __ballot_sync(kFull, bit);
  int rank = 0;
  for (int i = 0; i < b; ++i) {
    const float di = __shfl_sync(kFull, dj, i);
    if (di < dj || (di == dj && i < lane)) ++rank;
  }
  // bit mask of the bit holding each rank: lane r gets 1 << pi[r]
  uint32_t rbit = 0;
  for (int j = 0; j < b; ++j) {
    const int rj = __shfl_sync(kFull, rank, j);
    if (rj == lane) rbit = 1u << j;
  }
  if (lane < b) ssd[rank] = dj;
  __syncwarp();

  uint32_t *out = codes + (size_t)q * P;
  if (lane == 0) out[0] = u0;
  int n = 1, hs = 0;
  if (P > 1 && bsel >= 1 && ssd[0] <= smax) {
    if (lane == 0) {
      hkey[0] = pack_key(ssd[0], 1u, 1u);
      hcp[0] = 0.0f;
    }
    hs = 1;
  }
  __syncwarp();
  while (n < P && hs > 0) {
    const uint64_t top = hkey[0];
    const float topcp = hcp[0];
    const uint32_t rmask = (uint32_t)top & 0xffffffu;
    const uint32_t size = ((uint32_t)top >> 24) & 0xffu;
    const float cost = __uint_as_float((uint32_t)(top >> 32));
    const uint32_t flips = __reduce_or_sync(kFull, ((rmask >> lane) & 1u) ? rbit : 0u);
    if (lane == 0) out[n] = u0 ^ flips;
    ++n;
    const int m = 31 - __clz((int)rmask);
    bool v1 = false, v2 = false;
    uint64_t k1 = kEmpty, k2 = kEmpty;
    float cp1 = 0.0f, cp2 = 0.0f;
    if (m + 1 < bsel) {
      const float sdn = ssd[m + 1];
      const float c1 = __fadd_rn(topcp, sdn);  // shift: rank m -> m + 1
      if (c1 <= smax) {
        v1 = true;
        k1 = pack_key(c1, size, rmask + (1u << m));
        cp1 = topcp;
      }
      if (rmax <= 0 || (int)size < rmax) {  // expand: add rank m + 1
        const float c2 = __fadd_rn(cost, sdn);
        if (c2 <= smax) {
          v2 = true;
          k2 = pack_key(c2, size + 1, rmask | (1u << (m + 1)));
          cp2 = cost;
        }
      }
    }
    uint64_t x = kEmpty;
    float xcp = 0.0f;
    if (v1) {
      x = k1;
      xcp = cp1;
    } else if (v2) {
      x = k2;
      xcp = cp2;
    } else {
      hs -= 1;
      if (hs > 0) {
        x = hkey[hs];
        xcp = hcp[hs];
      }
    }
    // sift-down of x from the root
    if (x != kEmpty) {
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
          const int mc = 32 * i + 1 + src;
          if (lane == src) {
            hkey[i] = mk;
            hcp[i] = hcp[mc];
          }
          i = mc;
          __syncwarp();
        } else {
          if (lane == 0) {
            hkey[i] = x;
            hcp[i] = xcp;
          }
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
          hcp[j] = hcp[pj];
          j = pj;
        }
        hkey[j] = k2;
        hcp[j] = cp2;
      }
      hs += 1;
    }
    __syncwarp();
  }
  for (int t = n + lane; t < P; t += 32) out[t] = 0xffffffffu;
  if (lane == 0) nprobe[q] = n;
}

}  // namespace

cudaError_t nr_launch_route(nr_index *ix, const float *d_logits, int64_t nq, int P,
                            uint32_t *d_codes, int32_t *d_nprobe, cudaStream_t s) {
  if (nq <= 0) return cudaSuccess;
  {
    const int cap = P + 2;
    const size_t per_warp = (size_t)cap * 12 + 128;
    int wpb = (int)((48u * 1024u) / per_warp);
    if (wpb > 4) wpb = 4;
    if (wpb < 1) wpb = 1;
    const size_t smem = per_warp * (size_t)wpb;
    cudaError_t e = cudaFuncSetAttribute(route_warp_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const nr_params &p = ix->params;
    const int bsel = (p.l_sel > 0 && p.l_sel < ix->b) ? p.l_sel : ix->b;
    const int64_t grid = (nq + wpb - 1) / wpb;
    route_warp_kernel<<<(unsigned)grid, 32 * wpb, smem, s>>>(d_logits, ix->tau, ix->b, bsel,
                                                              p.r_max, p.s_max, nq, P, cap, d_codes,
                                                              d_nprobe);
    ix->launches += 1;
    return cudaGetLastError();
  }
  const int cap = P + 2;
  const size_t per_group = (size_t)cap * 12 + 256;
  int wpb = (int)((96u * 1024u) / (per_group * kQPW));
  if (wpb > 4) wpb = 4;
  if (wpb < 1) wpb = 1;
  const size_t smem = per_group * (size_t)(wpb * kQPW);
  cudaError_t e = cudaFuncSetAttribute(route_heap_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  const nr_params &p = ix->params;
  const int bsel = (p.l_sel > 0 && p.l_sel < ix->b) ? p.l_sel : ix->b;
  const int64_t qpb = (int64_t)wpb * kQPW;
  const int64_t grid = (nq + qpb - 1) / qpb;
  route_heap_kernel<<<(unsigned)grid, 32 * wpb, smem, s>>>(d_logits, ix->tau, ix->b, bsel, p.r_max,
                                                            p.s_max, nq, P, cap, d_codes, d_nprobe);
  ix->launches += 1;
  return cudaGetLastError();
}
