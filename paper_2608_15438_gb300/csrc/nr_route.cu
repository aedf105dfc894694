// K2 route: binarisation (Eq. 10), deviation scores (Sec. 3.2.3) and the
// probe list of Algorithm 1 as an exact best-first enumeration of flip sets.
//
// One warp per query. Lane j holds bit j. Ranks order the bits by
// (delta_j, j); a flip set F is a set of ranks with key
//   (cost(F), |F|, rank mask),  cost = fp32 sum of delta over F, ascending rank.
// Flip sets form a tree rooted at {0}: a set whose largest rank is m has the
// children "shift" (m -> m+1) and "expand" (add m+1). Every child's key is
// larger than its parent's (delta sorted ascending, fp32 round-to-nearest is
// monotone), so popping the smallest key of the frontier P-1 times yields the
// first P sets in key order, the empty set (the base bucket) first. Costs are
// carried as (cost, cost without the largest rank), so each child's cost is
// one addition in the same left-to-right order a sequential sum would use.
//
// The frontier lives in shared memory; slot s belongs to lane s % 32, which
// keeps the minimum of its own slots in registers. A pop is two warp
// min-reductions, a ballot and one rescan by the owning lane.
#include <cuda_runtime.h>
#include <stdint.h>

#include "nr_internal.cuh"

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr uint64_t kEmpty = ~0ull;

__device__ __forceinline__ uint64_t pack_key(float cost, uint32_t size, uint32_t mask) {
  return ((uint64_t)__float_as_uint(cost) << 32) | ((uint64_t)size << 24) | (uint64_t)mask;
}

__global__ void route_kernel(const float *__restrict__ logits, const float *__restrict__ tau, int b,
                             int bsel, int rmax, float smax, int64_t nq, int P, int cap,
                             uint32_t *__restrict__ codes, int32_t *__restrict__ nprobe) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, wpb = blockDim.x >> 5;
  const int64_t q = (int64_t)blockIdx.x * wpb + warp;
  if (q >= nq) return;  // uniform per warp
  uint64_t *skey = reinterpret_cast<uint64_t *>(smem) + (size_t)warp * cap;
  float *scostp = reinterpret_cast<float *>(smem + (size_t)wpb * cap * 8) + (size_t)warp * cap;
  float *ssd = reinterpret_cast<float *>(smem + (size_t)wpb * cap * 12) + warp * 32;
  int *spi = reinterpret_cast<int *>(smem + (size_t)wpb * cap * 12 + (size_t)wpb * 128) + warp * 32;

  // Eq. 10: bit j set iff l_j >= tau_j; deviation delta_j = |l_j - tau_j|
  float dj = __int_as_float(0x7f800000);
  bool bit = false;
  if (lane < b) {
    const float l = logits[q * b + lane];
    const float tj = tau[lane];
    bit = l >= tj;
    dj = fabsf(__fsub_rn(l, tj));
  }
  const uint32_t u0 = __ballot_sync(kFull, bit);
  // rank of bit `lane` by (delta, bit index)
  int rank = 0;
  for (int i = 0; i < b; ++i) {
    const float di = __shfl_sync(kFull, dj, i);
    if (di < dj || (di == dj && i < lane)) ++rank;
  }
  if (lane < b) {
    ssd[rank] = dj;
    spi[rank] = lane;
  }
  __syncwarp();
  const float sd = lane < b ? ssd[lane] : 0.0f;  // delta of rank `lane`
  const int pi = lane < b ? spi[lane] : 0;        // bit index of rank `lane`

  uint32_t *out = codes + (size_t)q * P;
  if (lane == 0) out[0] = u0;
  int n = 1;
  int nslots = 0;
  uint32_t my_hi = 0xffffffffu, my_lo = 0xffffffffu;
  int my_slot = -1;

  const float sd0 = __shfl_sync(kFull, sd, 0);
  if (P > 1 && bsel >= 1 && sd0 <= smax) {
    if (lane == 0) {
      const uint64_t key = pack_key(sd0, 1u, 1u);
      skey[0] = key;
      scostp[0] = 0.0f;
      my_hi = (uint32_t)(key >> 32);
      my_lo = (uint32_t)key;
      my_slot = 0;
    }
    nslots = 1;
  }
  __syncwarp();

  while (n < P) {
    const uint32_t hmin = __reduce_min_sync(kFull, my_hi);
    const uint32_t lmin = __reduce_min_sync(kFull, my_hi == hmin ? my_lo : 0xffffffffu);
    if (hmin == 0xffffffffu && lmin == 0xffffffffu) break;  // frontier empty
    const unsigned own = __ballot_sync(kFull, my_slot >= 0 && my_hi == hmin && my_lo == lmin);
    const int owner = __ffs(own) - 1;
    const int slot = __shfl_sync(kFull, my_slot, owner);
    const float costp = scostp[slot];
    const uint32_t rmask = lmin & 0xffffffu;
    const uint32_t size = lmin >> 24;
    const float cost = __uint_as_float(hmin);
    // ApplyFlips: code = u0 XOR (bits of the ranks in F)
    const uint32_t flips =
        __reduce_or_sync(kFull, (lane < b && ((rmask >> lane) & 1u)) ? (1u << pi) : 0u);
    if (lane == 0) out[n] = u0 ^ flips;
    ++n;
    __syncwarp();
    if (lane == owner) {
      skey[slot] = kEmpty;
      uint64_t best = kEmpty;
      int bs = -1;
      for (int s = lane; s < nslots; s += 32) {
        const uint64_t kk = skey[s];
        if (kk < best) {
          best = kk;
          bs = s;
        }
      }
      my_hi = (uint32_t)(best >> 32);
      my_lo = (uint32_t)best;
      my_slot = bs;
    }
    const int m = 31 - __clz((int)rmask);  // largest rank in F
    if (m + 1 < bsel) {
      const float sdn = __shfl_sync(kFull, sd, m + 1);
      // shift: replace rank m by m + 1
      const float c1 = __fadd_rn(costp, sdn);
      if (c1 <= smax) {
        const int s = nslots++;
        if (lane == (s & 31)) {
          const uint64_t key = pack_key(c1, size, rmask + (1u << m));
          skey[s] = key;
          scostp[s] = costp;
          if (key < (((uint64_t)my_hi << 32) | my_lo)) {
            my_hi = (uint32_t)(key >> 32);
            my_lo = (uint32_t)key;
            my_slot = s;
          }
        }
      }
      // expand: add rank m + 1
      if (rmax <= 0 || (int)size < rmax) {
        const float c2 = __fadd_rn(cost, sdn);
        if (c2 <= smax) {
          const int s = nslots++;
          if (lane == (s & 31)) {
            const uint64_t key = pack_key(c2, size + 1, rmask | (1u << (m + 1)));
            skey[s] = key;
            scostp[s] = cost;
            if (key < (((uint64_t)my_hi << 32) | my_lo)) {
              my_hi = (uint32_t)(key >> 32);
              my_lo = (uint32_t)key;
              my_slot = s;
            }
          }
        }
      }
    }
    __syncwarp();
  }
  for (int i = n + lane; i < P; i += 32) out[i] = 0xffffffffu;
  if (lane == 0) nprobe[q] = n;
}

}  // namespace

cudaError_t nr_launch_route(nr_index *ix, const float *d_logits, int64_t nq, int P,
                            uint32_t *d_codes, int32_t *d_nprobe, cudaStream_t s) {
  if (nq <= 0) return cudaSuccess;
  const int cap = 2 * P;
  const size_t per_warp = (size_t)cap * 12 + 256;
  int wpb = (int)((96u * 1024u) / per_warp);
  if (wpb > 8) wpb = 8;
  if (wpb < 1) wpb = 1;
  const size_t smem = per_warp * (size_t)wpb;
  cudaError_t e = cudaFuncSetAttribute(route_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  const nr_params &p = ix->params;
  const int bsel = (p.l_sel > 0 && p.l_sel < ix->b) ? p.l_sel : ix->b;
  const int64_t grid = (nq + wpb - 1) / wpb;
  route_kernel<<<(unsigned)grid, 32 * wpb, smem, s>>>(d_logits, ix->tau, ix->b, bsel, p.r_max,
                                                       p.s_max, nq, P, cap, d_codes, d_nprobe);
  ix->launches += 1;
  return cudaGetLastError();
}
