// Index construction on the GPU (neuroute_build.h; paper Sec. 3.3, thresholds
// Sec. 3.2.3): per-bit lower medians by a radix select over order-preserving
// keys, codes, a stable sort of ids by code, bucket-local k-means with one
// warp per bucket (one CTA for large buckets), the two CSR levels, and the
// placement of the rows in stored order.
//
// The k-means arithmetic follows a fixed definition that does not depend on
// the order of parallel work: fp32 distances with every product and sum
// rounded, centroid sums in fixed-point integers, integer seeding weights with
// exact prefix sums. The host builder follows the same definition, so both
// write the same index from the same logits.
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include <cub/device/device_radix_sort.cuh>
#include <cub/device/device_scan.cuh>

#include <new>
#include <vector>

#include "neuroute.h"
#include "neuroute_build.h"
#include "nr_internal.cuh"

namespace {

constexpr int kBMax = 24;          // code bits
constexpr int kKMax = 64;          // clusters per bucket
constexpr int kMaxSample = 4096;   // sample_per_cluster
constexpr int64_t kWarpRows = 4096;  // buckets up to this size: one warp; larger: one CTA
constexpr int kCtaThreads = 256;

// ---------------------------------------------------------------------------
// Arithmetic of the build definition (identical on the host builder)
// ---------------------------------------------------------------------------

__host__ __device__ __forceinline__ uint32_t float_key(float x) {
  uint32_t u;
  memcpy(&u, &x, 4);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__host__ __device__ __forceinline__ float key_float(uint32_t k) {
  const uint32_t u = (k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k;
  float x;
  memcpy(&x, &u, 4);
  return x;
}
// e with v = f 2^e, f in [0.5, 1), for a positive finite double
__host__ __device__ __forceinline__ int exponent_of(double v) {
  uint64_t bits;
  memcpy(&bits, &v, 8);
  return (int)((bits >> 52) & 0x7FF) - 1022;
}
__host__ __device__ __forceinline__ double pow2(int e) {
  const uint64_t bits = (uint64_t)(e + 1023) << 52;
  double v;
  memcpy(&v, &bits, 8);
  return v;
}
__device__ __forceinline__ uint64_t splitmix64(uint64_t &s) {
  uint64_t z = (s += 0x9E3779B97F4A7C15ull);
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
__device__ __forceinline__ int64_t uniform_pick(uint64_t draw, int64_t m) {
  const double u = __dmul_rn((double)(draw >> 11), 1.0 / 9007199254740992.0);
  const int64_t p = (int64_t)__dmul_rn(u, (double)m);
  return p < m ? p : m - 1;
}
// fp32 squared distance, each product and sum rounded, j ascending
__device__ __forceinline__ float dist_rn(const float (&l)[kBMax], const float *c, int b) {
  float s = 0.0f;
#pragma unroll
  for (int j = 0; j < kBMax; ++j)
    if (j < b) {
      const float t = __fsub_rn(l[j], c[j]);
      s = __fadd_rn(s, __fmul_rn(t, t));
    }
  return s;
}
__device__ __forceinline__ void load_logits(const float *__restrict__ L, uint32_t r, int b,
                                            float (&l)[kBMax]) {
  const float *p = L + (size_t)r * b;
#pragma unroll
  for (int j = 0; j < kBMax; ++j) l[j] = j < b ? __ldg(p + j) : 0.0f;
}

// ---------------------------------------------------------------------------
// Step 1/2: fixed-point scale and medians
// ---------------------------------------------------------------------------

__global__ void absmax_kernel(const float *__restrict__ L, int64_t n, unsigned int *out) {
  unsigned int m = 0;
  const uint32_t *u = reinterpret_cast<const uint32_t *>(L);
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const unsigned int v = __ldg(u + i) & 0x7FFFFFFFu;
    m = v > m ? v : m;
  }
  for (int o = 16; o; o >>= 1) {
    const unsigned int w = __shfl_xor_sync(0xffffffffu, m, o);
    m = w > m ? w : m;
  }
  if ((threadIdx.x & 31) == 0 && m) atomicMax(out, m);
}

// histogram of key digit (key >> shift) & 255 per column, over the elements
// whose higher digits equal prefix[j]
__global__ void median_hist_kernel(const float *__restrict__ L, int64_t N, int b, int shift,
                                   const uint32_t *__restrict__ prefix, uint32_t *hist) {
  extern __shared__ uint32_t sh[];  // [b][256]
  __shared__ uint32_t spre[kBMax];
  for (int i = threadIdx.x; i < b * 256; i += blockDim.x) sh[i] = 0;
  if (threadIdx.x < b) spre[threadIdx.x] = prefix[threadIdx.x];
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int64_t nwarps = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t base = ((int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5)) * 32; base < N;
       base += nwarps * 32) {
    const int64_t r = base + lane;
    const bool valid = r < N;
    for (int j = 0; j < b; ++j) {
      const uint32_t key = valid ? float_key(__ldg(L + (size_t)r * b + j)) : 0u;
      const bool match = valid && (shift == 24 || (key >> (shift + 8)) == spre[j]);
      const int bin = match ? j * 256 + (int)((key >> shift) & 255u) : -1;
      const unsigned peers = __match_any_sync(0xffffffffu, bin);
      if (match && lane == __ffs(peers) - 1) atomicAdd(&sh[bin], (uint32_t)__popc(peers));
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < b * 256; i += blockDim.x)
    if (sh[i]) atomicAdd(&hist[i], sh[i]);
}

// per column: the digit holding rank[j]; rank and prefix move to it; the
// column's histogram is cleared for the next pass. After the last digit the
// prefix is the whole key: tau[j].
__global__ void median_pick_kernel(uint32_t *hist, uint32_t *prefix, uint32_t *rank, int b,
                                   int shift, float *tau) {
  const int j = threadIdx.x;
  if (j >= b) return;
  uint32_t *h = hist + j * 256;
  const uint32_t r = rank[j];
  uint32_t cum = 0;
  int digit = 255;
  for (int d = 0; d < 256; ++d) {
    if (cum + h[d] > r) {
      digit = d;
      break;
    }
    cum += h[d];
  }
  rank[j] = r - cum;
  prefix[j] = shift == 24 ? (uint32_t)digit : ((prefix[j] << 8) | (uint32_t)digit);
  for (int d = 0; d < 256; ++d) h[d] = 0;
  if (shift == 0) tau[j] = key_float(prefix[j]);
}

// ---------------------------------------------------------------------------
// Step 3: codes, bucket sizes and the bucket list
// ---------------------------------------------------------------------------

__global__ void codes_kernel(const float *__restrict__ L, int64_t N, int b,
                             const float *__restrict__ tau, uint32_t *codes, uint32_t *ids) {
  __shared__ float st[kBMax];
  if (threadIdx.x < b) st[threadIdx.x] = tau[threadIdx.x];
  __syncthreads();
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < N;
       r += (int64_t)gridDim.x * blockDim.x) {
    uint32_t u = 0;
    for (int j = 0; j < b; ++j)
      if (__ldg(L + (size_t)r * b + j) >= st[j]) u |= 1u << j;
    codes[r] = u;
    ids[r] = (uint32_t)r;
  }
}

__global__ void count_kernel(const uint32_t *__restrict__ codes, int64_t N, uint32_t *cnt) {
  const int lane = threadIdx.x & 31;
  for (int64_t base = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) & ~(int64_t)31; base < N;
       base += (int64_t)gridDim.x * blockDim.x) {
    const int64_t p = base + lane;
    const int64_t c = p < N ? (int64_t)codes[p] : -1;
    const unsigned peers = __match_any_sync(0xffffffffu, c);
    if (c >= 0 && lane == __ffs(peers) - 1) atomicAdd(&cnt[c], (uint32_t)__popc(peers));
  }
}

__global__ void flag_kernel(const uint32_t *__restrict__ cnt, int64_t nb, uint32_t *flag) {
  for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u <= nb;
       u += (int64_t)gridDim.x * blockDim.x)
    flag[u] = (u < nb && cnt[u] > 0) ? 1u : 0u;
}

// non-empty codes in order; clusters per bucket K_B; the large-bucket list
__global__ void bucket_list_kernel(const uint32_t *__restrict__ cnt, const uint32_t *__restrict__ pos,
                                   int64_t nb, int K_max, int t, uint32_t *ne_code, uint32_t *kcount,
                                   uint32_t *big_e, uint32_t *big_n, unsigned int *nbig) {
  for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < nb;
       u += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t n = cnt[u];
    if (n == 0) continue;
    const uint32_t e = pos[u];
    ne_code[e] = (uint32_t)u;
    int64_t K = ((int64_t)n + t - 1) / t;
    if (K > K_max) K = K_max;
    if (K > (int64_t)n) K = n;
    if (K < 1) K = 1;
    kcount[e] = (uint32_t)K;
    if ((int64_t)n > kWarpRows) {
      const unsigned int i = atomicAdd(nbig, 1u);
      big_e[i] = e;
      big_n[i] = n;
    }
  }
}

// ---------------------------------------------------------------------------
// Step 4: bucket-local k-means, one group (a warp or a CTA) per bucket
// ---------------------------------------------------------------------------

struct KmArgs {
  const float *L;          // logits [N x b]
  const uint32_t *ids_s;   // ids sorted by code (ascending within a code)
  const uint32_t *bstart;  // [2^b + 1] first stored row of each code
  const uint32_t *ne_code; // [ne] non-empty codes, ascending
  const uint32_t *kslot;   // [ne + 1] first cluster slot of each bucket
  const uint32_t *big_e;   // large buckets, largest first
  int64_t ne, nbig;
  uint8_t *labels;         // [N] cluster of each row, by sorted position
  uint32_t *out_ids;       // [N] ids in stored order
  float *slot_cent;        // [slots x b]
  uint32_t *slot_cnt;      // [slots] rows per kept cluster
  uint32_t *ncl;           // [ne] kept clusters per bucket
  float *dmin;             // [groups x mcap] seeding scratch
  int64_t mcap;
  unsigned int *counter;   // [2] work counters (warp buckets, CTA buckets)
  int b, K_max, t, iters, S;
  uint64_t seed;
  double scale, inv_scale;
};

// shared memory of one group
struct KmSmem {
  float *cent;                // [K_max * b]
  unsigned long long *sum;    // [K_max * b] fixed-point sums
  uint32_t *cnt;              // [K_max]
  int32_t *remap;             // [K_max] kept index or -1
  uint32_t *off;              // [K_max] placement cursor
  uint32_t *wcnt;             // [NW * K_max] per-warp label counts of a chunk
  unsigned long long *red;    // [NW] reduction scratch
  long long *misc;            // [4] broadcast slots
};

__host__ __device__ inline size_t km_smem_bytes(int K_max, int b, int nw) {
  size_t o = 0;
  o += (size_t)K_max * b * 8;   // sum
  o += (size_t)K_max * b * 4;   // cent
  o += (size_t)K_max * 4 * 3;   // cnt, remap, off
  o += (size_t)nw * K_max * 4;  // wcnt
  o = (o + 7) & ~(size_t)7;
  o += (size_t)nw * 8 + 32;     // red, misc
  return (o + 15) & ~(size_t)15;
}

__device__ inline KmSmem km_carve(unsigned char *p, int K_max, int b, int nw) {
  KmSmem m;
  m.sum = reinterpret_cast<unsigned long long *>(p);
  p += (size_t)K_max * b * 8;
  m.cent = reinterpret_cast<float *>(p);
  p += (size_t)K_max * b * 4;
  m.cnt = reinterpret_cast<uint32_t *>(p);
  p += (size_t)K_max * 4;
  m.remap = reinterpret_cast<int32_t *>(p);
  p += (size_t)K_max * 4;
  m.off = reinterpret_cast<uint32_t *>(p);
  p += (size_t)K_max * 4;
  m.wcnt = reinterpret_cast<uint32_t *>(p);
  p += (size_t)nw * K_max * 4;
  p = reinterpret_cast<unsigned char *>(((uintptr_t)p + 7) & ~(uintptr_t)7);
  m.red = reinterpret_cast<unsigned long long *>(p);
  p += (size_t)nw * 8;
  m.misc = reinterpret_cast<long long *>(p);
  return m;
}

template <int NT>
__device__ __forceinline__ void gsync() {
  if (NT == 32)
    __syncwarp();
  else
    __syncthreads();
}

template <int NT>
__device__ float group_max(float v, const KmSmem &m) {
  for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  if (NT == 32) return v;
  const int w = threadIdx.x >> 5, nw = NT / 32;
  gsync<NT>();
  if ((threadIdx.x & 31) == 0) reinterpret_cast<float *>(m.red)[w] = v;
  gsync<NT>();
  float r = reinterpret_cast<float *>(m.red)[0];
  for (int i = 1; i < nw; ++i) r = fmaxf(r, reinterpret_cast<float *>(m.red)[i]);
  gsync<NT>();
  return r;
}

// exclusive prefix of v over the group's threads in rank order; *total = sum
template <int NT>
__device__ unsigned long long group_excl_scan(unsigned long long v, const KmSmem &m,
                                              unsigned long long *total) {
  const int lane = threadIdx.x & 31;
  unsigned long long x = v;
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  const unsigned long long wtot = __shfl_sync(0xffffffffu, x, 31);
  if (NT == 32) {
    *total = wtot;
    return x - v;
  }
  const int w = threadIdx.x >> 5, nw = NT / 32;
  gsync<NT>();
  if (lane == 31) m.red[w] = wtot;
  gsync<NT>();
  unsigned long long before = 0, all = 0;
  for (int i = 0; i < nw; ++i) {
    if (i < w) before += m.red[i];
    all += m.red[i];
  }
  gsync<NT>();
  *total = all;
  return before + x - v;
}

// k-means of bucket e by a group of NT threads (rank g); dmin: this group's
// seeding scratch of at least min(n, S K) floats.
template <int NT>
__device__ void kmeans_bucket(const KmArgs &a, int64_t e, const KmSmem &m, float *dmin) {
  const int g = threadIdx.x % NT;
  const int b = a.b;
  const uint32_t code = a.ne_code[e];
  const int64_t lo = a.bstart[code];
  const int64_t n = (int64_t)a.bstart[code + 1] - lo;
  const uint32_t *mem = a.ids_s + lo;
  uint8_t *lab = a.labels + lo;
  const int K = (int)(a.kslot[e + 1] - a.kslot[e]);
  float l[kBMax];

  if (K > 1) {
    // k-means++ seeding on the strided sample (one splitmix64 stream per bucket)
    uint64_t s = a.seed * 0x100000001B3ull ^ ((uint64_t)code * 0x9E3779B97F4A7C15ull);
    int64_t mm = (int64_t)a.S * K;
    const int64_t ms = n < mm ? n : mm;
    const int64_t q = (ms + NT - 1) / NT;
    const int64_t i0 = (int64_t)g * q, i1 = i0 + q < ms ? i0 + q : ms;
    auto sample_row = [&](int64_t i) { return mem[(uint64_t)i * (uint64_t)n / (uint64_t)ms]; };
    if (g == 0) m.misc[0] = uniform_pick(splitmix64(s), ms);
    gsync<NT>();
    {
      const uint32_t r = sample_row(m.misc[0]);
      for (int j = g; j < b; j += NT) m.cent[j] = a.L[(size_t)r * b + j];
    }
    for (int64_t i = i0; i < i1; ++i) dmin[i] = __int_as_float(0x7f800000);
    for (int k = 1; k < K; ++k) {
      gsync<NT>();  // centroid k - 1 written
      float mx = 0.0f;
      for (int64_t i = i0; i < i1; ++i) {
        load_logits(a.L, sample_row(i), b, l);
        const float d = dist_rn(l, m.cent + (size_t)(k - 1) * b, b);
        const float dm = d < dmin[i] ? d : dmin[i];
        dmin[i] = dm;
        mx = dm > mx ? dm : mx;
      }
      mx = group_max<NT>(mx, m);
      if (g == 0) {
        m.misc[1] = (long long)splitmix64(s);
        m.misc[0] = -1;
      }
      gsync<NT>();
      const uint64_t draw = (uint64_t)m.misc[1];
      if (mx > 0.0f) {
        const double mult = pow2(50 - exponent_of((double)mx));
        unsigned long long local = 0;
        for (int64_t i = i0; i < i1; ++i) local += (unsigned long long)__dmul_rn((double)dmin[i], mult);
        unsigned long long tot;
        const unsigned long long ex = group_excl_scan<NT>(local, m, &tot);
        if (tot > 0) {
          const unsigned long long r = __umul64hi(draw, tot);
          if (ex <= r && r < ex + local) {
            unsigned long long acc = ex;
            for (int64_t i = i0; i < i1; ++i) {
              acc += (unsigned long long)__dmul_rn((double)dmin[i], mult);
              if (acc > r) {
                m.misc[0] = i;
                break;
              }
            }
          }
        }
      }
      gsync<NT>();
      if (g == 0 && m.misc[0] < 0) m.misc[0] = uniform_pick(draw, ms);
      gsync<NT>();
      const uint32_t r = sample_row(m.misc[0]);
      for (int j = g; j < b; j += NT) m.cent[(size_t)k * b + j] = a.L[(size_t)r * b + j];
    }
  }
  // Lloyd passes (K = 1: one pass, the mean)
  const int iters = K > 1 ? (a.iters > 0 ? a.iters : 1) : 1;
  for (int it = 0; it < iters; ++it) {
    gsync<NT>();
    for (int i = g; i < K * b; i += NT) m.sum[i] = 0ull;
    for (int i = g; i < K; i += NT) m.cnt[i] = 0u;
    gsync<NT>();
    for (int64_t i = g; i < n; i += NT) {
      load_logits(a.L, mem[i], b, l);
      int best = 0;
      if (K > 1) {
        float bd = dist_rn(l, m.cent, b);
        for (int k = 1; k < K; ++k) {
          const float d = dist_rn(l, m.cent + (size_t)k * b, b);
          if (d < bd) {
            bd = d;
            best = k;
          }
        }
        lab[i] = (uint8_t)best;
      }
      atomicAdd(&m.cnt[best], 1u);
#pragma unroll
      for (int j = 0; j < kBMax; ++j)
        if (j < b)
          atomicAdd(&m.sum[best * b + j],
                    (unsigned long long)__double2ll_rn(__dmul_rn((double)l[j], a.scale)));
    }
    gsync<NT>();
    for (int i = g; i < K * b; i += NT) {
      const uint32_t c = m.cnt[i / b];
      if (c > 0)
        m.cent[i] = __double2float_rn(__ddiv_rn(
            __dmul_rn(__ll2double_rn((long long)m.sum[i]), a.inv_scale), (double)c));
    }
  }
  gsync<NT>();
  // keep the clusters with members, in label order
  const int64_t slot = a.kslot[e];
  if (g == 0) {
    int kk = 0;
    uint32_t at = 0;
    for (int k = 0; k < K; ++k) {
      if (m.cnt[k] > 0) {
        m.remap[k] = kk;
        m.off[k] = at;
        a.slot_cnt[slot + kk] = m.cnt[k];
        at += m.cnt[k];
        ++kk;
      } else {
        m.remap[k] = -1;
      }
    }
    a.ncl[e] = (uint32_t)kk;
  }
  gsync<NT>();
  for (int i = g; i < K * b; i += NT) {
    const int rk = m.remap[i / b];
    if (rk >= 0) a.slot_cent[(size_t)(slot + rk) * b + (i % b)] = m.cent[i];
  }
  // rows in (cluster, id) order
  if (K == 1) {
    for (int64_t i = g; i < n; i += NT) a.out_ids[lo + i] = mem[i];
    return;
  }
  const int lane = threadIdx.x & 31, w = g >> 5, nw = NT / 32;
  for (int64_t c0 = 0; c0 < n; c0 += NT) {
    const int64_t i = c0 + g;
    const int k = i < n ? (int)lab[i] : -1;
    const unsigned peers = __match_any_sync(0xffffffffu, k);
    const int rank = __popc(peers & ((1u << lane) - 1u));
    if (k >= 0 && rank == 0) m.wcnt[w * a.K_max + k] = (uint32_t)__popc(peers);
    gsync<NT>();
    if (k >= 0) {
      uint32_t pos = m.off[k] + (uint32_t)rank;
      for (int v = 0; v < w; ++v) pos += m.wcnt[v * a.K_max + k];
      a.out_ids[lo + pos] = mem[i];
    }
    gsync<NT>();
    for (int kk = g; kk < K; kk += NT) {
      uint32_t add = 0;
      for (int v = 0; v < nw; ++v) {
        add += m.wcnt[v * a.K_max + kk];
        m.wcnt[v * a.K_max + kk] = 0;
      }
      m.off[kk] += add;
    }
    gsync<NT>();
  }
}

// one warp per bucket of at most kWarpRows rows; persistent warps
__global__ void kmeans_warp_kernel(KmArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const size_t per = km_smem_bytes(a.K_max, a.b, 1);
  const KmSmem m = km_carve(smem + (size_t)w * per, a.K_max, a.b, 1);
  const int64_t gw = (int64_t)blockIdx.x * (blockDim.x >> 5) + w;
  float *dmin = a.dmin + gw * a.mcap;
  for (;;) {
    for (int k = lane; k < a.K_max; k += 32) m.wcnt[k] = 0;
    int64_t e = 0;
    if (lane == 0) e = (int64_t)atomicAdd(&a.counter[0], 1u);
    e = __shfl_sync(0xffffffffu, e, 0);
    if (e >= a.ne) break;
    const uint32_t code = a.ne_code[e];
    if ((int64_t)a.bstart[code + 1] - (int64_t)a.bstart[code] > kWarpRows) continue;
    kmeans_bucket<32>(a, e, m, dmin);
    __syncwarp();
  }
}

// one CTA per large bucket, largest first; persistent CTAs
__global__ void __launch_bounds__(kCtaThreads) kmeans_cta_kernel(KmArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  const KmSmem m = km_carve(smem, a.K_max, a.b, kCtaThreads / 32);
  float *dmin = a.dmin + (int64_t)blockIdx.x * a.mcap;
  __shared__ long long item;
  for (;;) {
    for (int k = threadIdx.x; k < (kCtaThreads / 32) * a.K_max; k += kCtaThreads) m.wcnt[k] = 0;
    if (threadIdx.x == 0) item = (long long)atomicAdd(&a.counter[1], 1u);
    __syncthreads();
    const int64_t it = item;
    __syncthreads();
    if (it >= a.nbig) break;
    kmeans_bucket<kCtaThreads>(a, a.big_e[it], m, dmin);
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// Step 5: CSR levels, centroids, inverse permutation, row placement
// ---------------------------------------------------------------------------

__global__ void scatter_ncl_kernel(const uint32_t *__restrict__ ne_code,
                                   const uint32_t *__restrict__ ncl, int64_t ne, uint32_t *clc) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < ne;
       e += (int64_t)gridDim.x * blockDim.x)
    clc[ne_code[e]] = ncl[e];
}

__global__ void csr_kernel(const uint32_t *__restrict__ ne_code, const uint32_t *__restrict__ ncl,
                           const uint32_t *__restrict__ kslot, const uint32_t *__restrict__ bkt_off,
                           const uint32_t *__restrict__ bstart,
                           const uint32_t *__restrict__ slot_cnt,
                           const float *__restrict__ slot_cent, int64_t ne, int b, uint32_t *cl_off,
                           float *cent, unsigned int *stats) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < ne;
       e += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t u = ne_code[e];
    const uint32_t g0 = bkt_off[u], nk = ncl[e], sl = kslot[e];
    uint32_t r = bstart[u];
    atomicMax(&stats[0], bstart[u + 1] - bstart[u]);
    if (nk == 1) atomicAdd(&stats[2], 1u);
    for (uint32_t k = 0; k < nk; ++k) {
      cl_off[g0 + k] = r;
      r += slot_cnt[sl + k];
      atomicMax(&stats[1], slot_cnt[sl + k]);
      for (int j = 0; j < b; ++j) cent[(size_t)(g0 + k) * b + j] = slot_cent[(size_t)(sl + k) * b + j];
    }
  }
}

__global__ void inverse_kernel(const uint32_t *__restrict__ ids, int64_t N, uint32_t *inv) {
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < N;
       p += (int64_t)gridDim.x * blockDim.x)
    inv[ids[p]] = (uint32_t)p;
}

// rows [row0, row0 + n) to their stored positions, 16 bytes per thread
__global__ void place_kernel(const uint4 *__restrict__ src, int64_t row0, int64_t n, int chunks,
                             const uint32_t *__restrict__ inv, uint4 *vec) {
  const int64_t total = n * chunks;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / chunks;
    const int c = (int)(i - r * chunks);
    vec[(size_t)inv[row0 + r] * chunks + c] = src[i];
  }
}

}  // namespace

struct nr_builder {
  nr_index *ix = nullptr;
  nr_build_config cfg{};
  float *logits = nullptr;
  int64_t rows_set = 0;
  bool finished = false;
  bool failed = false;  // a finish call failed: the builder can only be freed
  uint32_t *inv = nullptr;
  int64_t placed = 0;
};

namespace {

// device buffers of one finish call, released on every exit
struct Scratch {
  std::vector<void *> ptrs;
  ~Scratch() {
    for (void *p : ptrs)
      if (p) cudaFree(p);
  }
  template <class T>
  cudaError_t alloc(T **p, size_t count) {
    *p = nullptr;
    void *v = nullptr;
    const cudaError_t e = cudaMalloc(&v, count * sizeof(T) > 0 ? count * sizeof(T) : 16);
    if (e != cudaSuccess) return e;
    ptrs.push_back(v);
    *p = static_cast<T *>(v);
    return cudaSuccess;
  }
  void release(void *p) {
    for (auto &q : ptrs)
      if (q == p) {
        cudaFree(q);
        q = nullptr;
      }
  }
};

int grid_for(int64_t work, int threads, int num_sms) {
  int64_t g = (work + threads - 1) / threads;
  const int64_t cap = (int64_t)num_sms * 16;
  if (g > cap) g = cap;
  return g < 1 ? 1 : (int)g;
}

#define NRB_TRY(x)                                \
  do {                                            \
    const cudaError_t e_ = (x);                   \
    if (e_ != cudaSuccess) return cuda_status(e_); \
  } while (0)

nr_status finish_impl(nr_builder *bd, int64_t *info, cudaStream_t s) {
  nr_index *ix = bd->ix;
  const int64_t N = ix->N;
  const int b = ix->b;
  const int nsm = ix->num_sms;
  const int64_t nb = (int64_t)1 << b;
  const float *L = bd->logits;
  Scratch sc;
  // fixed-point scale from the largest |logit|; rejects NaN and infinities
  unsigned int *d_small = nullptr;
  NRB_TRY(sc.alloc(&d_small, 16));
  NRB_TRY(cudaMemsetAsync(d_small, 0, 64, s));
  absmax_kernel<<<grid_for(N * b, 256, nsm), 256, 0, s>>>(L, N * b, d_small);
  NRB_TRY(cudaGetLastError());
  unsigned int amax = 0;
  NRB_TRY(cudaMemcpyAsync(&amax, d_small, 4, cudaMemcpyDeviceToHost, s));
  NRB_TRY(cudaStreamSynchronize(s));
  if (amax >= 0x7F800000u) return NR_ERR_INVALID_ARG;
  float am;
  memcpy(&am, &amax, 4);
  const int G = 30 - (am > 0.0f ? exponent_of((double)am) : 0);
  // medians: 4 radix passes of 8 bits
  uint32_t *hist, *prefix, *rank;
  NRB_TRY(sc.alloc(&hist, (size_t)b * 256));
  NRB_TRY(sc.alloc(&prefix, kBMax));
  NRB_TRY(sc.alloc(&rank, kBMax));
  NRB_TRY(cudaMemsetAsync(hist, 0, (size_t)b * 256 * 4, s));
  {
    std::vector<uint32_t> r0(kBMax, (uint32_t)((N - 1) / 2));
    NRB_TRY(cudaMemcpyAsync(rank, r0.data(), kBMax * 4, cudaMemcpyHostToDevice, s));
    NRB_TRY(cudaStreamSynchronize(s));
  }
  NRB_TRY(cudaMemsetAsync(prefix, 0, kBMax * 4, s));
  const int hist_blocks = grid_for(N, 256, nsm) < nsm * 4 ? grid_for(N, 256, nsm) : nsm * 4;
  for (int shift = 24; shift >= 0; shift -= 8) {
    median_hist_kernel<<<hist_blocks, 256, (size_t)b * 256 * 4, s>>>(L, N, b, shift, prefix, hist);
    NRB_TRY(cudaGetLastError());
    median_pick_kernel<<<1, 32, 0, s>>>(hist, prefix, rank, b, shift, ix->tau);
    NRB_TRY(cudaGetLastError());
  }
  // codes and the stable sort of ids by code
  uint32_t *codes, *ids, *codes_s, *ids_s;
  NRB_TRY(sc.alloc(&codes, N));
  NRB_TRY(sc.alloc(&ids, N));
  NRB_TRY(sc.alloc(&codes_s, N));
  NRB_TRY(sc.alloc(&ids_s, N));
  codes_kernel<<<grid_for(N, 256, nsm), 256, 0, s>>>(L, N, b, ix->tau, codes, ids);
  NRB_TRY(cudaGetLastError());
  {
    size_t tb = 0;
    NRB_TRY(cub::DeviceRadixSort::SortPairs(nullptr, tb, codes, codes_s, ids, ids_s, N, 0, b, s));
    void *tmp;
    NRB_TRY(sc.alloc(reinterpret_cast<unsigned char **>(&tmp), tb));
    NRB_TRY(cub::DeviceRadixSort::SortPairs(tmp, tb, codes, codes_s, ids, ids_s, N, 0, b, s));
    NRB_TRY(cudaStreamSynchronize(s));
    sc.release(tmp);
  }
  sc.release(codes);
  sc.release(ids);
  // bucket sizes, row starts, the non-empty list
  uint32_t *cnt, *bstart, *flag, *pos;
  NRB_TRY(sc.alloc(&cnt, nb + 1));
  NRB_TRY(sc.alloc(&bstart, nb + 1));
  NRB_TRY(cudaMemsetAsync(cnt, 0, (size_t)(nb + 1) * 4, s));
  count_kernel<<<grid_for(N, 256, nsm), 256, 0, s>>>(codes_s, N, cnt);
  NRB_TRY(cudaGetLastError());
  {
    size_t tb = 0;
    NRB_TRY(cub::DeviceScan::ExclusiveSum(nullptr, tb, cnt, bstart, nb + 1, s));
    void *tmp;
    NRB_TRY(sc.alloc(reinterpret_cast<unsigned char **>(&tmp), tb));
    NRB_TRY(cub::DeviceScan::ExclusiveSum(tmp, tb, cnt, bstart, nb + 1, s));
    NRB_TRY(cudaStreamSynchronize(s));
    sc.release(tmp);
  }
  sc.release(codes_s);
  NRB_TRY(sc.alloc(&flag, nb + 1));
  NRB_TRY(sc.alloc(&pos, nb + 1));
  flag_kernel<<<grid_for(nb + 1, 256, nsm), 256, 0, s>>>(cnt, nb, flag);
  NRB_TRY(cudaGetLastError());
  {
    size_t tb = 0;
    NRB_TRY(cub::DeviceScan::ExclusiveSum(nullptr, tb, flag, pos, nb + 1, s));
    void *tmp;
    NRB_TRY(sc.alloc(reinterpret_cast<unsigned char **>(&tmp), tb));
    NRB_TRY(cub::DeviceScan::ExclusiveSum(tmp, tb, flag, pos, nb + 1, s));
    NRB_TRY(cudaStreamSynchronize(s));
    sc.release(tmp);
  }
  uint32_t ne32 = 0;
  NRB_TRY(cudaMemcpy(&ne32, pos + nb, 4, cudaMemcpyDeviceToHost));
  const int64_t ne = ne32;
  uint32_t *ne_code, *kcount, *kslot, *big_e, *big_n, *big_e_s, *big_n_s;
  NRB_TRY(sc.alloc(&ne_code, ne + 1));
  NRB_TRY(sc.alloc(&kcount, ne + 1));
  NRB_TRY(sc.alloc(&kslot, ne + 1));
  NRB_TRY(sc.alloc(&big_e, ne + 1));
  NRB_TRY(sc.alloc(&big_n, ne + 1));
  NRB_TRY(cudaMemsetAsync(kcount, 0, (size_t)(ne + 1) * 4, s));
  NRB_TRY(cudaMemsetAsync(d_small, 0, 64, s));
  bucket_list_kernel<<<grid_for(nb, 256, nsm), 256, 0, s>>>(cnt, pos, nb, ix->K_max, ix->t, ne_code,
                                                            kcount, big_e, big_n, d_small);
  NRB_TRY(cudaGetLastError());
  {
    size_t tb = 0;
    NRB_TRY(cub::DeviceScan::ExclusiveSum(nullptr, tb, kcount, kslot, ne + 1, s));
    void *tmp;
    NRB_TRY(sc.alloc(reinterpret_cast<unsigned char **>(&tmp), tb));
    NRB_TRY(cub::DeviceScan::ExclusiveSum(tmp, tb, kcount, kslot, ne + 1, s));
    NRB_TRY(cudaStreamSynchronize(s));
    sc.release(tmp);
  }
  sc.release(flag);
  uint32_t nslots = 0, nbig = 0;
  NRB_TRY(cudaMemcpy(&nslots, kslot + ne, 4, cudaMemcpyDeviceToHost));
  NRB_TRY(cudaMemcpy(&nbig, d_small, 4, cudaMemcpyDeviceToHost));
  // large buckets largest first (the order only balances the load)
  NRB_TRY(sc.alloc(&big_e_s, (size_t)nbig + 1));
  NRB_TRY(sc.alloc(&big_n_s, (size_t)nbig + 1));
  if (nbig > 0) {
    size_t tb = 0;
    NRB_TRY(cub::DeviceRadixSort::SortPairsDescending(nullptr, tb, big_n, big_n_s, big_e, big_e_s,
                                                      (int64_t)nbig, 0, 32, s));
    void *tmp;
    NRB_TRY(sc.alloc(reinterpret_cast<unsigned char **>(&tmp), tb));
    NRB_TRY(cub::DeviceRadixSort::SortPairsDescending(tmp, tb, big_n, big_n_s, big_e, big_e_s,
                                                      (int64_t)nbig, 0, 32, s));
    NRB_TRY(cudaStreamSynchronize(s));
    sc.release(tmp);
  }
  // k-means
  KmArgs a;
  a.L = L;
  a.ids_s = ids_s;
  a.bstart = bstart;
  a.ne_code = ne_code;
  a.kslot = kslot;
  a.big_e = big_e_s;
  a.ne = ne;
  a.nbig = nbig;
  a.b = b;
  a.K_max = ix->K_max;
  a.t = ix->t;
  a.iters = bd->cfg.lloyd_iters;
  a.S = bd->cfg.sample_per_cluster;
  a.seed = bd->cfg.seed;
  a.scale = pow2(G);
  a.inv_scale = pow2(-G);
  uint32_t *out_ids;
  NRB_TRY(cudaMalloc((void **)&out_ids, (size_t)N * 4));
  ix->ids = out_ids;  // owned by the index from here on
  NRB_TRY(sc.alloc(&a.labels, N));
  NRB_TRY(sc.alloc(&a.slot_cent, (size_t)nslots * b + 1));
  NRB_TRY(sc.alloc(&a.slot_cnt, (size_t)nslots + 1));
  NRB_TRY(sc.alloc(&a.ncl, ne + 1));
  NRB_TRY(sc.alloc(&a.counter, 4));
  NRB_TRY(cudaMemsetAsync(a.counter, 0, 16, s));
  a.out_ids = out_ids;
  const int wpb = 8;
  const size_t wsm = km_smem_bytes(ix->K_max, b, 1) * wpb;
  const size_t csm = km_smem_bytes(ix->K_max, b, kCtaThreads / 32);
  NRB_TRY(cudaFuncSetAttribute(kmeans_warp_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)wsm));
  NRB_TRY(cudaFuncSetAttribute(kmeans_cta_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)csm));
  int occ_w = 0, occ_c = 0;
  NRB_TRY(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ_w, kmeans_warp_kernel, 32 * wpb, wsm));
  NRB_TRY(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ_c, kmeans_cta_kernel, kCtaThreads, csm));
  if (occ_w < 1 || occ_c < 1) return NR_ERR_INVALID_ARG;
  const int grid_w = occ_w * nsm;
  const int grid_c = (int)(nbig < (uint32_t)(occ_c * nsm) ? (nbig > 0 ? nbig : 1) : occ_c * nsm);
  // seeding scratch: a warp's bucket has at most kWarpRows members; a CTA's
  // sample at most sample_per_cluster * K_max
  const int64_t mcap_c = (int64_t)a.S * ix->K_max;
  const int64_t mcap_w = kWarpRows;
  float *dmin_w, *dmin_c;
  NRB_TRY(sc.alloc(&dmin_w, (size_t)grid_w * wpb * mcap_w));
  NRB_TRY(sc.alloc(&dmin_c, (size_t)grid_c * mcap_c));
  if (nbig > 0) {
    a.dmin = dmin_c;
    a.mcap = mcap_c;
    kmeans_cta_kernel<<<grid_c, kCtaThreads, csm, s>>>(a);
    NRB_TRY(cudaGetLastError());
  }
  a.dmin = dmin_w;
  a.mcap = mcap_w;
  kmeans_warp_kernel<<<grid_w, 32 * wpb, wsm, s>>>(a);
  NRB_TRY(cudaGetLastError());
  NRB_TRY(cudaStreamSynchronize(s));
  sc.release(dmin_w);
  sc.release(dmin_c);
  sc.release(a.labels);
  sc.release(ids_s);
  // bucket -> cluster CSR level: exclusive sum of kept clusters over all codes
  uint32_t *clc;
  NRB_TRY(sc.alloc(&clc, nb + 1));
  NRB_TRY(cudaMemsetAsync(clc, 0, (size_t)(nb + 1) * 4, s));
  scatter_ncl_kernel<<<grid_for(ne, 256, nsm), 256, 0, s>>>(ne_code, a.ncl, ne, clc);
  NRB_TRY(cudaGetLastError());
  {
    size_t tb = 0;
    NRB_TRY(cub::DeviceScan::ExclusiveSum(nullptr, tb, clc, ix->bkt_off, nb + 1, s));
    void *tmp;
    NRB_TRY(sc.alloc(reinterpret_cast<unsigned char **>(&tmp), tb));
    NRB_TRY(cub::DeviceScan::ExclusiveSum(tmp, tb, clc, ix->bkt_off, nb + 1, s));
    NRB_TRY(cudaStreamSynchronize(s));
    sc.release(tmp);
  }
  uint32_t ncl_total = 0;
  NRB_TRY(cudaMemcpy(&ncl_total, ix->bkt_off + nb, 4, cudaMemcpyDeviceToHost));
  ix->n_cl = ncl_total;
  if (ix->n_cl >= ((int64_t)1 << 31)) return NR_ERR_INVALID_ARG;  // cluster indices fill 31 bits of a sort key
  NRB_TRY(cudaMalloc((void **)&ix->cl_off, ((size_t)ix->n_cl + 1) * 4));
  NRB_TRY(cudaMalloc((void **)&ix->cent, (size_t)ix->n_cl * b * 4 + 16));
  NRB_TRY(cudaMemsetAsync(d_small, 0, 64, s));
  csr_kernel<<<grid_for(ne, 128, nsm), 128, 0, s>>>(ne_code, a.ncl, kslot, ix->bkt_off, bstart,
                                                    a.slot_cnt, a.slot_cent, ne, b, ix->cl_off,
                                                    ix->cent, d_small);
  NRB_TRY(cudaGetLastError());
  {
    const uint32_t nn = (uint32_t)N;
    NRB_TRY(cudaMemcpyAsync(ix->cl_off + ix->n_cl, &nn, 4, cudaMemcpyHostToDevice, s));
    NRB_TRY(cudaStreamSynchronize(s));
  }
  unsigned int st3[3] = {0, 0, 0};
  NRB_TRY(cudaMemcpy(st3, d_small, 12, cudaMemcpyDeviceToHost));
  // stored position of every id, for the row placement
  NRB_TRY(cudaMalloc((void **)&bd->inv, (size_t)N * 4));
  inverse_kernel<<<grid_for(N, 256, nsm), 256, 0, s>>>(ix->ids, N, bd->inv);
  NRB_TRY(cudaGetLastError());
  NRB_TRY(cudaStreamSynchronize(s));
  if (info) {
    info[0] = ix->n_cl;
    info[1] = ne;
    info[2] = st3[0];
    info[3] = st3[1];
    info[4] = st3[2];
  }
  return NR_OK;
}

}  // namespace

extern "C" {

nr_status nr_build_begin(const nr_build_config *cfg, int64_t N, const float *W1, const float *b1,
                         const float *W2, const float *b2, const float *Wm, int device,
                         nr_builder **out) {
  if (!cfg || !out || !W1 || !b1 || !W2 || !b2) return NR_ERR_INVALID_ARG;
  if (cfg->n_mid < 0 || cfg->n_mid > 7 || (cfg->n_mid > 0 && !Wm)) return NR_ERR_INVALID_ARG;
  for (int i = 0; i < cfg->n_mid; ++i)
    if (cfg->mid_w[i] < 1 || cfg->mid_w[i] > 4096) return NR_ERR_INVALID_ARG;
  *out = nullptr;
  const int64_t esz = cfg->dtype == 0 ? 1 : 4;
  const int64_t row_bytes = (int64_t)cfg->D * esz;
  if ((cfg->dtype != 0 && cfg->dtype != 1) || cfg->D < 1 || cfg->H < 1 || cfg->H > 4096 ||
      cfg->b < 1 || cfg->b > kBMax || cfg->K_max < 1 || cfg->K_max > kKMax || cfg->t < 1 ||
      cfg->sample_per_cluster < 1 || cfg->sample_per_cluster > kMaxSample || N < 1 ||
      N >= (int64_t)0xFFFFFFFFll || !nr_row_bytes_ok(cfg->dtype, row_bytes))
    return NR_ERR_INVALID_ARG;
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess) {
    cudaGetLastError();
    return NR_ERR_CUDA;
  }
  if (device < 0 || device >= ndev) return NR_ERR_INVALID_ARG;
  DeviceGuard g(device);
  auto *bd = new (std::nothrow) nr_builder();
  if (!bd) return NR_ERR_OOM;
  bd->cfg = *cfg;
  nr_index *ix = nr_index_alloc();
  if (!ix) {
    delete bd;
    return NR_ERR_OOM;
  }
  bd->ix = ix;
  ix->device = device;
  ix->dtype = cfg->dtype;
  ix->N = N;
  ix->D = cfg->D;
  ix->H = cfg->H;
  ix->b = cfg->b;
  ix->K_max = cfg->K_max;
  ix->t = cfg->t;
  ix->in_scale = cfg->in_scale;
  ix->row_bytes = row_bytes;
  ix->n_mid = cfg->n_mid;
  for (int i = 0; i < 7; ++i) ix->mid_w[i] = i < cfg->n_mid ? cfg->mid_w[i] : 0;
  nr_status st = nr_index_init_device(ix);
  if (st == NR_OK) st = nr_index_upload_encoder(ix, W1, b1, W2, b2, Wm);
  if (st == NR_OK) st = cuda_status(cudaMalloc((void **)&ix->tau, (size_t)cfg->b * 4));
  if (st == NR_OK)
    st = cuda_status(cudaMalloc((void **)&ix->bkt_off, (((size_t)1 << cfg->b) + 1) * 4));
  if (st == NR_OK) st = cuda_status(cudaMalloc((void **)&bd->logits, (size_t)N * cfg->b * 4));
  if (st != NR_OK) {
    nr_build_free(bd);
    return st;
  }
  *out = bd;
  return NR_OK;
}

nr_status nr_build_encode(nr_builder *bd, const void *d_rows, int64_t row0, int64_t n, void *stream) {
  if (!bd || bd->finished || bd->failed || row0 < 0 || n < 0 || row0 + n > bd->ix->N) return NR_ERR_INVALID_ARG;
  if (n == 0) return NR_OK;
  if (!d_rows) return NR_ERR_INVALID_ARG;
  DeviceGuard g(bd->ix->device);
  const nr_status st = cuda_status(nr_launch_encode(bd->ix, d_rows, n,
                                                    bd->logits + (size_t)row0 * bd->ix->b,
                                                    (cudaStream_t)stream));
  if (st == NR_OK) bd->rows_set += n;
  return st;
}

nr_status nr_build_set_logits(nr_builder *bd, const float *d_logits, int64_t row0, int64_t n,
                              void *stream) {
  if (!bd || bd->finished || bd->failed || row0 < 0 || n < 0 || row0 + n > bd->ix->N) return NR_ERR_INVALID_ARG;
  if (n == 0) return NR_OK;
  if (!d_logits) return NR_ERR_INVALID_ARG;
  DeviceGuard g(bd->ix->device);
  const size_t bytes = (size_t)n * bd->ix->b * 4;
  const nr_status st = cuda_status(cudaMemcpyAsync(bd->logits + (size_t)row0 * bd->ix->b, d_logits,
                                                   bytes, cudaMemcpyDeviceToDevice,
                                                   (cudaStream_t)stream));
  if (st == NR_OK) bd->rows_set += n;
  return st;
}

nr_status nr_build_finish(nr_builder *bd, int64_t *info) {
  if (!bd || bd->finished || bd->failed || bd->rows_set != bd->ix->N) return NR_ERR_INVALID_ARG;
  DeviceGuard g(bd->ix->device);
  if (cudaDeviceSynchronize() != cudaSuccess) {
    cudaGetLastError();
    return NR_ERR_CUDA;
  }
  cudaStream_t s;
  if (cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking) != cudaSuccess) {
    cudaGetLastError();
    return NR_ERR_CUDA;
  }
  const nr_status st = finish_impl(bd, info, s);
  cudaStreamSynchronize(s);
  cudaStreamDestroy(s);
  if (st != NR_OK) {
    bd->failed = true;
    return st;
  }
  cudaFree(bd->logits);
  bd->logits = nullptr;
  nr_index *ix = bd->ix;
  if (cudaMalloc(&ix->vec, (size_t)ix->N * ix->row_bytes) != cudaSuccess) {
    cudaGetLastError();
    ix->vec = nullptr;
    bd->failed = true;
    return NR_ERR_OOM;
  }
  bd->finished = true;
  return NR_OK;
}

nr_status nr_build_place(nr_builder *bd, const void *d_rows, int64_t row0, int64_t n, void *stream) {
  if (!bd || !bd->finished || row0 < 0 || n < 0 || row0 + n > bd->ix->N) return NR_ERR_INVALID_ARG;
  if (n == 0) return NR_OK;
  if (!d_rows || ((uintptr_t)d_rows & 15) != 0) return NR_ERR_INVALID_ARG;
  nr_index *ix = bd->ix;
  DeviceGuard g(ix->device);
  const int chunks = (int)(ix->row_bytes / 16);
  place_kernel<<<grid_for(n * chunks, 256, ix->num_sms), 256, 0, (cudaStream_t)stream>>>(
      static_cast<const uint4 *>(d_rows), row0, n, chunks, bd->inv, static_cast<uint4 *>(ix->vec));
  const nr_status st = cuda_status(cudaGetLastError());
  if (st == NR_OK) bd->placed += n;
  return st;
}

nr_status nr_build_end(nr_builder *bd, nr_index **out) {
  if (!bd || !out) {
    nr_build_free(bd);
    return NR_ERR_INVALID_ARG;
  }
  *out = nullptr;
  if (!bd->finished || bd->placed != bd->ix->N) {
    nr_build_free(bd);
    return NR_ERR_INVALID_ARG;
  }
  DeviceGuard g(bd->ix->device);
  if (cudaDeviceSynchronize() != cudaSuccess) {
    cudaGetLastError();
    nr_build_free(bd);
    return NR_ERR_CUDA;
  }
  cudaFree(bd->inv);
  bd->inv = nullptr;
  *out = bd->ix;
  bd->ix = nullptr;
  delete bd;
  return NR_OK;
}

void nr_build_free(nr_builder *bd) {
  if (!bd) return;
  if (bd->ix) {
    DeviceGuard g(bd->ix->device);
    if (bd->logits) cudaFree(bd->logits);
    if (bd->inv) cudaFree(bd->inv);
    nr_index_free(bd->ix);
  }
  delete bd;
}

}  // extern "C"
