// K3 select: bucket lookup through the CSR directory (Sec. 3.3) and the
// centroid stage of Sec. 3.4.2 / Algorithm 2.
//
// One CTA per query:
//   1. probe i -> cluster range [bkt_off[u_i], bkt_off[u_i + 1]) (range-checked);
//   2. every cluster c of every probed bucket gets its centroid distance
//      d_c = sum_j (l_j - mu_cj)^2 as a sequential fp32 fmaf chain over j;
//   3. buckets holding exactly one cluster go to C^dir; over the other clusters
//      d_min, the gate theta = d_min + fmaf(m1, d_min, m0), survivors d_c <= theta;
//   4. a bitonic sort of the 64-bit keys (d_c bits, c) of C^dir and the
//      survivors, the first C survivors kept (top-C by (d_c, c)), and the kept
//      list written in key order together with its refinement segments
//      (first row, stream position) for K4.
// Sorting by exact keys makes the result independent of thread scheduling.
#include <cuda_runtime.h>
#include <stdint.h>

#include <cmath>

#include "nr_internal.cuh"

namespace {

constexpr int kThreads = 128;
constexpr uint64_t kMaxKey = ~0ull;

__device__ __forceinline__ void set_err(int *err, int code) { atomicCAS(err, 0, code); }

// Exclusive scan of a[0..n) in shared memory; returns the total. All threads call.
__device__ int block_exclusive_scan(int *a, int n, int *warp_sums) {
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int per = (n + kThreads - 1) / kThreads;
  const int lo = tid * per, hi = min(n, lo + per);
  int local = 0;
  for (int i = lo; i < hi; ++i) local += a[i];
  int incl = local;
  for (int o = 1; o < 32; o <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) warp_sums[wid] = incl;
  __syncthreads();
  if (wid == 0) {
    int ws = lane < kThreads / 32 ? warp_sums[lane] : 0;
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, ws, o);
      if (lane >= o) ws += v;
    }
    if (lane < kThreads / 32) warp_sums[lane] = ws;  // inclusive
  }
  __syncthreads();
  int run = (wid > 0 ? warp_sums[wid - 1] : 0) + incl - local;
  for (int i = lo; i < hi; ++i) {
    const int v = a[i];
    a[i] = run;
    run += v;
  }
  const int total = warp_sums[kThreads / 32 - 1];
  __syncthreads();
  return total;
}

// Bitonic sort of k[0..n), n a power of two. Thread i owns the pairs
// (lo, lo + stride) with lo = 2i - (i mod stride); for strides up to 32 the
// pairs of one warp stay inside its own 64-element blocks, so consecutive
// such stages need only a warp barrier.
__device__ void bitonic_sort(uint64_t *k, int n) {
  for (int size = 2; size <= n; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < n / 2; i += kThreads) {
        const int lo = 2 * i - (i & (stride - 1));
        const int hi = lo + stride;
        const bool up = (lo & size) == 0;
        const uint64_t a = k[lo], c = k[hi];
        if ((a > c) == up) {
          k[lo] = c;
          k[hi] = a;
        }
      }
      // a block barrier whenever this stage or the next one crosses warps
      const int next = stride > 1 ? stride >> 1 : size;
      if (stride > 32 || next > 32) __syncthreads();
      else __syncwarp();
    }
  }
  __syncthreads();
}

struct SelectArgs {
  const float *logits;
  const uint32_t *codes;
  const int32_t *nprobe;
  int b, K_max, P, C, Lmax;
  int64_t n_cl, N;
  const uint32_t *bkt_off, *cl_off;
  const float *cent;
  const uint8_t *single;  // [n_cl] 1 if the cluster's bucket holds one cluster
  bool gate_off;
  float m0, m1;
  int32_t *L, *nL;
  nr_seg *seg;
  uint32_t *slen;
  int64_t *stats;
  int *err;
};

__global__ void __launch_bounds__(kThreads) select_kernel(SelectArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int q = blockIdx.x, tid = threadIdx.x;
  const int S_cap = a.P * a.K_max;  // power-of-two rounding done below
  int S_pow = 1;
  while (S_pow < S_cap) S_pow <<= 1;
  uint64_t *keys = reinterpret_cast<uint64_t *>(smem);                 // [S_pow]
  int *ibuf = reinterpret_cast<int *>(smem + (size_t)S_pow * 8);       // [max(S_pow, 2P + 1)]
  const int ib_n = max(S_pow, 2 * a.P + 1);
  float *slog = reinterpret_cast<float *>(smem + (size_t)S_pow * 8 + (size_t)ib_n * 4);  // [32]
  int *warp_sums = reinterpret_cast<int *>(slog + 32);                                   // [8]
  unsigned int *sred = reinterpret_cast<unsigned int *>(warp_sums + 8);                  // [4]

  const int np = a.nprobe[q];
  if (tid < a.b) slog[tid] = a.logits[(size_t)q * a.b + tid];
  if (tid == 0) sred[0] = 0xffffffffu;
  int *cnt = ibuf;            // [P] clusters per probe -> exclusive offsets
  int *c0s = ibuf + a.P;      // [P] first cluster per probe
  const uint32_t nb = 1u << a.b;
  for (int i = tid; i < np; i += kThreads) {
    const uint32_t u = a.codes[(size_t)q * a.P + i];
    int n = 0, c0 = 0;
    if (u >= nb) {
      set_err(a.err, NR_DEV_BAD_CODE);
    } else {
      const uint32_t lo = a.bkt_off[u], hi = a.bkt_off[u + 1];
      if (hi < lo || (int64_t)hi > a.n_cl) {
        set_err(a.err, NR_DEV_BAD_BUCKET);
      } else {
        n = (int)(hi - lo);
        c0 = (int)lo;
        if (n > a.K_max) {
          set_err(a.err, NR_DEV_TOO_MANY);
          n = a.K_max;
        }
      }
    }
    cnt[i] = n;
    c0s[i] = c0;
  }
  __syncthreads();
  const int M = block_exclusive_scan(cnt, np, warp_sums);
  // each probe writes its clusters' indices into the key slots
  for (int i = tid; i < np; i += kThreads) {
    const int o = cnt[i], n = (i + 1 < np ? cnt[i + 1] : M) - o;
    for (int j = 0; j < n; ++j) keys[o + j] = (uint64_t)(uint32_t)(c0s[i] + j);
  }
  __syncthreads();
  // centroid distances; keys of all candidates (exclusion decided after d_min)
  for (int s = tid; s < M; s += kThreads) {
    const uint32_t c = (uint32_t)keys[s];
    const float *mu = a.cent + (size_t)c * a.b;
    float acc = 0.0f;
    for (int j = 0; j < a.b; ++j) {
      const float t = __fsub_rn(slog[j], mu[j]);
      acc = __fmaf_rn(t, t, acc);
    }
    keys[s] = ((uint64_t)__float_as_uint(acc) << 32) | c;
    if (!a.single[c]) atomicMin(&sred[0], __float_as_uint(acc));  // d >= 0: bit order = value order
  }
  for (int s = M + tid; s < S_pow; s += kThreads) keys[s] = kMaxKey;
  __syncthreads();
  const uint32_t dmin_bits = sred[0];
  float theta = __int_as_float(0x7f800000);
  if (!a.gate_off && dmin_bits != 0xffffffffu) {
    const float dmin = __uint_as_float(dmin_bits);
    theta = __fadd_rn(dmin, __fmaf_rn(a.m1, dmin, a.m0));
  }
  // drop non-singleton clusters above the gate
  for (int s = tid; s < M; s += kThreads) {
    const uint64_t kk = keys[s];
    const uint32_t c = (uint32_t)kk;
    if (!a.single[c] && !(__uint_as_float((uint32_t)(kk >> 32)) <= theta)) keys[s] = kMaxKey;
  }
  __syncthreads();
  int Sn = 1;
  while (Sn < M) Sn <<= 1;
  bitonic_sort(keys, Sn);
  // keep C^dir and the first C survivors in key order
  int *keep = ibuf;  // [Sn]
  for (int s = tid; s < Sn; s += kThreads) {
    const uint64_t kk = keys[s];
    keep[s] = (s < M && kk != kMaxKey && !a.single[(uint32_t)kk]) ? 1 : 0;
  }
  __syncthreads();
  block_exclusive_scan(keep, Sn, warp_sums);  // survivor rank in key order
  for (int s = tid; s < Sn; s += kThreads) {
    const uint64_t kk = keys[s];
    int kp = 0;
    if (s < M && kk != kMaxKey) kp = a.single[(uint32_t)kk] ? 1 : (keep[s] < a.C ? 1 : 0);
    keep[s] = kp;
  }
  __syncthreads();
  const int nl = block_exclusive_scan(keep, Sn, warp_sums);  // output position
  // write the kept entries at their output positions (keep[] is now the exclusive prefix)
  for (int s = tid; s < Sn; s += kThreads) {
    const uint64_t kk = keys[s];
    if (s < M && kk != kMaxKey) {
      const bool sg = a.single[(uint32_t)kk] != 0;
      const int pos = keep[s];
      const bool kept = sg || (s + 1 < Sn ? keep[s + 1] > pos : nl > pos);
      if (kept) a.L[(size_t)q * a.Lmax + pos] = (int32_t)(uint32_t)kk;
    }
  }
  __syncthreads();
  // segments of the kept clusters, in list order
  int *len2 = ibuf;  // reuse: [nl] (keep[] no longer needed)
  for (int i = tid; i < nl; i += kThreads) {
    const uint32_t c = (uint32_t)a.L[(size_t)q * a.Lmax + i];
    const uint32_t r0 = a.cl_off[c], r1 = a.cl_off[c + 1];
    int len = 0;
    if (r1 < r0 || (int64_t)r1 > a.N) set_err(a.err, NR_DEV_BAD_CLUSTER);
    else len = (int)(r1 - r0);
    len2[i] = len;
    a.seg[(size_t)q * a.Lmax + i].row0 = r0;
  }
  __syncthreads();
  const int total = block_exclusive_scan(len2, nl, warp_sums);
  for (int i = tid; i < nl; i += kThreads) a.seg[(size_t)q * a.Lmax + i].pos = (uint32_t)len2[i];
  for (int i = nl + tid; i < a.Lmax; i += kThreads) a.L[(size_t)q * a.Lmax + i] = -1;
  if (tid == 0) {
    a.nL[q] = nl;
    a.slen[q] = (uint32_t)total;
    if (a.stats) {
      a.stats[(size_t)q * 4 + 2] = nl;
      a.stats[(size_t)q * 4 + 3] = np;
    }
  }
}

}  // namespace

size_t nr_select_smem_bytes(int P, int C, int K_max) {
  (void)C;
  size_t S = 1;
  while (S < (size_t)P * (size_t)K_max) S <<= 1;
  const size_t ib = S > (size_t)(2 * P + 1) ? S : (size_t)(2 * P + 1);
  return S * 8 + ib * 4 + 32 * 4 + 8 * 4 + 4 * 4;
}

// defined in nr_api.cu: per-cluster flag "its bucket holds exactly one cluster"
const uint8_t *nr_single_table(nr_index *ix);

cudaError_t nr_launch_select(nr_index *ix, const float *d_logits, const uint32_t *d_codes,
                             const int32_t *d_nprobe, int64_t nq, int P, int C, int32_t *d_L,
                             int32_t *d_nL, nr_seg *d_seg, uint32_t *d_slen, int64_t *d_stats,
                             cudaStream_t s) {
  if (nq <= 0) return cudaSuccess;
  const size_t smem = nr_select_smem_bytes(P, C, ix->K_max);
  cudaError_t e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  SelectArgs a;
  a.logits = d_logits;
  a.codes = d_codes;
  a.nprobe = d_nprobe;
  a.b = ix->b;
  a.K_max = ix->K_max;
  a.P = P;
  a.C = C;
  a.Lmax = P + C;
  a.n_cl = ix->n_cl;
  a.N = ix->N;
  a.bkt_off = ix->bkt_off;
  a.cl_off = ix->cl_off;
  a.cent = ix->cent;
  a.single = nr_single_table(ix);
  const float m0 = ix->params.gate_m0;
  a.gate_off = std::isinf(m0) && m0 > 0.0f;
  a.m0 = m0;
  a.m1 = ix->params.gate_m1;
  a.L = d_L;
  a.nL = d_nL;
  a.seg = d_seg;
  a.slen = d_slen;
  a.stats = d_stats;
  a.err = ix->d_err;
  select_kernel<<<(unsigned)nq, kThreads, smem, s>>>(a);
  ix->launches += 1;
  return cudaGetLastError();
}
