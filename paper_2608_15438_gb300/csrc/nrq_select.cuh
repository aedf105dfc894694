// select_block: one block per query looks up the probed buckets, scores
// their centroids, applies the gate and top-C and lays out the refinement
// segments of the kept clusters (Sec. 3.3, 3.4.2, Algorithm 2).
#pragma once

#include "nrq_block.cuh"

namespace nrq {

// ============================================================== select
struct SelectParams {
  int b, K_max, P, C;
  int64_t n_cl, N;
  const uint32_t *bkt_off, *cl_off;
  const float *cent;
  bool gate_off;
  float m0, m1;
  int *err;
  // the sequential centroid stage (mode 1)
  int mode, n_bins, b_batch, b_min, c_t_low, c_u_min, c_f_min;
  float s_max, c_alpha_front;
  const float *tau;
  // calibrated gate curve (gate_n >= 2), else M(x) = m0 + m1 x
  int gate_n;
  float gate_x[16], gate_y[16];
};

// The gate margin M(x): m0 + m1 x, or the calibrated monotone piecewise-linear
// curve, flat beyond its ends, each segment's value held within its end values
// so that M never decreases in fp32 (the definition of the oracle's
// gate_margin).
__device__ __forceinline__ float gate_margin(const SelectParams &sp, float x) {
  if (sp.gate_n < 2) return __fmaf_rn(sp.m1, x, sp.m0);
  int i = 0;
  while (i + 1 < sp.gate_n && sp.gate_x[i + 1] <= x) ++i;
  if (x <= sp.gate_x[0]) return sp.gate_y[0];
  if (i == sp.gate_n - 1) return sp.gate_y[i];
  const float s = __fdiv_rn(__fsub_rn(sp.gate_y[i + 1], sp.gate_y[i]),
                            __fsub_rn(sp.gate_x[i + 1], sp.gate_x[i]));
  const float v = __fmaf_rn(__fsub_rn(x, sp.gate_x[i]), s, sp.gate_y[i]);
  return fminf(fmaxf(v, sp.gate_y[i]), sp.gate_y[i + 1]);
}

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
// key capacity of the shared-memory scratch: S keys plus the merge sort's gaps
__host__ __device__ inline int select_smem_keys(int S) { return S + S / 16; }
__host__ __device__ inline size_t select_scratch_bytes(int P, int K_max) {
  const int S = select_smem_cap(P, K_max);
  const int ib = S > 2 * P + 1 ? S : 2 * P + 1;
  return (size_t)select_smem_keys(S) * 8 + (size_t)ib * 4;
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

// Probe of candidate slot s: slots are numbered probe by probe, off[i] the
// first slot of probe i (nondecreasing).
// Requests the 128-byte line holding p into L2 (no register result).
__device__ __forceinline__ void prefetch_l2(const void *p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

__device__ __forceinline__ int slot_probe(const int *off, int np, int s) {
  int lo = 0, hi = np - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (off[mid] <= s) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// Probes whose directory entries one thread loads at once.
constexpr int kSelLookups = 8;

// Sort keys of the order-independent stage: ((d bits) << 32) | (c << 1) |
// single, single = the cluster's bucket holds only it (C^dir). For distinct
// clusters (c < 2^31) they order exactly as (d, c) does; the flag rides along
// so that no lookup is needed to tell C^dir apart after the sort.
__device__ __forceinline__ uint64_t tagged_key(float d, uint32_t c, bool single) {
  return ((uint64_t)__float_as_uint(d) << 32) | ((uint64_t)c << 1) | (single ? 1u : 0u);
}
__device__ __forceinline__ uint32_t key_cluster(uint64_t k) { return (uint32_t)k >> 1; }
__device__ __forceinline__ bool key_single(uint64_t k) { return (k & 1u) != 0; }

// The kept list from the collected keys k[0..n) (n <= E * blockDim.x), sorted
// into registers: C^dir keys always, the others while their rank among the
// others is below C, in key order; then their segments (first row, stream
// position) and, when L is not null, their cluster indices (-1 padded to
// Lmax). Returns the list length; *total = stream length.
template <int E>
__device__ __forceinline__ int select_tail_regs(const SelectParams &sp, uint64_t *k, int n,
                                                int *warp_sums, nr_seg *seg, int32_t *L, int Lmax,
                                                uint32_t *total) {
  uint64_t r[E];
  merge_sort_regs<E>(k, n, r);
  uint32_t sg = 0, kp = 0;
  int ns = 0;
#pragma unroll
  for (int e = 0; e < E; ++e)
    if (r[e] != kEmpty) {
      if (key_single(r[e])) sg |= 1u << e;
      else ++ns;
    }
  int all;
  int rank = block_thread_scan(ns, warp_sums, &all);  // rank among the non-C^dir keys
  int nk = 0;
#pragma unroll
  for (int e = 0; e < E; ++e)
    if (r[e] != kEmpty) {
      bool keep = (sg >> e) & 1u;
      if (!keep) {
        keep = rank < sp.C;
        ++rank;
      }
      if (keep) {
        kp |= 1u << e;
        ++nk;
      }
    }
  int nl;
  int pos = block_thread_scan(nk, warp_sums, &nl);  // output position
  int lsum = 0;
#pragma unroll
  for (int e = 0; e < E; ++e)
    if ((kp >> e) & 1u) {
      const uint32_t c = key_cluster(r[e]);
      const uint32_t r0 = __ldg(&sp.cl_off[c]), r1 = __ldg(&sp.cl_off[c + 1]);
      if (r1 < r0 || (int64_t)r1 > sp.N) set_err(sp.err, NR_DEV_BAD_CLUSTER);
      else lsum += (int)(r1 - r0);
    }
  int tot;
  int spos = block_thread_scan(lsum, warp_sums, &tot);  // stream position
#pragma unroll
  for (int e = 0; e < E; ++e)
    if ((kp >> e) & 1u) {
      const uint32_t c = key_cluster(r[e]);
      const uint32_t r0 = __ldg(&sp.cl_off[c]), r1 = __ldg(&sp.cl_off[c + 1]);
      const int ln = (r1 < r0 || (int64_t)r1 > sp.N) ? 0 : (int)(r1 - r0);
      seg[pos].row0 = r0;
      seg[pos].pos = (uint32_t)spos;
      if (L) L[pos] = (int32_t)c;
      spos += ln;
      ++pos;
    }
  if (L)
    for (int i = nl + threadIdx.x; i < Lmax; i += blockDim.x) L[i] = -1;
  *total = (uint32_t)tot;
  return nl;
}

// select_tail_regs with the smallest run length E (a power of two) that covers n
__device__ __forceinline__ int select_tail_smem(const SelectParams &sp, uint64_t *k, int n,
                                                int *warp_sums, nr_seg *seg, int32_t *L, int Lmax,
                                                uint32_t *total) {
  const int nt = blockDim.x;
  if (n <= nt) return select_tail_regs<1>(sp, k, n, warp_sums, seg, L, Lmax, total);
  if (n <= 2 * nt) return select_tail_regs<2>(sp, k, n, warp_sums, seg, L, Lmax, total);
  if (n <= 4 * nt) return select_tail_regs<4>(sp, k, n, warp_sums, seg, L, Lmax, total);
  if (n <= 8 * nt) return select_tail_regs<8>(sp, k, n, warp_sums, seg, L, Lmax, total);
  return select_tail_regs<16>(sp, k, n, warp_sums, seg, L, Lmax, total);
}

// One query: codes[0..np) -> the kept clusters C^dir U C^cent in (d, cluster)
// order and their refinement segments. Writes seg[i] = (first row, stream
// position) for i < nl, and L[i] (cluster index, -1 padded to Lmax) when L is
// not null; *n_scored = the number of centroid distances evaluated (every
// cluster of every probed bucket). slog: the query's b logits in shared memory; scratch:
// select_scratch_bytes(P, K_max) bytes of shared memory; slab: this query's
// select_slab_bytes(P, K_max) bytes of global memory (null when that is 0);
// warp_sums: 32 ints; sred: 2 unsigned. Returns nl (*total = stream length),
// or -1 when the query is deferred to the overflow kernel. Whole block calls.
//
// The keys to sort (C^dir and the gate's survivors) are collected straight
// into shared memory: one pass over the candidate clusters computes their
// distances, keeps the single-cluster buckets' and takes d_min over the rest;
// a second pass recomputes the others' distances and keeps those within the
// gate. Only when they do not fit are the query's candidate keys written to
// its global slab and the query deferred (returns -1) to the overflow
// kernel, whose blocks sort more keys in shared memory. Both give the same
// keys, and the sort orders them by exact value.
__device__ __forceinline__ int select_block(const SelectParams &sp, const float *slog,
                                            const uint32_t *codes, int np, unsigned char *scratch,
                                            unsigned char *slab, int *warp_sums, unsigned *sred,
                                            nr_seg *seg, int32_t *L, int Lmax, uint32_t *total,
                                            int *n_scored) {
  const int tid = threadIdx.x, nt = blockDim.x;
  const int S_smem = select_smem_cap(sp.P, sp.K_max);
  const int S_full = select_sort_cap(sp.P, sp.K_max);
  uint64_t *keys = reinterpret_cast<uint64_t *>(scratch);
  int *ibuf = reinterpret_cast<int *>(scratch + (size_t)select_smem_keys(S_smem) * 8);
  if (tid == 0) {
    sred[0] = 0xffffffffu;  // d_min bits over non-singleton candidates
    sred[1] = 0u;           // keys collected
  }
  int *cnt = ibuf;        // [P] clusters per probe -> exclusive offsets
  int *c0s = ibuf + sp.P;  // [P] first cluster per probe
  const uint32_t nb = 1u << sp.b;
  // directory lookups eight probes a thread at a time, all loads issued before
  // any is used (they are independent random reads)
  for (int i0 = tid; i0 < np; i0 += kSelLookups * nt) {
    uint32_t u[kSelLookups], lo[kSelLookups], hi[kSelLookups];
#pragma unroll
    for (int e = 0; e < kSelLookups; ++e) {
      const int i = i0 + e * nt;
      u[e] = i < np ? codes[i] : 0u;
    }
#pragma unroll
    for (int e = 0; e < kSelLookups; ++e) {
      lo[e] = hi[e] = 0u;
      if (i0 + e * nt < np && u[e] < nb) {
        lo[e] = __ldg(&sp.bkt_off[u[e]]);
        hi[e] = __ldg(&sp.bkt_off[u[e] + 1]);
      }
    }
#pragma unroll
    for (int e = 0; e < kSelLookups; ++e) {
      const int i = i0 + e * nt;
      if (i >= np) break;
      int n = 0, c0 = 0;
      if (u[e] >= nb) {
        set_err(sp.err, NR_DEV_BAD_CODE);
      } else if (hi[e] < lo[e] || (int64_t)hi[e] > sp.n_cl) {
        set_err(sp.err, NR_DEV_BAD_BUCKET);
      } else {
        n = (int)(hi[e] - lo[e]);
        c0 = (int)lo[e];
        if (n > sp.K_max) {
          set_err(sp.err, NR_DEV_TOO_MANY);
          n = sp.K_max;
        }
      }
      cnt[i] = n;
      c0s[i] = c0;
    }
  }
  __syncthreads();
  int M = block_exclusive_scan(cnt, np, warp_sums);
  *n_scored = M;  // every cluster of every probed bucket gets its distance
  // One pass over the candidates. C^dir keys are collected from the back of
  // the key array; the other clusters from the front when they are within the
  // gate of the running d_min. That gate is never tighter than the final one
  // when theta(x) = x + M(x) does not decrease with x: for m1 >= 0
  // (x + fmaf(m1, x, m0)) and for a calibrated curve (non-decreasing y, each
  // segment held within its end values).
  // Without the gate every candidate is kept: more than fit in shared memory
  // go straight to the slab (one distance pass instead of two)
  const bool direct = sp.gate_off && M > S_smem && slab != nullptr;
  if (tid == 0) sred[2] = 0u;  // keys collected from the front
  __syncthreads();
  const float m1 = sp.m1;
  const bool prefilter = !sp.gate_off && (sp.gate_n >= 2 || m1 >= 0.0f);
  // Slots are strided over the threads; each thread requests the next slot's
  // centroid row into L2 before it reads the current one. (Deeper prefetch,
  // or one contiguous run of slots a thread, measured slower at 1e9 rows:
  // these random row reads run at the GPU's random-sector rate already.)
  int pi = tid < M ? slot_probe(cnt, np, tid) : 0;
  for (int s = tid; s < (direct ? 0 : M); s += nt) {
    const uint32_t c = (uint32_t)(c0s[pi] + (s - cnt[pi]));
    const bool single = (pi + 1 < np ? cnt[pi + 1] : M) - cnt[pi] == 1;  // C^dir
    const int sn = s + nt;
    if (sn < M) {
      pi = slot_probe(cnt, np, sn);
      const float *mn = sp.cent + (size_t)(uint32_t)(c0s[pi] + (sn - cnt[pi])) * sp.b;
      prefetch_l2(mn);
      prefetch_l2(mn + sp.b - 1);
    }
    const float d = centroid_dist(sp.cent + (size_t)c * sp.b, slog, sp.b);
    const uint64_t key = tagged_key(d, c, single);
    if (single) {
      const unsigned pos = atomicAdd(&sred[1], 1u);
      if (pos < (unsigned)S_smem) keys[S_smem - 1 - pos] = key;
    } else {
      const uint32_t db = __float_as_uint(d);
      const uint32_t prev = atomicMin(&sred[0], db);  // d >= 0: bits order as values
      bool maybe = true;
      if (prefilter) {
        const float dm = __uint_as_float(prev < db ? prev : db);
        maybe = d <= __fadd_rn(dm, gate_margin(sp, dm));
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
    theta = __fadd_rn(dmin, gate_margin(sp, dmin));  // theta = d_min + M(d_min)
  }
  const int nA = (int)sred[1], nB = (int)sred[2];
  int Mk = direct ? S_smem + 1 : nA + nB;
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
  if (Mk <= S_smem) return select_tail_smem(sp, keys, Mk, warp_sums, seg, L, Lmax, total);
  // more keys than shared memory holds: every candidate key goes to the
  // query's global slab (tagged, or kEmpty where the gate drops it), and the
  // query is finished by select_overflow_block in a kernel of its own, whose
  // blocks hold more keys (returns -1: deferred)
  if (slab == nullptr || M > S_full) {
    if (tid == 0) set_err(sp.err, NR_DEV_TOO_MANY);
    *total = 0;
    return 0;
  }
  uint64_t *gk = reinterpret_cast<uint64_t *>(slab);
  for (int i = tid; i < np; i += nt) {  // each probe fills its clusters' slots
    const int o = cnt[i], n = (i + 1 < np ? cnt[i + 1] : M) - o;
    for (int j = 0; j < n; ++j) gk[o + j] = ((uint64_t)(uint32_t)(c0s[i] + j) << 1) | (n == 1 ? 1u : 0u);
  }
  __syncthreads();
  for (int s = tid; s < M; s += nt) {
    const uint64_t kc = gk[s];
    const uint32_t c = key_cluster(kc);
    const float d = centroid_dist(sp.cent + (size_t)c * sp.b, slog, sp.b);
    const bool keep = key_single(kc) || d <= theta;
    gk[s] = keep ? tagged_key(d, c, key_single(kc)) : kEmpty;
  }
  __syncthreads();
  *total = 0;
  return -1;
}

// The kept list of a deferred query from its slab keys[0..M) (tagged keys
// or kEmpty) by a bitonic network over the slab itself: C^dir and the first
// C others in key order, their segments and (L not null) clusters. For
// queries whose kept keys exceed the overflow block's shared memory.
__device__ __noinline__ int select_slab_finish(const SelectParams &sp, unsigned char *slab, int M,
                                               int *warp_sums, nr_seg *seg, int32_t *L, int Lmax,
                                               uint32_t *total) {
  const int tid = threadIdx.x, nt = blockDim.x;
  const int S_full = select_sort_cap(sp.P, sp.K_max);
  int Sn = 1;
  while (Sn < M) Sn <<= 1;
  uint64_t *keys = reinterpret_cast<uint64_t *>(slab);
  int *ints = reinterpret_cast<int *>(slab + (size_t)S_full * 8);
  for (int s = M + tid; s < Sn; s += nt) keys[s] = kEmpty;
  __syncthreads();
  bitonic_sort(keys, Sn);
  // keep C^dir and the first C survivors in key order
  int *keep = ints;  // [Sn]
  for (int s = tid; s < Sn; s += nt) {
    const uint64_t kk = keys[s];
    keep[s] = (s < M && kk != kEmpty && !key_single(kk)) ? 1 : 0;
  }
  __syncthreads();
  block_exclusive_scan(keep, Sn, warp_sums);  // survivor rank in key order
  for (int s = tid; s < Sn; s += nt) {
    const uint64_t kk = keys[s];
    int kp = 0;
    if (s < M && kk != kEmpty) kp = key_single(kk) ? 1 : (keep[s] < sp.C ? 1 : 0);
    keep[s] = kp;
  }
  __syncthreads();
  const int nl = block_exclusive_scan(keep, Sn, warp_sums);  // output positions
  for (int s = tid; s < Sn; s += nt) {
    const uint64_t kk = keys[s];
    if (s < M && kk != kEmpty) {
      const int pos = keep[s];
      const bool kept = (s + 1 < Sn ? keep[s + 1] : nl) > pos;
      if (kept) seg[pos].row0 = key_cluster(kk);  // cluster index for now
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

// Keys a block of the overflow kernel sorts in shared memory (its merge sort
// runs of 16 keys a thread over kSelOvfThreads threads), and the buckets of
// its preselection histogram.
constexpr int kSelOvfThreads = 512;
constexpr int kSelOvfKeys = 16 * kSelOvfThreads;
constexpr int kSelOvfBuckets = 2048;
__host__ __device__ inline size_t select_overflow_smem_bytes() {
  return (size_t)select_smem_keys(kSelOvfKeys) * 8 + (size_t)kSelOvfBuckets * 4 + 32 * 4 + 32;
}

// A deferred query, from its slab keys[0..M) (tagged keys, or kEmpty where
// the gate dropped a cluster). Only the C^dir keys and the C smallest others
// can be in the list, so the others are preselected first: a histogram of
// their distances' float bits (non-negative floats order as their bits) over
// [lo, hi] in kSelOvfBuckets buckets (a key in a lower bucket is smaller),
// and z* the bucket in which the count of others reaches C. Every other key
// in a bucket above z* has at least C smaller others, so it cannot be kept;
// the C^dir keys and the others up to bucket z* are collected into shared
// memory in any order, and the list is made from them exactly as
// select_tail_smem makes it (sort order, top-C, segments). When the
// collection exceeds kSelOvfKeys, select_slab_finish sorts the whole slab.
// skeys: select_smem_keys(kSelOvfKeys) keys and hist: kSelOvfBuckets uints of
// shared memory; sctl: 4 unsigned. Whole block (kSelOvfThreads threads) calls.
__device__ __forceinline__ int select_overflow_block(const SelectParams &sp, unsigned char *slab,
                                                     int M, uint64_t *skeys, uint32_t *hist,
                                                     unsigned *sctl, int *warp_sums, nr_seg *seg,
                                                     int32_t *L, int Lmax, uint32_t *total) {
  const int tid = threadIdx.x, nt = blockDim.x, lane = tid & 31;
  const uint64_t *gk = reinterpret_cast<const uint64_t *>(slab);
  for (int z = tid; z < kSelOvfBuckets; z += nt) hist[z] = 0u;
  if (tid == 0) {
    sctl[0] = 0u;           // keys collected
    sctl[1] = 0xffffffffu;  // smallest distance bits of the others
    sctl[2] = 0u;           // largest
    sctl[3] = 0u;           // the others
  }
  __syncthreads();
  uint32_t lo = 0xffffffffu, hi = 0u, no = 0u;
  for (int s = tid; s < M; s += nt) {
    const uint64_t k = gk[s];
    if (k == kEmpty || key_single(k)) continue;
    const uint32_t db = (uint32_t)(k >> 32);
    lo = min(lo, db);
    hi = max(hi, db);
    ++no;
  }
  lo = __reduce_min_sync(kFull, lo);
  hi = __reduce_max_sync(kFull, hi);
  no = __reduce_add_sync(kFull, no);
  if (lane == 0) {
    atomicMin(&sctl[1], lo);
    atomicMax(&sctl[2], hi);
    atomicAdd(&sctl[3], no);
  }
  __syncthreads();
  lo = sctl[1];
  hi = sctl[2];
  const uint32_t n_other = sctl[3];
  int shift = 0;
  if (hi >= lo)
    while (((hi - lo) >> shift) >= (uint32_t)kSelOvfBuckets) ++shift;
  uint32_t zs = kSelOvfBuckets - 1;  // every other key kept
  if (n_other > (uint32_t)sp.C) {
    for (int s = tid; s < M; s += nt) {
      const uint64_t k = gk[s];
      if (k == kEmpty || key_single(k)) continue;
      atomicAdd(&hist[((uint32_t)(k >> 32) - lo) >> shift], 1u);
    }
    __syncthreads();
    if (tid < 32) {  // the bucket in which the running count reaches C
      constexpr int per = kSelOvfBuckets / 32;
      uint32_t loc = 0;
      for (int e = 0; e < per; ++e) loc += hist[lane * per + e];
      uint32_t incl = loc;
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t v = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += v;
      }
      const unsigned hit = __ballot_sync(kFull, incl >= (uint32_t)sp.C);
      const int src = __ffs(hit) - 1;  // hit != 0: the total exceeds C
      if (lane == src) {
        uint32_t run = incl - loc;
        int z = lane * per;
        for (;; ++z) {
          run += hist[z];
          if (run >= (uint32_t)sp.C) break;
        }
        sctl[1] = (unsigned)z;
      }
    }
    __syncthreads();
    zs = sctl[1];
  }
  for (int s = tid; s < M; s += nt) {
    const uint64_t k = gk[s];
    if (k == kEmpty) continue;
    if (!key_single(k) && (((uint32_t)(k >> 32) - lo) >> shift) > zs) continue;
    const unsigned pos = atomicAdd(&sctl[0], 1u);
    if (pos < (unsigned)kSelOvfKeys) skeys[pos] = k;
  }
  __syncthreads();
  const int n = (int)sctl[0];
  __syncthreads();  // every thread has read the count
  if (n <= kSelOvfKeys) return select_tail_smem(sp, skeys, n, warp_sums, seg, L, Lmax, total);
  return select_slab_finish(sp, slab, M, warp_sums, seg, L, Lmax, total);
}

// ============================================================== select, mode 1
// The sequential centroid stage of Algorithm 2 (cent_mode 1), one block per
// query: probe scores and score bins (Algorithm 1), bins in order, C^dir of
// every bin entered, the other clusters in batches of b_batch with the
// running d_min gate, a bounded heap H of C kept sorted by (d, c), the
// heap-quality stop. Limits: P <= 2048 (C^dir is sorted by one block merge
// sort), b_batch <= 2048.

__host__ __device__ inline int seq_pow2(int v) {
  int p = 128;
  while (p < v) p <<= 1;
  return p;
}
// shared memory of select_block_seq
__host__ __device__ inline size_t select_seq_bytes(int P, int C, int B) {
  return (size_t)2 * C * 8                               // H, two buffers
         + (size_t)select_smem_keys(seq_pow2(B)) * 8     // one batch
         + (size_t)select_smem_keys(seq_pow2(P)) * 8     // C^dir keys
         + (size_t)(4 * P + 1) * 4                       // clusters, first cluster, slots, bin per probe
         + 32 * 4 * 2 + 64;                              // deviations and bits by rank, state
}

// Bin(s; n_bins, s_max) of Algorithm 1: min(n_bins - 1, floor(s n_bins / s_max)),
// or 0 when there is one bin or no finite s_max
__device__ __forceinline__ int score_bin(float s, int n_bins, float s_max) {
  if (n_bins <= 1 || !(s_max < __int_as_float(0x7f800000))) return 0;
  const int z = (int)__fdiv_rn(__fmul_rn(s, (float)n_bins), s_max);
  return z < n_bins - 1 ? z : n_bins - 1;
}

// Index of the last element of the nondecreasing off[lo..hi) that is <= v.
__device__ __forceinline__ int last_le(const int *off, int lo, int hi, int v) {
  int a = lo, b = hi - 1;
  while (a < b) {
    const int mid = (a + b + 1) >> 1;
    if (off[mid] <= v) a = mid;
    else b = mid - 1;
  }
  return a;
}

// Merge path: how many of the first d outputs of merging A[0..na) and
// B[0..nb) (ascending, ties to A) come from A. A is read through pad16 when
// a_pad, B when b_pad.
__device__ __forceinline__ int merge_split(const uint64_t *A, int na, bool a_pad, const uint64_t *B,
                                           int nb, bool b_pad, int d) {
  int a = d > nb ? d - nb : 0, hi = d < na ? d : na;
  while (a < hi) {
    const int mid = (a + hi) >> 1;
    const uint64_t x = A[a_pad ? pad16(mid) : mid], y = B[b_pad ? pad16(d - 1 - mid) : d - 1 - mid];
    if (x > y) hi = mid;
    else a = mid + 1;
  }
  return a;
}

template <int E>
__device__ __forceinline__ void sort_to_padded(uint64_t *k, int n) {
  uint64_t r[E];
  merge_sort_regs<E>(k, n, r);
  __syncthreads();
#pragma unroll
  for (int e = 0; e < E; ++e) k[pad16(threadIdx.x * E + e)] = r[e];
  __syncthreads();
}
// Sorts k[0..n) (n <= 16 blockDim.x) into k's padded layout (pad16(i) holds
// the i-th smallest; kEmpty past n).
__device__ __forceinline__ void sort_padded(uint64_t *k, int n) {
  const int nt = blockDim.x;
  if (n <= nt) sort_to_padded<1>(k, n);
  else if (n <= 2 * nt) sort_to_padded<2>(k, n);
  else if (n <= 4 * nt) sort_to_padded<4>(k, n);
  else if (n <= 8 * nt) sort_to_padded<8>(k, n);
  else sort_to_padded<16>(k, n);
}

__device__ __forceinline__ int select_block_seq(const SelectParams &sp, const float *slog,
                                                const uint32_t *codes, int np, unsigned char *seq,
                                                int *warp_sums, unsigned *sred, nr_seg *seg,
                                                int32_t *L, int Lmax, uint32_t *total,
                                                int *n_scored) {
  const int tid = threadIdx.x, nt = blockDim.x;
  const int C = sp.C, B = sp.b_batch, b = sp.b;
  uint64_t *Hb0 = reinterpret_cast<uint64_t *>(seq);
  uint64_t *Hb1 = Hb0 + C;
  uint64_t *Bk = Hb1 + C;
  uint64_t *dirk = Bk + select_smem_keys(seq_pow2(B));
  int *cnt = reinterpret_cast<int *>(dirk + select_smem_keys(seq_pow2(sp.P)));
  int *c0s = cnt + sp.P;
  int *nsoff = c0s + sp.P;  // [P + 1]
  int *zb = nsoff + sp.P + 1;
  float *sdr = reinterpret_cast<float *>(zb + sp.P);  // deviation of rank r
  int *bitr = reinterpret_cast<int *>(sdr + 32);      // bit index of rank r
  unsigned *st = reinterpret_cast<unsigned *>(bitr + 32);  // [0] u0, [1] |C^dir|
  const uint32_t nbk = 1u << b;
  // bucket lookups
  for (int i = tid; i < np; i += nt) {
    const uint32_t u = codes[i];
    int n = 0, c0 = 0;
    if (u >= nbk) {
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
  // the base code and the rank order of the bits (Eq. 10, Algorithm 1)
  if (tid == 0) {
    uint32_t u0 = 0;
    for (int j = 0; j < b; ++j) {
      const float l = slog[j], t = __ldg(&sp.tau[j]);
      if (l >= t) u0 |= 1u << j;
      sdr[j] = fabsf(__fsub_rn(l, t));
      bitr[j] = j;
    }
    for (int r = 1; r < b; ++r) {  // insertion sort by (deviation, bit)
      const float dv = sdr[r];
      const int bj = bitr[r];
      int q = r - 1;
      while (q >= 0 && (sdr[q] > dv || (sdr[q] == dv && bitr[q] > bj))) {
        sdr[q + 1] = sdr[q];
        bitr[q + 1] = bitr[q];
        --q;
      }
      sdr[q + 1] = dv;
      bitr[q + 1] = bj;
    }
    st[0] = u0;
    st[1] = 0u;
  }
  __syncthreads();
  // each probe's score (summed deviation of its flip set, ranks ascending),
  // its bin, and its clusters outside C^dir
  const uint32_t u0 = st[0];
  for (int i = tid; i < np; i += nt) {
    const uint32_t flips = codes[i] ^ u0;
    float s = 0.0f;
    for (int r = 0; r < b; ++r)
      if ((flips >> bitr[r]) & 1u) s = __fadd_rn(s, sdr[r]);
    zb[i] = score_bin(s, sp.n_bins, sp.s_max);
    nsoff[i] = cnt[i] >= 2 ? cnt[i] : 0;
  }
  __syncthreads();
  const int NS = block_exclusive_scan(nsoff, np, warp_sums);
  if (tid == 0) nsoff[np] = NS;
  __syncthreads();
  const bool gate_off = sp.gate_off;
  float dmin = __int_as_float(0x7f800000);
  int hN = 0, t_low = 0, b_proc = 0, nbat = 0;  // nbat: clusters of the batches processed
  bool stop = false;
  uint64_t *H = Hb0, *Hn = Hb1;
  int i = 0;
  while (i < np && !stop) {
    const int z = zb[i];
    int a = i + 1, e = np;  // first probe of a later bin
    while (a < e) {
      const int mid = (a + e) >> 1;
      if (zb[mid] <= z) a = mid + 1;
      else e = mid;
    }
    const int j = a;
    b_proc += 1;
    for (int p = i + tid; p < j; p += nt)  // C^dir of this bin
      if (cnt[p] == 1) {
        const uint32_t c = (uint32_t)c0s[p];
        const float d = centroid_dist(sp.cent + (size_t)c * b, slog, b);
        const unsigned pos = atomicAdd(&st[1], 1u);
        dirk[pos] = ((uint64_t)__float_as_uint(d) << 32) | c;
      }
    const int sa = nsoff[i], sb = nsoff[j];
    for (int x = sa; x < sb && !stop; x += B) {
      const int nb = sb - x < B ? sb - x : B;
      nbat += nb;
      if (tid == 0) sred[0] = 0xffffffffu;
      __syncthreads();
      for (int t = tid; t < nb; t += nt) {
        const int slot = x + t;
        const int p = last_le(nsoff, i, j, slot);
        const uint32_t c = (uint32_t)(c0s[p] + (slot - nsoff[p]));
        const float d = centroid_dist(sp.cent + (size_t)c * b, slog, b);
        Bk[t] = ((uint64_t)__float_as_uint(d) << 32) | c;
        atomicMin(&sred[0], __float_as_uint(d));
      }
      __syncthreads();
      const float bmin = __uint_as_float(sred[0]);
      if (bmin < dmin) dmin = bmin;
      float theta = __int_as_float(0x7f800000), front_th = theta;
      if (!gate_off) {
        const float m = gate_margin(sp, dmin);  // M(d_min)
        theta = __fadd_rn(dmin, m);
        front_th = __fadd_rn(dmin, __fmul_rn(sp.c_alpha_front, m));
      }
      for (int t = tid; t < nb; t += nt)  // the gate
        if (!(__uint_as_float((uint32_t)(Bk[t] >> 32)) <= theta)) Bk[t] = kEmpty;
      __syncthreads();
      sort_padded(Bk, nb);
      // gated keys of the batch (sorted, kEmpty last) and of H (a prefix)
      int bk = 0;
      {
        int lo = 0, hi = nb;
        while (lo < hi) {
          const int mid = (lo + hi) >> 1;
          if (Bk[pad16(mid)] != kEmpty) lo = mid + 1;
          else hi = mid;
        }
        bk = lo;
      }
      int hf = 0;
      {
        int lo = 0, hi = hN;
        while (lo < hi) {
          const int mid = (lo + hi) >> 1;
          if (__uint_as_float((uint32_t)(H[mid] >> 32)) <= theta) lo = mid + 1;
          else hi = mid;
        }
        hf = lo;
      }
      const int hn = hf + bk < C ? hf + bk : C;
      // the first hn of merge(H[0..hf), batch[0..bk)) into Hn
      const int Q = (hn + nt - 1) / nt;
      const int o0 = tid * Q < hn ? tid * Q : hn, o1 = o0 + Q < hn ? o0 + Q : hn;
      int ia = merge_split(H, hf, false, Bk, bk, true, o0);
      int ib = o0 - ia;
      int upd = 0, fr = 0;
      for (int o = o0; o < o1; ++o) {
        const uint64_t xa = ia < hf ? H[ia] : kEmpty, xb = ib < bk ? Bk[pad16(ib)] : kEmpty;
        const bool takeA = ib >= bk || (ia < hf && xa <= xb);
        if (takeA) {
          Hn[o] = xa;
          ++ia;
        } else {
          Hn[o] = xb;
          ++ib;
          ++upd;
          if (__uint_as_float((uint32_t)(xb >> 32)) <= front_th) ++fr;
        }
      }
      int updates, front;
      block_thread_scan(upd, warp_sums, &updates);
      block_thread_scan(fr, warp_sums, &front);
      uint64_t *tmp = H;
      H = Hn;
      Hn = tmp;
      hN = hn;
      t_low = (updates < sp.c_u_min && front < sp.c_f_min) ? t_low + 1 : 0;
      stop = sp.c_t_low > 0 && hN == C && b_proc >= sp.b_min && t_low >= sp.c_t_low;
      __syncthreads();
    }
    i = j;
  }
  // L = C^dir U H in (d, c) order, with the clusters' segments
  __syncthreads();
  const int nd = (int)st[1];
  *n_scored = nd + nbat;  // C^dir of the bins entered and the batches processed
  sort_padded(dirk, nd);
  const int n = nd + hN;
  const int Q = (n + nt - 1) / nt;
  const int o0 = tid * Q < n ? tid * Q : n, o1 = o0 + Q < n ? o0 + Q : n;
  const int ia0 = merge_split(dirk, nd, true, H, hN, false, o0);
  int ia = ia0, ib = o0 - ia0;
  int lsum = 0;
  for (int o = o0; o < o1; ++o) {
    const uint64_t xa = ia < nd ? dirk[pad16(ia)] : kEmpty, xb = ib < hN ? H[ib] : kEmpty;
    const bool takeA = ib >= hN || (ia < nd && xa <= xb);
    const uint32_t c = (uint32_t)(takeA ? xa : xb);
    if (takeA) ++ia;
    else ++ib;
    const uint32_t r0 = __ldg(&sp.cl_off[c]), r1 = __ldg(&sp.cl_off[c + 1]);
    if (r1 < r0 || (int64_t)r1 > sp.N) set_err(sp.err, NR_DEV_BAD_CLUSTER);
    else lsum += (int)(r1 - r0);
  }
  int tot;
  int spos = block_thread_scan(lsum, warp_sums, &tot);
  ia = ia0;
  ib = o0 - ia0;
  for (int o = o0; o < o1; ++o) {
    const uint64_t xa = ia < nd ? dirk[pad16(ia)] : kEmpty, xb = ib < hN ? H[ib] : kEmpty;
    const bool takeA = ib >= hN || (ia < nd && xa <= xb);
    const uint32_t c = (uint32_t)(takeA ? xa : xb);
    if (takeA) ++ia;
    else ++ib;
    const uint32_t r0 = __ldg(&sp.cl_off[c]), r1 = __ldg(&sp.cl_off[c + 1]);
    const int ln = (r1 < r0 || (int64_t)r1 > sp.N) ? 0 : (int)(r1 - r0);
    seg[o].row0 = r0;
    seg[o].pos = (uint32_t)spos;
    if (L) L[o] = (int32_t)c;
    spos += ln;
  }
  if (L)
    for (int t = n + tid; t < Lmax; t += nt) L[t] = -1;
  *total = (uint32_t)tot;
  return n;
}

}  // namespace nrq
