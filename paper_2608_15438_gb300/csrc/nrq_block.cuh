// Block-wide building blocks shared by the route and select kernels: scans,
// a bitonic sort in shared memory and a merge sort through registers.
#pragma once

#include "nrq_common.cuh"

namespace nrq {

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

// Exclusive prefix of v over the block's threads; *all = the sum. Starts
// with a barrier (warp_sums may still be read by a previous call).
__device__ __forceinline__ int block_thread_scan(int v, int *warp_sums, int *all) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  int x = v;
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(kFull, x, o);
    if (lane >= o) x += y;
  }
  __syncthreads();
  if (lane == 31) warp_sums[w] = x;
  __syncthreads();
  int before = 0, tot = 0;
  for (int i = 0; i < nw; ++i) {
    const int t = warp_sums[i];
    before += i < w ? t : 0;
    tot += t;
  }
  *all = tot;
  return before + x - v;
}

// Shared-memory position of element i of the merge sort's runs: one 8-byte
// gap every 16 keys, so that threads reading or writing their runs (a stride
// of E keys) fall on different banks.
__device__ __forceinline__ int pad16(int i) { return i + (i >> 4); }

// Block merge sort of k[0..n) ascending, for keys that are distinct apart
// from kEmpty padding; n <= E * blockDim.x, blockDim.x a power of two; k must
// hold pad16(E * blockDim.x) keys. On return r[e] holds sorted element
// threadIdx.x * E + e (kEmpty past n); k is clobbered.
// The keys are read striped, each thread sorts its E keys in registers (a
// bitonic network with compile-time indices), and runs are merged pairwise:
// every thread finds where its E outputs start on the merge path of its pair
// of runs by binary search and merges E keys.
template <int E>
__device__ __forceinline__ void merge_sort_regs(uint64_t *k, int n, uint64_t (&r)[E]) {
  const int tid = threadIdx.x, nt = blockDim.x;
  const int N = E * nt;
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int i = e * nt + tid;
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
  for (int e = 0; e < E; ++e) k[pad16(tid * E + e)] = r[e];
  __syncthreads();
  for (int w = E; w < N; w <<= 1) {
    const int lo = (tid * E) & ~(2 * w - 1);  // first key of my pair of runs
    const int d = tid * E - lo;               // my first output on its merge path
    int a = d > w ? d - w : 0, hi = d < w ? d : w;
    while (a < hi) {
      const int mid = (a + hi) >> 1;
      if (k[pad16(lo + mid)] > k[pad16(lo + w + d - 1 - mid)]) hi = mid;
      else a = mid + 1;
    }
    int i = a, j = d - a;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      const uint64_t x = i < w ? k[pad16(lo + i)] : kEmpty;
      const uint64_t y = j < w ? k[pad16(lo + w + j)] : kEmpty;
      const bool takeA = j >= w || (i < w && x <= y);
      r[e] = takeA ? x : y;
      i += takeA ? 1 : 0;
      j += takeA ? 0 : 1;
    }
    if (2 * w < N) {  // the last level's outputs stay in registers
      __syncthreads();
#pragma unroll
      for (int e = 0; e < E; ++e) k[pad16(tid * E + e)] = r[e];
      __syncthreads();
    }
  }
}

}  // namespace nrq
