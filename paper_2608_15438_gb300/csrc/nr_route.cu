// K2 route: binarisation (Eq. 10), deviation scores (Sec. 3.2.3) and the
// probe list of Algorithm 1: one block per query by threshold enumeration
// (nrq::route_block) without the R_max filter, else one warp per query
// (nrq::route_warp).
#include <cuda_runtime.h>
#include <stdint.h>

#include "nr_internal.cuh"
#include "nrq_route.cuh"

namespace {

__global__ void route_kernel(nrq::RouteParams rp, const float *__restrict__ logits, int64_t nq,
                             uint32_t *__restrict__ codes, int32_t *__restrict__ nprobe) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, wpb = blockDim.x >> 5;
  const int64_t q = (int64_t)blockIdx.x * wpb + warp;
  if (q >= nq) return;  // uniform per warp
  unsigned char *heap = smem + (size_t)warp * nrq::route_heap_bytes(rp.Q);
  uint32_t *out = codes + (size_t)q * rp.P;
  const int n = nrq::route_warp(rp, logits + q * rp.b, heap, out);
  for (int t = n + lane; t < rp.P; t += 32) out[t] = 0xffffffffu;
  if (lane == 0) nprobe[q] = n;
}

// One 128-thread block per query: the threshold enumeration (route_block).
__global__ void __launch_bounds__(nrq::kRouteThreads) route_block_kernel(
    nrq::RouteParams rp, const float *__restrict__ logits, int64_t nq, uint32_t *__restrict__ codes,
    int32_t *__restrict__ nprobe) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int64_t q = blockIdx.x;
  if (q >= nq) return;
  uint32_t *out = codes + (size_t)q * rp.P;
  const int n = nrq::route_block(rp, logits + q * rp.b, smem, out);
  for (int t = n + (int)threadIdx.x; t < rp.P; t += nrq::kRouteThreads) out[t] = 0xffffffffu;
  if (threadIdx.x == 0) nprobe[q] = n;
}

}  // namespace

nrq::RouteParams nr_route_params(const nr_index *ix, int P) {
  const nr_params &p = ix->params;
  nrq::RouteParams rp;
  rp.tau = ix->tau;
  rp.b = ix->b;
  rp.bsel = (p.l_sel > 0 && p.l_sel < ix->b) ? p.l_sel : ix->b;
  rp.rmax = p.r_max;
  rp.smax = p.s_max;
  rp.P = P;
  rp.bkt_off = ix->bkt_off;
  rp.nonempty = p.nonempty_budget;
  rp.Q = p.nonempty_budget ? NR_NONEMPTY_SCAN * P : P;
  return rp;
}

size_t nr_route_heap_bytes(int Q) { return nrq::route_heap_bytes(Q); }

cudaError_t nr_launch_route(nr_index *ix, const float *d_logits, int64_t nq, int P,
                            uint32_t *d_codes, int32_t *d_nprobe, cudaStream_t s) {
  if (nq <= 0) return cudaSuccess;
  const nrq::RouteParams rpb = nr_route_params(ix, P);  // before the launch configuration
  if (ix->params.r_max <= 0) {  // threshold enumeration
    const size_t smem = nrq::route_block_bytes(P, rpb.nonempty, rpb.Q);
    cudaError_t e = cudaFuncSetAttribute(route_block_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    route_block_kernel<<<(unsigned)nq, nrq::kRouteThreads, smem, s>>>(rpb, d_logits, nq, d_codes,
                                                                       d_nprobe);
    ix->launches += 1;
    return cudaGetLastError();
  }
  const size_t per_warp = nr_route_heap_bytes(rpb.Q);
  // warps per block: the choice that packs the most warps into an SM's
  // shared memory (the heap is the limit at large probe budgets)
  const size_t sm_bytes = (size_t)227 * 1024;
  int wpb = 1, best = 0;
  for (int w = 4; w >= 1; w >>= 1) {
    const size_t blk = per_warp * (size_t)w;
    if (blk > sm_bytes) continue;
    int blocks = (int)(sm_bytes / (blk + 1024));
    if (blocks > 32) blocks = 32;
    const int warps = blocks * w > 64 ? 64 : blocks * w;
    if (warps > best) {
      best = warps;
      wpb = w;
    }
  }
  const size_t smem = per_warp * (size_t)wpb;
  cudaError_t e = cudaFuncSetAttribute(route_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  const int64_t grid = (nq + wpb - 1) / wpb;
  const nrq::RouteParams rp = nr_route_params(ix, P);  // before the launch configuration
  route_kernel<<<(unsigned)grid, 32 * wpb, smem, s>>>(rp, d_logits, nq,
                                                       d_codes, d_nprobe);
  ix->launches += 1;
  return cudaGetLastError();
}
