// nr_search_static: the whole query path with its scratch memory in a fixed,
// file-scope device array instead of the index's growable workspace, so the
// call itself allocates nothing.
//
// It exists for callers that are not allowed to allocate device memory while
// they serve queries: code that runs under a device-memory budget owned by a
// host framework or inference server (whose allocator must see every byte),
// and latency-critical loops where cudaMalloc / cudaFree, which may
// synchronise the device, are not acceptable. The paper has no counterpart;
// the kernels and their results are exactly those of nr_search.
//
// The array is NR_STATIC_SCRATCH_BYTES long and lives as long as the library
// is loaded, on every GPU that loads it. Host code cannot use the array's
// name as a device address (on the host it only names a stand-in), so the
// device address is looked up with cudaGetSymbolAddress once per device, on
// the first call made on that device, with that device current, and kept for
// the life of the process: a device reset (cudaDeviceReset) after that call
// leaves the kept address stale, so the library must not be used across one.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "neuroute.h"
#include "nr_internal.cuh"

#define NR_STATIC_SCRATCH_BYTES ((size_t)32 << 20)

static __device__ __align__(256) unsigned char g_nr_static_scratch[NR_STATIC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void *g_scratch_addr[kMaxDevices] = {};

size_t up256(size_t v) { return (v + 255) & ~(size_t)255; }

// Device address of the array on `device` (which must be current).
nr_status scratch_address(int device, void **out) {
  if (device < 0 || device >= kMaxDevices) return NR_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_scratch_addr[device]) {
    void *p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_nr_static_scratch);
    if (e != cudaSuccess || !p) {
      cudaGetLastError();
      return NR_ERR_CUDA;
    }
    g_scratch_addr[device] = p;
  }
  *out = g_scratch_addr[device];
  return NR_OK;
}

}  // namespace

extern "C" nr_status nr_search_static(nr_index *ix, const void *d_queries, int64_t nq, int k,
                                      int probe_budget, int cluster_budget, int64_t *d_out_ids,
                                      float *d_out_dists, void *stream) {
  if (!ix) return NR_ERR_INVALID_ARG;
  const int P = probe_budget, C = cluster_budget;
  // the checks of every other search entry point (budgets, k, batch size,
  // the sequential centroid stage's limits)
  nr_status st = nr_check_budgets(ix, nq, k, P, C);
  if (st != NR_OK) return st;
  if (nq == 0) return NR_OK;
  if (!d_queries || !d_out_ids || !d_out_dists) return NR_ERR_INVALID_ARG;
  // scratch layout: logits, codes, probe counts, cluster lists and their
  // counts, segments, stream lengths, the refinement order, per-query stats,
  // select's global sort slabs, the query counter, the activations of an
  // encoder with several hidden layers. nq < 2^31 and every
  // per-query size is bounded (P, C <= 4096, b <= 24, the slab <= 768 KiB),
  // so no product below overflows size_t.
  const size_t Lmax = (size_t)P + (size_t)C, q = (size_t)nq;
  size_t o = 0;
  const size_t o_logits = o; o = up256(o + q * ix->b * 4);
  const size_t o_codes = o;  o = up256(o + q * P * 4);
  const size_t o_nprobe = o; o = up256(o + q * 4);
  const size_t o_L = o;      o = up256(o + q * Lmax * 4);
  const size_t o_nL = o;     o = up256(o + q * 4);
  const size_t o_seg = o;    o = up256(o + q * Lmax * sizeof(nr_seg));
  const size_t o_slen = o;   o = up256(o + q * 4);
  const size_t o_perm = o;   o = up256(o + q * 4);
  const size_t o_stats = o;  o = up256(o + q * NR_QSTATS * 8);
  const size_t slab_q = nr_select_slab_bytes(P, ix->K_max);
  const size_t o_slab = o;   o = up256(o + nr_select_slab_total((int64_t)q, P, ix->K_max));
  const size_t o_count = o;  o = up256(o + 16);
  const size_t o_enc = o;    o = up256(o + nr_encode_scratch_bytes(ix, (int64_t)q));
  if (o > NR_STATIC_SCRATCH_BYTES) return NR_ERR_INVALID_ARG;  // request too large for the array
  DeviceGuard g(ix->device);
  if (!g.ok) return NR_ERR_CUDA;
  void *base = nullptr;
  st = scratch_address(ix->device, &base);
  if (st != NR_OK) return st;
  char *w = static_cast<char *>(base);
  cudaStream_t s = (cudaStream_t)stream;
  float *logits = (float *)(w + o_logits);
  int64_t *stats = (int64_t *)(w + o_stats);
  // every buffer below is fully written before it is read, except the
  // refine kernel's query counter, which its launcher clears on the stream
  cudaError_t e = nr_launch_encode(ix, d_queries, nq, logits, s, w + o_enc);
  if (e == cudaSuccess)
    e = nr_launch_route(ix, logits, nq, P, (uint32_t *)(w + o_codes), (int32_t *)(w + o_nprobe), s);
  if (e == cudaSuccess)
    e = nr_launch_select(ix, logits, (uint32_t *)(w + o_codes), (int32_t *)(w + o_nprobe), nq, P, C,
                         (int32_t *)(w + o_L), (int32_t *)(w + o_nL), (nr_seg *)(w + o_seg),
                         (uint32_t *)(w + o_slen), stats, slab_q ? w + o_slab : nullptr, s);
  if (e == cudaSuccess)
    e = nr_launch_refine(ix, d_queries, nq, k, (int)Lmax, (nr_seg *)(w + o_seg),
                         (int32_t *)(w + o_nL), (uint32_t *)(w + o_slen), d_out_ids, d_out_dists,
                         stats, (unsigned int *)(w + o_count), (int32_t *)(w + o_perm), s);
  // statistics of this call are read from the array by nr_last_stats / nr_query_stats
  ix->d_stats = stats;
  ix->last_nq = nq;
  ix->timed_last = false;
  return cuda_status(e);
}
