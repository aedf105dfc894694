// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "neuroute.h"

// Makes `dev` the current device for a scope and restores the caller's;
// ok tells whether `dev` could be made current.
struct DeviceGuard {
  int prev = -1;
  bool ok = true;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    if (prev != dev) ok = cudaSetDevice(dev) == cudaSuccess;
  }
  ~DeviceGuard() {
    int cur = -1;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
  }
};

// Library status of a CUDA result; clears the runtime's last error.
inline nr_status cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return NR_OK;
  cudaGetLastError();
  return e == cudaErrorMemoryAllocation ? NR_ERR_OOM : NR_ERR_CUDA;
}

// Byte offset of (row r, 16-byte K chunk c) in the operand layout of the
// tensor-core encoder: K-major without swizzle, 8-row x 16-byte core matrices,
// the core matrices of one 8-row group consecutive along K (kchunks per row).
// The host writes W1 and W2 in this order; the kernel stages X and the hidden
// chunks in it.
__host__ __device__ inline uint32_t nr_tc_kmajor_off(int r, int c, int kchunks) {
  return (uint32_t)((r & 7) * 16 + (r >> 3) * kchunks * 128 + c * 128);
}

// Device-side check codes (first one wins; the host maps any to NR_ERR_DEVICE_CHECK)
enum : int {
  NR_DEV_OK = 0,
  NR_DEV_BAD_BUCKET = 1,   // bkt_off range reversed or past n_clusters
  NR_DEV_BAD_CLUSTER = 2,  // cl_off range reversed or past N
  NR_DEV_TOO_MANY = 3,     // a bucket holds more than K_max clusters
  NR_DEV_BAD_CODE = 4,     // a probe code >= 2^b
  NR_DEV_TIMEOUT = 5       // a bounded wait on an MMA completion barrier expired
};

struct nr_index {
  int device = 0;
  int dtype = 0;  // 0 uint8, 1 fp32
  int64_t N = 0;
  int D = 0, H = 0, b = 0, K_max = 0, t = 0;
  // encoder hidden layers after the first: widths, weights as the file
  // stores them (W [w x previous] then bias, per layer) and, for the kernel,
  // each layer's W transposed [previous x w] followed by its bias
  int n_mid = 0;
  int mid_w[7] = {0, 0, 0, 0, 0, 0, 0};
  float *Wm = nullptr, *WmT = nullptr;
  int64_t n_cl = 0;
  float in_scale = 1.0f;
  int64_t row_bytes = 0;
  // device arrays
  float *W1 = nullptr, *b1 = nullptr, *W2 = nullptr, *b2 = nullptr, *tau = nullptr;
  float *cent = nullptr;
  float *W1T = nullptr;  // [D][H]
  // fp16 operands of the tensor-core encoder, in chunks of 128 hidden units,
  // each chunk in the nr_tc_kmajor_off order: W1 [128 x D] per chunk, W2
  // [16 or 32 x 128] per chunk (rows >= b zero)
  void *W1h = nullptr;
  void *W2h = nullptr;
  // encoders with hidden layers after the first, on tensor cores layer by
  // layer: every layer's fp16 weights in (column tile, 64-wide K slice)
  // blocks in the nr_tc_kmajor_off order (n_ly = 0: such an encoder runs on
  // CUDA cores); the activation scratch of nr_encode and the index build,
  // grown on demand
  int n_ly = 0;
  size_t ly_off[9] = {};  // element offset of layer l's weights in Wl
  int ly_nt[9] = {};      // its column tile (a multiple of 16, at most 256)
  void *Wl = nullptr;
  void *enc_ws = nullptr;
  size_t enc_ws_cap = 0;
  uint32_t *bkt_off = nullptr, *cl_off = nullptr, *ids = nullptr;
  void *vec = nullptr;
  int *d_err = nullptr;
  nr_params params{};
  // workspace (grows on demand)
  void *ws = nullptr;
  size_t ws_cap = 0;
  int64_t last_nq = 0;
  int64_t *d_stats = nullptr;  // into ws, [last_nq x 4]
  bool timing = false;
  bool timed_last = false;
  cudaEvent_t ev[5] = {nullptr, nullptr, nullptr, nullptr, nullptr};
  int64_t launches = 0;
  int num_sms = 0;
  int smem_optin = 0;  // shared memory a block may opt in to, bytes
};

// Per-query statistics, int64 each: candidates, rounds, |L|, probes, clusters
// scored (centroid distances evaluated).
constexpr int NR_QSTATS = 5;

// Argument and size checks shared by every search entry point (budgets, k,
// batch size, and the sequential centroid stage's limits); NR_OK or
// NR_ERR_INVALID_ARG.
nr_status nr_check_budgets(const nr_index *ix, int64_t nq, int k, int P, int C);

// Per-query refinement segment: rows [row0, row0 + len) of cluster L[i]
// start at stream position pos.
struct nr_seg {
  uint32_t row0;
  uint32_t pos;
};

// Row sizes the query path supports: a multiple of 16 bytes up to 1 KB, and
// for fp32 rows a multiple of 64 bytes up to 8 KB (D up to 2048, the long-row
// refinement).
inline bool nr_row_bytes_ok(int dtype, int64_t row_bytes) {
  if (row_bytes < 16 || row_bytes % 16 != 0) return false;
  if (row_bytes <= 1024) return true;
  return dtype == 1 && row_bytes % 64 == 0 && row_bytes <= 8192;
}

// Index object helpers shared by the file loader and the GPU builder
// (nr_api.cu). The device must be current.
nr_index *nr_index_alloc();  // zeroed object with default params and host extras
nr_status nr_index_init_device(nr_index *ix);  // num_sms and the device check flag
// uploads fp32 W1 [H x D], b1 [H], W2 [b x H_last], b2 [b] and the middle
// layers Wm (host; NULL without any) and the encoder's derived forms; needs
// D, H, b, n_mid and mid_w set
nr_status nr_index_upload_encoder(nr_index *ix, const float *W1, const float *b1, const float *W2,
                                  const float *b2, const float *Wm);
// last hidden width and the number of floats of the middle layers
int nr_hidden_last(const nr_index *ix);
size_t nr_mid_floats(const nr_index *ix);

// kernel launchers (each returns cudaGetLastError() after the launch)
bool nr_encode_uses_tensor_cores(const nr_index *ix);
// device scratch an encode of n rows needs (the activations of an encoder
// with several hidden layers on tensor cores), 0 when none
size_t nr_encode_scratch_bytes(const nr_index *ix, int64_t n);
// scratch: nr_encode_scratch_bytes(ix, nq) bytes, or null to use (and grow,
// synchronising the device) the index's own
cudaError_t nr_launch_encode(nr_index *ix, const void *d_x, int64_t nq, float *d_logits,
                             cudaStream_t s, void *scratch = nullptr);
cudaError_t nr_launch_route(nr_index *ix, const float *d_logits, int64_t nq, int P,
                            uint32_t *d_codes, int32_t *d_nprobe, cudaStream_t s);
// dynamic shared memory of the select kernel for budgets (P, C) under the
// index's current parameters
size_t nr_select_smem_bytes(const nr_index *ix, int P, int C);
// global scratch per query that select needs for probe budget P (0: none)
size_t nr_select_slab_bytes(int P, int K_max);
// the global scratch of a select launch over nq queries: their slabs and the
// list of the queries deferred to its overflow kernel (0: none needed)
size_t nr_select_slab_total(int64_t nq, int P, int K_max);
cudaError_t nr_launch_select(nr_index *ix, const float *d_logits, const uint32_t *d_codes,
                             const int32_t *d_nprobe, int64_t nq, int P, int C, int32_t *d_L,
                             int32_t *d_nL, nr_seg *d_seg, uint32_t *d_slen, int64_t *d_stats,
                             void *d_slab, cudaStream_t s);
cudaError_t nr_launch_refine(nr_index *ix, const void *d_q, int64_t nq, int k, int Lmax,
                             const nr_seg *d_seg, const int32_t *d_nL, const uint32_t *d_slen,
                             int64_t *d_ids, float *d_dists, int64_t *d_stats,
                             unsigned int *d_counter, int32_t *d_perm, cudaStream_t s);
