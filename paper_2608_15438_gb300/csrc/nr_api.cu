// C ABI of the query path: index loading, argument checks, workspace and the
// launch sequence encode -> route -> select -> refine (see neuroute.h).
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <cmath>
#include <new>
#include <vector>

#include "neuroute.h"
#include "nr_internal.cuh"

namespace {

constexpr int kMaxProbe = 4096;
constexpr int kMaxClusterBudget = 4096;
constexpr int kMaxSelect = 65536;  // probe_budget * K_max (beyond 2,048: sorted in a global slab)
constexpr int kMaxTopK = 256;
constexpr size_t kChunkBudget = (size_t)8 << 30;  // workspace bytes per query chunk

uint32_t rd32(const unsigned char *h, int o) {
  uint32_t v;
  memcpy(&v, h + o, 4);
  return v;
}
uint64_t rd64(const unsigned char *h, int o) {
  uint64_t v;
  memcpy(&v, h + o, 8);
  return v;
}

size_t align256(size_t v) { return (v + 255) & ~(size_t)255; }

// Per-chunk workspace layout of a search over qc queries.
struct Layout {
  size_t logits, codes, nprobe, L, nL, seg, slen, slab, perm, enc, total;
};
Layout chunk_layout(const nr_index *ix, int64_t qc, int P, int C) {
  Layout l;
  size_t o = 0;
  const size_t Lmax = (size_t)P + (size_t)C;
  l.logits = o; o = align256(o + (size_t)qc * ix->b * 4);
  l.codes = o;  o = align256(o + (size_t)qc * P * 4);
  l.nprobe = o; o = align256(o + (size_t)qc * 4);
  l.L = o;      o = align256(o + (size_t)qc * Lmax * 4);
  l.nL = o;     o = align256(o + (size_t)qc * 4);
  l.seg = o;    o = align256(o + (size_t)qc * Lmax * sizeof(nr_seg));
  l.slen = o;   o = align256(o + (size_t)qc * 4);
  l.slab = o;   o = align256(o + nr_select_slab_total(qc, P, ix->K_max));
  l.perm = o;   o = align256(o + (size_t)qc * 4);
  l.enc = o;    o = align256(o + nr_encode_scratch_bytes(ix, qc));
  l.total = o;
  return l;
}

nr_status ensure_ws(nr_index *ix, size_t bytes) {
  if (bytes <= ix->ws_cap) return NR_OK;
  if (ix->ws) {
    // earlier calls' kernels (on the caller's or the library's streams) may
    // still read the old workspace
    cudaDeviceSynchronize();
    cudaFree(ix->ws);
    ix->ws = nullptr;
    ix->ws_cap = 0;
    ix->d_stats = nullptr;
  }
  size_t want = bytes + bytes / 4;
  if (cudaMalloc(&ix->ws, want) != cudaSuccess) {
    cudaGetLastError();
    if (cudaMalloc(&ix->ws, bytes) != cudaSuccess) {
      cudaGetLastError();
      ix->ws = nullptr;
      return NR_ERR_OOM;
    }
    want = bytes;
  }
  ix->ws_cap = want;
  return NR_OK;
}

struct TimedStage {
  int stage;  // 0 encode, 1 route, 2 select, 3 refine; -1 unused
  cudaEvent_t a, b;
};

nr_status check_params(const nr_params *p) {
  if (!(p->round_size >= 32 && p->round_size <= 4096 && (p->round_size & (p->round_size - 1)) == 0))
    return NR_ERR_INVALID_ARG;
  if (p->t_low < 0 || p->r_min < 0 || p->u_min < 0 || p->f_min < 0) return NR_ERR_INVALID_ARG;
  if (!(p->alpha_front >= 0.0f && p->alpha_front <= 1.0f)) return NR_ERR_INVALID_ARG;
  if (std::isnan(p->s_max) || std::isnan(p->gate_m0) || std::isnan(p->gate_m1)) return NR_ERR_INVALID_ARG;
  if ((p->cent_mode != 0 && p->cent_mode != 1) || p->n_bins < 1 || p->b_batch < 1 ||
      p->b_batch > 2048 || p->b_min < 0 || p->c_t_low < 0 || p->c_u_min < 0 || p->c_f_min < 0 ||
      !(p->c_alpha_front >= 0.0f && p->c_alpha_front <= 1.0f))
    return NR_ERR_INVALID_ARG;
  if (p->pipe_chunk < 0 || p->refine_ctas < 0 || p->refine_ctas > 32) return NR_ERR_INVALID_ARG;
  if (p->nonempty_budget != 0 && p->nonempty_budget != 1) return NR_ERR_INVALID_ARG;
  if (p->wait_limit_us > 60000000) return NR_ERR_INVALID_ARG;
  if (p->gate_n != 0) {
    if (p->gate_n < 2 || p->gate_n > 16) return NR_ERR_INVALID_ARG;
    for (int i = 0; i < p->gate_n; ++i) {
      if (!std::isfinite(p->gate_x[i]) || !std::isfinite(p->gate_y[i])) return NR_ERR_INVALID_ARG;
      if (i > 0 && !(p->gate_x[i] > p->gate_x[i - 1] && p->gate_y[i] >= p->gate_y[i - 1]))
        return NR_ERR_INVALID_ARG;
    }
  }
  return NR_OK;
}

}  // namespace

// Host-side extras of an index: the per-cluster "bucket holds one cluster"
// table used by K3, stage timers, and the device staging buffer of
// nr_search_host.
constexpr int kPipeSlots = 3;  // chunk buffers of the pipelined search

// Streams and events of the pipelined search (created on first use):
// a runs encode, route and select, b the refinement; sel[s] / ref[s] mark the
// end of select and of refinement in chunk buffer s.
struct PipeStreams {
  cudaStream_t a = nullptr, b = nullptr;
  cudaEvent_t fork = nullptr, join_a = nullptr, join_b = nullptr;
  cudaEvent_t sel[kPipeSlots] = {}, ref[kPipeSlots] = {};
};

struct nr_index_ext {
  std::vector<TimedStage> timers;
  void *io = nullptr;
  size_t io_cap = 0;
  PipeStreams pipe;
};

// The extension lives right after the index object (allocated together).
struct nr_index_full {
  nr_index ix;
  nr_index_ext ext;
};

static nr_index_ext *ext_of(nr_index *ix) { return &reinterpret_cast<nr_index_full *>(ix)->ext; }

nr_index *nr_index_alloc() {
  auto *full = new (std::nothrow) nr_index_full();
  if (!full) return nullptr;
  nr_params_default(&full->ix.params);
  return &full->ix;
}

nr_status nr_index_init_device(nr_index *ix) {
  cudaDeviceProp prop;
  if (cudaGetDeviceProperties(&prop, ix->device) != cudaSuccess) {
    cudaGetLastError();
    return NR_ERR_CUDA;
  }
  ix->num_sms = prop.multiProcessorCount;
  ix->smem_optin = (int)prop.sharedMemPerBlockOptin;
  if (cudaMalloc((void **)&ix->d_err, 16) != cudaSuccess) {
    cudaGetLastError();
    ix->d_err = nullptr;
    return NR_ERR_OOM;
  }
  if (cudaMemset(ix->d_err, 0, 16) != cudaSuccess) return NR_ERR_CUDA;
  return NR_OK;
}

int nr_hidden_last(const nr_index *ix) { return ix->n_mid > 0 ? ix->mid_w[ix->n_mid - 1] : ix->H; }

size_t nr_mid_floats(const nr_index *ix) {
  size_t n = 0;
  for (int i = 0, prev = ix->H; i < ix->n_mid; prev = ix->mid_w[i], ++i)
    n += (size_t)ix->mid_w[i] * prev + ix->mid_w[i];
  return n;
}

nr_status nr_index_upload_encoder(nr_index *ix, const float *W1, const float *b1, const float *W2,
                                  const float *b2, const float *Wm) {
  const int D = ix->D, H = ix->H, b = ix->b, HL = nr_hidden_last(ix);
  auto up = [&](void **dptr, const void *src, size_t bytes) -> nr_status {
    if (cudaMalloc(dptr, bytes > 0 ? bytes : 16) != cudaSuccess) {
      cudaGetLastError();
      *dptr = nullptr;
      return NR_ERR_OOM;
    }
    if (src && bytes && cudaMemcpy(*dptr, src, bytes, cudaMemcpyHostToDevice) != cudaSuccess)
      return NR_ERR_CUDA;
    return NR_OK;
  };
  std::vector<float> W1T((size_t)D * H);
  for (int u = 0; u < H; ++u)
    for (int j = 0; j < D; ++j) W1T[(size_t)j * H + u] = W1[(size_t)u * D + j];
  nr_status st;
  if ((st = up((void **)&ix->W1, W1, (size_t)H * D * 4)) != NR_OK) return st;
  if ((st = up((void **)&ix->b1, b1, (size_t)H * 4)) != NR_OK) return st;
  if ((st = up((void **)&ix->W2, W2, (size_t)b * HL * 4)) != NR_OK) return st;
  if ((st = up((void **)&ix->b2, b2, (size_t)b * 4)) != NR_OK) return st;
  if ((st = up((void **)&ix->W1T, W1T.data(), W1T.size() * 4)) != NR_OK) return st;
  if (ix->n_mid > 0) {
    // the middle layers as stored, and transposed per layer for the kernel
    const size_t n = nr_mid_floats(ix);
    std::vector<float> t(n);
    size_t o = 0;
    for (int l = 0, prev = H; l < ix->n_mid; prev = ix->mid_w[l], ++l) {
      const int w = ix->mid_w[l];
      for (int u = 0; u < w; ++u)
        for (int j = 0; j < prev; ++j) t[o + (size_t)j * w + u] = Wm[o + (size_t)u * prev + j];
      for (int u = 0; u < w; ++u) t[o + (size_t)w * prev + u] = Wm[o + (size_t)w * prev + u];
      o += (size_t)w * prev + w;
    }
    if ((st = up((void **)&ix->Wm, Wm, n * 4)) != NR_OK) return st;
    if ((st = up((void **)&ix->WmT, t.data(), n * 4)) != NR_OK) return st;
    // the tensor-core layers: every K a multiple of 64, every hidden width a
    // multiple of 64, b <= 256 (padded to a multiple of 16)
    bool tc = D % 64 == 0 && H % 64 == 0 && b <= 256;
    for (int l = 0; l < ix->n_mid; ++l) tc = tc && ix->mid_w[l] % 64 == 0;
    if (!tc) return NR_OK;
    const int L = ix->n_mid + 2;
    std::vector<int> Kl(L), Nl(L);
    std::vector<const float *> Wsrc(L);
    Kl[0] = D, Nl[0] = H, Wsrc[0] = W1;
    size_t o2 = 0;
    for (int l = 0, prev = H; l < ix->n_mid; prev = ix->mid_w[l], ++l) {
      Kl[l + 1] = prev, Nl[l + 1] = ix->mid_w[l], Wsrc[l + 1] = Wm + o2;
      o2 += (size_t)ix->mid_w[l] * prev + ix->mid_w[l];
    }
    Kl[L - 1] = HL, Nl[L - 1] = b, Wsrc[L - 1] = W2;
    size_t total = 0;
    for (int l = 0; l < L; ++l) {
      const int Np = (Nl[l] + 15) / 16 * 16;
      int nt = 16;  // the largest multiple of 16 that divides Np, at most 256
      for (int c = 256; c >= 16; c -= 16)
        if (Np % c == 0) {
          nt = c;
          break;
        }
      ix->ly_nt[l] = nt;
      ix->ly_off[l] = total;
      total += (size_t)Np * Kl[l];
    }
    std::vector<__half> wl(total, __float2half_rn(0.0f));
    for (int l = 0; l < L; ++l) {
      const int K = Kl[l], N = Nl[l], nt = ix->ly_nt[l], nks = K / 64;
      for (int r = 0; r < N; ++r)
        for (int k = 0; k < K; ++k) {
          const int ct = r / nt, rr = r % nt, ks = k / 64, kk = k % 64;
          const size_t at = ix->ly_off[l] + ((size_t)ct * nks + ks) * nt * 64 +
                            nr_tc_kmajor_off(rr, kk / 8, 8) / 2 + kk % 8;
          wl[at] = __float2half_rn(Wsrc[l][(size_t)r * K + k]);
        }
    }
    if ((st = up(&ix->Wl, wl.data(), wl.size() * 2)) != NR_OK) return st;
    ix->n_ly = L;
    return NR_OK;
  }
  // fp16 operands of the tensor-core encoder in its chunked operand order;
  // layer 2 padded to 16 or 32 rows (only shapes that kernel takes)
  if (D % 16 != 0 || H % 128 != 0 || b > 32) return NR_OK;
  const int n2 = b <= 16 ? 16 : 32;
  std::vector<__half> w1h((size_t)H * D), w2h((size_t)n2 * H, __float2half_rn(0.0f));
  for (int u = 0; u < H; ++u)
    for (int j = 0; j < D; ++j)
      w1h[(size_t)(u / 128) * 128 * D + nr_tc_kmajor_off(u % 128, j / 8, D / 8) / 2 + j % 8] =
          __float2half_rn(W1[(size_t)u * D + j]);
  for (int o = 0; o < b; ++o)
    for (int u = 0; u < H; ++u)
      w2h[(size_t)(u / 128) * n2 * 128 + nr_tc_kmajor_off(o, (u % 128) / 8, 16) / 2 + u % 8] =
          __float2half_rn(W2[(size_t)o * H + u]);
  if ((st = up(&ix->W1h, w1h.data(), w1h.size() * 2)) != NR_OK) return st;
  if ((st = up(&ix->W2h, w2h.data(), w2h.size() * 2)) != NR_OK) return st;
  return NR_OK;
}

extern "C" {

const char *nr_status_string(nr_status s) {
  switch (s) {
    case NR_OK: return "NR_OK";
    case NR_ERR_INVALID_ARG: return "NR_ERR_INVALID_ARG";
    case NR_ERR_IO: return "NR_ERR_IO";
    case NR_ERR_FORMAT: return "NR_ERR_FORMAT";
    case NR_ERR_OOM: return "NR_ERR_OOM";
    case NR_ERR_CUDA: return "NR_ERR_CUDA";
    case NR_ERR_DEVICE_CHECK: return "NR_ERR_DEVICE_CHECK";
  }
  return "NR_ERR_UNKNOWN";
}

nr_status nr_params_default(nr_params *p) {
  if (!p) return NR_ERR_INVALID_ARG;
  p->l_sel = 0;
  p->r_max = 0;
  p->s_max = INFINITY;
  p->gate_m0 = INFINITY;
  p->gate_m1 = 0.0f;
  p->round_size = 256;
  p->t_low = 4;
  p->u_min = 1;
  p->f_min = 1;
  p->r_min = 1;
  p->alpha_front = 0.5f;
  p->cent_mode = 0;
  p->n_bins = 1;
  p->b_batch = 256;
  p->b_min = 1;
  p->c_t_low = 0;
  p->c_u_min = 1;
  p->c_f_min = 1;
  p->c_alpha_front = 0.5f;
  p->gate_n = 0;
  for (int i = 0; i < 16; ++i) p->gate_x[i] = p->gate_y[i] = 0.0f;
  p->pipe_chunk = 0;
  p->refine_ctas = 0;
  p->nonempty_budget = 0;
  p->wait_limit_us = 0;
  return NR_OK;
}

void nr_index_free(nr_index *ix) {
  if (!ix) return;
  DeviceGuard g(ix->device);
  nr_index_ext *e = ext_of(ix);
  for (auto &t : e->timers) {
    cudaEventDestroy(t.a);
    cudaEventDestroy(t.b);
  }
  PipeStreams &ps = e->pipe;
  for (cudaEvent_t ev : {ps.fork, ps.join_a, ps.join_b})
    if (ev) cudaEventDestroy(ev);
  for (int i = 0; i < kPipeSlots; ++i) {
    if (ps.sel[i]) cudaEventDestroy(ps.sel[i]);
    if (ps.ref[i]) cudaEventDestroy(ps.ref[i]);
  }
  if (ps.a) cudaStreamDestroy(ps.a);
  if (ps.b) cudaStreamDestroy(ps.b);
  void *ptrs[] = {ix->W1, ix->b1, ix->W2, ix->b2, ix->Wm, ix->WmT, ix->tau, ix->cent, ix->W1T, ix->W1h, ix->W2h, ix->bkt_off,
                  ix->cl_off, ix->ids, ix->vec, ix->d_err, ix->ws, e->io, ix->Wl, ix->enc_ws};
  for (void *p : ptrs)
    if (p) cudaFree(p);
  delete reinterpret_cast<nr_index_full *>(ix);
}

nr_status nr_index_load(const char *path, int device, nr_index **out) {
  if (!path || !out) return NR_ERR_INVALID_ARG;
  *out = nullptr;
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess) {
    cudaGetLastError();
    return NR_ERR_CUDA;
  }
  if (device < 0 || device >= ndev) return NR_ERR_INVALID_ARG;
  FILE *f = fopen(path, "rb");
  if (!f) return NR_ERR_IO;
  unsigned char h[256];
  if (fread(h, 1, 256, f) != 256) {
    fclose(f);
    return NR_ERR_FORMAT;
  }
  if (fseeko(f, 0, SEEK_END) != 0) {
    fclose(f);
    return NR_ERR_IO;
  }
  const uint64_t fsize = (uint64_t)ftello(f);
  const uint32_t version = rd32(h, 8);
  if (memcmp(h, "NRIXv001", 8) != 0 || (version != 1 && version != 2)) {
    fclose(f);
    return NR_ERR_FORMAT;
  }
  nr_index *ix = nr_index_alloc();
  if (!ix) {
    fclose(f);
    return NR_ERR_OOM;
  }
  ix->device = device;
  ix->dtype = (int)rd32(h, 12);
  ix->N = (int64_t)rd64(h, 16);
  ix->D = (int)rd32(h, 24);
  ix->H = (int)rd32(h, 28);
  ix->b = (int)rd32(h, 32);
  ix->K_max = (int)rd32(h, 36);
  ix->t = (int)rd32(h, 40);
  ix->n_cl = (int64_t)rd64(h, 48);
  memcpy(&ix->in_scale, h + 56, 4);
  uint64_t off[10];
  for (int i = 0; i < 10; ++i) off[i] = rd64(h, 64 + 8 * i);
  // version 2: the encoder's hidden layers after the first
  ix->n_mid = version == 2 ? (int)rd32(h, 152) : 0;
  bool mid_ok = ix->n_mid >= 0 && ix->n_mid <= 7;
  for (int i = 0; mid_ok && i < ix->n_mid; ++i) {
    ix->mid_w[i] = (int)rd32(h, 156 + 4 * i);
    mid_ok = ix->mid_w[i] >= 1 && ix->mid_w[i] <= 4096;
  }
  const uint64_t mid_off = rd64(h, 192);
  const size_t esz = ix->dtype == 0 ? 1 : 4;
  ix->row_bytes = (int64_t)ix->D * (int64_t)esz;
  auto bad = [&](nr_status st) {
    fclose(f);
    nr_index_free(ix);
    return st;
  };
  if ((ix->dtype != 0 && ix->dtype != 1) || ix->b < 1 || ix->b > 24 || ix->D < 1 || ix->H < 1 ||
      ix->H > 4096 || ix->N < 1 || ix->N >= (int64_t)0xFFFFFFFFll || ix->n_cl < 1 ||
      ix->n_cl >= ((int64_t)1 << 31) || !nr_row_bytes_ok(ix->dtype, ix->row_bytes) ||
      ix->K_max < 0 || !mid_ok)
    return bad(NR_ERR_FORMAT);
  const uint64_t nb = ((uint64_t)1 << ix->b) + 1;
  const uint64_t sz[10] = {(uint64_t)ix->H * ix->D * 4, (uint64_t)ix->H * 4,
                           (uint64_t)ix->b * nr_hidden_last(ix) * 4, (uint64_t)ix->b * 4,
                           (uint64_t)ix->b * 4,         nb * 4,
                           (uint64_t)(ix->n_cl + 1) * 4, (uint64_t)ix->n_cl * ix->b * 4,
                           (uint64_t)ix->N * 4,         (uint64_t)ix->N * ix->D * esz};
  for (int i = 0; i < 10; ++i)
    if (off[i] < 256 || off[i] + sz[i] > fsize) return bad(NR_ERR_FORMAT);
  const uint64_t mid_sz = (uint64_t)nr_mid_floats(ix) * 4;
  if (ix->n_mid > 0 && (mid_off < 256 || mid_off + mid_sz > fsize)) return bad(NR_ERR_FORMAT);
  // host copies of the small sections
  std::vector<float> W1((size_t)ix->H * ix->D), b1(ix->H), W2((size_t)ix->b * nr_hidden_last(ix)),
      b2(ix->b), tau(ix->b), Wm(mid_sz / 4);
  std::vector<uint32_t> bkt(nb);
  auto rd = [&](int i, void *dst) {
    return fseeko(f, (off_t)off[i], SEEK_SET) == 0 && fread(dst, 1, sz[i], f) == sz[i];
  };
  if (!rd(0, W1.data()) || !rd(1, b1.data()) || !rd(2, W2.data()) || !rd(3, b2.data()) ||
      !rd(4, tau.data()) || !rd(5, bkt.data()))
    return bad(NR_ERR_IO);
  if (ix->n_mid > 0 && (fseeko(f, (off_t)mid_off, SEEK_SET) != 0 ||
                        fread(Wm.data(), 1, mid_sz, f) != mid_sz))
    return bad(NR_ERR_IO);
  // clusters per bucket: K_max from the header, else from the directory
  int kmax_dir = 1;
  for (uint64_t u = 0; u + 1 < nb; ++u) {
    if (bkt[u + 1] >= bkt[u]) {
      const uint32_t n = bkt[u + 1] - bkt[u];
      if ((int64_t)n > kmax_dir && n <= 65536) kmax_dir = (int)n;
    }
  }
  if (ix->K_max < 1) ix->K_max = kmax_dir;
  DeviceGuard g(device);
  nr_status st = nr_index_init_device(ix);
  if (st != NR_OK) return bad(st);
  if ((st = nr_index_upload_encoder(ix, W1.data(), b1.data(), W2.data(), b2.data(),
                                    ix->n_mid > 0 ? Wm.data() : nullptr)) != NR_OK)
    return bad(st);
  auto up = [&](void **dptr, const void *src, size_t bytes) -> nr_status {
    if (cudaMalloc(dptr, bytes > 0 ? bytes : 16) != cudaSuccess) {
      cudaGetLastError();
      *dptr = nullptr;
      return NR_ERR_OOM;
    }
    if (src && bytes && cudaMemcpy(*dptr, src, bytes, cudaMemcpyHostToDevice) != cudaSuccess)
      return NR_ERR_CUDA;
    return NR_OK;
  };
  if ((st = up((void **)&ix->tau, tau.data(), sz[4])) != NR_OK) return bad(st);
  if ((st = up((void **)&ix->bkt_off, bkt.data(), sz[5])) != NR_OK) return bad(st);
  // large sections streamed through a pinned staging buffer
  const size_t stage_bytes = (size_t)64 << 20;
  void *stage = nullptr;
  if (cudaMallocHost(&stage, stage_bytes) != cudaSuccess) {
    cudaGetLastError();
    return bad(NR_ERR_OOM);
  }
  auto stream_up = [&](int i, void **dptr) -> nr_status {
    if (cudaMalloc(dptr, sz[i] > 0 ? sz[i] : 16) != cudaSuccess) {
      cudaGetLastError();
      *dptr = nullptr;
      return NR_ERR_OOM;
    }
    if (fseeko(f, (off_t)off[i], SEEK_SET) != 0) return NR_ERR_IO;
    for (uint64_t done = 0; done < sz[i];) {
      const size_t n = (size_t)((sz[i] - done) < stage_bytes ? (sz[i] - done) : stage_bytes);
      if (fread(stage, 1, n, f) != n) return NR_ERR_IO;
      if (cudaMemcpy((char *)*dptr + done, stage, n, cudaMemcpyHostToDevice) != cudaSuccess)
        return NR_ERR_CUDA;
      done += n;
    }
    return NR_OK;
  };
  st = stream_up(6, (void **)&ix->cl_off);
  if (st == NR_OK) st = stream_up(7, (void **)&ix->cent);
  if (st == NR_OK) st = stream_up(8, (void **)&ix->ids);
  if (st == NR_OK) st = stream_up(9, &ix->vec);
  cudaFreeHost(stage);
  if (st != NR_OK) return bad(st);
  fclose(f);
  *out = ix;
  return NR_OK;
}

}  // extern "C"

namespace {

// Writes an index file: header fields from `ix` with N and n_cl given, the
// ten sections from src[i] (device memory where dev[i], else host memory),
// and with middle encoder layers (version 2) an eleventh section from mid
// (device memory where mid_dev).
nr_status write_nrix(const nr_index *ix, int64_t N, int64_t n_cl, const void *const src[10],
                     const bool dev[10], const void *mid, bool mid_dev, const char *path) {
  const uint64_t nb = ((uint64_t)1 << ix->b) + 1;
  const uint64_t sz[10] = {(uint64_t)ix->H * ix->D * 4, (uint64_t)ix->H * 4,
                           (uint64_t)ix->b * nr_hidden_last(ix) * 4, (uint64_t)ix->b * 4,
                           (uint64_t)ix->b * 4,         nb * 4,
                           (uint64_t)(n_cl + 1) * 4,    (uint64_t)n_cl * ix->b * 4,
                           (uint64_t)N * 4,             (uint64_t)N * ix->row_bytes};
  uint64_t off[10], cur = 256;
  for (int i = 0; i < 10; ++i) {
    off[i] = cur;
    cur = (cur + sz[i] + 255) & ~(uint64_t)255;
  }
  const uint64_t mid_sz = (uint64_t)nr_mid_floats(ix) * 4, mid_off = ix->n_mid > 0 ? cur : 0;
  if (ix->n_mid > 0) cur = (cur + mid_sz + 255) & ~(uint64_t)255;
  unsigned char h[256];
  memset(h, 0, sizeof(h));
  memcpy(h, "NRIXv001", 8);
  auto w32 = [&](int o, uint32_t v) { memcpy(h + o, &v, 4); };
  auto w64 = [&](int o, uint64_t v) { memcpy(h + o, &v, 8); };
  w32(8, ix->n_mid > 0 ? 2 : 1);
  if (ix->n_mid > 0) {
    w32(152, (uint32_t)ix->n_mid);
    for (int i = 0; i < ix->n_mid; ++i) w32(156 + 4 * i, (uint32_t)ix->mid_w[i]);
    w64(192, mid_off);
  }
  w32(12, (uint32_t)ix->dtype);
  w64(16, (uint64_t)N);
  w32(24, (uint32_t)ix->D);
  w32(28, (uint32_t)ix->H);
  w32(32, (uint32_t)ix->b);
  w32(36, (uint32_t)ix->K_max);
  w32(40, (uint32_t)ix->t);
  w64(48, (uint64_t)n_cl);
  memcpy(h + 56, &ix->in_scale, 4);
  for (int i = 0; i < 10; ++i) w64(64 + 8 * i, off[i]);
  w64(144, cur);
  FILE *f = fopen(path, "wb");
  if (!f) return NR_ERR_IO;
  const size_t stage_bytes = (size_t)64 << 20;
  void *stage = nullptr;
  if (cudaMallocHost(&stage, stage_bytes) != cudaSuccess) {
    cudaGetLastError();
    fclose(f);
    return NR_ERR_OOM;
  }
  nr_status st = NR_OK;
  static const unsigned char zeros[256] = {0};
  uint64_t at = 0;
  auto put = [&](const void *p, size_t n) {
    if (st == NR_OK && n && fwrite(p, 1, n, f) != n) st = NR_ERR_IO;
    at += n;
  };
  put(h, 256);
  for (int i = 0; i < 10 && st == NR_OK; ++i) {
    put(zeros, (size_t)(off[i] - at));
    if (!dev[i]) {
      put(src[i], (size_t)sz[i]);
      continue;
    }
    for (uint64_t done = 0; done < sz[i] && st == NR_OK;) {
      const size_t n = (size_t)((sz[i] - done) < stage_bytes ? (sz[i] - done) : stage_bytes);
      if (cudaMemcpy(stage, (const char *)src[i] + done, n, cudaMemcpyDeviceToHost) != cudaSuccess) {
        cudaGetLastError();
        st = NR_ERR_CUDA;
        break;
      }
      put(stage, n);
      done += n;
    }
  }
  if (ix->n_mid > 0 && st == NR_OK) {
    put(zeros, (size_t)(mid_off - at));
    if (!mid_dev) put(mid, (size_t)mid_sz);
    for (uint64_t done = 0; mid_dev && done < mid_sz && st == NR_OK;) {
      const size_t n = (size_t)((mid_sz - done) < stage_bytes ? (mid_sz - done) : stage_bytes);
      if (cudaMemcpy(stage, (const char *)mid + done, n, cudaMemcpyDeviceToHost) != cudaSuccess) {
        cudaGetLastError();
        st = NR_ERR_CUDA;
        break;
      }
      put(stage, n);
      done += n;
    }
  }
  put(zeros, (size_t)(cur - at));
  cudaFreeHost(stage);
  if (fclose(f) != 0 && st == NR_OK) st = NR_ERR_IO;
  return st;
}

}  // namespace

nr_status nr_check_budgets(const nr_index *ix, int64_t nq, int k, int P, int C) {
  if (nq < 0 || P < 1 || P > kMaxProbe || C < 1 || C > kMaxClusterBudget) return NR_ERR_INVALID_ARG;
  if ((int64_t)P * ix->K_max > kMaxSelect) return NR_ERR_INVALID_ARG;
  if (k < 1 || k > kMaxTopK || nq > ((int64_t)1 << 31) - 1) return NR_ERR_INVALID_ARG;
  // the sequential centroid stage sorts C^dir in one block and keeps H in
  // shared memory
  if (ix->params.cent_mode == 1 && (P > 2048 || nr_select_smem_bytes(ix, P, C) > (size_t)220 * 1024))
    return NR_ERR_INVALID_ARG;
  return NR_OK;
}

extern "C" {

nr_status nr_index_save(nr_index *ix, const char *path) {
  if (!ix || !path) return NR_ERR_INVALID_ARG;
  DeviceGuard g(ix->device);
  if (cudaDeviceSynchronize() != cudaSuccess) {
    cudaGetLastError();
    return NR_ERR_CUDA;
  }
  const void *src[10] = {ix->W1, ix->b1, ix->W2, ix->b2, ix->tau, ix->bkt_off,
                         ix->cl_off, ix->cent, ix->ids, ix->vec};
  const bool dev[10] = {true, true, true, true, true, true, true, true, true, true};
  return write_nrix(ix, ix->N, ix->n_cl, src, dev, ix->Wm, true, path);
}

nr_status nr_index_extract(nr_index *ix, const uint32_t *h_codes, int64_t n, const char *path,
                           int64_t *info) {
  if (!ix || !path || n < 0 || (n > 0 && !h_codes)) return NR_ERR_INVALID_ARG;
  const uint64_t nb = (uint64_t)1 << ix->b;
  std::vector<uint32_t> codes(h_codes, h_codes + n);
  for (uint32_t u : codes)
    if (u >= nb) return NR_ERR_INVALID_ARG;
  std::sort(codes.begin(), codes.end());
  codes.erase(std::unique(codes.begin(), codes.end()), codes.end());
  DeviceGuard g(ix->device);
  if (cudaDeviceSynchronize() != cudaSuccess) {
    cudaGetLastError();
    return NR_ERR_CUDA;
  }
  auto d2h = [](void *dst, const void *src, size_t bytes) {
    if (bytes == 0) return true;
    if (cudaMemcpy(dst, src, bytes, cudaMemcpyDeviceToHost) == cudaSuccess) return true;
    cudaGetLastError();
    return false;
  };
  // cluster and row ranges of the listed buckets
  std::vector<uint32_t> c0(codes.size()), c1(codes.size());
  for (size_t i = 0; i < codes.size(); ++i) {
    uint32_t pair[2];
    if (!d2h(pair, ix->bkt_off + codes[i], 8)) return NR_ERR_CUDA;
    if (pair[1] < pair[0] || pair[1] > (uint64_t)ix->n_cl) return NR_ERR_DEVICE_CHECK;
    c0[i] = pair[0];
    c1[i] = pair[1];
  }
  int64_t ncl = 0, nrow = 0;
  std::vector<uint32_t> bkt(nb + 1, 0), cl(1, 0);
  std::vector<std::vector<uint32_t>> clo(codes.size());
  for (size_t i = 0; i < codes.size(); ++i) {
    clo[i].resize((size_t)(c1[i] - c0[i]) + 1);
    if (!d2h(clo[i].data(), ix->cl_off + c0[i], clo[i].size() * 4)) return NR_ERR_CUDA;
    for (size_t k = 0; k + 1 < clo[i].size(); ++k) {
      if (clo[i][k + 1] < clo[i][k] || clo[i][k + 1] > (uint64_t)ix->N) return NR_ERR_DEVICE_CHECK;
      nrow += clo[i][k + 1] - clo[i][k];
      cl.push_back((uint32_t)nrow);
    }
    ncl += c1[i] - c0[i];
  }
  if (nrow < 1 || ncl < 1) return NR_ERR_INVALID_ARG;  // the file format needs a row
  {
    size_t i = 0;
    int64_t c = 0;
    for (uint64_t u = 0; u < nb; ++u) {
      bkt[u] = (uint32_t)c;
      if (i < codes.size() && codes[i] == u) c += c1[i] - c0[i], ++i;
    }
    bkt[nb] = (uint32_t)c;
  }
  std::vector<float> cent((size_t)ncl * ix->b), W1((size_t)ix->H * ix->D), b1(ix->H),
      W2((size_t)ix->b * nr_hidden_last(ix)), b2(ix->b), tau(ix->b), Wm(nr_mid_floats(ix));
  std::vector<uint32_t> ids((size_t)nrow);
  std::vector<unsigned char> vec;
  try {
    vec.resize((size_t)nrow * ix->row_bytes);
  } catch (...) {
    return NR_ERR_OOM;
  }
  int64_t ci = 0, ri = 0;
  for (size_t i = 0; i < codes.size(); ++i) {
    const size_t k = c1[i] - c0[i];
    if (!d2h(&cent[(size_t)ci * ix->b], ix->cent + (size_t)c0[i] * ix->b, k * ix->b * 4))
      return NR_ERR_CUDA;
    const uint32_t r0 = clo[i].front(), r1 = clo[i].back();
    if (r1 > r0) {
      if (!d2h(&ids[(size_t)ri], ix->ids + r0, (size_t)(r1 - r0) * 4)) return NR_ERR_CUDA;
      if (!d2h(&vec[(size_t)ri * ix->row_bytes], (const char *)ix->vec + (size_t)r0 * ix->row_bytes,
               (size_t)(r1 - r0) * ix->row_bytes))
        return NR_ERR_CUDA;
    }
    ci += k;
    ri += r1 - r0;
  }
  if (!d2h(W1.data(), ix->W1, W1.size() * 4) || !d2h(b1.data(), ix->b1, b1.size() * 4) ||
      !d2h(W2.data(), ix->W2, W2.size() * 4) || !d2h(b2.data(), ix->b2, b2.size() * 4) ||
      !d2h(tau.data(), ix->tau, tau.size() * 4) ||
      (ix->n_mid > 0 && !d2h(Wm.data(), ix->Wm, Wm.size() * 4)))
    return NR_ERR_CUDA;
  const void *src[10] = {W1.data(), b1.data(), W2.data(), b2.data(), tau.data(), bkt.data(),
                         cl.data(), cent.data(), ids.data(), vec.data()};
  const bool dev[10] = {false, false, false, false, false, false, false, false, false, false};
  const nr_status st = write_nrix(ix, nrow, ncl, src, dev, Wm.data(), false, path);
  if (st == NR_OK && info) {
    info[0] = nrow;
    info[1] = ncl;
  }
  return st;
}

nr_status nr_index_thresholds(nr_index *ix, float *h_tau) {
  if (!ix || !h_tau) return NR_ERR_INVALID_ARG;
  DeviceGuard g(ix->device);
  if (cudaMemcpy(h_tau, ix->tau, (size_t)ix->b * 4, cudaMemcpyDeviceToHost) != cudaSuccess) {
    cudaGetLastError();
    return NR_ERR_CUDA;
  }
  return NR_OK;
}

nr_status nr_index_info(const nr_index *ix, int64_t *info) {
  if (!ix || !info) return NR_ERR_INVALID_ARG;
  info[0] = ix->N;
  info[1] = ix->D;
  info[2] = ix->H;
  info[3] = ix->b;
  info[4] = ix->n_cl;
  info[5] = ix->dtype;
  info[6] = ix->K_max;
  info[7] = ix->t;
  return NR_OK;
}

nr_status nr_set_params(nr_index *ix, const nr_params *p) {
  if (!ix) return NR_ERR_INVALID_ARG;
  nr_params d;
  nr_params_default(&d);
  if (!p) p = &d;
  nr_status st = check_params(p);
  if (st != NR_OK) return st;
  ix->params = *p;
  return NR_OK;
}

nr_status nr_encode(nr_index *ix, const void *d_x, int64_t nq, float *d_logits, void *stream) {
  if (!ix || nq < 0) return NR_ERR_INVALID_ARG;
  if (nq == 0) return NR_OK;
  if (!d_x || !d_logits) return NR_ERR_INVALID_ARG;
  DeviceGuard g(ix->device);
  return cuda_status(nr_launch_encode(ix, d_x, nq, d_logits, (cudaStream_t)stream));
}

nr_status nr_route(nr_index *ix, const float *d_logits, int64_t nq, int probe_budget,
                   uint32_t *d_codes, int32_t *d_nprobe, void *stream) {
  if (!ix || nq < 0 || probe_budget < 1 || probe_budget > kMaxProbe) return NR_ERR_INVALID_ARG;
  if (nq == 0) return NR_OK;
  if (!d_logits || !d_codes || !d_nprobe || nq > (int64_t)1 << 30) return NR_ERR_INVALID_ARG;
  DeviceGuard g(ix->device);
  return cuda_status(nr_launch_route(ix, d_logits, nq, probe_budget, d_codes, d_nprobe,
                                     (cudaStream_t)stream));
}


nr_status nr_debug_clusters(nr_index *ix, const float *d_logits, int64_t nq, int probe_budget,
                            int cluster_budget, int32_t *d_clusters, int32_t *d_ncl,
                            void *stream) {
  if (!ix) return NR_ERR_INVALID_ARG;
  nr_status st = nr_check_budgets(ix, nq, 1, probe_budget, cluster_budget);
  if (st != NR_OK) return st;
  if (nq == 0) return NR_OK;
  if (!d_logits || !d_clusters || !d_ncl) return NR_ERR_INVALID_ARG;
  DeviceGuard g(ix->device);
  cudaStream_t s = (cudaStream_t)stream;
  const int P = probe_budget, C = cluster_budget;
  Layout l = chunk_layout(ix, nq, P, C);
  if ((st = ensure_ws(ix, l.total)) != NR_OK) return st;
  char *w = (char *)ix->ws;
  cudaError_t e = nr_launch_route(ix, d_logits, nq, P, (uint32_t *)(w + l.codes),
                                  (int32_t *)(w + l.nprobe), s);
  if (e == cudaSuccess)
    e = nr_launch_select(ix, d_logits, (uint32_t *)(w + l.codes), (int32_t *)(w + l.nprobe), nq,
                         P, C, d_clusters, d_ncl, (nr_seg *)(w + l.seg), (uint32_t *)(w + l.slen),
                         nullptr, nr_select_slab_bytes(P, ix->K_max) ? w + l.slab : nullptr, s);
  return cuda_status(e);
}

// Streams and events of the pipelined search, created once per index.
static nr_status ensure_pipe(nr_index *ix) {
  PipeStreams &ps = ext_of(ix)->pipe;
  if (ps.a) return NR_OK;
  int lo = 0, hi = 0;
  cudaError_t e = cudaDeviceGetStreamPriorityRange(&lo, &hi);
  // encode, route and select at the higher priority: their blocks are
  // scheduled first whenever refinement blocks leave room
  if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&ps.a, cudaStreamNonBlocking, hi);
  if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&ps.b, cudaStreamNonBlocking, lo);
  cudaEvent_t *evs[] = {&ps.fork, &ps.join_a, &ps.join_b};
  for (cudaEvent_t *ev : evs)
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(ev, cudaEventDisableTiming);
  for (int i = 0; i < kPipeSlots && e == cudaSuccess; ++i) {
    e = cudaEventCreateWithFlags(&ps.sel[i], cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ps.ref[i], cudaEventDisableTiming);
  }
  return cuda_status(e);
}

static nr_status search_impl(nr_index *ix, const void *d_q, const float *d_logits_in, int64_t nq,
                             int k, int P, int C, int64_t *d_ids, float *d_d, cudaStream_t s) {
  nr_status st = nr_check_budgets(ix, nq, k, P, C);
  if (st != NR_OK) return st;
  // chunks of qc queries: as many as the workspace budget allows, or
  // pipe_chunk when pipelined (refinement of chunk i on stream b while stream
  // a encodes, routes and selects chunk i + 1, i + 2 into other buffers)
  const int64_t pc = ix->params.pipe_chunk;
  const bool pipe = pc > 0 && nq > pc;
  const int slots = pipe ? kPipeSlots : 1;
  Layout one = chunk_layout(ix, 1, P, C);
  int64_t qc = (int64_t)(kChunkBudget / slots / (one.total > 0 ? one.total : 1));
  if (qc < 1) qc = 1;
  if (pipe && qc > pc) qc = pc;
  if (qc > nq) qc = nq;
  Layout l = chunk_layout(ix, qc, P, C);
  const size_t slot_bytes = align256(l.total);
  // workspace: [per-query stats][one query counter per buffer][chunk buffers]
  const size_t stats_off = 0;
  const size_t cnt_off = align256(stats_off + (size_t)nq * NR_QSTATS * 8);
  const size_t chunk_off = align256(cnt_off + 16 * (size_t)slots);
  if ((st = ensure_ws(ix, chunk_off + slot_bytes * (size_t)slots)) != NR_OK) return st;
  if (pipe && (st = ensure_pipe(ix)) != NR_OK) return st;
  char *w = (char *)ix->ws;
  int64_t *stats = (int64_t *)(w + stats_off);
  ix->d_stats = stats;
  ix->last_nq = nq;
  nr_index_ext *ex = ext_of(ix);
  PipeStreams &ps = ex->pipe;
  cudaStream_t sa = pipe ? ps.a : s, sb = pipe ? ps.b : s;
  size_t tslot = 0;
  auto tstart = [&](int stage, cudaStream_t st) -> size_t {
    if (!ix->timing) return 0;
    if (tslot >= ex->timers.size()) {
      TimedStage t{stage, nullptr, nullptr};
      cudaEventCreate(&t.a);
      cudaEventCreate(&t.b);
      ex->timers.push_back(t);
    }
    ex->timers[tslot].stage = stage;
    cudaEventRecord(ex->timers[tslot].a, st);
    return tslot;
  };
  auto tend = [&](size_t slot, cudaStream_t st) {
    if (!ix->timing) return;
    cudaEventRecord(ex->timers[slot].b, st);
    ++tslot;
  };
  cudaError_t e = cudaSuccess;
  if (pipe) {  // both library streams start after the caller's earlier work
    e = cudaEventRecord(ps.fork, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(sa, ps.fork, 0);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(sb, ps.fork, 0);
  }
  const int64_t RB = ix->row_bytes;
  int64_t i = 0;
  for (int64_t q0 = 0; q0 < nq && e == cudaSuccess; q0 += qc, ++i) {
    const int64_t n = (nq - q0) < qc ? (nq - q0) : qc;
    const int slot = (int)(i % slots);
    char *cw = w + chunk_off + slot_bytes * (size_t)slot;
    unsigned int *counter = (unsigned int *)(w + cnt_off + 16 * (size_t)slot);
    // buffer `slot` is free again once the refinement that last read it ended
    if (pipe && i >= slots && (e = cudaStreamWaitEvent(sa, ps.ref[slot], 0)) != cudaSuccess) break;
    const void *qp = (const char *)d_q + q0 * RB;
    const float *lg = d_logits_in ? d_logits_in + q0 * ix->b : (const float *)(cw + l.logits);
    size_t ev;
    if (!d_logits_in) {
      ev = tstart(0, sa);
      e = nr_launch_encode(ix, qp, n, (float *)(cw + l.logits), sa, cw + l.enc);
      tend(ev, sa);
      if (e != cudaSuccess) break;
    }
    ev = tstart(1, sa);
    e = nr_launch_route(ix, lg, n, P, (uint32_t *)(cw + l.codes), (int32_t *)(cw + l.nprobe), sa);
    tend(ev, sa);
    if (e != cudaSuccess) break;
    ev = tstart(2, sa);
    e = nr_launch_select(ix, lg, (uint32_t *)(cw + l.codes), (int32_t *)(cw + l.nprobe), n, P, C,
                         (int32_t *)(cw + l.L), (int32_t *)(cw + l.nL), (nr_seg *)(cw + l.seg),
                         (uint32_t *)(cw + l.slen), stats + q0 * NR_QSTATS,
                         nr_select_slab_bytes(P, ix->K_max) ? cw + l.slab : nullptr, sa);
    tend(ev, sa);
    if (e != cudaSuccess) break;
    if (pipe) {
      e = cudaEventRecord(ps.sel[slot], sa);
      if (e == cudaSuccess) e = cudaStreamWaitEvent(sb, ps.sel[slot], 0);
      if (e != cudaSuccess) break;
    }
    ev = tstart(3, sb);
    e = nr_launch_refine(ix, qp, n, k, P + C, (nr_seg *)(cw + l.seg), (int32_t *)(cw + l.nL),
                         (uint32_t *)(cw + l.slen), d_ids + q0 * k, d_d + q0 * k, stats + q0 * NR_QSTATS,
                         counter, (int32_t *)(cw + l.perm), sb);
    tend(ev, sb);
    if (pipe && e == cudaSuccess) e = cudaEventRecord(ps.ref[slot], sb);
  }
  if (pipe) {  // the caller's stream waits for everything enqueued above, even after an error
    cudaError_t j = cudaEventRecord(ps.join_a, sa);
    if (j == cudaSuccess) j = cudaEventRecord(ps.join_b, sb);
    if (j == cudaSuccess) j = cudaStreamWaitEvent(s, ps.join_a, 0);
    if (j == cudaSuccess) j = cudaStreamWaitEvent(s, ps.join_b, 0);
    if (e == cudaSuccess) e = j;
  }
  ix->timed_last = ix->timing;
  for (size_t t = tslot; t < ex->timers.size(); ++t) ex->timers[t].stage = -1;
  return cuda_status(e);
}

nr_status nr_search(nr_index *ix, const void *d_queries, int64_t nq, int k, int probe_budget,
                    int cluster_budget, int64_t *d_out_ids, float *d_out_dists, void *stream) {
  if (!ix) return NR_ERR_INVALID_ARG;
  if (nq > 0 && (!d_queries || !d_out_ids || !d_out_dists)) return NR_ERR_INVALID_ARG;
  DeviceGuard g(ix->device);
  if (nq == 0) return nr_check_budgets(ix, nq, k, probe_budget, cluster_budget);
  return search_impl(ix, d_queries, nullptr, nq, k, probe_budget, cluster_budget, d_out_ids,
                     d_out_dists, (cudaStream_t)stream);
}

nr_status nr_search_logits(nr_index *ix, const void *d_queries, const float *d_logits, int64_t nq,
                           int k, int probe_budget, int cluster_budget, int64_t *d_out_ids,
                           float *d_out_dists, void *stream) {
  if (!ix) return NR_ERR_INVALID_ARG;
  if (nq > 0 && (!d_queries || !d_logits || !d_out_ids || !d_out_dists)) return NR_ERR_INVALID_ARG;
  DeviceGuard g(ix->device);
  if (nq == 0) return nr_check_budgets(ix, nq, k, probe_budget, cluster_budget);
  return search_impl(ix, d_queries, d_logits, nq, k, probe_budget, cluster_budget, d_out_ids,
                     d_out_dists, (cudaStream_t)stream);
}

nr_status nr_search_host(nr_index *ix, const void *h_queries, int64_t nq, int k, int probe_budget,
                         int cluster_budget, int64_t *h_out_ids, float *h_out_dists,
                         void *stream) {
  if (!ix) return NR_ERR_INVALID_ARG;
  nr_status st = nr_check_budgets(ix, nq, k, probe_budget, cluster_budget);
  if (st != NR_OK) return st;
  if (nq == 0) return NR_OK;
  if (!h_queries || !h_out_ids || !h_out_dists) return NR_ERR_INVALID_ARG;
  DeviceGuard g(ix->device);
  cudaStream_t s = (cudaStream_t)stream;
  // device staging for the inputs and outputs, kept by the index and grown on demand
  const size_t qb = align256((size_t)nq * ix->row_bytes);
  const size_t ib = align256((size_t)nq * k * 8);
  const size_t db = align256((size_t)nq * k * 4);
  nr_index_ext *ex = ext_of(ix);
  if (ex->io_cap < qb + ib + db) {
    if (ex->io) cudaFree(ex->io);
    ex->io = nullptr;
    ex->io_cap = 0;
    if (cudaMalloc(&ex->io, qb + ib + db) != cudaSuccess) {
      cudaGetLastError();
      ex->io = nullptr;
      return NR_ERR_OOM;
    }
    ex->io_cap = qb + ib + db;
  }
  char *d = (char *)ex->io;
  cudaError_t e = cudaMemcpyAsync(d, h_queries, (size_t)nq * ix->row_bytes, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) {
    st = search_impl(ix, d, nullptr, nq, k, probe_budget, cluster_budget, (int64_t *)(d + qb),
                     (float *)(d + qb + ib), s);
    if (st == NR_OK) {
      e = cudaMemcpyAsync(h_out_ids, d + qb, (size_t)nq * k * 8, cudaMemcpyDeviceToHost, s);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(h_out_dists, d + qb + ib, (size_t)nq * k * 4, cudaMemcpyDeviceToHost, s);
    }
  }
  const cudaError_t e2 = cudaStreamSynchronize(s);
  if (st != NR_OK) return st;
  if (e == cudaSuccess) e = e2;
  return cuda_status(e);
}

nr_status nr_query_stats(nr_index *ix, int64_t *d_stats, int64_t nq, void *stream) {
  if (!ix || nq < 0 || nq > ix->last_nq || (nq > 0 && (!d_stats || !ix->d_stats)))
    return NR_ERR_INVALID_ARG;
  if (nq == 0) return NR_OK;
  DeviceGuard g(ix->device);
  return cuda_status(cudaMemcpyAsync(d_stats, ix->d_stats, (size_t)nq * NR_QSTATS * 8,
                                     cudaMemcpyDeviceToDevice, (cudaStream_t)stream));
}

nr_status nr_last_stats(nr_index *ix, nr_stats *out) {
  if (!ix || !out) return NR_ERR_INVALID_ARG;
  DeviceGuard g(ix->device);
  memset(out, 0, sizeof(*out));
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_status(e);
  out->nq = ix->last_nq;
  if (ix->last_nq > 0 && ix->d_stats) {
    std::vector<int64_t> h((size_t)ix->last_nq * NR_QSTATS);
    e = cudaMemcpy(h.data(), ix->d_stats, h.size() * 8, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_status(e);
    for (int64_t i = 0; i < ix->last_nq; ++i) {
      const int64_t *r = &h[(size_t)i * NR_QSTATS];
      out->candidates += r[0];
      out->rounds += r[1];
      out->clusters += r[2];
      out->probes += r[3];
      out->scored += r[4];
    }
  }
  int flag = 0;
  e = cudaMemcpy(&flag, ix->d_err, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_status(e);
  if (flag != 0) {
    cudaMemset(ix->d_err, 0, sizeof(int));
    return NR_ERR_DEVICE_CHECK;
  }
  return NR_OK;
}

nr_status nr_enable_timing(nr_index *ix, int on) {
  if (!ix) return NR_ERR_INVALID_ARG;
  ix->timing = on != 0;
  return NR_OK;
}

nr_status nr_last_timing(nr_index *ix, float *ms) {
  if (!ix || !ms) return NR_ERR_INVALID_ARG;
  DeviceGuard g(ix->device);
  for (int i = 0; i < 4; ++i) ms[i] = 0.0f;
  if (!ix->timed_last) return NR_OK;
  for (auto &t : ext_of(ix)->timers) {
    if (t.stage < 0) continue;
    if (cudaEventSynchronize(t.b) != cudaSuccess) return NR_ERR_CUDA;
    float v = 0.0f;
    if (cudaEventElapsedTime(&v, t.a, t.b) != cudaSuccess) return NR_ERR_CUDA;
    ms[t.stage] += v;
  }
  return NR_OK;
}

int64_t nr_kernel_launches(const nr_index *ix) { return ix ? ix->launches : 0; }

}  // extern "C"
