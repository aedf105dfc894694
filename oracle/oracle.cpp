// NeuRoute query-path oracle (test infrastructure only; see oracle.h).
// Plain loops, one query at a time, no blocking or fusion. Each function names
// the part of the paper it restates.
#include "oracle.h"

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <functional>
#include <limits>
#include <queue>
#include <set>
#include <thread>
#include <unordered_set>
#include <utility>
#include <vector>

struct or_index {
  int dtype = 0;
  int64_t N = 0;
  int D = 0, H = 0, b = 0, K_max = 0, t = 0;
  int64_t n_cl = 0;
  float in_scale = 1.0f;
  std::vector<float> W1, b1, W2, b2, tau, cent;
  // hidden layers after the first (file version 2): widths, and per layer
  // W [width x previous width] then its bias, concatenated as in the file
  int n_mid = 0;
  std::vector<int> mid_w;
  std::vector<float> Wm;
  std::vector<uint32_t> bkt_off, cl_off, ids;
  std::vector<uint8_t> vec;  // N * D * elem bytes
};

static const float kInf = std::numeric_limits<float>::infinity();

extern "C" void or_params_default(or_params *p) {
  p->l_sel = 0;
  p->r_max = 0;
  p->s_max = kInf;
  p->gate_m0 = kInf;
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
  p->nonempty_budget = 0;
}

// The gate margin M(x) (Sec. 3.4): m0 + m1 x, or the calibrated monotone
// piecewise-linear curve: flat beyond its ends, on segment i (the last
// breakpoint with x_i <= x) y_i + (x - x_i) (y_{i+1} - y_i) / (x_{i+1} - x_i)
// in fp32, the last step fused, then held within [y_i, y_{i+1}]: the paper
// asks for a monotone curve, and this keeps it monotone after fp32 rounding.
static float gate_margin(const or_params *p, float x) {
  if (p->gate_n < 2) return std::fmaf(p->gate_m1, x, p->gate_m0);
  int i = 0;
  while (i + 1 < p->gate_n && p->gate_x[i + 1] <= x) ++i;
  if (x <= p->gate_x[0]) return p->gate_y[0];
  if (i == p->gate_n - 1) return p->gate_y[i];
  const float s = (p->gate_y[i + 1] - p->gate_y[i]) / (p->gate_x[i + 1] - p->gate_x[i]);
  const float v = std::fmaf(x - p->gate_x[i], s, p->gate_y[i]);
  return std::min(std::max(v, p->gate_y[i]), p->gate_y[i + 1]);
}
extern "C" float or_gate_margin(const or_params *p, float x) { return gate_margin(p, x); }
static bool gate_is_off(const or_params *p) {
  return p->gate_n < 2 && std::isinf(p->gate_m0) && p->gate_m0 > 0.0f;
}

// ---------------------------------------------------------------- index file
// Layout: 256-byte header, then ten 256-byte-aligned sections
// (W1, b1, W2, b2, tau, bkt_off, cl_off, cent, ids, vec).
template <class T>
static bool read_section(FILE *f, uint64_t off, size_t count, std::vector<T> &out) {
  out.resize(count);
  if (count == 0) return true;
  if (fseeko(f, (off_t)off, SEEK_SET) != 0) return false;
  return fread(out.data(), sizeof(T), count, f) == count;
}

static uint32_t rd32(const unsigned char *h, int o) {
  uint32_t v;
  memcpy(&v, h + o, 4);
  return v;
}
static uint64_t rd64(const unsigned char *h, int o) {
  uint64_t v;
  memcpy(&v, h + o, 8);
  return v;
}

extern "C" or_index *or_index_load(const char *path, char *err, int errlen) {
  auto fail = [&](const char *msg) -> or_index * {
    if (err && errlen > 0) snprintf(err, (size_t)errlen, "%s", msg);
    return nullptr;
  };
  FILE *f = fopen(path, "rb");
  if (!f) return fail("cannot open index file");
  unsigned char h[256];
  if (fread(h, 1, 256, f) != 256) {
    fclose(f);
    return fail("truncated header");
  }
  const uint32_t version = rd32(h, 8);
  if (memcmp(h, "NRIXv001", 8) != 0 || (version != 1 && version != 2)) {
    fclose(f);
    return fail("bad magic or version");
  }
  or_index *ix = new or_index();
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
  ix->n_mid = version == 2 ? (int)rd32(h, 152) : 0;
  bool widths_ok = ix->n_mid >= 0 && ix->n_mid <= 7;
  for (int i = 0; widths_ok && i < ix->n_mid; ++i) {
    ix->mid_w.push_back((int)rd32(h, 156 + 4 * i));
    widths_ok = ix->mid_w.back() >= 1;
  }
  const uint64_t mid_off = rd64(h, 192);
  if (ix->dtype < 0 || ix->dtype > 1 || ix->b < 1 || ix->b > 24 || ix->D < 1 || ix->H < 1 ||
      !widths_ok) {
    fclose(f);
    delete ix;
    return fail("bad header fields");
  }
  const int h_last = ix->n_mid > 0 ? ix->mid_w.back() : ix->H;
  size_t mid_n = 0;
  for (int i = 0, prev = ix->H; i < ix->n_mid; prev = ix->mid_w[i], ++i)
    mid_n += (size_t)ix->mid_w[i] * prev + ix->mid_w[i];
  size_t esz = ix->dtype == 0 ? 1 : 4;
  size_t nb = ((size_t)1 << ix->b) + 1;
  bool ok = read_section(f, off[0], (size_t)ix->H * ix->D, ix->W1) &&
            read_section(f, off[1], (size_t)ix->H, ix->b1) &&
            read_section(f, off[2], (size_t)ix->b * h_last, ix->W2) &&
            (ix->n_mid == 0 || read_section(f, mid_off, mid_n, ix->Wm)) &&
            read_section(f, off[3], (size_t)ix->b, ix->b2) &&
            read_section(f, off[4], (size_t)ix->b, ix->tau) &&
            read_section(f, off[5], nb, ix->bkt_off) &&
            read_section(f, off[6], (size_t)ix->n_cl + 1, ix->cl_off) &&
            read_section(f, off[7], (size_t)ix->n_cl * ix->b, ix->cent) &&
            read_section(f, off[8], (size_t)ix->N, ix->ids) &&
            read_section(f, off[9], (size_t)ix->N * ix->D * esz, ix->vec);
  fclose(f);
  if (!ok) {
    delete ix;
    return fail("truncated section");
  }
  return ix;
}

extern "C" void or_index_free(or_index *ix) { delete ix; }

extern "C" int or_index_mid(const or_index *ix, int32_t *widths) {
  for (int i = 0; i < ix->n_mid; ++i) widths[i] = ix->mid_w[i];
  return ix->n_mid;
}

extern "C" void or_index_info(const or_index *ix, int64_t *info) {
  info[0] = ix->N;
  info[1] = ix->D;
  info[2] = ix->H;
  info[3] = ix->b;
  info[4] = ix->n_cl;
  info[5] = ix->dtype;
  info[6] = ix->K_max;
  info[7] = ix->t;
}
extern "C" const uint32_t *or_index_bkt_off(const or_index *ix) { return ix->bkt_off.data(); }
extern "C" const uint32_t *or_index_cl_off(const or_index *ix) { return ix->cl_off.data(); }
extern "C" const uint32_t *or_index_ids(const or_index *ix) { return ix->ids.data(); }
extern "C" const float *or_index_tau(const or_index *ix) { return ix->tau.data(); }
extern "C" const float *or_index_cent(const or_index *ix) { return ix->cent.data(); }

// ---------------------------------------------------------------- threads
static void parallel_for(int64_t n, int nthreads, const std::function<void(int64_t)> &fn) {
  if (nthreads <= 1 || n <= 1) {
    for (int64_t i = 0; i < n; ++i) fn(i);
    return;
  }
  std::vector<std::thread> th;
  std::atomic_int64_t next{0};
  for (int t = 0; t < nthreads; ++t)
    th.emplace_back([&]() {
      for (;;) {
        int64_t i = next.fetch_add(1);
        if (i >= n) break;
        fn(i);
      }
    });
  for (auto &x : th) x.join();
}

// ---------------------------------------------------------------- encoder
// Sec. 3.2.1 and the encoder table of the appendix: l = E(x), an MLP whose
// hidden layers are linear then ReLU (BatchNorm folded into the linear map)
// and whose last layer is linear: h_1 = max(0, W1 (s x) + b1), h_i =
// max(0, W_i h_{i-1} + b_i), l = W2 h_L + b2, in double, rounded to fp32 at
// the end.
static void encode_one(const or_index *ix, const void *x, int64_t i, float *out) {
  const int D = ix->D, H = ix->H, b = ix->b;
  std::vector<double> xin(D), h(H);
  for (int j = 0; j < D; ++j) {
    double v = ix->dtype == 0 ? (double)((const uint8_t *)x)[(size_t)i * D + j]
                              : (double)((const float *)x)[(size_t)i * D + j];
    xin[j] = (double)ix->in_scale * v;
  }
  for (int u = 0; u < H; ++u) {
    double acc = (double)ix->b1[u];
    for (int j = 0; j < D; ++j) acc += (double)ix->W1[(size_t)u * D + j] * xin[j];
    h[u] = acc > 0.0 ? acc : 0.0;
  }
  size_t o = 0;  // walks the middle layers' weights and biases
  for (int l = 0; l < ix->n_mid; ++l) {
    const int prev = (int)h.size(), w = ix->mid_w[l];
    std::vector<double> g(w);
    const float *W = ix->Wm.data() + o, *bias = W + (size_t)w * prev;
    for (int u = 0; u < w; ++u) {
      double acc = (double)bias[u];
      for (int j = 0; j < prev; ++j) acc += (double)W[(size_t)u * prev + j] * h[j];
      g[u] = acc > 0.0 ? acc : 0.0;
    }
    o += (size_t)w * prev + w;
    h.swap(g);
  }
  const int hl = (int)h.size();
  for (int q = 0; q < b; ++q) {
    double acc = (double)ix->b2[q];
    for (int u = 0; u < hl; ++u) acc += (double)ix->W2[(size_t)q * hl + u] * h[u];
    out[q] = (float)acc;
  }
}

extern "C" void or_encode(const or_index *ix, const void *x, int64_t nq, float *logits, int nthreads) {
  parallel_for(nq, nthreads, [&](int64_t i) { encode_one(ix, x, i, logits + (size_t)i * ix->b); });
}

extern "C" void or_encode_mlp(int dtype, int D, int H, int b, int n_mid, const int *mid_w,
                              float in_scale, const float *W1, const float *b1, const float *W2,
                              const float *b2, const float *Wm, const void *x, int64_t nq,
                              float *logits, int nthreads) {
  or_index e;  // an index holding only the encoder
  e.dtype = dtype;
  e.D = D;
  e.H = H;
  e.b = b;
  e.in_scale = in_scale;
  e.n_mid = n_mid;
  size_t mid_n = 0;
  for (int i = 0, prev = H; i < n_mid; prev = mid_w[i], ++i) {
    e.mid_w.push_back(mid_w[i]);
    mid_n += (size_t)mid_w[i] * prev + mid_w[i];
  }
  const int hl = n_mid > 0 ? mid_w[n_mid - 1] : H;
  e.W1.assign(W1, W1 + (size_t)H * D);
  e.b1.assign(b1, b1 + H);
  e.W2.assign(W2, W2 + (size_t)b * hl);
  e.b2.assign(b2, b2 + b);
  if (n_mid > 0) e.Wm.assign(Wm, Wm + mid_n);
  or_encode(&e, x, nq, logits, nthreads);
}

extern "C" void or_encode_weights(int dtype, int D, int H, int b, float in_scale, const float *W1,
                                  const float *b1, const float *W2, const float *b2, const void *x,
                                  int64_t nq, float *logits, int nthreads) {
  or_encode_mlp(dtype, D, H, b, 0, nullptr, in_scale, W1, b1, W2, b2, nullptr, x, nq, logits,
                nthreads);
}

// ---------------------------------------------------------------- probe order
// Algorithm 1: flip sets F over the least-certain bits, scored by the summed
// deviation s = sum_{r in F} delta. Key = (cost, |F|, rank mask), cost added in
// fp32 from 0.0f over ascending rank.
static uint64_t probe_key(float cost, int size, uint32_t mask) {
  uint32_t cb;
  memcpy(&cb, &cost, 4);
  return ((uint64_t)cb << 32) | ((uint64_t)(uint32_t)size << 24) | (uint64_t)mask;
}

static float flip_cost(const float *sd, int b, uint32_t mask) {
  float acc = 0.0f;
  for (int r = 0; r < b; ++r)
    if ((mask >> r) & 1u) acc = acc + sd[r];
  return acc;
}

static int popcount32(uint32_t v) {
  int c = 0;
  while (v) {
    c += (int)(v & 1u);
    v >>= 1;
  }
  return c;
}

static int flippable_ranks(int b, const or_params *p) {
  return (p->l_sel > 0 && p->l_sel < b) ? p->l_sel : b;
}

extern "C" int or_probe_order(int b, const float *sd, int P, const or_params *p, uint64_t *keys) {
  if (b < 0 || b > 24 || P <= 0) return 0;
  const int bs = flippable_ranks(b, p);
  std::priority_queue<uint64_t, std::vector<uint64_t>, std::greater<uint64_t>> frontier;
  std::unordered_set<uint32_t> seen;
  frontier.push(probe_key(0.0f, 0, 0u));  // F = {} : the base bucket, score 0
  seen.insert(0u);
  int n = 0;
  while (n < P && !frontier.empty()) {
    uint64_t key = frontier.top();
    frontier.pop();
    keys[n++] = key;
    uint32_t mask = (uint32_t)(key & 0xFFFFFFu);
    int size = (int)((key >> 24) & 0xFFu);
    if (p->r_max > 0 && size >= p->r_max) continue;
    for (int r = 0; r < bs; ++r) {
      if ((mask >> r) & 1u) continue;
      uint32_t m2 = mask | (1u << r);
      if (seen.count(m2)) continue;
      float c = flip_cost(sd, b, m2);
      if (!(c <= p->s_max)) continue;  // supersets cost no less: prune
      seen.insert(m2);
      frontier.push(probe_key(c, size + 1, m2));
    }
  }
  return n;
}

extern "C" int or_probe_order_allsubsets(int b, const float *sd, int P, const or_params *p,
                                         uint64_t *keys) {
  if (b < 0 || b > 20 || P <= 0) return 0;
  const int bs = flippable_ranks(b, p);
  std::vector<uint64_t> all;
  for (uint32_t m = 0; m < (1u << b); ++m) {
    if (m >> bs) continue;
    int size = popcount32(m);
    if (p->r_max > 0 && size > p->r_max) continue;
    float c = flip_cost(sd, b, m);
    if (m != 0 && !(c <= p->s_max)) continue;
    all.push_back(probe_key(c, size, m));
  }
  std::sort(all.begin(), all.end());
  int n = (int)std::min<size_t>((size_t)P, all.size());
  for (int i = 0; i < n; ++i) keys[i] = all[i];
  return n;
}

// Eq. 10 (a_j = [l_j >= tau_j]), BucketId (bit j of the code = a_j),
// delta_j = |l_j - tau_j|, ranks by (delta, bit index), then Algorithm 1.
extern "C" int or_probe_list(int b, const float *logit, const float *tau, int P, const or_params *p,
                             uint32_t *codes, uint64_t *keys, int32_t *perm) {
  uint32_t u0 = 0;
  std::vector<float> delta(b);
  for (int j = 0; j < b; ++j) {
    if (logit[j] >= tau[j]) u0 |= 1u << j;
    float d = logit[j] - tau[j];
    delta[j] = std::fabs(d);
  }
  std::vector<int> pi(b);
  for (int j = 0; j < b; ++j) pi[j] = j;
  std::sort(pi.begin(), pi.end(), [&](int a, int c) {
    return delta[a] < delta[c] || (delta[a] == delta[c] && a < c);
  });
  std::vector<float> sd(b);
  for (int r = 0; r < b; ++r) sd[r] = delta[pi[r]];
  if (perm)
    for (int r = 0; r < b; ++r) perm[r] = pi[r];
  std::vector<uint64_t> k((size_t)std::max(P, 1));
  int n = or_probe_order(b, sd.data(), P, p, k.data());
  for (int i = 0; i < n; ++i) {
    uint32_t rmask = (uint32_t)(k[i] & 0xFFFFFFu);
    uint32_t flips = 0;
    for (int r = 0; r < b; ++r)
      if ((rmask >> r) & 1u) flips |= 1u << pi[r];  // ApplyFlips
    codes[i] = u0 ^ flips;
    if (keys) keys[i] = k[i];
  }
  return n;
}

// The probe list against the index: with the non-empty budget, the first P
// codes in key order whose buckets hold a cluster, among the first
// OR_NONEMPTY_SCAN * P flip sets (plain reading of the D3 variant: empty
// buckets are enumerated but not spent).
extern "C" int or_probe_list_index(const or_index *ix, const float *logit, int P, const or_params *p,
                                   uint32_t *codes, uint64_t *keys) {
  if (!p->nonempty_budget)
    return or_probe_list(ix->b, logit, ix->tau.data(), P, p, codes, keys, nullptr);
  const int scan = OR_NONEMPTY_SCAN * P;
  std::vector<uint32_t> c((size_t)scan);
  std::vector<uint64_t> k((size_t)scan);
  const int m = or_probe_list(ix->b, logit, ix->tau.data(), scan, p, c.data(), k.data(), nullptr);
  int n = 0;
  for (int i = 0; i < m && n < P; ++i) {
    if (ix->bkt_off[(size_t)c[i] + 1] == ix->bkt_off[c[i]]) continue;  // empty bucket
    codes[n] = c[i];
    if (keys) keys[n] = k[i];
    ++n;
  }
  return n;
}

// ---------------------------------------------------------------- centroid stage
// Sec. 3.4.2 / Algorithm 2: buckets holding one cluster go straight to C^dir;
// the other buckets' centroids are scored by squared L2 in logit space, gated
// by theta = d_min + M(d_min), and the C best survivors form C^cent.
static float centroid_distance(const float *logit, const float *mu, int b) {
  float acc = 0.0f;
  for (int j = 0; j < b; ++j) {
    float t = logit[j] - mu[j];
    acc = std::fmaf(t, t, acc);
  }
  return acc;
}

extern "C" float or_centroid_dist(const or_index *ix, const float *logit, int64_t c) {
  if (c < 0 || c >= ix->n_cl) return kInf;
  return centroid_distance(logit, &ix->cent[(size_t)c * ix->b], ix->b);
}

static bool dc_less(const std::pair<float, int64_t> &a, const std::pair<float, int64_t> &c) {
  return a.first < c.first || (a.first == c.first && a.second < c.second);
}

extern "C" int or_cluster_list(const or_index *ix, const float *logit, const uint32_t *codes,
                               int nprobe, int C, const or_params *p, int32_t *L, float *dL,
                               int32_t *n_dir, int64_t *n_scored) {
  const int b = ix->b;
  const uint64_t nbuckets = (uint64_t)1 << b;
  std::vector<std::pair<float, int64_t>> dir, cand;
  for (int i = 0; i < nprobe; ++i) {
    uint64_t u = codes[i];
    if (u >= nbuckets) return -1;
    uint32_t c0 = ix->bkt_off[u], c1 = ix->bkt_off[u + 1];
    if (c1 < c0 || (int64_t)c1 > ix->n_cl) return -1;
    if (c1 - c0 == 1) {
      dir.push_back({centroid_distance(logit, &ix->cent[(size_t)c0 * b], b), (int64_t)c0});
    } else {
      for (uint32_t c = c0; c < c1; ++c)
        cand.push_back({centroid_distance(logit, &ix->cent[(size_t)c * b], b), (int64_t)c});
    }
  }
  float dmin = kInf;
  for (auto &e : cand) dmin = std::min(dmin, e.first);
  const bool gate_off = gate_is_off(p);
  float theta = kInf;
  if (!gate_off && !cand.empty()) theta = dmin + gate_margin(p, dmin);
  std::vector<std::pair<float, int64_t>> surv;
  for (auto &e : cand)
    if (e.first <= theta) surv.push_back(e);
  std::sort(surv.begin(), surv.end(), dc_less);
  if ((int)surv.size() > C) surv.resize((size_t)C);
  std::vector<std::pair<float, int64_t>> all(dir);
  all.insert(all.end(), surv.begin(), surv.end());
  std::sort(all.begin(), all.end(), dc_less);
  for (size_t i = 0; i < all.size(); ++i) {
    L[i] = (int32_t)all[i].second;
    if (dL) dL[i] = all[i].first;
  }
  if (n_dir) *n_dir = (int32_t)dir.size();
  // every cluster of every probed bucket had its centroid distance evaluated
  if (n_scored) *n_scored = (int64_t)(dir.size() + cand.size());
  return (int)all.size();
}

// Algorithm 2 in its own order (Sec. 3.4.2): bins from Algorithm 1 in
// increasing score, each bin's single-cluster buckets to C^dir, its other
// clusters in batches; per batch the running d_min, the gate, the bounded
// heap kept under the gate, the heap/front update counts and the stop test.
extern "C" int or_cluster_list_seq(const or_index *ix, const float *logit, const uint32_t *codes,
                                   const float *score, int nprobe, int C, const or_params *p,
                                   int32_t *L, float *dL, int32_t *n_dir, int32_t *n_batches,
                                   int64_t *n_scored) {
  const int b = ix->b;
  const uint64_t nbuckets = (uint64_t)1 << b;
  const int nbins = p->n_bins > 1 ? p->n_bins : 1;
  const bool binned = nbins > 1 && p->s_max < kInf;
  auto bin_of = [&](float s) {
    if (!binned) return 0;
    const float z = (s * (float)nbins) / p->s_max;  // Bin(s; N_bins, S_max)
    const int zi = (int)z;
    return zi < nbins - 1 ? zi : nbins - 1;
  };
  const bool gate_off = gate_is_off(p);
  const int B = p->b_batch > 0 ? p->b_batch : 1;
  std::vector<std::pair<float, int64_t>> dir, H;
  float dmin = kInf;
  int b_proc = 0, t_low = 0, batches = 0;
  int64_t batch_clusters = 0;  // clusters of the batches processed
  bool stop = false;
  int i = 0;
  while (i < nprobe && !stop) {
    const int z = bin_of(score[i]);
    int j = i;
    while (j < nprobe && bin_of(score[j]) == z) ++j;  // the bin: probes [i, j)
    b_proc += 1;
    std::vector<int64_t> cz;  // MapBucketsToClusters
    for (int t = i; t < j; ++t) {
      const uint64_t u = codes[t];
      if (u >= nbuckets) return -1;
      const uint32_t c0 = ix->bkt_off[u], c1 = ix->bkt_off[u + 1];
      if (c1 < c0 || (int64_t)c1 > ix->n_cl) return -1;
      if (c1 - c0 == 1) {
        dir.push_back({centroid_distance(logit, &ix->cent[(size_t)c0 * b], b), (int64_t)c0});
      } else {
        for (uint32_t c = c0; c < c1; ++c) cz.push_back((int64_t)c);
      }
    }
    for (size_t s0 = 0; s0 < cz.size() && !stop; s0 += (size_t)B) {
      const size_t s1 = std::min(cz.size(), s0 + (size_t)B);
      std::vector<std::pair<float, int64_t>> batch;
      for (size_t t = s0; t < s1; ++t)
        batch.push_back({centroid_distance(logit, &ix->cent[(size_t)cz[t] * b], b), cz[t]});
      batch_clusters += (int64_t)batch.size();
      for (auto &e : batch) dmin = std::min(dmin, e.first);
      float theta = kInf, front_th = kInf;
      if (!gate_off) {
        const float m = gate_margin(p, dmin);  // M(d_min)
        theta = dmin + m;
        front_th = dmin + p->c_alpha_front * m;
      }
      // KeepTopKUnderGate: the C smallest of H U batch within the gate
      std::vector<std::pair<float, int64_t>> all;
      for (auto &e : H)
        if (e.first <= theta) all.push_back(e);
      for (auto &e : batch)
        if (e.first <= theta) all.push_back(e);
      std::sort(all.begin(), all.end(), dc_less);
      if ((int)all.size() > C) all.resize((size_t)C);
      int updates = 0, front = 0;
      for (auto &e : batch)
        for (auto &h : all)
          if (h == e) {
            updates += 1;
            if (e.first <= front_th) front += 1;
          }
      H.swap(all);
      batches += 1;
      const bool lowq = updates < p->c_u_min && front < p->c_f_min;
      t_low = lowq ? t_low + 1 : 0;
      if (p->c_t_low > 0 && (int)H.size() == C && b_proc >= p->b_min && t_low >= p->c_t_low)
        stop = true;
    }
    i = j;
  }
  std::vector<std::pair<float, int64_t>> out(dir);
  out.insert(out.end(), H.begin(), H.end());
  std::sort(out.begin(), out.end(), dc_less);
  for (size_t t = 0; t < out.size(); ++t) {
    L[t] = (int32_t)out[t].second;
    if (dL) dL[t] = out[t].first;
  }
  if (n_dir) *n_dir = (int32_t)dir.size();
  if (n_batches) *n_batches = batches;
  // distances evaluated: C^dir of every bin entered, and the batches processed
  if (n_scored) *n_scored = (int64_t)dir.size() + batch_clusters;
  return (int)out.size();
}

// ---------------------------------------------------------------- refinement
// Exact squared L2 in the original space (uint8 kept as integers, Sec. 4.1.1),
// top-k by (dist, id), candidates processed in rounds of R with the
// heap-quality stop rule of Algorithm 2 (T_low consecutive low-quality rounds).
struct Hit {
  uint32_t dkey;  // u8: the int32 distance; f32: the float's bits (non-negative)
  float dist;
  int64_t id;
  bool operator<(const Hit &o) const { return dkey < o.dkey || (dkey == o.dkey && id < o.id); }
  bool operator==(const Hit &o) const { return dkey == o.dkey && id == o.id; }
};

static Hit score_row(int dtype, int D, const void *q, const void *row, int64_t id) {
  Hit h;
  h.id = id;
  if (dtype == 0) {
    const uint8_t *a = (const uint8_t *)q, *x = (const uint8_t *)row;
    int32_t acc = 0;
    for (int j = 0; j < D; ++j) {
      int32_t t = (int32_t)x[j] - (int32_t)a[j];
      acc += t * t;
    }
    h.dkey = (uint32_t)acc;
    h.dist = (float)acc;
  } else {
    const float *a = (const float *)q, *x = (const float *)row;
    float acc = 0.0f;
    for (int j = 0; j < D; ++j) {
      float t = x[j] - a[j];
      acc = std::fmaf(t, t, acc);
    }
    h.dist = acc;
    memcpy(&h.dkey, &acc, 4);
  }
  return h;
}

static void topk_insert(std::vector<Hit> &H, const Hit &h, int k) {
  auto pos = std::lower_bound(H.begin(), H.end(), h);
  if ((int)H.size() < k) {
    H.insert(pos, h);
  } else if (pos != H.end()) {
    H.insert(pos, h);
    H.pop_back();
  }
}

static int front_slots(float alpha, int k) {
  double f = std::ceil((double)alpha * (double)k);
  if (f < 0.0) f = 0.0;
  if (f > (double)k) f = (double)k;
  return (int)f;
}

// Rows are produced by a callback so that or_search can walk clusters in place.
static void refine_rounds(int dtype, int D, const void *q, int64_t n,
                          const std::function<std::pair<const void *, int64_t>(int64_t)> &row_at,
                          int k, const or_params *p, int64_t *out_ids, float *out_d,
                          int64_t *stats) {
  const int R = p->round_size > 0 ? p->round_size : 256;
  const int nfront = front_slots(p->alpha_front, k);
  std::vector<Hit> H;
  int64_t scored = 0, rounds = 0;
  int low = 0;
  for (int64_t start = 0; start < n; start += R) {
    const int64_t end = std::min<int64_t>(n, start + R);
    std::vector<Hit> before(H);
    for (int64_t s = start; s < end; ++s) {
      auto rw = row_at(s);
      topk_insert(H, score_row(dtype, D, q, rw.first, rw.second), k);
    }
    scored += end - start;
    rounds += 1;
    // updates of this round: members of H after the round not in H before it
    std::set<std::pair<uint32_t, int64_t>> old;
    for (auto &h : before) old.insert({h.dkey, h.id});
    int newc = 0, frontc = 0;
    for (int i = 0; i < (int)H.size(); ++i) {
      if (old.count({H[i].dkey, H[i].id})) continue;
      newc += 1;
      if (i < nfront) frontc += 1;
    }
    const bool lowq = newc < p->u_min && frontc < p->f_min;
    low = lowq ? low + 1 : 0;
    if (p->t_low > 0 && (int)H.size() == k && rounds >= p->r_min && low >= p->t_low) break;
  }
  for (int i = 0; i < k; ++i) {
    if (i < (int)H.size()) {
      out_ids[i] = H[i].id;
      out_d[i] = H[i].dist;
    } else {
      out_ids[i] = -1;
      out_d[i] = kInf;
    }
  }
  if (stats) {
    stats[0] = scored;
    stats[1] = rounds;
  }
}

extern "C" void or_refine_stream(int dtype, int D, const void *q, const void *rows,
                                 const uint32_t *ids, int64_t n, int k, const or_params *p,
                                 int64_t *out_ids, float *out_d, int64_t *stats) {
  const size_t rb = (size_t)D * (dtype == 0 ? 1 : 4);
  refine_rounds(
      dtype, D, q, n,
      [&](int64_t s) {
        return std::make_pair((const void *)((const uint8_t *)rows + (size_t)s * rb),
                              (int64_t)ids[s]);
      },
      k, p, out_ids, out_d, stats);
}

// ---------------------------------------------------------------- whole search
extern "C" int or_search(const or_index *ix, const void *queries, const float *logits, int64_t nq,
                         int k, int P, int C, const or_params *p, int64_t *out_ids, float *out_d,
                         int64_t *stats, int nthreads) {
  const int b = ix->b, D = ix->D;
  const size_t esz = ix->dtype == 0 ? 1 : 4, rb = (size_t)D * esz;
  std::atomic_int bad{0};
  parallel_for(nq, nthreads, [&](int64_t qi) {
    const void *q = (const uint8_t *)queries + (size_t)qi * rb;
    std::vector<float> lg(b);
    if (logits)
      for (int j = 0; j < b; ++j) lg[j] = logits[(size_t)qi * b + j];
    else
      encode_one(ix, queries, qi, lg.data());
    std::vector<uint32_t> codes((size_t)P);
    std::vector<uint64_t> keys((size_t)P);
    int np = or_probe_list_index(ix, lg.data(), P, p, codes.data(), keys.data());
    std::vector<int32_t> L((size_t)np + (size_t)C);
    int nl;
    int64_t scored = 0;
    if (p->cent_mode == 1) {
      std::vector<float> score((size_t)np);  // summed deviation of each probe's flip set
      for (int t = 0; t < np; ++t) {
        const uint32_t cb = (uint32_t)(keys[t] >> 32);
        memcpy(&score[t], &cb, 4);
      }
      nl = or_cluster_list_seq(ix, lg.data(), codes.data(), score.data(), np, C, p, L.data(),
                               nullptr, nullptr, nullptr, &scored);
    } else {
      nl = or_cluster_list(ix, lg.data(), codes.data(), np, C, p, L.data(), nullptr, nullptr,
                           &scored);
    }
    if (nl < 0) {
      bad = 1;
      nl = 0;
    }
    // candidate stream: rows of the clusters of L, in L's order
    std::vector<int64_t> seg_start, seg_len;
    int64_t n = 0;
    for (int i = 0; i < nl; ++i) {
      uint32_t r0 = ix->cl_off[(size_t)L[i]], r1 = ix->cl_off[(size_t)L[i] + 1];
      if (r1 < r0 || (int64_t)r1 > ix->N) {
        bad = 1;
        continue;
      }
      seg_start.push_back(r0);
      seg_len.push_back((int64_t)r1 - r0);
      n += (int64_t)r1 - r0;
    }
    size_t seg = 0;
    int64_t seg_base = 0;
    auto row_at = [&](int64_t s) {
      while (s - seg_base >= seg_len[seg]) {
        seg_base += seg_len[seg];
        seg += 1;
      }
      int64_t r = seg_start[seg] + (s - seg_base);
      return std::make_pair((const void *)(ix->vec.data() + (size_t)r * rb), (int64_t)ix->ids[(size_t)r]);
    };
    int64_t st[2] = {0, 0};
    refine_rounds(ix->dtype, D, q, n, row_at, k, p, out_ids + (size_t)qi * k, out_d + (size_t)qi * k, st);
    if (stats) {
      int64_t *row = stats + (size_t)qi * 5;
      row[0] = st[0];
      row[1] = st[1];
      row[2] = nl;
      row[3] = np;
      row[4] = scored;
    }
  });
  return bad ? -1 : 0;
}

// ---------------------------------------------------------------- exact k-NN
// Sec. 3.1: the k base vectors nearest in Euclidean distance (squared L2 has
// the same order), ties by id.
extern "C" void or_bruteforce(int dtype, int D, const void *base, int64_t N, const void *queries,
                              int64_t nq, int k, int64_t *out_ids, float *out_d, int nthreads) {
  const size_t rb = (size_t)D * (dtype == 0 ? 1 : 4);
  parallel_for(nq, nthreads, [&](int64_t qi) {
    const void *q = (const uint8_t *)queries + (size_t)qi * rb;
    std::vector<Hit> H;
    for (int64_t i = 0; i < N; ++i)
      topk_insert(H, score_row(dtype, D, q, (const uint8_t *)base + (size_t)i * rb, i), k);
    for (int i = 0; i < k; ++i) {
      out_ids[(size_t)qi * k + i] = i < (int)H.size() ? H[i].id : -1;
      out_d[(size_t)qi * k + i] = i < (int)H.size() ? H[i].dist : kInf;
    }
  });
}
