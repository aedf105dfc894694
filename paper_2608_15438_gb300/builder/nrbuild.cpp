// NeuRoute index builder: a plain host routine run once, off the query path.
//
// Paper Sec. 3.3 (Index Construction) and Sec. 3.2.3 (Binarization):
//   1. encode every base vector with the encoder, l_i = E(x_i);
//   2. per-bit threshold tau_j = median of column j (lower median, exact, in
//      the total order of the fp32 bit patterns);
//   3. code u_i with bit j = [l_ij >= tau_j]; bucket = code;
//   4. per non-empty bucket B, K_B = min(K_max, ceil(|B| / t)) clusters found by
//      k-means++ seeding on a sample and a few Lloyd passes on the whole bucket,
//      in logit space; buckets with K_B = 1 stay a single cluster;
//   5. rows stored in (code, local label, id) order with two CSR levels:
//      bkt_off[code] -> cluster range, cl_off[cluster] -> row range.
// The file it writes is the input of the query path (format in neuroute.h).
//
// Host-only C++, threads over rows and buckets. It is deterministic for a
// given seed and thread count does not change the result. Given the same
// logits (nrb_build_logits), the library's GPU builder writes the same bytes.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstdio>
#include <cstring>
#include <functional>
#include <thread>
#include <vector>

extern "C" {
typedef struct {
  int dtype;        // 0 = uint8 vectors, 1 = fp32 vectors
  int D, H, b;      // input dim, hidden width, code bits (1..24)
  int K_max;        // max clusters per bucket
  int t;            // target cluster capacity
  float in_scale;   // encoder input scale (1/255 for uint8)
  int lloyd_iters;  // Lloyd passes on the whole bucket
  int sample_per_cluster;  // k-means++ sample size per cluster
  uint64_t seed;    // k-means seed
  int n_mid;        // hidden layers after the first (0..7)
  int mid_w[7];     // their widths; the last layer maps the last hidden width to b
} nrb_config;
}

namespace {

void parallel_for(int64_t n, int nthreads, const std::function<void(int64_t)> &fn) {
  if (nthreads <= 1 || n <= 1) {
    for (int64_t i = 0; i < n; ++i) fn(i);
    return;
  }
  std::vector<std::thread> th;
  std::atomic<int64_t> next{0};
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

uint64_t splitmix64(uint64_t &s) {
  uint64_t z = (s += 0x9E3779B97F4A7C15ull);
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Widths of the hidden layers: H, then the middle layers'.
int hidden_last(const nrb_config &c) { return c.n_mid > 0 ? c.mid_w[c.n_mid - 1] : c.H; }
size_t mid_floats(const nrb_config &c) {
  size_t n = 0;
  for (int i = 0, prev = c.H; i < c.n_mid; prev = c.mid_w[i], ++i) n += (size_t)c.mid_w[i] * prev + c.mid_w[i];
  return n;
}

// Encoder forward over rows [r0, r0 + n): blocks of 16 rows so the inner loop
// runs over independent accumulators. Hidden layers linear then ReLU, the
// last linear; Wm holds each middle layer's W [w x previous] then its bias.
void encode_block(const nrb_config &c, const void *x, int64_t r0, int n, const float *W1,
                  const float *b1, const float *W2, const float *b2, const float *Wm, float *out) {
  constexpr int BR = 16;
  const int D = c.D, B = c.b;
  int H = c.H;
  std::vector<float> xt((size_t)D * BR, 0.0f), h((size_t)H * BR, 0.0f);
  for (int r = 0; r < n; ++r)
    for (int j = 0; j < D; ++j) {
      float v = c.dtype == 0 ? (float)((const uint8_t *)x)[(size_t)(r0 + r) * D + j]
                             : ((const float *)x)[(size_t)(r0 + r) * D + j];
      xt[(size_t)j * BR + r] = v * c.in_scale;
    }
  for (int u = 0; u < H; ++u) {
    float acc[BR];
    for (int r = 0; r < BR; ++r) acc[r] = b1[u];
    const float *w = W1 + (size_t)u * D;
    for (int j = 0; j < D; ++j) {
      const float wj = w[j];
      const float *xr = &xt[(size_t)j * BR];
      for (int r = 0; r < BR; ++r) acc[r] += wj * xr[r];
    }
    for (int r = 0; r < BR; ++r) h[(size_t)u * BR + r] = acc[r] > 0.0f ? acc[r] : 0.0f;
  }
  const float *wl = Wm;
  for (int l = 0; l < c.n_mid; ++l) {
    const int w = c.mid_w[l];
    const float *bias = wl + (size_t)w * H;
    std::vector<float> g((size_t)w * BR, 0.0f);
    for (int u = 0; u < w; ++u) {
      float acc[BR];
      for (int r = 0; r < BR; ++r) acc[r] = bias[u];
      const float *wr = wl + (size_t)u * H;
      for (int j = 0; j < H; ++j) {
        const float wj = wr[j];
        const float *hr = &h[(size_t)j * BR];
        for (int r = 0; r < BR; ++r) acc[r] += wj * hr[r];
      }
      for (int r = 0; r < BR; ++r) g[(size_t)u * BR + r] = acc[r] > 0.0f ? acc[r] : 0.0f;
    }
    wl = bias + w;
    h.swap(g);
    H = w;
  }
  for (int o = 0; o < B; ++o) {
    float acc[BR];
    for (int r = 0; r < BR; ++r) acc[r] = b2[o];
    const float *w = W2 + (size_t)o * H;
    for (int u = 0; u < H; ++u) {
      const float wu = w[u];
      const float *hr = &h[(size_t)u * BR];
      for (int r = 0; r < BR; ++r) acc[r] += wu * hr[r];
    }
    for (int r = 0; r < n; ++r) out[(size_t)r * B + o] = acc[r];
  }
}

// ---------------------------------------------------------------------------
// Arithmetic of the build, fixed so that a parallel implementation reproduces
// it bit for bit (the library's GPU builder follows the same definition):
//  * distances in logit space are fp32 with every product and sum rounded
//    (t = a_j - c_j, s = s + t*t over j ascending from s = 0, no fused
//    multiply-add);
//  * a centroid is the mean of its members' logits, summed exactly as
//    integers in fixed point (x * 2^G rounded to nearest, G = 30 - e with
//    max |logit| = f 2^e, f in [0.5, 1)), then ((double)sum * 2^-G) / count
//    rounded to fp32 -- the order of the additions cannot change it;
//  * the k-means++ sample is every (n/m)-th member of the bucket (positions
//    floor(i n / m), members in id order), and the D^2-weighted draw uses
//    integer weights trunc(dmin_i * 2^F), F = 50 - e(max dmin), so the prefix
//    sums are exact.
// ---------------------------------------------------------------------------

// e with v = f * 2^e, f in [0.5, 1), for a positive finite double
int exponent_of(double v) {
  uint64_t bits;
  memcpy(&bits, &v, 8);
  return (int)((bits >> 52) & 0x7FF) - 1022;
}
double pow2(int e) {
  const uint64_t bits = (uint64_t)(e + 1023) << 52;
  double v;
  memcpy(&v, &bits, 8);
  return v;
}
uint64_t mulhi64(uint64_t a, uint64_t b) {
  return (uint64_t)(((unsigned __int128)a * (unsigned __int128)b) >> 64);
}

// order-preserving map of fp32 bit patterns to uint32 (total order, -0 < +0)
uint32_t float_key(float x) {
  uint32_t u;
  memcpy(&u, &x, 4);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
float key_float(uint32_t k) {
  const uint32_t u = (k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k;
  float x;
  memcpy(&x, &u, 4);
  return x;
}

float sqdist_f(const float *a, const float *c, int b) {
  float s = 0.0f;
  for (int j = 0; j < b; ++j) {
    const float t = a[j] - c[j];
    const float p = t * t;
    s = s + p;
  }
  return s;
}

struct Fixed {
  double scale, inv_scale;
};

// Fixed-point means of the labelled members; clusters without members keep
// their centroid. cnt[k] = members of cluster k.
void update_means(const float *logits, const uint32_t *rows, int64_t n, const uint8_t *lab, int K,
                  int b, const Fixed &fx, float *cent, std::vector<int64_t> &cnt) {
  std::vector<int64_t> sum((size_t)K * b, 0);
  cnt.assign((size_t)K, 0);
  for (int64_t i = 0; i < n; ++i) {
    const float *l = &logits[(size_t)rows[i] * b];
    const int k = lab[i];
    cnt[k] += 1;
    for (int j = 0; j < b; ++j) sum[(size_t)k * b + j] += llrint((double)l[j] * fx.scale);
  }
  for (int k = 0; k < K; ++k)
    if (cnt[k] > 0)
      for (int j = 0; j < b; ++j)
        cent[(size_t)k * b + j] =
            (float)(((double)sum[(size_t)k * b + j] * fx.inv_scale) / (double)cnt[k]);
}

// k-means in logit space for one bucket. rows: member ids, ascending.
// On return labels[i] in [0, kk) and cent_out / cnt_out hold the kk non-empty
// clusters in label order.
int cluster_bucket(const nrb_config &c, const float *logits, const uint32_t *rows, int64_t n,
                   uint32_t code, const Fixed &fx, std::vector<uint8_t> &labels,
                   std::vector<float> &cent_out, std::vector<int64_t> &cnt_out) {
  const int b = c.b;
  labels.assign((size_t)n, 0);
  int64_t K = (n + c.t - 1) / c.t;
  if (K > c.K_max) K = c.K_max;
  if (K > n) K = n;
  if (K < 1) K = 1;
  std::vector<float> cent((size_t)K * b, 0.0f);
  std::vector<int64_t> cnt;
  if (K > 1) {
    uint64_t s = c.seed * 0x100000001B3ull ^ ((uint64_t)code * 0x9E3779B97F4A7C15ull);
    const int64_t m = std::min<int64_t>(n, (int64_t)c.sample_per_cluster * K);
    auto sample = [&](int64_t i) {
      return &logits[(size_t)rows[(uint64_t)i * (uint64_t)n / (uint64_t)m] * b];
    };
    auto uniform_pick = [&](uint64_t draw) {
      int64_t p = (int64_t)((double)(draw >> 11) * (1.0 / 9007199254740992.0) * (double)m);
      return p < m ? p : m - 1;
    };
    memcpy(&cent[0], sample(uniform_pick(splitmix64(s))), sizeof(float) * b);
    std::vector<float> dmin((size_t)m, INFINITY);
    std::vector<uint64_t> w((size_t)m);
    for (int64_t k = 1; k < K; ++k) {
      float mx = 0.0f;
      for (int64_t i = 0; i < m; ++i) {
        const float d = sqdist_f(sample(i), &cent[(size_t)(k - 1) * b], b);
        if (d < dmin[i]) dmin[i] = d;
        if (dmin[i] > mx) mx = dmin[i];
      }
      const uint64_t draw = splitmix64(s);
      int64_t pick = -1;
      if (mx > 0.0f) {
        const double mult = pow2(50 - exponent_of((double)mx));
        uint64_t tot = 0;
        for (int64_t i = 0; i < m; ++i) {
          w[i] = (uint64_t)((double)dmin[i] * mult);
          tot += w[i];
        }
        if (tot > 0) {
          const uint64_t r = mulhi64(draw, tot);
          uint64_t acc = 0;
          for (int64_t i = 0; i < m; ++i) {
            acc += w[i];
            if (acc > r) {
              pick = i;
              break;
            }
          }
        }
      }
      if (pick < 0) pick = uniform_pick(draw);
      memcpy(&cent[(size_t)k * b], sample(pick), sizeof(float) * b);
    }
    // Lloyd passes on the whole bucket: assign (ties to the lower index), update
    const int iters = c.lloyd_iters > 0 ? c.lloyd_iters : 1;
    for (int it = 0; it < iters; ++it) {
      for (int64_t i = 0; i < n; ++i) {
        const float *l = &logits[(size_t)rows[i] * b];
        int best = 0;
        float bd = sqdist_f(l, &cent[0], b);
        for (int k = 1; k < K; ++k) {
          const float d = sqdist_f(l, &cent[(size_t)k * b], b);
          if (d < bd) {
            bd = d;
            best = k;
          }
        }
        labels[i] = (uint8_t)best;
      }
      update_means(logits, rows, n, labels.data(), (int)K, b, fx, cent.data(), cnt);
    }
  } else {
    update_means(logits, rows, n, labels.data(), 1, b, fx, cent.data(), cnt);
  }
  // drop empty clusters, renumber in label order
  std::vector<int> remap((size_t)K, -1);
  int kk = 0;
  for (int k = 0; k < K; ++k)
    if (cnt[k] > 0) remap[k] = kk++;
  cent_out.resize((size_t)kk * b);
  cnt_out.resize((size_t)kk);
  for (int k = 0; k < K; ++k)
    if (remap[k] >= 0) {
      memcpy(&cent_out[(size_t)remap[k] * b], &cent[(size_t)k * b], sizeof(float) * b);
      cnt_out[remap[k]] = cnt[k];
    }
  for (int64_t i = 0; i < n; ++i) labels[i] = (uint8_t)remap[labels[i]];
  return kk;
}

bool write_all(FILE *f, const void *p, size_t bytes) {
  return bytes == 0 || fwrite(p, 1, bytes, f) == bytes;
}

}  // namespace

extern "C" {

// Encode n rows with the builder's encoder (fp32). out: [n x b].
int nrb_encode(const nrb_config *c, const void *x, int64_t n, const float *W1, const float *b1,
               const float *W2, const float *b2, const float *Wm, float *out, int nthreads) {
  if (!c || !x || !out || n < 0 || c->n_mid < 0 || c->n_mid > 7 || (c->n_mid > 0 && !Wm)) return -1;
  const int64_t nblk = (n + 15) / 16;
  parallel_for(nblk, nthreads, [&](int64_t blk) {
    int64_t r0 = blk * 16;
    int cnt = (int)std::min<int64_t>(16, n - r0);
    encode_block(*c, x, r0, cnt, W1, b1, W2, b2, Wm, out + (size_t)r0 * c->b);
  });
  return 0;
}

// Build the index over base x [N x D] from the base's logits [N x b] and
// write it to path. Returns 0, -1 bad argument (including non-finite
// logits), -2 I/O error.
int nrb_build_logits(const nrb_config *c, const void *x, int64_t N, const float *logits_in,
                     const float *W1, const float *b1, const float *W2, const float *b2,
                     const float *Wm, const char *path, int nthreads, int64_t *info_out) {
  if (!c || !x || !logits_in || !path || N < 1 || N >= (int64_t)0xFFFFFFFFll || c->b < 1 ||
      c->b > 24 || c->D < 1 || c->H < 1 || c->K_max < 1 || c->K_max > 64 || c->t < 1 ||
      c->sample_per_cluster < 1 || (c->dtype != 0 && c->dtype != 1) || c->n_mid < 0 ||
      c->n_mid > 7 || (c->n_mid > 0 && !Wm))
    return -1;
  for (int i = 0; i < c->n_mid; ++i)
    if (c->mid_w[i] < 1) return -1;
  const int b = c->b, D = c->D;
  const size_t esz = c->dtype == 0 ? 1 : 4;
  const float *logits = logits_in;
  // fixed-point scale of the centroid sums from the largest |logit|
  uint32_t amax = 0;
  for (int64_t i = 0; i < N * b; ++i) {
    uint32_t u;
    memcpy(&u, &logits[i], 4);
    u &= 0x7FFFFFFFu;
    if (u > amax) amax = u;
  }
  if (amax >= 0x7F800000u) return -1;
  Fixed fx;
  {
    float am;
    memcpy(&am, &amax, 4);
    const int G = 30 - (am > 0.0f ? exponent_of((double)am) : 0);
    fx.scale = pow2(G);
    fx.inv_scale = pow2(-G);
  }
  // 2. per-bit lower median (rank floor((N-1)/2) in the total order of the
  // fp32 bit patterns)
  std::vector<float> tau((size_t)b);
  parallel_for(b, nthreads, [&](int64_t j) {
    std::vector<uint32_t> col((size_t)N);
    for (int64_t i = 0; i < N; ++i) col[i] = float_key(logits[(size_t)i * b + j]);
    size_t mid = (size_t)((N - 1) / 2);
    std::nth_element(col.begin(), col.begin() + mid, col.end());
    tau[j] = key_float(col[mid]);
  });
  // 3. codes and a stable counting sort of ids by code
  const size_t nb = (size_t)1 << b;
  std::vector<uint32_t> code((size_t)N);
  parallel_for((N + 65535) / 65536, nthreads, [&](int64_t blk) {
    int64_t lo = blk * 65536, hi = std::min<int64_t>(N, lo + 65536);
    for (int64_t i = lo; i < hi; ++i) {
      uint32_t u = 0;
      for (int j = 0; j < b; ++j)
        if (logits[(size_t)i * b + j] >= tau[j]) u |= 1u << j;
      code[i] = u;
    }
  });
  std::vector<int64_t> bstart(nb + 1, 0);
  for (int64_t i = 0; i < N; ++i) bstart[code[i] + 1] += 1;
  for (size_t u = 0; u < nb; ++u) bstart[u + 1] += bstart[u];
  std::vector<uint32_t> order((size_t)N);
  {
    std::vector<int64_t> fill(bstart.begin(), bstart.end() - 1);
    for (int64_t i = 0; i < N; ++i) order[fill[code[i]]++] = (uint32_t)i;
  }
  std::vector<uint32_t>().swap(code);
  // 4. bucket-local clustering
  std::vector<uint32_t> nonempty;
  for (size_t u = 0; u < nb; ++u)
    if (bstart[u + 1] > bstart[u]) nonempty.push_back((uint32_t)u);
  std::vector<std::vector<float>> bcent(nonempty.size());
  std::vector<std::vector<int64_t>> bcnt(nonempty.size());
  std::vector<int> ncl(nonempty.size());
  // largest buckets first for load balance
  std::vector<int64_t> sched(nonempty.size());
  for (size_t i = 0; i < sched.size(); ++i) sched[i] = (int64_t)i;
  std::sort(sched.begin(), sched.end(), [&](int64_t a, int64_t z) {
    int64_t na = bstart[nonempty[a] + 1] - bstart[nonempty[a]];
    int64_t nz = bstart[nonempty[z] + 1] - bstart[nonempty[z]];
    return na > nz || (na == nz && a < z);
  });
  parallel_for((int64_t)nonempty.size(), nthreads, [&](int64_t si) {
    int64_t i = sched[si];
    uint32_t u = nonempty[i];
    int64_t lo = bstart[u], n = bstart[u + 1] - lo;
    std::vector<uint8_t> lab;
    ncl[i] = cluster_bucket(*c, logits, &order[lo], n, u, fx, lab, bcent[i], bcnt[i]);
    // rows in (label, id) order inside the bucket: stable counting sort
    std::vector<int64_t> pos((size_t)ncl[i] + 1, 0);
    for (int k = 0; k < ncl[i]; ++k) pos[k + 1] = pos[k] + bcnt[i][k];
    std::vector<uint32_t> tmp((size_t)n);
    for (int64_t r = 0; r < n; ++r) tmp[pos[lab[r]]++] = order[lo + r];
    memcpy(&order[lo], tmp.data(), sizeof(uint32_t) * (size_t)n);
  });
  // 5. two CSR levels
  int64_t n_cl = 0;
  for (int k : ncl) n_cl += k;
  std::vector<uint32_t> bkt_off(nb + 1, 0), cl_off((size_t)n_cl + 1, 0);
  std::vector<float> cent((size_t)n_cl * b);
  {
    size_t e = 0;
    int64_t cidx = 0;
    for (size_t u = 0; u < nb; ++u) {
      bkt_off[u] = (uint32_t)cidx;
      if (e < nonempty.size() && nonempty[e] == u) {
        int64_t r = bstart[u];
        for (int k = 0; k < ncl[e]; ++k) {
          cl_off[cidx + k] = (uint32_t)r;
          r += bcnt[e][k];
          memcpy(&cent[(size_t)(cidx + k) * b], &bcent[e][(size_t)k * b], sizeof(float) * b);
        }
        cidx += ncl[e];
        ++e;
      }
    }
    bkt_off[nb] = (uint32_t)cidx;
    cl_off[n_cl] = (uint32_t)N;
  }
  const std::vector<uint32_t> &ids = order;
  // 6. write
  FILE *f = fopen(path, "wb");
  if (!f) return -2;
  auto align = [](uint64_t v) { return (v + 255) & ~(uint64_t)255; };
  const int hl = hidden_last(*c);
  uint64_t sz[10] = {(uint64_t)c->H * D * 4,  (uint64_t)c->H * 4, (uint64_t)b * hl * 4,
                     (uint64_t)b * 4,         (uint64_t)b * 4,    (uint64_t)(nb + 1) * 4,
                     (uint64_t)(n_cl + 1) * 4, (uint64_t)n_cl * b * 4, (uint64_t)N * 4,
                     (uint64_t)N * D * esz};
  uint64_t off[10];
  uint64_t cur = 256;
  for (int i = 0; i < 10; ++i) {
    off[i] = cur;
    cur = align(cur + sz[i]);
  }
  // the middle hidden layers (version 2): one more section after the vectors
  const uint64_t mid_sz = (uint64_t)mid_floats(*c) * 4, mid_off = c->n_mid > 0 ? cur : 0;
  if (c->n_mid > 0) cur = align(cur + mid_sz);
  unsigned char h[256];
  memset(h, 0, sizeof(h));
  memcpy(h, "NRIXv001", 8);
  uint32_t u32;
  uint64_t u64;
  u32 = c->n_mid > 0 ? 2 : 1; memcpy(h + 8, &u32, 4);
  u32 = (uint32_t)c->dtype; memcpy(h + 12, &u32, 4);
  u64 = (uint64_t)N; memcpy(h + 16, &u64, 8);
  u32 = (uint32_t)D; memcpy(h + 24, &u32, 4);
  u32 = (uint32_t)c->H; memcpy(h + 28, &u32, 4);
  u32 = (uint32_t)b; memcpy(h + 32, &u32, 4);
  u32 = (uint32_t)c->K_max; memcpy(h + 36, &u32, 4);
  u32 = (uint32_t)c->t; memcpy(h + 40, &u32, 4);
  u64 = (uint64_t)n_cl; memcpy(h + 48, &u64, 8);
  memcpy(h + 56, &c->in_scale, 4);
  for (int i = 0; i < 10; ++i) memcpy(h + 64 + 8 * i, &off[i], 8);
  memcpy(h + 144, &cur, 8);
  if (c->n_mid > 0) {
    u32 = (uint32_t)c->n_mid; memcpy(h + 152, &u32, 4);
    for (int i = 0; i < c->n_mid; ++i) {
      u32 = (uint32_t)c->mid_w[i];
      memcpy(h + 156 + 4 * i, &u32, 4);
    }
    memcpy(h + 192, &mid_off, 8);
  }
  bool ok = write_all(f, h, 256);
  const void *secs[9] = {W1, b1, W2, b2, tau.data(), bkt_off.data(), cl_off.data(), cent.data(), ids.data()};
  static const unsigned char zeros[256] = {0};
  uint64_t at = 256;
  for (int i = 0; i < 10 && ok; ++i) {
    ok = ok && write_all(f, zeros, (size_t)(off[i] - at));
    at = off[i];
    if (i < 9) {
      ok = ok && write_all(f, secs[i], (size_t)sz[i]);
    } else {
      // vectors in stored-row order, streamed in chunks
      const size_t rb = (size_t)D * esz;
      std::vector<uint8_t> buf;
      const int64_t CH = 65536;
      for (int64_t r0 = 0; r0 < N && ok; r0 += CH) {
        int64_t r1 = std::min<int64_t>(N, r0 + CH);
        buf.resize((size_t)(r1 - r0) * rb);
        for (int64_t r = r0; r < r1; ++r)
          memcpy(&buf[(size_t)(r - r0) * rb], (const uint8_t *)x + (size_t)ids[r] * rb, rb);
        ok = write_all(f, buf.data(), buf.size());
      }
    }
    at += sz[i];
  }
  if (c->n_mid > 0) {
    ok = ok && write_all(f, zeros, (size_t)(mid_off - at));
    ok = ok && write_all(f, Wm, (size_t)mid_sz);
    at = mid_off + mid_sz;
  }
  ok = ok && write_all(f, zeros, (size_t)(cur - at));
  ok = (fclose(f) == 0) && ok;
  if (!ok) return -2;
  if (info_out) {
    int64_t maxb = 0, maxc = 0, nsingle = 0;
    for (size_t i = 0; i < nonempty.size(); ++i) {
      maxb = std::max<int64_t>(maxb, bstart[nonempty[i] + 1] - bstart[nonempty[i]]);
      if (ncl[i] == 1) nsingle += 1;
    }
    for (int64_t k = 0; k < n_cl; ++k) maxc = std::max<int64_t>(maxc, (int64_t)cl_off[k + 1] - cl_off[k]);
    info_out[0] = n_cl;
    info_out[1] = (int64_t)nonempty.size();
    info_out[2] = maxb;
    info_out[3] = maxc;
    info_out[4] = nsingle;
  }
  return 0;
}

// Build the index over base x [N x D] with the builder's fp32 encoder and
// write it to path (nrb_build_logits on the encoded base).
int nrb_build(const nrb_config *c, const void *x, int64_t N, const float *W1, const float *b1,
              const float *W2, const float *b2, const float *Wm, const char *path, int nthreads,
              int64_t *info_out) {
  if (!c || !x || N < 1 || N >= (int64_t)0xFFFFFFFFll || c->b < 1 || c->b > 24) return -1;
  std::vector<float> logits;
  try {
    logits.resize((size_t)N * c->b);
  } catch (...) {
    return -1;
  }
  if (nrb_encode(c, x, N, W1, b1, W2, b2, Wm, logits.data(), nthreads) != 0) return -1;
  return nrb_build_logits(c, x, N, logits.data(), W1, b1, W2, b2, Wm, path, nthreads, info_out);
}

}  // extern "C"
