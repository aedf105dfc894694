// NeuRoute index builder: a plain host routine run once, off the query path.
//
// Paper Sec. 3.3 (Index Construction) and Sec. 3.2.3 (Binarization):
//   1. encode every base vector with the encoder, l_i = E(x_i);
//   2. per-bit threshold tau_j = median of column j (lower median, exact);
//   3. code u_i with bit j = [l_ij >= tau_j]; bucket = code;
//   4. per non-empty bucket B, K_B = min(K_max, ceil(|B| / t)) clusters found by
//      k-means++ seeding on a sample and a few Lloyd passes on the whole bucket,
//      in logit space; buckets with K_B = 1 stay a single cluster;
//   5. rows stored in (code, local label, id) order with two CSR levels:
//      bkt_off[code] -> cluster range, cl_off[cluster] -> row range.
// The file it writes is the input of the query path (format in neuroute.h).
//
// Host-only C++, threads over rows and buckets. It is deterministic for a
// given seed and thread count does not change the result.
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
double unif(uint64_t &s) { return (double)(splitmix64(s) >> 11) * (1.0 / 9007199254740992.0); }

// Encoder forward over rows [r0, r0 + n): blocks of 16 rows so the inner loop
// runs over independent accumulators.
void encode_block(const nrb_config &c, const void *x, int64_t r0, int n, const float *W1,
                  const float *b1, const float *W2, const float *b2, float *out) {
  constexpr int BR = 16;
  const int D = c.D, H = c.H, B = c.b;
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

double sqdist(const float *a, const double *m, int b) {
  double s = 0.0;
  for (int j = 0; j < b; ++j) {
    double t = (double)a[j] - m[j];
    s += t * t;
  }
  return s;
}

// k-means in logit space for one bucket. rows: member row numbers (ascending
// id). Returns the number of (non-empty) clusters; labels[i] in [0, K).
int cluster_bucket(const nrb_config &c, const float *logits, const int64_t *rows, int64_t n,
                   uint32_t code, std::vector<int> &labels, std::vector<float> &cent_out) {
  const int b = c.b;
  labels.assign((size_t)n, 0);
  int64_t K = (n + c.t - 1) / c.t;
  if (K > c.K_max) K = c.K_max;
  if (K < 1) K = 1;
  if (K > n) K = n;
  std::vector<double> cent((size_t)K * b, 0.0);
  if (K == 1) {
    for (int64_t i = 0; i < n; ++i)
      for (int j = 0; j < b; ++j) cent[j] += logits[(size_t)rows[i] * b + j];
    cent_out.resize((size_t)b);
    for (int j = 0; j < b; ++j) cent_out[j] = (float)(cent[j] / (double)n);
    return 1;
  }
  uint64_t s = c.seed * 0x100000001B3ull ^ ((uint64_t)code * 0x9E3779B97F4A7C15ull);
  // sample without replacement (partial Fisher-Yates on member positions)
  int64_t m = std::min<int64_t>(n, (int64_t)c.sample_per_cluster * K);
  std::vector<int64_t> pos((size_t)n);
  for (int64_t i = 0; i < n; ++i) pos[i] = i;
  for (int64_t i = 0; i < m; ++i) {
    int64_t j = i + (int64_t)(unif(s) * (double)(n - i));
    if (j >= n) j = n - 1;
    std::swap(pos[i], pos[j]);
  }
  // k-means++ seeding on the sample
  std::vector<double> dmin((size_t)m, 1e300);
  int64_t first = (int64_t)(unif(s) * (double)m);
  if (first >= m) first = m - 1;
  for (int j = 0; j < b; ++j) cent[j] = logits[(size_t)rows[pos[first]] * b + j];
  for (int64_t k = 1; k < K; ++k) {
    double tot = 0.0;
    for (int64_t i = 0; i < m; ++i) {
      double d = sqdist(&logits[(size_t)rows[pos[i]] * b], &cent[(size_t)(k - 1) * b], b);
      if (d < dmin[i]) dmin[i] = d;
      tot += dmin[i];
    }
    int64_t pick = m - 1;
    if (tot > 0.0) {
      double r = unif(s) * tot, acc = 0.0;
      for (int64_t i = 0; i < m; ++i) {
        acc += dmin[i];
        if (acc > r) {
          pick = i;
          break;
        }
      }
    } else {
      pick = (int64_t)(unif(s) * (double)m);
      if (pick >= m) pick = m - 1;
    }
    for (int j = 0; j < b; ++j) cent[(size_t)k * b + j] = logits[(size_t)rows[pos[pick]] * b + j];
  }
  // Lloyd passes on the whole bucket: assign (ties to the lower index), update
  std::vector<double> sum((size_t)K * b);
  std::vector<int64_t> cnt((size_t)K);
  const int iters = c.lloyd_iters > 0 ? c.lloyd_iters : 1;
  for (int it = 0; it < iters; ++it) {
    for (int64_t i = 0; i < n; ++i) {
      const float *l = &logits[(size_t)rows[i] * b];
      int best = 0;
      double bd = sqdist(l, &cent[0], b);
      for (int k = 1; k < K; ++k) {
        double d = sqdist(l, &cent[(size_t)k * b], b);
        if (d < bd) {
          bd = d;
          best = k;
        }
      }
      labels[i] = best;
    }
    std::fill(sum.begin(), sum.end(), 0.0);
    std::fill(cnt.begin(), cnt.end(), 0);
    for (int64_t i = 0; i < n; ++i) {
      cnt[labels[i]] += 1;
      for (int j = 0; j < b; ++j) sum[(size_t)labels[i] * b + j] += logits[(size_t)rows[i] * b + j];
    }
    for (int k = 0; k < K; ++k)
      if (cnt[k] > 0)
        for (int j = 0; j < b; ++j) cent[(size_t)k * b + j] = sum[(size_t)k * b + j] / (double)cnt[k];
  }
  // drop empty clusters, renumber in label order
  std::vector<int> remap((size_t)K, -1);
  int kk = 0;
  for (int k = 0; k < K; ++k)
    if (cnt[k] > 0) remap[k] = kk++;
  cent_out.resize((size_t)kk * b);
  for (int k = 0; k < K; ++k)
    if (remap[k] >= 0)
      for (int j = 0; j < b; ++j) cent_out[(size_t)remap[k] * b + j] = (float)cent[(size_t)k * b + j];
  for (int64_t i = 0; i < n; ++i) labels[i] = remap[labels[i]];
  return kk;
}

bool write_all(FILE *f, const void *p, size_t bytes) {
  return bytes == 0 || fwrite(p, 1, bytes, f) == bytes;
}

}  // namespace

extern "C" {

// Encode n rows with the builder's encoder (fp32). out: [n x b].
int nrb_encode(const nrb_config *c, const void *x, int64_t n, const float *W1, const float *b1,
               const float *W2, const float *b2, float *out, int nthreads) {
  if (!c || !x || !out || n < 0) return -1;
  const int64_t nblk = (n + 15) / 16;
  parallel_for(nblk, nthreads, [&](int64_t blk) {
    int64_t r0 = blk * 16;
    int cnt = (int)std::min<int64_t>(16, n - r0);
    encode_block(*c, x, r0, cnt, W1, b1, W2, b2, out + (size_t)r0 * c->b);
  });
  return 0;
}

// Build the index over base x [N x D] and write it to path.
// Returns 0, -1 bad argument, -2 I/O error.
int nrb_build(const nrb_config *c, const void *x, int64_t N, const float *W1, const float *b1,
              const float *W2, const float *b2, const char *path, int nthreads, int64_t *info_out) {
  if (!c || !x || !path || N < 1 || N >= (int64_t)0xFFFFFFFFll || c->b < 1 || c->b > 24 ||
      c->D < 1 || c->H < 1 || c->K_max < 1 || c->t < 1 || (c->dtype != 0 && c->dtype != 1))
    return -1;
  const int b = c->b, D = c->D;
  const size_t esz = c->dtype == 0 ? 1 : 4;
  // 1. logits of the whole base
  std::vector<float> logits((size_t)N * b);
  nrb_encode(c, x, N, W1, b1, W2, b2, logits.data(), nthreads);
  // 2. per-bit lower median
  std::vector<float> tau((size_t)b);
  parallel_for(b, nthreads, [&](int64_t j) {
    std::vector<float> col((size_t)N);
    for (int64_t i = 0; i < N; ++i) col[i] = logits[(size_t)i * b + j];
    size_t mid = (size_t)((N - 1) / 2);
    std::nth_element(col.begin(), col.begin() + mid, col.end());
    tau[j] = col[mid];
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
  std::vector<int64_t> order((size_t)N);
  {
    std::vector<int64_t> fill(bstart.begin(), bstart.end() - 1);
    for (int64_t i = 0; i < N; ++i) order[fill[code[i]]++] = i;
  }
  std::vector<uint32_t>().swap(code);
  // 4. bucket-local clustering
  std::vector<uint32_t> nonempty;
  for (size_t u = 0; u < nb; ++u)
    if (bstart[u + 1] > bstart[u]) nonempty.push_back((uint32_t)u);
  std::vector<std::vector<float>> bcent(nonempty.size());
  std::vector<int> ncl(nonempty.size());
  std::vector<int> label((size_t)N);  // by position in `order`
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
    std::vector<int> lab;
    ncl[i] = cluster_bucket(*c, logits.data(), &order[lo], n, u, lab, bcent[i]);
    // rows in (label, id) order inside the bucket: stable counting sort
    std::vector<int64_t> cnt((size_t)ncl[i] + 1, 0);
    for (int64_t r = 0; r < n; ++r) cnt[lab[r] + 1] += 1;
    for (int k = 0; k < ncl[i]; ++k) cnt[k + 1] += cnt[k];
    std::vector<int64_t> tmp((size_t)n);
    std::vector<int> tl((size_t)n);
    for (int64_t r = 0; r < n; ++r) {
      int64_t p = cnt[lab[r]]++;
      tmp[p] = order[lo + r];
      tl[p] = lab[r];
    }
    for (int64_t r = 0; r < n; ++r) {
      order[lo + r] = tmp[r];
      label[lo + r] = tl[r];
    }
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
        int64_t lo = bstart[u], n = bstart[u + 1] - lo;
        int64_t r = 0;
        for (int k = 0; k < ncl[e]; ++k) {
          cl_off[cidx + k] = (uint32_t)(lo + r);
          while (r < n && label[lo + r] == k) ++r;
          for (int j = 0; j < b; ++j) cent[(size_t)(cidx + k) * b + j] = bcent[e][(size_t)k * b + j];
        }
        cidx += ncl[e];
        ++e;
      }
    }
    bkt_off[nb] = (uint32_t)cidx;
    cl_off[n_cl] = (uint32_t)N;
  }
  std::vector<uint32_t> ids((size_t)N);
  for (int64_t r = 0; r < N; ++r) ids[r] = (uint32_t)order[r];
  // 6. write
  FILE *f = fopen(path, "wb");
  if (!f) return -2;
  auto align = [](uint64_t v) { return (v + 255) & ~(uint64_t)255; };
  uint64_t sz[10] = {(uint64_t)c->H * D * 4,  (uint64_t)c->H * 4, (uint64_t)b * c->H * 4,
                     (uint64_t)b * 4,         (uint64_t)b * 4,    (uint64_t)(nb + 1) * 4,
                     (uint64_t)(n_cl + 1) * 4, (uint64_t)n_cl * b * 4, (uint64_t)N * 4,
                     (uint64_t)N * D * esz};
  uint64_t off[10];
  uint64_t cur = 256;
  for (int i = 0; i < 10; ++i) {
    off[i] = cur;
    cur = align(cur + sz[i]);
  }
  unsigned char h[256];
  memset(h, 0, sizeof(h));
  memcpy(h, "NRIXv001", 8);
  uint32_t u32;
  uint64_t u64;
  u32 = 1; memcpy(h + 8, &u32, 4);
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

}  // extern "C"
