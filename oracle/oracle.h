/*
 * NeuRoute query-path ORACLE: a plain, slow, obviously-correct CPU
 * implementation of the batched search, written step by step from the paper
 * (NeuRoute, arxiv 2608.15438).
 *
 * This is TEST INFRASTRUCTURE. Only the test suite, the package smoke check and
 * the benchmark's CPU-baseline leg may load it. The product library never calls
 * it, and it shares no code, header, table or helper with the CUDA path: it
 * reads the index file with its own reader and implements every step itself.
 *
 * Steps and the passages they follow (paper section / equation / algorithm):
 *   or_encode          encoder forward l = E(x), one hidden ReLU layer (Sec. 3.2.1)
 *   or_probe_*         binarisation a_j = [l_j >= tau_j] (Eq. 10), deviation
 *                      delta_j = |l_j - tau_j| (Sec. 3.2.3), flip-set enumeration
 *                      ranked by summed deviation (Algorithm 1)
 *   or_cluster_list    bucket -> clusters (Sec. 3.3), singleton buckets to C^dir,
 *                      centroid distances, calibrated gate theta = d + M(d) and
 *                      top-C (Algorithm 2, Sec. 3.4.2)
 *   or_cluster_list_seq  the same stage in Algorithm 2's sequence: score bins,
 *                      centroid batches, running d_min, heap-quality early stop
 *   or_refine_stream   exact squared-L2 refinement into a top-k with heap-quality
 *                      early stopping counted in fixed rounds (Sec. 3.4.2, Alg. 2)
 *   or_search          all of the above per query, threads across queries
 *   or_bruteforce      exact k-NN by full scan (the problem statement, Sec. 3.1)
 *
 * Readings taken where the paper is silent (each is pinned by a test):
 *   - probe order key = (fp32 cost summed left to right over ascending rank,
 *     |F|, rank mask), exact top-P instead of score bins;
 *   - gate uses the final d_min over all probed non-singleton centroids,
 *     M(x) = m0 + m1 * x (gate off when m0 = +inf);
 *   - a round's "updates" = top-k members after the round that were not members
 *     before it; "front updates" = the same within the first ceil(alpha*k) slots.
 * Parity of the early-stop rule itself is unpinned by the paper (it prints no
 * worked example); it is pinned only by hand-built candidate streams.
 *
 * Compiled with -ffp-contract=off: the only fused multiply-adds are the
 * explicit std::fmaf chains.
 */
#ifndef NEUROUTE_ORACLE_H
#define NEUROUTE_ORACLE_H
#include <stdint.h>
#ifdef __cplusplus
extern "C" {
#endif

typedef struct or_index or_index;

typedef struct {
  int l_sel;          /* flippable ranks < l_sel; <= 0: all b bits */
  int r_max;          /* |F| <= r_max; <= 0: unbounded */
  float s_max;        /* summed deviation <= s_max; +inf: off */
  float gate_m0;      /* M(x) = m0 + m1 x; m0 = +inf: gate off */
  float gate_m1;
  int round_size;     /* candidates per early-stop round (R) */
  int t_low;          /* stop after t_low consecutive low-quality rounds; 0: never */
  int u_min;          /* round is low quality iff new < u_min and front < f_min */
  int f_min;
  int r_min;          /* no stop before r_min completed rounds */
  float alpha_front;  /* front = first ceil(alpha_front * k) slots of the top-k */
  /* centroid stage: 0 = order-independent (final d_min gate, top-C); 1 = the
   * sequential stage of Algorithm 2 (score bins, centroid batches, running
   * d_min gate, a bounded heap of C, early stop on heap quality) */
  int cent_mode;
  int n_bins;          /* score bins over [0, s_max] (Algorithm 1); one bin if s_max = +inf */
  int b_batch;         /* clusters per centroid batch (B_batch) */
  int b_min;           /* bins started before a stop is allowed (B_min) */
  int c_t_low;         /* stop after c_t_low consecutive low-quality batches; 0: never */
  int c_u_min, c_f_min; /* batch low quality iff updates < c_u_min and front < c_f_min */
  float c_alpha_front; /* front threshold d_min + c_alpha_front * M(d_min) */
  /* calibrated gate (Sec. 3.4): when gate_n >= 2, M is the piecewise-linear
   * curve through (gate_x[i], gate_y[i]) (x increasing, y non-decreasing),
   * flat beyond its ends, instead of gate_m0 + gate_m1 x */
  int gate_n;
  float gate_x[16], gate_y[16];
  /* 1: the probe budget counts non-empty buckets (the D3 variant): flip sets
   * in key order whose buckets hold no cluster are skipped, the first P
   * non-empty ones listed, at most OR_NONEMPTY_SCAN * P flip sets examined
   * (the base code included). 0 (default): P counts codes. */
  int nonempty_budget;
} or_params;

#define OR_NONEMPTY_SCAN 4

void or_params_default(or_params *p);

/* index file (format written by the package's builder); NULL on error */
or_index *or_index_load(const char *path, char *err, int errlen);
void or_index_free(or_index *ix);
/* info[0..7] = N, D, H, b, n_clusters, dtype (0 u8, 1 f32), K_max, t */
void or_index_info(const or_index *ix, int64_t *info);
/* pointers into the loaded index (read-only) */
const uint32_t *or_index_bkt_off(const or_index *ix);
const uint32_t *or_index_cl_off(const or_index *ix);
const uint32_t *or_index_ids(const or_index *ix);
const float *or_index_tau(const or_index *ix);
const float *or_index_cent(const or_index *ix);

/* logits [nq x b] (fp32, rounded from a double-precision forward pass) */
void or_encode(const or_index *ix, const void *x, int64_t nq, float *logits, int nthreads);

/* Widths of the hidden layers after the first (widths[0..n_mid), at most 7);
 * returns n_mid. */
int or_index_mid(const or_index *ix, int32_t *widths);

/* Logits of rows x under an encoder given by its weights: W1 [H x D], b1 [H],
 * then n_mid hidden layers of widths mid_w (Wm: per layer W [w x previous]
 * followed by its bias [w], concatenated), W2 [b x last hidden width], b2 [b]. */
void or_encode_mlp(int dtype, int D, int H, int b, int n_mid, const int *mid_w, float in_scale,
                   const float *W1, const float *b1, const float *W2, const float *b2,
                   const float *Wm, const void *x, int64_t nq, float *logits, int nthreads);
/* the same forward pass from explicit weights W1 [H x D], b1 [H], W2 [b x H],
 * b2 [b] (dtype 0 uint8 rows, 1 fp32 rows; inputs scaled by in_scale) */
void or_encode_weights(int dtype, int D, int H, int b, float in_scale, const float *W1,
                       const float *b1, const float *W2, const float *b2, const void *x,
                       int64_t nq, float *logits, int nthreads);

/* Probe order from a per-rank deviation vector sd[0..b-1] (sd sorted ascending
 * is NOT required here; rank r has cost sd[r]). Best-first over "add one rank"
 * with duplicate suppression. keys[i] = cost_bits << 32 | |F| << 24 | rankmask.
 * Returns the number of keys written (<= P). */
int or_probe_order(int b, const float *sd, int P, const or_params *p, uint64_t *keys);
/* Same order by sorting the keys of all 2^b subsets (b <= 20): a brute-force
 * cross-check of or_probe_order. */
int or_probe_order_allsubsets(int b, const float *sd, int P, const or_params *p, uint64_t *keys);

/* Full probe list of one query: codes[i] = u0 XOR flips of the i-th flip set.
 * keys (optional) as above; perm (optional) [b] = bit index of each rank. */
int or_probe_list(int b, const float *logit, const float *tau, int P, const or_params *p,
                  uint32_t *codes, uint64_t *keys, int32_t *perm);

/* The probe list of one query under p, against the index (for the
 * non-empty budget): codes [P], keys [P] (optional). Returns its length. */
int or_probe_list_index(const or_index *ix, const float *logit, int P, const or_params *p,
                        uint32_t *codes, uint64_t *keys);

/* Ordered cluster list L = C^dir U C^cent of one query. L has room for
 * nprobe + C entries; dL (optional) gets each entry's centroid distance.
 * n_dir (optional) gets |C^dir|; n_scored (optional) the number of centroid
 * distances evaluated (every cluster of every probed bucket). Returns |L|, or
 * -1 on an out-of-range index. */
int or_cluster_list(const or_index *ix, const float *logit, const uint32_t *codes, int nprobe,
                    int C, const or_params *p, int32_t *L, float *dL, int32_t *n_dir,
                    int64_t *n_scored);

/* The sequential centroid stage (Algorithm 2) of one query: probes in order
 * with scores score[i] (the summed deviation of their flip set), binned by
 * Bin(s) = min(n_bins - 1, floor(s n_bins / s_max)); bins processed in order;
 * single-cluster buckets of every bin entered go to C^dir; the other clusters
 * of a bin, in probe order, in batches of b_batch: d_min <- min(d_min, batch
 * min), theta = d_min + M(d_min), H <- the C smallest (d, c) of H U batch with
 * d <= theta; updates = batch entries in H, front = those with
 * d <= d_min + c_alpha_front M(d_min); stop when |H| = C, at least b_min bins
 * were entered and c_t_low consecutive batches had updates < c_u_min and
 * front < c_f_min. L = C^dir U H in (d, c) order. n_batches (optional) gets
 * the batches processed, n_scored (optional) the centroid distances evaluated
 * (C^dir of the bins entered plus the clusters of the batches processed).
 * Returns |L|, or -1 on an out-of-range index. */
int or_cluster_list_seq(const or_index *ix, const float *logit, const uint32_t *codes,
                        const float *score, int nprobe, int C, const or_params *p, int32_t *L,
                        float *dL, int32_t *n_dir, int32_t *n_batches, int64_t *n_scored);

/* The gate margin M(x) of the parameters p (linear, or the calibrated curve). */
float or_gate_margin(const or_params *p, float x);

/* Centroid distance (Eq. 12) of cluster c from one query's logits, the fmaf
 * chain of the centroid stage; +inf when c is out of range. */
float or_centroid_dist(const or_index *ix, const float *logit, int64_t c);

/* Refinement over an explicit candidate stream: rows [n x D] (u8 or f32 by
 * dtype), ids [n]. out_ids/out_d [k] sorted by (dist, id), padded (-1, +inf).
 * stats[0..1] = candidates scored, rounds. */
void or_refine_stream(int dtype, int D, const void *q, const void *rows, const uint32_t *ids,
                      int64_t n, int k, const or_params *p, int64_t *out_ids, float *out_d,
                      int64_t *stats);

/* Whole search. logits may be NULL (then computed by or_encode).
 * out_ids/out_d [nq x k]; stats (optional) [nq x 5] = candidates scored, rounds,
 * |L|, probes, centroid distances evaluated. Returns 0, or -1 on an
 * out-of-range index in the file. */
int or_search(const or_index *ix, const void *queries, const float *logits, int64_t nq, int k,
              int P, int C, const or_params *p, int64_t *out_ids, float *out_d, int64_t *stats,
              int nthreads);

/* Exact k-NN over base [N x D] (ids = row numbers), sorted by (dist, id). */
void or_bruteforce(int dtype, int D, const void *base, int64_t N, const void *queries, int64_t nq,
                   int k, int64_t *out_ids, float *out_d, int nthreads);

#ifdef __cplusplus
}
#endif
#endif
