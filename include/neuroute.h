/*
 * neuroute.h -- C ABI of the GB300 (sm_103a) NeuRoute batched query path.
 *
 * NeuRoute (arxiv 2608.15438) answers approximate k-nearest-neighbour queries
 * (problem statement: Sec. 3.1) from a bucketised index built on learned
 * binary codes. One search call runs, for every query, on the GPU:
 *   encode    l = E(q): MLP D -> H (ReLU) -> b logits               (Sec. 3.2.1)
 *   binarise  a_j = [l_j >= tau_j], base code u0 = sum_j a_j 2^j    (Eq. 10)
 *   probe     flip sets F ranked by summed deviation
 *             delta_j = |l_j - tau_j| -> probe codes u0 XOR F      (Sec. 3.2.3, Algorithm 1)
 *   lookup    code -> clusters -> rows through two CSR levels      (Sec. 3.3)
 *   select    singleton buckets to C^dir; centroid distances, gate
 *             theta = d_min + M(d_min), top-C -> C^cent            (Sec. 3.4.2, Algorithm 2)
 *   refine    exact squared L2 of the rows of C^dir U C^cent into a
 *             top-k, heap-quality early stop in fixed rounds      (Sec. 3.4, Algorithm 2)
 *
 * Conventions for every call
 *  - Pointers named d_* are DEVICE pointers on the index's device, row-major
 *    and contiguous; h_* are host pointers. The caller owns them.
 *  - `stream` is a cudaStream_t (NULL = the legacy default stream). Calls
 *    enqueue work on it and return; outputs are valid once the stream has
 *    synchronised. Argument and allocation errors are returned synchronously
 *    and enqueue nothing.
 *  - Device-side checks never trap: a bad index in the file, or a bounded
 *    wait inside a kernel that expires, sets a device flag that
 *    nr_last_stats reports as NR_ERR_DEVICE_CHECK (and clears).
 *  - One handle is not safe for concurrent calls (it owns one workspace).
 *  - Float arithmetic that decides an integer (bits, probe order, the gate,
 *    top-C, top-k membership) uses a fixed operation order, so results are
 *    bit-identical to a sequential CPU evaluation fed the same logits.
 *
 * Index file (little-endian), written by the package's builder:
 *   header 256 B: "NRIXv001", u32 version (1, or 2 with hidden layers after
 *     the first), u32 dtype (0 uint8, 1 fp32), u64 N (< 2^32 - 1), u32 D, H, b,
 *     K_max, t, u32 0, u64 n_clusters (< 2^31), f32 in_scale, u32 0,
 *     u64 section offsets[10], u64 file size; version 2 adds at byte 152
 *     u32 n_mid (1..7), u32 mid widths[7], u32 0, u64 offset of the eleventh
 *     section
 *   sections (256-byte aligned): W1 f32[H][D], b1 f32[H], W2 f32[b][H_last]
 *     (H_last = the last hidden width), b2 f32[b], tau f32[b], bkt_off
 *     u32[2^b + 1] (code -> cluster range), cl_off u32[n_clusters + 1]
 *     (cluster -> row range), cent f32[n_clusters][b], ids u32[N] (original id
 *     of each stored row), vec (uint8|fp32)[N][D] stored in (code, cluster, id)
 *     order; version 2: the middle layers, per layer W f32[w][previous width]
 *     then its bias f32[w]. Rows: uint8 or fp32 up to 1 KB, fp32 up to 8 KB
 *     (D <= 2048, a multiple of 64 bytes).
 */
#ifndef NEUROUTE_H
#define NEUROUTE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct nr_index nr_index; /* opaque, owned by the library */

typedef enum {
  NR_OK = 0,
  NR_ERR_INVALID_ARG = -1,  /* a bad argument or an unsupported size */
  NR_ERR_IO = -2,           /* the index file cannot be opened or read */
  NR_ERR_FORMAT = -3,       /* the index file is malformed or truncated */
  NR_ERR_OOM = -4,          /* device or host allocation failed */
  NR_ERR_CUDA = -5,         /* a CUDA runtime call failed */
  NR_ERR_DEVICE_CHECK = -6  /* a kernel found an out-of-range index in the file,
                               or a bounded wait inside a kernel expired */
} nr_status;

/* Query-time knobs. Defaults from nr_params_default().
 * Algorithm 1 filters (off by default): only the l_sel least-certain bits may
 * flip; |F| <= r_max; summed deviation <= s_max.
 * Gate of Algorithm 2: theta = d_min + M(d_min) with M(x) = gate_m0 + gate_m1 * x
 * (fp32 fmaf); gate_m0 = +inf turns the gate off.
 * Early stop (Sec. 3.4.2), counted in refinement rounds of round_size
 * candidates: after round t, "updates" = top-k members not present before the
 * round, "front updates" = those within the first ceil(alpha_front * k) slots;
 * the round is low quality iff updates < u_min and front updates < f_min; the
 * search stops once the top-k is full, t >= r_min and t_low consecutive rounds
 * were low quality (t_low = 0: never stop early). */
typedef struct {
  int l_sel;          /* <= 0: all b bits */
  int r_max;          /* <= 0: unbounded */
  float s_max;        /* +inf: off */
  float gate_m0;      /* +inf: gate off */
  float gate_m1;
  int round_size;     /* power of two in [32, 4096]; default 256 */
  int t_low;          /* default 4 */
  int u_min;          /* default 1 */
  int f_min;          /* default 1 */
  int r_min;          /* default 1 */
  float alpha_front;  /* in [0, 1]; default 0.5 */
  /* Centroid stage. cent_mode 0 (default): order independent, the gate uses
   * the final d_min over all probed non-singleton clusters and C^cent is the
   * top-C of the survivors. cent_mode 1: Algorithm 2's sequence: probes in
   * score bins Bin(s) = min(n_bins - 1, floor(s n_bins / s_max)) (one bin when
   * s_max = +inf); bins in order; single-cluster buckets of every bin entered
   * to C^dir; the other clusters of a bin, in probe order, in batches of
   * b_batch: d_min <- min(d_min, batch minimum), theta = d_min + M(d_min),
   * H <- the C smallest (d, c) of H U batch with d <= theta; a batch is low
   * quality iff fewer than c_u_min of its clusters are in H and fewer than
   * c_f_min of those have d <= d_min + c_alpha_front M(d_min); stop when
   * |H| = C, at least b_min bins were entered and c_t_low consecutive batches
   * were low quality (c_t_low = 0: never). C^cent = H. */
  int cent_mode;        /* 0 or 1; default 0. Mode 1 needs probe_budget <= 2048 and
                         * its shared memory (about 16 C + 12 P + 8 b_batch bytes)
                         * within 220 KB; searches outside are NR_ERR_INVALID_ARG */
  int n_bins;           /* >= 1; default 1 */
  int b_batch;          /* in [1, 2048]; default 256 */
  int b_min;            /* >= 0; default 1 */
  int c_t_low;          /* >= 0; default 0 */
  int c_u_min, c_f_min; /* >= 0; default 1, 1 */
  float c_alpha_front;  /* in [0, 1]; default 0.5 */
  /* Calibrated gate (Sec. 3.4): when gate_n >= 2 (at most 16), M is the
   * piecewise-linear curve through (gate_x[i], gate_y[i]), flat beyond its
   * ends: on segment i (the last breakpoint with gate_x[i] <= x),
   * M(x) = fmaf(x - x_i, (y_{i+1} - y_i) / (x_{i+1} - x_i), y_i) in fp32, held
   * within [y_i, y_{i+1}] so that M never decreases; the gate is then on and
   * gate_m0 / gate_m1 are unused. gate_x strictly increasing, gate_y
   * non-decreasing, all finite. gate_n = 0: M(x) = m0 + m1 x. */
  int gate_n;           /* 0, or 2..16; default 0 */
  float gate_x[16], gate_y[16];
  /* Execution only (results do not depend on these). pipe_chunk > 0: a batch
   * larger than pipe_chunk queries runs in chunks of pipe_chunk, the
   * refinement of a chunk (on a library-owned stream) overlapping encode,
   * route and select of the next chunks (on another), in up to three chunk
   * buffers; the caller's stream waits for both at the end of the call.
   * 0 (default): every stage on the caller's stream, one after the other.
   * refine_ctas: refinement blocks resident per SM, capped (0: as many as fit),
   * which leaves SM room to the overlapping stages. */
  int pipe_chunk;       /* >= 0; default 0 */
  int refine_ctas;      /* in [0, 32]; default 0 */
  /* 1: probe_budget counts non-empty buckets: flip sets in key order whose
   * buckets hold no cluster are skipped (not listed, not counted), the first
   * probe_budget non-empty ones listed, at most NR_NONEMPTY_SCAN *
   * probe_budget flip sets examined, the base code included. 0 (default):
   * probe_budget counts codes, empty buckets included. */
  int nonempty_budget;  /* 0 or 1; default 0 */
  /* Execution only: the limit of the tensor-core encoder's bounded hand-off
   * waits. 0 (default): 1 s; > 0: that many microseconds (at most 60 s);
   * < 0: a wait whose phase is not complete when first tested expires at
   * once, which exercises the failure path (the kernel stops, drains its
   * issued MMAs under its own 1 s bound, frees its tensor memory and sets the
   * device flag that nr_last_stats reports as NR_ERR_DEVICE_CHECK). */
  int wait_limit_us;
} nr_params;

#define NR_NONEMPTY_SCAN 4

/* Per-search statistics (sums over the queries of the last search call). */
typedef struct {
  int64_t nq;
  int64_t candidates; /* rows given an exact distance (rows of completed rounds) */
  int64_t rounds;     /* refinement rounds run */
  int64_t clusters;   /* |C^dir U C^cent| */
  int64_t probes;     /* probe codes generated */
  int64_t scored;     /* clusters whose centroid distance was evaluated */
} nr_stats;

/* Status name, static storage. */
const char *nr_status_string(nr_status s);

/* Fill *p with the defaults above. */
nr_status nr_params_default(nr_params *p);

/* Load an index file into device memory on `device` (CUDA ordinal): the
 * encoder and thresholds (Sec. 3.2.1, 3.2.3), the bucket directory and the
 * bucket-local clusters over the stored rows (Sec. 3.3).
 * Errors: NR_ERR_IO, NR_ERR_FORMAT (bad magic, sizes, truncation; b must be in
 * [1, 24]; a row must be a multiple of 16 bytes and at most 1024 bytes),
 * NR_ERR_OOM, NR_ERR_CUDA. On success *out owns all device memory of the
 * index; release it with nr_index_free. */
nr_status nr_index_load(const char *path, int device, nr_index **out);

/* Release the index and its workspace. NULL is a no-op. */
void nr_index_free(nr_index *ix);

/* info[0..7] = N, D, H, b, n_clusters, dtype (0 uint8, 1 fp32), K_max, t */
nr_status nr_index_info(const nr_index *ix, int64_t *info);

/* Copy the per-bit thresholds tau [b] (Sec. 3.2.3) to host memory h_tau.
 * Synchronous. Errors: NR_ERR_INVALID_ARG, NR_ERR_CUDA. */
nr_status nr_index_thresholds(nr_index *ix, float *h_tau);

/* Write the index to `path` in the file format above (the bytes nr_index_load
 * reads back). Waits for the device to finish its work first, then copies the
 * sections out through a pinned buffer. Errors: NR_ERR_IO (open or write),
 * NR_ERR_OOM, NR_ERR_CUDA. A failed call may leave a partial file. */
nr_status nr_index_save(nr_index *ix, const char *path);

/* Write to `path` a sub-index that holds only the buckets of the listed codes
 * (every other bucket empty), in the file format above. Clusters and rows keep
 * their order, so a query whose probe codes all lie in the list gets exactly
 * the results and statistics it gets from the whole index (cluster ties are
 * broken by cluster order, which is kept); it serves to check or time a CPU
 * evaluation of sample queries against an index too large for host memory.
 * h_codes: n host u32 codes < 2^b, any order, repeats allowed. info[0..1]
 * (may be NULL) = rows and clusters written. Errors: NR_ERR_INVALID_ARG (a code
 * out of range, or no row selected), NR_ERR_DEVICE_CHECK (inconsistent
 * offsets), NR_ERR_IO, NR_ERR_OOM, NR_ERR_CUDA. */
nr_status nr_index_extract(nr_index *ix, const uint32_t *h_codes, int64_t n, const char *path,
                           int64_t *info);

/* Where rows are stored, for calibrating the gate M and the score cutoff
 * S_max (Sec. 3.4: both are fitted on where a query's true neighbours lie).
 * d_ids: n device int64 row ids (any order, repeats allowed). d_out: n x 4
 * device int32, per id (cluster, bucket code, first cluster of that bucket,
 * clusters in that bucket), or (-1, -1, -1, 0) for an id not in the index.
 * Allocates O(n) device scratch; synchronous on `stream`. 0 <= n < 2^31.
 * Errors: NR_ERR_INVALID_ARG, NR_ERR_OOM, NR_ERR_CUDA. */
nr_status nr_index_locate(nr_index *ix, const int64_t *d_ids, int64_t n, int32_t *d_out,
                          void *stream);

/* Centroid distances (Eq. 12): d_out[q * m + j] = sum_i (l_qi - mu_ci)^2 with
 * c = d_clusters[q * m + j], evaluated as the query path evaluates it (fp32,
 * one fused multiply-add per coordinate in coordinate order), +inf where c is
 * out of range (-1 pads). d_logits [nq x b] fp32, d_clusters [nq x m] int32,
 * d_out [nq x m] fp32, all device. Asynchronous on `stream`.
 * Errors: NR_ERR_INVALID_ARG, NR_ERR_CUDA. */
nr_status nr_centroid_dists(nr_index *ix, const float *d_logits, int64_t nq,
                            const int32_t *d_clusters, int m, float *d_out, void *stream);

/* Calibration of the gate margin M and the bucket-score cutoff S_max from
 * held-out queries (Sec. 3.4: both are fitted on where a query's true
 * neighbours lie). Definitions, for a query with logits l, base code u0 and
 * deviations delta_j = |l_j - tau_j| ranked by (delta_j, j):
 *   score of bucket code u = the fp32 sum of delta over the ranks whose bit
 *     differs between u and u0, in ascending rank (Algorithm 1's cost);
 *   x = the smallest centroid distance over every cluster of the target
 *     buckets that hold two or more clusters (single-cluster buckets bypass
 *     the gate); y = the largest distance of such a target's own cluster,
 *     minus x (fp32); both NaN without such a target;
 *   S_max = the pair scores (NaN skipped) sorted, the entry at position
 *     ceil(coverage m) - 1 (clamped to [0, m - 1]);
 *   M = the queries with an x sorted by (x, y) in B = min(n_bins, n)
 *     equal-frequency bins [floor(i n / B), floor((i + 1) n / B)), a bin's
 *     point (x at its lower-median position, its y at sorted position
 *     ceil(q m) - 1), equal x merged (larger y), the y's running maximum; a
 *     single point (x0, y0) becomes (x0, y0), (next float above x0, y0).
 * Distances are the select kernel's fmaf chain. */

/* Scores of bucket codes: d_logits [nq x b] fp32, d_tau [b], d_codes
 * [nq x k] int32 (negative: none) -> d_scores [nq x k] fp32 (NaN for none);
 * all device, asynchronous on `stream`. 1 <= b <= 31.
 * Errors: NR_ERR_INVALID_ARG, NR_ERR_CUDA. */
nr_status nr_bucket_scores(const float *d_logits, const float *d_tau, int b, const int32_t *d_codes,
                           int64_t nq, int k, float *d_scores, void *stream);

/* Observations of nq calibration queries (device logits [nq x b]) with their
 * targets d_targets [nq x k] (device int64 row ids, -1 = none; typically
 * their top-k from a high-recall search): d_scores [nq x k] (NaN where the
 * target is not stored), d_x [nq], d_y [nq], all device fp32. Allocates
 * O(nq k) device scratch; synchronous on `stream`. nq k < 2^31.
 * Errors: NR_ERR_INVALID_ARG, NR_ERR_OOM, NR_ERR_CUDA. */
nr_status nr_calib_observe(nr_index *ix, const float *d_logits, const int64_t *d_targets, int64_t nq,
                           int k, float *d_scores, float *d_x, float *d_y, void *stream);

/* S_max from host scores [nq x k] at `coverage`; *pair_coverage = the
 * fraction of scores at or below it, *query_coverage = the fraction of the
 * queries with a score whose scores all are; *s_max = NaN (and both 0) when
 * no score is given. Host only. Errors: NR_ERR_INVALID_ARG. */
nr_status nr_calib_fit_s_max(const float *h_scores, int64_t nq, int k, double coverage,
                             float *s_max, double *pair_coverage, double *query_coverage);

/* The margin curve from host x, y [n] (NaN x skipped) at quantile q with
 * 1 <= n_bins <= 16 bins: *gate_n points (0 without observations, else 2..16)
 * in gate_x, gate_y [16]. Host only. Errors: NR_ERR_INVALID_ARG. */
nr_status nr_calib_fit_gate(const float *h_x, const float *h_y, int64_t n, int n_bins, double q,
                            int *gate_n, float *gate_x, float *gate_y);

/* All of the above: observations of the targets, S_max at `coverage` and the
 * curve at `quantile` written into *p (s_max, gate_n, gate_x, gate_y; the
 * other fields untouched; a fit without data leaves its fields as they
 * were); info (may be NULL) [3] = pair coverage, query coverage, queries with
 * an x. Pass *p to nr_set_params to search with them. Synchronous.
 * Errors: NR_ERR_INVALID_ARG, NR_ERR_OOM, NR_ERR_CUDA. */
nr_status nr_calibrate(nr_index *ix, const float *d_logits, const int64_t *d_targets, int64_t nq,
                       int k, int n_bins, double quantile, double coverage, nr_params *p,
                       double *info, void *stream);

/* Validate and set the query-time knobs (p = NULL restores the defaults).
 * NR_ERR_INVALID_ARG if a field is out of range. */
nr_status nr_set_params(nr_index *ix, const nr_params *p);

/* Encoder forward (Sec. 3.2.1): d_x [nq x D] (uint8 or fp32, the index dtype)
 * -> d_logits [nq x b] fp32, both device, row-major and contiguous.
 * h = ReLU(W1 (in_scale x) + b1), l = W2 h + b2 (with hidden layers after
 * the first, each h' = ReLU(W h + b) in turn). With d_x 16-byte aligned these
 * run on the tensor cores, operands fp16 (fp32 inputs and hidden activations
 * rounded to fp16, so magnitudes beyond 65504 do not fit), accumulation fp32
 * (logits agree with an exact evaluation to about 1e-3 of their norm): one
 * hidden layer with D % 16 == 0, D <= 128, H % 128 == 0, b <= 32, fused in one
 * kernel; several hidden layers with D and every hidden width multiples of
 * 64, layer by layer, each layer's activations in a scratch buffer the index
 * keeps (grown on demand: the first call of a larger batch, up to 2^18 rows,
 * allocates and synchronises the device). Other shapes and misaligned input
 * run on CUDA cores in fp32. nq = 0 is a no-op. Asynchronous on `stream`; a
 * device-side wait that expires sets the device flag (see nr_last_stats).
 * Errors: NR_ERR_INVALID_ARG, NR_ERR_CUDA. */
nr_status nr_encode(nr_index *ix, const void *d_x, int64_t nq, float *d_logits, void *stream);

/* Probe codes (Eq. 10 and Algorithm 1) from d_logits [nq x b]:
 * d_codes [nq x probe_budget] u32 receives, per query, the codes of the first
 * min(probe_budget, #admissible flip sets) flip sets in ascending
 * (cost, |F|, rank mask) order, the base code first; d_nprobe [nq] their count.
 * Unused slots are set to 0xFFFFFFFF. 1 <= probe_budget <= 4096. */
nr_status nr_route(nr_index *ix, const float *d_logits, int64_t nq, int probe_budget,
                   uint32_t *d_codes, int32_t *d_nprobe, void *stream);

/* Ordered cluster list C^dir U C^cent (Sec. 3.4.2) from d_logits:
 * d_clusters [nq x (probe_budget + cluster_budget)] int32 cluster indices sorted
 * by (centroid distance, cluster index), -1 padded; d_ncl [nq] their count.
 * Limits: 1 <= cluster_budget <= 4096; probe_budget * K_max <= 65536. */
nr_status nr_debug_clusters(nr_index *ix, const float *d_logits, int64_t nq, int probe_budget,
                            int cluster_budget, int32_t *d_clusters, int32_t *d_ncl,
                            void *stream);

/* Whole query path (the k-NN problem of Sec. 3.1, answered by the retrieval
 * of Sec. 3.4: encode, Eq. 10, Algorithm 1, Sec. 3.3 lookup, Algorithm 2,
 * exact refinement): d_queries [nq x D] (index dtype) -> d_out_ids [nq x k]
 * int64 original ids and d_out_dists [nq x k] fp32 squared L2 distances, each
 * row sorted by (distance, id), padded with (-1, +inf) when fewer than k rows
 * were scored. For uint8 indexes distances are the exact integer sums.
 * 1 <= k <= 256, 1 <= probe_budget <= 4096, 1 <= cluster_budget <= 4096,
 * probe_budget * K_max <= 65536. The library's workspace grows on demand. */
nr_status nr_search(nr_index *ix, const void *d_queries, int64_t nq, int k, int probe_budget,
                    int cluster_budget, int64_t *d_out_ids, float *d_out_dists, void *stream);

/* As nr_search, with the logits supplied by the caller (d_logits [nq x b]);
 * the encoder (Sec. 3.2.1) is not run, every later step of Sec. 3.4 is. */
nr_status nr_search_logits(nr_index *ix, const void *d_queries, const float *d_logits, int64_t nq,
                           int k, int probe_budget, int cluster_budget, int64_t *d_out_ids,
                           float *d_out_dists, void *stream);

/* As nr_search (Sec. 3.4) with HOST buffers: h_queries [nq x D] is copied to the device,
 * the search runs, and h_out_ids / h_out_dists are copied back; the call
 * returns after the stream has synchronised. Pinned host memory gives full
 * copy bandwidth; pageable memory works. */
nr_status nr_search_host(nr_index *ix, const void *h_queries, int64_t nq, int k, int probe_budget,
                         int cluster_budget, int64_t *h_out_ids, float *h_out_dists,
                         void *stream);

/* As nr_search, but the call allocates no memory: its scratch lives in one
 * fixed array of 32 MiB (NR_STATIC_SCRATCH_BYTES) compiled into the library,
 * which every GPU that loads the library holds until the process exits.
 * For callers that may not allocate device memory while serving queries:
 * code running under a device-memory budget owned by a host framework or an
 * inference server, and latency-critical loops in which cudaMalloc / cudaFree
 * (which can synchronise the device) are not acceptable. The paper has no
 * counterpart; the kernels, their order and their results are nr_search's.
 * Arguments are checked as nr_search checks them (the same budgets, k, batch
 * size and sequential-stage limits, NR_ERR_INVALID_ARG otherwise).
 * Size limit: with S = the smallest power of two >= probe_budget * K_max, a
 * call needs nq * (4 b + 4 P + 12 (P + C) + 56) bytes, plus nq * 12 S bytes
 * when S > 2048 (select's global sort slabs), each of its eleven buffers
 * rounded up to 256 bytes; a request beyond 32 MiB returns NR_ERR_INVALID_ARG
 * without enqueuing work. Splitting the batch brings nq down; a single query
 * needs about 12 S bytes, so every budget nr_search accepts (S <= 65536,
 * 768 KiB) fits for small enough batches.
 * The first call on a device looks up the array's device address with that
 * device made current and keeps it for the life of the process; make that
 * first call before any stream capture, and do not use the library across a
 * device reset (cudaDeviceReset), which would leave the kept address stale.
 * All calls share the one array and it keeps the last call's contents: two
 * calls whose work overlaps on the GPU (different streams, or different
 * indexes on the same device) race and corrupt each other; serialise them.
 * nr_last_stats and nr_query_stats after this call read its statistics from
 * the array; stage timing is not recorded. */
nr_status nr_search_static(nr_index *ix, const void *d_queries, int64_t nq, int k, int probe_budget,
                           int cluster_budget, int64_t *d_out_ids, float *d_out_dists,
                           void *stream);

/* Per-query statistics of the last search call: d_stats [nq x 5] int64 =
 * (candidates, rounds, |C^dir U C^cent|, probes, clusters scored), the last
 * being the number of centroid distances evaluated (Sec. 3.5's C_q).
 * Enqueued on `stream`. */
nr_status nr_query_stats(nr_index *ix, int64_t *d_stats, int64_t nq, void *stream);

/* Sums over the last search call (synchronises the device). Also returns
 * NR_ERR_DEVICE_CHECK, and clears the flag, if a kernel has flagged bad index
 * data or an expired wait since load or since the last such report. */
nr_status nr_last_stats(nr_index *ix, nr_stats *out);

/* Kernel time in milliseconds of the stages of the last search call
 * (ms[0..3] = encode, route, select, refine) measured with CUDA events on the
 * launch stream; enable with nr_enable_timing(ix, 1). Synchronises. */
nr_status nr_enable_timing(nr_index *ix, int on);
nr_status nr_last_timing(nr_index *ix, float *ms);

/* Measurement utility, not part of the search: the rate at which the GPU
 * `device` reads rows at random. n rows of row_bytes (a multiple of 16, at
 * most 1024) at well-mixed pseudo-random indices below `rows` are read from a
 * rows x row_bytes array, one row per thread, with L2 evicted before each of
 * reps runs; *h_gbs = row bytes read per second of the best run, in GB/s.
 * It bounds a kernel whose bytes are random row gathers, as the centroid
 * stage's are (Sec. 3.5: C_q centroid rows a query), the way the copy
 * bandwidth bounds a stream. Allocates rows * row_bytes + 4 n + 512 MiB of
 * device memory for the call and frees it; synchronous.
 * Errors: NR_ERR_INVALID_ARG, NR_ERR_OOM, NR_ERR_CUDA. */
nr_status nr_measure_gather(int device, int64_t rows, int row_bytes, int64_t n, int reps,
                            double *h_gbs);

/* Measurement utility, not part of the search: the rate at which the GPU
 * `device` reads a long contiguous array (`bytes`, a multiple of 16, at least
 * 1 MiB), sequentially, with no writes but one word a thread, L2 evicted
 * before each of reps runs; *h_gbs = bytes read per second of the best run,
 * in GB/s. It bounds a kernel whose bytes are reads of long runs, as the
 * refinement's are (Sec. 3.5: the candidate rows), more tightly than the
 * copy bandwidth, whose bytes are half writes. Allocates bytes + 512 MiB and
 * a few MB of device memory for the call and frees it; synchronous.
 * Errors: NR_ERR_INVALID_ARG, NR_ERR_OOM, NR_ERR_CUDA. */
nr_status nr_measure_read(int device, int64_t bytes, int reps, double *h_gbs);

/* Number of kernels the library launched since load (all entry points). */
int64_t nr_kernel_launches(const nr_index *ix);

#ifdef __cplusplus
}
#endif
#endif /* NEUROUTE_H */
