/*
 * neuroute_build.h -- index construction on the GPU (the step before the
 * query path of neuroute.h), for indexes too large for a host build.
 *
 * It builds the index of paper Sec. 3.3 (thresholds: Sec. 3.2.3):
 *   1. logits of every base row, l_i = E(x_i) (the library's tensor-core
 *      encoder, nr_build_encode) or given by the caller (nr_build_set_logits);
 *   2. tau_j = lower median of logit column j: the element of rank
 *      floor((N - 1) / 2) in the total order of fp32 bit patterns (-0 < +0);
 *   3. code u_i with bit j = [l_ij >= tau_j]; bucket = code;
 *   4. per non-empty bucket B (members in id order), K_B = min(K_max,
 *      ceil(|B| / t)) clusters (at most |B|) by k-means in logit space:
 *      k-means++ seeding on the members at positions floor(i |B| / m),
 *      m = min(|B|, sample_per_cluster * K_B), then lloyd_iters passes of
 *      (assign to the nearest centroid, ties to the lower index; move each
 *      centroid with members to their mean); clusters left without members
 *      are dropped;
 *   5. rows stored in (code, cluster, id) order under the two CSR levels.
 * Every float operation of step 4 has a fixed definition: fp32 distances with
 * each product and sum rounded (no fused multiply-add), means summed as
 * fixed-point integers (scale 2^G, G = 30 - e, max |logit| = f 2^e with
 * f in [0.5, 1)), seeding draws weighted by trunc(dmin * 2^(50 - e(max dmin)))
 * from a splitmix64 stream seeded by (seed, code). Fed the same logits, the
 * package's host builder (nrb_build_logits) writes the same bytes.
 *
 * A build runs in two passes over the base rows, so the caller never needs
 * the whole unsorted base on the device at once:
 *   nr_build_begin                  -> logits buffer [N x b] fp32 on the device
 *   nr_build_encode / _set_logits   -> any row ranges covering [0, N) once
 *   nr_build_finish                 -> steps 2-5 except the rows themselves
 *   nr_build_place                  -> any row ranges covering [0, N) once
 *   nr_build_end                    -> a query-ready nr_index (as nr_index_load)
 * Device memory: 4bN bytes of logits plus about 17N bytes of sort buffers
 * during nr_build_finish; after it, the index itself (N row_bytes + 4N ids +
 * the CSR levels and centroids) plus 4N bytes of row positions until
 * nr_build_end.
 *
 * Conventions as in neuroute.h (d_* device pointers on the builder's device,
 * row-major; `stream` a cudaStream_t; argument errors returned synchronously).
 * Limits: b in [1, 24], K_max in [1, 64], N in [1, 2^32 - 2], row bytes a
 * multiple of 16 and at most 1024.
 */
#ifndef NEUROUTE_BUILD_H
#define NEUROUTE_BUILD_H

#include <stdint.h>

#include "neuroute.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct nr_builder nr_builder; /* opaque, owned by the library */

/* Same fields and layout as the host builder's configuration. */
typedef struct {
  int dtype;              /* 0 = uint8 rows, 1 = fp32 rows */
  int D, H, b;            /* row dimension, encoder hidden width, code bits */
  int K_max;              /* clusters per bucket at most */
  int t;                  /* target cluster capacity */
  float in_scale;         /* encoder input scale (1/255 for uint8 rows) */
  int lloyd_iters;        /* Lloyd passes per bucket (< 1 means 1) */
  int sample_per_cluster; /* k-means++ sample per cluster (>= 1) */
  uint64_t seed;          /* k-means++ seed */
  int n_mid;              /* encoder hidden layers after the first (0..7) */
  int mid_w[7];           /* their widths */
} nr_build_config;

/* Start a build of N rows on `device`. W1 [H x D], b1 [H], W2 [b x H_last],
 * b2 [b] are host fp32 encoder weights, copied; H_last is the last hidden
 * width. Wm (NULL when n_mid = 0): the hidden layers after the first, for
 * each W [mid_w[i] x previous width] then its bias [mid_w[i]], concatenated.
 * Errors: NR_ERR_INVALID_ARG (a field out of range), NR_ERR_OOM, NR_ERR_CUDA. */
nr_status nr_build_begin(const nr_build_config *cfg, int64_t N, const float *W1, const float *b1,
                         const float *W2, const float *b2, const float *Wm, int device,
                         nr_builder **out);

/* Pass 1, encoder: logits of rows [row0, row0 + n) from d_rows [n x D]
 * (uint8 or fp32, cfg.dtype). Enqueued on `stream`. */
nr_status nr_build_encode(nr_builder *bd, const void *d_rows, int64_t row0, int64_t n,
                          void *stream);

/* Pass 1, given logits: copy d_logits [n x b] fp32 as the logits of rows
 * [row0, row0 + n). Enqueued on `stream`. */
nr_status nr_build_set_logits(nr_builder *bd, const float *d_logits, int64_t row0, int64_t n,
                              void *stream);

/* Steps 2-5 (all but copying the rows). The ranges given in pass 1 must add
 * up to exactly N rows, and their work must be complete (synchronise the
 * streams used) before this call; it runs on an internal stream and returns
 * when done. info[0..4] (may be NULL) = n_clusters, non-empty buckets, largest
 * bucket, largest cluster, buckets holding one cluster. Frees the logits.
 * Errors: NR_ERR_INVALID_ARG (pass 1 incomplete, or a logit that is not
 * finite), NR_ERR_OOM, NR_ERR_CUDA. */
nr_status nr_build_finish(nr_builder *bd, int64_t *info);

/* Pass 2: store rows [row0, row0 + n) from d_rows [n x D] at their positions.
 * Enqueued on `stream`; d_rows must stay valid until the stream reaches it. */
nr_status nr_build_place(nr_builder *bd, const void *d_rows, int64_t row0, int64_t n,
                         void *stream);

/* Finish: the ranges of pass 2 must add up to exactly N rows. Waits for the
 * device, then hands the index over in *out (release with nr_index_free) and
 * frees the builder, also on error. */
nr_status nr_build_end(nr_builder *bd, nr_index **out);

/* Abandon a build and free its memory. NULL is a no-op. */
void nr_build_free(nr_builder *bd);

#ifdef __cplusplus
}
#endif

#endif /* NEUROUTE_BUILD_H */
