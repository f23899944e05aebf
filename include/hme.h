/*
 * hme.h -- C ABI of the GB300 (sm_103a) gater library for hard mixtures of
 * experts (Gross, Ranzato, Szlam, "Hard Mixtures of Experts for Large Scale
 * Weakly Supervised Vision", arXiv 1704.06363).
 *
 * The gater of Section 2: K-means clustering of feature vectors z_j
 * (Lloyd iterations), the hard assignment of Eq. 2
 *     T(x)_i = 1  iff  i = argmin_j || z(x) - c_j ||_2 ,
 * and the split of the training set into per-expert shares ("each on its own
 * share of the training data", with no balancing of cluster sizes).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Every function returns an int status: HME_OK (0) or one of the HME_E*
 *   codes below.  On error nothing has been launched, and hme_last_error()
 *   returns a message (thread-local, valid until the next call on the thread).
 * - All array arguments are caller-owned DEVICE pointers (allocated by the
 *   caller, e.g. with torch).  The library allocates no device memory: all
 *   scratch lives in the caller's workspace `ws` of `ws_bytes` bytes, sized by
 *   hme_workspace_bytes().  ws must be 256-byte aligned.
 * - Work is enqueued asynchronously on `stream` (a cudaStream_t passed as
 *   void*; NULL = the legacy default stream).  Arguments are checked on the
 *   host before any launch.  Conditions only the device can see (a label out of
 *   range, a bounded device wait that expired) are recorded in a status word
 *   inside ws; hme_sync_status() waits for the stream and reports it.  Each
 *   call clears that word when it starts, so it reports on the last call made
 *   with that workspace.
 * - Feature matrices are row-major, N rows of d elements, row stride `ldx`
 *   elements (ldx >= d), element type HME_F32 (float) or HME_BF16 (bfloat16).
 *   For HME_BF16 the rows are read by TMA: the base must be 16-byte aligned and
 *   ldx * 2 a multiple of 16 bytes, otherwise HME_EINVAL.
 * - Centres C are K x d float32, row-major, contiguous (row stride d).
 * - Limits: 1 <= d <= 16384, 1 <= K <= 16384, 0 <= N < 2^31.
 * - All entry points may be called from several host threads on different
 *   workspaces; calls sharing one workspace must be ordered on one stream.
 */
#ifndef HME_H
#define HME_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define HME_API __attribute__((visibility("default")))
#else
#define HME_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ---------------------------------------------------- */
#define HME_OK 0
#define HME_EINVAL 1    /* bad argument (pointer, size, alignment, label range) */
#define HME_ENOMEM 2    /* ws_bytes smaller than hme_workspace_bytes() */
#define HME_ECUDA 3     /* a CUDA runtime or driver call failed */
#define HME_ETIMEOUT 4  /* a bounded device-side wait expired (see hme_sync_status) */
#define HME_EINTERNAL 5 /* internal inconsistency */

/* ---- element types of feature matrices ------------------------------- */
#define HME_F32 0
#define HME_BF16 1

/* ---- operations, for hme_workspace_bytes ----------------------------- */
#define HME_OP_INIT 0      /* hme_kmeans_init */
#define HME_OP_ASSIGN 1    /* hme_prepare_features, hme_assign, hme_update_centroids */
#define HME_OP_PARTITION 2 /* hme_partition (d and dtype ignored) */
#define HME_OP_ROUTE 3     /* hme_route */
#define HME_OP_TAG_HIST 4  /* hme_tag_cluster_hist (d = vocabulary size V; dtype ignored) */
#define HME_OP_STREAM 5    /* hme_kmeans_stream (N = chunk_rows) */
#define HME_OP_PCA 6       /* hme_pca_covariance, hme_pca_fit (K = r components); N = 0: hme_pca_transform only */

/* ---- k-means++ seeding variants -------------------------------------- */
#define HME_INIT_KMEANSPP 0           /* candidates = all N rows */
#define HME_INIT_KMEANSPP_SUBSAMPLE 1 /* candidates = min(N, 256 K) rows drawn with replacement */

/* ---- hme_assign flags ------------------------------------------------- */
#define HME_ASSIGN_DEFAULT 0
#define HME_ASSIGN_PREPARED 1 /* ws already holds this X, prepared by hme_prepare_features */
/* Not with HME_ASSIGN_PREPARED: the call also leaves this X prepared in ws, as
 * hme_prepare_features would, so that later calls can pass HME_ASSIGN_PREPARED.
 * An in-kernel split (see hme_prepare_features) writes the split rows as it
 * makes them: the first Lloyd iteration reads X once instead of twice. */
#define HME_ASSIGN_PREPARE_OUT 2
/* HME_F32 features with K > 256 and rows TMA can read (X on a 16-byte
 * boundary, ldx % 4 == 0): multiply x and c as tf32 operands (one product)
 * instead of the three products of the bf16 split; ignored otherwise.  The
 * wider operand error (see hme_assign) makes near ties, and so exact
 * re-scores, more frequent: on the 1.6e7 x 512, K = 1024 feature set at its
 * k-means++ centres the split was measured faster, so it is the default. */
#define HME_ASSIGN_TF32 4

/*
 * hme_workspace_bytes -- bytes of scratch an operation needs.
 * op is one of HME_OP_*; N is the number of rows (B for HME_OP_ROUTE).  The
 * HME_OP_ASSIGN size serves hme_prepare_features, hme_assign and
 * hme_update_centroids on the same (N, d, K, dtype), so one workspace can carry
 * prepared features from one Lloyd iteration to the next.  Returns 0 for
 * invalid arguments.
 */
HME_API size_t hme_workspace_bytes(int32_t op, int64_t N, int32_t d, int32_t K, int32_t dtype);

/* Message describing the last failed call on this host thread ("" if none). */
HME_API const char *hme_last_error(void);

/*
 * hme_sync_status -- wait for `stream`, then return the device-side status of
 * the last call made with workspace `ws`: HME_OK, HME_EINVAL (a label outside
 * [0, K) was seen and skipped), HME_ETIMEOUT (a bounded wait expired; outputs
 * of that call are undefined) or HME_ECUDA (an asynchronous CUDA error).
 */
HME_API int hme_sync_status(void *ws, void *stream);

/*
 * hme_kmeans_init -- k-means++ seeding (Arthur & Vassilvitskii 2007) of the
 * centres that Section 2 obtains by "K-means clustering" of the z_j; the paper
 * names no initialisation, so this is a stated reading.
 *   Candidates: all N rows (HME_INIT_KMEANSPP) or m = min(N, 256 K) rows
 *   (HME_INIT_KMEANSPP_SUBSAMPLE), candidate j = row floor(u_j N) with u_j from
 *   splitmix64 output j of (seed ^ 0xD1B54A32D192ED03).
 *   Picks use splitmix64 outputs 0, 1, ... of `seed`, u = top 53 bits / 2^53:
 *   the first centre is candidate floor(u m); each later centre is the
 *   smallest candidate whose running total of D^2 exceeds u * sum(D^2), where
 *   D^2 (fp64) is the squared distance to the nearest centre chosen so far; if
 *   that sum is 0, candidate floor(u m).
 * X: N x d (ldx, dtype), read only.  C_out: K x d float32, written (each row a
 * copy of a row of X).  Requires N >= 1.  Not on the timed Lloyd path: it
 * makes about 2K kernel launches.
 * Errors: HME_EINVAL for N < 1, an unknown method, sizes outside the limits, a
 * NULL X or C_out; HME_ENOMEM for a workspace smaller than
 * hme_workspace_bytes(HME_OP_INIT, ...).
 */
HME_API int hme_kmeans_init(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, int32_t K,
                    uint64_t seed, int32_t method, float *C_out, void *ws, size_t ws_bytes, void *stream);

/*
 * hme_prepare_features -- once per feature set: squared row norms ||x_i||^2
 * (fp32) and, for HME_F32, the split of every element into two bf16 parts
 * x = hi + lo + O(2^-16 |x|) that the tensor-core assign step consumes (the
 * norms are then those of hi + lo).  Writes
 * ws only.  Pass HME_ASSIGN_PREPARED to hme_assign to reuse it for every
 * iteration; the (N, d, K, dtype) of the later calls must be the same.
 * Without HME_ASSIGN_PREPARED, hme_assign and hme_route on HME_F32 features
 * with K <= 256 whose rows TMA can read (X on a 16-byte boundary,
 * ldx % 4 == 0) split each fp32 row inside the kernel as it arrives: one pass
 * over X instead of three for a one-off call.  With it they read the prepared
 * split, which streams faster when the same X is assigned many times.  (The
 * split and the norms are this library's evaluation of Eq. 2's distances,
 * not a step of the paper.)
 * Errors: HME_EINVAL for sizes outside the limits or a NULL or misaligned X;
 * HME_ENOMEM for a workspace smaller than hme_workspace_bytes(HME_OP_ASSIGN, ...).
 */
HME_API int hme_prepare_features(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, int32_t K,
                         void *ws, size_t ws_bytes, void *stream);

/*
 * hme_assign -- Eq. 2 (Section 2) for every row of X:
 *   labels_out[i] = argmin_k ||x_i - c_k||^2 , ties to the lowest k,
 *   mind_out[i]   = ||x_i - c_{labels[i]}||^2 (float32, >= 0)      (may be NULL),
 *   *objective_out = sum_i mind[i] in fp64 (one device double)     (may be NULL);
 *                   a tensor-core estimate: its fp32 accumulation is biased
 *                   by up to about (d/16) * nprod * 2^-24 (||x||^2 + ||c||^2)
 *                   per row; hme_update_centroids returns the exact J.
 * The distance is ||x||^2 - 2 x.c + ||c||^2 with x.c on the tcgen05 tensor
 * cores (fp32 accumulate): for HME_BF16 features, x.bf16(c) with c rounded to
 * bf16 (round to nearest even); for HME_F32 with HME_ASSIGN_TF32 (K > 256,
 * rows TMA can read), x as tf32 (10-bit significand, |x - x'| <= 2^-10 |x|)
 * against c rounded to tf32 (|c - c'| <= 2^-11 |c|), one product, with
 * ||c||^2 of the fp32 centres and ||x||^2 of the fp32 rows (with
 * HME_ASSIGN_PREPARED, the prepared norms); otherwise for HME_F32 the bf16
 * split x = xh + xl, c = ch + cl and the three products
 * xh.ch + xh.cl + xl.ch (nprod = 3; the dropped xl.cl is at most
 * 2^-16 (1 + 2^-8)^2 ||x|| ||c||), with the norms taken of the same split
 * values.  A row whose runner-up distance is within E of its best, E a bound
 * on the error of a difference of two computed distances
 * (steps * nprod * 2^-22 (||x||^2 + max_k ||c_k||^2), steps = ceil(d/16), or
 * ceil(d/8) for tf32 operands; plus, for split fp32 operands,
 * 2^-14 (||x|| + max ||c||) sqrt(D2) and 1.0625 * 2^-14 ||x|| max ||c||; for
 * tf32 operands 6.002 * 2^-10 ||x|| max ||c||), is re-scored
 * exactly on its candidates (all K when a third centre is also within E) with
 * direct differences, sum_j (x_j - c_j)^2 in fp32 (a sum of non-negative
 * terms).  The N x K distance matrix is never written.
 * X: N x d (ldx, dtype); C: K x d float32 (read only); labels_out: int32[N].
 * flags: HME_ASSIGN_DEFAULT, HME_ASSIGN_PREPARE_OUT (also leave X prepared in
 * ws), or HME_ASSIGN_PREPARED (skip the per-call hme_prepare_features pass; ws
 * must hold this X's preparation); PREPARED and PREPARE_OUT at once:
 * HME_EINVAL.  Either may be combined with HME_ASSIGN_TF32.
 */
HME_API int hme_assign(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, const float *C, int32_t K,
               int32_t flags, int32_t *labels_out, float *mind_out, double *objective_out,
               void *ws, size_t ws_bytes, void *stream);

/*
 * hme_assign_rows -- hme_assign (Eq. 2, Section 2) of rows [row0, row1) of an
 * N-row feature set, so that the assignment of a set can start on its first
 * rows while later ones are still being copied in (the first Lloyd iteration
 * of a set held in host memory: copy chunk j + 1 while chunk j is assigned).
 * X points to row 0 of all N rows; only rows [row0, row1) are read.
 * labels_out and mind_out (may be NULL) point to N-entry arrays; entries
 * [row0, row1) are written.  ws is an HME_OP_ASSIGN workspace for all N rows:
 * with HME_ASSIGN_PREPARE_OUT the preparation of these rows is left at their
 * place in it, so that once every row has been assigned this way, later
 * hme_assign calls on the whole set may pass HME_ASSIGN_PREPARED; with
 * HME_ASSIGN_PREPARED these rows must have been prepared.  *objective_out
 * (may be NULL) = the sum of mind over these rows.  Calls on one workspace
 * must be ordered on one stream (they share its queues and header).
 * Errors: as hme_assign, and HME_EINVAL unless 0 <= row0 <= row1 <= N.
 */
HME_API int hme_assign_rows(const void *X, int64_t N, int64_t row0, int64_t row1, int32_t d, int64_t ldx,
                            int32_t dtype, const float *C, int32_t K, int32_t flags, int32_t *labels_out,
                            float *mind_out, double *objective_out, void *ws, size_t ws_bytes, void *stream);

/*
 * hme_update_centroids -- the K-means centre step (Section 2, "K-means
 * clustering" of the z_j):
 *   counts_out[k] = |{i : labels[i] = k}| (int64, may be NULL),
 *   C_inout[k]    = (sum_{labels[i]=k} x_i) / counts[k] (fp64 sums, stored as
 *                   float32),
 *   *objective_out = sum_i ||x_i - c_{labels[i]}||^2 for the centres as they
 *                   were on entry (bf16-rounded for HME_BF16 features, as in
 *                   hme_assign), evaluated in fp64 as sum ||x||^2
 *                   - 2 sum_k c_k . S_k + sum_k n_k ||c_k||^2 from the
 *                   per-cluster sums S_k (one device double, may be NULL).
 *                   With the labels of the preceding hme_assign this is the
 *                   Lloyd objective J_t.
 * The per-cluster sums, counts and sum ||x||^2 stay in ws after the call.
 * prev_labels == NULL: they are recomputed from all N rows (segmented sums in
 * label order).  prev_labels != NULL: ws must hold the state left by the
 * previous hme_update_centroids call on the same X and ws, made with labels
 * equal to prev_labels (and no other call with this ws in between but
 * hme_assign / hme_prepare_features); only rows whose label differs from
 * prev_labels are read and moved between clusters.  Both give Lloyd's centres
 * (the same sums up to fp64 rounding order).
 * Empty clusters (the paper is silent; Section 4.5 reports every cluster used)
 * are re-seeded in ascending k: each takes the not-yet-taken row with the
 * largest mind[i], ties to the lowest i, as its centre (copied exactly); that
 * row stays counted in its own cluster.  mind may be NULL (then the lowest
 * untaken rows).  When every row is taken, a remaining empty centre is kept.
 * *n_reseeded_out (device int32, may be NULL) = clusters re-seeded.
 * Labels outside [0, K) are skipped and reported by hme_sync_status.
 * Errors: HME_EINVAL for sizes outside the limits, a NULL X, C_inout or (N > 0)
 * labels; HME_ENOMEM for a workspace smaller than hme_workspace_bytes(HME_OP_ASSIGN, ...).
 */
HME_API int hme_update_centroids(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype,
                                 const int32_t *labels, const int32_t *prev_labels, const float *mind, int32_t K,
                                 float *C_inout, int64_t *counts_out, int32_t *n_reseeded_out,
                                 double *objective_out, void *ws, size_t ws_bytes, void *stream);

/*
 * hme_partition -- each expert's share of the training set (Section 2: "each
 * on its own share"; no balancing, so buckets may be very unequal):
 *   hist_out[k]        = |{i : labels[i] = k}|                     (int64[K]),
 *   offsets_out        = exclusive prefix sum of hist              (int64[K+1]),
 *   perm_out[offsets[labels[i]] + |{j < i : labels[j] = labels[i]}|] = i
 *                        (a stable counting sort; int32[N]),
 *   sorted_labels_out[s] = labels[perm[s]]                         (int32[N], may be NULL).
 * Optional CSR multilabel lists (tag_off int64[N+1], tags int32[tag_off[N]])
 * move with their point: tag_off_out int64[N+1] and tags_out int32[tag_off[N]]
 * (all four NULL, or all four set).  Bit-exact; integer work only.
 * Labels outside [0, K) are skipped and reported by hme_sync_status.
 */
HME_API int hme_partition(const int32_t *labels, int64_t N, int32_t K, int64_t *hist_out, int64_t *offsets_out,
                  int32_t *perm_out, int32_t *sorted_labels_out, const int64_t *tag_off, const int32_t *tags,
                  int64_t *tag_off_out, int32_t *tags_out, void *ws, size_t ws_bytes, void *stream);

/*
 * hme_route -- evaluation-time gating (Section 2.1: the cost of an output is
 * the cost of T(x) plus one expert H_i(x)): Eq. 2 on a batch Q (B x d) with
 * frozen centres C, then the partition of its labels, so that each expert
 * receives a contiguous run of rows:
 *   expert_out[b] = label of Q row b (int32[B]), offsets_out (int64[K+1]),
 *   order_out (int32[B]) = rows of Q grouped by expert, ascending within one.
 * flags: HME_ASSIGN_DEFAULT, HME_ASSIGN_PREPARE_OUT, or HME_ASSIGN_PREPARED
 * when ws already holds Q prepared by hme_prepare_features or a PREPARE_OUT
 * call (e.g. routing the training set with the workspace of the Lloyd loop:
 * HME_OP_ROUTE and HME_OP_ASSIGN sizes agree).
 * Batches of at most 16384 rows: from the second call with the same
 * arguments (every pointer, size and flag, and the stream) on, the call's
 * launches are replayed as one CUDA graph captured at that second call (the
 * data behind the pointers may change freely between calls; it is read when
 * the graph runs).  Up to 8 argument sets are kept, the least recently used
 * replaced; a kept graph is used only in the CUDA context it was captured in.
 * The environment variable HME_NO_GRAPHS=1 turns this off.
 * Errors: HME_EINVAL for sizes outside the limits, a NULL or misaligned Q, a
 * NULL C or offsets_out, a NULL expert_out / order_out with B > 0, unknown or
 * conflicting flags; HME_ENOMEM for a workspace smaller than
 * hme_workspace_bytes(HME_OP_ROUTE, ...).
 */
HME_API int hme_route(const void *Q, int64_t B, int32_t d, int64_t ldq, int32_t dtype, const float *C, int32_t K,
                      int32_t flags, int32_t *expert_out, int64_t *offsets_out, int32_t *order_out, void *ws,
                      size_t ws_bytes, void *stream);

/*
 * hme_kmeans_stream -- Lloyd's iterations (Section 2, "K-means clustering")
 * for a feature set that stays outside HBM: X lives in page-locked host
 * memory (or anywhere device-accessible) and is streamed through two device
 * buffers of chunk_rows rows, the copy of one chunk overlapping the
 * clustering of the previous one.  Each of the `iters` iterations assigns
 * every chunk against the centres C_t (as hme_assign: Eq. 2, near ties
 * re-scored exactly), adds the chunk's rows to the fp64 per-cluster sums (as
 * hme_update_centroids' full pass), and then forms, from all N rows:
 *   objectives_out[t] = J(C_t, labels) in fp64               (may be NULL),
 *   C_inout = the new centres (S_k / n_k; the re-seed rule for empty
 *             clusters, whose picked rows are read from X in place),
 *   counts_out[k], *n_reseeded_out as hme_update_centroids   (may be NULL).
 * labels_out int32[N] and mind_out float32[N] (device memory) hold the last
 * iteration's assignment and distances.  The result is Lloyd's iteration
 * on all N rows; only the fp64 summation order differs from the in-HBM path.
 * X: N x d (ldx, dtype).  ws: hme_workspace_bytes(HME_OP_STREAM, chunk_rows,
 * d, K, dtype) bytes of device memory.  The call creates one stream and four
 * events of its own for the copies (so it cannot be captured into a graph);
 * the caller's stream is ordered after all of its work.
 * Errors: HME_EINVAL for N < 1, iters < 0, chunk_rows < 1, ldx < d, sizes
 * outside the limits, a NULL X, C_inout, labels_out or mind_out, X in pageable
 * host memory, a NULL or misaligned ws; HME_ENOMEM for a workspace smaller than
 * hme_workspace_bytes(HME_OP_STREAM, chunk_rows, ...); HME_ECUDA when creating
 * the copy stream or events or a copy fails.
 */
HME_API int hme_kmeans_stream(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, int32_t K,
                              int32_t iters, int64_t chunk_rows, float *C_inout, int32_t *labels_out, float *mind_out,
                              double *objectives_out, int64_t *counts_out, int32_t *n_reseeded_out, void *ws,
                              size_t ws_bytes, void *stream);

/*
 * hme_tag_cluster_hist -- the tag statistics of a clustering that Section 4.5
 * ("Analysis of YFCC100M clusters") reports: for every cluster k and tag t
 *   counts_out[k * V + t] = the number of times t occurs among the tags of the
 *                           points of cluster k (int64, K x V row-major: the
 *                           bars of the tag-over-cluster histograms),
 * and for every tag, with c(t) = counts[:, t] its distribution over clusters,
 *   sparsity_out[t] = ||c(t)||_1 / ||c(t)||_2 in fp64 (between 1 and
 *                     sqrt(K); 0 for a tag that never occurs)    (may be NULL).
 * Input is the partitioned form that hme_partition writes: offsets: int64[K+1]
 * point offsets of the clusters (offsets_out); tag_off: int64[N+1] and tags:
 * int32[tag_off[N]], the tag lists in that point order (tag_off_out,
 * tags_out), so each cluster's tags are one contiguous range.  Tags outside
 * [0, V) are skipped and reported by hme_sync_status (HME_EINVAL).  Integer
 * counts are exact; the ratio is the fp64 one of those counts.
 * ws: hme_workspace_bytes(HME_OP_TAG_HIST, N, V, K, 0) bytes.  All pointers
 * are device memory; asynchronous on stream.
 */
HME_API int hme_tag_cluster_hist(const int64_t *offsets, const int64_t *tag_off, const int32_t *tags, int64_t N,
                                 int32_t K, int32_t V, int64_t *counts_out, double *sparsity_out, void *ws,
                                 size_t ws_bytes, void *stream);

/*
 * hme_partition_noalloc -- the same stable partition as hme_partition (same
 * outputs, bit for bit; no tag lists) for callers that cannot allocate device
 * memory: code that must not call cudaMalloc/cudaFree where it routes a batch
 * (they can synchronise the whole device, e.g. a serving loop), or code whose
 * device memory is entirely owned by another framework's pool.  The paper has
 * no counterpart; this is a deployment convenience.
 *   No workspace: the scratch (status word + per-tile bucket counts) is a fixed
 *   16 MiB array in device memory that every GPU loading the library holds
 *   until exit.  The first call on a device, with that device current, looks up
 *   the array's address (cudaGetSymbolAddress); make that first call before any
 *   stream capture.  Calls share the array: calls that overlap on the GPU (two
 *   streams, two host threads) race and must not be issued.  The tile length
 *   grows so the counts fit; a size that still does not fit returns HME_EINVAL.
 *   *status_out (device int32, may be NULL) = 0, or 1 if a label outside
 *   [0, K) was seen and skipped.  Calls no cudaMalloc, cudaFree or allocating
 *   library routine.
 */
HME_API int hme_partition_noalloc(const int32_t *labels, int64_t N, int32_t K, int64_t *hist_out,
                                  int64_t *offsets_out, int32_t *perm_out, int32_t *sorted_labels_out,
                                  int32_t *status_out, void *stream);

/*
 * PCA before the gater (Section 4.2, "Model and training details": the gater
 * features Z = T^{L-1}(X) are projected onto their first 256 PCA dimensions
 * before the K-means).  The paper names the method and the dimension only;
 * readings: centred about the column mean, covariance normalised by N,
 * unwhitened projection, components in decreasing variance, each signed so
 * that its entry of largest magnitude (lowest index among equals) is positive.
 * fp32 features only (dtype HME_F32; anything else is HME_EINVAL).
 *
 * hme_pca_covariance -- mean_out[j] = (1/N) sum_i x_ij (fp64, d entries) and
 *   cov_out = (1/N) sum_i (x_i - mu)(x_i - mu)^T (fp64, d x d row-major, both
 *   triangles).  The centred values y = x - fp32(mu) are split into bf16
 *   y = yh + yl (|y - yh - yl| <= 2^-16 |y|) and the products
 *   yh yh' + yh yl' + yl yh' are summed on the tensor cores in fp32 over 512
 *   rows at a time (96 accumulation steps), up to 16 of those sums in fp32
 *   (round to nearest), and those in fp64, so that each entry is within
 *   (3 * 2^-16 + 98 * 2^-23 + 18 * 2^-24) (1/N) sum_i (|y_ia| + |mu_a|)
 *   (|y_ib| + |mu_b|) of the exact value (2^-23 per tensor-core step: one
 *   ulp, whatever the accumulator's rounding).  Requires N >= 1.
 *
 * hme_pca_fit -- the covariance as above, then its eigendecomposition by
 *   cyclic Jacobi in fp32 (until the off-diagonal norm is at most 2^-20 of
 *   the Frobenius norm, or stagnates below 2^-16 of it), then
 *   mean_out (fp32, d), components_out (fp32, r x d row-major, orthonormal
 *   rows), variances_out (fp32, r, the eigenvalues; may be NULL) and
 *   *sweeps_out (host int32, the Jacobi sweeps made; may be NULL).
 *   Synchronises `stream` once per sweep.  1 <= r <= d.  A matrix that does
 *   not converge in 40 sweeps returns HME_EINTERNAL.
 *
 * hme_pca_transform -- Z_out[i * ldz + j] = components_j . (x_i - mean)
 *   (fp32, N x r, ldz >= r): the assign kernel that splits fp32 rows inside
 *   the kernel, the components as its centres (bf16 hi/lo, three products),
 *   and mean.components_j (fp64, stored fp32) subtracted in the epilogue.
 *   1 <= r <= 256; X on a 16-byte boundary with ldx % 4 == 0 (TMA).
 *   Workspace: hme_workspace_bytes(HME_OP_PCA, 0, d, r, HME_F32) or larger.
 *
 * Errors of all three: HME_EINVAL for a dtype other than HME_F32, sizes
 * outside the limits or the bounds above (hme_pca_fit: d <= 8192), NULL
 * outputs, ldz < r, a misaligned X (hme_pca_transform); HME_ENOMEM for a
 * workspace smaller than hme_workspace_bytes(HME_OP_PCA, ...); HME_EINTERNAL
 * as above.
 */
HME_API int hme_pca_covariance(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, double *mean_out,
                               double *cov_out, void *ws, size_t ws_bytes, void *stream);
HME_API int hme_pca_fit(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, int32_t r, float *mean_out,
                        float *components_out, float *variances_out, int32_t *sweeps_out, void *ws, size_t ws_bytes,
                        void *stream);
HME_API int hme_pca_transform(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, const float *mean,
                              const float *components, int32_t r, float *Z_out, int64_t ldz, void *ws,
                              size_t ws_bytes, void *stream);

/* Number of kernels this library has launched in this process (diagnostic). */
HME_API int64_t hme_launch_count(void);

/*
 * hme_debug_bounded_wait -- test hook for the device-side bounded wait that
 * every pipeline wait in this library uses: launches one CTA that waits on a
 * shared-memory barrier nothing completes, with a limit of timeout_ns
 * nanoseconds (1 .. 10^9).  hme_sync_status(ws, stream) then returns
 * HME_ETIMEOUT and the context stays usable.
 */
HME_API int hme_debug_bounded_wait(uint64_t timeout_ns, void *ws, size_t ws_bytes, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* HME_H */
