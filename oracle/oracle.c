/*
 * oracle.c -- plain, slow, fp64 CPU oracle for the gater of
 * "Hard Mixtures of Experts for Large Scale Weakly Supervised Vision"
 * (Gross, Ranzato, Szlam; arXiv 1704.06363).
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load this library.  It shares
 * no code, header, table or helper with the CUDA path in
 * paper_1704_06363_gb300/, and it never calls into it.
 *
 * What the paper fixes (Section 2, "Models"):
 *   - the gater's centres c_1..c_K come from K-means clustering of the
 *     last-hidden-layer features z_j of every training point;
 *   - Eq. 2: T(x)_i = 1 iff i = argmin_j ||z(x) - c_j||_2, one expert per point;
 *   - no attempt is made to balance the number of points per cluster;
 *   - each expert is trained on its own share of the training data.
 * Section 4.2 fixes K = 50 on 256-dimensional PCA features; Section 4.5 shows
 * unbalanced cluster sizes with every cluster used.
 *
 * Everything the paper leaves open is a stated reading:
 *   init = k-means++ (Arthur & Vassilvitskii 2007) driven by splitmix64
 *   (Steele, Lea, Flood 2014); a fixed number of Lloyd iterations; ties in the
 *   argmin go to the lowest centre index; the argmin is taken on the squared
 *   distance (same minimiser as the unsquared norm); an empty cluster takes
 *   the farthest remaining point of the current assignment; buckets list their
 *   points in ascending index order; bf16 feature sets are assigned against
 *   the centres rounded to bf16 (round to nearest even).
 *
 * All distances are the direct sum of squared differences in fp64, with no
 * norm expansion, no blocking and no reordering.  Every function is a
 * straight transcription of the definition it cites.
 *
 * Parity status: every function below is pinned by tests/test_oracle_pins.py
 * (brute force, 1-D dynamic programming optimum, closed forms, invariants,
 * library routines, the published splitmix64 vector).
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <math.h>

#define ORC_F32 0
#define ORC_BF16 1

/* ---------------------------------------------------------------------- */
/* Random numbers: splitmix64 (Steele, Lea, Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014).  Output number j (j = 0, 1,
 * ...) of the generator seeded with s is mix(s + (j + 1) * gamma), so the
 * sequence can be indexed directly by a counter.                          */
/* ---------------------------------------------------------------------- */
static const uint64_t SM64_GAMMA = 0x9E3779B97F4A7C15ull;

uint64_t orc_splitmix64_at(uint64_t seed, uint64_t j)
{
    uint64_t z = seed + (j + 1) * SM64_GAMMA;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

/* u in [0,1) from the top 53 bits of r. */
double orc_unit(uint64_t r)
{
    return (double)(r >> 11) * (1.0 / 9007199254740992.0);
}

/* floor(u * n) for u = orc_unit(r), in exact integer arithmetic:
 * (top 53 bits of r) * n / 2^53. */
uint64_t orc_scaled_index(uint64_t r, uint64_t n)
{
    unsigned __int128 p = (unsigned __int128)(r >> 11) * (unsigned __int128)n;
    return (uint64_t)(p >> 53);
}

/* Domain constant separating the subsample stream from the pick stream. */
static const uint64_t SUBSAMPLE_STREAM = 0xD1B54A32D192ED03ull;

/* ---------------------------------------------------------------------- */
/* bf16: the top 16 bits of an IEEE binary32, rounded to nearest even.     */
/* ---------------------------------------------------------------------- */
uint16_t orc_f32_to_bf16_rne(float f)
{
    uint32_t u;
    memcpy(&u, &f, 4);
    if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu) != 0)
        return (uint16_t)((u >> 16) | 0x0040u); /* NaN stays NaN (quiet) */
    uint32_t lsb = (u >> 16) & 1u;
    u += 0x7FFFu + lsb;
    return (uint16_t)(u >> 16);
}

float orc_bf16_to_f32(uint16_t b)
{
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, 4);
    return f;
}

/* Element (i, j) of a row-major feature matrix with row stride ldx elements. */
static double feat(const void *X, int dtype, int64_t ldx, int64_t i, int64_t j)
{
    if (dtype == ORC_BF16)
        return (double)orc_bf16_to_f32(((const uint16_t *)X)[i * ldx + j]);
    return (double)((const float *)X)[i * ldx + j];
}

/* The centre coordinates the assign step compares against, as fp64: the stored
 * fp32 values, or their bf16 rounding when the features are bf16.  Returns a
 * malloc'd K x d table (NULL on allocation failure). */
static double *centre_table(const float *C, int64_t K, int64_t d, int dtype)
{
    double *T = (double *)malloc((size_t)(K * d > 0 ? K * d : 1) * sizeof(double));
    if (!T)
        return NULL;
    for (int64_t i = 0; i < K * d; ++i) {
        float c = C[i];
        T[i] = (dtype == ORC_BF16) ? (double)orc_bf16_to_f32(orc_f32_to_bf16_rne(c)) : (double)c;
    }
    return T;
}

/* ||x_i - y||^2 by the direct sum, j ascending, fp64. */
static double dist2_row_row(const void *X, int dtype, int64_t ldx, int64_t d,
                            int64_t i, int64_t i2)
{
    double s = 0.0;
    for (int64_t j = 0; j < d; ++j) {
        double t = feat(X, dtype, ldx, i, j) - feat(X, dtype, ldx, i2, j);
        s += t * t;
    }
    return s;
}

/* ---------------------------------------------------------------------- */
/* k-means++ seeding (Arthur & Vassilvitskii 2007).  The paper says only    */
/* "K-means clustering" (Section 2) and does not name an initialisation.    */
/*                                                                          */
/* Candidate rows: all N rows, or (subsample != 0) m = min(N, 256 K) rows   */
/* drawn with replacement, row r_j = floor(u * N) with u from splitmix64    */
/* output j of seed ^ SUBSAMPLE_STREAM.                                     */
/* Picks use splitmix64 outputs 0, 1, 2, ... of seed:                       */
/*   first centre: candidate floor(u * m);                                  */
/*   next centres: the smallest candidate j whose running total of D^2      */
/*   (in candidate order) exceeds u * (sum of D^2), D^2 = squared distance  */
/*   to the nearest centre chosen so far; if the sum is 0, floor(u * m).    */
/* C_out[k] is the chosen row (exact in fp32).  picked_out[k] = its row.    */
/* Returns 0, or -1 on bad arguments / allocation failure.                  */
/* ---------------------------------------------------------------------- */
int orc_kmeanspp(const void *X, int64_t N, int64_t d, int64_t ldx, int dtype,
                 int64_t K, uint64_t seed, int subsample,
                 float *C_out, int64_t *picked_out)
{
    if (N <= 0 || d <= 0 || K <= 0 || ldx < d)
        return -1;
    int64_t m = N;
    if (subsample && N > 256 * K)
        m = 256 * K;
    int64_t *rows = (int64_t *)malloc((size_t)m * sizeof(int64_t));
    double *D2 = (double *)malloc((size_t)m * sizeof(double));
    if (!rows || !D2) {
        free(rows);
        free(D2);
        return -1;
    }
    for (int64_t j = 0; j < m; ++j)
        rows[j] = (m == N) ? j
                           : (int64_t)orc_scaled_index(
                                 orc_splitmix64_at(seed ^ SUBSAMPLE_STREAM, (uint64_t)j), (uint64_t)N);

    uint64_t ctr = 0;
    int64_t pick = (int64_t)orc_scaled_index(orc_splitmix64_at(seed, ctr++), (uint64_t)m);
    for (int64_t k = 0; k < K; ++k) {
        if (k > 0) {
            double total = 0.0;
            for (int64_t j = 0; j < m; ++j)
                total += D2[j];
            uint64_t r = orc_splitmix64_at(seed, ctr++);
            if (total > 0.0) {
                double thr = orc_unit(r) * total;
                double run = 0.0;
                pick = -1;
                for (int64_t j = 0; j < m; ++j) {
                    run += D2[j];
                    if (run > thr) {
                        pick = j;
                        break;
                    }
                }
                if (pick < 0) { /* thr rounded past the last total: last positive */
                    for (int64_t j = m - 1; j >= 0; --j)
                        if (D2[j] > 0.0) {
                            pick = j;
                            break;
                        }
                }
            } else {
                pick = (int64_t)orc_scaled_index(r, (uint64_t)m);
            }
        }
        int64_t row = rows[pick];
        if (picked_out)
            picked_out[k] = row;
        for (int64_t j = 0; j < d; ++j)
            C_out[k * d + j] = (float)feat(X, dtype, ldx, row, j);
#pragma omp parallel for schedule(static)
        for (int64_t j = 0; j < m; ++j) {
            double dj = dist2_row_row(X, dtype, ldx, d, rows[j], row);
            if (k == 0 || dj < D2[j])
                D2[j] = dj;
        }
    }
    free(rows);
    free(D2);
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Assign (Eq. 2, Section 2): a_i = argmin_k ||x_i - c_k||.  The squared   */
/* distance D_ik = sum_j (x_ij - c_kj)^2 is summed directly in fp64; ties   */
/* go to the lowest k.  d1[i] = D_{i,a_i}, d2[i] = the second smallest      */
/* D_ik over k (equal to d1 when two centres tie; +inf when K = 1).         */
/* objective = sum_i d1[i], summed in ascending i.  Rows are independent,   */
/* so the loop over i may run on several threads without changing a value. */
/* ---------------------------------------------------------------------- */
int orc_assign(const void *X, int64_t N, int64_t d, int64_t ldx, int dtype,
               const float *C, int64_t K,
               int32_t *labels, double *d1, double *d2, double *objective)
{
    double *Ct = centre_table(C, K, d, dtype);
    if (!Ct)
        return -1;
#pragma omp parallel for schedule(dynamic, 64)
    for (int64_t i = 0; i < N; ++i) {
        double best = INFINITY, second = INFINITY;
        int64_t arg = 0;
        for (int64_t k = 0; k < K; ++k) {
            double s = 0.0;
            for (int64_t j = 0; j < d; ++j) {
                double t = feat(X, dtype, ldx, i, j) - Ct[k * d + j];
                s += t * t;
            }
            if (s < best) {
                second = best;
                best = s;
                arg = k;
            } else if (s < second) {
                second = s;
            }
        }
        labels[i] = (int32_t)arg;
        if (d1)
            d1[i] = best;
        if (d2)
            d2[i] = second;
    }
    if (objective) {
        double J = 0.0;
        if (d1) {
            for (int64_t i = 0; i < N; ++i)
                J += d1[i];
        }
        *objective = J;
    }
    free(Ct);
    return 0;
}

/* ---------------------------------------------------------------------- */
/* The K-means objective of a given assignment: J = sum_i ||x_i - c_{a_i}||^2 */
/* (the quantity Lloyd's iteration decreases), direct fp64 sums in ascending */
/* i and j, against the same centre values as orc_assign.  -1 on a bad label. */
/* ---------------------------------------------------------------------- */
int orc_objective(const void *X, int64_t N, int64_t d, int64_t ldx, int dtype,
                  const float *C, int64_t K, const int32_t *labels, double *objective)
{
    for (int64_t i = 0; i < N; ++i)
        if (labels[i] < 0 || labels[i] >= K)
            return -1;
    double *Ct = centre_table(C, K, d, dtype);
    if (!Ct)
        return -1;
    double J = 0.0;
    for (int64_t i = 0; i < N; ++i) {
        double s = 0.0;
        for (int64_t j = 0; j < d; ++j) {
            double t = feat(X, dtype, ldx, i, j) - Ct[(int64_t)labels[i] * d + j];
            s += t * t;
        }
        J += s;
    }
    free(Ct);
    *objective = J;
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Update (the K-means centre step behind Section 2's "K-means clustering   */
/* on the z_j"): c_k = mean of the x_i with a_i = k, summed in fp64 in       */
/* ascending i and rounded once to fp32.  counts[k] = |{i : a_i = k}|.      */
/* Empty clusters (the paper is silent; in its run every cluster is used,   */
/* Section 4.5): in ascending k, each empty cluster takes the point with the */
/* largest mind[i] (this assignment's distance to its own centre), ties to  */
/* the lowest i, no point twice; that point becomes the centre exactly.     */
/* It stays counted in its old cluster for this update.  When every point   */
/* has been used, a remaining empty cluster keeps its old centre.           */
/* Labels outside [0, K) return -1 and change nothing.                      */
/* ---------------------------------------------------------------------- */
int orc_update(const void *X, int64_t N, int64_t d, int64_t ldx, int dtype,
               const int32_t *labels, const double *mind, int64_t K,
               float *C_inout, int64_t *counts, int32_t *n_reseeded)
{
    for (int64_t i = 0; i < N; ++i)
        if (labels[i] < 0 || labels[i] >= K)
            return -1;
    double *sums = (double *)calloc((size_t)(K * d), sizeof(double));
    unsigned char *used = (unsigned char *)calloc((size_t)(N > 0 ? N : 1), 1);
    if (!sums || !used) {
        free(sums);
        free(used);
        return -1;
    }
    for (int64_t k = 0; k < K; ++k)
        counts[k] = 0;
    for (int64_t i = 0; i < N; ++i) {
        int64_t k = labels[i];
        counts[k] += 1;
        for (int64_t j = 0; j < d; ++j)
            sums[k * d + j] += feat(X, dtype, ldx, i, j);
    }
    for (int64_t k = 0; k < K; ++k)
        if (counts[k] > 0)
            for (int64_t j = 0; j < d; ++j)
                C_inout[k * d + j] = (float)(sums[k * d + j] / (double)counts[k]);

    int32_t reseeded = 0;
    for (int64_t k = 0; k < K; ++k) {
        if (counts[k] != 0)
            continue;
        int64_t far = -1;
        for (int64_t i = 0; i < N; ++i) {
            double mi = mind ? mind[i] : 0.0; /* no distances given: lowest unused i */
            if (!used[i] && (far < 0 || mi > (mind ? mind[far] : 0.0)))
                far = i;
        }
        if (far < 0)
            break; /* every point already used */
        used[far] = 1;
        for (int64_t j = 0; j < d; ++j)
            C_inout[k * d + j] = (float)feat(X, dtype, ldx, far, j);
        reseeded += 1;
    }
    if (n_reseeded)
        *n_reseeded = reseeded;
    free(sums);
    free(used);
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Partition (Section 2: each expert is optimised on its own share of the   */
/* training data; no balancing).  hist[k] = |{i : a_i = k}|,                */
/* offsets = exclusive prefix sum of hist (K + 1 entries), and the bucket   */
/* of expert k lists its points in ascending i:                             */
/*   perm[offsets[a_i] + |{j < i : a_j = a_i}|] = i,  sorted_labels[s] =    */
/*   a_{perm[s]}.                                                           */
/* Optional CSR tag lists (tag_off[N + 1], tags) move with their point:     */
/* slot s receives point perm[s]'s list, tag_off_out = running total.       */
/* Labels outside [0, K) return -1.                                         */
/* ---------------------------------------------------------------------- */
int orc_partition(const int32_t *labels, int64_t N, int64_t K,
                  int64_t *hist, int64_t *offsets, int32_t *perm, int32_t *sorted_labels,
                  const int64_t *tag_off, const int32_t *tags,
                  int64_t *tag_off_out, int32_t *tags_out)
{
    for (int64_t i = 0; i < N; ++i)
        if (labels[i] < 0 || labels[i] >= K)
            return -1;
    for (int64_t k = 0; k < K; ++k)
        hist[k] = 0;
    for (int64_t i = 0; i < N; ++i)
        hist[labels[i]] += 1;
    offsets[0] = 0;
    for (int64_t k = 0; k < K; ++k)
        offsets[k + 1] = offsets[k] + hist[k];
    int64_t *fill = (int64_t *)malloc((size_t)(K > 0 ? K : 1) * sizeof(int64_t));
    if (!fill)
        return -1;
    for (int64_t k = 0; k < K; ++k)
        fill[k] = offsets[k];
    for (int64_t i = 0; i < N; ++i) {
        int64_t s = fill[labels[i]]++;
        perm[s] = (int32_t)i;
        if (sorted_labels)
            sorted_labels[s] = labels[i];
    }
    free(fill);
    if (tag_off && tags && tag_off_out && tags_out) {
        tag_off_out[0] = 0;
        for (int64_t s = 0; s < N; ++s) {
            int64_t p = perm[s];
            int64_t len = tag_off[p + 1] - tag_off[p];
            for (int64_t t = 0; t < len; ++t)
                tags_out[tag_off_out[s] + t] = tags[tag_off[p] + t];
            tag_off_out[s + 1] = tag_off_out[s] + len;
        }
    }
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Tag statistics of a clustering (Section 4.5, "Analysis of YFCC100M       */
/* clusters"): counts[k * V + t] = number of times tag t occurs among the   */
/* tags of the points assigned to cluster k (the bars of the tag-over-      */
/* cluster histograms), and for every tag the sparsity of its distribution  */
/* over clusters c(t) = counts[., t]: ||c(t)||_1 / ||c(t)||_2 (the x axis of */
/* the sparsity-versus-accuracy figure); 0 for a tag that never occurs.     */
/* Straight from the definition: every point, every one of its tags.        */
/* Returns -1 on a label outside [0, K) or a tag outside [0, V).            */
/* ---------------------------------------------------------------------- */
int orc_tag_cluster_hist(const int32_t *labels, int64_t N, int64_t K,
                         const int64_t *tag_off, const int32_t *tags, int64_t V,
                         int64_t *counts, double *sparsity)
{
    for (int64_t i = 0; i < K * V; ++i)
        counts[i] = 0;
    for (int64_t i = 0; i < N; ++i) {
        int32_t k = labels[i];
        if (k < 0 || k >= K)
            return -1;
        for (int64_t j = tag_off[i]; j < tag_off[i + 1]; ++j) {
            int32_t t = tags[j];
            if (t < 0 || t >= V)
                return -1;
            counts[(int64_t)k * V + t] += 1;
        }
    }
    if (sparsity) {
        for (int64_t t = 0; t < V; ++t) {
            double l1 = 0.0, l2sq = 0.0;
            for (int64_t k = 0; k < K; ++k) {
                double c = (double)counts[k * V + t];
                l1 += c;
                l2sq += c * c;
            }
            sparsity[t] = l1 > 0.0 ? l1 / sqrt(l2sq) : 0.0;
        }
    }
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Lloyd's iteration, free running: T times { assign; update }, the gater's */
/* single round of K-means (Section 3 contrasts it with alternating rounds). */
/* objectives[t] = J of the assign step of iteration t; changed[t] = labels  */
/* that differ from iteration t - 1 (N for t = 0).  labels_out holds the    */
/* last assignment (made with the centres that entered the last update).    */
/* ---------------------------------------------------------------------- */
int orc_lloyd(const void *X, int64_t N, int64_t d, int64_t ldx, int dtype,
              float *C_inout, int64_t K, int64_t T,
              int32_t *labels_out, double *objectives, int64_t *changed,
              int64_t *counts_out)
{
    int32_t *prev = (int32_t *)malloc((size_t)(N > 0 ? N : 1) * sizeof(int32_t));
    double *d1 = (double *)malloc((size_t)(N > 0 ? N : 1) * sizeof(double));
    int64_t *counts = (int64_t *)malloc((size_t)(K > 0 ? K : 1) * sizeof(int64_t));
    if (!prev || !d1 || !counts) {
        free(prev);
        free(d1);
        free(counts);
        return -1;
    }
    int rc = 0;
    for (int64_t t = 0; t < T && rc == 0; ++t) {
        double J = 0.0;
        rc = orc_assign(X, N, d, ldx, dtype, C_inout, K, labels_out, d1, NULL, &J);
        if (rc != 0)
            break;
        if (objectives)
            objectives[t] = J;
        if (changed) {
            int64_t c = 0;
            for (int64_t i = 0; i < N; ++i)
                c += (t == 0) || (labels_out[i] != prev[i]);
            changed[t] = c;
        }
        memcpy(prev, labels_out, (size_t)N * sizeof(int32_t));
        int32_t nr = 0;
        rc = orc_update(X, N, d, ldx, dtype, labels_out, d1, K, C_inout, counts, &nr);
    }
    if (counts_out)
        memcpy(counts_out, counts, (size_t)K * sizeof(int64_t));
    free(prev);
    free(d1);
    free(counts);
    return rc;
}
