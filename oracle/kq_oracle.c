/*
 * kq_oracle.c -- plain, slow CPU oracle for the Kernel Quantization (KQ) hot path.
 *
 * TEST INFRASTRUCTURE ONLY. Only the test suite, the smoke check and the CPU
 * baseline leg of the benchmark may load this code. The product path (the CUDA
 * library) shares no code, header, table or helper with it.
 *
 * What it computes (paper: "Kernel Quantization for Efficient Network
 * Compression", arXiv 2003.05148):
 *   - kqo_assign        Sec. 3.1, Eq. 1: every kernel m_i (9 floats) goes to the
 *                       codeword c_k that minimises ||m_i - c_k||^2 (the sets S_k).
 *   - kqo_update        Sec. 3.1, Eq. 1: c_k = mean of S_k, the minimiser of Eq. 1
 *                       for fixed sets; z_k = |S_k|.
 *   - kqo_fit           Sec. 3.1 (k-means in Eq. 1): alternate assign / update.
 *   - kqo_level_fit     Sec. 3.2: 6-bit quantisation of the codebook by k-means over
 *                       all codebook scalars, each weighted by its entry's
 *                       appearance count z_k; then the 6-bit code of every scalar.
 *   - kqo_reconstruct   Sec. 3.2 (testing phase): recover the codebook from the
 *                       codes, then W from the kernel indices.
 *   - kqo_codebook_grad_step  Sec. 3.1, Eq. 2: retraining step of the codebook
 *                       with the element-wise average of the gradients of the
 *                       kernels mapped to each entry.
 *   - kqo_levels_grad_step    Sec. 3.2: the same averaged-gradient step for the
 *                       64 levels of the quantised codebook (average over every
 *                       weight whose value is that level).
 *   - kqo_level_fit_scalars   Sec. 3.2 (last step): 6-bit quantisation of a
 *                       fully-connected layer, the same k-means with weight 1 per
 *                       scalar.
 *
 * Readings where the paper is silent (each is also listed in the design notes):
 *   - Distance arithmetic: fp32, t_j = fl(x_j - c_j), acc = fmaf(t_j, t_j, acc)
 *     for j = 0..8 in that order, starting from acc = 0. The paper stores weights
 *     in fp32 (b_FP = 32, Eq. 5) and fixes no summation order; this one is fixed
 *     so that an argmin decision is taken in the same precision on both sides.
 *   - Argmin ties: strict '<' while scanning k = 0..K-1, so the lowest index wins.
 *     The running best starts at (+inf, 0), so a kernel whose distances are all
 *     +inf or NaN gets index 0.
 *   - Update: sums in fp64 in ascending row order, divided by z_k in fp64, rounded
 *     once to fp32. An empty cluster (z_k = 0) keeps its previous codeword.
 *   - 6-bit level fit: 64 levels initialised to linspace(min, max) over the
 *     scalars whose weight is positive (all scalars if none is); nearest level by
 *     fp32 |v - level|, ties to the lower level; level = weighted mean of its
 *     scalars computed from exact int64 fixed-point sums (scale 2^S, S = 62 - e
 *     where A*M = f * 2^e, f in [0.5, 1), A = total weight, M = max |v| over
 *     weighted scalars); an empty level keeps its value; stop when no code
 *     changes or after max_iters updates.
 *   - Averaged-gradient steps (Eq. 2): the mean gradient is the fp64 sum in
 *     ascending element order divided by the member count in fp64, rounded once
 *     to fp32; then step = fl32(lr * mean) and the new value = fl32(old - step).
 *     An entry (codeword or level) with no members keeps its value. A kernel
 *     whose index is outside [0, K) contributes nothing.
 *   - Fully-connected 6-bit quantisation: the level fit above with every scalar
 *     weighted 1.
 *
 * Build: gcc -O2 -ffp-contract=off -fno-fast-math -fPIC -shared -pthread
 *        kq_oracle.c -o libkq_oracle.so -lm
 * (-ffp-contract=off keeps the compiler from fusing x*y+z anywhere the source
 * did not write fmaf.)
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define KQO_D 9      /* omega^2 for 3x3 kernels */
#define KQO_LEVELS 64 /* 6-bit codebook quantisation */

/* ---------------------------------------------------------------------------
 * Eq. 1 distance, fp32 direct form in the fixed order j = 0..8.
 * ------------------------------------------------------------------------- */
static float dist_f32(const float *x, const float *c) {
    float acc = 0.0f;
    for (int j = 0; j < KQO_D; ++j) {
        float t = x[j] - c[j];
        acc = fmaf(t, t, acc);
    }
    return acc;
}

/* The same distance in fp64 (used only to report how close a decision was). */
static double dist_f64(const float *x, const float *c) {
    double acc = 0.0;
    for (int j = 0; j < KQO_D; ++j) {
        double t = (double)x[j] - (double)c[j];
        acc += t * t;
    }
    return acc;
}

typedef struct {
    const float *W;
    const float *C;
    int32_t K;
    int64_t lo, hi;
    int32_t *idx;
    float *dist;
    double *d1, *d2; /* optional fp64 best and second-best distances */
} assign_job;

static void *assign_rows(void *arg) {
    assign_job *a = (assign_job *)arg;
    for (int64_t i = a->lo; i < a->hi; ++i) {
        const float *x = a->W + i * KQO_D;
        float best = INFINITY;
        int32_t bk = 0;
        for (int32_t k = 0; k < a->K; ++k) {
            float d = dist_f32(x, a->C + (int64_t)k * KQO_D);
            if (d < best) {
                best = d;
                bk = k;
            }
        }
        a->idx[i] = bk;
        if (a->dist) a->dist[i] = best;
        if (a->d1) {
            double b1 = INFINITY, b2 = INFINITY;
            for (int32_t k = 0; k < a->K; ++k) {
                double d = dist_f64(x, a->C + (int64_t)k * KQO_D);
                if (d < b1) {
                    b2 = b1;
                    b1 = d;
                } else if (d < b2) {
                    b2 = d;
                }
            }
            a->d1[i] = b1;
            if (a->d2) a->d2[i] = b2;
        }
    }
    return NULL;
}

/* Eq. 1 assignment step. Rows are independent, so they are split over threads;
 * the result does not depend on the thread count. d1/d2 may be NULL. */
void kqo_assign(const float *W, int64_t n, const float *C, int32_t K, int32_t *idx, float *dist,
                double *d1, double *d2, int32_t nthreads) {
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    if ((int64_t)nthreads > n) nthreads = (int32_t)(n > 0 ? n : 1);
    pthread_t th[256];
    assign_job job[256];
    for (int t = 0; t < nthreads; ++t) {
        job[t].W = W;
        job[t].C = C;
        job[t].K = K;
        job[t].lo = n * t / nthreads;
        job[t].hi = n * (t + 1) / nthreads;
        job[t].idx = idx;
        job[t].dist = dist;
        job[t].d1 = d1;
        job[t].d2 = d2;
    }
    if (nthreads == 1) {
        assign_rows(&job[0]);
        return;
    }
    for (int t = 0; t < nthreads; ++t) pthread_create(&th[t], NULL, assign_rows, &job[t]);
    for (int t = 0; t < nthreads; ++t) pthread_join(th[t], NULL);
}

/* Eq. 1 update step: c_k = (1/z_k) * sum of the kernels in S_k. */
void kqo_update(const float *W, int64_t n, const int32_t *idx, int32_t K, const float *C_prev,
                float *C_next, int32_t *counts) {
    double *sum = (double *)calloc((size_t)K * KQO_D, sizeof(double));
    int64_t *z = (int64_t *)calloc((size_t)K, sizeof(int64_t));
    for (int64_t i = 0; i < n; ++i) {
        int32_t k = idx[i];
        z[k] += 1;
        for (int j = 0; j < KQO_D; ++j) sum[(int64_t)k * KQO_D + j] += (double)W[i * KQO_D + j];
    }
    for (int32_t k = 0; k < K; ++k) {
        for (int j = 0; j < KQO_D; ++j) {
            int64_t e = (int64_t)k * KQO_D + j;
            C_next[e] = z[k] > 0 ? (float)(sum[e] / (double)z[k]) : C_prev[e];
        }
        counts[k] = (int32_t)z[k];
    }
    free(sum);
    free(z);
}

/* Eq. 1 objective for given per-kernel distances: fp64 sum in ascending order. */
double kqo_objective(const float *dist, int64_t n) {
    double J = 0.0;
    for (int64_t i = 0; i < n; ++i) J += (double)dist[i];
    return J;
}

/* k-means of Eq. 1 from C_init: for t = 1..iters { assign(C_{t-1}); C_t = update }
 * then a final assign against C_iters. objective[t] (t = 0..iters) is the Eq. 1
 * objective of the assignment made against C_t. Returns the number of updates. */
int32_t kqo_fit(const float *W, int64_t n, int32_t K, const float *C_init, int32_t iters, float *C_out,
                int32_t *idx, int32_t *counts, double *objective, int32_t nthreads) {
    float *dist = (float *)malloc((size_t)(n > 0 ? n : 1) * sizeof(float));
    float *Ca = (float *)malloc((size_t)K * KQO_D * sizeof(float));
    float *Cb = (float *)malloc((size_t)K * KQO_D * sizeof(float));
    memcpy(Ca, C_init, (size_t)K * KQO_D * sizeof(float));
    for (int32_t t = 0; t < iters; ++t) {
        kqo_assign(W, n, Ca, K, idx, dist, NULL, NULL, nthreads);
        if (objective) objective[t] = kqo_objective(dist, n);
        kqo_update(W, n, idx, K, Ca, Cb, counts);
        float *tmp = Ca;
        Ca = Cb;
        Cb = tmp;
    }
    kqo_assign(W, n, Ca, K, idx, dist, NULL, NULL, nthreads);
    if (objective) objective[iters] = kqo_objective(dist, n);
    /* counts of the final assignment */
    memset(counts, 0, (size_t)K * sizeof(int32_t));
    for (int64_t i = 0; i < n; ++i) counts[idx[i]] += 1;
    memcpy(C_out, Ca, (size_t)K * KQO_D * sizeof(float));
    free(dist);
    free(Ca);
    free(Cb);
    return iters;
}

/* ---------------------------------------------------------------------------
 * Sec. 3.2: 6-bit codebook quantisation by weighted 1-D k-means.
 * ------------------------------------------------------------------------- */

/* Nearest of 64 levels by fp32 |v - level|, ties to the lower level index. */
static int nearest_level(float v, const float *levels) {
    float best = INFINITY;
    int bl = 0;
    for (int l = 0; l < KQO_LEVELS; ++l) {
        float d = fabsf(v - levels[l]);
        if (d < best) {
            best = d;
            bl = l;
        }
    }
    return bl;
}

/* Weight of scalar m in a level fit: w[m / group] when weights are given, else 1. */
static int64_t scalar_weight(const int32_t *w, int64_t group, int64_t m) { return w ? (int64_t)w[m / group] : 1; }

/* Fixed-point scale exponent S for the exact weighted sums (see header): N scalars,
 * weight of scalar m from scalar_weight. */
static int32_t level_scale_w(const float *v, int64_t N, const int32_t *w, int64_t group) {
    int64_t A = 0;
    float M = 0.0f;
    for (int64_t m = 0; m < N; ++m) {
        int64_t z = scalar_weight(w, group, m);
        if (z > 0) {
            A += z;
            float a = fabsf(v[m]);
            if (a > M) M = a;
        }
    }
    if (A == 0 || M == 0.0f) return 0;
    int e;
    frexp((double)A * (double)M, &e);
    return 62 - e;
}

int32_t kqo_level_scale(const float *C, int32_t K, const int32_t *counts) {
    return level_scale_w(C, (int64_t)K * KQO_D, counts, KQO_D);
}

/* Weighted 64-level k-means over N scalars (Sec. 3.2); writes the 64 levels and
 * the 6-bit code of each scalar. Returns the number of level updates made. */
static int32_t level_fit_w(const float *v, int64_t N, const int32_t *w, int64_t group, int32_t max_iters,
                           float *levels, uint8_t *codes) {
    /* initial levels: linspace(min, max, 64) over weighted scalars */
    int any = 0;
    for (int64_t m = 0; m < N; ++m) any |= scalar_weight(w, group, m) > 0;
    float lo = INFINITY, hi = -INFINITY;
    for (int64_t m = 0; m < N; ++m) {
        if (any && scalar_weight(w, group, m) <= 0) continue;
        if (v[m] < lo) lo = v[m];
        if (v[m] > hi) hi = v[m];
    }
    for (int l = 0; l < KQO_LEVELS; ++l)
        levels[l] = (float)((double)lo + ((double)hi - (double)lo) * (double)l / 63.0);

    const int32_t S = level_scale_w(v, N, w, group);
    const double up = ldexp(1.0, S), down = ldexp(1.0, -S);
    int64_t *q = (int64_t *)malloc((size_t)(N > 0 ? N : 1) * sizeof(int64_t));
    for (int64_t m = 0; m < N; ++m) q[m] = llrint((double)v[m] * up);

    uint8_t *prev = (uint8_t *)malloc((size_t)(N > 0 ? N : 1));
    uint8_t *cur = (uint8_t *)malloc((size_t)(N > 0 ? N : 1));
    int32_t updates = 0;
    for (int32_t it = 0; it < max_iters; ++it) {
        for (int64_t m = 0; m < N; ++m) cur[m] = (uint8_t)nearest_level(v[m], levels);
        if (it > 0 && memcmp(cur, prev, (size_t)N) == 0) break;
        int64_t wsum[KQO_LEVELS] = {0}, qsum[KQO_LEVELS] = {0};
        for (int64_t m = 0; m < N; ++m) {
            int64_t z = scalar_weight(w, group, m);
            if (z <= 0) continue;
            wsum[cur[m]] += z;
            qsum[cur[m]] += z * q[m];
        }
        for (int l = 0; l < KQO_LEVELS; ++l)
            if (wsum[l] > 0) levels[l] = (float)(((double)qsum[l] * down) / (double)wsum[l]);
        memcpy(prev, cur, (size_t)N);
        ++updates;
    }
    for (int64_t m = 0; m < N; ++m) codes[m] = (uint8_t)nearest_level(v[m], levels);
    free(q);
    free(prev);
    free(cur);
    return updates;
}

/* Sec. 3.2 codebook quantisation: the K*9 codebook scalars, each weighted by its
 * entry's appearance count z_k. */
int32_t kqo_level_fit(const float *C, int32_t K, const int32_t *counts, int32_t max_iters, float *levels,
                      uint8_t *codes) {
    return level_fit_w(C, (int64_t)K * KQO_D, counts, KQO_D, max_iters, levels, codes);
}

/* Sec. 3.2 fully-connected layers: m scalars, each weighted 1. */
int32_t kqo_level_fit_scalars(const float *v, int64_t m, int32_t max_iters, float *levels, uint8_t *codes) {
    return level_fit_w(v, m, NULL, 1, max_iters, levels, codes);
}

/* Sec. 3.2 testing phase: W'_i = decoded codebook row idx_i. With codes == NULL
 * the codebook C itself is used (kernel-level quantisation only). */
void kqo_reconstruct(const int32_t *idx, int64_t n, const float *C, const uint8_t *codes, const float *levels,
                     float *W_out) {
    for (int64_t i = 0; i < n; ++i) {
        int64_t k = idx[i];
        for (int j = 0; j < KQO_D; ++j)
            W_out[i * KQO_D + j] = codes ? levels[codes[k * KQO_D + j]] : C[k * KQO_D + j];
    }
}

/* Codeword init of the fit: C_0[j] = W[sel[j]] (the random draw sel is an input). */
void kqo_gather_rows(const float *W, const int64_t *sel, int32_t K, float *C0) {
    for (int32_t j = 0; j < K; ++j) memcpy(C0 + (int64_t)j * KQO_D, W + sel[j] * KQO_D, KQO_D * sizeof(float));
}

/* Sec. 3.2 encode: the 6-bit code (nearest level) of each of m values. */
void kqo_encode(const float *v, int64_t m, const float *levels, uint8_t *codes) {
    for (int64_t i = 0; i < m; ++i) codes[i] = (uint8_t)nearest_level(v[i], levels);
}

/* ---------------------------------------------------------------------------
 * Retraining with averaged gradients: Sec. 3.1 Eq. 2 and its use for the
 * quantised codebook in Sec. 3.2.
 * ------------------------------------------------------------------------- */

/* Eq. 2: every kernel i mapped to entry k (idx[i] == k, the set S_k) has a loss
 * gradient g_i = dL/dm_i (9 floats, row i of G); the entry moves against their
 * element-wise average:  c_k <- c_k - lr * (1 / z_k) * sum_{i in S_k} g_i,  z_k = |S_k|.
 * counts[k] receives z_k; an entry with z_k = 0 keeps its value. */
void kqo_codebook_grad_step(const float *G, int64_t n, const int32_t *idx, int32_t K, float lr, const float *C,
                            float *C_next, int32_t *counts) {
    double *sum = (double *)calloc((size_t)K * KQO_D, sizeof(double));
    int64_t *z = (int64_t *)calloc((size_t)K, sizeof(int64_t));
    for (int64_t i = 0; i < n; ++i) {
        int32_t k = idx[i];
        if (k < 0 || k >= K) continue;
        z[k] += 1;
        for (int j = 0; j < KQO_D; ++j) sum[(int64_t)k * KQO_D + j] += (double)G[i * KQO_D + j];
    }
    for (int32_t k = 0; k < K; ++k) {
        for (int j = 0; j < KQO_D; ++j) {
            int64_t e = (int64_t)k * KQO_D + j;
            if (z[k] > 0) {
                float mean = (float)(sum[e] / (double)z[k]);
                float step = lr * mean;
                C_next[e] = C[e] - step;
            } else {
                C_next[e] = C[e];
            }
        }
        counts[k] = (int32_t)z[k];
    }
    free(sum);
    free(z);
}

/* Sec. 3.2 retraining of the quantised codebook: the weights of the network are
 * W'_ij = levels[codes[idx_i][j]], so level l moves against the average gradient
 * of every weight whose value it is:
 *   levels[l] <- levels[l] - lr * mean{ G_ij : codes[idx_i * 9 + j] == l }.
 * counts[l] receives the number of such weights; a level with none keeps its value.
 * A kernel whose index is outside [0, K) contributes nothing. */
void kqo_levels_grad_step(const float *G, int64_t n, const int32_t *idx, int32_t K, const uint8_t *codes, float lr,
                          const float *levels, float *levels_next, int64_t *counts) {
    double sum[KQO_LEVELS] = {0};
    int64_t z[KQO_LEVELS] = {0};
    for (int64_t i = 0; i < n; ++i) {
        int32_t k = idx[i];
        if (k < 0 || k >= K) continue;
        for (int j = 0; j < KQO_D; ++j) {
            int l = codes[(int64_t)k * KQO_D + j];
            if (l >= KQO_LEVELS) continue;
            z[l] += 1;
            sum[l] += (double)G[i * KQO_D + j];
        }
    }
    for (int l = 0; l < KQO_LEVELS; ++l) {
        if (z[l] > 0) {
            float mean = (float)(sum[l] / (double)z[l]);
            float step = lr * mean;
            levels_next[l] = levels[l] - step;
        } else {
            levels_next[l] = levels[l];
        }
        counts[l] = z[l];
    }
}
