/*
 * nest_oracle.c -- plain fp64 CPU oracle for the kNN-LM step of Nearest
 * Neighbor Speculative Decoding (NEST, arXiv 2405.19325).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the CPU
 * baseline leg of the benchmark may load or call this code; the product
 * path (the CUDA library) never does, and the two share no code, header,
 * table or helper.  Nothing here is blocked, fused or reordered beyond what
 * the paper's definitions state: each function restates one definition in
 * double precision, with OpenMP only splitting independent outer loops.
 *
 *   nest_oracle_sqdist   squared l2 distance ||q - k||^2, whose negation is
 *                        the similarity s(q, k) of Sec. 2.2 (text after
 *                        Eq. 2) and App. A ("squared l2 distance")
 *   nest_oracle_topr     the r nearest neighbours pi (Sec. 2.2; the search
 *                        step of Algorithm 1): r smallest distances, ties
 *                        broken by the smaller key index
 *   nest_oracle_pknn     Eq. 2: p_kNN(w) proportional to the sum over pi of
 *                        1[w = v_i] exp(mu s_i); zero outside pi
 *   nest_oracle_mix      Eq. 3: p_M = lambda p_LM + (1 - lambda) p_kNN
 *   nest_oracle_rrc      Eq. 4: lambda_t = sigmoid((min|s|/max|s| - alpha)/tau)
 *
 * Inputs are the exact stored values: bf16 widens to double without
 * rounding, fp32 likewise.  Compile with -ffp-contract=off so that x86 and
 * Arm builds give the same bits.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_F32 0
#define ORACLE_BF16 1

/* A bf16 number is the upper 16 bits of an IEEE binary32 number. */
static double oracle_bf16_value(uint16_t bits)
{
    uint32_t word = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &word, sizeof f);
    return (double)f;
}

static double oracle_elem(const void* base, int dtype, int64_t pos)
{
    if (dtype == ORACLE_BF16)
        return oracle_bf16_value(((const uint16_t*)base)[pos]);
    return (double)((const float*)base)[pos];
}

/*
 * D[b * n + i] = sum_j (q[b][j] - K[i][j])^2 for b < B, i < n.
 * K is n x d row-major, q is B x d row-major, both of element type dtype.
 * The sum is taken term by term over j in order, in double precision.
 * Returns 0, or -1 on a bad argument.
 */
int nest_oracle_sqdist(const void* K, int dtype, int64_t n, int32_t d,
                       const void* q, int32_t B, double* D, int nthreads)
{
    if ((n > 0 && !K) || !q || !D || d <= 0 || B < 0 || n < 0) return -1;
    if (dtype != ORACLE_F32 && dtype != ORACLE_BF16) return -1;
    if (nthreads < 1) nthreads = 1;
#pragma omp parallel for num_threads(nthreads) schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        for (int32_t b = 0; b < B; ++b) {
            double acc = 0.0;
            for (int32_t j = 0; j < d; ++j) {
                double diff = oracle_elem(q, dtype, (int64_t)b * d + j)
                            - oracle_elem(K, dtype, i * (int64_t)d + j);
                acc += diff * diff;
            }
            D[(int64_t)b * n + i] = acc;
        }
    }
    return 0;
}

typedef struct {
    double dist;
    int64_t idx;
} oracle_pair;

/* Nearest first: smaller distance, then smaller key index. */
static int oracle_pair_cmp(const void* a, const void* b)
{
    const oracle_pair* x = (const oracle_pair*)a;
    const oracle_pair* y = (const oracle_pair*)b;
    if (x->dist < y->dist) return -1;
    if (x->dist > y->dist) return 1;
    if (x->idx < y->idx) return -1;
    if (x->idx > y->idx) return 1;
    return 0;
}

/*
 * The r nearest neighbours of one query among n candidates with distances
 * D[i] and key indices idx[i]: a full sort of (D, idx) pairs, nearest first,
 * of which the first min(r, n) are kept.  Slots past n are padded with
 * D = +inf and idx = -1.  Returns the number of real neighbours, or -1.
 */
int64_t nest_oracle_topr(const double* D, const int64_t* idx, int64_t n, int32_t r,
                         double* D_out, int64_t* idx_out)
{
    if (r < 1 || n < 0 || !D_out || !idx_out || (n > 0 && (!D || !idx))) return -1;
    oracle_pair* all = NULL;
    if (n > 0) {
        all = (oracle_pair*)malloc((size_t)n * sizeof(oracle_pair));
        if (!all) return -1;
        for (int64_t i = 0; i < n; ++i) {
            all[i].dist = D[i];
            all[i].idx = idx[i];
        }
        qsort(all, (size_t)n, sizeof(oracle_pair), oracle_pair_cmp);
    }
    int64_t keep = n < r ? n : r;
    for (int64_t i = 0; i < r; ++i) {
        if (i < keep) {
            D_out[i] = all[i].dist;
            idx_out[i] = all[i].idx;
        } else {
            D_out[i] = INFINITY;
            idx_out[i] = -1;
        }
    }
    free(all);
    return keep;
}

/*
 * Eq. 2 for one query.  s[i] is the similarity -||q - k||^2 of neighbour i
 * (i < r) and idx[i] its key index (-1 marks an empty slot, which carries no
 * weight).  values[] maps key index to token id (the datastore's V).
 *
 *   p_kNN(w) = sum_{i : v_i = w} exp(mu s_i) / sum_j exp(mu s_j)
 *
 * evaluated as exp(mu (s_i - s_max)) / sum_j exp(mu (s_j - s_max)), which is
 * the same number in exact arithmetic and keeps exp() from underflowing.
 * The normaliser runs over the r retrieved neighbours (Algorithm 1's
 * normaliser, whose printed lower limit "i = j" is read as j = 1).
 * p_knn has vocab entries and is overwritten.  Returns the number of real
 * neighbours, or -1 on a bad argument or an out-of-range index/value.
 */
int32_t nest_oracle_pknn(const double* s, const int64_t* idx, const int32_t* values,
                         int64_t N, int32_t r, double mu, int32_t vocab, double* p_knn)
{
    if (!s || !idx || !values || !p_knn || r < 1 || vocab < 1) return -1;
    for (int32_t w = 0; w < vocab; ++w) p_knn[w] = 0.0;
    double s_max = -INFINITY;
    int32_t real = 0;
    for (int32_t i = 0; i < r; ++i) {
        if (idx[i] < 0) continue;
        if (idx[i] >= N) return -1;
        int32_t v = values[idx[i]];
        if (v < 0 || v >= vocab) return -1;
        if (s[i] > s_max) s_max = s[i];
        ++real;
    }
    if (real == 0) return 0;
    double Z = 0.0;
    for (int32_t i = 0; i < r; ++i) {
        if (idx[i] < 0) continue;
        Z += exp(mu * (s[i] - s_max));
    }
    for (int32_t i = 0; i < r; ++i) {
        if (idx[i] < 0) continue;
        p_knn[values[idx[i]]] += exp(mu * (s[i] - s_max)) / Z;
    }
    return real;
}

/*
 * Eq. 3: p_m[w] = lambda p_lm[w] + (1 - lambda) p_knn[w], w < vocab.
 * n_real is the number of real neighbours behind p_knn.  The paper does not
 * cover an empty neighbour set (a candidate segment with no keys); there
 * p_kNN is all zeros and lambda is taken as 1, so that p_M = p_LM.
 */
int nest_oracle_mix(const float* p_lm, const double* p_knn, int32_t vocab,
                    double lambda, int32_t n_real, double* p_m)
{
    if (!p_lm || !p_knn || !p_m || vocab < 1) return -1;
    if (n_real == 0) lambda = 1.0;
    for (int32_t w = 0; w < vocab; ++w)
        p_m[w] = lambda * (double)p_lm[w] + (1.0 - lambda) * p_knn[w];
    return 0;
}

/*
 * Eq. 4 (relative retrieval confidence) for one query:
 *   lambda_t = sigmoid((min_i |s_i| / max_i |s_i| - alpha) / tau)
 * over the real neighbours (idx >= 0).  Eq. 4 takes absolute values; the
 * line of Algorithm 1 that repeats it drops them, and Eq. 4 is followed.
 * The paper does not cover two corner cases: with no real neighbour the
 * result is 1 (all weight on p_LM), and with max |s| = 0 (every neighbour
 * at distance 0) the ratio is taken as 1.  Returns NaN on a bad argument.
 */
double nest_oracle_rrc(const double* s, const int64_t* idx, int32_t r,
                       double alpha, double tau)
{
    if (!s || !idx || r < 1 || !(tau > 0.0)) return NAN;
    double lo = INFINITY, hi = 0.0;
    int32_t real = 0;
    for (int32_t i = 0; i < r; ++i) {
        if (idx[i] < 0) continue;
        double a = fabs(s[i]);
        if (a < lo) lo = a;
        if (a > hi) hi = a;
        ++real;
    }
    if (real == 0) return 1.0;
    double ratio = (hi == 0.0) ? 1.0 : lo / hi;
    return 1.0 / (1.0 + exp(-(ratio - alpha) / tau));
}

/*
 * Greedy token and span start for one row (Eq. 5 and Eq. 6, Sec. 3.3;
 * the span-selection steps of Algorithm 1).
 *
 *   token    = argmax_w p_m[w]; ties go to the smaller token id.
 *   span_key = the neighbour whose value is `token` and whose own term
 *              exp(mu s_i) is largest, i.e. the largest s_i (ties: smaller
 *              key index); -1 when no neighbour has that value.  Eq. 5 and
 *              Algorithm 1 write this as an argmax of p_kNN over neighbours
 *              with value w_t, which is one number for all of them; the
 *              max-pooling is read as pooling the neighbours' own terms.
 *   use_span = 1 when lambda <= delta and a span start exists (Eq. 6 emits
 *              the n-gram continuation), else 0 (emit the token).
 * p_m has vocab entries; s, idx are the r neighbours (idx < 0: empty slot).
 * Returns 0, or -1 on a bad argument.
 */
int nest_oracle_decide(const double* p_m, int32_t vocab, const double* s, const int64_t* idx,
                       const int32_t* values, int64_t N, int32_t r, double lambda, double delta,
                       int32_t* token, double* p_max, int64_t* span_key, int32_t* use_span)
{
    if (!p_m || vocab < 1 || !s || !idx || !values || r < 1 || !token || !p_max || !span_key ||
        !use_span)
        return -1;
    int32_t best = 0;
    for (int32_t w = 1; w < vocab; ++w)
        if (p_m[w] > p_m[best]) best = w;
    *token = best;
    *p_max = p_m[best];
    int64_t key = -1;
    double key_s = 0.0;
    for (int32_t i = 0; i < r; ++i) {
        if (idx[i] < 0 || idx[i] >= N) continue;
        if (values[idx[i]] != best) continue;
        if (key < 0 || s[i] > key_s || (s[i] == key_s && idx[i] < key)) {
            key = idx[i];
            key_s = s[i];
        }
    }
    *span_key = key;
    *use_span = (lambda <= delta && key >= 0) ? 1 : 0;
    return 0;
}

/*
 * Relaxed speculative decoding of drafted spans (Eq. 7, Sec. 3.4; the
 * verification loop of Algorithm 1).  Row b of p_m (rows x vocab) is p_M at
 * draft position b and draft[b] the drafted token there; span j covers rows
 * [span_off[j], span_off[j+1]).
 *
 *   ratio[b]    = p_m[b][draft[b]] / (gamma * max_w p_m[b][w])
 *   accept[b]   = 1 if min(1, ratio[b]) > 1/2, else 0 (Algorithm 1 stops at
 *                 the first position whose acceptance is at most 1/2)
 *   n_accept[j] = number of leading accepted positions of span j
 *
 * A row whose maximum is 0 has ratio 0.  Returns 0, or -1 on a bad argument.
 */
int nest_oracle_verify(const double* p_m, int32_t vocab, const int32_t* draft, int32_t rows,
                       const int32_t* span_off, int32_t spans, double gamma, double* ratio,
                       int32_t* accept, int32_t* n_accept)
{
    if (!p_m || vocab < 1 || !draft || rows < 0 || !span_off || spans < 0 || !(gamma > 0.0) ||
        !ratio || !accept || !n_accept)
        return -1;
    for (int32_t b = 0; b < rows; ++b) {
        if (draft[b] < 0 || draft[b] >= vocab) return -1;
        double mx = 0.0;
        for (int32_t w = 0; w < vocab; ++w)
            if (p_m[(int64_t)b * vocab + w] > mx) mx = p_m[(int64_t)b * vocab + w];
        const double p = p_m[(int64_t)b * vocab + draft[b]];
        ratio[b] = mx > 0.0 ? p / (gamma * mx) : 0.0;
        const double a = ratio[b] < 1.0 ? ratio[b] : 1.0;
        accept[b] = a > 0.5 ? 1 : 0;
    }
    for (int32_t j = 0; j < spans; ++j) {
        if (span_off[j] < 0 || span_off[j + 1] < span_off[j] || span_off[j + 1] > rows) return -1;
        int32_t n = 0;
        while (span_off[j] + n < span_off[j + 1] && accept[span_off[j] + n]) ++n;
        n_accept[j] = n;
    }
    return 0;
}
