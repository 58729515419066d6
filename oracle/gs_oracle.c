/*
 * gs_oracle.c -- plain, slow, single-threaded CPU oracle for gradient
 * sparsification (Wangni, Wang, Liu, Zhang, "Gradient Sparsification for
 * Communication-Efficient Distributed Optimization", arXiv:1710.09854).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may link, load or
 * call this file: only tests/, __graft_entry__.smoke() and bench.py's
 * cpu_baseline / reference leg use it.  It shares no code, header, table or
 * constant with the CUDA library; the two are compared, never combined.
 *
 * Everything is fp64 (the paper fixes no precision), evaluated in the order
 * the paper states it, with no blocking, fusion or reordering:
 *
 *   Section 3      Q(g)_i = Z_i g_i / p_i with Z_i ~ Bernoulli(p_i).
 *   Proposition 1  p_i = min(lambda |g_i|, 1).
 *   Algorithm 3    greedy rescaling of the active set {i : p_i != 1} until
 *                  the scaling factor c drops to <= 1 (or `iters` rescalings
 *                  have been made).
 *   Algorithm 1    step 6: the M sparse vectors are summed (gso_aggregate;
 *                  gso_average also divides by M); step 7 sparsifies the
 *                  average again (gso_sparsify on gso_average's output).
 *   Algorithm 2    the closed-form solution of problem (4) for a variance
 *                  budget epsilon: sort the magnitudes, take the smallest k
 *                  satisfying (6), set p by (7).
 *
 * Readings where the paper is silent, ambiguous or garbled:
 *   - `iters` is the maximum number of rescalings (Algorithm 3, steps 4-10);
 *     iters = 0 returns p^0.  Section 5 runs two.
 *   - A coordinate is active iff fl64(lambda |g_i|) < 1 (step 5 "p_i != 1").
 *   - g_i = 0 gives p_i = 0; such coordinates are never kept.
 *   - If the active mass sum_{i in I} p_i is 0 the loop stops.
 *   - If sum |g_i| = 0, lambda = 0 and nothing is kept.
 *   - Algorithm 2: the first display of section 3.2 squares g_(k) inside a
 *     sum over i; it is read as g_(i)^2 (the only reading under which (6)
 *     and (7) follow from it).  With g != 0 the smallest k of (6) is at most
 *     (number of non-zero g_i) - 1, so the suffix in (7) holds a non-zero
 *     entry and lambda is finite and positive; g = 0 gives lambda = 0.
 *   - The Bernoulli draw uses Philox4x32-10 (Salmon et al., SC'11), key =
 *     (seed lo, seed hi), counter = (q lo, q hi, worker, step) with q = i/4,
 *     word i mod 4; u_i = word * 2^-32 and Z_i = [u_i < p_i].
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define GSO_OK 0
#define GSO_INVALID 1
#define GSO_NONFINITE 4
#define GSO_INTERNAL 6

#if defined(__GNUC__)
#define GSO_EXPORT __attribute__((visibility("default")))
#else
#define GSO_EXPORT
#endif

/* ------------------------------------------------------------------------
 * Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel Random Numbers: As
 * Easy as 1, 2, 3", SC'11).  One round maps the counter (X0, X1, X2, X3)
 * under key (K0, K1) to
 *     (hi(M1*X2) ^ X1 ^ K0,  lo(M1*X2),  hi(M0*X0) ^ X3 ^ K1,  lo(M0*X0))
 * with the published multipliers M0 = 0xD2511F53, M1 = 0xCD9E8D57; between
 * rounds the key is bumped by the Weyl constants (0x9E3779B9, 0xBB67AE85).
 * Ten rounds.
 * ---------------------------------------------------------------------- */
GSO_EXPORT void gso_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4])
{
    uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
    uint32_t k0 = key[0], k1 = key[1];
    int r;
    for (r = 0; r < 10; r++) {
        uint64_t prod0 = (uint64_t)0xD2511F53u * (uint64_t)x0;
        uint64_t prod1 = (uint64_t)0xCD9E8D57u * (uint64_t)x2;
        uint32_t hi0 = (uint32_t)(prod0 >> 32), lo0 = (uint32_t)prod0;
        uint32_t hi1 = (uint32_t)(prod1 >> 32), lo1 = (uint32_t)prod1;
        uint32_t y0 = hi1 ^ x1 ^ k0;
        uint32_t y1 = lo1;
        uint32_t y2 = hi0 ^ x3 ^ k1;
        uint32_t y3 = lo0;
        x0 = y0; x1 = y1; x2 = y2; x3 = y3;
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/* The 32-bit random word that decides coordinate i of worker `worker` at
 * training step `step`. */
GSO_EXPORT uint32_t gso_word(uint64_t seed, uint32_t step, uint32_t worker, int64_t i)
{
    uint64_t q = (uint64_t)i / 4u;
    uint32_t ctr[4], key[2], out[4];
    ctr[0] = (uint32_t)(q & 0xFFFFFFFFu);
    ctr[1] = (uint32_t)(q >> 32);
    ctr[2] = worker;
    ctr[3] = step;
    key[0] = (uint32_t)(seed & 0xFFFFFFFFu);
    key[1] = (uint32_t)(seed >> 32);
    gso_philox4x32_10(ctr, key, out);
    return out[(uint64_t)i % 4u];
}

/* u_i in [0, 1): the word scaled by 2^-32 (exact in fp64). */
GSO_EXPORT double gso_uniform(uint64_t seed, uint32_t step, uint32_t worker, int64_t i)
{
    return (double)gso_word(seed, step, worker, i) * 0x1p-32;
}

/* Fill u[0..n) with the uniforms of coordinates i0 .. i0+n-1. */
GSO_EXPORT void gso_uniforms(uint64_t seed, uint32_t step, uint32_t worker, int64_t i0, int64_t n, double* u)
{
    int64_t k;
    for (k = 0; k < n; k++) u[k] = gso_uniform(seed, step, worker, i0 + k);
}

/* Result of the greedy solve. */
typedef struct {
    double lambda;     /* final lambda */
    int64_t capped;    /* #{i : p_i = 1} at the final lambda */
    int32_t iters_run; /* rescalings performed */
    int32_t pad;
    double sum_p;      /* sum_i p_i at the final lambda */
    double l1;         /* sum_i |g_i| */
} gso_info;

static int check_args(int64_t d, double kappa, int iters)
{
    if (d < 1) return GSO_INVALID;
    if (!(kappa > 0.0) || kappa > 1.0) return GSO_INVALID;
    if (iters < 0) return GSO_INVALID;
    return GSO_OK;
}

/* ------------------------------------------------------------------------
 * Algorithm 3 in the lambda form of Proposition 1.
 *
 * Step 3 sets p^0_i = min(rho d |g_i| / sum|g|, 1), i.e. lambda_0 = rho d / S.
 * At iteration j the active set is I = {i : lambda_j |g_i| < 1}; with
 * K = d - |I| capped coordinates and A = sum_{i in I} p_i^j the scaling
 * variable of step 6 is c = (rho d - d + |I|) / A = (rho d - K) / A.  Step 7
 * stops when c <= 1; otherwise step 8 rescales the active p by c, which is
 * lambda_{j+1} = c lambda_j (capped entries stay at 1 because c > 1).
 * ---------------------------------------------------------------------- */
GSO_EXPORT int gso_greedy_lambda(const float* g, int64_t d, double kappa, int iters, gso_info* info)
{
    int rc = check_args(d, kappa, iters);
    double S = 0.0, budget, lambda, A;
    int64_t i, K;
    int32_t j;
    if (rc != GSO_OK) return rc;

    for (i = 0; i < d; i++) S += fabs((double)g[i]);
    if (!isfinite(S)) return GSO_NONFINITE;

    memset(info, 0, sizeof(*info));
    info->l1 = S;
    if (S == 0.0) return GSO_OK; /* nothing to keep: lambda = 0 */

    budget = kappa * (double)d;
    lambda = budget / S; /* step 3 */
    j = 0;
    while (j < iters) {  /* steps 4-10 */
        K = 0;
        A = 0.0;
        for (i = 0; i < d; i++) {
            double x = lambda * fabs((double)g[i]);
            if (x >= 1.0) K++;     /* p_i = 1: outside the active set */
            else A += x;           /* p_i^j for i in I */
        }
        if (A == 0.0) break;       /* no active mass left */
        {
            double c = (budget - (double)K) / A; /* step 6 */
            if (c <= 1.0) break;                 /* step 7 */
            lambda = c * lambda;                 /* step 8 */
        }
        j++;                                     /* step 9 */
    }

    K = 0;
    A = 0.0;
    for (i = 0; i < d; i++) {
        double x = lambda * fabs((double)g[i]);
        if (x >= 1.0) K++;
        else A += x;
    }
    info->lambda = lambda;
    info->capped = K;
    info->iters_run = j;
    info->sum_p = (double)K + A;
    return GSO_OK;
}

/* ------------------------------------------------------------------------
 * Algorithm 3 exactly as printed: it carries the probability vector itself.
 * Step 3 computes p^0_i = min(rho d |g_i| / sum|g|, 1); each pass forms the
 * active set, the scaling variable c, stops on c <= 1, and replaces the
 * active entries by min(c p_i, 1).  Used to check the lambda form above.
 * ---------------------------------------------------------------------- */
GSO_EXPORT int gso_greedy_pvector(const float* g, int64_t d, double kappa, int iters, double* p, int32_t* iters_run)
{
    int rc = check_args(d, kappa, iters);
    double S = 0.0, rd;
    int64_t i;
    int32_t j = 0;
    if (rc != GSO_OK) return rc;

    for (i = 0; i < d; i++) S += fabs((double)g[i]);
    if (!isfinite(S)) return GSO_NONFINITE;
    if (S == 0.0) {
        for (i = 0; i < d; i++) p[i] = 0.0;
        *iters_run = 0;
        return GSO_OK;
    }
    rd = kappa * (double)d;
    for (i = 0; i < d; i++) {
        double t = rd * fabs((double)g[i]) / S;
        p[i] = t < 1.0 ? t : 1.0;
    }
    while (j < iters) {
        int64_t nI = 0;
        double sumI = 0.0, c;
        for (i = 0; i < d; i++) {
            if (p[i] != 1.0) { nI++; sumI += p[i]; }
        }
        if (sumI == 0.0) break;
        c = (rd - (double)d + (double)nI) / sumI;
        if (c <= 1.0) break;
        for (i = 0; i < d; i++) {
            if (p[i] != 1.0) {
                double t = c * p[i];
                p[i] = t < 1.0 ? t : 1.0;
            }
        }
        j++;
    }
    *iters_run = j;
    return GSO_OK;
}

/* p_i = min(lambda |g_i|, 1) (Proposition 1) with lambda from Algorithm 3. */
GSO_EXPORT int gso_probabilities(const float* g, int64_t d, double kappa, int iters, double* p, gso_info* info)
{
    int64_t i;
    int rc = gso_greedy_lambda(g, d, kappa, iters, info);
    if (rc != GSO_OK) return rc;
    for (i = 0; i < d; i++) {
        double x = info->lambda * fabs((double)g[i]);
        p[i] = x < 1.0 ? x : 1.0;
    }
    return GSO_OK;
}

/* ------------------------------------------------------------------------
 * Section 3: draw Z_i ~ Bernoulli(p_i), amplify kept entries to g_i / p_i,
 * and write them as (index, value) pairs in ascending index order (the plain
 * coding of the non-zero coordinates of Q(g), section 3.3).
 *
 * `i0` offsets both the Philox counter and the written index: coordinate k
 * of this vector is coordinate i0 + k of the worker's full vector (used for
 * layer-wise sparsification, where each layer is solved on its own but the
 * random stream follows the worker's flat index).
 * idx / val must hold d entries.
 * ---------------------------------------------------------------------- */
GSO_EXPORT int gso_sparsify(const float* g, int64_t d, double kappa, int iters, uint64_t seed, uint32_t step,
                            uint32_t worker, int64_t i0, int32_t* idx, float* val, int64_t* nnz, gso_info* info)
{
    int64_t i, n = 0;
    int rc = gso_greedy_lambda(g, d, kappa, iters, info);
    *nnz = 0;
    if (rc != GSO_OK) return rc;
    for (i = 0; i < d; i++) {
        double gi = (double)g[i];
        double x = info->lambda * fabs(gi);
        double p = x < 1.0 ? x : 1.0;
        double u;
        if (p == 0.0) continue; /* g_i = 0 is never kept */
        u = gso_uniform(seed, step, worker, i0 + i);
        if (u < p) {
            idx[n] = (int32_t)(i0 + i);
            val[n] = (float)(gi / p);
            n++;
        }
    }
    *nnz = n;
    return GSO_OK;
}

/* Layer-wise sparsification (section 5.2): each segment [off[l], off[l+1])
 * of the worker's vector gets its own Algorithm 3 with budget kappa * d_l.
 * The per-segment results are concatenated in index order; lambdas[l] (if
 * not NULL) receives each segment's lambda. */
GSO_EXPORT int gso_segmented_sparsify(const float* g, const int64_t* off, int L, double kappa, int iters, uint64_t seed,
                                      uint32_t step, uint32_t worker, int32_t* idx, float* val, int64_t* nnz,
                                      double* lambdas)
{
    int l;
    int64_t total = 0;
    *nnz = 0;
    if (L < 1 || off[0] != 0) return GSO_INVALID;
    for (l = 0; l < L; l++) {
        int64_t n = 0;
        gso_info info;
        int rc;
        if (off[l + 1] <= off[l]) return GSO_INVALID;
        rc = gso_sparsify(g + off[l], off[l + 1] - off[l], kappa, iters, seed, step, worker, off[l], idx + total,
                          val + total, &n, &info);
        if (rc != GSO_OK) return rc;
        if (lambdas) lambdas[l] = info.lambda;
        total += n;
    }
    *nnz = total;
    return GSO_OK;
}

/* ------------------------------------------------------------------------
 * Algorithm 1, step 6, as a sum: out_i = sum_{m=0}^{M-1} Q(g^m)_i, added in
 * fp32 in worker order m = 0, 1, ... .  Each worker's sparse vector is first
 * written out densely, then added to the running fp32 sum.
 * ---------------------------------------------------------------------- */
GSO_EXPORT int gso_aggregate(const int32_t* const* idx, const float* const* val, const int64_t* nnz, int M, int64_t d,
                             float* out)
{
    int m;
    int64_t i, e;
    float* dense;
    if (M < 1 || d < 1) return GSO_INVALID;
    dense = (float*)malloc((size_t)d * sizeof(float));
    if (!dense) return GSO_INTERNAL;
    for (i = 0; i < d; i++) out[i] = 0.0f;
    for (m = 0; m < M; m++) {
        for (i = 0; i < d; i++) dense[i] = 0.0f;
        for (e = 0; e < nnz[m]; e++) {
            int64_t k = idx[m][e];
            if (k < 0 || k >= d) { free(dense); return GSO_INVALID; }
            dense[k] = val[m][e];
        }
        for (i = 0; i < d; i++) out[i] = out[i] + dense[i];
    }
    free(dense);
    return GSO_OK;
}

/* ------------------------------------------------------------------------
 * Algorithm 1, step 6 as printed: the average v = (1/M) sum_m Q(g^m).  The
 * sum is gso_aggregate's (fp32, worker order); each coordinate is then divided
 * by M in fp32 (one correctly rounded division).  Step 7 sparsifies v again,
 * v = Q(v): that is gso_sparsify applied to this output, with a worker id of
 * its own for the random stream.
 * ---------------------------------------------------------------------- */
GSO_EXPORT int gso_average(const int32_t* const* idx, const float* const* val, const int64_t* nnz, int M, int64_t d,
                           float* out)
{
    int64_t i;
    const float fm = (float)M;
    int rc = gso_aggregate(idx, val, nnz, M, d, out);
    if (rc != GSO_OK) return rc;
    for (i = 0; i < d; i++) out[i] = out[i] / fm;
    return GSO_OK;
}

/* ------------------------------------------------------------------------
 * Section 3.3, eqs. (9)-(10): the hybrid coding of Q(g).  The kept
 * coordinates with p_i = 1 (the capped set S_k) go to Q_A as (index,
 * g_i / p_i = g_i); every other kept coordinate has p_i = lambda |g_i|, so its
 * value g_i / p_i is sign(g_i) / lambda and Q_B needs only its index and sign,
 * plus the one shared scalar 1 / lambda.
 *
 * Input is the plain coding (idx, val, nnz) that gso_sparsify made from g
 * with this lambda.  A Q_B entry is written as the code 2 * index + s with
 * s = 1 for a negative g_i.  Both lists keep ascending index order.
 * ---------------------------------------------------------------------- */
GSO_EXPORT int gso_hybrid_encode(const float* g, int64_t d, double lambda, const int32_t* idx, const float* val,
                                 int64_t nnz, int32_t* qa_idx, float* qa_val, int64_t* na, uint32_t* qb_code,
                                 int64_t* nb, double* inv_lambda)
{
    int64_t e, a = 0, b = 0;
    *na = 0;
    *nb = 0;
    if (d < 1 || nnz < 0 || nnz > d || !(lambda > 0.0)) return GSO_INVALID;
    for (e = 0; e < nnz; e++) {
        int64_t i = idx[e];
        double gi, x;
        if (i < 0 || i >= d) return GSO_INVALID;
        gi = (double)g[i];
        x = lambda * fabs(gi);
        if (x >= 1.0) {                 /* p_i = min(x, 1) = 1: i is in S_k */
            qa_idx[a] = (int32_t)i;
            qa_val[a] = val[e];
            a++;
        } else {
            qb_code[b] = (uint32_t)i * 2u + (gi < 0.0 ? 1u : 0u);
            b++;
        }
    }
    *na = a;
    *nb = b;
    *inv_lambda = 1.0 / lambda;
    return GSO_OK;
}

/* The inverse: merge Q_A and Q_B back into one ascending list of (index,
 * value), a Q_B entry taking the value +-fl32(1 / lambda). */
GSO_EXPORT int gso_hybrid_decode(const int32_t* qa_idx, const float* qa_val, int64_t na, const uint32_t* qb_code,
                                 int64_t nb, double inv_lambda, int32_t* idx, float* val, int64_t* nnz)
{
    int64_t a = 0, b = 0, n = 0;
    const float mag = (float)inv_lambda;
    while (a < na || b < nb) {
        int64_t ib = b < nb ? (int64_t)(qb_code[b] >> 1) : -1;
        if (b >= nb || (a < na && (int64_t)qa_idx[a] < ib)) {
            idx[n] = qa_idx[a];
            val[n] = qa_val[a];
            a++;
        } else {
            if (a < na && (int64_t)qa_idx[a] == ib) return GSO_INVALID; /* one index in both lists */
            idx[n] = (int32_t)ib;
            val[n] = (qb_code[b] & 1u) ? -mag : mag;
            b++;
        }
        n++;
    }
    *nnz = n;
    return GSO_OK;
}

/* Section 3.3 (last paragraph): the dense code q in {0, -1, +1, 2}^d (0: not
 * kept, -1/+1: the sign of a kept coordinate outside S_k, 2: a coordinate in
 * S_k) under standard entropy coding takes sum_l d_l log2(d / d_l) bits over
 * the symbols l with d_l > 0 -- at most 2d. */
GSO_EXPORT double gso_ternary_bits(int64_t d, int64_t n_neg, int64_t n_pos, int64_t n_cap)
{
    int64_t counts[4];
    double bits = 0.0;
    int l;
    counts[0] = d - n_neg - n_pos - n_cap;
    counts[1] = n_neg;
    counts[2] = n_pos;
    counts[3] = n_cap;
    for (l = 0; l < 4; l++) {
        if (counts[l] < 0) return -1.0;
        if (counts[l] > 0) bits += (double)counts[l] * log2((double)d / (double)counts[l]);
    }
    return bits;
}

/* Section 5: one worker's share of one step of the communication cost
 * H(T, M) of gradient sparsification:
 *   #{i : p_i = 1} (b + log2 d) + min(2d, log2 d * sum_{i : p_i < 1} p_i) + b
 * for b-bit floating point numbers. */
GSO_EXPORT double gso_comm_bits(int64_t d, int64_t n_capped, double sum_p_uncapped, int b)
{
    const double ld = log2((double)d);
    double q = ld * sum_p_uncapped;
    if (q > 2.0 * (double)d) q = 2.0 * (double)d;
    return (double)n_capped * ((double)b + ld) + q + (double)b;
}

/* ------------------------------------------------------------------------
 * Section 3.2, Algorithm 2: the closed-form solution of problem (4),
 *     min sum p_i  s.t.  sum g_i^2 / p_i <= (1 + eps) sum g_i^2,  0 < p_i <= 1.
 * With the magnitudes sorted from the largest, a_1 >= a_2 >= ... >= a_d,
 * step 1 takes the smallest k with
 *     a_{k+1} sum_{i>k} a_i <= eps sum_i g_i^2 + sum_{i>k} a_i^2      (6)
 * and step 2 sets p = 1 on the k largest and, on the rest,
 *     p_i = |g_i| lambda,  lambda = sum_{i>k} a_i / (eps sum g^2 + sum_{i>k} a_i^2)   (7).
 * The suffix sums are accumulated from the smallest magnitude up.
 * `capped` receives k, `sum_p` = k + lambda sum_{i>k} a_i, `l1` = sum |g_i|,
 * and *a_k the k-th largest magnitude (+inf when k = 0): p_i = 1 exactly
 * for |g_i| >= a_k.
 * ---------------------------------------------------------------------- */
static int cmp_desc(const void* x, const void* y)
{
    const double a = *(const double*)x, b = *(const double*)y;
    return (a < b) - (a > b);
}

static int closed_form(const float* g, int64_t d, double eps, gso_info* info, double* a_k)
{
    double *a, *A, *B, S = 0.0, l1 = 0.0;
    int64_t i, k;
    if (d < 1 || !(eps >= 0.0) || !isfinite(eps)) return GSO_INVALID;
    memset(info, 0, sizeof(*info));
    *a_k = INFINITY;
    for (i = 0; i < d; i++) {
        const double x = (double)g[i];
        S += x * x;
        l1 += fabs(x);
    }
    if (!isfinite(S) || !isfinite(l1)) return GSO_NONFINITE;
    info->l1 = l1;
    if (S == 0.0) return GSO_OK; /* g = 0: nothing to keep */

    a = (double*)malloc((size_t)d * sizeof(double));
    A = (double*)malloc((size_t)(d + 1) * sizeof(double));
    B = (double*)malloc((size_t)(d + 1) * sizeof(double));
    if (!a || !A || !B) { free(a); free(A); free(B); return GSO_INTERNAL; }
    for (i = 0; i < d; i++) a[i] = fabs((double)g[i]);
    qsort(a, (size_t)d, sizeof(double), cmp_desc);
    /* A[j] = sum_{i >= j} a_i and B[j] = sum_{i >= j} a_i^2 over the sorted
     * magnitudes (0-based j; A[d] = B[d] = 0). */
    A[d] = 0.0;
    B[d] = 0.0;
    for (i = d - 1; i >= 0; i--) {
        A[i] = A[i + 1] + a[i];
        B[i] = B[i + 1] + a[i] * a[i];
    }
    /* (6) for k = 0, 1, ...: a_{k+1} is a[k] and the sums over i > k start at a[k]. */
    for (k = 0; k < d; k++)
        if (a[k] * A[k] <= eps * S + B[k]) break;
    if (k == d) { free(a); free(A); free(B); return GSO_INTERNAL; } /* (6) holds at k = d - 1 when eps >= 0 */
    info->lambda = A[k] / (eps * S + B[k]);
    info->capped = k;
    info->sum_p = (double)k + info->lambda * A[k];
    if (k > 0) *a_k = a[k - 1];
    free(a);
    free(A);
    free(B);
    return GSO_OK;
}

GSO_EXPORT int gso_closed_form_lambda(const float* g, int64_t d, double eps, gso_info* info)
{
    double a_k;
    return closed_form(g, d, eps, info, &a_k);
}

/* p from (7): 1 on the k largest magnitudes, lambda |g_i| elsewhere. */
GSO_EXPORT int gso_probabilities_eps(const float* g, int64_t d, double eps, double* p, gso_info* info)
{
    double a_k;
    int64_t i;
    int rc = closed_form(g, d, eps, info, &a_k);
    if (rc != GSO_OK) return rc;
    for (i = 0; i < d; i++) {
        const double x = fabs((double)g[i]);
        p[i] = x >= a_k ? 1.0 : info->lambda * x;
    }
    return GSO_OK;
}

/* Section 3 with the p of Algorithm 2: the same Philox draw, amplification and
 * ascending (index, value) output as gso_sparsify. */
GSO_EXPORT int gso_sparsify_eps(const float* g, int64_t d, double eps, uint64_t seed, uint32_t step, uint32_t worker,
                                int64_t i0, int32_t* idx, float* val, int64_t* nnz, gso_info* info)
{
    double a_k;
    int64_t i, n = 0;
    int rc = closed_form(g, d, eps, info, &a_k);
    *nnz = 0;
    if (rc != GSO_OK) return rc;
    for (i = 0; i < d; i++) {
        const double gi = (double)g[i];
        const double x = fabs(gi);
        const double p = x >= a_k ? 1.0 : info->lambda * x;
        if (p == 0.0) continue;
        if (gso_uniform(seed, step, worker, i0 + i) < p) {
            idx[n] = (int32_t)(i0 + i);
            val[n] = (float)(gi / p);
            n++;
        }
    }
    *nnz = n;
    return GSO_OK;
}

/* ------------------------------------------------------------------------
 * Section 3.3, last paragraph: the dense code q~ in {0, +1, -1, 2}^d of
 * Q(g) -- q~_i = 0 where coordinate i is dropped, sign(g_i) where it is kept
 * with p_i < 1, and 2 where p_i = 1 -- entropy coded under the static model
 * the paper prices it with, P(s) = d_s / d (d_s = number of coordinates with
 * symbol s), whose ideal length is sum_s d_s log2(d / d_s) <= 2d bits.
 *
 * The coder writes that model as one event per non-zero symbol: the run of
 * zeros before it and its value.  Under the model the run length g is
 * geometric, P(g) = (1 - p0) p0^g with p0 = d_0 / d, and the value given
 * "non-zero" has P(t) = d_t / (d - d_0); the product P(g) P(t) is exactly
 * the model's probability p0^g (d_t / d) of "g zeros, then t", so coding the
 * events costs what coding the symbols one by one would.  The run is coded
 * through v = g + 1: first its bit length l = floor(log2 v), with
 * P(l) = p0^(2^l - 1) (1 - p0^(2^l)), then its l bits below the leading one,
 * each on its own, bit k being 1 with probability p0^(2^k) / (1 + p0^(2^k))
 * -- these are independent given l and multiply back to P(g) exactly.
 *
 * Layout of one vector's code (16-bit words, multi-word integers low word
 * first):
 *   header     d (2 words), d_{+1} (2), d_{-1} (2), d_2 (2), log2 K (1)
 *   directory  per chunk of K consecutive non-zero symbols: the index of its
 *              first non-zero (2 words) and its stream length in words (1)
 *   streams    one rANS stream per chunk, in chunk order.
 * A chunk's first non-zero is placed by the directory (its run is not
 * coded); every later one codes its run from the previous non-zero; the
 * zeros after the last non-zero are implied by d.
 *
 * rANS (Duda's asymmetric numeral systems, range variant): model
 * probabilities are integer frequencies f_s over M = 2^15 with cumulative
 * starts c_s; the state x lives in [2^15, 2^31); the encoder starts from
 * x = 2^15, visits the chunk's coding steps in reverse order, and before
 * each step emits the low 16 bits of x (x >>= 16) while x >= f_s 2^16, then
 * sets x = floor(x / f_s) M + (x mod f_s) + c_s; at the end it flushes x as
 * two words.  A chunk's stream is the flushed state (high word first)
 * followed by the emitted words in reverse order of emission, so that the
 * decoder reads it forward: slot = x mod M, s with c_s <= slot < c_s + f_s,
 * x = f_s (x >> 15) + slot - c_s, and one word x = (x << 16) | w whenever x
 * falls below 2^15; it must end at x = 2^15.
 *
 * Frequencies (fp64, correctly rounded, in the order written here):
 *   p0 = d_0 / d;  s_0 = p0, s_{k+1} = s_k s_k  (k < 30)
 *   bit k (k < 30): r = s_k / (1 + s_k), f_1 = (floor(r 2^16) + 1) >> 1
 *                   clamped to [1, 2^15 - 1], f_0 = 2^15 - f_1
 *   length l (l <= 30): P(l) = pi_l (1 - s_l), pi_0 = 1, pi_{l+1} = pi_l s_l
 *   value t (+1, -1, 2): P(t) = d_t / (d - d_0)
 *   multi-symbol models: f = max(1, floor(P 2^15)) for every symbol that can
 *   occur (every l; the values with d_t > 0), then the largest f (first on
 *   ties) absorbs 2^15 - sum f.
 * ---------------------------------------------------------------------- */
#define GSO_RANS_SCALE 15
#define GSO_RANS_M (1u << GSO_RANS_SCALE)
#define GSO_RANS_L (1u << 15)
#define GSO_DENSE_LMAX 31   /* bit lengths 0 .. 30 (v = g + 1 < 2^31) */
#define GSO_DENSE_BITS 30

typedef struct {
    uint32_t len_f[GSO_DENSE_LMAX], len_c[GSO_DENSE_LMAX + 1];
    uint32_t bit_f1[GSO_DENSE_BITS];
    uint32_t val_f[3], val_c[4];
} gso_dense_model;

static void gso_normalise(const double* P, const int* present, int n, uint32_t* f, uint32_t* c)
{
    int64_t sum = 0;
    int s, best = -1;
    for (s = 0; s < n; s++) {
        if (present[s]) {
            double q = floor(P[s] * (double)GSO_RANS_M);
            f[s] = q < 1.0 ? 1u : (uint32_t)q;
        } else {
            f[s] = 0;
        }
        sum += f[s];
        if (best < 0 || f[s] > f[best]) best = s;
    }
    f[best] = (uint32_t)((int64_t)f[best] + (int64_t)GSO_RANS_M - sum);
    c[0] = 0;
    for (s = 0; s < n; s++) c[s + 1] = c[s] + f[s];
}

/* The quantized model of one vector from its symbol counts. */
GSO_EXPORT int gso_dense_model_build(int64_t d, int64_t n_pos, int64_t n_neg, int64_t n_cap, gso_dense_model* m)
{
    double sq[GSO_DENSE_LMAX], P[GSO_DENSE_LMAX], Pv[3], pi, p0;
    int present[GSO_DENSE_LMAX], pv[3], k, l;
    const int64_t nz = n_pos + n_neg + n_cap;
    if (d < 1 || n_pos < 0 || n_neg < 0 || n_cap < 0 || nz > d) return GSO_INVALID;
    p0 = (double)(d - nz) / (double)d;
    sq[0] = p0;
    for (k = 1; k < GSO_DENSE_LMAX; k++) sq[k] = sq[k - 1] * sq[k - 1];
    for (k = 0; k < GSO_DENSE_BITS; k++) {
        const double r = sq[k] / (1.0 + sq[k]);
        uint32_t f1 = ((uint32_t)floor(r * 65536.0) + 1u) >> 1;
        if (f1 < 1u) f1 = 1u;
        if (f1 > GSO_RANS_M - 1u) f1 = GSO_RANS_M - 1u;
        m->bit_f1[k] = f1;
    }
    pi = 1.0;
    for (l = 0; l < GSO_DENSE_LMAX; l++) {
        P[l] = pi * (1.0 - sq[l]);
        pi = pi * sq[l];
        present[l] = 1;
    }
    gso_normalise(P, present, GSO_DENSE_LMAX, m->len_f, m->len_c);
    Pv[0] = nz > 0 ? (double)n_pos / (double)nz : 0.0;
    Pv[1] = nz > 0 ? (double)n_neg / (double)nz : 0.0;
    Pv[2] = nz > 0 ? (double)n_cap / (double)nz : 0.0;
    pv[0] = n_pos > 0;
    pv[1] = n_neg > 0;
    pv[2] = n_cap > 0;
    if (nz == 0) pv[0] = 1;   /* an unused model still sums to M */
    gso_normalise(Pv, pv, 3, m->val_f, m->val_c);
    return GSO_OK;
}

/* One coding step of a chunk: symbol s of a model given as (f, c). */
typedef struct { uint32_t f, c; } gso_sym;

/* Encoder of one chunk.  Steps are pushed in decode order into `st`, then
 * coded in reverse; words are written in reverse emission order at out. */
static int64_t gso_rans_chunk(const gso_sym* st, int64_t n_steps, uint16_t* out, int64_t cap)
{
    uint16_t* rev;
    int64_t n = 0, i;
    uint32_t x = GSO_RANS_L;
    rev = (uint16_t*)malloc((size_t)(n_steps + 2) * sizeof(uint16_t));
    if (!rev) return -1;
    for (i = n_steps - 1; i >= 0; i--) {
        const uint32_t f = st[i].f, c = st[i].c;
        if ((uint64_t)x >= ((uint64_t)f << 16)) {
            rev[n++] = (uint16_t)(x & 0xFFFFu);
            x >>= 16;
        }
        x = (x / f) * GSO_RANS_M + (x % f) + c;
    }
    /* stored: the state's high word, its low word, then the emitted words last-first */
    if (out && cap >= n + 2) {
        out[0] = (uint16_t)(x >> 16);
        out[1] = (uint16_t)(x & 0xFFFFu);
        for (i = 0; i < n; i++) out[2 + i] = rev[n - 1 - i];
    }
    free(rev);
    return n + 2;
}

static int gso_val_sym(int8_t q)
{
    return q == 1 ? 0 : (q == -1 ? 1 : 2);
}

static void put32(uint16_t* w, uint32_t v)
{
    w[0] = (uint16_t)(v & 0xFFFFu);
    w[1] = (uint16_t)(v >> 16);
}

static uint32_t get32(const uint16_t* w)
{
    return (uint32_t)w[0] | ((uint32_t)w[1] << 16);
}

/* Encode the dense vector qt (values 0, +1, -1, 2) with chunks of
 * K = 2^log2_k non-zero symbols.  Writes *n_words; out (capacity cap words)
 * is filled only when the code fits. */
GSO_EXPORT int gso_dense_encode(const int8_t* qt, int64_t d, int log2_k, uint16_t* out, int64_t cap,
                                int64_t* n_words)
{
    int64_t n_pos = 0, n_neg = 0, n_cap = 0, nz, n_chunks, i, j, total, head;
    int64_t* nzi;
    gso_dense_model m;
    gso_sym* st;
    const int64_t K = (int64_t)1 << log2_k;
    int rc;
    if (d < 1 || d >= ((int64_t)1 << 31) || log2_k < 4 || log2_k > 10 || !n_words) return GSO_INVALID;
    for (i = 0; i < d; i++) {
        if (qt[i] == 1) n_pos++;
        else if (qt[i] == -1) n_neg++;
        else if (qt[i] == 2) n_cap++;
        else if (qt[i] != 0) return GSO_INVALID;
    }
    rc = gso_dense_model_build(d, n_pos, n_neg, n_cap, &m);
    if (rc != GSO_OK) return rc;
    nz = n_pos + n_neg + n_cap;
    n_chunks = (nz + K - 1) / K;
    nzi = (int64_t*)malloc((size_t)(nz + 1) * sizeof(int64_t));
    st = (gso_sym*)malloc((size_t)(K * (2 + GSO_DENSE_BITS)) * sizeof(gso_sym));
    if (!nzi || !st) {
        free(nzi);
        free(st);
        return GSO_INTERNAL;
    }
    for (i = 0, j = 0; i < d; i++)
        if (qt[i] != 0) nzi[j++] = i;
    head = 9 + 3 * n_chunks;
    total = head;
    if (out && cap >= 9) {
        put32(out, (uint32_t)d);
        put32(out + 2, (uint32_t)n_pos);
        put32(out + 4, (uint32_t)n_neg);
        put32(out + 6, (uint32_t)n_cap);
        out[8] = (uint16_t)log2_k;
    }
    for (i = 0; i < n_chunks; i++) {
        const int64_t a = i * K, b = (a + K < nz) ? a + K : nz;
        int64_t n_steps = 0, len;
        for (j = a; j < b; j++) {
            if (j > a) {
                const uint32_t v = (uint32_t)(nzi[j] - nzi[j - 1]);   /* run of zeros + 1 */
                int l = 0, k;
                while ((v >> (l + 1)) != 0u) l++;
                st[n_steps].f = m.len_f[l];
                st[n_steps].c = m.len_c[l];
                n_steps++;
                for (k = l - 1; k >= 0; k--) {
                    const uint32_t bit = (v >> k) & 1u, f1 = m.bit_f1[k];
                    st[n_steps].f = bit ? f1 : GSO_RANS_M - f1;
                    st[n_steps].c = bit ? GSO_RANS_M - f1 : 0u;
                    n_steps++;
                }
            }
            {
                const int s = gso_val_sym(qt[nzi[j]]);
                st[n_steps].f = m.val_f[s];
                st[n_steps].c = m.val_c[s];
                n_steps++;
            }
        }
        len = gso_rans_chunk(st, n_steps, (out && cap >= total) ? out + total : NULL,
                             out ? cap - total : 0);
        if (len < 0) {
            free(nzi);
            free(st);
            return GSO_INTERNAL;
        }
        if (out && cap >= head) {
            put32(out + 9 + 3 * i, (uint32_t)nzi[a]);
            out[9 + 3 * i + 2] = (uint16_t)len;
        }
        total += len;
    }
    *n_words = total;
    free(nzi);
    free(st);
    return GSO_OK;
}

/* rANS decoder state over one chunk's words. */
typedef struct {
    const uint16_t* w;
    int64_t pos, n;
    uint32_t x;
    int bad;
} gso_rans_dec;

static uint32_t gso_rans_take(gso_rans_dec* r, const uint32_t* f, const uint32_t* c, int n_sym)
{
    const uint32_t slot = r->x & (GSO_RANS_M - 1u);
    int s = 0;
    while (s < n_sym - 1 && !(slot < c[s + 1])) s++;
    r->x = f[s] * (r->x >> GSO_RANS_SCALE) + slot - c[s];
    if (r->x < GSO_RANS_L) {
        if (r->pos < r->n) r->x = (r->x << 16) | r->w[r->pos++];
        else r->bad = 1;
    }
    return (uint32_t)s;
}

/* Decode a code written by gso_dense_encode into qt[0..d). */
GSO_EXPORT int gso_dense_decode(const uint16_t* in, int64_t n_words, int64_t d, int8_t* qt)
{
    gso_dense_model m;
    int64_t n_pos, n_neg, n_cap, nz, K, n_chunks, i, j, off;
    int rc, log2_k;
    if (n_words < 9 || d < 1 || (int64_t)get32(in) != d) return GSO_INVALID;
    n_pos = get32(in + 2);
    n_neg = get32(in + 4);
    n_cap = get32(in + 6);
    log2_k = in[8];
    if (log2_k < 4 || log2_k > 10) return GSO_INVALID;
    rc = gso_dense_model_build(d, n_pos, n_neg, n_cap, &m);
    if (rc != GSO_OK) return rc;
    nz = n_pos + n_neg + n_cap;
    K = (int64_t)1 << log2_k;
    n_chunks = (nz + K - 1) / K;
    if (n_words < 9 + 3 * n_chunks) return GSO_INVALID;
    memset(qt, 0, (size_t)d);
    off = 9 + 3 * n_chunks;
    for (i = 0; i < n_chunks; i++) {
        const int64_t cnt = (i + 1) * K <= nz ? K : nz - i * K;
        const int64_t len = in[9 + 3 * i + 2];
        int64_t idx = get32(in + 9 + 3 * i);
        uint32_t bitf[2], bitc[3];
        gso_rans_dec r;
        if (len < 2 || off + len > n_words) return GSO_INVALID;
        r.w = in + off;
        r.pos = 2;
        r.n = len;
        r.x = ((uint32_t)r.w[0] << 16) | r.w[1];
        r.bad = 0;
        for (j = 0; j < cnt; j++) {
            uint32_t s;
            if (j > 0) {
                const int l = (int)gso_rans_take(&r, m.len_f, m.len_c, GSO_DENSE_LMAX);
                uint32_t v = 1;
                int k;
                for (k = l - 1; k >= 0; k--) {
                    bitf[1] = m.bit_f1[k];
                    bitf[0] = GSO_RANS_M - bitf[1];
                    bitc[0] = 0;
                    bitc[1] = bitf[0];
                    bitc[2] = GSO_RANS_M;
                    v = 2u * v + gso_rans_take(&r, bitf, bitc, 2);
                }
                idx += v;
            }
            if (idx < 0 || idx >= d) return GSO_INVALID;
            s = gso_rans_take(&r, m.val_f, m.val_c, 3);
            qt[idx] = s == 0 ? 1 : (s == 1 ? -1 : 2);
        }
        if (r.bad || r.x != GSO_RANS_L || r.pos != r.n) return GSO_INVALID;
        off += len;
    }
    return off == n_words ? GSO_OK : GSO_INVALID;
}
