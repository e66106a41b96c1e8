/*
 * ecasq_oracle.c -- plain, slow, CPU reference for ECASQ (Entropy-Constrained
 * Adaptive Stochastic Quantization, arxiv 2608.18147).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may include, link or
 * call this file; only the test suite, the smoke check and the benchmark's CPU
 * baseline leg use it.  It shares no code with the CUDA library.
 *
 * Precision: every floating-point result is IEEE binary64.  The prefix sums
 * N(t), S(t), S2(t) of App. E are accumulated in IEEE binary128 (_Float128),
 * where they are exact for fp32 inputs of ordinary dynamic range, and every
 * per-interval quantity C_P, U_P, D_P is evaluated in binary128 from them and
 * rounded once to binary64.  Interval endpoints are unique input values
 * (P = X, Sec. 5), indices are 0-based, intervals are half-open (v_k, v_j]
 * (App. E convention) and the first value's own mass w_0 is added explicitly
 * (Phi^first, Sec. 5).
 *
 * Functions and the passages they follow:
 *   or_hist_new      Sec. 2 (sorted copy, weighted histogram), App. E (prefix sums)
 *   or_hist_new_grid Sec. 5 / App. E for a general permissible set P: the same
 *                    histogram view with P as the candidate values, first-value
 *                    set L = {a : p_a <= x_1} and last-value set R = {b : p_b >= x_d}
 *   pair_q           App. E: U_P, D_P, C_P from prefix differences
 *   h, or_phi        Sec. 4 (h), Sec. 5 (Phi, Phi^first)
 *   or_apx_dp        Sec. 5, eqs. apx_base / apx_rec / apx_final
 *   or_apx_dp_columns the same DP evaluated column by column (each pair's link
 *                    cost computed once for all layers), for full-size checks;
 *                    or_apx_dp_columns_prefix its tables for the first columns alone
 *   or_apx_dp_linear Sec. 5 (last paragraph): the codebook of the same DP in linear
 *                    space (forward and backward passes, split at a middle value)
 *   or_dp_decision,  one output / one candidate of eq. apx_rec (eq. apx_base with
 *   or_dp_candidate  `first`), for checking sampled outputs of large GPU runs
 *   or_eval_idx      Sec. 2 (MSE), Sec. 3 (H(Xhat)), Sec. 5 eq. apx_additive_entropy
 *   or_eval_direct   the per-entry definitions of Sec. 1-3 and Sec. 5 (no prefix sums)
 *   or_asq_dp        Sec. 2, eq. asqdp (ZipML/QUIVER recurrence, lambda = 0)
 *   or_opt_dp        Sec. 4 with the boundary conventions of App. E (naive O(s p^3))
 *   or_brute         exhaustive enumeration of spanning codebooks drawn from X
 *   or_brute_grid    the same over codebooks drawn from a permissible set P
 *   or_search        Sec. 3 / Sec. 5: tune lambda for a budget b (schedule below)
 *   or_timeshare     Sec. 7: two-way time-sharing between the evaluated points
 *                    around b; or_quantize_timeshare encodes with it
 *   or_refine        Sec. 6: three-colour refinement
 *   or_quantize      Sec. 2: unbiased stochastic rounding, Sec. 1 entropy
 *
 * Readings where the paper is silent (the same readings the CUDA library uses):
 *   - lambda search: lambda = 0 first; otherwise rounds of 7 geometric
 *     midpoints (built with correctly rounded sqrt only) inside [lo, hi];
 *     the bracket shrinks to the pair around the smallest feasible point;
 *     the answer is the minimum-MSE feasible evaluated point (ties: smaller
 *     lambda); feasibility is H(I,B) <= b.
 *   - refinement objective: the true Lagrangian MSE + lambda' H(Xhat); each
 *     moving value is placed at the best unique input value strictly between
 *     its neighbours (exhaustive scan; ties keep the current value, else the
 *     lowest index); with a budget, a colour step that lifts H(Xhat) above b
 *     is undone.
 *   - stochastic rounding decision: SplitMix64 (Steele, Lea and Flood,
 *     OOPSLA 2014) on seed + (i+1)*0x9E3779B97F4A7C15, k = top 24 bits;
 *     round up iff fl32(fl32(k*2^-24) * fl32(b-a)) < fl32(x-a).
 *
 * Parity unpinned by the paper: the multiplier schedule of or_search, the scan
 * and tie rules of or_refine and the random draw of or_quantize are the readings
 * above, not values the paper fixes.  The tests pin them to those readings only
 * (SplitMix64's published outputs, the exact rounding probability, refinement
 * monotonicity and coordinate optimality, the search's feasibility and least-MSE
 * choice among its evaluated points).
 *
 * Build: gcc -O2 -fopenmp -ffp-contract=off -fPIC -shared (see build.py).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef _Float128 q128;

#define OR_OK 0
#define OR_EINVAL (-1)
#define OR_ENONFINITE (-2)
#define OR_EINFEASIBLE (-3)
#define OR_ERANGE (-7)
#define OR_ENOMEM (-8)

typedef struct or_hist {
    int64_t d, p;
    float *v;      /* unique values, ascending */
    int64_t *w;    /* multiplicities */
    int64_t *N;    /* N[t] = sum_{r<t} w_r,        t = 0..p */
    q128 *S;       /* S[t] = sum_{r<t} w_r v_r */
    q128 *S2;      /* S2[t] = sum_{r<t} w_r v_r^2 */
    double norm2;  /* ||X||^2 */
    int64_t nL, nR;  /* L = {0..nL-1}, R = {p-nR..p-1} (Sec. 5); 1, 1 when P = X */
    /* optional memo of C and Phi for every pair k < j (upper triangle) */
    double *tC, *tPhi;
} or_hist;

/* ---------------------------------------------------------------- basics */

/* h(y) = -y log2 y, h(0) = 0 (Sec. 4). */
static double h(double y) { return y > 0.0 ? -y * log2(y) : 0.0; }

static int cmp_f32(const void *a, const void *b) {
    float x = *(const float *)a, y = *(const float *)b;
    return (x > y) - (x < y);
}

static inline size_t tri(int64_t k, int64_t j) { return (size_t)j * (size_t)(j - 1) / 2 + (size_t)k; }

void or_hist_free(or_hist *H) {
    if (!H) return;
    free(H->v); free(H->w); free(H->N); free(H->S); free(H->S2);
    free(H->tC); free(H->tPhi);
    free(H);
}

/* Sorted copy of X and its weighted histogram (Sec. 2: "we assume X is
 * sorted ... work with its weighted histogram"), plus the prefix sums of
 * App. E.  -0.0 and +0.0 are the same value. */
or_hist *or_hist_new(const float *x, int64_t d, int32_t *status) {
    *status = OR_OK;
    if (!x || d < 1) { *status = OR_EINVAL; return NULL; }
    for (int64_t i = 0; i < d; i++)
        if (!isfinite(x[i])) { *status = OR_ENONFINITE; return NULL; }
    float *xs = (float *)malloc(sizeof(float) * (size_t)d);
    or_hist *H = (or_hist *)calloc(1, sizeof(or_hist));
    if (!xs || !H) { free(xs); free(H); *status = OR_ENOMEM; return NULL; }
    for (int64_t i = 0; i < d; i++) xs[i] = (x[i] == 0.0f) ? 0.0f : x[i];
    qsort(xs, (size_t)d, sizeof(float), cmp_f32);
    int64_t p = 1;
    for (int64_t i = 1; i < d; i++) p += (xs[i] != xs[i - 1]);
    H->d = d; H->p = p;
    H->v = (float *)malloc(sizeof(float) * (size_t)p);
    H->w = (int64_t *)malloc(sizeof(int64_t) * (size_t)p);
    H->N = (int64_t *)malloc(sizeof(int64_t) * (size_t)(p + 1));
    H->S = (q128 *)malloc(sizeof(q128) * (size_t)(p + 1));
    H->S2 = (q128 *)malloc(sizeof(q128) * (size_t)(p + 1));
    if (!H->v || !H->w || !H->N || !H->S || !H->S2) { free(xs); or_hist_free(H); *status = OR_ENOMEM; return NULL; }
    int64_t u = 0;
    H->v[0] = xs[0]; H->w[0] = 1;
    for (int64_t i = 1; i < d; i++) {
        if (xs[i] != xs[i - 1]) { u++; H->v[u] = xs[i]; H->w[u] = 0; }
        H->w[u]++;
    }
    free(xs);
    H->N[0] = 0; H->S[0] = 0; H->S2[0] = 0;
    for (int64_t t = 0; t < p; t++) {
        q128 vv = (q128)H->v[t], ww = (q128)H->w[t];
        H->N[t + 1] = H->N[t] + H->w[t];
        H->S[t + 1] = H->S[t] + ww * vv;
        H->S2[t + 1] = H->S2[t] + ww * vv * vv;
    }
    H->norm2 = (double)H->S2[p];
    H->nL = 1;
    H->nR = 1;
    return H;
}

/* General permissible set P (Sec. 5, App. E): candidate values p_0 < ... < p_{n-1}
 * with p_0 <= min x and p_{n-1} >= max x (App. E: otherwise no unbiased quantizer
 * drawn from P spans X).  The first value may be any a in L = {a : p_a <= x_1} and
 * the last any b in R = {b : p_b >= x_d} (eqs. apx_base, apx_final); both are runs
 * of indices, L = {0..nL-1}, R = {n-nR..n-1}.  The histogram view takes v = P and,
 * for every t, w_t = |{x : p_{t-1} < x <= p_t}| (for a in L this is n_a =
 * |{x : x = p_a}|, the first value's own mass of Phi^first) and the prefix sums of App. E,
 *   N[t+1] = |{x <= p_t}|,  S[t+1] = sum_{x <= p_t} x,  S2[t+1] = sum_{x <= p_t} x^2,
 * accumulated entry by entry in binary128.  Every later function then reads
 * X_{a,b} = {x : p_a < x <= p_b} for a < b, as App. E defines it for P. */
or_hist *or_hist_new_grid(const float *x, int64_t d, const float *P, int64_t n, int32_t *status) {
    *status = OR_OK;
    if (!x || d < 1 || !P || n < 1) { *status = OR_EINVAL; return NULL; }
    for (int64_t i = 0; i < d; i++)
        if (!isfinite(x[i])) { *status = OR_ENONFINITE; return NULL; }
    for (int64_t t = 0; t < n; t++)
        if (!isfinite(P[t]) || (t > 0 && !(P[t] > P[t - 1]))) { *status = OR_EINVAL; return NULL; }
    float *xs = (float *)malloc(sizeof(float) * (size_t)d);
    or_hist *H = (or_hist *)calloc(1, sizeof(or_hist));
    if (!xs || !H) { free(xs); free(H); *status = OR_ENOMEM; return NULL; }
    for (int64_t i = 0; i < d; i++) xs[i] = (x[i] == 0.0f) ? 0.0f : x[i];
    qsort(xs, (size_t)d, sizeof(float), cmp_f32);
    float p0 = P[0] == 0.0f ? 0.0f : P[0], pl = P[n - 1] == 0.0f ? 0.0f : P[n - 1];
    if (!(p0 <= xs[0]) || !(pl >= xs[d - 1])) { free(xs); free(H); *status = OR_EINVAL; return NULL; }
    H->nL = 0;
    H->nR = 0;
    for (int64_t t = 0; t < n; t++) {
        float pt = P[t] == 0.0f ? 0.0f : P[t];
        H->nL += (pt <= xs[0]);
        H->nR += (pt >= xs[d - 1]);
    }
    H->d = d; H->p = n;
    H->v = (float *)malloc(sizeof(float) * (size_t)n);
    H->w = (int64_t *)malloc(sizeof(int64_t) * (size_t)n);
    H->N = (int64_t *)malloc(sizeof(int64_t) * (size_t)(n + 1));
    H->S = (q128 *)malloc(sizeof(q128) * (size_t)(n + 1));
    H->S2 = (q128 *)malloc(sizeof(q128) * (size_t)(n + 1));
    if (!H->v || !H->w || !H->N || !H->S || !H->S2) { free(xs); or_hist_free(H); *status = OR_ENOMEM; return NULL; }
    H->N[0] = 0; H->S[0] = 0; H->S2[0] = 0;
    int64_t i = 0;
    q128 sacc = 0, qacc = 0;
    for (int64_t t = 0; t < n; t++) {
        float pt = P[t] == 0.0f ? 0.0f : P[t];
        H->v[t] = pt;
        int64_t i0 = i;
        while (i < d && xs[i] <= pt) {
            q128 xv = (q128)xs[i];
            sacc += xv;
            qacc += xv * xv;
            i++;
        }
        H->w[t] = i - i0;
        H->N[t + 1] = i;
        H->S[t + 1] = sacc;
        H->S2[t + 1] = qacc;
    }
    free(xs);
    H->norm2 = (double)H->S2[n];
    return H;
}

void or_hist_info(const or_hist *H, int64_t *d, int64_t *p, double *norm2) {
    *d = H->d; *p = H->p; *norm2 = H->norm2;
}

void or_hist_ends(const or_hist *H, int64_t *nL, int64_t *nR) {
    *nL = H->nL; *nR = H->nR;
}

/* Copy out the histogram and the prefix sums (binary128 split as hi + lo). */
void or_hist_arrays(const or_hist *H, float *v, int64_t *w, int64_t *N,
                    double *S_hi, double *S_lo, double *S2_hi, double *S2_lo) {
    for (int64_t t = 0; t < H->p; t++) { v[t] = H->v[t]; w[t] = H->w[t]; }
    for (int64_t t = 0; t <= H->p; t++) {
        N[t] = H->N[t];
        double a = (double)H->S[t], b = (double)H->S2[t];
        S_hi[t] = a; S_lo[t] = (double)(H->S[t] - (q128)a);
        S2_hi[t] = b; S2_lo[t] = (double)(H->S2[t] - (q128)b);
    }
}

/* App. E: for k < j, over X_{k,j} = {x : v_k < x <= v_j},
 *   U = (S_kj - v_k N_kj)/(v_j - v_k),  D = (v_j N_kj - S_kj)/(v_j - v_k),
 *   C = (v_k + v_j) S_kj - S2_kj - v_k v_j N_kj.
 * The numerators are formed in binary128 and rounded once; the division is
 * one binary64 division by L = v_j - v_k (binary64 subtraction). */
static void pair_q(const or_hist *H, int64_t k, int64_t j, double *C, double *U, double *D) {
    int64_t dN = H->N[j + 1] - H->N[k + 1];
    q128 n = (q128)dN;
    q128 dS = H->S[j + 1] - H->S[k + 1];
    q128 dS2 = H->S2[j + 1] - H->S2[k + 1];
    q128 vk = (q128)H->v[k], vj = (q128)H->v[j];
    q128 A = dS - vk * n;             /* sum (x - v_k)   */
    q128 E = vj * n - dS;             /* sum (v_j - x)   */
    q128 Cq = (vk + vj) * dS - dS2 - vk * vj * n;
    double L = (double)H->v[j] - (double)H->v[k];
    *C = (double)Cq;
    *U = (double)A / L;
    *D = (double)E / L;
}

void or_pair(const or_hist *H, int64_t k, int64_t j, double *out3) {
    pair_q(H, k, j, &out3[0], &out3[1], &out3[2]);
}

/* Sec. 5: Phi = h(U/d) + h(D/d);  Phi^first[a, .] = h(U/d) + h((D + n_a)/d).
 * first_a < 0: an ordinary interval; otherwise the first interval, starting at a. */
static double phi_of(const or_hist *H, double U, double D, int64_t first_a) {
    double dd = (double)H->d;
    double Dm = first_a >= 0 ? D + (double)H->w[first_a] : D;
    return h(U / dd) + h(Dm / dd);
}

double or_phi(const or_hist *H, int64_t k, int64_t j, int32_t first) {
    double C, U, D;
    pair_q(H, k, j, &C, &U, &D);
    return phi_of(H, U, D, first ? k : -1);
}

/* Memoise C and Phi for every pair (only practical for p up to ~2e4). */
int32_t or_hist_cache(or_hist *H) {
    int64_t p = H->p;
    if (H->tC) return OR_OK;
    size_t n = (size_t)p * (size_t)(p - 1) / 2;
    if (n == 0) return OR_OK;
    H->tC = (double *)malloc(sizeof(double) * n);
    H->tPhi = (double *)malloc(sizeof(double) * n);
    if (!H->tC || !H->tPhi) { free(H->tC); free(H->tPhi); H->tC = H->tPhi = NULL; return OR_ENOMEM; }
#pragma omp parallel for schedule(dynamic, 16)
    for (int64_t j = 1; j < p; j++)
        for (int64_t k = 0; k < j; k++) {
            double C, U, D;
            pair_q(H, k, j, &C, &U, &D);
            H->tC[tri(k, j)] = C;
            H->tPhi[tri(k, j)] = phi_of(H, U, D, -1);
        }
    return OR_OK;
}

static inline void cphi(const or_hist *H, int64_t k, int64_t j, double *C, double *Phi) {
    if (H->tC) { *C = H->tC[tri(k, j)]; *Phi = H->tPhi[tri(k, j)]; return; }
    double U, D;
    pair_q(H, k, j, C, &U, &D);
    *Phi = phi_of(H, U, D, -1);
}

/* -------------------------------------------------------- evaluation */

/* Metrics of a codebook given as ascending candidate indices a[0..m-1]
 * with a[0] in L and a[m-1] in R (Q spans X, Q subset of P):
 *   out[0] MSE            = sum_r C[a_r, a_{r+1}]                     (Sec. 2)
 *   out[1] H(I,B)         = Phi^first[a_0,a_1] + sum_{r>=1} Phi[a_r,a_{r+1}] (eq. apx_additive_entropy)
 *   out[2] H(Xhat)        = sum_r h(f_r / d), f_r = U[a_{r-1},a_r] + D[a_r,a_{r+1}],
 *                           f_0 = n_{a_0} + D[a_0,a_1], f_{m-1} = U[a_{m-2},a_{m-1}] (Sec. 3, Sec. 5)
 */
int32_t or_eval_idx(const or_hist *H, const int64_t *a, int32_t m, double *out) {
    double dd = (double)H->d;
    if (m < 1 || a[0] < 0 || a[0] >= H->nL || a[m - 1] < H->p - H->nR || a[m - 1] >= H->p) return OR_EINVAL;
    for (int32_t r = 1; r < m; r++) if (a[r] <= a[r - 1]) return OR_EINVAL;
    if (m == 1) { out[0] = 0.0; out[1] = 0.0; out[2] = 0.0; return OR_OK; }
    double mse = 0.0, hs = 0.0, hx = 0.0;
    double prevU = 0.0;
    for (int32_t r = 0; r + 1 < m; r++) {
        double C, U, D;
        pair_q(H, a[r], a[r + 1], &C, &U, &D);
        mse += C;
        hs += phi_of(H, U, D, r == 0 ? a[0] : -1);
        double f = (r == 0) ? (double)H->w[a[0]] + D : prevU + D;
        hx += h(f / dd);
        prevU = U;
    }
    hx += h(prevU / dd);
    out[0] = mse; out[1] = hs; out[2] = hx;
    return OR_OK;
}

/* The same metrics straight from the per-entry definitions, for any
 * ascending codebook Q (double values) that spans x:
 *   a_x = max{q <= x}, b_x = min{q >= x}; Pr[up] = (x - a_x)/(b_x - a_x) (Sec. 2);
 *   MSE = sum (b_x - x)(x - a_x); f_q = sum_x Pr[xhat = q]; H(Xhat) = sum h(f_q/d) (Sec. 3);
 *   interval I_x: q_I < x <= q_{I+1}, I_x = first interval when x = q_1 (Sec. 5),
 *   H(I,B) = entropy of the joint law of (I_x, B_x).
 * out: [MSE, H(I,B), H(Xhat)]. */
int32_t or_eval_direct(const float *x, int64_t d, const double *Q, int32_t m, double *out) {
    if (m < 1) return OR_EINVAL;
    for (int32_t r = 1; r < m; r++) if (!(Q[r] > Q[r - 1])) return OR_EINVAL;
    double *f = (double *)calloc((size_t)m, sizeof(double));
    double *ib = (double *)calloc((size_t)(2 * m), sizeof(double));
    if (!f || !ib) { free(f); free(ib); return OR_ENOMEM; }
    double mse = 0.0;
    int32_t st = OR_OK;
    for (int64_t i = 0; i < d; i++) {
        double xv = (double)x[i];
        if (xv < Q[0] || xv > Q[m - 1]) { st = OR_ERANGE; break; }
        if (m == 1) { f[0] += 1.0; ib[0] += 1.0; continue; }
        /* interval index I: q_I < x <= q_{I+1}; x = q_0 goes to interval 0 */
        int32_t I = 0;
        while (I + 1 < m - 1 && xv > Q[I + 1]) I++;
        double a = Q[I], b = Q[I + 1];
        double pu = (xv - a) / (b - a);
        mse += (b - xv) * (xv - a);
        f[I] += 1.0 - pu;
        f[I + 1] += pu;
        ib[2 * I] += 1.0 - pu;
        ib[2 * I + 1] += pu;
    }
    if (st == OR_OK) {
        double dd = (double)d, hx = 0.0, hs = 0.0;
        for (int32_t r = 0; r < m; r++) hx += h(f[r] / dd);
        for (int32_t r = 0; r < 2 * m; r++) hs += h(ib[r] / dd);
        out[0] = mse; out[1] = hs; out[2] = hx;
    }
    free(f); free(ib);
    return st;
}

/* ------------------------------------------------------ approximate DP */

/* Sec. 5, lambda' = lam_prime, L = {0..nL-1}, R = {p-nR..p-1} ({0} and {p-1} when P = X):
 *   dp(2, j) = min_{a in L, a<j} C[a, j] + lambda' Phi^first[a, j]  (eq. apx_base)
 *   dp(i, j) = min_{k<j} dp(i-1, k) + C[k, j] + lambda' Phi[k, j]  (eq. apx_rec)
 *   answer   = min_{2<=i<=s} min_{j in R} dp(i, j)  (or i = s only) (eq. apx_final)
 * Each candidate is formed as dp(i-1,k) + (C + lambda' Phi); the argmin is the
 * lowest k (lowest a in the base layer) among exact binary64 minima; the final
 * selection is the smallest i, then the smallest j.
 * Arrays (optional, row-major (s+1) x p, rows 0 and 1 unused):
 *   dp (+inf where undefined), bp (-1 where undefined), margin = relative gap
 *   between the best and second-best candidate ((2nd - best)/best).
 * Q_idx receives the traced codebook (unique-value indices), m its size. */
int32_t or_apx_dp(const or_hist *H, int32_t s, double lam_prime, int32_t exact_s,
                  double *dp_out, int32_t *bp_out, double *margin_out,
                  int64_t *Q_idx, int32_t *m_out, double *best_out) {
    int64_t p = H->p;
    if (s < 2) return OR_EINVAL;
    if (p == 1) {
        Q_idx[0] = 0; *m_out = 1; *best_out = 0.0;
        return OR_OK;
    }
    size_t rows = (size_t)s + 1;
    double *dp = (double *)malloc(sizeof(double) * rows * (size_t)p);
    int32_t *bp = (int32_t *)malloc(sizeof(int32_t) * rows * (size_t)p);
    double *mg = (double *)malloc(sizeof(double) * rows * (size_t)p);
    if (!dp || !bp || !mg) { free(dp); free(bp); free(mg); return OR_ENOMEM; }
    for (size_t t = 0; t < rows * (size_t)p; t++) { dp[t] = INFINITY; bp[t] = -1; mg[t] = INFINITY; }
    /* base layer */
    for (int64_t j = 1; j < p; j++) {
        double best = INFINITY;
        int64_t arg = -1;
        for (int64_t a = 0; a < H->nL && a < j; a++) {
            double C, U, D;
            pair_q(H, a, j, &C, &U, &D);
            double c = C + lam_prime * phi_of(H, U, D, a);
            if (c < best) { best = c; arg = a; }
        }
        dp[2 * (size_t)p + (size_t)j] = best;
        bp[2 * (size_t)p + (size_t)j] = (int32_t)arg;
    }
    /* recurrence layers */
    for (int32_t i = 3; i <= s; i++) {
        const double *prev = dp + (size_t)(i - 1) * (size_t)p;
        double *cur = dp + (size_t)i * (size_t)p;
        int32_t *cbp = bp + (size_t)i * (size_t)p;
        double *cmg = mg + (size_t)i * (size_t)p;
#pragma omp parallel for schedule(dynamic, 8)
        for (int64_t j = i - 1; j < p; j++) {
            double best = INFINITY, second = INFINITY;
            int64_t arg = -1;
            for (int64_t k = i - 2; k < j; k++) {
                double C, Phi;
                cphi(H, k, j, &C, &Phi);
                double cand = prev[k] + (C + lam_prime * Phi);
                if (cand < best) { second = best; best = cand; arg = k; }
                else if (cand < second) second = cand;
            }
            cur[j] = best;
            cbp[j] = (int32_t)arg;
            cmg[j] = (best > 0.0) ? (second - best) / best : (second > best ? INFINITY : 0.0);
        }
    }
    /* final selection */
    int32_t istar = -1;
    int64_t jstar = -1;
    double best = INFINITY;
    int32_t ilo = exact_s ? s : 2;
    for (int32_t i = ilo; i <= s; i++)
        for (int64_t jr = p - H->nR; jr < p; jr++) {
            double v = dp[(size_t)i * (size_t)p + (size_t)jr];
            if (v < best) { best = v; istar = i; jstar = jr; }
        }
    if (istar < 0) { free(dp); free(bp); free(mg); return OR_EINFEASIBLE; }
    /* traceback */
    int64_t j = jstar;
    Q_idx[istar - 1] = j;
    for (int32_t i = istar; i >= 3; i--) {
        j = bp[(size_t)i * (size_t)p + (size_t)j];
        Q_idx[i - 2] = j;
    }
    Q_idx[0] = bp[2 * (size_t)p + (size_t)j];
    *m_out = istar;
    *best_out = best;
    if (dp_out) memcpy(dp_out, dp, sizeof(double) * rows * (size_t)p);
    if (bp_out) memcpy(bp_out, bp, sizeof(int32_t) * rows * (size_t)p);
    if (margin_out) memcpy(margin_out, mg, sizeof(double) * rows * (size_t)p);
    free(dp); free(bp); free(mg);
    return OR_OK;
}

/* Columns 1 <= j < jend of the column-by-column DP into dp, bp, mg ((s+1) x p,
 * preset to +inf / -1 / +inf): the base layer, then layers 3..s of each column in
 * increasing j; W holds one column's link costs. */
static void apx_columns_fill(const or_hist *H, int32_t s, double lam_prime, int64_t jend, double *dp, int32_t *bp,
                             double *mg, double *W) {
    int64_t p = H->p;
    /* base layer: as or_apx_dp */
    for (int64_t j = 1; j < jend; j++) {
        double best = INFINITY;
        int64_t arg = -1;
        for (int64_t a = 0; a < H->nL && a < j; a++) {
            double C, U, D;
            pair_q(H, a, j, &C, &U, &D);
            double c = C + lam_prime * phi_of(H, U, D, a);
            if (c < best) { best = c; arg = a; }
        }
        dp[2 * (size_t)p + (size_t)j] = best;
        bp[2 * (size_t)p + (size_t)j] = (int32_t)arg;
    }
    for (int64_t j = 1; j < jend; j++) {
        if (s < 3) break;
#pragma omp parallel for schedule(static)
        for (int64_t k = 0; k < j; k++) {
            double C, Phi;
            cphi(H, k, j, &C, &Phi);
            W[k] = C + lam_prime * Phi;
        }
        int32_t itop = s < (int32_t)(j + 1) ? s : (int32_t)(j + 1);  /* layers with j >= i - 1 */
#pragma omp parallel for schedule(dynamic, 1)
        for (int32_t i = 3; i <= itop; i++) {
            const double *prev = dp + (size_t)(i - 1) * (size_t)p;
            double best = INFINITY, second = INFINITY;
            int64_t arg = -1;
            for (int64_t k = i - 2; k < j; k++) {
                double cand = prev[k] + W[k];
                if (cand < best) { second = best; best = cand; arg = k; }
                else if (cand < second) second = cand;
            }
            size_t o = (size_t)i * (size_t)p + (size_t)j;
            dp[o] = best;
            bp[o] = (int32_t)arg;
            mg[o] = (best > 0.0) ? (second - best) / best : (second > best ? INFINITY : 0.0);
        }
    }
}

/* The same DP as or_apx_dp (same tables, same codebook), evaluated column by
 * column so that inputs far too large for the pair memo stay practical: for
 * each j, in increasing order, the link costs C[k, j] + lambda' Phi[k, j] of
 * every k < j are computed once (in parallel over k) and every layer
 * i = 3..s then takes its minimum over k in [i-2, j-1] of
 * dp(i-1, k) + (C + lambda' Phi) -- the binary64 candidate of or_apx_dp,
 * lowest k among exact minima, the same second-best margin.  dp(i-1, k) for
 * k < j is final when column j is reached, because every k < j was visited
 * earlier.  Memory: the (s+1) x p tables plus one column.
 * Used by the one-off full-size checks, where or_apx_dp would recompute each
 * pair once per layer. */
int32_t or_apx_dp_columns(const or_hist *H, int32_t s, double lam_prime, int32_t exact_s,
                          double *dp_out, int32_t *bp_out, double *margin_out,
                          int64_t *Q_idx, int32_t *m_out, double *best_out) {
    int64_t p = H->p;
    if (s < 2) return OR_EINVAL;
    if (p == 1) {
        Q_idx[0] = 0; *m_out = 1; *best_out = 0.0;
        return OR_OK;
    }
    size_t rows = (size_t)s + 1;
    double *dp = (double *)malloc(sizeof(double) * rows * (size_t)p);
    int32_t *bp = (int32_t *)malloc(sizeof(int32_t) * rows * (size_t)p);
    double *mg = (double *)malloc(sizeof(double) * rows * (size_t)p);
    double *W = (double *)malloc(sizeof(double) * (size_t)p);
    if (!dp || !bp || !mg || !W) { free(dp); free(bp); free(mg); free(W); return OR_ENOMEM; }
    for (size_t t = 0; t < rows * (size_t)p; t++) { dp[t] = INFINITY; bp[t] = -1; mg[t] = INFINITY; }
    apx_columns_fill(H, s, lam_prime, p, dp, bp, mg, W);
    free(W);
    int32_t istar = -1;
    int64_t jstar = -1;
    double best = INFINITY;
    int32_t ilo = exact_s ? s : 2;
    for (int32_t i = ilo; i <= s; i++)
        for (int64_t jr = p - H->nR; jr < p; jr++) {
            double v = dp[(size_t)i * (size_t)p + (size_t)jr];
            if (v < best) { best = v; istar = i; jstar = jr; }
        }
    if (istar < 0) { free(dp); free(bp); free(mg); return OR_EINFEASIBLE; }
    int64_t j = jstar;
    Q_idx[istar - 1] = j;
    for (int32_t i = istar; i >= 3; i--) {
        j = bp[(size_t)i * (size_t)p + (size_t)j];
        Q_idx[i - 2] = j;
    }
    Q_idx[0] = bp[2 * (size_t)p + (size_t)j];
    *m_out = istar;
    *best_out = best;
    if (dp_out) memcpy(dp_out, dp, sizeof(double) * rows * (size_t)p);
    if (bp_out) memcpy(bp_out, bp, sizeof(int32_t) * rows * (size_t)p);
    if (margin_out) memcpy(margin_out, mg, sizeof(double) * rows * (size_t)p);
    free(dp); free(bp); free(mg);
    return OR_OK;
}

/* The tables of or_apx_dp_columns for the columns j < jend alone (0 < jend <= p):
 * dp(i, j) reads only columns k < j, so these entries are the whole DP's.  For
 * full-size checks whose whole DP would take too long; the codebook (eq. apx_final)
 * needs every column and is not formed.  Entries of columns >= jend: +inf, -1, +inf. */
int32_t or_apx_dp_columns_prefix(const or_hist *H, int32_t s, double lam_prime, int64_t jend, double *dp_out,
                                 int32_t *bp_out, double *margin_out) {
    int64_t p = H->p;
    if (s < 2 || jend < 1 || jend > p || !dp_out || !bp_out || !margin_out) return OR_EINVAL;
    size_t rows = (size_t)s + 1;
    double *W = (double *)malloc(sizeof(double) * (size_t)p);
    if (!W) return OR_ENOMEM;
    for (size_t t = 0; t < rows * (size_t)p; t++) { dp_out[t] = INFINITY; bp_out[t] = -1; margin_out[t] = INFINITY; }
    apx_columns_fill(H, s, lam_prime, jend, dp_out, bp_out, margin_out, W);
    free(W);
    return OR_OK;
}

/* Linear-space traceback of the approximate DP (Sec. 5, last paragraph: Hirschberg's
 * method specialised to eq. apx_rec).  Link cost of consecutive values k < j:
 * C[k, j] + lambda' Phi[k, j], with Phi^first when k is the first value (index 0, P = X).
 *   1. A forward pass over the layers of eq. apx_rec keeping two rows finds the answer of
 *      eq. apx_final: m = the smallest i with the least dp(i, p-1).
 *   2. Subproblem (u, v, n): the n values of the chain with u and v fixed at its ends.
 *      For n >= 3 the middle position is t = (n + 1) / 2.  The forward pass from u gives
 *      G(c), the least cost of a chain of t values from u to c; the backward pass to v
 *      gives B(c), the least cost of a chain of n - t + 1 values from c to v (suffix
 *      costs, links taken from the right).  The middle value is the lowest c, u < c < v,
 *      among the exact binary64 minima of G(c) + B(c); recurse on (u, c, t) and
 *      (c, v, n - t + 1).  Each pass keeps two rows of p values.
 * Reading (the paper gives none): ties of G + B go to the lowest c.  The sums G + B add
 * a prefix and a suffix cost, in a different order from the forward recurrence, so at
 * exact or near ties the codebook may differ from or_apx_dp's (whose traceback takes
 * the lowest k at every step from the end); its objective is the same optimum.
 * Q_idx receives the codebook, m its size, best = dp(m, p-1) of the forward pass. */
static double link_cost(const or_hist *H, int64_t k, int64_t j, double lam_prime) {
    double C, U, D;
    pair_q(H, k, j, &C, &U, &D);
    return C + lam_prime * phi_of(H, U, D, k == 0 ? 0 : -1);
}

int32_t or_apx_dp_linear(const or_hist *H, int32_t s, double lam_prime, int32_t exact_s, int64_t *Q_idx,
                         int32_t *m_out, double *best_out) {
    int64_t p = H->p;
    if (s < 2 || H->nL != 1 || H->nR != 1) return OR_EINVAL;
    if (p == 1) { Q_idx[0] = 0; *m_out = 1; *best_out = 0.0; return OR_OK; }
    double *r0 = (double *)malloc(sizeof(double) * (size_t)p);
    double *r1 = (double *)malloc(sizeof(double) * (size_t)p);
    double *r2 = (double *)malloc(sizeof(double) * (size_t)p);
    double *r3 = (double *)malloc(sizeof(double) * (size_t)p);
    int64_t *stk = (int64_t *)malloc(sizeof(int64_t) * 3 * (size_t)(s + 2));
    if (!r0 || !r1 || !r2 || !r3 || !stk) { free(r0); free(r1); free(r2); free(r3); free(stk); return OR_ENOMEM; }
    /* 1. forward pass: dp(i, p-1) for every i */
    double best = INFINITY;
    int32_t m = -1;
    double *prev = r0, *cur = r1;
    for (int64_t j = 0; j < p; j++) prev[j] = INFINITY;
    for (int64_t j = 1; j < p; j++) prev[j] = link_cost(H, 0, j, lam_prime);  /* layer 2 */
    for (int32_t i = 2; i <= s; i++) {
        if (i > 2) {
            for (int64_t j = 0; j < p; j++) cur[j] = INFINITY;
#pragma omp parallel for schedule(dynamic, 8)
            for (int64_t j = i - 1; j < p; j++) {
                double b = INFINITY;
                for (int64_t k = i - 2; k < j; k++) {
                    double c = prev[k] + link_cost(H, k, j, lam_prime);
                    if (c < b) b = c;
                }
                cur[j] = b;
            }
            double *t = prev; prev = cur; cur = t;
        }
        if ((!exact_s || i == s) && prev[p - 1] < best) { best = prev[p - 1]; m = i; }
    }
    if (m < 0) { free(r0); free(r1); free(r2); free(r3); free(stk); return OR_EINFEASIBLE; }
    /* 2. the chain, by splitting at middle values */
    Q_idx[0] = 0;
    Q_idx[m - 1] = p - 1;
    int32_t top = 0;
    stk[0] = 0; stk[1] = p - 1; stk[2] = m;  /* (u, v, n); Q_idx position of u = pos below */
    int64_t *pos = (int64_t *)malloc(sizeof(int64_t) * (size_t)(s + 2));
    pos[0] = 0;
    top = 1;
    while (top > 0) {
        top--;
        int64_t u = stk[3 * top], v = stk[3 * top + 1], n = stk[3 * top + 2], pu = pos[top];
        if (n <= 2) continue;
        int64_t t = (n + 1) / 2;
        /* forward from u: G_r(c) for c in (u, v), r = 2..t */
        double *G = r0, *Gn = r1;
        for (int64_t c = u; c <= v; c++) G[c] = INFINITY;
        for (int64_t c = u + 1; c < v; c++) G[c] = link_cost(H, u, c, lam_prime);
        for (int64_t r = 3; r <= t; r++) {
            for (int64_t c = u; c <= v; c++) Gn[c] = INFINITY;
#pragma omp parallel for schedule(dynamic, 8)
            for (int64_t c = u + r - 1; c < v; c++) {
                double b = INFINITY;
                for (int64_t k = u + r - 2; k < c; k++) {
                    double x = G[k] + link_cost(H, k, c, lam_prime);
                    if (x < b) b = x;
                }
                Gn[c] = b;
            }
            double *tt = G; G = Gn; Gn = tt;
        }
        /* backward to v: B_r(c) for c in (u, v), r = 2..n-t+1 */
        double *B = r2, *Bn = r3;
        for (int64_t c = u; c <= v; c++) B[c] = INFINITY;
        for (int64_t c = u + 1; c < v; c++) B[c] = link_cost(H, c, v, lam_prime);
        for (int64_t r = 3; r <= n - t + 1; r++) {
            for (int64_t c = u; c <= v; c++) Bn[c] = INFINITY;
#pragma omp parallel for schedule(dynamic, 8)
            for (int64_t c = u + 1; c <= v - (r - 1); c++) {
                double b = INFINITY;
                for (int64_t j = c + 1; j <= v - (r - 2); j++) {
                    double x = link_cost(H, c, j, lam_prime) + B[j];
                    if (x < b) b = x;
                }
                Bn[c] = b;
            }
            double *tt = B; B = Bn; Bn = tt;
        }
        int64_t cs = -1;
        double sb = INFINITY;
        for (int64_t c = u + 1; c < v; c++) {
            double x = G[c] + B[c];
            if (x < sb) { sb = x; cs = c; }
        }
        if (cs < 0) { free(r0); free(r1); free(r2); free(r3); free(stk); free(pos); return OR_EINFEASIBLE; }
        Q_idx[pu + t - 1] = cs;
        stk[3 * top] = u; stk[3 * top + 1] = cs; stk[3 * top + 2] = t; pos[top] = pu; top++;
        stk[3 * top] = cs; stk[3 * top + 1] = v; stk[3 * top + 2] = n - t + 1; pos[top] = pu + t - 1; top++;
    }
    *m_out = m;
    *best_out = best;
    free(r0); free(r1); free(r2); free(r3); free(stk); free(pos);
    return OR_OK;
}

/* One decision of eq. apx_rec against a caller-given previous layer:
 * min over k in [i-2, j-1] of prev[k] + (C[k,j] + lambda' Phi[k,j]).
 * Used to check single outputs of large GPU runs. */
void or_dp_decision(const or_hist *H, const double *prev, int32_t i, int64_t j, double lam_prime,
                    double *best_out, int64_t *arg_out, double *second_out) {
    double best = INFINITY, second = INFINITY;
    int64_t arg = -1;
    for (int64_t k = i - 2; k < j; k++) {
        double C, Phi;
        cphi(H, k, j, &C, &Phi);
        double cand = prev[k] + (C + lam_prime * Phi);
        if (cand < best) { second = best; best = cand; arg = k; }
        else if (cand < second) second = cand;
    }
    *best_out = best; *arg_out = arg; *second_out = second;
}

/* Value of one candidate of eq. apx_rec (or eq. apx_base when first != 0). */
double or_dp_candidate(const or_hist *H, double prev_k, int64_t k, int64_t j, double lam_prime, int32_t first) {
    double C, U, D;
    pair_q(H, k, j, &C, &U, &D);
    if (first) return C + lam_prime * phi_of(H, U, D, k);
    return prev_k + (C + lam_prime * phi_of(H, U, D, -1));
}

/* ------------------------------------------------------------- ASQ DP */

/* Sec. 2, eq. asqdp: dp(2, j) = C[0, j]; dp(i, j) = min_{k<=j} dp(i-1,k) + C[k,j]
 * (C[j,j] = 0); answer dp(s, p-1), the least MSE with at most s values. */
int32_t or_asq_dp(const or_hist *H, int32_t s, double *best_out) {
    int64_t p = H->p;
    if (s < 2) return OR_EINVAL;
    if (p == 1) { *best_out = 0.0; return OR_OK; }
    double *a = (double *)malloc(sizeof(double) * (size_t)p);
    double *b = (double *)malloc(sizeof(double) * (size_t)p);
    if (!a || !b) { free(a); free(b); return OR_ENOMEM; }
    a[0] = 0.0;  /* a single value at v_0 quantizes the prefix {v_0} exactly */
    for (int64_t j = 1; j < p; j++) {
        double C, U, D;
        pair_q(H, 0, j, &C, &U, &D);
        a[j] = C;
    }
    for (int32_t i = 3; i <= s; i++) {
        for (int64_t j = 0; j < p; j++) {
            double best = a[j];  /* k = j */
            for (int64_t k = 0; k < j; k++) {
                double C, U, D;
                pair_q(H, k, j, &C, &U, &D);
                double c = a[k] + C;
                if (c < best) best = c;
            }
            b[j] = best;
        }
        double *t = a; a = b; b = t;
    }
    *best_out = a[p - 1];
    free(a); free(b);
    return OR_OK;
}

/* ---------------------------------------------------------- optimal DP */

/* Sec. 4 with App. E's conventions (L = {0..nL-1}, R = {p-nR..p-1}), naive O(s p^3):
 *   dp(2, a, j)  = C[a, j] + lambda' h((n_a + D[a, j]) / d),  a in L, a < j
 *   dp(i, l, j)  = C[l, j] + min_{k<l} dp(i-1, k, l) + lambda' h((U[k,l] + D[l,j]) / d),  i >= 3
 *   answer       = min_{2<=i<=s} min_{j in R} min_{l<j} dp(i, l, j) + lambda' h(U[l, j] / d)
 * Ties: lowest k; at the answer the smallest i, then j, then l.
 * The traced codebook goes to Q_idx / m.  Memory s p^2 doubles. */
int32_t or_opt_dp(const or_hist *H, int32_t s, double lam_prime, int32_t exact_s,
                  double *best_out, int64_t *Q_idx, int32_t *m_out) {
    int64_t p = H->p;
    double dd = (double)H->d;
    if (s < 2) return OR_EINVAL;
    if (p == 1) { *best_out = 0.0; Q_idx[0] = 0; *m_out = 1; return OR_OK; }
    size_t pp = (size_t)p * (size_t)p;
    double *U = (double *)malloc(sizeof(double) * pp);
    double *D = (double *)malloc(sizeof(double) * pp);
    double *C = (double *)malloc(sizeof(double) * pp);
    double *dp = (double *)malloc(sizeof(double) * pp * (size_t)(s + 1));
    int64_t *bk = (int64_t *)malloc(sizeof(int64_t) * pp * (size_t)(s + 1));
    if (!U || !D || !C || !dp || !bk) { free(U); free(D); free(C); free(dp); free(bk); return OR_ENOMEM; }
    for (int64_t k = 0; k < p; k++)
        for (int64_t j = 0; j < p; j++) {
            size_t t = (size_t)k * (size_t)p + (size_t)j;
            if (k < j) pair_q(H, k, j, &C[t], &U[t], &D[t]);
            else { C[t] = 0.0; U[t] = 0.0; D[t] = 0.0; }
        }
#define DPO(i, l, j) dp[((size_t)(i) * (size_t)p + (size_t)(l)) * (size_t)p + (size_t)(j)]
#define BKO(i, l, j) bk[((size_t)(i) * (size_t)p + (size_t)(l)) * (size_t)p + (size_t)(j)]
    for (size_t t = 0; t < pp * (size_t)(s + 1); t++) { dp[t] = INFINITY; bk[t] = -1; }
    for (int64_t a = 0; a < H->nL; a++)
        for (int64_t j = a + 1; j < p; j++)
            DPO(2, a, j) = C[(size_t)a * p + j] + lam_prime * h(((double)H->w[a] + D[(size_t)a * p + j]) / dd);
    for (int32_t i = 3; i <= s; i++) {
#pragma omp parallel for schedule(dynamic, 4)
        for (int64_t l = 1; l < p; l++)
            for (int64_t j = l + 1; j < p; j++) {
                double best = INFINITY;
                int64_t arg = -1;
                for (int64_t k = 0; k < l; k++) {
                    double prev = DPO(i - 1, k, l);
                    if (!(prev < INFINITY)) continue;
                    double c = prev + lam_prime * h((U[(size_t)k * p + l] + D[(size_t)l * p + j]) / dd);
                    if (c < best) { best = c; arg = k; }
                }
                if (arg >= 0) { DPO(i, l, j) = C[(size_t)l * p + j] + best; BKO(i, l, j) = arg; }
            }
    }
    double best = INFINITY;
    int32_t bi = -1;
    int64_t bl = -1, bj = -1;
    for (int32_t i = exact_s ? s : 2; i <= s; i++)
        for (int64_t jr = p - H->nR; jr < p; jr++)
            for (int64_t l = 0; l < jr; l++) {
                double v = DPO(i, l, jr);
                if (!(v < INFINITY)) continue;
                double c = v + lam_prime * h(U[(size_t)l * p + (size_t)jr] / dd);
                if (c < best) { best = c; bi = i; bl = l; bj = jr; }
            }
    if (bi < 0) { free(U); free(D); free(C); free(dp); free(bk); return OR_EINFEASIBLE; }
    /* traceback: state (i, l, j) -> (i-1, k, l) */
    int64_t l = bl, j = bj;
    Q_idx[bi - 1] = j;
    for (int32_t i = bi; i >= 3; i--) {
        Q_idx[i - 2] = l;
        int64_t k = BKO(i, l, j);
        j = l; l = k;
    }
    Q_idx[0] = l;
    *m_out = bi;
    *best_out = best;
#undef DPO
#undef BKO
    free(U); free(D); free(C); free(dp); free(bk);
    return OR_OK;
}

/* --------------------------------------------------------- brute force */

/* Enumerate every codebook Q subset of the unique values with v_0, v_{p-1} in Q
 * and |Q| <= s, scored with the per-entry definitions (or_eval_direct).
 * out[0] min MSE + lambda' H(I,B)        out[1] min MSE + lambda' H(Xhat)
 * out[2] min MSE s.t. H(I,B) <= b        out[3] min MSE s.t. H(Xhat) <= b - 1
 * out[4] H(Xhat) of the out[2] minimiser out[5] min MSE (no entropy term)
 * masks[0..3]: the interior-value bitmask attaining out[0..3] (first found).
 * Ties keep the first mask in increasing mask order.  p <= 20. */
int32_t or_brute(const float *x, int64_t d, int32_t s, double lam_prime, double budget,
                 double *out, int64_t *masks) {
    int32_t st;
    or_hist *H = or_hist_new(x, d, &st);
    if (!H) return st;
    int64_t p = H->p;
    if (p > 20 || s < 2) { or_hist_free(H); return OR_EINVAL; }
    double *Q = (double *)malloc(sizeof(double) * (size_t)p);
    for (int r = 0; r < 6; r++) out[r] = INFINITY;
    for (int r = 0; r < 4; r++) masks[r] = -1;
    out[4] = NAN;
    int64_t ni = p >= 2 ? p - 2 : 0;
    int64_t nmask = (int64_t)1 << ni;
    for (int64_t mask = 0; mask < nmask; mask++) {
        int32_t m = 0;
        Q[m++] = (double)H->v[0];
        for (int64_t t = 0; t < ni; t++)
            if (mask >> t & 1) Q[m++] = (double)H->v[t + 1];
        if (p >= 2) Q[m++] = (double)H->v[p - 1];
        if (m > s) continue;
        double ev[3];
        if (or_eval_direct(x, d, Q, m, ev) != OR_OK) continue;
        double js = ev[0] + lam_prime * ev[1], jt = ev[0] + lam_prime * ev[2];
        if (js < out[0]) { out[0] = js; masks[0] = mask; }
        if (jt < out[1]) { out[1] = jt; masks[1] = mask; }
        if (ev[1] <= budget && ev[0] < out[2]) { out[2] = ev[0]; masks[2] = mask; out[4] = ev[2]; }
        if (ev[2] <= budget - 1.0 && ev[0] < out[3]) { out[3] = ev[0]; masks[3] = mask; }
        if (ev[0] < out[5]) out[5] = ev[0];
    }
    free(Q);
    or_hist_free(H);
    return OR_OK;
}

/* The enumeration of or_brute over codebooks drawn from a permissible set P
 * (ascending, n <= 16): every subset of P with 2 <= |Q| <= s, Q[0] <= min x and
 * Q[last] >= max x (Sec. 5: q_1 <= x_1, q_t >= x_d), scored with the per-entry
 * definitions.  Outputs as or_brute; masks are bitmasks over all n values of P. */
int32_t or_brute_grid(const float *x, int64_t d, const float *P, int64_t n, int32_t s, double lam_prime,
                      double budget, double *out, int64_t *masks) {
    if (!x || d < 1 || !P || n < 1 || n > 16 || s < 2) return OR_EINVAL;
    float xmin = x[0], xmax = x[0];
    for (int64_t i = 1; i < d; i++) {
        if (x[i] < xmin) xmin = x[i];
        if (x[i] > xmax) xmax = x[i];
    }
    double Q[16];
    for (int r = 0; r < 6; r++) out[r] = INFINITY;
    for (int r = 0; r < 4; r++) masks[r] = -1;
    out[4] = NAN;
    for (int64_t mask = 1; mask < ((int64_t)1 << n); mask++) {
        int32_t m = 0;
        for (int64_t t = 0; t < n; t++)
            if (mask >> t & 1) Q[m++] = (double)P[t];
        if (m < 2 || m > s || !(Q[0] <= (double)xmin) || !(Q[m - 1] >= (double)xmax)) continue;
        double ev[3];
        if (or_eval_direct(x, d, Q, m, ev) != OR_OK) continue;
        double js = ev[0] + lam_prime * ev[1], jt = ev[0] + lam_prime * ev[2];
        if (js < out[0]) { out[0] = js; masks[0] = mask; }
        if (jt < out[1]) { out[1] = jt; masks[1] = mask; }
        if (ev[1] <= budget && ev[0] < out[2]) { out[2] = ev[0]; masks[2] = mask; out[4] = ev[2]; }
        if (ev[2] <= budget - 1.0 && ev[0] < out[3]) { out[3] = ev[0]; masks[3] = mask; }
        if (ev[0] < out[5]) out[5] = ev[0];
    }
    return OR_OK;
}

/* ------------------------------------------------------- lambda search */

/* The seven interior points of [lo, hi] from three levels of geometric
 * midpoints sqrt(a*b) (correctly rounded multiply and sqrt only). */
void or_midpoints7(double lo, double hi, double *t) {
    t[3] = sqrt(lo * hi);
    t[1] = sqrt(lo * t[3]);
    t[5] = sqrt(t[3] * hi);
    t[0] = sqrt(lo * t[1]);
    t[2] = sqrt(t[1] * t[3]);
    t[4] = sqrt(t[3] * t[5]);
    t[6] = sqrt(t[5] * hi);
}

typedef struct { double lam, mse, hs, hx; int32_t m; int32_t feasible; } or_point;

static int32_t eval_lambda(const or_hist *H, int32_t s, double lam, int32_t exact_s, double budget,
                           or_point *pt, int64_t *Qbuf) {
    int32_t m;
    double best, ev[3];
    int32_t st = or_apx_dp(H, s, lam * H->norm2, exact_s, NULL, NULL, NULL, Qbuf, &m, &best);
    if (st != OR_OK) return st;
    st = or_eval_idx(H, Qbuf, m, ev);
    if (st != OR_OK) return st;
    pt->lam = lam; pt->mse = ev[0]; pt->hs = ev[1]; pt->hx = ev[2]; pt->m = m;
    pt->feasible = ev[1] <= budget;
    return OR_OK;
}

/* Budgeted solve (Sec. 3: "by a binary search for lambda we can respect the
 * entropy constraint"; Sec. 5: keep the lowest-MSE solution whose surrogate
 * entropy H(I,B) is at most b).  Schedule:
 *   pass 1: lambda in {0} + midpoints7(lo, hi); if lambda = 0 is feasible it is the answer;
 *   passes 2..rounds: midpoints7 of the bracket [t_{f-1}, t_f] around the smallest
 *     feasible point t_f (t_0 = lo), or [t_7, hi] when none is feasible;
 *   if no evaluated point is feasible: evaluate hi; still infeasible -> OR_EINFEASIBLE
 *     (the hi solution is returned);
 *   answer: minimum MSE over the feasible evaluated points, ties to the smaller lambda.
 * trace (cap rows of 6 doubles): lam, mse, H(I,B), H(Xhat), m, feasible.
 * res: lam, mse, H(I,B), H(Xhat). */
/* plus: when not NULL, also the evaluated infeasible point of least H(I,B)
 * (ties: less MSE, then the smaller lambda) and its codebook (Sec. 7's Q+). */
typedef struct { or_point pt; int64_t *Q; int have; } or_plus;

static int32_t search_core(const or_hist *H, int32_t s, double budget, double lo, double hi, int32_t rounds,
                           int32_t exact_s, int64_t *Q_idx, int32_t *m_out, double *res,
                           double *trace, int32_t trace_cap, int32_t *n_trace, or_plus *plus) {
    if (!(budget >= 0.0) || !(lo > 0.0) || !(hi > lo) || rounds < 1 || s < 2) return OR_EINVAL;
    int64_t *Qb = (int64_t *)malloc(sizeof(int64_t) * (size_t)(s + 1));
    int64_t *Qbest = (int64_t *)malloc(sizeof(int64_t) * (size_t)(s + 1));
    or_point best = {0};
    int have = 0, nt = 0;
    int32_t st = OR_OK, status = OR_OK;
#define RECORD(pt)                                                                   \
    do {                                                                             \
        if (nt < trace_cap) {                                                        \
            double *r_ = trace + 6 * (size_t)nt;                                     \
            r_[0] = (pt).lam; r_[1] = (pt).mse; r_[2] = (pt).hs; r_[3] = (pt).hx;    \
            r_[4] = (pt).m; r_[5] = (pt).feasible;                                   \
        }                                                                            \
        nt++;                                                                        \
        if ((pt).feasible && (!have || (pt).mse < best.mse ||                        \
                              ((pt).mse == best.mse && (pt).lam < best.lam))) {      \
            best = (pt); have = 1; memcpy(Qbest, Qb, sizeof(int64_t) * (size_t)(pt).m); \
        }                                                                            \
        if (plus && !(pt).feasible &&                                                \
            (!plus->have || (pt).hs < plus->pt.hs ||                                 \
             ((pt).hs == plus->pt.hs && ((pt).mse < plus->pt.mse ||                  \
                                         ((pt).mse == plus->pt.mse && (pt).lam < plus->pt.lam))))) { \
            plus->pt = (pt); plus->have = 1;                                         \
            memcpy(plus->Q, Qb, sizeof(int64_t) * (size_t)(pt).m);                   \
        }                                                                            \
    } while (0)
    or_point pt;
    st = eval_lambda(H, s, 0.0, exact_s, budget, &pt, Qb);
    if (st != OR_OK) goto done;
    RECORD(pt);
    if (!pt.feasible) {
        for (int32_t r = 0; r < rounds; r++) {
            double t[7];
            or_midpoints7(lo, hi, t);
            int f = -1;
            for (int q = 0; q < 7; q++) {
                st = eval_lambda(H, s, t[q], exact_s, budget, &pt, Qb);
                if (st != OR_OK) goto done;
                RECORD(pt);
                if (pt.feasible && f < 0) f = q;
            }
            if (f >= 0) { double nlo = f > 0 ? t[f - 1] : lo; hi = t[f]; lo = nlo; }
            else lo = t[6];
        }
        if (!have) {
            st = eval_lambda(H, s, hi, exact_s, budget, &pt, Qb);
            if (st != OR_OK) goto done;
            RECORD(pt);
            if (!have) {
                status = OR_EINFEASIBLE;
                best = pt; memcpy(Qbest, Qb, sizeof(int64_t) * (size_t)pt.m);
            }
        }
    }
#undef RECORD
    memcpy(Q_idx, Qbest, sizeof(int64_t) * (size_t)best.m);
    *m_out = best.m;
    res[0] = best.lam; res[1] = best.mse; res[2] = best.hs; res[3] = best.hx;
    st = status;
done:
    *n_trace = nt;
    free(Qb); free(Qbest);
    return st;
}

int32_t or_search(const or_hist *H, int32_t s, double budget, double lo, double hi, int32_t rounds,
                  int32_t exact_s, int64_t *Q_idx, int32_t *m_out, double *res,
                  double *trace, int32_t trace_cap, int32_t *n_trace) {
    return search_core(H, s, budget, lo, hi, rounds, exact_s, Q_idx, m_out, res, trace, trace_cap, n_trace, NULL);
}

/* Two-way time-sharing (Sec. 7).  Q- is the budgeted solve's answer (least MSE with
 * H(I,B) = b- <= b); Q+ is the evaluated point of least rate b+ > b.  Each entry
 * uses Q+ with probability beta = (b - b-)/(b+ - b-), so the expected MSE and rate
 * are the beta-mixtures of the two.  Readings: the rate is H(I,B), the quantity the
 * budget constrains; beta = 0 (no Q+) when every evaluated point is feasible, when
 * b- = b, or when Q+ does not have less MSE than Q- (time-sharing cannot help).
 * out: beta, lam-, lam+, and the mixture's MSE, H(I,B), H(Xhat); m_plus = 0 without Q+.
 * The search runs as or_search; status as or_search. */
int32_t or_timeshare(const or_hist *H, int32_t s, double budget, double lo, double hi, int32_t rounds,
                     int32_t exact_s, int64_t *Qm_idx, int32_t *m_minus, int64_t *Qp_idx, int32_t *m_plus,
                     double *minus_met, double *plus_met, double *out) {
    double res[4];
    double trace[6];
    int32_t nt;
    or_plus plus;
    plus.have = 0;
    plus.Q = Qp_idx;
    int32_t st = search_core(H, s, budget, lo, hi, rounds, exact_s, Qm_idx, m_minus, res, trace, 0, &nt, &plus);
    if (st != OR_OK) return st;
    minus_met[0] = res[1]; minus_met[1] = res[2]; minus_met[2] = res[3];
    double beta = 0.0;
    if (plus.have && plus.pt.mse < res[1] && res[2] < budget)
        beta = (budget - res[2]) / (plus.pt.hs - res[2]);
    if (beta > 0.0) {
        *m_plus = plus.pt.m;
        plus_met[0] = plus.pt.mse; plus_met[1] = plus.pt.hs; plus_met[2] = plus.pt.hx;
        out[2] = plus.pt.lam;
    } else {
        *m_plus = 0;
        plus_met[0] = plus_met[1] = plus_met[2] = NAN;
        out[2] = NAN;
    }
    out[0] = beta;
    out[1] = res[0];
    for (int r = 0; r < 3; r++)
        out[3 + r] = beta > 0.0 ? (1.0 - beta) * minus_met[r] + beta * plus_met[r] : minus_met[r];
    return OR_OK;
}

/* ----------------------------------------------------------- refinement */

static double objective_true(const or_hist *H, const int64_t *a, int32_t m, double lam_prime, double *hx_out) {
    double ev[3];
    or_eval_idx(H, a, m, ev);
    if (hx_out) *hx_out = ev[2];
    return ev[0] + lam_prime * ev[2];
}

/* Local objective of Sec. 6 for moving a[l] to unique index c (a[l-1] < c < a[l+1]):
 * C[a_{l-1}, c] + C[c, a_{l+1}] + lambda' (h(f_{l-1}/d) + h(f_l/d) + h(f_{l+1}/d)). */
static double local_obj(const or_hist *H, const int64_t *a, int32_t m, int32_t l, int64_t c, double lam_prime) {
    double dd = (double)H->d;
    int64_t L = a[l - 1], R = a[l + 1];
    double C1, U1, D1, C2, U2, D2;
    pair_q(H, L, c, &C1, &U1, &D1);
    pair_q(H, c, R, &C2, &U2, &D2);
    double fl;
    if (l - 1 == 0) fl = (double)H->w[a[0]] + D1;
    else { double Cx, Ux, Dx; pair_q(H, a[l - 2], L, &Cx, &Ux, &Dx); fl = Ux + D1; }
    double fm = U1 + D2;
    double fr;
    if (l + 1 == m - 1) fr = U2;
    else { double Cx, Ux, Dx; pair_q(H, R, a[l + 2], &Cx, &Ux, &Dx); fr = U2 + Dx; }
    return (C1 + C2) + lam_prime * ((h(fl / dd) + h(fm / dd)) + h(fr / dd));
}

/* Three-colour refinement (Sec. 6).  a[0..m-1] (unique indices) is updated in
 * place.  Colour c moves the interior values l = 1..m-2 with l % 3 == c, each
 * to its best position strictly between its fixed neighbours.  With guard != 0
 * a colour step whose H(Xhat) exceeds budget is undone.  A round is the three
 * colour steps in order 0, 1, 2; refinement stops after a round that does not
 * lower J = MSE + lambda' H(Xhat) by more than tol * |J| (Sec. 6 evaluation:
 * stop once a complete round fails to decrease the objective), or after max_rounds.
 * J_trace (max_rounds + 1 entries) receives J before round 1 and after each. */
int32_t or_refine(const or_hist *H, int64_t *a, int32_t m, double lam_prime, double budget,
                  int32_t guard, int32_t max_rounds, double tol, int32_t *rounds_used, double *J_trace) {
    *rounds_used = 0;
    if (m < 3) { if (J_trace) J_trace[0] = objective_true(H, a, m, lam_prime, NULL); return OR_OK; }
    int64_t *nw = (int64_t *)malloc(sizeof(int64_t) * (size_t)m);
    double J = objective_true(H, a, m, lam_prime, NULL);
    if (J_trace) J_trace[0] = J;
    for (int32_t r = 0; r < max_rounds; r++) {
        double J0 = J;
        for (int32_t col = 0; col < 3; col++) {
            memcpy(nw, a, sizeof(int64_t) * (size_t)m);
            int moved = 0;
            for (int32_t l = 1; l <= m - 2; l++) {
                if (l % 3 != col) continue;
                double bestv = local_obj(H, a, m, l, a[l], lam_prime);
                int64_t bestc = a[l];
                for (int64_t c = a[l - 1] + 1; c < a[l + 1]; c++) {
                    if (c == a[l]) continue;
                    double v = local_obj(H, a, m, l, c, lam_prime);
                    if (v < bestv) { bestv = v; bestc = c; }
                }
                nw[l] = bestc;
                moved |= (bestc != a[l]);
            }
            if (!moved) continue;
            double hx;
            objective_true(H, nw, m, lam_prime, &hx);
            if (guard && hx > budget) continue;
            memcpy(a, nw, sizeof(int64_t) * (size_t)m);
        }
        J = objective_true(H, a, m, lam_prime, NULL);
        *rounds_used = r + 1;
        if (J_trace) J_trace[r + 1] = J;
        if (!(J0 - J > tol * fabs(J0))) break;
    }
    free(nw);
    return OR_OK;
}

/* ---------------------------------------------------------- quantization */

/* SplitMix64 output function (Steele, Lea and Flood, OOPSLA 2014). */
uint64_t or_splitmix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

/* Stochastic quantization (Sec. 2) of x[i] in its original order into Q
 * (ascending floats spanning x): a = max{q <= x}; if x == a the index of a,
 * else round up to the next value with the decision rule in the file header.
 * counts[m] receives the index histogram and h_emp its empirical entropy
 * (Sec. 1: -sum f log2 f with f the fraction of entries at each index). */
int32_t or_quantize(const float *x, int64_t d, const float *Q, int32_t m, uint64_t seed,
                    uint8_t *idx, uint32_t *counts, double *h_emp) {
    if (m < 1 || m > 256 || d < 1) return OR_EINVAL;
    for (int32_t r = 1; r < m; r++) if (!(Q[r] > Q[r - 1])) return OR_EINVAL;
    for (int32_t r = 0; r < m; r++) counts[r] = 0;
    for (int64_t i = 0; i < d; i++) {
        float xv = x[i];
        if (!(xv >= Q[0] && xv <= Q[m - 1])) return OR_ERANGE;
        int32_t lo = 0, hi = m - 1;       /* largest t with Q[t] <= x */
        while (lo < hi) {
            int32_t mid = (lo + hi + 1) / 2;
            if (Q[mid] <= xv) lo = mid; else hi = mid - 1;
        }
        int32_t t = lo;
        if (Q[t] != xv) {
            uint64_t z = or_splitmix64(seed + (uint64_t)(i + 1) * 0x9E3779B97F4A7C15ULL);
            float k = (float)(uint32_t)(z >> 40) * 0x1p-24f;
            float d1 = xv - Q[t];
            float d2 = Q[t + 1] - Q[t];
            float pr = k * d2;
            if (pr < d1) t += 1;
        }
        idx[i] = (uint8_t)t;
        counts[t]++;
    }
    double he = 0.0, dd = (double)d;
    for (int32_t r = 0; r < m; r++) he += h((double)counts[r] / dd);
    *h_emp = he;
    return OR_OK;
}

/* Time-shared stochastic quantization (Sec. 7 with Sec. 2): entry i (original order)
 * uses Q+ iff k_s * 2^-24 < beta, k_s the top 24 bits of SplitMix64(seed_ts +
 * (i+1)*0x9E3779B97F4A7C15) (binary64 compare, exact), then rounds within the chosen
 * codebook with the rule of or_quantize (seed, same counter i).  sel[i] = 1 for Q+.
 * counts: [mm] for Q-, then [mp] for Q+.  rate: the bits per entry of coding each
 * part with its own empirical law, -(1/d) sum_parts sum_r c_r log2(c_r / n_part). */
int32_t or_quantize_timeshare(const float *x, int64_t d, const float *Qm, int32_t mm, const float *Qp,
                              int32_t mp, double beta, uint64_t seed, uint64_t seed_ts, uint8_t *idx,
                              uint8_t *sel, uint32_t *counts, double *rate) {
    if (d < 1 || mm < 1 || mm > 256 || mp < 0 || mp > 256 || !(beta >= 0.0 && beta <= 1.0)) return OR_EINVAL;
    if (beta > 0.0 && mp < 1) return OR_EINVAL;
    for (int32_t r = 0; r < mm + mp; r++) counts[r] = 0;
    for (int64_t i = 0; i < d; i++) {
        uint64_t zs = or_splitmix64(seed_ts + (uint64_t)(i + 1) * 0x9E3779B97F4A7C15ULL);
        int use_plus = (double)(uint32_t)(zs >> 40) * 0x1p-24 < beta;
        const float *Q = use_plus ? Qp : Qm;
        int32_t m = use_plus ? mp : mm;
        float xv = x[i];
        if (!(xv >= Q[0] && xv <= Q[m - 1])) return OR_ERANGE;
        int32_t lo = 0, hi = m - 1;
        while (lo < hi) {
            int32_t mid = (lo + hi + 1) / 2;
            if (Q[mid] <= xv) lo = mid; else hi = mid - 1;
        }
        int32_t t = lo;
        if (Q[t] != xv) {
            uint64_t z = or_splitmix64(seed + (uint64_t)(i + 1) * 0x9E3779B97F4A7C15ULL);
            float k = (float)(uint32_t)(z >> 40) * 0x1p-24f;
            if (k * (Q[t + 1] - Q[t]) < xv - Q[t]) t += 1;
        }
        idx[i] = (uint8_t)t;
        if (sel) sel[i] = (uint8_t)use_plus;
        counts[(use_plus ? mm : 0) + t]++;
    }
    double bits = 0.0;
    for (int part = 0; part < 2; part++) {
        int32_t off = part ? mm : 0, m = part ? mp : mm;
        double n = 0.0;
        for (int32_t r = 0; r < m; r++) n += (double)counts[off + r];
        for (int32_t r = 0; r < m; r++)
            if (counts[off + r]) bits -= (double)counts[off + r] * log2((double)counts[off + r] / n);
    }
    *rate = bits / (double)d;
    return OR_OK;
}

/* Number of threads the OpenMP parts use. */
int32_t or_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
