/*
 * ecasq.h -- C ABI of the GB300 ECASQ library (Entropy-Constrained Adaptive
 * Stochastic Quantization, arxiv 2608.18147).
 *
 * Given x in R^d, a cap s on the codebook size and an entropy budget b
 * (bits per entry), ECASQ picks Q subset of X, |Q| <= s, spanning X, that
 * minimises the stochastic-quantization MSE subject to H(Xhat) <= b
 * (Sec. 1, "ECASQ solves ...").  The library implements the approximate
 * dynamic program of Sec. 5 (surrogate entropy H(I,B)), the multiplier search
 * of Sec. 3 / Sec. 5, the three-colour refinement of Sec. 6 and the unbiased
 * stochastic rounding of Sec. 2, on one GPU.
 *
 * Conventions shared by every entry point:
 *   - Pointers are DEVICE pointers unless the comment says "host".  The
 *     caller owns every buffer; the library never allocates device memory:
 *     all scratch comes from the caller's workspace (see ecasq_workspace_size).
 *     The workspace start must be 256-byte aligned.
 *   - Calls are ordered on `stream` (a cudaStream_t; NULL = legacy default).
 *     Entry points that return host results synchronise `stream` before
 *     returning.  Concurrent calls that share one workspace race.
 *   - x is fp32, length d >= 1, all finite (NaN/Inf -> ECASQ_ENONFINITE).
 *     -0.0 and +0.0 are the same value.  d < 2^31.
 *   - Q is an ascending fp32 codebook of m values, m <= s <= 256; Q[0] = min x
 *     and Q[m-1] = max x (Q spans X, Sec. 1).  m < s is allowed ("at most s",
 *     eq. apx_final).
 *   - lambda is on the vNMSE scale; the DP uses lambda' = lambda * ||X||^2
 *     (Sec. 3: vNMSE + lambda H  equals  MSE + lambda' H).
 *   - Return value: ECASQ_OK (0) or a negative status; ecasq_strerror names it.
 */
#ifndef ECASQ_H
#define ECASQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *ecasq_stream_t; /* same type as cudaStream_t */

#define ECASQ_OK 0
#define ECASQ_EINVAL (-1)      /* bad argument (d < 1, s outside [2,256], b < 0, null pointer, ...) */
#define ECASQ_ENONFINITE (-2)  /* x holds NaN or Inf */
#define ECASQ_EINFEASIBLE (-3) /* no evaluated multiplier meets the budget (result = largest multiplier's solution) */
#define ECASQ_EWORKSPACE (-4)  /* workspace smaller than ecasq_workspace_size() or misaligned */
#define ECASQ_ECUDA (-5)       /* a CUDA call failed (launch error, fault) */
#define ECASQ_ETIMEOUT (-6)    /* a bounded device-side wait ran out */
#define ECASQ_ERANGE (-7)      /* an entry of x lies outside [Q[0], Q[m-1]], or Q is not a subset of X */

/* flags */
#define ECASQ_EXACT_S 1u          /* use exactly s values (eq. apx_final with i = s only) */
#define ECASQ_NO_REFINE_GUARD 2u  /* refinement may raise H(Xhat) above the budget */
#define ECASQ_DP_REFERENCE 4u     /* run the fp64 reference DP kernel instead of the fast kernel */
#define ECASQ_TIME_KERNELS 8u     /* time the DP kernels with CUDA events (ecasq_result_t.dp_kernel_ms) */
#define ECASQ_EXACT_TABLES 16u    /* resolve every DP output exactly (default: only what eq. apx_final and the traceback read) */
#define ECASQ_RESIDENT_COSTS 32u  /* fast DP: compute the lambda-independent interval costs C and Phi (Sec. 5, App. E)
                                     once per call into the workspace and stream them to every pass (workspace:
                                     ecasq_workspace_size_flags with this flag; about 4.3 d^2 bytes extra) */
#define ECASQ_STREAMED_COSTS 64u  /* fast DP, for inputs whose full table does not fit: the interval-cost tiles of a
                                     band of column blocks at a time are built into a bounded buffer (about 64 columns
                                     of tiles, 2.3 MB x ceil(d / 64); ecasq_workspace_size_flags with this flag) and
                                     the wavefront runs band by band; rebuilt in every pass.  RESIDENT_COSTS wins
                                     when both are given.  Results are the same as with either other mode. */
#define ECASQ_ONE_PART_PUBLISH 128u /* fast DP with resident or streamed costs and 10 <= s <= 16: publish each column block
                                     of the wavefront once, after all its layers, instead of in two parts (rows 2..8
                                     after layer 8, then the rest); same results, for comparison */
#define ECASQ_UNSEEDED_SEARCH 256u /* fast DP with resident or streamed costs and tile skipping (10 <= s <= 18, 27 <= s <= 34): in the
                                     multiplier search, start every pass's tile skipping from scratch instead of from
                                     the fp32 minima of the bracket's evaluated upper end (an upper bound of every
                                     later pass's minima, Sec. 5's candidates being non-decreasing in lambda); same
                                     results, for comparison */
#define ECASQ_TEST_SELF_SEED (1u << 29) /* test hook for the seeded tile skipping: with a fixed multiplier and resident
                                     or streamed costs, the pass runs twice, the second time seeded with the first
                                     one's fp32 minima (the seed then equals every output's minimum, the tightest
                                     start the seeding allows); results must equal those without the flag.
                                     ecasq_result_t.passes counts both.  Not for production use. */
#define ECASQ_TEST_STALL (1u << 30) /* test hook for the bounded device waits: column block 0 of the fast DP's
                                     wavefront is never published and the flag waits give up after 2^14 spins, so
                                     the call must return ECASQ_ETIMEOUT (nothing else) and leave the workspace
                                     usable by the next call.  Not for production use. */

typedef struct ecasq_params {
    int32_t s;                 /* codebook cap, 2..256 */
    uint32_t flags;            /* ECASQ_* flags */
    double budget_bits;        /* b >= 0, bits per entry, compared with H(I,B) (Sec. 5) */
    double lambda;             /* < 0: search on the budget; >= 0: one fixed multiplier (vNMSE scale) */
    double lambda_lo;          /* search bracket (vNMSE scale); <= 0 selects 1e-8 */
    double lambda_hi;          /* <= 0 selects 1e3 */
    int32_t search_rounds;     /* rounds of 7 geometric midpoints; <= 0 selects 6 */
    int32_t refine_max_rounds; /* three-colour refinement rounds (Sec. 6); 0 = none */
    double refine_rel_tol;     /* stop once a round lowers J by <= tol*|J| (0: by nothing) */
} ecasq_params_t;

typedef struct ecasq_result {
    int32_t status;            /* same as the return value */
    int32_t m;                 /* |Q| */
    int32_t passes;            /* DP launches (each covers up to 8 multipliers) */
    int32_t lambdas_evaluated; /* multipliers evaluated by the search */
    int32_t refine_rounds;     /* refinement rounds executed */
    int32_t reserved;
    int64_t d, p;              /* entries, unique values */
    double lambda;             /* selected multiplier (vNMSE scale) */
    double lambda_prime;       /* lambda * ||X||^2 */
    double norm2;              /* ||X||^2 */
    double mse;                /* MSE(Q, X) = sum (b_x - x)(x - a_x)          (Sec. 2) */
    double vnmse;              /* mse / ||X||^2                               (Sec. 2) */
    double h_surrogate;        /* H(I,B), eq. apx_additive_entropy             (Sec. 5) */
    double h_exact;            /* H(Xhat)                                     (Sec. 3) */
    double r_tot;              /* H(Xhat) + 32 m / d                          (Sec. 3, 8) */
    double objective;          /* mse + lambda' * h_exact after refinement, else mse + lambda' * h_surrogate */
    int64_t candidates;        /* min-plus candidates evaluated by the DP (all passes) */
    int64_t rescored;          /* candidates re-scored in fp64 by the fast DP's exact stage */
    double dp_kernel_ms;       /* with ECASQ_TIME_KERNELS: summed duration of the min-plus kernel launches */
    int32_t dp_kernel_launches;/* with ECASQ_TIME_KERNELS: number of those launches */
    int32_t reserved2;
    double refine_last_rel;    /* (J_before - J_after) / |J_before| of the last refinement round (Sec. 6), 0 without
                                  refinement: at most refine_rel_tol when the stop rule ended it */
} ecasq_result_t;

/* Two-way time-sharing (Sec. 7): the mixture of the budgeted solution Q- (rate
 * b- <= b) and the evaluated point Q+ of least rate b+ > b, each entry using Q+
 * with probability beta = (b - b-)/(b+ - b-).  Rates are H(I,B), the quantity the
 * budget constrains; MSE and rates of the mixture are linear in beta. */
typedef struct ecasq_timeshare {
    double beta;               /* probability of Q+; 0 = Q- alone (no Q+, b- = b, or Q+ not better) */
    double lambda_plus;        /* multiplier of Q+ (vNMSE scale); NaN without Q+ */
    double mse, vnmse;         /* of the mixture */
    double h_surrogate;        /* H(I,B) of the mixture (= b when beta > 0) */
    double h_exact;            /* H(Xhat) of the mixture */
    double plus_mse, plus_h_surrogate, plus_h_exact;  /* of Q+; NaN without Q+ */
    int32_t m_plus;            /* |Q+|, 0 without Q+ */
    int32_t reserved;
} ecasq_timeshare_t;

/* Bytes of workspace needed by every entry point below for vectors of up to d
 * entries, codebook cap s, and `rows` independent rows (1 for single-vector
 * calls).  Returns 0 for invalid arguments. */
size_t ecasq_workspace_size(int64_t d, int32_t s, int64_t rows);

/* Workspace bytes for calls made with `flags`: ecasq_workspace_size plus, with
 * ECASQ_RESIDENT_COSTS, the resident interval-cost tiles (fp32 C and Phi of
 * every pair k < j in 64 x 64 tiles, and per tile each column's minimum C and
 * Phi: ceil(d/64)(ceil(d/64)+1)/2 tiles of 35328 bytes, e.g. 74 GB at
 * d = 2^17).  Returns 0 for invalid arguments or
 * a size that does not fit in size_t. */
size_t ecasq_workspace_size_flags(int64_t d, int32_t s, int64_t rows, uint32_t flags);

/* Budgeted (or fixed-multiplier) solve of one vector.
 * Pipeline: sort, weighted histogram and prefix sums (Sec. 2, App. E) ->
 * approximate DP (Sec. 5, eqs. apx_base, apx_rec, apx_final) over a multiplier
 * search (Sec. 3, Sec. 5: keep the lowest-MSE solution with H(I,B) <= b) ->
 * optional three-colour refinement (Sec. 6) at the selected multiplier.
 *   x   [d] device, input (not modified)
 *   Q   [s] device, output: Q[0..m-1] ascending, the rest untouched
 *   res host, output (may be NULL)
 * Search schedule: multiplier 0 first (if feasible it is the answer); else
 * rounds of the 7 geometric midpoints of [lo, hi] (sqrt only), the bracket
 * shrinking to the pair around the smallest feasible midpoint; if nothing is
 * feasible, hi itself; ECASQ_EINFEASIBLE when that fails too (Q then holds
 * the solution at hi).  Synchronises `stream`. */
int ecasq_solve(const float *x, int64_t d, const ecasq_params_t *prm, void *ws, size_t ws_bytes,
                float *Q, ecasq_result_t *res, ecasq_stream_t stream);

/* ecasq_solve with the codebook drawn from a caller-given permissible set P
 * instead of the unique values of x (Sec. 5 and App. E define the DP and C_P,
 * U_P, D_P, Phi_P for any sorted P; e.g. a uniform min-max grid or the values of
 * a narrow float format).  The same search, refinement and results, with every
 * codebook index referring to P.
 *   P   device [n] fp32, finite, strictly ascending, P[0] <= min x and
 *       P[n-1] >= max x (-0.0 counts as +0.0); otherwise ECASQ_EINVAL.  The first
 *       codebook value ranges over L = {P[a] <= min x} (eq. apx_base) and the last
 *       over R = {P[b] >= max x} (eq. apx_final); ties go to the smallest size,
 *       then the smallest last index, then the lowest first index.
 *   Q   device [s] output, values of P.  res->p = n.
 * Refinement moves interior values only; the first and last stay where the DP
 * put them.
 * DP: the interval costs of every pair of P are evaluated once per call in binary64
 * (24 bytes per pair, n <= 32768) and each layer is filtered in fp32 with a certified
 * band whose members are re-scored in binary64, so the result equals the binary64
 * reference kernel's (ECASQ_DP_REFERENCE forces that kernel; sets above 32768
 * values use it).  The fast kernel of ecasq_solve is not used: its recurrences need
 * every slab's mass at a candidate value, true only for P = X.  ECASQ_RESIDENT_COSTS
 * is ignored.
 * Workspace: ecasq_workspace_size_grid(d, n, s, flags).  Synchronises `stream`. */
size_t ecasq_workspace_size_grid(int64_t d, int64_t n, int32_t s, uint32_t flags);
int ecasq_solve_grid(const float *x, int64_t d, const float *P, int64_t n, const ecasq_params_t *prm, void *ws,
                     size_t ws_bytes, float *Q, ecasq_result_t *res, ecasq_stream_t stream);

/* Budgeted solve with two-way time-sharing (Sec. 7): the multiplier search of
 * ecasq_solve (or of ecasq_solve_grid when P is not NULL), then Q+ = the evaluated
 * point with the least H(I,B) above the budget (ties: less MSE, then the smaller
 * multiplier) and beta as in ecasq_timeshare_t.  Every evaluated point is a
 * minimiser of the surrogate Lagrangian, so the mixture reaches the budget exactly
 * with an MSE linear in beta.  prm->lambda must be < 0 (a budget) and
 * prm->refine_max_rounds 0, else ECASQ_EINVAL.
 *   P, n  as ecasq_solve_grid, or P = NULL for the unique values of x
 *   Qm    device [s] output: Q- (as ecasq_solve's Q)
 *   Qp    device [s] output: Q+ when ts->m_plus > 0, else untouched
 *   res   host (may be NULL): ecasq_solve's result for Q-
 *   ts    host output
 * Workspace: ecasq_workspace_size_flags(d, s, 1, flags), or with P
 * ecasq_workspace_size_grid(d, n, s, flags).  Synchronises `stream`. */
int ecasq_solve_timeshare(const float *x, int64_t d, const float *P, int64_t n, const ecasq_params_t *prm, void *ws,
                          size_t ws_bytes, float *Qm, float *Qp, ecasq_result_t *res, ecasq_timeshare_t *ts,
                          ecasq_stream_t stream);

/* Time-shared stochastic quantization (Sec. 7 with Sec. 2): entry i (original
 * order) uses Qp iff k_s 2^-24 < beta in binary64, k_s = top 24 bits of
 * SplitMix64(seed_ts + (i+1) 0x9E3779B97F4A7C15), then rounds within its codebook
 * exactly as ecasq_quantize with `seed` (same counter i).  A decoder that knows
 * seed_ts regenerates the partition; `sel` is a convenience copy of it.
 *   Qm [mm], Qp [mp]  device, ascending; mp may be 0 (and Qp NULL) when beta = 0
 *   idx     device [d] uint8 output: index into the entry's codebook
 *   sel     device [d] uint8 output (may be NULL): 1 where Qp was used
 *   counts  device [mm + mp] uint32 output: index histograms of Qm, then Qp
 *   ws      device, >= 256 bytes, 256-byte aligned (status record)
 *   rate    host (may be NULL): bits per entry of coding each part with its own
 *           empirical law, -(1/d) sum_parts sum_r c_r log2(c_r / n_part)
 * ECASQ_EINVAL for beta outside [0, 1], non-ascending codebooks or mp = 0 with
 * beta > 0; ECASQ_ERANGE if an entry lies outside its codebook's range.
 * Synchronises `stream`. */
int ecasq_quantize_timeshare(const float *x, int64_t d, const float *Qm, int32_t mm, const float *Qp, int32_t mp,
                             double beta, uint64_t seed, uint64_t seed_ts, uint8_t *idx, uint8_t *sel,
                             uint32_t *counts, void *ws, size_t ws_bytes, double *rate, ecasq_stream_t stream);


/* The optimal DP of Sec. 4 (App. E for a permissible set) at G <= 8 fixed
 * multipliers: the least MSE + lambda' H(Xhat) over codebooks drawn from P (or from
 * the unique values of x when P is NULL) with at most s values (exactly s with
 * ECASQ_EXACT_S), first value in L and last in R as in eq. apx_base / apx_final.
 * State (i, l, j) with the entropy of p_l charged once both neighbours are known:
 *   dp(2, a, j) = C[a, j] + lambda' h((n_a + D[a, j]) / d)                     (a in L)
 *   dp(i, l, j) = C[l, j] + min_{k<l} dp(i-1, k, l) + lambda' h((U[k, l] + D[l, j]) / d)
 *   optimum     = min_{i, j in R, l<j} dp(i, l, j) + lambda' h(U[l, j] / d)
 * Ties: lowest k; at the optimum the smallest i, then j, then l.  Every candidate is
 * filtered in fp32 and every one within a certified band is re-scored in binary64
 * with the formula above, so values and decisions are those of a binary64 evaluation.
 * O(p^3 s / 6) candidates and O(p^2 s G) table cells: meant for p up to a few
 * thousand (the candidate set is capped at 16384 values).
 *   lambdas   host [G], vNMSE scale (lambda' = lambda ||X||^2), >= 0 and finite
 *   P, n      device [n] permissible set (as ecasq_solve_grid) or NULL (n ignored)
 *   Q_out     device [G * s] (row g: codebook of multiplier g, m_out[g] values)
 *   m_out     host [G]
 *   metrics   host [G * 4]: optimum, MSE, H(I,B), H(Xhat) of the traced codebook
 * Workspace: ecasq_workspace_size_opt(d, n or d, s, G) (about 12 G s p^2 / 2 bytes of
 * tables plus 12 p^2 bytes of pair quantities).  Synchronises `stream`. */
size_t ecasq_workspace_size_opt(int64_t d, int64_t n, int32_t s, int32_t G);
int ecasq_opt_dp(const float *x, int64_t d, const float *P, int64_t n, int32_t s, const double *lambdas, int32_t G,
                 uint32_t flags, void *ws, size_t ws_bytes, float *Q_out, int32_t *m_out, double *metrics,
                 ecasq_stream_t stream);

/* One DP pass (Sec. 5) at G <= 8 fixed multipliers, the unit of the search.
 *   lambdas   host [G], vNMSE scale, >= 0
 *   Q_out     device [G * s] (row g: codebook of multiplier g, m_out[g] values)
 *   m_out     host [G]
 *   metrics   host [G * 4]: DP optimum (eq. apx_final), MSE, H(I,B), H(Xhat)
 * The DP tables stay in the workspace until the next call (ecasq_dp_tables).
 * Synchronises `stream`. */
int ecasq_dp_pass(const float *x, int64_t d, int32_t s, const double *lambdas, int32_t G, uint32_t flags,
                  void *ws, size_t ws_bytes, float *Q_out, int32_t *m_out, double *metrics,
                  ecasq_stream_t stream);

/* Copy the DP tables of multiplier g of the last ecasq_dp_pass on this
 * workspace: dp (fp64) and bp (int32, lowest argmin k; -1 where undefined),
 * each row-major [(s+1) x p], rows 0 and 1 unused, +inf / -1 where the layer
 * is undefined.  The fast kernel resolves exactly the outputs the final
 * selection and traceback depend on; elsewhere dp holds its fp32-filtered
 * value and bp = -2, unless the pass ran with ECASQ_EXACT_TABLES (or
 * ECASQ_DP_REFERENCE).  dp_out, bp_out device; p_out host.  Synchronises
 * `stream`. */
int ecasq_dp_tables(void *ws, size_t ws_bytes, int32_t g, double *dp_out, int32_t *bp_out, int64_t *p_out,
                    ecasq_stream_t stream);

/* Linear-space traceback of the approximate DP (Sec. 5, last paragraph: Hirschberg's
 * method on eq. apx_rec), one multiplier `lambda` (vNMSE scale, lambda' = lambda ||X||^2),
 * P = X.  Memory O(d): the workspace holds the histogram and prefix sums, four DP rows and
 * a few scalars (ecasq_workspace_size_linear(d), about 124 d bytes) -- no table of
 * backpointers.  A forward pass over the layers of eq. apx_rec (two rows) gives dp(i, p-1)
 * and the answer of eq. apx_final (m = the smallest i with the least value; ECASQ_EXACT_S:
 * i = s).  The chain of m values is then rebuilt by splitting subproblems (u, v, n) -- n
 * values with u and v fixed at the ends -- at the middle position t = (n + 1) / 2: the
 * middle value is the lowest c among the exact binary64 minima of G(c) + B(c), G the least
 * cost of a chain of t values from u to c (forward pass), B of n - t + 1 values from c to v
 * (backward pass over suffix costs).  All costs are binary64 with the reference interval
 * quantities (the values of ECASQ_DP_REFERENCE).  The optimum is the one of eq. apx_final;
 * at exact ties of G + B the codebook may differ from the backpointer traceback's (which
 * takes the lowest k at every step from the end).  Time O(s d^2) pair evaluations.
 * Q_out [s] device (first m entries), m_out host, metrics host [4]: dp(m, p-1) (the
 * surrogate Lagrangian of eq. apx_final), MSE, H(I,B), H(Xhat) of the codebook.
 * ECASQ_EINVAL for d < 1, s outside [2, 256] or a negative / non-finite lambda;
 * ECASQ_EINFEASIBLE when no codebook of the required size exists (ECASQ_EXACT_S with
 * s above the number of unique values).  Synchronises `stream`. */
size_t ecasq_workspace_size_linear(int64_t d);
int ecasq_dp_linear(const float *x, int64_t d, int32_t s, double lambda, uint32_t flags, void *ws, size_t ws_bytes,
                    float *Q_out, int32_t *m_out, double *metrics, ecasq_stream_t stream);

/* Three-colour refinement (Sec. 6) of a codebook Q subset of X at a fixed
 * multiplier, minimising MSE + lambda' H(Xhat): colours 0, 1, 2 in turn move
 * each interior value with index % 3 == colour to the best unique input value
 * strictly between its neighbours (ties keep the value, else the lowest);
 * with a budget (budget_bits >= 0 and no ECASQ_NO_REFINE_GUARD flag) a colour
 * step that lifts H(Xhat) above the budget is undone; stop after a round that
 * lowers J by <= rel_tol*|J| or after max_rounds.
 *   Q  device [m], in/out.  res host (may be NULL).  Synchronises `stream`. */
int ecasq_refine(const float *x, int64_t d, float *Q, int32_t m, double lambda, double budget_bits,
                 int32_t max_rounds, double rel_tol, uint32_t flags, void *ws, size_t ws_bytes,
                 ecasq_result_t *res, ecasq_stream_t stream);

/* MSE, H(I,B) and H(Xhat) of a codebook Q subset of X (Sec. 2, Sec. 3,
 * eq. apx_additive_entropy).  out host [3].  Synchronises `stream`. */
int ecasq_evaluate(const float *x, int64_t d, const float *Q, int32_t m, void *ws, size_t ws_bytes,
                   double *out, ecasq_stream_t stream);

/* Unbiased stochastic quantization (Sec. 2) of x in its original order:
 * a = max{q <= x}; an entry equal to a gets a's index, otherwise it is
 * rounded up to the next value iff fl32(fl32(k 2^-24) fl32(b - a)) <
 * fl32(x - a), k = top 24 bits of SplitMix64(seed + (i+1) 0x9E3779B97F4A7C15)
 * (Steele, Lea and Flood 2014) for entry i; so E[xhat] = x up to 2^-23 (b-a).
 *   idx     device [d] uint8 output
 *   counts  device [m] uint32 output: index histogram
 *   h_emp   host, output (may be NULL): empirical entropy of idx (Sec. 1)
 * ECASQ_ERANGE if an entry lies outside [Q[0], Q[m-1]].  Synchronises
 * `stream` only when h_emp is not NULL. */
int ecasq_quantize(const float *x, int64_t d, const float *Q, int32_t m, uint64_t seed, uint8_t *idx,
                   uint32_t *counts, void *ws, size_t ws_bytes, double *h_emp, ecasq_stream_t stream);

/* ecasq_quantize without a workspace: same arguments minus (ws, ws_bytes),
 * same kernel, same results (idx, counts and h_emp equal to ecasq_quantize's
 * for the same inputs and seed).  The paper has no counterpart: this is an
 * interface convenience around the quantizer of Sec. 2.
 *
 * Who needs it: callers that cannot hand the library device memory at the
 * point where they quantize -- a hook inside a training or serving framework
 * that runs where the framework forbids allocation (its caching allocator
 * may not be re-entered there), a latency-critical path that cannot afford an
 * allocation's synchronisation, or a process already at its memory limit.
 * The function itself calls no device allocator (no cudaMalloc/cudaFree, no
 * allocating library routine); idx and counts are the caller's buffers.
 *
 * Scratch: a fixed 256-byte block of device memory inside this library, one
 * per device, holding one status record.  Its range-error flag must be zero
 * when the kernel starts; every call zeroes it on `stream` before its launch.
 * Limits: m <= 256 (the codebook cap) and d < 2^31, as for ecasq_quantize;
 * larger sizes return ECASQ_EINVAL.  The scratch does not grow with d.
 *
 * Set-up: the first call on each device looks up the scratch's device address
 * (cudaGetSymbolAddress, which may load this library's device code) and keeps
 * it; an error there returns ECASQ_ECUDA.  Make that first call on each device
 * before any stream capture begins.  The kept address belongs to the device
 * context of that first call: resetting the device (cudaDeviceReset) after it
 * is not supported.  `stream` must belong to the current device (a stream of
 * another device returns ECASQ_EINVAL).
 *
 * Concurrency: all calls on one device share the one scratch block.  Calls
 * that overlap in time on the same device -- from several host threads, or on
 * streams not ordered with each other -- race on it (one call's reset can
 * erase another's error flag); serialise them.  Synchronises `stream`. */
int ecasq_quantize_noalloc(const float *x, int64_t d, const float *Q, int32_t m, uint64_t seed, uint8_t *idx,
                           uint32_t *counts, double *h_emp, ecasq_stream_t stream);

/* Budgeted solves of `rows` independent rows of length d (row-major X),
 * each exactly as ecasq_solve would do it on that row alone (same schedule,
 * same results).  Q [rows * s] device, m_out [rows] device, res host [rows]
 * (may be NULL).  Synchronises `stream`. */
int ecasq_solve_batched(const float *X, int64_t rows, int64_t d, const ecasq_params_t *prm, void *ws,
                        size_t ws_bytes, float *Q, int32_t *m_out, ecasq_result_t *res,
                        ecasq_stream_t stream);

/* Weighted histogram and App. E prefix sums of x (step 1 of every solve):
 *   v [p] fp32 unique values ascending, w [p] int64 multiplicities,
 *   N [p+1] int64, S and S2 [2*(p+1)] fp64 as (hi[0..p], lo[0..p]) with
 *   N[t] = sum_{r<t} w_r, S[t] = sum w_r v_r, S2[t] = sum w_r v_r^2.
 *   All device, sized for p = d; p_out host.  Workspace: ecasq_workspace_size_prep(d)
 *   (about 92 d bytes: the sort's keys, the histogram and the sums; the solves'
 *   workspace holds far more).  Synchronises `stream`. */
size_t ecasq_workspace_size_prep(int64_t d);
int ecasq_prepare(const float *x, int64_t d, void *ws, size_t ws_bytes, float *v, int64_t *w, int64_t *N,
                  double *S, double *S2, int64_t *p_out, ecasq_stream_t stream);

/* Kernels this library has launched in the calling process so far (all
 * threads, all entry points): a monotone counter for launch accounting. */
int64_t ecasq_kernel_launches(void);

const char *ecasq_strerror(int status);
int ecasq_version(void);

#ifdef __cplusplus
}
#endif
#endif /* ECASQ_H */
