// common.cuh -- shared internals of the ECASQ CUDA library (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <math_constants.h>
#include <stdint.h>
#include <stddef.h>

#include "../../include/ecasq.h"

namespace ecasq {

constexpr int kMaxS = 256;      // codebook cap
constexpr int kMaxG = 8;        // multipliers per DP pass
constexpr int kSortTile = 2048; // keys per radix-sort block
constexpr int kScanTile = 1024; // longest row of the batched path (one block of 256 threads)
constexpr int kHistPer = 16;    // sorted keys per thread in the histogram / prefix-sum blocks
constexpr int kHistTile = 256 * kHistPer;  // keys per histogram block

#define ECASQ_CUDA_TRY(expr)                          \
    do {                                              \
        cudaError_t e_ = (expr);                      \
        if (e_ != cudaSuccess) return ECASQ_ECUDA;    \
    } while (0)

#define ECASQ_LAUNCH_CHECK() ECASQ_CUDA_TRY(cudaGetLastError())

__host__ __device__ static inline int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }
// Row stride of every DP table: p rounded up to 64 entries, so each row starts
// 256-byte aligned (the fast kernel copies rows with 16-byte cp.async).
__host__ __device__ static inline int64_t table_stride(int64_t p) { return (p + 63) & ~(int64_t)63; }
static inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// ---------------------------------------------------------------- workspace
// Device-side status block at the start of the workspace.
struct DevStatus {
    int64_t p;            // number of unique values
    int32_t nonfinite;    // x held NaN/Inf
    int32_t range_err;    // quantize: entry outside [Q0, Qm-1]; refine: Q not in X
    int32_t timeout;      // a bounded wait ran out
    int32_t bound_viol;   // fast DP: fp32 minima outside their certified error bound
    double norm2;         // ||X||^2 (hi part of the double-double sum)
    int64_t rescored;     // fast DP: candidates re-scored in fp64
    int64_t overflow;     // fast DP: needed outputs whose band spans more than 32 tiles
    int32_t last_s;       // s and G of the last DP pass (for ecasq_dp_tables)
    int32_t last_G;
    int64_t last_d;       // d of the last DP pass
    int64_t members;      // fast DP: band members found (all outputs)
    int64_t big_bands;    // fast DP: outputs with more members than the inline list holds
    int64_t tiles_run;    // fast DP, resident costs: (warp, tile) units evaluated
    int64_t tiles_skipped; // ... and skipped by the lower bound
    int64_t grid_nL;      // permissible set: |L| = #{p_a <= min x}, |R| = #{p_b >= max x} (Sec. 5)
    int64_t grid_nR;
    int64_t tiles_fetched; // fast DP, resident costs: interval-cost tiles copied in from HBM
};

struct Layout {
    size_t status;         // DevStatus
    size_t keys0, keys1;   // uint32 [d]
    size_t rcount;         // uint32 [256 * nb] radix counts / offsets
    size_t head;           // int32 [d] unique index of each sorted position
    size_t v;              // float [d] unique values
    size_t w;              // int64 [d] multiplicities
    size_t N;              // int64 [d+1]
    size_t S, S2;          // double [2(d+1)] (hi | lo)
    size_t part;           // double-double scan partials
    size_t dp64;           // double [G (s+1) d]
    size_t bp;             // int32 [G (s+1) d]
    size_t dp32;           // float  [G (s+1) d]
    size_t qidx;           // int32 [G s]  traced codebooks (unique indices)
    size_t mcount;         // int32 [G]
    size_t metrics;        // double [G 4]
    size_t lam;            // double [G]   lambda' of each multiplier
    size_t refine;         // refinement scratch
    size_t refine_part;    // refinement per-chunk partial minima
    size_t band;           // fast DP band lists
    size_t costs;          // resident interval-cost tiles (ECASQ_RESIDENT_COSTS), after everything else
    size_t costs_bytes;    // 0 when absent
    bool costs_streamed;   // ECASQ_STREAMED_COSTS: the costs region holds one band of tiles at a time
    size_t gpairs;         // grid DP pair cache (permissible sets up to kGridPairsMax values)
    size_t gpairs_bytes;   // 0 when absent
    size_t total;
    int64_t d;
    int32_t s;
};

size_t make_layout(int64_t d, int32_t s, int64_t rows, Layout *L);

template <typename T>
static inline T *wsp(void *ws, size_t off) { return reinterpret_cast<T *>(static_cast<char *>(ws) + off); }

// ------------------------------------------------------------ double-double
// Error-free transformations (Knuth's TwoSum; TwoProd with fma) and the
// double-double sum used for the App. E prefix sums.  All operations are
// spelled with _rn intrinsics so the compiler cannot contract them.
struct dd { double hi, lo; };

__device__ __forceinline__ dd two_sum(double a, double b) {
    double s = __dadd_rn(a, b);
    double bb = __dsub_rn(s, a);
    double e = __dadd_rn(__dsub_rn(a, __dsub_rn(s, bb)), __dsub_rn(b, bb));
    return {s, e};
}
__device__ __forceinline__ dd fast_two_sum(double a, double b) {  // |a| >= |b|
    double s = __dadd_rn(a, b);
    return {s, __dsub_rn(b, __dsub_rn(s, a))};
}
__device__ __forceinline__ dd two_prod(double a, double b) {
    double p = __dmul_rn(a, b);
    return {p, __fma_rn(a, b, -p)};
}
__device__ __forceinline__ dd dd_add(dd a, dd b) {
    dd s = two_sum(a.hi, b.hi);
    dd t = two_sum(a.lo, b.lo);
    s.lo = __dadd_rn(s.lo, t.hi);
    s = fast_two_sum(s.hi, s.lo);
    s.lo = __dadd_rn(s.lo, t.lo);
    return fast_two_sum(s.hi, s.lo);
}
// a + b for a double b: the value dd_add(a, {b, 0}) gives (its second two_sum adds zero and
// its last renormalisation leaves a normalised pair unchanged), in half the operations.
__device__ __forceinline__ dd dd_add_d(dd a, double b) {
    dd s = two_sum(a.hi, b);
    s.lo = __dadd_rn(s.lo, a.lo);
    return fast_two_sum(s.hi, s.lo);
}
__device__ __forceinline__ dd dd_neg(dd a) { return {-a.hi, -a.lo}; }
__device__ __forceinline__ dd dd_sub(dd a, dd b) { return dd_add(a, dd_neg(b)); }
__device__ __forceinline__ dd dd_mul_d(dd a, double b) {
    dd p = two_prod(a.hi, b);
    p.lo = __fma_rn(a.lo, b, p.lo);
    return fast_two_sum(p.hi, p.lo);
}
__device__ __forceinline__ dd dd_mul(dd a, dd b) {
    dd p = two_prod(a.hi, b.hi);
    p.lo = __fma_rn(a.hi, b.lo, p.lo);
    p.lo = __fma_rn(a.lo, b.hi, p.lo);
    return fast_two_sum(p.hi, p.lo);
}
__device__ __forceinline__ double dd_round(dd a) { return __dadd_rn(a.hi, a.lo); }

// h(y) = -y log2 y, h(0) = 0 (Sec. 4).
__device__ __forceinline__ double hfun(double y) { return y > 0.0 ? -__dmul_rn(y, log2(y)) : 0.0; }

// Per-row prefix data of the batched path (rows of length d <= kScanTile): row r
// holds v[dcap], w[dcap], N[dcap+1], S and S2 [2(dcap+1)] packed as (hi[0..p], lo[0..p]).
struct RowsData {
    float *v;
    int64_t *w, *N;
    double *S, *S2;
    int64_t *p;       // [rows]
    double *norm2;    // [rows]
    int32_t *nonfinite;  // [rows]
    int64_t d, dcap;
};

// One search round of the batched path: block b runs row rows[b] at G multipliers.
constexpr int kRowsMaxP = 128;  // unique values per row the batched path holds in shared memory
struct RowsPass {
    RowsData R;
    const int32_t *rows;  // [nact] row of each block
    const double *lam;    // [nact][G] lambda' of the row
    int G, s, exact_s;
    int32_t *bp;          // [nact][G][s+1][dcap]
    int32_t *qidx;        // [nact][G][s]
    int32_t *mcount;      // [nact][G]
    double *metrics;      // [nact][G][4]
    double *pairs;        // [rows][pstride]: the row's binary64 {C, Phi} by pair, Phi^first and fp32
                          // {C scale, Phi} by pair, kept across rounds
    int64_t pstride;      // doubles per row: 3 npair(pmax) + pmax
    int pairs_ready;      // the rows' interval costs are already in `pairs`
    int bp_smem;          // backpointers in shared memory (set by the launcher)
};

// Prefix-sum view (App. E) used by every exact pair evaluation.
struct Prefix {
    const float *v;       // [p]
    const int64_t *w;     // [p]
    const int64_t *N;     // [p+1]
    const double *S;      // hi [p+1] | lo [p+1]
    const double *S2;
    int64_t p;
    int64_t d;
    int64_t ps;           // DP-table row stride, table_stride(p)
    int64_t nL = 1;       // first-value set L = {0..nL-1}, last-value set R = {p-nR..p-1}
    int64_t nR = 1;       // (Sec. 5); both 1 when the candidates are the unique values of x
    double scale32 = 1.0; // grid DP: power of two that brings ||X||^2 into [1, 2) for fp32 copies
};

// Largest permissible set whose pair costs the grid DP caches (24 bytes per pair).
constexpr int64_t kGridPairsMax = 32768;
// Largest candidate set of the optimal DP (Sec. 4): one block row per l in a launch.
constexpr int64_t kOptMax = 16384;

__device__ __forceinline__ dd load_dd(const double *a, int64_t p, int64_t t) { return {a[t], a[p + 1 + t]}; }

// App. E for k < j over X_{k,j} = {x : v_k < x <= v_j}:
//   A = S_kj - v_k N_kj, E = v_j N_kj - S_kj, C = (v_k+v_j) S_kj - S2_kj - v_k v_j N_kj,
//   U = A / (v_j - v_k), D = E / (v_j - v_k).
// Numerators in double-double, rounded once; one binary64 division each.
__device__ __forceinline__ void pair_exact(const Prefix &P, int64_t k, int64_t j, double &C, double &U,
                                           double &D) {
    double n = (double)(P.N[j + 1] - P.N[k + 1]);
    dd dS = dd_sub(load_dd(P.S, P.p, j + 1), load_dd(P.S, P.p, k + 1));
    dd dS2 = dd_sub(load_dd(P.S2, P.p, j + 1), load_dd(P.S2, P.p, k + 1));
    double vk = (double)P.v[k], vj = (double)P.v[j];
    dd A = dd_sub(dS, two_prod(vk, n));
    dd E = dd_sub(two_prod(vj, n), dS);
    dd sk = two_sum(vk, vj);
    dd Cd = dd_sub(dd_sub(dd_mul(sk, dS), dS2), two_prod(__dmul_rn(vk, vj), n));
    double L = __dsub_rn(vj, vk);
    C = dd_round(Cd);
    U = __ddiv_rn(dd_round(A), L);
    D = __ddiv_rn(dd_round(E), L);
}

// Sec. 5: Phi = h(U/d) + h(D/d); Phi^first adds the first value's mass w_0 to D.
__device__ __forceinline__ double phi_exact(const Prefix &P, double U, double D, bool first) {
    double dd_ = (double)P.d;
    double Dm = first ? __dadd_rn(D, (double)P.w[0]) : D;
    return __dadd_rn(hfun(__ddiv_rn(U, dd_)), hfun(__ddiv_rn(Dm, dd_)));
}

// Phi^first[a, .] for a first value a in L: the down symbol also holds n_a = w_a.
__device__ __forceinline__ double phi_first_at(const Prefix &P, int64_t a, double U, double D) {
    double dd_ = (double)P.d;
    return __dadd_rn(hfun(__ddiv_rn(U, dd_)), hfun(__ddiv_rn(__dadd_rn(D, (double)P.w[a]), dd_)));
}

// Metrics of codebook a[0..m-1] (unique indices): MSE, H(I,B), H(Xhat), summed
// in interval order exactly as the definitions list them (Sec. 2, Sec. 3,
// eq. apx_additive_entropy).  One warp; lanes evaluate intervals, lane 0 sums.
static __device__ __noinline__ void eval_codebook_warp(const Prefix &P, const int32_t *a, int m, double *out3, double *scratch) {
    // scratch: 4 * kMaxS doubles (C, Phi, U, D per interval)
    int lane = threadIdx.x & 31;
    for (int r = lane; r + 1 < m; r += 32) {
        double C, U, D;
        pair_exact(P, a[r], a[r + 1], C, U, D);
        scratch[r] = C;
        scratch[kMaxS + r] = r == 0 ? phi_first_at(P, a[0], U, D) : phi_exact(P, U, D, false);
        scratch[2 * kMaxS + r] = U;
        scratch[3 * kMaxS + r] = D;
    }
    __syncwarp();
    if (m < 2) {
        if (lane == 0) { out3[0] = 0.0; out3[1] = 0.0; out3[2] = 0.0; }
        __syncwarp();
        return;
    }
    // output-entropy terms in parallel: f_r = U_{r-1} + D_r (w of the first value + D_0 for
    // r = 0), term r = h(f_r / d), and term m-1 = h(U_{m-2} / d); each lane overwrites the
    // D slots it alone reads
    const double dd_ = (double)P.d;
    for (int r = lane; r < m; r += 32) {
        double f;
        if (r == m - 1) f = scratch[2 * kMaxS + m - 2];
        else f = (r == 0) ? __dadd_rn((double)P.w[a[0]], scratch[3 * kMaxS]) : __dadd_rn(scratch[2 * kMaxS + r - 1], scratch[3 * kMaxS + r]);
        scratch[3 * kMaxS + r] = hfun(__ddiv_rn(f, dd_));
    }
    __syncwarp();
    if (lane == 0) {
        // the sums in interval order, as a sequential evaluation adds them
        double mse = 0.0, hs = 0.0, hx = 0.0;
        for (int r = 0; r + 1 < m; r++) {
            mse = __dadd_rn(mse, scratch[r]);
            hs = __dadd_rn(hs, scratch[kMaxS + r]);
            hx = __dadd_rn(hx, scratch[3 * kMaxS + r]);
        }
        hx = __dadd_rn(hx, scratch[3 * kMaxS + m - 1]);
        out3[0] = mse; out3[1] = hs; out3[2] = hx;
    }
    __syncwarp();
}

// eval_codebook_warp for m <= 32 with no shared scratch: lane r holds interval r's C,
// Phi (Phi^first for r = 0), U and D, and term r of the output entropy (the neighbour's U
// by a shuffle); the three sums run in interval order from shuffled values, as there.
static __device__ __noinline__ void eval_codebook_lanes(const Prefix &P, const int32_t *a, int m, double *out3) {
    const int lane = threadIdx.x & 31;
    double C = 0.0, F = 0.0, U = 0.0, D = 0.0;
    if (lane + 1 < m) {
        pair_exact(P, a[lane], a[lane + 1], C, U, D);
        F = lane == 0 ? phi_first_at(P, a[0], U, D) : phi_exact(P, U, D, false);
    }
    const double Uprev = __shfl_up_sync(0xffffffffu, U, 1);
    const double Ulast = __shfl_sync(0xffffffffu, U, m >= 2 ? m - 2 : 0);
    double ht = 0.0;
    if (m >= 2 && lane < m) {
        const double f = lane == m - 1 ? Ulast : (lane == 0 ? __dadd_rn((double)P.w[a[0]], D) : __dadd_rn(Uprev, D));
        ht = hfun(__ddiv_rn(f, (double)P.d));
    }
    double mse = 0.0, hs = 0.0, hx = 0.0;
    for (int r = 0; r + 1 < m; r++) {
        mse = __dadd_rn(mse, __shfl_sync(0xffffffffu, C, r));
        hs = __dadd_rn(hs, __shfl_sync(0xffffffffu, F, r));
        hx = __dadd_rn(hx, __shfl_sync(0xffffffffu, ht, r));
    }
    if (m >= 2) hx = __dadd_rn(hx, __shfl_sync(0xffffffffu, ht, m - 1));
    if (lane == 0) { out3[0] = mse; out3[1] = hs; out3[2] = hx; }
    __syncwarp();
}

// -------------------------------------------------------------- host helpers
// Kernels launched by this library in this process (all threads).
void note_launch();

int prepare_device(const float *x, int64_t d, void *ws, const Layout &L, cudaStream_t st, int64_t *p_host,
                   double *norm2_host);

}  // namespace ecasq
