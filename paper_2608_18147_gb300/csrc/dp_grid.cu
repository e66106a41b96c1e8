// dp_grid.cu -- the approximate DP (Sec. 5) over a caller-given permissible set P
// of n values (App. E), for n up to kGridPairsMax.
//
// C_P and Phi_P of a pair k < j depend on neither the layer nor the multiplier, so
// k_grid_pairs evaluates every pair once per call with the reference formulas
// (pair_exact / phi_exact, binary64) into a triangle indexed j(j-1)/2 + k, next to
// fp32 copies {C * scale, Phi}; scale = 2^-e with 2^e <= ||X||^2 < 2^(e+1), which
// keeps the fp32 values near 1 (the DP is invariant under scaling X by a power of
// two when lambda' scales with ||X||^2, Sec. 3).
//
// Layer i >= 3 (eq. apx_rec) runs one block per output j for all G multipliers:
//  1. fp32 pass over k in [i-2, j-1]: val32 = fl(dp32(i-1,k) + fl(fma(lam32, Phi32, C32)))
//     gives the fp32 minimum m32 of each multiplier;
//  2. every k with val32 <= T = m32 (1 + 10u) + 3A is re-scored with the binary64
//     candidate of the reference kernel, dp(i-1,k) + (C + lambda' Phi); the lowest k
//     among the exact minima wins, as in k_dp_layer_ref.
// Why the band holds every exact minimiser: all terms are >= 0; each fp32 input is
// within u = 2^-24 (relative) of its binary64 value, or within 2^-150 (absolute) when
// subnormal; the fma and the add round once each.  So val32 is within (1 +- u)^4 of
// the exact sum v of the binary64 inputs, up to A = (70 + lam32) 2^-150 (the absolute
// errors of the six roundings, weighted by lam32 and by Phi <= 2 max h = 1.07).
// The binary64 candidate is within (1 +- 2^-53)^3 of v.  A k whose binary64 candidate
// is minimal therefore has val32 <= (m32 + A)(1 + 8.0001u) + A < T.  fp32 overflow
// only turns a candidate far above the minimum into +inf, which stays out of the band.
#include "common.cuh"

namespace ecasq {

void timer_begin(cudaStream_t st);
void timer_end(cudaStream_t st);

struct GridArgs {
    const double2 *pc64;   // {C, Phi} binary64, triangle j(j-1)/2 + k
    const float2 *pc32;    // {C * scale, Phi} fp32
    double *dp64;          // [G][s+1][ps]
    int32_t *bp;
    float *dp32;           // [G][s+1][ps], dp64 * scale rounded to fp32
    const int64_t *N;      // [n+1]: N[t+1] = #{x <= P_t}
    int64_t n, ps;
    int G, s;
    double scale;
    double lam64[kMaxG];   // lambda'
    float lam32[kMaxG];    // fl32(lambda' * scale)
    double slack[kMaxG];   // 3A of the band threshold
};

__device__ __forceinline__ size_t g_at(const GridArgs &A, int g, int i, int64_t j) {
    return ((size_t)g * (size_t)(A.s + 1) + (size_t)i) * (size_t)A.ps + (size_t)j;
}

__global__ void __launch_bounds__(256) k_grid_pairs(Prefix P, double scale, double2 *pc64, float2 *pc32) {
    const int64_t npair = P.p * (P.p - 1) / 2;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < npair; t += stride) {
        int64_t j = (int64_t)((1.0 + sqrt(1.0 + 8.0 * (double)t)) * 0.5);
        while (j * (j - 1) / 2 > t) j--;
        while ((j + 1) * j / 2 <= t) j++;
        int64_t k = t - j * (j - 1) / 2;
        double C, U, D;
        pair_exact(P, k, j, C, U, D);
        double F = phi_exact(P, U, D, false);
        pc64[t] = make_double2(C, F);
        pc32[t] = make_float2(__double2float_rn(__dmul_rn(C, scale)), __double2float_rn(F));
    }
}

// dp32 of one layer from dp64 (layer 2 comes from k_dp_base).
__global__ void k_grid_round(GridArgs A, int i) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < (int64_t)A.G * A.n; t += stride) {
        int g = (int)(t / A.n);
        int64_t j = t % A.n;
        A.dp32[g_at(A, g, i, j)] = __double2float_rn(__dmul_rn(A.dp64[g_at(A, g, i, j)], A.scale));
    }
}

// One block per output j (heavy outputs first), its threads splitting the k range, so
// that no output's scan is a long serial walk of one warp (the last outputs have n - 1
// candidates per multiplier, and each step of a walk waits on its loads from L2).
constexpr int kGridThreads = 256;
__global__ void __launch_bounds__(kGridThreads, 3) k_grid_layer(GridArgs A, int i) {
    __shared__ float sm[kGridThreads / 32][kMaxG];
    __shared__ double sb[kGridThreads / 32][kMaxG];
    __shared__ int32_t sa[kGridThreads / 32][kMaxG];
    __shared__ float sT[kMaxG];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const int64_t j = A.n - 1 - (int64_t)blockIdx.x;
    if (j < i - 1) return;  // block-uniform
    const size_t tb = (size_t)j * (size_t)(j - 1) / 2;
    const int G = A.G;
    float m[kMaxG];
#pragma unroll
    for (int g = 0; g < kMaxG; g++) m[g] = CUDART_INF_F;
    for (int64_t k = i - 2 + threadIdx.x; k < j; k += kGridThreads) {
        float2 cf = A.pc32[tb + k];
#pragma unroll
        for (int g = 0; g < kMaxG; g++)
            if (g < G) m[g] = fminf(m[g], __fadd_rn(A.dp32[g_at(A, g, i - 1, k)], __fmaf_rn(A.lam32[g], cf.y, cf.x)));
    }
#pragma unroll
    for (int g = 0; g < kMaxG; g++) {
        float v = m[g];
        for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
        if (lane == 0) sm[wid][g] = v;
    }
    __syncthreads();
    // the band limits, once per block (binary64 runs at 1/64 of the fp32 rate): rounded down
    // to fp32, so that for an fp32 candidate c, c <= T32 exactly when c <= T
    if (threadIdx.x < kMaxG) {
        const int g = threadIdx.x;
        float v = sm[0][g];
        for (int w = 1; w < kGridThreads / 32; w++) v = fminf(v, sm[w][g]);
        sT[g] = __double2float_rd(__dadd_rn(__dmul_rn((double)v, 1.0 + 10.0 * 0x1p-24), A.slack[g]));
    }
    __syncthreads();
    float T[kMaxG];
#pragma unroll
    for (int g = 0; g < kMaxG; g++) T[g] = sT[g];
    double best[kMaxG];
    int32_t arg[kMaxG];
#pragma unroll
    for (int g = 0; g < kMaxG; g++) { best[g] = CUDART_INF; arg[g] = -1; }
    const int64_t Nj = A.N[j + 1];
    for (int64_t k = i - 2 + threadIdx.x; k < j; k += kGridThreads) {
        float2 cf = A.pc32[tb + k];
        // no data in (P_k, P_j]: then App. E's sums are differences of equal prefix values,
        // so C = U = D = 0 and Phi = 0 exactly, and the candidate is dp(i-1, k) itself
        // (x + 0 = x for x >= +0, lambda' 0 = +0): no pair load, no binary64 arithmetic.
        // Grids with many empty intervals (heavy tails) have long runs of such candidates
        // in their bands.
        const bool empty = A.N[k + 1] == Nj;
#pragma unroll
        for (int g = 0; g < kMaxG; g++) {
            if (g < G) {
                float v = __fadd_rn(A.dp32[g_at(A, g, i - 1, k)], __fmaf_rn(A.lam32[g], cf.y, cf.x));
                if (v <= T[g]) {
                    const double dprev = A.dp64[g_at(A, g, i - 1, k)];
                    double c = dprev;
                    if (!empty) {
                        const double2 e = A.pc64[tb + k];
                        c = __dadd_rn(dprev, __dadd_rn(e.x, __dmul_rn(A.lam64[g], e.y)));
                    }
                    // integer compares of the bit patterns (binary64 compares run on the
                    // binary64 pipe)
                    const long long cb = __double_as_longlong(c), bb = __double_as_longlong(best[g]);
                    // non-negative doubles (+inf included) order like their bit patterns
                    const bool lt = (cb >= 0 && bb >= 0) ? cb < bb : c < best[g];
                    if (lt) { best[g] = c; arg[g] = (int32_t)k; }  // k ascends per thread
                }
            }
        }
    }
    // least value, then lowest k: over the lanes, then over the warps
#pragma unroll
    for (int g = 0; g < kMaxG; g++) {
        double b = best[g];
        int32_t a = arg[g];
        for (int o = 16; o > 0; o >>= 1) {
            double b2 = __shfl_xor_sync(0xffffffffu, b, o);
            int32_t a2 = __shfl_xor_sync(0xffffffffu, a, o);
            if (a2 >= 0 && (a < 0 || b2 < b || (b2 == b && a2 < a))) { b = b2; a = a2; }
        }
        if (lane == 0) { sb[wid][g] = b; sa[wid][g] = a; }
    }
    __syncthreads();
    if (threadIdx.x < G) {
        const int g = threadIdx.x;
        double b = sb[0][g];
        int32_t a = sa[0][g];
        for (int w = 1; w < kGridThreads / 32; w++) {
            const double b2 = sb[w][g];
            const int32_t a2 = sa[w][g];
            if (a2 >= 0 && (a < 0 || b2 < b || (b2 == b && a2 < a))) { b = b2; a = a2; }
        }
        A.dp64[g_at(A, g, i, j)] = b;
        A.bp[g_at(A, g, i, j)] = a;
        A.dp32[g_at(A, g, i, j)] = __double2float_rn(__dmul_rn(b, A.scale));
    }
}

size_t grid_pairs_bytes(int64_t n) {
    if (n < 2 || n > kGridPairsMax) return 0;
    size_t np = (size_t)n * (size_t)(n - 1) / 2;
    return align256(16 * np) + align256(8 * np);
}

int launch_dp_clear_base(const Prefix &P, const double *lamp, int G, int s, double *dp64, int32_t *bp,
                         cudaStream_t st);

// One DP pass over the grid; build_pairs: fill the pair cache first (once per call).
int launch_dp_grid(const Prefix &P, const double *lamp, int G, int s, double *dp64, int32_t *bp, float *dp32,
                   void *pairs, bool build_pairs, int num_sms, cudaStream_t st) {
    const int64_t n = P.p;
    size_t np = (size_t)n * (size_t)(n - 1) / 2;
    GridArgs A;
    A.pc64 = reinterpret_cast<const double2 *>(pairs);
    A.pc32 = reinterpret_cast<const float2 *>(static_cast<char *>(pairs) + align256(16 * np));
    A.dp64 = dp64; A.bp = bp; A.dp32 = dp32;
    A.N = P.N;
    A.n = n; A.ps = P.ps; A.G = G; A.s = s;
    A.scale = P.scale32;
    for (int g = 0; g < kMaxG; g++) {
        double l = g < G ? lamp[g] : 0.0;
        A.lam64[g] = l;
        A.lam32[g] = (float)(l * P.scale32);
        A.slack[g] = 3.0 * (70.0 + (double)A.lam32[g]) * 0x1p-150;
    }
    if (build_pairs && np > 0) {
        note_launch();
        k_grid_pairs<<<(unsigned)std::min<int64_t>(cdiv((int64_t)np, 256), (int64_t)num_sms * 16), 256, 0, st>>>(
            P, P.scale32, reinterpret_cast<double2 *>(pairs),
            reinterpret_cast<float2 *>(static_cast<char *>(pairs) + align256(16 * np)));
        ECASQ_LAUNCH_CHECK();
    }
    // clear the tables, then eq. apx_base (min over a in L) exactly as the reference kernel
    int rc = launch_dp_clear_base(P, lamp, G, s, dp64, bp, st);
    if (rc != ECASQ_OK) return rc;
    note_launch();
    k_grid_round<<<(unsigned)std::min<int64_t>(cdiv((int64_t)G * n, 256), (int64_t)num_sms * 8), 256, 0, st>>>(A, 2);
    ECASQ_LAUNCH_CHECK();
    timer_begin(st);
    for (int i = 3; i <= s; i++) {
        if (n < i) break;
        note_launch();
        k_grid_layer<<<(unsigned)n, kGridThreads, 0, st>>>(A, i);
        ECASQ_LAUNCH_CHECK();
    }
    timer_end(st);
    return ECASQ_OK;
}

}  // namespace ecasq
