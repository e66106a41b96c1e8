// dp_ref.cu -- fp64 reference kernels of the approximate DP (Sec. 5) and the
// traceback / evaluation that every DP pass ends with.
//
// The reference DP evaluates every candidate of eq. apx_rec in binary64 with
// interval costs from double-double prefix differences (App. E), one layer per
// launch.  It is the slow, exact path (ECASQ_DP_REFERENCE) against which the
// fast kernel is validated; the traceback and evaluation kernels serve both.
#include "common.cuh"

namespace ecasq {

void timer_begin(cudaStream_t st);
void timer_end(cudaStream_t st);

struct Lams { double v[kMaxG]; };

__device__ __forceinline__ size_t dp_at(int g, int i, int64_t j, int s, int64_t p) {
    return ((size_t)g * (size_t)(s + 1) + (size_t)i) * (size_t)p + (size_t)j;
}

// Rows 0, 1 and every undefined entry: dp = +inf, bp = -1.
__global__ void k_dp_clear(double *dp64, int32_t *bp, int G, int s, int64_t p) {
    size_t n = (size_t)G * (size_t)(s + 1) * (size_t)p;
    size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    size_t stride = (size_t)gridDim.x * blockDim.x;
    for (; i < n; i += stride) { dp64[i] = CUDART_INF; bp[i] = -1; }
}

// eq. apx_base: dp(2, j) = min over a in L, a < j, of C[a, j] + lambda' Phi^first[a, j]
// (lowest a among exact minima; L = {0} when P = X).
__global__ void k_dp_base(Prefix P, Lams lam, int G, int s, double *dp64, int32_t *bp) {
    int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x + 1;
    if (j >= P.p) return;
    double best[kMaxG];
    int32_t arg[kMaxG];
#pragma unroll
    for (int g = 0; g < kMaxG; g++) { best[g] = CUDART_INF; arg[g] = -1; }
    for (int64_t a = 0; a < P.nL && a < j; a++) {
        double C, U, D;
        pair_exact(P, a, j, C, U, D);
        double phi = phi_first_at(P, a, U, D);
#pragma unroll
        for (int g = 0; g < kMaxG; g++) {
            if (g < G) {
                double c = __dadd_rn(C, __dmul_rn(lam.v[g], phi));
                if (c < best[g]) { best[g] = c; arg[g] = (int32_t)a; }
            }
        }
    }
    for (int g = 0; g < G; g++) {
        dp64[dp_at(g, 2, j, s, P.ps)] = best[g];
        bp[dp_at(g, 2, j, s, P.ps)] = arg[g];
    }
}

// eq. apx_rec, one layer i >= 3 for all G multipliers: thread per j, every
// k in [i-2, j-1], candidate dp(i-1, k) + (C[k,j] + lambda' Phi[k,j]); the
// lowest k among exact minima wins.  Heavy (large-j) blocks launch first.
__global__ void __launch_bounds__(128) k_dp_layer_ref(Prefix P, Lams lam, int G, int s, int i, double *dp64,
                                                      int32_t *bp) {
    int64_t nblk = gridDim.x;
    int64_t j = (nblk - 1 - blockIdx.x) * blockDim.x + threadIdx.x;
    if (j < i - 1 || j >= P.p) return;
    double best[kMaxG];
    int32_t arg[kMaxG];
#pragma unroll
    for (int g = 0; g < kMaxG; g++) { best[g] = CUDART_INF; arg[g] = -1; }
    for (int64_t k = i - 2; k < j; k++) {
        double C, U, D;
        pair_exact(P, k, j, C, U, D);
        double phi = phi_exact(P, U, D, false);
#pragma unroll
        for (int g = 0; g < kMaxG; g++) {
            if (g < G) {
                double prev = dp64[dp_at(g, i - 1, k, s, P.ps)];
                double c = __dadd_rn(prev, __dadd_rn(C, __dmul_rn(lam.v[g], phi)));
                if (c < best[g]) { best[g] = c; arg[g] = (int32_t)k; }
            }
        }
    }
    for (int g = 0; g < G; g++) {
        dp64[dp_at(g, i, j, s, P.ps)] = best[g];
        bp[dp_at(g, i, j, s, P.ps)] = arg[g];
    }
}

// eq. apx_final over i and j in R (smallest i, then smallest j, among exact minima;
// i = s only with EXACT_S) and the backpointer walk down to the first value
// a = bp(2, .), then the metrics of the traced codebook.  Block g = one multiplier,
// one warp.
__global__ void k_traceback_eval(Prefix P, int G, int s, int exact_s, const double *dp64, const int32_t *bp,
                                 int32_t *qidx, int32_t *mcount, double *metrics) {
    __shared__ double scratch[4 * kMaxS];
    __shared__ int32_t a[kMaxS];
    __shared__ int sm_m;
    int g = blockIdx.x;
    int64_t p = P.p;
    if (threadIdx.x == 0) {
        int istar = -1;
        int64_t jstar = -1;
        double best = CUDART_INF;
        for (int i = exact_s ? s : 2; i <= s; i++)
            for (int64_t jr = p - P.nR; jr < p; jr++) {
                double v = dp64[dp_at(g, i, jr, s, P.ps)];
                if (v < best) { best = v; istar = i; jstar = jr; }
            }
        if (istar < 0) {
            sm_m = 0;
        } else {
            int64_t j = jstar;
            a[istar - 1] = (int32_t)j;
            bool ok = true;  // every output on the path carries a backpointer (not so after a timed-out wait)
            for (int i = istar; i >= 3 && ok; i--) {
                j = bp[dp_at(g, i, j, s, P.ps)];
                ok = j >= 0;
                a[i - 2] = (int32_t)j;
            }
            if (ok) a[0] = bp[dp_at(g, 2, j, s, P.ps)];
            sm_m = (ok && a[0] >= 0) ? istar : 0;
        }
        metrics[4 * g + 0] = best;
        mcount[g] = sm_m;
    }
    __syncwarp();
    int m = sm_m;
    for (int r = threadIdx.x; r < m; r += 32) qidx[g * s + r] = a[r];
    if (m > 0 && m <= 32)
        eval_codebook_lanes(P, a, m, &metrics[4 * g + 1]);  // the same values, one interval per lane
    else if (m > 0)
        eval_codebook_warp(P, a, m, &metrics[4 * g + 1], scratch);
}

// Metrics of a caller-given codebook (unique indices on the device); nothing when
// gate is given and holds 0 (the caller then reads no result).
__global__ void k_eval_codebook(Prefix P, const int32_t *a_in, int m, double *out3, const int32_t *gate) {
    __shared__ double scratch[4 * kMaxS];
    __shared__ int32_t a[kMaxS];
    if (gate && *gate == 0) return;
    for (int r = threadIdx.x; r < m; r += 32) a[r] = a_in[r];
    __syncwarp();
    if (m <= 32)
        eval_codebook_lanes(P, a, m, out3);  // the same values, one interval per lane
    else
        eval_codebook_warp(P, a, m, out3, scratch);
}

// Q[r] = v[a[r]] for every multiplier row g.
__global__ void k_gather_q(const float *v, const int32_t *qidx, const int32_t *mcount, int s, float *Q) {
    int g = blockIdx.x;
    int m = mcount[g];
    for (int r = threadIdx.x; r < m; r += blockDim.x) Q[g * s + r] = v[qidx[g * s + r]];
}

// Unique indices of a codebook given by value (binary search in v); -1 if absent.
__global__ void k_locate_q(const float *v, int64_t p, const float *Q, int m, int32_t *a, DevStatus *st) {
    for (int r = threadIdx.x; r < m; r += blockDim.x) {
        float q = Q[r];
        if (q == 0.0f) q = 0.0f;
        int64_t lo = 0, hi = p - 1;
        while (lo < hi) {
            int64_t mid = (lo + hi) >> 1;
            if (v[mid] < q) lo = mid + 1; else hi = mid;
        }
        bool ok = v[lo] == q;
        a[r] = ok ? (int32_t)lo : -1;
        if (!ok) st->range_err = 1;
    }
}

// ------------------------------------------------------------ short rows
// One DP pass of the search for many independent rows (p <= kRowsMaxP), one block
// per row: the interval costs of every pair k < j of the row are computed once into
// shared memory (pair_exact / phi_exact, the reference formulas), then eq. apx_base
// and apx_rec run for the row's G multipliers with two layers in shared memory
// (candidates, lowest k and smallest i exactly as k_dp_base, k_dp_layer_ref and
// k_traceback_eval), and each multiplier's codebook is traced and evaluated by
// eval_codebook_warp.  Backpointers go to the caller's scratch.
__host__ __device__ __forceinline__ int tri(int k, int j) { return j * (j - 1) / 2 + k; }

constexpr int kRowsThreads = 512;  // 16 warps: two blocks per SM fit the shared-memory pair caches
__global__ void __launch_bounds__(kRowsThreads) k_rows_pass(RowsPass A) {
    extern __shared__ __align__(16) double rsm[];
    const int b = blockIdx.x;
    const int64_t row = A.rows[b];
    const RowsData &R = A.R;
    const int64_t dcap = R.dcap;
    const int p = (int)R.p[row];
    const int G = A.G, s = A.s;
    Prefix P;
    P.v = R.v + row * dcap;
    P.w = R.w + row * dcap;
    P.N = R.N + row * (dcap + 1);
    P.S = R.S + row * 2 * (dcap + 1);
    P.S2 = R.S2 + row * 2 * (dcap + 1);
    P.p = p;
    P.d = R.d;
    P.ps = p;
    const int npair = p * (p - 1) / 2;
    double *PhF = rsm;                    // [p]   Phi^first[0, j]
    double *dpb = PhF + p;                // [2][G][p] binary64 layers
    double *last = dpb + 2 * G * p;       // [G][s+1] dp(i, p-1)
    double *scratch = last + G * (s + 1);  // [4 kMaxS] evaluation scratch
    // [npair] {C scale, Phi}, k-major: pair (k, j) at koff(k) + j - k - 1, koff(k) = k p - k (k + 1) / 2,
    // so the lanes of a warp (consecutive j, one k) read consecutive words
    float2 *pc32 = reinterpret_cast<float2 *>(scratch + 4 * kMaxS);
    float *d32 = reinterpret_cast<float *>(pc32 + npair);            // [2][G][p] dp scale, fp32
    // backpointers: read only by this block's traceback, so they stay in shared memory
    // (int8: a row has at most kRowsMaxP = 128 unique values) unless that does not fit
    int8_t *bps = reinterpret_cast<int8_t *>(d32 + 2 * (size_t)G * p);  // [G][s+1][p]
    __shared__ int32_t a_sm[kMaxS];
    __shared__ int sm_m;
    __shared__ int next_out[2];  // per layer parity: outputs handed out so far
    // the row's scale 2^-e (2^e <= ||X_row||^2 < 2^(e+1)) keeps the fp32 copies near 1
    const double n2 = R.norm2[row];
    const double scale = (n2 > 0.0 && isfinite(n2)) ? ldexp(1.0, -ilogb(n2)) : 1.0;
    __shared__ double lam[kMaxG], slack[kMaxG];
    __shared__ float lam32[kMaxG];
    if (threadIdx.x < kMaxG) {
        const int g = threadIdx.x;
        lam[g] = g < G ? A.lam[(size_t)b * G + g] : 0.0;
        lam32[g] = __double2float_rn(__dmul_rn(lam[g], scale));
        slack[g] = 3.0 * (70.0 + (double)lam32[g]) * 0x1p-150;
    }
    // the row's interval costs, kept across rounds in `pairs`: binary64 {C, Phi} by pair,
    // Phi^first, and the fp32 copies
    // (plain 8-byte accesses: a row's cache starts on a multiple of 8 bytes, not of 16)
    double *gp = A.pairs + row * A.pstride;
    double *gpc64 = gp;  // {C, Phi} of pair t at gpc64[2 t], gpc64[2 t + 1]
    double *gphf = gp + 2 * (size_t)npair;
    float2 *gpc32 = reinterpret_cast<float2 *>(gphf + p);
    if (A.pairs_ready) {
        for (int t = threadIdx.x; t < npair; t += blockDim.x) pc32[t] = gpc32[t];
        for (int t = threadIdx.x; t < p; t += blockDim.x) PhF[t] = gphf[t];
    } else {
        for (int t = threadIdx.x; t < npair; t += blockDim.x) {
            int j = (int)((1.0 + sqrt(1.0 + 8.0 * (double)t)) * 0.5);
            while (j * (j - 1) / 2 > t) j--;
            while ((j + 1) * j / 2 <= t) j++;
            int k = t - j * (j - 1) / 2;
            double C, U, D;
            pair_exact(P, k, j, C, U, D);
            const double F = phi_exact(P, U, D, false);
            gpc64[2 * (size_t)t] = C;
            gpc64[2 * (size_t)t + 1] = F;
            const float2 c32 = make_float2(__double2float_rn(__dmul_rn(C, scale)), __double2float_rn(F));
            const int r = k * p - k * (k + 1) / 2 + (j - k - 1);
            pc32[r] = c32;
            gpc32[r] = c32;
            if (k == 0) { PhF[j] = phi_exact(P, U, D, true); gphf[j] = PhF[j]; }
        }
    }
    for (int q = threadIdx.x; q < G * (s + 1); q += blockDim.x) last[q] = CUDART_INF;
    if (threadIdx.x < 2) next_out[threadIdx.x] = 0;
    int32_t *bp = A.bp + (size_t)b * G * (s + 1) * dcap;
    const bool bp_sm = A.bp_smem != 0;
    auto set_bp = [&](int g, int i, int j, int32_t v) {
        if (bp_sm) bps[((size_t)g * (s + 1) + i) * p + j] = (int8_t)v;
        else bp[((size_t)g * (s + 1) + i) * dcap + j] = v;
    };
    __syncthreads();
    // eq. apx_base: dp(2, j) = C[0, j] + lambda' Phi^first[0, j]
    for (int q = threadIdx.x; q < G * p; q += blockDim.x) {
        int g = q / p, j = q % p;
        double v = CUDART_INF;
        int32_t arg = -1;
        if (j >= 1) { v = __dadd_rn(gpc64[2 * (size_t)tri(0, j)], __dmul_rn(lam[g], PhF[j])); arg = 0; }
        dpb[g * p + j] = v;
        d32[g * p + j] = __double2float_rn(__dmul_rn(v, scale));
        set_bp(g, 2, j, arg);
        if (j == p - 1) last[g * (s + 1) + 2] = v;
    }
    __syncthreads();
    // eq. apx_rec, layers 3..s: an fp32 pass over k finds the fp32 minimum m32; every k whose
    // fp32 candidate is within the certified band of m32 is re-scored with the binary64
    // candidate, and the lowest k among the exact minima wins (the result of the binary64
    // recurrence, bit for bit).  The band, as in the grid DP: all terms are >= 0, each fp32
    // input is within u = 2^-24 (relative) of its binary64 value or 2^-150 (absolute) when
    // subnormal, the fma and the add round once each, so an exact minimiser has
    // val32 <= (m32 + A)(1 + 8.0001u) + A < m32 (1 + 10u) + 3A, A = (70 + lam32) 2^-150.
    // The outputs of a layer go to the warps in order of decreasing work (j descending, all
    // multipliers of one j together), 32 at a time from a shared counter, so no thread
    // waits on one that drew the longest scans.  Each output takes one fp32 pass over k:
    // the running minimum m32 and, for every k, whether its value is within a conservative
    // band of the running minimum, Tr(x) = ru(ru(x (1 + 2^-20)) + ru(2 slack)) >= T(x) for
    // x >= 0, non-decreasing in x; the running minimum only falls, so every k within the
    // final band T(m32) was within Tr of the minimum at its visit, and the bits marked hold
    // every member (the re-scoring re-checks each against T(m32)).
    const int lane = threadIdx.x & 31;
    const int nout = G * p;
    int cur = 0;
    for (int i = 3; i <= s; i++) {
        const double *prev = dpb + (size_t)cur * G * p;
        const float *prev32 = d32 + (size_t)cur * G * p;
        double *nxt = dpb + (size_t)(cur ^ 1) * G * p;
        float *nxt32 = d32 + (size_t)(cur ^ 1) * G * p;
        int *ctr = &next_out[i & 1];
        if (threadIdx.x == 0) next_out[(i + 1) & 1] = 0;  // the next layer's counter (unused until the barrier)
        for (;;) {
            int base = 0;
            if (lane == 0) base = atomicAdd(ctr, 32);
            base = __shfl_sync(0xffffffffu, base, 0);
            if (base >= nout) break;  // warp-uniform
            const int q = base + lane;
            if (q >= nout) continue;
            const int g = q % G, j = p - 1 - q / G;
            const int tb = j * (j - 1) / 2;
            const float l32 = lam32[g];
            const float sl = __double2float_ru(__dmul_rn(2.0, slack[g]));
            const float *pv = prev32 + g * p;
            float m32 = CUDART_INF_F, Tr = CUDART_INF_F;
            uint32_t mkw[4];
#pragma unroll
            for (int w = 0; w < 4; w++) {
                const int k0 = max(i - 2, 32 * w), k1 = min(j, 32 * w + 32);
                uint32_t mk = 0u;
                int ko = k0 * p - k0 * (k0 + 1) / 2 - 1;  // koff(k0) - 1: pair (k, j) at ko + j - k
                for (int k = k0; k < k1; ko += p - k - 1, k++) {
                    const float2 cf = pc32[ko + j - k];
                    const float v = __fadd_rn(pv[k], __fmaf_rn(l32, cf.y, cf.x));
                    if (v < m32) {
                        m32 = v;
                        Tr = __fadd_ru(__fmul_ru(v, 1.0f + 0x1p-20f), sl);
                    }
                    mk |= (v <= Tr ? 1u : 0u) << (k & 31);
                }
                mkw[w] = mk;
            }
            const float T = __double2float_rd(__dadd_rn(__dmul_rn((double)m32, 1.0 + 10.0 * 0x1p-24), slack[g]));
            // members re-scored in binary64 in increasing k (the lowest k among exact minima)
            double best = CUDART_INF;
            int32_t arg = -1;
#pragma unroll
            for (int w = 0; w < 4; w++) {
                uint32_t mk = mkw[w];
                while (mk) {
                    const int k = 32 * w + __ffs(mk) - 1;
                    mk &= mk - 1u;
                    const float2 cf = pc32[k * p - k * (k + 1) / 2 + j - k - 1];
                    if (!(__fadd_rn(pv[k], __fmaf_rn(l32, cf.y, cf.x)) <= T)) continue;
                    const double *e = gpc64 + 2 * (size_t)(tb + k);
                    const double c = __dadd_rn(prev[g * p + k], __dadd_rn(e[0], __dmul_rn(lam[g], e[1])));
                    if (c < best) { best = c; arg = k; }
                }
            }
            nxt[g * p + j] = best;
            nxt32[g * p + j] = __double2float_rn(__dmul_rn(best, scale));
            set_bp(g, i, j, arg);
            if (j == p - 1) last[g * (s + 1) + i] = best;
        }
        __syncthreads();
        cur ^= 1;
    }
    // eq. apx_final and the traceback of multiplier g into a[0..m-1] (lane 0); returns m
    auto trace = [&](int g, int32_t *a) -> int {
        int istar = -1;
        double best = CUDART_INF;
        for (int i = A.exact_s ? s : 2; i <= s; i++) {
            double v = last[g * (s + 1) + i];
            if (v < best) { best = v; istar = i; }
        }
        int m = 0;
        if (istar >= 0) {
            int64_t j = p - 1;
            a[istar - 1] = (int32_t)j;
            for (int i = istar; i >= 3; i--) {
                j = bp_sm ? (int64_t)bps[((size_t)g * (s + 1) + i) * p + j]
                          : (int64_t)bp[((size_t)g * (s + 1) + i) * dcap + j];
                a[i - 2] = (int32_t)j;
            }
            a[0] = 0;
            m = istar;
        }
        A.metrics[((size_t)b * G + g) * 4 + 0] = best;
        A.mcount[(size_t)b * G + g] = m;
        return m;
    };
    if (s <= 32) {
        // codebooks of at most 32 values: warp g takes multiplier g, its lanes holding one
        // interval each (eval_codebook_lanes), so no warp of the block waits on a serial tail
        __shared__ int32_t a_w[kMaxG][32];
        __shared__ int m_w[kMaxG];
        const int g = threadIdx.x >> 5;
        if (g < G) {
            if (lane == 0) m_w[g] = trace(g, a_w[g]);
            __syncwarp();
            const int m = m_w[g];
            if (lane < m) A.qidx[((size_t)b * G + g) * s + lane] = a_w[g][lane];
            if (m > 0) eval_codebook_lanes(P, a_w[g], m, &A.metrics[((size_t)b * G + g) * 4 + 1]);
        }
    } else if (threadIdx.x < 32) {  // one warp, multiplier by multiplier
        for (int g = 0; g < G; g++) {
            if (threadIdx.x == 0) sm_m = trace(g, a_sm);
            __syncwarp();
            const int m = sm_m;
            for (int r = threadIdx.x; r < m; r += 32) A.qidx[((size_t)b * G + g) * s + r] = a_sm[r];
            if (m > 0) eval_codebook_warp(P, a_sm, m, &A.metrics[((size_t)b * G + g) * 4 + 1], scratch);
            __syncwarp();
        }
    }
}

size_t rows_pass_smem(int p, int G, int s, bool bp_smem) {
    size_t npair = (size_t)p * (p - 1) / 2;
    return sizeof(double) * ((size_t)p + 2 * (size_t)G * p + (size_t)G * (s + 1) + 4 * (size_t)kMaxS) +
           sizeof(float2) * npair + sizeof(float) * 2 * (size_t)G * p +
           (bp_smem ? (size_t)G * (s + 1) * p : 0);
}
// Backpointers in shared memory when that still leaves room for two blocks per SM.
static bool rows_bp_in_smem(int p, int G, int s) { return rows_pass_smem(p, G, s, true) <= 110 * 1024; }

int launch_rows_pass(const RowsPass &A, int nact, int pmax, cudaStream_t st) {
    if (nact == 0) return ECASQ_OK;
    if (pmax > kRowsMaxP) return ECASQ_EINVAL;
    RowsPass B = A;
    B.bp_smem = rows_bp_in_smem(pmax, A.G, A.s) ? 1 : 0;
    size_t smem = rows_pass_smem(pmax, A.G, A.s, B.bp_smem != 0);
    ECASQ_CUDA_TRY(cudaFuncSetAttribute(k_rows_pass, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    note_launch();
    k_rows_pass<<<(unsigned)nact, kRowsThreads, smem, st>>>(B);
    ECASQ_LAUNCH_CHECK();
    return ECASQ_OK;
}

// Q[row][r] = v_row[a[row][r]] for the selected codebooks.
__global__ void k_rows_gather(RowsData R, const int32_t *a, const int32_t *m, int s, float *Q) {
    const int64_t row = blockIdx.x;
    const float *v = R.v + row * R.dcap;
    for (int r = threadIdx.x; r < m[row]; r += blockDim.x) Q[row * s + r] = v[a[row * s + r]];
}

int launch_rows_gather(const RowsData &R, const int32_t *a, const int32_t *m, int64_t rows, int s, float *Q,
                       cudaStream_t st) {
    note_launch();
    k_rows_gather<<<(unsigned)rows, 32, 0, st>>>(R, a, m, s, Q);
    ECASQ_LAUNCH_CHECK();
    return ECASQ_OK;
}

// ----------------------------------------------------------- host launchers
// Tables cleared (dp = +inf, bp = -1) and layer 2 (eq. apx_base) filled.
int launch_dp_clear_base(const Prefix &P, const double *lamp, int G, int s, double *dp64, int32_t *bp,
                         cudaStream_t st) {
    Lams lam{};
    for (int g = 0; g < G; g++) lam.v[g] = lamp[g];
    note_launch();
    k_dp_clear<<<4096, 256, 0, st>>>(dp64, bp, G, s, P.ps);
    ECASQ_LAUNCH_CHECK();
    if (P.p >= 2) {
        note_launch();
        k_dp_base<<<(unsigned)cdiv(P.p - 1, 128), 128, 0, st>>>(P, lam, G, s, dp64, bp);
        ECASQ_LAUNCH_CHECK();
    }
    return ECASQ_OK;
}

int launch_dp_reference(const Prefix &P, const double *lamp, int G, int s, double *dp64, int32_t *bp,
                        cudaStream_t st) {
    Lams lam{};
    for (int g = 0; g < G; g++) lam.v[g] = lamp[g];
    int rc = launch_dp_clear_base(P, lamp, G, s, dp64, bp, st);
    if (rc != ECASQ_OK) return rc;
    timer_begin(st);
    for (int i = 3; i <= s; i++) {
        if (P.p < i) break;
        note_launch();
        k_dp_layer_ref<<<(unsigned)cdiv(P.p, 128), 128, 0, st>>>(P, lam, G, s, i, dp64, bp);
        ECASQ_LAUNCH_CHECK();
    }
    timer_end(st);
    return ECASQ_OK;
}

int launch_traceback_eval(const Prefix &P, int G, int s, int exact_s, const double *dp64, const int32_t *bp,
                          int32_t *qidx, int32_t *mcount, double *metrics, cudaStream_t st) {
    note_launch();
    k_traceback_eval<<<G, 32, 0, st>>>(P, G, s, exact_s, dp64, bp, qidx, mcount, metrics);
    ECASQ_LAUNCH_CHECK();
    return ECASQ_OK;
}

int launch_eval_codebook(const Prefix &P, const int32_t *a, int m, double *out3, cudaStream_t st,
                         const int32_t *gate) {
    note_launch();
    k_eval_codebook<<<1, 32, 0, st>>>(P, a, m, out3, gate);
    ECASQ_LAUNCH_CHECK();
    return ECASQ_OK;
}

int launch_gather_q(const float *v, const int32_t *qidx, const int32_t *mcount, int G, int s, float *Q,
                    cudaStream_t st) {
    note_launch();
    k_gather_q<<<G, 64, 0, st>>>(v, qidx, mcount, s, Q);
    ECASQ_LAUNCH_CHECK();
    return ECASQ_OK;
}

int launch_locate_q(const float *v, int64_t p, const float *Q, int m, int32_t *a, DevStatus *ds, cudaStream_t st) {
    note_launch();
    k_locate_q<<<1, 256, 0, st>>>(v, p, Q, m, a, ds);
    ECASQ_LAUNCH_CHECK();
    return ECASQ_OK;
}

}  // namespace ecasq
