// dp_opt.cu -- the optimal DP of Sec. 4 (with App. E's first- and last-value sets
// L, R for a permissible set P) on the GPU, at up to 8 fixed multipliers per pass.
//
// State (i, l, j), l < j: the least cost of the prefix up to p_l with i-1 values
// ending at p_l, plus the MSE of (p_l, p_j] (Sec. 4).  With lambda' = lambda ||X||^2:
//   dp(2, a, j) = C[a, j] + lambda' h((n_a + D[a, j]) / d),                        a in L
//   dp(i, l, j) = C[l, j] + min_{k<l} dp(i-1, k, l) + lambda' h((U[k, l] + D[l, j]) / d)
//   answer      = min_{i <= s} min_{j in R} min_{l<j} dp(i, l, j) + lambda' h(U[l, j] / d)
// (ties: lowest k; at the answer the smallest i, then j, then l).  The entropy term
// depends on the triple (k, l, j), so a layer has about p^3 / 6 candidates; each
// candidate's h() is shared by the G multipliers.
//
// k_opt_layer: block (chunk, l) owns 256 outputs j of one l.  The column
// A_g(k) = dp(i-1, k, l) and u(k) = U[k, l] are staged in shared memory in fp32 (tiles
// of kOptTile k), A_g as its excess over the column minimum a_g = min_k A_g(k), so the
// filter's relative error applies to the excess, not to the whole prefix cost.  fp32
// pass: y = (u(k) + D[l, j]) / d, h = -y lg2(y), cand = fma(lam32, h, (A - a) scale);
// per-multiplier minimum m32.  Band pass: every k with cand <= T is re-scored in binary64
// with the oracle's formula dp(i-1,k,l) + lambda' h((U + D)/d); the lowest k among the
// exact minima wins.  Empty grid intervals make long runs of exact ties (U[k, l] = 0 for
// every k of the run, so y is the same), and the 32 outputs of a warp rarely agree on
// which k are in their bands, so band work must be cheap per lane: a member with the
// same U as the multiplier's current best and no smaller dp(i-1, k, l) cannot be strictly
// better (fl(a + c) is monotone in a), which integer compares of the bit patterns of the
// two non-negative doubles decide without fp64 arithmetic; the other members go to a
// per-lane queue in shared memory that the warp drains together (one binary64 sequence
// serves up to 32 lanes' members), in increasing k per lane, so the lowest-k rule holds
// (a skip decided against an earlier best stays valid: the best only improves); h(y) in
// binary64 is cached by the value of U[k, l]; at lambda' = 0 the candidate is
// dp(i-1, k, l) itself.
//
// Why the band holds every exact minimiser (scaled units, u = 2^-24): y32 is within
// 4.0001u of y (two input roundings, the add, the reciprocal of d and the product);
// __log2f is within 2^-22 absolute on [0.5, 2] and 2 ulp elsewhere (CUDA programming
// guide, intrinsic functions), so with |h'(t)| <= |log2 t| + log2 e the fp32 h is
// within E_h = 12u + 2^-90 of h(y) (y32 <= 2^-100 is taken as h = 0).  The staged excess
// fl32(fl64(A - a) scale) is within 1.0001u of (A - a) scale, lambda within u, and the fma
// rounds once, so |cand32 - c| <= 2.0001u c + 1.0002 lambda E_h + 2^-148 for the exact
// excess c = (A - a) scale + lambda h.  The binary64 candidate is within 2^-52 of
// A + lambda' h (relative) plus 2^-50 lambda', so an exact minimiser's excess exceeds the
// least excess by at most 2^-51 (a + c) + 2^-49 lambda.  Hence an exact minimiser has
// cand32 <= m32 (1 + 4.001u) + lambda (2.001 E_h + 2^-47) + 2^-50 a + 2^-146 < T =
// m32 (1 + 6u) + lam32 (2.1 E_h + 2^-40) + 2^-49 a + 2^-140.
#include "common.cuh"

namespace ecasq {

void timer_begin(cudaStream_t st);
void timer_end(cudaStream_t st);

constexpr int kOptTile = 1024;   // k per shared-memory tile
constexpr int kOptThreads = 256; // outputs j per block
constexpr int kOptQueue = 8;     // band members a lane holds before its warp drains the queues

struct OptArgs {
    const double *C, *U, *D;  // pair quantities, triangle j(j-1)/2 + k
    double *dp;               // [G][s-1][npair]: layer i at (i - 2)
    int32_t *bk;
    const int64_t *w;         // n_a of the base layer
    int64_t n, npair;
    int64_t nL, nR;
    int G, s;
    double dd;                // d
    float invd32;             // fl32(1 / d)
    double scale;             // 2^-e, 2^e <= ||X||^2 < 2^(e+1)
    double lam64[kMaxG];      // lambda'
    float lam32[kMaxG];       // fl32(lambda' scale)
    double slack[kMaxG];      // lam32 (2.1 E_h + 2^-40) + 2^-140
};

__host__ __device__ __forceinline__ size_t otri(int64_t k, int64_t j) { return (size_t)j * (size_t)(j - 1) / 2 + (size_t)k; }

__device__ __forceinline__ size_t oat(const OptArgs &A, int g, int i, size_t t) {
    return ((size_t)g * (size_t)(A.s - 1) + (size_t)(i - 2)) * (size_t)A.npair + t;
}

__global__ void __launch_bounds__(256) k_opt_pairs(Prefix P, double *C, double *U, double *D) {
    const int64_t npair = P.p * (P.p - 1) / 2;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < npair; t += stride) {
        int64_t j = (int64_t)((1.0 + sqrt(1.0 + 8.0 * (double)t)) * 0.5);
        while (j * (j - 1) / 2 > t) j--;
        while ((j + 1) * j / 2 <= t) j++;
        int64_t k = t - j * (j - 1) / 2;
        double c, u, dd_;
        pair_exact(P, k, j, c, u, dd_);
        C[t] = c; U[t] = u; D[t] = dd_;
    }
}

// Layer 2: dp(2, a, j) for a in L, +inf (bk = -1) for every other l.
__global__ void k_opt_base(OptArgs A) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < A.npair; t += stride) {
        int64_t j = (int64_t)((1.0 + sqrt(1.0 + 8.0 * (double)t)) * 0.5);
        while (j * (j - 1) / 2 > t) j--;
        while ((j + 1) * j / 2 <= t) j++;
        int64_t a = t - j * (j - 1) / 2;
        double hv = 0.0, c = 0.0;
        if (a < A.nL) {
            c = A.C[t];
            hv = hfun(__ddiv_rn(__dadd_rn((double)A.w[a], A.D[t]), A.dd));
        }
        for (int g = 0; g < A.G; g++) {
            A.dp[oat(A, g, 2, t)] = a < A.nL ? __dadd_rn(c, __dmul_rn(A.lam64[g], hv)) : CUDART_INF;
            A.bk[oat(A, g, 2, t)] = a < A.nL ? (int32_t)a : -1;
        }
    }
}

__device__ __forceinline__ float h32(float y) {
    return y > 0x1p-100f ? -__fmul_rn(y, __log2f(y)) : 0.0f;
}

__global__ void __launch_bounds__(kOptThreads) k_opt_layer(OptArgs A, int i) {
    __shared__ __align__(16) float sA[kOptTile][kMaxG];  // [k][g]: two 16-byte loads per k
    __shared__ float su[kOptTile];
    __shared__ long long sred[kOptThreads / 32][kMaxG];
    __shared__ int32_t qk[kOptQueue][kOptThreads];  // queued band members (k) per lane
    __shared__ uint8_t qg[kOptQueue][kOptThreads];  // ... and their multiplier masks
    __shared__ double amin[kMaxG];  // column minimum of dp(i-1, ., l) per multiplier
    const int64_t l = A.n - 2 - (int64_t)blockIdx.y;  // heavy l first
    const int64_t j0 = l + 1 + (int64_t)blockIdx.x * kOptThreads;
    if (l < 0 || j0 >= A.n) return;
    const int64_t j = j0 + threadIdx.x;
    const bool own = j < A.n;
    const int G = A.G;
    // finite predecessors: k in L at i = 3, k >= i - 3 above
    const int64_t klo = i == 3 ? 0 : i - 3;
    const int64_t khi = i == 3 ? min(A.nL, l) : l;
    const size_t tl = otri(0, l);            // U[k, l] = U[tl + k], dp(i-1, k, l) at tl + k
    const size_t tj = own ? otri(l, j) : 0;  // (l, j)
    const double D64 = own ? A.D[tj] : 0.0;
    const float D32 = __double2float_rn(D64);
    {   // column minima: integer minima of the bit patterns (the values are >= 0; -0 as +0)
        long long mn[kMaxG];
#pragma unroll
        for (int g = 0; g < kMaxG; g++) mn[g] = 0x7ff0000000000000ll;
        for (int64_t k = klo + threadIdx.x; k < khi; k += kOptThreads) {
#pragma unroll
            for (int g = 0; g < kMaxG; g++)
                if (g < G) mn[g] = min(mn[g], __double_as_longlong(A.dp[oat(A, g, i - 1, tl + k)]) & 0x7fffffffffffffffll);
        }
#pragma unroll
        for (int g = 0; g < kMaxG; g++) {
            for (int o = 16; o > 0; o >>= 1) mn[g] = min(mn[g], __shfl_xor_sync(0xffffffffu, mn[g], o));
            if ((threadIdx.x & 31) == 0) sred[threadIdx.x >> 5][g] = mn[g];
        }
        __syncthreads();
        if (threadIdx.x < kMaxG) {
            long long v = sred[0][threadIdx.x];
            for (int w = 1; w < kOptThreads / 32; w++) v = min(v, sred[w][threadIdx.x]);
            amin[threadIdx.x] = __longlong_as_double(v);
        }
        __syncthreads();
    }
    float m[kMaxG];
#pragma unroll
    for (int g = 0; g < kMaxG; g++) m[g] = CUDART_INF_F;
    auto stage = [&](int64_t kt, int nk) {
        for (int q = threadIdx.x; q < nk; q += kOptThreads) {
            su[q] = __double2float_rn(A.U[tl + kt + q]);
            for (int g = 0; g < G; g++) {
                double a = A.dp[oat(A, g, i - 1, tl + kt + q)];
                sA[q][g] = a < CUDART_INF ? __double2float_rn(__dmul_rn(__dsub_rn(a, amin[g]), A.scale)) : CUDART_INF_F;
            }
            for (int g = G; g < kMaxG; g++) sA[q][g] = CUDART_INF_F;
        }
    };
    for (int64_t kt = klo; kt < khi; kt += kOptTile) {
        const int nk = (int)min((int64_t)kOptTile, khi - kt);
        __syncthreads();
        stage(kt, nk);
        __syncthreads();
        if (own) {
            int q = 0;
            for (; q + 1 < nk; q += 2) {  // two k per step: independent lg2 chains
                float h0 = h32(__fmul_rn(__fadd_rn(su[q], D32), A.invd32));
                float h1 = h32(__fmul_rn(__fadd_rn(su[q + 1], D32), A.invd32));
                const float4 *p0 = reinterpret_cast<const float4 *>(sA[q]);
                const float4 *p1 = reinterpret_cast<const float4 *>(sA[q + 1]);
                float4 a0 = p0[0], b0 = p0[1], a1 = p1[0], b1 = p1[1];
                float v0[8] = {a0.x, a0.y, a0.z, a0.w, b0.x, b0.y, b0.z, b0.w};
                float v1[8] = {a1.x, a1.y, a1.z, a1.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
                for (int g = 0; g < kMaxG; g++)
                    m[g] = fminf(m[g], fminf(__fmaf_rn(A.lam32[g], h0, v0[g]), __fmaf_rn(A.lam32[g], h1, v1[g])));
            }
            if (q < nk) {
                float h0 = h32(__fmul_rn(__fadd_rn(su[q], D32), A.invd32));
#pragma unroll
                for (int g = 0; g < kMaxG; g++) m[g] = fminf(m[g], __fmaf_rn(A.lam32[g], h0, sA[q][g]));
            }
        }
    }
    // T rounded down to fp32: for an fp32 candidate c, c <= T32 exactly when c <= T
    float T[kMaxG];
    double best[kMaxG];
    int32_t arg[kMaxG];
    long long abest[kMaxG], ubest[kMaxG];  // bits of dp(i-1, arg, l) and U[arg, l] of the best
#pragma unroll
    for (int g = 0; g < kMaxG; g++) {
        double t = __dadd_rn(__dmul_rn((double)m[g], 1.0 + 6.0 * 0x1p-24), A.slack[g]);
        if (g < G && amin[g] < CUDART_INF) t = __dadd_rn(t, __dmul_rn(__dmul_rn(amin[g], A.scale), 0x1p-49));
        T[g] = g < G ? __double2float_rd(t) : -CUDART_INF_F;  // no member for absent multipliers
        best[g] = CUDART_INF;
        arg[g] = -1;
        abest[g] = -1;
        ubest[g] = -1;
    }
    long long ucache = -1;  // U bits whose h64 is in hcache
    double hcache = 0.0;
    int qn = 0;             // queued members of this lane
    const int tid = threadIdx.x;
    // exact evaluation of member k for the multipliers in gm (in increasing k per lane)
    auto exact = [&](int64_t k, unsigned gm) {
        const double u64 = A.U[tl + k];
        const long long ub = __double_as_longlong(u64);
#pragma unroll
        for (int g = 0; g < kMaxG; g++) {
            if (!(gm >> g & 1u)) continue;
            const double a64 = A.dp[oat(A, g, i - 1, tl + k)];
            const long long ab = __double_as_longlong(a64);
            if (ub == ubest[g] && ab >= abest[g] && ab >= 0 && abest[g] >= 0) continue;
            double c;
            if (A.lam64[g] == 0.0) {
                c = __dadd_rn(a64, 0.0);  // lambda' h = 0
            } else {
                if (ub != ucache) {
                    hcache = hfun(__ddiv_rn(__dadd_rn(u64, D64), A.dd));
                    ucache = ub;
                }
                c = __dadd_rn(a64, __dmul_rn(A.lam64[g], hcache));
            }
            if (c < best[g]) {
                best[g] = c;
                arg[g] = (int32_t)k;
                abest[g] = ab;
                ubest[g] = ub;
            }
        }
    };
    auto drain = [&]() {  // warp-uniform: every lane of the warp calls it
        int mx = __reduce_max_sync(0xffffffffu, qn);
        for (int r = 0; r < mx; r++)
            if (r < qn) exact(qk[r][tid], qg[r][tid]);
        qn = 0;
    };
    for (int64_t kt = klo; kt < khi; kt += kOptTile) {
        const int nk = (int)min((int64_t)kOptTile, khi - kt);
        if (khi - klo > kOptTile) {  // restage the tile (one tile stays resident)
            __syncthreads();
            stage(kt, nk);
            __syncthreads();
        }
        for (int q = 0; q < nk; q++) {
            if (own) {
                float h = h32(__fmul_rn(__fadd_rn(su[q], D32), A.invd32));
                const float4 *p0 = reinterpret_cast<const float4 *>(sA[q]);
                float4 a0 = p0[0], b0 = p0[1];
                float v0[8] = {a0.x, a0.y, a0.z, a0.w, b0.x, b0.y, b0.z, b0.w};
                unsigned gm = 0;
#pragma unroll
                for (int g = 0; g < kMaxG; g++)
                    if (g < G && __fmaf_rn(A.lam32[g], h, v0[g]) <= T[g]) gm |= 1u << g;
                if (gm) {
                    const int64_t k = kt + q;
                    const long long ub = __double_as_longlong(A.U[tl + k]);
                    // drop members an earlier best already rules out (same y, no smaller dp)
#pragma unroll
                    for (int g = 0; g < kMaxG; g++) {
                        if ((gm >> g & 1u) && ub == ubest[g] && abest[g] >= 0) {
                            long long ab = __double_as_longlong(A.dp[oat(A, g, i - 1, tl + k)]);
                            if (ab >= abest[g]) gm &= ~(1u << g);
                        }
                    }
                    if (gm) {
                        qk[qn][tid] = (int32_t)k;
                        qg[qn][tid] = (uint8_t)gm;
                        qn++;
                    }
                }
            }
            if (__any_sync(0xffffffffu, qn == kOptQueue)) drain();
        }
    }
    drain();
    if (!own) return;
    const double Cj = A.C[tj];
#pragma unroll
    for (int g = 0; g < kMaxG; g++) {
        if (g < G) {
            A.dp[oat(A, g, i, tj)] = arg[g] >= 0 ? __dadd_rn(Cj, best[g]) : CUDART_INF;
            A.bk[oat(A, g, i, tj)] = arg[g];
        }
    }
}

// Final selection, traceback and metrics, one block per multiplier.

__global__ void __launch_bounds__(1024) k_opt_final(OptArgs A, Prefix P, int exact_s, int32_t *qidx, int32_t *mcount,
                                                    double *metrics) {
    __shared__ double rv[1024];
    __shared__ int64_t rt[1024];
    __shared__ double scratch[4 * kMaxS];
    __shared__ int32_t a[kMaxS];
    __shared__ int sm_m;
    const int g = blockIdx.x;
    const int ilo = exact_s ? A.s : 2;
    const int64_t jlo = A.n - A.nR;
    const int64_t total = (int64_t)(A.s - ilo + 1) * A.nR * A.n;  // (i, j, l) in lexicographic order
    double bv = CUDART_INF;
    int64_t bt = -1;
    for (int64_t t = threadIdx.x; t < total; t += blockDim.x) {
        int64_t l = t % A.n;
        int64_t r = t / A.n;
        int64_t j = jlo + r % A.nR;
        int i = ilo + (int)(r / A.nR);
        if (l >= j) continue;
        size_t tj = otri(l, j);
        double v = A.dp[oat(A, g, i, tj)];
        if (!(v < CUDART_INF)) continue;
        double c = __dadd_rn(v, __dmul_rn(A.lam64[g], hfun(__ddiv_rn(A.U[tj], A.dd))));
        if (c < bv) { bv = c; bt = t; }  // t ascends per thread
    }
    rv[threadIdx.x] = bv;
    rt[threadIdx.x] = bt;
    __syncthreads();
    for (int o = 512; o > 0; o >>= 1) {
        if (threadIdx.x < o) {
            double v2 = rv[threadIdx.x + o];
            int64_t t2 = rt[threadIdx.x + o];
            if (t2 >= 0 && (rt[threadIdx.x] < 0 || v2 < rv[threadIdx.x] || (v2 == rv[threadIdx.x] && t2 < rt[threadIdx.x]))) {
                rv[threadIdx.x] = v2;
                rt[threadIdx.x] = t2;
            }
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        int64_t t = rt[0];
        if (t < 0) {
            sm_m = 0;
        } else {
            int64_t l = t % A.n, r = t / A.n;
            int64_t j = jlo + r % A.nR;
            int bi = ilo + (int)(r / A.nR);
            a[bi - 1] = (int32_t)j;
            for (int i = bi; i >= 3; i--) {
                a[i - 2] = (int32_t)l;
                int64_t k = A.bk[oat(A, g, i, otri(l, j))];
                j = l;
                l = k;
            }
            a[0] = (int32_t)l;
            sm_m = bi;
        }
        metrics[4 * g + 0] = rv[0];
        mcount[g] = sm_m;
    }
    __syncthreads();
    const int m = sm_m;
    if (threadIdx.x < 32) {
        for (int r = threadIdx.x; r < m; r += 32) qidx[g * A.s + r] = a[r];
        if (m > 0) eval_codebook_warp(P, a, m, &metrics[4 * g + 1], scratch);
    }
}

size_t opt_pairs_bytes(int64_t n) {
    size_t np = (size_t)n * (size_t)(n - 1) / 2;
    return 3 * align256(8 * np);
}

size_t opt_tables_bytes(int64_t n, int s, int G) {
    size_t np = (size_t)n * (size_t)(n - 1) / 2;
    size_t cells = (size_t)G * (size_t)(s - 1) * np;
    return align256(8 * cells) + align256(4 * cells);
}

// One optimal-DP pass: pair quantities (once per call when build_pairs), base layer,
// layers 3..s, final selection + traceback + metrics into qidx / mcount / metrics.
int launch_opt_dp(const Prefix &P, const double *lamp, int G, int s, int exact_s, void *pairs, bool build_pairs,
                  void *tables, int32_t *qidx, int32_t *mcount, double *metrics, int num_sms, cudaStream_t st) {
    const int64_t n = P.p;
    const size_t np = (size_t)n * (size_t)(n - 1) / 2;
    OptArgs A;
    char *pb = static_cast<char *>(pairs);
    A.C = reinterpret_cast<const double *>(pb);
    A.U = reinterpret_cast<const double *>(pb + align256(8 * np));
    A.D = reinterpret_cast<const double *>(pb + 2 * align256(8 * np));
    const size_t cells = (size_t)G * (size_t)(s - 1) * np;
    A.dp = static_cast<double *>(tables);
    A.bk = reinterpret_cast<int32_t *>(static_cast<char *>(tables) + align256(8 * cells));
    A.w = P.w;
    A.n = n; A.npair = (int64_t)np; A.nL = P.nL; A.nR = P.nR;
    A.G = G; A.s = s;
    A.dd = (double)P.d;
    A.invd32 = (float)(1.0 / (double)P.d);
    A.scale = P.scale32;
    const double Eh = 12.0 * 0x1p-24 + 0x1p-90;
    for (int g = 0; g < kMaxG; g++) {
        double l = g < G ? lamp[g] : 0.0;
        A.lam64[g] = l;
        A.lam32[g] = (float)(l * P.scale32);
        A.slack[g] = (double)A.lam32[g] * (2.1 * Eh + 0x1p-40) + 0x1p-140;
    }
    if (build_pairs) {
        note_launch();
        k_opt_pairs<<<(unsigned)std::min<int64_t>(cdiv((int64_t)np, 256), (int64_t)num_sms * 16), 256, 0, st>>>(
            P, const_cast<double *>(A.C), const_cast<double *>(A.U), const_cast<double *>(A.D));
        ECASQ_LAUNCH_CHECK();
    }
    note_launch();
    k_opt_base<<<(unsigned)std::min<int64_t>(cdiv((int64_t)np, 256), (int64_t)num_sms * 16), 256, 0, st>>>(A);
    ECASQ_LAUNCH_CHECK();
    timer_begin(st);
    const unsigned nchunk = (unsigned)cdiv(n - 1, kOptThreads);
    for (int i = 3; i <= s; i++) {
        note_launch();
        k_opt_layer<<<dim3(nchunk, (unsigned)(n - 1)), kOptThreads, 0, st>>>(A, i);
        ECASQ_LAUNCH_CHECK();
    }
    timer_end(st);
    note_launch();
    k_opt_final<<<G, 1024, 0, st>>>(A, P, exact_s, qidx, mcount, metrics);
    ECASQ_LAUNCH_CHECK();
    return ECASQ_OK;
}

}  // namespace ecasq
