// dp_linear.cu -- linear-space traceback of the approximate DP (Sec. 5, last paragraph:
// Hirschberg's method specialised to eq. apx_rec), in binary64 with the reference
// interval costs (pair_exact, phi_exact).
//
// Link cost of consecutive values k < j: C[k, j] + lambda' Phi[k, j], with Phi^first when
// k is the first value (index 0).  Every pass keeps two rows of p values:
//  * forward from u, layer r: G_r(c) = min over k in [u + r - 2, c - 1] of G_{r-1}(k) +
//    link(k, c) (G_2(c) = link(u, c)), the least cost of a chain of r values from u to c;
//  * backward to v, layer r: B_r(c) = min over j in [c + 1, v - r + 2] of link(c, j) +
//    B_{r-1}(j) (B_2(c) = link(c, v)), the least cost of a chain of r values from c to v.
// A forward pass from the first value over every layer gives dp(i, p-1) and the answer of
// eq. apx_final (m = the smallest i with the least value).  Then subproblem (u, v, n) --
// n values with u and v fixed at the ends -- is split at the middle position t = (n+1)/2:
// the middle value is the lowest c among the exact binary64 minima of G_t(c) +
// B_{n-t+1}(c), and (u, c, t), (c, v, n - t + 1) follow.  The host keeps the stack of
// subproblems (it reads one index per split); all arithmetic runs here.
#include <algorithm>
#include <vector>

#include "common.cuh"

namespace ecasq {

__device__ __forceinline__ double lin_link(const Prefix &P, int64_t k, int64_t j, double lam) {
    double C, U, D;
    pair_exact(P, k, j, C, U, D);
    return __dadd_rn(C, __dmul_rn(lam, phi_exact(P, U, D, k == 0)));
}

// Warp-wide minimum of a binary64 value (minima are exact: the order does not matter).
__device__ __forceinline__ double warp_min(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmin(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Forward layer r >= 3: outputs c in [c_lo, c_hi] (c_lo = u + r - 1), one warp each, the
// lanes splitting k in [u + r - 2, c - 1].  With col, the value at c = p - 1 also goes to col[r].
__global__ void __launch_bounds__(256) k_lin_fwd(Prefix P, const double *gin, double *gout, int64_t u, int r,
                                                 int64_t c_lo, int64_t c_hi, double lam, double *col) {
    const int64_t c = c_lo + (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (c > c_hi) return;  // warp-uniform
    double b = CUDART_INF;
    for (int64_t k = u + r - 2 + lane; k < c; k += 32) b = fmin(b, __dadd_rn(gin[k], lin_link(P, k, c, lam)));
    b = warp_min(b);
    if (lane == 0) {
        gout[c] = b;
        if (col && c == P.p - 1) col[r] = b;
    }
}

// Forward layer 2 from u: G_2(c) = link(u, c), c in [u + 1, c_hi].
__global__ void k_lin_fwd2(Prefix P, double *gout, int64_t u, int64_t c_hi, double lam, double *col) {
    const int64_t c = u + 1 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (c > c_hi) return;
    const double v = lin_link(P, u, c, lam);
    gout[c] = v;
    if (col && c == P.p - 1) col[2] = v;
}

// Backward layer r >= 3: outputs c in [c_lo, c_hi] (c_hi = v - r + 1), one warp each, the
// lanes splitting j in [c + 1, v - r + 2].
__global__ void __launch_bounds__(256) k_lin_bwd(Prefix P, const double *bin, double *bout, int64_t v, int r,
                                                 int64_t c_lo, int64_t c_hi, double lam) {
    const int64_t c = c_lo + (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (c > c_hi) return;
    double b = CUDART_INF;
    for (int64_t j = c + 1 + lane; j <= v - r + 2; j += 32) b = fmin(b, __dadd_rn(lin_link(P, c, j, lam), bin[j]));
    b = warp_min(b);
    if (lane == 0) bout[c] = b;
}

// Backward layer 2 to v: B_2(c) = link(c, v), c in [c_lo, v - 1].
__global__ void k_lin_bwd2(Prefix P, double *bout, int64_t v, int64_t c_lo, double lam) {
    const int64_t c = c_lo + (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= v) return;
    bout[c] = lin_link(P, c, v, lam);
}

// The middle value: the lowest c in [c_lo, c_hi] among the minima of G(c) + B(c) (one block).
__global__ void __launch_bounds__(1024) k_lin_split(const double *G, const double *B, int64_t c_lo, int64_t c_hi,
                                                    int64_t *out) {
    __shared__ double sv[32];
    __shared__ int64_t si[32];
    double bv = CUDART_INF;
    int64_t bi = INT64_MAX;
    for (int64_t c = c_lo + threadIdx.x; c <= c_hi; c += blockDim.x) {
        const double x = __dadd_rn(G[c], B[c]);
        if (x < bv) { bv = x; bi = c; }  // increasing c: the first of equal values is the lowest
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const double ov = __shfl_xor_sync(0xffffffffu, bv, o);
        const int64_t oi = __shfl_xor_sync(0xffffffffu, bi, o);
        if (ov < bv || (ov == bv && oi < bi)) { bv = ov; bi = oi; }
    }
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0) { sv[wid] = bv; si[wid] = bi; }
    __syncthreads();
    if (wid == 0) {
        const int nw = blockDim.x >> 5;
        bv = lane < nw ? sv[lane] : CUDART_INF;
        bi = lane < nw ? si[lane] : INT64_MAX;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const double ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int64_t oi = __shfl_xor_sync(0xffffffffu, bi, o);
            if (ov < bv || (ov == bv && oi < bi)) { bv = ov; bi = oi; }
        }
        if (lane == 0) *out = bv < CUDART_INF ? bi : -1;
    }
}

// eq. apx_final over col[2..s] (or col[s] alone): m = the smallest i with the least value;
// layers above p (no chain of that many values) do not exist.
__global__ void k_lin_pick(const double *col, int s, int exact_s, int64_t p, int32_t *m_out, double *best_out) {
    if (threadIdx.x != 0 || blockIdx.x != 0) return;
    double best = CUDART_INF;
    int m = -1;
    for (int i = exact_s ? s : 2; i <= s && i <= p; i++)
        if (col[i] < best) { best = col[i]; m = i; }
    *m_out = m;
    *best_out = best;
}

static int fwd_layers(const Prefix &P, double *r0, double *r1, int64_t u, int64_t c_hi, int t, double lam,
                      double *col, cudaStream_t st, double **last) {
    // layers 2..t of the forward pass from u over c <= c_hi; *last: the row holding layer t
    note_launch();
    k_lin_fwd2<<<(unsigned)cdiv(std::max<int64_t>(c_hi - u, 1), 256), 256, 0, st>>>(P, r0, u, c_hi, lam, col);
    ECASQ_LAUNCH_CHECK();
    double *a = r0, *b = r1;
    for (int r = 3; r <= t; r++) {
        const int64_t c_lo = u + r - 1;
        if (c_lo > c_hi) break;
        note_launch();
        k_lin_fwd<<<(unsigned)cdiv(c_hi - c_lo + 1, 8), 256, 0, st>>>(P, a, b, u, r, c_lo, c_hi, lam, col);
        ECASQ_LAUNCH_CHECK();
        std::swap(a, b);
    }
    *last = a;
    return ECASQ_OK;
}

static int bwd_layers(const Prefix &P, double *r0, double *r1, int64_t v, int64_t c_lo, int t, double lam,
                      cudaStream_t st, double **last) {
    note_launch();
    k_lin_bwd2<<<(unsigned)cdiv(std::max<int64_t>(v - c_lo, 1), 256), 256, 0, st>>>(P, r0, v, c_lo, lam);
    ECASQ_LAUNCH_CHECK();
    double *a = r0, *b = r1;
    for (int r = 3; r <= t; r++) {
        const int64_t c_hi = v - r + 1;
        if (c_hi < c_lo) break;
        note_launch();
        k_lin_bwd<<<(unsigned)cdiv(c_hi - c_lo + 1, 8), 256, 0, st>>>(P, a, b, v, r, c_lo, c_hi, lam);
        ECASQ_LAUNCH_CHECK();
        std::swap(a, b);
    }
    *last = a;
    return ECASQ_OK;
}

// rows: 4 device rows of at least p doubles; col: s + 1 doubles; small: 2 int64 + 1 int32 +
// 1 double of device scratch.  qidx_host receives the codebook (m entries), *m_out, *best.
int launch_dp_linear(const Prefix &P, double lam, int s, int exact_s, double *rows, double *col, void *small,
                     std::vector<int32_t> &qidx_host, int *m_out, double *best, cudaStream_t st) {
    const int64_t p = P.p;
    double *R0 = rows, *R1 = rows + p, *R2 = rows + 2 * p, *R3 = rows + 3 * p;
    int64_t *split = reinterpret_cast<int64_t *>(small);
    int32_t *md = reinterpret_cast<int32_t *>(split + 2);
    double *bd = reinterpret_cast<double *>(split + 3);
    if (p == 1) {
        qidx_host.assign(1, 0);
        *m_out = 1;
        *best = 0.0;
        return ECASQ_OK;
    }
    // 1. forward pass over every layer: dp(i, p-1) -> col, then eq. apx_final
    {
        double *last;
        int rc = fwd_layers(P, R0, R1, 0, p - 1, s, lam, col, st, &last);
        if (rc) return rc;
    }
    note_launch();
    k_lin_pick<<<1, 32, 0, st>>>(col, s, exact_s, p, md, bd);
    ECASQ_LAUNCH_CHECK();
    int32_t m = 0;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(&m, md, sizeof(m), cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(best, bd, sizeof(double), cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    if (m < 2) return ECASQ_EINFEASIBLE;
    // 2. split subproblems (u, v, n) at their middle values
    qidx_host.assign(m, -1);
    qidx_host[0] = 0;
    qidx_host[m - 1] = (int32_t)(p - 1);
    struct Sub { int64_t u, v; int n, pos; };
    std::vector<Sub> stack{{0, p - 1, m, 0}};
    while (!stack.empty()) {
        const Sub q = stack.back();
        stack.pop_back();
        if (q.n <= 2) continue;
        const int t = (q.n + 1) / 2;
        double *G, *B;
        int rc = fwd_layers(P, R0, R1, q.u, q.v - 1, t, lam, nullptr, st, &G);
        if (rc) return rc;
        rc = bwd_layers(P, R2, R3, q.v, q.u + 1, q.n - t + 1, lam, st, &B);
        if (rc) return rc;
        // G_t is valid from u + t - 1, B_{n-t+1} up to v - n + t
        const int64_t c_lo = q.u + t - 1, c_hi = q.v - q.n + t;
        if (c_lo > c_hi) return ECASQ_EINFEASIBLE;
        note_launch();
        k_lin_split<<<1, 1024, 0, st>>>(G, B, c_lo, c_hi, split);
        ECASQ_LAUNCH_CHECK();
        int64_t c = -1;
        ECASQ_CUDA_TRY(cudaMemcpyAsync(&c, split, sizeof(c), cudaMemcpyDeviceToHost, st));
        ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
        if (c < 0) return ECASQ_EINFEASIBLE;
        qidx_host[q.pos + t - 1] = (int32_t)c;
        stack.push_back({q.u, c, t, q.pos});
        stack.push_back({c, q.v, q.n - t + 1, q.pos + t - 1});
    }
    *m_out = m;
    return ECASQ_OK;
}

}  // namespace ecasq
