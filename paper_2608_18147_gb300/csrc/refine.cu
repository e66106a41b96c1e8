// refine.cu -- one colour step of the three-colour refinement (Sec. 6).
//
// Block b moves the b-th value of the colour class: q_l with l % 3 == colour,
// 1 <= l <= m-2.  Its candidates are the unique input values strictly between
// its fixed neighbours; the local objective of Sec. 6 (true entropy reading) is
//   C[q_{l-1}, c] + C[c, q_{l+1}] + lambda' (h(f_{l-1}/d) + h(f_l/d) + h(f_{l+1}/d)),
// f_{l-1} = U[q_{l-2}, q_{l-1}] + D[q_{l-1}, c]   (n_{q_0} + D[q_0, c] when l-1 = 0),
// f_l     = U[q_{l-1}, c] + D[c, q_{l+1}],
// f_{l+1} = U[c, q_{l+1}] + D[q_{l+1}, q_{l+2}]   (U[c, q_{m-1}] when l+1 = m-1).
// Values of one class never share a frequency term, so all of them move at
// once (Sec. 6, Fig. 3).  Ties keep the current value, else the lowest index.
//
// The scan of q_l is a function of (q_{l-2}, q_{l-1}, q_l, q_{l+1}, q_{l+2}) alone (and of
// lambda', fixed in a call).  ctx[l] records that context whenever a scan kept q_l
// where it was; while the context is unchanged the scan would keep it again, so the
// value is not scanned (same result, no candidate evaluated).  A value that moved has
// no record (its move may still be undone by the caller).
#include "common.cuh"

namespace ecasq {

constexpr int kCtx = 6;  // q_{l-2}, q_{l-1}, q_l, q_{l+1}, q_{l+2} (-1 past the ends), valid

__device__ __forceinline__ void context_of(const int32_t *a, int m, int l, int32_t c[5]) {
    c[0] = l >= 2 ? a[l - 2] : -1;
    c[1] = a[l - 1];
    c[2] = a[l];
    c[3] = a[l + 1];
    c[4] = l + 2 <= m - 1 ? a[l + 2] : -1;
}
__device__ __forceinline__ bool context_unchanged(const int32_t *a, int m, int l, const int32_t *ctx) {
    const int32_t *r = ctx + kCtx * l;
    if (!r[5]) return false;
    int32_t c[5];
    context_of(a, m, l, c);
    return c[0] == r[0] && c[1] == r[1] && c[2] == r[2] && c[3] == r[3] && c[4] == r[4];
}

struct Nbr {
    int64_t L, R, cur, a0;
    double Ux, Dx;   // outer neighbours' fixed halves of f_{l-1} and f_{l+1}
    int firstL, lastR;
};

__device__ __forceinline__ double local_obj(const Prefix &P, const Nbr &n, int64_t c, double lamp) {
    double dd_ = (double)P.d;
    double C1, U1, D1, C2, U2, D2;
    pair_exact(P, n.L, c, C1, U1, D1);
    pair_exact(P, c, n.R, C2, U2, D2);
    double fl = n.firstL ? __dadd_rn((double)P.w[n.a0], D1) : __dadd_rn(n.Ux, D1);
    double fm = __dadd_rn(U1, D2);
    double fr = n.lastR ? U2 : __dadd_rn(U2, n.Dx);
    double ent = __dadd_rn(__dadd_rn(hfun(__ddiv_rn(fl, dd_)), hfun(__ddiv_rn(fm, dd_))), hfun(__ddiv_rn(fr, dd_)));
    return __dadd_rn(__dadd_rn(C1, C2), __dmul_rn(lamp, ent));
}

constexpr int kRefineChunk = 256;   // candidates per block: one per thread, so a value's range spreads over many SMs

__device__ __forceinline__ Nbr make_nbr(const Prefix &P, const int32_t *a, int m, int l) {
    Nbr n;
    n.L = a[l - 1]; n.R = a[l + 1]; n.cur = a[l]; n.a0 = a[0];
    n.firstL = (l - 1 == 0); n.lastR = (l + 1 == m - 1);
    double C, U, D;
    n.Ux = 0.0; n.Dx = 0.0;
    if (!n.firstL) { pair_exact(P, a[l - 2], n.L, C, U, D); n.Ux = U; }
    if (!n.lastR) { pair_exact(P, n.R, a[l + 2], C, U, D); n.Dx = D; }
    return n;
}

// Block (chunk, b): the b-th value of the colour class, candidates
// L+1+chunk*kRefineChunk .. (excluding the current position); the best
// (value, lowest index) of the chunk goes to part[b * nchunk + chunk], and the
// objective at the current position to curval[b].
struct RefPart { double v; int64_t i; };
constexpr int kRefineValues = kMaxS / 3 + 1;  // values of one colour class, at most

__global__ void __launch_bounds__(256) k_refine_chunks(Prefix P, const int32_t *a, int m, int colour, double lamp,
                                                       RefPart *part, double *curval, int nchunk,
                                                       const int32_t *ctx) {
    __shared__ Nbr nb;
    __shared__ double rv[256];
    __shared__ int64_t ri[256];
    int l0 = colour == 0 ? 3 : colour;
    int l = l0 + 3 * blockIdx.y;
    if (l > m - 2) return;
    int64_t lo = (int64_t)a[l - 1] + 1 + (int64_t)blockIdx.x * kRefineChunk;
    int64_t hi = min((int64_t)a[l + 1], lo + kRefineChunk);
    if (lo >= hi || context_unchanged(a, m, l, ctx)) return;  // uniform over the block
    if (threadIdx.x == 0) nb = make_nbr(P, a, m, l);
    __syncthreads();
    Nbr n = nb;
    double bv = CUDART_INF;
    int64_t bi = -1;
    for (int64_t c = lo + threadIdx.x; c < hi; c += blockDim.x) {
        double v = local_obj(P, n, c, lamp);
        if (c == n.cur) { curval[blockIdx.y] = v; continue; }
        if (v < bv) { bv = v; bi = c; }  // c ascends per thread: keeps the lowest
    }
    rv[threadIdx.x] = bv; ri[threadIdx.x] = bi;
    __syncthreads();
    for (int o = 128; o > 0; o >>= 1) {
        if (threadIdx.x < o) {
            double v2 = rv[threadIdx.x + o];
            int64_t i2 = ri[threadIdx.x + o];
            if (v2 < rv[threadIdx.x] || (v2 == rv[threadIdx.x] && i2 >= 0 && (ri[threadIdx.x] < 0 || i2 < ri[threadIdx.x]))) {
                rv[threadIdx.x] = v2; ri[threadIdx.x] = i2;
            }
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) part[(size_t)blockIdx.y * nchunk + blockIdx.x] = {rv[0], ri[0]};
}

// One warp per moved value: best over the chunks (lowest index among equal
// values), then keep the current position unless the best is strictly lower.
__global__ void k_refine_pick(const int32_t *a, int m, int colour, const RefPart *part, const double *curval,
                              int nchunk, int32_t *a_new, int32_t *moved, int32_t *ctx) {
    int l0 = colour == 0 ? 3 : colour;
    int l = l0 + 3 * blockIdx.x;
    if (l > m - 2) return;
    if (context_unchanged(a, m, l, ctx)) return;  // a_new[l] == a[l] already
    int64_t range = (int64_t)a[l + 1] - (int64_t)a[l - 1] - 1;
    int nc = (int)cdiv(range, kRefineChunk);
    double bv = CUDART_INF;
    int64_t bi = -1;
    for (int c = threadIdx.x; c < nc; c += 32) {
        RefPart q = part[(size_t)blockIdx.x * nchunk + c];
        if (q.i >= 0 && (q.v < bv || (q.v == bv && q.i < bi))) { bv = q.v; bi = q.i; }
    }
    for (int o = 16; o > 0; o >>= 1) {
        double v2 = __shfl_down_sync(0xffffffffu, bv, o);
        int64_t i2 = __shfl_down_sync(0xffffffffu, bi, o);
        if (i2 >= 0 && (bi < 0 || v2 < bv || (v2 == bv && i2 < bi))) { bv = v2; bi = i2; }
    }
    if (threadIdx.x == 0) {
        const int64_t cur = a[l];
        const double vc = curval[blockIdx.x];  // local_obj at the current position (k_refine_chunks)
        int64_t nw = (bi >= 0 && bv < vc) ? bi : cur;
        a_new[l] = (int32_t)nw;
        if (nw != cur) atomicExch(moved, 1);
        int32_t *r = ctx + kCtx * l;
        if (nw == cur) {
            int32_t c[5];
            context_of(a, m, l, c);
            for (int q = 0; q < 5; q++) r[q] = c[q];
            r[5] = 1;
        } else {
            r[5] = 0;
        }
    }
}

// After a colour step: the step's codebook replaces the current one unless no value moved,
// or (with the guard) its H(Xhat), ev[2] from the gated evaluation, exceeds the budget
// (Sec. 6).  On the device, so that a refinement round needs no host round trip until
// its stop test.
// A value that moved went to the lowest-index minimiser of its local objective, which does
// not depend on the value itself, only on its four neighbours (other colours: they did not
// move in this step); a scan in its new context would keep it there, so a kept step gives
// it the record such a scan writes, and the next round does not scan it again unless a
// neighbour moves.
__global__ void k_refine_commit(int32_t *a, const int32_t *a_new, const int32_t *moved, const double *ev, int m,
                                int guard, double budget, int32_t *ctx) {
    if (!*moved) return;
    if (guard && ev[2] > budget) return;
    for (int l = threadIdx.x; l < m; l += blockDim.x) {
        if (a_new[l] == a[l]) continue;
        int32_t c[5];
        context_of(a_new, m, l, c);
        int32_t *r = ctx + kCtx * l;
        for (int q = 0; q < 5; q++) r[q] = c[q];
        r[5] = 1;
    }
    __syncwarp();  // every comparison with the old codebook is done
    for (int t = threadIdx.x; t < m; t += blockDim.x) a[t] = a_new[t];
}

int launch_refine_commit(int32_t *a, const int32_t *a_new, const int32_t *moved, const double *ev, int m, bool guard,
                         double budget, int32_t *ctx, cudaStream_t st) {
    note_launch();
    k_refine_commit<<<1, 32, 0, st>>>(a, a_new, moved, ev, m, guard ? 1 : 0, budget, ctx);
    ECASQ_LAUNCH_CHECK();
    return ECASQ_OK;
}

size_t refine_scratch_bytes(int64_t d) {
    return sizeof(double) * kRefineValues + sizeof(RefPart) * kRefineValues * (size_t)cdiv(d, kRefineChunk);
}

size_t refine_ctx_bytes() { return sizeof(int32_t) * kCtx * kMaxS; }

int launch_refine_colour(const Prefix &P, const int32_t *a, int m, int colour, double lamp, int32_t *a_new,
                         int32_t *moved, void *part_buf, int32_t *ctx, cudaStream_t st, int *nblocks_out) {
    int l0 = colour == 0 ? 3 : colour;
    int nblk = (m - 2 >= l0) ? (m - 2 - l0) / 3 + 1 : 0;
    *nblocks_out = nblk;
    if (nblk == 0) return ECASQ_OK;
    int nchunk = (int)cdiv(P.p, kRefineChunk);
    double *curval = reinterpret_cast<double *>(part_buf);  // then the chunks' partial results
    RefPart *part = reinterpret_cast<RefPart *>(curval + kRefineValues);
    note_launch();
    k_refine_chunks<<<dim3(nchunk, nblk), 256, 0, st>>>(P, a, m, colour, lamp, part, curval, nchunk, ctx);
    ECASQ_LAUNCH_CHECK();
    note_launch();
    k_refine_pick<<<nblk, 32, 0, st>>>(a, m, colour, part, curval, nchunk, a_new, moved, ctx);
    ECASQ_LAUNCH_CHECK();
    return ECASQ_OK;
}

}  // namespace ecasq
