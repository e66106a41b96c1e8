// dp_fast.cu -- fast approximate DP (Sec. 5, eqs. apx_base / apx_rec / apx_final).
//
// Three stages per DP pass, for up to 8 multipliers at once:
//
// 1. k_wavefront / k_wavefront_res: an fp32 filter over the whole (k, j)
//    triangle with every layer i = 3..s fused.  A persistent CTA owns a block of
//    64 columns j and sweeps 64-wide tiles of k in increasing order; the tile
//    k-block K may be used as soon as column block K has published all its
//    layers (a flag with release/acquire order, bounded waits).  The interval
//    costs C[k,j] and Phi[k,j] of a tile (App. E quantities rebuilt with
//    compensated fp32 recurrences that add one point at a time, all terms
//    non-negative, from a double-double anchor per tile and column) are either
//    computed by two producer warps next to the consumers (k_wavefront), or
//    computed once per call into a resident table (k_build_costs) and streamed
//    in with bulk copies (k_wavefront_res, ECASQ_RESIDENT_COSTS); the values are
//    bit-identical.  The consumer threads evaluate dp(i-1,k) + C + lambda' Phi
//    for their (layer, column, multiplier) outputs with packed f32x2 adds and
//    integer mins.  Per output the kernel keeps the fp32 minimum and up to two
//    runs of tiles whose minimum came within the certified error band of it.
// 2. k_need_layer (layers s down to 3): the outputs whose exact value the
//    answer depends on.  eq. apx_final needs dp(i, p-1) for every i; an output
//    resolved exactly needs the exact values of its band members in the layer
//    below.  For every needed output the kernel re-evaluates its listed tiles
//    (within the certified bound; bit-identically from the resident table), keeps the members k whose fp32 value lies within the
//    band (up to 8 inline, the count either way) and marks (i-1, k) needed.
//    With ECASQ_EXACT_TABLES every output is needed.
// 3. k_exact_small / k_exact_big (layers 3 up to s, over the lists the need
//    stage wrote; k_fill_unneeded first): re-score the members of every needed
//    output in binary64 with double-double interval costs (the reference
//    formulas) and take the lowest k among exact minima: dp64, bp.  Outputs
//    with more members re-scan their band's tiles in fp32 and re-score the
//    members they meet on the fly -- never a full binary64 scan.  Outputs not
//    needed keep their fp32 minimum (dp64 = m32, bp = -2).
//
// The fp32 band: with u = 2^-24, each fp32 candidate value carries a relative
// error of at most eps_i = max(eps_{i-1}, 24u) + 1.0001u (eps_2 = 1.0001u), so
// the exact argmin k* satisfies val32(k*) <= m32 (1 + eps_i)/(1 - eps_i) for
// ANY fp32 evaluation within that bound (the re-evaluations of stages 2 and 3
// need not be bit-identical to the wavefront's).  The 24u budget for one
// interval cost (about 21u used): column anchors within 2u (C: 4.5u) from a
// double-double corner and compensated scans of non-negative increments,
// compensated recurrences of non-negative point terms, correctly rounded
// reciprocal and products, and the documented error of __log2f (2^-22
// absolute on [0.5,2), 2 ulp elsewhere) amplified at most 2.44x through
// h(y) = -y log2 y for y <= 1/2; values y > 1/2 are evaluated through 1 - y
// computed from the complementary mass.  The exact stage re-checks
// |m32 - dp64| <= eps_i dp64 for every resolved output and counts violations.
#include <algorithm>

#include "common.cuh"

namespace ecasq {

int launch_dp_reference(const Prefix &P, const double *lamp, int G, int s, double *dp64, int32_t *bp,
                        cudaStream_t st);
void timer_begin(cudaStream_t st);
void timer_end(cudaStream_t st);

constexpr int BJ = 64;         // columns per block
constexpr int BK = 64;         // k per tile
constexpr int LPT = 7;         // layers per consumer thread
constexpr int JPT = 4;         // columns per consumer thread (stride 16)
constexpr int NJQ = BJ / JPT;  // 16 column groups
constexpr int NPROD = 64;      // producer threads: one per column of the block
constexpr int PSTR = BK + 4;   // padded row stride (floats) of the interval-cost buffers
constexpr int MAXCONS = 256;
constexpr int NMEM = 8;        // members kept inline per output
constexpr int64_t kMaxFastP = (int64_t)1 << 20;
constexpr uint32_t kSpinLimit = 1u << 26;
constexpr uint32_t kTestSpinLimit = 1u << 14;  // the ECASQ_TEST_STALL hook: about 10-20 ms of spinning
constexpr uint32_t kCopySpinLimit = 1u << 22;  // waits on bulk copies (microseconds when healthy)
constexpr int kMdpMax = 36;  // block-minimum row stride bound (s + 1 rounded up to 4): tile skipping for s <= 35
// Resident interval costs: per tile, C[64][PSTR] then Phi[64][PSTR] (the shared-memory layout).
constexpr int kCostHalfFloats = BJ * PSTR;
constexpr uint32_t kCostHalfBytes = (uint32_t)(kCostHalfFloats * sizeof(float));  // 17408, a multiple of 16
constexpr size_t kCostTileFloats = 2 * (size_t)kCostHalfFloats;

// Band of an output: up to two runs of tile indices K (< 2^14), tiles arriving in
// increasing K (the diagonal block, K = J, last).  Low word: run 1 as
// first << 16 | last; high word: run 2 the same way, 0 when absent (a second run
// starts at a tile >= 2).  A tile within the band extends run 1 when it follows
// run 1 directly and there is no run 2, else opens run 2, else extends run 2 to
// itself (the gap is then scanned too: a superset, never a miss).  A tile below
// the band restarts it: run 1 = [K, K], no run 2.
__device__ __forceinline__ void band_update(uint32_t &w1, uint32_t &w2, bool rst, bool app, uint32_t K,
                                            uint32_t KK) {
    const bool has2 = w2 != 0u;
    const bool ext1 = app && !has2 && ((w1 & 0xFFFFu) + 1u == K);
    const uint32_t n1 = ext1 ? ((w1 & 0xFFFF0000u) | K) : w1;
    const uint32_t n2 = (app && !ext1) ? (has2 ? ((w2 & 0xFFFF0000u) | K) : KK) : w2;
    w1 = rst ? KK : n1;
    w2 = rst ? 0u : n2;
}
__device__ __forceinline__ uint64_t band_pack(uint32_t w1, uint32_t w2) { return ((uint64_t)w2 << 32) | w1; }

// Fold the minimum c of tile K (>= +0, or +inf) into an output's running minimum
// bb and band: below bb - bb tau restarts the band, up to bb + bb tau joins it.
// Non-negative floats order like their bit patterns, so the tests are unsigned
// integer compares; bb = +inf makes bb - T a NaN, whose bits lie above every
// value, so the first tile restarts the band (an all-+inf tile too, harmlessly:
// outputs whose minimum stays +inf are never resolved).
__device__ __forceinline__ void band_fold(float c, float &bb, float tau, uint32_t &w1, uint32_t &w2, uint32_t K,
                                          uint32_t KK) {
    const float T = __fmul_rn(bb, tau);
    const uint32_t ci = __float_as_uint(c);
    const bool rst = ci < __float_as_uint(__fsub_rn(bb, T));
    const bool app = !rst && ci <= __float_as_uint(__fadd_rn(bb, T));
    band_update(w1, w2, rst, app, K, KK);
    bb = fminf(bb, c);
}

// Per-pass constants, copied once to device memory (kernels index them at run time).
struct FastParams {
    float tau[kMaxS + 1];  // per layer: band factor 2 eps_i / (1 - eps_i), with margin
    float eps[kMaxS + 1];  // per layer: eps_i
    float lam32[kMaxG];    // lambda'_g rounded to fp32
    double lam64[kMaxG];
};

struct FastArgs {
    const float *v;
    const float *wf;       // multiplicities as fp32 (exact below 2^24)
    const int64_t *N;
    const double *S, *S2;  // hi [p+1] | lo [p+1]
    int64_t p, d;
    int64_t ps;            // table row stride (multiple of 64)
    float invd;            // correctly rounded 1/d
    int G, s, lgc, Gc, nsplit, nJ, ncons;
    const FastParams *prm;
    float *dp32;           // tile-major fp32 copy of dp: see d32()
    uint64_t *band;        // [G][s+1][ps] tile runs per output
    int32_t *mcnt;         // [G][s+1][ps] band members
    int32_t *members;      // [G][s+1][ps][NMEM]
    uint8_t *need;         // [G][s+1][ps] output resolved exactly
    float *corner;         // [nJ(nJ-1)/2][8]: state of pair (64K+63, 64J), K < J (N, E, Ec, A, Ac, C, Cc)
    const float *costs;    // resident interval costs (tile (K, J) at J(J+1)/2 + K - tile_base), or null
    float2 *tsum;          // with costs: per tile, {min_k C, min_k Phi} of its 64 columns (the rows' padding)
    size_t tile_base;      // index of the first tile the costs hold: 0, or J0(J0+1)/2 for a band of blocks
    int J0, J1;            // the wavefront's column blocks [J0, J1): all of them, or one band (streamed costs)
    int32_t *lists;        // [s+1][2][G ps]: needed outputs of layer i (g << 24 | j); 0: <= NMEM members, 1: more
    int *list_cnt;         // [s+1][2]
    int32_t *wide;         // [G ps]: needed outputs of the layer being closed whose bands span more than
                           // kThreadTiles tiles (g << 24 | j), walked by a warp each (k_need_wide)
    int *wide_cnt;         // [s+1]
    float *mdp;            // [nJ][G][mdp_stride]: min over the block's 64 columns of dp32(g, i, .)
    int mdp_stride;        // s + 1 rounded up to a multiple of 4 (16-byte rows)
    int prune;             // skip tiles by the lower bound (resident or streamed costs)
    int stage_tiles;       // with prune: tiles per staged batch (32, or 16 off the parked diagonal)
    const float *seed;     // with prune: fp32 dp rows [nJ][s+1][64] of an earlier pass at a multiplier >= every
                           // multiplier of this one (upper bounds of this pass's fp32 minima), or null
    uint32_t spin_limit;   // flag waits give up after this many spins (kSpinLimit; lower in the test hook)
    int hold0;             // test hook: column block 0 is never published (its waiters time out)
    int split_pub;         // resident costs, two layer groups: blocks are published in two parts (below)
    int *done;             // [nsplit][nJ]: every row of the block is stored
    int *half;             // [nsplit][nJ]: rows 2..8 of the block are stored (split_pub)
    int *ticket;
    int *abort_flag;
    DevStatus *st;
};

// The fp32 copy of dp is stored tile-major, [column block][g][i][64], so that the
// rows (g, i = 2..s-1) one tile of k needs are one contiguous run per multiplier.
__device__ __forceinline__ size_t d32(const FastArgs &a, int g, int i, int64_t j) {
    return (((size_t)(j >> 6) * (size_t)a.G + (size_t)g) * (size_t)(a.s + 1) + (size_t)i) * BJ + (size_t)(j & 63);
}

__device__ __forceinline__ size_t oidx(const FastArgs &a, int g, int i, int64_t j) {
    return ((size_t)g * (size_t)(a.s + 1) + (size_t)i) * (size_t)a.ps + (size_t)j;
}

// ------------------------------------------------------------ named barriers
__device__ __forceinline__ void bar_sync(int id, int n) { asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory"); }
__device__ __forceinline__ void bar_arrive(int id, int n) { asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(n) : "memory"); }
enum { BAR_FULL = 1, BAR_EMPTY = 3, BAR_CONS = 5, BAR_PROD = 6 };

// ------------------------------------------------------------ fp32 numerics

// Sum2 step (Ogita, Rump, Oishi 2005): x + c carries the running sum of
// non-negative terms; TwoSum keeps the rounding error of each addition.
__device__ __forceinline__ void comp_add(float &x, float &c, float t) {
    float s = __fadd_rn(x, t);
    float bb = __fsub_rn(s, x);
    float e = __fadd_rn(__fsub_rn(x, __fsub_rn(s, bb)), __fsub_rn(t, bb));
    x = s;
    c = __fadd_rn(c, e);
}

// Reciprocal from rcp.approx plus one Newton step: relative error <= u/2 + 2^-46
// (no slow-path branch, unlike the IEEE-rounded intrinsic).
__device__ __forceinline__ float rcp_nr(float x) {
    float r;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
    float e = __fmaf_rn(-x, r, 1.0f);
    return __fmaf_rn(r, e, r);
}

// -log2(1 - z) for z in [0, 1/2], from log(1 - z) = -2 atanh(z / (2 - z)).
__device__ __forceinline__ float neg_log2_1m(float z) {
    float t = __fmul_rn(z, rcp_nr(__fsub_rn(2.0f, z)));  // t in [0, 1/3]
    float t2 = __fmul_rn(t, t);
    // 2 (t + t^3/3 + ... + t^15/15) / ln 2; the next term is below 2^-26 t
    float q = 1.0f / 15.0f;
    q = __fmaf_rn(q, t2, 1.0f / 13.0f);
    q = __fmaf_rn(q, t2, 1.0f / 11.0f);
    q = __fmaf_rn(q, t2, 1.0f / 9.0f);
    q = __fmaf_rn(q, t2, 1.0f / 7.0f);
    q = __fmaf_rn(q, t2, 1.0f / 5.0f);
    q = __fmaf_rn(q, t2, 1.0f / 3.0f);
    q = __fmaf_rn(q, t2, 1.0f);
    return __fmul_rn(__fmul_rn(t, q), 2.8853900817779268f);  // 2 / ln 2
}

// h(y) = -y log2 y for y in [0, 1/2] (y = 0 gives 0), without branches.
__device__ __forceinline__ float h32_small(float y) {
    float r = __fmul_rn(y, -__log2f(fmaxf(y, 1e-37f)));
    return (y > 0.0f) ? fmaxf(r, 0.0f) : 0.0f;
}
// h(y) for y in [0, 1], `comp` = 1 - y computed from the complementary mass.  The
// series for y > 1/2 is a branch: only intervals holding more than half of all entries
// reach it, and a warp whose lanes have none skips it.
__device__ __forceinline__ float h32_any(float y, float comp) {
    float l = -__log2f(fmaxf(y, 1e-37f));
    if (y > 0.5f) l = neg_log2_1m(fminf(fmaxf(comp, 0.0f), 0.5f));
    float r = __fmul_rn(y, l);
    return (y > 0.0f) ? fmaxf(r, 0.0f) : 0.0f;
}

// Recurrence state of one column j while k descends: N = sum w, E = sum w (v_j - v_t),
// A = sum w (v_t - v_k), C = sum w (v_j - v_t)(v_t - v_k) over t in (k, j].
struct Rec {
    float N, E, Ec, A, Ac, C, Cc;
};

// Interval cost of (k, j) from the state: C and Phi = h(U/d) + h(D/d) (Sec. 5).
// At most one of U, D exceeds d/2 (U + D <= d), so only the larger mass needs
// the 1 - y form.
__device__ __forceinline__ void rec_emit(const Rec &r, float vj, float vk, float d_f, float invd, float &Cout,
                                         float &Phi) {
    float Eu = __fadd_rn(r.E, r.Ec), Au = __fadd_rn(r.A, r.Ac);
    Cout = __fadd_rn(fmaxf(__fadd_rn(r.C, r.Cc), 0.0f), 0.0f);  // >= +0 (no -0)
    float L = __fsub_rn(vj, vk);
    float rL = rcp_nr(L);
    float D = __fmul_rn(Eu, rL), U = __fmul_rn(Au, rL);
    float mbig = fmaxf(U, D), msmall = fminf(U, D);
    float out = __fsub_rn(d_f, r.N);  // mass outside the interval (exact)
    float comp = __fmul_rn(__fadd_rn(out, msmall), invd);
    Phi = __fadd_rn(__fadd_rn(h32_small(__fmul_rn(msmall, invd)), h32_any(__fmul_rn(mbig, invd), comp)), 0.0f);
}

// Add point t = k+1 (moving from k+1 to k): vt = v_{k+1}, wt = w_{k+1}, dk = v_{k+1} - v_k.
__device__ __forceinline__ void rec_step(Rec &r, float vj, float vt, float wt, float dk) {
    r.N = __fadd_rn(r.N, wt);
    comp_add(r.E, r.Ec, __fmul_rn(wt, __fsub_rn(vj, vt)));
    float Eu = __fadd_rn(r.E, r.Ec);
    comp_add(r.A, r.Ac, __fmul_rn(dk, r.N));
    comp_add(r.C, r.Cc, __fmul_rn(dk, Eu));
}

// Anchor of a tile: the state of pair (k, j) from double-double prefix sums.
__device__ __forceinline__ void split_f(dd x, float &hi, float &lo) {
    double t = dd_round(x);
    hi = __double2float_rn(t);
    lo = __double2float_rn(__dadd_rn(__dsub_rn(x.hi, (double)hi), x.lo));
}

__device__ void rec_anchor(const FastArgs &a, int64_t k, int64_t j, Rec &r) {
    int64_t n = a.N[j + 1] - a.N[k + 1];
    double nd = (double)n;
    dd dS = dd_sub(load_dd(a.S, a.p, j + 1), load_dd(a.S, a.p, k + 1));
    dd dS2 = dd_sub(load_dd(a.S2, a.p, j + 1), load_dd(a.S2, a.p, k + 1));
    double vk = (double)a.v[k], vj = (double)a.v[j];
    dd A = dd_sub(dS, two_prod(vk, nd));
    dd E = dd_sub(two_prod(vj, nd), dS);
    dd Cd = dd_sub(dd_sub(dd_mul(two_sum(vk, vj), dS), dS2), two_prod(__dmul_rn(vk, vj), nd));
    r.N = (float)n;
    split_f(E, r.E, r.Ec);
    split_f(A, r.A, r.Ac);
    split_f(Cd, r.C, r.Cc);
}

__device__ __forceinline__ size_t corner_idx(int64_t K, int64_t J) { return (size_t)J * (size_t)(J - 1) / 2 + (size_t)K; }

// Corner states (double-double, rounded to fp32 pairs) for every tile below the
// diagonal: pair (k, j) = (64K + 63, 64J), K < J.
__global__ void k_corners(FastArgs a) {
    int64_t n = (int64_t)a.nJ * (a.nJ - 1) / 2;
    int64_t id = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (; id < n; id += stride) {
        // invert id = J(J-1)/2 + K
        int64_t J = (int64_t)((1.0 + sqrt(1.0 + 8.0 * (double)id)) * 0.5);
        while (J * (J - 1) / 2 > id) J--;
        while ((J + 1) * J / 2 <= id) J++;
        int64_t K = id - J * (J - 1) / 2;
        Rec r;
        rec_anchor(a, K * BK + BK - 1, J * BJ, r);
        float *o = a.corner + 8 * (size_t)id;
        o[0] = r.N; o[1] = r.E; o[2] = r.Ec; o[3] = r.A; o[4] = r.Ac; o[5] = r.C; o[6] = r.Cc; o[7] = 0.f;
    }
}

// Compensated (Sum2) exclusive scan over the 64 producer threads of (x, c) pairs.
__device__ __forceinline__ void pair_add(float &x, float &c, float y, float yc) {
    float s = __fadd_rn(x, y);
    float bb = __fsub_rn(s, x);
    float e = __fadd_rn(__fsub_rn(x, __fsub_rn(s, bb)), __fsub_rn(y, bb));
    x = s;
    c = __fadd_rn(__fadd_rn(c, yc), e);
}

__device__ void scan64_excl(float v, float &x_out, float &c_out, float (*wsum)[2]) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;  // producer threads 0..63
    float x = v, c = 0.f;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        float y = __shfl_up_sync(0xffffffffu, x, o), yc = __shfl_up_sync(0xffffffffu, c, o);
        if (lane >= o) pair_add(x, c, y, yc);
    }
    if (lane == 31) { wsum[wid][0] = x; wsum[wid][1] = c; }
    bar_sync(BAR_PROD, NPROD);
    if (wid == 1) pair_add(x, c, wsum[0][0], wsum[0][1]);
    // exclusive: shift by one
    float xe = __shfl_up_sync(0xffffffffu, x, 1), ce = __shfl_up_sync(0xffffffffu, c, 1);
    if (lane == 0) {
        if (wid == 0) { xe = 0.f; ce = 0.f; }
        else { xe = wsum[0][0]; ce = wsum[0][1]; }
    }
    x_out = xe;
    c_out = ce;
    bar_sync(BAR_PROD, NPROD);
}

__device__ __forceinline__ Rec rec_empty() { return {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f}; }

__device__ __forceinline__ int ld_acquire(const int *p) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_release(int *p, int v) {
    asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// packed fp32 pair arithmetic (sm_100+)
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rd;\n\tmov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\tmov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "mov.b64 rc, {%6, %7};\n\tfma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return d;
}
__device__ __forceinline__ float min3(float a, float b, float c) {
    float d;
    asm("min.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// ------------------------------------------- bulk copies (TMA engine) and mbarriers
__device__ __forceinline__ uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void mbar_init(unsigned long long *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_fence_init() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }
// arrive once and raise the phase's expected transaction count by `bytes`
__device__ __forceinline__ void mbar_expect_tx(unsigned long long *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_test(unsigned long long *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait for phase `parity` of `bar`: on expiry record a timeout, raise the abort flag and return.
__device__ __forceinline__ void mbar_wait_bounded(unsigned long long *bar, uint32_t parity, DevStatus *st, int *abort_flag) {
    uint32_t spins = 0;
    while (!mbar_test(bar, parity)) {
        if (++spins > kCopySpinLimit) {
            st->timeout = 1;
            atomicExch(abort_flag, 1);
            return;
        }
        __nanosleep(32);
    }
}
__device__ __forceinline__ uint64_t policy_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}
// global -> shared, completion counted on `bar` (bytes and both addresses multiples of 16)
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, unsigned long long *bar,
                                         uint64_t policy) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
            smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
        : "memory");
}
// shared -> global, bulk-group completion
__device__ __forceinline__ void bulk_s2g(void *dst, const void *src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(smem_u32(src)), "r"(bytes)
                 : "memory");
}
// global -> shared without a cache hint (rows every later block reads again)
__device__ __forceinline__ void bulk_g2s_nohint(void *dst, const void *src, uint32_t bytes, unsigned long long *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     smem_u32(dst)),
                 "l"(src), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}
// global writes seen through generic loads/acquire -> ordered before later bulk copies
__device__ __forceinline__ void fence_proxy_async_global() { asm volatile("fence.proxy.async.global;" ::: "memory"); }
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read_all() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// generic-proxy writes to shared memory -> visible to later bulk copies
__device__ __forceinline__ void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__host__ __device__ __forceinline__ size_t cost_tile_idx(int64_t K, int64_t J) {
    return (size_t)J * (size_t)(J + 1) / 2 + (size_t)K;
}

// ------------------------------------------------------------ shared memory
struct TileMeta {
    int J, K, split, kind;  // kind: 0 off-diagonal, 1 diagonal, 2 stop
};

struct __align__(16) Smem {
    float C[2][BJ][PSTR];
    float Phi[2][BJ][PSTR];
    float diag[2][kMaxG][BJ];             // dp32 of the previous / current layer inside the column
    float kv[BK], kw[BK], kd[BK];         // v_k (k0..k0+63), w_{k+1}, v_{k+1} - v_k
    TileMeta meta[2];
    float wsum[2][2];                     // producer scan: per-warp totals
    int ticket;
    int sfront[2];                        // resident costs: frontier of the minima in stage buffer sb
    int pad;
    uint32_t needw[2][MAXCONS / 32];      // resident costs: per warp, the tiles of the batch it needs
    unsigned long long mbar[2];           // resident costs: bulk-copy completion of buffer b
    unsigned long long smbar[2];          // resident costs: completion of stage buffer sb
    float tau[kMaxS + 1];                 // FastParams::tau and lam32, read on every tile
    float lam32[kMaxG];
    // staged dp32 block minima of a tile's column block (tile skipping): the split's
    // multipliers' rows of a.mdp_stride floats each, flat (up to kMaxG x 20 floats)
    __align__(16) float mdp[2][kMaxG][20];
    // followed by dp32 slices [2][Gc * (s-2)][BK] (dynamic)
};

// ------------------------------------------------------- one tile of interval costs
// Per-k constants of the tile starting at k0 (k = k0 + jl): v_k, w_{k+1}, v_{k+1} - v_k.
__device__ __forceinline__ void tile_consts(const FastArgs &a, int64_t k0, int jl, float *kv, float *kw, float *kd) {
    int64_t k = k0 + jl;
    kv[jl] = k < a.p ? a.v[k] : 0.f;
    kw[jl] = (k + 1 < a.p) ? a.wf[k + 1] : 0.f;
    kd[jl] = (k + 1 < a.p) ? __fsub_rn(a.v[k + 1], a.v[k]) : 0.f;
}

// Global inputs of column jl of tile (K, J), loaded by one of the 64 threads: the tile
// constants of k = 64K + jl (v_k, w_{k+1}, v_{k+1} - v_k), the column's increment
// (w_{jt+1}, v_{jt+1}, v_jt, jt = 64J + jl) and v_j, and off the diagonal the corner
// state of (K, J).
struct TileIn {
    float kv, kw, kd;
    float wn, vn, vt, vj;
    float c[7];
};
__device__ __forceinline__ void tile_load_consts(const FastArgs &a, int64_t K, int jl, TileIn &q) {
    const int64_t k = K * BK + jl;
    q.kv = k < a.p ? a.v[k] : 0.f;
    q.kw = (k + 1 < a.p) ? a.wf[k + 1] : 0.f;
    q.kd = (k + 1 < a.p) ? __fsub_rn(a.v[k + 1], a.v[k]) : 0.f;
}
__device__ __forceinline__ void tile_load(const FastArgs &a, int64_t K, int64_t J, int jl, TileIn &q) {
    const int64_t jt = J * BJ + jl;
    const bool okc = jt + 1 < a.p;
    q.wn = okc ? a.wf[jt + 1] : 0.f;
    q.vn = okc ? a.v[jt + 1] : 0.f;
    q.vt = okc ? a.v[jt] : 0.f;
    q.vj = jt < a.p ? a.v[jt] : 0.f;
#pragma unroll
    for (int r = 0; r < 7; r++) q.c[r] = 0.f;
    if (K != J) {
        const float *cp = a.corner + 8 * corner_idx(K, J);
#pragma unroll
        for (int r = 0; r < 7; r++) q.c[r] = cp[r];
    }
}

// Anchor of column jl at k = 64K + 63 (off the diagonal): the corner state of (K, J)
// advanced along j with compensated exclusive scans of non-negative increments.
// Threads 0..63 of the block all call it (the scans synchronise them on BAR_PROD);
// vk = v at k = 64K + 63.
__device__ Rec tile_anchor(const TileIn &q, int64_t J, int jl, float vk, const FastArgs &a, float (*wsum)[2]) {
    const bool okc = J * BJ + jl + 1 < a.p;
    const float wn = q.wn, vn = q.vn;
    const float dj = okc ? __fsub_rn(vn, q.vt) : 0.f;
    const float *cp = q.c;
    float nx, nc, ax, ac, ex, ec, cx, cc;
    scan64_excl(wn, nx, nc, wsum);                               // N (exact)
    scan64_excl(okc ? __fmul_rn(wn, __fsub_rn(vn, vk)) : 0.f, ax, ac, wsum);  // A
    float Nj = __fadd_rn(cp[0], __fadd_rn(nx, nc));
    float Aj = __fadd_rn(__fadd_rn(cp[3], ax), __fadd_rn(cp[4], ac));
    scan64_excl(__fmul_rn(dj, Nj), ex, ec, wsum);              // E
    scan64_excl(__fmul_rn(dj, Aj), cx, cc, wsum);              // C
    Rec anchor_r;
    anchor_r.N = Nj;
    anchor_r.E = cp[1]; anchor_r.Ec = cp[2];
    pair_add(anchor_r.E, anchor_r.Ec, ex, ec);
    anchor_r.A = cp[3]; anchor_r.Ac = cp[4];
    pair_add(anchor_r.A, anchor_r.Ac, ax, ac);
    anchor_r.C = cp[5]; anchor_r.Cc = cp[6];
    pair_add(anchor_r.C, anchor_r.Cc, cx, cc);
    return anchor_r;
}

// Interval costs C[k, j] and Phi[k, j] of column j = 64J + jl for the 64 k of tile K
// (k descending) into Cr[jl][.] and Pr[jl][.]; +inf / 0 where k >= j or j >= p.
// anchor_r: the column's state at k = 64K + 63 (off the diagonal); vj = v_j.
__device__ void tile_rows(const FastArgs &a, int64_t K, int64_t J, int jl, const Rec &anchor_r, float vj,
                          const float *kv, const float *kw, const float *kd, float (*Cr)[PSTR], float (*Pr)[PSTR]) {
    const bool diag = (K == J);
    const int64_t j0 = J * BJ;
    const int64_t j = j0 + jl;
    const float d_f = (float)a.d;
        // interval costs of column j for k in the tile (descending k); the row's
        // padding slot BK receives min_k C and min_k Phi (lower bounds for tile skipping)
        float mc = CUDART_INF_F, mp = CUDART_INF_F;
        if (j < a.p) {
            Rec r;
            int kl_hi;
            if (diag) {
                r = rec_empty();
                kl_hi = (int)(j - j0) - 1;  // k = j-1 first
                // state for k = j: empty; step to k = j-1 adds t = j
                for (int kl = BK - 1; kl > kl_hi; kl--) { Cr[jl][kl] = CUDART_INF_F; Pr[jl][kl] = 0.f; }
                if (kl_hi < BK - 1) mp = 0.f;
                for (int kl = kl_hi; kl >= 0; kl--) {
                    rec_step(r, vj, kv[kl + 1], kw[kl], kd[kl]);  // kl + 1 <= 63
                    float c, ph;
                    rec_emit(r, vj, kv[kl], d_f, a.invd, c, ph);
                    Cr[jl][kl] = c; Pr[jl][kl] = ph;
                    mc = fminf(mc, c); mp = fminf(mp, ph);
                }
            } else {
                r = anchor_r;
                Rec nxt = r;
                for (int kl = BK - 1; kl >= 0; kl--) {
                    Rec cur = nxt;
                    if (kl > 0) rec_step(nxt, vj, kv[kl], kw[kl - 1], kd[kl - 1]);  // state of k - 1
                    float c, ph;
                    rec_emit(cur, vj, kv[kl], d_f, a.invd, c, ph);
                    Cr[jl][kl] = c; Pr[jl][kl] = ph;
                    mc = fminf(mc, c); mp = fminf(mp, ph);
                }
            }
        } else {
            for (int kl = 0; kl < BK; kl++) { Cr[jl][kl] = CUDART_INF_F; Pr[jl][kl] = 0.f; }
            mp = 0.f;
        }
        Cr[jl][BK] = mc;
        Pr[jl][BK] = mp;
}

// tile_anchor and tile_rows for one tile (threads 0..63 of the block; kv, kw, kd hold
// the tile constants of tile K, visible to all 64).
__device__ void tile_columns(const FastArgs &a, int64_t K, int64_t J, int jl, const float *kv, const float *kw,
                             const float *kd, float (*wsum)[2], float (*Cr)[PSTR], float (*Pr)[PSTR]) {
    TileIn q;
    tile_load(a, K, J, jl, q);
    const Rec anchor_r = K == J ? rec_empty() : tile_anchor(q, J, jl, kv[BK - 1], a, wsum);
    tile_rows(a, K, J, jl, anchor_r, q.vj, kv, kw, kd, Cr, Pr);
}

// Resident interval costs: every tile (K <= J) computed once, exactly as the
// wavefront's own producer computes it (tile_anchor, tile_rows), staged in shared
// memory and written out by a bulk copy.  64 threads per block; blocks stride over
// the tiles.  A tile's global inputs are loaded while the previous tile's rows are
// computed, and the wait for the previous bulk store to have read the staging rows
// comes only just before they are overwritten.
struct __align__(16) BuildSmem {
    float C[BJ][PSTR];
    float Phi[BJ][PSTR];
    float kv[BK], kw[BK], kd[BK];
    float wsum[2][2];
};

__global__ void __launch_bounds__(NPROD) k_build_costs(FastArgs a, float *costs) {
    __shared__ BuildSmem S;
    const int jl = threadIdx.x;
    // the tiles of column blocks [J0, J1): indices J0(J0+1)/2 .. J1(J1+1)/2 - 1, stored from tile_base
    const int64_t ntiles = (int64_t)a.J1 * (a.J1 + 1) / 2;
    int64_t t = (int64_t)a.tile_base + blockIdx.x;
    if (t >= ntiles) return;
    // invert t = J(J+1)/2 + K, K <= J
    int64_t J = (int64_t)((sqrt(8.0 * (double)t + 1.0) - 1.0) * 0.5);
    while (J * (J + 1) / 2 > t) J--;
    while ((J + 1) * (J + 2) / 2 <= t) J++;
    int64_t K = t - J * (J + 1) / 2;
    TileIn cur;
    tile_load_consts(a, K, jl, cur);
    tile_load(a, K, J, jl, cur);
    for (;;) {
        S.kv[jl] = cur.kv; S.kw[jl] = cur.kw; S.kd[jl] = cur.kd;
        bar_sync(BAR_PROD, NPROD);
        const Rec anchor_r = K == J ? rec_empty() : tile_anchor(cur, J, jl, S.kv[BK - 1], a, S.wsum);
        // the next tile of this block: t + gridDim.x, walking (J, K) along the rows
        const int64_t tn = t + gridDim.x;
        int64_t Jn = J, Kn = K + gridDim.x;
        while (Kn > Jn) { Kn -= Jn + 1; Jn++; }
        TileIn nxt;
        if (tn < ntiles) {
            tile_load_consts(a, Kn, jl, nxt);
            tile_load(a, Kn, Jn, jl, nxt);
        }
        if (jl == 0) bulk_wait_read_all();  // the previous tile's bulk store has read the rows
        bar_sync(BAR_PROD, NPROD);
        tile_rows(a, K, J, jl, anchor_r, cur.vj, S.kv, S.kw, S.kd, S.C, S.Phi);
        a.tsum[((size_t)t - a.tile_base) * BJ + jl] = make_float2(S.C[jl][BK], S.Phi[jl][BK]);  // this thread's own row
        fence_proxy_async_smem();
        bar_sync(BAR_PROD, NPROD);
        if (jl == 0) {
            float *dst = costs + ((size_t)t - a.tile_base) * kCostTileFloats;
            bulk_s2g(dst, &S.C[0][0], kCostHalfBytes);
            bulk_s2g(dst + kCostHalfFloats, &S.Phi[0][0], kCostHalfBytes);
            bulk_commit();
        }
        if (tn >= ntiles) break;
        t = tn; J = Jn; K = Kn;
        cur = nxt;
    }
    if (jl == 0) bulk_wait_all();
}

// ------------------------------------------------------------ consumer side
// A consumer thread owns the outputs (g = split * Gc + gl, layers 3 + lg * LPT + l,
// columns jq + 16 q of the block) and keeps their band state in registers.
struct ConsId {
    int ct, jq, lg, gl;
    bool active;
};
__device__ __forceinline__ ConsId cons_id(const FastArgs &a, int ct) {
    ConsId id;
    id.ct = ct;
    id.jq = ct % NJQ;
    const int rest = ct / NJQ;
    id.lg = rest % a.lgc;
    id.gl = rest / a.lgc;
    id.active = ct < a.Gc * a.lgc * NJQ;
    return id;
}

// The outputs a consumer thread owns: LP layers x JPT columns (LP = LPT, or 8 for the
// generic path of the resident kernel at larger s: see launch_dp_fast).
template <int LP>
struct ConsStateT {
    float best[LP][JPT];
    uint32_t w1[LP][JPT], w2[LP][JPT];  // band runs (band_update)
};
using ConsState = ConsStateT<LPT>;
template <int LP>
__device__ __forceinline__ void cons_reset(ConsStateT<LP> &cs) {
#pragma unroll
    for (int l = 0; l < LP; l++)
#pragma unroll
        for (int q = 0; q < JPT; q++) { cs.best[l][q] = CUDART_INF_F; cs.w1[l][q] = 0u; cs.w2[l][q] = 0u; }
}

// Seeded running minima of block J.  Every fp32 candidate is monotone in lambda' (C and
// Phi are >= 0 and the roundings are monotone), so by induction over the layers an
// earlier pass's fp32 minimum at a multiplier >= this one's bounds this pass's minimum
// m from above.  Starting the running minimum at that bound changes no result: the
// tile holding m is never skipped (its lower bound is <= m <= the limit), so the final
// minimum is m itself; a tile the tighter limit skips has every candidate above
// m (1 + tau), outside the band; and band_fold keeps the band a superset of the tiles
// with a candidate within m (1 + tau) from any starting bb >= m (a reset drops only
// tiles whose candidates all lie above the band).  The band words keep their reset
// state, run 1 = tile 0: a seeded output whose walk never resets its band keeps tile 0
// in it (a superset again; a run opened at tile 0 could not be told from no run).
// Only the skip tests see the seed: more tiles are skipped, the tables are unchanged.
template <int LP>
__device__ __forceinline__ void cons_seed(const FastArgs &a, ConsStateT<LP> &cs, int J, const ConsId &id) {
    const float *sr = a.seed + (size_t)J * (size_t)(a.s + 1) * BJ;
#pragma unroll
    for (int l = 0; l < LP; l++) {
        // rows past the last layer repeat the last one (cons_offdiag): so does their seed
        const int i = 3 + min(id.lg * LP + l, a.s - 3);
#pragma unroll
        for (int q = 0; q < JPT; q++) {
            const int jl = id.jq + NJQ * q;
            const float v = ((int64_t)J * BJ + jl < a.p) ? sr[(size_t)i * BJ + jl] : CUDART_INF_F;
            if (v < CUDART_INF_F) cs.best[l][q] = v;
        }
    }
}

// Off-diagonal tile K: the fp32 minimum over the tile's 64 k of every output the
// thread owns (g must be a real multiplier), folded into its band state.
// Candidate values are >= +0, so their bit patterns order like the floats: the
// running minimum is kept as int bits and updated with integer min (ALU pipe)
// next to the packed adds (FMA pipe).
// Returns false when the warp skipped the tile (see below).
template <int LP>
__device__ __forceinline__ bool cons_offdiag(const FastArgs &a, const Smem &S, const float *sDPb, int b, uint32_t K,
                                             int g, const ConsId &id, ConsStateT<LP> &cs) {
    const int L = a.s - 2;
    int cm[LP][JPT];
#pragma unroll
    for (int l = 0; l < LP; l++)
#pragma unroll
        for (int q = 0; q < JPT; q++) cm[l][q] = 0x7f800000;  // +inf
    const float *dpb = sDPb + (size_t)id.gl * L * BK;
    const float lam = S.lam32[g];
    const float2 lam2 = make_float2(lam, lam);
    int rowl[LP];
#pragma unroll
    for (int l = 0; l < LP; l++) rowl[l] = min(id.lg * LP + l, L - 1);
    if (a.prune) {
        // Exact tile skipping.  Every candidate of the tile for output (l, q) is
        // >= lb = fl(min dp(i-1, .) + fl(fma(lam, min Phi, min C))) (rounding is monotone);
        // when lb exceeds the output's band limit bb + bb tau, the tile changes neither
        // its minimum nor its band.  The warp skips when that holds for all its outputs.
        const float *md = &S.mdp[b][0][0] + (size_t)id.gl * a.mdp_stride + 2;
        float lbq[JPT];
#pragma unroll
        for (int q = 0; q < JPT; q++) {
            const int jl = id.jq + NJQ * q;
            lbq[q] = __fmaf_rn(lam, S.Phi[b][jl][BK], S.C[b][jl][BK]);
        }
        bool need = false;
#pragma unroll
        for (int l = 0; l < LP; l++) {
            const float m = md[rowl[l]], tau = S.tau[3 + rowl[l]];
#pragma unroll
            for (int q = 0; q < JPT; q++) {
                const float bb = cs.best[l][q];
                need |= __fadd_rn(m, lbq[q]) <= __fadd_rn(bb, __fmul_rn(bb, tau));
            }
        }
        if (!__any_sync(__activemask(), need)) return false;
    }
#pragma unroll 1
    for (int kk = 0; kk < BK; kk += 4) {
        float2 W[JPT][2];
#pragma unroll
        for (int q = 0; q < JPT; q++) {
            float4 c4 = *reinterpret_cast<const float4 *>(&S.C[b][id.jq + NJQ * q][kk]);
            float4 f4 = *reinterpret_cast<const float4 *>(&S.Phi[b][id.jq + NJQ * q][kk]);
            W[q][0] = fma2(lam2, make_float2(f4.x, f4.y), make_float2(c4.x, c4.y));
            W[q][1] = fma2(lam2, make_float2(f4.z, f4.w), make_float2(c4.z, c4.w));
        }
#pragma unroll
        for (int l = 0; l < LP; l++) {
            // layer i = 3 + li uses dp row 2 + li; rows past the last layer are
            // clamped (their results are never used)
            const float4 d4 = *reinterpret_cast<const float4 *>(dpb + (size_t)rowl[l] * BK + kk);
            float2 da = make_float2(d4.x, d4.y), db = make_float2(d4.z, d4.w);
#pragma unroll
            for (int q = 0; q < JPT; q++) {
                float2 t0 = add2(da, W[q][0]);
                float2 t1 = add2(db, W[q][1]);
                int c = min(min(cm[l][q], __float_as_int(t0.x)), __float_as_int(t0.y));
                cm[l][q] = min(min(c, __float_as_int(t1.x)), __float_as_int(t1.y));
            }
        }
    }
    // band bookkeeping (branch-free; layers past the last one carry state that is never read)
    const uint32_t KK = (K << 16) | K;
#pragma unroll
    for (int l = 0; l < LP; l++) {
        const float tau = S.tau[3 + rowl[l]];
#pragma unroll
        for (int q = 0; q < JPT; q++) band_fold(__int_as_float(cm[l][q]), cs.best[l][q], tau, cs.w1[l][q], cs.w2[l][q], K, KK);
    }
    return true;
}

// Diagonal block J (its tile in buffer b): layers in order, each needing the
// previous layer's values inside the block; dp32 and the band words of the block
// go to global memory.  The owner of an output computes its minimum over the
// block's 64 k; when a.lgc == 2 the partner lane (lane ^ 16: same multiplier and
// columns, the other layer group) takes half of the k range and the halves meet
// by a shuffle.  All `a.ncons` consumer threads take part (BAR_CONS).
// staged: S.diag[0] already holds layer 2 of the block (bulk copy), else it is
// loaded here.
template <int LP>
__device__ __forceinline__ void cons_diag(const FastArgs &a, Smem &S, int b, int J, int split, const ConsId &id,
                                          ConsStateT<LP> &cs, bool staged) {
    const int L = a.s - 2;
    const int ct = id.ct;
    const int g = split * a.Gc + id.gl;
    const bool own = id.active && g < a.G;
    const int64_t j0 = (int64_t)J * BJ;
    if (!staged) {
        for (int q = ct; q < a.Gc * BJ; q += a.ncons) {
            int gg = q / BJ, jj = q % BJ;
            int g2 = split * a.Gc + gg;
            int64_t jx = j0 + jj;
            S.diag[0][gg][jj] = (g2 < a.G && jx < a.p) ? a.dp32[d32(a, g2, 2, jx)] : CUDART_INF_F;
        }
        bar_sync(BAR_CONS, a.ncons);
    }
    const bool pair = a.lgc == 2;  // warp-uniform
    const float lam = own ? S.lam32[g] : 0.f;
    const float2 lam2 = make_float2(lam, lam);
    const uint32_t K = (uint32_t)J, KK = (K << 16) | K;
    int cur = 0;
    for (int li = 0; li < L; li++) {
        if (LP != LPT && a.prune) {
            // block minimum of the layer below (row 2 + li) for later blocks' skip tests, by the
            // warp of that index (values >= +0: integer min on the bits); with LPT layers per
            // thread, skipping runs on the paired diagonal only, which writes its own minima
            const int w = ct >> 5, wl = ct & 31;
            const int gw = split * a.Gc + w;
            if (w < a.Gc && gw < a.G) {
                const int v = min(__float_as_int(S.diag[cur][w][wl]), __float_as_int(S.diag[cur][w][wl + 32]));
                const int mn = __reduce_min_sync(0xffffffffu, v);
                if (wl == 0) a.mdp[((size_t)J * a.G + gw) * a.mdp_stride + 2 + li] = __int_as_float(mn);
            }
        }
        const int i = 3 + li;
        const int olg = li / LP, l = li - olg * LP;
        const bool owner = own && id.lg == olg;
        const int kbeg = (pair && !owner) ? BJ / 2 : 0;
        const int kend = (pair && owner) ? BJ / 2 : BJ;
        int m0[JPT], m1[JPT];
#pragma unroll
        for (int q = 0; q < JPT; q++) { m0[q] = 0x7f800000; m1[q] = 0x7f800000; }
        if (own && (owner || pair)) {
            const float *prow = &S.diag[cur][id.gl][0];
#pragma unroll 2
            for (int kk = kbeg; kk < kend; kk += 4) {
                const float4 d4 = *reinterpret_cast<const float4 *>(prow + kk);
#pragma unroll
                for (int q = 0; q < JPT; q++) {
                    const int jl = id.jq + NJQ * q;
                    float4 c4 = *reinterpret_cast<const float4 *>(&S.C[b][jl][kk]);
                    float4 f4 = *reinterpret_cast<const float4 *>(&S.Phi[b][jl][kk]);
                    float2 v0 = fma2(lam2, make_float2(f4.x, f4.y), make_float2(c4.x, c4.y));
                    float2 v1 = fma2(lam2, make_float2(f4.z, f4.w), make_float2(c4.z, c4.w));
                    float2 t0 = add2(make_float2(d4.x, d4.y), v0);
                    float2 t1 = add2(make_float2(d4.z, d4.w), v1);
                    m0[q] = min(min(m0[q], __float_as_int(t0.x)), __float_as_int(t0.y));
                    m1[q] = min(min(m1[q], __float_as_int(t1.x)), __float_as_int(t1.y));
                }
            }
        }
#pragma unroll
        for (int q = 0; q < JPT; q++) {
            m0[q] = min(m0[q], m1[q]);
            if (pair) m0[q] = min(m0[q], __shfl_xor_sync(0xffffffffu, m0[q], 16));
        }
        if (owner) {
#pragma unroll
            for (int lx = 0; lx < LP; lx++) {
                if (lx != l) continue;
#pragma unroll
                for (int q = 0; q < JPT; q++) {
                    const int jl = id.jq + NJQ * q;
                    const int64_t j = j0 + jl;
                    band_fold(__int_as_float(m0[q]), cs.best[lx][q], S.tau[i], cs.w1[lx][q], cs.w2[lx][q], K, KK);
                    const float bb = cs.best[lx][q];
                    S.diag[cur ^ 1][id.gl][jl] = bb;
                    if (j < a.p) {
                        a.dp32[d32(a, g, i, j)] = bb;
                        a.band[oidx(a, g, i, j)] = band_pack(cs.w1[lx][q], cs.w2[lx][q]);
                    }
                }
            }
        }
        bar_sync(BAR_CONS, a.ncons);
        cur ^= 1;
    }
}

// Diagonal block when a.lgc == 2 (the usual s <= 16).  Only pairs k < j of the tile
// count, so each lane takes two whole columns of its column group jq, balanced on the
// triangle: lanes 0-15 column jq + 48 (k < 64) and column jq (k < 16), lanes 16-31
// column jq + 32 (k < 48) and column jq + 16 (k < 32): 80 pairs each, in 20 groups of
// four consecutive k (kdiag_group).  The costs W = C + lambda' Phi of those pairs stay
// in registers for all layers, so each layer reads only the previous layer's 64 values
// from shared memory, and every column's minimum is complete within one lane (pairs
// k >= j carry C = +inf in the tile and never win).  The band state is parked in `park`
// ([3][LPT][JPT][ncons] words: best, run 1, run 2) and folded there; the block
// ends with its diagonal, so the registers are not restored.  A warp holds one
// multiplier, and the rows of S.diag and the parked slots it reads and writes are
// that multiplier's alone, so the layers need only a warp barrier each.
// Group g4 of a diagonal lane (half 0: lanes 0-15, half 1: lanes 16-31): its column
// (q = 0: the long one, 1: the short one) and first k.  Groups 0-11 are k 0..47 of the
// long column for both halves; groups 12-15 are k 48..63 of the long column (half 0)
// or k 0..15 of the short one (half 1); groups 16-19 are k 0..15 (half 0) or 16..31
// (half 1) of the short column.
constexpr int kDiagGroups = 20;
__device__ __forceinline__ void kdiag_group(int g4, int half, int &q, int &k) {
    if (g4 < 12) { q = 0; k = 4 * g4; }
    else if (g4 < 16) { q = half; k = half ? 4 * (g4 - 12) : 4 * g4; }
    else { q = 1; k = half ? 4 * (g4 - 12) : 4 * (g4 - 16); }
}

// cons_diag_pair in three steps, so that the block can be published in two parts
// (diag_prepare; diag_layers over a range of layers; diag_store over a range of rows).
// diag_prepare: park the band state, store the block minimum of layer 2, and build the
// lane's costs W = C + lambda' Phi of its 80 pairs (kept in registers for all layers).
__device__ __forceinline__ void diag_prepare(const FastArgs &a, Smem &S, uint32_t *park, int b, int J, int split,
                                             const ConsId &id, const ConsState &cs, float2 (&W)[2 * kDiagGroups]) {
    const int ct = id.ct, nc = a.ncons;
    const int g = split * a.Gc + id.gl;
    const bool own = id.active && g < a.G;  // uniform over a warp (one multiplier per warp)
    constexpr int NS = LPT * JPT;
#pragma unroll
    for (int l = 0; l < LPT; l++)
#pragma unroll
        for (int q = 0; q < JPT; q++) {
            const int x = (l * JPT + q) * nc + ct;
            park[x] = __float_as_uint(cs.best[l][q]);
            park[NS * nc + x] = cs.w1[l][q];
            park[2 * NS * nc + x] = cs.w2[l][q];
        }
    asm volatile("" ::: "memory");  // the state leaves the registers before W is built
    const int lane = ct & 31;
    if (a.prune && own) {  // block minimum of layer 2 (values are >= +0: integer min on the bits)
        int v = min(__float_as_int(S.diag[0][id.gl][lane]), __float_as_int(S.diag[0][id.gl][lane + 32]));
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(0xffffffffu, v, o));
        if (lane == 0) a.mdp[((size_t)J * a.G + g) * a.mdp_stride + 2] = __int_as_float(v);
    }
    const int half = (ct >> 4) & 1;
    const int qb = 3 - half, qs = half;  // the lane's long and short columns (q of jq + 16 q)
    const float lam = own ? S.lam32[g] : 0.f;
    const float2 lam2 = make_float2(lam, lam);
#pragma unroll
    for (int g4 = 0; g4 < kDiagGroups; g4++) {  // W[2 g4], W[2 g4 + 1]: costs of group g4's four pairs
        int q, k;
        kdiag_group(g4, half, q, k);
        const int jl = id.jq + NJQ * (q ? qs : qb);
        float4 c4 = *reinterpret_cast<const float4 *>(&S.C[b][jl][k]);
        float4 f4 = *reinterpret_cast<const float4 *>(&S.Phi[b][jl][k]);
        W[2 * g4] = fma2(lam2, make_float2(f4.x, f4.y), make_float2(c4.x, c4.y));
        W[2 * g4 + 1] = fma2(lam2, make_float2(f4.z, f4.w), make_float2(c4.z, c4.w));
    }
}

// Layers li0 <= li < li1 (i = 3 + li) of the diagonal block; cur: the S.diag row
// holding layer i - 1 (in/out).
__device__ __forceinline__ void diag_layers(const FastArgs &a, Smem &S, uint32_t *park, int J, int split,
                                            const ConsId &id, const float2 (&W)[2 * kDiagGroups], int li0, int li1,
                                            int &cur) {
    const int ct = id.ct, nc = a.ncons;
    const int g = split * a.Gc + id.gl;
    const bool own = id.active && g < a.G;
    constexpr int NS = LPT * JPT;
    const int half = (ct >> 4) & 1;
    const int qb = 3 - half, qs = half;
    const uint32_t K = (uint32_t)J, KK = (K << 16) | K;
    for (int li = li0; li < li1; li++) {
        const int i = 3 + li;
        const int olg = li / LPT, l = li - olg * LPT;
        // minima (float bits; candidates are >= +0) of the long and the short column:
        // each group of four k reduces on its own, then the groups by a tree, so the
        // layer's dependency chain is a few mins deep
        int lmin = 0x7f800000, smin = 0x7f800000;
        if (own) {
            const float *prow = &S.diag[cur][id.gl][0];
            int m[kDiagGroups];
#pragma unroll
            for (int g4 = 0; g4 < kDiagGroups; g4++) {
                int q, k;
                kdiag_group(g4, half, q, k);
                const float4 d4 = *reinterpret_cast<const float4 *>(prow + k);
                const float2 t0 = add2(make_float2(d4.x, d4.y), W[2 * g4]);
                const float2 t1 = add2(make_float2(d4.z, d4.w), W[2 * g4 + 1]);
                m[g4] = min(min(__float_as_int(t0.x), __float_as_int(t0.y)), min(__float_as_int(t1.x), __float_as_int(t1.y)));
            }
            // groups 0-11: the long column; 12-15: long (half 0) or short (half 1); 16-19: short
            const int A = min(min(min(min(m[0], m[1]), min(m[2], m[3])), min(min(m[4], m[5]), min(m[6], m[7]))),
                              min(min(m[8], m[9]), min(m[10], m[11])));
            const int B = min(min(m[12], m[13]), min(m[14], m[15]));
            const int C = min(min(m[16], m[17]), min(m[18], m[19]));
            lmin = half ? A : min(A, B);
            smin = half ? min(B, C) : C;
        }
        if (own) {
            // each lane folds its two columns into the owner's slots (layer group olg,
            // same column group: lane jq + 16 olg of the warp)
            const int cto = (ct & ~31) | (olg << 4) | id.jq;
#pragma unroll
            for (int c = 0; c < 2; c++) {
                const int q = c ? qs : qb;
                const int mq = c ? smin : lmin;
                const int jl = id.jq + NJQ * q;
                const int x = (l * JPT + q) * nc + cto;
                float bb = __uint_as_float(park[x]);
                uint32_t w1 = park[NS * nc + x], w2 = park[2 * NS * nc + x];
                band_fold(__int_as_float(mq), bb, S.tau[i], w1, w2, K, KK);
                park[x] = __float_as_uint(bb);
                park[NS * nc + x] = w1;
                park[2 * NS * nc + x] = w2;
                S.diag[cur ^ 1][id.gl][jl] = bb;
            }
        }
        __syncwarp();  // the layer's row and parked state belong to this warp alone
        cur ^= 1;
    }
}

// The block's final values of layers ilo <= i <= ihi from the parked state, and the
// block minimum of each of those layers (over the 64 columns a half-warp holds).
__device__ __forceinline__ void diag_store(const FastArgs &a, const uint32_t *park, int J, int split,
                                           const ConsId &id, int ilo, int ihi) {
    const int ct = id.ct, nc = a.ncons;
    const int g = split * a.Gc + id.gl;
    const bool own = id.active && g < a.G;
    const int64_t j0 = (int64_t)J * BJ;
    if (own) {
#pragma unroll
        for (int l = 0; l < LPT; l++) {
            const int i = 3 + id.lg * LPT + l;
            const bool real = i <= a.s && i >= ilo && i <= ihi;
            int v = 0x7f800000;
#pragma unroll
            for (int q = 0; q < JPT; q++) {
                const int64_t j = j0 + id.jq + NJQ * q;
                const int x = (l * JPT + q) * nc + ct;
                v = min(v, (int)park[x]);
                if (real && j < a.p) a.dp32[d32(a, g, i, j)] = __uint_as_float(park[x]);
            }
            if (a.prune) {
#pragma unroll
                for (int o = 8; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(0xffffffffu, v, o));
                if (real && id.jq == 0) a.mdp[((size_t)J * a.G + g) * a.mdp_stride + i] = __int_as_float(v);
            }
        }
    }
}

// The whole diagonal block at once (the block is then published in one part).
__device__ __forceinline__ void cons_diag_pair(const FastArgs &a, Smem &S, uint32_t *park, int b, int J, int split,
                                               const ConsId &id, ConsState &cs) {
    float2 W[2 * kDiagGroups];
    diag_prepare(a, S, park, b, J, split, id, cs, W);
    int cur = 0;
    diag_layers(a, S, park, J, split, id, W, 0, a.s - 2, cur);
    diag_store(a, park, J, split, id, 3, a.s);
}

// Split publish (resident costs, two layer groups).  The chain of blocks runs through the
// last off-diagonal tile (J-1, J) and the diagonal block J.  Block J-1 is published in
// two parts -- rows 2..8 (layer group 0's inputs) after its layer 8, every row at the
// end -- and block J takes tile (J-1, J) in the same two parts, so its layers 3..9
// start as soon as block J-1 has finished layer 8.
// cons_lasttile_grp: tile (J-1, J) for layer group grp (0: layers 3..9 from rows 2..8;
// 1: layers 10..s from rows 9..s-1) by all 32 lanes of the warp -- lane 16 h + jq takes
// columns jq + 16 q, q in {2h, 2h+1}, over the group's seven layers -- after which the
// owners (the lanes of layer group grp) fold the tile minima of their four columns
// into their parked band state.  There is no skip test: this tile is on the chain.
__device__ __forceinline__ void cons_lasttile_grp(const FastArgs &a, const Smem &S, const float *sDPb, int b,
                                                  uint32_t *park, uint32_t K, int g, const ConsId &id, int grp) {
    const int L = a.s - 2;
    const int ct = id.ct, nc = a.ncons;
    const int h = (ct >> 4) & 1;
    constexpr int NS = LPT * JPT;
    int cm[LPT][2];
#pragma unroll
    for (int l = 0; l < LPT; l++) { cm[l][0] = 0x7f800000; cm[l][1] = 0x7f800000; }
    const float *dpb = sDPb + (size_t)id.gl * L * BK;
    const float lam = S.lam32[g];
    const float2 lam2 = make_float2(lam, lam);
    int rowl[LPT];
#pragma unroll
    for (int l = 0; l < LPT; l++) rowl[l] = min(grp * LPT + l, L - 1);
#pragma unroll 1
    for (int kk = 0; kk < BK; kk += 4) {
        float2 W[2][2];
#pragma unroll
        for (int c = 0; c < 2; c++) {
            const int jl = id.jq + NJQ * (2 * h + c);
            const float4 c4 = *reinterpret_cast<const float4 *>(&S.C[b][jl][kk]);
            const float4 f4 = *reinterpret_cast<const float4 *>(&S.Phi[b][jl][kk]);
            W[c][0] = fma2(lam2, make_float2(f4.x, f4.y), make_float2(c4.x, c4.y));
            W[c][1] = fma2(lam2, make_float2(f4.z, f4.w), make_float2(c4.z, c4.w));
        }
#pragma unroll
        for (int l = 0; l < LPT; l++) {
            const float4 d4 = *reinterpret_cast<const float4 *>(dpb + (size_t)rowl[l] * BK + kk);
            const float2 da = make_float2(d4.x, d4.y), db = make_float2(d4.z, d4.w);
#pragma unroll
            for (int c = 0; c < 2; c++) {
                const float2 t0 = add2(da, W[c][0]);
                const float2 t1 = add2(db, W[c][1]);
                const int m = min(min(cm[l][c], __float_as_int(t0.x)), __float_as_int(t0.y));
                cm[l][c] = min(min(m, __float_as_int(t1.x)), __float_as_int(t1.y));
            }
        }
    }
    const uint32_t KK = (K << 16) | K;
#pragma unroll
    for (int l = 0; l < LPT; l++) {
        const float tau = S.tau[3 + rowl[l]];
#pragma unroll
        for (int c = 0; c < 2; c++) {
            const int other = __shfl_xor_sync(0xffffffffu, cm[l][c], 16);  // the partner's column q ^ 2
            if (h == grp) {  // the owner of layer group grp (id.lg == h when there are two groups)
#pragma unroll
                for (int e = 0; e < 2; e++) {
                    const int q = e ? 2 * (1 - h) + c : 2 * h + c;
                    const int x = (l * JPT + q) * nc + ct;
                    float bb = __uint_as_float(park[x]);
                    uint32_t w1 = park[NS * nc + x], w2 = park[2 * NS * nc + x];
                    band_fold(__int_as_float(e ? other : cm[l][c]), bb, tau, w1, w2, K, KK);
                    park[x] = __float_as_uint(bb);
                    park[NS * nc + x] = w1;
                    park[2 * NS * nc + x] = w2;
                }
            }
        }
    }
}

// Band words of the diagonal block from the parked state (after cons_diag_pair).
__device__ __forceinline__ void diag_pair_bands(const FastArgs &a, const uint32_t *park, int J, int split,
                                                const ConsId &id) {
    const int ct = id.ct, nc = a.ncons;
    const int g = split * a.Gc + id.gl;
    if (!(id.active && g < a.G)) return;
    constexpr int NS = LPT * JPT;
    const int64_t j0 = (int64_t)J * BJ;
#pragma unroll
    for (int l = 0; l < LPT; l++) {
        const int i = 3 + id.lg * LPT + l;
#pragma unroll
        for (int q = 0; q < JPT; q++) {
            const int64_t j = j0 + id.jq + NJQ * q;
            const int x = (l * JPT + q) * nc + ct;
            const uint32_t w1 = park[NS * nc + x], w2 = park[2 * NS * nc + x];
            if (i <= a.s && j < a.p) a.band[oidx(a, g, i, j)] = band_pack(w1, w2);
        }
    }
}

// Bounded wait (one thread) until `flag` is set; false when the wait gave up
// (timeout or abort).
__device__ __forceinline__ bool wait_flag(const FastArgs &a, const int *flag) {
    uint32_t spins = 0;
    while (ld_acquire(flag) == 0) {
        // the abort flag and the spin limit are checked every 64 spins, so a spin costs
        // one flag load and a short sleep
        if ((++spins & 63u) == 0u) {
            if (*(volatile int *)a.abort_flag) return false;
            if (spins > a.spin_limit) {
                a.st->timeout = 1;
                atomicExch(a.abort_flag, 1);
                return false;
            }
        }
        __nanosleep(32);
    }
    return true;
}
// ... until column block K of `split` is published (every row), or its rows 2..8 are.
__device__ __forceinline__ bool wait_block(const FastArgs &a, int split, int K) {
    return wait_flag(a, a.done + (size_t)split * a.nJ + K);
}
__device__ __forceinline__ bool wait_lower(const FastArgs &a, int split, int K) {
    return wait_flag(a, a.half + (size_t)split * a.nJ + K);
}

// Publish column block J of `split` (one thread, after a barrier that follows every
// thread's stores of the block).  The release store orders everything that happens
// before it, the other threads' stores included through the barrier, before the flag
// (the pattern of an acq_rel fence plus a relaxed store); readers acquire the flag.
__device__ __forceinline__ void publish_block(const FastArgs &a, int split, int J) {
    if (a.hold0 && J == 0) return;  // test hook: the waiters on block 0 must give up
    st_release(a.done + (size_t)split * a.nJ + J, 1);
}
// The first part of a split publish: rows 2..8 of block J (and their block minima).
__device__ __forceinline__ void publish_lower(const FastArgs &a, int split, int J) {
    if (a.hold0 && J == 0) return;
    st_release(a.half + (size_t)split * a.nJ + J, 1);
}

// ------------------------------------------------------------------ kernels
// Fused producer: two producer warps compute each tile's interval costs
// (tile_columns) and stage the dp32 rows with cp.async while the consumer warps
// evaluate the previous tile (named barriers FULL / EMPTY per buffer).
template <int LP>
__global__ void __launch_bounds__(NPROD + MAXCONS, 1) k_wavefront(FastArgs a) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    Smem &S = *reinterpret_cast<Smem *>(smem_raw);
    float *sDP = reinterpret_cast<float *>(smem_raw + sizeof(Smem));
    const int L = a.s - 2;                // layers 3..s
    const int rowsDP = a.Gc * L;          // staged dp32 rows per tile (layers 2..s-1)
    const int tid = threadIdx.x;
    const int nall = NPROD + a.ncons;
    for (int q = tid; q <= kMaxS; q += blockDim.x) S.tau[q] = a.prm->tau[q];
    if (tid < kMaxG) S.lam32[tid] = a.prm->lam32[tid];
    __syncthreads();

    if (tid < NPROD) {
        // =========================== producer warps ===========================
        const int jl = tid;  // column within the block
        uint32_t n = 0;      // tile sequence number
        for (;;) {
            if (tid == 0) S.ticket = atomicAdd(a.ticket, 1);
            bar_sync(BAR_PROD, NPROD);
            int t = S.ticket;
            bar_sync(BAR_PROD, NPROD);
            bool stop = t >= a.nJ * a.nsplit;
            int J = stop ? 0 : t / a.nsplit, split = stop ? 0 : t % a.nsplit;
            int ntiles = stop ? 1 : J + 1;
            for (int K = 0; K < ntiles; K++) {
                int b = n & 1;
                if (n >= 2) bar_sync(BAR_EMPTY + b, nall);
                if (stop) {
                    if (tid == 0) S.meta[b] = {0, 0, 0, 2};
                    bar_arrive(BAR_FULL + b, nall);
                    n++;
                    break;
                }
                bool diag = (K == J);
                int64_t k0 = (int64_t)K * BK;
                // wait for column block K (bounded); the diagonal needs nothing
                if (!diag && tid == 0) wait_block(a, split, K);
                bar_sync(BAR_PROD, NPROD);
                tile_consts(a, k0, jl, S.kv, S.kw, S.kd);
                // dp32 slice of rows (g, layer 2..s-1) for k in the tile (cp.async, L2 only)
                if (!diag) {
                    int gbase = split * a.Gc;
                    int n16 = rowsDP * (BK / 4);
                    float *dst = sDP + (size_t)b * rowsDP * BK;
                    for (int q = tid; q < n16; q += NPROD) {
                        int row = q / (BK / 4), c4 = q % (BK / 4);
                        int gl = row / L, li = row % L;  // layer index li -> dp row i = 2 + li
                        int g = gbase + gl;
                        float *sp = dst + (size_t)row * BK + c4 * 4;
                        if (g < a.G) {
                            const float *gp = a.dp32 + d32(a, g, 2 + li, k0 + c4 * 4);
                            unsigned sa = (unsigned)__cvta_generic_to_shared(sp);
                            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(sa), "l"(gp) : "memory");
                        } else {
                            *reinterpret_cast<float4 *>(sp) = make_float4(CUDART_INF_F, CUDART_INF_F, CUDART_INF_F,
                                                                          CUDART_INF_F);
                        }
                    }
                    asm volatile("cp.async.commit_group;" ::: "memory");
                }
                bar_sync(BAR_PROD, NPROD);
                tile_columns(a, K, J, jl, S.kv, S.kw, S.kd, S.wsum, S.C[b], S.Phi[b]);
                if (!diag) asm volatile("cp.async.wait_all;" ::: "memory");
                if (tid == 0) S.meta[b] = {J, K, split, diag ? 1 : 0};
                bar_arrive(BAR_FULL + b, nall);
                n++;
            }
            if (stop) break;
        }
        // drain: wait until the consumers released the last two buffers
        for (uint32_t q = (n >= 2 ? n - 2 : 0); q < n; q++) bar_sync(BAR_EMPTY + (q & 1), nall);
        return;
    }

    // ============================= consumer warps =============================
    const ConsId id = cons_id(a, tid - NPROD);
    ConsStateT<LP> cs;
    uint32_t n = 0;
    for (;;) {
        int b = n & 1;
        bar_sync(BAR_FULL + b, nall);
        TileMeta m = S.meta[b];
        if (m.kind == 2) { bar_arrive(BAR_EMPTY + b, nall); break; }
        const int g = m.split * a.Gc + id.gl;
        if (m.K == 0) cons_reset(cs);
        if (m.kind == 0) {
            if (id.active && g < a.G) cons_offdiag(a, S, sDP + (size_t)b * rowsDP * BK, b, (uint32_t)m.K, g, id, cs);
            bar_arrive(BAR_EMPTY + b, nall);
        } else {
            cons_diag(a, S, b, m.J, m.split, id, cs, false);
            if (id.ct == 0) publish_block(a, m.split, m.J);
            bar_arrive(BAR_EMPTY + b, nall);
        }
        n++;
    }
}

// Bulk copies of tile (K, J) into buffer b of the resident-cost kernel: the interval
// costs from the resident table and, off the diagonal, the dp32 rows (g, layers
// 2..s-1) of the split's real multipliers (rows of other slots are never read) and
// their block minima; on the diagonal, row 2 of the block.  res_issue_costs (one
// thread) expects every byte of the tile on mbar[b] and copies the costs, which no
// block publishes; res_issue_rows(w) copies multiplier w's rows (w = 0 also the
// minima) and needs block K made visible to the issuing thread's copies first
// (res_probe / res_wait for warp 0, the fence after the stage wait for the others).
// A copy may land before the expectation is posted: the phase cannot complete
// before the single arrival, which carries the whole byte count.
__device__ __forceinline__ void res_issue_costs(const FastArgs &a, Smem &S, int b, int K, int J, int split,
                                                uint64_t policy) {
    const int L = a.s - 2;
    const int gbase = split * a.Gc;
    const bool diag = K == J;
    const int ngv = std::min(a.G - gbase, a.Gc);  // real multipliers of the split
    const uint32_t rows_bytes = (uint32_t)((diag ? 1 : L) * BK * sizeof(float));
    const uint32_t mdp_bytes = (a.prune && !diag) ? (uint32_t)(ngv * a.mdp_stride * sizeof(float)) : 0u;
    const float *src = a.costs + (cost_tile_idx(K, J) - a.tile_base) * kCostTileFloats;
    mbar_expect_tx(&S.mbar[b], 2 * kCostHalfBytes + (uint32_t)ngv * rows_bytes + mdp_bytes);
    bulk_g2s(&S.C[b][0][0], src, kCostHalfBytes, &S.mbar[b], policy);
    bulk_g2s(&S.Phi[b][0][0], src + kCostHalfFloats, kCostHalfBytes, &S.mbar[b], policy);
}
__device__ __forceinline__ void res_issue_rows(const FastArgs &a, Smem &S, float *sDP, int b, int K, int J, int split,
                                               int w) {
    const int L = a.s - 2, rowsDP = a.Gc * L;
    const int gbase = split * a.Gc;
    const bool diag = K == J;
    const int ngv = std::min(a.G - gbase, a.Gc);
    const uint32_t rows_bytes = (uint32_t)((diag ? 1 : L) * BK * sizeof(float));
    if (w == 0 && a.prune && !diag)
        bulk_g2s_nohint(&S.mdp[b][0][0], a.mdp + ((size_t)K * a.G + gbase) * a.mdp_stride,
                        (uint32_t)(ngv * a.mdp_stride * sizeof(float)), &S.mbar[b]);
    float *dst = diag ? &S.diag[0][w][0] : sDP + (size_t)b * rowsDP * BK + (size_t)w * L * BK;
    bulk_g2s_nohint(dst, a.dp32 + d32(a, gbase + w, 2, (int64_t)K * BK), rows_bytes, &S.mbar[b]);
}
// Warp 0 alone issues the whole tile.
__device__ __forceinline__ void res_issue(const FastArgs &a, Smem &S, float *sDP, int b, int K, int J, int split,
                                          uint64_t policy, int lane) {
    if (lane == 0) res_issue_costs(a, S, b, K, J, split, policy);
    __syncwarp();
    if (lane < std::min(a.G - split * a.Gc, a.Gc)) res_issue_rows(a, S, sDP, b, K, J, split, lane);
}

// Warp 0 of the resident-cost kernel tracks `frontier`: every column block <= frontier
// of the current split is published.  A block publishes only after the block before
// it (its last off-diagonal tile waits for that one), so one flag seen set vouches for
// every block below it, and most tiles need no flag load at all.  When the frontier
// advances, every lane of warp 0 fences the generic-proxy stores of the newly
// published blocks (dp32 rows, block minima) against its later bulk copies, so the
// copies themselves carry no fence.
// res_probe: is block K published?  If K is past the frontier, the 32 lanes load the
// flags of blocks K, K + st, K + 2 st, ... (below J) at once and the frontier moves to
// the highest block seen published.
__device__ __forceinline__ bool res_probe(const FastArgs &a, int split, int K, int J, int &frontier, int lane) {
    if (K <= frontier) return true;
    const int stride = (J - K + 31) / 32;
    const int m = K + lane * stride;
    const bool set = m < J && ld_acquire(a.done + (size_t)split * a.nJ + m) != 0;
    const unsigned bal = __ballot_sync(0xffffffffu, set);
    if (bal == 0u) return false;
    frontier = K + (31 - __clz(bal)) * stride;
    __syncwarp();
    fence_proxy_async_global();
    return true;
}
// res_wait: bounded wait until block K is published (after res_probe said no).
__device__ __forceinline__ void res_wait(const FastArgs &a, int split, int K, int &frontier, int lane) {
    int ok = 0;
    if (lane == 0) ok = wait_block(a, split, K) ? 1 : 0;
    ok = __shfl_sync(0xffffffffu, ok, 0);
    if (ok) frontier = max(frontier, K);
    __syncwarp();
    fence_proxy_async_global();
}

// Tile skipping in batches (resident or streamed costs).  A batch is up to a.stage_tiles
// (at most 32) consecutive off-diagonal tiles of block J; warp 0 stages their column
// summaries (a.tsum) and the block minima of their column blocks (a.mdp, all G
// multipliers) into a stage buffer with two bulk copies, one batch ahead.  The stage
// buffers follow the dp32 rows in shared memory: where the paired diagonal parks its
// band state (free until the diagonal; 32 tiles per batch), else in space of their own
// (16 tiles per batch, for the larger rows of more layers).
__host__ __device__ __forceinline__ size_t stage_floats(int G, int mdp_stride, int ntiles) {
    return (size_t)ntiles * BJ * 2 + (size_t)ntiles * G * mdp_stride;
}
// The batch after the one ending at K1: 1, 1, 2, 4, ... nt tiles (the band limits are
// +inf before the first tile and tighten fast).
__device__ __forceinline__ int batch_end(int K1, int J, int nt) { return min(J, K1 + min(nt, max(1, K1))); }

// Warp 0: stage tiles K0 <= K < K1 of block J into stage buffer sb.  Minima of blocks
// past `frontier` may be incomplete in the copy; need_mask does not read them.
template <int NT>
__device__ __forceinline__ void res_stage(const FastArgs &a, Smem &S, float *stg, int sb, int K0, int K1, int J,
                                          int frontier, uint64_t policy, int lane) {
    if (lane == 0) {
        const uint32_t tb = (uint32_t)((size_t)(K1 - K0) * BJ * sizeof(float2));
        const uint32_t mb = (uint32_t)((size_t)(K1 - K0) * a.G * a.mdp_stride * sizeof(float));
        S.sfront[sb] = frontier;  // ordered before the readers' wait by the arrive (release)
        mbar_expect_tx(&S.smbar[sb], tb + mb);
        bulk_g2s(stg, a.tsum + (cost_tile_idx(0, J) - a.tile_base + (size_t)K0) * BJ, tb, &S.smbar[sb], policy);
        bulk_g2s_nohint(stg + (size_t)NT * BJ * 2, a.mdp + (size_t)K0 * a.G * a.mdp_stride, mb, &S.smbar[sb]);
    }
}

// Batch skip test of one warp over the staged tiles K0 <= K < K1: bit K - K0 of the
// result is set when some output of the warp may take a candidate from tile K by the
// test of cons_offdiag, here evaluated on the staged column minima and block minima
// with the warp's band limits as they stand.  The limits only shrink as later tiles
// fold, and rounding is monotone, so a tile this test rules out is ruled out by
// cons_offdiag too: walking only the tiles some warp needs changes no result.  Blocks
// past `fr` had no published minima when staged and are always needed.
template <int NT, int LP>
__device__ __forceinline__ uint32_t need_mask(const FastArgs &a, const Smem &S, const float *stg, int K0, int K1, int fr,
                                              int g, const ConsId &id, const ConsStateT<LP> &cs) {
    const int L = a.s - 2;
    const float lam = S.lam32[g];
    int rowl[LP];
    float lim[LP][JPT];
#pragma unroll
    for (int l = 0; l < LP; l++) {
        rowl[l] = min(id.lg * LP + l, L - 1);
        const float tau = S.tau[3 + rowl[l]];
#pragma unroll
        for (int q = 0; q < JPT; q++) lim[l][q] = __fadd_rn(cs.best[l][q], __fmul_rn(cs.best[l][q], tau));
    }
    const float2 *ts = reinterpret_cast<const float2 *>(stg) + id.jq;
    const float *md = stg + (size_t)NT * BJ * 2 + (size_t)g * a.mdp_stride + 2;
    const int mstride = a.G * a.mdp_stride;
    uint32_t mask = 0;
#pragma unroll 2
    for (int K = K0; K < K1; K++) {
        bool need = true;
        if (K <= fr) {
            const int r = K - K0;
            float lbq[JPT];
#pragma unroll
            for (int q = 0; q < JPT; q++) {
                const float2 v = ts[r * BJ + NJQ * q];
                lbq[q] = __fmaf_rn(lam, v.y, v.x);
            }
            need = false;
#pragma unroll
            for (int l = 0; l < LP; l++) {
                const float m = md[r * mstride + rowl[l]];
#pragma unroll
                for (int q = 0; q < JPT; q++) need |= __fadd_rn(m, lbq[q]) <= lim[l][q];
            }
        }
        mask |= (__any_sync(0xffffffffu, need) ? 1u : 0u) << (K - K0);
    }
    return mask;
}

// Resident interval costs: no producer warps.  Warp 0 claims the column blocks,
// waits for the flags and issues the bulk copies of the next tile while the current
// one is evaluated (two buffers, one mbarrier each); all MAXCONS threads are
// consumers.  With tile skipping the off-diagonal tiles go in staged batches: every
// warp runs need_mask over the batch and only the tiles some warp needs are copied
// in and walked, so a tile every warp rules out costs neither HBM traffic nor a
// barrier; the next batch is staged while this one is walked.
template <int LP>
__global__ void __launch_bounds__(MAXCONS, 1) k_wavefront_res(FastArgs a) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    Smem &S = *reinterpret_cast<Smem *>(smem_raw);
    float *sDP = reinterpret_cast<float *>(smem_raw + sizeof(Smem));
    const int L = a.s - 2;
    const int rowsDP = a.Gc * L;
    const int ct = threadIdx.x;
    const int lane = ct & 31;
    for (int q = ct; q <= kMaxS; q += blockDim.x) S.tau[q] = a.prm->tau[q];
    if (ct < kMaxG) S.lam32[ct] = a.prm->lam32[ct];
    if (ct == 0) {
        mbar_init(&S.mbar[0], 1);
        mbar_init(&S.mbar[1], 1);
        mbar_init(&S.smbar[0], 1);
        mbar_init(&S.smbar[1], 1);
        mbar_fence_init();
    }
    __syncthreads();
    const ConsId id = cons_id(a, ct);
    ConsStateT<LP> cs;
    const uint64_t policy = policy_evict_first();
    uint32_t n = 0;   // tile sequence number: buffer n & 1
    uint32_t mph[2] = {0u, 0u};  // completed phases of mbar[0], mbar[1] (one per fill; two for a split last tile)
    uint32_t ns = 0;  // batch sequence number (tile skipping): stage buffer ns & 1, its fill ns >> 1
    float *stage = sDP + (size_t)2 * rowsDP * BK;  // the park area, free off the diagonal
    constexpr int NT = LP == LPT ? 32 : 16;  // tiles per staged batch (a.stage_tiles, set to match)
    const size_t sfl = stage_floats(a.G, a.mdp_stride, NT);
    unsigned long long n_run = 0, n_skip = 0;  // lane 0 of each warp: its (warp, tile) units
    int frontier = -1, fsplit = -1;            // warp 0 (res_probe)
    for (;;) {
        if (ct == 0) S.ticket = atomicAdd(a.ticket, 1);
        __syncthreads();
        const int t = S.ticket;
        if (t >= (a.J1 - a.J0) * a.nsplit) break;
        const int J = a.J0 + t / a.nsplit, split = t % a.nsplit;
        const int g = split * a.Gc + id.gl;
        const bool own = id.active && g < a.G;
        if (split != fsplit) { frontier = -1; fsplit = split; }
        cons_reset(cs);
        if (a.seed && own) cons_seed(a, cs, J, id);
        int issued = -1;  // the tile whose copies are in flight into buffer n & 1 (J: the diagonal), or -1
        const int ngv = min(a.G - split * a.Gc, a.Gc);  // real multipliers of the split
        // the tiles walked here: K < Kend (with a split publish the last one, J - 1, is the chain's)
        const int Kend = a.split_pub ? max(J - 1, 0) : J;
        if (a.prune && Kend > 0 && ct < 32) {  // stage the first batch
            if (frontier < 0) res_probe(a, split, 0, J, frontier, lane);
            res_stage<NT>(a, S, stage + (ns & 1) * sfl, ns & 1, 0, batch_end(0, Kend, NT), J, frontier, policy, lane);
        }
        for (int K0 = 0; K0 < Kend;) {
            const int K1 = a.prune ? batch_end(K0, Kend, NT) : min(Kend, K0 + 32);
            uint32_t wm = 0xffffffffu;  // the warp's tiles of the batch
            uint32_t U = 0xffffffffu;   // the tiles some warp needs
            int frb = -1;               // tiles <= frb: every warp issues its own rows (res_issue_rows)
            if (a.prune) {
                const int sb = ns & 1;
                mbar_wait_bounded(&S.smbar[sb], (ns >> 1) & 1u, a.st, a.abort_flag);
                frb = S.sfront[sb];
                if (lane == 0) fence_proxy_async_global();  // blocks <= frb, published, before this warp's copies
                wm = own ? need_mask<NT>(a, S, stage + sb * sfl, K0, K1, frb, g, id, cs) : 0u;
                if (lane == 0) S.needw[sb][ct >> 5] = wm;
                __syncthreads();  // needw; every read of stage buffer sb is done
                U = 0;
                for (int w = 0; w < (int)(blockDim.x >> 5); w++) U |= S.needw[sb][w];
                ns++;
                if (K1 < Kend && ct < 32) {  // stage the next batch while this one is walked
                    const int K2 = batch_end(K1, Kend, NT);
                    if (K2 - 1 > frontier) res_probe(a, split, frontier + 1, J, frontier, lane);
                    res_stage<NT>(a, S, stage + (ns & 1) * sfl, ns & 1, K1, K2, J, frontier, policy, lane);
                }
            }
            U &= (K1 - K0 == 32) ? 0xffffffffu : ((1u << (K1 - K0)) - 1u);
            if (own) n_skip += (unsigned long long)(K1 - K0 - __popc(U));
            if (U && issued < 0) {
                const int Kf = K0 + __ffs(U) - 1;
                if (Kf <= frb) {
                    if (ct == 0) res_issue_costs(a, S, n & 1, Kf, J, split, policy);
                    if (lane == 0 && (ct >> 5) < ngv) res_issue_rows(a, S, sDP, n & 1, Kf, J, split, ct >> 5);
                } else if (ct < 32) {
                    if (!res_probe(a, split, Kf, J, frontier, lane)) res_wait(a, split, Kf, frontier, lane);
                    res_issue(a, S, sDP, n & 1, Kf, J, split, policy, lane);
                }
            }
            while (U) {
                const int K = K0 + __ffs(U) - 1;
                U &= U - 1;
                // the next tile to copy: the batch's next needed one, else the diagonal after
                // the last batch (with a split publish the tail copies its own tiles), else (no
                // skipping) the next batch's first tile
                const int Kn = U ? K0 + __ffs(U) - 1 : (K1 == Kend ? (a.split_pub ? -1 : J) : (a.prune ? -1 : K1));
                const int b = n & 1;
                bool pending = false;  // warp 0: the rows of tile Kn still to be issued
                if (Kn >= 0 && Kn < J && Kn <= frb) {
                    if (ct == 0) res_issue_costs(a, S, b ^ 1, Kn, J, split, policy);
                    if (lane == 0 && (ct >> 5) < ngv) res_issue_rows(a, S, sDP, b ^ 1, Kn, J, split, ct >> 5);
                } else if (ct < 32 && Kn >= 0) {
                    const bool ready = Kn >= J || res_probe(a, split, Kn, J, frontier, lane);
                    if (ready)
                        res_issue(a, S, sDP, b ^ 1, Kn, J, split, policy, lane);
                    else if (lane == 0)
                        res_issue_costs(a, S, b ^ 1, Kn, J, split, policy);  // the costs publish nothing
                    pending = !ready;
                }
                issued = Kn;
                mbar_wait_bounded(&S.mbar[b], mph[b] & 1u, a.st, a.abort_flag);
                mph[b]++;
                if (own) {
                    const bool ran = ((wm >> (K - K0)) & 1u) &&
                                     cons_offdiag(a, S, sDP + (size_t)b * rowsDP * BK, b, (uint32_t)K, g, id, cs);
                    n_run += ran ? 1 : 0;
                    n_skip += ran ? 0 : 1;
                }
                __syncthreads();  // buffer b free for the tile after Kn
                if (ct < 32 && pending) {
                    res_wait(a, split, Kn, frontier, lane);
                    if (lane < ngv) res_issue_rows(a, S, sDP, b ^ 1, Kn, J, split, lane);
                }
                n++;
            }
            K0 = K1;
        }
        if constexpr (LP != LPT) {  // the generic diagonal (no split publish, no parked state)
            const int b = n & 1;
            if (issued != J && ct < 32) res_issue(a, S, sDP, b, J, J, split, policy, lane);
            mbar_wait_bounded(&S.mbar[b], mph[b] & 1u, a.st, a.abort_flag);
            mph[b]++;
            cons_diag(a, S, b, J, split, id, cs, true);
            __syncthreads();  // every thread's dp32 and layer minima of block J are stored
            if (ct == 0) publish_block(a, split, J);
            n++;
        } else if (a.split_pub) {
            // the chain's part: tile (J-1, J) in buffer bA, the diagonal in bD (the cost copies
            // depend on nothing published; the diagonal also copies row 2 of block J)
            uint32_t *park = reinterpret_cast<uint32_t *>(sDP + (size_t)2 * rowsDP * BK);
            const int bA = n & 1, bD = bA ^ 1;
            const int gbase = split * a.Gc;
            const uint32_t lo_bytes = (uint32_t)(LPT * BK * sizeof(float));        // rows 2..8
            const uint32_t hi_bytes = (uint32_t)((L - LPT) * BK * sizeof(float));  // rows 9..s-1
            float *rowsA = sDP + (size_t)bA * rowsDP * BK;
            if (ct < 32) {
                if (lane == 0) {
                    if (J > 0) {
                        mbar_expect_tx(&S.mbar[bA], 2 * kCostHalfBytes + (uint32_t)ngv * lo_bytes);
                        const float *src = a.costs + (cost_tile_idx(J - 1, J) - a.tile_base) * kCostTileFloats;
                        bulk_g2s(&S.C[bA][0][0], src, kCostHalfBytes, &S.mbar[bA], policy);
                        bulk_g2s(&S.Phi[bA][0][0], src + kCostHalfFloats, kCostHalfBytes, &S.mbar[bA], policy);
                    }
                    res_issue_costs(a, S, bD, J, J, split, policy);
                }
                __syncwarp();
                if (lane < ngv) res_issue_rows(a, S, sDP, bD, J, J, split, lane);
            }
            mbar_wait_bounded(&S.mbar[bD], mph[bD] & 1u, a.st, a.abort_flag);
            mph[bD]++;
            float2 W[2 * kDiagGroups];
            diag_prepare(a, S, park, bD, J, split, id, cs, W);
            int cur = 0;
            if (J > 0) {  // layer group 0 of tile (J-1, J): rows 2..8 of block J-1
                if (ct < 32) {
                    if (lane == 0) wait_lower(a, split, J - 1);
                    __syncwarp();
                    fence_proxy_async_global();
                    if (lane < ngv)
                        bulk_g2s_nohint(rowsA + (size_t)lane * L * BK, a.dp32 + d32(a, gbase + lane, 2, (int64_t)(J - 1) * BK),
                                        lo_bytes, &S.mbar[bA]);
                }
                mbar_wait_bounded(&S.mbar[bA], mph[bA] & 1u, a.st, a.abort_flag);
                mph[bA]++;
                if (own) cons_lasttile_grp(a, S, rowsA, bA, park, (uint32_t)(J - 1), g, id, 0);
                __syncwarp();
            }
            diag_layers(a, S, park, J, split, id, W, 0, LPT - 1, cur);  // layers 3..8
            diag_store(a, park, J, split, id, 3, 2 + LPT - 1);
            __syncthreads();  // rows 3..8 and their block minima are stored
            if (ct == 0) publish_lower(a, split, J);
            diag_layers(a, S, park, J, split, id, W, LPT - 1, LPT, cur);  // layer 9
            if (J > 0) {  // layer group 1: rows 9..s-1 of block J-1, after its full publish
                if (ct < 32) {
                    if (lane == 0) {
                        mbar_expect_tx(&S.mbar[bA], (uint32_t)ngv * hi_bytes);
                        wait_block(a, split, J - 1);
                    }
                    __syncwarp();
                    fence_proxy_async_global();
                    if (lane < ngv)
                        bulk_g2s_nohint(rowsA + (size_t)lane * L * BK + LPT * BK,
                                        a.dp32 + d32(a, gbase + lane, 2 + LPT, (int64_t)(J - 1) * BK), hi_bytes,
                                        &S.mbar[bA]);
                }
                mbar_wait_bounded(&S.mbar[bA], mph[bA] & 1u, a.st, a.abort_flag);
                mph[bA]++;
                if (own) cons_lasttile_grp(a, S, rowsA, bA, park, (uint32_t)(J - 1), g, id, 1);
                __syncwarp();
                if (own) n_run++;
            }
            diag_layers(a, S, park, J, split, id, W, LPT, L, cur);  // layers 10..s
            diag_store(a, park, J, split, id, 2 + LPT, a.s);
            __syncthreads();  // every row and block minimum of block J is stored
            if (ct == 0) publish_block(a, split, J);
            diag_pair_bands(a, park, J, split, id);
            n += 2;
        } else {  // the diagonal tile (issued with the last tile walked, else now)
            const int b = n & 1;
            if (issued != J && ct < 32) res_issue(a, S, sDP, b, J, J, split, policy, lane);
            mbar_wait_bounded(&S.mbar[b], mph[b] & 1u, a.st, a.abort_flag);
            mph[b]++;
            uint32_t *park = reinterpret_cast<uint32_t *>(sDP + (size_t)2 * rowsDP * BK);
            if (a.lgc == 2)
                cons_diag_pair(a, S, park, b, J, split, id, cs);
            else
                cons_diag(a, S, b, J, split, id, cs, true);
            __syncthreads();  // every thread's dp32 and layer minima of block J are stored
            if (ct == 0) publish_block(a, split, J);
            if (a.lgc == 2) diag_pair_bands(a, park, J, split, id);
            n++;
        }
    }
    if (lane == 0 && (n_run | n_skip)) {
        atomicAdd((unsigned long long *)&a.st->tiles_run, n_run);
        atomicAdd((unsigned long long *)&a.st->tiles_skipped, n_skip);
    }
    if (ct == 0 && n) atomicAdd((unsigned long long *)&a.st->tiles_fetched, (unsigned long long)n);  // one cost tile per buffer fill
}

// ------------------------------------------------------------ base layer
// eq. apx_base for every multiplier: exact dp64, bp and the fp32 copy; all
// other rows cleared (dp64 = +inf, bp = -1, dp32 = +inf).
__global__ void k_fast_clear(double *dp64, int32_t *bp, float *dp32, size_t n) {
    size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    size_t stride = (size_t)gridDim.x * blockDim.x;
    for (; i < n; i += stride) { dp64[i] = CUDART_INF; bp[i] = -1; dp32[i] = CUDART_INF_F; }
}

__global__ void k_fast_base(Prefix P, FastArgs a, double *dp64, int32_t *bp) {
    int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x + 1;
    if (j >= P.p) return;
    double C, U, D;
    pair_exact(P, 0, j, C, U, D);
    double phi = phi_exact(P, U, D, true);
    for (int g = 0; g < a.G; g++) {
        double v = __dadd_rn(C, __dmul_rn(a.prm->lam64[g], phi));
        dp64[oidx(a, g, 2, j)] = v;
        bp[oidx(a, g, 2, j)] = 0;
        a.dp32[d32(a, g, 2, j)] = __fadd_rn(__double2float_rn(v), 0.0f);  // >= +0 (no -0)
    }
}

// ------------------------------------------------------------- extraction
// fp32 value of candidate k for output (g, i, j), bit-identical to the wavefront.
__device__ __forceinline__ float cand32(float dprev, float lam, float C, float Phi) {
    return __fadd_rn(dprev, __fmaf_rn(lam, Phi, C));
}

// Visit the candidates k of tile K for output (g, i, j) in the wavefront's fp32
// arithmetic (k descending) and call f(k, value) for every k with value <= thr.
template <typename F>
__device__ void visit_tile(const FastArgs &a, int g, int i, int64_t j, int64_t K, float thr, F &&f) {
    int64_t J = j / BJ, j0 = J * BJ, k0 = K * BK;
    float lam = a.prm->lam32[g];
    const float *prev = a.dp32 + d32(a, g, i - 1, k0) - k0;  // prev[k] for k in tile K
    if (a.costs) {
        // the wavefront's own interval costs, read back from the resident table
        const float *cr = a.costs + (cost_tile_idx(K, J) - a.tile_base) * kCostTileFloats + (size_t)(j - j0) * PSTR;
        const float *pr = cr + kCostHalfFloats;
        int64_t khi = (K == J) ? j - 1 : k0 + BK - 1;
        for (int64_t k = khi; k >= k0; k--) {
            const float v = cand32(prev[k], lam, cr[k - k0], pr[k - k0]);
            if (v <= thr) f(k, v);
        }
        return;
    }
    float vj = a.v[j];
    const float d_f = (float)a.d;
    Rec r;
    int64_t khi;
    float c, ph;
    if (K == J) {
        r = rec_empty();
        khi = j;  // state of the empty interval (j, j]
    } else {
        khi = k0 + BK - 1;
        rec_anchor(a, khi, j, r);  // any evaluation within the certified bound will do
        rec_emit(r, vj, a.v[khi], d_f, a.invd, c, ph);
        const float v = cand32(prev[khi], lam, c, ph);
        if (v <= thr) f(khi, v);
    }
    for (int64_t k = khi - 1; k >= k0; k--) {
        rec_step(r, vj, a.v[k + 1], a.wf[k + 1], __fsub_rn(a.v[k + 1], a.v[k]));
        rec_emit(r, vj, a.v[k], d_f, a.invd, c, ph);
        const float v = cand32(prev[k], lam, c, ph);
        if (v <= thr) f(k, v);
    }
}

// Tiles listed by a band word (band_update), in increasing order.
template <typename F>
__device__ void visit_band(const FastArgs &a, int g, int i, int64_t j, uint64_t w, float thr, F &&f) {
    const uint32_t w1 = (uint32_t)w, w2 = (uint32_t)(w >> 32);
    for (uint32_t K = w1 >> 16; K <= (w1 & 0xFFFFu); K++) visit_tile(a, g, i, j, (int64_t)K, thr, f);
    if (w2)
        for (uint32_t K = w2 >> 16; K <= (w2 & 0xFFFFu); K++) visit_tile(a, g, i, j, (int64_t)K, thr, f);
}

// Tiles a band word spans (both runs).
__device__ __forceinline__ uint32_t band_tiles(uint64_t w) {
    const uint32_t w1 = (uint32_t)w, w2 = (uint32_t)(w >> 32);
    return (w1 & 0xFFFFu) - (w1 >> 16) + 1u + (w2 ? (w2 & 0xFFFFu) - (w2 >> 16) + 1u : 0u);
}

__device__ __forceinline__ float band_threshold(const FastArgs &a, int i, float m32) {
    return __fadd_rn(m32, __fmul_rn(m32, a.prm->tau[i]));
}

// The candidates of output (g, i, j)'s band, by the 32 lanes of a warp together, with
// visit_tile's decisions (fp32 value <= thr): f(in, k, v) is called by every lane at once
// (a warp-uniform call; `in` is false for a lane without a candidate in that step;
// `v` is the candidate's fp32 value, +inf for a lane without one).
// With resident costs the lanes split every tile's k (the table gives any pair
// directly); otherwise they take whole tiles and walk them in step along visit_tile's
// recurrence (k descending from the anchor at the tile's top pair, or from the empty
// interval (j, j] on the diagonal tile), so the values, and the decisions, are visit_tile's.
template <typename F>
__device__ __forceinline__ void warp_visit_band(const FastArgs &a, int g, int i, int64_t j, uint64_t w, float thr,
                                                F &&f) {
    const int lane = threadIdx.x & 31;
    const uint32_t w1 = (uint32_t)w, w2 = (uint32_t)(w >> 32);
    const uint32_t n1 = (w1 & 0xFFFFu) - (w1 >> 16) + 1u;
    const uint32_t ntile = n1 + (w2 ? (w2 & 0xFFFFu) - (w2 >> 16) + 1u : 0u);
    const float lam32 = a.prm->lam32[g];
    const int64_t J = j / BJ, j0 = J * BJ;
    if (a.costs) {
        for (uint32_t t = 0; t < ntile; t++) {
            const int64_t K = t < n1 ? (w1 >> 16) + t : (w2 >> 16) + (t - n1);
            const int64_t k0 = K * BK;
            const float *cr = a.costs + (cost_tile_idx(K, J) - a.tile_base) * kCostTileFloats + (size_t)(j - j0) * PSTR;
            const float *pr = cr + kCostHalfFloats;
            const float *prev32 = a.dp32 + d32(a, g, i - 1, k0) - k0;
            const int64_t khi = (K == J) ? j - 1 : k0 + BK - 1;
            for (int64_t kb = k0; kb <= khi; kb += 32) {  // warp-uniform
                const int64_t k = kb + lane;
                const float v = k <= khi ? cand32(prev32[k], lam32, cr[k - k0], pr[k - k0]) : CUDART_INF_F;
                f(v <= thr, k, v);
            }
        }
        return;
    }
    const float vj = a.v[j], d_f = (float)a.d;
    for (uint32_t tb = 0; tb < ntile; tb += 32) {  // warp-uniform
        const uint32_t t = tb + lane;
        // tile K of the band (lanes past the band's end take tile 0 and no candidate)
        const int64_t K = t >= ntile ? 0 : (int64_t)(t < n1 ? (w1 >> 16) + t : (w2 >> 16) + (t - n1));
        const int64_t k0 = K * BK;
        const float *prev32 = a.dp32 + d32(a, g, i - 1, k0) - k0;
        Rec r = rec_empty();
        int64_t kfirst = k0 + BK - 1;
        int nk = 0;  // candidates of the lane's tile: k = kfirst, kfirst - 1, ..., kfirst - nk + 1
        if (t < ntile) {
            if (K == J) {
                kfirst = j - 1;
                nk = (int)(j - k0);
            } else {
                nk = BK;
                rec_anchor(a, kfirst, j, r);
            }
        }
        for (int it = 0; it < BK; it++) {  // warp-uniform
            const int64_t k = kfirst - it;
            float v = CUDART_INF_F;
            if (it < nk) {
                if (it > 0 || K == J) rec_step(r, vj, a.v[k + 1], a.wf[k + 1], __fsub_rn(a.v[k + 1], a.v[k]));
                float c, ph;
                rec_emit(r, vj, a.v[k], d_f, a.invd, c, ph);
                v = cand32(prev32[k], lam32, c, ph);
            }
            f(it < nk && v <= thr, k, v);
        }
    }
}

// Outputs eq. apx_final reads: dp(i, p-1) for i in [ilo, s] (or every output).
__global__ void k_need_init(FastArgs a, int ilo, int all) {
    int64_t tot = (int64_t)a.G * (a.s + 1) * a.ps;
    int64_t id = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (; id < tot; id += stride) {
        int64_t j = id % a.ps;
        int i = (int)((id / a.ps) % (a.s + 1));
        uint8_t v = 0;
        if (i >= 3 && j < a.p && j >= i - 1) v = all ? 1 : (j == a.p - 1 && i >= ilo);
        a.need[id] = v;
    }
}

// Warp-aggregated append of `v` to list[*cnt] by the lanes of `mask` that want it.
__device__ __forceinline__ void warp_append(unsigned mask, bool want, int32_t v, int32_t *list, int *cnt) {
    const unsigned m = __ballot_sync(mask, want);
    if (!m) return;
    const int lane = threadIdx.x & 31;
    const int leader = __ffs(m) - 1;
    int base = 0;
    if (lane == leader) base = atomicAdd(cnt, __popc(m));
    base = __shfl_sync(mask, base, leader);
    if (want) list[base + __popc(m & ((1u << lane) - 1u))] = v;
}

__device__ __forceinline__ int32_t *layer_list(const FastArgs &a, int i, int kind) {
    return a.lists + ((size_t)i * 2 + kind) * (size_t)a.G * (size_t)a.ps;
}

// Backward closure, layer i: members of every needed output; mark (i-1, k) needed;
// list the needed outputs for the exact stage (inline members / big bands).  A thread
// walks an output's band when it spans at most kThreadTiles tiles; wider bands go to
// k_need_wide, a warp each (threads of one warp walking bands of very different widths
// would wait on the widest).
constexpr uint32_t kThreadTiles = 4;
__global__ void k_need_layer(FastArgs a, int i) {
    if (*(volatile const int *)a.abort_flag) return;  // a wait gave up: the tables are not valid
    const int64_t tot = (int64_t)a.G * a.p;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    unsigned long long nmem = 0, nbig = 0;
    int32_t *lsmall = layer_list(a, i, 0), *lbig = layer_list(a, i, 1);
    int *csmall = a.list_cnt + 2 * i, *cbig = csmall + 1;
    for (int64_t base = (int64_t)blockIdx.x * blockDim.x; base < tot; base += stride) {  // warp-uniform trip count
        const int64_t id = base + threadIdx.x;
        bool listed = false, wide = false;
        int cnt = 0;
        int32_t packed = 0;
        if (id < tot) {
            const int64_t j = id % a.p;
            const int g = (int)(id / a.p);
            const size_t o = oidx(a, g, i, j);
            if (j >= i - 1 && a.need[o]) {
                const float m32 = a.dp32[d32(a, g, i, j)];
                if (!(m32 < CUDART_INF_F)) {
                    a.mcnt[o] = 0;
                } else {
                    const uint64_t w = a.band[o];
                    packed = (int32_t)((g << 24) | (int32_t)j);
                    if (band_tiles(w) > kThreadTiles) {
                        wide = true;  // a warp walks it (k_need_wide): lanes' walks would diverge
                    } else {
                        int32_t *mem = a.members + o * NMEM;
                        uint8_t *below = a.need + oidx(a, g, i - 1, 0);
                        const bool mark = i - 1 >= 3;
                        float vmin = CUDART_INF_F;
                        int32_t kmin = -1;
                        visit_band(a, g, i, j, w, band_threshold(a, i, m32), [&](int64_t k, float v) {
                            if (cnt < NMEM) mem[cnt] = (int32_t)k;
                            cnt++;
                            if (mark) below[k] = 1;
                            if (v < vmin || (v == vmin && (int32_t)k < kmin)) { vmin = v; kmin = (int32_t)k; }
                        });
                        if (cnt > NMEM) mem[0] = kmin;  // a big output keeps its fp32 argmin (k_exact_big)
                        a.mcnt[o] = cnt;
                        nmem += cnt;
                        nbig += cnt > NMEM;
                        listed = true;
                    }
                }
            }
        }
        warp_append(0xffffffffu, listed && cnt <= NMEM, packed, lsmall, csmall);
        warp_append(0xffffffffu, listed && cnt > NMEM, packed, lbig, cbig);
        warp_append(0xffffffffu, wide, packed, a.wide, a.wide_cnt + i);
    }
    if (nmem) atomicAdd((unsigned long long *)&a.st->members, nmem);
    if (nbig) atomicAdd((unsigned long long *)&a.st->big_bands, nbig);
}

// The closure of layer i for the outputs k_need_layer deferred: a warp per output walks
// its band (warp_visit_band), marks (i-1, k) needed for every member, keeps the first
// NMEM members it meets (the exact stage's rule is order-free) and lists the output.
__global__ void __launch_bounds__(128) k_need_wide(FastArgs a, int i) {
    if (*(volatile const int *)a.abort_flag) return;  // a wait gave up: the tables are not valid
    const int n = a.wide_cnt[i];
    const int lane = threadIdx.x & 31;
    const unsigned lt = (1u << lane) - 1u;
    const int warps = gridDim.x * (blockDim.x >> 5);
    const bool mark = i - 1 >= 3;
    int32_t *lsmall = layer_list(a, i, 0), *lbig = layer_list(a, i, 1);
    int *csmall = a.list_cnt + 2 * i, *cbig = csmall + 1;
    unsigned long long nmem = 0, nbig = 0, nover = 0;  // lane 0
    for (int e = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); e < n; e += warps) {
        const int32_t v = a.wide[e];
        const int g = v >> 24;
        const int64_t j = v & 0xFFFFFF;
        const size_t o = oidx(a, g, i, j);
        const uint64_t w = a.band[o];
        int32_t *mem = a.members + o * NMEM;
        uint8_t *below = a.need + oidx(a, g, i - 1, 0);
        int cnt = 0;  // warp-uniform
        float vmin = CUDART_INF_F;  // per lane: its least member value, lowest k on ties
        int32_t kmin = INT32_MAX;
        warp_visit_band(a, g, i, j, w, band_threshold(a, i, a.dp32[d32(a, g, i, j)]), [&](bool in, int64_t k, float v) {
            const unsigned mask = __ballot_sync(0xffffffffu, in);
            if (in) {
                const int pos = cnt + __popc(mask & lt);
                if (pos < NMEM) mem[pos] = (int32_t)k;
                if (mark) below[k] = 1;
                if (v < vmin || (v == vmin && (int32_t)k < kmin)) { vmin = v; kmin = (int32_t)k; }
            }
            cnt += __popc(mask);
        });
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            const float v2 = __shfl_xor_sync(0xffffffffu, vmin, off);
            const int32_t k2 = __shfl_xor_sync(0xffffffffu, kmin, off);
            if (v2 < vmin || (v2 == vmin && k2 < kmin)) { vmin = v2; kmin = k2; }
        }
        __syncwarp();  // every lane's member stores are done before lane 0 overwrites slot 0
        if (lane == 0) {
            if (cnt > NMEM) mem[0] = kmin;  // a big output keeps its fp32 argmin (k_exact_big)
            a.mcnt[o] = cnt;
            nmem += cnt;
            nbig += cnt > NMEM;
            nover += band_tiles(w) > 32u ? 1 : 0;  // wide bands (diagnostic)
            if (cnt <= NMEM) lsmall[atomicAdd(csmall, 1)] = v;
            else lbig[atomicAdd(cbig, 1)] = v;
        }
        __syncwarp();
    }
    if (lane == 0) {
        if (nmem) atomicAdd((unsigned long long *)&a.st->members, nmem);
        if (nbig) atomicAdd((unsigned long long *)&a.st->big_bands, nbig);
        if (nover) atomicAdd((unsigned long long *)&a.st->overflow, nover);
    }
}

// Outputs the answer does not read keep their fp32 minimum: dp64 = m32, bp = -2.
__global__ void k_fill_unneeded(FastArgs a, double *dp64, int32_t *bp) {
    if (*(volatile const int *)a.abort_flag) return;  // a wait gave up: the tables are not valid
    const int64_t tot = (int64_t)a.G * (a.s + 1) * a.ps;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t o = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; o < tot; o += stride) {
        const int64_t j = o % a.ps;
        const int i = (int)((o / a.ps) % (a.s + 1));
        const int g = (int)(o / (a.ps * (a.s + 1)));
        if (i < 3 || j >= a.p || j < i - 1 || a.need[o]) continue;
        const float m32 = a.dp32[d32(a, g, i, j)];
        if (m32 < CUDART_INF_F) { dp64[o] = (double)m32; bp[o] = -2; }
    }
}

// ----------------------------------------------------------- exact layer
__device__ __forceinline__ double exact_value(const Prefix &P, const double *prev, int64_t k, int64_t j, double lam) {
    double C, U, D;
    pair_exact(P, k, j, C, U, D);
    return __dadd_rn(prev[k], __dadd_rn(C, __dmul_rn(lam, phi_exact(P, U, D, false))));
}
__device__ __forceinline__ void exact_candidate(const Prefix &P, const double *prev, int64_t k, int64_t j,
                                                double lam, double &best, int32_t &arg) {
    const double c = exact_value(P, prev, k, j, lam);
    if (c < best || (c == best && k < arg)) { best = c; arg = (int32_t)k; }
}

// Result of a resolved output and its certificate check: the fp32 minimum must lie
// within eps_i of the exact one.
__device__ __forceinline__ bool exact_store(const FastArgs &a, int g, int i, int64_t j, double best, int32_t arg,
                                            double *dp64, int32_t *bp) {
    const size_t o = oidx(a, g, i, j);
    dp64[o] = best;
    bp[o] = arg == INT32_MAX ? -1 : arg;
    const float m32 = a.dp32[d32(a, g, i, j)];
    const double e = (double)a.prm->eps[i];
    return fabs((double)m32 - best) <= e * best * 1.0001;
}

__device__ __forceinline__ void count_exact(const FastArgs &a, unsigned long long nres, int nviol) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        nres += __shfl_xor_sync(0xffffffffu, nres, o);
        nviol += __shfl_xor_sync(0xffffffffu, nviol, o);
    }
    if ((threadIdx.x & 31) == 0) {
        if (nres) atomicAdd((unsigned long long *)&a.st->rescored, nres);
        if (nviol) atomicAdd(&a.st->bound_viol, nviol);
    }
}

// Layer i, outputs with at most NMEM members: one thread each, binary64 re-scoring
// with double-double interval costs; the lowest k among exact minima wins.
__global__ void __launch_bounds__(128) k_exact_small(Prefix P, FastArgs a, int i, double *dp64, int32_t *bp) {
    if (*(volatile const int *)a.abort_flag) return;  // a wait gave up: the tables are not valid
    // A warp takes 32 listed outputs at a time and evaluates their members flattened
    // (member r of the 32 outputs' lists goes to lane r mod 32), so every lane of a
    // binary64 sequence does useful work; then each output's lane takes the least value,
    // lowest k on ties, over its own members (the per-output rule, which is order-free).
    __shared__ double sval[4][32 * NMEM];
    __shared__ int32_t sk[4][32 * NMEM];
    const int n = a.list_cnt[2 * i];
    const int32_t *list = layer_list(a, i, 0);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    unsigned long long nres = 0;
    int nviol = 0;
    const int wstride = gridDim.x * (blockDim.x >> 5) * 32;
    for (int base = (blockIdx.x * (blockDim.x >> 5) + wid) * 32; base < n; base += wstride) {  // warp-uniform
        const int e = base + lane;
        int g = 0, cnt = 0;
        int64_t j = 0;
        long long o = 0;
        if (e < n) {
            const int32_t v = list[e];
            g = v >> 24;
            j = v & 0xFFFFFF;
            o = (long long)oidx(a, g, i, j);
            cnt = a.mcnt[o];
        }
        int off = cnt;  // inclusive, then exclusive prefix of the member counts
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            const int t = __shfl_up_sync(0xffffffffu, off, d);
            if (lane >= d) off += t;
        }
        const int total = __shfl_sync(0xffffffffu, off, 31);
        off -= cnt;
        for (int rb = 0; rb < total; rb += 32) {  // warp-uniform
            const int r = rb + lane;
            int ow = 0;  // the last lane whose offset is <= r: the owner of member r
#pragma unroll
            for (int st = 16; st > 0; st >>= 1) {
                const int oc = __shfl_sync(0xffffffffu, off, ow + st);
                if (oc <= r) ow += st;
            }
            const int og = __shfl_sync(0xffffffffu, g, ow);
            const int64_t oj = __shfl_sync(0xffffffffu, j, ow);
            const long long oo = __shfl_sync(0xffffffffu, o, ow);
            const int q = r - __shfl_sync(0xffffffffu, off, ow);
            if (r < total) {
                const int32_t k = a.members[(size_t)oo * NMEM + q];
                sk[wid][r] = k;
                sval[wid][r] = exact_value(P, dp64 + oidx(a, og, i - 1, 0), k, oj, a.prm->lam64[og]);
            }
        }
        __syncwarp();
        if (cnt > 0) {
            double best = CUDART_INF;
            int32_t arg = INT32_MAX;
            for (int q = 0; q < cnt; q++) {
                const double c = sval[wid][off + q];
                const int32_t k = sk[wid][off + q];
                if (c < best || (c == best && k < arg)) { best = c; arg = k; }
            }
            nres += cnt;
            nviol += exact_store(a, g, i, j, best, arg, dp64, bp) ? 0 : 1;
        } else if (e < n) {
            nviol += exact_store(a, g, i, j, CUDART_INF, INT32_MAX, dp64, bp) ? 0 : 1;
        }
        __syncwarp();  // the staging slots are free for the next 32 outputs
    }
    count_exact(a, nres, nviol);
}

// Layer i, outputs with more members: one warp each (fp32 re-evaluation within the
// band by warp_visit_band, whose decisions are the closure stage's; exact re-scoring of
// the members met), then the lanes' results meet (value, then lowest k).  The members
// met wait in the warp's queue, and each time it holds 32 every lane re-scores one of
// them in binary64, so the binary64 sequence runs with all lanes busy (the result,
// least value then lowest k, does not depend on the order).
__global__ void __launch_bounds__(128) k_exact_big(Prefix P, FastArgs a, int i, double *dp64, int32_t *bp) {
    if (*(volatile const int *)a.abort_flag) return;  // a wait gave up: the tables are not valid
    __shared__ int32_t queue[4][32];  // per warp: band members waiting for binary64 re-scoring
    const int n = a.list_cnt[2 * i + 1];
    const int32_t *list = layer_list(a, i, 1);
    const int lane = threadIdx.x & 31;
    const unsigned lt = (1u << lane) - 1u;
    int32_t *qw = queue[threadIdx.x >> 5];
    const int warps = gridDim.x * (blockDim.x >> 5);
    unsigned long long nres = 0;
    int nviol = 0;
    for (int e = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); e < n; e += warps) {
        const int32_t v = list[e];
        const int g = v >> 24;
        const int64_t j = v & 0xFFFFFF;
        const size_t o = oidx(a, g, i, j);
        const float m32 = a.dp32[d32(a, g, i, j)];
        const float thr = band_threshold(a, i, m32);
        const uint64_t w = a.band[o];
        const double lam = a.prm->lam64[g];
        const double *prev = dp64 + oidx(a, g, i - 1, 0);
        double best = CUDART_INF;
        int32_t arg = INT32_MAX;
        int qn = 0;  // warp-uniform queue length
        // The closure stage kept the band's fp32 argmin kb in the member slot 0; its binary64
        // value b0 bounds the binary64 minimum from above.  Every fp32 candidate value is within
        // eps_i (relative) of the candidate's exact (real) value V, so V >= val32 / (1 + eps_i);
        // a binary64 candidate is within far less than 2^-40 of V (a few correctly rounded
        // operations per layer on non-negative terms, s <= 256 layers).  So a member with
        // val32 > b0 (1 + eps_i + 2^-30) has V > b0 (1 + 2^-31) and a binary64 value above b0:
        // it can neither be the minimum nor tie it, and is not re-scored.
        const int32_t kb = a.members[o * NMEM];
        double b0 = CUDART_INF;
        if (lane == 0 && kb >= 0) b0 = exact_value(P, prev, kb, j, lam);
        b0 = __shfl_sync(0xffffffffu, b0, 0);
        if (lane == 0 && kb >= 0) { best = b0; arg = kb; nres++; }
        const float thr2 = b0 < CUDART_INF
                               ? __double2float_ru(__dmul_ru(b0, __dadd_ru(1.0 + 0x1p-30, (double)a.prm->eps[i])))
                               : CUDART_INF_F;
        warp_visit_band(a, g, i, j, w, thr, [&](bool in0, int64_t k, float v) {
            const bool in = in0 && v <= thr2 && (int32_t)k != kb;
            const unsigned mask = __ballot_sync(0xffffffffu, in);
            if (!mask) return;
            const int cnt = __popc(mask), pos = qn + __popc(mask & lt);
            if (in && pos < 32) qw[pos] = (int32_t)k;
            __syncwarp();
            if (qn + cnt >= 32) {
                exact_candidate(P, prev, qw[lane], j, lam, best, arg);
                nres++;
                __syncwarp();
                if (in && pos >= 32) qw[pos - 32] = (int32_t)k;
                __syncwarp();
                qn += cnt - 32;
            } else {
                qn += cnt;
            }
        });
        if (lane < qn) {
            exact_candidate(P, prev, qw[lane], j, lam, best, arg);
            nres++;
        }
        __syncwarp();  // the queue is free for the warp's next output
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            const double b2 = __shfl_xor_sync(0xffffffffu, best, off);
            const int32_t a2 = __shfl_xor_sync(0xffffffffu, arg, off);
            if (b2 < best || (b2 == best && a2 < arg)) { best = b2; arg = a2; }
        }
        if (lane == 0) nviol += exact_store(a, g, i, j, best, arg, dp64, bp) ? 0 : 1;
    }
    count_exact(a, nres, nviol);
}

// ------------------------------------------------------------------ host
__global__ void k_weights_f32(const int64_t *w, float *wf, int64_t p) {
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i < p) wf[i] = (float)w[i];
}

__global__ void k_store_params(FastParams prm, FastParams *dst) {
    if (threadIdx.x == 0 && blockIdx.x == 0) *dst = prm;
}

static int mdp_stride(int s) { return (s + 1 + 3) & ~3; }

// The band region: band words, member lists, need marks, flags, constants, corner
// states, block minima, the exact stage's lists; then the seed rows (cons_seed).
static size_t band_core_bytes(int64_t d, int32_t s) {
    size_t rows = (size_t)kMaxG * (size_t)(s + 1) * (size_t)table_stride(d);
    size_t nJ = (size_t)cdiv(d, BJ);
    return align256(8 * rows) + align256(4 * rows) + align256(4 * NMEM * rows) + align256(rows) +
           align256(8 * (size_t)kMaxG * nJ + 64) + align256(sizeof(FastParams)) + align256(32 * nJ * (nJ + 1) / 2) +
           align256(4 * (size_t)kMaxG * (size_t)mdp_stride(s) * nJ) +
           align256(2 * 4 * (size_t)kMaxG * (size_t)(s + 1) * (size_t)table_stride(d)) +
           align256(4 * 2 * (size_t)(s + 1)) + align256(4 * (size_t)kMaxG * (size_t)table_stride(d)) +
           align256(4 * (size_t)(s + 1));
}
static size_t seed_rows_bytes(int64_t d, int32_t s) { return align256(4 * (size_t)cdiv(d, BJ) * BJ * (size_t)(s + 1)); }
size_t fast_dp_band_bytes(int64_t d, int32_t s) { return band_core_bytes(d, s) + seed_rows_bytes(d, s); }
static float *seed_rows(void *ws, const Layout &Lw) {
    return reinterpret_cast<float *>(wsp<char>(ws, Lw.band) + band_core_bytes(Lw.d, Lw.s));
}

// Keep the fp32 dp rows of multiplier g of the last pass (G multipliers over p values) as
// the seed rows of a later pass at multipliers <= this one's (cons_seed).
int save_dp_seed(void *ws, const Layout &Lw, int64_t p, int G, int s, int g, cudaStream_t st) {
    if (g < 0 || g >= G || s != Lw.s) return ECASQ_EINVAL;
    const size_t row = (size_t)(s + 1) * BJ * sizeof(float);
    const float *src = wsp<float>(ws, Lw.dp32) + (size_t)g * (s + 1) * BJ;
    ECASQ_CUDA_TRY(cudaMemcpy2DAsync(seed_rows(ws, Lw), row, src, row * (size_t)G, row, (size_t)cdiv(p, BJ),
                                     cudaMemcpyDeviceToDevice, st));
    return ECASQ_OK;
}

static size_t smem_bytes(int Gc, int s) { return sizeof(Smem) + (size_t)2 * Gc * (s - 2) * BK * sizeof(float); }

// Certified band factors (see the file header): eps_2 = 1.0001u, eps_i = max(eps_{i-1}, 24u) + 1.0001u.
static void band_factors(int s, FastParams &fp) {
    const double u = 1.0 / 16777216.0;
    for (int i = 0; i <= kMaxS; i++) { fp.tau[i] = 0.f; fp.eps[i] = 0.f; }
    double eps = 1.0001 * u;
    fp.eps[2] = (float)eps;
    for (int i = 3; i <= s; i++) {
        eps = std::max(eps, 24.0 * u) + 1.0001 * u;
        fp.eps[i] = (float)eps;
        fp.tau[i] = (float)(2.0 * eps / (1.0 - eps) * 1.001 + 2.0 * u);
    }
}

// The resident table: every tile's C and Phi rows, then every tile's column summary
// (BJ float2), both indexed by J(J+1)/2 + K with J < ceil(d / 64).
size_t resident_costs_bytes(int64_t d) {
    if (d < 1) return 0;
    double nJ = (double)cdiv(d, BJ);
    double bytes = nJ * (nJ + 1.0) * 0.5 * ((double)kCostTileFloats * sizeof(float) + BJ * sizeof(float2));
    if (!(bytes < 9.0e18)) return 0;
    size_t n = (size_t)cdiv(d, BJ);
    return n * (n + 1) / 2 * (kCostTileFloats * sizeof(float) + BJ * sizeof(float2));
}

// Streamed interval costs: the cost tiles of a band of column blocks at a time, in a
// buffer of streamed_costs_bytes(d) (tiles, then their column summaries).  The band
// holds up to 64 full columns of tiles, so a band near the end of the triangle still
// has 64 blocks (times the multiplier splits) to spread over the SMs.
static size_t tile_bytes_with_summary() { return kCostTileFloats * sizeof(float) + BJ * sizeof(float2); }
size_t streamed_costs_bytes(int64_t d) {
    if (d < 1) return 0;
    const size_t nJ = (size_t)cdiv(d, BJ);
    const size_t full = nJ * (nJ + 1) / 2, band = std::min(full, (size_t)64 * nJ);
    return band * tile_bytes_with_summary();
}

int launch_dp_fast(const Prefix &P, const double *lamp, int G, int s, void *ws, const Layout &Lw, cudaStream_t st,
                   bool exact_s, bool exact_tables, float *costs, bool build_costs, bool test_stall,
                   size_t chunk_bytes, bool split_off, bool seeded) {
    double *dp64 = wsp<double>(ws, Lw.dp64);
    int32_t *bp = wsp<int32_t>(ws, Lw.bp);
    // small inputs, very large ones and huge counts take the reference kernel
    if (P.p < 2 * BJ || P.p > kMaxFastP || P.d >= (1 << 24) || s < 3 || cdiv(s - 2, LPT) * NJQ > MAXCONS)
        return launch_dp_reference(P, lamp, G, s, dp64, bp, st);
    FastArgs a{};
    a.v = P.v;
    a.N = P.N;
    a.S = P.S;
    a.S2 = P.S2;
    a.p = P.p;
    a.d = P.d;
    a.ps = P.ps;
    a.invd = 1.0f / (float)P.d;  // IEEE division on the host: correctly rounded
    a.G = G;
    a.s = s;
    // Layers per consumer thread: LPT, or 8 on the generic path (the fused kernel, or the
    // resident one without the paired diagonal) when that costs fewer layer slots times
    // multiplier splits; at s = 32, 4 groups of 8 layers (64 threads per multiplier, 4
    // multipliers per split) against 5 of 7 (80 threads, 3 per split): 2 splits of 8
    // slots per pass instead of 3 of 7.  With resident or streamed costs, also when 8
    // layers give an even number of layer groups and LPT an odd one or more than two:
    // only then can the generic path skip tiles (s = 17, 18; s = 27..30 with several
    // multipliers, where the slots favour LPT).  A single multiplier at s = 27..34 keeps
    // LPT: with one warp pair per block the skipping did not pay for the eighth layer.
    int lp = LPT;
    if (!(costs && cdiv(s - 2, LPT) == 2 && mdp_stride(s) <= 20)) {
        auto slots = [&](int l) {
            const int lgc = (int)cdiv(s - 2, l), gc = std::max(1, std::min(G, MAXCONS / (lgc * NJQ)));
            return (int64_t)cdiv(G, gc) * l;
        };
        const int lg8 = (int)cdiv(s - 2, 8);
        const bool skip8 = costs && lg8 % 2 == 0 && mdp_stride(s) <= kMdpMax && (lg8 == 2 || G > 1);
        if (cdiv(s - 2, 8) * NJQ <= MAXCONS && (skip8 || slots(8) < slots(LPT))) lp = 8;
    }
    a.lgc = (int)cdiv(s - 2, lp);
    a.Gc = std::max(1, std::min(G, MAXCONS / (a.lgc * NJQ)));
    a.nsplit = (int)cdiv(G, a.Gc);
    a.nJ = (int)cdiv(P.p, BJ);
    a.ncons = (int)cdiv((int64_t)a.Gc * a.lgc * NJQ, 32) * 32;
    FastParams fp;
    band_factors(s, fp);
    for (int g = 0; g < kMaxG; g++) {
        fp.lam64[g] = g < G ? lamp[g] : 0.0;
        fp.lam32[g] = (float)fp.lam64[g];
    }
    size_t rows = (size_t)kMaxG * (size_t)(s + 1) * (size_t)table_stride(Lw.d);
    char *base = wsp<char>(ws, Lw.band);
    a.dp32 = wsp<float>(ws, Lw.dp32);
    a.band = reinterpret_cast<uint64_t *>(base);
    base += align256(8 * rows);
    a.mcnt = reinterpret_cast<int32_t *>(base);
    base += align256(4 * rows);
    a.members = reinterpret_cast<int32_t *>(base);
    base += align256(4 * NMEM * rows);
    a.need = reinterpret_cast<uint8_t *>(base);
    base += align256(rows);
    int *flags = reinterpret_cast<int *>(base);  // done [kMaxG][nJ], half [kMaxG][nJ], ticket, abort
    base += align256(8 * (size_t)kMaxG * (size_t)cdiv(Lw.d, BJ) + 64);
    FastParams *dprm = reinterpret_cast<FastParams *>(base);
    base += align256(sizeof(FastParams));
    a.corner = reinterpret_cast<float *>(base);
    {
        size_t nJd = (size_t)cdiv(Lw.d, BJ);
        char *q = base + align256(32 * nJd * (nJd + 1) / 2);
        a.mdp = reinterpret_cast<float *>(q);
        q += align256(4 * (size_t)kMaxG * (size_t)mdp_stride(s) * nJd);
        a.lists = reinterpret_cast<int32_t *>(q);
        q += align256(2 * 4 * (size_t)kMaxG * (size_t)(s + 1) * (size_t)table_stride(Lw.d));
        a.list_cnt = reinterpret_cast<int *>(q);
        q += align256(4 * 2 * (size_t)(s + 1));
        a.wide = reinterpret_cast<int32_t *>(q);
        q += align256(4 * (size_t)kMaxG * (size_t)table_stride(Lw.d));
        a.wide_cnt = reinterpret_cast<int *>(q);
    }
    a.mdp_stride = mdp_stride(s);
    a.spin_limit = test_stall ? kTestSpinLimit : kSpinLimit;
    // two-part publishing of each block (the chain's last tile in two layer groups)
    a.split_pub = (costs && lp == LPT && a.lgc == 2 && !split_off) ? 1 : 0;
    a.hold0 = test_stall ? 1 : 0;
    // Tile skipping needs every warp to hold whole multipliers (its batch test is a warp
    // vote), so an even number of layer groups (16-thread groups, 32-lane warps), and a
    // diagonal that writes the blocks' minima: the paired one (LPT layers per thread, two
    // groups) or the generic one with 8 layers per thread.
    a.prune = (costs && (lp == LPT ? a.lgc == 2 : a.lgc % 2 == 0) && a.mdp_stride <= kMdpMax &&
               a.Gc * a.mdp_stride <= kMaxG * 20) ? 1 : 0;
    const bool parked = costs && lp == LPT && a.lgc == 2;  // the paired diagonal and its parked state
    a.stage_tiles = lp == LPT ? 32 : 16;  // k_wavefront_res<LP>'s batch size
    a.seed = (seeded && a.prune && s == Lw.s) ? seed_rows(ws, Lw) : nullptr;
    a.costs = costs;
    a.tile_base = 0;
    a.J0 = 0;
    a.J1 = a.nJ;
    // tiles the costs buffer holds at once: the whole triangle, or (streamed) one band
    const size_t cap_tiles = chunk_bytes ? chunk_bytes / tile_bytes_with_summary()
                                         : (size_t)cdiv(Lw.d, BJ) * (size_t)(cdiv(Lw.d, BJ) + 1) / 2;
    if (costs) a.tsum = reinterpret_cast<float2 *>(costs + cap_tiles * kCostTileFloats);
    if (chunk_bytes && cap_tiles < (size_t)a.nJ) return ECASQ_EWORKSPACE;  // one column of tiles must fit
    a.prm = dprm;
    a.done = flags;
    a.half = flags + (size_t)kMaxG * a.nJ;
    a.ticket = a.half + (size_t)kMaxG * a.nJ;
    a.abort_flag = a.ticket + 1;
    a.st = wsp<DevStatus>(ws, Lw.status);
    float *wf = wsp<float>(ws, Lw.keys1);  // the sort's ping-pong buffer is free now
    a.wf = wf;
    size_t n = (size_t)G * (size_t)(s + 1) * (size_t)P.ps;
    note_launch();
    k_store_params<<<1, 32, 0, st>>>(fp, dprm);
    note_launch();
    k_fast_clear<<<4096, 256, 0, st>>>(dp64, bp, a.dp32, n);
    note_launch();
    k_weights_f32<<<(unsigned)cdiv(P.p, 256), 256, 0, st>>>(P.w, wf, P.p);
    ECASQ_LAUNCH_CHECK();
    ECASQ_CUDA_TRY(cudaMemsetAsync(flags, 0, sizeof(int) * (2 * (size_t)kMaxG * a.nJ + 2), st));
    note_launch();
    k_fast_base<<<(unsigned)cdiv(P.p - 1, 128), 128, 0, st>>>(P, a, dp64, bp);
    ECASQ_LAUNCH_CHECK();
    int dev = 0, nsm = 0;
    ECASQ_CUDA_TRY(cudaGetDevice(&dev));
    ECASQ_CUDA_TRY(cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev));
    // corner states: needed by every tile the producer computes (per pass, or once into the table)
    if (a.nJ > 1 && (!costs || build_costs)) {
        note_launch();
        k_corners<<<(unsigned)std::min<int64_t>(cdiv((int64_t)a.nJ * (a.nJ - 1) / 2, 128), 152 * 64), 128, 0, st>>>(a);
        ECASQ_LAUNCH_CHECK();
    }
    size_t smem = smem_bytes(a.Gc, s);
    const size_t stage_bytes = a.prune ? 2 * stage_floats(G, a.mdp_stride, a.stage_tiles) * sizeof(float) : 0;
    if (parked)  // parked band state; off the diagonal, the two stage buffers
        smem += std::max((size_t)3 * LPT * JPT * a.ncons * sizeof(uint32_t), stage_bytes);
    else
        smem += stage_bytes;
    auto wave = costs ? (lp == 8 ? k_wavefront_res<8> : k_wavefront_res<LPT>)
                      : (lp == 8 ? k_wavefront<8> : k_wavefront<LPT>);
    ECASQ_CUDA_TRY(cudaFuncSetAttribute(wave, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    int per_sm = 0;
    if (costs && build_costs)
        ECASQ_CUDA_TRY(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_build_costs, NPROD, 0));
    // one band of column blocks per round: [J0, J1) whose tiles fit the buffer (all of them
    // when the buffer holds the whole triangle); with streamed costs every band's tiles are
    // built just before its wavefront, else the table is built once per call.  The
    // timer covers the min-plus kernel; with streamed costs, every band's build and
    // wavefront together (the builds are then part of every pass)
    if (chunk_bytes) timer_begin(st);
    for (int J0 = 0; J0 < a.nJ;) {
        int J1 = a.nJ;
        if (chunk_bytes) {
            J1 = J0 + 1;
            const size_t T0 = (size_t)J0 * (J0 + 1) / 2;
            while (J1 < a.nJ && (size_t)(J1 + 1) * (J1 + 2) / 2 - T0 <= cap_tiles) J1++;
        }
        a.J0 = J0;
        a.J1 = J1;
        a.tile_base = chunk_bytes ? (size_t)J0 * (J0 + 1) / 2 : 0;
        if (costs && build_costs) {
            const int64_t ntiles = (int64_t)J1 * (J1 + 1) / 2 - (int64_t)a.tile_base;
            note_launch();
            k_build_costs<<<(unsigned)std::min<int64_t>(ntiles, (int64_t)nsm * std::max(per_sm, 1)), NPROD, 0, st>>>(
                a, costs);
            ECASQ_LAUNCH_CHECK();
        }
        if (J0 > 0) ECASQ_CUDA_TRY(cudaMemsetAsync(a.ticket, 0, sizeof(int), st));
        int grid = std::min(nsm, (J1 - J0) * a.nsplit);
        if (!chunk_bytes) timer_begin(st);
        note_launch();
        wave<<<grid, (costs ? 0 : NPROD) + a.ncons, smem, st>>>(a);
        if (!chunk_bytes) timer_end(st);
        ECASQ_LAUNCH_CHECK();
        J0 = J1;
    }
    if (chunk_bytes) timer_end(st);
    // a streamed band holds only the last band's tiles: the need and exact stages re-derive
    // the costs they read (any evaluation within the certified bound will do)
    if (chunk_bytes) {
        a.costs = nullptr;
        a.tile_base = 0;
    }
    const int ilo = exact_s ? s : 2;
    note_launch();
    k_need_init<<<(unsigned)std::min<int64_t>(cdiv((int64_t)G * (s + 1) * P.ps, 256), (int64_t)nsm * 32), 256, 0, st>>>(
        a, ilo, exact_tables ? 1 : 0);
    ECASQ_LAUNCH_CHECK();
    ECASQ_CUDA_TRY(cudaMemsetAsync(a.list_cnt, 0, sizeof(int) * 2 * (size_t)(s + 1), st));
    ECASQ_CUDA_TRY(cudaMemsetAsync(a.wide_cnt, 0, sizeof(int) * (size_t)(s + 1), st));
    const unsigned gl = (unsigned)std::min<int64_t>(cdiv((int64_t)G * P.p, 128), (int64_t)nsm * 64);
    for (int i = s; i >= 3; i--) {
        note_launch();
        k_need_layer<<<gl, 128, 0, st>>>(a, i);
        ECASQ_LAUNCH_CHECK();
        note_launch();
        k_need_wide<<<(unsigned)nsm * 16, 128, 0, st>>>(a, i);
        ECASQ_LAUNCH_CHECK();
    }
    note_launch();
    k_fill_unneeded<<<(unsigned)std::min<int64_t>(cdiv((int64_t)G * (s + 1) * P.ps, 256), (int64_t)nsm * 32), 256, 0,
                      st>>>(a, dp64, bp);
    ECASQ_LAUNCH_CHECK();
    for (int i = 3; i <= s; i++) {
        note_launch();
        k_exact_small<<<(unsigned)nsm * 8, 128, 0, st>>>(P, a, i, dp64, bp);
        ECASQ_LAUNCH_CHECK();
        note_launch();
        k_exact_big<<<(unsigned)nsm * 16, 128, 0, st>>>(P, a, i, dp64, bp);
        ECASQ_LAUNCH_CHECK();
    }
    return ECASQ_OK;
}

}  // namespace ecasq
