// api.cu -- the extern "C" entry points of include/ecasq.h and the host-side
// drivers: workspace carving, the multiplier search, the refinement loop.
#include <math.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <mutex>
#include <vector>

#include "common.cuh"

namespace ecasq {

// launchers defined in the other translation units
int launch_dp_reference(const Prefix &P, const double *lamp, int G, int s, double *dp64, int32_t *bp,
                        cudaStream_t st);
int launch_dp_fast(const Prefix &P, const double *lamp, int G, int s, void *ws, const Layout &L, cudaStream_t st,
                   bool exact_s, bool exact_tables, float *costs, bool build_costs, bool test_stall,
                   size_t chunk_bytes, bool split_off, bool seeded);
int save_dp_seed(void *ws, const Layout &Lw, int64_t p, int G, int s, int g, cudaStream_t st);
size_t resident_costs_bytes(int64_t d);
size_t streamed_costs_bytes(int64_t d);
int launch_rows_prepare(const float *X, int64_t rows, const RowsData &R, cudaStream_t st);
int launch_grid_prefix(const float *P, int64_t n, const float *vX, const int64_t *NX, const double *SX,
                       const double *S2X, int64_t pX, float *v, int64_t *w, int64_t *N, double *S, double *S2,
                       DevStatus *st, cudaStream_t stream);
int launch_rows_pass(const RowsPass &A, int nact, int pmax, cudaStream_t st);
int launch_rows_gather(const RowsData &R, const int32_t *a, const int32_t *m, int64_t rows, int s, float *Q,
                       cudaStream_t st);
int launch_traceback_eval(const Prefix &P, int G, int s, int exact_s, const double *dp64, const int32_t *bp,
                          int32_t *qidx, int32_t *mcount, double *metrics, cudaStream_t st);
int launch_eval_codebook(const Prefix &P, const int32_t *a, int m, double *out3, cudaStream_t st,
                         const int32_t *gate = nullptr);
int launch_gather_q(const float *v, const int32_t *qidx, const int32_t *mcount, int G, int s, float *Q,
                    cudaStream_t st);
int launch_locate_q(const float *v, int64_t p, const float *Q, int m, int32_t *a, DevStatus *ds, cudaStream_t st);
size_t refine_ctx_bytes();
int launch_refine_colour(const Prefix &P, const int32_t *a, int m, int colour, double lamp, int32_t *a_new,
                         int32_t *moved, void *part_buf, int32_t *ctx, cudaStream_t st, int *nblocks_out);
size_t refine_scratch_bytes(int64_t d);
int launch_refine_commit(int32_t *a, const int32_t *a_new, const int32_t *moved, const double *ev, int m, bool guard,
                         double budget, int32_t *ctx, cudaStream_t st);
int launch_quantize(const float *x, int64_t d, const float *Q, int m, uint64_t seed, uint8_t *idx, uint32_t *counts,
                    DevStatus *st, int num_sms, cudaStream_t stream);
int launch_quantize_timeshare(const float *x, int64_t d, const float *Qm, int mm, const float *Qp, int mp,
                              double beta, uint64_t seed, uint64_t seed_ts, uint8_t *idx, uint8_t *sel,
                              uint32_t *counts, DevStatus *st, int num_sms, cudaStream_t stream);
size_t fast_dp_band_bytes(int64_t d, int32_t s);
size_t grid_pairs_bytes(int64_t n);
int launch_dp_grid(const Prefix &P, const double *lamp, int G, int s, double *dp64, int32_t *bp, float *dp32,
                   void *pairs, bool build_pairs, int num_sms, cudaStream_t st);
size_t opt_pairs_bytes(int64_t n);
size_t opt_tables_bytes(int64_t n, int s, int G);
int launch_opt_dp(const Prefix &P, const double *lamp, int G, int s, int exact_s, void *pairs, bool build_pairs,
                  void *tables, int32_t *qidx, int32_t *mcount, double *metrics, int num_sms, cudaStream_t st);

int launch_dp_linear(const Prefix &P, double lam, int s, int exact_s, double *rows, double *col, void *small,
                     std::vector<int32_t> &qidx_host, int *m_out, double *best, cudaStream_t st);

static std::atomic<long long> g_launches{0};
void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

// CUDA events around the min-plus kernel when ECASQ_TIME_KERNELS is set.
struct KernelTimer {
    bool on = false;
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    double ms = 0.0;
    int launches = 0;
};
static thread_local KernelTimer g_timer;
void timer_begin(cudaStream_t st) {
    if (!g_timer.on) return;
    if (!g_timer.e0) { cudaEventCreate(&g_timer.e0); cudaEventCreate(&g_timer.e1); }
    cudaEventRecord(g_timer.e0, st);
}
void timer_end(cudaStream_t st) {
    if (!g_timer.on) return;
    cudaEventRecord(g_timer.e1, st);
}
static void timer_collect() {
    if (!g_timer.on || !g_timer.e0) return;
    float ms = 0.f;
    if (cudaEventSynchronize(g_timer.e1) == cudaSuccess && cudaEventElapsedTime(&ms, g_timer.e0, g_timer.e1) == cudaSuccess) {
        g_timer.ms += ms;
        g_timer.launches += 1;
    }
}

size_t make_layout(int64_t d, int32_t s, int64_t rows, Layout *L) {
    (void)rows;
    size_t off = 0;
    auto take = [&](size_t bytes) { size_t o = off; off += align256(bytes); return o; };
    int64_t nb = cdiv(d, kSortTile), nbs = cdiv(d, kScanTile);
    size_t rowsz = (size_t)kMaxG * (size_t)(s + 1) * (size_t)table_stride(d);
    L->status = take(sizeof(DevStatus));
    L->keys0 = take(4 * (size_t)d);
    L->keys1 = take(4 * (size_t)d);
    L->rcount = take(4 * 256 * (size_t)nb);
    L->head = 0;
    L->v = take(4 * (size_t)d);
    L->w = take(8 * (size_t)d);
    L->N = take(8 * (size_t)(d + 1));
    L->S = take(16 * (size_t)(d + 1));
    L->S2 = take(16 * (size_t)(d + 1));
    L->part = take(48 * (size_t)nbs);
    L->dp64 = take(8 * std::max(rowsz, (size_t)4 * (size_t)(d + 1)));
    L->bp = take(4 * rowsz);
    L->dp32 = take(4 * rowsz);
    L->qidx = take(4 * (size_t)kMaxG * kMaxS);
    L->mcount = take(4 * (size_t)kMaxG);
    L->metrics = take(8 * (size_t)kMaxG * 4);
    L->lam = take(8 * (size_t)kMaxG);
    L->refine = take(4 * 2 * kMaxS + 256 + 8 * 8 + refine_ctx_bytes());
    L->refine_part = take(refine_scratch_bytes(d));
    L->band = take(fast_dp_band_bytes(d, s));
    L->costs = 0;
    L->costs_bytes = 0;
    L->costs_streamed = false;
    L->gpairs = 0;
    L->gpairs_bytes = 0;
    L->total = off;
    L->d = d;
    L->s = s;
    return off;
}

// Only what the sort, histogram and prefix sums use (ecasq_prepare): the regions of
// make_layout up to the scan partials, then a 32 (d+1)-byte scratch in place of the
// DP tables (the fp64 sums before their double-double split).
static size_t make_prep_layout(int64_t d, Layout *L) {
    memset(L, 0, sizeof(*L));
    size_t off = 0;
    auto take = [&](size_t bytes) { size_t o = off; off += align256(bytes); return o; };
    int64_t nb = cdiv(d, kSortTile), nbs = cdiv(d, kScanTile);
    L->status = take(sizeof(DevStatus));
    L->keys0 = take(4 * (size_t)d);
    L->keys1 = take(4 * (size_t)d);
    L->rcount = take(4 * 256 * (size_t)nb);
    L->v = take(4 * (size_t)d);
    L->w = take(8 * (size_t)d);
    L->N = take(8 * (size_t)(d + 1));
    L->S = take(16 * (size_t)(d + 1));
    L->S2 = take(16 * (size_t)(d + 1));
    L->part = take(48 * (size_t)nbs);
    L->dp64 = take(8 * 4 * (size_t)(d + 1));
    L->total = off;
    L->d = d;
    L->s = 2;
    return off;
}

static int g_num_sms = 0;
static int num_sms() {
    if (g_num_sms == 0) {
        int dev = 0, n = 0;
        if (cudaGetDevice(&dev) == cudaSuccess && cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess)
            g_num_sms = n;
        else
            g_num_sms = 152;
    }
    return g_num_sms;
}

// Scratch of ecasq_quantize_noalloc: one status record in a fixed block of
// this library's device memory (no allocation at call time).  The record's
// range-error flag must read zero when the kernel starts.
constexpr size_t kNoAllocScratchBytes = 256;
static_assert(sizeof(DevStatus) <= kNoAllocScratchBytes, "status record larger than the fixed scratch block");
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];
constexpr int kNoAllocMaxDevices = 64;
static std::mutex g_noalloc_mu;
static void *g_noalloc_addr[kNoAllocMaxDevices];

// Device address of the scratch block on the current device, looked up once
// per device (cudaGetSymbolAddress) and kept.  `st` must belong to that device.
static int noalloc_scratch(cudaStream_t st, void **out) {
    int dev = -1, sdev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kNoAllocMaxDevices) return ECASQ_ECUDA;
    if (cudaStreamGetDevice(st, &sdev) != cudaSuccess) return ECASQ_ECUDA;
    if (sdev != dev) return ECASQ_EINVAL;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_addr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return ECASQ_ECUDA;
        g_noalloc_addr[dev] = p;
    }
    *out = g_noalloc_addr[dev];
    return ECASQ_OK;
}

// Batched short rows (d <= kScanTile): per-row prefix data, pass scratch and
// results, placed after the single-row layout (which the rows that cannot take the
// batched path still use).
struct RowsLayout {
    size_t v, w, N, S, S2, p, norm2, nonfinite, bp, lam, act, mcount, metrics, qidx, sel, m, pairs, total;
    int64_t pstride;
};
static size_t rows_layout(int64_t d, int32_t s, int64_t rows, RowsLayout *R) {
    size_t off = 0;
    auto take = [&](size_t bytes) { size_t o = off; off += align256(bytes); return o; };
    const size_t n = (size_t)rows, dc = (size_t)d;
    R->v = take(4 * n * dc);
    R->w = take(8 * n * dc);
    R->N = take(8 * n * (dc + 1));
    R->S = take(16 * n * (dc + 1));
    R->S2 = take(16 * n * (dc + 1));
    R->p = take(8 * n);
    R->norm2 = take(8 * n);
    R->nonfinite = take(4 * n);
    R->bp = take(4 * n * kMaxG * (size_t)(s + 1) * dc);
    R->lam = take(8 * n * kMaxG);
    R->act = take(4 * n);
    R->mcount = take(4 * n * kMaxG);
    R->metrics = take(32 * n * kMaxG);
    R->qidx = take(4 * n * kMaxG * (size_t)s);
    R->sel = take(4 * n * (size_t)s);
    R->m = take(4 * n);
    const int64_t pm = std::min<int64_t>(d, kRowsMaxP);
    // binary64 {C, Phi} by pair, Phi^first, fp32 {C, Phi} by pair; even, so rows start on 16 bytes
    R->pstride = (3 * (pm * (pm - 1) / 2) + pm + 1) & ~(int64_t)1;
    R->pairs = take(8 * n * (size_t)R->pstride);
    R->total = off;
    return off;
}
static size_t rows_region_bytes(int64_t d, int32_t s, int64_t rows) {
    if (d > kScanTile) return 0;
    RowsLayout R;
    return rows_layout(d, s, rows, &R);
}

// ECASQ_RESIDENT_COSTS: the interval-cost tiles follow the common layout;
// ECASQ_STREAMED_COSTS (without RESIDENT): a buffer for one band of tiles there instead.
static int add_resident_costs(uint32_t flags, Layout *L) {
    if (!(flags & (ECASQ_RESIDENT_COSTS | ECASQ_STREAMED_COSTS))) return ECASQ_OK;
    const bool streamed = !(flags & ECASQ_RESIDENT_COSTS);
    size_t cb = streamed ? streamed_costs_bytes(L->d) : resident_costs_bytes(L->d);
    if (!cb || L->total > SIZE_MAX - align256(cb)) return ECASQ_EINVAL;
    L->costs = L->total;
    L->costs_bytes = cb;
    L->costs_streamed = streamed;
    L->total += align256(cb);
    return ECASQ_OK;
}

static int check_ws(const void *ws, size_t bytes, const Layout &L) {
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255) != 0 || bytes < L.total) return ECASQ_EWORKSPACE;
    return ECASQ_OK;
}

static Prefix make_prefix(void *ws, const Layout &L, int64_t p, int64_t d) {
    Prefix P;
    P.v = wsp<float>(ws, L.v);
    P.w = wsp<int64_t>(ws, L.w);
    P.N = wsp<int64_t>(ws, L.N);
    P.S = wsp<double>(ws, L.S);
    P.S2 = wsp<double>(ws, L.S2);
    P.p = p;
    P.d = d;
    P.ps = table_stride(p);
    return P;
}

// The 7 interior points of [lo, hi] from three levels of geometric midpoints
// sqrt(a*b): correctly rounded multiply and sqrt only.
static void midpoints7(double lo, double hi, double *t) {
    t[3] = sqrt(lo * hi);
    t[1] = sqrt(lo * t[3]);
    t[5] = sqrt(t[3] * hi);
    t[0] = sqrt(lo * t[1]);
    t[2] = sqrt(t[1] * t[3]);
    t[4] = sqrt(t[3] * t[5]);
    t[6] = sqrt(t[5] * hi);
}

struct PassOut {
    std::vector<int32_t> qidx;  // G * s
    std::vector<int32_t> m;     // G
    std::vector<double> met;    // G * 4
};

// One DP pass over a prepared workspace: DP at lambda'_g (g < G), traceback,
// evaluation, results to the host.
// costs_built: in/out, whether the resident interval costs (if the layout has
// them) already hold this call's prefix data.
// seeded: the workspace's seed rows hold an earlier pass's fp32 minima at a multiplier
// >= every multiplier of this pass (save_dp_seed); the fast kernel's tile skipping
// starts from them.
static int dp_pass_prepared(void *ws, const Layout &L, const Prefix &P, int s, const double *lamp, int G,
                            uint32_t flags, cudaStream_t st, PassOut &out, bool *costs_built, bool seeded = false) {
    double *dp64 = wsp<double>(ws, L.dp64);
    int32_t *bp = wsp<int32_t>(ws, L.bp);
    int rc;
    if (flags & ECASQ_DP_REFERENCE) {
        rc = launch_dp_reference(P, lamp, G, s, dp64, bp, st);
    } else if (L.gpairs_bytes) {
        rc = launch_dp_grid(P, lamp, G, s, dp64, bp, wsp<float>(ws, L.dp32), wsp<void>(ws, L.gpairs), !*costs_built,
                            num_sms(), st);
        if (rc == ECASQ_OK) *costs_built = true;
    } else {
        float *costs = L.costs_bytes ? wsp<float>(ws, L.costs) : nullptr;
        // streamed costs are rebuilt band by band in every pass
        rc = launch_dp_fast(P, lamp, G, s, ws, L, st, (flags & ECASQ_EXACT_S) != 0, (flags & ECASQ_EXACT_TABLES) != 0,
                            costs, costs && (L.costs_streamed || !*costs_built), (flags & ECASQ_TEST_STALL) != 0,
                            L.costs_streamed ? L.costs_bytes : 0, (flags & ECASQ_ONE_PART_PUBLISH) != 0,
                            seeded && !(flags & ECASQ_UNSEEDED_SEARCH));
        if (costs && rc == ECASQ_OK) *costs_built = true;
    }
    if (rc != ECASQ_OK) return rc;
    timer_collect();
    rc = launch_traceback_eval(P, G, s, (flags & ECASQ_EXACT_S) ? 1 : 0, dp64, bp, wsp<int32_t>(ws, L.qidx),
                               wsp<int32_t>(ws, L.mcount), wsp<double>(ws, L.metrics), st);
    if (rc != ECASQ_OK) return rc;
    out.qidx.assign((size_t)G * s, 0);
    out.m.assign(G, 0);
    out.met.assign((size_t)G * 4, 0.0);
    ECASQ_CUDA_TRY(cudaMemcpyAsync(out.qidx.data(), wsp<int32_t>(ws, L.qidx), sizeof(int32_t) * G * s,
                                   cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(out.m.data(), wsp<int32_t>(ws, L.mcount), sizeof(int32_t) * G,
                                   cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(out.met.data(), wsp<double>(ws, L.metrics), sizeof(double) * G * 4,
                                   cudaMemcpyDeviceToHost, st));
    int32_t sg[2] = {s, G};
    int64_t dd_ = L.d;
    DevStatus *ds = wsp<DevStatus>(ws, L.status);
    ECASQ_CUDA_TRY(cudaMemcpyAsync(&ds->last_s, sg, sizeof(sg), cudaMemcpyHostToDevice, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(&ds->last_d, &dd_, sizeof(dd_), cudaMemcpyHostToDevice, st));
    DevStatus h;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(&h, ds, sizeof(DevStatus), cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    if (h.timeout) return ECASQ_ETIMEOUT;
    for (int g = 0; g < G; g++)
        if (out.m[g] < 1) return ECASQ_EINFEASIBLE;
    return ECASQ_OK;
}

static int64_t candidates_of(int64_t p, int s, int exact) {
    (void)exact;
    // eq. apx_rec evaluates, for layers i = 3..s, every k in [i-2, j-1], j in [i-1, p-1]
    int64_t c = 0;
    for (int i = 3; i <= s; i++) {
        int64_t n = p - (i - 1);  // number of j
        if (n <= 0) break;
        c += n * (n + 1) / 2;
    }
    return c;
}

// Upload a codebook (unique indices) and evaluate it: out3 = MSE, H(I,B), H(Xhat).
// With gate (device), the kernel evaluates only if *gate != 0 (else out3 is stale).
static int eval_device(void *ws, const Layout &L, const Prefix &P, const int32_t *a_dev, int m, cudaStream_t st,
                       double *out3_host, const int32_t *gate = nullptr) {
    double *o = reinterpret_cast<double *>(wsp<char>(ws, L.refine) + 4 * 2 * kMaxS + 256);
    int rc = launch_eval_codebook(P, a_dev, m, o, st, gate);
    if (rc != ECASQ_OK) return rc;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(out3_host, o, 3 * sizeof(double), cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    return ECASQ_OK;
}

// Three-colour refinement loop (Sec. 6) on the host; a_host in/out.
static int refine_device(void *ws, const Layout &L, const Prefix &P, std::vector<int32_t> &a_host, double lamp,
                         double budget, bool guard, int max_rounds, double tol, cudaStream_t st, int *rounds_used,
                         double *last_rel = nullptr) {
    int m = (int)a_host.size();
    *rounds_used = 0;
    if (last_rel) *last_rel = 0.0;
    if (m < 3 || max_rounds <= 0) return ECASQ_OK;
    int32_t *a = wsp<int32_t>(ws, L.refine);
    int32_t *an = a + kMaxS;
    int32_t *moved = an + kMaxS;
    // records of scans that kept their value (refine.cu), after the evaluation output
    int32_t *ctx = reinterpret_cast<int32_t *>(wsp<char>(ws, L.refine) + 4 * 2 * kMaxS + 256 + 8 * 8);
    ECASQ_CUDA_TRY(cudaMemsetAsync(ctx, 0, refine_ctx_bytes(), st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(a, a_host.data(), sizeof(int32_t) * m, cudaMemcpyHostToDevice, st));
    double ev[3];
    int rc = eval_device(ws, L, P, a, m, st, ev);
    if (rc != ECASQ_OK) return rc;
    double J = ev[0] + lamp * ev[2];
    double *evd = reinterpret_cast<double *>(wsp<char>(ws, L.refine) + 4 * 2 * kMaxS + 256);  // eval_device's output
    for (int r = 0; r < max_rounds; r++) {
        double J0 = J;
        for (int col = 0; col < 3; col++) {
            ECASQ_CUDA_TRY(cudaMemcpyAsync(an, a, sizeof(int32_t) * m, cudaMemcpyDeviceToDevice, st));
            ECASQ_CUDA_TRY(cudaMemsetAsync(moved, 0, sizeof(int32_t), st));
            int nblk = 0;
            rc = launch_refine_colour(P, a, m, col, lamp, an, moved, wsp<void>(ws, L.refine_part), ctx, st, &nblk);
            if (rc != ECASQ_OK) return rc;
            if (nblk == 0) continue;
            // only a step that moved a value is evaluated; the step is kept or dropped on the device
            rc = launch_eval_codebook(P, an, m, evd, st, moved);
            if (rc != ECASQ_OK) return rc;
            rc = launch_refine_commit(a, an, moved, evd, m, guard, budget, ctx, st);
            if (rc != ECASQ_OK) return rc;
        }
        rc = eval_device(ws, L, P, a, m, st, ev);
        if (rc != ECASQ_OK) return rc;
        J = ev[0] + lamp * ev[2];
        *rounds_used = r + 1;
        if (last_rel) *last_rel = J0 != 0.0 ? (J0 - J) / fabs(J0) : 0.0;
        if (!(J0 - J > tol * fabs(J0))) break;
    }
    ECASQ_CUDA_TRY(cudaMemcpyAsync(a_host.data(), a, sizeof(int32_t) * m, cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    return ECASQ_OK;
}

static int write_codebook(void *ws, const Layout &L, const std::vector<int32_t> &a, float *Q, cudaStream_t st) {
    int32_t *qi = wsp<int32_t>(ws, L.qidx);
    int32_t *mc = wsp<int32_t>(ws, L.mcount);
    int32_t m = (int32_t)a.size();
    ECASQ_CUDA_TRY(cudaMemcpyAsync(qi, a.data(), sizeof(int32_t) * m, cudaMemcpyHostToDevice, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(mc, &m, sizeof(int32_t), cudaMemcpyHostToDevice, st));
    int rc = launch_gather_q(wsp<float>(ws, L.v), qi, mc, 1, kMaxS, Q, st);
    if (rc != ECASQ_OK) return rc;
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    return ECASQ_OK;
}

static bool params_ok(const ecasq_params_t *prm) {
    if (!prm) return false;
    if (prm->s < 2 || prm->s > kMaxS) return false;
    if (prm->lambda < 0.0 && !(prm->budget_bits >= 0.0)) return false;
    if (prm->lambda >= 0.0 && !isfinite(prm->lambda)) return false;
    if (prm->refine_max_rounds < 0) return false;
    return true;
}

struct Eval { double lam, mse, hs, hx; int m; bool feas; std::vector<int32_t> a; };

}  // namespace ecasq

using namespace ecasq;

extern "C" {

int ecasq_version(void) { return 10000; }

int64_t ecasq_kernel_launches(void) { return (int64_t)g_launches.load(); }

const char *ecasq_strerror(int status) {
    switch (status) {
        case ECASQ_OK: return "ok";
        case ECASQ_EINVAL: return "invalid argument";
        case ECASQ_ENONFINITE: return "input holds NaN or Inf";
        case ECASQ_EINFEASIBLE: return "entropy budget infeasible for the evaluated multipliers";
        case ECASQ_EWORKSPACE: return "workspace too small or not 256-byte aligned";
        case ECASQ_ECUDA: return "CUDA error";
        case ECASQ_ETIMEOUT: return "bounded device wait timed out";
        case ECASQ_ERANGE: return "value outside the codebook range, or codebook value not in x";
        default: return "unknown status";
    }
}

size_t ecasq_workspace_size(int64_t d, int32_t s, int64_t rows) {
    if (d < 1 || d >= ((int64_t)1 << 31) || s < 2 || s > kMaxS || rows < 1) return 0;
    Layout L;
    return make_layout(d, s, rows, &L) + rows_region_bytes(d, s, rows);
}

size_t ecasq_workspace_size_flags(int64_t d, int32_t s, int64_t rows, uint32_t flags) {
    size_t base = ecasq_workspace_size(d, s, rows);
    if (!base || !(flags & (ECASQ_RESIDENT_COSTS | ECASQ_STREAMED_COSTS))) return base;
    size_t cb = (flags & ECASQ_RESIDENT_COSTS) ? resident_costs_bytes(d) : streamed_costs_bytes(d);
    if (!cb || base > SIZE_MAX - align256(cb)) return 0;
    return base + align256(cb);
}

size_t ecasq_workspace_size_prep(int64_t d) {
    if (d < 1 || d >= ((int64_t)1 << 31)) return 0;
    Layout L;
    return make_prep_layout(d, &L);
}

int ecasq_prepare(const float *x, int64_t d, void *ws, size_t ws_bytes, float *v, int64_t *w, int64_t *N,
                  double *S, double *S2, int64_t *p_out, ecasq_stream_t stream) {
    if (!x || d < 1 || d >= ((int64_t)1 << 31) || !v || !w || !N || !S || !S2 || !p_out) return ECASQ_EINVAL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    Layout L;
    make_prep_layout(d, &L);
    int rc = check_ws(ws, ws_bytes, L);
    if (rc) return rc;
    int64_t p;
    double n2;
    rc = prepare_device(x, d, ws, L, st, &p, &n2);
    if (rc) return rc;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(v, wsp<float>(ws, L.v), 4 * p, cudaMemcpyDeviceToDevice, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(w, wsp<int64_t>(ws, L.w), 8 * p, cudaMemcpyDeviceToDevice, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(N, wsp<int64_t>(ws, L.N), 8 * (p + 1), cudaMemcpyDeviceToDevice, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(S, wsp<double>(ws, L.S), 16 * (p + 1), cudaMemcpyDeviceToDevice, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(S2, wsp<double>(ws, L.S2), 16 * (p + 1), cudaMemcpyDeviceToDevice, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    *p_out = p;
    return ECASQ_OK;
}

int ecasq_dp_pass(const float *x, int64_t d, int32_t s, const double *lambdas, int32_t G, uint32_t flags, void *ws,
                  size_t ws_bytes, float *Q_out, int32_t *m_out, double *metrics, ecasq_stream_t stream) {
    if (!x || d < 1 || d >= ((int64_t)1 << 31) || s < 2 || s > kMaxS || !lambdas || G < 1 || G > kMaxG || !Q_out ||
        !m_out || !metrics)
        return ECASQ_EINVAL;
    for (int g = 0; g < G; g++)
        if (!(lambdas[g] >= 0.0) || !isfinite(lambdas[g])) return ECASQ_EINVAL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    Layout L;
    make_layout(d, s, 1, &L);
    int rc = add_resident_costs(flags, &L);
    if (rc) return rc;
    rc = check_ws(ws, ws_bytes, L);
    if (rc) return rc;
    int64_t p;
    double n2;
    rc = prepare_device(x, d, ws, L, st, &p, &n2);
    if (rc) return rc;
    Prefix P = make_prefix(ws, L, p, d);
    if (p == 1) {
        for (int g = 0; g < G; g++) {
            ECASQ_CUDA_TRY(cudaMemcpyAsync(Q_out + (size_t)g * s, P.v, 4, cudaMemcpyDeviceToDevice, st));
            m_out[g] = 1;
            for (int t = 0; t < 4; t++) metrics[4 * g + t] = 0.0;
        }
        ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
        return ECASQ_OK;
    }
    double lamp[kMaxG];
    for (int g = 0; g < G; g++) lamp[g] = lambdas[g] * n2;
    PassOut po;
    bool costs_built = false;
    rc = dp_pass_prepared(ws, L, P, s, lamp, G, flags, st, po, &costs_built);
    if (rc) return rc;
    rc = launch_gather_q(P.v, wsp<int32_t>(ws, L.qidx), wsp<int32_t>(ws, L.mcount), G, s, Q_out, st);
    if (rc) return rc;
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    for (int g = 0; g < G; g++) {
        m_out[g] = po.m[g];
        for (int t = 0; t < 4; t++) metrics[4 * g + t] = po.met[4 * g + t];
    }
    return ECASQ_OK;
}

int ecasq_dp_tables(void *ws, size_t ws_bytes, int32_t g, double *dp_out, int32_t *bp_out, int64_t *p_out,
                    ecasq_stream_t stream) {
    if (!ws || !dp_out || !bp_out || !p_out || g < 0 || g >= kMaxG) return ECASQ_EINVAL;
    if ((reinterpret_cast<uintptr_t>(ws) & 255) != 0 || ws_bytes < sizeof(DevStatus)) return ECASQ_EWORKSPACE;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    DevStatus h;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(&h, ws, sizeof(DevStatus), cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    if (h.last_s < 2 || g >= h.last_G || h.p < 2 || h.last_d < 1) return ECASQ_EINVAL;
    Layout L;
    make_layout(h.last_d, h.last_s, 1, &L);
    int rc = check_ws(ws, ws_bytes, L);
    if (rc) return rc;
    size_t ps = (size_t)table_stride(h.p), rowsn = (size_t)(h.last_s + 1);
    size_t off = (size_t)g * rowsn * ps;
    ECASQ_CUDA_TRY(cudaMemcpy2DAsync(dp_out, 8 * (size_t)h.p, wsp<double>(ws, L.dp64) + off, 8 * ps, 8 * (size_t)h.p,
                                     rowsn, cudaMemcpyDeviceToDevice, st));
    ECASQ_CUDA_TRY(cudaMemcpy2DAsync(bp_out, 4 * (size_t)h.p, wsp<int32_t>(ws, L.bp) + off, 4 * ps, 4 * (size_t)h.p,
                                     rowsn, cudaMemcpyDeviceToDevice, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    *p_out = h.p;
    return ECASQ_OK;
}

static void fill_result(ecasq_result_t *res, int status, int m, int64_t d, int64_t p, double lam, double n2,
                        const double *ev, double objective, int passes, int nlam, int rr, int64_t cand,
                        int64_t rescored) {
    if (!res) return;
    memset(res, 0, sizeof(*res));
    res->status = status;
    res->m = m;
    res->passes = passes;
    res->lambdas_evaluated = nlam;
    res->refine_rounds = rr;
    res->d = d;
    res->p = p;
    res->lambda = lam;
    res->lambda_prime = lam * n2;
    res->norm2 = n2;
    res->mse = ev[0];
    res->vnmse = n2 > 0.0 ? ev[0] / n2 : 0.0;
    res->h_surrogate = ev[1];
    res->h_exact = ev[2];
    res->r_tot = ev[2] + 32.0 * (double)m / (double)d;
    res->objective = objective;
    res->candidates = cand;
    res->rescored = rescored;
}

static int64_t read_rescored(void *ws, cudaStream_t st) {
    DevStatus h;
    if (cudaMemcpyAsync(&h, ws, sizeof(DevStatus), cudaMemcpyDeviceToHost, st) != cudaSuccess) return -1;
    if (cudaStreamSynchronize(st) != cudaSuccess) return -1;
    return h.rescored;
}

// The search, refinement and result of a solve over a prepared histogram view P
// (unique values of x, or a caller-given candidate set).
// Sec. 7: the evaluated infeasible point of least H(I,B) (ties: less MSE, then the
// smaller multiplier), the Q+ of two-way time-sharing.
struct PlusPoint { bool have = false; double lam = 0.0, mse = 0.0, hs = 0.0, hx = 0.0; std::vector<int32_t> a; };

static int solve_prepared(void *ws, const Layout &L, const Prefix &P, int64_t d, double n2, const ecasq_params_t *prm,
                          float *Q, ecasq_result_t *res, cudaStream_t st, PlusPoint *plus = nullptr) {
    const int s = prm->s;
    const int64_t p = P.p;
    int rc;
    double zero3[3] = {0.0, 0.0, 0.0};
    bool costs_built = false;
    if (p == 1) {
        ECASQ_CUDA_TRY(cudaMemcpyAsync(Q, P.v, 4, cudaMemcpyDeviceToDevice, st));
        ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
        fill_result(res, ECASQ_OK, 1, d, p, prm->lambda >= 0 ? prm->lambda : 0.0, n2, zero3, 0.0, 0, 0, 0, 0, 0);
        return ECASQ_OK;
    }
    int passes = 0, nlam = 0;
    int64_t cand_per = candidates_of(p, s, 0);
    int64_t cand = 0;
    std::vector<Eval> evals;
    // Seed rows (tile skipping of the fast kernel): the fp32 minima of the last pass at
    // seed_lam, kept while every later multiplier stays below it.  The search's upper
    // bracket end is such a multiplier once it has been evaluated.
    double seed_lam = -1.0;
    int last_G = 0;
    auto run = [&](const std::vector<double> &lams) -> int {
        double lamp[kMaxG];
        int G = (int)lams.size();
        bool seeded = seed_lam >= 0.0;
        for (int g = 0; g < G; g++) {
            lamp[g] = lams[g] * n2;
            seeded = seeded && lams[g] <= seed_lam;
        }
        PassOut po;
        int r = dp_pass_prepared(ws, L, P, s, lamp, G, prm->flags, st, po, &costs_built, seeded);
        if (r) return r;
        last_G = G;
        passes++;
        nlam += G;
        cand += cand_per * G;
        for (int g = 0; g < G; g++) {
            Eval e;
            e.lam = lams[g];
            e.m = po.m[g];
            e.mse = po.met[4 * g + 1];
            e.hs = po.met[4 * g + 2];
            e.hx = po.met[4 * g + 3];
            e.feas = prm->lambda >= 0.0 ? true : (e.hs <= prm->budget_bits);
            e.a.assign(po.qidx.begin() + (size_t)g * s, po.qidx.begin() + (size_t)g * s + e.m);
            evals.push_back(e);
        }
        return ECASQ_OK;
    };
    int status = ECASQ_OK;
    const Eval *sel = nullptr;
    if (prm->lambda >= 0.0) {
        if ((prm->flags & ECASQ_TEST_SELF_SEED) && L.costs_bytes && !L.gpairs_bytes &&
            !(prm->flags & (ECASQ_DP_REFERENCE | ECASQ_UNSEEDED_SEARCH))) {
            rc = run({prm->lambda});
            if (rc) return rc;
            rc = save_dp_seed(ws, L, p, 1, s, 0, st);
            if (rc) return rc;
            seed_lam = prm->lambda;
        }
        rc = run({prm->lambda});
        if (rc) return rc;
        sel = &evals.back();
    } else {
        double lo = prm->lambda_lo > 0.0 ? prm->lambda_lo : 1e-8;
        double hi = prm->lambda_hi > 0.0 ? prm->lambda_hi : 1e3;
        int R = prm->search_rounds > 0 ? prm->search_rounds : 6;
        if (!(hi > lo)) return ECASQ_EINVAL;
        double t[7];
        midpoints7(lo, hi, t);
        std::vector<double> l1 = {0.0};
        l1.insert(l1.end(), t, t + 7);
        rc = run(l1);
        if (rc) return rc;
        if (evals[0].feas) {
            sel = &evals[0];
        } else {
            for (int r = 0; r < R; r++) {
                if (r > 0) {
                    midpoints7(lo, hi, t);
                    rc = run(std::vector<double>(t, t + 7));
                    if (rc) return rc;
                }
                const Eval *pts = &evals[evals.size() - 7];
                int f = -1;
                for (int q = 0; q < 7; q++)
                    if (pts[q].feas) { f = q; break; }
                if (f >= 0) {
                    double nlo = f > 0 ? pts[f - 1].lam : lo;
                    hi = pts[f].lam;
                    lo = nlo;
                    // the next passes lie below hi: its fp32 minima bound theirs
                    if (L.costs_bytes && !L.gpairs_bytes && !(prm->flags & (ECASQ_DP_REFERENCE | ECASQ_UNSEEDED_SEARCH))) {
                        rc = save_dp_seed(ws, L, p, last_G, s, last_G - 7 + f, st);
                        if (rc) return rc;
                        seed_lam = hi;
                    }
                } else {
                    lo = pts[6].lam;
                }
            }
            for (const Eval &e : evals)
                if (e.feas && (!sel || e.mse < sel->mse || (e.mse == sel->mse && e.lam < sel->lam))) sel = &e;
            if (!sel) {
                rc = run({hi});
                if (rc) return rc;
                sel = &evals.back();
                if (!sel->feas) status = ECASQ_EINFEASIBLE;
            }
        }
    }
    if (plus) {
        for (const Eval &e : evals) {
            if (e.feas) continue;
            if (!plus->have || e.hs < plus->hs ||
                (e.hs == plus->hs && (e.mse < plus->mse || (e.mse == plus->mse && e.lam < plus->lam)))) {
                plus->have = true;
                plus->lam = e.lam; plus->mse = e.mse; plus->hs = e.hs; plus->hx = e.hx;
                plus->a = e.a;
            }
        }
    }
    std::vector<int32_t> a = sel->a;
    double lam = sel->lam;
    double lamp = lam * n2;
    int rr = 0;
    double last_rel = 0.0;
    if (status == ECASQ_OK && prm->refine_max_rounds > 0 && (int)a.size() >= 3) {
        bool guard = prm->lambda < 0.0 && !(prm->flags & ECASQ_NO_REFINE_GUARD);
        rc = refine_device(ws, L, P, a, lamp, prm->budget_bits, guard, prm->refine_max_rounds, prm->refine_rel_tol,
                           st, &rr, &last_rel);
        if (rc) return rc;
    }
    rc = write_codebook(ws, L, a, Q, st);
    if (rc) return rc;
    double ev[3];
    rc = eval_device(ws, L, P, wsp<int32_t>(ws, L.qidx), (int)a.size(), st, ev);
    if (rc) return rc;
    double obj = prm->refine_max_rounds > 0 ? ev[0] + lamp * ev[2] : ev[0] + lamp * ev[1];
    fill_result(res, status, (int)a.size(), d, p, lam, n2, ev, obj, passes, nlam, rr, cand, read_rescored(ws, st));
    if (res) {
        res->dp_kernel_ms = g_timer.ms;
        res->dp_kernel_launches = g_timer.launches;
        res->refine_last_rel = last_rel;
    }
    g_timer.on = false;
    return status;
}

// Layout, workspace check, sort / histogram / prefix sums of x (Sec. 2, App. E).
static int prepare_plain(const float *x, int64_t d, const ecasq_params_t *prm, void *ws, size_t ws_bytes, Layout *L,
                         Prefix *P, double *n2, cudaStream_t st) {
    make_layout(d, prm->s, 1, L);
    int rc = add_resident_costs(prm->flags, L);
    if (rc) return rc;
    rc = check_ws(ws, ws_bytes, *L);
    if (rc) return rc;
    int64_t p;
    rc = prepare_device(x, d, ws, *L, st, &p, n2);
    if (rc) return rc;
    *P = make_prefix(ws, *L, p, d);
    return ECASQ_OK;
}

static void timer_reset(const ecasq_params_t *prm) {
    g_timer.on = (prm->flags & ECASQ_TIME_KERNELS) != 0;
    g_timer.ms = 0.0;
    g_timer.launches = 0;
}

int ecasq_solve(const float *x, int64_t d, const ecasq_params_t *prm, void *ws, size_t ws_bytes, float *Q,
                ecasq_result_t *res, ecasq_stream_t stream) {
    if (!x || !Q || d < 1 || d >= ((int64_t)1 << 31) || !params_ok(prm)) return ECASQ_EINVAL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    timer_reset(prm);
    Layout L;
    Prefix P;
    double n2;
    int rc = prepare_plain(x, d, prm, ws, ws_bytes, &L, &P, &n2, st);
    if (rc) return rc;
    return solve_prepared(ws, L, P, d, n2, prm, Q, res, st);
}

size_t ecasq_workspace_size_grid(int64_t d, int64_t n, int32_t s, uint32_t flags) {
    (void)flags;  // the grid DP keeps its own pair cache; resident tiles are not used
    if (d < 1 || d >= ((int64_t)1 << 31) || n < 1 || n >= ((int64_t)1 << 31) || s < 2 || s > kMaxS) return 0;
    Layout L;
    make_layout(std::max(d, n), s, 1, &L);
    return L.total + align256(grid_pairs_bytes(n));
}

static int grid_view(const float *x, int64_t d, const float *Pg, int64_t n, void *ws, const Layout &L, Prefix *Po,
                     double *n2o, cudaStream_t st);
static double scale32_of(double n2);

// The histogram view over a permissible set P (Sec. 5, App. E): prepare x, then
// gather the prefix sums at the points of P; P->nL, P->nR receive |L|, |R|.
static int prepare_grid(const float *x, int64_t d, const float *Pg, int64_t n, const ecasq_params_t *prm, void *ws,
                        size_t ws_bytes, Layout *Lo, Prefix *Po, double *n2o, cudaStream_t st) {
    const int64_t dmax = std::max(d, n);
    Layout &L = *Lo;
    make_layout(dmax, prm->s, 1, &L);
    L.d = dmax;
    size_t gb = grid_pairs_bytes(n);
    if (gb) {
        L.gpairs = L.total;
        L.gpairs_bytes = gb;
        L.total += align256(gb);
    }
    int rc = check_ws(ws, ws_bytes, L);
    if (rc) return rc;
    return grid_view(x, d, Pg, n, ws, L, Po, n2o, st);
}

static double scale32_of(double n2) {
    return (n2 > 0.0 && std::isfinite(n2)) ? std::ldexp(1.0, -std::ilogb(n2)) : 1.0;
}

// Sort / histogram / prefix sums of x, then the grid view of P in place of the
// unique values (needs L.dp64 as scratch for the unique-value arrays).
static int grid_view(const float *x, int64_t d, const float *Pg, int64_t n, void *ws, const Layout &L, Prefix *Po,
                     double *n2o, cudaStream_t st) {
    int64_t pX;
    double n2;
    int rc = prepare_device(x, d, ws, L, st, &pX, &n2);
    if (rc) return rc;
    // the unique-value view moves to scratch (the fp64 DP table area), the grid view takes its place
    char *scr = wsp<char>(ws, L.dp64);
    float *vX = reinterpret_cast<float *>(scr);
    int64_t *NX = reinterpret_cast<int64_t *>(scr + align256(4 * (size_t)pX));
    double *SX = reinterpret_cast<double *>(scr + align256(4 * (size_t)pX) + align256(8 * (size_t)(pX + 1)));
    double *S2X = SX + 2 * (pX + 1);
    ECASQ_CUDA_TRY(cudaMemcpyAsync(vX, wsp<float>(ws, L.v), 4 * (size_t)pX, cudaMemcpyDeviceToDevice, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(NX, wsp<int64_t>(ws, L.N), 8 * (size_t)(pX + 1), cudaMemcpyDeviceToDevice, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(SX, wsp<double>(ws, L.S), 16 * (size_t)(pX + 1), cudaMemcpyDeviceToDevice, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(S2X, wsp<double>(ws, L.S2), 16 * (size_t)(pX + 1), cudaMemcpyDeviceToDevice, st));
    DevStatus *ds = wsp<DevStatus>(ws, L.status);
    rc = launch_grid_prefix(Pg, n, vX, NX, SX, S2X, pX, wsp<float>(ws, L.v), wsp<int64_t>(ws, L.w),
                            wsp<int64_t>(ws, L.N), wsp<double>(ws, L.S), wsp<double>(ws, L.S2), ds, st);
    if (rc) return rc;
    DevStatus h;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(&h, ds, sizeof(DevStatus), cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    if (h.range_err || h.grid_nL < 1 || h.grid_nR < 1) return ECASQ_EINVAL;
    int64_t pz = n;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(&ds->p, &pz, sizeof(pz), cudaMemcpyHostToDevice, st));
    *Po = make_prefix(ws, L, n, d);
    Po->nL = h.grid_nL;
    Po->nR = h.grid_nR;
    Po->scale32 = scale32_of(n2);
    *n2o = n2;
    return ECASQ_OK;
}

int ecasq_solve_grid(const float *x, int64_t d, const float *Pg, int64_t n, const ecasq_params_t *prm, void *ws,
                     size_t ws_bytes, float *Q, ecasq_result_t *res, ecasq_stream_t stream) {
    if (!x || !Q || !Pg || d < 1 || d >= ((int64_t)1 << 31) || n < 1 || n >= ((int64_t)1 << 31) || !params_ok(prm))
        return ECASQ_EINVAL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    timer_reset(prm);
    Layout L;
    Prefix P;
    double n2;
    int rc = prepare_grid(x, d, Pg, n, prm, ws, ws_bytes, &L, &P, &n2, st);
    if (rc) return rc;
    // The fast kernel's fp32 recurrences add one candidate at a time and assume each
    // slab's mass sits at its right end (true for the unique values of x only); a grid
    // runs the grid DP (cached pair costs), or beyond kGridPairsMax the reference DP.
    ecasq_params_t pg = *prm;
    if (!L.gpairs_bytes) pg.flags |= ECASQ_DP_REFERENCE;
    return solve_prepared(ws, L, P, d, n2, &pg, Q, res, st);
}

int ecasq_solve_timeshare(const float *x, int64_t d, const float *Pg, int64_t n, const ecasq_params_t *prm, void *ws,
                          size_t ws_bytes, float *Qm, float *Qp, ecasq_result_t *res, ecasq_timeshare_t *ts,
                          ecasq_stream_t stream) {
    if (!x || !Qm || !Qp || !ts || d < 1 || d >= ((int64_t)1 << 31) || !params_ok(prm) || !(prm->lambda < 0.0) ||
        prm->refine_max_rounds != 0)
        return ECASQ_EINVAL;
    if (Pg && (n < 1 || n >= ((int64_t)1 << 31))) return ECASQ_EINVAL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    timer_reset(prm);
    Layout L;
    Prefix P;
    double n2;
    ecasq_params_t pg = *prm;
    int rc;
    if (Pg) {
        rc = prepare_grid(x, d, Pg, n, prm, ws, ws_bytes, &L, &P, &n2, st);
        if (rc == ECASQ_OK && !L.gpairs_bytes) pg.flags |= ECASQ_DP_REFERENCE;
    } else {
        rc = prepare_plain(x, d, prm, ws, ws_bytes, &L, &P, &n2, st);
    }
    if (rc) return rc;
    PlusPoint plus;
    ecasq_result_t rm;
    int status = solve_prepared(ws, L, P, d, n2, &pg, Qm, &rm, st, &plus);
    if (res) *res = rm;
    memset(ts, 0, sizeof(*ts));
    ts->lambda_plus = NAN;
    ts->plus_mse = ts->plus_h_surrogate = ts->plus_h_exact = NAN;
    if (status != ECASQ_OK) return status;
    // Sec. 7: beta = (b - b-)/(b+ - b-) when Q+ exists, has less MSE and b- < b
    double beta = 0.0;
    if (plus.have && plus.mse < rm.mse && rm.h_surrogate < prm->budget_bits)
        beta = (prm->budget_bits - rm.h_surrogate) / (plus.hs - rm.h_surrogate);
    double mm[3] = {rm.mse, rm.h_surrogate, rm.h_exact};
    double mx[3] = {rm.mse, rm.h_surrogate, rm.h_exact};
    if (beta > 0.0) {
        rc = write_codebook(ws, L, plus.a, Qp, st);
        if (rc) return rc;
        double pm[3] = {plus.mse, plus.hs, plus.hx};
        for (int r = 0; r < 3; r++) mx[r] = (1.0 - beta) * mm[r] + beta * pm[r];
        ts->m_plus = (int32_t)plus.a.size();
        ts->lambda_plus = plus.lam;
        ts->plus_mse = plus.mse;
        ts->plus_h_surrogate = plus.hs;
        ts->plus_h_exact = plus.hx;
    }
    ts->beta = beta;
    ts->mse = mx[0];
    ts->vnmse = n2 > 0.0 ? mx[0] / n2 : 0.0;
    ts->h_surrogate = mx[1];
    ts->h_exact = mx[2];
    return ECASQ_OK;
}

int ecasq_refine(const float *x, int64_t d, float *Q, int32_t m, double lambda, double budget_bits,
                 int32_t max_rounds, double rel_tol, uint32_t flags, void *ws, size_t ws_bytes, ecasq_result_t *res,
                 ecasq_stream_t stream) {
    if (!x || !Q || d < 1 || d >= ((int64_t)1 << 31) || m < 1 || m > kMaxS || !(lambda >= 0.0) ||
        !isfinite(lambda) || max_rounds < 0)
        return ECASQ_EINVAL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    Layout L;
    make_layout(d, 2, 1, &L);
    int rc = check_ws(ws, ws_bytes, L);
    if (rc) return rc;
    int64_t p;
    double n2;
    rc = prepare_device(x, d, ws, L, st, &p, &n2);
    if (rc) return rc;
    Prefix P = make_prefix(ws, L, p, d);
    int32_t *a_dev = wsp<int32_t>(ws, L.qidx);
    DevStatus *ds = wsp<DevStatus>(ws, L.status);
    rc = launch_locate_q(P.v, p, Q, m, a_dev, ds, st);
    if (rc) return rc;
    std::vector<int32_t> a(m);
    DevStatus h;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(a.data(), a_dev, 4 * m, cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(&h, ds, sizeof(h), cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    if (h.range_err) return ECASQ_ERANGE;
    if (a[0] != 0 || a[m - 1] != p - 1) return ECASQ_ERANGE;
    for (int r = 1; r < m; r++)
        if (a[r] <= a[r - 1]) return ECASQ_EINVAL;
    double lamp = lambda * n2;
    bool guard = budget_bits >= 0.0 && !(flags & ECASQ_NO_REFINE_GUARD);
    int rr = 0;
    double last_rel = 0.0;
    rc = refine_device(ws, L, P, a, lamp, budget_bits, guard, max_rounds, rel_tol, st, &rr, &last_rel);
    if (rc) return rc;
    rc = write_codebook(ws, L, a, Q, st);
    if (rc) return rc;
    double ev[3];
    rc = eval_device(ws, L, P, wsp<int32_t>(ws, L.qidx), m, st, ev);
    if (rc) return rc;
    fill_result(res, ECASQ_OK, m, d, p, lambda, n2, ev, ev[0] + lamp * ev[2], 0, 0, rr, 0, 0);
    if (res) res->refine_last_rel = last_rel;
    return ECASQ_OK;
}

int ecasq_evaluate(const float *x, int64_t d, const float *Q, int32_t m, void *ws, size_t ws_bytes, double *out,
                   ecasq_stream_t stream) {
    if (!x || !Q || !out || d < 1 || d >= ((int64_t)1 << 31) || m < 1 || m > kMaxS) return ECASQ_EINVAL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    Layout L;
    make_layout(d, 2, 1, &L);
    int rc = check_ws(ws, ws_bytes, L);
    if (rc) return rc;
    int64_t p;
    double n2;
    rc = prepare_device(x, d, ws, L, st, &p, &n2);
    if (rc) return rc;
    Prefix P = make_prefix(ws, L, p, d);
    int32_t *a_dev = wsp<int32_t>(ws, L.qidx);
    DevStatus *ds = wsp<DevStatus>(ws, L.status);
    rc = launch_locate_q(P.v, p, Q, m, a_dev, ds, st);
    if (rc) return rc;
    std::vector<int32_t> a(m);
    DevStatus h;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(a.data(), a_dev, 4 * m, cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(&h, ds, sizeof(h), cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    if (h.range_err || a[0] != 0 || a[m - 1] != p - 1) return ECASQ_ERANGE;
    for (int r = 1; r < m; r++)
        if (a[r] <= a[r - 1]) return ECASQ_EINVAL;
    return eval_device(ws, L, P, a_dev, m, st, out);
}

int ecasq_quantize(const float *x, int64_t d, const float *Q, int32_t m, uint64_t seed, uint8_t *idx,
                   uint32_t *counts, void *ws, size_t ws_bytes, double *h_emp, ecasq_stream_t stream) {
    if (!x || !Q || !idx || !counts || d < 1 || d >= ((int64_t)1 << 31) || m < 1 || m > kMaxS) return ECASQ_EINVAL;
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255) != 0 || ws_bytes < sizeof(DevStatus)) return ECASQ_EWORKSPACE;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    DevStatus *ds = wsp<DevStatus>(ws, 0);
    std::vector<float> qh(m);
    ECASQ_CUDA_TRY(cudaMemcpyAsync(qh.data(), Q, 4 * m, cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaMemsetAsync(ds, 0, sizeof(DevStatus), st));
    ECASQ_CUDA_TRY(cudaMemsetAsync(counts, 0, 4 * (size_t)m, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    for (int r = 1; r < m; r++)
        if (!(qh[r] > qh[r - 1])) return ECASQ_EINVAL;
    int rc = launch_quantize(x, d, Q, m, seed, idx, counts, ds, num_sms(), st);
    if (rc) return rc;
    std::vector<uint32_t> ch(m);
    DevStatus h;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(&h, ds, sizeof(h), cudaMemcpyDeviceToHost, st));
    if (h_emp) ECASQ_CUDA_TRY(cudaMemcpyAsync(ch.data(), counts, 4 * (size_t)m, cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    if (h.range_err) return ECASQ_ERANGE;
    if (h_emp) {
        double he = 0.0, dd_ = (double)d;
        for (int r = 0; r < m; r++) {
            double f = (double)ch[r] / dd_;
            if (f > 0.0) he += -f * log2(f);
        }
        *h_emp = he;
    }
    return ECASQ_OK;
}

// Same checks, kernel and host arithmetic as ecasq_quantize; the status record
// lives in the fixed scratch block and host copies in fixed-size arrays.
int ecasq_quantize_noalloc(const float *x, int64_t d, const float *Q, int32_t m, uint64_t seed, uint8_t *idx,
                           uint32_t *counts, double *h_emp, ecasq_stream_t stream) {
    if (!x || !Q || !idx || !counts || d < 1 || d >= ((int64_t)1 << 31) || m < 1 || m > kMaxS) return ECASQ_EINVAL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    void *scratch = nullptr;
    int rc = noalloc_scratch(st, &scratch);
    if (rc) return rc;
    DevStatus *ds = reinterpret_cast<DevStatus *>(scratch);
    float qh[kMaxS];
    ECASQ_CUDA_TRY(cudaMemcpyAsync(qh, Q, 4 * (size_t)m, cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaMemsetAsync(ds, 0, sizeof(DevStatus), st));
    ECASQ_CUDA_TRY(cudaMemsetAsync(counts, 0, 4 * (size_t)m, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    for (int r = 1; r < m; r++)
        if (!(qh[r] > qh[r - 1])) return ECASQ_EINVAL;
    rc = launch_quantize(x, d, Q, m, seed, idx, counts, ds, num_sms(), st);
    if (rc) return rc;
    uint32_t ch[kMaxS];
    DevStatus h;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(&h, ds, sizeof(h), cudaMemcpyDeviceToHost, st));
    if (h_emp) ECASQ_CUDA_TRY(cudaMemcpyAsync(ch, counts, 4 * (size_t)m, cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    if (h.range_err) return ECASQ_ERANGE;
    if (h_emp) {
        double he = 0.0, dd_ = (double)d;
        for (int r = 0; r < m; r++) {
            double f = (double)ch[r] / dd_;
            if (f > 0.0) he += -f * log2(f);
        }
        *h_emp = he;
    }
    return ECASQ_OK;
}

// Linear-space traceback (Sec. 5, last paragraph): the preparation layout, then four DP
// rows of d + 1 doubles, the column dp(i, p-1), the codebook and a little scratch.
struct LinearLayout { Layout prep; size_t rows, col, qidx, mcount, small, total; };
static bool linear_layout(int64_t d, LinearLayout *LL) {
    if (d < 1 || d >= ((int64_t)1 << 31)) return false;
    size_t off = make_prep_layout(d, &LL->prep);
    auto take = [&](size_t bytes) { size_t o = off; off += align256(bytes); return o; };
    LL->rows = take(4 * 8 * (size_t)(d + 1));
    LL->col = take(8 * (size_t)(kMaxS + 1));
    LL->qidx = take(4 * (size_t)kMaxS);
    LL->mcount = take(4);
    LL->small = take(64);
    LL->total = off;
    return true;
}

size_t ecasq_workspace_size_linear(int64_t d) {
    LinearLayout LL;
    return linear_layout(d, &LL) ? LL.total : 0;
}

int ecasq_dp_linear(const float *x, int64_t d, int32_t s, double lambda, uint32_t flags, void *ws, size_t ws_bytes,
                    float *Q_out, int32_t *m_out, double *metrics, ecasq_stream_t stream) {
    if (!x || !Q_out || !m_out || !metrics || s < 2 || s > kMaxS || !(lambda >= 0.0) || !isfinite(lambda))
        return ECASQ_EINVAL;
    LinearLayout LL;
    if (!linear_layout(d, &LL)) return ECASQ_EINVAL;
    int rc = check_ws(ws, ws_bytes, LL.prep);
    if (rc) return rc;
    if (ws_bytes < LL.total) return ECASQ_EWORKSPACE;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    int64_t p;
    double n2;
    rc = prepare_device(x, d, ws, LL.prep, st, &p, &n2);
    if (rc) return rc;
    Prefix P = make_prefix(ws, LL.prep, p, d);
    std::vector<int32_t> a;
    int m = 0;
    double best = 0.0;
    rc = launch_dp_linear(P, lambda * n2, s, (flags & ECASQ_EXACT_S) ? 1 : 0, wsp<double>(ws, LL.rows),
                          wsp<double>(ws, LL.col), wsp<void>(ws, LL.small), a, &m, &best, st);
    if (rc) return rc;
    int32_t *qi = wsp<int32_t>(ws, LL.qidx);
    int32_t *mc = wsp<int32_t>(ws, LL.mcount);
    ECASQ_CUDA_TRY(cudaMemcpyAsync(qi, a.data(), sizeof(int32_t) * m, cudaMemcpyHostToDevice, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(mc, &m, sizeof(int32_t), cudaMemcpyHostToDevice, st));
    rc = launch_gather_q(P.v, qi, mc, 1, kMaxS, Q_out, st);
    if (rc) return rc;
    double ev[3] = {0.0, 0.0, 0.0};
    if (m >= 2) {
        double *o = wsp<double>(ws, LL.small) + 4;
        rc = launch_eval_codebook(P, qi, m, o, st);
        if (rc) return rc;
        ECASQ_CUDA_TRY(cudaMemcpyAsync(ev, o, 3 * sizeof(double), cudaMemcpyDeviceToHost, st));
    }
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    *m_out = m;
    metrics[0] = best;
    metrics[1] = ev[0];
    metrics[2] = ev[1];
    metrics[3] = ev[2];
    return ECASQ_OK;
}

// Optimal DP (Sec. 4): base layout, then the pair quantities C, U, D and the
// tables dp, bk of G multipliers.
static bool opt_layout(int64_t d, int64_t n, int32_t s, int32_t G, Layout *L, size_t *pairs_off, size_t *tables_off) {
    if (d < 1 || d >= ((int64_t)1 << 31) || n < 1 || n > kOptMax || s < 2 || s > kMaxS || G < 1 || G > kMaxG)
        return false;
    make_layout(std::max(d, n), s, 1, L);
    L->d = std::max(d, n);
    *pairs_off = L->total;
    *tables_off = *pairs_off + align256(opt_pairs_bytes(n));
    L->total = *tables_off + align256(opt_tables_bytes(n, s, G));
    return true;
}

size_t ecasq_workspace_size_opt(int64_t d, int64_t n, int32_t s, int32_t G) {
    Layout L;
    size_t po, to;
    return opt_layout(d, n, s, G, &L, &po, &to) ? L.total : 0;
}

int ecasq_opt_dp(const float *x, int64_t d, const float *Pg, int64_t n, int32_t s, const double *lambdas, int32_t G,
                 uint32_t flags, void *ws, size_t ws_bytes, float *Q_out, int32_t *m_out, double *metrics,
                 ecasq_stream_t stream) {
    if (!x || !lambdas || !Q_out || !m_out || !metrics || d < 1 || d >= ((int64_t)1 << 31) || G < 1 || G > kMaxG ||
        s < 2 || s > kMaxS)
        return ECASQ_EINVAL;
    for (int g = 0; g < G; g++)
        if (!(lambdas[g] >= 0.0) || !std::isfinite(lambdas[g])) return ECASQ_EINVAL;
    if (Pg && (n < 1 || n > kOptMax)) return ECASQ_EINVAL;
    if (!Pg && d > kOptMax) return ECASQ_EINVAL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const int64_t nmax = Pg ? n : d;
    Layout L;
    size_t pairs_off, tables_off;
    if (!opt_layout(d, nmax, s, G, &L, &pairs_off, &tables_off)) return ECASQ_EINVAL;
    int rc = check_ws(ws, ws_bytes, L);
    if (rc) return rc;
    Prefix P;
    double n2;
    if (Pg) {
        rc = grid_view(x, d, Pg, n, ws, L, &P, &n2, st);
        if (rc) return rc;
    } else {
        int64_t p;
        rc = prepare_device(x, d, ws, L, st, &p, &n2);
        if (rc) return rc;
        P = make_prefix(ws, L, p, d);
        P.scale32 = scale32_of(n2);
    }
    int32_t *qidx = wsp<int32_t>(ws, L.qidx);
    int32_t *mc = wsp<int32_t>(ws, L.mcount);
    double *met = wsp<double>(ws, L.metrics);
    if (P.p == 1) {
        ECASQ_CUDA_TRY(cudaMemcpyAsync(Q_out, P.v, 4, cudaMemcpyDeviceToDevice, st));
        ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
        for (int g = 0; g < G; g++) {
            m_out[g] = 1;
            for (int r = 0; r < 4; r++) metrics[4 * g + r] = 0.0;
        }
        return ECASQ_OK;
    }
    double lamp[kMaxG];
    for (int g = 0; g < G; g++) lamp[g] = lambdas[g] * n2;
    rc = launch_opt_dp(P, lamp, G, s, (flags & ECASQ_EXACT_S) ? 1 : 0, wsp<void>(ws, pairs_off), true,
                       wsp<void>(ws, tables_off), qidx, mc, met, num_sms(), st);
    if (rc) return rc;
    rc = launch_gather_q(P.v, qidx, mc, G, s, Q_out, st);
    if (rc) return rc;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(m_out, mc, sizeof(int32_t) * G, cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(metrics, met, sizeof(double) * 4 * G, cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    for (int g = 0; g < G; g++)
        if (m_out[g] < 1) return ECASQ_EINFEASIBLE;
    return ECASQ_OK;
}

int ecasq_quantize_timeshare(const float *x, int64_t d, const float *Qm, int32_t mm, const float *Qp, int32_t mp,
                             double beta, uint64_t seed, uint64_t seed_ts, uint8_t *idx, uint8_t *sel,
                             uint32_t *counts, void *ws, size_t ws_bytes, double *rate, ecasq_stream_t stream) {
    if (!x || !Qm || !idx || !counts || d < 1 || d >= ((int64_t)1 << 31) || mm < 1 || mm > kMaxS || mp < 0 ||
        mp > kMaxS || !(beta >= 0.0 && beta <= 1.0) || (beta > 0.0 && (mp < 1 || !Qp)))
        return ECASQ_EINVAL;
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255) != 0 || ws_bytes < sizeof(DevStatus)) return ECASQ_EWORKSPACE;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    DevStatus *ds = wsp<DevStatus>(ws, 0);
    float qh[2 * kMaxS];
    ECASQ_CUDA_TRY(cudaMemcpyAsync(qh, Qm, 4 * (size_t)mm, cudaMemcpyDeviceToHost, st));
    if (mp > 0) ECASQ_CUDA_TRY(cudaMemcpyAsync(qh + kMaxS, Qp, 4 * (size_t)mp, cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaMemsetAsync(ds, 0, sizeof(DevStatus), st));
    ECASQ_CUDA_TRY(cudaMemsetAsync(counts, 0, 4 * (size_t)(mm + mp), st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    for (int r = 1; r < mm; r++)
        if (!(qh[r] > qh[r - 1])) return ECASQ_EINVAL;
    for (int r = 1; r < mp; r++)
        if (!(qh[kMaxS + r] > qh[kMaxS + r - 1])) return ECASQ_EINVAL;
    int rc = launch_quantize_timeshare(x, d, Qm, mm, mp > 0 ? Qp : Qm, mp, beta, seed, seed_ts, idx, sel, counts, ds,
                                       num_sms(), st);
    if (rc) return rc;
    uint32_t ch[2 * kMaxS];
    DevStatus h;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(&h, ds, sizeof(h), cudaMemcpyDeviceToHost, st));
    if (rate) ECASQ_CUDA_TRY(cudaMemcpyAsync(ch, counts, 4 * (size_t)(mm + mp), cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    if (h.range_err) return ECASQ_ERANGE;
    if (rate) {
        // each part coded with its own empirical law: -(1/d) sum_parts sum_r c_r log2(c_r / n_part)
        double bits = 0.0;
        for (int part = 0; part < 2; part++) {
            int off = part ? mm : 0, m = part ? mp : mm;
            double np_ = 0.0;
            for (int r = 0; r < m; r++) np_ += (double)ch[off + r];
            for (int r = 0; r < m; r++)
                if (ch[off + r]) bits -= (double)ch[off + r] * log2((double)ch[off + r] / np_);
        }
        *rate = bits / (double)d;
    }
    return ECASQ_OK;
}

// Short rows (d <= kScanTile, no refinement): every row runs the multiplier search
// of ecasq_solve in lockstep with the others -- one k_rows_pass launch per round
// for all rows still searching -- with the per-row arithmetic of the reference DP,
// so each row's result equals ecasq_solve on that row alone.  Rows with more than
// kRowsMaxP unique values, longer rows and refinement take ecasq_solve row by row.
static int solve_rows_batched(const float *X, int64_t rows, int64_t d, const ecasq_params_t *prm, void *ws,
                              size_t ws_bytes, float *Q, int32_t *m_out, ecasq_result_t *res, cudaStream_t st) {
    const int s = prm->s;
    Layout L1;
    make_layout(d, s, 1, &L1);
    int rc = add_resident_costs(prm->flags, &L1);
    if (rc) return rc;
    RowsLayout RL;
    rows_layout(d, s, rows, &RL);
    const size_t roff = align256(L1.total);
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255) != 0 || ws_bytes < roff + RL.total) return ECASQ_EWORKSPACE;
    char *rb = static_cast<char *>(ws) + roff;
    RowsData R;
    R.v = reinterpret_cast<float *>(rb + RL.v);
    R.w = reinterpret_cast<int64_t *>(rb + RL.w);
    R.N = reinterpret_cast<int64_t *>(rb + RL.N);
    R.S = reinterpret_cast<double *>(rb + RL.S);
    R.S2 = reinterpret_cast<double *>(rb + RL.S2);
    R.p = reinterpret_cast<int64_t *>(rb + RL.p);
    R.norm2 = reinterpret_cast<double *>(rb + RL.norm2);
    R.nonfinite = reinterpret_cast<int32_t *>(rb + RL.nonfinite);
    R.d = d;
    R.dcap = d;
    rc = launch_rows_prepare(X, rows, R, st);
    if (rc) return rc;
    std::vector<int64_t> ph(rows);
    std::vector<double> n2h(rows);
    std::vector<int32_t> nfh(rows);
    ECASQ_CUDA_TRY(cudaMemcpyAsync(ph.data(), R.p, 8 * (size_t)rows, cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(n2h.data(), R.norm2, 8 * (size_t)rows, cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(nfh.data(), R.nonfinite, 4 * (size_t)rows, cudaMemcpyDeviceToHost, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    for (int64_t r = 0; r < rows; r++)
        if (nfh[r]) return ECASQ_ENONFINITE;

    // per-row search state (the schedule of ecasq_solve)
    struct Row {
        std::vector<Eval> evals;
        double lo, hi;
        bool done = false, failed = false;
        int sel = -1, status = ECASQ_OK, passes = 0, nlam = 0;
        int best = -1;  // the feasible evaluation the selection rule prefers so far
    };
    std::vector<Row> st_rows(rows);
    const bool fixed = prm->lambda >= 0.0;
    double lo0 = prm->lambda_lo > 0.0 ? prm->lambda_lo : 1e-8;
    double hi0 = prm->lambda_hi > 0.0 ? prm->lambda_hi : 1e3;
    const int Rn = prm->search_rounds > 0 ? prm->search_rounds : 6;
    if (!fixed && !(hi0 > lo0)) return ECASQ_EINVAL;
    std::vector<int64_t> slow;  // rows that take ecasq_solve
    for (int64_t r = 0; r < rows; r++) {
        st_rows[r].lo = lo0;
        st_rows[r].hi = hi0;
        if (ph[r] > kRowsMaxP) { slow.push_back(r); st_rows[r].done = true; }
        else if (ph[r] == 1) st_rows[r].done = true;
        else st_rows[r].evals.reserve(fixed ? 1 : 8 + 7 * (size_t)Rn + 1);
    }
    int32_t *actd = reinterpret_cast<int32_t *>(rb + RL.act);
    double *lamd = reinterpret_cast<double *>(rb + RL.lam);
    int32_t *mcd = reinterpret_cast<int32_t *>(rb + RL.mcount);
    double *metd = reinterpret_cast<double *>(rb + RL.metrics);
    int32_t *qid = reinterpret_cast<int32_t *>(rb + RL.qidx);
    bool pairs_ready = false;
    // one pass over `act` rows, G multipliers each (lams: row-major [nact][G], vNMSE scale)
    auto pass = [&](const std::vector<int32_t> &act, const std::vector<double> &lams, int G) -> int {
        const int nact = (int)act.size();
        if (!nact) return ECASQ_OK;
        std::vector<double> lamp((size_t)nact * G);
        int pmax = 2;
        for (int b = 0; b < nact; b++) {
            for (int g = 0; g < G; g++) lamp[(size_t)b * G + g] = lams[(size_t)b * G + g] * n2h[act[b]];
            pmax = std::max<int>(pmax, (int)ph[act[b]]);
        }
        ECASQ_CUDA_TRY(cudaMemcpyAsync(actd, act.data(), 4 * (size_t)nact, cudaMemcpyHostToDevice, st));
        ECASQ_CUDA_TRY(cudaMemcpyAsync(lamd, lamp.data(), 8 * lamp.size(), cudaMemcpyHostToDevice, st));
        RowsPass A;
        A.R = R;
        A.rows = actd;
        A.lam = lamd;
        A.G = G;
        A.s = s;
        A.exact_s = (prm->flags & ECASQ_EXACT_S) ? 1 : 0;
        A.bp = reinterpret_cast<int32_t *>(rb + RL.bp);
        A.qidx = qid;
        A.mcount = mcd;
        A.metrics = metd;
        A.pairs = reinterpret_cast<double *>(rb + RL.pairs);
        A.pstride = RL.pstride;
        A.pairs_ready = pairs_ready ? 1 : 0;
        int r2 = launch_rows_pass(A, nact, pmax, st);
        pairs_ready = true;  // every active row of a later round was active in this one
        if (r2) return r2;
        std::vector<int32_t> mh((size_t)nact * G), qh((size_t)nact * G * s);
        std::vector<double> meth((size_t)nact * G * 4);
        ECASQ_CUDA_TRY(cudaMemcpyAsync(mh.data(), mcd, 4 * mh.size(), cudaMemcpyDeviceToHost, st));
        ECASQ_CUDA_TRY(cudaMemcpyAsync(qh.data(), qid, 4 * qh.size(), cudaMemcpyDeviceToHost, st));
        ECASQ_CUDA_TRY(cudaMemcpyAsync(meth.data(), metd, 8 * meth.size(), cudaMemcpyDeviceToHost, st));
        ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
        for (int b = 0; b < nact; b++) {
            Row &w = st_rows[act[b]];
            w.passes++;
            w.nlam += G;
            bool bad = false;
            for (int g = 0; g < G; g++) {
                const size_t q = (size_t)b * G + g;
                Eval e;
                e.lam = lams[q];
                e.m = mh[q];
                e.mse = meth[4 * q + 1];
                e.hs = meth[4 * q + 2];
                e.hx = meth[4 * q + 3];
                e.feas = fixed ? true : (e.hs <= prm->budget_bits);
                // the codebook is kept only where it can be selected: a fixed multiplier, the
                // closing pass at the bracket's upper end, or the best feasible point so far
                // (least MSE, then the smaller multiplier: the final selection's rule)
                const bool lead = e.feas && (w.best < 0 || e.mse < w.evals[w.best].mse ||
                                             (e.mse == w.evals[w.best].mse && e.lam < w.evals[w.best].lam));
                if (lead) w.best = (int)w.evals.size();
                if (lead || fixed || G == 1)
                    e.a.assign(qh.begin() + q * s, qh.begin() + q * s + std::max(e.m, 0));
                w.evals.push_back(e);
                if (e.m < 1) bad = true;
            }
            if (bad) { w.failed = true; w.done = true; w.status = ECASQ_EINFEASIBLE; }
        }
        return ECASQ_OK;
    };
    auto active = [&]() {
        std::vector<int32_t> act;
        for (int64_t r = 0; r < rows; r++)
            if (!st_rows[r].done) act.push_back((int32_t)r);
        return act;
    };
    if (fixed) {
        std::vector<int32_t> act = active();
        rc = pass(act, std::vector<double>(act.size(), prm->lambda), 1);
        if (rc) return rc;
        for (int32_t r : act)
            if (!st_rows[r].failed) st_rows[r].sel = 0;
    } else {
        double t[7];
        {  // multiplier 0 and the first round together
            std::vector<int32_t> act = active();
            midpoints7(lo0, hi0, t);
            std::vector<double> lams;
            for (size_t b = 0; b < act.size(); b++) {
                lams.push_back(0.0);
                lams.insert(lams.end(), t, t + 7);
            }
            rc = pass(act, lams, 8);
            if (rc) return rc;
            for (int32_t r : act) {
                Row &w = st_rows[r];
                if (w.failed) continue;
                if (w.evals[0].feas) { w.sel = 0; w.done = true; }
            }
        }
        for (int rr = 0; rr < Rn; rr++) {
            std::vector<int32_t> act = active();
            if (rr > 0) {
                std::vector<double> lams;
                for (int32_t r : act) {
                    midpoints7(st_rows[r].lo, st_rows[r].hi, t);
                    lams.insert(lams.end(), t, t + 7);
                }
                rc = pass(act, lams, 7);
                if (rc) return rc;
            }
            for (int32_t r : act) {
                Row &w = st_rows[r];
                if (w.failed) continue;
                const Eval *pts = &w.evals[w.evals.size() - 7];
                int f = -1;
                for (int q = 0; q < 7; q++)
                    if (pts[q].feas) { f = q; break; }
                if (f >= 0) {
                    double nlo = f > 0 ? pts[f - 1].lam : w.lo;
                    w.hi = pts[f].lam;
                    w.lo = nlo;
                } else {
                    w.lo = pts[6].lam;
                }
            }
        }
        std::vector<int32_t> need_hi;
        std::vector<double> his;
        for (int32_t r : active()) {
            Row &w = st_rows[r];
            for (size_t q = 0; q < w.evals.size(); q++) {
                const Eval &e = w.evals[q];
                if (e.feas && (w.sel < 0 || e.mse < w.evals[w.sel].mse ||
                               (e.mse == w.evals[w.sel].mse && e.lam < w.evals[w.sel].lam)))
                    w.sel = (int)q;
            }
            if (w.sel < 0) { need_hi.push_back(r); his.push_back(w.hi); }
        }
        rc = pass(need_hi, his, 1);
        if (rc) return rc;
        for (int32_t r : need_hi) {
            Row &w = st_rows[r];
            if (w.failed) continue;
            w.sel = (int)w.evals.size() - 1;
            if (!w.evals[w.sel].feas) w.status = ECASQ_EINFEASIBLE;
        }
    }
    // selected codebooks -> Q, m; results
    std::vector<int32_t> selh((size_t)rows * s, 0), mh(rows, 0);
    int status = ECASQ_OK;
    for (int64_t r = 0; r < rows; r++) {
        Row &w = st_rows[r];
        if (std::find(slow.begin(), slow.end(), r) != slow.end()) continue;
        double zero3[3] = {0.0, 0.0, 0.0};
        if (ph[r] == 1) {
            mh[r] = 1;
            selh[(size_t)r * s] = 0;
            fill_result(res ? &res[r] : nullptr, ECASQ_OK, 1, d, 1, fixed ? prm->lambda : 0.0, n2h[r], zero3, 0.0, 0, 0,
                        0, 0, 0);
            continue;
        }
        if (w.failed || w.sel < 0) {
            status = ECASQ_EINFEASIBLE;
            if (res) { memset(&res[r], 0, sizeof(res[r])); res[r].status = ECASQ_EINFEASIBLE; res[r].d = d; res[r].p = ph[r]; }
            continue;
        }
        const Eval &e = w.evals[w.sel];
        mh[r] = e.m;
        for (int q = 0; q < e.m; q++) selh[(size_t)r * s + q] = e.a[q];
        const double ev[3] = {e.mse, e.hs, e.hx};
        const double lamp = e.lam * n2h[r];
        if (w.status != ECASQ_OK) status = w.status;
        fill_result(res ? &res[r] : nullptr, w.status, e.m, d, ph[r], e.lam, n2h[r], ev, ev[0] + lamp * ev[1], w.passes,
                    w.nlam, 0, candidates_of(ph[r], s, 0) * w.nlam, 0);
    }
    int32_t *seld = reinterpret_cast<int32_t *>(rb + RL.sel);
    int32_t *md = reinterpret_cast<int32_t *>(rb + RL.m);
    ECASQ_CUDA_TRY(cudaMemcpyAsync(seld, selh.data(), 4 * selh.size(), cudaMemcpyHostToDevice, st));
    ECASQ_CUDA_TRY(cudaMemcpyAsync(md, mh.data(), 4 * mh.size(), cudaMemcpyHostToDevice, st));
    rc = launch_rows_gather(R, seld, md, rows, s, Q, st);
    if (rc) return rc;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(m_out, md, 4 * (size_t)rows, cudaMemcpyDeviceToDevice, st));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    // rows with many unique values: the single-row path (its layout sits before the row data)
    for (int64_t r : slow) {
        ecasq_result_t one;
        rc = ecasq_solve(X + r * d, d, prm, ws, roff, Q + r * s, &one, reinterpret_cast<ecasq_stream_t>(st));
        if (rc != ECASQ_OK && rc != ECASQ_EINFEASIBLE) return rc;
        if (rc == ECASQ_EINFEASIBLE) status = rc;
        ECASQ_CUDA_TRY(cudaMemcpyAsync(m_out + r, &one.m, sizeof(int32_t), cudaMemcpyHostToDevice, st));
        if (res) res[r] = one;
    }
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    return status;
}

int ecasq_solve_batched(const float *X, int64_t rows, int64_t d, const ecasq_params_t *prm, void *ws,
                        size_t ws_bytes, float *Q, int32_t *m_out, ecasq_result_t *res, ecasq_stream_t stream) {
    if (!X || !Q || !m_out || rows < 1 || d < 1 || d >= ((int64_t)1 << 31) || !params_ok(prm)) return ECASQ_EINVAL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (d <= kScanTile && prm->refine_max_rounds == 0)
        return solve_rows_batched(X, rows, d, prm, ws, ws_bytes, Q, m_out, res, st);
    int status = ECASQ_OK;
    for (int64_t r = 0; r < rows; r++) {
        ecasq_result_t one;
        int rc = ecasq_solve(X + r * d, d, prm, ws, ws_bytes, Q + r * prm->s, &one, stream);
        if (rc != ECASQ_OK && rc != ECASQ_EINFEASIBLE) return rc;
        if (rc == ECASQ_EINFEASIBLE) status = rc;
        ECASQ_CUDA_TRY(cudaMemcpyAsync(m_out + r, &one.m, sizeof(int32_t), cudaMemcpyHostToDevice, st));
        if (res) res[r] = one;
    }
    ECASQ_CUDA_TRY(cudaStreamSynchronize(st));
    return status;
}

}  // extern "C"
