// prep.cu -- step 1 of every solve: sorted copy of x, weighted histogram
// (Sec. 2: "we assume X is sorted ... work with its weighted histogram") and the
// prefix sums N, S, S2 of App. E, accumulated in double-double.
//
// Sort: LSD radix sort, 4 passes of 8 bits over order-preserving uint32 keys
// (-0.0 folded into +0.0).  Each pass: per-block digit counts, one scan of the
// [digit][block] count matrix, and a stable scatter whose in-block ranks come
// from warp match masks.
#include <algorithm>

#include "common.cuh"

namespace ecasq {

__device__ __forceinline__ uint32_t f2key(float f) {
    uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float key2f(uint32_t k) {
    uint32_t u = (k & 0x80000000u) ? (k & 0x7fffffffu) : ~k;
    return __uint_as_float(u);
}

__global__ void k_make_keys(const float *__restrict__ x, int64_t d, uint32_t *__restrict__ keys,
                            DevStatus *st) {
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (; i < d; i += stride) {
        float f = x[i];
        if (!isfinite(f)) st->nonfinite = 1;
        if (f == 0.0f) f = 0.0f;
        keys[i] = f2key(f);
    }
}

// counts[digit * nb + block] = number of keys of the block with that digit.
__global__ void __launch_bounds__(256) k_radix_count(const uint32_t *__restrict__ keys, int64_t d, int shift,
                                                     uint32_t *__restrict__ counts, int nb) {
    __shared__ uint32_t h[256];
    h[threadIdx.x] = 0;
    __syncthreads();
    int64_t base = (int64_t)blockIdx.x * kSortTile;
    for (int r = 0; r < kSortTile / 256; r++) {
        int64_t i = base + r * 256 + threadIdx.x;
        if (i < d) atomicAdd(&h[(keys[i] >> shift) & 255u], 1u);
    }
    __syncthreads();
    counts[(size_t)threadIdx.x * nb + blockIdx.x] = h[threadIdx.x];
}

// In-place exclusive scan of uint32 values.  Block b scans a[b*chunk .. min(n, (b+1)*chunk))
// by 1024 threads, in coalesced tiles of 4096 (four consecutive values per thread) with a
// running carry that starts at carry_in[b] (0 when carry_in is null).  One block with
// chunk = n scans the whole array; with several blocks, carry_in holds the exclusive
// prefix of the chunks' totals (k_scan_chunk_sums, then a one-block scan of those).
__global__ void __launch_bounds__(1024) k_scan_u32(uint32_t *a, int64_t n, int64_t chunk,
                                                   const uint32_t *carry_in) {
    __shared__ uint32_t wsum[32];
    __shared__ uint32_t carry;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const int64_t lo = (int64_t)blockIdx.x * chunk, hi = min(n, lo + chunk);
    if (threadIdx.x == 0) carry = carry_in ? carry_in[blockIdx.x] : 0u;
    __syncthreads();
    for (int64_t base = lo; base < hi; base += 4 * 1024) {
        const int64_t i0 = base + 4 * (int64_t)threadIdx.x;
        uint32_t v[4];
#pragma unroll
        for (int e = 0; e < 4; e++) v[e] = i0 + e < hi ? a[i0 + e] : 0u;
        const uint32_t s = v[0] + v[1] + v[2] + v[3];
        uint32_t incl = s;
        for (int o = 1; o < 32; o <<= 1) {
            uint32_t t = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += t;
        }
        if (lane == 31) wsum[wid] = incl;
        __syncthreads();
        if (wid == 0) {
            uint32_t w = wsum[lane], wi = w;
            for (int o = 1; o < 32; o <<= 1) {
                uint32_t t = __shfl_up_sync(0xffffffffu, wi, o);
                if (lane >= o) wi += t;
            }
            wsum[lane] = wi - w;
        }
        __syncthreads();
        uint32_t run = carry + wsum[wid] + incl - s;
#pragma unroll
        for (int e = 0; e < 4; e++) {
            if (i0 + e < hi) a[i0 + e] = run;
            run += v[e];
        }
        __syncthreads();  // every thread has read carry and wsum
        if (threadIdx.x == blockDim.x - 1) carry = run;  // the old carry plus this tile's total
        __syncthreads();
    }
}

// Totals of the chunks a[b*chunk .. min(n, (b+1)*chunk)), one block of 1024 per chunk.
__global__ void __launch_bounds__(1024) k_scan_chunk_sums(const uint32_t *__restrict__ a, int64_t n, int64_t chunk,
                                                          uint32_t *__restrict__ sums) {
    __shared__ uint32_t wsum[32];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const int64_t lo = (int64_t)blockIdx.x * chunk, hi = min(n, lo + chunk);
    uint32_t t = 0;
    for (int64_t i = lo + threadIdx.x; i < hi; i += blockDim.x) t += a[i];
    for (int o = 16; o; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (lane == 0) wsum[wid] = t;
    __syncthreads();
    if (wid == 0) {
        t = wsum[lane];
        for (int o = 16; o; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (lane == 0) sums[blockIdx.x] = t;
    }
}

// Exclusive scan of the n radix counts: one block while n is small, else the chunks'
// totals, a one-block scan of them and a scan of every chunk from its offset
// (sums: scratch of at least 1024 uint32 values).
static void scan_counts(uint32_t *a, int64_t n, uint32_t *sums, cudaStream_t stream) {
    constexpr int64_t kOneBlock = 1 << 16;
    if (n <= kOneBlock) {
        note_launch();
        k_scan_u32<<<1, 1024, 0, stream>>>(a, n, n, nullptr);
        return;
    }
    const int64_t nchunks = std::min<int64_t>(1024, cdiv(n, 16384));
    const int64_t chunk = cdiv(cdiv(n, nchunks), 4096) * 4096;
    const int64_t nc = cdiv(n, chunk);
    note_launch();
    k_scan_chunk_sums<<<(unsigned)nc, 1024, 0, stream>>>(a, n, chunk, sums);
    note_launch();
    k_scan_u32<<<1, 1024, 0, stream>>>(sums, nc, nc, nullptr);
    note_launch();
    k_scan_u32<<<(unsigned)nc, 1024, 0, stream>>>(a, n, chunk, sums);
}

// Stable scatter of one radix pass.  Positions inside a tile are visited in
// rounds of 256 (round r covers tile positions r*256 .. r*256+255, thread t
// holding position r*256 + t), so (round, warp, lane) is the input order.
__global__ void __launch_bounds__(256) k_radix_scatter(const uint32_t *__restrict__ kin, uint32_t *__restrict__ kout,
                                                       int64_t d, int shift, const uint32_t *__restrict__ offs,
                                                       int nb) {
    __shared__ uint32_t cnt[8][256];
    __shared__ uint32_t base[8][256];
    __shared__ uint32_t run[256];
    int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    uint32_t lt_mask = (1u << lane) - 1u;
    run[threadIdx.x] = offs[(size_t)threadIdx.x * nb + blockIdx.x];
    int64_t tbase = (int64_t)blockIdx.x * kSortTile;
    for (int r = 0; r < kSortTile / 256; r++) {
        for (int w = 0; w < 8; w++) cnt[w][threadIdx.x] = 0;
        __syncthreads();
        int64_t i = tbase + r * 256 + threadIdx.x;
        bool valid = i < d;
        uint32_t key = valid ? kin[i] : 0u;
        uint32_t dig = valid ? ((key >> shift) & 255u) : (256u + (uint32_t)lane);
        uint32_t peers = __match_any_sync(0xffffffffu, dig);
        uint32_t rank = __popc(peers & lt_mask);
        if (valid && rank == 0) cnt[wid][dig] = __popc(peers);
        __syncthreads();
        {
            uint32_t acc = run[threadIdx.x];
            for (int w = 0; w < 8; w++) {
                base[w][threadIdx.x] = acc;
                acc += cnt[w][threadIdx.x];
            }
            run[threadIdx.x] = acc;
        }
        __syncthreads();
        if (valid) kout[base[wid][dig] + rank] = key;
        __syncthreads();
    }
}

// Pass A of the histogram scan: per tile of kScanTile sorted keys, the number
// of unique-value heads and the double-double sums of x and x^2.
struct DDPart { double s_hi, s_lo, q_hi, q_lo; int64_t heads; int64_t pad; };


template <typename T>
__device__ __forceinline__ T shfl_up(T v, int o) { return __shfl_up_sync(0xffffffffu, v, o); }

struct ScanVal { dd s, q; int64_t h; };

__device__ __forceinline__ ScanVal sv_add(const ScanVal &a, const ScanVal &b) {
    return {dd_add(a.s, b.s), dd_add(a.q, b.q), a.h + b.h};
}

// Block-wide inclusive scan of one ScanVal per thread (256 threads).
__device__ ScanVal block_scan_incl(ScanVal v, ScanVal *wtot, ScanVal &total) {
    int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    for (int o = 1; o < 32; o <<= 1) {
        ScanVal t;
        t.s.hi = shfl_up(v.s.hi, o); t.s.lo = shfl_up(v.s.lo, o);
        t.q.hi = shfl_up(v.q.hi, o); t.q.lo = shfl_up(v.q.lo, o);
        t.h = shfl_up(v.h, o);
        if (lane >= o) v = sv_add(t, v);
    }
    if (lane == 31) wtot[wid] = v;
    __syncthreads();
    if (threadIdx.x == 0) {
        ScanVal acc = wtot[0];
        for (int w = 1; w < 8; w++) { acc = sv_add(acc, wtot[w]); wtot[w] = acc; }
    }
    __syncthreads();
    if (wid > 0) v = sv_add(wtot[wid - 1], v);
    total = wtot[7];
    __syncthreads();
    return v;
}

// The thread's kHistPer consecutive sorted keys starting at base (positions >= d are
// left out): x as binary64, the sums of x and x^2 in double-double (x^2 of a binary32
// value is exact in binary64) and the number of heads.  One fixed order per thread, so
// the single-row and the batched paths, which both call it, give the same bits.
__device__ __forceinline__ ScanVal hist_thread_sums(const uint32_t *keys, int64_t d, int64_t base) {
    ScanVal v{{0.0, 0.0}, {0.0, 0.0}, 0};
    uint32_t prev = base > 0 && base - 1 < d ? keys[base - 1] : 0u;
#pragma unroll 4
    for (int e = 0; e < kHistPer; e++) {
        const int64_t i = base + e;
        if (i < d) {
            const uint32_t k = keys[i];
            const double x = (double)key2f(k);
            v.s = dd_add_d(v.s, x);
            v.q = dd_add_d(v.q, __dmul_rn(x, x));
            v.h += (i == 0 || k != prev) ? 1 : 0;
            prev = k;
        }
    }
    return v;
}

// Pass C for the thread's keys: from the exclusive prefix `run` before them, every head
// i writes its unique index u = run.h, v[u], N[u] = i, S[u] and S2[u] (hi at [u], lo at
// [lo_off + u]); the last position d - 1 also writes the totals at index p and returns
// p and ||X||^2 through p_out and norm2_out.
__device__ __forceinline__ void hist_thread_fill(const uint32_t *keys, int64_t d, int64_t base, ScanVal run,
                                                 float *v, int64_t *N, double *S, double *S2, int64_t lo_off,
                                                 int64_t *p_out, double *norm2_out) {
    uint32_t prev = base > 0 && base - 1 < d ? keys[base - 1] : 0u;
#pragma unroll 4
    for (int e = 0; e < kHistPer; e++) {
        const int64_t i = base + e;
        if (i >= d) break;
        const uint32_t k = keys[i];
        const double x = (double)key2f(k);
        const bool head = i == 0 || k != prev;
        prev = k;
        if (head) {
            const int64_t u = run.h;
            v[u] = (float)x;
            N[u] = i;
            S[u] = run.s.hi; S[lo_off + u] = run.s.lo;
            S2[u] = run.q.hi; S2[lo_off + u] = run.q.lo;
        }
        run.s = dd_add_d(run.s, x);
        run.q = dd_add_d(run.q, __dmul_rn(x, x));
        run.h += head ? 1 : 0;
        if (i == d - 1) {
            const int64_t p = run.h;
            N[p] = d;
            S[p] = run.s.hi; S[lo_off + p] = run.s.lo;
            S2[p] = run.q.hi; S2[lo_off + p] = run.q.lo;
            *p_out = p;
            *norm2_out = run.q.hi;
        }
    }
}

__global__ void __launch_bounds__(256) k_hist_partials(const uint32_t *__restrict__ keys, int64_t d, DDPart *part) {
    __shared__ ScanVal wtot[8];
    const ScanVal v = hist_thread_sums(keys, d, (int64_t)blockIdx.x * kHistTile + (int64_t)threadIdx.x * kHistPer);
    ScanVal tot;
    block_scan_incl(v, wtot, tot);
    if (threadIdx.x == 0) part[blockIdx.x] = {tot.s.hi, tot.s.lo, tot.q.hi, tot.q.lo, tot.h, 0};
}

// Exclusive scan of the tile partials (one thread, in order; nb is small).
// Exclusive scan of the tiles' partials by one block of 256 threads: each thread sums a
// contiguous run of tiles in order, the runs' totals are scanned across the block
// (block_scan_incl), and each thread then writes its run's exclusive prefixes.
__global__ void __launch_bounds__(256) k_hist_scan_partials(DDPart *part, int64_t nb) {
    __shared__ ScanVal wtot[8];
    __shared__ ScanVal incl_all[256];
    const int64_t per = cdiv(nb, (int64_t)blockDim.x);
    const int64_t lo = min((int64_t)threadIdx.x * per, nb), hi = min(lo + per, nb);
    ScanVal s{{0.0, 0.0}, {0.0, 0.0}, 0};
    for (int64_t b = lo; b < hi; b++) {
        ScanVal t{{part[b].s_hi, part[b].s_lo}, {part[b].q_hi, part[b].q_lo}, part[b].heads};
        s = sv_add(s, t);
    }
    ScanVal total;
    incl_all[threadIdx.x] = block_scan_incl(s, wtot, total);
    __syncthreads();
    ScanVal acc = threadIdx.x > 0 ? incl_all[threadIdx.x - 1] : ScanVal{{0.0, 0.0}, {0.0, 0.0}, 0};
    for (int64_t b = lo; b < hi; b++) {
        ScanVal t{{part[b].s_hi, part[b].s_lo}, {part[b].q_hi, part[b].q_lo}, part[b].heads};
        part[b] = {acc.s.hi, acc.s.lo, acc.q.hi, acc.q.lo, acc.h, 0};
        acc = sv_add(acc, t);
    }
}

// Pass C: per sorted position i that starts a run of equal keys (a head), the
// unique index u and v[u], N[u] = i, S[u], S2[u] (exclusive prefix sums).
// The last position also writes N[p] = d, S[p], S2[p], p and ||X||^2.
__global__ void __launch_bounds__(256) k_hist_fill(const uint32_t *__restrict__ keys, int64_t d, const DDPart *part,
                                                   float *v, int64_t *N, double *S, double *S2, DevStatus *st,
                                                   int64_t pcap) {
    __shared__ ScanVal wtot[8];
    const int64_t base = (int64_t)blockIdx.x * kHistTile + (int64_t)threadIdx.x * kHistPer;
    const ScanVal loc = hist_thread_sums(keys, d, base);
    ScanVal tot;
    const ScanVal incl = block_scan_incl(loc, wtot, tot);
    const DDPart &pb = part[blockIdx.x];
    const ScanVal off{{pb.s_hi, pb.s_lo}, {pb.q_hi, pb.q_lo}, pb.heads};
    // exclusive prefix before this thread's first element
    ScanVal run{dd_sub(incl.s, loc.s), dd_sub(incl.q, loc.q), incl.h - loc.h};
    run = sv_add(off, run);
    hist_thread_fill(keys, d, base, run, v, N, S, S2, pcap + 1, &st->p, &st->norm2);
}

// The arrays were written with lo parts at offset pcap+1 (pcap = d); repack
// them to offset p+1 so that every later kernel indexes (hi[0..p], lo[0..p]).
__global__ void k_hist_finish(int64_t *N, int64_t *w, double *S, double *S2, const DevStatus *st, int64_t pcap,
                              double *Sp, double *S2p) {
    int64_t p = st->p;
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (; i <= p; i += stride) {
        if (i < p) w[i] = N[i + 1] - N[i];
        Sp[i] = S[i]; Sp[p + 1 + i] = S[pcap + 1 + i];
        S2p[i] = S2[i]; S2p[p + 1 + i] = S2[pcap + 1 + i];
    }
}

// ------------------------------------------------------------ short rows
// One block per row of length d <= kScanTile: the sorted keys (bitonic sort in
// shared memory; the order is unique, so any exact sort gives the same keys) and
// then the arithmetic of k_hist_fill for a single tile (zero tile offset), so that
// v, w, N, S, S2, p and ||X||^2 of every row equal what prepare_device gives for
// that row alone.
__global__ void __launch_bounds__(256) k_rows_prepare(const float *__restrict__ X, RowsData R) {
    __shared__ uint32_t keys[kScanTile];
    __shared__ ScanVal wtot[8];
    __shared__ int nonfin;
    const int64_t row = blockIdx.x;
    const int d = (int)R.d;
    const float *x = X + row * R.d;
    if (threadIdx.x == 0) nonfin = 0;
    __syncthreads();
    for (int i = threadIdx.x; i < kScanTile; i += blockDim.x) {
        uint32_t k = 0xFFFFFFFFu;  // above every finite key: padding sorts last
        if (i < d) {
            float f = x[i];
            if (!isfinite(f)) nonfin = 1;
            if (f == 0.0f) f = 0.0f;
            k = f2key(f);
        }
        keys[i] = k;
    }
    __syncthreads();
    int n2 = 1;
    while (n2 < d) n2 <<= 1;
    for (int kk = 2; kk <= n2; kk <<= 1) {
        for (int jj = kk >> 1; jj > 0; jj >>= 1) {
            for (int i = threadIdx.x; i < n2; i += blockDim.x) {
                int l = i ^ jj;
                if (l > i) {
                    uint32_t a = keys[i], b = keys[l];
                    bool up = (i & kk) == 0;
                    if ((a > b) == up) { keys[i] = b; keys[l] = a; }
                }
            }
            __syncthreads();
        }
    }
    const int64_t dcap = R.dcap;
    float *v = R.v + row * dcap;
    int64_t *N = R.N + row * (dcap + 1), *w = R.w + row * dcap;
    double *S = R.S + row * 2 * (dcap + 1), *S2 = R.S2 + row * 2 * (dcap + 1);
    // k_hist_fill, one tile
    const int64_t base = (int64_t)threadIdx.x * kHistPer;
    const ScanVal loc = hist_thread_sums(keys, d, base);
    ScanVal tot;
    const ScanVal incl = block_scan_incl(loc, wtot, tot);
    const int64_t p = tot.h;
    const ScanVal off{{0.0, 0.0}, {0.0, 0.0}, 0};
    ScanVal run{dd_sub(incl.s, loc.s), dd_sub(incl.q, loc.q), incl.h - loc.h};
    run = sv_add(off, run);
    hist_thread_fill(keys, d, base, run, v, N, S, S2, p + 1, R.p + row, R.norm2 + row);
    __syncthreads();
    for (int u = threadIdx.x; u < p; u += blockDim.x) w[u] = N[u + 1] - N[u];
    if (threadIdx.x == 0) R.nonfinite[row] = nonfin;
}

int launch_rows_prepare(const float *X, int64_t rows, const RowsData &R, cudaStream_t st) {
    if (R.d < 1 || R.d > kScanTile) return ECASQ_EINVAL;
    note_launch();
    k_rows_prepare<<<(unsigned)rows, 256, 0, st>>>(X, R);
    ECASQ_LAUNCH_CHECK();
    return ECASQ_OK;
}

// ------------------------------------------------------------ general P
// The histogram view over a caller-given candidate set P (Sec. 5, App. E): for
// every grid point t, u_t = #{unique x <= p_t}; N, S, S2 at t+1 are the unique-value
// prefix sums at u_t (the sums of all entries x <= p_t), so w_t = #{p_(t-1) < x <= p_t}.
// Flags st->range_err when P is not strictly ascending and finite, starts above min x
// or ends below max x (App. E: then no quantizer drawn from P spans X), and records
// the sizes of the first- and last-value sets L = {a : p_a <= min x} and
// R = {b : p_b >= max x} of eqs. apx_base and apx_final in st->grid_nL, grid_nR.
// vX, NX, SX, S2X: the unique-value arrays (pX values, packed hi | lo).
__global__ void k_grid_prefix(const float *__restrict__ P, int64_t n, const float *__restrict__ vX,
                              const int64_t *__restrict__ NX, const double *__restrict__ SX,
                              const double *__restrict__ S2X, int64_t pX, float *v, int64_t *w, int64_t *N, double *S,
                              double *S2, DevStatus *st) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < n; t += stride) {
        float pt = P[t];
        if (pt == 0.0f) pt = 0.0f;
        bool bad = !isfinite(pt);
        if (t > 0 && !(P[t] > P[t - 1])) bad = true;
        if (t == 0 && !(pt <= vX[0])) bad = true;
        if (t == n - 1 && !(pt >= vX[pX - 1])) bad = true;
        if (bad) st->range_err = 1;
        // L = {a : p_a <= min x} and R = {b : p_b >= max x} are runs at the two ends
        // (P ascending): the last member of L and the first of R record the sizes
        if (pt <= vX[0] && (t == n - 1 || !(P[t + 1] <= vX[0]))) st->grid_nL = t + 1;
        if (pt >= vX[pX - 1] && (t == 0 || !(P[t - 1] >= vX[pX - 1]))) st->grid_nR = n - t;
        // u = #{unique values <= pt} (binary search)
        int64_t lo = 0, hi = pX;
        while (lo < hi) {
            int64_t mid = (lo + hi) >> 1;
            if (vX[mid] <= pt) lo = mid + 1; else hi = mid;
        }
        v[t] = pt;
        N[t + 1] = NX[lo];
        S[t + 1] = SX[lo]; S[n + 1 + t + 1] = SX[pX + 1 + lo];
        S2[t + 1] = S2X[lo]; S2[n + 1 + t + 1] = S2X[pX + 1 + lo];
        if (t == 0) { N[0] = 0; S[0] = 0.0; S[n + 1] = 0.0; S2[0] = 0.0; S2[n + 1] = 0.0; }
    }
}

__global__ void k_grid_weights(const int64_t *N, int64_t n, int64_t *w) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < n; t += stride) w[t] = N[t + 1] - N[t];
}

int launch_grid_prefix(const float *P, int64_t n, const float *vX, const int64_t *NX, const double *SX,
                       const double *S2X, int64_t pX, float *v, int64_t *w, int64_t *N, double *S, double *S2,
                       DevStatus *st, cudaStream_t stream) {
    const unsigned blocks = (unsigned)std::min<int64_t>(cdiv(n, 256), 4096);
    note_launch();
    k_grid_prefix<<<blocks, 256, 0, stream>>>(P, n, vX, NX, SX, S2X, pX, v, w, N, S, S2, st);
    ECASQ_LAUNCH_CHECK();
    note_launch();
    k_grid_weights<<<blocks, 256, 0, stream>>>(N, n, w);
    ECASQ_LAUNCH_CHECK();
    return ECASQ_OK;
}

int prepare_device(const float *x, int64_t d, void *ws, const Layout &L, cudaStream_t stream, int64_t *p_host,
                   double *norm2_host) {
    DevStatus *st = wsp<DevStatus>(ws, L.status);
    uint32_t *k0 = wsp<uint32_t>(ws, L.keys0), *k1 = wsp<uint32_t>(ws, L.keys1);
    uint32_t *cnt = wsp<uint32_t>(ws, L.rcount);
    ECASQ_CUDA_TRY(cudaMemsetAsync(st, 0, sizeof(DevStatus), stream));
    int nb = (int)cdiv(d, kSortTile);
    note_launch();
    k_make_keys<<<(unsigned)std::min<int64_t>(cdiv(d, 256), 4096), 256, 0, stream>>>(x, d, k0, st);
    ECASQ_LAUNCH_CHECK();
    uint32_t *a = k0, *b = k1;
    for (int shift = 0; shift < 32; shift += 8) {
        note_launch();
        k_radix_count<<<nb, 256, 0, stream>>>(a, d, shift, cnt, nb);
        scan_counts(cnt, (int64_t)256 * nb, wsp<uint32_t>(ws, L.v), stream);  // v is free until the histogram
        note_launch();
        k_radix_scatter<<<nb, 256, 0, stream>>>(a, b, d, shift, cnt, nb);
        ECASQ_LAUNCH_CHECK();
        uint32_t *t = a; a = b; b = t;
    }
    // a == k0 holds the sorted keys
    int64_t nbs = cdiv(d, kHistTile);  // the layout holds cdiv(d, kScanTile) >= nbs partials
    DDPart *part = wsp<DDPart>(ws, L.part);
    // scratch copies of N/S/S2 with lo parts at offset d+1 live in keys1 / dp area
    double *Stmp = wsp<double>(ws, L.dp64);
    double *S2tmp = Stmp + 2 * (d + 1);
    note_launch();
    k_hist_partials<<<(unsigned)nbs, 256, 0, stream>>>(a, d, part);
    note_launch();
    k_hist_scan_partials<<<1, 256, 0, stream>>>(part, nbs);
    note_launch();
    k_hist_fill<<<(unsigned)nbs, 256, 0, stream>>>(a, d, part, wsp<float>(ws, L.v), wsp<int64_t>(ws, L.N), Stmp,
                                                 S2tmp, st, d);
    ECASQ_LAUNCH_CHECK();
    note_launch();
    k_hist_finish<<<(unsigned)std::min<int64_t>(cdiv(d + 1, 256), 4096), 256, 0, stream>>>(
        wsp<int64_t>(ws, L.N), wsp<int64_t>(ws, L.w), Stmp, S2tmp, st, d, wsp<double>(ws, L.S),
        wsp<double>(ws, L.S2));
    ECASQ_LAUNCH_CHECK();
    DevStatus h;
    ECASQ_CUDA_TRY(cudaMemcpyAsync(&h, st, sizeof(DevStatus), cudaMemcpyDeviceToHost, stream));
    ECASQ_CUDA_TRY(cudaStreamSynchronize(stream));
    if (h.nonfinite) return ECASQ_ENONFINITE;
    *p_host = h.p;
    *norm2_host = h.norm2;
    return ECASQ_OK;
}

}  // namespace ecasq
