// quantize.cu -- unbiased stochastic quantization (Sec. 2) and the index
// histogram behind the empirical entropy (Sec. 1).
//
// Entry i (original order) with a = max{q <= x}: if x == a it keeps a's index;
// otherwise it rounds up to the next value iff
//   fl32(fl32(k * 2^-24) * fl32(b - a)) < fl32(x - a),
// k = top 24 bits of SplitMix64(seed + (i+1) * 0x9E3779B97F4A7C15)
// (Steele, Lea and Flood 2014).  HBM-bound: 4 B read + 1 B written per entry;
// the codebook and the histogram live in shared memory.
#include <algorithm>

#include "common.cuh"

namespace ecasq {

__device__ __forceinline__ uint64_t splitmix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;

// half: the largest power of two <= m - 1 (0 when m = 1); q[m .. 2 half - 1] hold +inf, so
// the search needs no bound test.  zc = seed + (i + 1) * gamma (mod 2^64) for entry i.
__device__ __forceinline__ int search_half(int m) { return m > 1 ? 1 << (31 - __clz(m - 1)) : 0; }

__device__ __forceinline__ int quant_one(float xv, uint64_t zc, const float *q, int m, int half, bool &bad) {
    if (!(xv >= q[0] && xv <= q[m - 1])) { bad = true; return 0; }
    int t = 0;  // largest t with q[t] <= x: one step per bit of m - 1, the same count in every lane
    for (int b = half; b; b >>= 1)
        if (q[t + b] <= xv) t += b;
    if (q[t] != xv) {
        uint64_t z = splitmix64(zc);
        float k = __fmul_rn((float)(uint32_t)(z >> 40), 0x1p-24f);
        float d1 = __fsub_rn(xv, q[t]);
        float d2 = __fsub_rn(q[t + 1], q[t]);
        if (__fmul_rn(k, d2) < d1) t += 1;
    }
    return t;
}

// Codebooks of at most kPrivBins values count their indices in per-thread
// histograms: 16-bit counters packed in pairs, word w of thread t at
// ph[w * 256 + t] (each thread its own bank column: no conflicts, no atomics).  A
// thread folds its counters into the block's 32-bit totals after every
// kFoldEntries of its entries, before any counter could pass 65535 (only inputs of
// more than about 10^10 entries get that far).
constexpr int kPrivBins = 32;
constexpr int kQThreads = 256;
constexpr int kFoldEntries = 32768;

__device__ __forceinline__ void priv_count(uint32_t *ph, int t) {
    ph[(t >> 1) * kQThreads + threadIdx.x] += 1u << ((t & 1) << 4);
}
__device__ __forceinline__ void priv_fold(uint32_t *ph, uint32_t *hcount, int m) {
    for (int w = 0; w < (m + 1) >> 1; w++) {
        const uint32_t v = ph[w * kQThreads + threadIdx.x];
        if (v) {
            if (v & 0xffffu) atomicAdd(&hcount[2 * w], v & 0xffffu);
            if (v >> 16) atomicAdd(&hcount[2 * w + 1], v >> 16);
            ph[w * kQThreads + threadIdx.x] = 0;
        }
    }
}

// Encode.  Vector path: each thread takes two groups of four entries per step (two
// 16-byte loads in flight before any arithmetic), writes four indices per group.
template <bool PRIV>
__global__ void __launch_bounds__(kQThreads) k_quantize(const float *__restrict__ x, int64_t d,
                                                        const float *__restrict__ Q, int m, uint64_t seed,
                                                        uint8_t *__restrict__ idx, uint32_t *__restrict__ counts,
                                                        DevStatus *st) {
    __shared__ float q[kMaxS];
    __shared__ uint32_t hcount[kMaxS];
    __shared__ uint32_t ph[PRIV ? (kPrivBins / 2) * kQThreads : 1];
    for (int r = threadIdx.x; r < kMaxS; r += blockDim.x) {
        q[r] = r < m ? Q[r] : CUDART_INF_F;
        hcount[r] = 0;
    }
    const int half = search_half(m);
    if (PRIV)
        for (int w = 0; w < kPrivBins / 2; w++) ph[w * kQThreads + threadIdx.x] = 0;
    __syncthreads();
    auto count = [&](int t) {
        if (PRIV) priv_count(ph, t); else atomicAdd(&hcount[t], 1u);
    };
    bool bad = false;
    const bool vec = ((reinterpret_cast<uintptr_t>(x) & 15) == 0) && ((reinterpret_cast<uintptr_t>(idx) & 3) == 0);
    const int64_t ngroups = vec ? d / 4 : 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t g0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const float4 *x4 = reinterpret_cast<const float4 *>(x);
    uchar4 *i4 = reinterpret_cast<uchar4 *>(idx);
    int since_fold = 0;  // entries counted since the last fold
    for (int64_t g = g0; g < ngroups; g += 2 * stride) {
        const int64_t h = g + stride;
        const bool two = h < ngroups;
        const float4 xa = x4[g];
        const float4 xb = two ? x4[h] : make_float4(0.f, 0.f, 0.f, 0.f);
        {
            const uint64_t z0 = seed + (uint64_t)(4 * g + 1) * kGamma;  // entries 4g .. 4g+3: z0 + r gamma
            const int t0 = quant_one(xa.x, z0, q, m, half, bad), t1 = quant_one(xa.y, z0 + kGamma, q, m, half, bad);
            const int t2 = quant_one(xa.z, z0 + 2 * kGamma, q, m, half, bad);
            const int t3 = quant_one(xa.w, z0 + 3 * kGamma, q, m, half, bad);
            i4[g] = make_uchar4((uint8_t)t0, (uint8_t)t1, (uint8_t)t2, (uint8_t)t3);
            count(t0); count(t1); count(t2); count(t3);
        }
        if (two) {
            const uint64_t z0 = seed + (uint64_t)(4 * h + 1) * kGamma;
            const int t0 = quant_one(xb.x, z0, q, m, half, bad), t1 = quant_one(xb.y, z0 + kGamma, q, m, half, bad);
            const int t2 = quant_one(xb.z, z0 + 2 * kGamma, q, m, half, bad);
            const int t3 = quant_one(xb.w, z0 + 3 * kGamma, q, m, half, bad);
            i4[h] = make_uchar4((uint8_t)t0, (uint8_t)t1, (uint8_t)t2, (uint8_t)t3);
            count(t0); count(t1); count(t2); count(t3);
        }
        if (PRIV && (since_fold += 8) >= kFoldEntries) {
            priv_fold(ph, hcount, m);
            since_fold = 0;
        }
    }
    for (int64_t i = 4 * ngroups + g0; i < d; i += stride) {
        const int t = quant_one(x[i], seed + (uint64_t)(i + 1) * kGamma, q, m, half, bad);
        idx[i] = (uint8_t)t;
        count(t);
        if (PRIV && ++since_fold >= kFoldEntries) {
            priv_fold(ph, hcount, m);
            since_fold = 0;
        }
    }
    if (bad) st->range_err = 1;
    __syncthreads();
    if (PRIV) {
        // bins of the per-thread counters, summed over the block: warp w takes words w, w + 8, ...
        const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
        for (int w = wid; w < (m + 1) >> 1; w += kQThreads / 32) {
            uint32_t lo = 0, hi = 0;
            for (int c = lane; c < kQThreads; c += 32) {
                const uint32_t v = ph[w * kQThreads + c];
                lo += v & 0xffffu;
                hi += v >> 16;
            }
            for (int o = 16; o; o >>= 1) {
                lo += __shfl_xor_sync(0xffffffffu, lo, o);
                hi += __shfl_xor_sync(0xffffffffu, hi, o);
            }
            if (lane == 0) {
                hcount[2 * w] += lo;  // only warp wid writes these two bins after the barrier
                if (2 * w + 1 < m) hcount[2 * w + 1] += hi;
            }
        }
        __syncthreads();
    }
    for (int r = threadIdx.x; r < m; r += blockDim.x)
        if (hcount[r]) atomicAdd(&counts[r], hcount[r]);
}

// ------------------------------------------------ short codebooks (m <= 16)
// The same decisions as k_quantize with fewer instructions per entry:
//  * the search takes STEPS = ceil(log2 m) unrolled steps (a template argument), and the
//    range test compares with q[0] and q[m-1] held in registers;
//  * the draw computes only bits 32..63 of SplitMix64's second product, the bits the
//    rule reads (k = bits 40..63 of the output, and the final xor-shift by 31 leaves
//    bits 40..63 unchanged), with 32-bit limbs: each 64-bit multiply modulo 2^64 is a
//    wide 32 x 32 product plus two 32-bit multiply-adds, and the top word of the second
//    one a high product plus two;
//  * the index counts are per-thread 32-bit counters in shared memory (one column per
//    thread, no packing and no folding).
constexpr int kFastBins = 16;
constexpr uint32_t kC1lo = 0x1CE4E5B9u, kC1hi = 0xBF58476Du;  // SplitMix64 multipliers (Steele, Lea, Flood 2014)
constexpr uint32_t kC2lo = 0x133111EBu, kC2hi = 0x94D049BBu;

// Bits 32..63 of the SplitMix64 output for state z = (zh:zl).
__device__ __forceinline__ uint32_t splitmix64_hi(uint32_t zl, uint32_t zh) {
    const uint32_t xl = zl ^ __funnelshift_r(zl, zh, 30), xh = zh ^ (zh >> 30);  // z ^ (z >> 30)
    const uint64_t w = (uint64_t)xl * kC1lo;                                       // (xh:xl) * C1 mod 2^64
    const uint32_t al = (uint32_t)w;
    const uint32_t ah = (uint32_t)(w >> 32) + xl * kC1hi + xh * kC1lo;
    const uint32_t yl = al ^ __funnelshift_r(al, ah, 27), yh = ah ^ (ah >> 27);   // a ^ (a >> 27)
    return __umulhi(yl, kC2lo) + yl * kC2hi + yh * kC2lo;                         // top word of y * C2
}

template <int STEPS>
__device__ __forceinline__ int quant_fast(float xv, uint32_t zl, uint32_t zh, const float *q, float q0, float qm,
                                          bool &bad) {
    const bool in = xv >= q0 && xv <= qm;  // outside the codebook's range: index 0 and the error flag
    bad |= !in;
    int t = 0;
#pragma unroll
    for (int s = STEPS - 1; s >= 0; s--)
        if (q[t + (1 << s)] <= xv) t += 1 << s;
    const float a = q[t];
    const float k = __fmul_rn((float)(splitmix64_hi(zl, zh) >> 8), 0x1p-24f);
    const bool up = a != xv && __fmul_rn(k, __fsub_rn(q[t + 1], a)) < __fsub_rn(xv, a);
    return in ? t + (up ? 1 : 0) : 0;
}

// 64-bit counter state (zh:zl) advanced by gamma.
__device__ __forceinline__ void add_gamma(uint32_t &zl, uint32_t &zh) {
    const uint64_t z = (((uint64_t)zh << 32) | zl) + kGamma;
    zl = (uint32_t)z;
    zh = (uint32_t)(z >> 32);
}

template <int STEPS>
__global__ void __launch_bounds__(kQThreads) k_quantize_short(const float *__restrict__ x, int64_t d,
                                                              const float *__restrict__ Q, int m, uint64_t seed,
                                                              uint8_t *__restrict__ idx,
                                                              uint32_t *__restrict__ counts, DevStatus *st) {
    __shared__ float q[2 * kFastBins + 1];
    __shared__ uint32_t ph[kFastBins * kQThreads];  // ph[t * kQThreads + thread]
    for (int r = threadIdx.x; r < 2 * kFastBins + 1; r += blockDim.x) q[r] = r < m ? Q[r] : CUDART_INF_F;
#pragma unroll
    for (int t = 0; t < kFastBins; t++) ph[t * kQThreads + threadIdx.x] = 0u;
    __syncthreads();
    const float q0 = q[0], qm = q[m - 1];
    uint32_t *myc = ph + threadIdx.x;
    bool bad = false;
    const bool vec = ((reinterpret_cast<uintptr_t>(x) & 15) == 0) && ((reinterpret_cast<uintptr_t>(idx) & 3) == 0);
    const int64_t ngroups = vec ? d / 4 : 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t g0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const float4 *x4 = reinterpret_cast<const float4 *>(x);
    uchar4 *i4 = reinterpret_cast<uchar4 *>(idx);
    for (int64_t g = g0; g < ngroups; g += 2 * stride) {
        const int64_t h = g + stride;
        const bool two = h < ngroups;
        const float4 xa = x4[g];
        const float4 xb = two ? x4[h] : make_float4(q0, q0, q0, q0);
        const float xs[8] = {xa.x, xa.y, xa.z, xa.w, xb.x, xb.y, xb.z, xb.w};
        int ts[8];
        uint64_t za = seed + (uint64_t)(4 * g + 1) * kGamma;  // entry 4g: seed + (4g + 1) gamma
        uint64_t zb = seed + (uint64_t)(4 * h + 1) * kGamma;
        uint32_t al = (uint32_t)za, ah = (uint32_t)(za >> 32), bl = (uint32_t)zb, bh = (uint32_t)(zb >> 32);
#pragma unroll
        for (int r = 0; r < 4; r++) {
            ts[r] = quant_fast<STEPS>(xs[r], al, ah, q, q0, qm, bad);
            ts[4 + r] = quant_fast<STEPS>(xs[4 + r], bl, bh, q, q0, qm, bad);
            add_gamma(al, ah);
            add_gamma(bl, bh);
        }
        i4[g] = make_uchar4((uint8_t)ts[0], (uint8_t)ts[1], (uint8_t)ts[2], (uint8_t)ts[3]);
#pragma unroll
        for (int r = 0; r < 4; r++) myc[ts[r] * kQThreads] += 1u;
        if (two) {
            i4[h] = make_uchar4((uint8_t)ts[4], (uint8_t)ts[5], (uint8_t)ts[6], (uint8_t)ts[7]);
#pragma unroll
            for (int r = 4; r < 8; r++) myc[ts[r] * kQThreads] += 1u;
        }
    }
    for (int64_t i = 4 * ngroups + g0; i < d; i += stride) {
        const uint64_t z = seed + (uint64_t)(i + 1) * kGamma;
        const int t = quant_fast<STEPS>(x[i], (uint32_t)z, (uint32_t)(z >> 32), q, q0, qm, bad);
        idx[i] = (uint8_t)t;
        myc[t * kQThreads] += 1u;
    }
    if (bad) st->range_err = 1;
    __syncthreads();
    // bin t summed over the block's threads: warp w takes bins w, w + 8
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    for (int t = wid; t < m; t += kQThreads / 32) {
        uint32_t c = 0;
        for (int u = lane; u < kQThreads; u += 32) c += ph[t * kQThreads + u];
        for (int o = 16; o; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
        if (lane == 0 && c) atomicAdd(&counts[t], c);
    }
}

int launch_quantize(const float *x, int64_t d, const float *Q, int m, uint64_t seed, uint8_t *idx, uint32_t *counts,
                    DevStatus *st, int num_sms, cudaStream_t stream) {
    const int64_t groups = cdiv(d, 4);
    int64_t blocks = std::min<int64_t>(cdiv(groups, 2 * kQThreads), (int64_t)num_sms * 8);
    if (blocks < 1) blocks = 1;
    note_launch();
    if (m <= kFastBins) {
        // STEPS = ceil(log2 m): the search visits q[t + 2^s] for s < STEPS
        const int steps = m > 1 ? 32 - __builtin_clz((unsigned)(m - 1)) : 0;
        switch (steps) {
            case 0: k_quantize_short<0><<<(unsigned)blocks, kQThreads, 0, stream>>>(x, d, Q, m, seed, idx, counts, st); break;
            case 1: k_quantize_short<1><<<(unsigned)blocks, kQThreads, 0, stream>>>(x, d, Q, m, seed, idx, counts, st); break;
            case 2: k_quantize_short<2><<<(unsigned)blocks, kQThreads, 0, stream>>>(x, d, Q, m, seed, idx, counts, st); break;
            case 3: k_quantize_short<3><<<(unsigned)blocks, kQThreads, 0, stream>>>(x, d, Q, m, seed, idx, counts, st); break;
            default: k_quantize_short<4><<<(unsigned)blocks, kQThreads, 0, stream>>>(x, d, Q, m, seed, idx, counts, st); break;
        }
    } else if (m <= kPrivBins)
        k_quantize<true><<<(unsigned)blocks, kQThreads, 0, stream>>>(x, d, Q, m, seed, idx, counts, st);
    else
        k_quantize<false><<<(unsigned)blocks, kQThreads, 0, stream>>>(x, d, Q, m, seed, idx, counts, st);
    ECASQ_LAUNCH_CHECK();
    return ECASQ_OK;
}

// Two-way time-sharing (Sec. 7): entry i uses Q+ iff k_s * 2^-24 < beta (binary64,
// exact), k_s = top 24 bits of SplitMix64(seed_ts + (i+1) * 0x9E3779B97F4A7C15),
// then rounds within its codebook exactly as k_quantize (seed, same counter i).
// counts: [mm] for Q-, then [mp] for Q+; sel (may be null): 1 where Q+ was used.
__global__ void __launch_bounds__(256) k_quantize_timeshare(const float *__restrict__ x, int64_t d,
                                                            const float *__restrict__ Qm, int mm,
                                                            const float *__restrict__ Qp, int mp, double beta,
                                                            uint64_t seed, uint64_t seed_ts, uint8_t *__restrict__ idx,
                                                            uint8_t *__restrict__ sel, uint32_t *__restrict__ counts,
                                                            DevStatus *st) {
    __shared__ float q[2][kMaxS];
    __shared__ uint32_t hcount[2 * kMaxS];
    for (int r = threadIdx.x; r < kMaxS; r += blockDim.x) {
        q[0][r] = r < mm ? Qm[r] : CUDART_INF_F;
        q[1][r] = r < mp ? Qp[r] : CUDART_INF_F;
        hcount[r] = 0;
        hcount[kMaxS + r] = 0;
    }
    __syncthreads();
    bool bad = false;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < d; i += stride) {
        uint64_t zs = splitmix64(seed_ts + (uint64_t)(i + 1) * kGamma);
        int part = __dmul_rn((double)(uint32_t)(zs >> 40), 0x1p-24) < beta ? 1 : 0;
        const int mq = part ? mp : mm;
        int t = quant_one(x[i], seed + (uint64_t)(i + 1) * kGamma, q[part], mq, search_half(mq), bad);
        idx[i] = (uint8_t)t;
        if (sel) sel[i] = (uint8_t)part;
        atomicAdd(&hcount[part * kMaxS + t], 1u);
    }
    if (bad) st->range_err = 1;
    __syncthreads();
    for (int r = threadIdx.x; r < mm; r += blockDim.x)
        if (hcount[r]) atomicAdd(&counts[r], hcount[r]);
    for (int r = threadIdx.x; r < mp; r += blockDim.x)
        if (hcount[kMaxS + r]) atomicAdd(&counts[mm + r], hcount[kMaxS + r]);
}

int launch_quantize_timeshare(const float *x, int64_t d, const float *Qm, int mm, const float *Qp, int mp,
                              double beta, uint64_t seed, uint64_t seed_ts, uint8_t *idx, uint8_t *sel,
                              uint32_t *counts, DevStatus *st, int num_sms, cudaStream_t stream) {
    int64_t blocks = std::min<int64_t>(cdiv(d, 256), (int64_t)num_sms * 8);
    if (blocks < 1) blocks = 1;
    note_launch();
    k_quantize_timeshare<<<(unsigned)blocks, 256, 0, stream>>>(x, d, Qm, mm, Qp, mp, beta, seed, seed_ts, idx, sel,
                                                               counts, st);
    ECASQ_LAUNCH_CHECK();
    return ECASQ_OK;
}

}  // namespace ecasq
