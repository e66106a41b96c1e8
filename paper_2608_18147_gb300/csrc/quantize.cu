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

__device__ __forceinline__ int quant_one(float xv, int64_t i, const float *q, int m, uint64_t seed, bool &bad) {
    if (!(xv >= q[0] && xv <= q[m - 1])) { bad = true; return 0; }
    int lo = 0, hi = m - 1;  // largest t with q[t] <= x
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (q[mid] <= xv) lo = mid; else hi = mid - 1;
    }
    int t = lo;
    if (q[t] != xv) {
        uint64_t z = splitmix64(seed + (uint64_t)(i + 1) * 0x9E3779B97F4A7C15ull);
        float k = __fmul_rn((float)(uint32_t)(z >> 40), 0x1p-24f);
        float d1 = __fsub_rn(xv, q[t]);
        float d2 = __fsub_rn(q[t + 1], q[t]);
        if (__fmul_rn(k, d2) < d1) t += 1;
    }
    return t;
}

__global__ void __launch_bounds__(256) k_quantize(const float *__restrict__ x, int64_t d, const float *__restrict__ Q,
                                                  int m, uint64_t seed, uint8_t *__restrict__ idx,
                                                  uint32_t *__restrict__ counts, DevStatus *st) {
    __shared__ float q[kMaxS];
    __shared__ uint32_t hcount[kMaxS];
    for (int r = threadIdx.x; r < kMaxS; r += blockDim.x) {
        q[r] = r < m ? Q[r] : 0.0f;
        hcount[r] = 0;
    }
    __syncthreads();
    bool bad = false;
    bool vec = ((reinterpret_cast<uintptr_t>(x) & 15) == 0) && ((reinterpret_cast<uintptr_t>(idx) & 3) == 0);
    int64_t ngroups = d / 4;
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    int64_t g0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (vec) {
        for (int64_t g = g0; g < ngroups; g += stride) {
            float4 xv = reinterpret_cast<const float4 *>(x)[g];
            int64_t i = 4 * g;
            int t0 = quant_one(xv.x, i, q, m, seed, bad);
            int t1 = quant_one(xv.y, i + 1, q, m, seed, bad);
            int t2 = quant_one(xv.z, i + 2, q, m, seed, bad);
            int t3 = quant_one(xv.w, i + 3, q, m, seed, bad);
            reinterpret_cast<uchar4 *>(idx)[g] = make_uchar4((uint8_t)t0, (uint8_t)t1, (uint8_t)t2, (uint8_t)t3);
            atomicAdd(&hcount[t0], 1u); atomicAdd(&hcount[t1], 1u);
            atomicAdd(&hcount[t2], 1u); atomicAdd(&hcount[t3], 1u);
        }
    }
    int64_t start = vec ? 4 * ngroups : 0;
    for (int64_t i = start + g0; i < d; i += stride) {
        int t = quant_one(x[i], i, q, m, seed, bad);
        idx[i] = (uint8_t)t;
        atomicAdd(&hcount[t], 1u);
    }
    if (bad) st->range_err = 1;
    __syncthreads();
    for (int r = threadIdx.x; r < m; r += blockDim.x)
        if (hcount[r]) atomicAdd(&counts[r], hcount[r]);
}

int launch_quantize(const float *x, int64_t d, const float *Q, int m, uint64_t seed, uint8_t *idx, uint32_t *counts,
                    DevStatus *st, int num_sms, cudaStream_t stream) {
    int64_t groups = cdiv(d, 4);
    int64_t blocks = std::min<int64_t>(cdiv(groups, 256), (int64_t)num_sms * 8);
    if (blocks < 1) blocks = 1;
    note_launch();
    k_quantize<<<(unsigned)blocks, 256, 0, stream>>>(x, d, Q, m, seed, idx, counts, st);
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
        q[0][r] = r < mm ? Qm[r] : 0.0f;
        q[1][r] = r < mp ? Qp[r] : 0.0f;
        hcount[r] = 0;
        hcount[kMaxS + r] = 0;
    }
    __syncthreads();
    bool bad = false;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < d; i += stride) {
        uint64_t zs = splitmix64(seed_ts + (uint64_t)(i + 1) * 0x9E3779B97F4A7C15ull);
        int part = __dmul_rn((double)(uint32_t)(zs >> 40), 0x1p-24) < beta ? 1 : 0;
        int t = quant_one(x[i], i, q[part], part ? mp : mm, seed, bad);
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
