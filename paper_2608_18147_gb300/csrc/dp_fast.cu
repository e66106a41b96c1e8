// dp_fast.cu -- fast approximate-DP kernel (Sec. 5).  Placeholder that routes
// to the fp64 reference kernel until the fp32-filter kernel lands.
#include "common.cuh"

namespace ecasq {

int launch_dp_reference(const Prefix &P, const double *lamp, int G, int s, double *dp64, int32_t *bp,
                        cudaStream_t st);

size_t fast_dp_band_bytes(int64_t d, int32_t s) {
    (void)d; (void)s;
    return 256;
}

int launch_dp_fast(const Prefix &P, const double *lamp, int G, int s, void *ws, const Layout &L, cudaStream_t st) {
    return launch_dp_reference(P, lamp, G, s, wsp<double>(ws, L.dp64), wsp<int32_t>(ws, L.bp), st);
}

}  // namespace ecasq
