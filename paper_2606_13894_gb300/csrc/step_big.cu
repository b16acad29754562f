// Instances of the streamed step kernel (step_kernels.cuh) over the tiles of
// big blocks whose factors a finalisation kernel kept (4096-element tiles).
#include "step_kernels.cuh"

namespace gefen {
namespace stepk {

namespace {
template <typename C, int MODE, int HB>
cudaError_t big_by_fmt(int fmt, const Launch& L, const Ptrs& P, int* err, cudaStream_t st) {
    switch (fmt) {
        case 0: return stream_kernel<C, MODE, HB, 0, true, kShapeAny>(L, P, err, st);
        case 1: return stream_kernel<C, MODE, HB, 1, true, kShapeAny>(L, P, err, st);
        case 2: return stream_kernel<C, MODE, HB, 2, true, kShapeAny>(L, P, err, st);
        case 3: return stream_kernel<C, MODE, HB, 3, true, kShapeAny>(L, P, err, st);
        default: return cudaErrorInvalidValue;
    }
}
}  // namespace

cudaError_t stream_big(int mode, int hb, int fmt, const Launch& L, const Ptrs& P, int* err, cudaStream_t st) {
    if (mode == kPlain) return big_by_fmt<S4KCfg, kPlain, 0>(fmt, L, P, err, st);
    if (mode == kHist) {
        if (hb) return big_by_fmt<S4KHistCfg, kHist, kFusedBins>(fmt, L, P, err, st);
        if (fmt != 0) return cudaErrorNotSupported;
        return stream_kernel<S4KCfg, kHist, 0, 0, true, kShapeAny>(L, P, err, st);
    }
    if (mode == kGradOnly) {
        if (fmt != 0) return cudaErrorInvalidValue;
        if (hb) return stream_kernel<S4KHistCfg, kGradOnly, kFusedBins, 0, true, kShapeAny>(L, P, err, st);
        return stream_kernel<S4KCfg, kGradOnly, 0, 0, true, kShapeAny>(L, P, err, st);
    }
    return cudaErrorInvalidValue;
}

}  // namespace stepk
}  // namespace gefen
