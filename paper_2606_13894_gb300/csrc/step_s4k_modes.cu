// Instances of the streamed step kernel (step_kernels.cuh): 4096-element
// tiles of refit steps (x counted in shared-memory cells, or staged for the
// histogram kernel) and of first-gradient histogram steps.  Staged x (more
// cells than shared memory holds) is served by one instance for all shapes.
#include "step_kernels.cuh"

namespace gefen {
namespace stepk {

cudaError_t stream_s4k_modes(int mode, int hb, int fmt, int shape, const Launch& L, const Ptrs& P, int* err,
                             cudaStream_t st) {
    if (mode == kHist) {
        if (hb) return stream_by_fmt_shape<S4KHistCfg, kHist, kFusedBins, false, true>(fmt, shape, L, P, err, st);
        if (fmt != 0) return cudaErrorNotSupported;
        return stream_kernel<S4KCfg, kHist, 0, 0, false, kShapeAny>(L, P, err, st);
    }
    if (mode == kGradOnly) {
        if (fmt != 0) return cudaErrorInvalidValue;
        if (hb) return stream_by_shape<S4KHistCfg, kGradOnly, kFusedBins, false, 0, true>(shape, L, P, err, st);
        return stream_kernel<S4KCfg, kGradOnly, 0, 0, false, kShapeAny>(L, P, err, st);
    }
    return cudaErrorInvalidValue;
}

}  // namespace stepk
}  // namespace gefen
