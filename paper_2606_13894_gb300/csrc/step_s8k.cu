// Instances of the streamed step kernel (step_kernels.cuh): 8192-element
// tiles (blocks of 4096 < p <= 8192, so no block of 16 to 256 elements), for
// every step mode.
#include "step_kernels.cuh"

namespace gefen {
namespace stepk {

cudaError_t stream_s8k(int mode, int hb, int fmt, int shape, const Launch& L, const Ptrs& P, int* err,
                       cudaStream_t st) {
    if (mode == kPlain) return stream_by_fmt_shape<S8KCfg, kPlain, 0, false, false>(fmt, shape, L, P, err, st);
    if (mode == kHist) {
        if (hb) return stream_by_fmt_shape<S8KHistCfg, kHist, kFusedBins, false, false>(fmt, shape, L, P, err, st);
        if (fmt != 0) return cudaErrorNotSupported;
        return stream_kernel<S8KCfg, kHist, 0, 0, false, kShapeAny>(L, P, err, st);
    }
    if (mode == kGradOnly) {
        if (fmt != 0) return cudaErrorInvalidValue;
        if (hb) return stream_by_shape<S8KHistCfg, kGradOnly, kFusedBins, false, 0, false>(shape, L, P, err, st);
        return stream_kernel<S8KCfg, kGradOnly, 0, 0, false, kShapeAny>(L, P, err, st);
    }
    return cudaErrorInvalidValue;
}

}  // namespace stepk
}  // namespace gefen
