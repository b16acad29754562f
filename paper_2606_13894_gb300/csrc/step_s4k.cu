// Instances of the streamed step kernel (step_kernels.cuh): 4096-element
// tiles of plain steps, every storage format and block shape.
#include "step_kernels.cuh"

namespace gefen {
namespace stepk {

cudaError_t stream_s4k_plain(int fmt, int shape, const Launch& L, const Ptrs& P, int* err, cudaStream_t st) {
    return stream_by_fmt_shape<S4KCfg, kPlain, 0, false, true>(fmt, shape, L, P, err, st);
}

}  // namespace stepk
}  // namespace gefen
