// Host-side declarations shared between the translation units of libgefen.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "gefen.h"

namespace gefen {

constexpr size_t kWsAlign = 256;
inline size_t align_up(size_t x, size_t a = kWsAlign) { return (x + a - 1) / a * a; }

// One contiguous run of fp32 values to histogram.
struct HistRange {
    int64_t offset;
    int64_t count;
};

// Adds the cell counts of every non-NaN value of the listed runs of `x`
// to hist[bins] (u64, device).  Enqueued on `stream`; returns a CUDA status.
cudaError_t launch_histogram(const float* x, const HistRange* ranges, int nranges,
                             int bins, uint64_t* hist, cudaStream_t stream);

// Loads the histogram kernels on the current device (so that a later launch
// needs nothing more from the driver).
cudaError_t prepare_histogram();

// Multiprocessor count of the current device (cached per device).
int device_sm_count();

// GEFEN_EUNSUPPORTED unless the current device is compute capability 10.3.
gefen_status_t check_device();

}  // namespace gefen
