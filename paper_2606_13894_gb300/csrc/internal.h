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

// C = alpha * A * B^T + beta * D (row-major; A: M x K, B: N x K, C, D: M x N),
// written as C and/or as its transpose CT (N x M); bf16 storage with fp32
// accumulation (tcgen05 when TMA can address A and B), or fp32 throughout.
// D, C, CT nullable.  err: device word set when a bounded wait gave up.
// sym: the result is symmetric (M == N, C given, CT not): on the tensor cores
// only the tiles on or above the diagonal are computed and mirrored.
cudaError_t gemm_bf16_nt(int M, int N, int K, float alpha, const void* A, int lda, const void* B, int ldb,
                         float beta, const void* D, int ldd, void* C, int ldc, void* CT, int ldct, int* err,
                         cudaStream_t st, bool sym = false);
cudaError_t gemm_f32_nt(int M, int N, int K, float alpha, const float* A, int lda, const float* B, int ldb,
                        float beta, const float* D, int ldd, float* C, int ldc, float* CT, int ldct,
                        cudaStream_t st);
// Whether the bf16 product takes the tcgen05 path for these operands.
bool gemm_tc_usable(int lda, int ldb, const void* A, const void* B);

// Multiprocessor count of the current device (cached per device).
int device_sm_count();

// GEFEN_EUNSUPPORTED unless the current device is compute capability 10.3.
gefen_status_t check_device();

}  // namespace gefen
