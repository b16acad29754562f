// Histogram of normalised values over [-1, 1] (Algorithm 3, "accumulate all
// entries of Z into histogram counts").
//
// HBM-bound: 4 bytes read per value.  Counts are privatised in shared memory
// and flushed to the u64 result once per CTA.  Up to 16384 cells: u32
// counters.  Up to 65536 cells: two 16-bit counters per u32 word (128 KB for
// 65536 cells, one CTA per SM), kept below 2^16 by construction: after every
// kPackedUnits units (at most 49152 values) the CTA moves each counter that
// has reached 2^14 to the u64 result, so between checks none can pass
// 2^14 - 1 + 49152 = 65535.  NaN values are skipped.
#include <algorithm>
#include <vector>

#include "common.cuh"
#include "internal.h"

namespace gefen {

namespace {

constexpr int kHistThreads = 1024;
constexpr int kHistMaxRanges = 512;
constexpr int64_t kHistUnit = 16384;  // values per work unit
constexpr int kHistLoads = 4;         // float4 loads in flight per thread
constexpr int kPacked = 16;           // hist_body mode: two 16-bit counters per word
constexpr int kPackedUnits = 3;       // units between checks of the 16-bit counters
constexpr unsigned kSpillAt = 1u << 14;

struct HistLaunch {
    int32_t nranges;
    int32_t bins;
    int64_t nunits;
    int64_t off[kHistMaxRanges];
    int64_t cnt[kHistMaxRanges];
    int64_t unit_begin[kHistMaxRanges];
};

__device__ __forceinline__ int find_range(const HistLaunch& L, int64_t unit) {
    int lo = 0, hi = L.nranges - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (L.unit_begin[mid] <= unit) lo = mid; else hi = mid - 1;
    }
    return lo;
}

template <int CL>
__device__ __forceinline__ void count_one(float x, float halfB, int B, unsigned* local) {
    if (isnan(x)) return;
    const int c = hist_cell(x, halfB, B);
    if (CL == kPacked)
        atomicAdd(local + (c >> 1), 1u << ((c & 1) << 4));  // cell c: half c & 1 of word c / 2
    else
        atomicAdd(local + c, 1u);
}

// Moves every 16-bit counter that has reached kSpillAt to the u64 result
// (between two CTA barriers: no count is in flight).
__device__ __forceinline__ void spill_packed(unsigned* words, int B, uint64_t* __restrict__ hist) {
    const int nw = (B + 1) >> 1;
    for (int i = threadIdx.x; i < nw; i += blockDim.x) {
        const unsigned w = words[i];
        const unsigned lo = w & 0xFFFFu, hi = w >> 16;
        if (lo < kSpillAt && hi < kSpillAt) continue;
        unsigned keep = w;
        if (lo >= kSpillAt) {
            atomicAdd(reinterpret_cast<unsigned long long*>(hist + 2 * i), static_cast<unsigned long long>(lo));
            keep &= 0xFFFF0000u;
        }
        if (hi >= kSpillAt) {
            atomicAdd(reinterpret_cast<unsigned long long*>(hist + 2 * i + 1), static_cast<unsigned long long>(hi));
            keep &= 0x0000FFFFu;
        }
        words[i] = keep;
    }
}

template <int CL>
__device__ __forceinline__ void hist_body(const float* __restrict__ x, const HistLaunch& L,
                                          uint64_t* __restrict__ hist, unsigned* s_hist) {
    const int B = L.bins;
    const float halfB = 0.5f * static_cast<float>(B);
    int since = 0;  // units since the last check of the 16-bit counters (uniform)
    for (int64_t u = blockIdx.x; u < L.nunits; u += gridDim.x) {
        const int r = find_range(L, u);
        const int64_t s0 = L.off[r] + (u - L.unit_begin[r]) * kHistUnit;
        const int64_t s1 = min(s0 + kHistUnit, L.off[r] + L.cnt[r]);
        if (s0 >= s1) continue;
        // 16-byte aligned body with float4 loads; scalar head/tail.
        int64_t h = (s0 + 3) & ~int64_t(3);
        if (h > s1) h = s1;
        for (int64_t e = s0 + threadIdx.x; e < h; e += blockDim.x)
            count_one<CL>(__ldcg(x + e), halfB, B, s_hist);
        const int64_t nv = (s1 - h) >> 2;
        const float4* xv = reinterpret_cast<const float4*>(x + h);
        // kHistLoads float4 loads in flight per thread before any count (a
        // missing load reads as NaN, which is not counted)
        for (int64_t j0 = threadIdx.x; j0 < nv; j0 += kHistLoads * blockDim.x) {
            float4 q[kHistLoads];
#pragma unroll
            for (int u = 0; u < kHistLoads; ++u) {
                const int64_t j = j0 + static_cast<int64_t>(u) * blockDim.x;
                q[u] = j < nv ? __ldcg(xv + j) : make_float4(NAN, NAN, NAN, NAN);
            }
#pragma unroll
            for (int u = 0; u < kHistLoads; ++u) {
                count_one<CL>(q[u].x, halfB, B, s_hist);
                count_one<CL>(q[u].y, halfB, B, s_hist);
                count_one<CL>(q[u].z, halfB, B, s_hist);
                count_one<CL>(q[u].w, halfB, B, s_hist);
            }
        }
        for (int64_t e = h + nv * 4 + threadIdx.x; e < s1; e += blockDim.x)
            count_one<CL>(__ldcg(x + e), halfB, B, s_hist);
        if (CL == kPacked && ++since == kPackedUnits) {
            since = 0;
            __syncthreads();
            spill_packed(s_hist, B, hist);
            __syncthreads();
        }
    }
}

__global__ void __launch_bounds__(kHistThreads) k_hist1(const float* __restrict__ x, const __grid_constant__ HistLaunch L,
                                                       uint64_t* __restrict__ hist) {
    extern __shared__ unsigned s_hist[];
    const int B = L.bins;
    for (int i = threadIdx.x; i < B; i += blockDim.x) s_hist[i] = 0u;
    __syncthreads();
    hist_body<1>(x, L, hist, s_hist);
    __syncthreads();
    for (int i = threadIdx.x; i < B; i += blockDim.x) {
        const unsigned c = s_hist[i];
        if (c) atomicAdd(reinterpret_cast<unsigned long long*>(hist + i), static_cast<unsigned long long>(c));
    }
}

__global__ void __launch_bounds__(kHistThreads) k_hist16(const float* __restrict__ x,
                                                        const __grid_constant__ HistLaunch L,
                                                        uint64_t* __restrict__ hist) {
    extern __shared__ unsigned s_words[];  // cell c: half c & 1 of word c / 2
    const int B = L.bins;
    const int nw = (B + 1) >> 1;
    for (int i = threadIdx.x; i < nw; i += blockDim.x) s_words[i] = 0u;
    __syncthreads();
    hist_body<kPacked>(x, L, hist, s_words);
    __syncthreads();
    for (int i = threadIdx.x; i < nw; i += blockDim.x) {
        const unsigned w = s_words[i];
        const unsigned lo = w & 0xFFFFu, hi = w >> 16;
        if (lo) atomicAdd(reinterpret_cast<unsigned long long*>(hist + 2 * i), static_cast<unsigned long long>(lo));
        if (hi && 2 * i + 1 < B)
            atomicAdd(reinterpret_cast<unsigned long long*>(hist + 2 * i + 1), static_cast<unsigned long long>(hi));
    }
}

}  // namespace

cudaError_t prepare_histogram() {
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, k_hist1);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, k_hist16);
    return e;
}

cudaError_t launch_histogram(const float* x, const HistRange* ranges, int nranges, int bins, uint64_t* hist,
                             cudaStream_t stream) {
    // One launch sees at most 2^36 values, so a CTA's u32 counters (it handles
    // a 1/(number of CTAs) share) stay far below 2^32.
    constexpr int64_t kMaxPerLaunch = int64_t(1) << 36;
    static thread_local HistLaunch L;
    const int sms = device_sm_count();
    std::vector<HistRange> pieces;
    for (int i = 0; i < nranges; ++i)
        for (int64_t o = 0; o < ranges[i].count; o += kMaxPerLaunch)
            pieces.push_back({ranges[i].offset + o, std::min(kMaxPerLaunch, ranges[i].count - o)});
    size_t i = 0;
    while (i < pieces.size()) {
        L.nranges = 0;
        L.bins = bins;
        int64_t units = 0, vals = 0;
        for (; i < pieces.size() && L.nranges < kHistMaxRanges && vals + pieces[i].count <= kMaxPerLaunch; ++i) {
            const int64_t c = pieces[i].count;
            L.off[L.nranges] = pieces[i].offset;
            L.cnt[L.nranges] = c;
            L.unit_begin[L.nranges] = units;
            units += (c + kHistUnit - 1) / kHistUnit;
            vals += c;
            ++L.nranges;
        }
        L.nunits = units;
        if (units == 0) continue;
        cudaError_t e;
        if (bins <= 16384) {
            const size_t smem = static_cast<size_t>(bins) * sizeof(unsigned);
            e = cudaFuncSetAttribute(k_hist1, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
            if (e != cudaSuccess) return e;
            const int64_t grid = std::min<int64_t>(units, 2 * static_cast<int64_t>(sms));
            k_hist1<<<dim3(static_cast<unsigned>(grid)), kHistThreads, smem, stream>>>(x, L, hist);
        } else {
            const size_t smem = static_cast<size_t>((bins + 1) / 2) * sizeof(unsigned);
            e = cudaFuncSetAttribute(k_hist16, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
            if (e != cudaSuccess) return e;
            // resident CTAs per SM for this size (asked once per size)
            static thread_local size_t fit_smem = 0;
            static thread_local int per_sm = 1;
            if (fit_smem != smem) {
                if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_hist16, kHistThreads, smem) !=
                        cudaSuccess || per_sm < 1) {
                    (void)cudaGetLastError();
                    per_sm = 1;
                }
                fit_smem = smem;
            }
            const int64_t grid = std::min<int64_t>(units, static_cast<int64_t>(per_sm) * sms);
            k_hist16<<<dim3(static_cast<unsigned>(grid)), kHistThreads, smem, stream>>>(x, L, hist);
        }
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace gefen
