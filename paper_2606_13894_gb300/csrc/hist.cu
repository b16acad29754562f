// Histogram of normalised values over [-1, 1] (Algorithm 3, "accumulate all
// entries of Z into histogram counts").
//
// HBM-bound: 4 bytes read per value.  Counts are privatised in shared memory
// (u32) and flushed to the u64 result once per CTA.  Up to 16384 cells fit in
// one CTA; for up to 65536 cells a cluster of two CTAs splits the cells, each
// CTA owning half in its shared memory.  Both CTAs of the pair read every value
// of their unit (the second read is an L2 hit: the pair runs together) and each
// counts only the values of its own cells, so no count crosses between CTAs.
// NaN values are skipped.
#include <cooperative_groups.h>

#include <algorithm>
#include <vector>

#include "common.cuh"
#include "internal.h"

namespace cg = cooperative_groups;

namespace gefen {

namespace {

constexpr int kHistThreads = 1024;
constexpr int kHistMaxRanges = 512;
constexpr int64_t kHistUnit = 16384;  // values per work unit
constexpr int kHistLoads = 4;         // float4 loads in flight per thread

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
__device__ __forceinline__ void count_one(float x, float halfB, int B, int per, unsigned* local, unsigned rank) {
    if (isnan(x)) return;
    const int c = hist_cell(x, halfB, B);
    if (CL == 1) {
        atomicAdd(local + c, 1u);
    } else {
        const int li = c - static_cast<int>(rank) * per;  // this CTA's cells: [rank per, (rank+1) per)
        if (static_cast<unsigned>(li) < static_cast<unsigned>(per)) atomicAdd(local + li, 1u);
    }
}

template <int CL>
__device__ __forceinline__ void hist_body(const float* __restrict__ x, const HistLaunch& L,
                                          uint64_t* __restrict__ hist, unsigned* s_hist, unsigned rank) {
    const int B = L.bins;
    const int per = (B + CL - 1) / CL;  // cells owned by each CTA of the cluster
    const float halfB = 0.5f * static_cast<float>(B);
    const int64_t nclusters = gridDim.x / CL;
    const int64_t cid = blockIdx.x / CL;
    // every CTA of a cluster reads the whole unit
    for (int64_t u = cid; u < L.nunits; u += nclusters) {
        const int r = find_range(L, u);
        const int64_t s0 = L.off[r] + (u - L.unit_begin[r]) * kHistUnit;
        const int64_t s1 = min(s0 + kHistUnit, L.off[r] + L.cnt[r]);
        if (s0 >= s1) continue;
        // 16-byte aligned body with float4 loads; scalar head/tail.
        int64_t h = (s0 + 3) & ~int64_t(3);
        if (h > s1) h = s1;
        for (int64_t e = s0 + threadIdx.x; e < h; e += blockDim.x)
            count_one<CL>(__ldcg(x + e), halfB, B, per, s_hist, rank);
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
                count_one<CL>(q[u].x, halfB, B, per, s_hist, rank);
                count_one<CL>(q[u].y, halfB, B, per, s_hist, rank);
                count_one<CL>(q[u].z, halfB, B, per, s_hist, rank);
                count_one<CL>(q[u].w, halfB, B, per, s_hist, rank);
            }
        }
        for (int64_t e = h + nv * 4 + threadIdx.x; e < s1; e += blockDim.x)
            count_one<CL>(__ldcg(x + e), halfB, B, per, s_hist, rank);
    }
}

__global__ void __launch_bounds__(kHistThreads) k_hist1(const float* __restrict__ x, const __grid_constant__ HistLaunch L,
                                                       uint64_t* __restrict__ hist) {
    extern __shared__ unsigned s_hist[];
    const int B = L.bins;
    for (int i = threadIdx.x; i < B; i += blockDim.x) s_hist[i] = 0u;
    __syncthreads();
    hist_body<1>(x, L, hist, s_hist, 0u);
    __syncthreads();
    for (int i = threadIdx.x; i < B; i += blockDim.x) {
        const unsigned c = s_hist[i];
        if (c) atomicAdd(reinterpret_cast<unsigned long long*>(hist + i), static_cast<unsigned long long>(c));
    }
}

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kHistThreads)
    k_hist2(const float* __restrict__ x, const __grid_constant__ HistLaunch L, uint64_t* __restrict__ hist) {
    extern __shared__ unsigned s_hist[];
    cg::cluster_group cluster = cg::this_cluster();
    const unsigned rank = cluster.block_rank();
    const int B = L.bins;
    const int per = (B + 1) / 2;
    for (int i = threadIdx.x; i < per; i += blockDim.x) s_hist[i] = 0u;
    __syncthreads();
    hist_body<2>(x, L, hist, s_hist, rank);
    __syncthreads();
    const int base = static_cast<int>(rank) * per;
    for (int i = threadIdx.x; i < per && base + i < B; i += blockDim.x) {
        const unsigned c = s_hist[i];
        if (c) atomicAdd(reinterpret_cast<unsigned long long*>(hist + base + i), static_cast<unsigned long long>(c));
    }
}

}  // namespace

cudaError_t launch_histogram(const float* x, const HistRange* ranges, int nranges, int bins, uint64_t* hist,
                             cudaStream_t stream) {
    // One launch sees at most 2^36 values, so a CTA's u32 counters (it handles
    // a 1/(number of clusters) share) stay far below 2^32.
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
            e = cudaFuncSetAttribute(k_hist2, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
            if (e != cudaSuccess) return e;
            // all clusters co-resident (units are dealt out statically): the
            // number of SM pairs the hardware can place, not sms / 2
            // (a property of the kernel and its shared memory: asked once per size)
            static thread_local size_t fit_smem = 0;
            static thread_local int fit = 0;
            if (fit_smem != smem) {
                cudaLaunchConfig_t cfg = {};
                cfg.gridDim = dim3(2 * static_cast<unsigned>(std::max(1, sms / 2)));
                cfg.blockDim = dim3(kHistThreads);
                cfg.dynamicSmemBytes = smem;
                if (cudaOccupancyMaxActiveClusters(&fit, k_hist2, &cfg) != cudaSuccess || fit < 1) {
                    (void)cudaGetLastError();
                    fit = std::max(1, sms / 2);
                }
                fit_smem = smem;
            }
            const int64_t clusters = std::min<int64_t>(units, fit);
            k_hist2<<<dim3(static_cast<unsigned>(2 * clusters)), kHistThreads, smem, stream>>>(x, L, hist);
        }
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace gefen
