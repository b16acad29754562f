// Histogram of normalised values over [-1, 1] (Algorithm 3, "accumulate all
// entries of Z into histogram counts").
//
// HBM-bound: 4 bytes read per value.  Counts are privatised in shared memory
// and flushed to the u64 result once per CTA.  Up to 16384 cells: u32
// counters, two CTAs per SM.  Up to 65536 cells, one CTA per SM: u32 counters
// for the (at most 57344) central cells, where normalised momentum piles up,
// and for the kEdge cells at each end (every block's largest |x| is 1 and
// lands there); the sparse shoulders between them are added straight to the
// u64 result.  That path computes a cell in seven instructions (a round-down
// add of 1.5 * 2^23 takes the floor), lets a warp whose 512 values of a round
// share one cell count them with a single atomic, and asks L2 for its next
// units ahead of the loads.  NaN values are skipped.
#include <algorithm>
#include <mutex>
#include <vector>

#include "common.cuh"
#include "internal.h"

namespace gefen {

namespace {

constexpr int kHistThreads = 1024;
constexpr int kHistMaxRanges = 512;
constexpr int64_t kHistUnit = 32768;  // values per work unit
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

__device__ __forceinline__ void count_one(float x, float halfB, int B, unsigned* local) {
    if (isnan(x)) return;
    atomicAdd(local + hist_cell(x, halfB, B), 1u);
}

__device__ __forceinline__ void hist_body(const float* __restrict__ x, const HistLaunch& L,
                                          uint64_t* __restrict__ hist, unsigned* s_hist) {
    const int B = L.bins;
    const float halfB = 0.5f * static_cast<float>(B);
    for (int64_t u = blockIdx.x; u < L.nunits; u += gridDim.x) {
        const int r = find_range(L, u);
        const int64_t s0 = L.off[r] + (u - L.unit_begin[r]) * kHistUnit;
        const int64_t s1 = min(s0 + kHistUnit, L.off[r] + L.cnt[r]);
        if (s0 >= s1) continue;
        // 16-byte aligned body with float4 loads; scalar head/tail.
        int64_t h = (s0 + 3) & ~int64_t(3);
        if (h > s1) h = s1;
        for (int64_t e = s0 + threadIdx.x; e < h; e += blockDim.x)
            count_one(__ldcg(x + e), halfB, B, s_hist);
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
                count_one(q[u].x, halfB, B, s_hist);
                count_one(q[u].y, halfB, B, s_hist);
                count_one(q[u].z, halfB, B, s_hist);
                count_one(q[u].w, halfB, B, s_hist);
            }
        }
        for (int64_t e = h + nv * 4 + threadIdx.x; e < s1; e += blockDim.x)
            count_one(__ldcg(x + e), halfB, B, s_hist);
    }
}

__global__ void __launch_bounds__(kHistThreads) k_hist1(const float* __restrict__ x, const __grid_constant__ HistLaunch L,
                                                       uint64_t* __restrict__ hist) {
    extern __shared__ unsigned s_hist[];
    const int B = L.bins;
    for (int i = threadIdx.x; i < B; i += blockDim.x) s_hist[i] = 0u;
    __syncthreads();
    hist_body(x, L, hist, s_hist);
    __syncthreads();
    for (int i = threadIdx.x; i < B; i += blockDim.x) {
        const unsigned c = s_hist[i];
        if (c) atomicAdd(reinterpret_cast<unsigned long long*>(hist + i), static_cast<unsigned long long>(c));
    }
}

// ------------------------------------------------- 65536-cell path
// Cells of the 65536-cell path as the bits of a float: the floor of the cell
// coordinate is taken by a round-down add of 1.5 * 2^23, so that the sum's
// bits minus kMagicBits are the cell (coordinates below 2^22 here).  With B a
// power of two the scaling by B/2 is exact, so RN(x + 1) * B/2 floored by one
// round-down fma is the cell definition's floor(RN(RN(x + 1) * B/2)), clamped
// in the integer domain; other B take the definition's two roundings, clamped
// in fp32.  NaN maps to nan_bits (the caller's marker of a skipped value).
constexpr float kMagic = 12582912.0f;  // 1.5 * 2^23
constexpr uint32_t kMagicBits = 0x4B400000u;

template <bool POW2>
__device__ __forceinline__ uint32_t cell_bits(float x, float halfB, float top, int top_bits, uint32_t nan_bits) {
    uint32_t c;
    if (POW2) {
        const float f = __fmaf_rd(__fadd_rn(x, 1.0f), halfB, kMagic);
        c = static_cast<uint32_t>(max(min(__float_as_int(f), top_bits), static_cast<int>(kMagicBits)));
    } else {
        const float u = __fmul_rn(__fadd_rn(x, 1.0f), halfB);
        c = __float_as_uint(__fadd_rd(fminf(fmaxf(u, 0.0f), top), kMagic));
    }
    return isnan(x) ? nan_bits : c;
}

// Counters of the 16384 < B <= 65536 path: u32 counters in shared memory for
// the ncen central cells [c_lo, c_lo + ncen) and the `edge` cells at each end
// ([0, edge) then [B - edge, B)); a cell between them is added to the u64
// result directly.  Normalised momentum piles up near 0, and each block's
// largest |x| is 1 (an end cell), so the cells left to global atomics hold
// the few values between.
struct Cells {
    unsigned* cen;
    unsigned* ext;
    uint32_t c_lo, ncen, edge, B;
};

constexpr uint32_t kMaxCentral = 57344;  // 224 KB of u32 counters
constexpr uint32_t kEdge = 32;

__host__ __device__ constexpr uint32_t central_cells(uint32_t B) { return B < kMaxCentral ? B : kMaxCentral; }
__host__ __device__ constexpr uint32_t edge_cells(uint32_t B) {
    return (B - central_cells(B)) / 2 < kEdge ? (B - central_cells(B)) / 2 : kEdge;
}

// Adds n counts to cell c (0xFFFFFFFF: a NaN value, skipped).
__device__ __forceinline__ void count_cell(const Cells& S, uint64_t* __restrict__ hist, uint32_t c, unsigned n) {
    const uint32_t d = c - S.c_lo;
    if (d < S.ncen) {
        atomicAdd(S.cen + d, n);
    } else if (c < S.B) {
        if (c < S.edge)
            atomicAdd(S.ext + c, n);
        else if (c >= S.B - S.edge)
            atomicAdd(S.ext + S.edge + (c - (S.B - S.edge)), n);
        else
            atomicAdd(reinterpret_cast<unsigned long long*>(hist + c), static_cast<unsigned long long>(n));
    }
}

// Asks L2 to fetch the 16-byte aligned body of unit u (no registers or
// shared memory held while it is in flight).
__device__ __forceinline__ void prefetch_unit_l2(const float* __restrict__ x, const HistLaunch& L, int64_t u) {
    const int r = find_range(L, u);
    const int64_t s0 = L.off[r] + (u - L.unit_begin[r]) * kHistUnit;
    const int64_t s1 = min(s0 + kHistUnit, L.off[r] + L.cnt[r]);
    const int64_t h = (s0 + 3) & ~int64_t(3);
    if (s1 - h < 4) return;
    const uint32_t bytes = static_cast<uint32_t>(((s1 - h) >> 2) * 16);
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(x + h), "r"(bytes) : "memory");
}

constexpr int kPrefetchUnits = 2;  // units of this CTA ahead of the one it counts

// 16384 < B <= 65536 cells (Cells: u32 counters for the central and end
// cells, 224 KB at 65536 cells, one CTA per SM).  Shared memory leaves room
// for no second CTA, so the loads in flight come from L2: thread 0 asks L2
// for this CTA's unit kPrefetchUnits ahead while the CTA counts, and each
// thread keeps four 16-byte loads in flight.  When all 512 values of a warp's
// round fall in one cell (or are all NaN) the warp adds them with one atomic,
// else every value is one atomic.
// n counts for a value whose cell, before any clamp, is raw (see the kernel):
// a central cell at once, the rest through count_cell.  With B a power of
// two, raw >= B is a value outside [-1, 1) or NaN: raw + kMagicBits are the
// bits of the round-down fma, which is NaN for NaN (skipped), below 1.5 *
// 2^23 for x < -1 (cell 0) and above it for x >= 1 (cell B - 1), as the cell
// definition clamps; other B pass the clamped cell, and raw >= B is NaN.
// (The kernel passes d = raw - c_lo.)
template <bool POW2>
__device__ __forceinline__ void count_raw(const Cells& S, uint64_t* __restrict__ hist, uint32_t d, unsigned n) {
    if (d < S.ncen) {
        atomicAdd(S.cen + d, n);
        return;
    }
    const uint32_t raw = d + S.c_lo;
    uint32_t c = raw;
    if (raw >= S.B) {
        if (!POW2) return;
        const float f = __uint_as_float(raw + kMagicBits);
        if (isnan(f)) return;
        c = f < kMagic ? 0u : S.B - 1;
    }
    count_cell(S, hist, c, n);
}

template <bool POW2>
__global__ void __launch_bounds__(kHistThreads, 1) k_hist16(const float* __restrict__ x,
                                                           const __grid_constant__ HistLaunch L,
                                                           uint64_t* __restrict__ hist) {
    extern __shared__ uint4 s_dyn[];
    const int B = L.bins;
    Cells S;
    S.B = static_cast<uint32_t>(B);
    S.ncen = central_cells(S.B);
    S.c_lo = (S.B - S.ncen) / 2;
    S.edge = edge_cells(S.B);
    S.cen = reinterpret_cast<unsigned*>(s_dyn);
    S.ext = S.cen + S.ncen;
    for (int i = threadIdx.x; i < static_cast<int>(S.ncen + 2 * S.edge); i += blockDim.x) S.cen[i] = 0u;
    // a NaN value's cell bits: kMagicBits - 1, cell 0xFFFFFFFF
    const uint32_t nan_bits = kMagicBits - 1u;
    const int top_bits = static_cast<int>(kMagicBits) + B - 1;
    if (threadIdx.x == 0)
        for (int p = 0; p < kPrefetchUnits; ++p) {
            const int64_t u = blockIdx.x + static_cast<int64_t>(p) * gridDim.x;
            if (u < L.nunits) prefetch_unit_l2(x, L, u);
        }
    __syncthreads();
    const float halfB = 0.5f * static_cast<float>(B), top = static_cast<float>(B - 1);
    const int lane = threadIdx.x & 31;
    // B a power of two: the cell of x in [-1, 1) before any clamp, one add and
    // one round-down fma (x >= 1, x < -1, infinities and NaN all give raw >= B
    // and are settled by count_raw); other B: the clamped cell.
    // (returned relative to the central run: raw - c_lo, one subtraction)
    const uint32_t base_bits = kMagicBits + S.c_lo;
    auto cell = [&](float v) -> uint32_t {
        if (POW2) return __float_as_uint(__fmaf_rd(__fadd_rn(v, 1.0f), halfB, kMagic)) - base_bits;
        return cell_bits<false>(v, halfB, top, top_bits, nan_bits) - base_bits;
    };
    for (int64_t u = blockIdx.x; u < L.nunits; u += gridDim.x) {
        if (threadIdx.x == 0) {
            const int64_t un = u + static_cast<int64_t>(kPrefetchUnits) * gridDim.x;
            if (un < L.nunits) prefetch_unit_l2(x, L, un);
        }
        const int r = find_range(L, u);
        const int64_t s0 = L.off[r] + (u - L.unit_begin[r]) * kHistUnit;
        const int64_t s1 = min(s0 + kHistUnit, L.off[r] + L.cnt[r]);
        if (s0 < s1) {
            // 16-byte aligned body with float4 loads; scalar head and tail
            int64_t h = (s0 + 3) & ~int64_t(3);
            if (h > s1) h = s1;
            for (int64_t e = s0 + threadIdx.x; e < h; e += blockDim.x) {
                count_raw<POW2>(S, hist, cell(__ldcg(x + e)), 1u);
            }
            const int64_t nv = (s1 - h) >> 2;
            const float4* xv = reinterpret_cast<const float4*>(x + h);
            for (int64_t jw = threadIdx.x & ~31; jw < nv; jw += kHistLoads * blockDim.x) {
                float4 q[kHistLoads];
#pragma unroll
                for (int k = 0; k < kHistLoads; ++k) {
                    const int64_t j = jw + lane + static_cast<int64_t>(k) * blockDim.x;
                    q[k] = j < nv ? __ldcg(xv + j) : make_float4(NAN, NAN, NAN, NAN);
                }
                uint32_t c[4 * kHistLoads];
#pragma unroll
                for (int k = 0; k < kHistLoads; ++k) {
                    c[4 * k] = cell(q[k].x);
                    c[4 * k + 1] = cell(q[k].y);
                    c[4 * k + 2] = cell(q[k].z);
                    c[4 * k + 3] = cell(q[k].w);
                }
                // one cell for the whole round?  Three of each lane's values
                // first (random data fails there), then all of them
                const uint32_t c0 = __shfl_sync(0xffffffffu, c[0], 0);
                bool one = __all_sync(0xffffffffu, c[0] == c0 && c[2 * kHistLoads] == c0 && c[4 * kHistLoads - 1] == c0);
                if (one) {
                    uint32_t diff = 0;
#pragma unroll
                    for (int k = 1; k < 4 * kHistLoads; ++k) diff |= c[k] ^ c0;
                    one = __all_sync(0xffffffffu, diff == 0u);
                }
                if (one) {
                    // equal raw cells are one cell (or all NaN, or all clamped alike)
                    if (lane == 0) count_raw<POW2>(S, hist, c0, 32u * 4u * kHistLoads);
                } else {
#pragma unroll
                    for (int k = 0; k < 4 * kHistLoads; ++k) count_raw<POW2>(S, hist, c[k], 1u);
                }
            }
            for (int64_t e = h + nv * 4 + threadIdx.x; e < s1; e += blockDim.x) {
                count_raw<POW2>(S, hist, cell(__ldcg(x + e)), 1u);
            }
        }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < static_cast<int>(S.ncen); i += blockDim.x) {
        const unsigned c = S.cen[i];
        if (c) atomicAdd(reinterpret_cast<unsigned long long*>(hist + S.c_lo + i), static_cast<unsigned long long>(c));
    }
    for (int i = threadIdx.x; i < static_cast<int>(2 * S.edge); i += blockDim.x) {
        const unsigned c = S.ext[i];
        const uint32_t cl = i < static_cast<int>(S.edge) ? static_cast<uint32_t>(i) : S.B - 2 * S.edge + i;
        if (c) atomicAdd(reinterpret_cast<unsigned long long*>(hist + cl), static_cast<unsigned long long>(c));
    }
}

}  // namespace

cudaError_t prepare_histogram() {
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, k_hist1);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, k_hist16<true>);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, k_hist16<false>);
    return e;
}

// Resident CTAs per SM of k16 with `smem` bytes of shared memory on the
// current device (1 if the query fails), cached per (device, kernel, size).
static int hist16_per_sm(void (*k16)(const float*, HistLaunch, uint64_t*), bool pow2, size_t smem) {
    static std::mutex mu;
    static std::vector<std::pair<std::pair<int, size_t>, int>> cache;  // ((device * 2 + pow2, smem), CTAs)
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    const int key = 2 * dev + (pow2 ? 1 : 0);
    std::lock_guard<std::mutex> g(mu);
    for (const auto& kv : cache)
        if (kv.first.first == key && kv.first.second == smem) return kv.second;
    int n = 1;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k16, kHistThreads, smem) != cudaSuccess || n < 1) {
        (void)cudaGetLastError();
        n = 1;
    }
    cache.push_back({{key, smem}, n});
    return n;
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
            // u32 counters for the central cells and the cells at both ends
            const uint32_t b32 = static_cast<uint32_t>(bins);
            const size_t smem = static_cast<size_t>(central_cells(b32) + 2 * edge_cells(b32)) * sizeof(unsigned);
            const bool pow2 = (bins & (bins - 1)) == 0;
            auto k16 = pow2 ? k_hist16<true> : k_hist16<false>;
            e = cudaFuncSetAttribute(k16, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
            if (e != cudaSuccess) return e;
            // resident CTAs per SM for this size, asked once per device and size
            const int per_sm = hist16_per_sm(k16, pow2, smem);
            const int64_t grid = std::min<int64_t>(units, static_cast<int64_t>(per_sm) * sms);
            k16<<<dim3(static_cast<unsigned>(grid)), kHistThreads, smem, stream>>>(x, L, hist);
        }
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace gefen
