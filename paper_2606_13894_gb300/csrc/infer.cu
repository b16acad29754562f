// gefen_infer_blocks: Automatic Block Partitioning (Algorithm 2; the partition
// score of Sec. 5.1).
//
//   z_j = log(g_j^2 + eps),  mu_i(p) = mean of z over run i of p elements,
//   S(p) = (1/(n/p - 1)) sum_i |mu_{i+1}(p) - mu_i(p)|,
// strict local maxima of S over the ascending divisors 1 < p < n, largest wins
// (smallest p on ties), else 1.
//
// A bf16 |g| takes at most 32768 values, so z comes from a table computed once
// per call in fp64.  z is held in fixed point (z * 2^48; |z| < 746 for any
// double, so 16-value partial sums fit int64) and one
// pass builds exact 128-bit prefix sums P.  Then
//   mu_{i+1} - mu_i = (P[(i+2)p] - 2 P[(i+1)p] + P[ip]) / (2^48 p)
// is an exact integer divided once, so each score costs n/p loads instead of n
// additions, and the sums do not depend on the order of evaluation.
#include <algorithm>
#include <cmath>
#include <vector>

#include "common.cuh"
#include "internal.h"

namespace gefen {

namespace {

constexpr int kInferThreads = 256;
constexpr int kInferPer = 16;          // elements per thread in the scan
constexpr int kInferTile = kInferThreads * kInferPer;
constexpr int kScoreMaxCtas = 512;
constexpr int64_t kInferMaxN = int64_t(1) << 32;

struct i128s {  // two's complement 128-bit value
    uint64_t lo;
    int64_t hi;
};

__device__ __forceinline__ i128s add_i(i128s a, i128s b) {
    i128s r;
    r.lo = a.lo + b.lo;
    r.hi = a.hi + b.hi + (r.lo < a.lo ? 1 : 0);
    return r;
}
__device__ __forceinline__ i128s sub_i(i128s a, i128s b) {
    i128s r;
    r.lo = a.lo - b.lo;
    r.hi = a.hi - b.hi - (a.lo < b.lo ? 1 : 0);
    return r;
}
__device__ __forceinline__ i128s from64(int64_t v) {
    i128s r;
    r.lo = static_cast<uint64_t>(v);
    r.hi = v < 0 ? -1 : 0;
    return r;
}
__device__ __forceinline__ double abs_to_double(i128s v) {
    u128 m;
    if (v.hi < 0) {  // negate
        m.lo = ~v.lo + 1ull;
        m.hi = ~static_cast<uint64_t>(v.hi) + (m.lo == 0 ? 1ull : 0ull);
    } else {
        m.lo = v.lo;
        m.hi = static_cast<uint64_t>(v.hi);
    }
    return u128_to_double_rn(m);
}

struct InferHdr {
    int64_t period;
    int32_t status;  // 0 ok; 1 a gradient gave a non-finite log
    int32_t pad;
};

struct InferWs {
    InferHdr* hdr;
    int64_t* ztab;     // 32768 fixed-point z values
    i128s* tile_sum;   // per scan tile, then its exclusive prefix
    i128s* P;          // n + 1 prefix sums
    double* partial;   // ndiv x kScoreMaxCtas
    double* scores;    // ndiv
    int64_t* divs;     // ndiv (device copy)
};

struct InferLayout {
    size_t hdr, ztab, tile, P, partial, scores, divs, total;
};

InferLayout infer_layout(int64_t n, int64_t ndiv) {
    InferLayout L;
    size_t o = 0;
    const int64_t ntiles = (n + kInferTile - 1) / kInferTile;
    L.hdr = o; o += align_up(sizeof(InferHdr));
    L.ztab = o; o += align_up(32768 * sizeof(int64_t));
    L.tile = o; o += align_up(static_cast<size_t>(ntiles + 1) * sizeof(i128s));
    L.P = o; o += align_up(static_cast<size_t>(n + 1) * sizeof(i128s));
    L.partial = o; o += align_up(static_cast<size_t>(ndiv) * kScoreMaxCtas * sizeof(double));
    L.scores = o; o += align_up(static_cast<size_t>(ndiv) * sizeof(double));
    L.divs = o; o += align_up(static_cast<size_t>(ndiv) * sizeof(int64_t));
    L.total = o;
    return L;
}

std::vector<int64_t> divisors_of(int64_t n) {
    std::vector<int64_t> lo, hi;
    for (int64_t d = 1; d * d <= n; ++d) {
        if (n % d) continue;
        lo.push_back(d);
        if (d * d != n) hi.push_back(n / d);
    }
    lo.insert(lo.end(), hi.rbegin(), hi.rend());
    return lo;
}

__global__ void k_infer_ztab(double eps, InferWs W) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t == 0) { W.hdr->status = 0; W.hdr->period = 1; }
    if (t >= 32768) return;
    const double g = static_cast<double>(bf16_bits_to_f32(static_cast<uint16_t>(t)));
    const double z = log(g * g + eps);
    if (!isfinite(z)) {
        W.ztab[t] = 0;
        return;
    }
    W.ztab[t] = __double2ll_rn(z * 281474976710656.0);  // z * 2^48
}

__device__ __forceinline__ int64_t zfix(const int64_t* __restrict__ ztab, uint16_t bits, int* bad) {
    const uint16_t a = bits & 0x7FFFu;
    if ((a & 0x7F80u) == 0x7F80u) *bad = 1;  // inf or NaN gradient
    return __ldg(ztab + a);
}

// Per-thread sums of 16 consecutive z, then the tile's sum.
__device__ __forceinline__ int64_t thread_sum16(const uint16_t* __restrict__ g, int64_t n, int64_t e0,
                                                const int64_t* __restrict__ ztab, int64_t* z, int* bad) {
    int64_t s = 0;
    if (e0 + kInferPer <= n && ((reinterpret_cast<uintptr_t>(g + e0) & 15u) == 0)) {
        const uint4 a = __ldg(reinterpret_cast<const uint4*>(g + e0));
        const uint4 b = __ldg(reinterpret_cast<const uint4*>(g + e0) + 1);
        const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            z[2 * i] = zfix(ztab, static_cast<uint16_t>(w[i] & 0xFFFFu), bad);
            z[2 * i + 1] = zfix(ztab, static_cast<uint16_t>(w[i] >> 16), bad);
        }
    } else {
#pragma unroll
        for (int i = 0; i < kInferPer; ++i) z[i] = (e0 + i < n) ? zfix(ztab, g[e0 + i], bad) : 0;
    }
#pragma unroll
    for (int i = 0; i < kInferPer; ++i) s += z[i];
    return s;
}

// Inclusive block scan of 128-bit values (Hillis-Steele in shared memory).
__device__ __forceinline__ i128s block_scan_incl(i128s v, i128s* s) {
    const int t = threadIdx.x;
    s[t] = v;
    __syncthreads();
    for (int o = 1; o < blockDim.x; o <<= 1) {
        i128s a = from64(0);
        if (t >= o) a = s[t - o];
        __syncthreads();
        if (t >= o) s[t] = add_i(s[t], a);
        __syncthreads();
    }
    return s[t];
}

__global__ void __launch_bounds__(kInferThreads) k_infer_tilesum(const uint16_t* __restrict__ g, int64_t n,
                                                                  InferWs W) {
    __shared__ i128s s[kInferThreads];
    int bad = 0;
    int64_t z[kInferPer];
    const int64_t e0 = static_cast<int64_t>(blockIdx.x) * kInferTile + threadIdx.x * kInferPer;
    const int64_t ts = thread_sum16(g, n, e0, W.ztab, z, &bad);
    if (bad) W.hdr->status = 1;
    const i128s tot = block_scan_incl(from64(ts), s);
    if (threadIdx.x == blockDim.x - 1) W.tile_sum[blockIdx.x] = tot;
}

// Exclusive prefix of the tile sums (one CTA, chunks of blockDim.x).
__global__ void __launch_bounds__(1024) k_infer_scan_tiles(int64_t ntiles, InferWs W) {
    __shared__ i128s s[1024];
    i128s carry = from64(0);
    for (int64_t base = 0; base < ntiles; base += blockDim.x) {
        const int64_t i = base + threadIdx.x;
        const i128s v = i < ntiles ? W.tile_sum[i] : from64(0);
        const i128s inc = block_scan_incl(v, s);
        const i128s total = s[blockDim.x - 1];
        if (i < ntiles) W.tile_sum[i] = add_i(carry, sub_i(inc, v));
        carry = add_i(carry, total);
        __syncthreads();
    }
}

__global__ void __launch_bounds__(kInferThreads) k_infer_prefix(const uint16_t* __restrict__ g, int64_t n,
                                                                 InferWs W) {
    __shared__ i128s s[kInferThreads];
    int bad = 0;
    int64_t z[kInferPer];
    const int64_t e0 = static_cast<int64_t>(blockIdx.x) * kInferTile + threadIdx.x * kInferPer;
    const int64_t ts = thread_sum16(g, n, e0, W.ztab, z, &bad);
    const i128s inc = block_scan_incl(from64(ts), s);
    i128s run = add_i(W.tile_sum[blockIdx.x], sub_i(inc, from64(ts)));
    if (blockIdx.x == 0 && threadIdx.x == 0) W.P[0] = from64(0);
#pragma unroll
    for (int i = 0; i < kInferPer; ++i) {
        if (e0 + i >= n) break;
        run = add_i(run, from64(z[i]));
        W.P[e0 + i + 1] = run;
    }
}

// Per-CTA partial sums of |mu_{i+1} - mu_i| for divisor q (p = divs[q]).
__global__ void __launch_bounds__(kInferThreads) k_infer_score(int64_t n, int q, int64_t p, InferWs W) {
    __shared__ double s[kInferThreads];
    const int64_t nb = n / p;
    const double scale = 1.0 / (281474976710656.0 * static_cast<double>(p));
    double acc = 0.0;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i + 1 < nb;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const i128s a = W.P[i * p], b = W.P[(i + 1) * p], c = W.P[(i + 2) * p];
        const i128s d2 = sub_i(add_i(a, c), add_i(b, b));
        acc += abs_to_double(d2) * scale;
    }
    s[threadIdx.x] = acc;
    __syncthreads();
    for (int o = blockDim.x / 2; o > 0; o >>= 1) {
        if (threadIdx.x < o) s[threadIdx.x] += s[threadIdx.x + o];
        __syncthreads();
    }
    if (threadIdx.x == 0) W.partial[static_cast<size_t>(q) * kScoreMaxCtas + blockIdx.x] = s[0];
}

// Scores from the partials, then the selection rule (one CTA).
__global__ void __launch_bounds__(256) k_infer_select(int64_t n, int ndiv, const int* __restrict__ nctas, InferWs W) {
    for (int q = threadIdx.x; q < ndiv; q += blockDim.x) {
        const int64_t p = W.divs[q], nb = n / p;
        double s = 0.0;
        const int c = nctas[q];
        for (int j = 0; j < c; ++j) s += W.partial[static_cast<size_t>(q) * kScoreMaxCtas + j];
        W.scores[q] = nb > 1 ? s / static_cast<double>(nb - 1) : __longlong_as_double(0x7ff8000000000000ll);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int64_t best_p = 1;
        double best_s = 0.0;
        bool have = false;
        for (int q = 1; q + 1 < ndiv; ++q) {
            const double sq = W.scores[q];
            if (sq > W.scores[q - 1] && sq > W.scores[q + 1]) {
                if (!have || sq > best_s) { best_s = sq; best_p = W.divs[q]; have = true; }
            }
        }
        W.hdr->period = have ? best_p : 1;
    }
}

InferWs infer_ws(void* base, int64_t n, int64_t ndiv) {
    const InferLayout L = infer_layout(n, ndiv);
    char* p = static_cast<char*>(base);
    InferWs w;
    w.hdr = reinterpret_cast<InferHdr*>(p + L.hdr);
    w.ztab = reinterpret_cast<int64_t*>(p + L.ztab);
    w.tile_sum = reinterpret_cast<i128s*>(p + L.tile);
    w.P = reinterpret_cast<i128s*>(p + L.P);
    w.partial = reinterpret_cast<double*>(p + L.partial);
    w.scores = reinterpret_cast<double*>(p + L.scores);
    w.divs = reinterpret_cast<int64_t*>(p + L.divs);
    return w;
}

}  // namespace

}  // namespace gefen

using namespace gefen;

extern "C" size_t gefen_infer_workspace_size(int64_t numel) {
    if (numel < 1 || numel > kInferMaxN) return 0;
    const int64_t nd = static_cast<int64_t>(divisors_of(numel).size());
    // the per-divisor CTA counts travel in the workspace too
    return infer_layout(numel, nd).total + align_up(static_cast<size_t>(nd) * sizeof(int));
}

extern "C" gefen_status_t gefen_infer_blocks(const uint16_t* grad, int64_t numel, double eps, int64_t* period_out,
                                             double* scores_out, int64_t scores_cap, int64_t* ndiv_out,
                                             void* workspace, size_t workspace_bytes, gefen_stream_t stream) {
    if (grad == nullptr || period_out == nullptr || numel < 1 || numel > kInferMaxN) return GEFEN_EINVAL;
    if (!(eps > 0.0) || !std::isfinite(eps)) return GEFEN_EINVAL;
    if (scores_out != nullptr && scores_cap < 0) return GEFEN_EINVAL;
    const size_t need = gefen_infer_workspace_size(numel);
    if (workspace == nullptr || workspace_bytes < need) return GEFEN_ENOMEM;
    if (reinterpret_cast<uintptr_t>(workspace) % kWsAlign) return GEFEN_EINVAL;
    if (gefen_status_t s = check_device(); s != GEFEN_OK) return s;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const std::vector<int64_t> divs = divisors_of(numel);
    const int nd = static_cast<int>(divs.size());
    const InferLayout L = infer_layout(numel, nd);
    InferWs W = infer_ws(workspace, numel, nd);
    int* d_nctas = reinterpret_cast<int*>(static_cast<char*>(workspace) + L.total);
    std::vector<int> nctas(nd);
    for (int q = 0; q < nd; ++q) {
        const int64_t nb = numel / divs[q];
        const int64_t work = std::max<int64_t>(0, nb - 1);
        nctas[q] = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(kScoreMaxCtas, (work + 4095) / 4096)));
    }
    // small host tables travel with the stream (pageable copies are staged)
    if (cudaMemcpyAsync(W.divs, divs.data(), nd * sizeof(int64_t), cudaMemcpyHostToDevice, st) != cudaSuccess ||
        cudaMemcpyAsync(d_nctas, nctas.data(), nd * sizeof(int), cudaMemcpyHostToDevice, st) != cudaSuccess)
        return GEFEN_ECUDA;
    const int64_t ntiles = (numel + kInferTile - 1) / kInferTile;
    k_infer_ztab<<<128, 256, 0, st>>>(eps, W);
    k_infer_tilesum<<<dim3(static_cast<unsigned>(ntiles)), kInferThreads, 0, st>>>(grad, numel, W);
    k_infer_scan_tiles<<<1, 1024, 0, st>>>(ntiles, W);
    k_infer_prefix<<<dim3(static_cast<unsigned>(ntiles)), kInferThreads, 0, st>>>(grad, numel, W);
    for (int q = 0; q < nd; ++q) k_infer_score<<<nctas[q], kInferThreads, 0, st>>>(numel, q, divs[q], W);
    k_infer_select<<<1, 256, 0, st>>>(numel, nd, d_nctas, W);
    if (cudaGetLastError() != cudaSuccess) return GEFEN_ECUDA;
    InferHdr h;
    if (cudaMemcpyAsync(&h, W.hdr, sizeof(h), cudaMemcpyDeviceToHost, st) != cudaSuccess) return GEFEN_ECUDA;
    std::vector<double> sc;
    if (scores_out && scores_cap > 0) {
        sc.resize(nd);
        if (cudaMemcpyAsync(sc.data(), W.scores, nd * sizeof(double), cudaMemcpyDeviceToHost, st) != cudaSuccess)
            return GEFEN_ECUDA;
    }
    if (cudaStreamSynchronize(st) != cudaSuccess) return GEFEN_ECUDA;
    if (h.status) return GEFEN_EDEVICE;
    *period_out = h.period;
    if (ndiv_out) *ndiv_out = nd;
    if (scores_out)
        for (int q = 0; q < nd && q < scores_cap; ++q) scores_out[q] = sc[q];
    return GEFEN_OK;
}
