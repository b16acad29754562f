// gefen_muon_step: Gefen-Muon (the paper's appendix "Gefen-Muon") on sm_103a.
//
// Muon's momentum buffer is kept as Gefen codes with a per-block absmax scale
// (Algorithm 1, Quantize); the orthogonalisation is Muon's:
//   m    = mu * Cdec[c] * s_b + (1 - mu) * g           (buffer, decoded + EMA)
//   s'_b = max |m|, c = nearest level of m / s'_b in Cenc, s_b = s'_b
//   U    = g + mu (m - g) with Nesterov, else m
//   X    = U / max(||U||_F, eps); X <- a X + (b A + c A A) X, A = X X^T,
//          on the smaller side (ns_steps times)
//   theta = theta (1 - lr wd) - lr sqrt(max(1, rows/cols)) X
// The element-wise parts and the Newton-Schulz products are this library's
// kernels: with bf16 storage (as Muon runs them) the products are the tcgen05
// GEMM of gemm.cu, with fp32 storage its CUDA-core fallback.
//
// The working matrix X is s x n with s = min(rows, cols) on the small side:
// X = U for rows <= cols, X = U^T otherwise.  Both X and T = X^T are kept,
// row-major, so that every product reads K-contiguous operands:
//   A  = X X^T                      (s x s, K = n)
//   B  = c A A^T + b A              (A is symmetric: A A^T = A A)
//   X' = B X + a X = B T^T + a X    (s x n, K = s), written with T' = X'^T
// One of the two layouts is U's own (rows x cols row-major), so the update
// reads the result in place.
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace gefen {

namespace {

constexpr int kMuThreads = 256;
constexpr int kMuPartials = 1024;  // CTAs of the encode kernel (norm partials)

struct MuonLayout {
    size_t hdr, snew, part, p0, p1, q0, q1, ga, gb, total;
};

// header (256 B; word 0: a bounded wait gave up; byte 16: 1 / ||U||) | new scales | norm
// partials | two rows x cols buffers (U's layout) | two cols x rows buffers
// (transposed) | A | B
MuonLayout muon_layout(int64_t rows, int64_t cols, int64_t period, bool bf16) {
    MuonLayout L;
    const int64_t n = rows * cols, s = std::min(rows, cols);
    const size_t eb = bf16 ? 2 : 4;
    size_t o = 0;
    L.hdr = o; o += kWsAlign;
    L.snew = o; o += align_up(static_cast<size_t>(n / period) * sizeof(float));
    L.part = o; o += align_up(static_cast<size_t>(kMuPartials) * sizeof(double));
    L.p0 = o; o += align_up(static_cast<size_t>(n) * eb);
    L.p1 = o; o += align_up(static_cast<size_t>(n) * eb);
    L.q0 = o; o += align_up(static_cast<size_t>(n) * eb);
    L.q1 = o; o += align_up(static_cast<size_t>(n) * eb);
    L.ga = o; o += align_up(static_cast<size_t>(s * s) * eb);
    L.gb = o; o += align_up(static_cast<size_t>(s * s) * eb);
    L.total = o;
    return L;
}

struct MuonArgs {
    int64_t n, period;
    float mu, omm;  // momentum, 1 - momentum
    int nesterov, k;
    const uint16_t* grads;
    uint8_t* codes;
    float* scale;
    const float* cb_dec;
    const float* cb_enc;
    float* snew;
    double* part;
    void* u;  // update buffer (fp32 or bf16)
};

// Block of element e (a 32-bit division whenever n < 2^32, the usual case).
__device__ __forceinline__ int64_t muon_block(const MuonArgs& A, int64_t e) {
    if (A.n < (int64_t(1) << 32))
        return static_cast<uint32_t>(e) / static_cast<uint32_t>(A.period);
    return e / A.period;
}

__device__ __forceinline__ float muon_m(const MuonArgs& A, const float* s_dec, int64_t e, int64_t bi) {
    const float g = bf16_bits_to_f32(A.grads[e]);
    return fmaf(A.omm, g, A.mu * A.scale[bi] * s_dec[A.codes[e]]);
}

// s'_b = max |m| over each block (atomic max of non-negative float bits:
// exact and order-independent).  A warp whose 32 elements lie in one block
// takes their maximum first and sends one atomic.
__global__ void __launch_bounds__(kMuThreads) k_muon_absmax(MuonArgs A) {
    __shared__ float s_dec[kMaxLevels];
    if (threadIdx.x < kMaxLevels) s_dec[threadIdx.x] = threadIdx.x < A.k ? A.cb_dec[threadIdx.x] : 0.0f;
    __syncthreads();
    for (int64_t e = blockIdx.x * static_cast<int64_t>(kMuThreads) + threadIdx.x; e < A.n;
         e += static_cast<int64_t>(gridDim.x) * kMuThreads) {
        const int64_t bi = muon_block(A, e);
        const unsigned am = __float_as_uint(fabsf(muon_m(A, s_dec, e, bi)));
        unsigned* dst = reinterpret_cast<unsigned int*>(A.snew) + bi;
        const unsigned live = __activemask();
        const int first = __ffs(live) - 1;
        const long long b0 = __shfl_sync(live, static_cast<long long>(bi), first);
        if (__all_sync(live, bi == b0)) {
            const unsigned wm = __reduce_max_sync(live, am);
            if ((threadIdx.x & 31) == first) atomicMax(dst, wm);
        } else {
            atomicMax(dst, am);
        }
    }
}

// Vector forms (period % 8 == 0, n % 8 == 0, codes 8-byte aligned): a thread
// takes eight consecutive elements -- one 16-byte load of g, one 8-byte load
// of codes, all in one block -- with the same arithmetic per element as the
// scalar forms.
__device__ __forceinline__ void load8(const MuonArgs& A, int64_t v, float (&g)[8], uint32_t (&c)[8]) {
    const uint4 gw = reinterpret_cast<const uint4*>(A.grads)[v];
    const uint2 cw = reinterpret_cast<const uint2*>(A.codes)[v];
    const uint32_t gg[4] = {gw.x, gw.y, gw.z, gw.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        g[2 * i] = bf16_lo(gg[i]);
        g[2 * i + 1] = bf16_hi(gg[i]);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        c[i] = (cw.x >> (8 * i)) & 0xFFu;
        c[4 + i] = (cw.y >> (8 * i)) & 0xFFu;
    }
}

__global__ void __launch_bounds__(kMuThreads) k_muon_absmax8(MuonArgs A) {
    __shared__ float s_dec[kMaxLevels];
    if (threadIdx.x < kMaxLevels) s_dec[threadIdx.x] = threadIdx.x < A.k ? A.cb_dec[threadIdx.x] : 0.0f;
    __syncthreads();
    const int64_t nv = A.n >> 3;
    for (int64_t v = blockIdx.x * static_cast<int64_t>(kMuThreads) + threadIdx.x; v < nv;
         v += static_cast<int64_t>(gridDim.x) * kMuThreads) {
        const int64_t bi = muon_block(A, v << 3);
        float g[8];
        uint32_t c[8];
        load8(A, v, g, c);
        const float mus = A.mu * A.scale[bi];
        float am = 0.0f;
#pragma unroll
        for (int i = 0; i < 8; ++i) am = fmaxf(am, fabsf(fmaf(A.omm, g[i], mus * s_dec[c[i]])));
        unsigned* dst = reinterpret_cast<unsigned int*>(A.snew) + bi;
        const unsigned live = __activemask();
        const int first = __ffs(live) - 1;
        const long long b0 = __shfl_sync(live, static_cast<long long>(bi), first);
        const unsigned ab = __float_as_uint(am);
        if (__all_sync(live, bi == b0)) {
            const unsigned wm = __reduce_max_sync(live, ab);
            if ((threadIdx.x & 31) == first) atomicMax(dst, wm);
        } else {
            atomicMax(dst, ab);
        }
    }
}

// Encoding as the step kernels do it: x = m * (1 / s'), its level from the
// cell records (four copies), the binary search when a cell holds more than
// three midpoints.
constexpr int kMuLutR = 4;

template <bool BF16>
__global__ void __launch_bounds__(kMuThreads) k_muon_encode8(MuonArgs A) {
    __shared__ float s_dec[kMaxLevels], s_mid[kMaxLevels + 4];
    __shared__ float4 s_lut[(kLutCells + 2) * kMuLutR];
    __shared__ double s_red[kMuThreads / 32];
    const int t = threadIdx.x;
    if (t < kMaxLevels) s_dec[t] = t < A.k ? A.cb_dec[t] : 0.0f;
    for (int i = t; i < kMaxLevels + 4; i += kMuThreads)
        s_mid[i] = (i < A.k - 1) ? 0.5f * (A.cb_enc[i] + A.cb_enc[i + 1]) : INFINITY;
    __syncthreads();
    const bool lut = !__syncthreads_or(build_cell_records<kMuLutR>(s_mid, s_lut, t, kMuThreads));
    const int zero_code = level_search(s_mid, 0.0f);
    const int copy = t % kMuLutR;
    double acc = 0.0;
    const int64_t nv = A.n >> 3;
    for (int64_t v = blockIdx.x * static_cast<int64_t>(kMuThreads) + t; v < nv;
         v += static_cast<int64_t>(gridDim.x) * kMuThreads) {
        const int64_t bi = muon_block(A, v << 3);
        float g[8];
        uint32_t c[8];
        load8(A, v, g, c);
        const float mus = A.mu * A.scale[bi];
        const float sn = A.snew[bi];
        const float inv = sn > 0.0f ? __frcp_rn(sn) : 0.0f;
        float u[8];
        uint32_t cw[2] = {0u, 0u};
        float sq = 0.0f;  // squares of the stored update, exact in fp32 for bf16 values
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const float m = fmaf(A.omm, g[i], mus * s_dec[c[i]]);
            const float x = m * inv;
            const uint32_t code = sn <= 0.0f ? static_cast<uint32_t>(zero_code)
                                  : lut      ? lut_encode<kMuLutR>(s_lut, copy, x)
                                             : static_cast<uint32_t>(level_search(s_mid, x));
            cw[i >> 2] |= code << (8 * (i & 3));
            u[i] = A.nesterov ? fmaf(A.mu, m - g[i], g[i]) : m;
            if (BF16) u[i] = __bfloat162float(__float2bfloat16_rn(u[i]));
        }
        reinterpret_cast<uint2*>(A.codes)[v] = make_uint2(cw[0], cw[1]);
        if (BF16) {
            __nv_bfloat162 h[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(u[2 * i], u[2 * i + 1]);
            reinterpret_cast<uint4*>(A.u)[v] = *reinterpret_cast<uint4*>(h);
#pragma unroll
            for (int i = 0; i < 8; ++i) sq = fmaf(u[i], u[i], sq);
            acc += static_cast<double>(sq);
        } else {
            float4* uo = reinterpret_cast<float4*>(A.u) + 2 * v;
            uo[0] = make_float4(u[0], u[1], u[2], u[3]);
            uo[1] = make_float4(u[4], u[5], u[6], u[7]);
#pragma unroll
            for (int i = 0; i < 8; ++i) acc += static_cast<double>(u[i]) * u[i];
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if ((t & 31) == 0) s_red[t >> 5] = acc;
    __syncthreads();
    if (t == 0) {
        double sum = 0.0;
        for (int w = 0; w < kMuThreads / 32; ++w) sum += s_red[w];
        A.part[blockIdx.x] = sum;
    }
}

// 1 / max(||U||, eps) from the partials, summed in one fixed order.
__global__ void __launch_bounds__(kMuThreads) k_muon_inv(const double* __restrict__ part, int nparts, double eps,
                                                        float* __restrict__ inv_out) {
    __shared__ double s_sum[kMuThreads];
    double ps = 0.0;
    for (int i = threadIdx.x; i < nparts; i += kMuThreads) ps += part[i];
    s_sum[threadIdx.x] = ps;
    __syncthreads();
    for (int w = kMuThreads / 2; w > 0; w >>= 1) {
        if (threadIdx.x < w) s_sum[threadIdx.x] += s_sum[threadIdx.x + w];
        __syncthreads();
    }
    if (threadIdx.x == 0) *inv_out = static_cast<float>(1.0 / fmax(sqrt(s_sum[0]), eps));
}

// X = U / ||U|| in place (rows x cols) and, when ut is given, its transpose
// (cols x rows), 32 x 32 tiles through shared memory; the new scales are
// committed on the way.
template <typename T>
__global__ void __launch_bounds__(256) k_muon_scale_t(T* __restrict__ u, T* __restrict__ ut, int rows, int cols,
                                                     const float* __restrict__ inv_p, float* __restrict__ scale,
                                                     const float* __restrict__ snew, int64_t nb) {
    __shared__ T tile[32][33];
    const float inv = *inv_p;
    const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    for (int i = ty; i < 32; i += 8) {
        if (r0 + i < rows && c0 + tx < cols) {
            T* p = u + static_cast<int64_t>(r0 + i) * cols + c0 + tx;
            T y;
            if constexpr (sizeof(T) == 2) y = __float2bfloat16_rn(__bfloat162float(*p) * inv);
            else y = *p * inv;
            *p = y;
            tile[i][tx] = y;
        }
    }
    const int64_t cta = static_cast<int64_t>(blockIdx.y) * gridDim.x + blockIdx.x;
    const int64_t ncta = static_cast<int64_t>(gridDim.x) * gridDim.y;
    for (int64_t b = cta * 256 + threadIdx.x; b < nb; b += ncta * 256) scale[b] = snew[b];
    if (ut == nullptr) return;
    __syncthreads();
    for (int i = ty; i < 32; i += 8)
        if (c0 + i < cols && r0 + tx < rows) ut[static_cast<int64_t>(c0 + i) * rows + r0 + tx] = tile[tx][i];
}

// The bf16 form for even rows and cols: 64 x 64 tiles, each lane moving two
// elements (four bytes), so a warp reads and writes whole 128-byte rows of U
// and of U^T; the tile's rows are 66 elements apart in shared memory (the
// column reads of the transpose meet at most two lanes per bank).
__global__ void __launch_bounds__(256) k_muon_scale_t2(__nv_bfloat16* __restrict__ u, __nv_bfloat16* __restrict__ ut,
                                                      int rows, int cols, const float* __restrict__ inv_p,
                                                      float* __restrict__ scale, const float* __restrict__ snew,
                                                      int64_t nb) {
    __shared__ __nv_bfloat162 tile[64][33];  // row i: columns 2 j, 2 j + 1 in entry j
    const float inv = *inv_p;
    const int c0 = blockIdx.x * 64, r0 = blockIdx.y * 64;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int i = warp; i < 64; i += 8) {
        const int r = r0 + i, c = c0 + 2 * lane;
        if (r < rows && c < cols) {
            __nv_bfloat162* p = reinterpret_cast<__nv_bfloat162*>(u + static_cast<int64_t>(r) * cols + c);
            const float2 f = __bfloat1622float2(*p);
            const __nv_bfloat162 y = __floats2bfloat162_rn(f.x * inv, f.y * inv);
            *p = y;
            tile[i][lane] = y;
        }
    }
    const int64_t cta = static_cast<int64_t>(blockIdx.y) * gridDim.x + blockIdx.x;
    const int64_t ncta = static_cast<int64_t>(gridDim.x) * gridDim.y;
    for (int64_t b = cta * 256 + threadIdx.x; b < nb; b += ncta * 256) scale[b] = snew[b];
    if (ut == nullptr) return;
    __syncthreads();
    // row c0 + j of U^T: lane l writes its elements r0 + 2 l and r0 + 2 l + 1
    for (int j = warp; j < 64; j += 8) {
        const int c = c0 + j, r = r0 + 2 * lane;
        if (c < cols && r < rows) {
            const __nv_bfloat162 a = tile[2 * lane][j >> 1], b = tile[2 * lane + 1][j >> 1];
            const __nv_bfloat162 o = (j & 1) ? __halves2bfloat162(a.y, b.y) : __halves2bfloat162(a.x, b.x);
            *reinterpret_cast<__nv_bfloat162*>(ut + static_cast<int64_t>(c) * rows + r) = o;
        }
    }
}

// theta = theta * decay - step * X, four elements per thread.
template <bool BF16>
__global__ void __launch_bounds__(kMuThreads) k_muon_update4(float* __restrict__ theta, const void* __restrict__ x,
                                                          int64_t n4, float decay, float step) {
    for (int64_t v = blockIdx.x * static_cast<int64_t>(kMuThreads) + threadIdx.x; v < n4;
         v += static_cast<int64_t>(gridDim.x) * kMuThreads) {
        float xv[4];
        if (BF16) {
            const uint2 w = reinterpret_cast<const uint2*>(x)[v];
            xv[0] = bf16_lo(w.x);
            xv[1] = bf16_hi(w.x);
            xv[2] = bf16_lo(w.y);
            xv[3] = bf16_hi(w.y);
        } else {
            const float4 f = reinterpret_cast<const float4*>(x)[v];
            xv[0] = f.x; xv[1] = f.y; xv[2] = f.z; xv[3] = f.w;
        }
        float4 t4 = reinterpret_cast<float4*>(theta)[v];
        t4.x = fmaf(-step, xv[0], decay * t4.x);
        t4.y = fmaf(-step, xv[1], decay * t4.y);
        t4.z = fmaf(-step, xv[2], decay * t4.z);
        t4.w = fmaf(-step, xv[3], decay * t4.w);
        reinterpret_cast<float4*>(theta)[v] = t4;
    }
}

// Re-encode, write the update U and each CTA's partial sum of U^2.
template <bool BF16>
__global__ void __launch_bounds__(kMuThreads) k_muon_encode(MuonArgs A) {
    __shared__ float s_dec[kMaxLevels], s_mid[kMaxLevels];
    __shared__ double s_red[kMuThreads / 32];
    const int t = threadIdx.x;
    if (t < kMaxLevels) {
        s_dec[t] = t < A.k ? A.cb_dec[t] : 0.0f;
        s_mid[t] = (t < A.k - 1) ? 0.5f * (A.cb_enc[t] + A.cb_enc[t + 1]) : INFINITY;
    }
    __syncthreads();
    const int zero_code = level_search(s_mid, 0.0f);
    double acc = 0.0;
    for (int64_t e = blockIdx.x * static_cast<int64_t>(kMuThreads) + t; e < A.n;
         e += static_cast<int64_t>(gridDim.x) * kMuThreads) {
        const int64_t bi = muon_block(A, e);
        const float g = bf16_bits_to_f32(A.grads[e]);
        const float m = fmaf(A.omm, g, A.mu * A.scale[bi] * s_dec[A.codes[e]]);
        const float sn = A.snew[bi];
        A.codes[e] = static_cast<uint8_t>(sn > 0.0f ? level_search(s_mid, __fdiv_rn(m, sn)) : zero_code);
        const float u = A.nesterov ? fmaf(A.mu, m - g, g) : m;
        if (BF16) {
            const __nv_bfloat16 ub = __float2bfloat16_rn(u);
            reinterpret_cast<__nv_bfloat16*>(A.u)[e] = ub;
            const double ud = static_cast<double>(__bfloat162float(ub));
            acc += ud * ud;
        } else {
            reinterpret_cast<float*>(A.u)[e] = u;
            acc += static_cast<double>(u) * u;
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if ((t & 31) == 0) s_red[t >> 5] = acc;
    __syncthreads();
    if (t == 0) {
        double s = 0.0;
        for (int w = 0; w < kMuThreads / 32; ++w) s += s_red[w];
        A.part[blockIdx.x] = s;
    }
}

template <bool BF16>
__global__ void __launch_bounds__(kMuThreads) k_muon_update(float* __restrict__ theta, const void* __restrict__ x,
                                                         int64_t n, float decay, float step) {
    for (int64_t e = blockIdx.x * static_cast<int64_t>(kMuThreads) + threadIdx.x; e < n;
         e += static_cast<int64_t>(gridDim.x) * kMuThreads) {
        const float xv = BF16 ? __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(x)[e])
                              : reinterpret_cast<const float*>(x)[e];
        theta[e] = fmaf(-step, xv, decay * theta[e]);
    }
}

}  // namespace

}  // namespace gefen

using namespace gefen;

extern "C" size_t gefen_muon_workspace_size(int64_t rows, int64_t cols, int64_t period, uint32_t flags) {
    if (rows < 1 || cols < 1 || period < 1 || (rows * cols) % period != 0) return 0;
    if (rows > (int64_t(1) << 31) - 1 || cols > (int64_t(1) << 31) - 1) return 0;
    return muon_layout(rows, cols, period, (flags & GEFEN_MUON_BF16_GEMM) != 0).total;
}

extern "C" gefen_status_t gefen_muon_step(int64_t rows, int64_t cols, int64_t period, float* params,
                                          const uint16_t* grads, uint8_t* codes, float* scale,
                                          const float* codebook_dec, const float* codebook_enc, int32_t k,
                                          gefen_muon_hparams_t hp, void* workspace, size_t workspace_bytes,
                                          gefen_stream_t stream) {
    if (rows < 1 || cols < 1 || period < 1 || (rows * cols) % period != 0) return GEFEN_EINVAL;
    if (rows > (int64_t(1) << 31) - 1 || cols > (int64_t(1) << 31) - 1) return GEFEN_EINVAL;
    if (!params || !grads || !codes || !scale || !codebook_dec || !codebook_enc) return GEFEN_EINVAL;
    if (k < 2 || k > GEFEN_MAX_LEVELS) return GEFEN_EINVAL;
    if (hp.flags & ~GEFEN_MUON_BF16_GEMM) return GEFEN_EINVAL;
    if (!(hp.momentum >= 0.0 && hp.momentum < 1.0) || !std::isfinite(hp.lr) || !std::isfinite(hp.weight_decay) ||
        !(hp.eps > 0.0) || hp.ns_steps < 0 || hp.ns_steps > 100 || !std::isfinite(hp.ns_a) ||
        !std::isfinite(hp.ns_b) || !std::isfinite(hp.ns_c))
        return GEFEN_EINVAL;
    if ((reinterpret_cast<uintptr_t>(params) | reinterpret_cast<uintptr_t>(grads)) & 15u) return GEFEN_EINVAL;
    const bool bf16 = (hp.flags & GEFEN_MUON_BF16_GEMM) != 0;
    const MuonLayout L = muon_layout(rows, cols, period, bf16);
    if (workspace == nullptr || workspace_bytes < L.total) return GEFEN_ENOMEM;
    if (reinterpret_cast<uintptr_t>(workspace) % kWsAlign) return GEFEN_EINVAL;
    if (gefen_status_t s = check_device(); s != GEFEN_OK) return s;

    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    char* ws = static_cast<char*>(workspace);
    const int64_t n = rows * cols;
    MuonArgs A;
    A.n = n;
    A.period = period;
    A.mu = static_cast<float>(hp.momentum);
    A.omm = static_cast<float>(1.0 - hp.momentum);
    A.nesterov = hp.nesterov ? 1 : 0;
    A.k = k;
    A.grads = grads;
    A.codes = codes;
    A.scale = scale;
    A.cb_dec = codebook_dec;
    A.cb_enc = codebook_enc;
    A.snew = reinterpret_cast<float*>(ws + L.snew);
    A.part = reinterpret_cast<double*>(ws + L.part);
    void* P0 = ws + L.p0;
    void* P1 = ws + L.p1;
    void* Q0 = ws + L.q0;
    void* Q1 = ws + L.q1;
    void* GA = ws + L.ga;
    void* GB = ws + L.gb;
    int* err = reinterpret_cast<int*>(ws + L.hdr);
    A.u = P0;

    const int grid = static_cast<int>(std::min<int64_t>(kMuPartials, (n + kMuThreads - 1) / kMuThreads));
    // eight elements per thread when whole groups of eight share a block
    const bool vec = period % 8 == 0 && n % 8 == 0 && (reinterpret_cast<uintptr_t>(codes) & 7u) == 0;
    if (cudaMemsetAsync(A.snew, 0, static_cast<size_t>(n / period) * sizeof(float), st) != cudaSuccess)
        return GEFEN_ECUDA;
    if (vec) k_muon_absmax8<<<grid, kMuThreads, 0, st>>>(A);
    else k_muon_absmax<<<grid, kMuThreads, 0, st>>>(A);
    if (bf16) {
        if (vec) k_muon_encode8<true><<<grid, kMuThreads, 0, st>>>(A);
        else k_muon_encode<true><<<grid, kMuThreads, 0, st>>>(A);
    } else {
        if (vec) k_muon_encode8<false><<<grid, kMuThreads, 0, st>>>(A);
        else k_muon_encode<false><<<grid, kMuThreads, 0, st>>>(A);
    }
    float* inv = reinterpret_cast<float*>(ws + L.hdr + 16);
    k_muon_inv<<<1, kMuThreads, 0, st>>>(A.part, grid, hp.eps, inv);
    if (cudaGetLastError() != cudaSuccess) return GEFEN_ECUDA;
    // X = U / ||U|| in place, with its transpose when Newton-Schulz follows
    {
        const dim3 tg(static_cast<unsigned>((cols + 31) / 32), static_cast<unsigned>((rows + 31) / 32));
        void* ut = hp.ns_steps > 0 ? Q0 : nullptr;
        if (bf16 && rows % 2 == 0 && cols % 2 == 0)
            k_muon_scale_t2<<<dim3(static_cast<unsigned>((cols + 63) / 64), static_cast<unsigned>((rows + 63) / 64)),
                              256, 0, st>>>(static_cast<__nv_bfloat16*>(P0), static_cast<__nv_bfloat16*>(ut),
                                            static_cast<int>(rows), static_cast<int>(cols), inv, scale, A.snew,
                                            n / period);
        else if (bf16)
            k_muon_scale_t<__nv_bfloat16><<<tg, 256, 0, st>>>(static_cast<__nv_bfloat16*>(P0),
                                                              static_cast<__nv_bfloat16*>(ut), static_cast<int>(rows),
                                                              static_cast<int>(cols), inv, scale, A.snew, n / period);
        else
            k_muon_scale_t<float><<<tg, 256, 0, st>>>(static_cast<float*>(P0), static_cast<float*>(ut),
                                                     static_cast<int>(rows), static_cast<int>(cols), inv, scale,
                                                     A.snew, n / period);
        if (cudaGetLastError() != cudaSuccess) return GEFEN_ECUDA;
    }

    // Newton-Schulz on X (s x n) and T = X^T (n x s): the P buffers hold U's
    // layout (rows x cols), the Q buffers the transposed one
    const bool wide = rows <= cols;
    const int s = static_cast<int>(std::min(rows, cols)), nn = static_cast<int>(std::max(rows, cols));
    const float a = static_cast<float>(hp.ns_a), b = static_cast<float>(hp.ns_b), c = static_cast<float>(hp.ns_c);
    void* U = P0;
    if (hp.ns_steps > 0) {
        void *X = wide ? P0 : Q0, *T = wide ? Q0 : P0, *Xn = wide ? P1 : Q1, *Tn = wide ? Q1 : P1;
        for (int it = 0; it < hp.ns_steps; ++it) {
            cudaError_t e;
            if (bf16) {
                e = gemm_bf16_nt(s, s, nn, 1.0f, X, nn, X, nn, 0.0f, nullptr, 0, GA, s, nullptr, 0, err, st, true);
                if (e == cudaSuccess)
                    e = gemm_bf16_nt(s, s, s, c, GA, s, GA, s, b, GA, s, GB, s, nullptr, 0, err, st, true);
                if (e == cudaSuccess)
                    e = gemm_bf16_nt(s, nn, s, 1.0f, GB, s, T, s, a, X, nn, Xn, nn, Tn, s, err, st);
            } else {
                const float *fx = static_cast<const float*>(X), *ft = static_cast<const float*>(T);
                float *fa = static_cast<float*>(GA), *fb = static_cast<float*>(GB);
                e = gemm_f32_nt(s, s, nn, 1.0f, fx, nn, fx, nn, 0.0f, nullptr, 0, fa, s, nullptr, 0, st);
                if (e == cudaSuccess) e = gemm_f32_nt(s, s, s, c, fa, s, fa, s, b, fa, s, fb, s, nullptr, 0, st);
                if (e == cudaSuccess)
                    e = gemm_f32_nt(s, nn, s, 1.0f, fb, s, ft, s, a, fx, nn, static_cast<float*>(Xn), nn,
                                    static_cast<float*>(Tn), s, st);
            }
            if (e != cudaSuccess) return GEFEN_ECUDA;
            std::swap(X, Xn);
            std::swap(T, Tn);
        }
        U = wide ? X : T;
    }
    const double adj = hp.lr * std::sqrt(std::max(1.0, static_cast<double>(rows) / static_cast<double>(cols)));
    const float decay = static_cast<float>(1.0 - hp.lr * hp.weight_decay);
    if (n % 4 == 0) {
        if (bf16) k_muon_update4<true><<<grid, kMuThreads, 0, st>>>(params, U, n / 4, decay, static_cast<float>(adj));
        else k_muon_update4<false><<<grid, kMuThreads, 0, st>>>(params, U, n / 4, decay, static_cast<float>(adj));
    } else {
        if (bf16) k_muon_update<true><<<grid, kMuThreads, 0, st>>>(params, U, n, decay, static_cast<float>(adj));
        else k_muon_update<false><<<grid, kMuThreads, 0, st>>>(params, U, n, decay, static_cast<float>(adj));
    }
    if (cudaGetLastError() != cudaSuccess) return GEFEN_ECUDA;
    return GEFEN_OK;
}
