// gefen_step: the fused optimizer step of Algorithm 1 (loop body) on sm_103a.
//
// Per block b of p elements (Algorithm 1; Sec. 5.1.1 Quantize):
//   m_i  = beta1 * Cdec[c_i] * s_b + (1 - beta1) * g_i       (decode + momentum)
//   s'_b = max |m_i|,  G_b = mean g_i^2                       (block reductions)
//   v_b  = beta2 v_b + (1 - beta2) G_b                         (shared second moment)
//   theta_i = theta_i (1 - lr wd) - lr/(1-beta1^t) / (sqrt(v_b/(1-beta2^t)) + eps) * m_i
//   c_i  = nearest level of m_i / s'_b in Cenc,  s_b = s'_b    (re-encode)
//
// The step is bound by HBM traffic (12 bytes per parameter: theta read+write,
// bf16 g, u8 code read+write).  Every element's write needs its block's final
// reductions, so the kernels differ by block size:
//   p == 1                 k_step_p1       elementwise, v and s per element
//   p % 16 == 0, p <= 8K   k_step_stream   persistent CTAs stream tiles of
//                                          whole blocks through shared memory
//                                          (bulk copies): one HBM pass
//   p % 16 == 0, p <= 16K  k_step_tile16   one CTA holds whole blocks in
//                                          registers: one HBM pass
//   other p <= 2048        k_step_generic  the same with scalar accesses
//   larger p               k_big_*         chunked: partial reductions, block
//                                          finalise, apply (re-reads g, codes)
#include <algorithm>
#include <cmath>
#include <cstring>
#include <vector>

#include <cuda_bf16.h>

#include "common.cuh"
#include "internal.h"

namespace gefen {

namespace {

constexpr int kThreads = 256;
constexpr int kMaxSegs = 300;
constexpr int kGenericTile = 2048;  // elements per CTA in the generic tile path
constexpr int kChunk = 8192;        // elements per CTA in the big-block path
constexpr int64_t kTile16Max = 16384;

enum Mode { kPlain = 0, kHist = 1, kGradOnly = 2 };

// Storage formats: bit 0 = two 4-bit codes per byte (element i in byte i/2,
// low nibble for even i), bit 1 = bf16 theta.  The arithmetic is fp32 in all.
template <int FMT>
struct Format {
    static constexpr bool kC4 = (FMT & 1) != 0;
    static constexpr bool kTB = (FMT & 2) != 0;
    static constexpr int kThetaBytes = kTB ? 2 : 4;
};

// The four codes of a group of four elements starting at element e (e % 4 == 0).
template <int FMT>
__device__ __forceinline__ uint32_t codes4_at(const unsigned char* base, int64_t e) {
    if (Format<FMT>::kC4) return *reinterpret_cast<const uint16_t*>(base + (e >> 1));
    return *reinterpret_cast<const uint32_t*>(base + e);
}
template <int FMT>
__device__ __forceinline__ uint32_t code_of(uint32_t w, int i) {
    if (Format<FMT>::kC4) return (w >> (4 * i)) & 0xFu;
    return __byte_perm(w, 0u, 0x4440u + i);
}
template <int FMT>
__device__ __forceinline__ uint32_t pack_codes4(const uint32_t (&c)[4]) {
    if (Format<FMT>::kC4) return c[0] | (c[1] << 4) | (c[2] << 8) | (c[3] << 12);
    return __byte_perm(__byte_perm(c[0], c[1], 0x0040u), __byte_perm(c[2], c[3], 0x0040u), 0x5410u);
}
template <int FMT>
__device__ __forceinline__ void store_codes4(uint8_t* codes, int64_t e, uint32_t packed) {
    if (Format<FMT>::kC4)
        __stcs(reinterpret_cast<unsigned short*>(codes + (e >> 1)), static_cast<unsigned short>(packed));
    else
        __stcs(reinterpret_cast<unsigned int*>(codes + e), packed);
}
// Four theta values starting at element e of an fp32 or bf16 array.
template <int FMT>
__device__ __forceinline__ float4 theta4_global(const float* params, int64_t e) {
    if (Format<FMT>::kTB) {
        const uint2 w = __ldcs(reinterpret_cast<const uint2*>(reinterpret_cast<const uint16_t*>(params) + e));
        return make_float4(bf16_lo(w.x), bf16_hi(w.x), bf16_lo(w.y), bf16_hi(w.y));
    }
    return __ldcs(reinterpret_cast<const float4*>(params + e));
}
template <int FMT>
__device__ __forceinline__ float4 theta4_smem(const unsigned char* base, int e) {
    if (Format<FMT>::kTB) {
        const uint2 w = *reinterpret_cast<const uint2*>(base + 2 * e);
        return make_float4(bf16_lo(w.x), bf16_hi(w.x), bf16_lo(w.y), bf16_hi(w.y));
    }
    return *reinterpret_cast<const float4*>(base + 4 * e);
}
__device__ __forceinline__ uint32_t bf16_pair_rn(float lo, float hi) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);  // .x = lo (low half), .y = hi
    return *reinterpret_cast<const uint32_t*>(&v);
}
template <int FMT>
__device__ __forceinline__ void theta4_store(float* params, int64_t e, float4 t) {
    if (Format<FMT>::kTB)
        __stcs(reinterpret_cast<uint2*>(reinterpret_cast<uint16_t*>(params) + e),
               make_uint2(bf16_pair_rn(t.x, t.y), bf16_pair_rn(t.z, t.w)));
    else
        __stcs(reinterpret_cast<float4*>(params + e), t);
}

struct Seg {
    int64_t elem_off;
    int64_t numel;
    int64_t period;
    int64_t block_off;
    int64_t unit_begin;  // first work unit (CTA) of this tensor in the launch
    int64_t per_unit;    // tile paths: blocks per tile; big path: chunks per block
    int64_t aux_begin;   // big path: first big-block index of this tensor
    int64_t nblocks;     // numel / period
    uint32_t pmagic;     // floor(2^32 / period) + 1: e / p == umulhi(e, pmagic) for e * p < 2^32
    uint32_t flags;  // kSegBigTiles: tiles of big blocks whose factors come from blk_state
};

constexpr uint32_t kSegBigTiles = 1u;

inline void seg_fill(Seg& s, const gefen_tensor_t& x) {
    s.elem_off = x.offset;
    s.numel = x.numel;
    s.period = x.period;
    s.block_off = x.block_offset;
    s.nblocks = x.numel / x.period;
    s.pmagic = static_cast<uint32_t>((uint64_t(1) << 32) / static_cast<uint64_t>(x.period)) + 1u;
    s.flags = 0;
}

struct HP {
    float beta1, omb1;  // beta1, 1 - beta1
    float beta2, omb2;  // beta2, 1 - beta2
    float inv_bc2;      // 1 / (1 - beta2^t)
    float lr_bc1;       // lr / (1 - beta1^t)
    float eps;
    float decay;        // 1 - lr * weight_decay
};

struct Launch {
    int32_t nseg;
    int64_t nunits;
    HP hp;
    Seg seg[kMaxSegs];
};

struct Ptrs {
    float* params;
    const uint16_t* grads;
    uint8_t* codes;
    float* v;
    float* scale;
    const float* cb_dec;
    const float* cb_enc;
    int k;
    float* xstage;      // histogram input staging (HIST modes, kernels that do not count in place)
    uint64_t* hist;     // the histogram (HIST modes)
    int bins;
    double* part_g2;    // big path: per-chunk sum of g^2
    float* part_mx;     // big path: per-chunk max
    float4* blk_state;  // big path: per big block (s_old, s_new, fac, -)
};

__device__ __forceinline__ int find_seg(const Launch& L, int64_t unit) {
    int lo = 0, hi = L.nseg - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (L.seg[mid].unit_begin <= unit) lo = mid; else hi = mid - 1;
    }
    return lo;
}

__device__ __forceinline__ int find_seg_aux(const Launch& L, int64_t idx) {
    int lo = 0, hi = L.nseg - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (L.seg[mid].aux_begin <= idx) lo = mid; else hi = mid - 1;
    }
    return lo;
}

// Decode table (Cdec) and sorted midpoints of Cenc in shared memory; returns
// the code of the level nearest 0 (ties to the lower index).
__device__ __forceinline__ void load_codebooks(const Ptrs& P, float* s_dec, float* s_mid) {
    const int t = threadIdx.x;
    if (t < kMaxLevels) {
        s_dec[t] = t < P.k ? P.cb_dec[t] : 0.0f;
        s_mid[t] = (t < P.k - 1) ? 0.5f * (P.cb_enc[t] + P.cb_enc[t + 1]) : INFINITY;
    }
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}
__device__ __forceinline__ double warp_sum_d(double x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}
__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
    return x;
}

// Shared-v update and the per-block step factor lr/(1-beta1^t)/(sqrt(vhat)+eps).
__device__ __forceinline__ float block_update(const HP& hp, float* v, int64_t bi, float G) {
    const float vn = fmaf(hp.beta2, v[bi], hp.omb2 * G);
    v[bi] = vn;
    return hp.lr_bc1 / (sqrtf(vn * hp.inv_bc2) + hp.eps);
}

__device__ __forceinline__ void unpack16_bf16(uint4 a, uint4 b, float* g) {
    const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        g[2 * i] = bf16_lo(w[i]);
        g[2 * i + 1] = bf16_hi(w[i]);
    }
}

__device__ __forceinline__ uint32_t byte_of(uint4 c, int i) {
    const uint32_t w = (i < 4) ? c.x : (i < 8) ? c.y : (i < 12) ? c.z : c.w;
    return (w >> (8 * (i & 3))) & 0xFFu;
}

// ------------------------------------------------------------------ p == 1
// Every element is its own block: v and s are per element, x = m/|m| = +-1,
// so its level is one of two, found once per CTA (an infinite m gives x = NaN
// and level 0, m = 0 the level of 0).  With two codes per byte a thread owns
// both elements of a byte (a pair); the nibble of an element past the
// tensor's end is left as it was.  fp32 theta and 8-bit codes whose blocks
// start on a multiple of four take four elements per thread with 16-byte
// accesses.
template <int MODE, int FMT>
__global__ void __launch_bounds__(kThreads) k_step_p1(const __grid_constant__ Launch L, const Ptrs P) {
    constexpr int EPC = Format<FMT>::kC4 ? 2 : 1;  // elements per thread and step
    __shared__ float s_dec[kMaxLevels], s_mid[kMaxLevels];
    if (MODE != kGradOnly) load_codebooks(P, s_dec, s_mid);
    __syncthreads();
    const int64_t unit = blockIdx.x;
    const Seg& S = L.seg[find_seg(L, unit)];
    const int64_t base = (unit - S.unit_begin) * (4 * kThreads * EPC);
    const HP& hp = L.hp;
    const int zero_code = (MODE != kGradOnly) ? level_search(s_mid, 0.0f) : 0;
    const int cpos = (MODE != kGradOnly) ? level_search(s_mid, 1.0f) : 0;
    const int cneg = (MODE != kGradOnly) ? level_search(s_mid, -1.0f) : 0;
    // the level of m (and x = m / |m| for the histogram)
    auto level = [&](float m, float am, float& x) -> int {
        if (am > 0.0f) {
            x = __fdiv_rn(m, am);
            return isinf(m) ? 0 : (m > 0.0f ? cpos : cneg);
        }
        x = __int_as_float(0x7fffffff);
        return zero_code;
    };
    if (FMT == 0 && MODE != kGradOnly && ((S.block_off & 3) | (S.elem_off & 3)) == 0 &&
        ((reinterpret_cast<uintptr_t>(P.v) | reinterpret_cast<uintptr_t>(P.scale)) & 15u) == 0) {
        const int64_t le = base + 4 * static_cast<int64_t>(threadIdx.x);
        if (le + 4 <= S.numel) {
            const int64_t e = S.elem_off + le, bi = S.block_off + le;
            const uint2 gw = __ldcs(reinterpret_cast<const uint2*>(P.grads + e));
            const uint32_t cw = __ldcs(reinterpret_cast<const unsigned int*>(P.codes + e));
            const float4 sc = *reinterpret_cast<const float4*>(P.scale + bi);
            const float4 vv = *reinterpret_cast<const float4*>(P.v + bi);
            const float4 tt = __ldcs(reinterpret_cast<const float4*>(P.params + e));
            const float g[4] = {bf16_lo(gw.x), bf16_hi(gw.x), bf16_lo(gw.y), bf16_hi(gw.y)};
            const float s4[4] = {sc.x, sc.y, sc.z, sc.w}, v4[4] = {vv.x, vv.y, vv.z, vv.w};
            const float t4[4] = {tt.x, tt.y, tt.z, tt.w};
            float mo[4], vo[4], to[4], xo[4];
            uint32_t co = 0u;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float m = fmaf(hp.omb1, g[q], hp.beta1 * s4[q] * s_dec[(cw >> (8 * q)) & 0xFFu]);
                const float vn = fmaf(hp.beta2, v4[q], hp.omb2 * (g[q] * g[q]));
                const float fac = hp.lr_bc1 / (sqrtf(vn * hp.inv_bc2) + hp.eps);
                mo[q] = fabsf(m);
                vo[q] = vn;
                to[q] = fmaf(-fac, m, hp.decay * t4[q]);
                co |= static_cast<uint32_t>(level(m, mo[q], xo[q])) << (8 * q);
            }
            *reinterpret_cast<float4*>(P.v + bi) = make_float4(vo[0], vo[1], vo[2], vo[3]);
            *reinterpret_cast<float4*>(P.scale + bi) = make_float4(mo[0], mo[1], mo[2], mo[3]);
            __stcs(reinterpret_cast<float4*>(P.params + e), make_float4(to[0], to[1], to[2], to[3]));
            __stcs(reinterpret_cast<unsigned int*>(P.codes + e), co);
            if (MODE == kHist) __stcs(reinterpret_cast<float4*>(P.xstage + e), make_float4(xo[0], xo[1], xo[2], xo[3]));
            return;
        }
        if (le >= S.numel) return;
        // the tensor's last one to three elements: the scalar form below, by this thread
    }
    const bool vec = FMT == 0 && MODE != kGradOnly && ((S.block_off & 3) | (S.elem_off & 3)) == 0 &&
                     ((reinterpret_cast<uintptr_t>(P.v) | reinterpret_cast<uintptr_t>(P.scale)) & 15u) == 0;
    uint16_t* th16 = reinterpret_cast<uint16_t*>(P.params);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t c0 = vec ? base + 4 * static_cast<int64_t>(threadIdx.x) + i
                               : base + (threadIdx.x + i * kThreads) * static_cast<int64_t>(EPC);
        if (c0 >= S.numel) break;
        uint32_t cbyte = 0u;
        if (MODE != kGradOnly && Format<FMT>::kC4) cbyte = P.codes[(S.elem_off + c0) >> 1];
#pragma unroll
        for (int q = 0; q < EPC; ++q) {
            const int64_t le = c0 + q;
            if (le >= S.numel) break;
            const int64_t e = S.elem_off + le;
            const int64_t bi = S.block_off + le;
            const float g = bf16_bits_to_f32(__ldcs(P.grads + e));
            if (MODE == kGradOnly) {
                P.xstage[e] = g != 0.0f ? __fdiv_rn(g, fabsf(g)) : __int_as_float(0x7fffffff);
                continue;
            }
            const uint32_t cold = Format<FMT>::kC4 ? ((cbyte >> (4 * q)) & 0xFu) : __ldcs(P.codes + e);
            const float m = fmaf(hp.omb1, g, hp.beta1 * P.scale[bi] * s_dec[cold]);
            const float fac = block_update(hp, P.v, bi, g * g);
            const float am = fabsf(m);
            P.scale[bi] = am;
            const float th = Format<FMT>::kTB ? bf16_bits_to_f32(__ldcs(th16 + e)) : __ldcs(P.params + e);
            const float tn = fmaf(-fac, m, hp.decay * th);
            if (Format<FMT>::kTB)
                __stcs(th16 + e, __bfloat16_as_ushort(__float2bfloat16_rn(tn)));
            else
                __stcs(P.params + e, tn);
            float x;
            const int c = level(m, am, x);
            if (Format<FMT>::kC4)
                cbyte = (cbyte & ~(0xFu << (4 * q))) | (static_cast<uint32_t>(c) << (4 * q));
            else
                P.codes[e] = static_cast<uint8_t>(c);
            if (MODE == kHist) P.xstage[e] = x;
        }
        if (MODE != kGradOnly && Format<FMT>::kC4) P.codes[(S.elem_off + c0) >> 1] = static_cast<uint8_t>(cbyte);
    }
}

// -------------------------------------------------- p % 16 == 0, p <= 16K
// One CTA processes a tile of whole blocks (<= kThreads*V*16 elements); each
// thread owns V vectors of 16 elements (16-byte loads of codes, 2 x 16 bytes
// of bf16 grads, 4 x 16 bytes of fp32 params).  Phase 1 decodes m into
// registers and writes per-vector partials; the block reductions run in shared
// memory; phase 2 updates theta (prefetched into L2 by one bulk prefetch at the
// start) and re-encodes.  One HBM pass: 12 bytes per parameter.
template <int V, int MODE>
__global__ void __launch_bounds__(kThreads) k_step_tile16(const __grid_constant__ Launch L, const Ptrs P) {
    __shared__ float s_dec[kMaxLevels], s_mid[kMaxLevels];
    __shared__ float2 s_part[kThreads * V];
    __shared__ float2 s_blk[kThreads * V];
    const int tid = threadIdx.x;
    const int64_t unit = blockIdx.x;
    const Seg& S = L.seg[find_seg(L, unit)];
    const HP& hp = L.hp;
    const int64_t p = S.period;
    const int64_t blk0 = (unit - S.unit_begin) * S.per_unit;
    const int nblk = static_cast<int>(min(S.per_unit, S.nblocks - blk0));
    const int64_t e0 = S.elem_off + blk0 * p;
    const int q = static_cast<int>(p >> 4);  // vectors per block
    const int nvec = nblk * q;
    const int64_t bo = S.block_off + blk0;

    if (MODE != kGradOnly) {
        load_codebooks(P, s_dec, s_mid);
        if (tid == 0) {
            const uint32_t bytes = static_cast<uint32_t>(nvec) * 64u;
            asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(P.params + e0), "r"(bytes)
                         : "memory");
        }
    }
    __syncthreads();

    float m[V][16];
#pragma unroll
    for (int i = 0; i < V; ++i) {
        const int j = tid + i * kThreads;
        float g2 = 0.0f, mx = 0.0f;
        if (j < nvec) {
            const int64_t e = e0 + static_cast<int64_t>(j) * 16;
            const uint4 ga = __ldcs(reinterpret_cast<const uint4*>(P.grads + e));
            const uint4 gb = __ldcs(reinterpret_cast<const uint4*>(P.grads + e) + 1);
            float g[16];
            unpack16_bf16(ga, gb, g);
            if (MODE == kGradOnly) {
#pragma unroll
                for (int t = 0; t < 16; ++t) {
                    m[i][t] = g[t];
                    mx = fmaxf(mx, fabsf(g[t]));
                }
            } else {
                const uint4 cw = __ldcs(reinterpret_cast<const uint4*>(P.codes + e));
                const float b1s = hp.beta1 * P.scale[bo + j / q];
#pragma unroll
                for (int t = 0; t < 16; ++t) {
                    const float mm = fmaf(hp.omb1, g[t], b1s * s_dec[byte_of(cw, t)]);
                    m[i][t] = mm;
                    g2 = fmaf(g[t], g[t], g2);
                    mx = fmaxf(mx, fabsf(mm));
                }
            }
        }
        s_part[j] = make_float2(g2, mx);
    }
    __syncthreads();

    // Block reductions over the per-vector partials (fixed order).
    const float pf = static_cast<float>(p);
    if (q <= 8) {
        for (int b = tid; b < nblk; b += kThreads) {
            float g2 = 0.0f, mx = 0.0f;
            for (int t = 0; t < q; ++t) {
                const float2 pp = s_part[b * q + t];
                g2 += pp.x;
                mx = fmaxf(mx, pp.y);
            }
            float fac = 0.0f;
            if (MODE != kGradOnly) {
                fac = block_update(hp, P.v, bo + b, g2 / pf);
                P.scale[bo + b] = mx;
            }
            s_blk[b] = make_float2(fac, mx);
        }
    } else {
        const int warp = tid >> 5, lane = tid & 31;
        for (int b = warp; b < nblk; b += kThreads / 32) {
            float g2 = 0.0f, mx = 0.0f;
            for (int t = lane; t < q; t += 32) {
                const float2 pp = s_part[b * q + t];
                g2 += pp.x;
                mx = fmaxf(mx, pp.y);
            }
            g2 = warp_sum(g2);
            mx = warp_max(mx);
            if (lane == 0) {
                float fac = 0.0f;
                if (MODE != kGradOnly) {
                    fac = block_update(hp, P.v, bo + b, g2 / pf);
                    P.scale[bo + b] = mx;
                }
                s_blk[b] = make_float2(fac, mx);
            }
        }
    }
    __syncthreads();

    if (MODE == kGradOnly) {
#pragma unroll
        for (int i = 0; i < V; ++i) {
            const int j = tid + i * kThreads;
            if (j >= nvec) continue;
            const int64_t e = e0 + static_cast<int64_t>(j) * 16;
            const float a = s_blk[j / q].y;
            float x[16];
#pragma unroll
            for (int t = 0; t < 16; ++t) x[t] = a > 0.0f ? __fdiv_rn(m[i][t], a) : __int_as_float(0x7fffffff);
            float4* xs = reinterpret_cast<float4*>(P.xstage + e);
#pragma unroll
            for (int t = 0; t < 4; ++t) __stcs(xs + t, make_float4(x[4 * t], x[4 * t + 1], x[4 * t + 2], x[4 * t + 3]));
        }
        return;
    }

    const int zero_code = level_search(s_mid, 0.0f);
    float4 th[V][4];
#pragma unroll
    for (int i = 0; i < V; ++i) {
        const int j = tid + i * kThreads;
        if (j < nvec) {
            const float4* src = reinterpret_cast<const float4*>(P.params + e0 + static_cast<int64_t>(j) * 16);
#pragma unroll
            for (int t = 0; t < 4; ++t) th[i][t] = __ldcg(src + t);
        }
    }
#pragma unroll
    for (int i = 0; i < V; ++i) {
        const int j = tid + i * kThreads;
        if (j >= nvec) continue;
        const int64_t e = e0 + static_cast<int64_t>(j) * 16;
        const float2 bs = s_blk[j / q];
        const float fac = bs.x, sn = bs.y;
        float* thf = reinterpret_cast<float*>(th[i]);
#pragma unroll
        for (int t = 0; t < 16; ++t) thf[t] = fmaf(-fac, m[i][t], hp.decay * thf[t]);
        float4* dst = reinterpret_cast<float4*>(P.params + e);
#pragma unroll
        for (int t = 0; t < 4; ++t) __stcs(dst + t, th[i][t]);
        uint32_t w[4] = {0u, 0u, 0u, 0u};
        float x[16];
#pragma unroll
        for (int t = 0; t < 16; ++t) {
            int c;
            if (sn > 0.0f) {
                x[t] = __fdiv_rn(m[i][t], sn);
                c = level_search(s_mid, x[t]);
            } else {
                x[t] = __int_as_float(0x7fffffff);
                c = zero_code;
            }
            w[t >> 2] |= static_cast<uint32_t>(c) << (8 * (t & 3));
        }
        __stcs(reinterpret_cast<uint4*>(P.codes + e), make_uint4(w[0], w[1], w[2], w[3]));
        if (MODE == kHist) {
            float4* xs = reinterpret_cast<float4*>(P.xstage + e);
#pragma unroll
            for (int t = 0; t < 4; ++t) __stcs(xs + t, make_float4(x[4 * t], x[4 * t + 1], x[4 * t + 2], x[4 * t + 3]));
        }
    }
}

// ------------------------------------------------ streamed tiles (bulk copy)
// Persistent CTAs stream tiles of whole blocks (p % 16 == 0, p <= TILE).
// Thread 0 keeps STAGES tiles of g and codes in flight through a ring of
// shared-memory stages (cp.async.bulk, completion on an mbarrier) and asks L2
// to prefetch the same tiles' theta.  A warp owns 512 consecutive elements of
// a tile; lane l owns the four groups of four at 128 j + 4 l (j < 4), so every
// warp-wide access of theta, g, codes or x is one contiguous run.
// Theta is read straight from global memory (an L2 hit) and theta' and the
// new codes are stored straight from registers, so a stage is free again as
// soon as its tile is decoded.
//
// Decoding reads a shared table; encoding maps x = m / s' to its cell of a
// uniform grid over [-1, 1] whose record holds the number of midpoints below
// the cell and the next three midpoints, so the nearest level is base + three
// compares (identical to the binary search, which remains the fallback when a
// cell holds more than three midpoints).  Both tables are replicated (LUTR,
// DECR copies, lane l reading copy l % R) so the gathers of one warp spread
// over more shared-memory banks.

struct TileInfo {
    int64_t e0;    // first element
    int64_t bo;    // first block index into v / scale (big-block tiles: index into blk_state)
    int nelem;
    int nblk;
    int p;
    uint32_t pmagic;  // floor(2^32 / p) + 1: e / p == umulhi(e, pmagic) for e, p < 2^16
    int ext;          // a tile of a big block: its factors were finalised beforehand
    float rp;         // 1 / p (fp32, round to nearest), computed by the issuing thread
};

template <int LUTR, int DECR>
struct alignas(16) StreamTables {
    float4 lut[(kLutCells + 2) * LUTR];  // copy r of record c+1 (cell c in [-1, kLutCells]) at (c+1) LUTR + r
    float dec[kMaxLevels * DECR];        // copy r of level c at c DECR + r
    float mid[kMaxLevels + 4];
};

// Stage layout: [theta (THS only) | g bf16 | codes].
template <int TILE, bool THS, int FMT>
struct StageLayout {
    static constexpr int kG = THS ? Format<FMT>::kThetaBytes * TILE : 0;
    static constexpr int kC = kG + 2 * TILE;
    static constexpr int kBytes = kC + (Format<FMT>::kC4 ? TILE / 2 : TILE);
};

template <int TILE, int THREADS, int STAGES, int LUTR, int DECR, bool THS, int HB, int FMT>
struct alignas(128) StreamSmem {
    static constexpr int kHistCells = HB;  // cells counted in shared memory (0: x is staged instead)
    unsigned char stage[STAGES][StageLayout<TILE, THS, FMT>::kBytes];
    uint32_t hist[HB > 0 ? HB : 1];
    StreamTables<LUTR, DECR> tab;
    float2 part[THREADS / 32];  // per warp: (sum g^2, max |m|)
    float2 blk[TILE / 16];      // per block, irregular shapes: (step factor, 1/s')  [grad-only: (-, absmax)]
    TileInfo tile[STAGES];      // the tile each stage holds, written by the issuing thread
    TileInfo next;              // the issuing thread's next descriptor, prepared during a tile
    unsigned long long bar[STAGES];
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
// Waits for the barrier phase with the given parity; gives up after ~2^31
// cycles (about a second) and returns false, so a lost copy cannot hang the GPU.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
    const long long t0 = clock64();
    while (true) {
        uint32_t ok;
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(ok)
            : "r"(bar), "r"(parity)
            : "memory");
        if (ok) return true;
        if (clock64() - t0 > (1ll << 31)) return false;
    }
}
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}
__device__ __forceinline__ void prefetch_l2(const void* src, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

// Decode table, midpoints (padded with +inf) and the cell records.
template <int THREADS, int LUTR, int DECR>
__device__ __forceinline__ int build_tables(const Ptrs& P, StreamTables<LUTR, DECR>& T, bool grad_only) {
    const int t = threadIdx.x;
    if (grad_only) return 0;
    for (int i = t; i < kMaxLevels * DECR; i += THREADS) {
        const int c = i / DECR;
        T.dec[i] = c < P.k ? P.cb_dec[c] : 0.0f;
    }
    for (int i = t; i < kMaxLevels + 4; i += THREADS)
        T.mid[i] = (i < P.k - 1) ? 0.5f * (P.cb_enc[i] + P.cb_enc[i + 1]) : INFINITY;
    __syncthreads();
    return build_cell_records<LUTR>(T.mid, T.lut, t, THREADS);
}

// The issuing thread walks the segment table forward: a CTA's tiles come in
// increasing unit order, so its segment cursor only grows.
__device__ __forceinline__ TileInfo tile_info(const Launch& L, int64_t unit, int& seg) {
    while (seg + 1 < L.nseg && L.seg[seg + 1].unit_begin <= unit) ++seg;
    const Seg& S = L.seg[seg];
    const int64_t p = S.period;
    TileInfo ti;
    ti.rp = 0.0f;
    if (S.flags & kSegBigTiles) {
        // per_unit tiles per block, each p / per_unit consecutive elements
        const int64_t local = unit - S.unit_begin;
        const int64_t tsz = p / S.per_unit;
        ti.ext = 1;
        ti.nblk = 1;
        ti.p = static_cast<int>(min(p, static_cast<int64_t>(1) << 30));
        ti.nelem = static_cast<int>(tsz);
        ti.e0 = S.elem_off + local * tsz;
        ti.bo = S.aux_begin + local / S.per_unit;
        ti.pmagic = 0u;
        return ti;
    }
    ti.ext = 0;
    const int64_t blk0 = (unit - S.unit_begin) * S.per_unit;
    ti.nblk = static_cast<int>(min(S.per_unit, S.nblocks - blk0));
    ti.p = static_cast<int>(p);
    ti.nelem = ti.nblk * ti.p;
    ti.e0 = S.elem_off + blk0 * p;
    ti.bo = S.block_off + blk0;
    ti.pmagic = S.pmagic;
    ti.rp = __frcp_rn(static_cast<float>(p));
    return ti;
}

// A tile fits its stage iff it holds at most TILE elements, a multiple of 16
// (so every copy is a whole number of 16-byte units).
template <int TILE>
__device__ __forceinline__ bool tile_fits(const TileInfo& ti) {
    return ti.nelem > 0 && ti.nelem <= TILE && (ti.nelem & 15) == 0;
}

// Publishes the tile's descriptor in its stage and starts its copies.
template <int TILE, int MODE, bool THS, int FMT, typename Smem>
__device__ __forceinline__ void issue_tile(Smem& sm, int s, const TileInfo& ti, const Ptrs& P) {
    using SL = StageLayout<TILE, THS, FMT>;
    constexpr uint32_t TB = Format<FMT>::kThetaBytes;
    sm.tile[s] = ti;
    if (!tile_fits<TILE>(ti)) return;  // never copied; the consumer stops before waiting on it
    const uint32_t n = static_cast<uint32_t>(ti.nelem);
    const uint32_t bar = smem_u32(&sm.bar[s]);
    unsigned char* st = sm.stage[s];
    if (MODE == kGradOnly) {
        mbar_expect_tx(bar, 2u * n);
        bulk_g2s(smem_u32(st + SL::kG), P.grads + ti.e0, 2u * n, bar);
    } else {
        // codes: n bytes, or n/2 with two per byte (tiles start and end on
        // multiples of 32 elements then, so every copy is whole 16-byte units)
        const uint32_t cn = Format<FMT>::kC4 ? n / 2 : n;
        const unsigned char* cs = P.codes + (Format<FMT>::kC4 ? ti.e0 / 2 : ti.e0);
        const unsigned char* ts = reinterpret_cast<const unsigned char*>(P.params) + TB * ti.e0;
        mbar_expect_tx(bar, (THS ? TB * n : 0u) + 2u * n + cn);
        if (THS) bulk_g2s(smem_u32(st), ts, TB * n, bar);
        bulk_g2s(smem_u32(st + SL::kG), P.grads + ti.e0, 2u * n, bar);
        bulk_g2s(smem_u32(st + SL::kC), cs, cn, bar);
        if (!THS) prefetch_l2(ts, TB * n);
    }
}

// Block state (s and v before the step) of the blocks of the thread's NG
// groups, whose first elements are eb + 128 j.
template <int NG>
__device__ __forceinline__ void load_state(const Ptrs& P, const TileInfo& ti, int eb, float (&s)[NG], float (&v)[NG]) {
    if (ti.ext) {  // a big block: s before the step was kept by its finalisation
        const float s0 = P.blk_state[ti.bo].x;
#pragma unroll
        for (int j = 0; j < NG; ++j) { s[j] = s0; v[j] = 0.0f; }
        return;
    }
    if (ti.p > 65535) return;              // only a tile that does not fit; never processed
    if (ti.p % (128 * NG) == 0) {          // one block per warp slice
        if (eb < ti.nelem) {
            const int64_t bi = ti.bo + __umulhi(static_cast<uint32_t>(eb), ti.pmagic);
            const float s0 = P.scale[bi], v0 = P.v[bi];
#pragma unroll
            for (int j = 0; j < NG; ++j) { s[j] = s0; v[j] = v0; }
        }
        return;
    }
#pragma unroll
    for (int j = 0; j < NG; ++j) {
        const int e = eb + 128 * j;
        if (e < ti.nelem) {
            const int64_t bi = ti.bo + __umulhi(static_cast<uint32_t>(e), ti.pmagic);
            s[j] = P.scale[bi];
            v[j] = P.v[bi];
        }
    }
}

__device__ __forceinline__ void butterfly(float& s2, float& mx, int lanes) {
    for (int o = lanes >> 1; o > 0; o >>= 1) {
        s2 += __shfl_xor_sync(0xffffffffu, s2, o);
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    }
}

// Warp maxima and sums for block reductions.  A maximum of magnitudes (>= 0,
// never NaN: fmaxf drops NaN) is one integer max over the float bits, which
// order like the values; a sum is a five-level butterfly.
__device__ __forceinline__ float warp_max_nonneg(float x) {
    return __uint_as_float(__reduce_max_sync(0xffffffffu, __float_as_uint(x)));
}
__device__ __forceinline__ float warp_sum_bfly(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}
// Hardware approximations (about 1 ulp): the step factor and the scale's
// reciprocal feed the parameter update and the nearest-level decision, both
// far inside the 1e-5 parameter and 1e-6 decision-margin tolerances.
__device__ __forceinline__ float rcp_approx(float x) {
    float r;
    asm("rcp.approx.f32 %0, %1;" : "=f"(r) : "f"(x));
    return r;
}
__device__ __forceinline__ float sqrt_approx(float x) {
    float r;
    asm("sqrt.approx.f32 %0, %1;" : "=f"(r) : "f"(x));
    return r;
}

// 0xFFFFFFFF if a < b else 0 (one compare that yields an integer mask)

// Nearest levels of four values, packed as four code bytes.  With the cell
// records (LUT): |x| <= 1 up to rounding (x = m / max|m|, or 0 for a zero
// block), so the record index floor(256 x + 257) lies in [0, 513].  The floor
// is one round-down fma against 1.5 * 2^23, where the float grid is the
// integers: y = floor(256 x + 257) + 1.5 * 2^23 exactly, and the index is the
// bit pattern of y minus that of 1.5 * 2^23.  The unsigned clamp keeps a NaN
// or a corrupted value inside the table.
template <bool LUT, int LUTR, int DECR>
__device__ __forceinline__ void encode4(const StreamTables<LUTR, DECR>& T, int copy, const float (&x)[4],
                                        uint32_t (&c)[4]) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        if (LUT) {
            c[i] = lut_encode<LUTR>(T.lut, copy, x[i]);
        } else {
            c[i] = static_cast<uint32_t>(level_search(T.mid, x[i]));
        }
    }
}

// One tile of the streamed step.  FULL: every group of the tile is live (the
// tile holds TILE elements), so no group needs a bounds predicate.
template <int TILE, int THREADS, int LUTR, int DECR, int MODE, bool THS, int FMT, bool LUT, bool FULL, typename Smem>
__device__ __forceinline__ void stream_tile(Smem& sm, const Ptrs& P, const HP& hp, const TileInfo& ti,
                                            unsigned char* st, int eb, const float (&r_s)[4], const float (&r_v)[4],
                                            const float4 (&th)[4]) {
    using SL = StageLayout<TILE, THS, FMT>;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int lut_copy = lane % LUTR, dec_copy = lane % DECR;
    const int p = ti.p;
    const float rp = ti.rp;
    bool live[4];
    int blk[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const int e = eb + 128 * j;
        live[j] = FULL || e < ti.nelem;
        blk[j] = static_cast<int>(__umulhi(static_cast<uint32_t>(e), ti.pmagic));
    }
    const int64_t ge0 = ti.e0 + eb;  // element of group 0; group j at + 128 j

    // phase 1: decode m, partials per group of four
    float m[16], g2[4], mx[4];
    const float* dec = sm.tab.dec + dec_copy;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        g2[j] = 0.0f;
        mx[j] = 0.0f;
        const int e = eb + 128 * j;
        const uint2 gw = live[j] ? *reinterpret_cast<const uint2*>(st + SL::kG + 2 * e) : make_uint2(0u, 0u);
        const float g[4] = {bf16_lo(gw.x), bf16_hi(gw.x), bf16_lo(gw.y), bf16_hi(gw.y)};
        if (MODE == kGradOnly) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                m[4 * j + i] = g[i];
                mx[j] = fmaxf(mx[j], fabsf(g[i]));
            }
        } else {
            const uint32_t cw = live[j] ? codes4_at<FMT>(st + SL::kC, e) : 0u;
            const float b1s = hp.beta1 * r_s[j];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const uint32_t c = code_of<FMT>(cw, i);
                const float mm = fmaf(hp.omb1, g[i], b1s * dec[c * DECR]);
                m[4 * j + i] = mm;
                g2[j] = fmaf(g[i], g[i], g2[j]);
                mx[j] = fmaxf(mx[j], fabsf(mm));
            }
        }
    }

    // block reductions: every lane holding a block ends with the same sums
    // (butterflies are exact under commutation; lists of partials are summed
    // in one fixed order), so each derives the block's factors
    float fac[4], inv[4];  // grad-only: inv = max |g|
    auto finish = [&](float s2, float sx, float v_old, int64_t bi, bool writer, float& f, float& iv) {
        if (MODE == kGradOnly) {
            iv = sx;
            f = 0.0f;
        } else {
            const float vn = fmaf(hp.beta2, v_old, hp.omb2 * (s2 * rp));
            f = hp.lr_bc1 * rcp_approx(sqrt_approx(vn * hp.inv_bc2) + hp.eps);
            iv = sx > 0.0f ? rcp_approx(sx) : 0.0f;
            if (writer) {
                P.v[bi] = vn;
                P.scale[bi] = sx;
            }
        }
    };
    if (ti.ext) {
        // a tile of a big block: v, s and the step factor were finalised
        const float4 bs = P.blk_state[ti.bo];  // (s before, s after, step factor, -)
        const float iv = (MODE == kGradOnly) ? bs.y : (bs.y > 0.0f ? __frcp_rn(bs.y) : 0.0f);
#pragma unroll
        for (int j = 0; j < 4; ++j) { fac[j] = bs.z; inv[j] = iv; }
    } else if ((p & 511) == 0) {
        // a warp's 512 elements lie in one block
        float s2 = warp_sum_bfly((g2[0] + g2[1]) + (g2[2] + g2[3]));
        float sx = warp_max_nonneg(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])));
        const int nw = p >> 9;  // warps per block
        const int w0 = blk[0] * nw;  // the block's first warp (its blocks are whole warps)
        if (nw > 1) {
            if (lane == 0) sm.part[warp] = make_float2(s2, sx);
            __syncthreads();
            s2 = 0.0f;
            sx = 0.0f;
#pragma unroll
            for (int t = 0; t < THREADS / 32; ++t) {
                if (t < nw && w0 + t < THREADS / 32) {  // idle warps of a partial tile stay in range
                    const float2 pp = sm.part[w0 + t];
                    s2 += pp.x;
                    sx = fmaxf(sx, pp.y);
                }
            }
        }
        finish(s2, sx, r_v[0], ti.bo + blk[0], live[0] && lane == 0 && warp == w0, fac[0], inv[0]);
#pragma unroll
        for (int j = 1; j < 4; ++j) { fac[j] = fac[0]; inv[j] = inv[0]; }
    } else if (p == 256) {
        // groups 0,1 and 2,3 form one block each
        const float s0 = warp_sum_bfly(g2[0] + g2[1]), x0 = warp_max_nonneg(fmaxf(mx[0], mx[1]));
        const float s1 = warp_sum_bfly(g2[2] + g2[3]), x1 = warp_max_nonneg(fmaxf(mx[2], mx[3]));
        finish(s0, x0, r_v[0], ti.bo + blk[0], live[0] && lane == 0, fac[0], inv[0]);
        finish(s1, x1, r_v[2], ti.bo + blk[2], live[2] && lane == 0, fac[2], inv[2]);
        fac[1] = fac[0]; inv[1] = inv[0];
        fac[3] = fac[2]; inv[3] = inv[2];
    } else if ((p & (p - 1)) == 0) {
        // p in {16, 32, 64, 128}: a block spans p/4 lanes of one group.
        // Reduce-scatter over the four groups: the two halves of a span swap
        // the sums of two groups (each keeps a pair), the quarters swap one
        // more, and a butterfly over the remaining lanes completes the one
        // group a lane keeps -- the pairs combine as in a butterfly per group,
        // so the sums are the same.  The lane derives that block's factors
        // once; each lane then gathers its four groups' factors.
        const int lanes = p >> 2, oa = lanes >> 1, ob = lanes >> 2;
        const bool hi = (lane & oa) != 0, lo = (lane & ob) != 0;
        float k0 = hi ? g2[2] : g2[0], k1 = hi ? g2[3] : g2[1];
        float q0 = hi ? mx[2] : mx[0], q1 = hi ? mx[3] : mx[1];
        k0 += __shfl_xor_sync(0xffffffffu, hi ? g2[0] : g2[2], oa);
        k1 += __shfl_xor_sync(0xffffffffu, hi ? g2[1] : g2[3], oa);
        q0 = fmaxf(q0, __shfl_xor_sync(0xffffffffu, hi ? mx[0] : mx[2], oa));
        q1 = fmaxf(q1, __shfl_xor_sync(0xffffffffu, hi ? mx[1] : mx[3], oa));
        float s2 = (lo ? k1 : k0) + __shfl_xor_sync(0xffffffffu, lo ? k0 : k1, ob);
        float sx = fmaxf(lo ? q1 : q0, __shfl_xor_sync(0xffffffffu, lo ? q0 : q1, ob));
        butterfly(s2, sx, ob);
        const int g = (hi ? 2 : 0) + (lo ? 1 : 0);  // the group this lane completed
        const float vg = g == 0 ? r_v[0] : g == 1 ? r_v[1] : g == 2 ? r_v[2] : r_v[3];
        const int bg = g == 0 ? blk[0] : g == 1 ? blk[1] : g == 2 ? blk[2] : blk[3];
        const bool lg = g == 0 ? live[0] : g == 1 ? live[1] : g == 2 ? live[2] : live[3];
        float f, iv;
        finish(s2, sx, vg, ti.bo + bg, lg && (lane & (ob - 1)) == 0, f, iv);
        const int base = lane & ~(oa | ob);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int src = base | ((j & 2) ? oa : 0) | ((j & 1) ? ob : 0);
            fac[j] = __shfl_sync(0xffffffffu, f, src);
            inv[j] = __shfl_sync(0xffffffffu, iv, src);
        }
    } else {
        // any other shape: each group's partial goes over the thread's own
        // (already decoded) g bytes of that group, then one warp per block
        float2* part4 = reinterpret_cast<float2*>(st + SL::kG);  // partial of group e/4 at byte 2e of g
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if (live[j]) part4[(eb + 128 * j) >> 2] = make_float2(g2[j], mx[j]);
        // the stage is refilled by bulk copies (async proxy) after these writes
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncthreads();
        const int q4 = p >> 2;  // groups per block
        for (int bb = warp; bb < ti.nblk; bb += THREADS / 32) {
            float s2 = 0.0f, sx = 0.0f;
            for (int t = lane; t < q4; t += 32) {
                const float2 pp = part4[bb * q4 + t];
                s2 += pp.x;
                sx = fmaxf(sx, pp.y);
            }
            s2 = warp_sum(s2);
            sx = warp_max(sx);
            if (lane == 0) {
                float f = 0.0f, iv = 0.0f;
                finish(s2, sx, MODE == kGradOnly ? 0.0f : P.v[ti.bo + bb], ti.bo + bb, true, f, iv);
                sm.blk[bb] = make_float2(f, iv);
            }
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float2 bs = live[j] ? sm.blk[blk[j]] : make_float2(0.0f, 0.0f);
            fac[j] = bs.x;
            inv[j] = bs.y;
        }
    }

    // phase 2: theta', the new codes (and x for the histogram), stored
    // straight from registers.  A zero block (inv = 0) encodes x = 0, the
    // level nearest 0, and stages NaN for the histogram.
    float* xsp = (MODE != kPlain && Smem::kHistCells == 0) ? P.xstage + ti.e0 + eb : nullptr;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        if (!live[j]) continue;
        float x[4];
        if (MODE == kGradOnly) {
#pragma unroll
            for (int i = 0; i < 4; ++i)
                x[i] = inv[j] > 0.0f ? __fdiv_rn(m[4 * j + i], inv[j]) : __int_as_float(0x7fffffff);
        } else {
            float4 t = THS ? theta4_smem<FMT>(st, eb + 128 * j) : th[j];
            t.x = fmaf(-fac[j], m[4 * j], hp.decay * t.x);
            t.y = fmaf(-fac[j], m[4 * j + 1], hp.decay * t.y);
            t.z = fmaf(-fac[j], m[4 * j + 2], hp.decay * t.z);
            t.w = fmaf(-fac[j], m[4 * j + 3], hp.decay * t.w);
            theta4_store<FMT>(P.params, ge0 + 128 * j, t);
#pragma unroll
            for (int i = 0; i < 4; ++i) x[i] = m[4 * j + i] * inv[j];
            uint32_t c[4];
            encode4<LUT>(sm.tab, lut_copy, x, c);
            store_codes4<FMT>(P.codes, ge0 + 128 * j, pack_codes4<FMT>(c));
            if (MODE == kHist) {
#pragma unroll
                for (int i = 0; i < 4; ++i) x[i] = inv[j] > 0.0f ? x[i] : __int_as_float(0x7fffffff);
            }
        }
        if (MODE != kPlain) {
            if (Smem::kHistCells > 0) {
                // count x of nonzero blocks in the CTA's cells (NaN skipped)
                if (inv[j] > 0.0f) {
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        if (!isnan(x[i])) atomicAdd(&sm.hist[hist_cell(x[i], 0.5f * P.bins, P.bins)], 1u);
                }
            } else {
                __stcs(reinterpret_cast<float4*>(xsp + 128 * j), make_float4(x[0], x[1], x[2], x[3]));
            }
        }
    }
}

template <int TILE, int THREADS, int STAGES, int LUTR, int DECR, int MODE, bool THS, int FMT, bool LUT, typename Smem>
__device__ __forceinline__ void stream_loop(Smem& sm, const Launch& L, const Ptrs& P, int* err, int seg) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t G = gridDim.x;
    const int eb = warp * 512 + lane * 4;  // first element of the thread's group 0 within a tile

    float r_s[4] = {0.0f, 0.0f, 0.0f, 0.0f}, r_v[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    if (MODE != kGradOnly && blockIdx.x < L.nunits) load_state<4>(P, sm.tile[0], eb, r_s, r_v);

    for (int it = 0;; ++it) {
        const int64_t u = blockIdx.x + static_cast<int64_t>(it) * G;
        if (u >= L.nunits) break;
        const int s = it % STAGES;
        const uint32_t parity = static_cast<uint32_t>((it / STAGES) & 1);
        const TileInfo ti = sm.tile[s];
        if (!tile_fits<TILE>(ti)) {
            // a tile the host planned too large (uniform: every thread reads
            // the same descriptor): nothing was copied for it.  Wait, bounded,
            // for the copies already issued for later tiles, flag, stop.
            __syncthreads();  // descriptors the issuing thread wrote since the last barrier
            for (int j = 1; j < STAGES; ++j) {
                const int64_t uj = u + static_cast<int64_t>(j) * G;
                if (uj >= L.nunits || !tile_fits<TILE>(sm.tile[(it + j) % STAGES])) continue;
                mbar_wait(smem_u32(&sm.bar[(it + j) % STAGES]), static_cast<uint32_t>(((it + j) / STAGES) & 1));
            }
            if (tid == 0) atomicExch(err, 2);
            break;
        }
        // the descriptor of the tile that refills this stage.  With two CTAs
        // per SM (three stages) it is prepared here, off the critical path
        // (only the issuing thread reads it back); with one CTA per SM a late
        // warp 0 holds up the block exchange, so it is prepared after the
        // tile's last barrier instead.
        const int64_t un = u + static_cast<int64_t>(STAGES) * G;
        if (STAGES >= 3 && tid == 0 && un < L.nunits) sm.next = tile_info(L, un, seg);
        // theta from global memory (an L2 hit: prefetched when the tile was
        // issued) is requested before the stage wait; from the stage, just
        // before use
        float4 th[4];
        if (MODE != kGradOnly && !THS) {
#pragma unroll
            for (int j = 0; j < 4; ++j)
                if (eb + 128 * j < ti.nelem) th[j] = theta4_global<FMT>(P.params, ti.e0 + eb + 128 * j);
        }
        // each thread waits for the stage itself; a wait that gives up is
        // acted on, uniformly, at the end of the tile
        const bool ok = mbar_wait(smem_u32(&sm.bar[s]), parity);
        // block state of the next tile, one tile ahead: with three or more
        // stages its descriptor was published before the last barrier
        float n_s[4] = {0.0f, 0.0f, 0.0f, 0.0f}, n_v[4] = {0.0f, 0.0f, 0.0f, 0.0f};
        if (STAGES >= 3 && MODE != kGradOnly && u + G < L.nunits)
            load_state<4>(P, sm.tile[(it + 1) % STAGES], eb, n_s, n_v);

        if (ti.nelem == TILE)
            stream_tile<TILE, THREADS, LUTR, DECR, MODE, THS, FMT, LUT, true>(sm, P, L.hp, ti, sm.stage[s], eb, r_s, r_v, th);
        else
            stream_tile<TILE, THREADS, LUTR, DECR, MODE, THS, FMT, LUT, false>(sm, P, L.hp, ti, sm.stage[s], eb, r_s, r_v, th);

        // every thread is done with stage s: refill it with tile it + STAGES
        if (__syncthreads_or(!ok)) {
            // a copy that never completed (the tile's outputs are undefined):
            // wait, bounded, for the copies still in flight, flag, stop
            for (int j = 0; j < STAGES; ++j) {
                const int64_t uj = u + static_cast<int64_t>(j) * G;
                if (uj >= L.nunits || !tile_fits<TILE>(sm.tile[(it + j) % STAGES])) continue;
                mbar_wait(smem_u32(&sm.bar[(it + j) % STAGES]), static_cast<uint32_t>(((it + j) / STAGES) & 1));
            }
            if (tid == 0) atomicExch(err, 1);
            break;
        }
        if (tid == 0 && un < L.nunits) {
            if (STAGES < 3) sm.next = tile_info(L, un, seg);
            issue_tile<TILE, MODE, THS, FMT>(sm, s, sm.next, P);
        }
        if (STAGES < 3 && MODE != kGradOnly && u + G < L.nunits)
            load_state<4>(P, sm.tile[(it + 1) % STAGES], eb, n_s, n_v);
#pragma unroll
        for (int j = 0; j < 4; ++j) { r_s[j] = n_s[j]; r_v[j] = n_v[j]; }
    }
}

template <int TILE, int THREADS, int STAGES, int LUTR, int DECR, bool THS, int HB, int FMT, int MODE, int MINB>
__global__ void __launch_bounds__(THREADS, MINB) k_step_stream(const __grid_constant__ Launch L, const Ptrs P, int* err) {
    using Smem = StreamSmem<TILE, THREADS, STAGES, LUTR, DECR, THS, HB, FMT>;
    static_assert(TILE == 16 * THREADS && THREADS % 32 == 0 && STAGES >= 2, "tile shape");
    static_assert(32 % LUTR == 0 && 32 % DECR == 0, "table copies");
    extern __shared__ __align__(128) unsigned char smem_raw[];
    Smem& sm = *reinterpret_cast<Smem*>(smem_raw);
    const int64_t G = gridDim.x;
    int seg = 0;  // the issuing thread's cursor into L.seg

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) mbar_init(smem_u32(&sm.bar[s]), 1u);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        for (int s = 0; s < STAGES; ++s) {
            const int64_t u = blockIdx.x + s * G;
            if (u < L.nunits) issue_tile<TILE, MODE, THS, FMT>(sm, s, tile_info(L, u, seg), P);
        }
    }
    if (HB > 0)
        for (int i = threadIdx.x; i < HB; i += THREADS) sm.hist[i] = 0u;
    const int bad = build_tables<THREADS>(P, sm.tab, MODE == kGradOnly);
    const bool lut_ok = !__syncthreads_or(bad);
    if (MODE != kGradOnly && lut_ok)
        stream_loop<TILE, THREADS, STAGES, LUTR, DECR, MODE, THS, FMT, true>(sm, L, P, err, seg);
    else
        stream_loop<TILE, THREADS, STAGES, LUTR, DECR, MODE, THS, FMT, false>(sm, L, P, err, seg);
    if (HB > 0) {
        // add the CTA's counts to the histogram
        __syncthreads();
        for (int c = threadIdx.x; c < P.bins; c += THREADS) {
            const uint32_t n = sm.hist[c];
            if (n) atomicAdd(reinterpret_cast<unsigned long long*>(P.hist) + c, static_cast<unsigned long long>(n));
        }
    }
}

// ------------------------------------------- generic p <= 2048 (scalar)
// Any period: a tile of whole blocks (<= kGenericTile elements), element
// partials in shared memory, per-block reductions, then the update.
template <int MODE>
__global__ void __launch_bounds__(kThreads) k_step_generic(const __grid_constant__ Launch L, const Ptrs P) {
    constexpr int PER = kGenericTile / kThreads;
    __shared__ float s_dec[kMaxLevels], s_mid[kMaxLevels];
    __shared__ float s_g2[kGenericTile], s_mx[kGenericTile];
    __shared__ float2 s_blk[kGenericTile / 2];  // p >= 2 on this path
    const int tid = threadIdx.x;
    const int64_t unit = blockIdx.x;
    const Seg& S = L.seg[find_seg(L, unit)];
    const HP& hp = L.hp;
    const int64_t p = S.period;
    const int64_t blk0 = (unit - S.unit_begin) * S.per_unit;
    const int nblk = static_cast<int>(min(S.per_unit, S.nblocks - blk0));
    const int ne = nblk * static_cast<int>(p);
    const int64_t e0 = S.elem_off + blk0 * p;
    const int64_t bo = S.block_off + blk0;
    const int pi = static_cast<int>(p);
    if (MODE != kGradOnly) load_codebooks(P, s_dec, s_mid);
    __syncthreads();

    float m[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        const int le = tid + i * kThreads;
        m[i] = 0.0f;
        if (le < ne) {
            const float g = bf16_bits_to_f32(__ldcs(P.grads + e0 + le));
            if (MODE == kGradOnly) {
                m[i] = g;
                s_mx[le] = fabsf(g);
            } else {
                const float sold = P.scale[bo + le / pi];
                m[i] = fmaf(hp.omb1, g, hp.beta1 * sold * s_dec[__ldcs(P.codes + e0 + le)]);
                s_g2[le] = g * g;
                s_mx[le] = fabsf(m[i]);
            }
        }
    }
    __syncthreads();
    const float pf = static_cast<float>(p);
    const int warp = tid >> 5, lane = tid & 31;
    if (pi < 32) {
        for (int b = tid; b < nblk; b += kThreads) {
            float g2 = 0.0f, mx = 0.0f;
            for (int t = 0; t < pi; ++t) {
                if (MODE != kGradOnly) g2 += s_g2[b * pi + t];
                mx = fmaxf(mx, s_mx[b * pi + t]);
            }
            float fac = 0.0f;
            if (MODE != kGradOnly) {
                fac = block_update(hp, P.v, bo + b, g2 / pf);
                P.scale[bo + b] = mx;
            }
            s_blk[b] = make_float2(fac, mx);
        }
    } else {
        for (int b = warp; b < nblk; b += kThreads / 32) {
            float g2 = 0.0f, mx = 0.0f;
            for (int t = lane; t < pi; t += 32) {
                if (MODE != kGradOnly) g2 += s_g2[b * pi + t];
                mx = fmaxf(mx, s_mx[b * pi + t]);
            }
            g2 = warp_sum(g2);
            mx = warp_max(mx);
            if (lane == 0) {
                float fac = 0.0f;
                if (MODE != kGradOnly) {
                    fac = block_update(hp, P.v, bo + b, g2 / pf);
                    P.scale[bo + b] = mx;
                }
                s_blk[b] = make_float2(fac, mx);
            }
        }
    }
    __syncthreads();
    const int zero_code = (MODE != kGradOnly) ? level_search(s_mid, 0.0f) : 0;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        const int le = tid + i * kThreads;
        if (le >= ne) continue;
        const int64_t e = e0 + le;
        const float2 bs = s_blk[le / pi];
        if (MODE == kGradOnly) {
            P.xstage[e] = bs.y > 0.0f ? __fdiv_rn(m[i], bs.y) : __int_as_float(0x7fffffff);
            continue;
        }
        const float th = __ldcs(P.params + e);
        __stcs(P.params + e, fmaf(-bs.x, m[i], hp.decay * th));
        float x;
        int c;
        if (bs.y > 0.0f) {
            x = __fdiv_rn(m[i], bs.y);
            c = level_search(s_mid, x);
        } else {
            x = __int_as_float(0x7fffffff);
            c = zero_code;
        }
        P.codes[e] = static_cast<uint8_t>(c);
        if (MODE == kHist) P.xstage[e] = x;
    }
}

// --------------------------------------------------------- big blocks
// Blocks longer than a tile: each block is cut into chunks of kChunk elements.
// (1) k_big_partial: per chunk, sum g^2 (double across threads) and max|m|.
// (2) k_big_finalize: per block, reduce its chunks in a fixed order, update v
//     and s, and keep (s_old, s_new, factor) for the apply pass.
// (3) k_big_apply: per chunk, recompute m from the kept s_old, update theta,
//     re-encode with s_new.  g and codes are read twice: 15 bytes per param.
struct ChunkRange {
    int64_t c0, c1;     // element range
    int64_t bigblk;     // global big-block index (into blk_state)
    int64_t bi;         // block index into v/scale
};

__device__ __forceinline__ ChunkRange chunk_range(const Launch& L, int64_t unit) {
    const Seg& S = L.seg[find_seg(L, unit)];
    const int64_t local = unit - S.unit_begin;
    const int64_t b = local / S.per_unit, c = local % S.per_unit;
    const int64_t bs = S.elem_off + b * S.period;
    ChunkRange r;
    r.c0 = bs + c * kChunk;
    r.c1 = min(r.c0 + kChunk, bs + S.period);
    r.bigblk = S.aux_begin + b;
    r.bi = S.block_off + b;
    return r;
}

template <typename F>
__device__ __forceinline__ void for_chunk_elems(int64_t c0, int64_t c1, bool aligned, F&& f) {
    // f(e, g, code_or_0) for every element; 16-element vectors when aligned.
    if (aligned) {
        const int nv = static_cast<int>((c1 - c0) >> 4);
        for (int j = threadIdx.x; j < nv; j += kThreads) {
            const int64_t e = c0 + static_cast<int64_t>(j) * 16;
            f(e, true);
        }
    } else {
        for (int64_t e = c0 + threadIdx.x; e < c1; e += kThreads) f(e, false);
    }
}

template <int MODE, int FMT>
__global__ void __launch_bounds__(kThreads) k_big_partial(const __grid_constant__ Launch L, const Ptrs P, int aligned) {
    __shared__ float s_dec[kMaxLevels];
    __shared__ double s_red[kThreads / 32];
    __shared__ float s_redm[kThreads / 32];
    if (MODE != kGradOnly && threadIdx.x < kMaxLevels)
        s_dec[threadIdx.x] = threadIdx.x < P.k ? P.cb_dec[threadIdx.x] : 0.0f;
    __syncthreads();
    const int64_t unit = blockIdx.x;
    const ChunkRange R = chunk_range(L, unit);
    const HP& hp = L.hp;
    const float b1s = (MODE != kGradOnly) ? hp.beta1 * P.scale[R.bi] : 0.0f;
    float g2 = 0.0f, mx = 0.0f;
    for_chunk_elems(R.c0, R.c1, aligned != 0, [&](int64_t e, bool vec) {
        if (vec) {
            const uint4 ga = __ldcg(reinterpret_cast<const uint4*>(P.grads + e));
            const uint4 gb = __ldcg(reinterpret_cast<const uint4*>(P.grads + e) + 1);
            float g[16];
            unpack16_bf16(ga, gb, g);
            if (MODE == kGradOnly) {
#pragma unroll
                for (int t = 0; t < 16; ++t) mx = fmaxf(mx, fabsf(g[t]));
            } else {
                uint32_t cv[16];
                if (Format<FMT>::kC4) {
                    const uint2 cw = __ldcg(reinterpret_cast<const uint2*>(P.codes + (e >> 1)));
#pragma unroll
                    for (int t = 0; t < 16; ++t) cv[t] = ((t < 8 ? cw.x : cw.y) >> (4 * (t & 7))) & 0xFu;
                } else {
                    const uint4 cw = __ldcg(reinterpret_cast<const uint4*>(P.codes + e));
#pragma unroll
                    for (int t = 0; t < 16; ++t) cv[t] = byte_of(cw, t);
                }
#pragma unroll
                for (int t = 0; t < 16; ++t) {
                    const float mm = fmaf(hp.omb1, g[t], b1s * s_dec[cv[t]]);
                    g2 = fmaf(g[t], g[t], g2);
                    mx = fmaxf(mx, fabsf(mm));
                }
            }
        } else {
            const float g = bf16_bits_to_f32(P.grads[e]);
            if (MODE == kGradOnly) {
                mx = fmaxf(mx, fabsf(g));
            } else {
                const float mm = fmaf(hp.omb1, g, b1s * s_dec[P.codes[e]]);
                g2 = fmaf(g, g, g2);
                mx = fmaxf(mx, fabsf(mm));
            }
        }
    });
    double d = warp_sum_d(static_cast<double>(g2));
    mx = warp_max(mx);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) { s_red[warp] = d; s_redm[warp] = mx; }
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        float m2 = 0.0f;
        for (int w = 0; w < kThreads / 32; ++w) { t += s_red[w]; m2 = fmaxf(m2, s_redm[w]); }
        P.part_g2[unit] = t;
        P.part_mx[unit] = m2;
    }
}

template <int MODE>
__global__ void __launch_bounds__(kThreads) k_big_finalize(const __grid_constant__ Launch L, const Ptrs P) {
    __shared__ double s_red[kThreads / 32];
    __shared__ float s_redm[kThreads / 32];
    const int64_t gb = blockIdx.x;  // global big-block index
    const Seg& S = L.seg[find_seg_aux(L, gb)];
    const int64_t b = gb - S.aux_begin;
    const int64_t u0 = S.unit_begin + b * S.per_unit;
    double d = 0.0;
    float mx = 0.0f;
    for (int64_t c = threadIdx.x; c < S.per_unit; c += kThreads) {
        d += P.part_g2[u0 + c];
        mx = fmaxf(mx, P.part_mx[u0 + c]);
    }
    d = warp_sum_d(d);
    mx = warp_max(mx);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) { s_red[warp] = d; s_redm[warp] = mx; }
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        float m2 = 0.0f;
        for (int w = 0; w < kThreads / 32; ++w) { t += s_red[w]; m2 = fmaxf(m2, s_redm[w]); }
        const int64_t bi = S.block_off + b;
        if (MODE == kGradOnly) {
            P.blk_state[gb] = make_float4(0.0f, m2, 0.0f, 0.0f);
        } else {
            const float sold = P.scale[bi];
            const float G = static_cast<float>(t / static_cast<double>(S.period));
            const float fac = block_update(L.hp, P.v, bi, G);
            P.scale[bi] = m2;
            P.blk_state[gb] = make_float4(sold, m2, fac, 0.0f);
        }
    }
}

template <int MODE>
__global__ void __launch_bounds__(kThreads) k_big_apply(const __grid_constant__ Launch L, const Ptrs P, int aligned) {
    __shared__ float s_dec[kMaxLevels], s_mid[kMaxLevels];
    if (MODE != kGradOnly) load_codebooks(P, s_dec, s_mid);
    __syncthreads();
    const int64_t unit = blockIdx.x;
    const ChunkRange R = chunk_range(L, unit);
    const HP& hp = L.hp;
    const float4 st = P.blk_state[R.bigblk];
    const float b1s = hp.beta1 * st.x, sn = st.y, fac = st.z;
    const int zero_code = (MODE != kGradOnly) ? level_search(s_mid, 0.0f) : 0;
    const float nanv = __int_as_float(0x7fffffff);
    // x = value / s_new and its code (zero block: NaN and the code of 0)
    auto encode = [&](float val, float& x) -> int {
        if (sn > 0.0f) {
            x = __fdiv_rn(val, sn);
            return level_search(s_mid, x);
        }
        x = nanv;
        return zero_code;
    };
    if (aligned) {
        const int nv = static_cast<int>((R.c1 - R.c0) >> 4);
        for (int j = threadIdx.x; j < nv; j += kThreads) {
            const int64_t e = R.c0 + static_cast<int64_t>(j) * 16;
            const uint4 ga = __ldcs(reinterpret_cast<const uint4*>(P.grads + e));
            const uint4 gb = __ldcs(reinterpret_cast<const uint4*>(P.grads + e) + 1);
            float g[16], x[16];
            unpack16_bf16(ga, gb, g);
            if (MODE == kGradOnly) {
#pragma unroll
                for (int t = 0; t < 16; ++t) x[t] = sn > 0.0f ? __fdiv_rn(g[t], sn) : nanv;
            } else {
                const uint4 cw = __ldcs(reinterpret_cast<const uint4*>(P.codes + e));
                float4 th[4];
                const float4* src = reinterpret_cast<const float4*>(P.params + e);
#pragma unroll
                for (int t = 0; t < 4; ++t) th[t] = __ldcs(src + t);
                float* thf = reinterpret_cast<float*>(th);
                uint32_t w[4] = {0u, 0u, 0u, 0u};
#pragma unroll
                for (int t = 0; t < 16; ++t) {
                    const float mm = fmaf(hp.omb1, g[t], b1s * s_dec[byte_of(cw, t)]);
                    thf[t] = fmaf(-fac, mm, hp.decay * thf[t]);
                    w[t >> 2] |= static_cast<uint32_t>(encode(mm, x[t])) << (8 * (t & 3));
                }
                float4* dst = reinterpret_cast<float4*>(P.params + e);
#pragma unroll
                for (int t = 0; t < 4; ++t) __stcs(dst + t, th[t]);
                __stcs(reinterpret_cast<uint4*>(P.codes + e), make_uint4(w[0], w[1], w[2], w[3]));
            }
            if (MODE != kPlain) {
                float4* xs = reinterpret_cast<float4*>(P.xstage + e);
#pragma unroll
                for (int t = 0; t < 4; ++t) __stcs(xs + t, make_float4(x[4 * t], x[4 * t + 1], x[4 * t + 2], x[4 * t + 3]));
            }
        }
    } else {
        for (int64_t e = R.c0 + threadIdx.x; e < R.c1; e += kThreads) {
            const float g = bf16_bits_to_f32(P.grads[e]);
            float x;
            if (MODE == kGradOnly) {
                x = sn > 0.0f ? __fdiv_rn(g, sn) : nanv;
            } else {
                const float mm = fmaf(hp.omb1, g, b1s * s_dec[P.codes[e]]);
                P.params[e] = fmaf(-fac, mm, hp.decay * P.params[e]);
                P.codes[e] = static_cast<uint8_t>(encode(mm, x));
            }
            if (MODE != kPlain) P.xstage[e] = x;
        }
    }
}

// ------------------------------------------------------------- host side
enum PathClass { kP1 = 0, kS4K, kS8K, kT16V4, kGeneric, kBigAligned, kBigUnaligned, kNumClasses };

template <int TILE_, int THREADS_, int STAGES_, int LUTR_, int DECR_, bool THS_, int MINB_>
struct StreamCfg {
    static constexpr int TILE = TILE_, THREADS = THREADS_, STAGES = STAGES_, LUTR = LUTR_, DECR = DECR_, MINB = MINB_;
    static constexpr bool THS = THS_;
};
// p <= 4096: two 256-thread CTAs per SM, 3-stage rings of 12 KB tiles (g,
// codes; theta read from global memory), cell records in 8 copies and the
// decode table in 8;
// p <= 8192: one 512-thread CTA per SM, a 2-stage ring of 56 KB tiles
// (theta staged too), cell records in 8 copies and the decode table in 32.
using S4KCfg = StreamCfg<4096, 256, 3, 8, 8, false, 2>;
using S8KCfg = StreamCfg<8192, 512, 2, 8, 32, true, 1>;
// Steps that also histogram x (refit steps) count up to kFusedBins cells in
// shared memory; the tables give up copies to make room.
constexpr int kFusedBins = 4096;
using S4KHistCfg = StreamCfg<4096, 256, 3, 4, 8, false, 2>;
using S8KHistCfg = StreamCfg<8192, 512, 2, 2, 4, true, 1>;
constexpr int kS4KTile = S4KCfg::TILE, kS8KTile = S8KCfg::TILE;

PathClass classify(int64_t p) {
    if (p == 1) return kP1;
    if (p % 16 == 0 && p <= kS4KTile) return kS4K;
    if (p % 16 == 0 && p <= kS8KTile) return kS8K;
    if (p % 16 == 0 && p <= kTile16Max) return kT16V4;
    if (p <= kGenericTile) return kGeneric;
    return (p % 16 == 0) ? kBigAligned : kBigUnaligned;
}

// p1_epc: elements each thread of k_step_p1 handles per round (2 with two
// codes per byte).
int64_t units_of(PathClass c, const gefen_tensor_t& t, int64_t* per_unit, int64_t tile_cap = 0, int p1_epc = 1) {
    const int64_t p = t.period, nb = t.numel / p;
    if (tile_cap > 0) {  // streamed classes: whole blocks per tile of the kernel's own size
        *per_unit = std::max<int64_t>(1, tile_cap / p);
        return (nb + *per_unit - 1) / *per_unit;
    }
    switch (c) {
        case kP1:
            *per_unit = 1;
            return (t.numel + 4 * kThreads * p1_epc - 1) / (4 * kThreads * p1_epc);
        case kS4K:
        case kS8K:
        case kT16V4: {
            const int64_t cap = (c == kS4K) ? kS4KTile : (c == kS8K) ? kS8KTile : kThreads * 4 * 16;
            *per_unit = std::max<int64_t>(1, cap / p);
            return (nb + *per_unit - 1) / *per_unit;
        }
        case kGeneric:
            *per_unit = std::max<int64_t>(1, kGenericTile / p);
            return (nb + *per_unit - 1) / *per_unit;
        default:
            *per_unit = (p + kChunk - 1) / kChunk;  // chunks per block
            return nb * *per_unit;
    }
}

struct Plan {
    std::vector<int> idx[kNumClasses];
    int64_t big_chunks = 0, big_blocks = 0, max_elem = 0;
};

Plan make_plan(const gefen_tensor_t* t, int32_t n) {
    Plan pl;
    for (int i = 0; i < n; ++i) {
        if (t[i].numel == 0) continue;
        PathClass c = classify(t[i].period);
        pl.idx[c].push_back(i);
        int64_t per = 0;
        int64_t u = units_of(c, t[i], &per);
        if (c == kBigAligned || c == kBigUnaligned) {
            pl.big_chunks += u;
            pl.big_blocks += t[i].numel / t[i].period;
        }
        pl.max_elem = std::max(pl.max_elem, t[i].offset + t[i].numel);
    }
    return pl;
}

struct WsLayout {
    size_t header, part_g2, part_mx, blk_state, xstage, total;
};

// Workspace: a 256-byte header (word 0: set when a bounded device wait gave
// up), then big-block partials and block state, then the histogram staging.
WsLayout ws_layout(const Plan& pl, uint32_t flags) {
    WsLayout w;
    size_t o = 0;
    w.header = o;
    o += kWsAlign;
    w.part_g2 = o;
    o += align_up(static_cast<size_t>(pl.big_chunks) * sizeof(double));
    w.part_mx = o;
    o += align_up(static_cast<size_t>(pl.big_chunks) * sizeof(float));
    w.blk_state = o;
    o += align_up(static_cast<size_t>(pl.big_blocks) * sizeof(float4));
    w.xstage = o;
    if (flags & (GEFEN_HIST | GEFEN_HIST_GRAD_ONLY)) o += align_up(static_cast<size_t>(pl.max_elem) * sizeof(float));
    w.total = o;
    return w;
}

bool validate_tensors(const gefen_tensor_t* t, int32_t n) {
    if (n < 0 || (n > 0 && t == nullptr)) return false;
    std::vector<std::pair<int64_t, int64_t>> er, br;
    for (int i = 0; i < n; ++i) {
        const gefen_tensor_t& x = t[i];
        if (x.offset < 0 || x.offset % 16 != 0 || x.numel < 0 || x.period < 1 || x.block_offset < 0) return false;
        if (x.numel % x.period != 0) return false;
        if (x.numel > (int64_t(1) << 40) || x.offset > (int64_t(1) << 42)) return false;
        if (x.numel == 0) continue;
        er.emplace_back(x.offset, x.offset + x.numel);
        br.emplace_back(x.block_offset, x.block_offset + x.numel / x.period);
    }
    for (auto* v : {&er, &br}) {
        std::sort(v->begin(), v->end());
        for (size_t i = 1; i < v->size(); ++i)
            if ((*v)[i].first < (*v)[i - 1].second) return false;
    }
    return true;
}

// Fills L.seg with up to kMaxSegs tensors at a time and launches one grid
// per group through `kernel(L, units)`.
template <typename K>
cudaError_t launch_class(K kernel, Launch& L, const std::vector<int>& ids, const gefen_tensor_t* t,
                         PathClass c, int64_t tile_cap = 0, int p1_epc = 1) {
    size_t i = 0;
    while (i < ids.size()) {
        L.nseg = 0;
        int64_t units = 0;
        for (; i < ids.size() && L.nseg < kMaxSegs; ++i) {
            const gefen_tensor_t& x = t[ids[i]];
            Seg& s = L.seg[L.nseg++];
            seg_fill(s, x);
            s.unit_begin = units;
            s.aux_begin = 0;
            if (tile_cap > 0 && x.period > tile_cap) return cudaErrorInvalidValue;  // planning error
            units += units_of(c, x, &s.per_unit, tile_cap, p1_epc);
        }
        L.nunits = units;
        if (units == 0) continue;
        kernel(L, units);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

// One launch of the streamed kernel over the units of a prepared Launch.
template <typename C, int MODE, int HB, int FMT>
cudaError_t stream_kernel(const Launch& L, const Ptrs& P, int* err, cudaStream_t st) {
    auto kern = k_step_stream<C::TILE, C::THREADS, C::STAGES, C::LUTR, C::DECR, C::THS, HB, FMT, MODE, C::MINB>;
    const int smem =
        static_cast<int>(sizeof(StreamSmem<C::TILE, C::THREADS, C::STAGES, C::LUTR, C::DECR, C::THS, HB, FMT>));
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, C::THREADS, smem);
    if (e != cudaSuccess) return e;
    const int64_t cap = static_cast<int64_t>(std::max(1, per_sm)) * device_sm_count();
    kern<<<dim3(static_cast<unsigned>(std::min(L.nunits, cap))), C::THREADS, smem, st>>>(L, P, err);
    return cudaGetLastError();
}

template <typename C, int MODE, int HB, int FMT>
cudaError_t launch_stream(Launch& L, const std::vector<int>& ids, const gefen_tensor_t* t, PathClass c,
                          const Ptrs& P, int* err, cudaStream_t st) {
    cudaError_t e2 = cudaSuccess;
    cudaError_t e = launch_class(
        [&](Launch& LL, int64_t) {
            if (e2 == cudaSuccess) e2 = stream_kernel<C, MODE, HB, FMT>(LL, P, err, st);
        },
        L, ids, t, c, C::TILE);
    return e != cudaSuccess ? e : e2;
}

// Big blocks whose size is a multiple of the streamed tile are applied by the
// streamed kernel, tile by tile, with the factors their finalisation kept.
inline bool big_streamable(int64_t p) { return p > kTile16Max && p % kS4KTile == 0; }

// fused: the streamed kernels count the histogram in shared memory (the
// other kernels stage x for launch_histogram).  FMT: storage format (only
// the classes the host validated for it occur).
template <int MODE, int FMT>
cudaError_t run_step(const Plan& pl, const gefen_tensor_t* t, Launch& L, const Ptrs& P, int* err, cudaStream_t st,
                     bool fused) {
    cudaError_t e;
    e = launch_class([&](Launch& LL, int64_t u) { k_step_p1<MODE, FMT><<<dim3(u), kThreads, 0, st>>>(LL, P); },
                     L, pl.idx[kP1], t, kP1, 0, Format<FMT>::kC4 ? 2 : 1);
    if (e != cudaSuccess) return e;
    auto streamed = [&](auto cfg, auto hist_cfg, PathClass c) -> cudaError_t {
        using C = decltype(cfg);
        using CH = decltype(hist_cfg);
        if constexpr (MODE != kPlain) {
            if (fused) return launch_stream<CH, MODE, kFusedBins, FMT>(L, pl.idx[c], t, c, P, err, st);
            if constexpr (FMT == 0) return launch_stream<C, MODE, 0, 0>(L, pl.idx[c], t, c, P, err, st);
            return pl.idx[c].empty() ? cudaSuccess : cudaErrorNotSupported;
        } else {
            return launch_stream<C, MODE, 0, FMT>(L, pl.idx[c], t, c, P, err, st);
        }
    };
    if ((e = streamed(S4KCfg{}, S4KHistCfg{}, kS4K)) != cudaSuccess) return e;
    if ((e = streamed(S8KCfg{}, S8KHistCfg{}, kS8K)) != cudaSuccess) return e;
    if constexpr (FMT == 0) {
        e = launch_class([&](Launch& LL, int64_t u) { k_step_tile16<4, MODE><<<dim3(u), kThreads, 0, st>>>(LL, P); },
                         L, pl.idx[kT16V4], t, kT16V4);
        if (e != cudaSuccess) return e;
        e = launch_class([&](Launch& LL, int64_t u) { k_step_generic<MODE><<<dim3(u), kThreads, 0, st>>>(LL, P); },
                         L, pl.idx[kGeneric], t, kGeneric);
        if (e != cudaSuccess) return e;
    }
    // Big blocks: partial, finalize, apply per group of tensors.  Chunk and
    // block counters run across groups so workspace slots never collide.
    for (int cls : {kBigAligned, kBigUnaligned}) {
        const int aligned = (cls == kBigAligned) ? 1 : 0;
        const std::vector<int>& ids = pl.idx[cls];
        size_t i = 0;
        while (i < ids.size()) {
            L.nseg = 0;
            int64_t units = 0, blocks = 0;
            for (; i < ids.size() && L.nseg < kMaxSegs; ++i) {
                const gefen_tensor_t& x = t[ids[i]];
                Seg& s = L.seg[L.nseg++];
                seg_fill(s, x);
                s.unit_begin = units;
                s.aux_begin = blocks;
                units += units_of(static_cast<PathClass>(cls), x, &s.per_unit);
                blocks += x.numel / x.period;
            }
            L.nunits = units;
            if (units == 0) continue;
            k_big_partial<MODE, FMT><<<dim3(units), kThreads, 0, st>>>(L, P, aligned);
            k_big_finalize<MODE><<<dim3(blocks), kThreads, 0, st>>>(L, P);
            if ((e = cudaGetLastError()) != cudaSuccess) return e;
            // apply: streamed tiles where the block size allows, chunks otherwise
            // (same big-block numbering, so both read the finalised state)
            static thread_local Launch LS, LA;
            LS.hp = LA.hp = L.hp;
            LS.nseg = LA.nseg = 0;
            LS.nunits = LA.nunits = 0;
            for (int j = 0; j < L.nseg; ++j) {
                const Seg& sj = L.seg[j];
                if (big_streamable(sj.period)) {
                    Seg& d = LS.seg[LS.nseg++];
                    d = sj;
                    d.flags = kSegBigTiles;
                    d.per_unit = sj.period / kS4KTile;
                    d.unit_begin = LS.nunits;
                    LS.nunits += sj.nblocks * d.per_unit;
                } else {
                    Seg& d = LA.seg[LA.nseg++];
                    d = sj;
                    d.unit_begin = LA.nunits;
                    LA.nunits += sj.nblocks * sj.per_unit;
                }
            }
            if (LS.nunits > 0) {
                if constexpr (MODE != kPlain) {
                    if (fused)
                        e = stream_kernel<S4KHistCfg, MODE, kFusedBins, FMT>(LS, P, err, st);
                    else if constexpr (FMT == 0)
                        e = stream_kernel<S4KCfg, MODE, 0, 0>(LS, P, err, st);
                    else
                        e = cudaErrorNotSupported;
                } else {
                    e = stream_kernel<S4KCfg, MODE, 0, FMT>(LS, P, err, st);
                }
                if (e != cudaSuccess) return e;
            }
            if constexpr (FMT == 0) {
                if (LA.nunits > 0) k_big_apply<MODE><<<dim3(LA.nunits), kThreads, 0, st>>>(LA, P, aligned);
            } else {
                if (LA.nunits > 0) return cudaErrorNotSupported;
            }
            if ((e = cudaGetLastError()) != cudaSuccess) return e;
        }
    }
    return cudaSuccess;
}

// Whether every tensor's path can store this format: p == 1, the streamed
// tiles (p a multiple of 32 with two codes per byte) and big blocks applied
// as streamed tiles.
bool format_supported(const gefen_tensor_t* t, int32_t n, int fmt) {
    for (int i = 0; i < n; ++i) {
        if (t[i].numel == 0) continue;
        const int64_t p = t[i].period;
        const PathClass c = classify(p);
        bool ok = c == kP1 || c == kS4K || c == kS8K || (c == kBigAligned && big_streamable(p));
        if ((fmt & 1) && (c == kS4K || c == kS8K) && p % 32 != 0) ok = false;
        if (!ok) return false;
    }
    return true;
}

}  // namespace

}  // namespace gefen

using namespace gefen;

extern "C" size_t gefen_step_workspace_size(const gefen_tensor_t* tensors, int32_t ntensors, uint32_t flags) {
    if (!validate_tensors(tensors, ntensors)) return 0;
    return ws_layout(make_plan(tensors, ntensors), flags).total;
}

extern "C" gefen_status_t gefen_step(const gefen_tensor_t* tensors, int32_t ntensors, float* params,
                                     const uint16_t* grads, uint8_t* codes, float* v, float* scale,
                                     const float* codebook_dec, const float* codebook_enc, int32_t k,
                                     gefen_hparams_t hp, uint64_t* hist, int32_t hist_bins, void* workspace,
                                     size_t workspace_bytes, gefen_stream_t stream) {
    if (!validate_tensors(tensors, ntensors)) return GEFEN_EINVAL;
    const uint32_t flags = hp.flags;
    if (flags & ~(GEFEN_HIST | GEFEN_HIST_GRAD_ONLY | GEFEN_CODES_4BIT | GEFEN_PARAMS_BF16)) return GEFEN_EINVAL;
    if ((flags & GEFEN_HIST) && (flags & GEFEN_HIST_GRAD_ONLY)) return GEFEN_EINVAL;
    const bool grad_only = (flags & GEFEN_HIST_GRAD_ONLY) != 0;
    const bool want_hist = (flags & (GEFEN_HIST | GEFEN_HIST_GRAD_ONLY)) != 0;
    if (grads == nullptr) return GEFEN_EINVAL;
    if (!grad_only) {
        if (!params || !codes || !v || !scale || !codebook_dec || !codebook_enc) return GEFEN_EINVAL;
        if (k < 2 || k > GEFEN_MAX_LEVELS) return GEFEN_EINVAL;
        if (hp.step < 1) return GEFEN_EINVAL;
        if (!(hp.beta1 >= 0.0 && hp.beta1 < 1.0 && hp.beta2 >= 0.0 && hp.beta2 < 1.0)) return GEFEN_EINVAL;
        if (!std::isfinite(hp.lr) || !std::isfinite(hp.eps) || !std::isfinite(hp.weight_decay) || hp.eps < 0.0)
            return GEFEN_EINVAL;
        if ((reinterpret_cast<uintptr_t>(params) | reinterpret_cast<uintptr_t>(codes)) & 15u) return GEFEN_EINVAL;
    }
    if (reinterpret_cast<uintptr_t>(grads) & 15u) return GEFEN_EINVAL;
    if (want_hist && (hist == nullptr || hist_bins < 1 || hist_bins > GEFEN_MAX_BINS)) return GEFEN_EINVAL;
    // storage formats (the first-gradient histogram reads g only)
    const int fmt = grad_only ? 0 : ((flags & GEFEN_CODES_4BIT) ? 1 : 0) | ((flags & GEFEN_PARAMS_BF16) ? 2 : 0);
    if (fmt & 1) {
        if (k > 16) return GEFEN_EINVAL;
        for (int i = 0; i < ntensors; ++i)
            if (tensors[i].offset % 32 != 0) return GEFEN_EINVAL;
    }
    if (fmt != 0) {
        if (!format_supported(tensors, ntensors, fmt)) return GEFEN_EUNSUPPORTED;
        if (want_hist && hist_bins > kFusedBins) return GEFEN_EUNSUPPORTED;
    }
    const Plan pl = make_plan(tensors, ntensors);
    const WsLayout wl = ws_layout(pl, flags);
    if (workspace_bytes < wl.total || workspace == nullptr) return GEFEN_ENOMEM;
    if (reinterpret_cast<uintptr_t>(workspace) % kWsAlign) return GEFEN_EINVAL;
    if (gefen_status_t s = check_device(); s != GEFEN_OK) return s;

    char* ws = static_cast<char*>(workspace);
    Ptrs P;
    P.params = params;
    P.grads = grads;
    P.codes = codes;
    P.v = v;
    P.scale = scale;
    P.cb_dec = codebook_dec;
    P.cb_enc = codebook_enc;
    P.k = grad_only ? 2 : k;
    P.xstage = want_hist ? reinterpret_cast<float*>(ws + wl.xstage) : nullptr;
    P.hist = hist;
    P.bins = hist_bins;
    P.part_g2 = reinterpret_cast<double*>(ws + wl.part_g2);
    P.part_mx = reinterpret_cast<float*>(ws + wl.part_mx);
    P.blk_state = reinterpret_cast<float4*>(ws + wl.blk_state);

    static thread_local Launch L;  // ~15 KB parameter block, reused per thread
    std::memset(&L.hp, 0, sizeof(L.hp));
    if (!grad_only) {
        const double t = static_cast<double>(hp.step);
        const double bc1 = 1.0 - std::pow(hp.beta1, t), bc2 = 1.0 - std::pow(hp.beta2, t);
        L.hp.beta1 = static_cast<float>(hp.beta1);
        L.hp.omb1 = static_cast<float>(1.0 - hp.beta1);
        L.hp.beta2 = static_cast<float>(hp.beta2);
        L.hp.omb2 = static_cast<float>(1.0 - hp.beta2);
        L.hp.inv_bc2 = static_cast<float>(1.0 / bc2);
        L.hp.lr_bc1 = static_cast<float>(hp.lr / bc1);
        L.hp.eps = static_cast<float>(hp.eps);
        L.hp.decay = static_cast<float>(1.0 - hp.lr * hp.weight_decay);
    }
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e;
    int* err = reinterpret_cast<int*>(ws + wl.header);
    const bool fused = want_hist && hist_bins <= kFusedBins;
    if (grad_only) {
        e = run_step<kGradOnly, 0>(pl, tensors, L, P, err, st, fused);
    } else if (flags & GEFEN_HIST) {
        switch (fmt) {
            case 0: e = run_step<kHist, 0>(pl, tensors, L, P, err, st, fused); break;
            case 1: e = run_step<kHist, 1>(pl, tensors, L, P, err, st, fused); break;
            case 2: e = run_step<kHist, 2>(pl, tensors, L, P, err, st, fused); break;
            default: e = run_step<kHist, 3>(pl, tensors, L, P, err, st, fused); break;
        }
    } else {
        switch (fmt) {
            case 0: e = run_step<kPlain, 0>(pl, tensors, L, P, err, st, false); break;
            case 1: e = run_step<kPlain, 1>(pl, tensors, L, P, err, st, false); break;
            case 2: e = run_step<kPlain, 2>(pl, tensors, L, P, err, st, false); break;
            default: e = run_step<kPlain, 3>(pl, tensors, L, P, err, st, false); break;
        }
    }
    if (e != cudaSuccess) return GEFEN_ECUDA;
    if (want_hist) {
        std::vector<HistRange> rr;
        for (int i = 0; i < ntensors; ++i) {
            if (tensors[i].numel == 0) continue;
            const PathClass c = classify(tensors[i].period);
            if (fused && (c == kS4K || c == kS8K || (c == kBigAligned && big_streamable(tensors[i].period))))
                continue;  // counted in place
            rr.push_back({tensors[i].offset, tensors[i].numel});
        }
        if (!rr.empty() && launch_histogram(P.xstage, rr.data(), static_cast<int>(rr.size()), hist_bins, hist, st) !=
                               cudaSuccess)
            return GEFEN_ECUDA;
    }
    return GEFEN_OK;
}

extern "C" gefen_status_t gefen_step_status(void* workspace, gefen_stream_t stream) {
    if (workspace == nullptr || reinterpret_cast<uintptr_t>(workspace) % kWsAlign) return GEFEN_EINVAL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    int word = 0;
    if (cudaMemcpyAsync(&word, workspace, sizeof(word), cudaMemcpyDeviceToHost, st) != cudaSuccess) return GEFEN_ECUDA;
    if (cudaStreamSynchronize(st) != cudaSuccess) return GEFEN_ECUDA;
    if (word == 0) return GEFEN_OK;
    if (cudaMemsetAsync(workspace, 0, sizeof(word), st) != cudaSuccess) return GEFEN_ECUDA;
    return GEFEN_ETIMEOUT;
}
