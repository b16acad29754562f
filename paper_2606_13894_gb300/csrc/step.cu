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
//                                          (step_kernels.cuh; one launch per
//                                          block shape)
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

#include "step_kernels.cuh"

namespace gefen {

namespace {

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
// (1) k_big_partial: per chunk, sum g^2 and max|m| (fp32 within the chunk, as
//     in a streamed block; FP64 on every thread would cost this GPU more
//     than the chunk's loads).
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

template <int MODE, int FMT>
__global__ void __launch_bounds__(kThreads) k_big_partial(const __grid_constant__ Launch L, const Ptrs P, int aligned) {
    __shared__ float s_dec[kMaxLevels];
    __shared__ float s_red[kThreads / 32];
    __shared__ float s_redm[kThreads / 32];
    if (MODE != kGradOnly && threadIdx.x < kMaxLevels)
        s_dec[threadIdx.x] = threadIdx.x < P.k ? P.cb_dec[threadIdx.x] : 0.0f;
    __syncthreads();
    const int64_t unit = blockIdx.x;
    const ChunkRange R = chunk_range(L, unit);
    const HP& hp = L.hp;
    const float b1s = (MODE != kGradOnly) ? hp.beta1 * P.scale[R.bi] : 0.0f;
    float g2 = 0.0f, mx = 0.0f;
    auto add16 = [&](const uint4& ga, const uint4& gb, const uint32_t (&cv)[16]) {
        float g[16];
        unpack16_bf16(ga, gb, g);
#pragma unroll
        for (int t = 0; t < 16; ++t) {
            if (MODE == kGradOnly) {
                mx = fmaxf(mx, fabsf(g[t]));
            } else {
                const float mm = fmaf(hp.omb1, g[t], b1s * s_dec[cv[t]]);
                g2 = fmaf(g[t], g[t], g2);
                mx = fmaxf(mx, fabsf(mm));
            }
        }
    };
    if (aligned) {
        const int nv = static_cast<int>((R.c1 - R.c0) >> 4);
        for (int j = threadIdx.x; j < nv; j += kThreads) {
            const int64_t e = R.c0 + static_cast<int64_t>(j) * 16;
            const uint4 ga = __ldcg(reinterpret_cast<const uint4*>(P.grads + e));
            const uint4 gb = __ldcg(reinterpret_cast<const uint4*>(P.grads + e) + 1);
            uint32_t cv[16];
            if (MODE != kGradOnly) {
                if (Format<FMT>::kC4) {
                    const uint2 cw = __ldcg(reinterpret_cast<const uint2*>(P.codes + (e >> 1)));
#pragma unroll
                    for (int t = 0; t < 16; ++t) cv[t] = ((t < 8 ? cw.x : cw.y) >> (4 * (t & 7))) & 0xFu;
                } else {
                    const uint4 cw = __ldcg(reinterpret_cast<const uint4*>(P.codes + e));
#pragma unroll
                    for (int t = 0; t < 16; ++t) cv[t] = byte_of(cw, t);
                }
            }
            add16(ga, gb, cv);
        }
    } else {
        for (int64_t e = R.c0 + threadIdx.x; e < R.c1; e += kThreads) {
            const float g = bf16_bits_to_f32(P.grads[e]);
            if (MODE == kGradOnly) {
                mx = fmaxf(mx, fabsf(g));
            } else {
                const float mm = fmaf(hp.omb1, g, b1s * s_dec[P.codes[e]]);
                g2 = fmaf(g, g, g2);
                mx = fmaxf(mx, fabsf(mm));
            }
        }
    }
    const float d = warp_sum_bfly(g2);
    mx = warp_max_nonneg(mx);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) { s_red[warp] = d; s_redm[warp] = mx; }
    __syncthreads();
    if (threadIdx.x == 0) {
        float t = 0.0f, m2 = 0.0f;
#pragma unroll
        for (int w = 0; w < kThreads / 32; ++w) { t += s_red[w]; m2 = fmaxf(m2, s_redm[w]); }
        P.part_g2[unit] = t;
        P.part_mx[unit] = m2;
    }
}

// (a thread adds its chunks in fp64, the warps and the CTA in fp32)
template <int MODE>
__global__ void __launch_bounds__(kThreads) k_big_finalize(const __grid_constant__ Launch L, const Ptrs P) {
    __shared__ float s_red[kThreads / 32];
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
    const float df = warp_sum_bfly(static_cast<float>(d));
    mx = warp_max_nonneg(mx);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) { s_red[warp] = df; s_redm[warp] = mx; }
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

// Below this many elements a streamed class takes a single launch: a second
// launch's fixed cost (table build, ramp and tail, about 10 us) exceeds what
// a shape's own instance saves.
constexpr int64_t kShapeSplitElems = int64_t(1) << 28;

// The streamed kernel over the tensors `ids` of class c (kS4K or kS8K): one
// launch (per segment-table group) for each block shape among them, or one
// launch in all for a class of under kShapeSplitElems elements (its shape's
// instance when the shapes agree, else the instance for any shape).
cudaError_t launch_stream(Launch& L, const std::vector<int>& ids, const gefen_tensor_t* t, PathClass c, int mode,
                          int hb, int fmt, const Ptrs& P, int* err, cudaStream_t st) {
    std::vector<int> by[3];
    int64_t total = 0;
    for (int id : ids) total += t[id].numel;
    for (int id : ids) by[shape_of(t[id].period)].push_back(id);
    if (total < kShapeSplitElems && (by[0].size() != ids.size() && by[1].size() != ids.size() &&
                                     by[2].size() != ids.size())) {
        by[kShapeAny] = ids;
        by[kShapeWarp].clear();
        by[kShapeSub].clear();
    }
    const int64_t cap = (c == kS4K) ? kS4KTile : kS8KTile;
    for (int shape : {kShapeWarp, kShapeSub, kShapeAny}) {
        cudaError_t e2 = cudaSuccess;
        cudaError_t e = launch_class(
            [&](Launch& LL, int64_t) {
                if (e2 != cudaSuccess) return;
                if (c == kS4K)
                    e2 = (mode == kPlain) ? stream_s4k_plain(fmt, shape, LL, P, err, st)
                                          : stream_s4k_modes(mode, hb, fmt, shape, LL, P, err, st);
                else
                    e2 = stream_s8k(mode, hb, fmt, shape, LL, P, err, st);
            },
            L, by[shape], t, c, cap);
        if (e != cudaSuccess) return e;
        if (e2 != cudaSuccess) return e2;
    }
    return cudaSuccess;
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
    // the streamed classes: shared-memory cells on fused histogram steps; an
    // unfused histogram step supports the plain format only
    const int hb = (MODE != kPlain && fused) ? kFusedBins : 0;
    for (PathClass c : {kS4K, kS8K}) {
        if (MODE != kPlain && !fused && FMT != 0) {
            if (!pl.idx[c].empty()) return cudaErrorNotSupported;
            continue;
        }
        if ((e = launch_stream(L, pl.idx[c], t, c, MODE, hb, FMT, P, err, st)) != cudaSuccess) return e;
    }
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
                if (MODE != kPlain && !fused && FMT != 0) return cudaErrorNotSupported;
                if ((e = stream_big(MODE, hb, FMT, LS, P, err, st)) != cudaSuccess) return e;
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
