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
//   p % 16 == 0, p <= 16K  k_step_tile16   one CTA holds whole blocks in
//                                          registers: one HBM pass
//   other p <= 2048        k_step_generic  the same with scalar accesses
//   larger p               k_big_*         chunked: partial reductions, block
//                                          finalise, apply (re-reads g, codes)
#include <algorithm>
#include <cmath>
#include <cstring>
#include <vector>

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
    uint32_t pad;
};

inline void seg_fill(Seg& s, const gefen_tensor_t& x) {
    s.elem_off = x.offset;
    s.numel = x.numel;
    s.period = x.period;
    s.block_off = x.block_offset;
    s.nblocks = x.numel / x.period;
    s.pmagic = static_cast<uint32_t>((uint64_t(1) << 32) / static_cast<uint64_t>(x.period)) + 1u;
    s.pad = 0;
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
    float* xstage;      // histogram input staging (HIST modes)
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
// Every element is its own block: v and s are per element, x = m/|m| = +-1.
template <int MODE>
__global__ void __launch_bounds__(kThreads) k_step_p1(const __grid_constant__ Launch L, const Ptrs P) {
    __shared__ float s_dec[kMaxLevels], s_mid[kMaxLevels];
    if (MODE != kGradOnly) load_codebooks(P, s_dec, s_mid);
    __syncthreads();
    const int64_t unit = blockIdx.x;
    const Seg& S = L.seg[find_seg(L, unit)];
    const int64_t base = (unit - S.unit_begin) * (4 * kThreads);
    const HP& hp = L.hp;
    const int zero_code = (MODE != kGradOnly) ? level_search(s_mid, 0.0f) : 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t le = base + threadIdx.x + i * kThreads;
        if (le >= S.numel) break;
        const int64_t e = S.elem_off + le;
        const int64_t bi = S.block_off + le;
        const float g = bf16_bits_to_f32(__ldcs(P.grads + e));
        if (MODE == kGradOnly) {
            P.xstage[e] = g != 0.0f ? __fdiv_rn(g, fabsf(g)) : __int_as_float(0x7fffffff);
            continue;
        }
        const float m = fmaf(hp.omb1, g, hp.beta1 * P.scale[bi] * s_dec[__ldcs(P.codes + e)]);
        const float fac = block_update(hp, P.v, bi, g * g);
        const float am = fabsf(m);
        P.scale[bi] = am;
        const float th = __ldcs(P.params + e);
        __stcs(P.params + e, fmaf(-fac, m, hp.decay * th));
        float x;
        int c;
        if (am > 0.0f) {
            x = __fdiv_rn(m, am);
            c = level_search(s_mid, x);
        } else {
            x = __int_as_float(0x7fffffff);
            c = zero_code;
        }
        P.codes[e] = static_cast<uint8_t>(c);
        if (MODE == kHist) P.xstage[e] = x;
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
// Persistent CTAs stream tiles of whole blocks (p % 16 == 0, p <= TILE)
// through a STAGES-deep shared-memory ring: thread 0 issues cp.async.bulk
// copies of theta, g and codes for tile i+STAGES-1 while every thread works on
// tile i, and writes theta' and codes' back with bulk stores.  Decoding uses a
// shared table; encoding maps x = m / s' to its cell of a uniform grid over
// [-1, 1] whose record holds the number of midpoints below the cell and the next
// three midpoints, so the nearest level is base + three compares (identical to
// the binary search, which remains the fallback when a cell holds more than
// three midpoints).
constexpr int kLutCells = 512;
constexpr float kLutGuard = 2.384185791015625e-07f;  // 2^-22, below every cell edge

struct alignas(16) StreamTables {
    float4 lut[kLutCells + 2];  // record c+1 for cell c in [-1, kLutCells]
    float dec[kMaxLevels];
    float mid[kMaxLevels + 4];
};

template <int TILE, int THREADS, int STAGES>
struct alignas(128) StreamSmem {
    unsigned char stage[STAGES][TILE * 7];  // theta f32 | g bf16 | codes u8
    StreamTables tab;
    float2 part[TILE / 8];   // per 8-element group (or per warp): (sum g^2, max |m|)
    float2 blk[TILE / 16];   // per block: (step factor, 1/s')  [grad-only: (-, absmax)]
    float sold[TILE / 16];   // per block: scale before the step
    float vold[TILE / 16];   // per block: v before the step
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
__device__ __forceinline__ void bulk_s2g(void* dst, uint32_t src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(src), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read_all() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// Decode table, midpoints (padded with +inf) and the cell records.
template <int THREADS>
__device__ __forceinline__ int build_tables(const Ptrs& P, StreamTables& T, bool grad_only) {
    const int t = threadIdx.x;
    if (grad_only) return 0;
    for (int i = t; i < kMaxLevels + 4; i += THREADS) {
        if (i < kMaxLevels) T.dec[i] = i < P.k ? P.cb_dec[i] : 0.0f;
        T.mid[i] = (i < P.k - 1) ? 0.5f * (P.cb_enc[i] + P.cb_enc[i + 1]) : INFINITY;
    }
    __syncthreads();
    int bad = 0;
    // cell(x) = floor(fma(x, G/2, G/2)) is within 2^-24 of exact in x: each
    // record counts the midpoints below its cell minus a 2^-22 guard and holds
    // the next three; its cell plus the guard on both sides may hold at most
    // three midpoints, or the binary search is used instead.
    for (int c = t - 1; c <= kLutCells; c += THREADS) {
        const float lo = -1.0f + 2.0f * static_cast<float>(c) / kLutCells - kLutGuard;
        const float hi = -1.0f + 2.0f * static_cast<float>(c + 1) / kLutCells + kLutGuard;
        const int base = level_search(T.mid, lo);
        const int upto = level_search(T.mid, hi);
        bad |= (upto - base > 3);
        T.lut[c + 1] = make_float4(__int_as_float(base), T.mid[base], T.mid[base + 1], T.mid[base + 2]);
    }
    return bad;
}

__device__ __forceinline__ int encode_lut(const StreamTables& T, bool lut_ok, float x) {
    if (lut_ok) {
        int c = __float2int_rd(__fmaf_rn(x, 0.5f * kLutCells, 0.5f * kLutCells));
        c = min(max(c, -1), kLutCells);
        const float4 r = T.lut[c + 1];
        return __float_as_int(r.x) + (r.y < x) + (r.z < x) + (r.w < x);
    }
    return level_search(T.mid, x);
}

struct TileInfo {
    int64_t e0;    // first element
    int64_t bo;    // first block index into v / scale
    int nelem;
    int nblk;
    int p;
    uint32_t pmagic;  // floor(2^32 / p) + 1: e / p == umulhi(e, pmagic) for e, p < 2^16
};

__device__ __forceinline__ TileInfo tile_info(const Launch& L, int64_t unit) {
    const Seg& S = L.seg[find_seg(L, unit)];
    const int64_t p = S.period;
    const int64_t blk0 = (unit - S.unit_begin) * S.per_unit;
    TileInfo ti;
    ti.nblk = static_cast<int>(min(S.per_unit, S.nblocks - blk0));
    ti.p = static_cast<int>(p);
    ti.nelem = ti.nblk * ti.p;
    ti.e0 = S.elem_off + blk0 * p;
    ti.bo = S.block_off + blk0;
    ti.pmagic = S.pmagic;
    return ti;
}

// A tile fits its stage iff it holds at most TILE elements, a multiple of 16
// (so every copy is a whole number of 16-byte units).
template <int TILE>
__device__ __forceinline__ bool tile_fits(const TileInfo& ti) {
    return ti.nelem > 0 && ti.nelem <= TILE && (ti.nelem & 15) == 0;
}

template <int TILE, int MODE>
__device__ __forceinline__ void issue_tile(unsigned char* stage, uint32_t bar, const TileInfo& ti, const Ptrs& P) {
    if (!tile_fits<TILE>(ti)) return;  // never copied; the consumer stops before waiting on it
    const uint32_t n = static_cast<uint32_t>(ti.nelem);
    if (MODE == kGradOnly) {
        mbar_expect_tx(bar, 2u * n);
        bulk_g2s(smem_u32(stage + 4 * TILE), P.grads + ti.e0, 2u * n, bar);
    } else {
        mbar_expect_tx(bar, 7u * n);
        bulk_g2s(smem_u32(stage), P.params + ti.e0, 4u * n, bar);
        bulk_g2s(smem_u32(stage + 4 * TILE), P.grads + ti.e0, 2u * n, bar);
        bulk_g2s(smem_u32(stage + 6 * TILE), P.codes + ti.e0, n, bar);
    }
}

template <int TILE, int THREADS, int STAGES, int MODE, int MINB>
__global__ void __launch_bounds__(THREADS, MINB) k_step_stream(const __grid_constant__ Launch L, const Ptrs P, int* err) {
    using Smem = StreamSmem<TILE, THREADS, STAGES>;
    // each thread owns one group of 8 consecutive elements of the tile
    static_assert(TILE == 8 * THREADS && THREADS >= TILE / 16 && THREADS % 32 == 0, "tile shape");
    extern __shared__ __align__(128) unsigned char smem_raw[];
    Smem& sm = *reinterpret_cast<Smem*>(smem_raw);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const HP& hp = L.hp;
    const int64_t G = gridDim.x;

    if (tid == 0) {
        for (int s = 0; s < STAGES; ++s) mbar_init(smem_u32(&sm.bar[s]), 1u);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    const int bad = build_tables<THREADS>(P, sm.tab, MODE == kGradOnly);
    const bool lut_ok = !__syncthreads_or(bad);
    const int zero_code = (MODE != kGradOnly) ? level_search(sm.tab.mid, 0.0f) : 0;

    if (tid == 0) {
        for (int s = 0; s < STAGES - 1; ++s) {
            const int64_t u = blockIdx.x + s * G;
            if (u < L.nunits) issue_tile<TILE, MODE>(sm.stage[s], smem_u32(&sm.bar[s]), tile_info(L, u), P);
        }
    }
    // block state of the first tile; later tiles' state is loaded one tile ahead
    float r_sold = 0.0f, r_vold = 0.0f;
    if (MODE != kGradOnly && blockIdx.x < L.nunits) {
        const TileInfo t0 = tile_info(L, blockIdx.x);
        if (tid < t0.nblk) { r_sold = P.scale[t0.bo + tid]; r_vold = P.v[t0.bo + tid]; }
    }

    for (int it = 0;; ++it) {
        const int64_t u = blockIdx.x + static_cast<int64_t>(it) * G;
        if (u >= L.nunits) break;
        const int s = it % STAGES;
        const uint32_t parity = static_cast<uint32_t>((it / STAGES) & 1);
        const TileInfo ti = tile_info(L, u);
        if (!tile_fits<TILE>(ti)) {
            // a tile the host planned too large: nothing was copied for it.
            // Wait (bounded) for the copies already issued for later tiles,
            // flag the error and stop.
            for (int j = 1; j < STAGES; ++j) {
                const int64_t uj = u + static_cast<int64_t>(j) * G;
                if (uj >= L.nunits || !tile_fits<TILE>(tile_info(L, uj))) continue;
                mbar_wait(smem_u32(&sm.bar[(it + j) % STAGES]), static_cast<uint32_t>(((it + j) / STAGES) & 1));
            }
            if (tid == 0) atomicExch(err, 2);
            break;
        }
        if (MODE != kGradOnly) {
            if (tid < ti.nblk) { sm.sold[tid] = r_sold; sm.vold[tid] = r_vold; }
            if (u + G < L.nunits) {
                const TileInfo tn = tile_info(L, u + G);
                if (tid < tn.nblk) { r_sold = P.scale[tn.bo + tid]; r_vold = P.v[tn.bo + tid]; }
            }
        }
        const bool ok = mbar_wait(smem_u32(&sm.bar[s]), parity);
        if (__syncthreads_or(!ok)) {
            if (tid == 0) atomicExch(err, 1);
            break;
        }
        unsigned char* st = sm.stage[s];
        float* sth = reinterpret_cast<float*>(st);
        const uint16_t* sg = reinterpret_cast<const uint16_t*>(st + 4 * TILE);
        uint8_t* sc = st + 6 * TILE;
        const int q = ti.p >> 3;  // 8-element groups per block (p % 16 == 0)
        const float pf = static_cast<float>(ti.p);
        // a block whose groups all sit in one warp finishes in phase 1
        const bool seg = (q <= 32) && ((32 % q) == 0);
        const bool warp_part = !seg && (q % 32 == 0);
        auto finish = [&](int b, float g2, float mx) {
            if (MODE == kGradOnly) {
                sm.blk[b] = make_float2(0.0f, mx);
            } else {
                const float vn = fmaf(hp.beta2, sm.vold[b], hp.omb2 * (g2 / pf));
                P.v[ti.bo + b] = vn;
                P.scale[ti.bo + b] = mx;
                const float fac = hp.lr_bc1 / (sqrtf(vn * hp.inv_bc2) + hp.eps);
                sm.blk[b] = make_float2(fac, mx > 0.0f ? 1.0f / mx : 0.0f);
            }
        };

        // phase 1: decode m, partials over the thread's 8 elements
        const int e = tid * 8;
        const bool live = e < ti.nelem;
        const int b = static_cast<int>(__umulhi(static_cast<uint32_t>(e), ti.pmagic));
        float m[8];
        float g2 = 0.0f, mx = 0.0f;
        if (live) {
            const uint4 gw = *reinterpret_cast<const uint4*>(sg + e);
            const uint32_t gws[4] = {gw.x, gw.y, gw.z, gw.w};
            if (MODE == kGradOnly) {
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    m[2 * j] = bf16_lo(gws[j]);
                    m[2 * j + 1] = bf16_hi(gws[j]);
                }
#pragma unroll
                for (int j = 0; j < 8; ++j) mx = fmaxf(mx, fabsf(m[j]));
            } else {
                const uint2 cw = *reinterpret_cast<const uint2*>(sc + e);
                const float b1s = hp.beta1 * sm.sold[b];
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const float g = (j & 1) ? bf16_hi(gws[j >> 1]) : bf16_lo(gws[j >> 1]);
                    const uint32_t c = ((j < 4 ? cw.x : cw.y) >> (8 * (j & 3))) & 0xFFu;
                    const float mm = fmaf(hp.omb1, g, b1s * sm.tab.dec[c]);
                    m[j] = mm;
                    g2 = fmaf(g, g, g2);
                    mx = fmaxf(mx, fabsf(mm));
                }
            }
        }
        if (seg) {
            for (int o = q >> 1; o > 0; o >>= 1) {
                g2 += __shfl_xor_sync(0xffffffffu, g2, o);
                mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
            }
            if (live && (tid % q) == 0) finish(b, g2, mx);
        } else if (warp_part) {
            g2 = warp_sum(g2);
            mx = warp_max(mx);
            if (lane == 0) sm.part[tid >> 5] = make_float2(g2, mx);
        } else {
            sm.part[tid] = make_float2(g2, mx);
        }
        __syncthreads();
        if (!seg) {
            // remaining block reductions over the stored partials (fixed order)
            const int per = warp_part ? (q >> 5) : q;
            for (int bb = warp; bb < ti.nblk; bb += THREADS / 32) {
                float s2 = 0.0f, sx = 0.0f;
                for (int t = lane; t < per; t += 32) {
                    const float2 pp = sm.part[bb * per + t];
                    s2 += pp.x;
                    sx = fmaxf(sx, pp.y);
                }
                s2 = warp_sum(s2);
                sx = warp_max(sx);
                if (lane == 0) finish(bb, s2, sx);
            }
            __syncthreads();
        }

        // phase 2: update and re-encode into the stage, x to the staging buffer
        if (live) {
            const float2 bs = sm.blk[b];
            float x[8];
            if (MODE == kGradOnly) {
#pragma unroll
                for (int j = 0; j < 8; ++j) x[j] = bs.y > 0.0f ? __fdiv_rn(m[j], bs.y) : __int_as_float(0x7fffffff);
            } else {
                float4* tp = reinterpret_cast<float4*>(sth + e);
                float4 t0 = tp[0], t1 = tp[1];
                t0.x = fmaf(-bs.x, m[0], hp.decay * t0.x);
                t0.y = fmaf(-bs.x, m[1], hp.decay * t0.y);
                t0.z = fmaf(-bs.x, m[2], hp.decay * t0.z);
                t0.w = fmaf(-bs.x, m[3], hp.decay * t0.w);
                t1.x = fmaf(-bs.x, m[4], hp.decay * t1.x);
                t1.y = fmaf(-bs.x, m[5], hp.decay * t1.y);
                t1.z = fmaf(-bs.x, m[6], hp.decay * t1.z);
                t1.w = fmaf(-bs.x, m[7], hp.decay * t1.w);
                tp[0] = t0;
                tp[1] = t1;
                uint32_t w0 = 0, w1 = 0;
                if (bs.y > 0.0f) {
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        x[j] = m[j] * bs.y;
                        const uint32_t c = static_cast<uint32_t>(encode_lut(sm.tab, lut_ok, x[j]));
                        if (j < 4) w0 |= c << (8 * j); else w1 |= c << (8 * (j - 4));
                    }
                } else {
                    const uint32_t z = static_cast<uint32_t>(zero_code) * 0x01010101u;
                    w0 = w1 = z;
#pragma unroll
                    for (int j = 0; j < 8; ++j) x[j] = __int_as_float(0x7fffffff);
                }
                *reinterpret_cast<uint2*>(sc + e) = make_uint2(w0, w1);
            }
            if (MODE != kPlain) {
                float4* xs = reinterpret_cast<float4*>(P.xstage + ti.e0 + e);
                __stcs(xs, make_float4(x[0], x[1], x[2], x[3]));
                __stcs(xs + 1, make_float4(x[4], x[5], x[6], x[7]));
            }
        }
        if (MODE != kGradOnly) fence_proxy_async();
        __syncthreads();
        if (tid == 0) {
            if (MODE != kGradOnly) {
                const uint32_t n = static_cast<uint32_t>(ti.nelem);
                bulk_s2g(P.params + ti.e0, smem_u32(sth), 4u * n);
                bulk_s2g(P.codes + ti.e0, smem_u32(sc), n);
            }
            bulk_commit();
            // Refill the stage tile it-1 used with tile it+STAGES-1.  Its store
            // was committed an iteration ago: wait until only this tile's
            // store may still be reading shared memory.
            const int64_t un = u + static_cast<int64_t>(STAGES - 1) * G;
            if (un < L.nunits) {
                asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
                const int sn = (it + STAGES - 1) % STAGES;
                issue_tile<TILE, MODE>(sm.stage[sn], smem_u32(&sm.bar[sn]), tile_info(L, un), P);
            }
        }
    }
    if (tid == 0) bulk_wait_all();
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

template <int MODE>
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
                const uint4 cw = __ldcg(reinterpret_cast<const uint4*>(P.codes + e));
#pragma unroll
                for (int t = 0; t < 16; ++t) {
                    const float mm = fmaf(hp.omb1, g[t], b1s * s_dec[byte_of(cw, t)]);
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

// p <= 4096: two 512-thread CTAs per SM, 3-stage rings of 28 KB tiles;
// p <= 8192: one 1024-thread CTA per SM, 3-stage ring of 56 KB tiles
constexpr int kS4KTile = 4096, kS4KThreads = 512, kS4KStages = 3, kS4KMinBlocks = 2;
constexpr int kS8KTile = 8192, kS8KThreads = 1024, kS8KStages = 3, kS8KMinBlocks = 1;

PathClass classify(int64_t p) {
    if (p == 1) return kP1;
    if (p % 16 == 0 && p <= kS4KTile) return kS4K;
    if (p % 16 == 0 && p <= kS8KTile) return kS8K;
    if (p % 16 == 0 && p <= kTile16Max) return kT16V4;
    if (p <= kGenericTile) return kGeneric;
    return (p % 16 == 0) ? kBigAligned : kBigUnaligned;
}

int64_t units_of(PathClass c, const gefen_tensor_t& t, int64_t* per_unit, int64_t tile_cap = 0) {
    const int64_t p = t.period, nb = t.numel / p;
    if (tile_cap > 0) {  // streamed classes: whole blocks per tile of the kernel's own size
        *per_unit = std::max<int64_t>(1, tile_cap / p);
        return (nb + *per_unit - 1) / *per_unit;
    }
    switch (c) {
        case kP1:
            *per_unit = 1;
            return (t.numel + 4 * kThreads - 1) / (4 * kThreads);
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
                         PathClass c, int64_t tile_cap = 0) {
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
            units += units_of(c, x, &s.per_unit, tile_cap);
        }
        L.nunits = units;
        if (units == 0) continue;
        kernel(L, units);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

template <int TILE, int THREADS, int STAGES, int MINB, int MODE>
cudaError_t launch_stream(Launch& L, const std::vector<int>& ids, const gefen_tensor_t* t, PathClass c,
                          const Ptrs& P, int* err, cudaStream_t st) {
    auto kern = k_step_stream<TILE, THREADS, STAGES, MODE, MINB>;
    const int smem = static_cast<int>(sizeof(StreamSmem<TILE, THREADS, STAGES>));
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, THREADS, smem);
    if (e != cudaSuccess) return e;
    const int64_t cap = static_cast<int64_t>(std::max(1, per_sm)) * device_sm_count();
    return launch_class(
        [&](Launch& LL, int64_t u) {
            kern<<<dim3(static_cast<unsigned>(std::min(u, cap))), THREADS, smem, st>>>(LL, P, err);
        },
        L, ids, t, c, TILE);
}

template <int MODE>
cudaError_t run_step(const Plan& pl, const gefen_tensor_t* t, Launch& L, const Ptrs& P, int* err, cudaStream_t st) {
    cudaError_t e;
    e = launch_class([&](Launch& LL, int64_t u) { k_step_p1<MODE><<<dim3(u), kThreads, 0, st>>>(LL, P); },
                     L, pl.idx[kP1], t, kP1);
    if (e != cudaSuccess) return e;
    e = launch_stream<kS4KTile, kS4KThreads, kS4KStages, kS4KMinBlocks, MODE>(L, pl.idx[kS4K], t, kS4K, P, err, st);
    if (e != cudaSuccess) return e;
    e = launch_stream<kS8KTile, kS8KThreads, kS8KStages, kS8KMinBlocks, MODE>(L, pl.idx[kS8K], t, kS8K, P, err, st);
    if (e != cudaSuccess) return e;
    e = launch_class([&](Launch& LL, int64_t u) { k_step_tile16<4, MODE><<<dim3(u), kThreads, 0, st>>>(LL, P); },
                     L, pl.idx[kT16V4], t, kT16V4);
    if (e != cudaSuccess) return e;
    e = launch_class([&](Launch& LL, int64_t u) { k_step_generic<MODE><<<dim3(u), kThreads, 0, st>>>(LL, P); },
                     L, pl.idx[kGeneric], t, kGeneric);
    if (e != cudaSuccess) return e;
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
            k_big_partial<MODE><<<dim3(units), kThreads, 0, st>>>(L, P, aligned);
            k_big_finalize<MODE><<<dim3(blocks), kThreads, 0, st>>>(L, P);
            k_big_apply<MODE><<<dim3(units), kThreads, 0, st>>>(L, P, aligned);
            if ((e = cudaGetLastError()) != cudaSuccess) return e;
        }
    }
    return cudaSuccess;
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
    if (flags & ~(GEFEN_HIST | GEFEN_HIST_GRAD_ONLY)) return GEFEN_EINVAL;
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
    if (grad_only) e = run_step<kGradOnly>(pl, tensors, L, P, err, st);
    else if (flags & GEFEN_HIST) e = run_step<kHist>(pl, tensors, L, P, err, st);
    else e = run_step<kPlain>(pl, tensors, L, P, err, st);
    if (e != cudaSuccess) return GEFEN_ECUDA;
    if (want_hist) {
        std::vector<HistRange> rr;
        for (int i = 0; i < ntensors; ++i)
            if (tensors[i].numel > 0) rr.push_back({tensors[i].offset, tensors[i].numel});
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
