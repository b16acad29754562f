// Shared part of the step kernels (gefen_step, Algorithm 1's loop body):
// the launch and pointer records, the storage formats, device helpers and the
// streamed-tile kernel (k_step_stream).  The streamed kernel's instances are
// compiled in several translation units (step_s4k.cu, step_s4k_modes.cu,
// step_s8k.cu, step_big.cu), each behind one launcher declared here, so that
// they build in parallel; step.cu plans the launches and holds the other
// step kernels.
#pragma once

#include <algorithm>
#include <cstdint>

#include <cuda_bf16.h>

#include "common.cuh"
#include "internal.h"

namespace gefen {
namespace stepk {

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
// shared memory.  To make room, the 4096 tiles run two stages and keep the
// decode table in 4 copies (the cell records keep 8: a refit step 2% faster
// than with three stages and the records in 4), and the 8192 tiles read
// theta from global memory (an L2 hit after the issuing thread's prefetch)
// instead of staging it: 8 copies of each table fit then, and a refit step's
// 8192 tiles ran 6% faster than with theta staged and the tables in 2 and 4
// copies.
constexpr int kFusedBins = 4096;
using S4KHistCfg = StreamCfg<4096, 256, 2, 8, 4, false, 2>;
using S8KHistCfg = StreamCfg<8192, 512, 2, 8, 8, false, 1>;
constexpr int kS4KTile = S4KCfg::TILE, kS8KTile = S8KCfg::TILE;

// Block shapes a streamed launch serves (every segment of the launch has one):
// blocks of whole warps' slices (p % 512 == 0), blocks of 16 to 256
// elements (a power of two), or any p % 16 == 0 up to the tile.
constexpr int kShapeAny = 0, kShapeWarp = 1, kShapeSub = 2;

inline int shape_of(int64_t p) {
    if (p % 512 == 0) return kShapeWarp;
    if (p >= 16 && p <= 256 && (p & (p - 1)) == 0) return kShapeSub;
    return kShapeAny;
}

// Launchers of the streamed kernel.  hb: cells counted in shared memory (0 or
// kFusedBins); shape: kShapeWarp, kShapeSub or kShapeAny; fmt: storage format.
cudaError_t stream_s4k_plain(int fmt, int shape, const Launch& L, const Ptrs& P, int* err, cudaStream_t st);
cudaError_t stream_s4k_modes(int mode, int hb, int fmt, int shape, const Launch& L, const Ptrs& P, int* err,
                             cudaStream_t st);
cudaError_t stream_s8k(int mode, int hb, int fmt, int shape, const Launch& L, const Ptrs& P, int* err,
                       cudaStream_t st);
// Tiles of big blocks with finalised factors (4096-element tiles).
cudaError_t stream_big(int mode, int hb, int fmt, const Launch& L, const Ptrs& P, int* err, cudaStream_t st);

}  // namespace stepk

namespace {

using namespace stepk;

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
// increasing unit order, so its segment cursor only grows.  BIG: a launch
// over tiles of big blocks.
template <bool BIG>
__device__ __forceinline__ TileInfo tile_info(const Launch& L, int64_t unit, int& seg) {
    while (seg + 1 < L.nseg && L.seg[seg + 1].unit_begin <= unit) ++seg;
    const Seg& S = L.seg[seg];
    const int64_t p = S.period;
    TileInfo ti;
    ti.rp = 0.0f;
    if (BIG && (S.flags & kSegBigTiles)) {
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
template <int NG, bool BIG>
__device__ __forceinline__ void load_state(const Ptrs& P, const TileInfo& ti, int eb, float (&s)[NG], float (&v)[NG]) {
    if (BIG && ti.ext) {  // a big block: s before the step was kept by its finalisation
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
template <int TILE, int THREADS, int LUTR, int DECR, int MODE, bool THS, int FMT, bool LUT, bool FULL, bool BIG,
          int SHAPE, typename Smem>
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
    if constexpr (BIG) {
        // a tile of a big block: v, s and the step factor were finalised
        const float4 bs = P.blk_state[ti.bo];  // (s before, s after, step factor, -)
        const float iv = (MODE == kGradOnly) ? bs.y : (bs.y > 0.0f ? __frcp_rn(bs.y) : 0.0f);
#pragma unroll
        for (int j = 0; j < 4; ++j) { fac[j] = bs.z; inv[j] = iv; }
    } else if (SHAPE != kShapeSub && (p & 511) == 0) {
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
    } else if (SHAPE != kShapeWarp && p == 256) {
        // groups 0,1 and 2,3 form one block each
        const float s0 = warp_sum_bfly(g2[0] + g2[1]), x0 = warp_max_nonneg(fmaxf(mx[0], mx[1]));
        const float s1 = warp_sum_bfly(g2[2] + g2[3]), x1 = warp_max_nonneg(fmaxf(mx[2], mx[3]));
        finish(s0, x0, r_v[0], ti.bo + blk[0], live[0] && lane == 0, fac[0], inv[0]);
        finish(s1, x1, r_v[2], ti.bo + blk[2], live[2] && lane == 0, fac[2], inv[2]);
        fac[1] = fac[0]; inv[1] = inv[0];
        fac[3] = fac[2]; inv[3] = inv[2];
    } else if (SHAPE != kShapeWarp && (p & (p - 1)) == 0) {
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
    } else if (SHAPE == kShapeAny) {
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

template <int TILE, int THREADS, int STAGES, int LUTR, int DECR, int MODE, bool THS, int FMT, bool LUT, bool BIG,
          int SHAPE, typename Smem>
__device__ __forceinline__ void stream_loop(Smem& sm, const Launch& L, const Ptrs& P, int* err, int seg) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t G = gridDim.x;
    const int eb = warp * 512 + lane * 4;  // first element of the thread's group 0 within a tile

    float r_s[4] = {0.0f, 0.0f, 0.0f, 0.0f}, r_v[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    if (MODE != kGradOnly && blockIdx.x < L.nunits) load_state<4, BIG>(P, sm.tile[0], eb, r_s, r_v);

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
        if (STAGES >= 3 && tid == 0 && un < L.nunits) sm.next = tile_info<BIG>(L, un, seg);
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
            load_state<4, BIG>(P, sm.tile[(it + 1) % STAGES], eb, n_s, n_v);

        if (ti.nelem == TILE)
            stream_tile<TILE, THREADS, LUTR, DECR, MODE, THS, FMT, LUT, true, BIG, SHAPE>(sm, P, L.hp, ti, sm.stage[s], eb, r_s, r_v,
                                                                                th);
        else
            stream_tile<TILE, THREADS, LUTR, DECR, MODE, THS, FMT, LUT, false, BIG, SHAPE>(sm, P, L.hp, ti, sm.stage[s], eb, r_s,
                                                                                 r_v, th);

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
            if (STAGES < 3) sm.next = tile_info<BIG>(L, un, seg);
            issue_tile<TILE, MODE, THS, FMT>(sm, s, sm.next, P);
        }
        if (STAGES < 3 && MODE != kGradOnly && u + G < L.nunits)
            load_state<4, BIG>(P, sm.tile[(it + 1) % STAGES], eb, n_s, n_v);
#pragma unroll
        for (int j = 0; j < 4; ++j) { r_s[j] = n_s[j]; r_v[j] = n_v[j]; }
    }
}

// BIG: a launch over the tiles of big blocks (factors finalised beforehand);
// SHAPE: the block shapes of the launch's other tiles (kShapeWarp, kShapeSub
// or kShapeAny).  A launch carries code for its own tiles only.
template <int TILE, int THREADS, int STAGES, int LUTR, int DECR, bool THS, int HB, int FMT, int MODE, int MINB, bool BIG,
          int SHAPE>
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
            if (u < L.nunits) issue_tile<TILE, MODE, THS, FMT>(sm, s, tile_info<BIG>(L, u, seg), P);
        }
    }
    if (HB > 0)
        for (int i = threadIdx.x; i < HB; i += THREADS) sm.hist[i] = 0u;
    const int bad = build_tables<THREADS>(P, sm.tab, MODE == kGradOnly);
    const bool lut_ok = !__syncthreads_or(bad);
    if (MODE != kGradOnly && lut_ok)
        stream_loop<TILE, THREADS, STAGES, LUTR, DECR, MODE, THS, FMT, true, BIG, SHAPE>(sm, L, P, err, seg);
    else
        stream_loop<TILE, THREADS, STAGES, LUTR, DECR, MODE, THS, FMT, false, BIG, SHAPE>(sm, L, P, err, seg);
    if (HB > 0) {
        // add the CTA's counts to the histogram
        __syncthreads();
        for (int c = threadIdx.x; c < P.bins; c += THREADS) {
            const uint32_t n = sm.hist[c];
            if (n) atomicAdd(reinterpret_cast<unsigned long long*>(P.hist) + c, static_cast<unsigned long long>(n));
        }
    }
}

// One launch of the streamed kernel over the units of a prepared Launch.
template <typename C, int MODE, int HB, int FMT, bool BIG, int SHAPE>
cudaError_t stream_kernel(const Launch& L, const Ptrs& P, int* err, cudaStream_t st) {
    auto kern = k_step_stream<C::TILE, C::THREADS, C::STAGES, C::LUTR, C::DECR, C::THS, HB, FMT, MODE, C::MINB, BIG, SHAPE>;
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

// Dispatch of a launch's storage format and block shapes to an instance.
// SUB: the class has blocks of 16 to 256 elements.
template <typename C, int MODE, int HB, bool BIG, int FMT, bool SUB>
cudaError_t stream_by_shape(int shape, const Launch& L, const Ptrs& P, int* err, cudaStream_t st) {
    if (shape == kShapeWarp) return stream_kernel<C, MODE, HB, FMT, BIG, kShapeWarp>(L, P, err, st);
    if constexpr (SUB) {
        if (shape == kShapeSub) return stream_kernel<C, MODE, HB, FMT, BIG, kShapeSub>(L, P, err, st);
    }
    return stream_kernel<C, MODE, HB, FMT, BIG, kShapeAny>(L, P, err, st);
}
template <typename C, int MODE, int HB, bool BIG, bool SUB>
cudaError_t stream_by_fmt_shape(int fmt, int shape, const Launch& L, const Ptrs& P, int* err, cudaStream_t st) {
    switch (fmt) {
        case 0: return stream_by_shape<C, MODE, HB, BIG, 0, SUB>(shape, L, P, err, st);
        case 1: return stream_by_shape<C, MODE, HB, BIG, 1, SUB>(shape, L, P, err, st);
        case 2: return stream_by_shape<C, MODE, HB, BIG, 2, SUB>(shape, L, P, err, st);
        case 3: return stream_by_shape<C, MODE, HB, BIG, 3, SUB>(shape, L, P, err, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace

}  // namespace gefen
