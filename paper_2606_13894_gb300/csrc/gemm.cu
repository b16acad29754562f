// Matrix products of Gefen-Muon's Newton-Schulz iteration (the paper's
// appendix "Gefen-Muon"), on sm_103a:
//
//   C = alpha * A * B^T + beta * D      A: M x K, B: N x K, C, D: M x N
//
// all row-major (K contiguous in A and B), written as C and/or as its
// transpose CT (N x M).
//
// bf16 storage, fp32 accumulation: a persistent tcgen05 kernel, one CTA per
// SM taking 128 x BN tiles of C (BN 256, or 128 when there are too few
// tiles).  Warp 0 loads 128 x 64 k-tiles of A and BN x 64 of B with TMA
// (128-byte swizzle) into a ring of shared-memory stages; warp 1 issues
// tcgen05.mma (M 128, N BN, K 16; four per stage) into one of two tensor-memory
// accumulators and frees each stage with tcgen05.commit; warps 2-5 read the
// other accumulator with tcgen05.ld, apply alpha and beta * D and store C, and
// CT through a per-warp transpose buffer, while the next tile accumulates.
// A symmetric product (A = X X^T and c A A^T + b A in Newton-Schulz) computes
// only the tiles on or above the diagonal and writes each element twice, so
// its result is exactly symmetric.  Every wait on an mbarrier gives up after
// about a second and flags the error word instead.
//
// Any other case (fp32 storage, or leading dimensions that TMA cannot
// address): a tiled CUDA-core kernel with fp32 arithmetic.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace gefen {

namespace {

constexpr int kBM = 128, kBK = 64;
constexpr long long kSpin = 1ll << 31;

__device__ __forceinline__ uint32_t saddr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
// Waits for the phase with this parity; false after about kSpin cycles.
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
        if (clock64() - t0 > kSpin) return false;
    }
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int c0, int c1, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
        : "memory");
}

// Shared-memory matrix descriptor of a K-major operand tile stored as TMA's
// 128-byte swizzle writes it: rows of 64 bf16 (128 B), eight-row swizzle
// atoms 1024 B apart (the stride offset); the leading offset is not used by
// this layout; bits 46-47 carry the descriptor version, 61-63 the swizzle.
__device__ __forceinline__ uint64_t desc_sw128(uint32_t addr) {
    uint64_t d = static_cast<uint64_t>((addr & 0x3FFFFu) >> 4);
    d |= static_cast<uint64_t>(1) << 16;            // leading byte offset 16 B (unused)
    d |= static_cast<uint64_t>(1024 >> 4) << 32;    // stride byte offset
    d |= static_cast<uint64_t>(1) << 46;            // version
    d |= static_cast<uint64_t>(2) << 61;            // 128-byte swizzle
    return d;
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}
// TMA store of a 32 x 32 bf16 block from shared memory to global (x: column,
// y: row of the tensor map's matrix); out-of-range parts are not written.
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, uint32_t src, int x, int y) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(x), "r"(y), "r"(src)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// Until at most one committed store group is still reading shared memory.
__device__ __forceinline__ void bulk_wait_read1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }
// Until every committed store group has completed.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// Generic-proxy writes to shared memory become visible to the TMA unit.
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 32 consecutive fp32 accumulator columns of the calling thread's row.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr)
        : "memory");
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

struct GemmArgs {
    int M, N, K;
    float alpha, beta;
    const __nv_bfloat16* D;
    int ldd;
    __nv_bfloat16* C;
    int ldc;
    __nv_bfloat16* CT;
    int ldct;
    int sym;  // C is symmetric (M == N): only tiles on or above the diagonal are computed, each written twice
    int nfull;  // tiles taken whole; the rest (a last, partial wave) as two halves of BN / 2 columns each
    int* err;
};

// Per tile width BN: ring depth, bytes per stage, tensor-memory columns (two
// accumulators, so the epilogue of one tile overlaps the next tile's MMAs).
template <int BN>
struct TcCfg {
    static constexpr int kStagesN = BN == 256 ? 4 : 6;
    static constexpr uint32_t kTileAB = kBM * kBK * 2, kTileBB = BN * kBK * 2;
    static constexpr uint32_t kCols = 2 * BN;
    // kind::f16 instruction descriptor: fp32 accumulator, bf16 A and B, both
    // K-major, N / 8 at bit 17, M / 16 at bit 24
    static constexpr uint32_t kIdescN = (1u << 4) | (1u << 7) | (1u << 10) |
                                        (static_cast<uint32_t>(BN >> 3) << 17) |
                                        (static_cast<uint32_t>(kBM >> 4) << 24);
    // the same with N = BN / 2 (half tiles)
    static constexpr uint32_t kIdescHalf = (1u << 4) | (1u << 7) | (1u << 10) |
                                           (static_cast<uint32_t>(BN >> 4) << 17) |
                                           (static_cast<uint32_t>(kBM >> 4) << 24);
};

template <int BN>
struct alignas(1024) TcSmem {
    using C = TcCfg<BN>;
    unsigned char a[C::kStagesN][C::kTileAB];  // 1024-byte aligned tiles (swizzle atoms)
    unsigned char b[C::kStagesN][C::kTileBB];
    // per epilogue warp, two buffers each: a 32 x 32 block of C and of its
    // transpose, row-major, as the TMA stores read them
    __nv_bfloat16 stc[4][2][32][32];
    __nv_bfloat16 stt[4][2][32][32];
    unsigned long long full[C::kStagesN], empty[C::kStagesN], acc_full[2], acc_empty[2];
    uint32_t tmem;
    int abort;
    int consumed;  // k-tiles the MMA issuer took from the ring
};

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void umma_bf16_n(uint32_t tmem, uint64_t da, uint64_t db, uint32_t idesc,
                                            uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem),
        "l"(da), "l"(db), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Tile t of the CTA's schedule: (m block, n block).  Symmetric products take
// the tiles with m block <= n block only (BN == BM), n block by n block.
__device__ __forceinline__ void tile_of(int t, int ntm, bool sym, int& mb, int& nb) {
    if (!sym) {
        mb = t % ntm;
        nb = t / ntm;
        return;
    }
    int j = static_cast<int>((sqrtf(8.0f * static_cast<float>(t) + 1.0f) - 1.0f) * 0.5f);
    while (j * (j + 1) / 2 > t) --j;
    while ((j + 1) * (j + 2) / 2 <= t) ++j;
    nb = j;
    mb = t - j * (j + 1) / 2;
}

// Two bf16 (round to nearest even) in one word, the first in the low half.
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&h);
}

// Row `row` of D, columns col0 .. col0 + 31 as bf16 pairs (zero outside D).
__device__ __forceinline__ void load_d(uint32_t (&d)[16], const GemmArgs& G, int row, int col0) {
    if (row < G.M && col0 + 32 <= G.N) {
        const uint4* p = reinterpret_cast<const uint4*>(G.D + static_cast<int64_t>(row) * G.ldd + col0);
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) {
            const uint4 w = __ldg(p + qq);
            d[4 * qq] = w.x;
            d[4 * qq + 1] = w.y;
            d[4 * qq + 2] = w.z;
            d[4 * qq + 3] = w.w;
        }
    } else {
        const unsigned short* p = reinterpret_cast<const unsigned short*>(G.D) + static_cast<int64_t>(row) * G.ldd;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int c = col0 + 2 * j;
            const uint32_t lo = (row < G.M && c < G.N) ? p[c] : 0u;
            const uint32_t hi = (row < G.M && c + 1 < G.N) ? p[c + 1] : 0u;
            d[j] = lo | (hi << 16);
        }
    }
}

// Work item `it` of the schedule: a whole tile (it < nfull, and every tile of
// a symmetric product) or one half of a tile of the last wave, BN / 2 columns
// wide.  Gives its row block, first column and width.
template <int BN>
__device__ __forceinline__ void item_of(int it, int ntm, bool sym, int nfull, int& mb, int& n0, int& ncols) {
    int nb;
    if (sym || it < nfull) {
        tile_of(it, ntm, sym, mb, nb);
        n0 = nb * BN;
        ncols = BN;
    } else {
        const int h = it - nfull;
        tile_of(nfull + (h >> 1), ntm, false, mb, nb);
        n0 = nb * BN + (h & 1) * (BN / 2);
        ncols = BN / 2;
    }
}

constexpr int kTcThreads = 192;  // warp 0: TMA, warp 1: MMA, warps 2-5: epilogue

// Persistent tcgen05 GEMM: each CTA takes tiles blockIdx.x, + gridDim.x, ...
template <int BN>
__global__ void __launch_bounds__(kTcThreads, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
              const __grid_constant__ CUtensorMap mapBh, const __grid_constant__ CUtensorMap mapC,
              const __grid_constant__ CUtensorMap mapCT, const GemmArgs G) {
    using Cf = TcCfg<BN>;
    constexpr int S = Cf::kStagesN;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    // aligned to 1024 bytes here: the launch asks for 1024 bytes of slack
    TcSmem<BN>& sm = *reinterpret_cast<TcSmem<BN>*>(smem_raw + ((1024 - (saddr(smem_raw) & 1023)) & 1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int KT = (G.K + kBK - 1) / kBK;
    const int ntm = (G.M + kBM - 1) / kBM, ntn = (G.N + BN - 1) / BN;
    const bool sym = G.sym != 0;
    const int ntiles = sym ? ntn * (ntn + 1) / 2 : ntm * ntn;
    const int nfull = sym ? ntiles : G.nfull;
    const int nitems = nfull + 2 * (ntiles - nfull);

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(saddr(&sm.full[s]), 1);
            mbar_init(saddr(&sm.empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(saddr(&sm.acc_full[b]), 1);
            mbar_init(saddr(&sm.acc_empty[b]), 4);  // one arrival per epilogue warp
        }
        sm.abort = 0;
        sm.consumed = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapA)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapB)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapBh)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapC)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapCT)) : "memory");
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(saddr(&sm.tmem)),
                     "r"(Cf::kCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sm.tmem;
    volatile int* abort = &sm.abort;
    // Launched as a programmatic dependent of the previous kernel on the
    // stream: everything above overlapped its end; the operands (and the
    // buffers written) may be that kernel's, so wait for it to complete.
    // Then let the next product start its own prologue.
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    int issued = 0;  // thread 0: k-tiles whose loads were started
    if (threadIdx.x == 0) {
        // producer: the A and B k-tiles of every tile of this CTA, in order
        int ring = 0;
        for (int t = blockIdx.x; t < nitems && !*abort; t += gridDim.x) {
            int mb, n0, ncols;
            item_of<BN>(t, ntm, sym, nfull, mb, n0, ncols);
            const bool whole = ncols == BN;
            for (int kt = 0; kt < KT; ++kt, ++ring) {
                const int s = ring % S;
                if (ring >= S && !mbar_wait(saddr(&sm.empty[s]), static_cast<uint32_t>((ring / S - 1) & 1))) {
                    atomicExch(&sm.abort, 1);
                    break;
                }
                const uint32_t bar = saddr(&sm.full[s]);
                mbar_expect_tx(bar, Cf::kTileAB + (whole ? Cf::kTileBB : Cf::kTileBB / 2));
                tma_load_2d(saddr(sm.a[s]), &mapA, kt * kBK, mb * kBM, bar);
                tma_load_2d(saddr(sm.b[s]), whole ? &mapB : &mapBh, kt * kBK, n0, bar);
                issued = ring + 1;
            }
        }
    } else if (threadIdx.x == 32) {
        // MMA issuer: accumulator b = i & 1 for the CTA's i-th tile, reused
        // once the epilogue has drained it
        int ring = 0, i = 0;
        for (int t = blockIdx.x; t < nitems && !*abort; t += gridDim.x, ++i) {
            const uint32_t idesc = (sym || t < nfull) ? Cf::kIdescN : Cf::kIdescHalf;
            const int b = i & 1;
            if (i >= 2 && !mbar_wait(saddr(&sm.acc_empty[b]), static_cast<uint32_t>(((i >> 1) - 1) & 1))) {
                atomicExch(&sm.abort, 1);
                break;
            }
            tc_fence_after();
            const uint32_t acc = tmem + static_cast<uint32_t>(b * BN);
            bool ok = true;
            for (int kt = 0; kt < KT; ++kt, ++ring) {
                const int s = ring % S;
                if (!mbar_wait(saddr(&sm.full[s]), static_cast<uint32_t>((ring / S) & 1))) {
                    atomicExch(&sm.abort, 1);
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t a0 = saddr(sm.a[s]), b0 = saddr(sm.b[s]);
#pragma unroll
                for (int kk = 0; kk < kBK / 16; ++kk)
                    umma_bf16_n(acc, desc_sw128(a0 + kk * 32), desc_sw128(b0 + kk * 32), idesc,
                                (kt | kk) != 0 ? 1u : 0u);
                umma_commit(saddr(&sm.empty[s]));
            }
            umma_commit(saddr(&sm.acc_full[b]));  // arrives once this tile's MMAs have completed
            if (!ok) break;
        }
        sm.consumed = ring;
    } else if (warp >= 2) {
        // epilogue: this warp reads accumulator rows 32 q .. 32 q + 31 (the
        // TMEM lanes of warp id % 4), 32 columns at a time: a 32 x 32 block
        // that it stages in shared memory, as C and as its transpose, and
        // writes with TMA stores.  In a symmetric product a block above the
        // diagonal is stored at its place and mirrored; a block on the
        // diagonal takes its upper triangle for both halves; a block below
        // it is left to the mirror of the block above.
        const int q = warp & 3, e = warp - 2;
        const bool hasC = G.C != nullptr, hasT = sym || G.CT != nullptr;
        const bool useD = G.beta != 0.0f && G.D != nullptr;
        int nst = 0;  // blocks this warp has staged (their buffer alternates)
        int i = 0;
        for (int t = blockIdx.x; t < nitems; t += gridDim.x, ++i) {
            const int b = i & 1;
            const bool ok = mbar_wait(saddr(&sm.acc_full[b]), static_cast<uint32_t>((i >> 1) & 1));
            tc_fence_after();
            if (!__all_sync(0xffffffffu, ok) || *abort) {
                atomicExch(&sm.abort, 1);
                break;
            }
            int mb, n0, ncols;
            item_of<BN>(t, ntm, sym, nfull, mb, n0, ncols);
            const int i0 = mb * kBM + 32 * q, row = i0 + lane;
            // first column block of this warp: in a symmetric product the
            // blocks left of the diagonal are skipped
            const int cfirst = sym ? max(0, i0 - n0) : 0;
            uint32_t dn[16];  // D of the next block, loaded one block ahead
            if (useD) load_d(dn, G, row, n0 + cfirst);
            for (int c0 = cfirst; c0 < ncols; c0 += 32) {
                const int col0 = n0 + c0;
                uint32_t dc[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) dc[j] = dn[j];
                if (useD && c0 + 32 < ncols) load_d(dn, G, row, col0 + 32);
                float v[32];
                tmem_ld32(tmem + static_cast<uint32_t>(b * BN + c0) + (static_cast<uint32_t>(32 * q) << 16), v);
                if (useD) {
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        v[2 * j] = G.alpha * v[2 * j] + G.beta * __uint_as_float(dc[j] << 16);
                        v[2 * j + 1] = G.alpha * v[2 * j + 1] + G.beta * __uint_as_float(dc[j] & 0xFFFF0000u);
                    }
                } else {
#pragma unroll
                    for (int k = 0; k < 32; ++k) v[k] *= G.alpha;
                }
                const bool ondiag = sym && col0 == i0;
                const int p = nst & 1;
                __nv_bfloat16(*bc)[32] = sm.stc[e][p];
                __nv_bfloat16(*bt)[32] = sm.stt[e][p];
                // the stores that last read buffer p have finished reading it
                if (lane == 0) bulk_wait_read1();
                __syncwarp();
                if (hasC) {
#pragma unroll
                    for (int qq = 0; qq < 4; ++qq) {
                        uint4 w;
                        w.x = pack_bf16(v[8 * qq], v[8 * qq + 1]);
                        w.y = pack_bf16(v[8 * qq + 2], v[8 * qq + 3]);
                        w.z = pack_bf16(v[8 * qq + 4], v[8 * qq + 5]);
                        w.w = pack_bf16(v[8 * qq + 6], v[8 * qq + 7]);
                        *reinterpret_cast<uint4*>(&bc[lane][8 * qq]) = w;
                    }
                }
                if (hasT) {
#pragma unroll
                    for (int k = 0; k < 32; ++k) bt[k][lane] = __float2bfloat16_rn(v[k]);
                }
                if (ondiag) {
                    // row lane, columns left of the diagonal: the transpose
                    __syncwarp();
                    for (int k = 0; k < lane; ++k) bc[lane][k] = bt[lane][k];
                }
                fence_async_smem();
                __syncwarp();
                if (lane == 0) {
                    if (hasC) tma_store_2d(&mapC, saddr(&bc[0][0]), col0, i0);
                    if (hasT && !ondiag) tma_store_2d(&mapCT, saddr(&bt[0][0]), i0, col0);
                    bulk_commit();
                }
                ++nst;
            }
            // this accumulator is drained: the MMA issuer may reuse it
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(saddr(&sm.acc_empty[b]));
        }
        // every store of this warp has completed before the CTA exits
        if (lane == 0) bulk_wait_all();
    }
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (*abort) {
        if (threadIdx.x == 0) {
            atomicExch(G.err, 1);
            // wait (bounded) for the loads still in flight
            for (int k = sm.consumed; k < issued; ++k)
                mbar_wait(saddr(&sm.full[k % S]), static_cast<uint32_t>((k / S) & 1));
        }
    }
    if (warp == 0) {
        __syncwarp();
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(Cf::kCols)
                     : "memory");
    }
}

// ------------------------------------------------- CUDA-core fallback
// 64 x 64 tiles, 256 threads with 4 x 4 results each, K in steps of 16
// through shared memory; fp32 arithmetic on fp32 or bf16 storage.
template <typename T>
__device__ __forceinline__ float ld_f(const T* p) {
    if constexpr (sizeof(T) == 2) return __bfloat162float(*reinterpret_cast<const __nv_bfloat16*>(p));
    else return *p;
}
template <typename T>
__device__ __forceinline__ void st_f(T* p, float v) {
    if constexpr (sizeof(T) == 2) *reinterpret_cast<__nv_bfloat16*>(p) = __float2bfloat16_rn(v);
    else *p = v;
}

template <typename T>
__global__ void __launch_bounds__(256) k_gemm_simt(int M, int N, int K, float alpha, const T* __restrict__ A, int lda,
                                                  const T* __restrict__ B, int ldb, float beta, const T* D, int ldd,
                                                  T* C, int ldc, T* CT, int ldct) {
    __shared__ float As[16][64 + 4], Bs[16][64 + 4];
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
    float acc[4][4] = {};
    for (int k0 = 0; k0 < K; k0 += 16) {
        for (int i = threadIdx.x; i < 64 * 16; i += 256) {
            const int rr = i >> 4, kk = i & 15;
            const int ra = m0 + rr, rb = n0 + rr, k = k0 + kk;
            As[kk][rr] = (ra < M && k < K) ? ld_f(A + static_cast<int64_t>(ra) * lda + k) : 0.0f;
            Bs[kk][rr] = (rb < N && k < K) ? ld_f(B + static_cast<int64_t>(rb) * ldb + k) : 0.0f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < 16; ++kk) {
            float a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                a[i] = As[kk][ty + 16 * i];
                b[i] = Bs[kk][tx + 16 * i];
            }
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int row = m0 + ty + 16 * i;
        if (row >= M) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int col = n0 + tx + 16 * j;
            if (col >= N) continue;
            float v = alpha * acc[i][j];
            if (beta != 0.0f && D != nullptr) v += beta * ld_f(D + static_cast<int64_t>(row) * ldd + col);
            if (C != nullptr) st_f(C + static_cast<int64_t>(row) * ldc + col, v);
            if (CT != nullptr) st_f(CT + static_cast<int64_t>(col) * ldct + row, v);
        }
    }
}

// cuTensorMapEncodeTiled from the driver, looked up once.
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static std::once_flag once;
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
        else
            (void)cudaGetLastError();
    });
    return fn;
}

// TMA map of a row-major rows x cols bf16 matrix (leading dimension ld).
// Operands: box 64 columns x box_rows rows, 128-byte swizzle, zero fill out
// of range.  Results (box_rows 0): box 32 x 32, no swizzle.
bool make_map(CUtensorMap* map, const void* base, int rows, int cols, int ld, int box_rows) {
    const auto fn = encode_fn();
    if (!fn) return false;
    const bool operand = box_rows > 0;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(operand ? kBK : 32),
                               static_cast<cuuint32_t>(operand ? box_rows : 32)};
    const cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, operand ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
              operand ? CU_TENSOR_MAP_L2_PROMOTION_L2_256B : CU_TENSOR_MAP_L2_PROMOTION_NONE,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// A bf16 matrix that TMA can address: 16-byte aligned base and row stride.
bool tma_ok(const void* p, int ld) { return p == nullptr || (ld % 8 == 0 && (reinterpret_cast<uintptr_t>(p) & 15u) == 0); }

}  // namespace

bool gemm_tc_usable(int lda, int ldb, const void* A, const void* B) {
    // TMA: 16-byte aligned bases and row strides
    return lda % 8 == 0 && ldb % 8 == 0 && (reinterpret_cast<uintptr_t>(A) & 15u) == 0 &&
           (reinterpret_cast<uintptr_t>(B) & 15u) == 0 && encode_fn() != nullptr;
}

static_assert(sizeof(TcSmem<128>) + 1024 <= 232448 && sizeof(TcSmem<256>) + 1024 <= 232448,
              "shared memory per CTA");

template <int BN>
cudaError_t launch_tc(const CUtensorMap& ma, const CUtensorMap& mb, const CUtensorMap& mbh, const CUtensorMap& mc,
                      const CUtensorMap& mct, GemmArgs G, cudaStream_t st) {
    const int smem = static_cast<int>(sizeof(TcSmem<BN>)) + 1024;
    cudaError_t e = cudaFuncSetAttribute(k_gemm_tc<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const int ntm = (G.M + kBM - 1) / kBM, ntn = (G.N + BN - 1) / BN;
    const int ntiles = G.sym ? ntn * (ntn + 1) / 2 : ntm * ntn;
    const int sms = device_sm_count();
    // a last wave that fills at most half the SMs runs as half tiles on
    // twice as many (symmetric products keep whole tiles)
    const int tail = ntiles % sms;
    G.nfull = (!G.sym && ntiles > sms && tail > 0 && 2 * tail <= sms) ? ntiles - tail : ntiles;
    const int nitems = G.nfull + 2 * (ntiles - G.nfull);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(std::min(nitems, sms)));
    cfg.blockDim = dim3(kTcThreads);
    cfg.dynamicSmemBytes = static_cast<size_t>(smem);
    cfg.stream = st;
    // programmatic dependent launch: the prologue overlaps the previous kernel
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, k_gemm_tc<BN>, ma, mb, mbh, mc, mct, G);
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t gemm_bf16_nt(int M, int N, int K, float alpha, const void* A, int lda, const void* B, int ldb,
                         float beta, const void* D, int ldd, void* C, int ldc, void* CT, int ldct, int* err,
                         cudaStream_t st, bool sym) {
    if (M <= 0 || N <= 0) return cudaSuccess;
    if (sym && (M != N || CT != nullptr || C == nullptr)) return cudaErrorInvalidValue;
    const bool results_ok = tma_ok(C, ldc) && tma_ok(CT, ldct) && (beta == 0.0f || tma_ok(D, ldd));
    if (K > 0 && results_ok && gemm_tc_usable(lda, ldb, A, B)) {
        // 256-wide tiles when there are enough of them for every SM, else
        // (and for symmetric products) 128-wide ones
        const int64_t tiles256 = static_cast<int64_t>((M + kBM - 1) / kBM) * ((N + 255) / 256);
        const int bn = (sym || tiles256 < device_sm_count()) ? 128 : 256;
        CUtensorMap ma, mb, mbh, mc{}, mct{};
        if (!make_map(&ma, A, M, K, lda, kBM) || !make_map(&mb, B, N, K, ldb, bn) ||
            !make_map(&mbh, B, N, K, ldb, bn / 2))
            return cudaErrorInvalidValue;
        if (C != nullptr && !make_map(&mc, C, M, N, ldc, 0)) return cudaErrorInvalidValue;
        if (CT != nullptr && !make_map(&mct, CT, N, M, ldct, 0)) return cudaErrorInvalidValue;
        if (sym) mct = mc;  // the mirrored blocks go to C itself
        GemmArgs G;
        G.M = M;
        G.N = N;
        G.K = K;
        G.alpha = alpha;
        G.beta = beta;
        G.D = static_cast<const __nv_bfloat16*>(D);
        G.ldd = ldd;
        G.C = static_cast<__nv_bfloat16*>(C);
        G.ldc = ldc;
        G.CT = static_cast<__nv_bfloat16*>(CT);
        G.ldct = ldct;
        G.sym = sym ? 1 : 0;
        G.err = err;
        G.nfull = 0;  // set by the launch
        return bn == 128 ? launch_tc<128>(ma, mb, mbh, mc, mct, G, st) : launch_tc<256>(ma, mb, mbh, mc, mct, G, st);
    }
    const dim3 grid((N + 63) / 64, (M + 63) / 64);
    k_gemm_simt<__nv_bfloat16><<<grid, 256, 0, st>>>(
        M, N, K, alpha, static_cast<const __nv_bfloat16*>(A), lda, static_cast<const __nv_bfloat16*>(B), ldb, beta,
        static_cast<const __nv_bfloat16*>(D), ldd, static_cast<__nv_bfloat16*>(C), ldc,
        static_cast<__nv_bfloat16*>(CT), ldct);
    return cudaGetLastError();
}

cudaError_t gemm_f32_nt(int M, int N, int K, float alpha, const float* A, int lda, const float* B, int ldb,
                        float beta, const float* D, int ldd, float* C, int ldc, float* CT, int ldct,
                        cudaStream_t st) {
    if (M <= 0 || N <= 0) return cudaSuccess;
    const dim3 grid((N + 63) / 64, (M + 63) / 64);
    k_gemm_simt<float><<<grid, 256, 0, st>>>(M, N, K, alpha, A, lda, B, ldb, beta, D, ldd, C, ldc, CT, ldct);
    return cudaGetLastError();
}

}  // namespace gefen

// Exposed for tests: C = alpha A B^T + beta D in bf16 (see gefen.h).
extern "C" gefen_status_t gefen_gemm_bf16(int32_t M, int32_t N, int32_t K, float alpha, const uint16_t* A,
                                          int32_t lda, const uint16_t* B, int32_t ldb, float beta, const uint16_t* D,
                                          int32_t ldd, uint16_t* C, int32_t ldc, uint16_t* CT, int32_t ldct,
                                          void* workspace, size_t workspace_bytes, gefen_stream_t stream) {
    using namespace gefen;
    if (M < 0 || N < 0 || K < 0 || !A || !B || (!C && !CT)) return GEFEN_EINVAL;
    if ((C && ldc < N) || (CT && ldct < M) || lda < K || ldb < K || (beta != 0.0f && (!D || ldd < N)))
        return GEFEN_EINVAL;
    if (workspace == nullptr || workspace_bytes < kWsAlign) return GEFEN_ENOMEM;
    if (reinterpret_cast<uintptr_t>(workspace) % kWsAlign) return GEFEN_EINVAL;
    if (gefen_status_t s = check_device(); s != GEFEN_OK) return s;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    int* err = static_cast<int*>(workspace);
    if (gemm_bf16_nt(M, N, K, alpha, A, lda, B, ldb, beta, D, ldd, C, ldc, CT, ldct, err, st, false) != cudaSuccess)
        return GEFEN_ECUDA;
    return GEFEN_OK;
}

// Exposed for tests: C = alpha A A^T + beta D, symmetric (see gefen.h).
extern "C" gefen_status_t gefen_gemm_bf16_sym(int32_t N, int32_t K, float alpha, const uint16_t* A, int32_t lda,
                                              float beta, const uint16_t* D, int32_t ldd, uint16_t* C, int32_t ldc,
                                              void* workspace, size_t workspace_bytes, gefen_stream_t stream) {
    using namespace gefen;
    if (N < 0 || K < 0 || !A || !C || ldc < N || lda < K || (beta != 0.0f && (!D || ldd < N))) return GEFEN_EINVAL;
    if (workspace == nullptr || workspace_bytes < kWsAlign) return GEFEN_ENOMEM;
    if (reinterpret_cast<uintptr_t>(workspace) % kWsAlign) return GEFEN_EINVAL;
    if (gefen_status_t s = check_device(); s != GEFEN_OK) return s;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    int* err = static_cast<int*>(workspace);
    if (gemm_bf16_nt(N, N, K, alpha, A, lda, A, lda, beta, D, ldd, C, ldc, nullptr, 0, err, st, true) != cudaSuccess)
        return GEFEN_ECUDA;
    return GEFEN_OK;
}
