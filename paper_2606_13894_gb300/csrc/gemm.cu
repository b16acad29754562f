// Matrix products of Gefen-Muon's Newton-Schulz iteration (the paper's
// appendix "Gefen-Muon"), on sm_103a:
//
//   C = alpha * A * B^T + beta * D      A: M x K, B: N x K, C, D: M x N
//
// all row-major (K contiguous in A and B), written as C and/or as its
// transpose CT (N x M).
//
// bf16 storage, fp32 accumulation: a tcgen05 kernel.  One CTA computes a
// 128 x 256 tile of C in tensor memory (256 of its 512 columns).  Thread 0
// loads 128 x 64 tiles of A and 256 x 64 tiles of B with TMA (128-byte
// swizzle) into a ring of four shared-memory stages; thread 32 issues
// tcgen05.mma (M 128, N 256, K 16; four per stage) as each stage lands and
// frees it with tcgen05.commit; all four warps then read the accumulator rows
// with tcgen05.ld, apply alpha and beta * D and store C directly, or CT
// through shared memory so that its rows go out coalesced.  Every wait on an
// mbarrier gives up after about a second and flags the error word instead.
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

constexpr int kBM = 128, kBN = 256, kBK = 64, kStages = 4;
constexpr int kGemmThreads = 128;
constexpr uint32_t kTileA = kBM * kBK * 2, kTileB = kBN * kBK * 2;  // bytes
constexpr uint32_t kTmemCols = 256;
constexpr long long kSpin = 1ll << 31;

struct alignas(1024) GemmSmem {
    unsigned char a[kStages][kTileA];  // each 1024-byte aligned (swizzle atoms)
    unsigned char b[kStages][kTileB];
    unsigned long long full[kStages], empty[kStages], done;
    uint32_t tmem;
    int abort;
    int consumed;  // k-tiles the MMA issuer took from the ring
};
// The transposed epilogue stages a 256 x 128 bf16 tile over the operand ring.
static_assert(sizeof(GemmSmem::a) + sizeof(GemmSmem::b) >= kBN * kBM * 2, "staging fits the ring");

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
// Instruction descriptor of kind::f16: fp32 accumulator (bits 4-5 = 1), bf16
// A and B (bits 7-9, 10-12 = 1), both K-major, N / 8 at bit 17, M / 16 at 24.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(kBN >> 3) << 17) |
                            (static_cast<uint32_t>(kBM >> 4) << 24);

__device__ __forceinline__ void umma_bf16(uint32_t tmem, uint64_t da, uint64_t db, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem),
        "l"(da), "l"(db), "r"(kIdesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}
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
    int* err;
};

__global__ void __launch_bounds__(kGemmThreads, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB, const GemmArgs G) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    // aligned to 1024 bytes here: the launch asks for 1024 bytes of slack
    GemmSmem& sm = *reinterpret_cast<GemmSmem*>(smem_raw + ((1024 - (saddr(smem_raw) & 1023)) & 1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.y * kBM, n0 = blockIdx.x * kBN;
    const int KT = (G.K + kBK - 1) / kBK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(saddr(&sm.full[s]), 1);
            mbar_init(saddr(&sm.empty[s]), 1);
        }
        mbar_init(saddr(&sm.done), 1);
        sm.abort = 0;
        sm.consumed = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapA)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapB)) : "memory");
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(saddr(&sm.tmem)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sm.tmem;

    int issued = 0;  // thread 0: k-tiles whose loads were started
    if (threadIdx.x == 0) {
        // producer: TMA loads of A and B k-tiles into the ring
        for (int kt = 0; kt < KT; ++kt) {
            const int s = kt % kStages;
            if (kt >= kStages && !mbar_wait(saddr(&sm.empty[s]), static_cast<uint32_t>((kt / kStages - 1) & 1))) {
                atomicExch(&sm.abort, 1);
                break;
            }
            if (*static_cast<volatile int*>(&sm.abort)) break;
            const uint32_t bar = saddr(&sm.full[s]);
            mbar_expect_tx(bar, kTileA + kTileB);
            tma_load_2d(saddr(sm.a[s]), &mapA, kt * kBK, m0, bar);
            tma_load_2d(saddr(sm.b[s]), &mapB, kt * kBK, n0, bar);
            issued = kt + 1;
        }
    } else if (threadIdx.x == 32) {
        // MMA issuer: four K = 16 steps per stage, the stage freed by commit
        int kt = 0;
        for (; kt < KT; ++kt) {
            const int s = kt % kStages;
            if (!mbar_wait(saddr(&sm.full[s]), static_cast<uint32_t>((kt / kStages) & 1))) {
                atomicExch(&sm.abort, 1);
                break;
            }
            tc_fence_after();
            const uint32_t a0 = saddr(sm.a[s]), b0 = saddr(sm.b[s]);
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk)
                umma_bf16(tmem, desc_sw128(a0 + kk * 32), desc_sw128(b0 + kk * 32), (kt | kk) != 0 ? 1u : 0u);
            umma_commit(saddr(&sm.empty[s]));
        }
        sm.consumed = kt;
        umma_commit(saddr(&sm.done));  // arrives once every MMA issued above has completed
    }
    __syncwarp();

    // epilogue: warp w holds accumulator rows 32 w .. 32 w + 31 (TMEM lanes)
    const bool ok = mbar_wait(saddr(&sm.done), 0u);
    tc_fence_after();
    // one decision for the whole CTA (the transposed store has a barrier)
    if (!__syncthreads_and(ok && *static_cast<volatile int*>(&sm.abort) == 0)) {
        if (threadIdx.x == 0) atomicExch(G.err, 1);
    } else {
        const int r = 32 * warp + lane, row = m0 + r;
        __nv_bfloat16* stage = reinterpret_cast<__nv_bfloat16*>(sm.a[0]);  // CT staging: [col][row], 256 x 128
        for (int c0 = 0; c0 < kBN; c0 += 32) {
            float v[32];
            tmem_ld32(tmem + (static_cast<uint32_t>(32 * warp) << 16) + static_cast<uint32_t>(c0), v);
            if (row < G.M) {
                if (G.beta != 0.0f && G.D != nullptr) {
                    const __nv_bfloat16* d = G.D + static_cast<int64_t>(row) * G.ldd + n0 + c0;
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        v[i] = G.alpha * v[i] + (n0 + c0 + i < G.N ? G.beta * __bfloat162float(d[i]) : 0.0f);
                } else {
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] *= G.alpha;
                }
                if (G.C != nullptr) {
                    __nv_bfloat16* c = G.C + static_cast<int64_t>(row) * G.ldc + n0 + c0;
                    if (n0 + c0 + 32 <= G.N && ((reinterpret_cast<uintptr_t>(c) & 15u) == 0)) {
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            __nv_bfloat162 h[4];
#pragma unroll
                            for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(v[8 * q + 2 * i], v[8 * q + 2 * i + 1]);
                            *reinterpret_cast<uint4*>(c + 8 * q) = *reinterpret_cast<uint4*>(h);
                        }
                    } else {
                        for (int i = 0; i < 32 && n0 + c0 + i < G.N; ++i) c[i] = __float2bfloat16_rn(v[i]);
                    }
                }
            }
            if (G.CT != nullptr) {
#pragma unroll
                for (int i = 0; i < 32; ++i) stage[(c0 + i) * kBM + r] = __float2bfloat16_rn(v[i]);
            }
        }
        if (G.CT != nullptr) {
            __syncthreads();
            // rows of CT: column n0 + j of C, elements m0 .. m0 + 127 (256 bytes)
            for (int j = warp; j < kBN; j += kGemmThreads / 32) {
                const int col = n0 + j;
                if (col >= G.N) break;
                __nv_bfloat16* ct = G.CT + static_cast<int64_t>(col) * G.ldct + m0;
                const __nv_bfloat16* src = stage + j * kBM;
                for (int i = lane; i < kBM; i += 32)
                    if (m0 + i < G.M) ct[i] = src[i];
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0 && sm.consumed < issued) {
        // an aborted pipeline: wait (bounded) for the loads still in flight
        for (int kt = sm.consumed; kt < issued; ++kt)
            mbar_wait(saddr(&sm.full[kt % kStages]), static_cast<uint32_t>((kt / kStages) & 1));
    }
    if (warp == 0) {
        __syncwarp();
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
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

// TMA map of a row-major rows x cols bf16 matrix (leading dimension ld), box
// 64 columns x box_rows rows, 128-byte swizzle, zero fill out of range.
bool make_map(CUtensorMap* map, const void* base, int rows, int cols, int ld, int box_rows) {
    const auto fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), static_cast<cuuint32_t>(box_rows)};
    const cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool gemm_tc_usable(int lda, int ldb, const void* A, const void* B) {
    // TMA: 16-byte aligned bases and row strides
    return lda % 8 == 0 && ldb % 8 == 0 && (reinterpret_cast<uintptr_t>(A) & 15u) == 0 &&
           (reinterpret_cast<uintptr_t>(B) & 15u) == 0 && encode_fn() != nullptr;
}

cudaError_t gemm_bf16_nt(int M, int N, int K, float alpha, const void* A, int lda, const void* B, int ldb,
                         float beta, const void* D, int ldd, void* C, int ldc, void* CT, int ldct, int* err,
                         cudaStream_t st) {
    if (M <= 0 || N <= 0) return cudaSuccess;
    if (K > 0 && gemm_tc_usable(lda, ldb, A, B)) {
        CUtensorMap ma, mb;
        if (!make_map(&ma, A, M, K, lda, kBM) || !make_map(&mb, B, N, K, ldb, kBN)) return cudaErrorInvalidValue;
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
        G.err = err;
        const int smem = static_cast<int>(sizeof(GemmSmem)) + 1024;
        cudaError_t e = cudaFuncSetAttribute(k_gemm_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        const dim3 grid((N + kBN - 1) / kBN, (M + kBM - 1) / kBM);
        k_gemm_tc<<<grid, kGemmThreads, smem, st>>>(ma, mb, G);
        return cudaGetLastError();
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
    if (gemm_bf16_nt(M, N, K, alpha, A, lda, B, ldb, beta, D, ldd, C, ldc, CT, ldct, err, st) != cudaSuccess)
        return GEFEN_ECUDA;
    return GEFEN_OK;
}
