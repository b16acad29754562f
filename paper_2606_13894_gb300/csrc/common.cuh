// Shared device helpers for the Gefen kernels (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "gefen.h"

namespace gefen {

constexpr int kMaxLevels = GEFEN_MAX_LEVELS;
constexpr int kMaxBins = GEFEN_MAX_BINS;

// ---------------------------------------------------------------- bf16
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ float bf16_bits_to_f32(uint16_t b) {
    return __uint_as_float(static_cast<uint32_t>(b) << 16);
}

// ------------------------------------------------------------ histogram
// Cell of a normalised value among B uniform cells over [-1, 1] (Algorithm 3):
// floor((x + 1) * (B/2)) with the add and the multiply each rounded to fp32,
// clamped to [0, B-1].  Callers skip NaN before calling.
__device__ __forceinline__ int hist_cell(float x, float halfB, int B) {
    float t = __fadd_rn(x, 1.0f);
    float u = __fmul_rn(t, halfB);
    float f = floorf(u);
    f = fminf(fmaxf(f, 0.0f), static_cast<float>(B - 1));
    return static_cast<int>(f);
}

// ------------------------------------------------- nearest codebook level
// Number of midpoints strictly below x among 256 sorted midpoints (entries
// past k-1 are +inf): the index of the nearest level, ties to the lower one.
__device__ __forceinline__ int level_search(const float* __restrict__ mids, float x) {
    int c = 0;
#pragma unroll
    for (int s = 128; s >= 1; s >>= 1) c += (mids[c + s - 1] < x) ? s : 0;
    return c;
}

// The same level through cell records: x = m / s' lies in [-1, 1]; a record
// per cell of a uniform grid of kLutCells over [-1, 1] (two guard cells at
// the ends) holds the number of midpoints below the cell and the next three
// midpoints, so the level is the base plus three compares.  Identical to
// level_search whenever build_cell_records reports no cell (widened by a
// 2^-22 guard on both sides) with more than three midpoints; the callers use
// level_search otherwise.  R copies of each record spread a warp's gathers
// over more shared-memory banks (copy r of record c + 1 at (c + 1) R + r).
constexpr int kLutCells = 512;
constexpr float kLutGuard = 2.384185791015625e-07f;  // 2^-22, below every cell edge

__device__ __forceinline__ uint32_t lt_mask(float a, float b) {
    uint32_t r;
    asm("set.lt.u32.f32 %0, %1, %2;" : "=r"(r) : "f"(a), "f"(b));
    return r;
}

// Fills lut[(kLutCells + 2) * R] from mid (padded with +inf to kMaxLevels + 4
// entries, already in shared memory behind a barrier); thread t of nthreads.
// Returns nonzero when some cell holds more than three midpoints.
template <int R>
__device__ __forceinline__ int build_cell_records(const float* mid, float4* lut, int t, int nthreads) {
    int bad = 0;
    // cell(x) = floor(fma(x, G/2, G/2)) is within 2^-24 of exact in x: each
    // record counts the midpoints below its cell minus the guard and holds
    // the next three
    for (int i = t; i < kLutCells + 2; i += nthreads) {
        const int c = i - 1;
        const float lo = -1.0f + 2.0f * static_cast<float>(c) / kLutCells - kLutGuard;
        const float hi = -1.0f + 2.0f * static_cast<float>(c + 1) / kLutCells + kLutGuard;
        const int base = level_search(mid, lo);
        const int upto = level_search(mid, hi);
        bad |= (upto - base > 3);
        const float4 rec = make_float4(__int_as_float(base), mid[base], mid[base + 1], mid[base + 2]);
#pragma unroll
        for (int r = 0; r < R; ++r) lut[i * R + r] = rec;
    }
    return bad;
}

// The level of x from the records (copy `copy`).
template <int R>
__device__ __forceinline__ uint32_t lut_encode(const float4* lut, int copy, float x) {
    constexpr float kMagicCell = 12582912.0f;  // 1.5 * 2^23: the round-down add leaves the cell in the low bits
    const float y = __fmaf_rd(x, 0.5f * kLutCells, 0.5f * kLutCells + 1.0f + kMagicCell);
    const uint32_t r = static_cast<uint32_t>(__float_as_int(y)) - 0x4B400000u;
    const float4 rec = lut[min(r, static_cast<uint32_t>(kLutCells + 1)) * R + copy];
    return static_cast<uint32_t>(__float_as_int(rec.x)) - lt_mask(rec.y, x) - lt_mask(rec.z, x) - lt_mask(rec.w, x);
}

// --------------------------------------------------- 128-bit integers
struct u128 {
    uint64_t hi, lo;
};

__device__ __forceinline__ u128 mul_u64(uint64_t a, uint64_t b) {
    u128 r;
    r.lo = a * b;
    r.hi = __umul64hi(a, b);
    return r;
}

__device__ __forceinline__ u128 sub_u128(u128 a, u128 b) {
    u128 r;
    r.lo = a.lo - b.lo;
    r.hi = a.hi - b.hi - (a.lo < b.lo ? 1ull : 0ull);
    return r;
}

__device__ __forceinline__ u128 add_u128(u128 a, u128 b) {
    u128 r;
    r.lo = a.lo + b.lo;
    r.hi = a.hi + b.hi + (r.lo < a.lo ? 1ull : 0ull);
    return r;
}

// Signed 64-bit value sign-extended to 128 bits (two's complement).
__device__ __forceinline__ u128 from_i64(int64_t v) {
    u128 r;
    r.lo = static_cast<uint64_t>(v);
    r.hi = v < 0 ? ~0ull : 0ull;
    return r;
}

// 2^e as a double for 0 <= e <= 1023 (exact).
__device__ __forceinline__ double pow2d(int e) {
    return __longlong_as_double(static_cast<long long>(1023 + e) << 52);
}

// Correctly rounded (to nearest, ties to even) conversion of an unsigned
// 128-bit integer to double.  The top 64 bits are normalised and every bit
// below them is folded into bit 0 as a sticky bit; bit 0 lies below the
// rounding position of a 64-bit integer's conversion, so the result of the
// 64-bit conversion is the correctly rounded value, then scaled exactly.
__device__ __forceinline__ double u128_to_double_rn(u128 v) {
    if (v.hi == 0) return __ull2double_rn(v.lo);
    int sh = __clzll(static_cast<long long>(v.hi));
    uint64_t top = sh ? (v.hi << sh) | (v.lo >> (64 - sh)) : v.hi;
    uint64_t rest = v.lo << sh;
    top |= (rest != 0) ? 1ull : 0ull;
    return __ull2double_rn(top) * pow2d(64 - sh);
}

// Approximate conversion to float: relative error below 2^-24 + 2^-62.
__device__ __forceinline__ float u128_to_float_approx(u128 v) {
    if (v.hi == 0) return __ull2float_rn(v.lo);
    int sh = __clzll(static_cast<long long>(v.hi));
    uint64_t top = sh ? (v.hi << sh) | (v.lo >> (64 - sh)) : v.hi;
    return __ull2float_rn(top) * __int_as_float((127 + 64 - sh) << 23);
}

}  // namespace gefen
