// gefen_refit_codebook: exact histogram DP quantizer (Algorithm 3; Appendix D).
//
// Nonempty cells j = 1..b (centre u_j / B, u_j = 2 i_j + 1 - B).  Exact integer
// prefix moments P0 = sum c, P1 = sum c u, P2 = sum c u^2 give any run [l..r]
// its s0, s1, s2.  Canonical costs (units of 1/B^2, round to nearest):
//   interior  (double)(s0 s2 - s1^2) / (double)s0
//   first     (double)(s2 + 2B s1 + B^2 s0)      (centre -1)
//   last      (double)(s2 - 2B s1 + B^2 s0)      (centre +1)
// D[r][k'] = min_{k' <= l <= r} D[l-1][k'-1] + cost(l..r), ties to the smallest l.
//
// Levels 2..k in one cooperative launch with a grid barrier between levels,
// one warp per end position r at a time.  fp64 is slow on this
// part, so candidates are screened in float-float arithmetic (a pair of fp32
// values, about 2^-43 relative error): D[.][k'-1] is kept as a (hi, lo) pair
// and each cost comes from its exact 128-bit integer numerator.  Whole runs of
// candidates are excluded with two exact facts: the interior cost of [l..r]
// does not increase as l grows (a subset has no larger squared error) and
// D[.][k'-1] does not decrease along r (more cells for the same levels never
// cost less).  So for l in [a, e]:  value(l) >= D[a-1][k'-1] + cost(e..r).
// A 32-wide window around a hint (the previous level's split at r, moved by
// its share of the last cell; on level 2, the best of 32 evenly spaced
// candidates) gives the best screened value u, one candidate per lane; the
// rest of [k', r] is searched by 32-way subdivision (one run bound per lane),
// dropping every run whose bound exceeds u by more than 2^-34 relative, and
// the narrow runs left are screened 32 candidates to a round.  Survivors
// (near-ties only) get the
// canonical fp64 value once the final bound is known; their minimum, ties to
// the smallest l, equals the full scan bit for bit.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace gefen {

namespace {

constexpr int kDpThreads = 64;
constexpr float kEps = 5.820766091346741e-11f;  // 2^-34: exclusion margin (screen error < 2^-41)

struct Header {
    int32_t status;  // 0 ok, 1 moment overflow (N (B-1)^2 >= 2^64), 2 a level barrier timed out
    int32_t b;       // nonempty cells
    int32_t k_eff;   // levels the DP uses (b <= 1: b)
    int32_t pad;
    uint64_t total;
};

struct DpWs {
    Header* hdr;
    int32_t* idx;  // idx[j], j = 1..b: bin of the j-th nonempty cell
    uint64_t* P0;
    int64_t* P1;
    uint64_t* P2;
    double* D;     // (k+1) x (B+1)
    int32_t* A;    // (k+1) x (B+1)
    float2* E;     // (k+1) x (B+2): row kk, entry l = (hi, lo) of D[kk][l-1], read by level kk+1
    int2* NS;      // B+1: near-optimal run starts [lo, hi] of each anchor row of the current level
    uint32_t* sync;  // [0]: barrier arrivals; [1 + 3 kk + phase]: next row of level kk in that phase
};

// Counters: one barrier-arrival word, then three row counters per level.
__host__ __device__ constexpr int sync_words(int k) { return 3 * (k + 1) + 2; }

struct DpLayout {
    size_t hdr, hist, idx, P0, P1, P2, D, A, E, NS, sync, total;
};

constexpr size_t cx_align(size_t x) { return (x + kWsAlign - 1) / kWsAlign * kWsAlign; }

// Workspace: status header at offset 0 (so it can be read without knowing the
// sizes), the histogram copy, then the DP arrays.
constexpr DpLayout dp_layout(int B, int k) {
    DpLayout L{};
    size_t o = 0;
    const size_t n1 = static_cast<size_t>(B) + 1;
    L.hdr = o; o += cx_align(sizeof(Header));
    L.hist = o; o += cx_align(static_cast<size_t>(B) * sizeof(uint64_t));
    L.idx = o; o += cx_align(n1 * sizeof(int32_t));
    L.P0 = o;  o += cx_align(n1 * sizeof(uint64_t));
    L.P1 = o;  o += cx_align(n1 * sizeof(int64_t));
    L.P2 = o;  o += cx_align(n1 * sizeof(uint64_t));
    L.D = o;   o += cx_align(static_cast<size_t>(k + 1) * n1 * sizeof(double));
    L.A = o;   o += cx_align(static_cast<size_t>(k + 1) * n1 * sizeof(int32_t));
    L.E = o;   o += cx_align(static_cast<size_t>(k + 1) * (n1 + 1) * sizeof(float2));
    L.NS = o;  o += cx_align(n1 * sizeof(int2));
    L.sync = o; o += cx_align(static_cast<size_t>(sync_words(k)) * sizeof(uint32_t));
    L.total = o;
    return L;
}

DpWs dp_ws(void* base, int B, int k) {
    const DpLayout L = dp_layout(B, k);
    char* p = static_cast<char*>(base);
    DpWs w;
    w.hdr = reinterpret_cast<Header*>(p + L.hdr);
    w.idx = reinterpret_cast<int32_t*>(p + L.idx);
    w.P0 = reinterpret_cast<uint64_t*>(p + L.P0);
    w.P1 = reinterpret_cast<int64_t*>(p + L.P1);
    w.P2 = reinterpret_cast<uint64_t*>(p + L.P2);
    w.D = reinterpret_cast<double*>(p + L.D);
    w.A = reinterpret_cast<int32_t*>(p + L.A);
    w.E = reinterpret_cast<float2*>(p + L.E);
    w.NS = reinterpret_cast<int2*>(p + L.NS);
    w.sync = reinterpret_cast<uint32_t*>(p + L.sync);
    return w;
}

// ------------------------------------------------------------ exact costs
__device__ __forceinline__ u128 interior_num(uint64_t s0, int64_t s1, uint64_t s2) {
    const uint64_t a1 = s1 < 0 ? static_cast<uint64_t>(-s1) : static_cast<uint64_t>(s1);
    return sub_u128(mul_u64(s0, s2), mul_u64(a1, a1));
}

// s2 + sign*2B*s1 + B^2*s0 (sign = +1: centre -1; sign = -1: centre +1); >= 0.
__device__ __forceinline__ u128 fixed_num(uint64_t s0, int64_t s1, uint64_t s2, int B, int sign) {
    const uint64_t Bu = static_cast<uint64_t>(B);
    u128 t = mul_u64(Bu * Bu, s0);
    t = add_u128(t, u128{0ull, s2});
    const uint64_t a1 = s1 < 0 ? static_cast<uint64_t>(-s1) : static_cast<uint64_t>(s1);
    const u128 m = mul_u64(2ull * Bu, a1);
    const bool neg = (sign > 0) ? (s1 < 0) : (s1 > 0);
    return neg ? sub_u128(t, m) : add_u128(t, m);
}

struct Run {
    uint64_t s0;
    int64_t s1;
    uint64_t s2;
};

__device__ __forceinline__ Run run_of(const DpWs& W, int l, uint64_t P0r, int64_t P1r, uint64_t P2r) {
    Run q;
    q.s0 = P0r - __ldg(W.P0 + l - 1);
    q.s1 = P1r - __ldg(W.P1 + l - 1);
    q.s2 = P2r - __ldg(W.P2 + l - 1);
    return q;
}

// ---------------------------------------------------- float-float values
struct ff {
    float hi, lo;
};

__device__ __forceinline__ ff ff_quick(float a, float b) {  // |a| >= |b|
    const float s = __fadd_rn(a, b);
    return ff{s, __fsub_rn(b, __fsub_rn(s, a))};
}
__device__ __forceinline__ ff ff_add(ff x, ff y) {
    const float s = __fadd_rn(x.hi, y.hi);
    const float bb = __fsub_rn(s, x.hi);
    const float e = __fadd_rn(__fsub_rn(x.hi, __fsub_rn(s, bb)), __fsub_rn(y.hi, bb));
    return ff_quick(s, __fadd_rn(e, __fadd_rn(x.lo, y.lo)));
}
__device__ __forceinline__ ff ff_sub(ff x, ff y) { return ff_add(x, ff{-y.hi, -y.lo}); }
// n / d: one reciprocal, an exact product error by fma, one correction.
__device__ __forceinline__ ff ff_div(ff n, ff d) {
    const float r = __frcp_rn(d.hi);
    const float q1 = __fmul_rn(n.hi, r);
    const float p = __fmul_rn(q1, d.hi);
    const float pe = __fmaf_rn(q1, d.hi, -p);
    float rem = __fsub_rn(n.hi, p);
    rem = __fsub_rn(rem, pe);
    rem = __fadd_rn(rem, n.lo);
    rem = __fsub_rn(rem, __fmul_rn(q1, d.lo));
    return ff_quick(q1, __fmul_rn(rem, r));
}
// An unsigned 128-bit integer as hi + lo (top 64 bits kept: error < 2^-47).
// Built from bit fields and 32-bit conversions only: 64-bit integer to float
// conversions would run on the slow fp64 pipe of this part.
__device__ __forceinline__ ff u128_to_ff(u128 v) {
    uint64_t T;
    int e2;  // value = T * 2^e2
    if (v.hi) {
        const int sh = __clzll(static_cast<long long>(v.hi));
        T = sh ? (v.hi << sh) | (v.lo >> (64 - sh)) : v.hi;
        e2 = 64 - sh;
    } else if (v.lo) {
        const int sh = __clzll(static_cast<long long>(v.lo));
        T = v.lo << sh;
        e2 = -sh;
    } else {
        return ff{0.0f, 0.0f};
    }
    // hi: the top 24 bits exactly (T has bit 63 set)
    const uint32_t mant = static_cast<uint32_t>(T >> 40) & 0x7FFFFFu;
    const float hi = __int_as_float(((127 + 63 + e2) << 23) | static_cast<int>(mant));
    // lo: the remaining 40 bits, rounded once
    const uint64_t R = T & 0xFFFFFFFFFFull;
    const float r = __fmaf_rn(__uint2float_rn(static_cast<uint32_t>(R >> 32)), 4294967296.0f,
                              __uint2float_rn(static_cast<uint32_t>(R)));
    return ff_quick(hi, r * __int_as_float((127 + e2) << 23));
}
// ------------------------------------------- doubles handled as integer bits
// Non-negative doubles order like their bit patterns, so the search converts,
// compares and reduces them with integer operations: this part's fp64 pipe has
// a small fraction of its integer and fp32 throughput.
constexpr uint64_t kInfBits = 0x7FF0000000000000ull;

__host__ __device__ __forceinline__ int clz64(uint64_t x) {  // x != 0
#ifdef __CUDA_ARCH__
    return __clzll(static_cast<long long>(x));
#else
    return __builtin_clzll(x);
#endif
}

// Bits of the correctly rounded (to nearest, ties to even) double of an
// unsigned 128-bit integer.
__host__ __device__ __forceinline__ uint64_t u128_to_dbits(u128 v) {
    int lz;
    uint64_t top, rest;
    if (v.hi) {
        lz = clz64(v.hi);
        top = lz ? (v.hi << lz) | (v.lo >> (64 - lz)) : v.hi;
        rest = v.lo << lz;
    } else if (v.lo) {
        lz = 64 + clz64(v.lo);
        top = v.lo << (lz - 64);
        rest = 0;
    } else {
        return 0;
    }
    // value = top * 2^(64 - lz) with bit 63 of top set: keep 53 bits, round on
    // the 11 below them and every bit of rest
    uint64_t m = top >> 11;
    const uint32_t g = static_cast<uint32_t>(top) & 0x7FFu;
    m += (g > 0x400u || (g == 0x400u && (rest != 0 || (m & 1)))) ? 1 : 0;
    int e = 127 - lz;  // exponent of the leading bit
    if (m >> 53) {
        m >>= 1;
        ++e;
    }
    return (static_cast<uint64_t>(e + 1023) << 52) | (m & 0xFFFFFFFFFFFFFull);
}

constexpr uint64_t kMant = 0xFFFFFFFFFFFFFull;  // the 52 stored significand bits
constexpr uint64_t kHidden = 1ull << 52;

// Bits of RN(N / D) for positive normal doubles N, D (bits nb, db; N may be
// +0) whose quotient is normal: the significand quotient by long division in
// five 11-bit digits, each estimated in fp32 and corrected by one exact
// integer step, then rounded to nearest (ties to even) with the remainder as
// sticky bit.  Equal to IEEE division; integer and fp32 operations only.
__host__ __device__ __forceinline__ uint64_t div_dbits(uint64_t nb, uint64_t db) {
    if (nb == 0) return 0;
    uint64_t Nm = (nb & kMant) | kHidden, Dm = (db & kMant) | kHidden;
    int e = static_cast<int>(nb >> 52) - static_cast<int>(db >> 52);
    if (Nm < Dm) {  // Nm / Dm in [1, 2) from here on
        Nm <<= 1;
        --e;
    }
    uint64_t R = Nm - Dm, Q = 1;
#ifdef __CUDA_ARCH__
    const float rd = __frcp_rn(__uint2float_rn(static_cast<uint32_t>(Dm >> 21)) * 2097152.0f);
#else
    const float rd = 1.0f / (static_cast<float>(static_cast<uint32_t>(Dm >> 21)) * 2097152.0f);
#endif
    for (int i = 0; i < 5; ++i) {
        R <<= 11;  // R < Dm < 2^53 before the shift
#ifdef __CUDA_ARCH__
        const float rf = __uint2float_rn(static_cast<uint32_t>(R >> 32)) * 4294967296.0f;
        uint64_t q = __float2uint_rz(rf * rd);
#else
        const float rf = static_cast<float>(static_cast<uint32_t>(R >> 32)) * 4294967296.0f;
        uint64_t q = static_cast<uint64_t>(static_cast<uint32_t>(rf * rd));
#endif
        uint64_t p = q * Dm;  // q <= 2^11, so no overflow
        if (p > R) {
            --q;
            p -= Dm;
        }
        R -= p;
        if (R >= Dm) {
            ++q;
            R -= Dm;
        }
        Q = (Q << 11) | q;
    }
    // Q in [2^55, 2^56): 53 significand bits and three below them
    uint64_t m = Q >> 3;
    const uint32_t g = static_cast<uint32_t>(Q) & 7u;
    m += (g > 4u || (g == 4u && (R != 0 || (m & 1)))) ? 1 : 0;
    if (m >> 53) {
        m >>= 1;
        ++e;
    }
    return (static_cast<uint64_t>(e + 1023) << 52) | (m & kMant);
}

// Bits of RN(a + b) for non-negative normal (or zero) doubles a, b with a
// finite sum: align with three extra bits (guard, round, sticky), add, round
// to nearest (ties to even).  Equal to IEEE addition; integer operations only.
__host__ __device__ __forceinline__ uint64_t add_dbits(uint64_t a, uint64_t b) {
    if (a < b) {
        const uint64_t t = a;
        a = b;
        b = t;
    }
    if (b == 0) return a;
    int ea = static_cast<int>(a >> 52);
    const int d = ea - static_cast<int>(b >> 52);
    if (d > 54) return a;  // b below half an ulp of a
    const uint64_t ma = ((a & kMant) | kHidden) << 3, mb = ((b & kMant) | kHidden) << 3;
    uint64_t sm = ma + ((mb >> d) | (((mb & ((1ull << d) - 1)) != 0) ? 1 : 0));
    if (sm >> 56) {
        sm = (sm >> 1) | (sm & 1);
        ++ea;
    }
    uint64_t m = sm >> 3;
    const uint32_t g = static_cast<uint32_t>(sm) & 7u;
    m += (g > 4u || (g == 4u && (m & 1))) ? 1 : 0;
    if (m >> 53) {
        m >>= 1;
        ++ea;
    }
    return (static_cast<uint64_t>(ea) << 52) | (m & kMant);
}

// A non-negative double (bits) as a float-float value: hi holds its top 24
// significant bits, lo the other 29 rounded once (relative error below
// 2^-47).  DP values are 0, +inf, or at least 2^-62 (an integer numerator over
// a count below 2^62) and below 2^127.
__device__ __forceinline__ ff dbits_to_ff(uint64_t b) {
    if (b >= kInfBits) return ff{INFINITY, 0.0f};
    if (b == 0) return ff{0.0f, 0.0f};
    const int e = static_cast<int>(b >> 52) - 1023;
    const float hi = __uint_as_float((static_cast<uint32_t>(e + 127) << 23) | (static_cast<uint32_t>(b >> 29) & 0x7FFFFFu));
    const float lo = __uint2float_rn(static_cast<uint32_t>(b) & 0x1FFFFFFFu) *
                     __uint_as_float(static_cast<uint32_t>(e - 52 + 127) << 23);
    return ff{hi, lo};
}

__device__ __forceinline__ ff cost_ff_interior(const Run& q) {
    return ff_div(u128_to_ff(interior_num(q.s0, q.s1, q.s2)), u128_to_ff(u128{0ull, q.s0}));
}
// Whether every value bounded below by lb is certainly above the best
// screened value u by more than da (margin 2^-34 relative, far above the
// screening error, plus da).
__device__ __forceinline__ bool excluded(ff lb, ff u, float da = 0.0f) {
    return ff_sub(lb, u).hi > kEps * (lb.hi + u.hi) + da;
}
// Every level writes its own rows of D, A and E once, past L1, and they are
// read only by later levels (after the grid barrier), so no SM can hold a stale
// copy and the reads may go through L1.
__device__ __forceinline__ ff ld_ff(const float2* E, int l) {
    const float2 e = __ldca(E + l);
    return ff{e.x, e.y};
}


// ---------------------------------------------------------------- kernels
// Compaction of nonempty cells and exact prefix moments (one CTA).
constexpr int kPrefixThreads = 1024;

__global__ void __launch_bounds__(kPrefixThreads) k_dp_prefix(const uint64_t* __restrict__ hist, int B, int k,
                                                             DpWs W) {
    __shared__ uint64_t s_cnt[kPrefixThreads], s_p0[kPrefixThreads], s_p2[kPrefixThreads];
    __shared__ int64_t s_p1[kPrefixThreads];
    __shared__ uint64_t s_hi[kPrefixThreads];
    const int t = threadIdx.x;
    if (t < sync_words(k)) W.sync[t] = 0u;
    const int per = (B + kPrefixThreads - 1) / kPrefixThreads;
    const int i0 = min(B, t * per), i1 = min(B, i0 + per);
    uint64_t cnt = 0, p0 = 0, p2 = 0, hi = 0;
    int64_t p1 = 0;
    for (int i = i0; i < i1; ++i) {
        const uint64_t c = hist[i];
        if (!c) continue;
        const int64_t u = 2 * static_cast<int64_t>(i) + 1 - B;
        ++cnt;
        const uint64_t np0 = p0 + c;
        hi += (np0 < p0) ? 1ull : 0ull;  // carry: total count past 2^64
        p0 = np0;
        p1 += static_cast<int64_t>(c) * u;
        p2 += c * static_cast<uint64_t>(u * u);
    }
    s_cnt[t] = cnt; s_p0[t] = p0; s_p1[t] = p1; s_p2[t] = p2; s_hi[t] = hi;
    __syncthreads();
    // inclusive scan (Hillis-Steele) over the 1024 thread sums
    for (int o = 1; o < kPrefixThreads; o <<= 1) {
        uint64_t a = 0, b0 = 0, b2 = 0, h = 0;
        int64_t b1 = 0;
        if (t >= o) { a = s_cnt[t - o]; b0 = s_p0[t - o]; b1 = s_p1[t - o]; b2 = s_p2[t - o]; h = s_hi[t - o]; }
        __syncthreads();
        if (t >= o) {
            s_cnt[t] += a;
            const uint64_t np0 = s_p0[t] + b0;
            s_hi[t] += h + ((np0 < b0) ? 1ull : 0ull);
            s_p0[t] = np0;
            s_p1[t] += b1;
            s_p2[t] += b2;
        }
        __syncthreads();
    }
    const uint64_t N = s_p0[kPrefixThreads - 1];
    const bool overflow_n = s_hi[kPrefixThreads - 1] != 0;
    const int b = static_cast<int>(s_cnt[kPrefixThreads - 1]);
    // exact moments need N (B-1)^2 < 2^64
    const uint64_t bb = static_cast<uint64_t>(B - 1) * static_cast<uint64_t>(B - 1);
    // exact signed first moments need N < 2^62 as well
    const bool bad = overflow_n || (N >> 62) != 0 || (bb != 0 && __umul64hi(N, bb) != 0);
    if (t == 0) {
        W.hdr->status = bad ? 1 : 0;
        W.hdr->b = bad ? 0 : b;
        W.hdr->k_eff = bad ? -1 : (b <= 1 ? b : min(k, b));
        W.hdr->total = N;
        W.P0[0] = 0; W.P1[0] = 0; W.P2[0] = 0;
        W.idx[0] = -1;
    }
    if (bad) return;
    // write this thread's entries at its exclusive prefix
    int j = static_cast<int>(t ? s_cnt[t - 1] : 0);
    uint64_t q0 = t ? s_p0[t - 1] : 0, q2 = t ? s_p2[t - 1] : 0;
    int64_t q1 = t ? s_p1[t - 1] : 0;
    for (int i = i0; i < i1; ++i) {
        const uint64_t c = hist[i];
        if (!c) continue;
        const int64_t u = 2 * static_cast<int64_t>(i) + 1 - B;
        ++j;
        q0 += c;
        q1 += static_cast<int64_t>(c) * u;
        q2 += c * static_cast<uint64_t>(u * u);
        W.idx[j] = i;
        W.P0[j] = q0;
        W.P1[j] = q1;
        W.P2[j] = q2;
    }
}

// Level 0 (D[0][0] = 0) and level 1 (first level, centre -1: D[1][r] =
// cost_first(1..r)); thread g covers r = g - 1 and writes E[g] = float(D[1][g-1]).
__global__ void __launch_bounds__(kDpThreads) k_dp_level1(int B, DpWs W) {
    const int g = blockIdx.x * blockDim.x + threadIdx.x;
    if (g > B + 1) return;
    const int n1 = B + 1;
    const Header h = *W.hdr;
    if (h.status) return;
    const int r = g - 1;
    if (r >= 0) {
        W.D[r] = (r == 0) ? 0.0 : INFINITY;
        W.A[r] = 0;
    }
    uint64_t d = kInfBits;
    if (r >= 1 && r <= h.b) d = u128_to_dbits(fixed_num(W.P0[r], W.P1[r], W.P2[r], B, +1));
    if (r >= 0) {
        W.D[n1 + r] = __longlong_as_double(static_cast<long long>(d));
        W.A[n1 + r] = (r >= 1 && r <= h.b) ? 1 : 0;
    }
    const ff e = dbits_to_ff(d);
    W.E[1 * (n1 + 1) + g] = make_float2(e.hi, e.lo);  // row 1 of E
}

// Candidate screen + canonical evaluation for one (r, level).
struct Best {
    uint64_t v;  // bits of a non-negative double
    int l;
};

__device__ __forceinline__ void take(Best& b, uint64_t v, int l) {
    if (v < b.v || (v == b.v && l < b.l)) { b.v = v; b.l = l; }
}

// Lexicographic (hi, lo) minimum over the warp.  Screened values are >= 0 or
// +inf, so hi orders like its bit pattern; lo has either sign and is mapped to
// an order-preserving signed key.  Two integer warp reductions.
__device__ __forceinline__ int lo_key(float x) {
    const int b = __float_as_int(x);
    return b >= 0 ? b : (b ^ 0x7FFFFFFF);
}
__device__ __forceinline__ ff warp_min_ff(ff v) {
    const unsigned hb = __float_as_uint(v.hi);
    const unsigned hm = __reduce_min_sync(0xffffffffu, hb);
    const int lk = __reduce_min_sync(0xffffffffu, hb == hm ? lo_key(v.lo) : 0x7FFFFFFF);
    return ff{__uint_as_float(hm), __int_as_float(lk >= 0 ? lk : (lk ^ 0x7FFFFFFF))};
}
// Lexicographic (value, l) minimum over the warp: three integer reductions.
__device__ __forceinline__ Best warp_min_best(Best b) {
    const unsigned h = static_cast<unsigned>(b.v >> 32), lo = static_cast<unsigned>(b.v);
    const unsigned hm = __reduce_min_sync(0xffffffffu, h);
    const unsigned lm = __reduce_min_sync(0xffffffffu, h == hm ? lo : 0xFFFFFFFFu);
    const unsigned l = __reduce_min_sync(0xffffffffu, (h == hm && lo == lm) ? static_cast<unsigned>(b.l) : 0x7FFFFFFFu);
    return Best{(static_cast<uint64_t>(hm) << 32) | lm, static_cast<int>(l)};
}

// Warps (end positions at a time) per CTA of the levels kernel: 16 up to
// kDpSmallBins cells (every row has its own warp), 8 above (anchored levels:
// smaller CTAs wait at their block barrier for fewer rows; 65536 x 256 26.8
// -> 26.1 ms, while 4096 x 256 took 2.92 ms against 2.83 with 16).
constexpr int kDpWarpsSmall = 16, kDpWarpsLarge = 8, kDpSmallBins = 8192;
constexpr int kStackCap = 192;   // runs pending per warp

// Everything one warp needs to screen and evaluate candidates for one r.
struct RowCtx {
    const DpWs* W;
    const double* Dp;
    const float2* Ep;
    uint64_t P0r, P2r;
    int64_t P1r;
    int B, r;
    bool last;  // +1-centred cost of the last level
};

// Screened value of the run [l..r] as the last cell (value of candidate l).
__device__ __forceinline__ ff run_cost_ff(const RowCtx& c, int l) {
    const Run q = run_of(*c.W, l, c.P0r, c.P1r, c.P2r);
    return c.last ? u128_to_ff(fixed_num(q.s0, q.s1, q.s2, c.B, -1)) : cost_ff_interior(q);
}

// Canonical value of candidate l (bits): D[l-1] + cost(l..r), each rounded
// as the oracle rounds them -- the conversions, the division and the sum in
// integer arithmetic that reproduces IEEE round-to-nearest (this part's fp64
// pipe is slow).  Used only for candidates near the minimum.
__device__ __forceinline__ uint64_t canonical(const RowCtx& c, int l) {
    const Run q = run_of(*c.W, l, c.P0r, c.P1r, c.P2r);
    const uint64_t dprev = __ldca(reinterpret_cast<const unsigned long long*>(c.Dp) + l - 1);
    const uint64_t cost = c.last ? u128_to_dbits(fixed_num(q.s0, q.s1, q.s2, c.B, -1))
                                 : div_dbits(u128_to_dbits(interior_num(q.s0, q.s1, q.s2)),
                                             u128_to_dbits(u128{0ull, q.s0}));
    return add_dbits(dprev, cost);
}

// Search state of one warp: u is the best screened value seen; each lane
// keeps at most one pending candidate (one not excluded when it was screened),
// whose canonical value is taken only if the final u still does not exclude
// it.  A second pending candidate in the same lane first settles the first.
// Every candidate the final u does not exclude thus gets its canonical value,
// and the best of those is the full scan's.
//
// An anchor row also records the extent [nlo, nhi] of its near-optimal
// candidates: every l whose exact value is within da of the row minimum (runs
// and candidates are then excluded only beyond the relative margin plus da).
struct Search {
    ff u;
    int pl;  // pending candidate of this lane, 0 if none
    ff pv;   // its screened value
    Best bst;
    float da;      // absolute margin of the near-optimal extent (0: not recorded)
    int nlo, nhi;  // extent of the near-optimal candidates this lane settled
};

__device__ __forceinline__ void search_init(Search& S, float da) {
    S.u = ff{INFINITY, 0.0f};
    S.pl = 0;
    S.pv = ff{INFINITY, 0.0f};
    S.bst = Best{kInfBits, 0};
    S.da = da;
    S.nlo = 0x7FFFFFFF;
    S.nhi = 0;
}

__device__ __forceinline__ void settle(const RowCtx& c, Search& S) {
    if (S.pl != 0 && !excluded(S.pv, S.u, S.da)) {
        S.nlo = min(S.nlo, S.pl);
        S.nhi = max(S.nhi, S.pl);
        if (!excluded(S.pv, S.u)) take(S.bst, canonical(c, S.pl), S.pl);
    }
    S.pl = 0;
}

// One round over up to 32 candidates, one per lane (l = 0: none; every
// candidate is >= 2).
__device__ __forceinline__ void eval_lanes(const RowCtx& c, int l, Search& S) {
    const bool in = l != 0;
    ff v{INFINITY, 0.0f};
    if (in) v = ff_add(ld_ff(c.Ep, l), run_cost_ff(c, l));
    const ff vm = warp_min_ff(v);
    if (vm.hi < S.u.hi || (vm.hi == S.u.hi && vm.lo < S.u.lo)) S.u = vm;
    if (in && !excluded(v, S.u, S.da)) {
        settle(c, S);
        S.pl = l;
        S.pv = v;
    }
}
// One round over the candidates a, a+st, ..., up to e (at most 32).
__device__ __forceinline__ void eval_candidates(const RowCtx& c, int a, int e, int lane, Search& S, int st = 1) {
    const int l = a + lane * st;
    eval_lanes(c, l <= e ? l : 0, S);
}

// Every candidate l in [lo, hi] of one row, pruned: a 32-wide window around
// the hint, then the rest by 32-way subdivision.  Leaves the result in S.
__device__ void search_row(const RowCtx& c, int kk, int lo, int hi, int hint, int lane, int2* stack, Search& S) {
    if (kk == 2 && hi - lo >= 64) {
        // level 2: the previous level's split (always 1) says nothing, so
        // sample 32 evenly spaced candidates and centre the window on the best
        const int st = (hi - lo) / 31;
        eval_candidates(c, lo, hi, lane, S, st);
        const unsigned at = __ballot_sync(0xffffffffu, S.pl != 0 && S.pv.hi == S.u.hi && S.pv.lo == S.u.lo);
        hint = at ? __shfl_sync(0xffffffffu, S.pl, __ffs(at) - 1) : lo + (hi - lo) / 2;
    }
    hint = min(max(hint, lo), hi);
    int w0 = max(lo, hint - 8);
    const int w1 = min(hi, w0 + 31);
    w0 = max(lo, w1 - 31);
    eval_candidates(c, w0, w1, lane, S);
    int sp = 0;  // warp-uniform
    if (lane == 0) {
        if (w1 < hi) stack[sp] = make_int2(w1 + 1, hi);
        if (w0 > lo) stack[sp + (w1 < hi ? 1 : 0)] = make_int2(lo, w0 - 1);
    }
    sp = (w1 < hi ? 1 : 0) + (w0 > lo ? 1 : 0);
    __syncwarp();
    while (sp > 0) {
        if (stack[sp - 1].y - stack[sp - 1].x < 32) {
            // runs of at most 32 candidates from the top of the stack, packed
            // into one round as long as they fit
            int n = 0, l = 0;
            while (sp > 0) {
                const int2 q = stack[sp - 1];
                const int w = q.y - q.x + 1;
                if (n + w > 32) break;
                if (lane >= n && lane < n + w) l = q.x + (lane - n);
                n += w;
                --sp;
            }
            __syncwarp();
            eval_lanes(c, l, S);
            continue;
        }
        const int2 run = stack[--sp];
        __syncwarp();
        const int a = run.x, e = run.y, width = e - a + 1;
        // 32 sub-runs; lane i bounds [ca, ce] by D[ca-1] + cost(ce..r)
        const int cw = (width + 31) >> 5;
        const int ca = a + lane * cw, ce = min(e, ca + cw - 1);
        bool keep = false;
        if (ca <= e) keep = !excluded(ff_add(ld_ff(c.Ep, ca), run_cost_ff(c, ce)), S.u, S.da);
        const unsigned mask = __ballot_sync(0xffffffffu, keep);
        const int cnt = __popc(mask);
        if (sp + cnt > kStackCap) {
            // no room to split: screen the run directly (never expected)
            for (int b = a; b <= e; b += 32) eval_candidates(c, b, min(e, b + 31), lane, S);
            continue;
        }
        // nearest the window on top: left of the window -> highest sub-run last
        const int below = __popc(mask & ((1u << lane) - 1u));
        const int pos = (e < w0) ? below : (cnt - 1 - below);
        if (keep) stack[sp + pos] = make_int2(ca, ce);
        sp += cnt;
        __syncwarp();
    }
    settle(c, S);
}

// How a row of a level is searched.
enum RowMode {
    kRowFull = 0,     // every run start in [kk, r]
    kRowAnchor = 1,   // the same, recording the near-optimal extent in NS[r]
    kRowBracket = 2,  // only the run starts between the extents of the two nearest anchors
};

// Anchored bracketing.  With V(r, l) = D[kk-1][l-1] + cost(l..r) in exact
// arithmetic, the interior cost satisfies the quadrangle inequality
// cost(a..c) + cost(b..d) <= cost(a..d) + cost(b..c) for a <= b <= c <= d (the
// squared error of contiguous cells of points on a line), and the D terms
// cancel, so for r1 < r2 and l < l':  V(r1,l) + V(r2,l') <= V(r1,l') + V(r2,l).
// Take an anchor row a < r and a minimiser l* of row a.  For l < l*:
// V(r,l) - V(r,l*) >= V(a,l) - V(a,l*), so every l below the anchor's
// near-optimal extent (V(a,l) > min_a + da) has V(r,l) > min_r + da; likewise,
// with an anchor a' > r, every l above its extent.  da is 2^-39 of the largest
// D[kk-1][x] over the rows the anchor serves, and min_r <= D[kk-1][r-1] (the
// run [r..r] costs 0), so da exceeds 2^9 times the rounding of the canonical
// fp64 values (under 2^-49 relative): no run start outside the bracket can
// win or tie the canonical minimum, and the bracketed rows give the full
// scan's result bit for bit.
__device__ void level_row(int B, int kk, int r, int stride, int mode, const DpWs& W, const Header& h, int lane,
                          int2* stack) {
    const int n1 = B + 1;
    const bool last = (kk == h.k_eff);
    const bool active = kk <= h.k_eff && r <= h.b && (last ? (r == h.b) : (r >= kk));
    uint64_t d = kInfBits;
    int al = 0;
    if (active) {
        RowCtx c;
        c.W = &W;
        c.Dp = W.D + static_cast<size_t>(kk - 1) * n1;
        c.Ep = W.E + static_cast<size_t>(kk - 1) * (n1 + 1);
        c.P0r = W.P0[r];
        c.P1r = W.P1[r];
        c.P2r = W.P2[r];
        c.B = B;
        c.r = r;
        c.last = last;
        float da = 0.0f;
        int lo = kk, hi = r;
        if (mode == kRowAnchor) {
            // rows served: (r - stride, r + stride), whose minima are at most
            // D[kk-1][x] for x in [r - stride, r + stride - 2]
            float dm = 0.0f;
            const int x0 = max(kk - 1, r - stride), x1 = min(h.b, r + stride - 2);
            for (int x = x0 + lane; x <= x1; x += 32) dm = fmaxf(dm, __ldca(&c.Ep[x + 1].x));
            dm = __uint_as_float(__reduce_max_sync(0xffffffffu, __float_as_uint(dm)));  // dm >= 0
            da = dm * 0x1p-39f;
        } else if (mode == kRowBracket) {
            const int a1 = (r / stride) * stride, a2 = min(a1 + stride, h.b);
            if (a1 >= kk) lo = max(lo, __ldcg(W.NS + a1).x);
            hi = min(hi, __ldcg(W.NS + a2).y);
            if (lo > hi) { lo = kk; hi = r; }  // never expected: the whole range
        }
        // hint: the previous level's split at r, moved by its share of the last cell
        const int hp = max(kk, __ldca(W.A + static_cast<size_t>(kk - 1) * n1 + r));
        const int hint = hp + (r - hp) / kk;
        Search S;
        search_init(S, da);
        search_row(c, kk, lo, hi, hint, lane, stack, S);
        const Best b = warp_min_best(S.bst);
        d = b.v;
        al = b.l;
        if (mode == kRowAnchor) {
            const int nlo = __reduce_min_sync(0xffffffffu, S.nlo);
            const int nhi = __reduce_max_sync(0xffffffffu, S.nhi);
            if (lane == 0) __stcg(W.NS + r, make_int2(nlo, nhi));
        }
    }
    if (lane == 0) {
        // stored past L1 (.cg): no SM may cache part of a row before the level ends
        __stcg(reinterpret_cast<unsigned long long*>(W.D) + static_cast<size_t>(kk) * n1 + r,
               static_cast<unsigned long long>(d));
        __stcg(W.A + static_cast<size_t>(kk) * n1 + r, al);
        const ff e = dbits_to_ff(d);
        float2* En = W.E + static_cast<size_t>(kk) * (n1 + 1);
        __stcg(En + r + 1, make_float2(e.hi, e.lo));
        if (r == 0) __stcg(En, make_float2(INFINITY, 0.0f));
    }
}

__device__ __forceinline__ uint32_t ld_acquire(const void* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

struct DpLaunch {
    int B, k;
    int stride;              // anchor spacing; 0: every row searched over its whole range
    uint32_t barrier_extra;  // added to every barrier target (0; a test hook makes it unreachable)
    long long spin;          // cycles a barrier wait may take before it gives up
};

// Grid barrier of the cooperative launch.  The wait gives up after P.spin
// cycles, or as soon as another CTA has given up (status 2), so a lost CTA
// cannot hang the GPU.  Returns true when the CTA must stop.
__device__ __forceinline__ bool grid_barrier(const DpWs& W, uint32_t target, long long spin, int* s_abort) {
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();  // this CTA's rows before its arrival
        atomicAdd(W.sync, 1u);
        const long long t0 = clock64();
        int ab = 0;
        while (ld_acquire(W.sync) < target) {
            if (ld_acquire(&W.hdr->status) != 0u || clock64() - t0 > spin) {
                ab = 1;
                atomicCAS(&W.hdr->status, 0, 2);
                break;
            }
        }
        *s_abort = ab;
    }
    __syncthreads();
    return *s_abort != 0;
}

// Rows 0..n-1 of one phase over the grid's warps: warp w of CTA c takes row
// w G + c (a CTA's warps spread over the whole range of end positions, so
// each SM holds wide and narrow searches alike), the rest come from the
// phase's counter.
template <int WARPS, class F>
__device__ __forceinline__ void for_rows(int n, uint32_t* counter, int gw, int nwarps, int lane, F&& f) {
    int i = (gw % WARPS) * static_cast<int>(gridDim.x) + gw / WARPS;
    while (i < n) {
        f(i);
        if (nwarps >= n) break;
        int ni = 0;
        if (lane == 0) ni = nwarps + static_cast<int>(atomicAdd(counter, 1u));
        i = __shfl_sync(0xffffffffu, ni, 0);
    }
}

// Levels 2..k in one cooperative launch (every CTA resident), a grid barrier
// between levels.  With anchors (P.stride > 0, interior levels), a level runs
// in two phases: the anchor rows r = 0, stride, 2 stride, ... and b, then
// (after a barrier) every other row, bracketed by its two anchors.
template <int WARPS>
__global__ void __launch_bounds__(WARPS * 32) k_dp_levels(DpLaunch P, DpWs W) {
    __shared__ int2 s_stack[WARPS][kStackCap];
    __shared__ int s_abort;
    const Header h = *W.hdr;
    if (h.status) return;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t G = gridDim.x;
    const int nwarps = static_cast<int>(G) * WARPS;
    const int gw = static_cast<int>(blockIdx.x) * WARPS + warp;
    const int B = P.B, S = P.stride;
    int2* stack = s_stack[warp];
    uint32_t nbar = 0;
    for (int kk = 2; kk <= P.k; ++kk) {
        uint32_t* ctr = W.sync + 1 + 3 * kk;
        if (S > 0 && kk < h.k_eff && h.b > S) {
            const int nA = h.b / S + 1 + (h.b % S ? 1 : 0);
            for_rows<WARPS>(nA, ctr + 1, gw, nwarps, lane,
                     [&](int i) { level_row(B, kk, min(i * S, h.b), S, kRowAnchor, W, h, lane, stack); });
            if (grid_barrier(W, ++nbar * G + P.barrier_extra, P.spin, &s_abort)) return;
            for_rows<WARPS>(B + 1, ctr + 2, gw, nwarps, lane, [&](int r) {
                if (r <= h.b && (r % S == 0 || r == h.b)) return;  // an anchor
                level_row(B, kk, r, S, kRowBracket, W, h, lane, stack);
            });
        } else {
            for_rows<WARPS>(B + 1, ctr, gw, nwarps, lane,
                     [&](int r) { level_row(B, kk, r, S, kRowFull, W, h, lane, stack); });
        }
        if (kk == P.k) break;
        if (grid_barrier(W, ++nbar * G + P.barrier_extra, P.spin, &s_abort)) return;
    }
}

// Backtrack the splits into cell starts and levels.  One CTA: thread 0 follows the split positions back from (k_eff, b) -- a
// chain of dependent loads -- and every thread then derives its levels (the
// count-weighted mean of each run of cells, two fp64 divisions) in parallel.
__global__ void k_dp_backtrack(int B, int k, DpWs W, float* __restrict__ codebook, int32_t* __restrict__ cell_start,
                               double* __restrict__ cost) {
    if (blockIdx.x != 0) return;
    __shared__ int start[kMaxLevels + 2];
    const Header h = *W.hdr;
    if (h.status) return;
    const int n1 = B + 1;
    const int b = h.b, ke = h.k_eff;
    if (b <= 1) {
        if (threadIdx.x != 0) return;
        for (int j = 0; j < k; ++j) {
            codebook[j] = 1.0f;
            if (cell_start) cell_start[j] = -1;
        }
        codebook[0] = -1.0f;
        if (cell_start && b == 1) cell_start[0] = W.idx[1];
        if (cost) {
            double c = 0.0;
            if (b == 1) c = u128_to_double_rn(fixed_num(W.P0[1], W.P1[1], W.P2[1], B, +1));
            *cost = c;
        }
        return;
    }
    if (threadIdx.x == 0) {
        int r = b;
        for (int kk = ke; kk >= 1; --kk) {
            const int l = W.A[static_cast<size_t>(kk) * n1 + r];
            start[kk] = l;
            r = l - 1;
        }
        if (cost) *cost = W.D[static_cast<size_t>(ke) * n1 + b];
    }
    __syncthreads();
    // level j = kk - 1; levels past k_eff repeat +1 (they are never the nearest)
    for (int j = threadIdx.x; j < k; j += blockDim.x) {
        const int kk = j + 1;
        if (kk > ke) {
            codebook[j] = 1.0f;
            if (cell_start) cell_start[j] = -1;
            continue;
        }
        const int l = start[kk];
        const int rr = (kk == ke) ? b : start[kk + 1] - 1;
        if (cell_start) cell_start[j] = W.idx[l];
        if (kk == 1) {
            codebook[j] = -1.0f;
        } else if (kk == ke) {
            codebook[j] = 1.0f;
        } else {
            const uint64_t s0 = W.P0[rr] - W.P0[l - 1];
            const int64_t s1 = W.P1[rr] - W.P1[l - 1];
            const double mu = __ddiv_rn(__ddiv_rn(__ll2double_rn(s1), __ull2double_rn(s0)), static_cast<double>(B));
            codebook[j] = __double2float_rn(mu);
        }
    }
}

}  // namespace

}  // namespace gefen

using namespace gefen;

namespace {

constexpr int kAnchorStride = 16;           // rows between anchors (automatic choice)
constexpr long long kBarrierSpin = 1ll << 31;  // about a second at the SM clock

// Test hooks (gefen_refit_debug): anchor stride (-1 automatic), barrier target
// offset, barrier wait limit (0: kBarrierSpin).
std::atomic<int> g_dbg_stride{-1};
std::atomic<uint32_t> g_dbg_barrier_extra{0};
std::atomic<long long> g_dbg_spin{0};

// Resident CTAs per SM of k_dp_levels<WARPS>, asked once per device.
template <int WARPS>
int dp_levels_per_sm() {
    static std::mutex mu;
    static int cached[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    std::lock_guard<std::mutex> g(mu);
    if (cached[dev] == 0) {
        int n = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_dp_levels<WARPS>, WARPS * 32, 0) != cudaSuccess) {
            (void)cudaGetLastError();
            return 0;
        }
        cached[dev] = n;
    }
    return cached[dev];
}

// Levels 2..k: one cooperative launch of k_dp_levels<WARPS>.
template <int WARPS>
cudaError_t launch_levels(int bins, int k, const DpWs& W, cudaStream_t st) {
    const int per_sm = dp_levels_per_sm<WARPS>();
    if (per_sm < 1) return cudaErrorLaunchFailure;
    const int rows = (bins + 1 + WARPS - 1) / WARPS;  // CTAs with a row each
    const int grid = std::max(1, std::min(per_sm * device_sm_count(), rows));
    DpLaunch P;
    P.B = bins;
    P.k = k;
    // anchors pay off once the rows outnumber the grid's warps: each warp
    // then searches one anchor row in full and brackets the rest
    const int auto_stride = (bins + 1 > 2 * grid * WARPS) ? kAnchorStride : 0;
    const int forced = g_dbg_stride.load();
    P.stride = forced >= 0 ? forced : auto_stride;
    P.barrier_extra = g_dbg_barrier_extra.load();
    const long long spin = g_dbg_spin.load();
    P.spin = spin > 0 ? spin : kBarrierSpin;
    DpWs w = W;
    void* args[] = {&P, &w};
    return cudaLaunchCooperativeKernel(reinterpret_cast<const void*>(k_dp_levels<WARPS>), dim3(grid), dim3(WARPS * 32),
                                       args, 0, st);
}

}  // namespace

extern "C" size_t gefen_refit_workspace_size(int32_t bins, int32_t k) {
    if (bins < 1 || bins > GEFEN_MAX_BINS || k < 2 || k > GEFEN_MAX_LEVELS) return 0;
    return dp_layout(bins, k).total;
}

extern "C" gefen_status_t gefen_refit_codebook(const float* x, int64_t n, const uint64_t* hist_in, int32_t bins,
                                               int32_t k, float* codebook_out, uint64_t* hist_out,
                                               int32_t* cell_start_out, double* cost_out, void* workspace,
                                               size_t workspace_bytes, gefen_stream_t stream) {
    if (bins < 1 || bins > GEFEN_MAX_BINS || k < 2 || k > GEFEN_MAX_LEVELS) return GEFEN_EINVAL;
    if (codebook_out == nullptr) return GEFEN_EINVAL;
    if (x == nullptr && hist_in == nullptr) return GEFEN_EINVAL;
    if (x != nullptr && (n < 0 || n > (int64_t(1) << 40) || (reinterpret_cast<uintptr_t>(x) & 15u))) return GEFEN_EINVAL;
    const size_t need = gefen_refit_workspace_size(bins, k);
    if (workspace == nullptr || workspace_bytes < need) return GEFEN_ENOMEM;
    if (reinterpret_cast<uintptr_t>(workspace) % kWsAlign) return GEFEN_EINVAL;
    if (gefen_status_t s = check_device(); s != GEFEN_OK) return s;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const DpLayout L = dp_layout(bins, k);
    uint64_t* wh = reinterpret_cast<uint64_t*>(static_cast<char*>(workspace) + L.hist);
    const DpWs W = dp_ws(workspace, bins, k);
    const uint64_t* h = hist_in;
    if (x != nullptr) {
        uint64_t* dst = hist_out ? hist_out : wh;
        if (cudaMemsetAsync(dst, 0, static_cast<size_t>(bins) * sizeof(uint64_t), st) != cudaSuccess) return GEFEN_ECUDA;
        if (n > 0) {
            HistRange rr{0, n};
            if (launch_histogram(x, &rr, 1, bins, dst, st) != cudaSuccess) return GEFEN_ECUDA;
        }
        h = dst;
    } else if (hist_out != nullptr && hist_out != hist_in) {
        if (cudaMemcpyAsync(hist_out, hist_in, static_cast<size_t>(bins) * sizeof(uint64_t), cudaMemcpyDeviceToDevice,
                            st) != cudaSuccess)
            return GEFEN_ECUDA;
    }
    k_dp_prefix<<<1, kPrefixThreads, 0, st>>>(h, bins, k, W);
    const int grid1 = (bins + 2 + kDpThreads - 1) / kDpThreads;
    k_dp_level1<<<grid1, kDpThreads, 0, st>>>(bins, W);
    const cudaError_t el = (bins > kDpSmallBins) ? launch_levels<kDpWarpsLarge>(bins, k, W, st)
                                                 : launch_levels<kDpWarpsSmall>(bins, k, W, st);
    if (el != cudaSuccess) return GEFEN_ECUDA;
    k_dp_backtrack<<<1, 256, 0, st>>>(bins, k, W, codebook_out, cell_start_out, cost_out);
    if (cudaGetLastError() != cudaSuccess) return GEFEN_ECUDA;
    return GEFEN_OK;
}

extern "C" gefen_status_t gefen_refit_status(const void* workspace, int32_t* k_eff_out, gefen_stream_t stream) {
    if (workspace == nullptr) return GEFEN_EINVAL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    Header h;
    if (cudaMemcpyAsync(&h, workspace, sizeof(h), cudaMemcpyDeviceToHost, st) != cudaSuccess) return GEFEN_ECUDA;
    if (cudaStreamSynchronize(st) != cudaSuccess) return GEFEN_ECUDA;
    if (k_eff_out) *k_eff_out = h.k_eff;
    if (h.status == 2) return GEFEN_ETIMEOUT;
    return h.status ? GEFEN_EDEVICE : GEFEN_OK;
}

extern "C" gefen_status_t gefen_refit_tables(const void* workspace, int32_t bins, int32_t k, double* dtable_out,
                                             int32_t* argl_out, gefen_stream_t stream) {
    if (workspace == nullptr || bins < 1 || bins > GEFEN_MAX_BINS || k < 2 || k > GEFEN_MAX_LEVELS)
        return GEFEN_EINVAL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const char* ws = static_cast<const char*>(workspace);
    const DpLayout L = dp_layout(bins, k);
    const size_t cnt = static_cast<size_t>(k + 1) * (static_cast<size_t>(bins) + 1);
    if (dtable_out &&
        cudaMemcpyAsync(dtable_out, ws + L.D, cnt * sizeof(double), cudaMemcpyDeviceToDevice, st) != cudaSuccess)
        return GEFEN_ECUDA;
    if (argl_out &&
        cudaMemcpyAsync(argl_out, ws + L.A, cnt * sizeof(int32_t), cudaMemcpyDeviceToDevice, st) != cudaSuccess)
        return GEFEN_ECUDA;
    return GEFEN_OK;
}

// ---------------------------------------------------------------------------
// Refit without a caller workspace.  The scratch the refit needs lives in one
// file-scope device array sized for the largest request it accepts: 4096
// histogram cells (16 cells per level at 256 levels) and 256 levels.  Every
// device that loads this library holds the array until the process exits.
namespace {

constexpr int kStaticMaxBins = 4096;
constexpr int kStaticMaxLevels = 256;

constexpr size_t kStaticScratchBytes = dp_layout(kStaticMaxBins, kStaticMaxLevels).total;

__device__ __align__(256) unsigned char g_refit_scratch[kStaticScratchBytes];

// Device address of the array, looked up once per device.
std::mutex g_scratch_mu;
void* g_scratch_addr[64] = {nullptr};

gefen_status_t static_scratch(void** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return GEFEN_ECUDA;
    std::lock_guard<std::mutex> g(g_scratch_mu);
    if (g_scratch_addr[dev] == nullptr) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_refit_scratch) != cudaSuccess || p == nullptr) {
            (void)cudaGetLastError();
            return GEFEN_ECUDA;
        }
        // load the refit's kernels now as well, so that a later call needs
        // nothing more from the driver
        cudaFuncAttributes fa;
        if (cudaFuncGetAttributes(&fa, k_dp_prefix) != cudaSuccess ||
            cudaFuncGetAttributes(&fa, k_dp_level1) != cudaSuccess ||
            cudaFuncGetAttributes(&fa, k_dp_levels<kDpWarpsSmall>) != cudaSuccess ||
            cudaFuncGetAttributes(&fa, k_dp_levels<kDpWarpsLarge>) != cudaSuccess ||
            cudaFuncGetAttributes(&fa, k_dp_backtrack) != cudaSuccess || dp_levels_per_sm<kDpWarpsSmall>() < 1 ||
            dp_levels_per_sm<kDpWarpsLarge>() < 1 ||
            prepare_histogram() != cudaSuccess) {
            (void)cudaGetLastError();
            return GEFEN_ECUDA;
        }
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return GEFEN_OK;
}

}  // namespace

extern "C" gefen_status_t gefen_refit_static_init(void) {
    if (gefen_status_t s = check_device(); s != GEFEN_OK) return s;
    void* scratch = nullptr;
    return static_scratch(&scratch);
}

extern "C" gefen_status_t gefen_refit_codebook_static(const float* x, int64_t n, const uint64_t* hist_in,
                                                      int32_t bins, int32_t k, float* codebook_out,
                                                      uint64_t* hist_out, int32_t* cell_start_out,
                                                      double* cost_out, gefen_stream_t stream) {
    if (bins < 1 || k < 2 || codebook_out == nullptr || (x == nullptr && hist_in == nullptr)) return GEFEN_EINVAL;
    if (bins > kStaticMaxBins || k > kStaticMaxLevels) return GEFEN_EUNSUPPORTED;
    if (dp_layout(bins, k).total > kStaticScratchBytes) return GEFEN_EUNSUPPORTED;
    void* scratch = nullptr;
    if (gefen_status_t s = static_scratch(&scratch); s != GEFEN_OK) return s;
    return gefen_refit_codebook(x, n, hist_in, bins, k, codebook_out, hist_out, cell_start_out, cost_out, scratch,
                                kStaticScratchBytes, stream);
}

extern "C" gefen_status_t gefen_refit_static_status(int32_t* k_eff_out, gefen_stream_t stream) {
    void* scratch = nullptr;
    if (gefen_status_t s = static_scratch(&scratch); s != GEFEN_OK) return s;
    return gefen_refit_status(scratch, k_eff_out, stream);
}

extern "C" gefen_status_t gefen_refit_debug(int32_t anchor_stride, uint32_t barrier_extra,
                                            int64_t barrier_spin_cycles) {
    if (anchor_stride < -1 || anchor_stride > GEFEN_MAX_BINS || barrier_spin_cycles < 0) return GEFEN_EINVAL;
    g_dbg_stride.store(anchor_stride);
    g_dbg_barrier_extra.store(barrier_extra);
    g_dbg_spin.store(barrier_spin_cycles);
    return GEFEN_OK;
}
