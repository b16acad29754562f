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
// One launch per level, one thread per end position r.  Instead of evaluating
// all O(r) candidates in fp64 (slow on this part), each candidate is screened
// in fp32 from the exact 128-bit numerator: the screened value v32 is within
// 4e-7 relative of the canonical value, so [v32(1-2^-20), v32(1+2^-20)]
// brackets it.  Whole runs of candidates are excluded with two exact facts:
// the interior cost of [l..r] does not increase as l grows (a subset has no
// larger squared error) and D[.][k'-1] does not decrease along r (more cells
// for the same levels never cost less).  So for l in [a, e]:
//   value(l) >= D[a-1][k'-1] + cost(e..r),   and for l >= a: value(l) >= D[a-1].
// Candidates that survive (typically a handful near the optimum) are evaluated
// with the canonical fp64 formula; the minimum over them, with ties to the
// smallest l, equals the full scan bit for bit.
#include <algorithm>
#include <cmath>

#include "common.cuh"
#include "internal.h"

namespace gefen {

namespace {

constexpr int kDpThreads = 128;
constexpr float kMLo = 1.0f - 9.5367431640625e-07f;  // 1 - 2^-20
constexpr float kMHi = 1.0f + 9.5367431640625e-07f;  // 1 + 2^-20

struct Header {
    int32_t status;  // 0 ok, 1 moment overflow (N (B-1)^2 >= 2^64)
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
    float* E;      // 2 x (B+2): E[l] = float(D[level][l-1]) for the next level
};

struct DpLayout {
    size_t hdr, hist, idx, P0, P1, P2, D, A, E, total;
};

// Workspace: status header at offset 0 (so it can be read without knowing the
// sizes), the histogram copy, then the DP arrays.
DpLayout dp_layout(int B, int k) {
    DpLayout L;
    size_t o = 0;
    const size_t n1 = static_cast<size_t>(B) + 1;
    L.hdr = o; o += align_up(sizeof(Header));
    L.hist = o; o += align_up(static_cast<size_t>(B) * sizeof(uint64_t));
    L.idx = o; o += align_up(n1 * sizeof(int32_t));
    L.P0 = o;  o += align_up(n1 * sizeof(uint64_t));
    L.P1 = o;  o += align_up(n1 * sizeof(int64_t));
    L.P2 = o;  o += align_up(n1 * sizeof(uint64_t));
    L.D = o;   o += align_up(static_cast<size_t>(k + 1) * n1 * sizeof(double));
    L.A = o;   o += align_up(static_cast<size_t>(k + 1) * n1 * sizeof(int32_t));
    L.E = o;   o += align_up(2 * (n1 + 1) * sizeof(float));
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
    w.E = reinterpret_cast<float*>(p + L.E);
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

__device__ __forceinline__ float cost32_interior(const Run& q) {
    return u128_to_float_approx(interior_num(q.s0, q.s1, q.s2)) * __frcp_rn(__ull2float_rn(q.s0));
}

__device__ __forceinline__ double cost64_interior(const Run& q) {
    return __ddiv_rn(u128_to_double_rn(interior_num(q.s0, q.s1, q.s2)), __ull2double_rn(q.s0));
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
    double d = INFINITY;
    if (r >= 1 && r <= h.b) {
        d = u128_to_double_rn(fixed_num(W.P0[r], W.P1[r], W.P2[r], B, +1));
    }
    if (r >= 0) {
        W.D[n1 + r] = d;
        W.A[n1 + r] = (r >= 1 && r <= h.b) ? 1 : 0;
    }
    W.E[1 * (n1 + 1) + g] = __double2float_rn(d);  // row 1 of the rolling E buffer
}

// Candidate screen + canonical evaluation for one (r, level) -- interior.
struct Best {
    double v;
    int l;
};

__device__ __forceinline__ void take(Best& b, double v, int l) {
    if (v < b.v || (v == b.v && l < b.l)) { b.v = v; b.l = l; }
}

__device__ __forceinline__ Best search_interior(const DpWs& W, const double* __restrict__ Dp,
                                                const float* __restrict__ Ep, int kk, int r, int hint) {
    const uint64_t P0r = W.P0[r], P2r = W.P2[r];
    const int64_t P1r = W.P1[r];
    float best_hi = INFINITY;
    Best bst{INFINITY, 0};
    // 1. a window of 32 candidates around the hint
    int w0 = max(kk, hint - 8);
    const int w1 = min(r, w0 + 31);
    w0 = max(kk, w1 - 31);
    for (int l = w0; l <= w1; ++l) {
        const float v = __ldg(Ep + l) + cost32_interior(run_of(W, l, P0r, P1r, P2r));
        best_hi = fminf(best_hi, v * kMHi);
    }
    auto eval = [&](int l) {
        const Run q = run_of(W, l, P0r, P1r, P2r);
        const float v = __ldg(Ep + l) + cost32_interior(q);
        best_hi = fminf(best_hi, v * kMHi);
        if (v * kMLo <= best_hi) take(bst, __dadd_rn(__ldg(Dp + l - 1), cost64_interior(q)), l);
    };
    for (int l = w0; l <= w1; ++l) eval(l);
    // 2. runs of 32 to the left: stop once even the smallest D plus the cost of
    //    [e..r] exceeds the best (it only grows leftwards)
    const float e_min = __ldg(Ep + kk);
    for (int e = w0 - 1; e >= kk;) {
        const int a = max(kk, e - 31);
        const float ce = cost32_interior(run_of(W, e, P0r, P1r, P2r));
        if ((e_min + ce) * kMLo > best_hi) break;
        if ((__ldg(Ep + a) + ce) * kMLo <= best_hi)
            for (int l = e; l >= a; --l) eval(l);
        e = a - 1;
    }
    // 3. runs of 32 to the right: stop once D alone exceeds the best
    for (int a = w1 + 1; a <= r;) {
        const float ea = __ldg(Ep + a);
        if (ea * kMLo > best_hi) break;
        const int e = min(r, a + 31);
        const float ce = cost32_interior(run_of(W, e, P0r, P1r, P2r));
        if ((ea + ce) * kMLo <= best_hi)
            for (int l = a; l <= e; ++l) eval(l);
        a = e + 1;
    }
    return bst;
}

// Interior level kk (2 <= kk < k_eff), or the last level kk == k_eff (only
// r = b, scanned by CTA 0), or nothing (kk > k_eff).  Thread g covers r = g-1.
__global__ void __launch_bounds__(kDpThreads) k_dp_level(int B, int kk, DpWs W) {
    const Header h = *W.hdr;
    if (h.status) return;
    const int n1 = B + 1;
    const int g = blockIdx.x * blockDim.x + threadIdx.x;
    const int r = g - 1;
    const double* Dp = W.D + static_cast<size_t>(kk - 1) * n1;
    const float* Ep = W.E + static_cast<size_t>((kk - 1) & 1) * (n1 + 1);
    float* En = W.E + static_cast<size_t>(kk & 1) * (n1 + 1);
    double* Dk = W.D + static_cast<size_t>(kk) * n1;
    int32_t* Ak = W.A + static_cast<size_t>(kk) * n1;

    if (kk == h.k_eff) {
        // Last level (centre +1): one r = b, candidates split over CTA 0.
        if (blockIdx.x == 0) {
            __shared__ float s_hi[kDpThreads];
            __shared__ double s_v[kDpThreads];
            __shared__ int s_l[kDpThreads];
            const int b = h.b;
            const uint64_t P0r = W.P0[b], P2r = W.P2[b];
            const int64_t P1r = W.P1[b];
            float hi = INFINITY;
            for (int l = kk + threadIdx.x; l <= b; l += blockDim.x) {
                const Run q = run_of(W, l, P0r, P1r, P2r);
                const float v = Ep[l] + u128_to_float_approx(fixed_num(q.s0, q.s1, q.s2, B, -1));
                hi = fminf(hi, v * kMHi);
            }
            s_hi[threadIdx.x] = hi;
            __syncthreads();
            for (int o = blockDim.x / 2; o > 0; o >>= 1) {
                if (threadIdx.x < o) s_hi[threadIdx.x] = fminf(s_hi[threadIdx.x], s_hi[threadIdx.x + o]);
                __syncthreads();
            }
            const float best_hi = s_hi[0];
            Best bst{INFINITY, 0};
            for (int l = kk + threadIdx.x; l <= b; l += blockDim.x) {
                const Run q = run_of(W, l, P0r, P1r, P2r);
                const u128 num = fixed_num(q.s0, q.s1, q.s2, B, -1);
                const float v = Ep[l] + u128_to_float_approx(num);
                if (v * kMLo <= best_hi) take(bst, __dadd_rn(Dp[l - 1], u128_to_double_rn(num)), l);
            }
            s_v[threadIdx.x] = bst.v;
            s_l[threadIdx.x] = bst.l;
            __syncthreads();
            for (int o = blockDim.x / 2; o > 0; o >>= 1) {
                if (threadIdx.x < o) {
                    Best a{s_v[threadIdx.x], s_l[threadIdx.x]};
                    take(a, s_v[threadIdx.x + o], s_l[threadIdx.x + o]);
                    s_v[threadIdx.x] = a.v;
                    s_l[threadIdx.x] = a.l;
                }
                __syncthreads();
            }
            if (threadIdx.x == 0) {
                Dk[b] = s_v[0];
                Ak[b] = s_l[0];
            }
        }
        if (r >= 0 && r <= B && r != h.b) {
            Dk[r] = INFINITY;
            Ak[r] = 0;
        }
        return;
    }
    if (g > B + 1) return;
    double d = INFINITY;
    int al = 0;
    if (kk < h.k_eff && r >= kk && r <= h.b) {
        // hint: the previous level's split at r, moved right by its share of
        // the last cell
        const int hp = max(kk, W.A[static_cast<size_t>(kk - 1) * n1 + r]);
        const int hint = hp + (r - hp) / kk;
        const Best bst = search_interior(W, Dp, Ep, kk, r, hint);
        d = bst.v;
        al = bst.l;
    }
    if (r >= 0) {
        Dk[r] = d;
        Ak[r] = al;
    }
    En[g] = __double2float_rn(d);
}

// Backtrack the splits into cell starts and levels (one thread).
__global__ void k_dp_backtrack(int B, int k, DpWs W, float* __restrict__ codebook, int32_t* __restrict__ cell_start,
                               double* __restrict__ cost) {
    if (threadIdx.x != 0 || blockIdx.x != 0) return;
    const Header h = *W.hdr;
    if (h.status) return;
    const int n1 = B + 1;
    const int b = h.b, ke = h.k_eff;
    for (int j = 0; j < k; ++j) {
        codebook[j] = 1.0f;
        if (cell_start) cell_start[j] = -1;
    }
    codebook[0] = -1.0f;
    if (b <= 1) {
        if (cell_start && b == 1) cell_start[0] = W.idx[1];
        if (cost) {
            double c = 0.0;
            if (b == 1) c = u128_to_double_rn(fixed_num(W.P0[1], W.P1[1], W.P2[1], B, +1));
            *cost = c;
        }
        return;
    }
    int r = b;
    int start[kMaxLevels + 1];
    for (int kk = ke; kk >= 1; --kk) {
        const int l = W.A[static_cast<size_t>(kk) * n1 + r];
        start[kk] = l;
        r = l - 1;
    }
    for (int kk = 1; kk <= ke; ++kk) {
        const int l = start[kk];
        const int rr = (kk == ke) ? b : start[kk + 1] - 1;
        if (cell_start) cell_start[kk - 1] = W.idx[l];
        if (kk == 1) {
            codebook[0] = -1.0f;
        } else if (kk == ke) {
            codebook[kk - 1] = 1.0f;
        } else {
            const uint64_t s0 = W.P0[rr] - W.P0[l - 1];
            const int64_t s1 = W.P1[rr] - W.P1[l - 1];
            const double mu = __ddiv_rn(__ddiv_rn(__ll2double_rn(s1), __ull2double_rn(s0)), static_cast<double>(B));
            codebook[kk - 1] = __double2float_rn(mu);
        }
    }
    if (cost) *cost = W.D[static_cast<size_t>(ke) * n1 + b];
}

}  // namespace

}  // namespace gefen

using namespace gefen;

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
    const int grid = (bins + 2 + kDpThreads - 1) / kDpThreads;
    k_dp_level1<<<grid, kDpThreads, 0, st>>>(bins, W);
    for (int kk = 2; kk <= k; ++kk) k_dp_level<<<grid, kDpThreads, 0, st>>>(bins, kk, W);
    k_dp_backtrack<<<1, 32, 0, st>>>(bins, k, W, codebook_out, cell_start_out, cost_out);
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
