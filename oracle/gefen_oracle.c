/*
 * Gefen CPU oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, obviously-correct restatement of what the Gefen paper
 * (arXiv 2606.13894, "Gefen: Optimized Stochastic Optimizer") defines for its
 * data-parallel hot path.  Only the test suite, the smoke check and the CPU
 * baseline leg of the benchmark may load this file's library; the product
 * path (the CUDA library) never does, and shares no code with it.
 *
 * Everything is computed in double precision unless a decision that yields an
 * integer is defined on fp32 inputs (histogram bins of fp32 values, Sec. 5.1.1 /
 * Algorithm 3), where the fp32 formula is spelled out.  Build with
 * -ffp-contract=off so that no multiply-add is fused.
 *
 * Parity status of each function (what pins it, other than itself) is listed in
 * tests/ and summarised in the design notes:
 *   oracle_step              pinned (closed-form AdamW reduction, invariants)
 *   oracle_step_unquantized  pinned (torch AdamW, closed form at t=1)
 *   oracle_histogram         pinned (hand-made edge values, counts sum to N)
 *   oracle_dp                pinned (brute force over partitions/labelings,
 *                                    centroid condition, Lloyd-Max bound)
 *   oracle_infer_blocks      pinned (planted periods, prime n, direct S(p),
 *                                    divisor-count maxima printed in Sec. 5.1)
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef unsigned __int128 u128;
typedef __int128 i128;

int oracle_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Threads of the parallel loops below (blocks of a step, divisors, rows of a
 * DP level); every result is the same for any count. */
void oracle_set_num_threads(int32_t n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* bf16 bit pattern -> float (exact: bf16 is the upper half of an fp32). */
static double bf16_to_double(uint16_t b) {
    uint32_t u = ((uint32_t)b) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* ------------------------------------------------------------------------ */
/* Histogram bin of a normalised value (Algorithm 3: "histogram counts over   */
/* [-1,1]").  B uniform cells; bin(x) = clamp(floor((x + 1) * (B/2)), 0, B-1) */
/* with the add and the multiply each rounded to fp32.  +1 lands in the last  */
/* cell.  NaN is counted in no cell (returns -1).                             */
/* ------------------------------------------------------------------------ */
int64_t oracle_bin(float x, int32_t B) {
    if (isnan(x)) return -1;
    float t = x + 1.0f;
    float u = t * (0.5f * (float)B);
    float f = floorf(u);
    if (f < 0.0f) return 0;
    if (f > (float)(B - 1)) return B - 1;
    return (int64_t)f;
}

/* Plain histogram of an fp32 array (Algorithm 3, "accumulate all entries"). */
void oracle_histogram(const float* x, int64_t n, int32_t B, uint64_t* hist) {
    for (int64_t i = 0; i < n; ++i) {
        int64_t b = oracle_bin(x[i], B);
        if (b >= 0) hist[b] += 1;
    }
}

/* ------------------------------------------------------------------------ */
/* Nearest codebook level (Sec. 5.1.1: Quantize).  argmin_j |x - C[j]|,      */
/* ties to the lower index.  Distances are taken in double.                  */
/* ------------------------------------------------------------------------ */
static int nearest_level(double x, const float* C, int k) {
    int best = 0;
    double bd = fabs(x - (double)C[0]);
    for (int j = 1; j < k; ++j) {
        double d = fabs(x - (double)C[j]);
        if (d < bd) { bd = d; best = j; }
    }
    return best;
}

int32_t oracle_nearest_level(double x, const float* C, int32_t k) {
    return nearest_level(x, C, k);
}

/* ------------------------------------------------------------------------ */
/* One Gefen step on one flattened tensor (Algorithm 1, loop body).          */
/*                                                                          */
/* Blocks are consecutive runs of p elements (p | n).  Per block b:          */
/*   m_i   = beta1 * Cdec[c_i] * s_b + (1 - beta1) * g_i        (momentum)  */
/*   s'_b  = max_i |m_i|                                        (Quantize)  */
/*   v'_b  = beta2 * v_b + (1 - beta2) * mean_i g_i^2           (shared v)  */
/*   theta_i -= lr * ( (m_i / (1-beta1^t)) / (sqrt(v'_b/(1-beta2^t)) + eps) */
/*                     + wd * theta_i )                         (update)    */
/*   c'_i  = nearest level of m_i / s'_b in Cenc ; s_b = s'_b               */
/* The update uses the unquantised m_i.  A block with s'_b = 0 stores the   */
/* level nearest to 0 for every element and contributes nothing to the      */
/* histogram.  hist_mode: 0 none; 1 histogram x_i = m_i/s'_b (refit input);  */
/* 2 histogram g_i / max|g| of each nonzero block and update nothing else   */
/* (Algorithm 3's input built from the first gradient).                     */
/* Histogram decisions take x rounded to fp32, the binning precision.       */
/* Returns 0 on success, -1 on bad arguments.                               */
/* ------------------------------------------------------------------------ */
int oracle_step(int64_t n, int64_t p, float* theta, const uint16_t* grad,
                uint8_t* codes, float* v, float* s, const float* cb_dec,
                const float* cb_enc, int32_t k, double lr, double beta1,
                double beta2, double eps, double wd, int64_t t,
                uint64_t* hist, int32_t bins, int32_t hist_mode) {
    if (n < 0 || p < 1 || (n % p) != 0 || k < 2 || k > 256 || t < 1) return -1;
    if (hist_mode != 0 && (hist == NULL || bins < 1)) return -1;
    const int64_t nb = n / p;
    const double bc1 = 1.0 - pow(beta1, (double)t);
    const double bc2 = 1.0 - pow(beta2, (double)t);
    const int zero_code = nearest_level(0.0, cb_enc, k);
    int failed = 0;
    /* blocks are independent (each thread keeps its own m); histogram
     * counts are added atomically, so every result is the serial one */
    #pragma omp parallel reduction(|:failed)
    {
    double* m = (double*)malloc(sizeof(double) * (size_t)(p > 0 ? p : 1));
    if (!m) failed = 1;
    #pragma omp for schedule(static)
    for (int64_t b = 0; b < nb; ++b) {
        if (!m) continue;
        const int64_t o = b * p;
        if (hist_mode == 2) {
            double amax = 0.0;
            for (int64_t i = 0; i < p; ++i) {
                double g = fabs(bf16_to_double(grad[o + i]));
                if (g > amax) amax = g;
            }
            if (amax > 0.0) {
                float a32 = (float)amax; /* exact: amax is an fp32 value */
                for (int64_t i = 0; i < p; ++i) {
                    float x = (float)bf16_to_double(grad[o + i]) / a32;
                    int64_t bi = oracle_bin(x, bins);
                    if (bi >= 0) {
                        #pragma omp atomic
                        hist[bi] += 1;
                    }
                }
            }
            continue;
        }
        double smax = 0.0, g2 = 0.0;
        const double sb = (double)s[b];
        for (int64_t i = 0; i < p; ++i) {
            double g = bf16_to_double(grad[o + i]);
            double mi = beta1 * ((double)cb_dec[codes[o + i]] * sb) + (1.0 - beta1) * g;
            m[i] = mi;
            if (fabs(mi) > smax) smax = fabs(mi);
            g2 += g * g;
        }
        const double G = g2 / (double)p;
        const double vnew = beta2 * (double)v[b] + (1.0 - beta2) * G;
        const double vhat = vnew / bc2;
        const double denom = sqrt(vhat) + eps;
        for (int64_t i = 0; i < p; ++i) {
            double th = (double)theta[o + i];
            double mhat = m[i] / bc1;
            th = th - lr * (mhat / denom + wd * th);
            theta[o + i] = (float)th;
        }
        if (smax > 0.0) {
            for (int64_t i = 0; i < p; ++i) {
                double x = m[i] / smax;
                codes[o + i] = (uint8_t)nearest_level(x, cb_enc, k);
                if (hist_mode == 1) {
                    int64_t bi = oracle_bin((float)x, bins);
                    if (bi >= 0) {
                        #pragma omp atomic
                        hist[bi] += 1;
                    }
                }
            }
        } else {
            for (int64_t i = 0; i < p; ++i) codes[o + i] = (uint8_t)zero_code;
        }
        v[b] = (float)vnew;
        s[b] = (float)smax;
    }
    free(m);
    }
    return failed ? -1 : 0;
}

/* Momenta (unquantised) of one step, for margin checks: m_i as in
 * oracle_step, and s'_b.  Writes m (n doubles) and smax (n/p doubles). */
int oracle_step_momentum(int64_t n, int64_t p, const uint16_t* grad,
                         const uint8_t* codes, const float* s,
                         const float* cb_dec, double beta1, double* m,
                         double* smax) {
    if (n < 0 || p < 1 || (n % p) != 0) return -1;
    for (int64_t b = 0; b < n / p; ++b) {
        double mx = 0.0;
        for (int64_t i = b * p; i < (b + 1) * p; ++i) {
            double g = bf16_to_double(grad[i]);
            m[i] = beta1 * ((double)cb_dec[codes[i]] * (double)s[b]) + (1.0 - beta1) * g;
            if (fabs(m[i]) > mx) mx = fabs(m[i]);
        }
        smax[b] = mx;
    }
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Unquantised variant: m kept in double, one v per block.  With p = 1 this */
/* is textbook AdamW (Sec. 3, Adam/AdamW equations with decoupled decay).   */
/* ------------------------------------------------------------------------ */
int oracle_step_unquantized(int64_t n, int64_t p, double* theta,
                            const double* g, double* m, double* v, double lr,
                            double beta1, double beta2, double eps, double wd,
                            int64_t t) {
    if (n < 0 || p < 1 || (n % p) != 0 || t < 1) return -1;
    const double bc1 = 1.0 - pow(beta1, (double)t);
    const double bc2 = 1.0 - pow(beta2, (double)t);
    for (int64_t b = 0; b < n / p; ++b) {
        double g2 = 0.0;
        for (int64_t i = b * p; i < (b + 1) * p; ++i) {
            m[i] = beta1 * m[i] + (1.0 - beta1) * g[i];
            g2 += g[i] * g[i];
        }
        v[b] = beta2 * v[b] + (1.0 - beta2) * (g2 / (double)p);
        const double denom = sqrt(v[b] / bc2) + eps;
        for (int64_t i = b * p; i < (b + 1) * p; ++i) {
            theta[i] = theta[i] - lr * ((m[i] / bc1) / denom + wd * theta[i]);
        }
    }
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Exact histogram DP quantizer (Algorithm 3; Appendix D).                   */
/*                                                                          */
/* Nonempty bins j = 1..b in ascending order, bin centre m_j = u_j / B with */
/* the odd integer u_j = 2*i_j + 1 - B.  Costs are in units of 1/B^2 and are */
/* built from exact integer moments of a run of bins [l..r]:                */
/*   s0 = sum c, s1 = sum c*u, s2 = sum c*u^2                               */
/*   interior level (free centre = weighted mean):                          */
/*       cost = (double)(s0*s2 - s1^2) / (double)s0                         */
/*   first level (centre -1, i.e. u = -B):  (double)(s2 + 2B s1 + B^2 s0)    */
/*   last level  (centre +1, i.e. u = +B):  (double)(s2 - 2B s1 + B^2 s0)    */
/* Each integer is exact (128-bit) and converted once with round-to-nearest; */
/* Appendix D's S2 - S1^2/S0 and S2 - 2aS1 + a^2S0 are these expressions.    */
/*                                                                          */
/* Recurrence (levels k' = 1..k; every level holds >= 1 nonempty bin):     */
/*   D[r][1]  = cost_first(1..r)                                            */
/*   D[r][k'] = min_{k' <= l <= r} D[l-1][k'-1] + cost_interior(l..r)       */
/*   D[b][k]  = min_{k  <= l <= b} D[l-1][k-1]  + cost_last(l..b)           */
/* Ties go to the smallest l.  Backtracking gives each level's first bin.   */
/* Levels: C[0] = -1, C[k-1] = +1, interior C = (s1/s0)/B rounded to fp32.   */
/*                                                                          */
/* If fewer than k bins are nonempty, the DP runs with k_eff = b levels      */
/* (b >= 2) and the codebook is padded with +1; with b <= 1 the codebook is  */
/* [-1, +1, +1, ...].  Returns k_eff, or -1 on bad arguments.               */
/*                                                                          */
/* dtable (nullable, (k_eff+1) x (b+1) doubles, row-major by level) receives */
/* every D[r][k'] the loops define (others = +inf); argl (nullable, same    */
/* shape, int32) receives the minimising l (1-based), or 0 where undefined.  */
/* ------------------------------------------------------------------------ */
typedef struct {
    int64_t b;
    int32_t B;
    uint64_t* P0;
    int64_t* P1;
    uint64_t* P2;
} dp_moments;

static void dp_cell(const dp_moments* M, int64_t l, int64_t r, uint64_t* s0,
                    int64_t* s1, uint64_t* s2) {
    *s0 = M->P0[r] - M->P0[l - 1];
    *s1 = M->P1[r] - M->P1[l - 1];
    *s2 = M->P2[r] - M->P2[l - 1];
}

static double cost_interior(const dp_moments* M, int64_t l, int64_t r) {
    uint64_t s0, s2;
    int64_t s1;
    dp_cell(M, l, r, &s0, &s1, &s2);
    u128 a = (u128)s0 * (u128)s2;
    uint64_t as1 = (uint64_t)(s1 < 0 ? -s1 : s1);
    u128 c = (u128)as1 * (u128)as1;
    u128 num = a - c; /* >= 0 by Cauchy-Schwarz */
    return (double)num / (double)s0;
}

static double cost_fixed(const dp_moments* M, int64_t l, int64_t r, int sign) {
    uint64_t s0, s2;
    int64_t s1;
    dp_cell(M, l, r, &s0, &s1, &s2);
    i128 B = (i128)M->B;
    i128 val = (i128)s2 + (i128)(2 * sign) * B * (i128)s1 + B * B * (i128)s0;
    return (double)(u128)val;
}

int32_t oracle_dp(const uint64_t* hist, int32_t B, int32_t k, float* codebook,
                  int32_t* cell_start, double* cost_out, double* dtable,
                  int32_t* argl) {
    if (B < 1 || k < 2 || k > 256) return -1;
    int64_t b = 0;
    u128 N = 0;
    for (int32_t i = 0; i < B; ++i) { b += (hist[i] != 0); N += hist[i]; }
    /* exact 64-bit moments need N * (B-1)^2 < 2^64 */
    if (N * (u128)((uint64_t)(B - 1) * (uint64_t)(B - 1)) >= ((u128)1 << 64)) return -1;
    for (int32_t j = 0; j < k; ++j) { codebook[j] = 1.0f; if (cell_start) cell_start[j] = -1; }
    codebook[0] = -1.0f;
    if (b <= 1) {
        if (cell_start && b == 1) {
            for (int32_t i = 0; i < B; ++i) if (hist[i]) { cell_start[0] = i; break; }
        }
        if (cost_out) {
            double c = 0.0;
            for (int32_t i = 0; i < B; ++i) if (hist[i]) {
                int64_t u = 2 * (int64_t)i + 1 - B;
                c = (double)((u128)hist[i] * (u128)((u + B) * (u + B)));
            }
            *cost_out = c;
        }
        return b == 1 ? 1 : 0;
    }
    const int32_t ke = (b < k) ? (int32_t)b : k;

    int32_t* idx = (int32_t*)malloc(sizeof(int32_t) * (size_t)(b + 1));
    dp_moments M;
    M.b = b; M.B = B;
    M.P0 = (uint64_t*)calloc((size_t)(b + 1), sizeof(uint64_t));
    M.P1 = (int64_t*)calloc((size_t)(b + 1), sizeof(int64_t));
    M.P2 = (uint64_t*)calloc((size_t)(b + 1), sizeof(uint64_t));
    /* D and argmin, (ke+1) x (b+1), row k' */
    double* D = (double*)malloc(sizeof(double) * (size_t)(ke + 1) * (size_t)(b + 1));
    int32_t* A = (int32_t*)calloc((size_t)(ke + 1) * (size_t)(b + 1), sizeof(int32_t));
    if (!idx || !M.P0 || !M.P1 || !M.P2 || !D || !A) {
        free(idx); free(M.P0); free(M.P1); free(M.P2); free(D); free(A);
        return -1;
    }
    int64_t j = 0;
    for (int32_t i = 0; i < B; ++i) {
        if (!hist[i]) continue;
        ++j;
        idx[j] = i;
        int64_t u = 2 * (int64_t)i + 1 - B;
        M.P0[j] = M.P0[j - 1] + hist[i];
        M.P1[j] = M.P1[j - 1] + (int64_t)hist[i] * u;
        M.P2[j] = M.P2[j - 1] + hist[i] * (uint64_t)(u * u);
    }
#define DAT(kk, rr) D[(size_t)(kk) * (size_t)(b + 1) + (size_t)(rr)]
#define AAT(kk, rr) A[(size_t)(kk) * (size_t)(b + 1) + (size_t)(rr)]
    for (size_t q = 0; q < (size_t)(ke + 1) * (size_t)(b + 1); ++q) D[q] = INFINITY;
    DAT(0, 0) = 0.0;
    for (int64_t r = 1; r <= b; ++r) { DAT(1, r) = cost_fixed(&M, 1, r, +1); AAT(1, r) = 1; }
    for (int32_t kk = 2; kk <= ke; ++kk) {
        const int last = (kk == ke);
        const int64_t r_lo = last ? b : kk;
        #pragma omp parallel for schedule(dynamic, 16)
        for (int64_t r = r_lo; r <= b; ++r) {
            double best = INFINITY;
            int64_t bl = 0;
            for (int64_t l = kk; l <= r; ++l) {
                double c = last ? cost_fixed(&M, l, r, -1) : cost_interior(&M, l, r);
                double val = DAT(kk - 1, l - 1) + c;
                if (val < best) { best = val; bl = l; }
            }
            DAT(kk, r) = best;
            AAT(kk, r) = (int32_t)bl;
        }
    }
    /* backtrack */
    int64_t r = b;
    int64_t* start = (int64_t*)malloc(sizeof(int64_t) * (size_t)(ke + 1));
    for (int32_t kk = ke; kk >= 1; --kk) {
        int64_t l = AAT(kk, r);
        start[kk] = l;
        r = l - 1;
    }
    for (int32_t kk = 1; kk <= ke; ++kk) {
        int64_t l = start[kk];
        int64_t rr = (kk == ke) ? b : start[kk + 1] - 1;
        if (cell_start) cell_start[kk - 1] = idx[l];
        if (kk == 1) codebook[0] = -1.0f;
        else if (kk == ke) codebook[kk - 1] = 1.0f;
        else {
            uint64_t s0, s2;
            int64_t s1;
            dp_cell(&M, l, rr, &s0, &s1, &s2);
            double mu = ((double)s1 / (double)s0) / (double)B;
            codebook[kk - 1] = (float)mu;
        }
    }
    if (cost_out) *cost_out = DAT(ke, b);
    if (dtable) memcpy(dtable, D, sizeof(double) * (size_t)(ke + 1) * (size_t)(b + 1));
    if (argl) memcpy(argl, A, sizeof(int32_t) * (size_t)(ke + 1) * (size_t)(b + 1));
#undef DAT
#undef AAT
    free(start); free(idx); free(M.P0); free(M.P1); free(M.P2); free(D); free(A);
    return ke;
}

/* One DP cell evaluated on its own: exposes the three canonical cell costs to
 * the tests (kind 0 interior, 1 first level at -1, 2 last level at +1) for a
 * run of nonempty bins [l..r] (1-based ranks among nonempty bins). */
double oracle_dp_cell_cost(const uint64_t* hist, int32_t B, int64_t l, int64_t r,
                           int32_t kind) {
    int64_t b = 0;
    for (int32_t i = 0; i < B; ++i) b += (hist[i] != 0);
    if (l < 1 || r > b || l > r) return NAN;
    dp_moments M;
    M.b = b; M.B = B;
    M.P0 = (uint64_t*)calloc((size_t)(b + 1), sizeof(uint64_t));
    M.P1 = (int64_t*)calloc((size_t)(b + 1), sizeof(int64_t));
    M.P2 = (uint64_t*)calloc((size_t)(b + 1), sizeof(uint64_t));
    int64_t j = 0;
    for (int32_t i = 0; i < B; ++i) {
        if (!hist[i]) continue;
        ++j;
        int64_t u = 2 * (int64_t)i + 1 - B;
        M.P0[j] = M.P0[j - 1] + hist[i];
        M.P1[j] = M.P1[j - 1] + (int64_t)hist[i] * u;
        M.P2[j] = M.P2[j - 1] + hist[i] * (uint64_t)(u * u);
    }
    double c = kind == 0 ? cost_interior(&M, l, r)
             : kind == 1 ? cost_fixed(&M, l, r, +1)
                         : cost_fixed(&M, l, r, -1);
    free(M.P0); free(M.P1); free(M.P2);
    return c;
}

/* Sampled DP entries: given a previous-level row Dprev[0..b] (as produced by
 * any implementation), recompute D[r][kk] and its argmin for the listed r by
 * the full scan of Algorithm 3.  kind_last selects the +1-centred cost.      */
int oracle_dp_entries(const uint64_t* hist, int32_t B, int32_t kk,
                      int32_t kind_last, const double* Dprev, const int64_t* rs,
                      int64_t nr, double* out_val, int32_t* out_arg) {
    int64_t b = 0;
    for (int32_t i = 0; i < B; ++i) b += (hist[i] != 0);
    dp_moments M;
    M.b = b; M.B = B;
    M.P0 = (uint64_t*)calloc((size_t)(b + 1), sizeof(uint64_t));
    M.P1 = (int64_t*)calloc((size_t)(b + 1), sizeof(int64_t));
    M.P2 = (uint64_t*)calloc((size_t)(b + 1), sizeof(uint64_t));
    int64_t j = 0;
    for (int32_t i = 0; i < B; ++i) {
        if (!hist[i]) continue;
        ++j;
        int64_t u = 2 * (int64_t)i + 1 - B;
        M.P0[j] = M.P0[j - 1] + hist[i];
        M.P1[j] = M.P1[j - 1] + (int64_t)hist[i] * u;
        M.P2[j] = M.P2[j - 1] + hist[i] * (uint64_t)(u * u);
    }
    #pragma omp parallel for schedule(dynamic, 1)
    for (int64_t q = 0; q < nr; ++q) {
        int64_t r = rs[q];
        double best = INFINITY;
        int64_t bl = 0;
        for (int64_t l = kk; l <= r; ++l) {
            double c = kind_last ? cost_fixed(&M, l, r, -1) : cost_interior(&M, l, r);
            double val = Dprev[l - 1] + c;
            if (val < best) { best = val; bl = l; }
        }
        out_val[q] = best;
        out_arg[q] = (int32_t)bl;
    }
    free(M.P0); free(M.P1); free(M.P2);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Automatic Block Partitioning (Algorithm 2; Sec. 5.1 partition score).     */
/*                                                                          */
/* z_j = log(g_j^2 + eps).  For every divisor p of n (ascending):            */
/*   mu_i(p) = mean of z over block i (consecutive run of p),               */
/*   S(p)    = (1/(n/p - 1)) * sum_{i} |mu_{i+1}(p) - mu_i(p)|              */
/* (S(n) is 0/0 = NaN.)  Candidates: 1 < p < n whose S(p) is strictly larger */
/* than both neighbours in the sorted divisor list; the result is the        */
/* candidate with the largest S (smallest p on ties), or 1 if none.         */
/* divisors/scores (nullable, capacity cap) receive the list and S(p).       */
/* Returns the number of divisors, or -1 on bad arguments / small cap.       */
/* ------------------------------------------------------------------------ */
int64_t oracle_divisors(int64_t n, int64_t* out, int64_t cap) {
    if (n < 1) return -1;
    int64_t lo_cnt = 0;
    for (int64_t d = 1; d * d <= n; ++d) lo_cnt += (n % d == 0);
    int64_t* lo = (int64_t*)malloc(sizeof(int64_t) * (size_t)lo_cnt);
    int64_t q = 0;
    for (int64_t d = 1; d * d <= n; ++d) if (n % d == 0) lo[q++] = d;
    int64_t cnt = 0;
    for (q = 0; q < lo_cnt; ++q) { if (out && cnt < cap) out[cnt] = lo[q]; ++cnt; }
    for (q = lo_cnt - 1; q >= 0; --q) {
        if (lo[q] * lo[q] == n) continue;
        if (out && cnt < cap) out[cnt] = n / lo[q];
        ++cnt;
    }
    free(lo);
    return cnt;
}

int64_t oracle_infer_blocks(const uint16_t* grad, int64_t n, double eps,
                            int64_t* period_out, int64_t* divisors,
                            double* scores, int64_t cap) {
    if (n < 1) return -1;
    int64_t nd = oracle_divisors(n, NULL, 0);
    int64_t* P = (int64_t*)malloc(sizeof(int64_t) * (size_t)nd);
    double* S = (double*)malloc(sizeof(double) * (size_t)nd);
    double* z = (double*)malloc(sizeof(double) * (size_t)n);
    oracle_divisors(n, P, nd);
    #pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < n; ++j) {
        double g = bf16_to_double(grad[j]);
        z[j] = log(g * g + eps);
    }
    #pragma omp parallel for schedule(dynamic, 1)
    for (int64_t q = 0; q < nd; ++q) {
        const int64_t p = P[q], nb = n / p;
        double acc = 0.0, prev = 0.0;
        for (int64_t i = 0; i < nb; ++i) {
            double sum = 0.0;
            for (int64_t e = i * p; e < (i + 1) * p; ++e) sum += z[e];
            double mu = sum / (double)p;
            if (i > 0) acc += fabs(mu - prev);
            prev = mu;
        }
        S[q] = nb > 1 ? acc / (double)(nb - 1) : NAN;
    }
    int64_t best_p = 1;
    double best_s = -INFINITY;
    int have = 0;
    for (int64_t q = 1; q + 1 < nd; ++q) {
        /* strict local maximum over the sorted divisor list; NaN never wins */
        if (S[q] > S[q - 1] && S[q] > S[q + 1]) {
            if (!have || S[q] > best_s) { best_s = S[q]; best_p = P[q]; have = 1; }
        }
    }
    *period_out = have ? best_p : 1;
    if (divisors) for (int64_t q = 0; q < nd && q < cap; ++q) divisors[q] = P[q];
    if (scores) for (int64_t q = 0; q < nd && q < cap; ++q) scores[q] = S[q];
    free(P); free(S); free(z);
    return nd;
}
