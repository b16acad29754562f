/*
 * gefen.h -- C ABI of libgefen.so, the GB300 (sm_103a) implementation of the
 * hot path of the Gefen optimizer (arXiv 2606.13894, "Gefen: Optimized
 * Stochastic Optimizer").
 *
 * Conventions shared by every call
 * --------------------------------
 *  - Plain C types only.  Device pointers point to CUDA global memory of the
 *    current device; "host" pointers to ordinary host memory.  bf16 values are
 *    passed as their uint16_t bit patterns.
 *  - The caller owns every buffer.  The library never allocates device memory:
 *    scratch comes from a caller-provided workspace whose size the matching
 *    *_workspace_size() call returns (0 means none is needed; a NULL workspace
 *    is then allowed).  Calls keep no state between invocations, except the
 *    static refit's own array and the refit's test hook (both below).
 *  - All work is enqueued on `stream` (a cudaStream_t; NULL is the legacy
 *    default stream) and returns without waiting, unless a call's description
 *    says it synchronises.
 *  - Arguments are validated on the host before anything is enqueued; a bad
 *    argument returns GEFEN_EINVAL (or GEFEN_ENOMEM for a short workspace) and
 *    leaves every buffer untouched.  A failed launch returns GEFEN_ECUDA.  A
 *    fault that happens later on the device surfaces from the next CUDA call
 *    or from gefen_sync_status().
 *  - Calls on different streams that write the same buffers race; the library
 *    does not order them.
 */
#ifndef GEFEN_H
#define GEFEN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* gefen_stream_t; /* same type as cudaStream_t */

typedef enum {
    GEFEN_OK = 0,
    GEFEN_EINVAL = 1,       /* bad argument (host-side check, nothing enqueued) */
    GEFEN_ECUDA = 2,        /* a CUDA runtime call or kernel launch failed */
    GEFEN_ENOMEM = 3,       /* workspace smaller than the size query requires */
    GEFEN_ETIMEOUT = 4,     /* a bounded device wait gave up (the call's outputs are not valid) */
    GEFEN_EUNSUPPORTED = 5, /* not an sm_103 device, or a size past a stated limit */
    GEFEN_EDEVICE = 6       /* the device-side check of a call's data failed */
} gefen_status_t;

/* One parameter tensor inside the flat arenas of gefen_step().
 * Its elements are params[offset .. offset+numel) (likewise grads and codes);
 * its blocks are the consecutive runs [offset + b*period, offset + (b+1)*period)
 * for b = 0 .. numel/period - 1 (Algorithm 2 reshapes the flattened tensor into
 * (n/p) x p), and block b's state is v[block_offset + b], scale[block_offset + b].
 * Requirements: offset % 16 == 0, numel >= 0, period >= 1, numel % period == 0;
 * element ranges of different tensors do not overlap, nor do block ranges. */
typedef struct {
    int64_t offset;
    int64_t numel;
    int64_t period;
    int64_t block_offset;
} gefen_tensor_t;

/* Hyperparameters of Algorithm 1 (AdamW's: stepsize alpha = lr, weight decay
 * lambda, decay rates beta1, beta2 in [0,1), eps) and the step counter t >= 1
 * used by both bias corrections.  flags: GEFEN_HIST* and the storage formats
 * GEFEN_CODES_4BIT, GEFEN_PARAMS_BF16 (below). */
typedef struct {
    double lr;
    double beta1;
    double beta2;
    double eps;
    double weight_decay;
    int64_t step;
    uint32_t flags;
} gefen_hparams_t;

/* Also histogram x_i = m_i / s'_b of every element of every block with
 * s'_b > 0 into `hist` during the step (the input of a codebook refit). */
#define GEFEN_HIST 1u
/* Only histogram g_i / max_{j in block}|g_j| of every nonzero block and write
 * nothing else: the histogram of Algorithm 3 built from the first gradient. */
#define GEFEN_HIST_GRAD_ONLY 2u
/* Storage formats (the four-bit codes of the Ablation Study, "Getting Down to
 * Four Bits", and the 16-bit parameters of the mixed-precision runs in the
 * Experiments; the arithmetic stays fp32):
 * GEFEN_CODES_4BIT: k <= 16 and two codes per byte -- element i of the arena
 * in byte i/2, the low nibble for even i; every tensor offset a multiple of
 * 32.  GEFEN_PARAMS_BF16: params holds bf16 values (the update is computed in
 * fp32 and rounded to nearest-even).  Either format is available for blocks
 * of 1 element, blocks of p <= 8192 with p % 16 == 0 (p % 32 == 0 with 4-bit
 * codes) and larger blocks with p % 4096 == 0; other tensors, and histograms
 * of more than 4096 cells, return GEFEN_EUNSUPPORTED. */
#define GEFEN_CODES_4BIT 4u
#define GEFEN_PARAMS_BF16 8u

/* Largest histogram supported by every call (bins), and largest codebook. */
#define GEFEN_MAX_BINS 65536
#define GEFEN_MAX_LEVELS 256

/* Text for a status code (static storage). */
const char* gefen_status_string(gefen_status_t s);

/* Waits for `stream`, then reports a pending CUDA error as GEFEN_ECUDA. */
gefen_status_t gefen_sync_status(gefen_stream_t stream);

/* -------------------------------------------------------------------------
 * gefen_step -- one iteration of Algorithm 1's loop body for every tensor.
 *
 * For each block b of each tensor, with codes c_i, scale s_b, shared v_b:
 *   m_i  = beta1 * codebook_dec[c_i] * s_b + (1 - beta1) * g_i
 *   s'_b = max_i |m_i|                                      (Quantize, absmax)
 *   v_b  = beta2 * v_b + (1 - beta2) * mean_i g_i^2         (one v per block)
 *   theta_i -= lr * ( m_i/(1-beta1^t) / (sqrt(v_b/(1-beta2^t)) + eps)
 *                     + weight_decay * theta_i )
 *   c_i  = index of the level of codebook_enc nearest to m_i / s'_b (ties to
 *          the lower index); s_b = s'_b.
 * The update uses the unquantised m_i.  A block with s'_b = 0 stores the level
 * nearest to 0 in every c_i.  Initial state (Algorithm 1, "m_0 <- 0",
 * "v_0 <- 0"): codes at the level nearest 0, scale = 0, v = 0.  After a
 * codebook refit, pass the old codebook as codebook_dec and the new one as
 * codebook_enc for one step.
 *
 * params  f32[*] (bf16 with GEFEN_PARAMS_BF16) device, in/out
 * grads   bf16[*] device, in
 * codes   u8[*] (two per byte with GEFEN_CODES_4BIT) device, in/out
 * v, scale f32[*] device, in/out (per block)
 * codebook_dec, codebook_enc  f32[k] device, sorted ascending, 2 <= k <= 256
 * hist    u64[hist_bins] device, counts are ADDED (caller zeroes); required
 *         when a GEFEN_HIST* flag is set, else ignored (may be NULL).
 *         1 <= hist_bins <= GEFEN_MAX_BINS.  Cell i of B is
 *         [-1 + 2i/B, -1 + 2(i+1)/B), +1 in the last (fp32 arithmetic).
 * params, grads, codes must be 16-byte aligned.  With GEFEN_HIST_GRAD_ONLY
 * only grads, hist and the tensor table are used.
 * workspace: gefen_step_workspace_size() bytes (at least 256), 256-byte
 * aligned; its first 256 bytes must be zero before the first call (they hold
 * the flag gefen_step_status() reads).
 * ------------------------------------------------------------------------- */
size_t gefen_step_workspace_size(const gefen_tensor_t* tensors, int32_t ntensors,
                                 uint32_t flags);
gefen_status_t gefen_step(const gefen_tensor_t* tensors, int32_t ntensors,
                          float* params, const uint16_t* grads, uint8_t* codes,
                          float* v, float* scale, const float* codebook_dec,
                          const float* codebook_enc, int32_t k,
                          gefen_hparams_t hp, uint64_t* hist, int32_t hist_bins,
                          void* workspace, size_t workspace_bytes,
                          gefen_stream_t stream);

/* Synchronises `stream` and reports whether a step that used this workspace
 * gave up a bounded wait for its own shared-memory copies (GEFEN_ETIMEOUT; the
 * step's outputs are then not valid).  Reading the flag clears it.  The same
 * call reads the flag of a gefen_muon_step or gefen_gemm_bf16 workspace. */
gefen_status_t gefen_step_status(void* workspace, gefen_stream_t stream);

/* -------------------------------------------------------------------------
 * gefen_refit_codebook -- Algorithm 3 (Exact DP Quantization Codebook
 * Learning) with Appendix D's interval costs.
 *
 * Input: either n fp32 values x (device; each counted in the cell above, NaN
 * in none) or, when x == NULL, a histogram hist_in u64[bins] (device).
 * The nonempty cells j = 1..b (ascending, centre u_j/bins with the odd integer
 * u_j = 2*i_j + 1 - bins) are split into k contiguous runs minimising the
 * squared error with the first level fixed at -1, the last at +1 and every
 * other level at its run's count-weighted mean; every level gets >= 1
 * nonempty cell.  Costs use exact integer moments:
 *   interior run:  (double)(s0*s2 - s1^2) / (double)s0
 *   first level:   (double)(s2 + 2B*s1 + B^2*s0),  last: (double)(s2 - 2B*s1 + B^2*s0)
 * (round-to-nearest double, units of 1/B^2), D[r][k'] = min over the run
 * start l of D[l-1][k'-1] + cost, ties to the smallest l.  The result equals
 * the full O(b^2 k) scan bit for bit.  With b < k nonempty cells the DP runs
 * with b levels and the codebook is padded with +1 (b <= 1: [-1,+1,+1,...]).
 *
 * codebook_out   f32[k] device: C[0] = -1, C[k_eff-1] = +1, interior levels
 *                = (s1/s0)/bins rounded to fp32.
 * hist_out       u64[bins] device, nullable: the histogram used.
 * cell_start_out i32[k] device, nullable: first cell index of each level (-1
 *                for padding).
 * cost_out       f64[1] device, nullable: the optimum D[b][k_eff].
 * Requirements: 1 <= bins <= GEFEN_MAX_BINS, 2 <= k <= GEFEN_MAX_LEVELS,
 * n >= 0, x 16-byte aligned, total count N < 2^62 with N*(bins-1)^2 < 2^64
 * (checked on the device: on failure the outputs are left untouched and
 * gefen_refit_status() reports GEFEN_EDEVICE).  The DP's levels are separated
 * by grid-wide barriers whose waits are bounded (about a second); if one gives
 * up, the outputs are left untouched and gefen_refit_status() reports
 * GEFEN_ETIMEOUT.  workspace: gefen_refit_workspace_size() bytes.
 * ------------------------------------------------------------------------- */
size_t gefen_refit_workspace_size(int32_t bins, int32_t k);
gefen_status_t gefen_refit_codebook(const float* x, int64_t n, const uint64_t* hist_in,
                                    int32_t bins, int32_t k, float* codebook_out,
                                    uint64_t* hist_out, int32_t* cell_start_out,
                                    double* cost_out, void* workspace,
                                    size_t workspace_bytes, gefen_stream_t stream);

/* Device-side status of the last gefen_refit_codebook() that used this
 * workspace; synchronises `stream`.  k_eff_out (host, nullable) receives the
 * number of levels the DP used.  GEFEN_EDEVICE: the moment bound above was
 * exceeded; GEFEN_ETIMEOUT: a bounded wait between DP levels gave up.  Either
 * way the codebook, cell starts and cost were left untouched. */
gefen_status_t gefen_refit_status(const void* workspace, int32_t* k_eff_out,
                                  gefen_stream_t stream);

/* The full DP tables of the last refit in this workspace, for inspection:
 * D (f64) and the minimising run start l (i32, 1-based; 0 where undefined),
 * both (k+1) x (bins+1) row-major by level; entries the recurrence does not
 * define are +inf / 0.  Copies device to device on `stream`. */
gefen_status_t gefen_refit_tables(const void* workspace, int32_t bins, int32_t k,
                                  double* dtable_out, int32_t* argl_out,
                                  gefen_stream_t stream);

/* Test hook of gefen_refit_codebook (the paper has no counterpart): a
 * process-wide setting read by every later refit launch.
 * anchor_stride: -1 chooses automatically (the default), 0 searches every end
 * position over its whole range, s >= 1 puts an anchor every s positions
 * (results are identical in every case).  barrier_extra: 0 normally; any other
 * value makes every level barrier wait for arrivals that never come, so the
 * refit gives up after barrier_spin_cycles (0: the default of about 2^31
 * cycles) and gefen_refit_status() reports GEFEN_ETIMEOUT.  Call it again
 * with (-1, 0, 0) to restore the defaults.  Not for concurrent use with
 * refits on other threads. */
gefen_status_t gefen_refit_debug(int32_t anchor_stride, uint32_t barrier_extra,
                                 int64_t barrier_spin_cycles);

/* -------------------------------------------------------------------------
 * gefen_refit_codebook_static -- gefen_refit_codebook without a workspace.
 * The paper has no counterpart: this entry point exists for callers that
 * cannot allocate device memory when they refit -- a host program whose
 * memory is reserved up front by a framework's caching allocator or a serving
 * runtime (so no workspace can be carved out), or a caller that must not
 * synchronise the device, which cudaFree (and at times cudaMalloc) do.
 *
 * Same inputs, outputs and results as gefen_refit_codebook(); the scratch is
 * one device array inside the library, sized for bins <= 4096 and k <= 256
 * (about 21.5 MB).  Larger requests return GEFEN_EUNSUPPORTED.  The call
 * allocates nothing: no cudaMalloc, cudaFree or allocating library call.
 *
 * The array exists on a device once the library's refit module is loaded
 * there, which CUDA's lazy loading delays to the first use, and it stays
 * until the process exits.  So call gefen_refit_static_init() once per device
 * (with that device current) before a caching allocator or runtime reserves
 * the device's memory, and before any stream capture: it loads the module,
 * looks up the array's device address and loads the refit's kernels.
 * Otherwise the first gefen_refit_codebook_static() on a device does the same.
 * All calls share the one array and it keeps the last call's contents (the
 * refit clears what it needs); calls whose work overlaps on the GPU --
 * different streams, or different host threads -- race on it and must be
 * ordered by the caller.
 * gefen_refit_static_status() reads the device-side status of the last static
 * refit (synchronises `stream`): GEFEN_EDEVICE if the moment bound was
 * exceeded, GEFEN_ETIMEOUT if a bounded wait gave up; in both cases the
 * outputs were left untouched.
 * ------------------------------------------------------------------------- */
gefen_status_t gefen_refit_static_init(void);
gefen_status_t gefen_refit_codebook_static(const float* x, int64_t n, const uint64_t* hist_in,
                                           int32_t bins, int32_t k, float* codebook_out,
                                           uint64_t* hist_out, int32_t* cell_start_out,
                                           double* cost_out, gefen_stream_t stream);
gefen_status_t gefen_refit_static_status(int32_t* k_eff_out, gefen_stream_t stream);

/* -------------------------------------------------------------------------
 * gefen_infer_blocks -- Algorithm 2 (Automatic Block Partitioning) for one
 * flattened gradient tensor g (bf16 bits, device, numel elements).
 *
 * z_j = log(g_j^2 + eps).  For every divisor p of n (ascending):
 *   mu_i(p) = mean of z over the i-th run of p elements,
 *   S(p)    = mean over i of |mu_{i+1}(p) - mu_i(p)|      (S(n) undefined)
 * (the partition-score equation of Sec. 5.1).  The period is the divisor
 * 1 < p < n whose score is a strict local maximum over the sorted divisor list
 * and is the largest such (smallest p on ties); 1 if there is none.
 * Synchronises `stream` and writes period_out (host).  scores_out (host,
 * nullable, scores_cap entries) receives S(p) for the divisors in ascending
 * order; ndiv_out (host, nullable) the divisor count.  1 <= numel <= 2^32,
 * eps > 0, grad 16-byte aligned.  A non-finite gradient returns GEFEN_EDEVICE.
 * workspace: gefen_infer_workspace_size(numel) bytes.
 * ------------------------------------------------------------------------- */
size_t gefen_infer_workspace_size(int64_t numel);
gefen_status_t gefen_infer_blocks(const uint16_t* grad, int64_t numel, double eps,
                                  int64_t* period_out, double* scores_out,
                                  int64_t scores_cap, int64_t* ndiv_out,
                                  void* workspace, size_t workspace_bytes,
                                  gefen_stream_t stream);

/* -------------------------------------------------------------------------
 * gefen_muon_step -- Gefen-Muon (the paper's appendix "Gefen-Muon"): Muon's
 * momentum buffer kept as Gefen codes with a per-block absmax scale
 * (Algorithm 1, Quantize), Muon's orthogonalisation unchanged.  For one
 * rows x cols matrix (row-major), blocks of `period` consecutive elements:
 *   m    = momentum * codebook_dec[c_i] * s_b + (1 - momentum) * g_i
 *   s'_b = max |m_i|; c_i = level of codebook_enc nearest m_i / s'_b (ties to
 *          the lower index; level nearest 0 for s'_b = 0); s_b = s'_b
 *   U    = g + momentum * (m - g) with nesterov, else m
 *   X    = U / max(||U||_F, eps), then ns_steps times on the smaller side:
 *          X <- ns_a X + (ns_b A + ns_c A A) X with A = X X^T
 *   theta <- theta (1 - lr weight_decay) - lr sqrt(max(1, rows/cols)) X
 * (Muon as in PyTorch's torch.optim.Muon: momentum 0.95, Nesterov, 5 steps of
 * (3.4445, -4.7750, 2.0315), eps 1e-7 are its defaults).  The matrix
 * products are this library's: with GEFEN_MUON_BF16_GEMM bf16 storage and
 * fp32 accumulation on the tensor cores (gefen_gemm_bf16, as Muon runs them),
 * else fp32 throughout on the CUDA cores.  Word 0 of the workspace is set if
 * a bounded wait of the products gave up (gefen_step_status reads and clears
 * it; the outputs are then not valid).
 *
 * params f32[rows*cols], grads bf16[rows*cols] (16-byte aligned), codes
 * u8[rows*cols], scale f32[rows*cols/period] (device, in/out); codebooks
 * f32[k] (2 <= k <= 256).  workspace: gefen_muon_workspace_size() bytes,
 * 256-byte aligned.  rows, cols < 2^31; period divides rows*cols.
 * ------------------------------------------------------------------------- */
#define GEFEN_MUON_BF16_GEMM 1u

typedef struct {
    double lr;
    double momentum;
    double weight_decay;
    double eps;
    int32_t nesterov;
    int32_t ns_steps;
    double ns_a, ns_b, ns_c;
    uint32_t flags;
} gefen_muon_hparams_t;

size_t gefen_muon_workspace_size(int64_t rows, int64_t cols, int64_t period, uint32_t flags);

/* The product Gefen-Muon's Newton-Schulz iteration runs on (the paper has no
 * counterpart; exposed for tests and for callers who want it):
 *   C = alpha * A * B^T + beta * D
 * A: M x K, B: N x K, C and D: M x N, all row-major bf16 (bit patterns) with
 * leading dimensions lda >= K, ldb >= K, ldd >= N, ldc >= N; CT (nullable)
 * receives C transposed (N x M, ldct >= M); C may be NULL when CT is given; D
 * is read only when beta != 0.  fp32 accumulation; each output rounded once
 * to bf16.  When every matrix it touches (A, B, C, CT, and D if read) is
 * 16-byte aligned with a leading dimension that is a multiple of 8, the
 * product runs on the tensor cores (tcgen05; operands staged and results
 * written by TMA), else on the CUDA cores.  workspace: >= 256 bytes, 256-byte aligned; its word 0 is
 * set if a bounded wait gave up (read it with gefen_step_status). */
gefen_status_t gefen_gemm_bf16(int32_t M, int32_t N, int32_t K, float alpha, const uint16_t* A,
                               int32_t lda, const uint16_t* B, int32_t ldb, float beta,
                               const uint16_t* D, int32_t ldd, uint16_t* C, int32_t ldc,
                               uint16_t* CT, int32_t ldct, void* workspace, size_t workspace_bytes,
                               gefen_stream_t stream);
/* The symmetric product of the same iteration (X X^T and its powers):
 *   C = alpha * A * A^T + beta * D
 * A: N x K, C and D: N x N, row-major bf16, lda >= K, ldc >= N, ldd >= N; D
 * is read only when beta != 0 and must then be symmetric.  C is symmetric bit
 * for bit: on the tensor cores (conditions as for gefen_gemm_bf16) only the
 * tiles on or above the diagonal are computed and each is also written
 * mirrored; on the CUDA cores C[i][j] and C[j][i] sum the same products in the
 * same order.  C must not overlap A or D.  workspace as for gefen_gemm_bf16. */
gefen_status_t gefen_gemm_bf16_sym(int32_t N, int32_t K, float alpha, const uint16_t* A, int32_t lda,
                                   float beta, const uint16_t* D, int32_t ldd, uint16_t* C, int32_t ldc,
                                   void* workspace, size_t workspace_bytes, gefen_stream_t stream);
gefen_status_t gefen_muon_step(int64_t rows, int64_t cols, int64_t period, float* params,
                               const uint16_t* grads, uint8_t* codes, float* scale,
                               const float* codebook_dec, const float* codebook_enc, int32_t k,
                               gefen_muon_hparams_t hp, void* workspace, size_t workspace_bytes,
                               gefen_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* GEFEN_H */
