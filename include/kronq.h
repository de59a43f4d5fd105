/*
 * libkronq -- the per-layer quantization path of KronQ ("KronQ: LLM Quantization via
 * Kronecker-Factored Hessian") as a C ABI over hand-written CUDA kernels for sm_103a.
 *
 * One linear layer W [d_out x d_in] is processed in four stages:
 *   1. Kronecker factors  H_X = X^T X, H_G = G^T G            (kq_accum_factor, kq_traces)
 *   2. bidirectional incoherence processing (BiIP)            (kq_compute_scales,
 *                                                              kq_rotate_in, kq_rotate_out)
 *   3. damped inverse Cholesky                                (kq_chol_inv)
 *   4. column-wise OBS sweep with b-bit asymmetric grids      (kq_obs_quantize)
 * with the GPTAQ drift correction as an option (kq_accum_drift, kq_gptaq_p, and the Pt
 * argument of kq_obs_quantize), inference with the quantized layer (kq_pack_codes,
 * kq_infer), plus two check-only calls (kq_dequant_revert, kq_proxy_loss).
 *
 * Conventions shared by every call
 *   - Tokens are rows: X is [T x d_in], G is [T x d_out]; the paper stacks tokens as
 *     columns, so its X X^T is X^T X here.
 *   - All pointers are DEVICE pointers owned by the caller unless stated otherwise. The
 *     library allocates no memory; scratch space is passed in as `ws` with a size from
 *     the matching *_workspace() query.
 *   - Matrices are dense row-major. Only kq_accum_factor takes a leading dimension (for
 *     its input); every other matrix is contiguous (leading dimension = row length).
 *   - Every call is asynchronous on `stream` (NULL = the legacy default stream) and
 *     returns a kq_status for errors detected on the host (bad arguments, launch
 *     failures). Errors detected by kernels are written to the optional device word
 *     `info` (first error wins) and read back with kq_check().
 *   - bf16 inputs are passed as their 16-bit patterns (uint16_t).
 *   - Supported rotation sizes are n = 2^k (0 <= k <= 15) and n = 28 * 2^k (2^k <= 1024).
 */
#ifndef KRONQ_H
#define KRONQ_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define KQ_API __attribute__((visibility("default")))
#else
#define KQ_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t. */
typedef struct CUstream_st* kq_stream_t;

typedef enum kq_status {
    KQ_OK = 0,
    KQ_ERR_INVALID_ARG = 1,  /* null pointer, negative size, size mismatch, bad alignment */
    KQ_ERR_UNSUPPORTED = 2,  /* dimension without a Hadamard construction, group not in {0, block} */
    KQ_ERR_NOT_PD = 3,       /* non-positive pivot in kq_chol_inv (reported through `info`) */
    KQ_ERR_CUDA = 4,         /* a CUDA runtime/driver call failed */
    KQ_ERR_TIMEOUT = 5,      /* a kernel gave up a bounded wait (reported through `info`) */
    KQ_ERR_WORKSPACE = 6,    /* ws is NULL or smaller than the *_workspace() size */
    KQ_ERR_NONFINITE = 7     /* a NaN or infinity reached the quantizer (kq_obs_quantize, `info`) */
} kq_status;

/* Text of the last host-side error of the calling thread ("" when none). */
KQ_API const char* kq_last_error(void);
/* Name of a status code. */
KQ_API const char* kq_status_name(int status);
/* Library version: major * 10000 + minor * 100 + patch. */
KQ_API int kq_version(void);
/* Number of kernels this library has launched in this process (all threads, all devices). */
KQ_API uint64_t kq_launch_count(void);

/*
 * Graph helpers (runtime plumbing, no counterpart in the paper). kq_graph_instantiate: an
 *   executable graph from a captured graph (cudaGraph_t passed as a pointer), with
 *   use_node_priority != 0 honouring the priority each kernel node was captured with (the
 *   capturing stream's): without it every node takes the priority of the stream the graph
 *   is launched into, and a two-stream schedule loses its ordering between the critical
 *   path and the side work. *exec receives the cudaGraphExec_t; the caller keeps the graph
 *   alive while exec is used and destroys exec with kq_graph_exec_destroy.
 *   kq_graph_launch: one launch of exec on the stream. CUDA errors give KQ_ERR_CUDA.
 */
KQ_API kq_status kq_graph_instantiate(void* graph, int use_node_priority, void** exec);
KQ_API kq_status kq_graph_launch(void* exec, kq_stream_t stream);
KQ_API kq_status kq_graph_exec_destroy(void* exec);

/*
 * Synchronize `stream`, then read the device error word `info` (may be NULL) and map it:
 * 0 -> KQ_OK, > 0 -> KQ_ERR_NOT_PD (the value is the 1-based index of the first
 * non-positive pivot), < 0 -> the status -info. Resets *info to 0 when `reset` != 0.
 * `pivot_out` (host, may be NULL) receives the raw word.
 */
KQ_API kq_status kq_check(int* info, int reset, int* pivot_out, kq_stream_t stream);

/*
 * kq_selftest_timeout: a diagnostic with no counterpart in the paper. Launches one kernel
 *   that waits on an mbarrier nothing arrives on, using the same bounded wait as every
 *   pipeline kernel (TMA/tcgen05 producers, consumers and epilogues), which gives up after
 *   limit_us microseconds (1 .. 2e6) and records -KQ_ERR_TIMEOUT in *info (device int). Read
 *   it with kq_check. It shows, without faulting or hanging the GPU, that a stalled pipeline
 *   returns an error status and leaves the context usable.
 */
KQ_API kq_status kq_selftest_timeout(int* info, int64_t limit_us, kq_stream_t stream);

/*
 * Debug build (no counterpart in the paper). libkronq_debug.so is the same library compiled
 * with -DKQ_DEBUG: before their global-memory stores the kernels check each index against
 * the size of the buffer it belongs to, and a failed check skips the store and records the
 * source line (first failure per source file) instead of faulting. A stand-in for a memory
 * checker on machines where none may run.
 * kq_debug_build: 1 for the debug build, 0 otherwise.
 * kq_debug_status: synchronizes the device, then *unit = the first source file (0 api,
 *   1 syrk, 2 biip, 3 chol, 4 obs, 5 trail_tc, 6 gptaq, 7 infer, 8 check) whose checks
 *   failed and *line = its first failing line, or *unit = -1 and *line = 0 when none did
 *   (always so in the normal build); reset clears the recorded lines.
 * kq_selftest_bounds: writes buf[i] = i for i = 0 .. n under a check against n; buf must
 *   hold n + 1 floats, so every write stays inside it in either build. The debug build skips
 *   index n and records it (the check itself is what this exercises).
 */
KQ_API int kq_debug_build(void);
KQ_API kq_status kq_debug_status(int* unit, int* line, int reset);
KQ_API kq_status kq_selftest_bounds(float* buf, int64_t n, kq_stream_t stream);

/*
 * kq_selftest_div: a diagnostic with no counterpart in the paper. The OBS sweep (Sec. 2.1
 *   Eq. (obs_update)) divides by the grid scale and by [H^-1]_pp on its sequential chain; it
 *   does so with a reciprocal and two Markstein corrections, which must equal IEEE
 *   round-to-nearest division bit for bit. For n pairs a[i], b[i] (device fp32) this adds to
 *   *mismatches (device uint64) the number of i where that division differs from the
 *   correctly rounded a[i] / b[i] in any bit. n = 0 is a no-op; NULL pointers or n < 0 give
 *   KQ_ERR_INVALID_ARG.
 */
KQ_API kq_status kq_selftest_div(const float* a, const float* b, int64_t n, unsigned long long* mismatches,
                                 kq_stream_t stream);

/* ------------------------------------------------------------------------------------
 * Stage 1: Kronecker factors.
 * Paper: Sec. 2.1 Eq. (ptq_obj) defines H_X = X X^T; Sec. 3.1 Eq. (kfac) the factor pair
 * H_X (x) H_G; Algorithm 1 computes H_X as an online statistic and loads a precomputed H_G.
 *
 * kq_accum_factor: H (+)= A^T A for A [T x d] bf16 (row t = token t, row stride `lda`
 *   elements). The sum is raw (no 1/T). H is [d x d] fp32, full symmetric storage (both
 *   triangles written). accumulate = 0 overwrites H, 1 adds to it (for token chunks
 *   streamed through several calls). If `trace` (device double*) is non-NULL it receives
 *   tr(H) of the resulting H, summed in fp64.
 *   Products of bf16 values are exact in fp32; sums are fp32 with the tensor-core
 *   accumulator drained into an fp32 running sum every `KQ_SYRK_CHUNK_TOKENS` tokens.
 *   Requirements: A 16-byte aligned, lda % 8 == 0, lda >= d, T >= 0, 1 <= d <= 65536.
 *   T == 0 gives H = 0 (accumulate = 0) or leaves H unchanged. `info` (nullable) receives
 *   -KQ_ERR_TIMEOUT if a pipeline wait gave up.
 * ---------------------------------------------------------------------------------- */
#define KQ_SYRK_CHUNK_TOKENS 512
KQ_API kq_status kq_accum_factor(const uint16_t* A, int64_t T, int64_t d, int64_t lda, float* H,
                          int accumulate, double* trace, int* info, kq_stream_t stream);

/* ------------------------------------------------------------------------------------
 * GPTAQ drift statistic (optional; the full objective of Sec. 3.1 Eq. kronq_full).
 * Paper: Sec. 2.1 Eq. (gptaq_obj) (Delta X = X~ - X, X~ the full-precision model's input to
 * the layer, X the running quantized model's); Algorithm 1 computes Delta X X^T online.
 *
 * kq_accum_drift: D (+)= (X~ - X)^T X for X~, X [T x d] bf16 (row t = token t, common row
 *   stride `ld` elements); D [d x d] fp32 row-major, D[a][b] = sum_t (x~_t[a] - x_t[a]) x_t[b]
 *   (not symmetric). The drift is split exactly into a bf16 pair hi + lo (x~ - x is exact
 *   in fp32; the pair holds it to 16 significant bits, exactly unless the two exponents are
 *   more than 8 apart), and D = hi^T X + lo^T X runs on the tensor cores (bf16 products,
 *   exact in fp32; fp32 sums drained every KQ_SYRK_CHUNK_TOKENS tokens).
 *   accumulate = 0 overwrites D, 1 adds to it. Requirements: X~, X 16-byte aligned,
 *   d % 8 == 0, ld % 8 == 0, ld >= d, 1 <= d <= 65536, 0 <= T < 2^31. T == 0 gives D = 0
 *   (accumulate = 0) or leaves D unchanged.
 *   ws (256-byte aligned) holds the split drift of a chunk of tokens: with
 *   kq_accum_drift_workspace(T, d) bytes all T tokens go through one pass; a smaller ws
 *   (at least 4 * d * 64 bytes) processes the tokens in chunks of what it holds.
 *   info (nullable): -KQ_ERR_TIMEOUT if a pipeline wait gave up.
 * The drift statistic is rescaled and rotated like H_X (Algorithm 1): pass D as the
 * H_X argument of kq_rotate_in (W = NULL, dir = KQ_FWD) to get D' = V S_X^-1 D S_X^-1 V^T.
 * ---------------------------------------------------------------------------------- */
KQ_API size_t kq_accum_drift_workspace(int64_t T, int64_t d);
KQ_API kq_status kq_accum_drift(const uint16_t* Xt, const uint16_t* X, int64_t T, int64_t d, int64_t ld,
                                float* D, int accumulate, int* info, void* ws, size_t ws_bytes,
                                kq_stream_t stream);

/* ------------------------------------------------------------------------------------
 * Stage 2: bidirectional incoherence processing.
 * Paper: Sec. 3.2 Eq. (rescale) gives S_X = diag(H_X_jj / ||W_:,j||^2)^(1/4) and
 * S_G = diag(H_G_ii / ||W_i,:||^2)^(1/4); Eq. (biip) the rotations W <- U W V^T,
 * H_X <- V H_X V^T, H_G <- U H_G U^T with randomized Hadamard transforms; Algorithm 1
 * applies the rescale first, then the rotations, then releases H_G.
 *
 * The randomized Hadamard transform of size n is V = H_n diag(sigma) / sqrt(n) with
 * sigma in {-1, +1}^n (int8, caller-drawn) and H_n the Sylvester matrix for n = 2^k, or
 * H_28 (x) H_{2^k} for n = 28 * 2^k, where H_28 is Paley's second construction over
 * GF(13) and index j = a * 2^k + b (b fastest). H_n is symmetric, so V^-1 = V^T.
 *
 * kq_compute_scales: s_x [d_in] and s_g [d_out] (fp32) from the ORIGINAL W [d_out x d_in]
 *   fp32 and the diagonals of the raw H_X [d_in x d_in] and H_G [d_out x d_out]. Norms are
 *   summed in fp64; s = sqrt(sqrt(h / a)), and s = 1 when h == 0 or a == 0 (a dead
 *   channel). Must run before either rotation. Each side is computed only if its output
 *   is non-NULL (s_x needs H_X); with H_G NULL, s_g = 1 (the one-sided variant). So the
 *   two sides can run on two streams as soon as their own factor exists.
 *
 * kq_traces: the sensitivity statistics of Sec. 3.3 Eq. (sensitivity), from the raw
 *   factors' diagonals and the scales (call before the rotations overwrite H_X / H_G).
 *   out [6] (device double): tr(H_X), tr(H_G), tr(H_X) tr(H_G), and the post-BiIP
 *   tr(H_X'), tr(H_G'), tr(H_X') tr(H_G') with tr(H') = sum_j H_jj / s_j^2 (the rotations
 *   preserve the trace). A NULL factor leaves its side of out untouched and the products
 *   use the values already in out, so the sides may come from two calls (X side first).
 *
 * kq_rotate_in (input side, length d_in, sign_v = sigma_V):
 *   dir = KQ_FWD: W <- (W S_X) V^T, and if H_X != NULL: H_X <- V S_X^-1 H_X S_X^-1 V^T
 *   (H_X any square matrix, e.g. the drift statistic D). dir = KQ_FWD_SYM: the same for a
 *   symmetric H_X, which lets the two-sided transform skip its last transposition: the
 *   result is the transpose of KQ_FWD's up to rounding (both equal the exact V M V^T to
 *   fp32 rounding). The same holds for kq_rotate_out's H_G.
 *   dir = KQ_INV: W <- (W V) S_X^-1 (undoes the forward map; H_X untouched).
 * kq_rotate_out (output side, length d_out, sign_u = sigma_U):
 *   dir = KQ_FWD: W <- U (S_G W), and if H_G != NULL: H_G <- U S_G^-1 H_G S_G^-1 U^T.
 *   dir = KQ_INV: W <- S_G^-1 (U^T W).
 *   All in place, fp32. s_x / s_g may be NULL for a pure rotation (S = I). In the FWD
 *   direction W may be NULL to transform only the factor (H_X or H_G).
 *   Returns KQ_ERR_UNSUPPORTED if the length has no Hadamard construction.
 * ---------------------------------------------------------------------------------- */
KQ_API kq_status kq_compute_scales_exp(const float* W, int64_t d_out, int64_t d_in, const float* H_X,
                                       const float* H_G, float* s_x, float* s_g, float ex, float eg,
                                       kq_stream_t stream);

/* BiIP statistics (Prop. 2 and Sec. 3.2; no counterpart in the quantization path itself):
 * kq_compute_scales_exp: the scales of kq_compute_scales with the exponent as a parameter,
 *   s_x = (h_x / a)^ex, s_g = (h_g / r)^eg, ex, eg in [0, 1] (1/4 gives kq_compute_scales'
 *   bits exactly; 0 gives no rescale). Prop. 2's exponent sweep varies eg.
 * kq_biip_stats: out [4] (device double) = [CV_in, CV_out, rho_in, rho_out]: the coefficient
 *   of variation (population standard deviation over mean) of the column norms and of the
 *   row norms of W [d_out x d_in], and rho = (sum sqrt(h a))^2 / (sum h sum a) <= 1 (Prop. 2's
 *   gain of the rescale over none) from the diagonal h of H_X (input side, a = squared
 *   column norms) or H_G (output side, a = squared row norms); a NULL factor leaves its rho
 *   entry untouched. fp64 sums. ws: kq_biip_stats_workspace(d_out, d_in) bytes. */
KQ_API size_t kq_biip_stats_workspace(int64_t d_out, int64_t d_in);
KQ_API kq_status kq_biip_stats(const float* W, int64_t d_out, int64_t d_in, const float* H_X, const float* H_G,
                               double* out, void* ws, size_t ws_bytes, kq_stream_t stream);

#define KQ_FWD 0
#define KQ_INV 1
#define KQ_FWD_SYM 2   /* KQ_FWD for a symmetric H_X / H_G (see kq_rotate_in) */
KQ_API kq_status kq_compute_scales(const float* W, int64_t d_out, int64_t d_in, const float* H_X,
                            const float* H_G, float* s_x, float* s_g, kq_stream_t stream);
KQ_API kq_status kq_traces(const float* H_X, const float* s_x, int64_t d_in, const float* H_G,
                    const float* s_g, int64_t d_out, double* out, kq_stream_t stream);
/*
 * kq_factor_diag: diag(A^T A) alone (the per-channel sums of squares; for G these are the
 *   only entries of H_G that the quantization reads, through S_G and the traces -- Prop. 1).
 *   diag [d] fp32 from fp64 sums in a fixed order (deterministic), trace (device double,
 *   nullable) = their fp64 total. Reads A once. ws: kq_factor_diag_workspace(T, d) bytes.
 * kq_compute_scales_diag / kq_traces_diag: kq_compute_scales / kq_traces with the factors'
 *   diagonals given as vectors (stride 1) instead of the full matrices.
 */
KQ_API size_t kq_factor_diag_workspace(int64_t T, int64_t d);
KQ_API kq_status kq_factor_diag(const uint16_t* A, int64_t T, int64_t d, int64_t lda, float* diag, double* trace,
                                void* ws, size_t ws_bytes, kq_stream_t stream);
KQ_API kq_status kq_compute_scales_diag(const float* W, int64_t d_out, int64_t d_in, const float* hx_diag,
                                        const float* hg_diag, float* s_x, float* s_g, kq_stream_t stream);
KQ_API kq_status kq_traces_diag(const float* hx_diag, const float* s_x, int64_t d_in, const float* hg_diag,
                                const float* s_g, int64_t d_out, double* out, kq_stream_t stream);
KQ_API kq_status kq_rotate_in(float* W, int64_t d_out, int64_t d_in, float* H_X, const float* s_x,
                       const int8_t* sign_v, int dir, kq_stream_t stream);
KQ_API kq_status kq_rotate_out(float* W, int64_t d_out, int64_t d_in, float* H_G, const float* s_g,
                        const int8_t* sign_u, int dir, kq_stream_t stream);

/* ------------------------------------------------------------------------------------
 * Stage 3: damped inverse Cholesky.
 * Paper: Algorithm 2 damps H_X <- H_X + lambda * mean(diag(H_X)) I and takes
 * L = Inverse_Cholesky(H_X); Proposition 1 defines L by H_X^-1 = L L^T (L lower).
 *
 * kq_chol_inv: H [n x n] fp32 symmetric (read only; the lower triangle is used) ->
 *   Lt [n x n] fp32, the lower-triangular L with (H + damp_rel * mean(diag H) I)^-1 = L L^T
 *   and positive diagonal; the strict upper triangle of Lt is written with zeros. R = L^T
 *   is the upper factor whose row j drives the OBS update of column j. Computed as the
 *   Cholesky factorization of the index-reversed matrix with its triangular inverse formed in
 *   the same sweep (2 n^3 / 3 flops): fp32 on the diagonal blocks, the products on the tensor
 *   cores with the 3xTF32 split (fp32-accurate products, fp32 sums). When n > 1024 the
 *   128-column steps of each 1024-column super-panel stay inside its diagonal block, its
 *   panel below and its rows of the inverse to the left come from two products with that
 *   block's inverse, and the tiles beyond take one K = 1024 update per super-panel.
 *   On a non-positive pivot, *info (required for that report) receives the 1-based index
 *   (in H's own indexing) of the failing pivot; Lt is then undefined. The caller may retry
 *   with a larger damp_rel.
 *   ws: kq_chol_inv_workspace(n) bytes.
 * ---------------------------------------------------------------------------------- */
KQ_API size_t kq_chol_inv_workspace(int64_t n);
KQ_API kq_status kq_chol_inv(const float* H, int64_t n, float damp_rel, float* Lt, int* info, void* ws,
                      size_t ws_bytes, kq_stream_t stream);

/*
 * kq_chol_inv_noalloc: the same computation and results as kq_chol_inv, for callers that
 *   cannot hand the library a workspace because they may not allocate device memory when
 *   they call it -- for example a plugin running inside another runtime that owns every
 *   device allocation, or a latency-bound loop where a cudaMalloc would synchronize the
 *   device. The paper has no counterpart; this is a convenience of this library.
 *   Scratch comes from a fixed array in device memory that the library owns:
 *   KQ_CHOL_NOALLOC_SCRATCH_BYTES = 2 N^2 * 4 + 256 bytes with N = KQ_CHOL_NOALLOC_MAX_N
 *   (the padded matrix and its inverse factor): 8 MiB + 256 bytes, held by every device that loads
 *   the library until the process exits. n > KQ_CHOL_NOALLOC_MAX_N is rejected with
 *   KQ_ERR_WORKSPACE and a message; no allocation is ever made.
 *   The first call on each device looks up the array's device address (cudaGetSymbolAddress,
 *   with that device current); make that first call before any stream capture.
 *   All calls share the one array and it keeps the previous call's contents (every byte a
 *   call reads is written by that call first), so calls whose work overlaps on the GPU --
 *   on different streams, or from different host threads -- race: serialize them.
 */
#define KQ_CHOL_NOALLOC_MAX_N 1024
#define KQ_CHOL_NOALLOC_SCRATCH_BYTES ((2ull * 1024 * 1024) * 4 + 256)
KQ_API kq_status kq_chol_inv_noalloc(const float* H, int64_t n, float damp_rel, float* Lt, int* info,
                                     kq_stream_t stream);

/* ------------------------------------------------------------------------------------
 * GPTAQ correction matrix (optional).
 * Paper: Proposition 1 and Algorithm 2: P = alpha ((D' L) o M_U) L^T with D' the rescaled,
 * rotated drift statistic, H^-1 = L L^T (L from kq_chol_inv of the damped H_X') and M_U
 * the strictly upper-triangular mask. Row p of P (alpha = 1) holds the least-squares
 * coefficients of column p's drift on the later columns.
 *
 * kq_gptaq_p: Pt [n x n] fp32 row-major receives P^T (strictly lower triangular; the upper
 *   triangle and the diagonal are written as 0). Dp = D' [n x n], Lt = L [n x n] row-major
 *   (lower; its strict upper triangle must be 0, as kq_chol_inv leaves it). Both triangular
 *   products run on the tensor cores with the 3xTF32 split (fp32-accurate products, fp32
 *   sums). Requirements: n % 4 == 0, 1 <= n <= 65536, Dp and Lt 16-byte aligned.
 *   ws: kq_gptaq_p_workspace(n) bytes (6 n^2 floats), 256-byte aligned.
 *   info (nullable): -KQ_ERR_TIMEOUT if a pipeline wait gave up.
 * ---------------------------------------------------------------------------------- */
KQ_API size_t kq_gptaq_p_workspace(int64_t n);
KQ_API kq_status kq_gptaq_p(const float* Dp, const float* Lt, int64_t n, float alpha, float* Pt, int* info,
                            void* ws, size_t ws_bytes, kq_stream_t stream);

/* ------------------------------------------------------------------------------------
 * Stage 4: column-wise OBS sweep, GPTQ mode (Pt = NULL) or with the GPTAQ correction P.
 * Paper: Sec. 2.1 Eq. (obs_update); Algorithm 2's inner column loop and lazy trailing
 * update; Proposition 1 (H_G cancels, so the sweep reads only L, and P with the drift).
 *
 * kq_obs_quantize: W [d_out x d_in] fp32 (the rotated, rescaled W'; destroyed), Lt from
 *   kq_chol_inv, Pt from kq_gptaq_p or NULL. For each block of `block` columns and each
 *   column j of it:
 *     q_j = clamp(rint(w_j / scale) + zero, 0, 2^bits - 1)        (round half to even)
 *     E_j = (w_j - scale * (q_j - zero)) / R_jj,  w_k -= E_j R_jk for k in (j, block end)
 *     with P:  w_k += w_j P_jk as well (w_j = column j's value just before quantization)
 *   then W[:, block end:] -= E_block R[block, block end:]
 *     with P:  W[:, block end:] += Wpre_block P[block, block end:] as well.
 *   Grid (asymmetric min-max): xmin = min(0, min x), xmax = max(0, max x), (-1, 1) if both
 *   are 0; scale = (xmax - xmin) / (2^bits - 1); zero = rint(-xmin / scale).
 *   group = 0: one grid per row from the whole row before the sweep (scale/zero [d_out]).
 *   group = block: one grid per row and block from the current, compensated block at
 *   block start (scale/zero [d_out x ceil(d_in / block)]).
 *   Outputs: codes [d_out x d_in] uint8; scale fp32 and zero int32 as above; col_loss
 *   [d_in] (nullable) = sum over rows of E_j^2; pre_q [d_out x d_in] (nullable) = the value
 *   w_j just before it was quantized.
 *   mode selects the arithmetic of the lazy trailing update (the column loop is the same):
 *   KQ_TRAIL_FP32: every fp32 operation and its order are fixed (IEEE division, rintf, one
 *     fmaf per intra-block update, with P w_k = fmaf(w_j, P_jk, fmaf(-E_j, R_jk, w_k));
 *     trailing update as acc = fmaf(E_k, R_kc, acc) over ascending k, with P continuing
 *     acc = fmaf(-wpre_k, P_kc, acc) over ascending k, then w_c - acc), so results are
 *     reproducible bit for bit and equal to the fp32-ordered definition.
 *   KQ_TRAIL_3XTF32: the trailing update runs on the tensor cores with the 3xTF32 split
 *     (E R ~= E_hi R_hi + E_hi R_lo + E_lo R_hi, hi = rounded to tf32, lo = the exact
 *     remainder; fp32 accumulation). Its sums differ from the fp32 order in the last bits,
 *     so a code can differ from the fp32-ordered definition where w / scale falls on a
 *     rounding tie, and the rest of that row then follows a slightly different error path.
 *     Needs d_in % 4 == 0 and a 16-byte aligned W.
 *   Requirements: 1 <= bits <= 8, block == 128, group in {0, block}; with P also
 *   d_in % 16 == 0 and W, codes, Pt 16-byte aligned.
 *   info (nullable, device int): -KQ_ERR_TIMEOUT if a tensor-core pipeline wait gave up;
 *   -KQ_ERR_NONFINITE if a value about to be quantized was NaN or infinite (a non-finite W',
 *   for example from a NaN weight; that row's codes and grids are then meaningless).
 *   ws: kq_obs_quantize_workspace(d_out, d_in, block, mode, with_p) bytes (with_p = 1 when
 *   Pt will be passed), 256-byte aligned.
 * ---------------------------------------------------------------------------------- */
#define KQ_TRAIL_FP32 0
#define KQ_TRAIL_3XTF32 1
KQ_API size_t kq_obs_quantize_workspace(int64_t d_out, int64_t d_in, int block, int mode, int with_p);
KQ_API kq_status kq_obs_quantize(float* W, int64_t d_out, int64_t d_in, const float* Lt, const float* Pt,
                                 int bits, int group, int block, int mode, uint8_t* codes, float* scale,
                                 int32_t* zero, float* col_loss, float* pre_q, int* info, void* ws,
                                 size_t ws_bytes, kq_stream_t stream);

/* ------------------------------------------------------------------------------------
 * Inference with a quantized layer.
 * Paper: Algorithm 2's revert W^ = S_G^-1 U^T Q' V S_X^-1 (Q' the dequantized codes) and
 * Sec. 3.2 (at inference the diagonal scales are reverted elementwise and U, V cost
 * O(d log d) per layer). y = W^ x is computed without forming W^:
 *   x' = V S_X^-1 x (fast Hadamard transform), y' = Q' x' (dequantizing product over the
 *   packed codes), y = S_G^-1 U^T y' (fast Hadamard transform).
 *
 * kq_pack_codes: codes [d_out x d_in] uint8 (from kq_obs_quantize) -> packed, 32-bit words
 *   along each row: word w of a row holds codes w * (32 / pb) .. + 32 / pb - 1, code t of the
 *   word in bits [t pb, t pb + pb), pb = bits for 2-, 4- and 8-bit codes and 4 for 3-bit
 *   codes. kq_packed_codes_bytes(d_out, d_in, bits) bytes (0 for unsupported bits).
 *   Requirements: bits in {2, 3, 4, 8}, d_in % 128 == 0, packed 16-byte aligned.
 * kq_infer: y [B x d_out] fp32 = W^ x for B tokens x [B x d_in] fp32 (1 <= B <= 8), from
 *   the packed codes, scale fp32 and zero int32 ([d_out] for group 0, [d_out x d_in / 128]
 *   for group 128), s_x [d_in], s_g [d_out] and the RHT signs of the quantization.
 *   All arithmetic fp32 (codes are exact as floats; per group scale (sum q x' - zero sum x')).
 *   ws: kq_infer_workspace(B, d_in, d_out) bytes, 256-byte aligned. packed, x, y, s_x, s_g
 *   16-byte aligned, the signs 4-byte aligned, d_out % 4 == 0; s_x, s_g required (not NULL). d_in and d_out need Hadamard constructions (2^k or 28 * 2^k).
 *   info: optional device error word (see kq_check). The weight stream waits on its copies
 *   with a time limit; a wait that runs out records -KQ_ERR_TIMEOUT there and leaves that
 *   part of y as NaN.
 * ---------------------------------------------------------------------------------- */
KQ_API size_t kq_packed_codes_bytes(int64_t d_out, int64_t d_in, int bits);
KQ_API kq_status kq_pack_codes(const uint8_t* codes, int64_t d_out, int64_t d_in, int bits, uint32_t* packed,
                               kq_stream_t stream);
KQ_API size_t kq_infer_workspace(int64_t B, int64_t d_in, int64_t d_out);
KQ_API kq_status kq_infer(const uint32_t* packed, const float* scale, const int32_t* zero, int64_t d_out,
                          int64_t d_in, int bits, int group, const float* s_x, const float* s_g,
                          const int8_t* sign_u, const int8_t* sign_v, const float* x, int64_t B, float* y,
                          int* info, void* ws, size_t ws_bytes, kq_stream_t stream);

/* ------------------------------------------------------------------------------------
 * Check-only calls (not part of the timed path).
 *
 * kq_dequant_revert: Algorithm 2's revert. Q' = scale * (codes - zero) on each row/group
 *   grid, then W_hat = S_G^-1 U^T Q' V S_X^-1, written to W_hat [d_out x d_in] fp32.
 * kq_proxy_loss: Sec. 3.1 Eq. (kron_obj), loss = tr(H_G dW H_X dW^T), dW = W - W_hat, with
 *   H_G = NULL meaning the identity. Result in *loss (device double). ws:
 *   kq_proxy_loss_workspace(d_out, d_in) bytes.
 * ---------------------------------------------------------------------------------- */
KQ_API kq_status kq_dequant_revert(const uint8_t* codes, const float* scale, const int32_t* zero,
                            int64_t d_out, int64_t d_in, int group, const float* s_x,
                            const float* s_g, const int8_t* sign_u, const int8_t* sign_v,
                            float* W_hat, kq_stream_t stream);
KQ_API size_t kq_proxy_loss_workspace(int64_t d_out, int64_t d_in);
KQ_API kq_status kq_proxy_loss(const float* W, const float* W_hat, int64_t d_out, int64_t d_in,
                        const float* H_X, const float* H_G, double* loss, void* ws,
                        size_t ws_bytes, kq_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* KRONQ_H */
