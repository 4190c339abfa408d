/*
 * xpress.h -- C ABI of the GB300 (sm_103a) implementation of the xPress
 * parallel refinement pass (arXiv 2608.02438, "xPress: Parallel Refinement for
 * Diffusion Drafters in Speculative Decoding").
 *
 * Conventions for every entry point
 *   - Tensors are DEVICE pointers to row-major, contiguous arrays owned by the
 *     caller; the library never frees them and keeps no reference to them
 *     after a call returns, except the weights given to xpress_refiner_create
 *     (which must outlive the refiner).
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *     Calls are asynchronous on that stream; results are valid after the
 *     stream is synchronised.
 *   - The return value reports argument validation and launch errors only
 *     (xpress_status).  Errors detected by the kernels themselves (a token id
 *     out of range, a bounded wait that timed out) are recorded in a status
 *     word inside the workspace; read it with xpress_get_device_status after
 *     synchronising.
 *   - Storage dtype: XPRESS_BF16 (bf16 bit patterns, 2 bytes) or XPRESS_F32.
 *     Weights, drafter hidden states h, base logits s and target logits all
 *     use the refiner's dtype.  Accumulation is fp32 throughout.  In the bf16
 *     case the activations that feed a tensor-core product are rounded to bf16
 *     (round to nearest even): c before W_1, sigma(W_1 c) before W_2, z before
 *     W_r.  Logits l = s + delta, log-sum-exp and sampling are fp32.
 *   - Supported shapes: r = 256, 1 <= B <= 32, V >= 32, V % 8 == 0,
 *     H % 8 == 0; otherwise XPRESS_ERR_UNSUPPORTED.
 *   - A refiner handle is not thread-safe: calls that use the same handle from
 *     several host threads must be serialised by the caller.
 */
#ifndef XPRESS_H
#define XPRESS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum { XPRESS_F32 = 0, XPRESS_BF16 = 1 } xpress_dtype;

/* sigma in Trans (Sec. 4.1 calls it "a pointwise nonlinearity"). */
typedef enum { XPRESS_ACT_SILU = 0, XPRESS_ACT_GELU = 1, XPRESS_ACT_RELU = 2 } xpress_act;

typedef enum {
    XPRESS_OK = 0,
    XPRESS_ERR_INVALID_ARG = -1,   /* NULL pointer, bad size, misaligned pointer */
    XPRESS_ERR_UNSUPPORTED = -2,   /* shape or dtype outside the supported set */
    XPRESS_ERR_CUDA = -3,          /* a CUDA runtime call failed */
    XPRESS_ERR_WORKSPACE = -4,     /* workspace NULL, too small or misaligned */
    XPRESS_ERR_TIMEOUT = -5,       /* device: a bounded wait gave up */
    XPRESS_ERR_DEVICE_CHECK = -6   /* device: an input failed a bounds check */
} xpress_status;

/* Opaque refiner: derived device tensors built once from the weights. */
typedef struct xpress_refiner xpress_refiner;

/* Refiner weights R_theta (Sec. 4.1, Eq. fuse / mix / mlp / read), device
 * pointers in the refiner dtype, row-major:
 *   W_e  [V, r]    token embedding; row x is the paper's column W_e[x]
 *   W_h  [r, H]    down-projection of h_k
 *   W_g  [r, H]    down-projection of the block mean g
 *   W_in [r, 3r]   fusion of [W_h h_k || W_g g || W_e[x_{k-1}]] (in that order)
 *   L    [r, B, B] per-channel causal mixer, L[d][k][j] = L^(d)_{k,j}; only the
 *                  strictly lower triangle (j < k) is read
 *   W1   [2r, r], W2 [r, 2r]   Trans MLP
 *   W_r  [V, r]    readout head (shared over positions, not tied to W_e)   */
typedef struct {
    int H, V, r, B;
    int dtype; /* xpress_dtype */
    int act;   /* xpress_act */
    const void *W_e, *W_h, *W_g, *W_in, *L, *W1, *W2, *W_r;
} xpress_weights;

/* Builds the derived tensors (the folded embedding E' = W_in[:, 2r:3r] W_e,
 * fp32 [V, r], and the TMA descriptors) on `stream` and synchronises it.
 * Allocates device memory (released by xpress_refiner_destroy).
 * Errors: INVALID_ARG (NULL), UNSUPPORTED (shape/dtype), CUDA. */
int xpress_refiner_create(const xpress_weights *w, void *stream, xpress_refiner **out);
int xpress_refiner_destroy(xpress_refiner *refiner);

/* One refinement call over b independent blocks (Sec. 4.2, Algorithm 1).
 *   h           [b, B, H]   drafter hidden states h_1..h_B (Sec. 4.1)
 *   s           [b, B, V]   drafter base logits s_k (Eq. correct)
 *   draft       [b, B]      Y^(0), int32 token ids; NULL => argmax_v s_k,v
 *                           (Algorithm 1's seed)
 *   anchor      [b]         x_0, the fixed anchor token (the last verified token)
 *   temperature [b]         T per sequence; T <= 0 re-selects by argmax
 *                           (Algorithm 1), T > 0 by the fixed-noise
 *                           hierarchical Gumbel-max draw of softmax(l/T)
 *   seed        [b]         Philox4x32-10 key per sequence
 *   offset                  per speculative round (counter word 3)
 *   K_max                   maximum number of refiner passes, >= 1
 *   fixed_K                 0: stop a block when a pass leaves it unchanged
 *                           (Algorithm 1's break); 1: run exactly K_max
 *                           passes on every block (Table 3 style timing)
 *   mode                    XPRESS_MODE_JACOBI: Algorithm 1 (parallel passes);
 *                           XPRESS_MODE_SEQUENTIAL: the sequential decode of
 *                           Theorem 1, y*_k = Select(R(y*_<k))_k for
 *                           k = 1..B, one position per pass (B dependent
 *                           passes; needs K_max >= B; draft and fixed_K are
 *                           not used; iters = B, converged = 1).  Both modes
 *                           reach the same block (Theorem 1); the second is
 *                           the serial baseline the paper compares against
 *                           (Table 3).                                      */
typedef enum { XPRESS_MODE_JACOBI = 0, XPRESS_MODE_SEQUENTIAL = 1 } xpress_mode;

typedef struct {
    int b;
    const void *h;
    const void *s;
    const int32_t *draft;
    const int32_t *anchor;
    const float *temperature;
    const uint64_t *seed;
    uint32_t offset;
    int K_max;
    int fixed_K;
    int mode; /* xpress_mode */
} xpress_block_in;

/* Outputs (device pointers; each may be NULL except tokens):
 *   tokens    [b, B]  refined block Y (int32)
 *   iters     [b]     refiner passes executed for the block (1..K_max)
 *   converged [b]     1 if the last pass left the block unchanged
 *   lse       [b, B]  T > 0: log sum_v exp(l_k,v / T) of the pass that last
 *                     evaluated position k; T <= 0: NaN
 *   logit_sel [b, B]  l_k,y / T at the selected token (T <= 0: l_k,y)
 *   z_final   [b, B, r] fp32 z_k of that pass (the W_r operand before rounding)
 *   refined_logits [b, B, V] fp32 l_k (debug; slows the pass down)
 *   trajectory [b, K_max, B] int32 (debug): trajectory[s][j][k] is the token
 *                     pass j + 1 selected for position k of block s, written
 *                     only where that pass evaluated position k (a pass
 *                     evaluates the positions after the first one the previous
 *                     pass changed, Theorem 1); every other entry keeps what
 *                     the caller stored there.  Y^(j) of Algorithm 1 is
 *                     recovered by carrying each position's last written
 *                     token forward from Y^(0).                             */
typedef struct {
    int32_t *tokens;
    int32_t *iters;
    int32_t *converged;
    float *lse;
    float *logit_sel;
    float *z_final;
    float *refined_logits;
    int32_t *trajectory;
} xpress_block_out;

/* Bytes of device workspace xpress_refine_block needs for b blocks. */
size_t xpress_refine_workspace_size(const xpress_refiner *refiner, int b);

/* Runs Algorithm 1 on all b blocks with no host synchronisation: the
 * iteration loop runs on the device.  Calls of a bf16 refiner (H a multiple of
 * 64) that evaluate at most 32 tokens (b * B <= 32) run as one persistent
 * cooperative kernel whose CTAs apply the stopping rule themselves; other
 * calls run a CUDA graph whose
 * WHILE conditional node repeats the per-pass kernels until the device clears
 * its condition.  Blocks that have converged drop out of later passes, and a
 * pass re-evaluates only the positions after the first token the previous
 * pass changed (by Theorem 1 the others cannot change).  workspace: >= the
 * size above, 256-byte aligned, owned by the caller, not shared by concurrent
 * calls.
 * Errors: INVALID_ARG, UNSUPPORTED, WORKSPACE, CUDA. */
int xpress_refine_block(const xpress_refiner *refiner, const xpress_block_in *in,
                        const xpress_block_out *out, void *workspace, size_t ws_bytes,
                        void *stream);

/* Acceptance of refined blocks against the target's logits (Sec. 3.1).
 *   target      [b, B+1, V] target logits for positions 1..B and the bonus
 *   s, tokens, lse, logit_sel, z_final: as passed to / returned by
 *               xpress_refine_block for the same blocks
 *   temperature [b] T <= 0: greedy -- accept the longest prefix equal to the
 *               target argmax, then emit the target's token;  T > 0: lossless
 *               rejection sampling -- accept y_k when u_k q_k(y_k) < p_k(y_k),
 *               else emit a draw of max(0, p_k - q_k) (p_k if that is empty);
 *               after B acceptances emit a draw of p_{B+1}
 *   seed, offset: as for refinement (streams 2 and 3)
 * All input pointers are required (lossless draws read lse, logit_sel, z_final
 * and s).
 * Outputs: accept_len [b] (0..B accepted draft tokens) and out_tokens
 * [b, B+1] (accepted tokens, then the correction or bonus token, then -1).
 * Errors: INVALID_ARG, WORKSPACE, CUDA. */
typedef struct {
    int b;
    const void *target;
    const void *s;
    const int32_t *tokens;
    const float *lse;
    const float *logit_sel;
    const float *z_final;
    const float *temperature;
    const uint64_t *seed;
    uint32_t offset;
} xpress_accept_in;

size_t xpress_accept_workspace_size(const xpress_refiner *refiner, int b);
int xpress_accept(const xpress_refiner *refiner, const xpress_accept_in *in, int32_t *accept_len,
                  int32_t *out_tokens, void *workspace, size_t ws_bytes, void *stream);

/* xpress_accept for callers that cannot allocate device memory (code that
 * runs while another thread captures a CUDA graph, allocators that forbid
 * device allocations after start-up, hosts that only hand out pre-registered
 * buffers).  It takes no workspace: the acceptance kernels keep their scratch
 * in a fixed 256 KiB array inside this library (a file-scope __device__
 * array, held by every GPU that loads the library until the process exits).
 * The paper has no counterpart to this entry point; it exists for such
 * callers only.
 *   - Same inputs, outputs and results as xpress_accept.
 *   - Size limit: the scratch of the batch must fit the array, which holds
 *     any batch with b * (B + 1) <= 8192 target rows on a 152-SM GB300;
 *     larger batches return XPRESS_ERR_UNSUPPORTED (use xpress_accept).
 *   - Allocates nothing: no cudaMalloc, no cudaFree, no allocating library
 *     call.  Its first call on a device looks up the array's device address
 *     (cudaGetSymbolAddress, once per device, with that device current);
 *     make that first call before any stream capture.
 *   - The refiner's device must be the current device; a call made with
 *     another device current returns XPRESS_ERR_INVALID_ARG.
 *   - Every call shares the one array, which keeps the previous call's
 *     contents: calls that overlap on the GPU (other streams, other threads)
 *     race on it and must be serialised by the caller.  Calls issued back to
 *     back on one stream are serialised by that stream.  The device status of
 *     these calls is not reported (xpress_get_device_status needs a
 *     workspace).
 * Errors: INVALID_ARG, UNSUPPORTED (batch too large), CUDA. */
int xpress_accept_noalloc(const xpress_refiner *refiner, const xpress_accept_in *in, int32_t *accept_len,
                          int32_t *out_tokens, void *stream);

/* Synchronises `stream`, then reads (and clears) the device status word kept
 * in `workspace` by xpress_refine_block / xpress_accept / xpress_train_step.  *status_out is an
 * xpress_status (XPRESS_OK, XPRESS_ERR_TIMEOUT or XPRESS_ERR_DEVICE_CHECK). */
int xpress_get_device_status(void *workspace, void *stream, int32_t *status_out);

/* Base logits of the drafter (Sec. 4.1, Fig. 2a: the target-sized LM head
 * that produces s_k, the Correct term of the refiner) and Algorithm 1's seed
 * Y^(0) = argmax_v s_k,v, for N hidden states.
 *   W_lm        [V, H] bf16, row v = the LM head's row for token v
 *   h           [N, H] bf16 hidden states (e.g. [b, B, H] flattened)
 *   s_out       [N, V] bf16 (may be NULL): s[n][v] = sum_i h[n][i] W_lm[v][i],
 *               accumulated in fp32 on tensor cores and rounded once to bf16
 *               (nearest even) -- the storage format xpress_refine_block
 *               reads
 *   argmax_out  [N] int32 (may be NULL): the first maximum of the stored s
 *               row (smallest id on ties), as xpress_refine_block takes it
 *               when no draft is given
 * At least one output must be given.  bf16 only; H % 8 == 0; W_lm and h
 * 16-byte aligned.  workspace: >= xpress_lm_head_workspace_size(V, N) bytes,
 * 256-byte aligned (per-CTA partial maxima).  Asynchronous on `stream`; two
 * kernel launches.
 * Errors: INVALID_ARG, WORKSPACE, CUDA. */
size_t xpress_lm_head_workspace_size(int V, int N);
int xpress_lm_head(const void *W_lm, int V, int H, const void *h, int N, void *s_out, int32_t *argmax_out,
                   void *workspace, size_t ws_bytes, void *stream);

/* Failure detection: every wait of the persistent small-batch kernel for
 * another CTA's progress (a monotone counter in the workspace) gives up after
 * `limit_ns` nanoseconds of wall time (2 s by default, 0 <= limit_ns <= 60 s);
 * the kernel then records XPRESS_ERR_TIMEOUT in the workspace's status word,
 * every CTA lets its own copies and tensor-core work drain, frees its tensor
 * memory and returns, and the next call on the workspace starts clean.  Waits
 * of a CTA on its own copies keep their own bounds.  Applies to the calls
 * made after it on this refiner (the paper has no counterpart; it exists so
 * that the timeout path can be exercised).
 * Errors: INVALID_ARG (NULL refiner, limit above 60 s). */
int xpress_set_wait_limit(xpress_refiner *refiner, uint64_t limit_ns);

/* Synchronises `stream`, then reads how many refiner passes the device loop
 * of the last xpress_refine_block call on `workspace` executed (the largest
 * per-block pass count that involved a kernel launch). */
int xpress_get_pass_count(void *workspace, void *stream, int32_t *passes_out);

/* Profiling hooks (benchmarks only).  After an xpress_refine_block call on
 * `workspace`, _prepare marks the first n_tokens positions of the b blocks as
 * evaluated, and xpress_profile_read launches the Read + Correct + selection
 * kernel alone on `stream` (its results overwrite the call's scratch), so
 * that it can be timed with CUDA events.  The inputs of that call must still
 * be alive.  Errors: INVALID_ARG, WORKSPACE, CUDA. */
int xpress_profile_read_prepare(const xpress_refiner *refiner, void *workspace, int b, int n_tokens,
                                void *stream);
int xpress_profile_read(const xpress_refiner *refiner, void *workspace, int b, void *stream);

/* ------------------------------------------------------------------------
 * Refiner training step (Sec. 4.3): the loss of one batch of b blocks and its
 * gradient with respect to every refiner weight, at T = 1:
 *   L_total = L(p^r) + lambda L(p^b) + beta L(p^r-hat)
 *   L(p)    = sum_k w_k [a_ce (-log p_k(y*_k)) + a_l1 |p_k - p^t_k|_1],
 *             w_k = exp(-(k-1)/gamma), k = 1..B, p^t_k = softmax(target_k)
 *   p^r      the refiner's p_k = softmax(s_k + W_r z_k) under teacher forcing
 *            (inputs x_0 = anchor, x_k = y*_k for k >= 1, 0-based)
 *   p^b      the drafter's base distribution softmax(s_k): the drafter-anchor
 *            term (no refiner weight enters it)
 *   p^r-hat  the refiner fed the drafter's argmax tokens (x_k = argmax s_{k-1}):
 *            the consistency term
 * lambda weighs the anchor term and beta the consistency term, as in the total
 * loss equation.  The bf16 operand roundings of the forward (c, sigma(W_1 c)
 * and z, as in refinement) pass the gradient straight through; sgn(0) = 0 in
 * the L1 subgradient.  u_h and u_g enter W_in as bf16 hi + lo pairs (about 16
 * bits).  The backward products take bf16 operands (dL/dl, dL/dz, dL/dt,
 * dL/da and the Fuse operand rounded to bf16) with fp32 accumulation.
 * Refiner dtype XPRESS_BF16 only (UNSUPPORTED otherwise); in->B must equal the
 * refiner's B. */
typedef struct {
    int b, B;
    const void *h;           /* [b, B, H] bf16 drafter hidden states */
    const void *s;           /* [b, B, V] bf16 drafter base logits */
    const void *target;      /* [b, B, V] bf16 target logits of the same positions */
    const int32_t *ystar;    /* [b, B] ground-truth tokens */
    const int32_t *anchor;   /* [b] x_0 */
    const int32_t *xhat;     /* [b, B] the drafter's argmax tokens, or NULL: the first
                                argmax of each s row is computed on the device */
    float a_ce, a_l1;        /* weights of the cross-entropy and L1 terms */
    float gamma;             /* position-weight decay (> 0) */
    float lambda, beta;      /* anchor and consistency weights */
} xpress_train_in;

/* Gradients are ADDED into the caller's fp32 buffers (zero them to start a
 * step; leave them to accumulate over several batches), each shaped like its
 * weight (xpress_weights); gL's upper triangle and diagonal are left alone.
 * loss: [b, 4] per block L(p^r), L(p^b), L(p^r-hat), L_total (overwritten). */
typedef struct {
    float *loss;
    float *gW_e, *gW_h, *gW_g, *gW_in, *gL, *gW1, *gW2, *gW_r;
} xpress_train_out;

/* Workspace of xpress_train_step for b blocks of B positions. */
size_t xpress_train_workspace_size(const xpress_refiner *refiner, int b, int B);

/* One training step on `stream` (asynchronous; about 30 kernel launches:
 * one pass over s and target for the drafter's statistics and argmax, the
 * forward products, four Read passes over the vocabulary -- log-sum-exp,
 * total-variation sums, dL/dz, dL/dW_r -- and the backward products).  Token
 * ids out of [0, V) are clamped to 0 and reported by the status word
 * (XPRESS_ERR_DEVICE_CHECK); a bounded wait that gives up reports
 * XPRESS_ERR_TIMEOUT there.
 * Errors: INVALID_ARG (NULL pointer, h / s / target not 16-byte aligned,
 * b < 1, B mismatch, gamma <= 0), UNSUPPORTED (fp32 refiner), WORKSPACE, CUDA. */
int xpress_train_step(const xpress_refiner *refiner, const xpress_train_in *in, const xpress_train_out *out,
                      void *workspace, size_t ws_bytes, void *stream);

/* Profiling hook (benchmarks only): after an xpress_train_step call on
 * `workspace` with the same arguments, launches one of its four vocabulary
 * passes alone on `stream` so that it can be timed with CUDA events:
 * pass 0 the log-sum-exp statistics, 1 the total-variation sums, 2 dL/dz,
 * 3 dL/dW_r (which adds into out->gW_r once more).
 * Errors: as xpress_train_step; INVALID_ARG for another pass number. */
int xpress_profile_train(const xpress_refiner *refiner, const xpress_train_in *in, const xpress_train_out *out,
                         void *workspace, size_t ws_bytes, int pass, void *stream);

/* Test hook (not part of the method): C (+)= A B^T for bf16 device matrices
 * through the tensor-core product the training step uses, A [M, K] stored
 * with rows along M (a_mn = 0) or as [K, M] (a_mn = 1), B [N, K] or [K, N]
 * likewise, C [M, N] fp32: overwritten (accumulate = 0) or added into
 * (accumulate = 1, the K range then split over CTAs).  Rows of an operand
 * stored with rows along K need a multiple of 8 elements.
 * Errors: INVALID_ARG, CUDA. */
int xpress_debug_gemm(const void *A, int a_mn, const void *B, int b_mn, int M, int N, int K, float *C, int accumulate,
                      void *stream);

const char *xpress_status_string(int status);
int xpress_version(void);

#ifdef __cplusplus
}
#endif
#endif /* XPRESS_H */
