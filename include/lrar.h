/*
 * lrar.h -- C ABI of liblrar.so, the GB300 (sm_103a) depth-attention mix of
 * "Low-Rank Attention Residuals" (arxiv 2607.09694).
 *
 * At a residual read site every token x mixes the outputs of earlier
 * sub-layers ("sources") i = 0..n_src-1 with a softmax over depth:
 *
 *   kbar_i = RMSNorm(k_i)            Eq. (8),  parameter-free (App. A.5)
 *   alpha_i = softmax_i(q . kbar_i)  Eq. (9),  static per-site query q
 *   h = sum_i alpha_i o_i            Eq. (10), full-width values
 *
 * where the routing key k_i is
 *   LRAR_PROJECTED  a learned r-dim key from the output projection (§3.3, Eq. 12),
 *   LRAR_SLICED     the last r coordinates of o_i (§3.4, Eq. 14),
 *   LRAR_FULL       o_i itself with r = d, i.e. standard AttnRes (§3.1, Eq. 2).
 *
 * RMSNorm is k / sqrt(mean_j k_j^2 + eps); eps is an argument because the
 * paper does not state it.  Scores carry no temperature.
 *
 * Layout (all row-major, all device memory owned by the caller):
 *   values  [n_src, T, d]   source-major stack of sub-layer outputs
 *   keys    [n_src, T, r]   P-LR keys (LRAR_PROJECTED only)
 *   query   [r] float32     (r = d for LRAR_FULL)
 *   h, dh   [T, d]          mixed output and its upstream gradient
 *   lse     [T] float32     log sum_i exp(score_i), saved by the forward
 *
 * Conventions shared by every entry point:
 *   - Calls are asynchronous and ordered on `stream` (a cudaStream_t; NULL is
 *     the legacy default stream).  No call synchronises the host or allocates
 *     memory, and no call keeps state between calls except
 *     lrar_backward_noalloc (its fixed scratch array and the cached address of
 *     it, described there); the library is thread-safe.
 *   - Return value: LRAR_OK (0) or a negative LRAR_ERR_* code.  Argument
 *     checks run before anything is launched; on error nothing is launched and
 *     outputs are untouched.  lrar_last_error() gives a message for the
 *     calling thread's most recent failure.
 *   - Tensor pointers must be 16-byte aligned (query, lse and dq: 4-byte),
 *     and d * sizeof(input element) must be a multiple of 16 bytes
 *     (LRAR_ERR_ALIGNMENT otherwise).
 *   - Element types: LRAR_F32 or LRAR_BF16; arithmetic is float32 throughout
 *     and every bfloat16 store rounds to nearest even.
 */
#ifndef LRAR_H
#define LRAR_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define LRAR_VERSION 2
#define LRAR_MAX_SOURCES 128
#define LRAR_MAX_BLOCK_SITES 64

/*
 * Bits a kernel may OR into a caller's optional device status word (the
 * `status` arguments below).  The library never clears the word: the caller
 * zeroes it, runs the calls, and reads it back when it wants to know.
 */
#define LRAR_STATUS_WAIT_TIMEOUT 1 /* a bounded wait inside a kernel gave up (about 2 s); outputs are invalid */
#define LRAR_STATUS_LSE_MISMATCH 2 /* a backward that took alpha from a supplied lse found a token whose
                                      weights sum to more than 1e-3 away from 1 (an lse of other inputs) */

enum lrar_variant { LRAR_FULL = 0, LRAR_SLICED = 1, LRAR_PROJECTED = 2 };
enum lrar_dtype { LRAR_F32 = 0, LRAR_BF16 = 1 };
enum lrar_status {
    LRAR_OK = 0,
    LRAR_ERR_INVALID_ARG = -1, /* null required pointer, bad enum, n_src < 1, r < 1, r > d,
                                  FULL with r != d, T < 0, eps <= 0 or not finite */
    LRAR_ERR_ALIGNMENT = -2,   /* pointer not 16-byte aligned or row size not a multiple of 16 bytes */
    LRAR_ERR_UNSUPPORTED = -3, /* n_src > LRAR_MAX_SOURCES, d beyond the kernel's width limit */
    LRAR_ERR_CUDA = -4,        /* a CUDA call or launch failed; lrar_last_error() has its text */
    LRAR_ERR_WORKSPACE = -5    /* workspace NULL or smaller than lrar_backward_workspace_size() */
};

/*
 * Forward mix at one residual site: Eq. (8)-(10) for all T tokens.
 *
 *   variant   LRAR_FULL / LRAR_SLICED / LRAR_PROJECTED
 *   in_dtype  element type of values and keys
 *   out_dtype element type of h
 *   values    [n_src, T, d] in_dtype, read only
 *   keys      [n_src, T, r] in_dtype, read only; LRAR_PROJECTED only, ignored otherwise
 *   query     [r] float32; may be NULL only when n_src == 1 (the softmax is then 1)
 *   n_src     number of sources, 1..LRAR_MAX_SOURCES (site t of Full AttnRes has t)
 *   T         tokens (batch x sequence); T == 0 is a no-op
 *   d, r      value width and key width; r == d for LRAR_FULL
 *             (d <= 2048 for bfloat16 input, <= 1024 for float32)
 *   eps       RMSNorm epsilon, > 0
 *   h         [T, d] out_dtype, written
 *   lse       [T] float32, written when non-NULL (LRAR_FULL's backward needs it;
 *             LRAR_SLICED's writing backward uses it to skip its routing stage)
 *   stream    cudaStream_t
 */
int lrar_forward(int variant, int in_dtype, int out_dtype, const void *values, const void *keys,
                 const float *query, int n_src, int64_t T, int d, int r, float eps, void *h, float *lse,
                 void *stream);

/*
 * Bytes of device workspace lrar_backward needs: the per-CTA partial sums of
 * dq, reduced in a fixed order so that dq is bitwise reproducible.  Depends
 * only on the arguments (not on the device).
 */
size_t lrar_backward_workspace_size(int variant, int n_src, int64_t T, int d, int r);

/*
 * Backward of lrar_forward: gradients of a loss L given dh = dL/dh.
 * The paper prints no gradient formulas; these are the chain rule through
 * Eq. (8)-(10):
 *   g_i = <dh, o_i>,  gbar = sum_i alpha_i g_i,  ds_i = alpha_i (g_i - gbar)
 *   dL/do_i  = alpha_i dh  (+ the key gradient where the key lives in o_i)
 *   dL/dk_i  = ds_i rho_i (q - (s_i / r) kbar_i),  rho_i = 1/sqrt(mean k_i^2 + eps)
 *   dL/dq    = sum over tokens and sources of ds_i kbar_i
 * SLICED adds dL/dk_i into the last r coordinates of dvalues; FULL adds it to
 * all of dvalues; PROJECTED writes it to dkeys.
 *
 *   in_dtype   element type of values, keys and dh
 *   grad_dtype element type of dvalues and dkeys
 *   dh         [T, d] in_dtype
 *   h          [T, d] h_dtype, the forward output; required for LRAR_FULL
 *              (gbar = <dh, h> lets FULL finish in one pass), ignored otherwise.
 *              gbar is exact for a float32 h; a bfloat16 h carries its rounding
 *              into gbar (as FlashAttention's backward does with its stored
 *              output): at most alpha_i rho_i |q - (s_i/d) kbar_i| sum_j |dh_j|
 *              ulp(h_j)/2 per gradient element
 *   h_dtype    element type of h
 *   lse        [T] float32 from the forward (4-byte aligned); required for LRAR_FULL.
 *              LRAR_SLICED may take it: when the gradients are written
 *              (accumulate = 0) and in_dtype == grad_dtype, alpha_i = exp(s_i - lse)
 *              comes from each value row's own key slice and the backward makes one
 *              pass over the values instead of a routing stage, a value pass and a
 *              key pass (same results up to fp32 rounding order).  It must be the
 *              forward's lse of the same values and query.  NULL: the sliced
 *              backward recomputes the routing.  Ignored for LRAR_PROJECTED.
 *   dvalues    [n_src, T, d] grad_dtype, written (accumulate = 0) or added into
 *   dkeys      [n_src, T, r] grad_dtype; LRAR_PROJECTED only, same accumulate rule
 *   dq         [r] float32, written or added into; summed over all T tokens
 *   accumulate 0: overwrite dvalues/dkeys/dq; 1: add into them (a source
 *              receives gradient from every later site)
 *   workspace  device scratch of at least lrar_backward_workspace_size() bytes,
 *              16-byte aligned; contents on entry are ignored
 *   status     optional device int (4-byte aligned), may be NULL: where alpha is
 *              taken from the supplied lse (LRAR_FULL; LRAR_SLICED's one-pass
 *              form), each token checks that its weights sum to 1 within 1e-3 and
 *              ORs LRAR_STATUS_LSE_MISMATCH in when they do not -- the sign of an
 *              lse that belongs to other values or another query.  The gradients
 *              are then not valid.  Never written otherwise.
 *   Other arguments as for lrar_forward.  values, dvalues and dkeys must not overlap.
 */
int lrar_backward(int variant, int in_dtype, int grad_dtype, const void *values, const void *keys,
                  const float *query, int n_src, int64_t T, int d, int r, float eps, const void *dh,
                  const void *h, int h_dtype, const float *lse, void *dvalues, void *dkeys, float *dq,
                  int accumulate, void *workspace, size_t workspace_bytes, int *status, void *stream);

/*
 * lrar_backward for callers that cannot allocate device memory.  The paper has
 * no counterpart: this is a deployment variant of lrar_backward.
 *
 * Some callers cannot hand lrar_backward a workspace: plugin callbacks of
 * inference or training runtimes that must not allocate while they run,
 * services held to a fixed device-memory budget, and C hosts that receive
 * device pointers from another component and have no device allocator.  This
 * call takes the same arguments minus the workspace and allocates nothing: its
 * scratch is a fixed 4 MiB array compiled into the library, which every GPU
 * that loads the library holds until the process exits.
 *   - Problems whose workspace would exceed 4 MiB (lrar_backward_workspace_size()
 *     > 4 MiB, i.e. a dq width -- r, or d for LRAR_FULL -- above 1024) are
 *     rejected with LRAR_ERR_UNSUPPORTED before anything runs.
 *   - The first call on each device that passes the argument checks looks up
 *     the scratch's device address with that device current, and keeps it for
 *     the life of the process; make that first call before any stream capture.
 *     A reset of the device (cudaDeviceReset, or a reset of its primary
 *     context) invalidates the kept address: do not use this call on a device
 *     after such a reset.
 *   - All calls on a device share the one scratch array.  None of it needs to
 *     start at zero (every partial sum is written before it is read), but calls
 *     that may run at the same time on the GPU (different streams, or host
 *     threads without ordering between them) race on it: serialise them.
 * Results, errors and all other rules are those of lrar_backward; arguments
 * are checked (with lrar_backward's codes and messages) before the device is
 * touched.
 */
int lrar_backward_noalloc(int variant, int in_dtype, int grad_dtype, const void *values, const void *keys,
                          const float *query, int n_src, int64_t T, int d, int r, float eps, const void *dh,
                          const void *h, int h_dtype, const float *lse, void *dvalues, void *dkeys, float *dq,
                          int accumulate, int *status, void *stream);

/*
 * Block AttnRes source assembly (§3.1, Eq. 5-6) and its gradient fan-out:
 *   dst[e] = beta * dst[e] + alpha * src[e]   for e = 0..count-1
 * beta == 0 does not read dst (opens a new block summary: dst = alpha * src).
 * After sub-layer j writes o_j, `dst = partial summary slot, src = o_j, beta = 1`
 * extends the partial block; in the backward `dst = d(o_j), src = d(slot)`
 * hands each member its summary's gradient.  For P-LR the same call sums keys
 * (the paper does not define a summary's key; this library reads it as the
 * sum of the members' keys).
 *   dst_dtype, src_dtype  element types (may differ, e.g. float32 summaries of
 *                         bfloat16 outputs)
 *   count                 elements (T * width); 0 is a no-op
 */
int lrar_block_accumulate(int dst_dtype, void *dst, int src_dtype, const void *src, int64_t count,
                          float alpha, float beta, void *stream);

/*
 * Block AttnRes two-phase batched sites (§3.5), low-rank keys only.  The
 * n_sites read sites inside one block all see the block's completed sources
 * (the embedding and the completed block summaries, Eq. 5) plus a partial
 * summary that grows by one output per site (Eq. 6).  Because the queries are
 * static, one pass over the completed sources serves every site of the block
 * (phase 1), and each site then folds in its partial summary with an
 * online-softmax update (phase 2).  The completed sources are read once per
 * block instead of once per site; the result equals lrar_forward over
 * [completed sources, partial summary].
 *
 * Phase 1:
 *   values      [n_completed, T, d] in_dtype: the completed sources (a stack prefix)
 *   keys        [n_completed, T, r] in_dtype, LRAR_PROJECTED only
 *   queries     [n_sites, r] float32, one static query per site
 *   h_pre       [n_sites, T, d] pre_dtype, written: softmax mix over the completed
 *               sources only (float32 keeps phase 2 exact; bfloat16 rounds it)
 *   lse_pre     [n_sites, T] float32, written: log sum_i exp(score) over them
 *   n_sites     1..LRAR_MAX_BLOCK_SITES
 *   status      optional device int (4-byte aligned), may be NULL: the kernel
 *               stages each token's keys with bulk copies and waits for them
 *               with a bound (about 2 s); a wait that runs out ORs
 *               LRAR_STATUS_WAIT_TIMEOUT in, stops the launch's further copies,
 *               and the launch drains the copies in flight and returns (h_pre
 *               and lse_pre are then not valid).  Never written otherwise.
 * Phase 2 (one site):
 *   h_pre, lse_pre  that site's rows of the phase-1 outputs ([T, d], [T])
 *   partial     [T, d] in_dtype: the partial-block summary (for the first site
 *               of a block the partial block is empty: use h_pre as h directly)
 *   partial_key [T, r] in_dtype: its projected key (LRAR_PROJECTED), else ignored
 *   query       [r] float32: the site's query
 *   h           [T, d] out_dtype, written; lse [T] float32, written when non-NULL.
 *               h may be h_pre and lse may be lse_pre (in place, pre_dtype ==
 *               out_dtype): each element is read before it is written.
 * Other arguments and errors as for lrar_forward; LRAR_FULL is LRAR_ERR_UNSUPPORTED.
 */
int lrar_block_phase1(int variant, int in_dtype, int pre_dtype, const void *values, const void *keys,
                      const float *queries, int n_completed, int n_sites, int64_t T, int d, int r, float eps,
                      void *h_pre, float *lse_pre, int *status, void *stream);
/* Phase 1 with the completed sources as separate tensors: values (and, for
 * LRAR_PROJECTED, keys) are HOST arrays of n_completed device pointers to [T, d]
 * (keys: [T, r]) matrices, 16-byte aligned, read during the call (the rules of
 * lrar_forward_ptrs).  Everything else as lrar_block_phase1. */
int lrar_block_phase1_ptrs(int variant, int in_dtype, int pre_dtype, const void *const *values,
                           const void *const *keys, const float *queries, int n_completed, int n_sites, int64_t T,
                           int d, int r, float eps, void *h_pre, float *lse_pre, int *status, void *stream);
int lrar_block_phase2(int variant, int in_dtype, int pre_dtype, int out_dtype, const void *h_pre,
                      const float *lse_pre, const void *partial, const void *partial_key, const float *query,
                      int64_t T, int d, int r, float eps, void *h, float *lse, void *stream);
/* Phase 2 that also assembles the partial summary it reads (Eq. 6): with the
 * open block's running sum through the previous member, prev_partial, and the
 * newest member's output, member, the partial summary is b = prev_partial +
 * member (float32 sum rounded once to in_dtype, bit for bit the result of
 * lrar_block_accumulate(member, prev_partial, alpha = beta = 1)).  b is written
 * over member, and the site's h and lse are those of lrar_block_phase2 with
 * partial = b.  For LRAR_PROJECTED, member_key is likewise replaced by
 * prev_partial_key + member_key.  The accumulate + phase-2 pair it replaces
 * reads b twice; this call reads its two terms once.
 *   prev_partial      [T, d] in_dtype, read
 *   member            [T, d] in_dtype, read and overwritten with b
 *   prev_partial_key  [T, r] in_dtype (LRAR_PROJECTED), read; else ignored
 *   member_key        [T, r] in_dtype (LRAR_PROJECTED), read and overwritten; else ignored
 * member (and member_key) must not overlap prev_partial, h_pre or h.
 * Everything else, and the errors, as lrar_block_phase2; prev_partial (and,
 * for LRAR_PROJECTED, prev_partial_key) NULL with T > 0 is LRAR_ERR_INVALID_ARG.
 */
int lrar_block_phase2_assemble(int variant, int in_dtype, int pre_dtype, int out_dtype, const void *h_pre,
                               const float *lse_pre, const void *prev_partial, void *member,
                               const void *prev_partial_key, void *member_key, const float *query, int64_t T,
                               int d, int r, float eps, void *h, float *lse, void *stream);

/*
 * Routing diagnostics of one site (§4.5-4.6): the effective number of sources
 * of every token, N_eff = exp(H(alpha)) with H = -sum_i alpha_i log alpha_i
 * (Eq. 16; 0 log 0 = 0), and alpha averaged over the T tokens (one row of the
 * mean-attention heatmap).  alpha is that of lrar_forward with the same
 * arguments (Eq. 8-9); for low-rank keys only the keys are read.
 *   neff        [T] float32, written; may be NULL
 *   mean_alpha  [n_src] float32, written; may be NULL (then no workspace is needed)
 *   workspace   >= lrar_diagnostics_workspace_size(n_src) bytes, 16-byte aligned,
 *               when mean_alpha is requested; contents on entry are ignored.
 *               The mean is summed in a fixed order (bitwise reproducible).
 * Other arguments, layouts and errors as for lrar_forward; T == 0 sets mean_alpha to 0.
 */
size_t lrar_diagnostics_workspace_size(int n_src);
int lrar_diagnostics(int variant, int in_dtype, const void *values, const void *keys, const float *query,
                     int n_src, int64_t T, int d, int r, float eps, float *neff, float *mean_alpha, void *workspace,
                     size_t workspace_bytes, void *stream);

/*
 * Sources as separate tensors (a pointer table instead of one stacked buffer):
 * every argument and rule is that of lrar_forward / lrar_backward, except
 *   values   HOST array of n_src device pointers; values[i] is source i's
 *            row-major [T, d] matrix (16-byte aligned)
 *   keys     HOST array of n_src pointers to [T, r] P-LR key matrices
 *            (LRAR_PROJECTED only, else ignored)
 *   dvalues, dkeys  HOST arrays of n_src pointers to the matching gradient
 *            matrices (each [T, d] / [T, r] of grad_dtype)
 * The arrays are read during the call and copied into the launch, so they
 * may be reused as soon as the call returns (a captured CUDA graph keeps the
 * pointers it saw).  A NULL array, a NULL entry or an unaligned entry is
 * rejected (LRAR_ERR_INVALID_ARG / LRAR_ERR_ALIGNMENT) before anything runs.
 * Gradient matrices of different sources must not overlap.
 */
int lrar_forward_ptrs(int variant, int in_dtype, int out_dtype, const void *const *values, const void *const *keys,
                      const float *query, int n_src, int64_t T, int d, int r, float eps, void *h, float *lse,
                      void *stream);
int lrar_backward_ptrs(int variant, int in_dtype, int grad_dtype, const void *const *values,
                       const void *const *keys, const float *query, int n_src, int64_t T, int d, int r, float eps,
                       const void *dh, const void *h, int h_dtype, const float *lse, void *const *dvalues,
                       void *const *dkeys, float *dq, int accumulate, void *workspace, size_t workspace_bytes,
                       int *status, void *stream);

/*
 * P-LR fused output projection (§3.3, Eq. 11-12) on the tensor cores:
 *   [o ; k] = [W_O ; W_K] a    for every token, i.e.  Y = A W^T,  Y [T, d + r]
 * Columns 0..d-1 of Y go to o, columns d..d+r-1 to keys, so a sub-layer's
 * output projection writes its value slot and its key slot in one pass (the
 * keys are never re-read to build the key stack).  With d = 0 it is Eq. 13's
 * embedding key k_0 = W_0^K o_0.  bfloat16 operands, float32 accumulation,
 * bfloat16 outputs rounded to nearest even.
 *   a       [T, m] row-major activations entering the output projection
 *           (m = d for attention, the SwiGLU hidden width for the FFN)
 *   w       [d + r, m] row-major: the d rows of W_O, then the r rows of W_K
 *   o       [T, d] (may be NULL when d == 0);  keys [T, r] (NULL when r == 0)
 *   status  optional device int (4-byte aligned): LRAR_STATUS_WAIT_TIMEOUT is
 *           ORed in if a pipeline wait inside the kernel gave up (about 2 s; the
 *           outputs are then not valid).  Never written otherwise.
 * in_dtype must be LRAR_BF16 (LRAR_ERR_UNSUPPORTED otherwise); m, d and r must
 * be multiples of 8 and a, w, o, keys 16-byte aligned (LRAR_ERR_ALIGNMENT).
 * T == 0 is a no-op.  No counterpart of the depth mix's other rules: the call
 * reads a and w, writes o and keys, and is ordered on `stream` like every call.
 */
int lrar_project(int in_dtype, const void *a, const void *w, int64_t T, int m, int d, int r, void *o, void *keys,
                 int *status, void *stream);

/* Static text for a status code. */
const char *lrar_strerror(int code);

/* Message of the calling thread's most recent failed call ("" if none). */
const char *lrar_last_error(void);

/* LRAR_VERSION of the built library. */
int lrar_version(void);

#ifdef __cplusplus
}
#endif

#endif /* LRAR_H */
