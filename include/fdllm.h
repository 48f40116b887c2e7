/*
 * fdllm.h -- C interface of the GB300 (sm_103a) commit-set selection library for
 * Frechet profile decoding of masked diffusion LLMs (Fast-dLLM++).
 *
 * One decode step of the paper's Algorithm 1, from logits at the masked positions of the
 * active block to the committed tokens and the updated mask:
 *   (a1) per masked position i: x_hat_i = argmax_v p_i(v) (lowest v on ties) and the
 *        confidence c_i = max_v p_i(v) = exp(M_i - logsumexp_i), p_i = softmax of row i
 *        (Sec. 3 "Notation"; Alg. 1 confidence loop);
 *   (a2) sort the masked confidences of each batch row in descending order, equal
 *        confidences lower position first (Alg. 1 sort);
 *   (a3) for every prefix size n: L_n = max{0, sum_{j<=n} c_(j) - (n-1)}, U_n = 1 - c_(n),
 *        G_n = L_n - U_n (Sec. 3 "Frechet profile quantities", Eq. frechet_Ln_Un);
 *   (a4) n* = max{n : G_n > delta}, n* = 1 when no n qualifies (Sec. 3; Alg. 1 select);
 *   (a5) reveal the n* most confident masked positions (Alg. 1 reveal).
 * Fast-dLLM's rules are available as alternative modes: factor, accept n iff
 * (n+1)(1 - c_(n)) < f (Sec. 1, Cor. factor-reduction); threshold, commit {i : c_i >= tau}
 * or the single most confident position when that set is empty (Sec. 2).
 *
 * Conventions for every entry point:
 *   - Pointers named logits, mask, out_*, conf, argmax and workspace are DEVICE pointers
 *     owned by the caller; the library never frees them.  `stream` is a cudaStream_t
 *     (NULL = legacy default stream) passed as void* so this header needs no CUDA headers.
 *   - logits is [B, L, V] row-major with V contiguous; dtype FDLLM_BF16 (bfloat16),
 *     FDLLM_FP16 (IEEE half) or FDLLM_FP32.  The base must be 16-byte aligned and
 *     V * sizeof(dtype) a multiple of 16 (V % 8 == 0 for bf16 and fp16, V % 4 == 0 for
 *     fp32); otherwise FDLLM_ERR_ALIGN.  A vocabulary
 *     that is not a multiple can be padded with -inf columns, which change nothing.
 *   - mask is uint8 [B, L], nonzero = masked.  Only masked positions are read from logits.
 *   - Limits: 1 <= B, 1 <= L <= FDLLM_MAX_L, B * L <= FDLLM_MAX_ROWS, V >= 1.
 *   - Work is enqueued asynchronously on `stream`; the return value reports only argument
 *     and launch errors, detected on the host.  Per-row data errors are reported in out_n
 *     (see FDLLM_ROW_NONFINITE) and, for calls that use a workspace, in its sticky status
 *     word, which fdllm_device_status / fdllm_workspace_status / fdllm_static_status read
 *     as FDLLM_ERR_NONFINITE.
 *   - All kernels are deterministic: the same inputs on the same GPU model give
 *     bit-identical outputs.  A position's confidence depends only on its logits and the
 *     call's shape (B * L, V, dtype), which fix how rows are cut into reduction units, so
 *     identical rows of one call give identical confidences (exact ties stay ties).
 *   - Arithmetic: confidences are reduced in fp32 (relative error within 1e-5 of the exact
 *     value); the rules are evaluated on those fp32 confidences with exact 64-bit fixed-point
 *     prefix sums of 1 - c in units of 2^-52 (delta = 1 - f formed from the same integer as
 *     f, so a flat profile gives the factor rule's decision bit for bit), and the threshold
 *     compares c with the smallest fp32 value >= tau, which decides c >= tau exactly.
 */
#ifndef FDLLM_H
#define FDLLM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define FDLLM_MAX_L 1024       /* positions per batch row (one CTA sorts a row in smem) */
#define FDLLM_MAX_ROWS 65536   /* B * L: masked-row compaction lives in shared memory */

typedef enum { FDLLM_BF16 = 0, FDLLM_FP32 = 1, FDLLM_FP16 = 2 } fdllm_dtype;

typedef enum {
    FDLLM_PROFILE = 0,   /* Frechet profile rule, Sec. 3: param = f, margin delta = 1 - f */
    FDLLM_FACTOR = 1,    /* Fast-dLLM factor rule: param = f                              */
    FDLLM_THRESHOLD = 2  /* Fast-dLLM threshold rule: param = tau                         */
} fdllm_mode;

typedef enum {
    FDLLM_OK = 0,
    FDLLM_ERR_ARG = 1,       /* a null pointer, a size out of range, an unknown enum, a
                                non-finite param                                         */
    FDLLM_ERR_ALIGN = 2,     /* logits base not 16-byte aligned or V*sizeof(dtype) % 16 */
    FDLLM_ERR_NONFINITE = 3, /* a selection met a row of FDLLM_ROW_NONFINITE (status word) */
    FDLLM_ERR_CUDA = 4,      /* a CUDA runtime call or kernel launch failed             */
    FDLLM_ERR_WORKSPACE = 5, /* caller workspace too small or misaligned                */
    FDLLM_ERR_DEVICE = 6     /* a kernel's bounded wait gave up (see fdllm_device_status) */
} fdllm_status;

/* out_n value of a batch row whose masked logits are unusable: a NaN anywhere in a masked
 * position's row, or a maximum of +inf or -inf.  Such a row commits nothing and its mask
 * is left unchanged; a call with a workspace also records it in the workspace's status word
 * (FDLLM_ERR_NONFINITE from the status calls).  (The paper defines confidences only for
 * proper distributions.) */
#define FDLLM_ROW_NONFINITE (-1)
/* out_n value of every row when a kernel of the step gave up a bounded wait. */
#define FDLLM_ROW_DEVICE_ERROR (-2)

/* ---------------------------------------------------------------------------------- */
/* One whole selection step (steps a1-a5 above; Alg. 1 from the model's logits to the
 * reveal), with a workspace the library owns.
 *
 *   logits      [B, L, V] device, dtype as given, read only at masked positions.
 *   mask        [B, L] uint8 device, nonzero = masked.  UPDATED IN PLACE: committed
 *               positions become 0 (Alg. 1 reveal).
 *   param       profile: f, the rule accepts n iff G_n > delta with delta = 1 - f (the
 *               matched parameter of Cor. factor-reduction; the paper's operating point
 *               delta = 0.25 is f = 0.75).  factor: f.  threshold: tau.  Any finite value
 *               is accepted; the paper states delta in [0, 1] (f in [0, 1]).
 *   out_tokens  [B, L] int32 device: written ONLY at committed positions, with x_hat.
 *   out_commit  [B, L] uint8 device: fully written, 1 = committed this step.
 *   out_n       [B] int32 device: number committed in each row; 0 iff the row had no
 *               masked position; FDLLM_ROW_NONFINITE / FDLLM_ROW_DEVICE_ERROR as above.
 *
 * The library's workspace is allocated on the current device at the first call that
 * needs more than it holds (cudaMalloc, which synchronises), then reused; make one call
 * of the largest shape before capturing the step in a CUDA graph.  Calls that share the
 * library workspace must be ordered on the GPU (one stream, or events); for concurrent
 * steps use fdllm_select_ws with a workspace per stream. */
fdllm_status fdllm_select(const void *logits, int dtype, int B, int L, int V, uint8_t *mask,
                          double param, int mode, int32_t *out_tokens, uint8_t *out_commit,
                          int32_t *out_n, void *stream);

/* Bytes of caller workspace fdllm_select_ws needs for this shape (a pure host function). */
size_t fdllm_workspace_bytes(int B, int L, int V, int dtype);

/* fdllm_select with a caller-provided workspace (device, 256-byte aligned, at least
 * fdllm_workspace_bytes(B, L, V, dtype) bytes).  The workspace must be zero-filled before
 * its first use; every call that completes leaves it ready for the next call, so it is
 * zeroed once, not per call.  The library never allocates on this path. */
fdllm_status fdllm_select_ws(const void *logits, int dtype, int B, int L, int V, uint8_t *mask,
                             double param, int mode, int32_t *out_tokens, uint8_t *out_commit,
                             int32_t *out_n, void *workspace, size_t workspace_bytes,
                             void *stream);

/* The profile rule on calibration-robust confidences (App. C, "Calibration-Robust Frechet
 * Certificates"): every masked confidence c_hat is replaced by the lower confidence
 * c_low = max{0, c_hat - eta_i} (Eq. robust_L_U), the masked positions are ranked by c_low
 * (ties: lower position first), L_eta(n) = max{0, sum_{j<=n} c_low_(j) - (n-1)},
 * U_eta(n) = 1 - c_low_(n), n is accepted iff L_eta(n) - U_eta(n) > delta = 1 - param, and
 * n* = max accepted, or 1 (the paper defines the robust certificate; this selection rule on
 * it is the library's reading).  With uniform eta and no clipping the score is the plain
 * one minus (n+1) eta (Cor. calibration-penalty).
 *   eta               uniform allowance, finite and >= 0 (App. C; otherwise FDLLM_ERR_ARG),
 *                     used when eta_per_position is NULL.
 *   eta_per_position  [B, L] fp32 device array of per-position allowances, or NULL; a
 *                     negative or NaN entry is read as 0 (device data: not checked on the
 *                     host).
 * Everything else as fdllm_select (the same library workspace).  eta = 0 gives exactly
 * fdllm_select's profile rule. */
fdllm_status fdllm_select_robust(const void *logits, int dtype, int B, int L, int V,
                                 uint8_t *mask, double param, double eta,
                                 const float *eta_per_position, int32_t *out_tokens,
                                 uint8_t *out_commit, int32_t *out_n, void *stream);

/* Scratch of fdllm_select_static: a fixed device array of this many bytes. */
#define FDLLM_STATIC_SCRATCH_BYTES (8u << 20)

/* fdllm_select without any allocation, for callers that must not allocate device memory
 * while they run steps: a serving process that reserves all of its memory up front and
 * forbids allocation afterwards, code running under an external allocator that owns the
 * device (a framework's memory pool, a fixed memory budget), or a caller that cannot hand
 * the library a workspace of its own.  (The paper has no counterpart: this is a property
 * of the library, not of the method.)
 *
 * Arguments and results are exactly those of fdllm_select.  The scratch memory is a fixed
 * array of FDLLM_STATIC_SCRATCH_BYTES bytes compiled into the library; every GPU that loads
 * the library holds it until the process exits.  A shape whose scratch need,
 * fdllm_workspace_bytes(B, L, V, dtype), exceeds that size is rejected with
 * FDLLM_ERR_WORKSPACE before anything is enqueued.  8 MiB covers, for example, every shape
 * with V <= 126464 in any dtype (up to B * L = 65536 rows), and fp32 V = 2^20 up to
 * B * L = 16383 rows.
 * The call allocates nothing: no cudaMalloc, no cudaFree, no allocating library routine.
 *
 * The first call on a device looks up the array's device address (cudaGetSymbolAddress)
 * with that device current and caches it; make that first call before any stream capture.
 * Every call clears the array's status word and work counter on `stream` before its
 * kernels run.  All calls on a device share the one array, which keeps the last call's
 * contents: calls whose work overlaps on the GPU (different streams without ordering
 * between them) race on it and produce wrong results; order such calls on one stream or
 * with events. */
fdllm_status fdllm_select_static(const void *logits, int dtype, int B, int L, int V,
                                 uint8_t *mask, double param, int mode, int32_t *out_tokens,
                                 uint8_t *out_commit, int32_t *out_n, void *stream);

/* The sticky device error of fdllm_select_static's array on the current device, as
 * fdllm_device_status reports the library workspace's: synchronises `stream`, returns
 * FDLLM_ERR_DEVICE if a kernel of a static call gave up a bounded wait (every row of that
 * call also reports out_n = -2), else FDLLM_ERR_NONFINITE if its selection found a row of
 * FDLLM_ROW_NONFINITE, FDLLM_OK otherwise, and clears the status.  Call it after a
 * static call and before the next one, which clears the array's status word itself.
 * Allocates nothing. */
fdllm_status fdllm_static_status(void *stream);

/* Step a1 alone (Sec. 3 "Notation"; Alg. 1 confidence loop): for every masked position,
 * out_conf = c = max softmax probability (fp32) and out_argmax = x_hat (int32, lowest index
 * among equal maxima).  Both [B, L] device arrays, written only at masked positions; a
 * row with non-finite logits (see FDLLM_ROW_NONFINITE) gets out_conf = NaN and
 * out_argmax = -1.  Uses the library workspace like fdllm_select. */
fdllm_status fdllm_confidence(const void *logits, int dtype, int B, int L, int V,
                              const uint8_t *mask, float *out_conf, int32_t *out_argmax,
                              void *stream);

/* Step a1's vocabulary reduction alone: the per-unit (max, sum of exp, first index)
 * partials of every masked position, written into the library workspace and not folded
 * into (c, x_hat).  One kernel.  Its use is timing the reduction kernel by itself (a CUDA
 * graph of these calls); arguments and errors as for fdllm_confidence. */
fdllm_status fdllm_vocab_reduce(const void *logits, int dtype, int B, int L, int V,
                                const uint8_t *mask, void *stream);

/* Steps a2-a5 alone (Alg. 1 sort, scan, select, reveal) on given confidences.
 *   conf    [B, L] fp32 device, read at masked positions; a masked value outside (0, 1]
 *           (NaN included) makes the row FDLLM_ROW_NONFINITE.
 *   argmax  [B, L] int32 device, the token revealed at each committed position.
 * mask, param, mode and the outputs as in fdllm_select.  Needs no workspace. */
fdllm_status fdllm_select_from_conf(const float *conf, const int32_t *argmax, int B, int L,
                                    uint8_t *mask, double param, int mode,
                                    int32_t *out_tokens, uint8_t *out_commit, int32_t *out_n,
                                    void *stream);

/* Input movement for the end-to-end path (the paper has no counterpart: it moves data, it
 * computes nothing): copies the rows of the masked positions of `src` [B, L, V] (dtype as
 * given) to the same offsets of `dst`, a device buffer of the same shape; rows of unmasked
 * positions of dst are not written.  src may be device memory or page-locked host memory
 * (cudaHostAlloc / torch pin_memory), which the GPU reads directly over the host link, so
 * that only the masked rows cross it.  mask [B, L] uint8 device.  Pageable host memory is
 * rejected (FDLLM_ERR_ARG); src and dst 16-byte aligned, V * sizeof(dtype) a multiple of 16
 * (FDLLM_ERR_ALIGN).  Asynchronous on `stream`. */
fdllm_status fdllm_gather_masked_rows(const void *src, void *dst, int dtype, int B, int L, int V,
                                      const uint8_t *mask, void *stream);

/* One selection step end to end on host buffers (Alg. 1's step as fdllm_select computes it;
 * this entry only moves data around it): the call a host program makes when its logits
 * are in host memory.  Arguments as in fdllm_select, except:
 *   logits  [B, L, V] in page-locked host memory (cudaHostAlloc / cudaHostRegister / torch
 *           pin_memory): the GPU reads the rows of masked positions over the host link and
 *           nothing else; pageable host memory is copied whole first (slower); device
 *           memory is read in place.  16-byte aligned.
 *   mask, out_tokens, out_commit, out_n  host (or device) arrays of fdllm_select's shapes;
 *           mask is updated in place and out_tokens keeps its values at positions not
 *           committed, as in fdllm_select.
 * The library copies mask and out_tokens to a device staging buffer of its own (per device,
 * grown on demand with cudaMalloc, released by fdllm_release_workspace), runs the step on
 * `stream` with the library workspace, copies out_tokens, out_commit, out_n and the mask
 * back and synchronises `stream` before it returns: the results are in place when the call
 * returns.  Argument errors are reported before anything is enqueued; the same device
 * errors as fdllm_select (fdllm_device_status).  Not for stream capture (it synchronises).
 * Calls share the staging buffer and the library workspace of their device: calls from
 * several host threads at once must be serialised by the caller.  The paper has no
 * counterpart. */
fdllm_status fdllm_select_host(const void *logits, int dtype, int B, int L, int V,
                               uint8_t *mask, double param, int mode, int32_t *out_tokens,
                               uint8_t *out_commit, int32_t *out_n, void *stream);

/* Step a1 fused with the LM head (the projection that produces the logits, Sec. 3
 * "Notation": p_i = softmax of the logits of position i), then steps a2-a5 as in
 * fdllm_select.  For every masked position the logits x = W h are computed on the tensor
 * cores (bf16 inputs, fp32 accumulation) and reduced to (c, x_hat) in the GEMM's epilogue:
 * the B*L*V logits are never written to memory.
 *   hidden   [B, L, H] bf16 device, the final hidden state of each position (read at masked
 *            positions only); 16-byte aligned.
 *   w_vocab  [V, H] bf16 device, the vocabulary projection, row v = the weights of token v;
 *            16-byte aligned.
 *   H        hidden size, a multiple of 8 (16-byte rows); V >= 1, any value.
 * mask, param, mode and the outputs as in fdllm_select (B*L <= FDLLM_MAX_ROWS, L <=
 * FDLLM_MAX_L).  Uses the library-owned workspace (at most B*L*(2H + 16*ceil(V/208) + 12)
 * bytes and a header), allocated outside the step as for fdllm_select.  Asynchronous on
 * `stream`.  The GEMM's tiling (row tiles of 128, CTA pairs, or vocabulary slabs for at most
 * 32 rows) is chosen from B*L and V; the environment variables FDLLM_LMHEAD_GEMM (solo,
 * pair, slab) and FDLLM_LMHEAD_BN (256, 208) force one, for measurements.
 * Results agree with fdllm_select applied to the fp32 logits fdllm_lmhead_logits writes
 * under the same tiling (the same tensor-core accumulation): tokens bit-exact, confidences
 * within 1e-5. */
fdllm_status fdllm_lmhead_select(const void *hidden, const void *w_vocab, int B, int L, int H,
                                 int V, uint8_t *mask, double param, int mode,
                                 int32_t *out_tokens, uint8_t *out_commit, int32_t *out_n,
                                 void *stream);

/* Step a1 alone on the LM head: out_conf (fp32) and out_argmax (int32), [B, L] device, written
 * at masked positions (NaN and -1 for a row whose logits hold a NaN or an infinite maximum).
 * Arguments as fdllm_lmhead_select. */
fdllm_status fdllm_lmhead_confidence(const void *hidden, const void *w_vocab, int B, int L,
                                     int H, int V, const uint8_t *mask, float *out_conf,
                                     int32_t *out_argmax, void *stream);

/* The same tensor-core GEMM with its accumulators stored instead of reduced: out_logits
 * [B, L, V] fp32 device, written at the masked positions' rows only (the unfused path, and
 * the exact inputs against which the fused reduction is checked). */
fdllm_status fdllm_lmhead_logits(const void *hidden, const void *w_vocab, int B, int L, int H,
                                 int V, const uint8_t *mask, float *out_logits, void *stream);

/* Model forward pass used by fdllm_decode_loop.  It must only enqueue stream-ordered GPU
 * work on `stream`: it is called while the loop body is being captured into a CUDA graph
 * (once, or twice when the driver rejects the first capture and the body is captured again
 * without programmatic dependent launches), and the captured work is replayed at every
 * step.  It must not synchronise or allocate.  It writes logits [B, block_len, V]
 * of the current block into `logits` for the rows with block_mask != 0.  loop_state is a
 * device pointer to two int32 values read at run time: [0] the global step (forward passes
 * so far), [1] the current block.  Return 0 on success. */
typedef int (*fdllm_forward_fn)(void *user, const int32_t *loop_state,
                                const uint8_t *block_mask, void *logits, void *stream);

/* Algorithm 1's outer loop on the GPU, with no host round trip per step: for each of
 * gen_len / block_len blocks, start with the block fully masked and repeat {forward pass;
 * selection with (mode, param) as in fdllm_select; reveal} while the block has masked
 * positions (Alg. 1: a block's steps go on until none of its positions is masked), then
 * move to the next block.
 * The loop is one CUDA graph with a conditional WHILE node; the forward pass, the two
 * selection kernels and a controller kernel form its body.
 *   logits          [B, block_len, V] device buffer the forward pass writes (dtype as given).
 *   seq_tokens      [B, gen_len] int32 device output: the committed tokens (-1 if none).
 *   nfe_per_block   [gen_len / block_len] int32 device output: steps (NFE) per block.
 *   max_steps       bound on the total number of steps; reaching it ends the loop early
 *                   and returns FDLLM_ERR_DEVICE.
 * A step whose selection reports a row as FDLLM_ROW_NONFINITE ends the loop after that
 * step with FDLLM_ERR_NONFINITE (such a row commits nothing, so its block would never
 * finish); a step that reports FDLLM_ROW_DEVICE_ERROR ends it with FDLLM_ERR_DEVICE.
 * nfe_per_block then holds the steps of the blocks reached and out_steps the steps taken.
 *   out_steps       host int: total steps taken.
 * Synchronous: returns when the generation is finished.  Allocates its own small buffers
 * and the library workspace (outside the graph).  Limits as fdllm_select with L = block_len;
 * modes FDLLM_PROFILE, FDLLM_FACTOR and FDLLM_THRESHOLD.  Errors: FDLLM_ERR_ARG for a bad
 * argument (checked before any device work) or a forward pass that returned nonzero;
 * FDLLM_ERR_CUDA for a failed graph build or launch.  Uses the library-owned workspace of
 * fdllm_select: no other selection may run on this device from another thread meanwhile.
 * Every step commits at least one position of each row that still has masked positions, so
 * each block ends after at most block_len steps. */
fdllm_status fdllm_decode_loop(int B, int gen_len, int block_len, int V, int dtype,
                               double param, int mode, fdllm_forward_fn forward, void *user,
                               void *logits, int32_t *seq_tokens, int32_t *nfe_per_block,
                               int max_steps, int *out_steps, void *stream);

/* fdllm_decode_loop with the LM head inside the loop body: the forward pass writes the final
 * hidden states [B, block_len, H] bf16 into `hidden` (rows with block_mask != 0), and each
 * step's selection is fdllm_lmhead_select against w_vocab [V, H] bf16 (the logits never
 * reach memory).  Arguments, limits and errors otherwise as fdllm_decode_loop and
 * fdllm_lmhead_select (H a multiple of 8; w_vocab NULL: FDLLM_ERR_ARG). */
fdllm_status fdllm_decode_loop_lmhead(int B, int gen_len, int block_len, int H, int V,
                                      const void *w_vocab, double param, int mode,
                                      fdllm_forward_fn forward, void *user, void *hidden,
                                      int32_t *seq_tokens, int32_t *nfe_per_block, int max_steps,
                                      int *out_steps, void *stream);

/* Heterogeneity-bonus diagnostics (Prop. heterogeneity-bonus, Eq. heterogeneity_decomp,
 * Remark adaptive-factor).  For each batch row, the masked confidences are sorted as the
 * selection sorts them (descending, ties: lower position first); at rank n = 1..m_b:
 *   out_G[b, n-1]     = G_n = max{0, sum_{j<=n} c_(j) - (n-1)} - (1 - c_(n))
 *   out_F[b, n-1]     = F_n = (n+1) c_(n) - n                (factor core)
 *   out_B[b, n-1]     = B_n = sum_{j<n} (c_(j) - c_(n))       (heterogeneity bonus)
 *   out_feff[b, n-1]  = f_eff(n) = 1 - delta + B_n           (Remark adaptive-factor)
 *   out_order[b, n-1] = the position holding c_(n)
 * Ranks n > m_b get NaN (order -1).  G_n = F_n + B_n wherever the lower bound is positive,
 * so the profile rule with margin delta behaves as the factor rule with the effective
 * factor f_eff(n).
 *   conf   [B, L] fp32 device (e.g. from fdllm_confidence), read at masked positions:
 *          values in [0, 1], or NaN (a NaN ranks after every number, so the terms of its
 *          rank and of every later rank are NaN); other values give unspecified terms.
 *   mask   [B, L] uint8 device, nonzero = masked (not modified).
 *   delta  the profile rule's margin (delta = 1 - param of fdllm_select), finite.
 *   out_G, out_F, out_B, out_feff  [B, L] fp64 device, each nullable; out_order [B, L]
 *   int32, nullable.
 * Asynchronous on `stream`; needs no workspace. */
fdllm_status fdllm_profile_terms(const float *conf, const uint8_t *mask, int B, int L,
                                 double delta, double *out_G, double *out_F, double *out_B,
                                 double *out_feff, int32_t *out_order, void *stream);

/* Health check of the library's failure detection: every wait inside the kernels is
 * bounded, and a wait that runs out records a device error and lets the kernel return
 * instead of hanging.  This launches one thread that waits on a barrier nobody completes,
 * with a limit of `seconds` (0 < seconds <= 10), synchronises `stream` and returns
 * FDLLM_ERR_DEVICE when the wait ran out and was reported as it should (FDLLM_OK would mean
 * the wait did not run out).  The device stays usable afterwards.  The paper has no
 * counterpart. */
fdllm_status fdllm_check_bounded_wait(double seconds, void *stream);

/* Synchronises `stream`, then reports (and clears) the sticky device error of the library
 * workspace on the current device: FDLLM_ERR_DEVICE if a kernel gave up a bounded wait
 * since the last call, else FDLLM_ERR_NONFINITE if a selection since the last call found a
 * row of FDLLM_ROW_NONFINITE, FDLLM_OK otherwise.  For fdllm_select_ws, pass the workspace to
 * fdllm_workspace_status instead.  Clearing an error also resets the workspace's work
 * counter, which a launch that gave up may have left mid-queue, so that the next call
 * starts from a clean header. */
fdllm_status fdllm_device_status(void *stream);
fdllm_status fdllm_workspace_status(void *workspace, void *stream);

/* Frees the library workspace of the current device (synchronises the device). */
void fdllm_release_workspace(void);

/* A static English description of a status code. */
const char *fdllm_status_string(int status);

/* Library version, major * 10000 + minor * 100 + patch. */
int fdllm_version(void);

#ifdef __cplusplus
}
#endif

#endif /* FDLLM_H */
