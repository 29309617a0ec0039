/*
 * xcache.h -- C ABI of the X-Cache chunk step on one GB300 (sm_103a).
 *
 * X-Cache (arXiv 2604.20289) accelerates autoregressive (AR) video-diffusion
 * inference: chunk n of latent video starts from noise and is refined by S
 * denoising passes, each through all B DiT blocks (Section 2.1, Eq. 1); a KV-update
 * pass on the clean latent then writes keys/values into a rolling KV cache
 * (Section 2.1).  X-Cache keeps, for every (denoising step t, block b), the
 * residual the block added the last time it computed (Eq. 2-3) and reuses it
 * (Eq. 4) when a dual-metric gate (Eq. 5-7, adaptive threshold Eq. 8-9) finds
 * the block input close to the cached fingerprint (Section 2.3).
 *
 * One xc_chunk_step call runs ONE forward pass (a denoising pass t or the
 * KV-update pass) over all blocks; the gate decisions stay on the device.
 *
 * Conventions
 *  - All calls return xc_status; no exception crosses the ABI.  On error the
 *    context state is unchanged and xc_last_error() describes the failure.
 *  - Work is asynchronous on the stream given to xc_init (a cudaStream_t,
 *    NULL = legacy default stream) unless a call says otherwise.
 *  - Pointers marked "host or device" are classified with
 *    cudaPointerGetAttributes; host buffers are staged through the context
 *    and a call given a host buffer synchronises with its stream before it
 *    returns, so the caller may reuse or read that buffer immediately.
 *  - The context owns its copies of the weights, the KV ring, the residual
 *    and fingerprint caches and all scratch; callers own every buffer they pass.
 */
#ifndef XCACHE_H
#define XCACHE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define XC_MAX_BLOCKS 64
#define XC_MAX_GROUPS 4

typedef enum {
    XC_OK = 0,
    XC_EINVAL = 1,     /* bad argument, shape or configuration */
    XC_ESTATE = 2,     /* call out of order (step index, KV pass) or no context */
    XC_ENOMEM = 3,     /* device or pinned-host allocation failed */
    XC_ECUDA = 4,      /* a CUDA runtime / driver call failed */
    XC_ENUMERIC = 5,   /* non-finite value in an input */
    XC_ETIMEOUT = 6    /* a kernel's bounded wait expired (device error word set) */
} xc_status;

typedef enum { XC_F32 = 0, XC_BF16 = 1 } xc_dtype;

/* Per-block decision of one pass (stats.decision). */
typedef enum {
    XC_DEC_FORCED = 0,   /* computed without evaluating the gate (KV pass, warmup,
                            anchor, step-0 protection, gating off, empty cache)   */
    XC_DEC_COMPUTE = 1,  /* gate evaluated: recompute                             */
    XC_DEC_SKIP = 2      /* gate evaluated: reuse x + r_hat (Eq. 4)               */
} xc_decision;

/* Model shape (Section 2.1; block internals are this library's reading of the
 * WAN-style DiT the paper builds on, Section 3.1.2).  A chunk holds
 * L = n_cams*frames*grid_h*grid_w tokens in (camera, frame, h, w) row-major
 * order.  kv_window_chunks counts ring slots INCLUDING the current chunk.
 * Constraints: d_model = n_heads*head_dim; head_dim % 16 == 0; for XC_BF16
 * head_dim in {64, 128}, d_model % 256 == 0 and d_ffn % 256 == 0;
 * n_blocks <= XC_MAX_BLOCKS; t_freq_dim even and <= 512.
 *
 * View groups (Section 2.3.1): with n_groups = 0 all cameras share the grid
 * (grid_h, grid_w).  With 1 <= n_groups <= XC_MAX_GROUPS, group g holds
 * group_cams[g] cameras of grid (group_h[g], group_w[g]); the groups' tokens
 * follow one another in group order (each group camera by camera, then
 * (frame, h, w) row-major), n_cams must equal the sum of group_cams, the
 * RoPE camera coordinate counts on across groups, and grid_h / grid_w are not
 * used.  The gate keeps one spatial and one global fingerprint entry per group.
 *
 * kv_period (Section 2.5 (3)): 0 = every chunk ends with a KV-update pass, the
 * only pass forced to compute every block.  P > 0 = only chunks n with
 * n mod P == P - 1 have a KV-update pass; their denoising passes run in
 * force-compute mode (every block computes, the gate is not evaluated, the
 * residual and fingerprint caches are refreshed), and a chunk without one
 * ends after its last denoising pass.  The ring then holds the clean K/V of
 * the last kv_window_chunks - 1 KV-update chunks.
 *
 * Cross-attention conditioning (condition tokens such as dynamic objects,
 * lanes and text, Sections 2.1 and 2.5): with d_ctx > 0 every block gets a
 * cross-attention layer between its self-attention and its FFN,
 *   x1 <- x1 + softmax(q K_c^T / sqrt(head_dim)) V_c W_o + b_o,
 *   q = (LN(x1) * gamma + beta) W_q + b_q,  [K_c | V_c] = C W_kv + b_kv,
 * over the up to max_ctx condition tokens C [n_ctx][d_ctx] given by
 * xc_set_context (no modulation, no gate, no RoPE).  XC_BF16 needs
 * d_ctx % 64 == 0, XC_F32 d_ctx % 16 == 0.  d_ctx = 0: no cross-attention. */
typedef struct {
    int n_blocks, d_model, n_heads, head_dim, d_ffn, c_latent, action_dim;
    int n_cams, frames, grid_h, grid_w;
    int kv_window_chunks, n_denoise_steps, dtype, t_freq_dim;
    float ln_eps, rope_theta;
    int kv_period;
    int n_groups;
    int group_cams[XC_MAX_GROUPS], group_h[XC_MAX_GROUPS], group_w[XC_MAX_GROUPS];
    int d_ctx, max_ctx;
} xc_model_cfg;

/* Float32 weights, host or device pointers (each classified on its own),
 * math convention y = x @ W with W stored [in][out] row-major.  For XC_BF16
 * models the values are rounded to bf16 on upload.
 * Shapes (d = d_model, F = d_ffn, B = n_blocks, C = c_latent, A = action_dim,
 * T = t_freq_dim):
 *   pe_w [C][d] pe_b [d]                 patch embedding
 *   t_w1 [T][d] t_b1 [d] t_w2 [d][d] t_b2 [d]   timestep MLP
 *   a_w1 [A][d] a_b1 [d] a_w2 [d][d] a_b2 [d]   action MLP
 *   mod_w [d][6d] mod_b [6d]  blk_mod [B][6][d]   adaLN-Zero (shift1, scale1,
 *                                                 gate1, shift2, scale2, gate2)
 *   qkv_w [B][d][3d] qkv_b [B][3d]  o_w [B][d][d] o_b [B][d]
 *   f1_w [B][d][F] f1_b [B][F]      f2_w [B][F][d] f2_b [B][d]
 *   head_w [d][2d] head_b [2d] head_tab [2][d]    head (shift, scale)
 *   out_w [d][C] out_b [C]
 * Cross-attention (d_ctx > 0 only, else ignored; D = d_ctx):
 *   ca_ln_w [B][d] ca_ln_b [B][d]   LN gain gamma and bias beta
 *   ca_q_w [B][d][d] ca_q_b [B][d]  ca_kv_w [B][D][2d] ca_kv_b [B][2d]
 *   ca_o_w [B][d][d] ca_o_b [B][d]
 * The pointers are only read during xc_init; device weights never pass
 * through host memory. */
typedef struct {
    const float *pe_w, *pe_b, *t_w1, *t_b1, *t_w2, *t_b2, *a_w1, *a_b1, *a_w2, *a_b2;
    const float *mod_w, *mod_b, *blk_mod;
    const float *qkv_w, *qkv_b, *o_w, *o_b, *f1_w, *f1_b, *f2_w, *f2_b;
    const float *head_w, *head_b, *head_tab, *out_w, *out_b;
    const float *ca_ln_w, *ca_ln_b, *ca_q_w, *ca_q_b, *ca_kv_w, *ca_kv_b, *ca_o_w, *ca_o_b;
} xc_weights;

/* Gate knobs (Section 2.3-2.5); xc_gate_params_default() gives Table 1:
 * F_n = 1, B_n = 0, W = 1, tau_floor = 0.97, m = 0.02, alpha = 0.30,
 * tau_dev = 2.0, M = off, step-0 protection off, K = 32 fingerprint tokens.
 * KV-update protection is always on: the KV pass never evaluates the gate.
 *   fp_refresh  0: cached fingerprint refreshed when the block computes;
 *               1: refreshed on every evaluation.
 *   fp_linear   0: spatial sample on the 3-D (frame, h, w) grid of each view
 *               group; 1: the 1-D fallback -- fp_tokens uniformly spaced,
 *               cell-centred indices along each camera's token axis
 *               (Section 2.3.1).  Changing fp_tokens or fp_linear between calls
 *               rebuilds the sample and clears every gate cell.
 *   chain       0: a skipped block writes x + r_hat at once (Eq. 4);
 *               1: lazy residual chaining -- a run of skipped blocks writes
 *               nothing; the gate of the next block takes the fingerprint of
 *               the chained input from the sampled rows and the cached
 *               residuals' per-camera means, and the input is written only
 *               before a block that computes (or the head), as the last
 *               written activation plus the run's residuals summed in fp32 in
 *               block order and rounded once.  Switching chaining on clears
 *               every gate cell; with a block trace set, passes do not chain.
 *   replay_skip host [n_blocks] or NULL: decision-replay mode -- for blocks the
 *               gate evaluates, the decision is replay_skip[b] != 0 instead of
 *               Eq. 7 (metrics, EMA and staleness are still updated).
 *   replay_table device uint8 [n_denoise_steps][n_blocks] or NULL: the same
 *               replay, read by the gate on the device from entry (t, b) when
 *               the pass runs (takes precedence over replay_skip), so a
 *               whole chunk's decisions can be set once without host copies.
 *               The caller keeps the table alive and unchanged until the
 *               passes that read it have completed. */
typedef struct {
    int enabled;
    float tau_floor, margin, alpha, tau_dev, eps_dev;
    int front_anchors, back_anchors, warmup_chunks, max_skips;
    int protect_step0;
    float step0_strict_tau;
    int fp_tokens, fp_refresh, fp_linear;
    int chain;
    const uint8_t *replay_skip;
    const uint8_t *replay_table;
} xc_gate_params;

/* Filled by xc_chunk_step when non-NULL (the call then synchronises with its
 * stream).  Metrics are NaN for blocks whose gate was not evaluated. */
typedef struct {
    int n_blocks;
    int chunk_index;          /* n of the pass just run */
    uint8_t decision[XC_MAX_BLOCKS];
    float s_cos[XC_MAX_BLOCKS];   /* Eq. 5, min over entries */
    float d_max[XC_MAX_BLOCKS];   /* Eq. 6 */
    float tau_cos[XC_MAX_BLOCKS]; /* Eq. 9 threshold used */
} xc_step_stats;

typedef struct xc_ctx xc_ctx;

/* Table 1 defaults.  p must be non-NULL. */
void xc_gate_params_default(xc_gate_params *p);

/* Validates cfg, allocates the context on the current CUDA device and uploads
 * the weights.  `cuda_stream` is a cudaStream_t (may be NULL).  On success
 * *out owns all device state; free it with xc_destroy.
 * Errors: XC_EINVAL (cfg/weights), XC_ENOMEM, XC_ECUDA. */
xc_status xc_init(const xc_model_cfg *cfg, const xc_weights *w, void *cuda_stream,
                  xc_ctx **out);

/* One forward pass of chunk n (the context's chunk counter).
 *   latent  host or device float32 [L][c_latent]: x at sigma (denoising pass)
 *           or the clean latent (KV-update pass, sigma = 0).
 *   action  host float32 [action_dim]: the chunk's action (condition channel,
 *           Section 2.3.2; adaLN-Zero conditioning).
 *   step_index  t in [0, n_denoise_steps) for a denoising pass; ignored when
 *           is_kv_update != 0.  Passes of a chunk must come in order
 *           t = 0..S-1, then the KV-update pass (which may also come alone at
 *           the start of a chunk); otherwise XC_ESTATE.  With kv_period P > 0
 *           a chunk without a KV-update pass (n mod P != P - 1) ends after
 *           pass S-1 and a KV-update call on it returns XC_ESTATE.
 *   is_kv_update  the KV-update pass: every block computes (KV-update
 *           protection, Section 2.5 (3)), clean K/V go to ring slot
 *           k mod kv_window_chunks (k = KV-update passes so far; k = n when
 *           kv_period = 0), and the chunk counter advances.
 *   gate    NULL = Table 1 defaults.
 *   v_out   host or device float32 [L][c_latent] velocity, or NULL.  A
 *           KV-update pass with v_out NULL (and no block trace set) computes
 *           only what the ring needs: the last block stops after its K/V
 *           projection and the output head is not run.
 *   stats   NULL or filled as documented above (synchronising).
 * Execution: the conditioning and the chunk's RoPE table are launched
 * directly; the rest of the pass (patch embedding, every block, the head)
 * is captured into a CUDA graph the first time its host inputs (pass index,
 * ring slot and fill, gate parameters and replay bits, latent / v_out /
 * trace pointers) occur, and replayed whenever they recur.  Gate decisions
 * stay on the device, so one graph serves every decision pattern.  While
 * profiling (xc_profile_start) passes are launched directly.
 * Errors: XC_EINVAL, XC_ESTATE, XC_ECUDA, XC_ETIMEOUT (device wait expired). */
xc_status xc_chunk_step(xc_ctx *ctx, const float *latent, const float *action, float sigma,
                        int step_index, int is_kv_update, const xc_gate_params *gate,
                        float *v_out, xc_step_stats *stats);

/* Condition tokens for the following passes (cross-attention models):
 * context host or device float32 [n_ctx][d_ctx], 1 <= n_ctx <= max_ctx.
 * Computes every block's condition keys and values on the context's stream;
 * the tokens stay in use until the next call (and across xc_reset).  Passes
 * of a cross-attention model before the first call return XC_ESTATE.
 * Errors: XC_EINVAL (no cross-attention, bad n_ctx or NULL), XC_ENUMERIC
 * (non-finite host value), XC_ECUDA. */
xc_status xc_set_context(xc_ctx *ctx, const float *context, int n_ctx);

/* Clears the KV ring, residual / fingerprint caches, EMA, staleness and the
 * chunk counter (the next chunk is a warmup chunk again, Section 2.2.3).
 * Weights and condition tokens are kept. */
xc_status xc_reset(xc_ctx *ctx);

/* Frees everything the context owns.  NULL is a no-op. */
void xc_destroy(xc_ctx *ctx);

/* Message of the last failing call on ctx (or of the last failing call that
 * had no context when ctx is NULL).  Never NULL. */
const char *xc_last_error(const xc_ctx *ctx);

/* Euler step of the flow-matching sampler (driver side of Section 2.1):
 * x[i] += dsigma * v[i] for i < n, float32, device pointers, on ctx's stream. */
xc_status xc_euler_update(xc_ctx *ctx, float *x, const float *v, float dsigma, long n);

/* Debug trace: when dev_buf != NULL every following pass copies each block's
 * output x_{t,b} into dev_buf + b*L*d (activation dtype: float32 or bf16).
 * NULL switches the trace off. */
xc_status xc_set_block_trace(xc_ctx *ctx, void *dev_buf);

/* Blocks until the context's stream is idle, then reports a device-side
 * error word (bounded-wait timeouts) as XC_ETIMEOUT. */
xc_status xc_sync(xc_ctx *ctx);

/* Chunk counter n (chunks completed since reset). */
int xc_chunk_index(const xc_ctx *ctx);

/* ---- measurement (no counterpart in the paper; used by the benchmark) ---- */

/* Kernel kinds of one forward pass (XC_K_XATTN: the four launches of a
 * cross-attention layer -- LN, q projection, attention, output projection;
 * XC_K_CHAIN: lazy chaining -- the per-camera means of a new cached
 * residual and the write of a chained input). */
typedef enum {
    XC_K_COND = 0, XC_K_EMBED, XC_K_GATE, XC_K_LN, XC_K_QKV, XC_K_ATTN, XC_K_OPROJ,
    XC_K_FFN1, XC_K_FFN2, XC_K_REUSE, XC_K_HEAD, XC_K_XATTN, XC_K_CHAIN, XC_K_COUNT
} xc_kernel_kind;

/* One timed launch: CUDA-event duration on the context's stream, the block
 * and pass it belongs to, the gate decision of that block in that pass
 * (xc_decision; kernels of a skipped block exit at once), the chunk index
 * and the number of resident keys the pass attended to (condition tokens
 * for XC_K_XATTN). */
typedef struct {
    int kind, block, pass_seq, decision, chunk, n_keys;
    float ms;
} xc_profile_rec;

/* Starts recording events around every launch whose kind bit is set in
 * kind_mask (1 << xc_kernel_kind), for at most `capacity` launches; resets
 * the pass sequence.  Errors: XC_EINVAL (capacity < 1), XC_ENOMEM. */
xc_status xc_profile_start(xc_ctx *ctx, unsigned kind_mask, int capacity);

/* Stops recording, synchronises and copies up to `max` records to `out`
 * (host); *n_out receives the number recorded.  Frees the events. */
xc_status xc_profile_stop(xc_ctx *ctx, xc_profile_rec *out, int max, int *n_out);

/* Number of kernel launches this context has issued since xc_init
 * (including early-exit launches of skipped blocks). */
long long xc_launch_count(const xc_ctx *ctx);

/* ---- testing hook (no counterpart in the paper) ----
 * With n > 0 the n-th device allocation made by the library from now on
 * (xc_init's weights, ring, caches and scratch; a rebuilt fingerprint
 * sample) fails as if the device were out of memory: the call reports
 * XC_ENOMEM and releases everything it had allocated.  n <= 0 switches the
 * hook off.  Process-wide; for tests of the error paths. */
void xc_debug_fail_alloc(int n);

/* Runs out one bounded device wait on purpose: a one-thread kernel waits on
 * a barrier phase that nothing completes, gives up after the library's wait
 * limit (2 s), records the expiry in the error word of ctx (NULL: the error
 * word of the operator entry points) and returns -- the path every bounded
 * wait of the library takes on expiry.  xc_sync(ctx) then reports
 * XC_ETIMEOUT (xc_op_device_error() a non-zero word) and clears it; the
 * context stays usable.  For tests of that path. */
xc_status xc_debug_expire_wait(xc_ctx *ctx);

#ifdef __cplusplus
}
#endif
#endif /* XCACHE_H */
