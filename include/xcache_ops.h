/*
 * xcache_ops.h -- operator-level entry points of the X-Cache hot path.
 *
 * These run ONE kernel of the chunk step on caller-owned device buffers, so
 * that each step of the path can be checked against the CPU oracle at full
 * size.  xc_chunk_step runs exactly these kernels.  All pointers are DEVICE
 * pointers; `stream` is a cudaStream_t (NULL = legacy default stream);
 * every call is asynchronous.  Activations use `dtype` (XC_F32: float32,
 * XC_BF16: bfloat16); vectors such as bias / gate / shift / scale are float32.
 * Weights are K-major: Wt [N][K] holds W^T of y = x W.
 * Errors: XC_EINVAL for a bad shape or pointer, XC_ECUDA for a launch
 * failure.  Kernels with bounded waits record expiry in a device error word
 * that xc_op_device_error() returns.
 */
#ifndef XCACHE_OPS_H
#define XCACHE_OPS_H

#include "xcache.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    XC_EPI_BIAS = 0,        /* out = A W + b                                     */
    XC_EPI_GELU = 1,        /* out = GELU_tanh(A W + b)  (FFN up-projection)     */
    XC_EPI_RESID_GATE = 2,  /* out = resid + gate * (A W + b)  (adaLN-Zero gated
                               residual of Eq. 1; O-projection / FFN down)       */
    XC_EPI_RESID_CACHE = 3  /* as XC_EPI_RESID_GATE and additionally
                               rhat = round(out) - xin (block residual, Eq. 2-3) */
} xc_epilogue;

/* C[M][N] = epilogue(A[M][K] @ Wt[N][K]^T).  M >= 1; N % 256 == 0 and K % 64 == 0
 * for XC_BF16 (tcgen05 path), N % 16 == 0 for XC_F32.  `gate`, `resid`,
 * `xin`, `rhat` may be NULL when the epilogue does not use them. */
xc_status xc_op_linear(int dtype, int epilogue, int M, int N, int K, const void *A,
                       const void *Wt, const float *bias, const float *gate,
                       const void *resid, const void *xin, void *out, void *rhat,
                       void *stream);

/* QKV projection with RoPE (Section 2.1 block, reading of RoPE over
 * (camera, absolute frame, h, w)).  A [M][d] with M = n_cams*frames*gh*gw,
 * Wt [3d][d], bias [3d]; writes q, k, v [M][d] (heads interleaved by column:
 * head h owns columns h*head_dim ...).  Token row r of chunk `chunk` sits at
 * camera r / (frames*gh*gw), absolute frame chunk*frames + f, grid (h, w). */
xc_status xc_op_qkv_rope(int dtype, int n_cams, int frames, int gh, int gw, int chunk,
                         int d, int head_dim, float rope_theta, const void *A,
                         const void *Wt, const float *bias, void *q, void *k, void *v,
                         void *stream);

/* o = softmax(q k^T / sqrt(head_dim)) v per head, no mask (every query sees
 * every key: full attention within the chunk and over all resident cached
 * keys).  q, o [Lq][H*hd]; k, v [n_keys][H*hd] (bf16: 16-byte aligned rows).
 *   workspace  device, optional.  With at least
 *              xc_op_attention_workspace_bytes() bytes and more (head,
 *              256-query) units than SMs, the work is spread evenly over the
 *              SMs: either the (unit, key tile) space is cut into equal
 *              shares, or -- with 8 or more waves of units and the K / V of
 *              all heads larger than L2 -- whole units run in waves and only
 *              the remaining units are cut; a second kernel merges the
 *              partials of the cut units.  With NULL (or too small) every
 *              unit runs whole on one SM.  Contents on entry are ignored; it
 *              must not be shared by calls that overlap in time.
 * bf16 needs head_dim 64 or 128; fp32 head_dim 16, 32 or 64. */
size_t xc_op_attention_workspace_bytes(int dtype, int head_dim);
xc_status xc_op_attention(int dtype, int Lq, int n_keys, int n_heads, int head_dim,
                          const void *q, const void *k, const void *v, void *o,
                          void *workspace, size_t workspace_bytes, void *stream);

/* out = LayerNorm(x) * (1 + scale) + shift over rows of length d (no affine,
 * population variance, eps), adaLN-Zero modulation.  x, out [M][d]. */
xc_status xc_op_ln_mod(int dtype, int M, int d, float eps, const void *x,
                       const float *shift, const float *scale, void *out, void *stream);

/* Reuse path of Eq. 4: out = round(x + rhat), n elements. */
xc_status xc_op_residual_reuse(int dtype, long n, const void *x, const void *rhat, void *out,
                               void *stream);

/* Per-(t, b) gate state kept on the device (32 bytes): EMA of the cosine
 * (Eq. 8), has-history bit, consecutive-skip counter (Section 2.5 (4)),
 * cache-valid bit, and which half of the double-buffered cached fingerprint
 * is active. */
typedef struct {
    double ema;
    int has_hist, stale, valid, active;
    int pad[2];
} xc_gate_cell;

/* Bytes of device workspace xc_op_gate needs for this geometry on the current
 * device (the gate's grid splits each camera's rows over the device's SMs). */
size_t xc_op_gate_workspace_bytes(int dtype, int n_cams, int tokens_per_cam, int d);

/* One gate evaluation of one (t, b) cell (Section 2.3-2.5): fingerprint of the
 * block input x (spatial sample, per-camera token mean, action), min-cosine
 * s_cos (Eq. 5) and max token deviation d_max (Eq. 6) against the cached
 * fingerprint, adaptive threshold (Eq. 9), decision (Eq. 7), EMA (Eq. 8) and
 * staleness updates.
 *   x        device [n_cams * tokens_per_cam][d] activation dtype
 *   fp_rows  device int [n_cams][kfp]: token rows of the spatial sample
 *   phi      device float [2][n_cams*kfp*d + n_cams*d]: the two halves of the
 *            cached fingerprint (spatial entries, then per-camera means); the
 *            current fingerprint is written into the inactive half
 *   phi_act  device float [2][8]: cached action halves
 *   cell     device xc_gate_cell, updated in place
 *   action   host float [action_dim] (action_dim <= 8)
 *   mode     1 evaluate the gate, 0 refresh only (forced compute)
 *   step     denoising step t (strict step-0 threshold)
 *   gate     knobs (NULL = Table 1); replay_skip[0], when set, replaces the
 *            decision (decision-replay mode)
 *   flag     device uint8 decision (xc_decision); s_cos, d_max, tau device float
 *   workspace device, >= xc_op_gate_workspace_bytes(); its counters are
 *            cleared by the call (cudaMemsetAsync), nothing is allocated
 * Asynchronous on `stream`.  Errors: XC_EINVAL. */
xc_status xc_op_gate(int dtype, int n_cams, int tokens_per_cam, int d, const void *x, const int *fp_rows,
                     int kfp, float *phi, float *phi_act, xc_gate_cell *cell, const float *action,
                     int action_dim, int mode, int step, const xc_gate_params *gate, uint8_t *flag,
                     float *s_cos, float *d_max, float *tau, void *workspace, size_t workspace_bytes,
                     void *stream);

/* Allocation-free variant of xc_op_gate.  The paper has no counterpart; this
 * is an interface of this library, for callers that cannot call cudaMalloc
 * when they call in: a runtime that owns the only device allocator of the
 * process (a plugin or embedding host), code held to a device-memory budget
 * fixed at start-up, or a latency-critical loop where an allocation and the
 * device synchronisation it may bring are not acceptable.
 * Same arguments, checks and results as xc_op_gate minus the workspace: the
 * gate's scratch (per-CTA partial metrics and column sums, and the tickets)
 * lives in one file-scope device array of 1 MiB (GATE_STATIC_SCRATCH_BYTES)
 * that every GPU which loads the library keeps until the process exits.
 * Nothing is allocated or freed; the tickets are cleared with
 * cudaMemsetAsync on each call.
 * The first call on a device looks up the array's device address
 * (cudaGetSymbolAddress) and caches it for that device for the rest of the
 * process; that first call should come before any stream capture.  The
 * cached address belongs to the device's primary context: do not use this
 * entry point after cudaDeviceReset() on that device, or from a context other
 * than the primary one.
 * All calls share the one array and it keeps the last call's contents:
 * calls that overlap on the GPU (different streams, no ordering) race; calls
 * ordered on one stream are safe.
 * Errors: XC_EINVAL for bad arguments (as xc_op_gate) or a geometry whose
 * scratch exceeds 1 MiB (the message states the bytes needed), XC_ECUDA if
 * the device or the array's address cannot be obtained. */
xc_status xc_op_gate_static(int dtype, int n_cams, int tokens_per_cam, int d, const void *x,
                            const int *fp_rows, int kfp, float *phi, float *phi_act, xc_gate_cell *cell,
                            const float *action, int action_dim, int mode, int step,
                            const xc_gate_params *gate, uint8_t *flag, float *s_cos, float *d_max,
                            float *tau, void *stream);

/* Reads and clears the process-wide device error word of operator calls
 * (synchronising).  0 = no error. */
int xc_op_device_error(void);

#ifdef __cplusplus
}
#endif
#endif /* XCACHE_OPS_H */
