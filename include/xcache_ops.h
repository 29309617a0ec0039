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
 * keys).  q, o [Lq][H*hd]; k, v [n_keys][H*hd]. */
xc_status xc_op_attention(int dtype, int Lq, int n_keys, int n_heads, int head_dim,
                          const void *q, const void *k, const void *v, void *o,
                          void *stream);

/* out = LayerNorm(x) * (1 + scale) + shift over rows of length d (no affine,
 * population variance, eps), adaLN-Zero modulation.  x, out [M][d]. */
xc_status xc_op_ln_mod(int dtype, int M, int d, float eps, const void *x,
                       const float *shift, const float *scale, void *out, void *stream);

/* Reuse path of Eq. 4: out = round(x + rhat), n elements. */
xc_status xc_op_residual_reuse(int dtype, long n, const void *x, const void *rhat, void *out,
                               void *stream);

/* Reads and clears the process-wide device error word of operator calls
 * (synchronising).  0 = no error. */
int xc_op_device_error(void);

#ifdef __cplusplus
}
#endif
#endif /* XCACHE_OPS_H */
