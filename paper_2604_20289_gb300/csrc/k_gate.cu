// Fused X-Cache gate of one (denoising step t, block b): fingerprint of the
// block input, both gating metrics against the cached fingerprint, adaptive
// threshold and the skip / recompute flag -- all on the device.
//
// Fingerprint (Section 2.3.1-2.3.2), one view group of V cameras:
//   spatial entry  x at the K-token 3-D grid sample of every camera  [V, k, d]
//   global channel per-camera mean of x over its tokens                 [V, d]
//   condition      the chunk's action vector                            [A]
// Metrics: s_cos = min over entries of the cosine (Eq. 5); d_max = max|cur -
// prev| / (mean|prev| + eps) over the spatial entry (Eq. 6).  Decision Eq. 7
// with tau_cos = max(tau_floor, ema - m) (Eq. 9), EMA update (Eq. 8) and the
// consecutive-skip cap (Section 2.5 (4)).
//
// Grid: one CTA per (camera c, 64-column slice s, row split r).  Each CTA
// streams its rows once (16-byte loads) for the column sums of the global
// channel and picks out the spatial-sample rows that fall in its range.
// Reduction without any spin-wait: the last CTA of each (c, s) (atomic
// ticket) finishes that slice's means; the last slice finisher makes the
// decision in fp64.  Partial results are combined in a fixed order, so the
// decision is deterministic.  The cached fingerprint is double-buffered per
// (t, b): the current fingerprint is written to the inactive half, which
// becomes active when the block recomputes (refresh on compute).
#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "xc_kernels.cuh"

namespace xc {

constexpr int GATE_CW = 64;
constexpr int GATE_THREADS = 256;

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ double warp_max_d(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmax(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Deterministic block reduction of N values per thread (op 0 = sum, 1 = max);
// result valid in thread 0.
template <int N>
__device__ __forceinline__ void block_reduce(double (&v)[N], const int (&op)[N], double (*sh)[N]) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int k = 0; k < N; ++k) v[k] = op[k] ? warp_max_d(v[k]) : warp_sum_d(v[k]);
    if (lane == 0) {
#pragma unroll
        for (int k = 0; k < N; ++k) sh[warp][k] = v[k];
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < GATE_THREADS / 32; ++w) {
#pragma unroll
            for (int k = 0; k < N; ++k) v[k] = op[k] ? fmax(v[k], sh[w][k]) : v[k] + sh[w][k];
        }
    }
    __syncthreads();
}

// Cosine of one entry from its dot product and squared norms (Eq. 5):
// both norms < 1e-12 -> 1, exactly one -> 0, NaN -> 0.
__device__ __forceinline__ double cos_rule(double dot, double n1sq, double n2sq) {
    const double a = sqrt(n1sq), b = sqrt(n2sq);
    if (isnan(a) || isnan(b) || isnan(dot)) return 0.0;
    if (a < 1e-12 && b < 1e-12) return 1.0;
    if (a < 1e-12 || b < 1e-12) return 0.0;
    return dot / (a * b);
}

template <typename T>
__global__ void __launch_bounds__(GATE_THREADS) gate_kernel(const GateArgs g) {
    constexpr int VEC = 16 / sizeof(T);
    constexpr int TPR = GATE_CW / VEC;
    constexpr int RPAR = GATE_THREADS / TPR;
    __shared__ float red[RPAR * GATE_CW];
    __shared__ double sh5[GATE_THREADS / 32][5];
    __shared__ double sh3[GATE_THREADS / 32][3];
    __shared__ int s_last;

    const int tid = threadIdx.x;
    const int blk = blockIdx.x;
    const int r = blk % g.R;
    const int cs = blk / g.R;
    const int s = cs % g.n_slices;
    const int c = cs / g.n_slices;
    const int d = g.d;
    const int col0 = s * GATE_CW;
    const int rbeg = c * g.npc + (int)(((long)r * g.npc) / g.R);
    const int rend = c * g.npc + (int)(((long)(r + 1) * g.npc) / g.R);
    const T *x = reinterpret_cast<const T *>(g.x);
    const int active = g.cell->active;
    const int n_sp = g.V * g.kfp * d;
    const int n_all = n_sp + g.V * d;
    const float *phi_prev = g.phi + (size_t)active * n_all;
    float *phi_next = g.phi + (size_t)(active ^ 1) * n_all;

    __shared__ int s_i0, s_i1;
    if (tid == 0) {
        s_i0 = g.kfp;
        s_i1 = 0;
    }
    __syncthreads();
    // fingerprint rows of this camera that fall in [rbeg, rend) (rows ascend)
    for (int i = tid; i < g.kfp; i += GATE_THREADS) {
        const int row = g.fp_rows[c * g.kfp + i];
        if (row >= rbeg && row < rend) {
            atomicMin(&s_i0, i);
            atomicMax(&s_i1, i + 1);
        }
    }

    // 1. column sums of this CTA's rows (global channel partials); 4 rows in
    //    flight per thread
    {
        const int ty = tid / TPR, tx = tid % TPR;
        float acc[VEC];
#pragma unroll
        for (int i = 0; i < VEC; ++i) acc[i] = 0.0f;
        auto add16 = [&](const uint4 u) {
            if constexpr (VEC == 8) {
                const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&w[j]));
                    acc[2 * j] += f.x;
                    acc[2 * j + 1] += f.y;
                }
            } else {
                acc[0] += __uint_as_float(u.x);
                acc[1] += __uint_as_float(u.y);
                acc[2] += __uint_as_float(u.z);
                acc[3] += __uint_as_float(u.w);
            }
        };
        const T *base = x + (size_t)col0 + tx * VEC;
        int row = rbeg + ty;
        for (; row + 3 * RPAR < rend; row += 4 * RPAR) {
            uint4 u[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) u[k] = *reinterpret_cast<const uint4 *>(base + (size_t)(row + k * RPAR) * d);
#pragma unroll
            for (int k = 0; k < 4; ++k) add16(u[k]);
        }
        for (; row < rend; row += RPAR) add16(*reinterpret_cast<const uint4 *>(base + (size_t)row * d));
#pragma unroll
        for (int i = 0; i < VEC; ++i) red[ty * GATE_CW + tx * VEC + i] = acc[i];
        __syncthreads();
        if (tid < GATE_CW) {
            float sum = 0.0f;
            for (int t = 0; t < RPAR; ++t) sum += red[t * GATE_CW + tid];
            g.colsum[((size_t)c * g.R + r) * d + col0 + tid] = sum;
        }
    }

    // 2. spatial-sample rows inside [rbeg, rend): metric partials, and the
    //    current fingerprint into the inactive buffer
    {
        double v[5] = {0.0, 0.0, 0.0, 0.0, 0.0};   // dot, |cur|^2, |prev|^2, max|diff|, sum|prev|
        const int i0 = s_i0, n_in = s_i1 > s_i0 ? s_i1 - s_i0 : 0;   // read after the barrier above
        for (int it = tid; it < n_in * GATE_CW; it += GATE_THREADS) {
            const int i = i0 + it / GATE_CW, j = it % GATE_CW;
            const int row = g.fp_rows[c * g.kfp + i];
            const size_t e = ((size_t)c * g.kfp + i) * d + col0 + j;
            const double cur = (double)to_f(x[(size_t)row * d + col0 + j]);
            const double prev = (double)phi_prev[e];
            phi_next[e] = (float)cur;
            v[0] += cur * prev;
            v[1] += cur * cur;
            v[2] += prev * prev;
            v[3] = fmax(v[3], fabs(cur - prev));
            v[4] += fabs(prev);
        }
        const int op[5] = {0, 0, 0, 1, 0};
        block_reduce<5>(v, op, sh5);
        if (tid == 0) {
#pragma unroll
            for (int k = 0; k < 5; ++k) g.sp_part[(size_t)blk * 5 + k] = v[k];
        }
    }

    // 3. last CTA of this (camera, slice): per-camera means of the slice
    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = atomicAdd(&g.cnt_cs[cs], 1u) == (unsigned)(g.R - 1);
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    {
        double v[3] = {0.0, 0.0, 0.0};
        if (tid < GATE_CW) {
            double sum = 0.0;
            for (int rr = 0; rr < g.R; ++rr) sum += (double)__ldcg(&g.colsum[((size_t)c * g.R + rr) * d + col0 + tid]);
            const float mean = (float)(sum / (double)g.npc);
            const size_t e = (size_t)n_sp + (size_t)c * d + col0 + tid;
            const double prev = (double)phi_prev[e];
            phi_next[e] = mean;
            v[0] = (double)mean * prev;
            v[1] = (double)mean * (double)mean;
            v[2] = prev * prev;
        }
        const int op[3] = {0, 0, 0};
        block_reduce<3>(v, op, sh3);
        if (tid == 0) {
#pragma unroll
            for (int k = 0; k < 3; ++k) g.gl_part[(size_t)cs * 3 + k] = v[k];
            g.cnt_cs[cs] = 0;
        }
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = atomicAdd(g.cnt_all, 1u) == (unsigned)(g.V * g.n_slices - 1);
    __syncthreads();
    if (!s_last) return;
    __threadfence();

    // 4. final: combine partials in a fixed order, decide (fp64)
    const int n_blk = g.V * g.n_slices * g.R;
    const int n_cs = g.V * g.n_slices;
    double v5[5] = {0.0, 0.0, 0.0, 0.0, 0.0};
    for (int i = tid; i < n_blk; i += GATE_THREADS) {
#pragma unroll
        for (int k = 0; k < 5; ++k) {
            const double p = __ldcg(&g.sp_part[(size_t)i * 5 + k]);
            v5[k] = k == 3 ? fmax(v5[k], p) : v5[k] + p;
        }
    }
    const int op5[5] = {0, 0, 0, 1, 0};
    block_reduce<5>(v5, op5, sh5);
    double v3[3] = {0.0, 0.0, 0.0};
    for (int i = tid; i < n_cs; i += GATE_THREADS) {
#pragma unroll
        for (int k = 0; k < 3; ++k) v3[k] += __ldcg(&g.gl_part[(size_t)i * 3 + k]);
    }
    const int op3[3] = {0, 0, 0};
    block_reduce<3>(v3, op3, sh3);
    if (tid != 0) return;
    *g.cnt_all = 0;

    double da = 0.0, na = 0.0, nb = 0.0;
    for (int i = 0; i < g.A; ++i) {
        const double a = (double)g.action[i];
        const double b = (double)g.phi_act[active * 8 + i];
        da += a * b;
        na += a * a;
        nb += b * b;
        g.phi_act[(active ^ 1) * 8 + i] = g.action[i];
    }
    const double cos_sp = cos_rule(v5[0], v5[1], v5[2]);
    const double cos_gl = cos_rule(v3[0], v3[1], v3[2]);
    const double cos_a = cos_rule(da, na, nb);
    const double s_min = fmin(fmin(cos_sp, cos_gl), cos_a);
    double dmax = v5[3] / (v5[4] / (double)n_sp + (double)g.eps_dev);
    if (isnan(dmax)) dmax = INFINITY;

    GateCell cell = *g.cell;
    uint8_t dec;
    bool flip;
    if (g.mode == 1 && cell.valid) {
        double tau = cell.has_hist ? fmax((double)g.tau_floor, cell.ema - (double)g.margin) : (double)g.tau_floor;
        if (g.strict_tau > 0.0f && g.step == 0) tau = fmax(tau, (double)g.strict_tau);
        bool skip = (s_min >= tau) && (dmax < (double)g.tau_dev);
        if (g.max_skips > 0 && cell.stale >= g.max_skips) skip = false;
        if (g.replay >= 0) skip = g.replay != 0;
        cell.ema = cell.has_hist ? (double)g.alpha * s_min + (1.0 - (double)g.alpha) * cell.ema : s_min;
        cell.has_hist = 1;
        cell.stale = skip ? cell.stale + 1 : 0;
        dec = skip ? XC_DEC_SKIP : XC_DEC_COMPUTE;
        flip = !skip || g.fp_refresh == 1;
        *g.s_cos = (float)s_min;
        *g.d_max = (float)dmax;
        *g.tau_out = (float)tau;
    } else {
        dec = XC_DEC_FORCED;
        flip = true;
        cell.valid = 1;
    }
    if (flip) cell.active ^= 1;
    *g.cell = cell;
    *g.flag = dec;
}

// Grid geometry shared by the launcher and the context (scratch sizing).
void gate_geometry(int V, int npc, int d, int n_sm, int *n_slices, int *R) {
    *n_slices = d / GATE_CW;
    const int base = V * *n_slices;
    int rr = (2 * n_sm + base - 1) / base;
    if (rr > npc) rr = npc;
    if (rr < 1) rr = 1;
    *R = rr;
}

template <typename T>
cudaError_t gate_launch(const GateArgs &g, cudaStream_t st) {
    const int blocks = g.V * g.n_slices * g.R;
    gate_kernel<T><<<blocks, GATE_THREADS, 0, st>>>(g);
    return cudaGetLastError();
}
template cudaError_t gate_launch<float>(const GateArgs &, cudaStream_t);
template cudaError_t gate_launch<bf16>(const GateArgs &, cudaStream_t);

// ---------------------------------------------------------------------------
// Allocation-free gate (xc_op_gate_static).  The gate kernel needs scratch for
// its column sums, partial metrics and tickets.  Here that scratch is one
// file-scope device array: every GPU that loads the library holds it until
// the process exits, and no call allocates or frees anything.  In host code
// the array's name is only a host-side stand-in, so its device address is
// looked up once per device with cudaGetSymbolAddress (the first call on a
// device does this set-up) and passed to the kernel.
// ---------------------------------------------------------------------------
constexpr size_t GATE_STATIC_SCRATCH_BYTES = 1u << 20;   // 1 MiB
static __device__ __align__(256) unsigned char g_gate_scratch[GATE_STATIC_SCRATCH_BYTES];

static std::mutex g_static_mu;
static void *g_static_ptr[64];                          // device address per device ordinal

// Device address of g_gate_scratch on the current device (set-up once per device).
static cudaError_t static_scratch(void **out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_static_mu);
    if (g_static_ptr[dev] == nullptr) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_gate_scratch);
        if (e != cudaSuccess) return e;
        g_static_ptr[dev] = p;
    }
    *out = g_static_ptr[dev];
    return cudaSuccess;
}

}  // namespace xc

using xc::GateArgs;
using xc::GateCell;

extern "C" xc_status xc_op_gate_static(int dtype, int n_cams, int tokens_per_cam, int d, const void *x,
                                       const int *fp_rows, int kfp, float *phi, float *phi_act,
                                       xc_gate_cell *cell, const float *action, int action_dim, int mode,
                                       int step, const xc_gate_params *gate, uint8_t *flag, float *s_cos,
                                       float *d_max, float *tau, void *stream) {
    char msg[256];
    auto fail = [&](xc_status s, const char *m) {
        snprintf(msg, sizeof msg, "xc_op_gate_static: %s", m);
        xc::set_global_error(msg);
        return s;
    };
    if (dtype != XC_F32 && dtype != XC_BF16) return fail(XC_EINVAL, "dtype");
    if (n_cams < 1 || tokens_per_cam < 1 || d < 64 || d % 64 != 0 || kfp < 1 || kfp > tokens_per_cam ||
        action_dim < 1 || action_dim > 8 || (mode != 0 && mode != 1) || step < 0)
        return fail(XC_EINVAL, "bad shape or mode (d % 64 == 0, 1 <= kfp <= tokens_per_cam, action_dim <= 8)");
    if (x == nullptr || fp_rows == nullptr || phi == nullptr || phi_act == nullptr || cell == nullptr ||
        action == nullptr || flag == nullptr || s_cos == nullptr || d_max == nullptr || tau == nullptr)
        return fail(XC_EINVAL, "NULL pointer");
    xc_gate_params p;
    if (gate != nullptr)
        p = *gate;
    else
        xc_gate_params_default(&p);
    const float knobs[] = {p.tau_floor, p.margin, p.alpha, p.tau_dev, p.eps_dev, p.step0_strict_tau};
    for (float v : knobs)
        if (isnan(v)) return fail(XC_EINVAL, "NaN gate knob");
    if (p.alpha < 0.0f || p.alpha > 1.0f || p.max_skips < 0 || (p.fp_refresh != 0 && p.fp_refresh != 1))
        return fail(XC_EINVAL, "gate knob out of range");

    // scratch layout, as for the caller-workspace gate
    int dev = 0, n_sm = 152;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return fail(XC_ECUDA, "no CUDA device");
    int ns = 0, R = 0;
    xc::gate_geometry(n_cams, tokens_per_cam, d, n_sm, &ns, &R);
    auto al = [](size_t v) { return (v + 255) & ~(size_t)255; };
    const size_t off_sp = al((size_t)n_cams * R * d * sizeof(float));
    const size_t off_gl = al(off_sp + (size_t)n_cams * ns * R * 5 * sizeof(double));
    const size_t off_cnt = al(off_gl + (size_t)n_cams * ns * 3 * sizeof(double));
    const size_t cnt_bytes = (size_t)(n_cams * ns + 1) * sizeof(unsigned);
    const size_t need = off_cnt + cnt_bytes;
    if (need > xc::GATE_STATIC_SCRATCH_BYTES) {
        snprintf(msg, sizeof msg,
                 "xc_op_gate_static: this geometry needs %zu bytes of scratch, more than the %zu-byte "
                 "static maximum (use xc_op_gate with a workspace)",
                 need, xc::GATE_STATIC_SCRATCH_BYTES);
        xc::set_global_error(msg);
        return XC_EINVAL;
    }
    void *scratch = nullptr;
    if (xc::static_scratch(&scratch) != cudaSuccess) return fail(XC_ECUDA, "cudaGetSymbolAddress failed");
    char *w = reinterpret_cast<char *>(scratch);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    // the tickets must start at zero; the rest of the array is overwritten
    if (cudaMemsetAsync(w + off_cnt, 0, cnt_bytes, st) != cudaSuccess) return fail(XC_ECUDA, "cudaMemsetAsync");

    GateArgs g;
    memset(&g, 0, sizeof g);
    g.x = x;
    g.d = d;
    g.V = n_cams;
    g.npc = tokens_per_cam;
    g.fp_rows = fp_rows;
    g.kfp = kfp;
    g.n_slices = ns;
    g.R = R;
    g.phi = phi;
    g.phi_act = phi_act;
    for (int i = 0; i < action_dim; ++i) g.action[i] = action[i];
    g.A = action_dim;
    g.cell = reinterpret_cast<GateCell *>(cell);
    g.mode = mode;
    g.step = step;
    g.tau_floor = p.tau_floor;
    g.margin = p.margin;
    g.alpha = p.alpha;
    g.tau_dev = p.tau_dev;
    g.eps_dev = p.eps_dev;
    g.strict_tau = p.step0_strict_tau;
    g.max_skips = p.max_skips;
    g.fp_refresh = p.fp_refresh;
    g.replay = p.replay_skip != nullptr ? (p.replay_skip[0] != 0 ? 1 : 0) : -1;
    g.flag = flag;
    g.s_cos = s_cos;
    g.d_max = d_max;
    g.tau_out = tau;
    g.colsum = reinterpret_cast<float *>(w);
    g.sp_part = reinterpret_cast<double *>(w + off_sp);
    g.gl_part = reinterpret_cast<double *>(w + off_gl);
    g.cnt_cs = reinterpret_cast<unsigned *>(w + off_cnt);
    g.cnt_all = g.cnt_cs + n_cams * ns;
    const cudaError_t e = dtype == XC_BF16 ? xc::gate_launch<xc::bf16>(g, st) : xc::gate_launch<float>(g, st);
    if (e != cudaSuccess) return fail(XC_ECUDA, cudaGetErrorString(e));
    return XC_OK;
}
