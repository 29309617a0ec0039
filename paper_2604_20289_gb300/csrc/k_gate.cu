// Fused X-Cache gate of one (denoising step t, block b): fingerprint of the
// block input, both gating metrics against the cached fingerprint, adaptive
// threshold and the skip / recompute flag -- all on the device.
//
// Fingerprint (Section 2.3.1-2.3.2), per view group g of V_g cameras:
//   spatial entry  x at the K-token sample of every camera of g        [V_g, k_g, d]
//   global channel per-camera mean of x over its tokens                 [V_g, d]
// plus the condition entry, the chunk's action vector                   [A]
// Metrics: s_cos = min over all entries of the cosine (Eq. 5); d_max = max
// over the groups of max|cur - prev| / (mean|prev| + eps) over the group's
// spatial entry (Eq. 6).  Decision Eq. 7 with tau_cos = max(tau_floor, ema -
// m) (Eq. 9), EMA update (Eq. 8) and the consecutive-skip cap (Section 2.5 (4)).
//
// Grid: one CTA (512 threads) per (camera c, 64-column slice s).  The CTA
// streams all of camera c's rows of its slice once (16-byte loads, 8 rows in
// flight per thread), so it completes that slice's per-camera means by
// itself; it also takes the slice of the spatial sample.  All reductions run
// in fp32; each CTA writes 8 partials and takes an atomic ticket; the last
// CTA combines the partials of each group in a fixed order and makes the
// decision (the EMA state is kept in fp64).  No spin-wait anywhere; deterministic.  The cached
// fingerprint is double-buffered per (t, b): the current fingerprint goes to
// the inactive half, which becomes active when the block recomputes.
#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "xc_kernels.cuh"

namespace xc {

constexpr int GATE_CW = 64;          // columns per CTA
constexpr int GATE_THREADS = 512;
constexpr int GATE_UNROLL = 8;       // rows in flight per thread
constexpr int GATE_PARTS = 8;        // dot, |cur|^2, |prev|^2, max|diff|, sum|prev| (spatial); dot, |cur|^2, |prev|^2 (global)

// Cosine of one entry from its dot product and squared norms (Eq. 5):
// both norms < 1e-12 -> 1, exactly one -> 0, NaN -> 0.
__device__ __forceinline__ float cos_rule_f(float dot, float n1sq, float n2sq) {
    const float a = sqrtf(n1sq), b = sqrtf(n2sq);
    if (isnan(a) || isnan(b) || isnan(dot)) return 0.0f;
    if (a < 1e-12f && b < 1e-12f) return 1.0f;
    if (a < 1e-12f || b < 1e-12f) return 0.0f;
    return dot / (a * b);
}

template <typename T>
__device__ __forceinline__ void add_vec16(float *acc, const uint4 u) {
    if constexpr (sizeof(T) == 2) {
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
}

template <typename T>
__global__ void __launch_bounds__(GATE_THREADS) gate_kernel(const GateArgs g) {
    pdl_wait();
    pdl_release();
    constexpr int VEC = 16 / sizeof(T);
    constexpr int TPR = GATE_CW / VEC;          // threads per row
    constexpr int RPAR = GATE_THREADS / TPR;    // rows per sweep
    constexpr int NW = GATE_THREADS / 32;
    __shared__ float red[RPAR * GATE_CW];
    __shared__ float wpart[NW][GATE_PARTS];
    __shared__ int s_last;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int blk = blockIdx.x;
    const int c = blk / g.n_slices, s = blk % g.n_slices;
    const int d = g.d;
    // camera c's group (unrolled compare chain: constant parameter indices)
    int tok0 = g.g_tok0[0], cam0 = g.g_cam0[0], npc = g.g_npc[0], fp0 = g.g_fp0[0], kfp = g.g_kfp[0];
#pragma unroll
    for (int q = 1; q < XC_MAX_GROUPS; ++q)
        if (q < g.n_groups && c >= g.g_cam0[q]) {
            tok0 = g.g_tok0[q];
            cam0 = g.g_cam0[q];
            npc = g.g_npc[q];
            fp0 = g.g_fp0[q];
            kfp = g.g_kfp[q];
        }
    const size_t ctok0 = (size_t)tok0 + (size_t)(c - cam0) * npc;   // camera c's first token
    const int crow0 = fp0 + (c - cam0) * kfp;                        // and first sample row
    const int col0 = s * GATE_CW;
    const T *x = reinterpret_cast<const T *>(g.x);
    const int active = g.cell->active;
    const int n_sp = g.n_rows * d;
    const int n_all = n_sp + g.V * d;
    const float *phi_prev = g.phi + (size_t)active * n_all;
    float *phi_next = g.phi + (size_t)(active ^ 1) * n_all;

    // 1. column sums of camera c, columns [col0, col0 + 64)
    float acc[VEC];
#pragma unroll
    for (int i = 0; i < VEC; ++i) acc[i] = 0.0f;
    {
        const int ty = tid / TPR, tx = tid % TPR;
        const T *base = x + ctok0 * d + col0 + tx * VEC;
        // GATE_UNROLL guarded loads in flight per step, the ragged end included
        for (int r = ty; r < npc; r += GATE_UNROLL * RPAR) {
            uint4 u[GATE_UNROLL];
#pragma unroll
            for (int k = 0; k < GATE_UNROLL; ++k)
                u[k] = r + k * RPAR < npc ? *reinterpret_cast<const uint4 *>(base + (size_t)(r + k * RPAR) * d)
                                          : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
            for (int k = 0; k < GATE_UNROLL; ++k) add_vec16<T>(acc, u[k]);
        }
#pragma unroll
        for (int i = 0; i < VEC; ++i) red[ty * GATE_CW + tx * VEC + i] = acc[i];
    }
    __syncthreads();

    float p[GATE_PARTS] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    // 2. global channel of this slice: per-camera means (threads 0..63)
    if (tid < GATE_CW) {
        float sum = 0.0f;
        for (int t = 0; t < RPAR; ++t) sum += red[t * GATE_CW + tid];
        const float mean = sum / (float)npc;
        const size_t e = (size_t)n_sp + (size_t)c * d + col0 + tid;
        const float prev = phi_prev[e];
        phi_next[e] = mean;
        p[5] = mean * prev;
        p[6] = mean * mean;
        p[7] = prev * prev;
    }
    // 3. spatial sample rows of camera c in this slice
    for (int it = tid; it < kfp * GATE_CW; it += GATE_THREADS) {
        const int i = it / GATE_CW, j = it % GATE_CW;
        const int row = g.fp_rows[crow0 + i];
        const size_t e = ((size_t)crow0 + i) * d + col0 + j;
        const float cur = to_f(x[(size_t)row * d + col0 + j]);
        const float prev = phi_prev[e];
        phi_next[e] = cur;
        p[0] = fmaf(cur, prev, p[0]);
        p[1] = fmaf(cur, cur, p[1]);
        p[2] = fmaf(prev, prev, p[2]);
        p[3] = fmaxf(p[3], fabsf(cur - prev));
        p[4] += fabsf(prev);
    }
    // CTA reduction: within warps, then across warps in a fixed order
#pragma unroll
    for (int k = 0; k < GATE_PARTS; ++k) {
        float v = p[k];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float w = __shfl_xor_sync(0xffffffffu, v, o);
            v = k == 3 ? fmaxf(v, w) : v + w;
        }
        if (lane == 0) wpart[warp][k] = v;
    }
    __syncthreads();
    if (tid < GATE_PARTS) {
        float v = 0.0f;
        for (int w = 0; w < NW; ++w) v = tid == 3 ? fmaxf(v, wpart[w][tid]) : v + wpart[w][tid];
        g.part[(size_t)blk * GATE_PARTS + tid] = v;
    }

    // 4. ticket: the last CTA combines all partials and decides
    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = atomicAdd(g.ticket, 1u) == (unsigned)(gridDim.x - 1);
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    // Per view group: fold the partials of the group's CTAs (cameras
    // [g_cam0[q], g_cam0[q + 1]), every slice) in a fixed order; thread 0
    // keeps the running min of the cosines and max of the deviations.
    float cos_min = INFINITY, dmax = 0.0f;
#pragma unroll
    for (int q = 0; q < XC_MAX_GROUPS; ++q) {
        if (q >= g.n_groups) break;
        const int b0 = g.g_cam0[q] * g.n_slices, b1 = g.g_cam0[q + 1] * g.n_slices;
        float v[GATE_PARTS] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        for (int b = b0 + tid; b < b1; b += GATE_THREADS) {
#pragma unroll
            for (int k = 0; k < GATE_PARTS; ++k) {
                const float w = __ldcg(&g.part[(size_t)b * GATE_PARTS + k]);
                v[k] = k == 3 ? fmaxf(v[k], w) : v[k] + w;
            }
        }
#pragma unroll
        for (int k = 0; k < GATE_PARTS; ++k) {
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const float w = __shfl_xor_sync(0xffffffffu, v[k], o);
                v[k] = k == 3 ? fmaxf(v[k], w) : v[k] + w;
            }
            if (lane == 0) wpart[warp][k] = v[k];
        }
        __syncthreads();
        if (tid == 0) {
            for (int k = 0; k < GATE_PARTS; ++k) {
                float a = wpart[0][k];
                for (int w = 1; w < NW; ++w) a = k == 3 ? fmaxf(a, wpart[w][k]) : a + wpart[w][k];
                v[k] = a;
            }
            const int n_sp_q = (g.g_cam0[q + 1] - g.g_cam0[q]) * g.g_kfp[q] * d;
            float dq = v[3] / (v[4] / (float)n_sp_q + g.eps_dev);
            if (isnan(dq)) dq = INFINITY;
            cos_min = fminf(cos_min, fminf(cos_rule_f(v[0], v[1], v[2]), cos_rule_f(v[5], v[6], v[7])));
            dmax = fmaxf(dmax, dq);
        }
        __syncthreads();
    }
    if (tid != 0) return;
    *g.ticket = 0;

    // All sums and metrics are fp32 (relative error ~1e-7, far inside the
    // 1e-3 band around a threshold): FP64 arithmetic, square roots and divides
    // are slow on this part; only the EMA state stays fp64.
    float da = 0.0f, na = 0.0f, nb = 0.0f;
    for (int i = 0; i < g.A; ++i) {
        const float a = g.action_dev != nullptr ? g.action_dev[i] : g.action[i];
        const float b = g.phi_act[active * 8 + i];
        da = fmaf(a, b, da);
        na = fmaf(a, a, na);
        nb = fmaf(b, b, nb);
        g.phi_act[(active ^ 1) * 8 + i] = g.action_dev != nullptr ? g.action_dev[i] : g.action[i];
    }
    const float cos_a = cos_rule_f(da, na, nb);
    const double s_min = (double)fminf(cos_min, cos_a);

    GateCell cell = *g.cell;
    uint8_t dec;
    bool flip;
    if (g.mode == 1 && cell.valid) {
        double tau = cell.has_hist ? fmax((double)g.tau_floor, cell.ema - (double)g.margin) : (double)g.tau_floor;
        if (g.strict_tau > 0.0f && g.step == 0) tau = fmax(tau, (double)g.strict_tau);
        bool skip = (s_min >= tau) && (dmax < g.tau_dev);
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

// Scratch of one gate launch: GATE_PARTS fp32 partials per CTA, then one
// 32-bit ticket (which must be zero before the launch; the kernel leaves it
// zero).  Returns the total bytes; *ticket_off receives the ticket's offset.
size_t gate_scratch(int V, int d, int *n_slices, size_t *ticket_off) {
    *n_slices = d / GATE_CW;
    const size_t part = (size_t)V * *n_slices * GATE_PARTS * sizeof(float);
    *ticket_off = (part + 255) & ~(size_t)255;
    return *ticket_off + 256;
}

template <typename T>
cudaError_t gate_launch(const GateArgs &g, cudaStream_t st) {
    return launch_pdl(gate_kernel<T>, dim3(g.V * g.n_slices), dim3(GATE_THREADS), 0, st, g);
}
template cudaError_t gate_launch<float>(const GateArgs &, cudaStream_t);
template cudaError_t gate_launch<bf16>(const GateArgs &, cudaStream_t);

// ---------------------------------------------------------------------------
// Allocation-free gate (xc_op_gate_static).  The gate kernel needs scratch for
// its partial metrics and its ticket.  Here that scratch is one file-scope
// device array: every GPU that loads the library holds it until the process
// exits, and no call allocates or frees anything.  In host code the array's
// name is only a host-side stand-in, so its device address is looked up once
// per device with cudaGetSymbolAddress (the first call on a device does this
// set-up) and passed to the kernel.
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

    int ns = 0;
    size_t ticket_off = 0;
    const size_t need = xc::gate_scratch(n_cams, d, &ns, &ticket_off);
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
    // the ticket must start at zero; the partials are overwritten
    if (cudaMemsetAsync(w + ticket_off, 0, sizeof(unsigned), st) != cudaSuccess)
        return fail(XC_ECUDA, "cudaMemsetAsync");

    GateArgs g;
    memset(&g, 0, sizeof g);
    g.x = x;
    g.d = d;
    xc::gate_single_group(g, n_cams, tokens_per_cam, kfp);
    g.fp_rows = fp_rows;
    g.n_slices = ns;
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
    g.part = reinterpret_cast<float *>(w);
    g.ticket = reinterpret_cast<unsigned *>(w + ticket_off);
    const cudaError_t e = dtype == XC_BF16 ? xc::gate_launch<xc::bf16>(g, st) : xc::gate_launch<float>(g, st);
    if (e != cudaSuccess) return fail(XC_ECUDA, cudaGetErrorString(e));
    return XC_OK;
}
