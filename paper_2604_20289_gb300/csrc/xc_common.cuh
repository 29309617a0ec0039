// Common device helpers of the X-Cache CUDA path (sm_103a).
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/xcache.h"
#include "../../include/xcache_ops.h"

namespace xc {

// Programmatic dependent launch.  Kernels of the chunk step are launched with
// programmatic stream serialisation: a kernel may be scheduled while its
// predecessor is still running, and pdl_wait() -- the first statement of each
// such kernel -- blocks until the predecessor has completed and its memory
// is visible (so everything earlier in the stream is complete as well).
// pdl_release() then lets the successor be scheduled.  Without the launch
// attribute both are no-ops.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_release() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                              Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
}

typedef __nv_bfloat16 bf16;

// Device error word bits (bounded waits that expired, bad launch state).
enum : int {
    ERR_WAIT_TMA = 1,
    ERR_WAIT_MMA = 2,
    ERR_WAIT_EPI = 4,
    ERR_WAIT_SOFTMAX = 8,
    ERR_WAIT_PRODUCER = 16,
    ERR_BAD_LAUNCH = 32,
};

// Wait limit of every spin on an mbarrier: 2 s of global time, and a hard
// iteration cap in case the timer does not advance.
constexpr unsigned long long WAIT_NS = 2000000000ull;
constexpr unsigned int WAIT_MAX_ITERS = 1u << 30;

// ---------------------------------------------------------------- storage
__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(bf16 v) { return __bfloat162float(v); }

template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }

// Round a float to the storage type and back (the value a store would keep).
template <typename T> __device__ __forceinline__ float round_to(float v) { return to_f(from_f<T>(v)); }

// Load / store a run of 16 consecutive elements (row-major, 16-element aligned).
template <typename T> __device__ __forceinline__ void load16(const T *p, float (&v)[16]);
template <> __device__ __forceinline__ void load16<float>(const float *p, float (&v)[16]) {
    const float4 *q = reinterpret_cast<const float4 *>(p);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        float4 t = q[i];
        v[4 * i] = t.x; v[4 * i + 1] = t.y; v[4 * i + 2] = t.z; v[4 * i + 3] = t.w;
    }
}
template <> __device__ __forceinline__ void load16<bf16>(const bf16 *p, float (&v)[16]) {
    const uint4 *q = reinterpret_cast<const uint4 *>(p);
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        uint4 t = q[i];
        uint32_t w[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            __nv_bfloat162 h = *reinterpret_cast<__nv_bfloat162 *>(&w[j]);
            float2 f = __bfloat1622float2(h);
            v[8 * i + 2 * j] = f.x;
            v[8 * i + 2 * j + 1] = f.y;
        }
    }
}
template <typename T> __device__ __forceinline__ void store16(T *p, const float (&v)[16]);
template <> __device__ __forceinline__ void store16<float>(float *p, const float (&v)[16]) {
    float4 *q = reinterpret_cast<float4 *>(p);
#pragma unroll
    for (int i = 0; i < 4; ++i) q[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
}
template <> __device__ __forceinline__ void store16<bf16>(bf16 *p, const float (&v)[16]) {
    uint4 *q = reinterpret_cast<uint4 *>(p);
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        uint32_t w[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            __nv_bfloat162 h = __floats2bfloat162_rn(v[8 * i + 2 * j], v[8 * i + 2 * j + 1]);
            w[j] = *reinterpret_cast<uint32_t *>(&h);
        }
        q[i] = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

__device__ __forceinline__ float gelu_tanh(float x) {
    const float k0 = 0.7978845608028654f;   // sqrt(2/pi)
    return 0.5f * x * (1.0f + tanhf(k0 * (x + 0.044715f * x * x * x)));
}
__device__ __forceinline__ float gelu_tanh_approx(float x) {
    const float k0 = 0.7978845608028654f;
    const float u = k0 * fmaf(0.044715f * x, x * x, x);
    float t;
    asm("tanh.approx.f32 %0, %1;" : "=f"(t) : "f"(u));
    const float hx = 0.5f * x;
    return fmaf(hx, t, hx);
}
__device__ __forceinline__ float silu(float x) { return x / (1.0f + expf(-x)); }

// ------------------------------------------------------------ GEMM epilogue
// Everything a fused GEMM epilogue may need.  One call processes the run of
// 16 consecutive output columns [col, col + 16) of one row.
struct EpiParams {
    int M, N;
    const float *bias;         // [N]
    const float *gate;         // [N]   adaLN-Zero gate (resid kinds)
    const void *resid;         // [M][N] residual stream input
    const void *xin;           // [M][N] block input (residual cache)
    void *out;                 // [M][N]  (q for the QKV kind)
    void *out_k;               // [M][d]  QKV kind
    void *out_v;               // [M][d]  QKV kind
    void *rhat;                // [M][N]  residual cache slot or nullptr
    // RoPE geometry (QKV kind): view group g covers tokens [g_tok0[g],
    // g_tok0[g + 1]) with cameras g_cam0[g].. of g_npc[g] = frames * g_gh[g]
    // * g_gw[g] tokens each
    int d, head_dim, frames, frame0;
    int n_groups;
    int g_tok0[XC_MAX_GROUPS], g_cam0[XC_MAX_GROUPS], g_npc[XC_MAX_GROUPS], g_gh[XC_MAX_GROUPS],
        g_gw[XC_MAX_GROUPS];
    const int *rope_axis;      // [head_dim/2] 0 camera, 1 frame, 2 h, 3 w
    const int *rope_off;       // [head_dim/2] table entry of position 0 of each pair
    const float2 *rope_cs;     // (cos, sin) table of this chunk (rope_table_kernel)
};

// One view group covering every camera (grid gh x gw).
inline void epi_single_grid(EpiParams &p, int frames, int gh, int gw) {
    p.frames = frames;
    p.n_groups = 1;
    p.g_tok0[0] = 0;
    p.g_cam0[0] = 0;
    p.g_npc[0] = frames * gh * gw;
    p.g_gh[0] = gh;
    p.g_gw[0] = gw;
}

// (camera, frame within the chunk, h, w) of token `row`.  The group is picked
// by an unrolled compare chain, so the parameter arrays are only read at
// constant indices.
__device__ __forceinline__ int4 token_pos(const EpiParams &p, int row) {
    int tok0 = p.g_tok0[0], cam0 = p.g_cam0[0], npc = p.g_npc[0], gh = p.g_gh[0], gw = p.g_gw[0];
#pragma unroll
    for (int g = 1; g < XC_MAX_GROUPS; ++g)
        if (g < p.n_groups && row >= p.g_tok0[g]) {
            tok0 = p.g_tok0[g];
            cam0 = p.g_cam0[g];
            npc = p.g_npc[g];
            gh = p.g_gh[g];
            gw = p.g_gw[g];
        }
    const int r = row - tok0;
    const int cl = r / npc;
    const int rem = r - cl * npc;
    return make_int4(cam0 + cl, rem / (gh * gw), (rem / gw) % gh, rem % gw);
}

enum { EPI_BIAS = XC_EPI_BIAS, EPI_GELU = XC_EPI_GELU, EPI_RESID_GATE = XC_EPI_RESID_GATE,
       EPI_RESID_CACHE = XC_EPI_RESID_CACHE, EPI_QKV_ROPE = 16 };

// Runs of W = 8 or 16 consecutive elements (16-byte aligned).
template <typename T, int W>
__device__ __forceinline__ void loadW(const T *p, float (&v)[W]) {
    if constexpr (W == 16) {
        load16<T>(p, v);
    } else if constexpr (sizeof(T) == 2) {
        const uint4 u = *reinterpret_cast<const uint4 *>(p);
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&w[j]));
            v[2 * j] = f.x;
            v[2 * j + 1] = f.y;
        }
    } else {
        const float4 a = reinterpret_cast<const float4 *>(p)[0], b = reinterpret_cast<const float4 *>(p)[1];
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
        v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
}
template <typename T, int W>
__device__ __forceinline__ void storeW(T *p, const float (&v)[W]) {
    if constexpr (W == 16) {
        store16<T>(p, v);
    } else if constexpr (sizeof(T) == 2) {
        uint32_t w[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            __nv_bfloat162 h = __floats2bfloat162_rn(v[2 * j], v[2 * j + 1]);
            w[j] = *reinterpret_cast<uint32_t *>(&h);
        }
        *reinterpret_cast<uint4 *>(p) = make_uint4(w[0], w[1], w[2], w[3]);
    } else {
        reinterpret_cast<float4 *>(p)[0] = make_float4(v[0], v[1], v[2], v[3]);
        reinterpret_cast<float4 *>(p)[1] = make_float4(v[4], v[5], v[6], v[7]);
    }
}

// Fused GEMM epilogue on one run of W consecutive output columns
// [col, col + W) of one row (W = 8 or 16, col a multiple of W).
template <int EPI, typename T, int W>
__device__ __forceinline__ void epilogue_run(const EpiParams &p, int row, int col, float (&acc)[W]) {
    if (row >= p.M) return;
    {
        float b[W];
        loadW<float, W>(p.bias + col, b);
#pragma unroll
        for (int i = 0; i < W; ++i) acc[i] += b[i];
    }
    const size_t off = (size_t)row * p.N + col;
    if constexpr (EPI == EPI_BIAS) {
        storeW<T, W>(reinterpret_cast<T *>(p.out) + off, acc);
    } else if constexpr (EPI == EPI_GELU) {
        if constexpr (sizeof(T) == 2) {
            // bf16 output: the hardware tanh (rel. error ~2^-11) is below the
            // output rounding (2^-9)
#pragma unroll
            for (int i = 0; i < W; ++i) acc[i] = gelu_tanh_approx(acc[i]);
        } else {
#pragma unroll
            for (int i = 0; i < W; ++i) acc[i] = gelu_tanh(acc[i]);
        }
        storeW<T, W>(reinterpret_cast<T *>(p.out) + off, acc);
    } else if constexpr (EPI == EPI_RESID_GATE || EPI == EPI_RESID_CACHE) {
        float r[W], g[W];
        loadW<T, W>(reinterpret_cast<const T *>(p.resid) + off, r);
        loadW<float, W>(p.gate + col, g);
#pragma unroll
        for (int i = 0; i < W; ++i) acc[i] = r[i] + g[i] * acc[i];
        storeW<T, W>(reinterpret_cast<T *>(p.out) + off, acc);
        if constexpr (EPI == EPI_RESID_CACHE) {
            if (p.rhat != nullptr) {
                float xi[W];
                loadW<T, W>(reinterpret_cast<const T *>(p.xin) + off, xi);
#pragma unroll
                for (int i = 0; i < W; ++i) acc[i] = round_to<T>(acc[i]) - xi[i];
                storeW<T, W>(reinterpret_cast<T *>(p.rhat) + off, acc);
            }
        }
    } else if constexpr (EPI == EPI_QKV_ROPE) {
        const int d = p.d;
        const int part = col / d;          // 0 q, 1 k, 2 v (runs never straddle: d % 16 == 0)
        const int c = col - part * d;
        if (part < 2) {
            const int4 tp = token_pos(p, row);
            const int pos[4] = {tp.x, tp.y, tp.z, tp.w};      // frame: index within the chunk
            const int pair0 = (c % p.head_dim) >> 1;
#pragma unroll
            for (int j = 0; j < W / 2; ++j) {
                const int pr = pair0 + j;
                const float2 t = p.rope_cs[p.rope_off[pr] + pos[p.rope_axis[pr]]];
                const float x0 = acc[2 * j], x1 = acc[2 * j + 1];
                acc[2 * j] = x0 * t.x - x1 * t.y;
                acc[2 * j + 1] = x0 * t.y + x1 * t.x;
            }
        }
        T *dst = reinterpret_cast<T *>(part == 0 ? p.out : (part == 1 ? p.out_k : p.out_v));
        storeW<T, W>(dst + (size_t)row * d + c, acc);
    }
}
template <int EPI, typename T>
__device__ __forceinline__ void epilogue16(const EpiParams &p, int row, int col, float (&acc)[16]) {
    epilogue_run<EPI, T, 16>(p, row, col, acc);
}

}  // namespace xc
