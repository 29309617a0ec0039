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
// Grid: one CTA (256 threads) per (camera c, column slice s, row block r).
// The slice is as wide as still fills the SMs (64 to 512 columns: the wider,
// the longer each row's contiguous run), the row blocks split each camera's
// tokens so that the grid fills the SMs (up to four CTAs per SM), and the R
// row blocks of one (camera, slice) form a thread-block cluster.  A CTA
// streams its rows of its slice once (16-byte streaming loads, batches of 8
// rows in flight per thread) into column sums, and takes every R-th row of
// the camera's spatial sample in its slice.  Two folds follow, each in a
// fixed order (deterministic; the only waits are one cluster barrier, which
// every CTA of the cluster reaches, and no spin-wait):
//   1. every rank stores its column sums into rank 0's shared memory
//      (distributed shared memory); after the cluster barrier rank 0 adds
//      them in rank order, giving the slice of the camera's mean, and its
//      global-channel products; every CTA then writes 8 partial metrics (its
//      sample products, rank 0 also the global-channel products);
//   2. the last CTA of the grid (global ticket) adds the partials of each
//      view group in CTA order and thread 0 applies Eq. 5-9 (metrics in fp32,
//      EMA state in fp64), writing the decision byte every later kernel of the
//      block reads.
// The ticket is left at zero for the next launch.  The cached fingerprint
// is double-buffered per (t, b): the current fingerprint goes to the inactive
// half, which becomes active when the block recomputes.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>

#include <cooperative_groups.h>

#include "xc_kernels.cuh"

namespace cg = cooperative_groups;

namespace xc {

constexpr int GATE_MAX_CW = 512;     // widest column slice of one CTA (64, 128, 256 or 512 columns)
constexpr int GATE_THREADS = 256;
constexpr int GATE_UNROLL = 8;       // rows in flight per thread (one unguarded batch)
constexpr int GATE_PARTS = 8;        // dot, |cur|^2, |prev|^2, max|diff|, sum|prev| (spatial); dot, |cur|^2, |prev|^2 (global)
constexpr int GATE_CTAS_PER_SM = 4;  // target CTAs per SM of the row split
constexpr int GATE_MAX_CLUSTER = 8;  // row blocks of one (camera, slice): one cluster (portable size)

// Cosine of one entry from its dot product and squared norms (Eq. 5):
// both norms < 1e-12 -> 1, exactly one -> 0, NaN -> 0.
__device__ __forceinline__ float cos_rule_f(float dot, float n1sq, float n2sq) {
    const float a = sqrtf(n1sq), b = sqrtf(n2sq);
    if (isnan(a) || isnan(b) || isnan(dot)) return 0.0f;
    if (a < 1e-12f && b < 1e-12f) return 1.0f;
    if (a < 1e-12f || b < 1e-12f) return 0.0f;
    return dot / (a * b);
}

// Adds one 16-byte vector to running fp32 pair sums: bf16 elements are
// widened by placing their 16 bits in the high half of an fp32 word (exact).
template <typename T>
__device__ __forceinline__ void add_pairs(float2 (&acc)[16 / sizeof(T) / 2], const uint4 u) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
    if constexpr (sizeof(T) == 2) {
#pragma unroll
        for (int j = 0; j < 4; ++j)
            acc[j] = __fadd2_rn(acc[j], make_float2(__uint_as_float(w[j] << 16), __uint_as_float(w[j] & 0xFFFF0000u)));
    } else {
        acc[0] = __fadd2_rn(acc[0], make_float2(__uint_as_float(w[0]), __uint_as_float(w[1])));
        acc[1] = __fadd2_rn(acc[1], make_float2(__uint_as_float(w[2]), __uint_as_float(w[3])));
    }
}

// Sum (or, for part 3, max) of the 8 partials over the CTA in a fixed order:
// butterfly within each warp, then warps in index order by thread 0.
__device__ __forceinline__ void cta_fold8(float (&v)[GATE_PARTS], float (*wpart)[GATE_PARTS], int lane, int warp,
                                          int nw) {
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
    if (threadIdx.x == 0) {
#pragma unroll
        for (int k = 0; k < GATE_PARTS; ++k) {
            float a = wpart[0][k];
            for (int w = 1; w < nw; ++w) a = k == 3 ? fmaxf(a, wpart[w][k]) : a + wpart[w][k];
            v[k] = a;
        }
    }
}

// Column sums of rows [rb0, rb1) (tokens from ctok0) over columns [col0,
// col0 + cw) of x [.][d]: cw / VEC threads cover a row (16 bytes each),
// the rest of the CTA takes further rows; full batches of GATE_UNROLL rows go
// out unguarded (32-bit byte offsets), the sums are kept as fp32 pairs (bf16
// halves widened by shifts, packed adds).  The CTA's sums land in cluster
// rank 0's call[r] (distributed shared memory).
template <typename T>
__device__ __forceinline__ void slice_colsums(const T *x, size_t ctok0, int d, int col0, int cw, int rb0, int rb1,
                                              int r, float *red, float (*call)[GATE_MAX_CW],
                                              cg::cluster_group &cluster) {
    constexpr int VEC = 16 / sizeof(T);
    const int tid = threadIdx.x;
    const int TPR = cw / VEC, RPAR = GATE_THREADS / TPR;
    const int ty = tid / TPR, tx = tid % TPR;
    const int first = rb0 + ty;
    const int n = first < rb1 ? (rb1 - first + RPAR - 1) / RPAR : 0;     // rows of this thread
    const char *p = reinterpret_cast<const char *>(x + (ctok0 + first) * d + col0 + tx * VEC);
    const uint32_t stride = (uint32_t)RPAR * (uint32_t)d * (uint32_t)sizeof(T);
    float2 acc2[VEC / 2];
#pragma unroll
    for (int i = 0; i < VEC / 2; ++i) acc2[i] = make_float2(0.0f, 0.0f);
    int i = 0;
    for (; i + GATE_UNROLL <= n; i += GATE_UNROLL) {
        uint4 u[GATE_UNROLL];
#pragma unroll
        for (int k = 0; k < GATE_UNROLL; ++k) u[k] = __ldcs(reinterpret_cast<const uint4 *>(p + k * stride));
        p += GATE_UNROLL * stride;
#pragma unroll
        for (int k = 0; k < GATE_UNROLL; ++k) add_pairs<T>(acc2, u[k]);
    }
    for (; i < n; ++i) {
        add_pairs<T>(acc2, __ldcs(reinterpret_cast<const uint4 *>(p)));
        p += stride;
    }
#pragma unroll
    for (int i2 = 0; i2 < VEC / 2; ++i2) {
        red[ty * cw + tx * VEC + 2 * i2] = acc2[i2].x;
        red[ty * cw + tx * VEC + 2 * i2 + 1] = acc2[i2].y;
    }
    __syncthreads();
    for (int j = tid; j < cw; j += GATE_THREADS) {
        float sum = 0.0f;
        for (int t = 0; t < RPAR; ++t) sum += red[t * cw + j];
        *cluster.map_shared_rank(&call[r][j], 0) = sum;
    }
}

// Camera c's view group: first token, first camera, tokens per camera,
// first sample row and sample rows per camera (unrolled compare chain:
// constant parameter indices).
struct CamGroup {
    int tok0, cam0, npc, fp0, kfp;
};
__device__ __forceinline__ CamGroup cam_group(const GateArgs &g, int c) {
    CamGroup q0{g.g_tok0[0], g.g_cam0[0], g.g_npc[0], g.g_fp0[0], g.g_kfp[0]};
#pragma unroll
    for (int q = 1; q < XC_MAX_GROUPS; ++q)
        if (q < g.n_groups && c >= g.g_cam0[q]) q0 = CamGroup{g.g_tok0[q], g.g_cam0[q], g.g_npc[q], g.g_fp0[q], g.g_kfp[q]};
    return q0;
}

template <typename T>
__global__ void __launch_bounds__(GATE_THREADS, GATE_CTAS_PER_SM) gate_kernel(const GateArgs g) {
    pdl_wait();
    pdl_release();
    constexpr int VEC = 16 / sizeof(T);
    constexpr int NW = GATE_THREADS / 32;
    __shared__ float red[GATE_THREADS * VEC];
    __shared__ float wpart[NW][GATE_PARTS];
    __shared__ float call[GATE_MAX_CLUSTER][GATE_MAX_CW];   // column sums of every rank (rank 0's copy is used)
    __shared__ int s_last;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int blk = blockIdx.x;
    const int R = g.R, cw = g.cw;
    const int r = blk % R, cs = blk / R;
    const int c = cs / g.n_slices, s = cs % g.n_slices;
    const int d = g.d;
    const CamGroup cg0 = cam_group(g, c);
    const int npc = cg0.npc, kfp = cg0.kfp;
    const size_t ctok0 = (size_t)cg0.tok0 + (size_t)(c - cg0.cam0) * npc;   // camera c's first token
    const int crow0 = cg0.fp0 + (c - cg0.cam0) * kfp;                        // and first sample row
    const int col0 = s * cw;
    const T *x = reinterpret_cast<const T *>(g.x);
    const int active = g.cell->active;
    const int n_sp = g.n_rows * d;
    const int n_all = n_sp + g.V * d;
    const float *phi_prev = g.phi + (size_t)active * n_all;
    float *phi_next = g.phi + (size_t)(active ^ 1) * n_all;
    cg::cluster_group cluster = cg::this_cluster();

    // 1. column sums of rows [rb0, rb1) of camera c, columns [col0, col0 + cw),
    //    into rank 0's shared memory -- unless the previous block was skipped
    //    under lazy chaining (Section 2.2, reading c27): then the input is not
    //    materialised and its per-camera mean is the running chained mean
    const bool chained = g.chain && g.prev_flag != nullptr && *g.prev_flag == XC_DEC_SKIP;
    if (!chained)
        slice_colsums<T>(x, ctok0, d, col0, cw, r * g.rows_per, min(npc, r * g.rows_per + g.rows_per), r, red, call,
                         cluster);

    float p[GATE_PARTS] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    // 2. sample rows r, r + R, ... of camera c in this slice
    {
        const int n_mine = r < kfp ? (kfp - r + R - 1) / R : 0;
        for (int it = tid; it < n_mine * cw; it += GATE_THREADS) {
            const int i = r + (it / cw) * R, j = it % cw;
            const int row = g.fp_rows[crow0 + i];
            const size_t e = ((size_t)crow0 + i) * d + col0 + j;
            float cur;
            if (chained) {
                // chained input on the sampled rows: running fp32 sum of the last
                // materialised rows and the pending residuals, rounded once
                const float sum = g.csp_in[e] + to_f(reinterpret_cast<const T *>(g.rhat_prev)[(size_t)row * d + col0 + j]);
                g.csp_out[e] = sum;
                cur = round_to<T>(sum);
            } else {
                cur = to_f(x[(size_t)row * d + col0 + j]);
                if (g.chain) g.csp_out[e] = cur;
            }
            const float prev = phi_prev[e];
            phi_next[e] = cur;
            p[0] = fmaf(cur, prev, p[0]);
            p[1] = fmaf(cur, cur, p[1]);
            p[2] = fmaf(prev, prev, p[2]);
            p[3] = fmaxf(p[3], fabsf(cur - prev));
            p[4] += fabsf(prev);
        }
    }

    // 3. the R CTAs of (c, s) form one thread-block cluster; after the
    //    cluster barrier rank 0 holds every rank's column sums and adds them
    //    in rank order (the other ranks do not touch shared memory again)
    cluster.sync();
    if (r == 0) {
        for (int j = tid; j < cw; j += GATE_THREADS) {
            const size_t cm = (size_t)c * d + col0 + j;
            float mean;
            if (chained) {
                mean = g.cgm_in[cm] + g.rmean_prev[cm];      // mean(x_{j-1}) + sum of the residuals' means
            } else {
                float sum = call[0][j];
                for (int rr = 1; rr < R; ++rr) sum += call[rr][j];
                mean = sum / (float)npc;
            }
            if (g.chain) g.cgm_out[cm] = mean;
            const size_t e = (size_t)n_sp + cm;
            const float prev = phi_prev[e];
            phi_next[e] = mean;
            p[5] = fmaf(mean, prev, p[5]);
            p[6] = fmaf(mean, mean, p[6]);
            p[7] = fmaf(prev, prev, p[7]);
        }
    }
    cta_fold8(p, wpart, lane, warp, NW);
    if (tid == 0) {
        float4 *dst = reinterpret_cast<float4 *>(g.part + (size_t)blk * GATE_PARTS);
        dst[0] = make_float4(p[0], p[1], p[2], p[3]);
        dst[1] = make_float4(p[4], p[5], p[6], p[7]);
    }

    // 4. global ticket: the last CTA combines all partials and decides.  The
    //    partials are written by thread 0, which fences (release) before its
    //    ticket; the last CTA's thread 0 fences (acquire) before the barrier.
    if (tid == 0) {
        __threadfence();
        s_last = atomicAdd(g.ticket, 1u) == (unsigned)(gridDim.x - 1);
        if (s_last) __threadfence();
    }
    __syncthreads();
    if (!s_last) return;
    // Per view group: fold the partials of the group's CTAs (cameras
    // [g_cam0[q], g_cam0[q + 1]), every slice and row block) in CTA order;
    // thread 0 keeps the running min of the cosines and max of the deviations.
    float cos_min = INFINITY, dmax = 0.0f;
#pragma unroll
    for (int q = 0; q < XC_MAX_GROUPS; ++q) {
        if (q >= g.n_groups) break;
        const int b0 = g.g_cam0[q] * g.n_slices * R, b1 = g.g_cam0[q + 1] * g.n_slices * R;
        float v[GATE_PARTS] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
        for (int b = b0 + tid; b < b1; b += GATE_THREADS) {
            const float4 lo = __ldcg(reinterpret_cast<const float4 *>(g.part + (size_t)b * GATE_PARTS));
            const float4 hi = __ldcg(reinterpret_cast<const float4 *>(g.part + (size_t)b * GATE_PARTS + 4));
            v[0] += lo.x;
            v[1] += lo.y;
            v[2] += lo.z;
            v[3] = fmaxf(v[3], lo.w);
            v[4] += hi.x;
            v[5] += hi.y;
            v[6] += hi.z;
            v[7] += hi.w;
        }
        cta_fold8(v, wpart, lane, warp, NW);
        if (tid == 0) {
            const int n_sp_q = (g.g_cam0[q + 1] - g.g_cam0[q]) * g.g_kfp[q] * d;
            float dq = v[3] / (v[4] / (float)n_sp_q + g.eps_dev);
            if (isnan(dq)) dq = INFINITY;
            cos_min = fminf(cos_min, fminf(cos_rule_f(v[0], v[1], v[2]), cos_rule_f(v[5], v[6], v[7])));
            dmax = fmaxf(dmax, dq);
        }
        __syncthreads();
    }
    if (tid != 0) return;
    *g.ticket = 0u;

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
        g.phi_act[(active ^ 1) * 8 + i] = a;
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
        if (g.replay_dev != nullptr)
            skip = *g.replay_dev != 0;
        else if (g.replay >= 0)
            skip = g.replay != 0;
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

// Per-camera column means of a cached residual r_hat [L][d] (lazy chaining,
// reading c27): the same grid, streaming and cluster fold as the gate's
// global channel; rank 0 writes mean[c][col].  Runs after the block's FFN
// down-projection and exits at once unless the block computed.
template <typename T>
__global__ void __launch_bounds__(GATE_THREADS, GATE_CTAS_PER_SM) camera_mean_kernel(const GateArgs g) {
    pdl_wait();
    pdl_release();
    constexpr int VEC = 16 / sizeof(T);
    __shared__ float red[GATE_THREADS * VEC];
    __shared__ float call[GATE_MAX_CLUSTER][GATE_MAX_CW];
    if (g.flag != nullptr && *g.flag == XC_DEC_SKIP) return;     // uniform over the grid
    const int blk = blockIdx.x, R = g.R, cw = g.cw;
    const int r = blk % R, cs = blk / R;
    const int c = cs / g.n_slices, s = cs % g.n_slices;
    const CamGroup cg0 = cam_group(g, c);
    const size_t ctok0 = (size_t)cg0.tok0 + (size_t)(c - cg0.cam0) * cg0.npc;
    cg::cluster_group cluster = cg::this_cluster();
    slice_colsums<T>(reinterpret_cast<const T *>(g.x), ctok0, g.d, s * cw, cw, r * g.rows_per,
                     min(cg0.npc, r * g.rows_per + g.rows_per), r, red, call, cluster);
    cluster.sync();
    if (r == 0)
        for (int j = threadIdx.x; j < cw; j += GATE_THREADS) {
            float sum = call[0][j];
            for (int rr = 1; rr < R; ++rr) sum += call[rr][j];
            g.cam_mean_out[(size_t)c * g.d + s * cw + j] = sum / (float)cg0.npc;
        }
}

static size_t align256(size_t v) { return (v + 255) & ~(size_t)255; }

// Grid and scratch of one gate launch for V cameras of at most max_npc tokens
// each, d columns, on a device with n_sm SMs.  The row blocks R of one
// (camera, slice) form a thread-block cluster, so R <= GATE_MAX_CLUSTER.
// Scratch: 8 fp32 partials per CTA, then one 32-bit ticket (zero before the
// first launch; every launch leaves it zero).
GateGeom gate_geometry(int V, int max_npc, int d, int n_sm) {
    GateGeom gg;
    const int target = GATE_CTAS_PER_SM * (n_sm > 0 ? n_sm : 1);   // resident CTA slots
    const int most = (max_npc + 63) / 64;                  // at least 64 rows per row block
    // the widest slice (longest contiguous run of each row) that still gives
    // at least 5/8 of the resident slots with clusters of at most 8 row
    // blocks (measured at the 14B shape: 512 columns x 8 row blocks, 480 CTAs,
    // 37 us against 53 us for 256 x 5 = 600 CTAs, one nearly full wave)
    gg.cw = 64;
    for (int cw = GATE_MAX_CW; cw > 64; cw /= 2)
        if (d % cw == 0 && (long long)V * (d / cw) * std::min(GATE_MAX_CLUSTER, most) * 8 >= 5LL * target) {
            gg.cw = cw;
            break;
        }
    gg.n_slices = d / gg.cw;
    const int cs = V * gg.n_slices;
    int R = target / cs;
    if (R > most) R = most;
    if (R > GATE_MAX_CLUSTER) R = GATE_MAX_CLUSTER;
    gg.R = R < 1 ? 1 : R;
    gg.rows_per = (max_npc + gg.R - 1) / gg.R;
    gg.n_ctas = cs * gg.R;
    gg.tickets_off = align256((size_t)gg.n_ctas * GATE_PARTS * sizeof(float));
    gg.n_tickets = 1;
    gg.total = gg.tickets_off + 256;
    return gg;
}

void gate_bind_scratch(GateArgs &g, const GateGeom &gg, void *scratch) {
    char *w = reinterpret_cast<char *>(scratch);
    g.n_slices = gg.n_slices;
    g.cw = gg.cw;
    g.R = gg.R;
    g.rows_per = gg.rows_per;
    g.part = reinterpret_cast<float *>(w);
    g.ticket = reinterpret_cast<unsigned *>(w + gg.tickets_off);
}

template <typename T>
static cudaError_t cluster_launch(void (*kern)(GateArgs), const GateArgs &g, cudaStream_t st) {
    if (g.R < 1 || g.R > GATE_MAX_CLUSTER) return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(g.V * g.n_slices * g.R);
    cfg.blockDim = dim3(GATE_THREADS);
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = (unsigned)g.R;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kern, g);
}
template <typename T>
cudaError_t gate_launch(const GateArgs &g, cudaStream_t st) {
    return cluster_launch<T>(gate_kernel<T>, g, st);
}
template <typename T>
cudaError_t camera_mean_launch(const GateArgs &g, cudaStream_t st) {
    return cluster_launch<T>(camera_mean_kernel<T>, g, st);
}
template cudaError_t gate_launch<float>(const GateArgs &, cudaStream_t);
template cudaError_t gate_launch<bf16>(const GateArgs &, cudaStream_t);
template cudaError_t camera_mean_launch<float>(const GateArgs &, cudaStream_t);
template cudaError_t camera_mean_launch<bf16>(const GateArgs &, cudaStream_t);

static int current_sm_count() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) return 1;
    return n;
}

// Checks the arguments of one operator-level gate evaluation (xc_op_gate and
// xc_op_gate_static take the same ones) and packs them, scratch not bound.
// Returns XC_OK or XC_EINVAL with the reason in msg.
static xc_status gate_op_args(int dtype, int n_cams, int tokens_per_cam, int d, const void *x, const int *fp_rows,
                              int kfp, float *phi, float *phi_act, xc_gate_cell *cell, const float *action,
                              int action_dim, int mode, int step, const xc_gate_params *gate, uint8_t *flag,
                              float *s_cos, float *d_max, float *tau, GateArgs *out, char *msg, size_t msg_n) {
    if (dtype != XC_F32 && dtype != XC_BF16) {
        snprintf(msg, msg_n, "dtype");
        return XC_EINVAL;
    }
    if (n_cams < 1 || tokens_per_cam < 1 || d < 64 || d % 64 != 0 || kfp < 1 || kfp > tokens_per_cam ||
        action_dim < 1 || action_dim > 8 || (mode != 0 && mode != 1) || step < 0) {
        snprintf(msg, msg_n, "bad shape or mode (d %% 64 == 0, 1 <= kfp <= tokens_per_cam, action_dim <= 8)");
        return XC_EINVAL;
    }
    if (x == nullptr || fp_rows == nullptr || phi == nullptr || phi_act == nullptr || cell == nullptr ||
        action == nullptr || flag == nullptr || s_cos == nullptr || d_max == nullptr || tau == nullptr) {
        snprintf(msg, msg_n, "NULL pointer");
        return XC_EINVAL;
    }
    xc_gate_params p;
    if (gate != nullptr)
        p = *gate;
    else
        xc_gate_params_default(&p);
    if (!gate_ok(&p, 1, msg, msg_n)) return XC_EINVAL;
    GateArgs &g = *out;
    memset(&g, 0, sizeof g);
    g.x = x;
    g.d = d;
    gate_single_group(g, n_cams, tokens_per_cam, kfp);
    g.fp_rows = fp_rows;
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
    return XC_OK;
}

// ---------------------------------------------------------------------------
// Allocation-free gate (xc_op_gate_static).  The gate kernel needs scratch for
// its partial metrics, column sums and tickets.  Here that scratch is one
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
using xc::GateGeom;

extern "C" {

size_t xc_op_gate_workspace_bytes(int dtype, int n_cams, int tokens_per_cam, int d) {
    (void)dtype;
    if (n_cams < 1 || tokens_per_cam < 1 || d < 64 || d % 64 != 0) return 0;
    return xc::gate_geometry(n_cams, tokens_per_cam, d, xc::current_sm_count()).total;
}

static_assert(sizeof(xc_gate_cell) == sizeof(xc::GateCell), "gate cell layout");

xc_status xc_op_gate(int dtype, int n_cams, int tokens_per_cam, int d, const void *x, const int *fp_rows, int kfp,
                     float *phi, float *phi_act, xc_gate_cell *cell, const float *action, int action_dim, int mode,
                     int step, const xc_gate_params *gate, uint8_t *flag, float *s_cos, float *d_max, float *tau,
                     void *workspace, size_t workspace_bytes, void *stream) {
    char why[200], msg[256];
    GateArgs g;
    xc_status st = xc::gate_op_args(dtype, n_cams, tokens_per_cam, d, x, fp_rows, kfp, phi, phi_act, cell, action,
                                    action_dim, mode, step, gate, flag, s_cos, d_max, tau, &g, why, sizeof why);
    if (st == XC_OK && workspace == nullptr) {
        snprintf(why, sizeof why, "NULL workspace");
        st = XC_EINVAL;
    }
    const GateGeom gg = xc::gate_geometry(n_cams, tokens_per_cam, d, xc::current_sm_count());
    if (st == XC_OK && workspace_bytes < gg.total) {
        snprintf(why, sizeof why, "workspace %zu bytes < %zu needed", workspace_bytes, gg.total);
        st = XC_EINVAL;
    }
    if (st != XC_OK) {
        snprintf(msg, sizeof msg, "xc_op_gate: %s", why);
        xc::set_global_error(msg);
        return st;
    }
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    xc::gate_bind_scratch(g, gg, workspace);
    cudaError_t e = cudaMemsetAsync(g.ticket, 0, sizeof(unsigned), s);
    if (e == cudaSuccess) e = dtype == XC_BF16 ? xc::gate_launch<xc::bf16>(g, s) : xc::gate_launch<float>(g, s);
    if (e != cudaSuccess) {
        snprintf(msg, sizeof msg, "xc_op_gate: %s", cudaGetErrorString(e));
        xc::set_global_error(msg);
        return XC_ECUDA;
    }
    return XC_OK;
}

xc_status xc_op_gate_static(int dtype, int n_cams, int tokens_per_cam, int d, const void *x, const int *fp_rows,
                            int kfp, float *phi, float *phi_act, xc_gate_cell *cell, const float *action,
                            int action_dim, int mode, int step, const xc_gate_params *gate, uint8_t *flag,
                            float *s_cos, float *d_max, float *tau, void *stream) {
    char why[200], msg[320];
    GateArgs g;
    const xc_status st = xc::gate_op_args(dtype, n_cams, tokens_per_cam, d, x, fp_rows, kfp, phi, phi_act, cell,
                                          action, action_dim, mode, step, gate, flag, s_cos, d_max, tau, &g, why,
                                          sizeof why);
    if (st != XC_OK) {
        snprintf(msg, sizeof msg, "xc_op_gate_static: %s", why);
        xc::set_global_error(msg);
        return st;
    }
    const GateGeom gg = xc::gate_geometry(n_cams, tokens_per_cam, d, xc::current_sm_count());
    if (gg.total > xc::GATE_STATIC_SCRATCH_BYTES) {
        snprintf(msg, sizeof msg,
                 "xc_op_gate_static: this geometry needs %zu bytes of scratch, more than the %zu-byte "
                 "static maximum (use xc_op_gate with a workspace)",
                 gg.total, xc::GATE_STATIC_SCRATCH_BYTES);
        xc::set_global_error(msg);
        return XC_EINVAL;
    }
    void *scratch = nullptr;
    if (xc::static_scratch(&scratch) != cudaSuccess) {
        xc::set_global_error("xc_op_gate_static: cudaGetSymbolAddress failed");
        return XC_ECUDA;
    }
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    xc::gate_bind_scratch(g, gg, scratch);
    // the tickets must start at zero; partials and column sums are overwritten
    cudaError_t e = cudaMemsetAsync(g.ticket, 0, sizeof(unsigned), s);
    if (e == cudaSuccess) e = dtype == XC_BF16 ? xc::gate_launch<xc::bf16>(g, s) : xc::gate_launch<float>(g, s);
    if (e != cudaSuccess) {
        snprintf(msg, sizeof msg, "xc_op_gate_static: %s", cudaGetErrorString(e));
        xc::set_global_error(msg);
        return XC_ECUDA;
    }
    return XC_OK;
}

}  // extern "C"
