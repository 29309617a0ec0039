// Host runtime of the X-Cache chunk step: the C ABI of include/xcache.h and
// include/xcache_ops.h.  Owns device memory for weights, the rolling KV ring,
// the per-(t, b) residual / fingerprint caches and scratch; sequences the
// kernels of one forward pass on the context's stream.  Gate decisions stay
// on the device: every recompute kernel of block b reads flag[b] and exits
// early when the gate chose reuse; the reuse kernel runs only then.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "xc_kernels.cuh"


using namespace xc;

// ------------------------------------------------------------------ helpers
namespace {

std::mutex g_err_mu;
std::string g_global_err = "no error";

struct Fail {
    xc_status st;
};

// RoPE pair table: head_dim split hd/8 (camera) : 3hd/8 (absolute frame) :
// hd/4 (h) : hd/4 (w); pair j of an axis with D dims rotates at theta^(-2j/D).
// For the per-chunk (cos, sin) table (rope_table_kernel): the axis of every
// pair and the table entry of its position 0; npos = positions per axis
// (cameras, frames per chunk, h, w).  Returns the number of table entries.
int rope_layout(int hd, const int npos[4], std::vector<int> &axis, std::vector<int> &off) {
    const int dims[4] = {hd / 8, 3 * hd / 8, hd / 4, hd / 4};
    axis.clear();
    off.clear();
    int base = 0;
    for (int a = 0; a < 4; ++a)
        for (int j = 0; j < dims[a] / 2; ++j) {
            axis.push_back(a);
            off.push_back(base);
            base += npos[a];
        }
    return base;
}

// 1-D fallback of the spatial sample (Section 2.3.1): K uniformly spaced,
// cell-centred indices floor((2j+1) N / (2K)) along each camera's N tokens,
// every token when N <= K.
std::vector<int> linear_rows(int V, long long N, int K, int *kfp) {
    std::vector<int> rows;
    const int k = N <= K ? (int)N : K;
    *kfp = k;
    for (int c = 0; c < V; ++c)
        for (int j = 0; j < k; ++j)
            rows.push_back((int)(c * N + (N <= K ? j : ((2LL * j + 1) * N) / (2LL * K))));
    return rows;
}

// Spatial sample of the fingerprint (Section 2.3.1): per axis
// k_a = clamp(floor(dim_a * (K / (F H W))^(1/3)), 1, dim_a), taken exactly as the
// largest k with k^3 * F*H*W <= K * dim_a^3; indices floor((2j+1) dim / (2k));
// Cartesian product per camera; cameras with <= K tokens keep every token.
std::vector<int> fingerprint_rows(int V, int Fr, int gh, int gw, int K, int *kfp) {
    const long long N = (long long)Fr * gh * gw;
    std::vector<int> rows;
    if (N <= K) {
        *kfp = (int)N;
        for (int c = 0; c < V; ++c)
            for (long long i = 0; i < N; ++i) rows.push_back((int)(c * N + i));
        return rows;
    }
    const int dims[3] = {Fr, gh, gw};
    int k[3];
    for (int a = 0; a < 3; ++a) {
        long long kk = 0;
        const long long dm = dims[a];
        while (kk + 1 <= dm && (kk + 1) * (kk + 1) * (kk + 1) * N <= (long long)K * dm * dm * dm) ++kk;
        if (kk < 1) kk = 1;
        k[a] = (int)kk;
    }
    *kfp = k[0] * k[1] * k[2];
    for (int c = 0; c < V; ++c)
        for (int i = 0; i < k[0]; ++i) {
            const int f = (int)(((2LL * i + 1) * Fr) / (2LL * k[0]));
            for (int j = 0; j < k[1]; ++j) {
                const int h = (int)(((2LL * j + 1) * gh) / (2LL * k[1]));
                for (int l = 0; l < k[2]; ++l) {
                    const int w = (int)(((2LL * l + 1) * gw) / (2LL * k[2]));
                    rows.push_back((int)(c * N + ((long long)f * gh + h) * gw + w));
                }
            }
        }
    return rows;
}

bool is_host_ptr(const void *p) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return true;
    }
    return a.type == cudaMemoryTypeHost || a.type == cudaMemoryTypeUnregistered;
}

}  // namespace

// Everything the per-pass block loop takes from the host (besides buffers
// that stay fixed for the context's lifetime).
struct PassSig {
    int t, kv, eval_mode, slot, n_keys, replay, n_ctx, want_v;
    uint64_t replay_bits;
    xc_gate_params p;                 // replay_skip pointer cleared
    const void *lat, *v, *trace;
};
struct GraphEntry {
    PassSig sig;
    cudaGraphExec_t exec;
    long long launches;
};

struct xc_ctx {
    xc_model_cfg cfg;
    int L, d, F, B, S, H, hd, Wkv, C, A, V;
    bool bf;
    size_t esz;
    cudaStream_t st;
    int n_sm;
    std::vector<void *> allocs;

    // weights
    float *pe_w, *pe_b, *t_w1, *t_b1, *t_w2, *t_b2, *a_w1, *a_b1, *a_w2, *a_b2;
    float *mod_w, *mod_b, *blk_mod, *head_w, *head_b, *head_tab, *out_w, *out_b;
    void *qkv_wt, *o_wt, *f1_wt, *f2_wt;      // [B][N][K] activation dtype
    float *qkv_b, *o_b, *f1_b, *f2_b;          // [B][N]
    int *rope_axis, *rope_off;                 // per pair
    float2 *rope_cs;                           // per-chunk (cos, sin) table
    int rope_n, rope_h, rope_w;               // table extent (largest grid of the view groups)

    // activations / conditioning
    void *xb[2], *x1, *hbuf, *q, *o, *u;
    float *lat, *vout;
    float *ht, *ha, *e, *mods, *hmod;

    // rolling KV ring [B][Wkv][L][d] and caches
    void *ring_k, *ring_v;
    void *rhat;                                // [S][B][L][d]
    float *phi;                                // [S][B][2][n_all]
    float *phi_act;                            // [S][B][2][8]
    GateCell *cells;                           // [S][B]
    int *fp_rows;                              // sample rows, group by group, camera by camera
    int fp_K, fp_lin, n_rows;
    int g_kfp[XC_MAX_GROUPS], g_fp0[XC_MAX_GROUPS];
    size_t phi_n_all;

    // view groups (Section 2.3.1): cameras [g_cam0[g], g_cam0[g+1]) of grid
    // g_gh[g] x g_gw[g], tokens from g_tok0[g]
    int G;
    int g_cam0[XC_MAX_GROUPS + 1], g_tok0[XC_MAX_GROUPS], g_npc[XC_MAX_GROUPS], g_gh[XC_MAX_GROUPS],
        g_gw[XC_MAX_GROUPS];

    // KV-update chunks (Section 2.5 (3)): period (0 = every chunk) and the
    // number of KV-update passes so far (the ring's write count)
    int kv_period, kvc;

    // cross-attention conditioning (d_ctx > 0): per-block weights, the
    // current condition tokens and their per-block keys / values
    bool xattn;
    int d_ctx, max_ctx, n_ctx;                 // n_ctx: current condition tokens (0 = none yet)
    float *ca_scale, *ca_shift;                // [B][d] gamma - 1 and beta (LN affine run as ln_mod)
    void *ca_q_wt, *ca_kv_wt, *ca_o_wt;        // [B][d][d], [B][2d][d_ctx], [B][d][d] activation dtype
    float *ca_q_b, *ca_kv_b, *ca_o_b;          // [B][d], [B][2d], [B][d]
    float *ones;                               // [d] gate of the ungated residual epilogue
    float *ctx_in;                             // [max_ctx][d_ctx] fp32 staging
    void *ctx_act;                             // [max_ctx][d_ctx] bf16 copy (bf16 models)
    void *ctx_k, *ctx_v;                       // [B][max_ctx][d] condition keys / values

    // per pass
    uint8_t *flags;
    float *s_cos, *d_max, *tau;
    uint8_t *h_flags;
    float *h_stats;                            // pinned [3][B]
    int *d_err;

    // lazy residual chaining: per-camera means of every cached residual
    // [S][B][V][d]; running chained sample rows [2][n_rows][d] and means
    // [2][V][d] of the current pass; the chain setting of the last pass
    float *rmean, *chain_sp, *chain_gm;
    int chain_last;

    // gate scratch (grid and layout in g_geom)
    GateGeom g_geom;
    char *g_scratch;

    // attention split workspace (partials of units cut between CTAs)
    void *attn_ws;
    size_t attn_ws_bytes;

    // device copy of the chunk's action (written by the conditioning kernel)
    float *act_dev;

    // CUDA graphs of the per-pass block loop, keyed by everything the loop
    // takes from the host (see PassSig).  The context's first pass runs
    // directly (one-time kernel set-up such as shared-memory attributes
    // happens outside any capture); every later new signature is captured.
    std::vector<struct GraphEntry> graphs;
    bool graphs_on;
    bool warm;
    cudaStream_t cap_st;                       // capture stream (the caller's may be the legacy default)

    // tensor maps (bf16); output tile width of each GEMM
    CUtensorMap tm_h, tm_o, tm_u, tm_q;
    int bn_qkv, bn_o, bn_f1, bn_f2;
    std::vector<CUtensorMap> tm_wqkv, tm_wo, tm_w1, tm_w2, tm_rk, tm_rv;
    std::vector<CUtensorMap> tm_caq, tm_cao, tm_cak, tm_cav, tm_ck, tm_cv;   // cross-attention

    int n, next_step;
    void *trace;
    std::string err;

    // measurement: launch counter, optional per-launch CUDA events
    long long launches;
    bool prof_on;
    unsigned prof_mask;
    int prof_cap, prof_n, pass_seq, cur_keys;
    std::vector<cudaEvent_t> prof_ev;
    std::vector<xc_profile_rec> prof_rec;
    uint8_t *dec_log;                          // device [prof_cap][B]
};

namespace {

void set_err(xc_ctx *c, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (c != nullptr) c->err = buf;
    std::lock_guard<std::mutex> g(g_err_mu);
    g_global_err = buf;
}

}  // namespace

void xc::set_global_error(const char *msg) { set_err(nullptr, "%s", msg); }

bool xc::gate_ok(const xc_gate_params *p, int B, char *why, size_t n) {
    auto bad = [&](const char *m) { snprintf(why, n, "invalid gate params: %s", m); return false; };
    const float f[] = {p->tau_floor, p->margin, p->alpha, p->tau_dev, p->eps_dev, p->step0_strict_tau};
    for (float v : f)
        if (std::isnan(v)) return bad("NaN threshold");
    if (p->alpha < 0.0f || p->alpha > 1.0f) return bad("alpha out of [0, 1]");
    if (p->front_anchors < 0 || p->back_anchors < 0 || p->warmup_chunks < 0 || p->max_skips < 0)
        return bad("negative count");
    if (p->fp_tokens < 1) return bad("fp_tokens < 1");
    if (p->fp_refresh != 0 && p->fp_refresh != 1) return bad("fp_refresh must be 0 or 1");
    if (p->fp_linear != 0 && p->fp_linear != 1) return bad("fp_linear must be 0 or 1");
    if (p->chain != 0 && p->chain != 1) return bad("chain must be 0 or 1");
    (void)B;
    return true;
}

namespace {

#define CK(call)                                                                            \
    do {                                                                                    \
        cudaError_t e_ = (call);                                                            \
        if (e_ != cudaSuccess) {                                                            \
            set_err(ctx, "%s failed: %s (%s:%d)", #call, cudaGetErrorString(e_), __FILE__, __LINE__); \
            throw Fail{e_ == cudaErrorMemoryAllocation ? XC_ENOMEM : XC_ECUDA};             \
        }                                                                                   \
    } while (0)

// Test hook (xc_debug_fail_alloc): when positive, the device allocation that
// brings the count to zero fails as if the device were out of memory.
std::atomic<int> g_fail_alloc{0};

void maybe_fail_alloc(xc_ctx *ctx) {
    int n = g_fail_alloc.load();
    while (n > 0 && !g_fail_alloc.compare_exchange_weak(n, n - 1)) {
    }
    if (n == 1) {
        set_err(ctx, "device allocation failed (injected by xc_debug_fail_alloc)");
        throw Fail{XC_ENOMEM};
    }
}

template <typename P>
P *dalloc(xc_ctx *ctx, size_t bytes) {
    void *p = nullptr;
    maybe_fail_alloc(ctx);
    CK(cudaMalloc(&p, bytes < 16 ? 16 : bytes));
    ctx->allocs.push_back(p);
    return reinterpret_cast<P *>(p);
}

// Host or device source: cudaMemcpyDefault classifies the pointer (unified addressing).
void upload(xc_ctx *ctx, float *dst, const float *src, size_t n) {
    CK(cudaMemcpy(dst, src, n * sizeof(float), cudaMemcpyDefault));
}

bool cfg_ok(const xc_model_cfg *c, char *why, size_t n) {
    auto bad = [&](const char *m) { snprintf(why, n, "invalid model cfg: %s", m); return false; };
    if (c->n_blocks < 1 || c->n_blocks > XC_MAX_BLOCKS) return bad("n_blocks out of [1, 64]");
    if (c->d_model < 16 || c->n_heads < 1 || c->head_dim < 16) return bad("sizes too small");
    if (c->n_heads * c->head_dim != c->d_model) return bad("d_model != n_heads * head_dim");
    if (c->head_dim % 16 != 0) return bad("head_dim % 16 != 0");
    if (c->d_model % 64 != 0 || c->d_ffn % 16 != 0 || c->d_ffn < 16) return bad("d_model % 64 or d_ffn % 16");
    if (c->c_latent != 16) return bad("c_latent must be 16");
    if (c->action_dim < 1 || c->action_dim > 8) return bad("action_dim out of [1, 8]");
    if (c->n_groups < 0 || c->n_groups > XC_MAX_GROUPS) return bad("n_groups out of [0, XC_MAX_GROUPS]");
    if (c->n_cams < 1 || c->frames < 1) return bad("empty latent grid");
    long long tokens = 0;
    if (c->n_groups == 0) {
        if (c->grid_h < 1 || c->grid_w < 1) return bad("empty latent grid");
        tokens = (long long)c->n_cams * c->frames * c->grid_h * c->grid_w;
    } else {
        long long cams = 0;
        for (int g = 0; g < c->n_groups; ++g) {
            if (c->group_cams[g] < 1 || c->group_h[g] < 1 || c->group_w[g] < 1) return bad("empty view group");
            cams += c->group_cams[g];
            tokens += (long long)c->group_cams[g] * c->frames * c->group_h[g] * c->group_w[g];
            if (tokens > (1LL << 24)) break;
        }
        if (cams != c->n_cams) return bad("n_cams != sum of group_cams");
    }
    if (tokens > (1LL << 24)) return bad("chunk too large");
    if (c->kv_period < 0) return bad("kv_period < 0");
    if (c->kv_window_chunks < 1 || c->n_denoise_steps < 1 || c->n_denoise_steps > 64) return bad("window / steps");
    if (c->t_freq_dim < 2 || c->t_freq_dim % 2 != 0 || c->t_freq_dim > COND_TEMB_MAX)
        return bad("t_freq_dim must be even and at most 512");
    if (!(c->ln_eps > 0.0f) || !(c->rope_theta > 1.0f)) return bad("ln_eps / rope_theta");
    if (c->dtype == XC_BF16) {
        if (c->head_dim != 64 && c->head_dim != 128) return bad("bf16 needs head_dim 64 or 128");
        if (c->d_model % 256 != 0 || c->d_ffn % 256 != 0) return bad("bf16 needs d_model, d_ffn % 256 == 0");
    } else if (c->dtype == XC_F32) {
        if (c->head_dim > 64) return bad("f32 path supports head_dim 16, 32, 64");
        if (c->head_dim != 16 && c->head_dim != 32 && c->head_dim != 64) return bad("f32 head_dim");
    } else {
        return bad("dtype must be XC_F32 or XC_BF16");
    }
    if (c->d_ctx < 0 || c->max_ctx < 0) return bad("d_ctx / max_ctx < 0");
    if (c->d_ctx > 0) {
        if (c->max_ctx < 1) return bad("cross-attention needs max_ctx >= 1");
        if (c->d_ctx % 16 != 0) return bad("d_ctx % 16 != 0");
        if (c->dtype == XC_BF16 && c->d_ctx % 64 != 0) return bad("bf16 cross-attention needs d_ctx % 64 == 0");
        if ((long long)c->max_ctx * c->d_ctx > (1LL << 28) || c->max_ctx > (1 << 24)) return bad("context too large");
    }
    return true;
}

// (Re)build the spatial sample for a token budget K; resets every gate cell.
void drop_graphs(xc_ctx *ctx) {
    for (GraphEntry &e : ctx->graphs) cudaGraphExecDestroy(e.exec);
    ctx->graphs.clear();
}

void ensure_fp(xc_ctx *ctx, int K, int linear) {
    if (ctx->fp_K == K && ctx->fp_lin == linear) return;
    std::vector<int> rows;
    for (int g = 0; g < ctx->G; ++g) {
        const int Vg = ctx->g_cam0[g + 1] - ctx->g_cam0[g];
        int kfp = 0;
        std::vector<int> r = linear ? linear_rows(Vg, ctx->g_npc[g], K, &kfp)
                                    : fingerprint_rows(Vg, ctx->cfg.frames, ctx->g_gh[g], ctx->g_gw[g], K, &kfp);
        ctx->g_fp0[g] = (int)rows.size();
        ctx->g_kfp[g] = kfp;
        for (int v : r) rows.push_back(v + ctx->g_tok0[g]);
    }
    const size_t n_all = rows.size() * (size_t)ctx->d + (size_t)ctx->V * ctx->d;
    if (ctx->fp_rows != nullptr) {
        CK(cudaStreamSynchronize(ctx->st));
        drop_graphs(ctx);                        // the captured passes point at the old buffers
        for (auto it = ctx->allocs.begin(); it != ctx->allocs.end();) {
            if (*it == ctx->fp_rows || *it == ctx->phi || *it == ctx->chain_sp) {
                cudaFree(*it);
                it = ctx->allocs.erase(it);
            } else {
                ++it;
            }
        }
    }
    ctx->fp_rows = dalloc<int>(ctx, rows.size() * sizeof(int));
    CK(cudaMemcpy(ctx->fp_rows, rows.data(), rows.size() * sizeof(int), cudaMemcpyHostToDevice));
    ctx->phi = dalloc<float>(ctx, (size_t)ctx->S * ctx->B * 2 * n_all * sizeof(float));
    ctx->chain_sp = dalloc<float>(ctx, 2 * rows.size() * (size_t)ctx->d * sizeof(float));
    CK(cudaMemsetAsync(ctx->phi, 0, (size_t)ctx->S * ctx->B * 2 * n_all * sizeof(float), ctx->st));
    CK(cudaMemsetAsync(ctx->cells, 0, (size_t)ctx->S * ctx->B * sizeof(GateCell), ctx->st));
    CK(cudaMemsetAsync(ctx->phi_act, 0, (size_t)ctx->S * ctx->B * 16 * sizeof(float), ctx->st));
    ctx->n_rows = (int)rows.size();
    ctx->phi_n_all = n_all;
    ctx->fp_K = K;
    ctx->fp_lin = linear;
}

// Chunk n has a KV-update pass (always when kv_period = 0).
bool kv_chunk(const xc_ctx *ctx, int n) { return ctx->kv_period == 0 || n % ctx->kv_period == ctx->kv_period - 1; }

// The gate is evaluated on denoising pass t of the current chunk: past the
// warmup chunks, not a protected step 0, not a force-compute (KV-update)
// chunk of a periodic schedule.
bool eval_pass(const xc_ctx *ctx, const xc_gate_params &p, int t) {
    const int n = ctx->n;
    return n >= p.warmup_chunks && !(p.protect_step0 && t == 0) && !(ctx->kv_period > 0 && kv_chunk(ctx, n));
}

void clear_state(xc_ctx *ctx) {
    const size_t ring = (size_t)ctx->B * ctx->Wkv * ctx->L * ctx->d * ctx->esz;
    CK(cudaMemsetAsync(ctx->ring_k, 0, ring, ctx->st));
    CK(cudaMemsetAsync(ctx->ring_v, 0, ring, ctx->st));
    CK(cudaMemsetAsync(ctx->rhat, 0, (size_t)ctx->S * ctx->B * ctx->L * ctx->d * ctx->esz, ctx->st));
    CK(cudaMemsetAsync(ctx->cells, 0, (size_t)ctx->S * ctx->B * sizeof(GateCell), ctx->st));
    CK(cudaMemsetAsync(ctx->phi_act, 0, (size_t)ctx->S * ctx->B * 16 * sizeof(float), ctx->st));
    if (ctx->phi != nullptr)
        CK(cudaMemsetAsync(ctx->phi, 0, (size_t)ctx->S * ctx->B * 2 * ctx->phi_n_all * sizeof(float), ctx->st));
    CK(cudaMemsetAsync(ctx->g_scratch + ctx->g_geom.tickets_off, 0, ctx->g_geom.n_tickets * sizeof(unsigned),
                       ctx->st));
    CK(cudaStreamSynchronize(ctx->st));
    ctx->n = 0;
    ctx->kvc = 0;
    ctx->next_step = 0;
}

// Per-block weight upload: W [K][N] float32 (host) -> Wt [N][K] activation dtype.
void upload_blocks(xc_ctx *ctx, void *dst, const float *src, int K, int N, float *tmp) {
    for (int b = 0; b < ctx->B; ++b) {
        CK(cudaMemcpy(tmp, src + (size_t)b * K * N, (size_t)K * N * sizeof(float), cudaMemcpyDefault));
        char *out = reinterpret_cast<char *>(dst) + (size_t)b * K * N * ctx->esz;
        if (ctx->bf)
            CK(transpose_convert<bf16>(tmp, reinterpret_cast<bf16 *>(out), K, N, ctx->st));
        else
            CK(transpose_convert<float>(tmp, reinterpret_cast<float *>(out), K, N, ctx->st));
        CK(cudaStreamSynchronize(ctx->st));
    }
}

void tmap(xc_ctx *ctx, CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint32_t box) {
    if (!make_tmap_bf16(m, base, rows, cols, box)) {
        set_err(ctx, "cuTensorMapEncodeTiled failed (rows %llu cols %llu)", (unsigned long long)rows,
                (unsigned long long)cols);
        throw Fail{XC_ECUDA};
    }
}

// Profiling hooks: an event pair around one launch when its kind is selected.
int prof_begin(xc_ctx *ctx, int kind, int block) {
    if (!ctx->prof_on || !(ctx->prof_mask & (1u << kind)) || ctx->prof_n >= ctx->prof_cap) return -1;
    const int i = ctx->prof_n++;
    CK(cudaEventRecord(ctx->prof_ev[2 * i], ctx->st));
    xc_profile_rec &r = ctx->prof_rec[i];
    r.kind = kind;
    r.block = block;
    r.pass_seq = ctx->pass_seq;
    r.decision = -1;
    r.chunk = ctx->n;
    r.n_keys = kind == XC_K_XATTN ? ctx->n_ctx : ctx->cur_keys;
    r.ms = 0.0f;
    return i;
}
void prof_end(xc_ctx *ctx, int i) {
    if (i >= 0) CK(cudaEventRecord(ctx->prof_ev[2 * i + 1], ctx->st));
}

// Launch `call` (n_launch kernels) with optional events and the launch count.
#define LAUNCH(kind, block, n_launch, call)        \
    do {                                           \
        const int pi_ = prof_begin(ctx, kind, block); \
        CK(call);                                  \
        prof_end(ctx, pi_);                        \
        ctx->launches += (n_launch);               \
    } while (0)

// Replays the graph of `sig`, or captures `body` into a new one and
// replays it (the context's very first pass runs directly instead).
template <typename F>
void run_graph(xc_ctx *ctx, const PassSig &sig, F &&body) {
    auto same = [&](const PassSig &a) { return memcmp(&a, &sig, sizeof sig) == 0; };
    for (GraphEntry &e : ctx->graphs)
        if (same(e.sig)) {
            CK(cudaGraphLaunch(e.exec, ctx->st));
            ctx->launches += e.launches;
            return;
        }
    if (!ctx->warm) {
        body(ctx->st);
        ctx->warm = true;
        return;
    }
    if (ctx->graphs.size() >= 128) drop_graphs(ctx);
    const long long l0 = ctx->launches;
    CK(cudaStreamBeginCapture(ctx->cap_st, cudaStreamCaptureModeThreadLocal));
    cudaGraph_t g = nullptr;
    try {
        body(ctx->cap_st);
    } catch (...) {
        cudaStreamEndCapture(ctx->cap_st, &g);
        if (g != nullptr) cudaGraphDestroy(g);
        ctx->launches = l0;
        throw;
    }
    CK(cudaStreamEndCapture(ctx->cap_st, &g));
    cudaGraphExec_t ex = nullptr;
    const cudaError_t e = cudaGraphInstantiate(&ex, g, 0);
    cudaGraphDestroy(g);
    CK(e);
    const long long n = ctx->launches - l0;
    ctx->launches = l0;
    ctx->graphs.push_back(GraphEntry{sig, ex, n});
    CK(cudaGraphLaunch(ex, ctx->st));
    ctx->launches += n;
}

template <typename T>
void run_pass(xc_ctx *ctx, const float *lat_dev, const float *action, float sigma, int t, bool kv,
              const xc_gate_params &p, float *v_dev, bool want_v) {
    const int L = ctx->L, d = ctx->d, F = ctx->F, B = ctx->B, hd = ctx->hd;
    cudaStream_t st = ctx->st;
    const size_t Ld = (size_t)L * d;
    const int n = ctx->n;
    // ring: the clean K/V of the last Wkv - 1 KV-update chunks plus this
    // chunk's own, written to the slot the next KV-update pass fills
    const int slot = ctx->kvc % ctx->Wkv;
    const int n_res = (ctx->kvc + 1 < ctx->Wkv ? ctx->kvc + 1 : ctx->Wkv);
    const int n_keys = n_res * L;
    ctx->cur_keys = n_keys;

    // conditioning c_t: timestep + action embeddings -> adaLN-Zero vectors
    {
        CondArgs ca{};
        // sinusoid of the flow time 1000 sigma: [cos(s f_i), sin(s f_i)],
        // f_i = 10000^(-i/half), in double precision (angles reach 1000 rad)
        const int half = ctx->cfg.t_freq_dim / 2;
        for (int i = 0; i < half; ++i) {
            const double a = 1000.0 * (double)sigma * std::exp(-std::log(10000.0) * (double)i / (double)half);
            ca.temb[i] = (float)std::cos(a);
            ca.temb[half + i] = (float)std::sin(a);
        }
        for (int i = 0; i < ctx->A; ++i) ca.act[i] = action[i];
        ca.A = ctx->A;
        ca.tf = ctx->cfg.t_freq_dim;
        ca.d = d;
        ca.B = B;
        ca.t_w1 = ctx->t_w1; ca.t_b1 = ctx->t_b1; ca.a_w1 = ctx->a_w1; ca.a_b1 = ctx->a_b1;
        ca.t_w2 = ctx->t_w2; ca.t_b2 = ctx->t_b2; ca.a_w2 = ctx->a_w2; ca.a_b2 = ctx->a_b2;
        ca.mod_w = ctx->mod_w; ca.mod_b = ctx->mod_b; ca.blk_mod = ctx->blk_mod;
        ca.head_w = ctx->head_w; ca.head_b = ctx->head_b; ca.head_tab = ctx->head_tab;
        ca.ht = ctx->ht; ca.ha = ctx->ha; ca.e = ctx->e; ca.mods = ctx->mods; ca.hmod = ctx->hmod;
        ca.act_out = ctx->act_dev;
        LAUNCH(XC_K_COND, -1, 3, conditioning(ca, st));
    }
    // RoPE table of this chunk (absolute frames n*F .. n*F + F - 1)
    LAUNCH(XC_K_EMBED, -1, 1,
           rope_table(hd, (double)ctx->cfg.rope_theta, n * ctx->cfg.frames,
                      make_int4(ctx->V, ctx->cfg.frames, ctx->rope_h, ctx->rope_w), ctx->rope_cs,
                      ctx->rope_n, st));

    // Everything below takes from the host only what PassSig holds, so it is
    // captured into a CUDA graph and replayed for passes with the same
    // signature (the gate decisions are device-side, so a graph serves every
    // decision pattern).
    auto body = [&](cudaStream_t st) {

    T *X[2] = {reinterpret_cast<T *>(ctx->xb[0]), reinterpret_cast<T *>(ctx->xb[1])};
    // A KV-update pass whose velocity nobody reads (and with no block trace)
    // only needs every block's K/V: the last block stops after its K/V
    // projection and the head is not run.
    const bool kv_tail_off = kv && !want_v && ctx->trace == nullptr;
    LAUNCH(XC_K_EMBED, -1, 1, patch_embed<T>(lat_dev, ctx->pe_w, ctx->pe_b, X[0], L, ctx->C, d, st));
    CK(cudaMemsetAsync(ctx->flags, 0, B, st));
    CK(cudaMemsetAsync(ctx->s_cos, 0xFF, 3 * B * sizeof(float), st));   // NaN

    const bool gating = p.enabled != 0 && !kv;
    const bool eval_mode = eval_pass(ctx, p, t);
    // lazy residual chaining (reading c27); a block trace needs every block's
    // output written, so traced passes do not chain
    const bool chain = gating && p.chain != 0 && ctx->trace == nullptr;
    auto gated_at = [&](int b) { return gating && b >= p.front_anchors && b < B - p.back_anchors; };
    T *x1 = reinterpret_cast<T *>(ctx->x1);
    T *hb = reinterpret_cast<T *>(ctx->hbuf);
    T *qb = reinterpret_cast<T *>(ctx->q);
    T *ob = reinterpret_cast<T *>(ctx->o);
    T *ub = reinterpret_cast<T *>(ctx->u);

    for (int b = 0; b < B; ++b) {
        T *xin = X[b & 1], *xout = X[(b + 1) & 1];
        const uint8_t *flag = ctx->flags + b;
        const bool gated = gated_at(b);
        const float *mb = ctx->mods + (size_t)b * 6 * d;   // shift1 scale1 gate1 shift2 scale2 gate2
        T *rk = reinterpret_cast<T *>(ctx->ring_k) + ((size_t)b * ctx->Wkv + slot) * Ld;
        T *rv = reinterpret_cast<T *>(ctx->ring_v) + ((size_t)b * ctx->Wkv + slot) * Ld;
        T *rh = gated ? reinterpret_cast<T *>(ctx->rhat) + ((size_t)t * B + b) * Ld : nullptr;

        if (gated) {
            GateArgs g;
            memset(&g, 0, sizeof g);
            g.x = xin;
            g.d = d;
            g.V = ctx->V;
            g.fp_rows = ctx->fp_rows;
            g.n_groups = ctx->G;
            g.n_rows = ctx->n_rows;
            for (int q = 0; q < ctx->G; ++q) {
                g.g_cam0[q] = ctx->g_cam0[q];
                g.g_tok0[q] = ctx->g_tok0[q];
                g.g_npc[q] = ctx->g_npc[q];
                g.g_fp0[q] = ctx->g_fp0[q];
                g.g_kfp[q] = ctx->g_kfp[q];
            }
            g.g_cam0[ctx->G] = ctx->V;
            const size_t cell = (size_t)t * B + b;
            g.phi = ctx->phi + cell * 2 * ctx->phi_n_all;
            g.phi_act = ctx->phi_act + cell * 16;
            g.action_dev = ctx->act_dev;
            g.A = ctx->A;
            g.cell = ctx->cells + cell;
            g.mode = eval_mode ? 1 : 0;
            g.step = t;
            g.tau_floor = p.tau_floor;
            g.margin = p.margin;
            g.alpha = p.alpha;
            g.tau_dev = p.tau_dev;
            g.eps_dev = p.eps_dev;
            g.strict_tau = p.step0_strict_tau;
            g.max_skips = p.max_skips;
            g.fp_refresh = p.fp_refresh;
            g.replay = p.replay_skip != nullptr ? (p.replay_skip[b] != 0 ? 1 : 0) : -1;
            g.replay_dev = p.replay_table != nullptr ? p.replay_table + (size_t)t * B + b : nullptr;
            g.flag = ctx->flags + b;
            g.s_cos = ctx->s_cos + b;
            g.d_max = ctx->d_max + b;
            g.tau_out = ctx->tau + b;
            gate_bind_scratch(g, ctx->g_geom, ctx->g_scratch);
            if (chain) {
                const size_t nsp = (size_t)ctx->n_rows * d, nm = (size_t)ctx->V * d;
                g.chain = 1;
                g.prev_flag = b >= 1 && gated_at(b - 1) ? ctx->flags + b - 1 : nullptr;
                g.rhat_prev = b >= 1 ? reinterpret_cast<const T *>(ctx->rhat) + ((size_t)t * B + b - 1) * Ld : nullptr;
                g.rmean_prev = b >= 1 ? ctx->rmean + ((size_t)t * B + b - 1) * nm : nullptr;
                g.csp_in = ctx->chain_sp + (size_t)((b + 1) & 1) * nsp;
                g.csp_out = ctx->chain_sp + (size_t)(b & 1) * nsp;
                g.cgm_in = ctx->chain_gm + (size_t)((b + 1) & 1) * nm;
                g.cgm_out = ctx->chain_gm + (size_t)(b & 1) * nm;
            }
            LAUNCH(XC_K_GATE, b, 1, gate_launch<T>(g, st));
        }
        // lazy chaining: write the input of block b if the blocks before it were skipped
        if (chain && b >= 1)
            LAUNCH(XC_K_CHAIN, b, 1,
                   chain_apply<T>(X[0], X[1], reinterpret_cast<const T *>(ctx->rhat) + (size_t)t * B * Ld, ctx->flags,
                                  b, B, (long)Ld, ctx->n_sm, st));

        // ---- recompute path (early-exits when flag[b] == skip)
        LAUNCH(XC_K_LN, b, 1, ln_mod<T>(xin, mb + 0 * d, mb + 1 * d, hb, L, d, ctx->cfg.ln_eps, flag, st));
        EpiParams ep;
        memset(&ep, 0, sizeof ep);
        ep.M = L;
        ep.N = 3 * d;
        ep.bias = ctx->qkv_b + (size_t)b * 3 * d;
        ep.out = qb;
        ep.out_k = rk;
        ep.out_v = rv;
        ep.d = d;
        ep.head_dim = hd;
        ep.n_groups = ctx->G;
        for (int q = 0; q < ctx->G; ++q) {
            ep.g_tok0[q] = ctx->g_tok0[q];
            ep.g_cam0[q] = ctx->g_cam0[q];
            ep.g_npc[q] = ctx->g_npc[q];
            ep.g_gh[q] = ctx->g_gh[q];
            ep.g_gw[q] = ctx->g_gw[q];
        }
        ep.frames = ctx->cfg.frames;
        ep.frame0 = n * ctx->cfg.frames;
        ep.rope_axis = ctx->rope_axis;
        ep.rope_off = ctx->rope_off;
        ep.rope_cs = ctx->rope_cs;
        if constexpr (sizeof(T) == 2) {
            LAUNCH(XC_K_QKV, b, 1, gemm_tc(EPI_QKV_ROPE, ctx->bn_qkv, ctx->tm_h, ctx->tm_wqkv[b], ep, d, flag, ctx->d_err, st));
        } else {
            const float *W = reinterpret_cast<const float *>(ctx->qkv_wt) + (size_t)b * 3 * d * d;
            LAUNCH(XC_K_QKV, b, 1, gemm_simt(EPI_QKV_ROPE, ep, reinterpret_cast<const float *>(hb), W, d, flag, st));
        }
        if (kv_tail_off && b == B - 1) break;       // the ring has this block's K/V
        if constexpr (sizeof(T) == 2) {
            int n_attn = 1;
            LAUNCH(XC_K_ATTN, b, n_attn,
                   attn_tc(hd, ctx->tm_q, ctx->tm_rk[b], ctx->tm_rv[b], reinterpret_cast<bf16 *>(ob), L, n_keys,
                           ctx->H, d, ctx->attn_ws, ctx->attn_ws_bytes, flag, ctx->d_err, &n_attn, st));
        } else {
            const float *Kr = reinterpret_cast<const float *>(ctx->ring_k) + (size_t)b * ctx->Wkv * Ld;
            const float *Vr = reinterpret_cast<const float *>(ctx->ring_v) + (size_t)b * ctx->Wkv * Ld;
            LAUNCH(XC_K_ATTN, b, 1, attn_simt(hd, reinterpret_cast<const float *>(qb), Kr, Vr, reinterpret_cast<float *>(ob), L, n_keys,
                         ctx->H, flag, st));
        }
        // O projection + gated residual: x1 = x + gate1 * (o W_o + b_o)
        memset(&ep, 0, sizeof ep);
        ep.M = L;
        ep.N = d;
        ep.bias = ctx->o_b + (size_t)b * d;
        ep.gate = mb + 2 * d;
        ep.resid = xin;
        ep.out = x1;
        if constexpr (sizeof(T) == 2) {
            LAUNCH(XC_K_OPROJ, b, 1, gemm_tc(EPI_RESID_GATE, ctx->bn_o, ctx->tm_o, ctx->tm_wo[b], ep, d, flag, ctx->d_err, st));
        } else {
            const float *W = reinterpret_cast<const float *>(ctx->o_wt) + (size_t)b * d * d;
            LAUNCH(XC_K_OPROJ, b, 1, gemm_simt(EPI_RESID_GATE, ep, reinterpret_cast<const float *>(ob), W, d, flag, st));
        }
        if (ctx->xattn) {
            // cross-attention layer over the condition tokens, in place on x1:
            // x1 <- x1 + attn((LN(x1) gamma + beta) W_q + b_q, K_c, V_c) W_o + b_o
            const size_t cb = (size_t)b * ctx->max_ctx * d;
            LAUNCH(XC_K_XATTN, b, 1,
                   ln_mod<T>(x1, ctx->ca_shift + (size_t)b * d, ctx->ca_scale + (size_t)b * d, hb, L, d,
                             ctx->cfg.ln_eps, flag, st));
            memset(&ep, 0, sizeof ep);
            ep.M = L;
            ep.N = d;
            ep.bias = ctx->ca_q_b + (size_t)b * d;
            ep.out = qb;
            if constexpr (sizeof(T) == 2) {
                LAUNCH(XC_K_XATTN, b, 1,
                       gemm_tc(EPI_BIAS, ctx->bn_o, ctx->tm_h, ctx->tm_caq[b], ep, d, flag, ctx->d_err, st));
                int n_x = 1;
                LAUNCH(XC_K_XATTN, b, n_x,
                       attn_tc(hd, ctx->tm_q, ctx->tm_ck[b], ctx->tm_cv[b], reinterpret_cast<bf16 *>(ob), L,
                               ctx->n_ctx, ctx->H, d, ctx->attn_ws, ctx->attn_ws_bytes, flag, ctx->d_err, &n_x, st));
            } else {
                const float *W = reinterpret_cast<const float *>(ctx->ca_q_wt) + (size_t)b * d * d;
                LAUNCH(XC_K_XATTN, b, 1, gemm_simt(EPI_BIAS, ep, reinterpret_cast<const float *>(hb), W, d, flag, st));
                LAUNCH(XC_K_XATTN, b, 1,
                       attn_simt(hd, reinterpret_cast<const float *>(qb),
                                 reinterpret_cast<const float *>(ctx->ctx_k) + cb,
                                 reinterpret_cast<const float *>(ctx->ctx_v) + cb, reinterpret_cast<float *>(ob), L,
                                 ctx->n_ctx, ctx->H, flag, st));
            }
            memset(&ep, 0, sizeof ep);
            ep.M = L;
            ep.N = d;
            ep.bias = ctx->ca_o_b + (size_t)b * d;
            ep.gate = ctx->ones;
            ep.resid = x1;
            ep.out = x1;
            if constexpr (sizeof(T) == 2) {
                LAUNCH(XC_K_XATTN, b, 1,
                       gemm_tc(EPI_RESID_GATE, ctx->bn_o, ctx->tm_o, ctx->tm_cao[b], ep, d, flag, ctx->d_err, st));
            } else {
                const float *W = reinterpret_cast<const float *>(ctx->ca_o_wt) + (size_t)b * d * d;
                LAUNCH(XC_K_XATTN, b, 1,
                       gemm_simt(EPI_RESID_GATE, ep, reinterpret_cast<const float *>(ob), W, d, flag, st));
            }
        }
        LAUNCH(XC_K_LN, b, 1, ln_mod<T>(x1, mb + 3 * d, mb + 4 * d, hb, L, d, ctx->cfg.ln_eps, flag, st));
        // FFN up: u = GELU_tanh(h2 W1 + b1)
        memset(&ep, 0, sizeof ep);
        ep.M = L;
        ep.N = F;
        ep.bias = ctx->f1_b + (size_t)b * F;
        ep.out = ub;
        if constexpr (sizeof(T) == 2) {
            LAUNCH(XC_K_FFN1, b, 1, gemm_tc(EPI_GELU, ctx->bn_f1, ctx->tm_h, ctx->tm_w1[b], ep, d, flag, ctx->d_err, st));
        } else {
            const float *W = reinterpret_cast<const float *>(ctx->f1_wt) + (size_t)b * F * d;
            LAUNCH(XC_K_FFN1, b, 1, gemm_simt(EPI_GELU, ep, reinterpret_cast<const float *>(hb), W, d, flag, st));
        }
        // FFN down + gated residual; residual cache write r_hat = x2 - x (Eq. 2-3)
        memset(&ep, 0, sizeof ep);
        ep.M = L;
        ep.N = d;
        ep.bias = ctx->f2_b + (size_t)b * d;
        ep.gate = mb + 5 * d;
        ep.resid = x1;
        ep.xin = xin;
        ep.out = xout;
        ep.rhat = rh;
        if constexpr (sizeof(T) == 2) {
            LAUNCH(XC_K_FFN2, b, 1, gemm_tc(EPI_RESID_CACHE, ctx->bn_f2, ctx->tm_u, ctx->tm_w2[b], ep, F, flag, ctx->d_err, st));
        } else {
            const float *W = reinterpret_cast<const float *>(ctx->f2_wt) + (size_t)b * d * F;
            LAUNCH(XC_K_FFN2, b, 1, gemm_simt(EPI_RESID_CACHE, ep, reinterpret_cast<const float *>(ub), W, F, flag, st));
        }
        // ---- reuse path (Eq. 4), only when the gate chose skip; with lazy
        // chaining the skipped block writes nothing, and a computed gated
        // block records the per-camera means of its new residual
        if (gated && !chain) LAUNCH(XC_K_REUSE, b, 1, residual_reuse<T>(xin, rh, xout, (long)Ld, flag, ctx->n_sm, st));
        if (gated && chain) {
            GateArgs gm;
            memset(&gm, 0, sizeof gm);
            gm.x = rh;
            gm.d = d;
            gm.V = ctx->V;
            gm.n_groups = ctx->G;
            for (int q = 0; q < ctx->G; ++q) {
                gm.g_cam0[q] = ctx->g_cam0[q];
                gm.g_tok0[q] = ctx->g_tok0[q];
                gm.g_npc[q] = ctx->g_npc[q];
            }
            gm.g_cam0[ctx->G] = ctx->V;
            gate_bind_scratch(gm, ctx->g_geom, ctx->g_scratch);
            gm.flag = ctx->flags + b;
            gm.cam_mean_out = ctx->rmean + ((size_t)t * B + b) * (size_t)ctx->V * d;
            LAUNCH(XC_K_CHAIN, b, 1, camera_mean_launch<T>(gm, st));
        }
        if (ctx->trace != nullptr)
            CK(cudaMemcpyAsync(reinterpret_cast<char *>(ctx->trace) + (size_t)b * Ld * sizeof(T), xout,
                               Ld * sizeof(T), cudaMemcpyDeviceToDevice, st));
    }
    if (chain)
        LAUNCH(XC_K_CHAIN, -1, 1,
               chain_apply<T>(X[0], X[1], reinterpret_cast<const T *>(ctx->rhat) + (size_t)t * B * Ld, ctx->flags, B,
                              B, (long)Ld, ctx->n_sm, st));
    if (!kv_tail_off)
        LAUNCH(XC_K_HEAD, -1, 1, head<T>(X[B & 1], ctx->hmod, ctx->out_w, ctx->out_b, v_dev, L, d, ctx->cfg.ln_eps, st));
    };   // body

    if (ctx->prof_on || !ctx->graphs_on) {
        body(st);                                    // profiling records events per launch
    } else {
        PassSig sig;
        memset(&sig, 0, sizeof sig);
        sig.t = t;
        sig.kv = kv ? 1 : 0;
        sig.eval_mode = eval_pass(ctx, p, t) ? 1 : 0;
        sig.slot = slot;
        sig.n_keys = n_keys;
        sig.n_ctx = ctx->n_ctx;
        sig.want_v = want_v ? 1 : 0;
        sig.p = p;
        sig.p.replay_skip = nullptr;
        sig.replay = p.replay_skip != nullptr ? 1 : 0;
        if (p.replay_skip != nullptr)
            for (int b = 0; b < B; ++b)
                if (p.replay_skip[b]) sig.replay_bits |= 1ull << b;
        sig.lat = lat_dev;
        sig.v = v_dev;
        sig.trace = ctx->trace;
        run_graph(ctx, sig, body);
    }
    if (ctx->prof_on) {
        if (ctx->pass_seq < ctx->prof_cap)
            CK(cudaMemcpyAsync(ctx->dec_log + (size_t)ctx->pass_seq * B, ctx->flags, B, cudaMemcpyDeviceToDevice, st));
        ctx->pass_seq += 1;
    }
}

}  // namespace

// ======================================================================= ABI
extern "C" {

void xc_gate_params_default(xc_gate_params *p) {
    if (p == nullptr) return;
    memset(p, 0, sizeof *p);
    p->enabled = 1;
    p->tau_floor = 0.97f;
    p->margin = 0.02f;
    p->alpha = 0.30f;
    p->tau_dev = 2.0f;
    p->eps_dev = 1e-6f;
    p->front_anchors = 1;
    p->back_anchors = 0;
    p->warmup_chunks = 1;
    p->max_skips = 0;
    p->protect_step0 = 0;
    p->step0_strict_tau = 0.0f;
    p->fp_tokens = 32;
    p->fp_refresh = 0;
    p->replay_skip = nullptr;
    p->replay_table = nullptr;
}

const char *xc_last_error(const xc_ctx *ctx) {
    if (ctx != nullptr) return ctx->err.c_str();
    std::lock_guard<std::mutex> g(g_err_mu);
    return g_global_err.c_str();
}

static void prof_free(xc_ctx *ctx);

void xc_destroy(xc_ctx *ctx) {
    if (ctx == nullptr) return;
    cudaStreamSynchronize(ctx->st);
    drop_graphs(ctx);
    if (ctx->cap_st != nullptr) cudaStreamDestroy(ctx->cap_st);
    prof_free(ctx);
    for (void *p : ctx->allocs) cudaFree(p);
    if (ctx->h_flags) cudaFreeHost(ctx->h_flags);
    if (ctx->h_stats) cudaFreeHost(ctx->h_stats);
    delete ctx;
}

xc_status xc_init(const xc_model_cfg *cfg, const xc_weights *w, void *cuda_stream, xc_ctx **out) {
    xc_ctx *ctx = nullptr;
    if (out == nullptr || cfg == nullptr || w == nullptr) {
        set_err(nullptr, "xc_init: NULL argument");
        return XC_EINVAL;
    }
    *out = nullptr;
    char why[256];
    if (!cfg_ok(cfg, why, sizeof why)) {
        set_err(nullptr, "%s", why);
        return XC_EINVAL;
    }
    const float *const req[] = {w->pe_w, w->pe_b, w->t_w1, w->t_b1, w->t_w2, w->t_b2, w->a_w1, w->a_b1, w->a_w2,
                                w->a_b2, w->mod_w, w->mod_b, w->blk_mod, w->qkv_w, w->qkv_b, w->o_w, w->o_b,
                                w->f1_w, w->f1_b, w->f2_w, w->f2_b, w->head_w, w->head_b, w->head_tab, w->out_w,
                                w->out_b};
    for (const float *p : req)
        if (p == nullptr) {
            set_err(nullptr, "xc_init: NULL weight pointer");
            return XC_EINVAL;
        }
    if (cfg->d_ctx > 0) {
        const float *const req_ca[] = {w->ca_ln_w, w->ca_ln_b, w->ca_q_w, w->ca_q_b,
                                       w->ca_kv_w, w->ca_kv_b, w->ca_o_w, w->ca_o_b};
        for (const float *p : req_ca)
            if (p == nullptr) {
                set_err(nullptr, "xc_init: NULL cross-attention weight pointer");
                return XC_EINVAL;
            }
    }
    ctx = new xc_ctx();
    try {
        ctx->cfg = *cfg;
        ctx->B = cfg->n_blocks;
        ctx->d = cfg->d_model;
        ctx->F = cfg->d_ffn;
        ctx->H = cfg->n_heads;
        ctx->hd = cfg->head_dim;
        ctx->S = cfg->n_denoise_steps;
        ctx->Wkv = cfg->kv_window_chunks;
        ctx->C = cfg->c_latent;
        ctx->A = cfg->action_dim;
        ctx->V = cfg->n_cams;
        ctx->G = cfg->n_groups == 0 ? 1 : cfg->n_groups;
        ctx->L = 0;
        ctx->g_cam0[0] = 0;
        ctx->rope_h = ctx->rope_w = 1;
        for (int g = 0; g < ctx->G; ++g) {
            const int Vg = cfg->n_groups == 0 ? cfg->n_cams : cfg->group_cams[g];
            ctx->g_gh[g] = cfg->n_groups == 0 ? cfg->grid_h : cfg->group_h[g];
            ctx->g_gw[g] = cfg->n_groups == 0 ? cfg->grid_w : cfg->group_w[g];
            ctx->g_npc[g] = cfg->frames * ctx->g_gh[g] * ctx->g_gw[g];
            ctx->g_tok0[g] = ctx->L;
            ctx->g_cam0[g + 1] = ctx->g_cam0[g] + Vg;
            ctx->L += Vg * ctx->g_npc[g];
            ctx->rope_h = std::max(ctx->rope_h, ctx->g_gh[g]);
            ctx->rope_w = std::max(ctx->rope_w, ctx->g_gw[g]);
        }
        ctx->kv_period = cfg->kv_period;
        ctx->kvc = 0;
        ctx->bf = cfg->dtype == XC_BF16;
        ctx->esz = ctx->bf ? 2 : 4;
        ctx->st = reinterpret_cast<cudaStream_t>(cuda_stream);
        int dev = 0;
        CK(cudaGetDevice(&dev));
        CK(cudaDeviceGetAttribute(&ctx->n_sm, cudaDevAttrMultiProcessorCount, dev));
        const int L = ctx->L, d = ctx->d, F = ctx->F, B = ctx->B, C = ctx->C, A = ctx->A, Tf = cfg->t_freq_dim;
        const size_t Ld = (size_t)L * d, es = ctx->esz;

        // weights
        auto up = [&](float *&dst, const float *src, size_t n) {
            dst = dalloc<float>(ctx, n * sizeof(float));
            upload(ctx, dst, src, n);
        };
        up(ctx->pe_w, w->pe_w, (size_t)C * d);
        up(ctx->pe_b, w->pe_b, d);
        up(ctx->t_w1, w->t_w1, (size_t)Tf * d);
        up(ctx->t_b1, w->t_b1, d);
        up(ctx->t_w2, w->t_w2, (size_t)d * d);
        up(ctx->t_b2, w->t_b2, d);
        up(ctx->a_w1, w->a_w1, (size_t)A * d);
        up(ctx->a_b1, w->a_b1, d);
        up(ctx->a_w2, w->a_w2, (size_t)d * d);
        up(ctx->a_b2, w->a_b2, d);
        up(ctx->mod_w, w->mod_w, (size_t)d * 6 * d);
        up(ctx->mod_b, w->mod_b, 6 * (size_t)d);
        up(ctx->blk_mod, w->blk_mod, (size_t)B * 6 * d);
        up(ctx->head_w, w->head_w, (size_t)d * 2 * d);
        up(ctx->head_b, w->head_b, 2 * (size_t)d);
        up(ctx->head_tab, w->head_tab, 2 * (size_t)d);
        up(ctx->out_w, w->out_w, (size_t)d * C);
        up(ctx->out_b, w->out_b, C);
        up(ctx->qkv_b, w->qkv_b, (size_t)B * 3 * d);
        up(ctx->o_b, w->o_b, (size_t)B * d);
        up(ctx->f1_b, w->f1_b, (size_t)B * F);
        up(ctx->f2_b, w->f2_b, (size_t)B * d);
        ctx->qkv_wt = dalloc<void>(ctx, (size_t)B * 3 * d * d * es);
        ctx->o_wt = dalloc<void>(ctx, (size_t)B * d * d * es);
        ctx->f1_wt = dalloc<void>(ctx, (size_t)B * F * d * es);
        ctx->f2_wt = dalloc<void>(ctx, (size_t)B * d * F * es);
        ctx->xattn = cfg->d_ctx > 0;
        ctx->d_ctx = cfg->d_ctx;
        ctx->max_ctx = cfg->max_ctx;
        ctx->n_ctx = 0;
        if (ctx->xattn) {
            const size_t Bd = (size_t)B * d;
            std::vector<float> gm1(Bd);
            CK(cudaMemcpy(gm1.data(), w->ca_ln_w, Bd * sizeof(float), cudaMemcpyDefault));
            for (size_t i = 0; i < Bd; ++i) gm1[i] -= 1.0f;                  // exact for gains in [0.5, 2]
            up(ctx->ca_shift, w->ca_ln_b, Bd);
            up(ctx->ca_scale, gm1.data(), Bd);
            up(ctx->ca_q_b, w->ca_q_b, Bd);
            up(ctx->ca_kv_b, w->ca_kv_b, 2 * Bd);
            up(ctx->ca_o_b, w->ca_o_b, Bd);
            std::vector<float> one((size_t)d, 1.0f);
            up(ctx->ones, one.data(), d);
            ctx->ca_q_wt = dalloc<void>(ctx, Bd * d * es);
            ctx->ca_kv_wt = dalloc<void>(ctx, 2 * Bd * ctx->d_ctx * es);
            ctx->ca_o_wt = dalloc<void>(ctx, Bd * d * es);
            const size_t nc = (size_t)ctx->max_ctx * ctx->d_ctx;
            ctx->ctx_in = dalloc<float>(ctx, nc * sizeof(float));
            ctx->ctx_act = ctx->bf ? dalloc<void>(ctx, nc * es) : nullptr;
            ctx->ctx_k = dalloc<void>(ctx, Bd * ctx->max_ctx * es);
            ctx->ctx_v = dalloc<void>(ctx, Bd * ctx->max_ctx * es);
            CK(cudaMemset(ctx->ctx_k, 0, Bd * ctx->max_ctx * es));     // rows past n_ctx stay finite
            CK(cudaMemset(ctx->ctx_v, 0, Bd * ctx->max_ctx * es));
        }
        {
            size_t mx = (size_t)3 * d * d;
            if ((size_t)d * F > mx) mx = (size_t)d * F;
            if (ctx->xattn && (size_t)2 * d * ctx->d_ctx > mx) mx = (size_t)2 * d * ctx->d_ctx;
            float *tmp = nullptr;
            maybe_fail_alloc(ctx);
            CK(cudaMalloc(&tmp, mx * sizeof(float)));
            try {
                upload_blocks(ctx, ctx->qkv_wt, w->qkv_w, d, 3 * d, tmp);
                upload_blocks(ctx, ctx->o_wt, w->o_w, d, d, tmp);
                upload_blocks(ctx, ctx->f1_wt, w->f1_w, d, F, tmp);
                upload_blocks(ctx, ctx->f2_wt, w->f2_w, F, d, tmp);
                if (ctx->xattn) {
                    upload_blocks(ctx, ctx->ca_q_wt, w->ca_q_w, d, d, tmp);
                    upload_blocks(ctx, ctx->ca_kv_wt, w->ca_kv_w, ctx->d_ctx, 2 * d, tmp);
                    upload_blocks(ctx, ctx->ca_o_wt, w->ca_o_w, d, d, tmp);
                }
            } catch (...) {
                cudaFree(tmp);
                throw;
            }
            cudaFree(tmp);
        }
        {
            std::vector<int> ax, off;
            const int npos[4] = {cfg->n_cams, cfg->frames, ctx->rope_h, ctx->rope_w};
            ctx->rope_n = rope_layout(ctx->hd, npos, ax, off);
            ctx->rope_axis = dalloc<int>(ctx, ax.size() * sizeof(int));
            ctx->rope_off = dalloc<int>(ctx, off.size() * sizeof(int));
            ctx->rope_cs = dalloc<float2>(ctx, (size_t)ctx->rope_n * sizeof(float2));
            CK(cudaMemcpy(ctx->rope_axis, ax.data(), ax.size() * sizeof(int), cudaMemcpyHostToDevice));
            CK(cudaMemcpy(ctx->rope_off, off.data(), off.size() * sizeof(int), cudaMemcpyHostToDevice));
        }

        // activations
        ctx->xb[0] = dalloc<void>(ctx, Ld * es);
        ctx->xb[1] = dalloc<void>(ctx, Ld * es);
        ctx->x1 = dalloc<void>(ctx, Ld * es);
        ctx->hbuf = dalloc<void>(ctx, Ld * es);
        ctx->q = dalloc<void>(ctx, Ld * es);
        ctx->o = dalloc<void>(ctx, Ld * es);
        ctx->u = dalloc<void>(ctx, (size_t)L * F * es);
        ctx->lat = dalloc<float>(ctx, (size_t)L * C * sizeof(float));
        ctx->vout = dalloc<float>(ctx, (size_t)L * C * sizeof(float));
        ctx->ht = dalloc<float>(ctx, d * sizeof(float));
        ctx->ha = dalloc<float>(ctx, d * sizeof(float));
        ctx->e = dalloc<float>(ctx, d * sizeof(float));
        ctx->mods = dalloc<float>(ctx, (size_t)B * 6 * d * sizeof(float));
        ctx->hmod = dalloc<float>(ctx, 2 * (size_t)d * sizeof(float));
        ctx->act_dev = dalloc<float>(ctx, 8 * sizeof(float));
        CK(cudaStreamCreateWithFlags(&ctx->cap_st, cudaStreamNonBlocking));
        ctx->graphs_on = true;

        // ring and caches
        ctx->ring_k = dalloc<void>(ctx, (size_t)B * ctx->Wkv * Ld * es);
        ctx->ring_v = dalloc<void>(ctx, (size_t)B * ctx->Wkv * Ld * es);
        ctx->rhat = dalloc<void>(ctx, (size_t)ctx->S * B * Ld * es);
        ctx->cells = dalloc<GateCell>(ctx, (size_t)ctx->S * B * sizeof(GateCell));
        ctx->phi_act = dalloc<float>(ctx, (size_t)ctx->S * B * 16 * sizeof(float));
        ctx->rmean = dalloc<float>(ctx, (size_t)ctx->S * B * ctx->V * d * sizeof(float));
        ctx->chain_gm = dalloc<float>(ctx, 2 * (size_t)ctx->V * d * sizeof(float));
        ctx->chain_last = 0;
        ctx->fp_K = -1;
        ctx->fp_lin = 0;
        ctx->fp_rows = nullptr;
        ctx->phi = nullptr;
        ctx->chain_sp = nullptr;
        ensure_fp(ctx, 32, 0);

        // per pass
        ctx->flags = dalloc<uint8_t>(ctx, XC_MAX_BLOCKS);
        ctx->s_cos = dalloc<float>(ctx, 3 * XC_MAX_BLOCKS * sizeof(float));
        ctx->d_max = ctx->s_cos + B;
        ctx->tau = ctx->s_cos + 2 * B;
        ctx->d_err = dalloc<int>(ctx, sizeof(int));
        CK(cudaMemset(ctx->d_err, 0, sizeof(int)));
        CK(cudaMallocHost(reinterpret_cast<void **>(&ctx->h_flags), XC_MAX_BLOCKS));
        CK(cudaMallocHost(reinterpret_cast<void **>(&ctx->h_stats), 3 * XC_MAX_BLOCKS * sizeof(float)));

        // gate scratch
        {
            int max_npc = 1;
            for (int g = 0; g < ctx->G; ++g) max_npc = std::max(max_npc, ctx->g_npc[g]);
            ctx->g_geom = gate_geometry(ctx->V, max_npc, d, ctx->n_sm);
            ctx->g_scratch = dalloc<char>(ctx, ctx->g_geom.total);
        }
        if (ctx->bf) {
            ctx->attn_ws_bytes = attn_workspace_bytes(ctx->hd);
            ctx->attn_ws = dalloc<char>(ctx, ctx->attn_ws_bytes);
        }

        // tensor maps of the bf16 path
        if (ctx->bf) {
            ctx->bn_qkv = gemm_tc_bn(L, 3 * d);
            ctx->bn_o = gemm_tc_bn(L, d);
            ctx->bn_f1 = gemm_tc_bn(L, F);
            ctx->bn_f2 = gemm_tc_bn(L, d);
            tmap(ctx, &ctx->tm_h, ctx->hbuf, L, d, 128);
            tmap(ctx, &ctx->tm_o, ctx->o, L, d, 128);
            tmap(ctx, &ctx->tm_u, ctx->u, L, F, 128);
            tmap(ctx, &ctx->tm_q, ctx->q, L, d, 128);
            ctx->tm_wqkv.resize(B);
            ctx->tm_wo.resize(B);
            ctx->tm_w1.resize(B);
            ctx->tm_w2.resize(B);
            ctx->tm_rk.resize(B);
            ctx->tm_rv.resize(B);
            for (int b = 0; b < B; ++b) {
                const char *wq = reinterpret_cast<const char *>(ctx->qkv_wt) + (size_t)b * 3 * d * d * es;
                const char *wo = reinterpret_cast<const char *>(ctx->o_wt) + (size_t)b * d * d * es;
                const char *w1 = reinterpret_cast<const char *>(ctx->f1_wt) + (size_t)b * F * d * es;
                const char *w2 = reinterpret_cast<const char *>(ctx->f2_wt) + (size_t)b * d * F * es;
                tmap(ctx, &ctx->tm_wqkv[b], wq, 3 * (uint64_t)d, d, ctx->bn_qkv);
                tmap(ctx, &ctx->tm_wo[b], wo, d, d, ctx->bn_o);
                tmap(ctx, &ctx->tm_w1[b], w1, F, d, ctx->bn_f1);
                tmap(ctx, &ctx->tm_w2[b], w2, d, F, ctx->bn_f2);
                const char *rk = reinterpret_cast<const char *>(ctx->ring_k) + (size_t)b * ctx->Wkv * Ld * es;
                const char *rv = reinterpret_cast<const char *>(ctx->ring_v) + (size_t)b * ctx->Wkv * Ld * es;
                tmap(ctx, &ctx->tm_rk[b], rk, (uint64_t)ctx->Wkv * L, d, 128);
                tmap(ctx, &ctx->tm_rv[b], rv, (uint64_t)ctx->Wkv * L, d, 128);
            }
            if (ctx->xattn) {
                const int D = ctx->d_ctx;
                for (auto *v : {&ctx->tm_caq, &ctx->tm_cao, &ctx->tm_cak, &ctx->tm_cav, &ctx->tm_ck, &ctx->tm_cv})
                    v->resize(B);
                for (int b = 0; b < B; ++b) {
                    const char *wq = reinterpret_cast<const char *>(ctx->ca_q_wt) + (size_t)b * d * d * es;
                    const char *wo = reinterpret_cast<const char *>(ctx->ca_o_wt) + (size_t)b * d * d * es;
                    const char *wkv = reinterpret_cast<const char *>(ctx->ca_kv_wt) + (size_t)b * 2 * d * D * es;
                    tmap(ctx, &ctx->tm_caq[b], wq, d, d, ctx->bn_o);
                    tmap(ctx, &ctx->tm_cao[b], wo, d, d, ctx->bn_o);
                    tmap(ctx, &ctx->tm_cak[b], wkv, d, D, 128);                      // rows [0, d): W_k^T
                    tmap(ctx, &ctx->tm_cav[b], wkv + (size_t)d * D * es, d, D, 128);  // rows [d, 2d): W_v^T
                    const size_t cb = (size_t)b * ctx->max_ctx * d * es;
                    tmap(ctx, &ctx->tm_ck[b], reinterpret_cast<const char *>(ctx->ctx_k) + cb, ctx->max_ctx, d, 128);
                    tmap(ctx, &ctx->tm_cv[b], reinterpret_cast<const char *>(ctx->ctx_v) + cb, ctx->max_ctx, d, 128);
                }
            }
        }
        ctx->trace = nullptr;
        clear_state(ctx);
        CK(cudaDeviceSynchronize());
    } catch (Fail &f) {
        std::string msg = ctx->err;
        xc_destroy(ctx);
        set_err(nullptr, "%s", msg.c_str());
        return f.st;
    }
    ctx->err = "no error";
    *out = ctx;
    return XC_OK;
}

xc_status xc_reset(xc_ctx *ctx) {
    if (ctx == nullptr) {
        set_err(nullptr, "xc_reset: NULL context");
        return XC_ESTATE;
    }
    try {
        clear_state(ctx);
    } catch (Fail &f) {
        return f.st;
    }
    return XC_OK;
}

int xc_chunk_index(const xc_ctx *ctx) { return ctx == nullptr ? -1 : ctx->n; }

void xc_debug_fail_alloc(int n) { g_fail_alloc.store(n > 0 ? n : 0); }

static int *op_err_word();

xc_status xc_debug_expire_wait(xc_ctx *ctx) {
    int *err = ctx != nullptr ? ctx->d_err : op_err_word();
    if (err == nullptr) {
        set_err(nullptr, "xc_debug_expire_wait: no device error word");
        return XC_ECUDA;
    }
    const cudaError_t e = expire_wait(err, ERR_WAIT_TMA, ctx != nullptr ? ctx->st : nullptr);
    if (e != cudaSuccess) {
        set_err(ctx, "xc_debug_expire_wait: %s", cudaGetErrorString(e));
        return XC_ECUDA;
    }
    return XC_OK;
}

long long xc_launch_count(const xc_ctx *ctx) { return ctx == nullptr ? -1 : ctx->launches; }

static void prof_free(xc_ctx *ctx) {
    for (cudaEvent_t e : ctx->prof_ev) cudaEventDestroy(e);
    ctx->prof_ev.clear();
    ctx->prof_rec.clear();
    if (ctx->dec_log != nullptr) cudaFree(ctx->dec_log);
    ctx->dec_log = nullptr;
    ctx->prof_on = false;
    ctx->prof_cap = ctx->prof_n = 0;
}

xc_status xc_profile_start(xc_ctx *ctx, unsigned kind_mask, int capacity) {
    if (ctx == nullptr) {
        set_err(nullptr, "xc_profile_start: NULL context");
        return XC_ESTATE;
    }
    if (capacity < 1) {
        set_err(ctx, "xc_profile_start: capacity < 1");
        return XC_EINVAL;
    }
    try {
        CK(cudaStreamSynchronize(ctx->st));
        prof_free(ctx);
        ctx->prof_ev.resize(2 * (size_t)capacity);
        for (auto &e : ctx->prof_ev) CK(cudaEventCreate(&e));
        ctx->prof_rec.resize(capacity);
        CK(cudaMalloc(&ctx->dec_log, (size_t)capacity * ctx->B));
        ctx->prof_cap = capacity;
        ctx->prof_n = 0;
        ctx->pass_seq = 0;
        ctx->prof_mask = kind_mask;
        ctx->prof_on = true;
    } catch (Fail &f) {
        prof_free(ctx);
        return f.st;
    }
    return XC_OK;
}

xc_status xc_profile_stop(xc_ctx *ctx, xc_profile_rec *out, int max, int *n_out) {
    if (ctx == nullptr) {
        set_err(nullptr, "xc_profile_stop: NULL context");
        return XC_ESTATE;
    }
    if (!ctx->prof_on) {
        set_err(ctx, "xc_profile_stop: profiling not started");
        return XC_ESTATE;
    }
    xc_status status = XC_OK;
    try {
        CK(cudaStreamSynchronize(ctx->st));
        const int passes = ctx->pass_seq < ctx->prof_cap ? ctx->pass_seq : ctx->prof_cap;
        std::vector<uint8_t> dec((size_t)passes * ctx->B + 1);
        if (passes > 0) CK(cudaMemcpy(dec.data(), ctx->dec_log, (size_t)passes * ctx->B, cudaMemcpyDeviceToHost));
        const int n = ctx->prof_n < max ? ctx->prof_n : max;
        for (int i = 0; i < n; ++i) {
            xc_profile_rec r = ctx->prof_rec[i];
            CK(cudaEventElapsedTime(&r.ms, ctx->prof_ev[2 * i], ctx->prof_ev[2 * i + 1]));
            if (r.block >= 0 && r.pass_seq < passes) r.decision = dec[(size_t)r.pass_seq * ctx->B + r.block];
            if (out != nullptr) out[i] = r;
        }
        if (n_out != nullptr) *n_out = ctx->prof_n;
    } catch (Fail &f) {
        status = f.st;
    }
    prof_free(ctx);
    return status;
}

xc_status xc_set_block_trace(xc_ctx *ctx, void *dev_buf) {
    if (ctx == nullptr) {
        set_err(nullptr, "xc_set_block_trace: NULL context");
        return XC_ESTATE;
    }
    ctx->trace = dev_buf;
    return XC_OK;
}

xc_status xc_sync(xc_ctx *ctx) {
    if (ctx == nullptr) {
        set_err(nullptr, "xc_sync: NULL context");
        return XC_ESTATE;
    }
    try {
        CK(cudaStreamSynchronize(ctx->st));
        int e = 0;
        CK(cudaMemcpy(&e, ctx->d_err, sizeof(int), cudaMemcpyDeviceToHost));
        if (e != 0) {
            CK(cudaMemset(ctx->d_err, 0, sizeof(int)));
            set_err(ctx, "device wait expired (error bits 0x%x)", e);
            return XC_ETIMEOUT;
        }
    } catch (Fail &f) {
        return f.st;
    }
    return XC_OK;
}

xc_status xc_euler_update(xc_ctx *ctx, float *x, const float *v, float dsigma, long n) {
    if (ctx == nullptr) {
        set_err(nullptr, "xc_euler_update: NULL context");
        return XC_ESTATE;
    }
    if (x == nullptr || v == nullptr || n < 0) {
        set_err(ctx, "xc_euler_update: bad argument");
        return XC_EINVAL;
    }
    if (n == 0) return XC_OK;
    try {
        CK(euler_update(x, v, dsigma, n, ctx->st));
        ctx->launches += 1;
    } catch (Fail &f) {
        return f.st;
    }
    return XC_OK;
}

xc_status xc_set_context(xc_ctx *ctx, const float *context, int n_ctx) {
    if (ctx == nullptr) {
        set_err(nullptr, "xc_set_context: NULL context");
        return XC_ESTATE;
    }
    if (!ctx->xattn) {
        set_err(ctx, "xc_set_context: the model has no cross-attention (d_ctx = 0)");
        return XC_EINVAL;
    }
    if (context == nullptr || n_ctx < 1 || n_ctx > ctx->max_ctx) {
        set_err(ctx, "xc_set_context: NULL tokens or n_ctx %d out of [1, %d]", n_ctx, ctx->max_ctx);
        return XC_EINVAL;
    }
    const int d = ctx->d, D = ctx->d_ctx, B = ctx->B;
    const size_t n = (size_t)n_ctx * D;
    try {
        cudaStream_t st = ctx->st;
        if (is_host_ptr(context)) {
            for (size_t i = 0; i < n; ++i)
                if (!std::isfinite(context[i])) {
                    set_err(ctx, "xc_set_context: non-finite condition token value");
                    return XC_ENUMERIC;
                }
            CK(cudaMemcpyAsync(ctx->ctx_in, context, n * sizeof(float), cudaMemcpyHostToDevice, st));
            CK(cudaStreamSynchronize(st));           // host buffer consumed before returning
        } else {
            CK(cudaMemcpyAsync(ctx->ctx_in, context, n * sizeof(float), cudaMemcpyDeviceToDevice, st));
        }
        CUtensorMap tm_a;
        if (ctx->bf) {
            CK(convert_f32<bf16>(ctx->ctx_in, reinterpret_cast<bf16 *>(ctx->ctx_act), (long)n, ctx->n_sm, st));
            if (!make_tmap_bf16(&tm_a, ctx->ctx_act, n_ctx, D, 128)) {
                set_err(ctx, "xc_set_context: tensor map encoding failed");
                return XC_ECUDA;
            }
        }
        // [K_c | V_c] = C W_kv + b_kv, one GEMM per half and block
        for (int b = 0; b < B; ++b)
            for (int half = 0; half < 2; ++half) {
                EpiParams ep;
                memset(&ep, 0, sizeof ep);
                ep.M = n_ctx;
                ep.N = d;
                ep.bias = ctx->ca_kv_b + (size_t)b * 2 * d + (size_t)half * d;
                ep.out = reinterpret_cast<char *>(half ? ctx->ctx_v : ctx->ctx_k) +
                         (size_t)b * ctx->max_ctx * d * ctx->esz;
                if (ctx->bf) {
                    CK(gemm_tc(EPI_BIAS, 128, tm_a, half ? ctx->tm_cav[b] : ctx->tm_cak[b], ep, D, nullptr,
                               ctx->d_err, st));
                } else {
                    const float *W = reinterpret_cast<const float *>(ctx->ca_kv_wt) + ((size_t)b * 2 + half) * d * D;
                    CK(gemm_simt(EPI_BIAS, ep, ctx->ctx_in, W, D, nullptr, st));
                }
                ctx->launches += 1;
            }
        ctx->n_ctx = n_ctx;
    } catch (Fail &f) {
        return f.st;
    }
    return XC_OK;
}

xc_status xc_chunk_step(xc_ctx *ctx, const float *latent, const float *action, float sigma, int step_index,
                        int is_kv_update, const xc_gate_params *gate, float *v_out, xc_step_stats *stats) {
    if (ctx == nullptr) {
        set_err(nullptr, "xc_chunk_step: NULL context");
        return XC_ESTATE;
    }
    if (latent == nullptr || action == nullptr) {
        set_err(ctx, "xc_chunk_step: NULL latent or action");
        return XC_EINVAL;
    }
    xc_gate_params p;
    if (gate != nullptr)
        p = *gate;
    else
        xc_gate_params_default(&p);
    char why[256];
    if (!gate_ok(&p, ctx->B, why, sizeof why)) {
        set_err(ctx, "%s", why);
        return XC_EINVAL;
    }
    for (int i = 0; i < ctx->A; ++i)
        if (!std::isfinite(action[i])) {
            set_err(ctx, "xc_chunk_step: non-finite action");
            return XC_ENUMERIC;
        }
    if (!std::isfinite(sigma)) {
        set_err(ctx, "xc_chunk_step: non-finite sigma");
        return XC_ENUMERIC;
    }
    const bool kv = is_kv_update != 0;
    if (kv) {
        if (ctx->next_step != 0 && ctx->next_step != ctx->S) {
            set_err(ctx, "KV-update pass before all %d denoising passes of chunk %d", ctx->S, ctx->n);
            return XC_ESTATE;
        }
        if (!kv_chunk(ctx, ctx->n)) {
            set_err(ctx, "chunk %d has no KV-update pass (kv_period %d)", ctx->n, ctx->kv_period);
            return XC_ESTATE;
        }
    } else if (step_index != ctx->next_step || step_index >= ctx->S) {
        set_err(ctx, "denoising pass %d out of order (expected %d)", step_index, ctx->next_step);
        return XC_ESTATE;
    }
    if (ctx->xattn && ctx->n_ctx == 0) {
        set_err(ctx, "cross-attention model without condition tokens: call xc_set_context first");
        return XC_ESTATE;
    }
    const int t = kv ? 0 : step_index;
    try {
        ensure_fp(ctx, p.fp_tokens, p.fp_linear);
        if (p.chain != 0 && ctx->chain_last == 0 && !kv) {
            // residuals cached before chaining have no per-camera means:
            // every gate cell starts over (the blocks recompute once)
            CK(cudaMemsetAsync(ctx->cells, 0, (size_t)ctx->S * ctx->B * sizeof(GateCell), ctx->st));
        }
        if (!kv) ctx->chain_last = p.chain;
        const size_t lat_bytes = (size_t)ctx->L * ctx->C * sizeof(float);
        const float *lat_dev = latent;
        if (is_host_ptr(latent)) {
            CK(cudaMemcpyAsync(ctx->lat, latent, lat_bytes, cudaMemcpyHostToDevice, ctx->st));
            lat_dev = ctx->lat;
        }
        const bool v_host = v_out != nullptr && is_host_ptr(v_out);
        float *v_dev = (v_out == nullptr || v_host) ? ctx->vout : v_out;
        if (ctx->bf)
            run_pass<bf16>(ctx, lat_dev, action, sigma, t, kv, p, v_dev, v_out != nullptr);
        else
            run_pass<float>(ctx, lat_dev, action, sigma, t, kv, p, v_dev, v_out != nullptr);
        if (v_host) CK(cudaMemcpyAsync(v_out, ctx->vout, lat_bytes, cudaMemcpyDeviceToHost, ctx->st));
        // Host buffers are consumed / produced synchronously: the caller may
        // reuse them as soon as the call returns.
        if (v_host || lat_dev != latent) CK(cudaStreamSynchronize(ctx->st));
        if (stats != nullptr) {
            CK(cudaMemcpyAsync(ctx->h_flags, ctx->flags, ctx->B, cudaMemcpyDeviceToHost, ctx->st));
            CK(cudaMemcpyAsync(ctx->h_stats, ctx->s_cos, 3 * ctx->B * sizeof(float), cudaMemcpyDeviceToHost,
                               ctx->st));
            CK(cudaStreamSynchronize(ctx->st));
            int e = 0;
            CK(cudaMemcpy(&e, ctx->d_err, sizeof(int), cudaMemcpyDeviceToHost));
            if (e != 0) {
                CK(cudaMemset(ctx->d_err, 0, sizeof(int)));
                set_err(ctx, "device wait expired (error bits 0x%x)", e);
                return XC_ETIMEOUT;
            }
            memset(stats, 0, sizeof *stats);
            stats->n_blocks = ctx->B;
            stats->chunk_index = ctx->n;
            for (int b = 0; b < ctx->B; ++b) {
                stats->decision[b] = ctx->h_flags[b];
                stats->s_cos[b] = ctx->h_stats[b];
                stats->d_max[b] = ctx->h_stats[ctx->B + b];
                stats->tau_cos[b] = ctx->h_stats[2 * ctx->B + b];
            }
        }
    } catch (Fail &f) {
        return f.st;
    }
    if (kv) {
        ctx->n += 1;
        ctx->kvc += 1;
        ctx->next_step = 0;
    } else if (step_index == ctx->S - 1 && !kv_chunk(ctx, ctx->n)) {
        ctx->n += 1;                                 // chunk without a KV-update pass ends here
        ctx->next_step = 0;
    } else {
        ctx->next_step = step_index + 1;
    }
    return XC_OK;
}

// ---------------------------------------------------------------- op entries
static int *op_err_word() {
    static int *p = nullptr;
    if (p == nullptr) {
        if (cudaMalloc(&p, sizeof(int)) != cudaSuccess) return nullptr;
        cudaMemset(p, 0, sizeof(int));
    }
    return p;
}

int xc_op_device_error(void) {
    int *p = op_err_word();
    if (p == nullptr) return -1;
    cudaDeviceSynchronize();
    int e = 0;
    cudaMemcpy(&e, p, sizeof(int), cudaMemcpyDeviceToHost);
    cudaMemset(p, 0, sizeof(int));
    return e;
}

#define OP_FAIL(code, ...)              \
    do {                                \
        set_err(nullptr, __VA_ARGS__);  \
        return code;                    \
    } while (0)
#define OP_CK(call)                                                                        \
    do {                                                                                   \
        cudaError_t e_ = (call);                                                           \
        if (e_ != cudaSuccess) OP_FAIL(XC_ECUDA, "%s: %s", #call, cudaGetErrorString(e_)); \
    } while (0)

xc_status xc_op_linear(int dtype, int epilogue, int M, int N, int K, const void *A, const void *Wt,
                       const float *bias, const float *gate, const void *resid, const void *xin, void *out,
                       void *rhat, void *stream) {
    if (M < 1 || N < 16 || K < 1 || A == nullptr || Wt == nullptr || bias == nullptr || out == nullptr)
        OP_FAIL(XC_EINVAL, "xc_op_linear: bad shape or NULL pointer");
    if (epilogue < XC_EPI_BIAS || epilogue > XC_EPI_RESID_CACHE) OP_FAIL(XC_EINVAL, "xc_op_linear: epilogue");
    if ((epilogue == XC_EPI_RESID_GATE || epilogue == XC_EPI_RESID_CACHE) && (gate == nullptr || resid == nullptr))
        OP_FAIL(XC_EINVAL, "xc_op_linear: gated residual needs gate and resid");
    if (epilogue == XC_EPI_RESID_CACHE && rhat != nullptr && xin == nullptr)
        OP_FAIL(XC_EINVAL, "xc_op_linear: residual cache needs xin");
    EpiParams ep;
    memset(&ep, 0, sizeof ep);
    ep.M = M;
    ep.N = N;
    ep.bias = bias;
    ep.gate = gate;
    ep.resid = resid;
    ep.xin = xin;
    ep.out = out;
    ep.rhat = rhat;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (dtype == XC_BF16) {
        if (N % 256 != 0 || K % 64 != 0) OP_FAIL(XC_EINVAL, "xc_op_linear: bf16 needs N %% 256 == 0, K %% 64 == 0");
        CUtensorMap ta, tb;
        const int bn = gemm_tc_bn(M, N);
        if (!make_tmap_bf16(&ta, A, M, K, 128) || !make_tmap_bf16(&tb, Wt, N, K, bn))
            OP_FAIL(XC_EINVAL, "xc_op_linear: tensor map (alignment?)");
        OP_CK(gemm_tc(epilogue, bn, ta, tb, ep, K, nullptr, op_err_word(), st));
    } else if (dtype == XC_F32) {
        if (N % 16 != 0) OP_FAIL(XC_EINVAL, "xc_op_linear: f32 needs N %% 16 == 0");
        OP_CK(gemm_simt(epilogue, ep, reinterpret_cast<const float *>(A), reinterpret_cast<const float *>(Wt), K,
                        nullptr, st));
    } else {
        OP_FAIL(XC_EINVAL, "xc_op_linear: dtype");
    }
    return XC_OK;
}

xc_status xc_op_qkv_rope(int dtype, int n_cams, int frames, int gh, int gw, int chunk, int d, int head_dim,
                         float rope_theta, const void *A, const void *Wt, const float *bias, void *q, void *k,
                         void *v, void *stream) {
    if (n_cams < 1 || frames < 1 || gh < 1 || gw < 1 || chunk < 0 || head_dim < 16 || head_dim % 16 != 0 ||
        d % head_dim != 0 || A == nullptr || Wt == nullptr || bias == nullptr || q == nullptr || k == nullptr ||
        v == nullptr)
        OP_FAIL(XC_EINVAL, "xc_op_qkv_rope: bad argument");
    // per-call RoPE layout and table (operator path; the chunk step keeps its own)
    static int *axis = nullptr, *off = nullptr;
    static float2 *cs = nullptr;
    static size_t cap_pairs = 0, cap_entries = 0;
    std::vector<int> ax, of;
    const int npos[4] = {n_cams, frames, gh, gw};
    const int n_entries = rope_layout(head_dim, npos, ax, of);
    cudaStream_t st0 = reinterpret_cast<cudaStream_t>(stream);
    if (ax.size() > cap_pairs || (size_t)n_entries > cap_entries) {
        OP_CK(cudaDeviceSynchronize());
        if (axis) cudaFree(axis);
        if (off) cudaFree(off);
        if (cs) cudaFree(cs);
        cap_pairs = ax.size();
        cap_entries = (size_t)n_entries;
        OP_CK(cudaMalloc(&axis, cap_pairs * sizeof(int)));
        OP_CK(cudaMalloc(&off, cap_pairs * sizeof(int)));
        OP_CK(cudaMalloc(&cs, cap_entries * sizeof(float2)));
    }
    OP_CK(cudaMemcpyAsync(axis, ax.data(), ax.size() * sizeof(int), cudaMemcpyHostToDevice, st0));
    OP_CK(cudaMemcpyAsync(off, of.data(), of.size() * sizeof(int), cudaMemcpyHostToDevice, st0));
    OP_CK(rope_table(head_dim, (double)rope_theta, chunk * frames, make_int4(n_cams, frames, gh, gw), cs, n_entries,
                     st0));
    const int npc = frames * gh * gw, M = n_cams * npc;
    EpiParams ep;
    memset(&ep, 0, sizeof ep);
    ep.M = M;
    ep.N = 3 * d;
    ep.bias = bias;
    ep.out = q;
    ep.out_k = k;
    ep.out_v = v;
    ep.d = d;
    ep.head_dim = head_dim;
    epi_single_grid(ep, frames, gh, gw);
    ep.frame0 = chunk * frames;
    ep.rope_axis = axis;
    ep.rope_off = off;
    ep.rope_cs = cs;
    cudaStream_t st = st0;
    if (dtype == XC_BF16) {
        if ((3 * d) % 256 != 0 || d % 64 != 0) OP_FAIL(XC_EINVAL, "xc_op_qkv_rope: bf16 needs 3d %% 256, d %% 64");
        CUtensorMap ta, tb;
        const int bn = gemm_tc_bn(M, 3 * d);
        if (!make_tmap_bf16(&ta, A, M, d, 128) || !make_tmap_bf16(&tb, Wt, 3 * (uint64_t)d, d, bn))
            OP_FAIL(XC_EINVAL, "xc_op_qkv_rope: tensor map");
        OP_CK(gemm_tc(EPI_QKV_ROPE, bn, ta, tb, ep, d, nullptr, op_err_word(), st));
    } else if (dtype == XC_F32) {
        OP_CK(gemm_simt(EPI_QKV_ROPE, ep, reinterpret_cast<const float *>(A), reinterpret_cast<const float *>(Wt), d,
                        nullptr, st));
    } else {
        OP_FAIL(XC_EINVAL, "xc_op_qkv_rope: dtype");
    }
    return XC_OK;
}

size_t xc_op_attention_workspace_bytes(int dtype, int head_dim) {
    if (dtype != XC_BF16 || (head_dim != 64 && head_dim != 128)) return 0;
    return attn_workspace_bytes(head_dim);
}

xc_status xc_op_attention(int dtype, int Lq, int n_keys, int n_heads, int head_dim, const void *q, const void *k,
                          const void *v, void *o, void *workspace, size_t workspace_bytes, void *stream) {
    if (Lq < 1 || n_keys < 1 || n_heads < 1 || q == nullptr || k == nullptr || v == nullptr || o == nullptr)
        OP_FAIL(XC_EINVAL, "xc_op_attention: bad argument");
    const int d = n_heads * head_dim;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (dtype == XC_BF16) {
        if (head_dim != 64 && head_dim != 128) OP_FAIL(XC_EINVAL, "xc_op_attention: bf16 head_dim 64 or 128");
        CUtensorMap tq, tk, tv;
        if (!make_tmap_bf16(&tq, q, Lq, d, 128) || !make_tmap_bf16(&tk, k, n_keys, d, 128) ||
            !make_tmap_bf16(&tv, v, n_keys, d, 128))
            OP_FAIL(XC_EINVAL, "xc_op_attention: tensor map");
        OP_CK(attn_tc(head_dim, tq, tk, tv, reinterpret_cast<bf16 *>(o), Lq, n_keys, n_heads, d, workspace,
                      workspace_bytes, nullptr, op_err_word(), nullptr, st));
    } else if (dtype == XC_F32) {
        OP_CK(attn_simt(head_dim, reinterpret_cast<const float *>(q), reinterpret_cast<const float *>(k),
                        reinterpret_cast<const float *>(v), reinterpret_cast<float *>(o), Lq, n_keys, n_heads,
                        nullptr, st));
    } else {
        OP_FAIL(XC_EINVAL, "xc_op_attention: dtype");
    }
    return XC_OK;
}

xc_status xc_op_ln_mod(int dtype, int M, int d, float eps, const void *x, const float *shift, const float *scale,
                       void *out, void *stream) {
    if (M < 1 || d < 16 || d % 16 != 0 || x == nullptr || shift == nullptr || scale == nullptr || out == nullptr)
        OP_FAIL(XC_EINVAL, "xc_op_ln_mod: bad argument");
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (dtype == XC_BF16)
        OP_CK(ln_mod<bf16>(reinterpret_cast<const bf16 *>(x), shift, scale, reinterpret_cast<bf16 *>(out), M, d, eps,
                           nullptr, st));
    else if (dtype == XC_F32)
        OP_CK(ln_mod<float>(reinterpret_cast<const float *>(x), shift, scale, reinterpret_cast<float *>(out), M, d,
                            eps, nullptr, st));
    else
        OP_FAIL(XC_EINVAL, "xc_op_ln_mod: dtype");
    return XC_OK;
}

xc_status xc_op_residual_reuse(int dtype, long n, const void *x, const void *rhat, void *out, void *stream) {
    if (n < 0 || n % 16 != 0 || x == nullptr || rhat == nullptr || out == nullptr)
        OP_FAIL(XC_EINVAL, "xc_op_residual_reuse: bad argument (n %% 16 == 0 required)");
    if (n == 0) return XC_OK;
    int dev = 0, n_sm = 152;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (dtype == XC_BF16)
        OP_CK(residual_reuse<bf16>(reinterpret_cast<const bf16 *>(x), reinterpret_cast<const bf16 *>(rhat),
                                   reinterpret_cast<bf16 *>(out), n, nullptr, n_sm, st));
    else if (dtype == XC_F32)
        OP_CK(residual_reuse<float>(reinterpret_cast<const float *>(x), reinterpret_cast<const float *>(rhat),
                                    reinterpret_cast<float *>(out), n, nullptr, n_sm, st));
    else
        OP_FAIL(XC_EINVAL, "xc_op_residual_reuse: dtype");
    return XC_OK;
}

}  // extern "C"
