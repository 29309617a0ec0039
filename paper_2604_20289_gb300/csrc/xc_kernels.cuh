// Launchers of the X-Cache kernels (k_*.cu) and the gate's device structs.
#pragma once
#include <cuda.h>

#include "xc_common.cuh"

namespace xc {
// Per-(t, b) gate state: EMA of the cosine (Eq. 8), has-history bit,
// consecutive-skip counter, cache-valid bit, active fingerprint half.
struct GateCell {
    double ema;
    int has_hist, stale, valid, active;
    int pad[2];
};
struct GateArgs {
    const void *x;
    int d, V;                // V: cameras of all view groups
    const int *fp_rows;      // spatial-sample token rows, group by group, camera by camera
    // view group g: cameras [g_cam0[g], g_cam0[g + 1]) of g_npc[g] tokens each
    // from token g_tok0[g]; g_kfp[g] sample rows per camera from row g_fp0[g]
    int n_groups, n_rows;    // n_rows: sample rows of all cameras
    int g_cam0[XC_MAX_GROUPS + 1], g_tok0[XC_MAX_GROUPS], g_npc[XC_MAX_GROUPS], g_fp0[XC_MAX_GROUPS],
        g_kfp[XC_MAX_GROUPS];
    int n_slices, cw;        // column slices of cw columns
    int R, rows_per;         // row blocks per camera and rows per row block: one CTA per (camera, slice, row block)
    float *phi;
    float *phi_act;
    float action[8];
    const float *action_dev;      // if set, the action is read from device memory (chunk step)
    int A;
    GateCell *cell;
    int mode;
    int step;
    float tau_floor, margin, alpha, tau_dev, eps_dev, strict_tau;
    int max_skips, fp_refresh, replay;   // replay: -1 off, 0 / 1 the replayed decision
    const uint8_t *replay_dev;           // device replay entry of this (t, b), or NULL
    uint8_t *flag;
    float *s_cos, *d_max, *tau_out;
    float *part;             // scratch [V * n_slices * R][8] partial metrics
    unsigned *ticket;        // scratch, zero before the launch (left zero)
    // lazy residual chaining (chain = 1): when *prev_flag (the previous
    // block's decision) is skip, the input is x_{j-1} + the pending residuals:
    // its sampled rows are csp_in + rhat_prev rows (running fp32 sums, [n_rows][d])
    // and its per-camera means cgm_in + rmean_prev ([V][d]); every chained
    // gate writes its own sums to csp_out / cgm_out
    int chain;
    const uint8_t *prev_flag;
    const void *rhat_prev;
    const float *rmean_prev;
    const float *csp_in, *cgm_in;
    float *csp_out, *cgm_out;
    float *cam_mean_out;     // camera_mean_launch: [V][d] per-camera means of x
};
// Grid and scratch layout of one gate launch (k_gate.cu).
struct GateGeom {
    int n_slices, cw, R, rows_per, n_ctas;
    size_t tickets_off, n_tickets, total;
};
// One view group of V cameras, npc tokens and kfp sample rows each.
inline void gate_single_group(GateArgs &g, int V, int npc, int kfp) {
    g.V = V;
    g.n_groups = 1;
    g.n_rows = V * kfp;
    g.g_cam0[0] = 0;
    g.g_cam0[1] = V;
    g.g_tok0[0] = 0;
    g.g_npc[0] = npc;
    g.g_fp0[0] = 0;
    g.g_kfp[0] = kfp;
}
// Gate grid for V cameras of at most max_npc tokens, d columns, n_sm SMs; the
// scratch holds the per-CTA partials and the ticket (see GateGeom).
GateGeom gate_geometry(int V, int max_npc, int d, int n_sm);
// Points the scratch fields (and grid fields) of g into `scratch`.
void gate_bind_scratch(GateArgs &g, const GateGeom &gg, void *scratch);
// Validates the gate knobs (NaN thresholds, ranges, counts); the reason goes to why.
bool gate_ok(const xc_gate_params *p, int B, char *why, size_t n);
template <typename T> cudaError_t gate_launch(const GateArgs &g, cudaStream_t st);
// Per-camera column means of g.x into g.cam_mean_out (same grid as the gate;
// exits at once when *g.flag is skip).
template <typename T> cudaError_t camera_mean_launch(const GateArgs &g, cudaStream_t st);
// Lazy chaining (reading c27): before block b (b = n_blocks: before the head)
// computes, when the blocks before it back to j were skipped, writes
// round(X[j & 1] + rhat[t][j] + ... + rhat[t][b - 1]) (fp32 sum in block
// order) to X[b & 1].  Exits at once otherwise.
template <typename T>
cudaError_t chain_apply(T *x0, T *x1, const T *rhat_t, const uint8_t *flags, int b, int n_blocks, long ld,
                        int n_sm, cudaStream_t st);
bool make_tmap_bf16(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint32_t box_rows);
int gemm_tc_bn(int M, int N);
cudaError_t gemm_tc(int epi, int bn, const CUtensorMap &ta, const CUtensorMap &tb, const EpiParams &ep, int K,
                    const uint8_t *skip, int *err, cudaStream_t st);
cudaError_t attn_tc(int head_dim, const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &tv, bf16 *o,
                    int Lq, int n_keys, int n_heads, int d, void *ws, size_t ws_bytes, const uint8_t *skip, int *err,
                    int *n_launched, cudaStream_t st);
size_t attn_workspace_bytes(int head_dim);
cudaError_t gemm_simt(int epi, const EpiParams &ep, const float *A, const float *Wt, int K, const uint8_t *skip,
                      cudaStream_t st);
cudaError_t attn_simt(int head_dim, const float *q, const float *k, const float *v, float *o, int Lq, int n_keys,
                      int H, const uint8_t *skip, cudaStream_t st);
template <typename T>
cudaError_t patch_embed(const float *z, const float *w, const float *b, T *out, int L, int C, int d, cudaStream_t st);
template <typename T>
cudaError_t ln_mod(const T *x, const float *shift, const float *scale, T *out, int M, int d, float eps,
                   const uint8_t *skip, cudaStream_t st);
template <typename T>
cudaError_t residual_reuse(const T *x, const T *r, T *out, long n, const uint8_t *skip, int n_sm, cudaStream_t st);
cudaError_t euler_update(float *x, const float *v, float ds, long n, cudaStream_t st);
template <typename T>
cudaError_t convert_f32(const float *in, T *out, long n, int n_sm, cudaStream_t st);
// Fused conditioning (three launches), see k_elem.cu.
constexpr int COND_TEMB_MAX = 512;
struct CondArgs {
    float temb[COND_TEMB_MAX];    // sinusoidal embedding of 1000 sigma (host, double precision)
    float act[8];
    int A, tf, d, B;
    const float *t_w1, *t_b1, *a_w1, *a_b1, *t_w2, *t_b2, *a_w2, *a_b2;
    const float *mod_w, *mod_b, *blk_mod, *head_w, *head_b, *head_tab;
    float *ht, *ha, *e, *mods, *hmod;
    float *act_out;               // device copy of the action (read by the gate kernels)
};
cudaError_t conditioning(const CondArgs &c, cudaStream_t st);
template <typename T>
cudaError_t head(const T *x, const float *hm, const float *w, const float *b, float *v, int L, int d, float eps,
                 cudaStream_t st);
template <typename T> cudaError_t transpose_convert(const float *W, T *Wt, int K, int N, cudaStream_t st);
cudaError_t rope_table(int hd, double theta, int frame0, int4 npos, float2 *out, int n, cudaStream_t st);
// Test of the bounded waits: a one-thread kernel whose wait runs out (after
// WAIT_NS) and records `code` in *err.
cudaError_t expire_wait(int *err, int code, cudaStream_t st);
// Records the message returned by xc_last_error(NULL).
void set_global_error(const char *msg);
}  // namespace xc
