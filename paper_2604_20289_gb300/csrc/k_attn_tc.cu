// Flash attention on the tcgen05 tensor core (bf16 in, fp32 softmax / accumulate).
//
//   o = softmax(q k^T / sqrt(hd)) v   per head, no mask inside the window:
//   the current chunk's queries see every resident key of the rolling KV
//   cache (past chunks' clean K/V plus the current chunk's own K/V).
//
// One CTA = one 128-query tile of one head.  Warp roles (192 threads):
//   warps 0..3 : softmax; thread r owns query row r = TMEM lane r.  Reads the
//                score row S (fp32, TMEM), online max / sum in the exp2 domain,
//                writes P (bf16, 128B-swizzled, K-major) to shared memory and
//                rescales its O row in TMEM when the running max grows;
//   warp 4     : TMA producer (Q once; K and V tiles of 128 keys, STAGES deep);
//   warp 5     : TMEM allocation; lane 0 issues S = Q K^T (M=128, N=128) into
//                one of two TMEM score buffers and O += P V (M=128, N=hd, V
//                read MN-major straight from its [keys][hd] tile).
// TMEM columns: S0 [0,128), S1 [128,256), O [256, 256+hd).
// S_{j+1} is computed while the softmax warps work on S_j; P V_j overlaps the
// score read of S_{j+1}.  Keys beyond n_keys are masked to -inf (their K/V
// rows are finite: the ring is zero-initialised and TMA zero-fills past the
// end of the tensor).
#include "xc_ptx.cuh"

namespace xc {

template <int HD>
struct AttnTile {
    static constexpr int BQ = 128, BKV = 128;
    static constexpr int NR = HD / 64;                 // 64-wide swizzle regions per row
    static constexpr int REGION = 128 * 128;           // [128 rows][64 bf16] bytes
    static constexpr int Q_BYTES = NR * REGION;
    static constexpr int KV_BYTES = NR * REGION;
    static constexpr int STAGES = HD == 64 ? 3 : 2;
    static constexpr int P_BYTES = 2 * REGION;
    static constexpr int OFF_K = Q_BYTES;
    static constexpr int OFF_V = OFF_K + STAGES * KV_BYTES;
    static constexpr int OFF_P = OFF_V + STAGES * KV_BYTES;
    static constexpr int OFF_BAR = OFF_P + P_BYTES;
    static constexpr int SMEM_BYTES = OFF_BAR + 256 + 1024;
    static constexpr int TMEM_COLS = 512;
    static constexpr int O_COL = 256;
};

__device__ __forceinline__ uint8_t *align1024_a(uint8_t *p) {
    const uint32_t s = smem_u32(p);
    return p + ((1024u - (s & 1023u)) & 1023u);
}

template <int HD>
__global__ void __launch_bounds__(192, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV, bf16 *__restrict__ o, const int Lq,
                   const int n_keys, const int d, const uint8_t *__restrict__ skip_flag, int *err) {
    using A = AttnTile<HD>;
    if (skip_flag != nullptr && *skip_flag == XC_DEC_SKIP) return;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = align1024_a(smem_raw);
    uint8_t *sQ = smem;
    uint8_t *sK = smem + A::OFF_K;
    uint8_t *sV = smem + A::OFF_V;
    uint8_t *sP = smem + A::OFF_P;
    uint64_t *bar = reinterpret_cast<uint64_t *>(smem + A::OFF_BAR);
    uint64_t *q_full = bar;
    uint64_t *kv_full = bar + 1;
    uint64_t *kv_empty = kv_full + A::STAGES;
    uint64_t *s_full = kv_empty + A::STAGES;   // [2]
    uint64_t *s_free = s_full + 2;             // [2]
    uint64_t *p_full = s_free + 2;
    uint64_t *pv_done = p_full + 1;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(pv_done + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int q0 = blockIdx.x * A::BQ;
    const int h = blockIdx.y;
    const int nkt = (n_keys + A::BKV - 1) / A::BKV;

    if (threadIdx.x == 0) {
        mbar_init(q_full, 1);
        for (int s = 0; s < A::STAGES; ++s) {
            mbar_init(&kv_full[s], 1);
            mbar_init(&kv_empty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&s_full[s], 1);
            mbar_init(&s_free[s], 128);
        }
        mbar_init(p_full, 128);
        mbar_init(pv_done, 1);
        mbar_fence_init();
    }
    if (warp == 5) tmem_alloc(tmem_slot, A::TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 4) {
        if (lane == 0) {
            mbar_expect_tx(q_full, A::Q_BYTES);
            for (int r = 0; r < A::NR; ++r) tma_load_2d(sQ + r * A::REGION, &tmQ, q_full, h * HD + 64 * r, q0);
            int issued = 0;
            for (int j = 0; j < nkt; ++j) {
                const int st = j % A::STAGES;
                if (!mbar_wait(&kv_empty[st], ((j / A::STAGES) & 1) ^ 1, err, ERR_WAIT_PRODUCER)) break;
                mbar_expect_tx(&kv_full[st], 2 * A::KV_BYTES);
                for (int r = 0; r < A::NR; ++r) {
                    tma_load_2d(sK + st * A::KV_BYTES + r * A::REGION, &tmK, &kv_full[st], h * HD + 64 * r,
                                j * A::BKV);
                    tma_load_2d(sV + st * A::KV_BYTES + r * A::REGION, &tmV, &kv_full[st], h * HD + 64 * r,
                                j * A::BKV);
                }
                issued = j + 1;
            }
            mbar_wait(q_full, 0, err, ERR_WAIT_PRODUCER);
            for (int j = issued - A::STAGES < 0 ? 0 : issued - A::STAGES; j < issued; ++j)
                mbar_wait(&kv_full[j % A::STAGES], (j / A::STAGES) & 1, err, ERR_WAIT_PRODUCER);
        }
    } else if (warp == 5) {
        if (lane == 0) {
            constexpr uint32_t idesc_s = idesc_bf16(128, 128, false, false);
            constexpr uint32_t idesc_o = idesc_bf16(128, HD, false, true);
            bool ok = mbar_wait(q_full, 0, err, ERR_WAIT_MMA);
            const uint32_t aQ = smem_u32(sQ), aK = smem_u32(sK), aV = smem_u32(sV), aP = smem_u32(sP);
            for (int j = 0; ok && j <= nkt; ++j) {
                if (j < nkt) {
                    const int st = j % A::STAGES;
                    const int sb = j & 1;
                    if (!mbar_wait(&kv_full[st], (j / A::STAGES) & 1, err, ERR_WAIT_MMA)) break;
                    if (j >= 2 && !mbar_wait(&s_free[sb], ((j - 2) >> 1) & 1, err, ERR_WAIT_MMA)) break;
                    tc_fence_after();
#pragma unroll
                    for (int ks = 0; ks < HD / 16; ++ks) {
                        const uint32_t off = (ks >> 2) * A::REGION + (ks & 3) * 32;
                        tc_mma(tmem + sb * 128, sdesc_sw128(aQ + off, 16, 1024),
                               sdesc_sw128(aK + st * A::KV_BYTES + off, 16, 1024), idesc_s, ks > 0 ? 1u : 0u);
                    }
                    tc_commit(&s_full[sb]);
                }
                if (j >= 1) {
                    const int jj = j - 1;
                    const int st = jj % A::STAGES;
                    if (!mbar_wait(p_full, jj & 1, err, ERR_WAIT_MMA)) break;
                    tc_fence_after();
#pragma unroll
                    for (int ks = 0; ks < A::BKV / 16; ++ks) {
                        const uint32_t pa = aP + (ks >> 2) * A::REGION + (ks & 3) * 32;
                        const uint32_t vb = aV + st * A::KV_BYTES + ks * 16 * 128;
                        tc_mma(tmem + A::O_COL, sdesc_sw128(pa, 16, 1024), sdesc_sw128(vb, A::REGION, 1024),
                               idesc_o, (jj > 0 || ks > 0) ? 1u : 0u);
                    }
                    tc_commit(pv_done);
                    tc_commit(&kv_empty[st]);
                }
            }
        }
    } else {
        // ---------------------------------------------------------- softmax
        const int r = warp * 32 + lane;
        const uint32_t tl = tmem + ((uint32_t)(warp * 32) << 16);
        const float sl2 = rsqrtf((float)HD) * 1.4426950408889634f;
        float m = -INFINITY, l = 0.0f;
        bool ok = true;
        for (int j = 0; j < nkt && ok; ++j) {
            const int sb = j & 1;
            ok = mbar_wait(&s_full[sb], (j >> 1) & 1, err, ERR_WAIT_SOFTMAX);
            __syncwarp();
            if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
            tc_fence_after();
            float s[128];
            tmem_ld128_sync(tl + sb * 128, s);
            tc_fence_before();
            mbar_arrive(&s_free[sb]);
            const int kbase = j * A::BKV;
            float mx = -INFINITY;
#pragma unroll
            for (int c = 0; c < 128; ++c) {
                if (kbase + c >= n_keys) s[c] = -INFINITY;
                mx = fmaxf(mx, s[c]);
            }
            const float m_new = fmaxf(m, mx * sl2);
            if (j >= 1) {
                ok = mbar_wait(pv_done, (j - 1) & 1, err, ERR_WAIT_SOFTMAX);
                __syncwarp();
                if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
                tc_fence_after();
                if (__any_sync(0xffffffffu, m_new > m)) {
                    const float alpha = exp2f(m - m_new);
#pragma unroll 1
                    for (int c = 0; c < HD / 16; ++c) {
                        float t[16];
                        tmem_ld16_sync(tl + A::O_COL + 16 * c, t);
#pragma unroll
                        for (int i = 0; i < 16; ++i) t[i] *= alpha;
                        tmem_st16_sync(tl + A::O_COL + 16 * c, t);
                    }
                    l *= alpha;
                }
            }
            m = m_new;
            float rs = 0.0f;
            uint8_t *prow = sP + r * 128;
#pragma unroll
            for (int c16 = 0; c16 < 16; ++c16) {
                uint32_t w[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float p0 = exp2f(fmaf(s[8 * c16 + 2 * i], sl2, -m));
                    const float p1 = exp2f(fmaf(s[8 * c16 + 2 * i + 1], sl2, -m));
                    rs += p0 + p1;
                    __nv_bfloat162 hh = __floats2bfloat162_rn(p0, p1);
                    w[i] = *reinterpret_cast<uint32_t *>(&hh);
                }
                const int region = c16 >> 3, cc = c16 & 7;
                *reinterpret_cast<uint4 *>(prow + region * A::REGION + ((cc ^ (r & 7)) << 4)) =
                    make_uint4(w[0], w[1], w[2], w[3]);
            }
            l += rs;
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(p_full);
        }
        if (ok) ok = mbar_wait(pv_done, (nkt - 1) & 1, err, ERR_WAIT_SOFTMAX);
        __syncwarp();
        if (__all_sync(0xffffffffu, ok)) {
            tc_fence_after();
            const float inv = 1.0f / l;
            const int row = q0 + r;
#pragma unroll 1
            for (int c = 0; c < HD / 16; ++c) {
                float t[16];
                tmem_ld16_sync(tl + A::O_COL + 16 * c, t);
#pragma unroll
                for (int i = 0; i < 16; ++i) t[i] *= inv;
                if (row < Lq) store16<bf16>(o + (size_t)row * d + h * HD + 16 * c, t);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 5) {
        tc_fence_after();
        tmem_dealloc(tmem, A::TMEM_COLS);
    }
}

bool make_tmap_bf16(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint32_t box_rows);

template <int HD>
static cudaError_t launch_attn(const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &tv, bf16 *o,
                               int Lq, int n_keys, int n_heads, int d, const uint8_t *skip, int *err,
                               cudaStream_t st) {
    using A = AttnTile<HD>;
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e =
            cudaFuncSetAttribute(attn_tc_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, A::SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    dim3 grid((Lq + A::BQ - 1) / A::BQ, n_heads);
    attn_tc_kernel<HD><<<grid, 192, A::SMEM_BYTES, st>>>(tq, tk, tv, o, Lq, n_keys, d, skip, err);
    return cudaGetLastError();
}

// q [Lq][d], k / v maps over [>= n_keys][d] (box 128 rows), o [Lq][d]; hd in {64, 128}.
cudaError_t attn_tc(int head_dim, const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &tv,
                    bf16 *o, int Lq, int n_keys, int n_heads, int d, const uint8_t *skip, int *err,
                    cudaStream_t st) {
    if (n_keys < 1 || Lq < 1) return cudaErrorInvalidValue;
    if (head_dim == 64) return launch_attn<64>(tq, tk, tv, o, Lq, n_keys, n_heads, d, skip, err, st);
    if (head_dim == 128) return launch_attn<128>(tq, tk, tv, o, Lq, n_keys, n_heads, d, skip, err, st);
    return cudaErrorInvalidValue;
}

}  // namespace xc
