// Flash attention on the tcgen05 tensor core (bf16 in, fp32 softmax / accumulate).
//
//   o = softmax(q k^T / sqrt(hd)) v   per head, no mask inside the window:
//   the current chunk's queries see every resident key of the rolling KV
//   cache (past chunks' clean K/V plus the current chunk's own K/V).
//
// One CTA = two 128-query tiles (Q0, Q1) of one head, 352 threads:
//   warps 0..3  softmax WG 0 (tile Q0), thread = query row = TMEM lane;
//   warps 4..7  softmax WG 1 (tile Q1);
//   warp 8      TMA producer: Q0/Q1 once, then 128-key K and V tiles through
//               a STAGES-deep ring (separate K and V barriers);
//   warp 9      TMEM allocation; MMA issue (hd 64: tile Q0; hd 128: both);
//   warp 10     hd 64: MMA issue for tile Q1 (MMA warps run converged, one
//               elected lane issuing each instruction).
// TMEM: S0 [0,128), S1 [128,256), O0 [256, 256+hd), O1 after it.  P (bf16)
// goes back into TMEM and feeds tcgen05.mma as the A operand straight from
// tensor memory (no shared-memory round trip); V is read MN-major from its
// [keys][hd] tile.
//   hd = 64 : P0 / P1 have their own 64 columns ([384,448), [448,512)), so
//             S_{j+1} is issued as soon as the softmax has READ S_j and runs on
//             the tensor core while the softmax computes P_j.
//   hd = 128: TMEM is full (S0 S1 O0 O1 = 512 columns); P_i overwrites S_i and
//             S_{j+1} waits until P_j V has been issued; the two tiles
//             ping-pong so the tensor core still has the other tile's work.
// At head_dim 64 the two softmax warps of each SM sub-partition (one per
// tile) take turns on the MUFU-bound exponential phase.
// Online softmax in the exp2 domain with lazy rescaling: a row's O and sum
// are rescaled only when its running max grows by more than 8 (2^8 headroom
// in fp32 / bf16).  Score scaling and row sums use packed fp32 pairs
// (FFMA2 / FADD2).  Keys beyond n_keys (ragged last tile) are masked to -inf;
// their K/V rows are finite (zero-initialised ring, TMA zero fill).
#include "xc_ptx.cuh"

namespace xc {

template <int HD>
struct AttnTile {
    static constexpr int BQ = 128, BKV = 128, QT = 2;
    static constexpr int NR = HD / 64;                 // 64-wide swizzle regions per row
    static constexpr int REGION = 128 * 128;           // [128 rows][64 bf16]
    static constexpr int Q_BYTES = NR * REGION;        // one 128-row Q tile
    static constexpr int KV_BYTES = NR * REGION;       // one 128-key K or V tile
    static constexpr int STAGES = HD == 64 ? 4 : 2;
    static constexpr int OFF_K = QT * Q_BYTES;
    static constexpr int OFF_V = OFF_K + STAGES * KV_BYTES;
    static constexpr int OFF_BAR = OFF_V + STAGES * KV_BYTES;
    static constexpr int SMEM_BYTES = OFF_BAR + 512 + 1024;
    static constexpr int TMEM_COLS = 512;
    static constexpr int THREADS = 352;            // 8 softmax, 1 TMA, 2 MMA warps
    static constexpr bool SEP_P = HD == 64;            // P has its own TMEM columns
    static constexpr int ISSUERS = SEP_P ? 2 : 1;      // MMA-issuing warps (9, 10)
    __host__ __device__ static constexpr int S_COL(int i) { return 128 * i; }
    __host__ __device__ static constexpr int O_COL(int i) { return 256 + HD * i; }
    __host__ __device__ static constexpr int P_COL(int i) { return SEP_P ? 256 + 2 * HD + 64 * i : 128 * i; }
    static constexpr float LAZY = 8.0f;                // rescale threshold (log2 units)
};

__device__ __forceinline__ uint8_t *align1024_a(uint8_t *p) {
    const uint32_t s = smem_u32(p);
    return p + ((1024u - (s & 1023u)) & 1023u);
}

__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float y;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(y) : "f"(a), "f"(b), "f"(c));
    return y;
}

__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Work split.  A unit is (head, pair of 128-query tiles), u = head * n_qblk +
// qblk, with n_kt key tiles.  Without a split (G = n_units CTAs) every CTA
// runs one whole unit.  With G = number of SMs < n_units, two orders:
//  * contiguous (WAVE = false): the (unit, key tile) iteration space, T =
//    n_units * n_kt, is cut into the contiguous shares [c T / G,
//    (c + 1) T / G).  A unit cut by the boundary between CTAs c - 1 and c is
//    finished by both as an unnormalised partial O with its running max m
//    and sum l (a flash-decoding partial, slot (boundary c, head / tail)),
//    and attn_combine_kernel merges the two.  Every share is at least one
//    unit, so a unit is cut at most once.  The units in flight span every
//    head, so each unit streams its head's K / V from DRAM once the heads'
//    K / V exceed L2.
//  * waves (WAVE = true, for many waves of units whose K / V exceed L2):
//    W = n_units / G waves of whole units -- CTA c runs units c, c + G, ...,
//    c + (W - 1) G, so the CTAs running at one time share a few heads and
//    each K / V tile comes from DRAM once per wave -- then the R = n_units -
//    W G remaining units, T2 = R n_kt key tiles, are split evenly: CTA c
//    takes [c T2 / G, (c + 1) T2 / G), less than one unit, touching at most
//    two units (its pieces W and W + 1, partial slots 2 c and 2 c + 1),
//    merged per remaining unit by attn_combine_kernel.
// Each role walks the CTA's key tiles with a cursor (TileCursor): tile
// counter g, unit u and its key tile k; in the wave order also the piece
// index p and the unit step du.
struct AttnSplit {
    long long T;          // contiguous: total iterations
    long long T2;         // waves: key tiles of the remaining units
    int n_kt, n_qblk, G, W;
    __host__ __device__ long long begin(int c) const { return T * c / G; }
    __host__ __device__ long long begin2(int c) const { return T2 * c / G; }
};
struct TileCursor {
    int g, u, k;          // tile counter, unit, key tile of the unit
    int p, du;            // waves: piece index, unit step (G over the waves, 1 in the remainder)
};
// Waves: pieces W and W + 1 of CTA c (its share of the remaining units) --
// first key tile of piece W, end key tiles of both (0: no such piece), and
// the unit of piece W.
struct RemSeg {
    int k0, k1a, k1b, u;
};
__device__ __forceinline__ RemSeg rem_seg(const AttnSplit &sp, int c) {
    const int nkt = sp.n_kt;
    RemSeg r{0, 0, 0, 0};
    const long long b = sp.begin2(c), e = sp.begin2(c + 1);
    if (b == e) return r;
    const long long ub = b / nkt, bnd = (ub + 1) * nkt;
    r.u = sp.W * sp.G + (int)ub;
    r.k0 = (int)(b - ub * nkt);
    r.k1a = (int)(e < bnd ? e - ub * nkt : nkt);
    r.k1b = (int)(e > bnd ? e - bnd : 0);
    return r;
}

template <int HD, bool WAVE>
__global__ void __launch_bounds__(352, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV, bf16 *__restrict__ o, const int Lq,
                   const int n_keys, const int d, const AttnSplit sp, float *__restrict__ ws_o,
                   float2 *__restrict__ ws_ml, const uint8_t *__restrict__ skip_flag, int *err) {
    pdl_wait();
    using A = AttnTile<HD>;
    if (skip_flag != nullptr && *skip_flag == XC_DEC_SKIP) return;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = align1024_a(smem_raw);
    uint8_t *sQ = smem;
    uint8_t *sK = smem + A::OFF_K;
    uint8_t *sV = smem + A::OFF_V;
    uint64_t *bar = reinterpret_cast<uint64_t *>(smem + A::OFF_BAR);
    uint64_t *q_full = bar;                    // Q of piece p landed (phase p)
    uint64_t *q_empty = bar + 1;               // every S MMA of piece p done (phase p)
    uint64_t *k_full = bar + 2;
    uint64_t *k_empty = k_full + A::STAGES;
    uint64_t *v_full = k_empty + A::STAGES;
    uint64_t *v_empty = v_full + A::STAGES;
    uint64_t *s_full = v_empty + A::STAGES;    // [2] S_i computed
    uint64_t *s_cons = s_full + 2;             // [2] S_i read by its softmax WG (hd 64)
    uint64_t *p_full = s_cons + 2;             // [2] P_i written, O_i corrected
    uint64_t *pv_done = p_full + 2;            // [2] P_i V done (hd 64: every tile; hd 128: last of a piece)
    uint64_t *o_free = pv_done + 2;            // [2] O_i of piece p read out (phase p)
    uint64_t *turn = o_free + 2;               // [2][4] exponential-phase hand-off per (WG, quadrant)
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(turn + 8);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nkt = sp.n_kt;
    const int cta = blockIdx.x;
    long long it0 = 0;
    int n_t;                                       // key tiles of this CTA (>= 1)
    if constexpr (WAVE) {
        n_t = sp.W * nkt + (int)(sp.begin2(cta + 1) - sp.begin2(cta));
    } else {
        it0 = sp.begin(cta);
        n_t = (int)(sp.begin(cta + 1) - it0);
    }
    const int u0 = (int)(it0 / nkt);
    // Waves: this CTA's remainder pieces (registers of the cursor roles),
    // and the tile at which its remainder begins.  The cursor steps like the
    // contiguous one -- next unit after a unit's last key tile -- with a jump
    // to the remainder at tile gw, so the per-tile tests stay the same.
    RemSeg rem{0, 0, 0, 0};
    if constexpr (WAVE) rem = rem_seg(sp, cta);
    const int gw = WAVE ? sp.W * nkt : -1;
    TileCursor c0{0, u0, (int)(it0 % nkt), 0, 1};
    if constexpr (WAVE) c0 = sp.W > 0 ? TileCursor{0, cta, 0, 0, sp.G} : TileCursor{0, rem.u, rem.k0, 0, 1};
    auto piece_of = [&](const TileCursor &c) {    // index of the cursor's piece in this CTA
        if constexpr (WAVE) return c.p;
        else return c.u - u0;
    };
    auto first_of = [&](const TileCursor &c) {
        if constexpr (WAVE) return c.k == 0 || c.g == gw;
        else return c.g == 0 || c.k == 0;
    };
    auto last_of = [&](const TileCursor &c) { return c.g == n_t - 1 || c.k == nkt - 1; };
    auto next = [&](TileCursor &c) {
        ++c.g;
        if (++c.k == nkt) {
            c.k = 0;
            if constexpr (WAVE) {
                c.u += c.du;
                ++c.p;
            } else {
                ++c.u;
            }
        }
        if constexpr (WAVE) {
            if (c.g == gw) {
                c.u = rem.u;
                c.k = rem.k0;
                c.du = 1;
                c.p = sp.W;
            }
        }
    };

    if (threadIdx.x == 0) {
        mbar_init(q_full, 1);
        mbar_init(q_empty, A::ISSUERS);
        for (int s = 0; s < A::STAGES; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&k_empty[s], A::ISSUERS);   // freed by every MMA warp
            mbar_init(&v_full[s], 1);
            mbar_init(&v_empty[s], A::ISSUERS);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&s_full[i], 1);
            mbar_init(&s_cons[i], 128);
            mbar_init(&p_full[i], 128);
            mbar_init(&pv_done[i], 1);
            mbar_init(&o_free[i], 128);
            for (int qd = 0; qd < 4; ++qd) mbar_init(&turn[4 * i + qd], 1);
        }
        mbar_fence_init();
    }
    if (warp == 9) tmem_alloc(tmem_slot, A::TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 8) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            int q_loads = 0, k_issued = 0, v_issued = 0;
            int h = 0;
            for (TileCursor c = c0; c.g < n_t; next(c)) {
                const int g = c.g;
                if (first_of(c)) {
                    const int u = c.u;
                    h = u / sp.n_qblk;
                    const int q0 = (u % sp.n_qblk) * (A::QT * A::BQ);
                    // the previous piece's Q stays until its last S MMA is done
                    if (q_loads > 0 && !mbar_wait(q_empty, (q_loads - 1) & 1, err, ERR_WAIT_PRODUCER)) break;
                    mbar_expect_tx(q_full, A::QT * A::Q_BYTES);
                    for (int i = 0; i < A::QT; ++i)
                        for (int r = 0; r < A::NR; ++r)
                            tma_load_2d(sQ + i * A::Q_BYTES + r * A::REGION, &tmQ, q_full, h * HD + 64 * r,
                                        q0 + i * A::BQ);
                    ++q_loads;
                }
                const int st = g % A::STAGES, kt = c.k;
                const uint32_t ph = ((g / A::STAGES) & 1) ^ 1;
                if (!mbar_wait(&k_empty[st], ph, err, ERR_WAIT_PRODUCER)) break;
                mbar_expect_tx(&k_full[st], A::KV_BYTES);
                for (int r = 0; r < A::NR; ++r)
                    tma_load_2d(sK + st * A::KV_BYTES + r * A::REGION, &tmK, &k_full[st], h * HD + 64 * r,
                                kt * A::BKV);
                k_issued = g + 1;
                if (!mbar_wait(&v_empty[st], ph, err, ERR_WAIT_PRODUCER)) break;
                mbar_expect_tx(&v_full[st], A::KV_BYTES);
                for (int r = 0; r < A::NR; ++r)
                    tma_load_2d(sV + st * A::KV_BYTES + r * A::REGION, &tmV, &v_full[st], h * HD + 64 * r,
                                kt * A::BKV);
                v_issued = g + 1;
            }
            // Drain: every copy this thread started has landed before exit.
            if (q_loads > 0) mbar_wait(q_full, (q_loads - 1) & 1, err, ERR_WAIT_PRODUCER);
            for (int g = k_issued - A::STAGES < 0 ? 0 : k_issued - A::STAGES; g < k_issued; ++g)
                mbar_wait(&k_full[g % A::STAGES], (g / A::STAGES) & 1, err, ERR_WAIT_PRODUCER);
            for (int g = v_issued - A::STAGES < 0 ? 0 : v_issued - A::STAGES; g < v_issued; ++g)
                mbar_wait(&v_full[g % A::STAGES], (g / A::STAGES) & 1, err, ERR_WAIT_PRODUCER);
        }
    } else if (warp >= 9) {
        // ------------------------------------------------------ MMA issue
        // hd 64: warp 9 issues every MMA of Q tile 0, warp 10 those of tile 1,
        // so the issue work is spread over two SM sub-partitions and neither
        // tile waits on the other's softmax.  hd 128: warp 9 alone.  The
        // whole warp runs the loop (converged); one elected lane issues each
        // tcgen05 instruction.
        if (warp == 9 || A::ISSUERS == 2) {
            constexpr uint32_t idesc_s = idesc_bf16(128, 128, false, false);
            constexpr uint32_t idesc_o = idesc_bf16(128, HD, false, true);
            // Descriptors are built once; each MMA adds a constant to the
            // start-address field (addresses stay below 256 KB, so the
            // 14-bit field never carries).
            const uint64_t dQ0 = sdesc_sw128(smem_u32(sQ), 16, 1024);
            const uint64_t dK0 = sdesc_sw128(smem_u32(sK), 16, 1024);
            const uint64_t dV0 = sdesc_sw128(smem_u32(sV), A::REGION, 1024);
            auto issue_s = [&](int i, int g) {        // S_i = Q_i K_g^T
                const uint64_t dq = dQ0 + (uint64_t)((i * A::Q_BYTES) >> 4);
                const uint64_t dk = dK0 + (uint64_t)(((g % A::STAGES) * A::KV_BYTES) >> 4);
#pragma unroll
                for (int ks = 0; ks < HD / 16; ++ks) {
                    const uint32_t off = ((ks >> 2) * A::REGION + (ks & 3) * 32) >> 4;
                    tc_mma_warp(tmem + A::S_COL(i), dq + off, dk + off, idesc_s, ks > 0 ? 1u : 0u);
                }
                tc_commit_warp(&s_full[i]);
            };
            auto issue_pv = [&](int i, const TileCursor &c) {   // O_i (+)= P_i V_g, P_i in TMEM
                const uint64_t dv = dV0 + (uint64_t)(((c.g % A::STAGES) * A::KV_BYTES) >> 4);
                const bool fresh = first_of(c);        // first tile of a piece: O_i = P_i V_g
#pragma unroll
                for (int ks = 0; ks < A::BKV / 16; ++ks)
                    tc_mma_tmem_a_warp(tmem + A::O_COL(i), tmem + A::P_COL(i) + 8 * ks, dv + ((ks * 16 * 128) >> 4),
                                       idesc_o, (!fresh || ks > 0) ? 1u : 0u);
            };
            auto wait = [&](uint64_t *b, int parity) -> bool {
                const bool r = mbar_wait(b, parity & 1, err, ERR_WAIT_MMA);
                return __all_sync(0xffffffffu, r) != 0;
            };
            // S of tile g needs its piece's Q (and, after a piece's last S,
            // the producer may replace Q); P V of the first tile of a piece
            // overwrites O, so it waits until the softmax has read O out.
            auto s_ready = [&](const TileCursor &c) -> bool {
                if (first_of(c) && !wait(q_full, piece_of(c))) return false;
                return wait(&k_full[c.g % A::STAGES], c.g / A::STAGES);
            };
            auto pv_ready = [&](int i, const TileCursor &c) -> bool {
                if (first_of(c) && piece_of(c) > 0 && !wait(&o_free[i], piece_of(c) - 1)) return false;
                return wait(&p_full[i], c.g) && wait(&v_full[c.g % A::STAGES], c.g / A::STAGES);
            };
            if constexpr (A::SEP_P) {
                // hd 64: S_i(g+1) is issued once the softmax has read S_i(g) (P
                // has its own columns), then P_i V_g once P_i is ready.
                const int i = warp - 9;
                bool ok = s_ready(c0);
                if (ok) {
                    tc_fence_after();
                    issue_s(i, 0);
                    tc_commit_warp(&k_empty[0]);
                    if (last_of(c0)) tc_commit_warp(q_empty);
                }
                TileCursor cs = c0;                    // next S tile is cs + 1
                for (TileCursor c = c0; ok && c.g < n_t; next(c)) {
                    const int g = c.g;
                    if (g + 1 < n_t) {
                        next(cs);
                        if (!(wait(&s_cons[i], g) && s_ready(cs))) break;
                        tc_fence_after();
                        issue_s(i, g + 1);
                        tc_commit_warp(&k_empty[(g + 1) % A::STAGES]);
                        if (last_of(cs)) tc_commit_warp(q_empty);
                    }
                    if (!pv_ready(i, c)) break;
                    tc_fence_after();
                    issue_pv(i, c);
                    tc_commit_warp(&pv_done[i]);
                    tc_commit_warp(&v_empty[g % A::STAGES]);
                }
            } else {
                // hd 128: one warp issues P0V(g), S0(g+1), P1V(g), S1(g+1) -- the
                // order in which the warpgroups finish their turns; P_i
                // overwrites S_i, so S_i(g+1) follows P_i V_g.
                bool ok = s_ready(c0);
                if (ok) {
                    tc_fence_after();
                    issue_s(0, 0);
                    issue_s(1, 0);
                    tc_commit_warp(&k_empty[0]);
                    if (last_of(c0)) tc_commit_warp(q_empty);
                }
                TileCursor cs = c0;                    // next S tile is cs + 1
                for (TileCursor c = c0; ok && c.g < n_t; next(c)) {
                    const int g = c.g;
                    const bool more = g + 1 < n_t;
                    if (more) next(cs);
                    if (!pv_ready(0, c)) break;
                    tc_fence_after();
                    issue_pv(0, c);
                    if (last_of(c)) tc_commit_warp(&pv_done[0]);
                    if (more) {
                        if (!s_ready(cs)) break;
                        tc_fence_after();
                        issue_s(0, g + 1);
                    }
                    if (!pv_ready(1, c)) break;
                    tc_fence_after();
                    issue_pv(1, c);
                    tc_commit_warp(&v_empty[g % A::STAGES]);
                    if (last_of(c)) tc_commit_warp(&pv_done[1]);
                    if (more) {
                        issue_s(1, g + 1);
                        tc_commit_warp(&k_empty[(g + 1) % A::STAGES]);
                        if (last_of(cs)) tc_commit_warp(q_empty);
                    }
                }
            }
        }
    } else {
        // ------------------------------------------------------------ softmax
        const int wg = warp >> 2;                          // tile of this warpgroup
        const int q = warp & 3;                            // TMEM lane quadrant
        const int r_tile = wg * A::BQ + q * 32 + lane;     // row within the unit (0..255)
        const uint32_t tl = tmem + ((uint32_t)(q * 32) << 16);
        const uint32_t tS = tl + A::S_COL(wg);
        const uint32_t tP = tl + A::P_COL(wg);
        const uint32_t tO = tl + A::O_COL(wg);
        const float sl2 = rsqrtf((float)HD) * 1.4426950408889634f;
        const int tail = n_keys - (nkt - 1) * A::BKV;      // valid keys in the last tile
        // One key tile g (key tile kt of its unit): S_i -> running max m,
        // P_i = 2^(S_i sl2 - m) into TMEM, running sum l.  false: a wait ran out.
        auto tile = [&](int g, int kt, bool fresh, float &m, float &l) -> bool {
            bool ok = mbar_wait(&s_full[wg], g & 1, err, ERR_WAIT_SOFTMAX);
            __syncwarp();
            if (!__all_sync(0xffffffffu, ok)) return false;
            tc_fence_after();
            float s[128];
            tmem_ld128_sync(tS, s);
            if constexpr (A::SEP_P) {
                tc_fence_before();
                mbar_arrive(&s_cons[wg]);
            }
            if (kt == nkt - 1 && tail < A::BKV) {
#pragma unroll
                for (int c = 0; c < 128; ++c)
                    if (c >= tail) s[c] = -INFINITY;
            }
            // row max: 16 independent chains of three-input max over columns
            // 0..111, the last 16 columns, then a tree
            float mx[16];
#pragma unroll
            for (int k = 0; k < 16; ++k) mx[k] = s[k];
#pragma unroll
            for (int c = 16; c < 112; c += 32) {
#pragma unroll
                for (int k = 0; k < 16; ++k) mx[k] = fmax3(mx[k], s[c + k], s[c + 16 + k]);
            }
#pragma unroll
            for (int k = 0; k < 16; ++k) mx[k] = fmaxf(mx[k], s[112 + k]);
#pragma unroll
            for (int k = 0; k < 5; ++k) mx[k] = fmax3(mx[k], mx[k + 5], mx[k + 10]);
            const float m_new = fmax3(fmax3(mx[0], mx[1], mx[2]), fmax3(mx[3], mx[4], mx[15]), mx[0]) * sl2;
            if (fresh) m = m_new;
            const bool grow = !fresh && m_new > m + A::LAZY;
            const float alpha = grow ? ex2_approx(m - m_new) : 1.0f;
            if (grow) m = m_new;
            if constexpr (A::SEP_P) {
                // P_i buffer free and O_i stable once P V of the previous tile is done
                if (g >= 1) {
                    ok = mbar_wait(&pv_done[wg], (g - 1) & 1, err, ERR_WAIT_SOFTMAX);
                    __syncwarp();
                    if (!__all_sync(0xffffffffu, ok)) return false;
                    tc_fence_after();
                }
            }
            // (hd 128: the commit behind s_full already covers P V of tile g-1)
            if (__any_sync(0xffffffffu, grow)) {
#pragma unroll 1
                for (int c = 0; c < HD / 16; ++c) {
                    float t[16];
                    tmem_ld16_sync(tO + 16 * c, t);
#pragma unroll
                    for (int i = 0; i < 16; ++i) t[i] *= alpha;
                    tmem_st16_sync(tO + 16 * c, t);
                }
            }
            // The two warps of each SM sub-partition (quadrant q of WG 0 and
            // of WG 1) take turns on the exponential phase, which is bound
            // by the sub-partition's MUFU: WG 0 does tile g, then WG 1 tile
            // g, then WG 0 tile g + 1 ... so that one warp's exponentials
            // overlap the other's loads, max and MMA waits.  The hand-off is
            // per quadrant, so a slower sub-partition does not hold up the
            // others.
            // (hd 128: the turns cost more than they save -- the exponential
            // phase is a smaller share of a key tile's work; 7.27 -> 7.16 ms
            // at the 14B shape, 1.91 -> 1.85 ms at the 1.3B shape)
            if constexpr (A::SEP_P) {
                if (wg == 1 || g > 0) {
                    ok = mbar_wait(&turn[4 * wg + q], (wg == 1 ? g : g - 1) & 1, err, ERR_WAIT_SOFTMAX);
                    __syncwarp();
                    if (!__all_sync(0xffffffffu, ok)) return false;
                }
            }
            // probabilities p = 2^(s * sl2 - m), packed bf16 pairs + row sum,
            // stored to TMEM in four 32-key quarters
            const float2 sc2 = make_float2(sl2, sl2), nm2 = make_float2(-m, -m);
            float2 rs0 = make_float2(0.f, 0.f), rs1 = make_float2(0.f, 0.f);
#pragma unroll
            for (int qt = 0; qt < 4; ++qt) {
                uint32_t w[16];
#pragma unroll
                for (int k = 0; k < 16; k += 2) {
                    const int c = 32 * qt + 2 * k;
                    const float2 a = __ffma2_rn(make_float2(s[c], s[c + 1]), sc2, nm2);
                    const float2 b = __ffma2_rn(make_float2(s[c + 2], s[c + 3]), sc2, nm2);
                    const float2 pa = make_float2(ex2_approx(a.x), ex2_approx(a.y));
                    const float2 pb = make_float2(ex2_approx(b.x), ex2_approx(b.y));
                    rs0 = __fadd2_rn(rs0, pa);
                    rs1 = __fadd2_rn(rs1, pb);
                    __nv_bfloat162 h0 = __floats2bfloat162_rn(pa.x, pa.y);
                    __nv_bfloat162 h1 = __floats2bfloat162_rn(pb.x, pb.y);
                    w[k] = *reinterpret_cast<uint32_t *>(&h0);
                    w[k + 1] = *reinterpret_cast<uint32_t *>(&h1);
                }
                tmem_st16u_sync(tP + 16 * qt, w);
            }
            const float2 rs = __fadd2_rn(rs0, rs1);
            l = l * alpha + (rs.x + rs.y);
            tc_fence_before();
            mbar_arrive(&p_full[wg]);
            __syncwarp();
            if (lane == 0) mbar_arrive(&turn[4 * (wg ^ 1) + q]);
            return true;
        };
        // End of a piece (its last tile g, unit u, piece p of this CTA): O_i
        // complete -> output (whole unit) or partial.
        auto end_piece = [&](int g, int u, int p, bool head_part, bool cut_front, float m, float l) -> bool {
            const bool ok = mbar_wait(&pv_done[wg], (A::SEP_P ? g : p) & 1, err, ERR_WAIT_SOFTMAX);
            __syncwarp();
            if (!__all_sync(0xffffffffu, ok)) return false;
            tc_fence_after();
            const int h = u / sp.n_qblk;
            const int row = (u % sp.n_qblk) * (A::QT * A::BQ) + r_tile;
            if (!head_part && !cut_front) {
                const float inv = 1.0f / l;
#pragma unroll 1
                for (int c = 0; c < HD / 16; ++c) {
                    float t[16];
                    tmem_ld16_sync(tO + 16 * c, t);
#pragma unroll
                    for (int i = 0; i < 16; ++i) t[i] *= inv;
                    if (row < Lq) store16<bf16>(o + (size_t)row * d + h * HD + 16 * c, t);
                }
            } else {
                const int slot = WAVE ? 2 * cta + (p - sp.W)                       // remainder piece 0 / 1
                                      : (head_part ? 2 * (cta + 1) : 2 * cta + 1);   // boundary c + 1 head / c tail
                float *wo = ws_o + ((size_t)slot * (A::QT * A::BQ) + r_tile) * HD;
#pragma unroll 1
                for (int c = 0; c < HD / 16; ++c) {
                    float t[16];
                    tmem_ld16_sync(tO + 16 * c, t);
                    store16<float>(wo + 16 * c, t);
                }
                ws_ml[(size_t)slot * (A::QT * A::BQ) + r_tile] = make_float2(m, l);
            }
            tc_fence_before();
            mbar_arrive(&o_free[wg]);
            return true;
        };
        bool ok = true;
        TileCursor cur = c0;
        while (ok && cur.g < n_t) {
            const bool cut_front = cur.k != 0;     // the piece's unit began in another CTA
            float m = -INFINITY, l = 0.0f;
            bool fresh = true;
            for (;;) {
                ok = tile(cur.g, cur.k, fresh, m, l);
                if (!ok) break;
                fresh = false;
                if (last_of(cur)) break;
                next(cur);
            }
            if (!ok) break;
            ok = end_piece(cur.g, cur.u, piece_of(cur), cur.k != nkt - 1, cut_front, m, l);
            next(cur);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc_fence_after();
        tmem_dealloc(tmem, A::TMEM_COLS);
    }
}

// Merges the partials of the units cut between CTAs (see AttnSplit): m =
// max_p m_p, O = sum_p O_p 2^(m_p - m) / sum_p l_p 2^(m_p - m).  Contiguous
// order: grid.x = CTA boundaries, two partials (head and tail) of the unit
// the boundary cuts.  Waves: grid.x = remaining units, the partials of the
// CTAs whose pieces touch it, in CTA order (up to G / R of them).  grid.y
// picks 32 of the head's columns, grid.z 64 of the unit's 256 query rows;
// one thread per row.
constexpr int COMBINE_ROWS = 64, COMBINE_COLS = 32;
template <int HD, bool WAVE>
__global__ void __launch_bounds__(COMBINE_ROWS)
    attn_combine_kernel(bf16 *__restrict__ o, const int Lq, const int d, const AttnSplit sp,
                        const float *__restrict__ ws_o, const float2 *__restrict__ ws_ml,
                        const uint8_t *__restrict__ skip_flag) {
    pdl_wait();
    if (skip_flag != nullptr && *skip_flag == XC_DEC_SKIP) return;
    int u, c_lo, c_hi;
    long long ub = 0;
    if constexpr (WAVE) {
        const int rr = blockIdx.x;                     // remaining unit
        ub = (long long)rr * sp.n_kt;
        const long long ue = ub + sp.n_kt;
        c_lo = (int)(ub * sp.G / sp.T2);               // begin2(c_lo) <= ub
        while (c_lo + 1 < sp.G && sp.begin2(c_lo + 1) <= ub) ++c_lo;
        c_hi = c_lo;                                   // last CTA whose piece touches the unit
        while (c_hi + 1 < sp.G && sp.begin2(c_hi + 1) < ue) ++c_hi;
        if (c_hi == c_lo) return;                      // one CTA ran the whole unit and wrote it
        u = sp.W * sp.G + rr;
    } else {
        const int b = blockIdx.x + 1;                  // boundary between CTAs b-1 and b
        const long long it = sp.begin(b);
        if (it % sp.n_kt == 0) return;                 // the boundary falls between units
        u = (int)(it / sp.n_kt);
        c_lo = b - 1;
        c_hi = b;
    }
    const int h = u / sp.n_qblk;
    const int r = blockIdx.z * COMBINE_ROWS + threadIdx.x;     // row of the unit
    const int k0 = blockIdx.y * COMBINE_COLS;
    const int row = (u % sp.n_qblk) * 256 + r;
    if (row >= Lq) return;
    // slot of CTA c's partial of this unit
    auto slot = [&](int c) {
        if constexpr (WAVE) return 2 * c + (sp.begin2(c) >= ub ? 0 : 1);
        else return c == c_lo ? 2 * c_hi : 2 * c_hi + 1;
    };
    auto has = [&](int c) {
        if constexpr (WAVE) return sp.begin2(c + 1) > sp.begin2(c);
        else return true;
    };
    float mm = -INFINITY;
    for (int c = c_lo; c <= c_hi; ++c)
        if (has(c)) mm = fmaxf(mm, ws_ml[(size_t)slot(c) * 256 + r].x);
    float den = 0.0f;
    float acc[COMBINE_COLS];
#pragma unroll
    for (int i = 0; i < COMBINE_COLS; ++i) acc[i] = 0.0f;
#pragma unroll 2
    for (int c = c_lo; c <= c_hi; ++c) {
        if (!has(c)) continue;
        const int sl = slot(c);
        const float2 ml = ws_ml[(size_t)sl * 256 + r];
        const float w = exp2f(ml.x - mm);
        den += ml.y * w;
        const float *src = ws_o + ((size_t)sl * 256 + r) * HD + k0;
#pragma unroll
        for (int j = 0; j < COMBINE_COLS; j += 16) {
            float x[16];
            load16<float>(src + j, x);
#pragma unroll
            for (int i = 0; i < 16; ++i) acc[j + i] = fmaf(x[i], w, acc[j + i]);
        }
    }
    const float inv = 1.0f / den;
#pragma unroll
    for (int j = 0; j < COMBINE_COLS; j += 16) {
        float y[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) y[i] = acc[j + i] * inv;
        store16<bf16>(o + (size_t)row * d + h * HD + k0 + j, y);
    }
}

bool make_tmap_bf16(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint32_t box_rows);

static int sm_count() {
    static int n = 0;
    if (n == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) n = 1;
    }
    return n;
}

size_t attn_workspace_bytes(int head_dim) {
    const size_t slots = 2 * ((size_t)sm_count() + 1);
    return slots * 256 * ((size_t)head_dim * sizeof(float) + sizeof(float2));
}

template <int HD, bool WAVE>
static cudaError_t launch_attn_(const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &tv, bf16 *o,
                                int Lq, int n_keys, int d, const AttnSplit &sp, bool split, int n_combine, void *ws,
                                const uint8_t *skip, int *err, int *n_launched, cudaStream_t st) {
    using A = AttnTile<HD>;
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<HD, WAVE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             A::SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const int n_sm = sm_count();
    float *ws_o = split ? reinterpret_cast<float *>(ws) : nullptr;
    float2 *ws_ml = split ? reinterpret_cast<float2 *>(ws_o + 2 * ((size_t)n_sm + 1) * 256 * HD) : nullptr;
    cudaError_t e = launch_pdl(attn_tc_kernel<HD, WAVE>, dim3(sp.G), dim3(A::THREADS), A::SMEM_BYTES, st, tq, tk,
                               tv, o, Lq, n_keys, d, sp, ws_o, ws_ml, skip, err);
    if (e != cudaSuccess) return e;
    if (n_launched) *n_launched = 1;
    if (split && n_combine > 0) {
        e = launch_pdl(attn_combine_kernel<HD, WAVE>, dim3(n_combine, HD / COMBINE_COLS, 256 / COMBINE_ROWS),
                       dim3(COMBINE_ROWS), 0, st, o, Lq, d, sp,
                       static_cast<const float *>(ws_o), static_cast<const float2 *>(ws_ml), skip);
        if (n_launched) *n_launched = 2;
    }
    return e;
}

// Work order (see AttnSplit): waves when there are many of them (W >= 8)
// and the K / V of all heads exceed L2 -- measured at the 14B shape (40
// heads x 20 MB of K / V, W = 13): 40.7 -> 1.2 GB of DRAM traffic per launch
// at the same attention time, the GPU's power then allowing a higher clock
// under its cap (1500 -> 1965 MHz, 0.766 -> 0.801 chunks/s); at the 1.3B
// shape (W = 4) the waves were 28 % slower per launch, the contiguous order
// stays.
template <int HD>
static cudaError_t launch_attn(const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &tv, bf16 *o,
                               int Lq, int n_keys, int n_heads, int d, void *ws, size_t ws_bytes,
                               const uint8_t *skip, int *err, int *n_launched, cudaStream_t st) {
    using A = AttnTile<HD>;
    AttnSplit sp;
    sp.n_kt = (n_keys + A::BKV - 1) / A::BKV;
    sp.n_qblk = (Lq + A::QT * A::BQ - 1) / (A::QT * A::BQ);
    const int n_units = sp.n_qblk * n_heads;
    sp.T = (long long)n_units * sp.n_kt;
    const int n_sm = sm_count();
    const bool split = n_units > n_sm && ws != nullptr && ws_bytes >= attn_workspace_bytes(HD);
    sp.G = split ? n_sm : n_units;
    sp.W = n_units / sp.G;
    const int n_rem = n_units - sp.W * sp.G;
    sp.T2 = (long long)n_rem * sp.n_kt;
    const double kv_bytes = 2.0 * n_keys * (double)d * sizeof(bf16);
    const bool wave = split && sp.W >= 8 && kv_bytes > 128.0 * 1024 * 1024;
    if (wave)
        return launch_attn_<HD, true>(tq, tk, tv, o, Lq, n_keys, d, sp, split, n_rem, ws, skip, err, n_launched, st);
    return launch_attn_<HD, false>(tq, tk, tv, o, Lq, n_keys, d, sp, split, sp.G - 1, ws, skip, err, n_launched,
                                   st);
}

// q [Lq][d], k / v maps over [>= n_keys][d] (box 128 rows), o [Lq][d]; hd in {64, 128}.
// ws: attn_workspace_bytes(hd) bytes enable the balanced split over the SMs
// when there are more units than SMs (nullptr: one CTA per unit).
cudaError_t attn_tc(int head_dim, const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &tv,
                    bf16 *o, int Lq, int n_keys, int n_heads, int d, void *ws, size_t ws_bytes,
                    const uint8_t *skip, int *err, int *n_launched, cudaStream_t st) {
    if (n_keys < 1 || Lq < 1) return cudaErrorInvalidValue;
    if (head_dim == 64)
        return launch_attn<64>(tq, tk, tv, o, Lq, n_keys, n_heads, d, ws, ws_bytes, skip, err, n_launched, st);
    if (head_dim == 128)
        return launch_attn<128>(tq, tk, tv, o, Lq, n_keys, n_heads, d, ws, ws_bytes, skip, err, n_launched, st);
    return cudaErrorInvalidValue;
}

}  // namespace xc
