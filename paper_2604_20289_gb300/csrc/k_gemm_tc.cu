// bf16 GEMM on the 5th-generation tensor core (tcgen05), fed by TMA.
//
//   C[M][N] = epilogue(A[M][K] @ Wt[N][K]^T), fp32 accumulation in TMEM.
//
// Persistent: one CTA per SM walks the 128 x BN output tiles round-robin
// (n fastest, so the CTAs running at the same time share A tiles in L2).
// Warp roles (320 threads):
//   warp 0, lane 0 : TMA producer, STAGES-deep ring of (A 128x64, B BNx64)
//                    tiles in 128B-swizzled shared memory, continuous across
//                    output tiles;
//   warp 1         : allocates TMEM (two BN-column accumulators) and issues
//                    tcgen05.mma (M=128, N=BN, K=16; 4 per 64-wide k-tile)
//                    into the free accumulator from a converged warp;
//   warps 2..9     : epilogue, two warps per TMEM lane quadrant, half of the
//                    columns each, in 32 x 32 blocks: thread = row, the
//                    block's residual operands arrive in shared memory by
//                    TMA, the fused epilogue (bias / GELU / gated residual /
//                    residual cache / RoPE) runs in registers, and the bf16
//                    block leaves by a TMA store from a 64B-swizzled staging
//                    buffer.  The accumulator is released after its last
//                    TMEM read, so the epilogue of tile i overlaps the main
//                    loop of tile i + 1.
// The skip flag of the block lets the whole recompute path early-exit when
// the gate chose reuse (Eq. 4), so decisions never return to the host.
#include <cstring>
#include <mutex>
#include <unordered_map>

#include "xc_ptx.cuh"

namespace xc {

constexpr int GEMM_BM = 128;
constexpr int GEMM_BK = 64;
constexpr int GEMM_SMEM_LIMIT = 232448;        // dynamic shared memory per CTA on this part
constexpr int EPI_BLOCK_BYTES = 32 * 32 * 2;   // one 32 x 32 bf16 block

// Residual-cache epilogue with 256-wide tiles: the residual and block-input
// blocks are loaded into the two buffers that then stage the output and
// r_hat, so the main loop keeps four pipeline stages in shared memory (the
// next blocks' loads wait until the stores have read the buffers).
template <int EPI, int BN>
__host__ __device__ constexpr bool epi_shared() {
    return EPI == EPI_RESID_CACHE && BN == 256;
}
// Staging blocks per epilogue warp: residual cache: out, r_hat, resid, x_in
// (2 when shared); gated residual: out, resid; the others: out,
// double-buffered.
template <int EPI, int BN>
__host__ __device__ constexpr int epi_blocks() {
    return (EPI == EPI_RESID_CACHE && !epi_shared<EPI, BN>()) ? 4 : 2;
}

template <int BN, int EPI>
struct GemmTile {
    static constexpr int A_BYTES = GEMM_BM * GEMM_BK * 2;
    static constexpr int B_BYTES = BN * GEMM_BK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int EPI_BYTES = 8 * epi_blocks<EPI, BN>() * EPI_BLOCK_BYTES;
    static constexpr int BAR_BYTES = 512;
    static constexpr int FIT = (GEMM_SMEM_LIMIT - 1024 - BAR_BYTES - EPI_BYTES) / STAGE_BYTES;
    static constexpr int STAGES = FIT > 6 ? 6 : FIT;
    static constexpr int OFF_EPI = STAGES * STAGE_BYTES;                // 1024-aligned
    static constexpr int BAR_OFFSET = OFF_EPI + EPI_BYTES;
    static constexpr int SMEM_BYTES = BAR_OFFSET + BAR_BYTES + 1024;   // + alignment slack
    static constexpr int TMEM_COLS = 2 * BN;                             // double-buffered accumulator
    static constexpr int EPI_THREADS = 256;
    static_assert(STAGES >= 3, "main-loop ring too shallow");
    static_assert(SMEM_BYTES <= GEMM_SMEM_LIMIT, "shared memory");
};

// Tensor maps of the epilogue (32 x 32 bf16 boxes, 64-byte swizzle):
// out[0..2] = q, k, v for the QKV epilogue, out[0] otherwise.
struct EpiMaps {
    CUtensorMap out[3];
    CUtensorMap rhat, resid, xin;
};

__device__ __forceinline__ uint8_t *align1024(uint8_t *p) {
    const uint32_t s = smem_u32(p);
    return p + ((1024u - (s & 1023u)) & 1023u);
}

// Byte offset of 16-byte chunk k (0..3) of row r in a 64B-swizzled 32 x 32
// bf16 block (the layout TMA reads and writes with CU_TENSOR_MAP_SWIZZLE_64B).
__device__ __forceinline__ uint32_t sw64(int r, int k) { return (uint32_t)(r * 64 + ((k ^ ((r >> 1) & 3)) << 4)); }

__device__ __forceinline__ void tma_store_2d(const CUtensorMap *tm, const void *src, int x, int y) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];"
                 ::"l"(reinterpret_cast<uint64_t>(tm)), "r"(smem_u32(src)), "r"(x), "r"(y)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// 32 bf16 of row r from a swizzled block -> float
__device__ __forceinline__ void read_row32(const uint8_t *blk, int r, float (&v)[32]) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint4 u = *reinterpret_cast<const uint4 *>(blk + sw64(r, k));
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float2 t = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&w[j]));
            v[8 * k + 2 * j] = t.x;
            v[8 * k + 2 * j + 1] = t.y;
        }
    }
}
// float -> 32 bf16 (round to nearest) into row r of a swizzled block
__device__ __forceinline__ void write_row32(uint8_t *blk, int r, const float (&v)[32]) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        uint32_t w[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            __nv_bfloat162 h = __floats2bfloat162_rn(v[8 * k + 2 * j], v[8 * k + 2 * j + 1]);
            w[j] = *reinterpret_cast<uint32_t *>(&h);
        }
        *reinterpret_cast<uint4 *>(blk + sw64(r, k)) = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

// Persistent tile order: tile t -> (m block, n block).  Tiles go in
// super-rows of GEMM_GROUP_M m blocks with m varying fastest inside a
// super-row, so the tiles in flight at one time (one per SM) share
// GEMM_GROUP_M row blocks of A and a few column blocks of B -- an
// L2-resident working set -- instead of all of B streaming through L2 for
// every row of m blocks (row-major order re-read B from DRAM once per 2-3
// m-block rows on the large-N projections).
constexpr int GEMM_GROUP_M = 16;
__device__ __forceinline__ void tile_mn(int tile, int tiles_m, int tiles_n, int &mb, int &nb) {
    const int per = GEMM_GROUP_M * tiles_n;
    const int grp = tile / per;
    const int first = grp * GEMM_GROUP_M;
    const int gm = min(GEMM_GROUP_M, tiles_m - first);
    const int loc = tile - grp * per;
    mb = first + loc % gm;
    nb = loc / gm;
}

template <int BN, int EPI>
__global__ void __launch_bounds__(320, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ EpiMaps em, const EpiParams ep, const int K,
                   const uint8_t *__restrict__ skip_flag, int *err) {
    pdl_wait();
    using G = GemmTile<BN, EPI>;
    if (skip_flag != nullptr && *skip_flag == XC_DEC_SKIP) return;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = align1024(smem_raw);
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + G::BAR_OFFSET);
    uint64_t *empty = full + G::STAGES;
    uint64_t *acc_full = empty + G::STAGES;    // [2]
    uint64_t *acc_empty = acc_full + 2;        // [2]
    uint64_t *ld_bar = acc_empty + 2;          // [8] residual operands of an epilogue warp landed
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(ld_bar + 8);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int KT = K / GEMM_BK;
    const int tiles_n = ep.N / BN;
    const int tiles_m = (ep.M + GEMM_BM - 1) / GEMM_BM;
    const int n_tiles = tiles_m * tiles_n;

    if (threadIdx.x == 0) {
        for (int s = 0; s < G::STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], G::EPI_THREADS);
        }
        for (int w = 0; w < 8; ++w) mbar_init(&ld_bar[w], 1);
        mbar_fence_init();
    }
    if (warp == 1) tmem_alloc(tmem_slot, G::TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            int it = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < n_tiles; tile += gridDim.x) {
                int mb, nb;
                tile_mn(tile, tiles_m, tiles_n, mb, nb);
                const int m0 = mb * GEMM_BM, n0 = nb * BN;
                for (int kt = 0; kt < KT; ++kt, ++it) {
                    const int s = it % G::STAGES;
                    const uint32_t ph = (it / G::STAGES) & 1;
                    if (!mbar_wait(&empty[s], ph ^ 1, err, ERR_WAIT_PRODUCER)) {
                        ok = false;
                        break;
                    }
                    uint8_t *sa = smem + s * G::STAGE_BYTES;
                    mbar_expect_tx(&full[s], G::STAGE_BYTES);
                    tma_load_2d(sa, &tmA, &full[s], kt * GEMM_BK, m0);
                    tma_load_2d(sa + G::A_BYTES, &tmB, &full[s], kt * GEMM_BK, n0);
                }
            }
            // Drain: every copy this thread started has landed before exit.
            for (int j = it - G::STAGES < 0 ? 0 : it - G::STAGES; j < it; ++j)
                mbar_wait(&full[j % G::STAGES], (j / G::STAGES) & 1, err, ERR_WAIT_PRODUCER);
        }
    } else if (warp == 1) {
        // MMA issue: the whole warp runs the loop (converged) and one elected
        // lane issues each tcgen05 instruction, so issue keeps pace while the
        // epilogue warps of the same sub-partitions are busy.
        {
            constexpr uint32_t idesc = idesc_bf16(GEMM_BM, BN, false, false);
            auto wait = [&](uint64_t *b, uint32_t parity) {
                const bool r = mbar_wait(b, parity, err, ERR_WAIT_MMA);
                return __all_sync(0xffffffffu, r);
            };
            // start-address field += offset >> 4 (shared addresses < 256 KB: no carry)
            const uint64_t d0 = sdesc_sw128(smem_u32(smem), 16, 1024);
            int it = 0, local = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < n_tiles; tile += gridDim.x, ++local) {
                const int buf = local & 1;
                const uint32_t use = (uint32_t)(local >> 1);
                if (!wait(&acc_empty[buf], (use & 1) ^ 1)) break;
                tc_fence_after();
                const uint32_t acc = tmem + buf * BN;
                for (int kt = 0; kt < KT; ++kt, ++it) {
                    const int s = it % G::STAGES;
                    if (!wait(&full[s], (it / G::STAGES) & 1)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t da = d0 + (uint64_t)((s * G::STAGE_BYTES) >> 4);
                    const uint64_t db = da + (uint64_t)(G::A_BYTES >> 4);
#pragma unroll
                    for (int k = 0; k < GEMM_BK / 16; ++k)
                        tc_mma_warp(acc, da + 2 * k, db + 2 * k, idesc, (kt | k) != 0 ? 1u : 0u);
                    tc_commit_warp(&empty[s]);
                }
                tc_commit_warp(&acc_full[buf]);
            }
        }
    } else {
        // ---------------------------------------------------------- epilogue
        // Warp ew = warp - 2 owns TMEM lane quadrant q (rows q*32 .. q*32+31 of
        // the tile; thread = row) and column half `half`, in 32-column blocks.
        constexpr bool RES = EPI == EPI_RESID_GATE || EPI == EPI_RESID_CACHE;
        constexpr bool CACHE = EPI == EPI_RESID_CACHE;
        constexpr bool SHARED = epi_shared<EPI, BN>();
        const int ew = warp - 2;
        const int q = warp & 3;
        const int half = ew >> 2;
        const uint32_t tq = tmem + ((uint32_t)(q * 32) << 16);
        uint8_t *eb = smem + G::OFF_EPI + ew * epi_blocks<EPI, BN>() * EPI_BLOCK_BYTES;
        uint8_t *s_out0 = eb;
        uint8_t *s_aux = eb + EPI_BLOCK_BYTES;          // r_hat (cache) / resid (gate) / second out
        uint8_t *s_res = (CACHE && !SHARED) ? eb + 2 * EPI_BLOCK_BYTES : (SHARED ? s_out0 : s_aux);
        uint8_t *s_xin = SHARED ? s_aux : eb + 3 * EPI_BLOCK_BYTES;
        uint64_t *lb = &ld_bar[ew];
        const bool has_rhat = CACHE && ep.rhat != nullptr;
        const uint32_t ld_bytes = (uint32_t)EPI_BLOCK_BYTES * (has_rhat ? 2u : 1u);
        uint32_t n_ld = 0;                               // TMA loads issued on lb (its phases)
        int n_st = 0;                                    // staging blocks written (out double-buffering)
        auto load_res = [&](int m0, int col) {           // resid (+ x_in) block -> shared memory
            if (lane == 0) {
                mbar_expect_tx(lb, ld_bytes);
                tma_load_2d(s_res, &em.resid, lb, col, m0 + q * 32);
                if (has_rhat) tma_load_2d(s_xin, &em.xin, lb, col, m0 + q * 32);
            }
            ++n_ld;
        };
        int local = 0;
        bool ok = true;
        for (int tile = blockIdx.x; ok && tile < n_tiles; tile += gridDim.x, ++local) {
            const int buf = local & 1;
            const uint32_t use = (uint32_t)(local >> 1);
            int mb, nb;
            tile_mn(tile, tiles_m, tiles_n, mb, nb);
            const int m0 = mb * GEMM_BM, n0 = nb * BN;
            const int row = m0 + q * 32 + lane;
            if constexpr (SHARED) {
                if (lane == 0) bulk_wait_read<0>();
                __syncwarp();
            }
            if constexpr (RES) load_res(m0, n0 + half * (BN / 2));
            // RoPE position of this thread's row (camera, frame, h, w), once per tile
            int pos0 = 0, pos1 = 0, pos2 = 0, pos3 = 0;
            if constexpr (EPI == EPI_QKV_ROPE) {
                const int4 tp = token_pos(ep, row);
                pos0 = tp.x;
                pos1 = tp.y;
                pos2 = tp.z;
                pos3 = tp.w;
            }
            // bias (and gate) of this thread's columns, one value per lane,
            // fetched one 32-column block ahead and broadcast by shuffles
            const int colw = n0 + half * (BN / 2);
            float b_next = ep.bias[colw + lane];
            float g_next = 0.0f;
            if constexpr (RES) g_next = ep.gate[colw + lane];
            ok = mbar_wait(&acc_full[buf], use & 1, err, ERR_WAIT_EPI);
            __syncwarp();
            if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
            tc_fence_after();
#pragma unroll 1
            for (int j = 0; j < BN / 64; ++j) {
                const int c = half * (BN / 2) + 32 * j;
                const int col = n0 + c;
                const float b_cur = b_next, g_cur = g_next;
                if (j + 1 < BN / 64) {
                    b_next = ep.bias[col + 32 + lane];
                    if constexpr (RES) g_next = ep.gate[col + 32 + lane];
                }
                float v[32];
                tmem_ld32_sync(tq + buf * BN + c, v);
                if (j == BN / 64 - 1) {
                    // last TMEM read of this tile: hand the accumulator back
                    tc_fence_before();
                    mbar_arrive(&acc_empty[buf]);
                }
#pragma unroll
                for (int i = 0; i < 32; ++i) v[i] += __shfl_sync(0xffffffffu, b_cur, i);
                float xi[32];
                if constexpr (RES) {
                    ok = mbar_wait(lb, (n_ld - 1) & 1, err, ERR_WAIT_EPI);
                    __syncwarp();
                    if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
                    float r[32];
                    read_row32(s_res, lane, r);
                    if constexpr (CACHE)
                        if (has_rhat) read_row32(s_xin, lane, xi);
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = r[i] + __shfl_sync(0xffffffffu, g_cur, i) * v[i];
                    __syncwarp();                      // every lane has read the block
                    if (!SHARED && j + 1 < BN / 64) load_res(m0, col + 32);
                }
                if constexpr (EPI == EPI_GELU) {
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = gelu_tanh_approx(v[i]);
                }
                int part = 0, cl = col;
                if constexpr (EPI == EPI_QKV_ROPE) {
                    part = col / ep.d;
                    cl = col - part * ep.d;
                    if (part < 2 && row < ep.M) {
                        const int pair0 = (cl % ep.head_dim) >> 1;
#pragma unroll
                        for (int k = 0; k < 16; ++k) {
                            const int pr = pair0 + k;
                            const int ax = ep.rope_axis[pr];
                            const int pa = ax == 0 ? pos0 : (ax == 1 ? pos1 : (ax == 2 ? pos2 : pos3));
                            const float2 t = ep.rope_cs[ep.rope_off[pr] + pa];
                            const float x0 = v[2 * k], x1 = v[2 * k + 1];
                            v[2 * k] = x0 * t.x - x1 * t.y;
                            v[2 * k + 1] = x0 * t.y + x1 * t.x;
                        }
                    }
                }
                // staging: out is double-buffered unless the block also carries
                // residual operands; a buffer is rewritten once the TMA store
                // that used it has read it
                uint8_t *s_out = (RES || (n_st & 1) == 0) ? s_out0 : s_aux;
                if (lane == 0) {
                    if constexpr (RES) bulk_wait_read<0>();
                    else bulk_wait_read<1>();
                }
                __syncwarp();
                write_row32(s_out, lane, v);
                if constexpr (CACHE) {
                    if (has_rhat) {
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] = round_to<bf16>(v[i]) - xi[i];
                        write_row32(s_aux, lane, v);
                    }
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_2d(&em.out[part], s_out, cl, m0 + q * 32);
                    if constexpr (CACHE)
                        if (has_rhat) tma_store_2d(&em.rhat, s_aux, col, m0 + q * 32);
                    bulk_commit();
                }
                ++n_st;
                if constexpr (SHARED) {
                    if (j + 1 < BN / 64) {
                        if (lane == 0) bulk_wait_read<0>();
                        __syncwarp();
                        load_res(m0, col + 32);
                    }
                }
            }
        }
        // every TMA store of this warp has completed before the CTA exits
        if (lane == 0) bulk_wait_all();
        __syncwarp();
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, G::TMEM_COLS);
    }
}

// ---------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *,
                                  CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                  CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    if (fn == nullptr) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

// 2-D bf16 tensor map over a row-major [rows][cols] matrix, box [box_rows][64],
// 128-byte swizzle, zero fill outside the matrix.
bool make_tmap_bf16(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (fn == nullptr) return false;
    if ((reinterpret_cast<uintptr_t>(base) & 15) != 0 || (cols * 2) % 16 != 0) return false;
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {cols * 2};
    cuuint32_t box[2] = {64, box_rows};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 2-D bf16 map with a 32 x 32 box and 64-byte swizzle (epilogue blocks).
static bool make_tmap_epi(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols) {
    EncodeTiledFn fn = encode_fn();
    if (fn == nullptr) return false;
    if ((reinterpret_cast<uintptr_t>(base) & 15) != 0 || (cols * 2) % 16 != 0 || cols % 32 != 0) return false;
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {cols * 2};
    cuuint32_t box[2] = {32, 32};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Encoded epilogue maps, looked up by (base, rows, cols): the chunk step
// reuses the same activation buffers on every pass, so encoding happens once
// per buffer.
namespace {
struct MapKey {
    const void *base;
    uint64_t rows, cols;
    bool operator==(const MapKey &o) const { return base == o.base && rows == o.rows && cols == o.cols; }
};
struct MapKeyHash {
    size_t operator()(const MapKey &k) const {
        return std::hash<const void *>()(k.base) ^ (size_t)(k.rows * 0x9E3779B97F4A7C15ull) ^ (size_t)(k.cols << 17);
    }
};
std::mutex g_map_mu;
std::unordered_map<MapKey, CUtensorMap, MapKeyHash> g_maps;
}  // namespace

static bool epi_map(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols) {
    if (base == nullptr) {                         // unused slot: any valid map
        memset(m, 0, sizeof(*m));
        return true;
    }
    std::lock_guard<std::mutex> lk(g_map_mu);
    const MapKey key{base, rows, cols};
    auto it = g_maps.find(key);
    if (it != g_maps.end()) {
        *m = it->second;
        return true;
    }
    if (g_maps.size() > 4096) g_maps.clear();
    if (!make_tmap_epi(m, base, rows, cols)) return false;
    g_maps.emplace(key, *m);
    return true;
}

template <int EPI>
static bool build_epi_maps(EpiMaps &em, const EpiParams &ep) {
    memset(&em, 0, sizeof(em));
    if constexpr (EPI == EPI_QKV_ROPE) {
        return epi_map(&em.out[0], ep.out, ep.M, ep.d) && epi_map(&em.out[1], ep.out_k, ep.M, ep.d) &&
               epi_map(&em.out[2], ep.out_v, ep.M, ep.d);
    } else {
        bool ok = epi_map(&em.out[0], ep.out, ep.M, ep.N);
        if constexpr (EPI == EPI_RESID_GATE || EPI == EPI_RESID_CACHE) ok = ok && epi_map(&em.resid, ep.resid, ep.M, ep.N);
        if constexpr (EPI == EPI_RESID_CACHE) {
            if (ep.rhat != nullptr)
                ok = ok && epi_map(&em.rhat, ep.rhat, ep.M, ep.N) && epi_map(&em.xin, ep.xin, ep.M, ep.N);
        }
        return ok;
    }
}

static int gemm_sm_count() {
    static int n = 0;
    if (n == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) n = 1;
    }
    return n;
}

// Output tile width for an M x N GEMM.  128 when 128 x 256 tiles would leave
// SMs idle.  Otherwise the persistent grid runs ceil(tiles / SMs) rounds of
// tiles; a 128 x 256 tile costs about 1.75 times a 128 x 128 one (it reuses
// each A tile for twice the columns), so 256 is taken when its rounds cost no
// more than the 128-wide tiles' rounds.
int gemm_tc_bn(int M, int N) {
    if (N % 256 != 0) return 128;
    const long m_tiles = (M + GEMM_BM - 1) / GEMM_BM, n_sm = gemm_sm_count();
    if (m_tiles * (N / 256) < n_sm) return 128;
    const long r256 = (m_tiles * (N / 256) + n_sm - 1) / n_sm;
    const long r128 = (m_tiles * (N / 128) + n_sm - 1) / n_sm;
    return 7 * r256 <= 4 * r128 ? 256 : 128;
}

template <int EPI, int BN>
static cudaError_t launch_tc(const CUtensorMap &ta, const CUtensorMap &tb, const EpiParams &ep, int K,
                             const uint8_t *skip, int *err, cudaStream_t st) {
    using G = GemmTile<BN, EPI>;
    auto kern = gemm_tc_kernel<BN, EPI>;
    EpiMaps em;
    if (!build_epi_maps<EPI>(em, ep)) return cudaErrorInvalidValue;
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, G::SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const int n_sm = gemm_sm_count();
    const int n_tiles = (ep.N / BN) * ((ep.M + GEMM_BM - 1) / GEMM_BM);
    const int grid = n_tiles < n_sm ? n_tiles : n_sm;
    return launch_pdl(kern, dim3(grid), dim3(320), G::SMEM_BYTES, st, ta, tb, em, ep, K, skip, err);
}

template <int BN>
static cudaError_t gemm_tc_bn_(int epi, const CUtensorMap &ta, const CUtensorMap &tb, const EpiParams &ep, int K,
                               const uint8_t *skip, int *err, cudaStream_t st) {
    switch (epi) {
        case EPI_BIAS: return launch_tc<EPI_BIAS, BN>(ta, tb, ep, K, skip, err, st);
        case EPI_GELU: return launch_tc<EPI_GELU, BN>(ta, tb, ep, K, skip, err, st);
        case EPI_RESID_GATE: return launch_tc<EPI_RESID_GATE, BN>(ta, tb, ep, K, skip, err, st);
        case EPI_RESID_CACHE: return launch_tc<EPI_RESID_CACHE, BN>(ta, tb, ep, K, skip, err, st);
        case EPI_QKV_ROPE: return launch_tc<EPI_QKV_ROPE, BN>(ta, tb, ep, K, skip, err, st);
        default: return cudaErrorInvalidValue;
    }
}

// Entry used by the chunk step and xc_op_linear / xc_op_qkv_rope (bf16 only).
// `ta` covers A [M][K] (box 128 rows), `tb` covers Wt [N][K] with box rows
// = bn (gemm_tc_bn(M, N)); N % bn == 0, K % 64 == 0.
cudaError_t gemm_tc(int epi, int bn, const CUtensorMap &ta, const CUtensorMap &tb, const EpiParams &ep, int K,
                    const uint8_t *skip, int *err, cudaStream_t st) {
    if (bn == 256) return gemm_tc_bn_<256>(epi, ta, tb, ep, K, skip, err, st);
    if (bn == 128) return gemm_tc_bn_<128>(epi, ta, tb, ep, K, skip, err, st);
    return cudaErrorInvalidValue;
}

}  // namespace xc
