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
//   warp 1         : allocates TMEM (two BN-column accumulators); lane 0
//                    issues tcgen05.mma (M=128, N=BN, K=16; 4 per 64-wide
//                    k-tile) into the free accumulator and commits each stage
//                    back to the producer;
//   warps 2..9     : epilogue -- tcgen05.ld of their 32-lane TMEM quadrant
//                    (two warps per quadrant, half of the columns each),
//                    fused bias / GELU / gated residual / residual-cache /
//                    RoPE, vectorised stores; then they release the
//                    accumulator, so the epilogue of tile i overlaps the
//                    main loop of tile i + 1.
// The skip flag of the block lets the whole recompute path early-exit when
// the gate chose reuse (Eq. 4), so decisions never return to the host.
#include "xc_ptx.cuh"

namespace xc {

constexpr int GEMM_BM = 128;
constexpr int GEMM_BK = 64;

template <int BN>
struct GemmTile {
    static constexpr int STAGES = BN == 256 ? 4 : 6;
    static constexpr int A_BYTES = GEMM_BM * GEMM_BK * 2;
    static constexpr int B_BYTES = BN * GEMM_BK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int STAGE_EPI = STAGES * STAGE_BYTES;       // 8 warps x [32 rows][32 fp32]
    static constexpr int EPI_BYTES = 8 * 32 * 32 * 4;
    static constexpr int BAR_OFFSET = STAGE_EPI + EPI_BYTES;
    static constexpr int SMEM_BYTES = BAR_OFFSET + 256 + 1024;   // barriers + alignment slack
    static constexpr int TMEM_COLS = 2 * BN;                      // double-buffered accumulator
    static constexpr int EPI_THREADS = 256;
};

__device__ __forceinline__ uint8_t *align1024(uint8_t *p) {
    const uint32_t s = smem_u32(p);
    return p + ((1024u - (s & 1023u)) & 1023u);
}

// Epilogue operands of one 32-column block of a warp: the thread owns rows
// r = it * 8 + lane / 4 (it = 0..3) of its 32-row quadrant and the 8 columns
// [col, col + 8).  They are loaded into registers ahead of use (bf16 path).
template <int EPI>
struct EpiPrefetch {
    float bias[8];
    float gate[8];
    uint4 resid[4];
    uint4 xin[4];
    float2 cs[4][4];      // RoPE (cos, sin) of the 4 pairs, per row
};

__device__ __forceinline__ uint4 ld_u4(const void *p) { return *reinterpret_cast<const uint4 *>(p); }

template <int EPI>
__device__ __forceinline__ void epi_prefetch(const EpiParams &p, int row0, int col, int lane, EpiPrefetch<EPI> &f) {
    loadW<float, 8>(p.bias + col, f.bias);
    if constexpr (EPI == EPI_RESID_GATE || EPI == EPI_RESID_CACHE) {
        loadW<float, 8>(p.gate + col, f.gate);
#pragma unroll
        for (int it = 0; it < 4; ++it) {
            const int row = row0 + it * 8 + (lane >> 2);
            if (row < p.M) {
                f.resid[it] = ld_u4(reinterpret_cast<const bf16 *>(p.resid) + (size_t)row * p.N + col);
                if constexpr (EPI == EPI_RESID_CACHE)
                    if (p.rhat != nullptr) f.xin[it] = ld_u4(reinterpret_cast<const bf16 *>(p.xin) + (size_t)row * p.N + col);
            }
        }
    }
    if constexpr (EPI == EPI_QKV_ROPE) {
        const int part = col / p.d;
        const int c = col - part * p.d;
        if (part < 2) {
            const int pair0 = (c % p.head_dim) >> 1;
            int off[4], axis[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                off[j] = p.rope_off[pair0 + j];
                axis[j] = p.rope_axis[pair0 + j];
            }
#pragma unroll
            for (int it = 0; it < 4; ++it) {
                const int row = row0 + it * 8 + (lane >> 2);
                if (row < p.M) {
                    const int cam = row / p.npc;
                    const int rem = row - cam * p.npc;
                    const int pos[4] = {cam, rem / (p.gh * p.gw), (rem / p.gw) % p.gh, rem % p.gw};
#pragma unroll
                    for (int j = 0; j < 4; ++j) f.cs[it][j] = p.rope_cs[off[j] + pos[axis[j]]];
                }
            }
        }
    }
}

__device__ __forceinline__ void unpack8(uint4 u, float (&v)[8]) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const float2 t = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&w[j]));
        v[2 * j] = t.x;
        v[2 * j + 1] = t.y;
    }
}

// Same arithmetic as epilogue_run<EPI, bf16, 8> on prefetched operands.
template <int EPI>
__device__ __forceinline__ void epi_apply(const EpiParams &p, int row, int col, float (&acc)[8],
                                          const EpiPrefetch<EPI> &f, int it) {
    if (row >= p.M) return;
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[i] += f.bias[i];
    const size_t off = (size_t)row * p.N + col;
    if constexpr (EPI == EPI_BIAS) {
        storeW<bf16, 8>(reinterpret_cast<bf16 *>(p.out) + off, acc);
    } else if constexpr (EPI == EPI_GELU) {
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] = gelu_tanh_approx(acc[i]);
        storeW<bf16, 8>(reinterpret_cast<bf16 *>(p.out) + off, acc);
    } else if constexpr (EPI == EPI_RESID_GATE || EPI == EPI_RESID_CACHE) {
        float r[8];
        unpack8(f.resid[it], r);
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] = r[i] + f.gate[i] * acc[i];
        storeW<bf16, 8>(reinterpret_cast<bf16 *>(p.out) + off, acc);
        if constexpr (EPI == EPI_RESID_CACHE) {
            if (p.rhat != nullptr) {
                float xi[8];
                unpack8(f.xin[it], xi);
#pragma unroll
                for (int i = 0; i < 8; ++i) acc[i] = round_to<bf16>(acc[i]) - xi[i];
                storeW<bf16, 8>(reinterpret_cast<bf16 *>(p.rhat) + off, acc);
            }
        }
    } else if constexpr (EPI == EPI_QKV_ROPE) {
        const int part = col / p.d;
        const int c = col - part * p.d;
        if (part < 2) {
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float2 t = f.cs[it][j];
                const float x0 = acc[2 * j], x1 = acc[2 * j + 1];
                acc[2 * j] = x0 * t.x - x1 * t.y;
                acc[2 * j + 1] = x0 * t.y + x1 * t.x;
            }
        }
        bf16 *dst = reinterpret_cast<bf16 *>(part == 0 ? p.out : (part == 1 ? p.out_k : p.out_v));
        storeW<bf16, 8>(dst + (size_t)row * p.d + c, acc);
    }
}

template <int BN, int EPI, typename T>
__global__ void __launch_bounds__(320, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const EpiParams ep, const int K, const uint8_t *__restrict__ skip_flag, int *err) {
    using G = GemmTile<BN>;
    if (skip_flag != nullptr && *skip_flag == XC_DEC_SKIP) return;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = align1024(smem_raw);
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + G::BAR_OFFSET);
    uint64_t *empty = full + G::STAGES;
    uint64_t *acc_full = empty + G::STAGES;    // [2]
    uint64_t *acc_empty = acc_full + 2;        // [2]
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_empty + 2);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int KT = K / GEMM_BK;
    const int tiles_n = ep.N / BN;
    const int n_tiles = ((ep.M + GEMM_BM - 1) / GEMM_BM) * tiles_n;

    if (threadIdx.x == 0) {
        for (int s = 0; s < G::STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], G::EPI_THREADS);
        }
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
                const int m0 = (tile / tiles_n) * GEMM_BM, n0 = (tile % tiles_n) * BN;
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
        // warps 2..9: two warps per TMEM lane quadrant, each half of the columns.
        // Each 32-row x 32-column block goes TMEM -> registers (thread = row) ->
        // XOR-swizzled shared memory -> registers (4 lanes per row, 8 columns
        // each), so the epilogue's global loads and stores are row-contiguous.
        const int q = warp & 3;   // TMEM lane quadrant this warp may access
        const int half = (warp - 2) >> 2;
        const uint32_t tq = tmem + ((uint32_t)(q * 32) << 16);
        float *stg = reinterpret_cast<float *>(smem + G::STAGE_EPI) + (warp - 2) * 32 * 32;
        int local = 0;
        for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x, ++local) {
            const int buf = local & 1;
            const uint32_t use = (uint32_t)(local >> 1);
            const int m0 = (tile / tiles_n) * GEMM_BM, n0 = (tile % tiles_n) * BN;
            const int c8 = (lane & 3) * 8;
            // The global operands of this warp's first column block are
            // requested before the accumulator is ready; those of block
            // j + 1 right after block j is stored, so they are in flight
            // while block j + 1 comes out of TMEM.
            EpiPrefetch<EPI> pf;
            epi_prefetch<EPI>(ep, m0 + q * 32, n0 + half * (BN / 2) + c8, lane, pf);
            const bool ok = mbar_wait(&acc_full[buf], use & 1, err, ERR_WAIT_EPI);
            __syncwarp();
            if (!__all_sync(0xffffffffu, ok)) break;
            tc_fence_after();
#pragma unroll
            for (int j = 0; j < BN / 64; ++j) {
                const int c = half * (BN / 2) + 32 * j;
                float v[16];
                tmem_ld16_sync(tq + buf * BN + c, v);
#pragma unroll
                for (int i = 0; i < 16; ++i) stg[lane * 32 + (i ^ lane)] = v[i];
                tmem_ld16_sync(tq + buf * BN + c + 16, v);
#pragma unroll
                for (int i = 0; i < 16; ++i) stg[lane * 32 + ((16 + i) ^ lane)] = v[i];
                __syncwarp();
#pragma unroll
                for (int it = 0; it < 4; ++it) {
                    const int r = it * 8 + (lane >> 2);
                    float a[8];
#pragma unroll
                    for (int k = 0; k < 8; ++k) a[k] = stg[r * 32 + ((c8 + k) ^ r)];
                    epi_apply<EPI>(ep, m0 + q * 32 + r, n0 + c + c8, a, pf, it);
                }
                if (j + 1 < BN / 64) epi_prefetch<EPI>(ep, m0 + q * 32, n0 + c + 32 + c8, lane, pf);
                __syncwarp();
            }
            tc_fence_before();
            mbar_arrive(&acc_empty[buf]);
        }
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

static int gemm_sm_count() {
    static int n = 0;
    if (n == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) n = 1;
    }
    return n;
}

// Output tile width for an M x N GEMM: 256, unless 128 x 256 tiles would
// leave SMs idle (fewer tiles than SMs) and N allows 128-wide tiles.
int gemm_tc_bn(int M, int N) {
    const long tiles256 = (long)((M + GEMM_BM - 1) / GEMM_BM) * (N / 256);
    return (N % 256 != 0 || (tiles256 < gemm_sm_count() && N % 128 == 0)) ? 128 : 256;
}

template <int EPI, int BN>
static cudaError_t launch_tc(const CUtensorMap &ta, const CUtensorMap &tb, const EpiParams &ep, int K,
                             const uint8_t *skip, int *err, cudaStream_t st) {
    using G = GemmTile<BN>;
    auto kern = gemm_tc_kernel<BN, EPI, bf16>;
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, G::SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const int n_sm = gemm_sm_count();
    const int n_tiles = (ep.N / BN) * ((ep.M + GEMM_BM - 1) / GEMM_BM);
    const int grid = n_tiles < n_sm ? n_tiles : n_sm;
    kern<<<grid, 320, G::SMEM_BYTES, st>>>(ta, tb, ep, K, skip, err);
    return cudaGetLastError();
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
