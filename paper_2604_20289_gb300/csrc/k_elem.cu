// Bandwidth-bound and small kernels of the chunk step: patch embedding,
// adaLN-Zero LayerNorm modulation, the reuse path (Eq. 4), the conditioning
// GEMVs, the output head, the Euler update and weight layout conversion.
#include "xc_kernels.cuh"
#include "xc_ptx.cuh"

namespace xc {

// ------------------------------------------------------- bounded-wait test
// One thread waits on an mbarrier phase that nothing completes: the bounded
// wait gives up after WAIT_NS, records `code` in *err and the kernel
// returns (the error path of every wait in the library, made to run out on
// purpose for its test).
__global__ void expire_wait_kernel(int *err, int code) {
    __shared__ uint64_t bar;
    if (threadIdx.x != 0) return;
    mbar_init(&bar, 1);
    mbar_fence_init();
    mbar_wait(&bar, 0, err, code);
}
cudaError_t expire_wait(int *err, int code, cudaStream_t st) {
    expire_wait_kernel<<<1, 32, 0, st>>>(err, code);
    return cudaGetLastError();
}

static int n_sm_elem() {
    static int n = 0;
    if (n == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) n = 1;
    }
    return n;
}

// ------------------------------------------------------------ patch embed
// X0[r][c] = round(sum_k z[r][k] * pe_w[k][c] + pe_b[c]), z float32 [L][16].
// Each lane owns 4 columns for the whole kernel and keeps their 16 x 4 block
// of pe_w and 4 biases in registers; a warp covers 128 consecutive columns
// and writes 128 columns of a row per store instruction.  CTA = 8 warps over
// one column block and a range of rows, walked in chunks of 64 latent rows
// (4 KB) staged in shared memory: the next chunk is loaded into registers
// (one float4 per thread) while the current one is computed, so the global
// load latency overlaps the arithmetic.
constexpr int PE_COLS = 128, PE_WARPS = 8, PE_CHUNK = 64;
template <typename T>
__global__ void __launch_bounds__(PE_WARPS * 32)
    patch_embed_kernel(const float *__restrict__ z, const float *__restrict__ w, const float *__restrict__ b,
                       T *__restrict__ out, int L, int d, int rows_per_cta) {
    pdl_wait();
    pdl_release();
    __shared__ __align__(16) float zs[2][PE_CHUNK * 16];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int col = blockIdx.x * PE_COLS + 4 * lane;
    const bool active = col < d;
    float2 wr[16][2], bias[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
    for (int k = 0; k < 16; ++k) {
        float4 t = make_float4(0.f, 0.f, 0.f, 0.f);
        if (active) t = *reinterpret_cast<const float4 *>(w + (size_t)k * d + col);
        wr[k][0] = make_float2(t.x, t.y);
        wr[k][1] = make_float2(t.z, t.w);
    }
    if (active) {
        const float4 t = *reinterpret_cast<const float4 *>(b + col);
        bias[0] = make_float2(t.x, t.y);
        bias[1] = make_float2(t.z, t.w);
    }
    const int r0 = blockIdx.y * rows_per_cta;
    const int r1 = min(L, r0 + rows_per_cta);
    // thread t stages float4 t of a chunk: row t / 4, quarter t % 4
    auto fetch = [&](int c0) {
        const int row = c0 + (threadIdx.x >> 2);
        return row < r1 ? __ldg(reinterpret_cast<const float4 *>(z + (size_t)row * 16) + (threadIdx.x & 3))
                        : make_float4(0.f, 0.f, 0.f, 0.f);
    };
    float4 nxt = fetch(r0);
    int buf = 0;
    for (int c0 = r0; c0 < r1; c0 += PE_CHUNK, buf ^= 1) {
        reinterpret_cast<float4 *>(zs[buf])[threadIdx.x] = nxt;
        __syncthreads();
        if (c0 + PE_CHUNK < r1) nxt = fetch(c0 + PE_CHUNK);
        const int n = min(PE_CHUNK, r1 - c0);
        if (active) {
            for (int rr = warp; rr < n; rr += PE_WARPS) {
                const float4 *zr = reinterpret_cast<const float4 *>(zs[buf] + rr * 16);
                float2 a01 = bias[0], a23 = bias[1];           // packed fp32 pairs: two FMAs per instruction
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float4 zq = zr[q];
                    const float zv[4] = {zq.x, zq.y, zq.z, zq.w};
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const float2 zz = make_float2(zv[i], zv[i]);
                        a01 = __ffma2_rn(zz, wr[4 * q + i][0], a01);
                        a23 = __ffma2_rn(zz, wr[4 * q + i][1], a23);
                    }
                }
                const float acc[4] = {a01.x, a01.y, a23.x, a23.y};
                T *dst = out + (size_t)(c0 + rr) * d + col;
                if constexpr (sizeof(T) == 2) {
                    __nv_bfloat162 lo = __floats2bfloat162_rn(acc[0], acc[1]);
                    __nv_bfloat162 hi = __floats2bfloat162_rn(acc[2], acc[3]);
                    uint2 pk;
                    pk.x = *reinterpret_cast<uint32_t *>(&lo);
                    pk.y = *reinterpret_cast<uint32_t *>(&hi);
                    *reinterpret_cast<uint2 *>(dst) = pk;
                } else {
                    *reinterpret_cast<float4 *>(dst) = make_float4(acc[0], acc[1], acc[2], acc[3]);
                }
            }
        }
    }
}

template <typename T>
cudaError_t patch_embed(const float *z, const float *w, const float *b, T *out, int L, int C, int d, cudaStream_t st) {
    if (C != 16 || d % 16 != 0) return cudaErrorInvalidValue;
    const int n_sm = n_sm_elem();
    const int n_cb = (d + PE_COLS - 1) / PE_COLS;
    int n_rb = (16 * n_sm + n_cb - 1) / n_cb;          // many short CTAs: no tail wave to speak of
    const int rows = ((L + n_rb - 1) / n_rb + PE_CHUNK - 1) / PE_CHUNK * PE_CHUNK;
    n_rb = (L + rows - 1) / rows;
    return launch_pdl(patch_embed_kernel<T>, dim3(n_cb, n_rb < 1 ? 1 : n_rb), dim3(PE_WARPS * 32), 0, st, z, w, b,
                      out, L, d, rows);
}
template cudaError_t patch_embed<float>(const float *, const float *, const float *, float *, int, int, int, cudaStream_t);
template cudaError_t patch_embed<bf16>(const float *, const float *, const float *, bf16 *, int, int, int, cudaStream_t);

// ------------------------------------------------------------- row stats
// A row is walked in 16-element runs; lane l owns runs l, l + 32, ...  Each
// lane reduces its own values to (count, mean, M2) in registers, the warp
// merges the lanes pairwise (Chan, Golub & LeVeque), so no per-element divide.
struct Moments {
    float n, mean, m2;
};
__device__ __forceinline__ Moments merge(Moments a, Moments b) {
    if (b.n == 0.0f) return a;
    if (a.n == 0.0f) return b;
    Moments r;
    r.n = a.n + b.n;
    const float dlt = b.mean - a.mean;
    const float f = b.n / r.n;
    r.mean = a.mean + dlt * f;
    r.m2 = a.m2 + b.m2 + dlt * dlt * a.n * f;
    return r;
}
__device__ __forceinline__ Moments warp_moments(Moments a) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        Moments b;
        b.n = __shfl_xor_sync(0xffffffffu, a.n, o);
        b.mean = __shfl_xor_sync(0xffffffffu, a.mean, o);
        b.m2 = __shfl_xor_sync(0xffffffffu, a.m2, o);
        a = merge(a, b);
    }
    return a;
}
// Moments of the first n_valid of the NCH runs a lane holds in registers.
template <int NCH>
__device__ __forceinline__ Moments lane_moments(const float (&v)[NCH][16], int n_valid) {
    float s = 0.0f;
#pragma unroll
    for (int k = 0; k < NCH; ++k)
        if (k < n_valid) {
#pragma unroll
            for (int i = 0; i < 16; ++i) s += v[k][i];
        }
    Moments m = {16.0f * n_valid, 0.0f, 0.0f};
    if (n_valid == 0) return m;
    m.mean = s / m.n;
#pragma unroll
    for (int k = 0; k < NCH; ++k)
        if (k < n_valid) {
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const float t = v[k][i] - m.mean;
                m.m2 = fmaf(t, t, m.m2);
            }
        }
    return m;
}

// ----------------------------------------------------------------- ln_mod
// One warp per row, the row held in registers (d <= 512 * NCH):
// h = round(LN(x) * (1 + scale) + shift).
template <typename T, int NCH>
__global__ void __launch_bounds__(256)
    ln_mod_kernel(const T *__restrict__ x, const float *__restrict__ shift, const float *__restrict__ scale,
                  T *__restrict__ out, int M, int d, float eps, const uint8_t *__restrict__ skip_flag) {
    pdl_wait();
    pdl_release();
    if (skip_flag != nullptr && *skip_flag == XC_DEC_SKIP) return;
    const int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (row >= M) return;
    const T *xr = x + (size_t)row * d;
    const int runs = d / 16;
    const int mine = runs > lane ? (runs - lane + 31) / 32 : 0;
    float v[NCH][16];
#pragma unroll
    for (int k = 0; k < NCH; ++k)
        if (k < mine) load16<T>(xr + 16 * (lane + 32 * k), v[k]);
    // the modulation vectors do not depend on the moments: fetch them while
    // the row reduction runs (one chunk ahead for wide rows)
    float sc[16], sh[16];
    if (mine > 0) {
        load16<float>(scale + 16 * lane, sc);
        load16<float>(shift + 16 * lane, sh);
    }
    const Moments mo = warp_moments(lane_moments<NCH>(v, mine));
    const float rstd = rsqrtf(mo.m2 / (float)d + eps);
    T *orow = out + (size_t)row * d;
#pragma unroll
    for (int k = 0; k < NCH; ++k) {
        if (k < mine) {
            const int c = 16 * (lane + 32 * k);
            if (k > 0) {
                load16<float>(scale + c, sc);
                load16<float>(shift + c, sh);
            }
#pragma unroll
            for (int i = 0; i < 16; ++i) v[k][i] = (v[k][i] - mo.mean) * rstd * (1.0f + sc[i]) + sh[i];
            store16<T>(orow + c, v[k]);
        }
    }
}

// d <= 512 (one 16-element run per lane): persistent warps walk rows
// row, row + n_warps, ... with the next row's load in flight while the
// current one is reduced; the modulation vectors stay in registers.
template <typename T>
__global__ void __launch_bounds__(256)
    ln_mod_row_kernel(const T *__restrict__ x, const float *__restrict__ shift, const float *__restrict__ scale,
                      T *__restrict__ out, int M, int d, float eps, const uint8_t *__restrict__ skip_flag) {
    pdl_wait();
    pdl_release();
    if (skip_flag != nullptr && *skip_flag == XC_DEC_SKIP) return;
    const int lane = threadIdx.x & 31;
    const int nw = (gridDim.x * blockDim.x) >> 5;
    const bool act = lane < d / 16;
    float sc[16], sh[16], cur[16], nxt[16];
    if (act) {
        load16<float>(scale + 16 * lane, sc);
        load16<float>(shift + 16 * lane, sh);
    }
    int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (row < M && act) load16<T>(x + (size_t)row * d + 16 * lane, cur);
    for (; row < M; row += nw) {
        const int nrow = row + nw;
        if (nrow < M && act) load16<T>(x + (size_t)nrow * d + 16 * lane, nxt);
        // two passes over the register-resident row: the mean, then the
        // squared deviations from it (butterfly sums, no Welford merges)
        float sum = 0.0f;
        if (act) {
#pragma unroll
            for (int i = 0; i < 16; ++i) sum += cur[i];
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
        const float mean = sum / (float)d;
        float m2 = 0.0f;
        if (act) {
#pragma unroll
            for (int i = 0; i < 16; ++i) m2 = fmaf(cur[i] - mean, cur[i] - mean, m2);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m2 += __shfl_xor_sync(0xffffffffu, m2, o);
        const float rstd = rsqrtf(m2 / (float)d + eps);
        if (act) {
#pragma unroll
            for (int i = 0; i < 16; ++i) cur[i] = (cur[i] - mean) * rstd * (1.0f + sc[i]) + sh[i];
            store16<T>(out + (size_t)row * d + 16 * lane, cur);
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) cur[i] = nxt[i];
    }
}

// d > 512: one CTA of LN_CTA threads per row.  The row is loaded once into
// registers as packed 16-byte vectors (KMAX per thread, all loads in flight),
// the mean and then the squared deviations are reduced over the CTA (warp
// butterflies, then the warps in order), and the modulated row is written
// back; many rows per SM are in flight at once.
constexpr int LN_CTA = 128;

template <typename T>
__device__ __forceinline__ void unpack16B(const uint4 u, float (&f)[16 / sizeof(T)]) {
    if constexpr (sizeof(T) == 2) {
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float2 t = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&w[j]));
            f[2 * j] = t.x;
            f[2 * j + 1] = t.y;
        }
    } else {
        f[0] = __uint_as_float(u.x);
        f[1] = __uint_as_float(u.y);
        f[2] = __uint_as_float(u.z);
        f[3] = __uint_as_float(u.w);
    }
}
template <typename T>
__device__ __forceinline__ uint4 pack16B(const float (&f)[16 / sizeof(T)]) {
    if constexpr (sizeof(T) == 2) {
        uint32_t w[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const __nv_bfloat162 h = __floats2bfloat162_rn(f[2 * j], f[2 * j + 1]);
            w[j] = *reinterpret_cast<const uint32_t *>(&h);
        }
        return make_uint4(w[0], w[1], w[2], w[3]);
    } else {
        return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]), __float_as_uint(f[2]), __float_as_uint(f[3]));
    }
}

// Sum over the CTA in a fixed order (deterministic).
__device__ __forceinline__ float cta_sum(float v, float *red) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    float s = red[0];
#pragma unroll
    for (int w = 1; w < LN_CTA / 32; ++w) s += red[w];
    return s;
}

template <typename T, int KMAX>
__global__ void __launch_bounds__(LN_CTA)
    ln_mod_cta_kernel(const T *__restrict__ x, const float *__restrict__ shift, const float *__restrict__ scale,
                      T *__restrict__ out, int M, int d, float eps, const uint8_t *__restrict__ skip_flag) {
    pdl_wait();
    pdl_release();
    if (skip_flag != nullptr && *skip_flag == XC_DEC_SKIP) return;
    constexpr int VEC = 16 / sizeof(T);
    __shared__ float red[2][LN_CTA / 32];
    const int row = blockIdx.x, tid = threadIdx.x;
    if (row >= M) return;
    const int nch = d / VEC;
    const uint4 *xr = reinterpret_cast<const uint4 *>(x + (size_t)row * d);
    uint4 raw[KMAX];
#pragma unroll
    for (int k = 0; k < KMAX; ++k) {
        const int c = tid + k * LN_CTA;
        raw[k] = c < nch ? xr[c] : make_uint4(0u, 0u, 0u, 0u);
    }
    float s = 0.0f;
#pragma unroll
    for (int k = 0; k < KMAX; ++k) {
        float f[VEC];
        unpack16B<T>(raw[k], f);
#pragma unroll
        for (int i = 0; i < VEC; ++i) s += f[i];
    }
    const float mean = cta_sum(s, red[0]) / (float)d;
    float m2 = 0.0f;
#pragma unroll
    for (int k = 0; k < KMAX; ++k) {
        if (tid + k * LN_CTA < nch) {
            float f[VEC];
            unpack16B<T>(raw[k], f);
#pragma unroll
            for (int i = 0; i < VEC; ++i) m2 = fmaf(f[i] - mean, f[i] - mean, m2);
        }
    }
    const float rstd = rsqrtf(cta_sum(m2, red[1]) / (float)d + eps);
    uint4 *orow = reinterpret_cast<uint4 *>(out + (size_t)row * d);
#pragma unroll
    for (int k = 0; k < KMAX; ++k) {
        const int c = tid + k * LN_CTA;
        if (c < nch) {
            float f[VEC], sc[VEC], sh[VEC];
            unpack16B<T>(raw[k], f);
#pragma unroll
            for (int i = 0; i < VEC; i += 4) {
                const float4 a = *reinterpret_cast<const float4 *>(scale + (size_t)c * VEC + i);
                const float4 b = *reinterpret_cast<const float4 *>(shift + (size_t)c * VEC + i);
                sc[i] = a.x; sc[i + 1] = a.y; sc[i + 2] = a.z; sc[i + 3] = a.w;
                sh[i] = b.x; sh[i + 1] = b.y; sh[i + 2] = b.z; sh[i + 3] = b.w;
            }
#pragma unroll
            for (int i = 0; i < VEC; ++i) f[i] = (f[i] - mean) * rstd * (1.0f + sc[i]) + sh[i];
            orow[c] = pack16B<T>(f);
        }
    }
}

template <typename T, int KMAX>
static cudaError_t ln_mod_cta(const T *x, const float *shift, const float *scale, T *out, int M, int d, float eps,
                              const uint8_t *skip, cudaStream_t st) {
    return launch_pdl(ln_mod_cta_kernel<T, KMAX>, dim3(M), dim3(LN_CTA), 0, st, x, shift, scale, out, M, d, eps,
                      skip);
}

template <typename T, int NCH>
static cudaError_t ln_mod_n(const T *x, const float *shift, const float *scale, T *out, int M, int d, float eps,
                            const uint8_t *skip, cudaStream_t st) {
    return launch_pdl(ln_mod_kernel<T, NCH>, dim3((M + 7) / 8), dim3(256), 0, st, x, shift, scale, out, M, d, eps, skip);
}

template <typename T>
cudaError_t ln_mod(const T *x, const float *shift, const float *scale, T *out, int M, int d, float eps,
                   const uint8_t *skip, cudaStream_t st) {
    if (d % 16 != 0) return cudaErrorInvalidValue;
    if (d <= 512) {
        const int want = (M + 7) / 8, cap = 2 * n_sm_elem();
        return launch_pdl(ln_mod_row_kernel<T>, dim3(want < cap ? want : cap), dim3(256), 0, st, x, shift, scale, out, M, d, eps, skip);
    }
    // one CTA per row: 16-byte vectors per thread
    const int per = (d / (16 / (int)sizeof(T)) + LN_CTA - 1) / LN_CTA;
    if (per <= 2) return ln_mod_cta<T, 2>(x, shift, scale, out, M, d, eps, skip, st);
    if (per <= 4) return ln_mod_cta<T, 4>(x, shift, scale, out, M, d, eps, skip, st);
    if (per <= 5) return ln_mod_cta<T, 5>(x, shift, scale, out, M, d, eps, skip, st);
    if (per <= 6) return ln_mod_cta<T, 6>(x, shift, scale, out, M, d, eps, skip, st);
    if (per <= 8) return ln_mod_cta<T, 8>(x, shift, scale, out, M, d, eps, skip, st);
    if (per <= 12) return ln_mod_cta<T, 12>(x, shift, scale, out, M, d, eps, skip, st);
    switch ((d + 511) / 512) {
        case 9: case 10: case 11: case 12: return ln_mod_n<T, 12>(x, shift, scale, out, M, d, eps, skip, st);
        default: return cudaErrorInvalidValue;
    }
}
template cudaError_t ln_mod<float>(const float *, const float *, const float *, float *, int, int, float,
                                   const uint8_t *, cudaStream_t);
template cudaError_t ln_mod<bf16>(const bf16 *, const float *, const float *, bf16 *, int, int, float,
                                  const uint8_t *, cudaStream_t);

// ------------------------------------------------------------ reuse (Eq. 4)
// out = round(x + rhat), 16-element vectors; runs only when the gate chose
// reuse (skip_flag == XC_DEC_SKIP) or unconditionally (skip_flag == nullptr).
template <typename T>
__global__ void __launch_bounds__(256)
    reuse_kernel(const T *__restrict__ x, const T *__restrict__ r, T *__restrict__ out, long n16,
                 const uint8_t *__restrict__ skip_flag) {
    pdl_wait();
    pdl_release();
    if (skip_flag != nullptr && *skip_flag != XC_DEC_SKIP) return;
    const long stride = (long)gridDim.x * blockDim.x;
    for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < n16; i += stride) {
        float a[16], b[16];
        load16<T>(x + i * 16, a);
        load16<T>(r + i * 16, b);
#pragma unroll
        for (int j = 0; j < 16; ++j) a[j] += b[j];
        store16<T>(out + i * 16, a);
    }
}

template <typename T>
cudaError_t residual_reuse(const T *x, const T *r, T *out, long n, const uint8_t *skip, int n_sm, cudaStream_t st) {
    const long n16 = n / 16;
    long blocks = (n16 + 255) / 256;
    const long cap = (long)n_sm * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    return launch_pdl(reuse_kernel<T>, dim3((unsigned)blocks), dim3(256), 0, st, x, r, out, n16, skip);
}
template cudaError_t residual_reuse<float>(const float *, const float *, float *, long, const uint8_t *, int, cudaStream_t);
template cudaError_t residual_reuse<bf16>(const bf16 *, const bf16 *, bf16 *, long, const uint8_t *, int, cudaStream_t);

// -------------------------------------------------- lazy chaining (Eq. 4)
// Before block b computes (b = n_blocks: before the head): if blocks j..b-1
// were all skipped (and block j-1 was not), x_{b-1} has not been
// materialised; it is x_{j-1} (buffer X[j & 1], written by block j-1 or the
// patch embedding) plus the cached residuals of the run.  Computed here in
// fp32 in block order, rounded once, into X[b & 1] (in place when the two are
// the same buffer: every element is read before it is written, by the same
// thread).  The decisions are read from the device, so one launch serves
// every pattern; the kernel exits at once when there is nothing to add.
template <typename T>
__global__ void __launch_bounds__(256)
    chain_apply_kernel(T *__restrict__ x0, T *__restrict__ x1, const T *__restrict__ rhat_t,
                       const uint8_t *__restrict__ flags, int b, int n_blocks, long n16, long ld) {
    pdl_wait();
    pdl_release();
    if (b < n_blocks && flags[b] == XC_DEC_SKIP) return;
    if (b == 0 || flags[b - 1] != XC_DEC_SKIP) return;
    int j = b - 1;
    while (j > 0 && flags[j - 1] == XC_DEC_SKIP) --j;
    const T *base = (j & 1) ? x1 : x0;
    T *out = (b & 1) ? x1 : x0;
    const long stride = (long)gridDim.x * blockDim.x;
    for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < n16; i += stride) {
        float a[16];
        load16<T>(base + i * 16, a);
        for (int k = j; k < b; ++k) {
            float r[16];
            load16<T>(rhat_t + (size_t)k * ld + i * 16, r);
#pragma unroll
            for (int e = 0; e < 16; ++e) a[e] += r[e];
        }
        store16<T>(out + i * 16, a);
    }
}

template <typename T>
cudaError_t chain_apply(T *x0, T *x1, const T *rhat_t, const uint8_t *flags, int b, int n_blocks, long ld,
                        int n_sm, cudaStream_t st) {
    const long n16 = ld / 16;
    long blocks = (n16 + 255) / 256;
    const long cap = (long)n_sm * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    return launch_pdl(chain_apply_kernel<T>, dim3((unsigned)blocks), dim3(256), 0, st, x0, x1, rhat_t, flags, b,
                      n_blocks, n16, ld);
}
template cudaError_t chain_apply<float>(float *, float *, const float *, const uint8_t *, int, int, long, int,
                                        cudaStream_t);
template cudaError_t chain_apply<bf16>(bf16 *, bf16 *, const bf16 *, const uint8_t *, int, int, long, int,
                                       cudaStream_t);

// -------------------------------------------------------------- Euler step
__global__ void euler_kernel(float *__restrict__ x, const float *__restrict__ v, float ds, long n) {
    pdl_wait();
    pdl_release();
    const long i = blockIdx.x * (long)blockDim.x + threadIdx.x;
    if (i < n) x[i] = fmaf(ds, v[i], x[i]);
}
cudaError_t euler_update(float *x, const float *v, float ds, long n, cudaStream_t st) {
    return launch_pdl(euler_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, st, x, v, ds, n);
}

// ----------------------------------------------------------- conditioning
constexpr int GEMV_WARPS = 16;

// Fused conditioning (a2), three launches per pass:
//   stage 1: ht = SiLU(W_t1 temb + b_t1), ha = SiLU(W_a1 a + b_a1)
//   stage 2: e  = (W_t2 ht + b_t2) + (W_a2 ha + b_a2)
//   stage 3: mods[b] = W_m SiLU(e) + b_m + table_b (every block b),
//            hmod    = W_h SiLU(e) + b_h + table_head
// The action and the sinusoidal timestep embedding (computed on the host in
// double precision, see xc_api.cu) ride in the kernel arguments.  Each CTA
// owns 32 output columns: the input is staged in shared memory and each of
// 16 warps keeps eight independent weight rows in flight.
__device__ __forceinline__ float gemv_col(const float *xs, const float *__restrict__ W, int n_in, int n_out, int j,
                                          int warp) {
    float a[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) a[k] = 0.0f;
    const float *wj = W + j;
    int i = warp;
    for (; i + 7 * GEMV_WARPS < n_in; i += 8 * GEMV_WARPS) {
        float w[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) w[k] = wj[(size_t)(i + k * GEMV_WARPS) * n_out];
#pragma unroll
        for (int k = 0; k < 8; ++k) a[k] = fmaf(xs[i + k * GEMV_WARPS], w[k], a[k]);
    }
    for (; i < n_in; i += GEMV_WARPS) a[0] = fmaf(xs[i], wj[(size_t)i * n_out], a[0]);
    return ((a[0] + a[1]) + (a[2] + a[3])) + ((a[4] + a[5]) + (a[6] + a[7]));
}

template <int STAGE>
__global__ void __launch_bounds__(GEMV_WARPS * 32) cond_kernel(const CondArgs c) {
    pdl_wait();
    pdl_release();
    extern __shared__ float xs[];
    __shared__ float part[GEMV_WARPS][33];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int d = c.d;
    const int nb_d = (d + 31) / 32;
    int j = 0, n_out = d;
    float acc = 0.0f;
    if constexpr (STAGE == 1) {
        const bool tpath = (int)blockIdx.x < nb_d;
        j = (tpath ? blockIdx.x : blockIdx.x - nb_d) * 32 + lane;
        const int n_in = tpath ? c.tf : c.A;
        if (tpath) {
            for (int i = threadIdx.x; i < c.tf; i += blockDim.x) xs[i] = c.temb[i];
        } else {
            for (int i = threadIdx.x; i < c.A; i += blockDim.x) {
                xs[i] = c.act[i];
                if (blockIdx.x == nb_d && c.act_out != nullptr) c.act_out[i] = c.act[i];
            }
        }
        __syncthreads();
        if (j < d) acc = gemv_col(xs, tpath ? c.t_w1 : c.a_w1, n_in, d, j, warp);
        part[warp][lane] = acc;
        __syncthreads();
        if (warp == 0 && j < d) {
            float s = 0.0f;
#pragma unroll
            for (int w = 0; w < GEMV_WARPS; ++w) s += part[w][lane];
            s += (tpath ? c.t_b1 : c.a_b1)[j];
            (tpath ? c.ht : c.ha)[j] = silu(s);
        }
    } else if constexpr (STAGE == 2) {
        j = blockIdx.x * 32 + lane;
        for (int i = threadIdx.x; i < d; i += blockDim.x) {
            xs[i] = c.ht[i];
            xs[d + i] = c.ha[i];
        }
        __syncthreads();
        if (j < d) acc = gemv_col(xs, c.t_w2, d, d, j, warp) + gemv_col(xs + d, c.a_w2, d, d, j, warp);
        part[warp][lane] = acc;
        __syncthreads();
        if (warp == 0 && j < d) {
            float s = 0.0f;
#pragma unroll
            for (int w = 0; w < GEMV_WARPS; ++w) s += part[w][lane];
            c.e[j] = s + c.t_b2[j] + c.a_b2[j];
        }
    } else {
        const int nb_m = (6 * d + 31) / 32;
        const bool mpath = (int)blockIdx.x < nb_m;
        n_out = mpath ? 6 * d : 2 * d;
        j = (mpath ? blockIdx.x : blockIdx.x - nb_m) * 32 + lane;
        for (int i = threadIdx.x; i < d; i += blockDim.x) xs[i] = silu(c.e[i]);
        __syncthreads();
        if (j < n_out) acc = gemv_col(xs, mpath ? c.mod_w : c.head_w, d, n_out, j, warp);
        part[warp][lane] = acc;
        __syncthreads();
        if (warp == 0 && j < n_out) {
            float s = 0.0f;
#pragma unroll
            for (int w = 0; w < GEMV_WARPS; ++w) s += part[w][lane];
            if (mpath) {
                s += c.mod_b[j];
                for (int b = 0; b < c.B; ++b) c.mods[(size_t)b * 6 * d + j] = s + c.blk_mod[(size_t)b * 6 * d + j];
            } else {
                c.hmod[j] = s + c.head_b[j] + c.head_tab[j];
            }
        }
    }
}

cudaError_t conditioning(const CondArgs &c, cudaStream_t st) {
    const int d = c.d, nb_d = (d + 31) / 32;
    if (c.A < 1 || c.A > 8 || c.tf < 2 || c.tf > COND_TEMB_MAX || (size_t)2 * d * sizeof(float) > 48 * 1024)
        return cudaErrorInvalidValue;
    const int in1 = c.tf > c.A ? c.tf : c.A;
    cudaError_t e = launch_pdl(cond_kernel<1>, dim3(2 * nb_d), dim3(GEMV_WARPS * 32), in1 * sizeof(float), st, c);
    if (e != cudaSuccess) return e;
    e = launch_pdl(cond_kernel<2>, dim3(nb_d), dim3(GEMV_WARPS * 32), 2 * d * sizeof(float), st, c);
    if (e != cudaSuccess) return e;
    return launch_pdl(cond_kernel<3>, dim3((6 * d + 31) / 32 + (2 * d + 31) / 32), dim3(GEMV_WARPS * 32),
                      d * sizeof(float), st, c);
}

// RoPE (cos, sin) table of one chunk, double precision.  Axes (camera, frame,
// h, w) own hd/16, 3hd/16, hd/8, hd/8 consecutive pairs; pair j of an axis
// with D = 2 * pairs dims rotates at theta^(-2j/D).  Axis a has npos[a]
// positions (frame: the chunk's frames, absolute frame = frame0 + p); entry
// base_a + j * npos[a] + p holds (cos, sin)(pos * freq).
__global__ void rope_table_kernel(int hd, double theta, int frame0, int4 npos, float2 *__restrict__ out, int n) {
    pdl_wait();
    pdl_release();
    const int e = blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= n) return;
    const int pairs[4] = {hd / 16, 3 * hd / 16, hd / 8, hd / 8};
    const int np[4] = {npos.x, npos.y, npos.z, npos.w};
    int base = 0;
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        const int span = pairs[a] * np[a];
        if (e < base + span) {
            const int j = (e - base) / np[a];
            const int p = (e - base) % np[a];
            const double freq = pow(theta, -2.0 * j / (2.0 * pairs[a]));
            const double ang = (double)(p + (a == 1 ? frame0 : 0)) * freq;
            out[e] = make_float2((float)cos(ang), (float)sin(ang));
            return;
        }
        base += span;
    }
}
cudaError_t rope_table(int hd, double theta, int frame0, int4 npos, float2 *out, int n, cudaStream_t st) {
    return launch_pdl(rope_table_kernel, dim3((n + 127) / 128), dim3(128), 0, st, hd, theta, frame0, npos, out, n);
}

// ------------------------------------------------------------------- head
// Output head (a10): v = round(LN(x) * (1 + scale) + shift) W_out + b,
// W_out [d][16].  CTA = 32 rows, 256 threads.  Pass 1: warp w reduces the
// moments of rows 4w..4w+3 (two loads in flight per lane).  Pass 2 walks the
// columns in chunks of 128 (the next chunk's loads in flight meanwhile): the
// CTA writes the modulated chunk h (rounded to the storage type) to shared
// memory transposed, hT[k][row] (lane = row when staging, so the stores are
// conflict-free), and the chunk's 128 x 16 block of W_out beside it; warp w
// then takes keys 16w..16w+15 of the chunk, lane (r4, c4) accumulating rows
// 4 r4..4 r4+3 x outputs 4 c4..4 c4+3 from one float4 of hT and one of W_out
// per key (16 FMA, as 8 packed fp32-pair FMAs, per two shared loads).  The 8 warps' partial sums are
// added in shared memory at the end, in warp order.
__device__ __forceinline__ void fma4(float2 (&a)[2], float h, const float4 &w) {
    const float2 hh = make_float2(h, h);
    a[0] = __ffma2_rn(hh, make_float2(w.x, w.y), a[0]);
    a[1] = __ffma2_rn(hh, make_float2(w.z, w.w), a[1]);
}
constexpr int HEAD_ROWS = 32, HEAD_CH = 128, HEAD_LD = HEAD_ROWS + 4;
template <typename T>
__global__ void __launch_bounds__(256)
    head_kernel(const T *__restrict__ x, const float *__restrict__ hm, const float *__restrict__ w,
                const float *__restrict__ b, float *__restrict__ v, int L, int d, float eps) {
    pdl_wait();
    pdl_release();
    __shared__ __align__(16) float hT[HEAD_CH * HEAD_LD];
    __shared__ __align__(16) float ws[HEAD_CH * 16];
    __shared__ float2 stats[HEAD_ROWS];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int row0 = blockIdx.x * HEAD_ROWS;
    const int runs = d / 16;
    // moments of one 16-element run, merged into mo
    auto add_run = [](Moments &mo, const float (&t)[16]) {
        float sum = 0.0f;
#pragma unroll
        for (int i = 0; i < 16; ++i) sum += t[i];
        Moments m1{16.0f, sum * (1.0f / 16.0f), 0.0f};
#pragma unroll
        for (int i = 0; i < 16; ++i) m1.m2 += (t[i] - m1.mean) * (t[i] - m1.mean);
        mo = merge(mo, m1);
    };
    for (int rr = 0; rr < 4; ++rr) {
        const int r = warp * 4 + rr, row = row0 + r;
        Moments mo{0.0f, 0.0f, 0.0f};
        if (row < L) {
            const T *xr = x + (size_t)row * d;
            int run = lane;
            for (; run + 32 < runs; run += 64) {         // two runs in flight
                float t0[16], t1[16];
                load16<T>(xr + 16 * run, t0);
                load16<T>(xr + 16 * (run + 32), t1);
                add_run(mo, t0);
                add_run(mo, t1);
            }
            if (run < runs) {
                float t0[16];
                load16<T>(xr + 16 * run, t0);
                add_run(mo, t0);
            }
        }
        mo = warp_moments(mo);
        if (lane == 0) stats[r] = make_float2(mo.mean, rsqrtf(mo.m2 / (float)d + eps));
    }
    __syncthreads();
    const float *shift = hm, *scale = hm + d;
    const int r4 = lane >> 2, c4 = lane & 3;
    float2 acc[4][2];                                     // [row][column pair]
#pragma unroll
    for (int i = 0; i < 4; ++i) acc[i][0] = acc[i][1] = make_float2(0.f, 0.f);
    const int my_row = row0 + lane;
    const float2 my_st = stats[lane];
    // warp w stages keys [16 w, 16 w + 16) of each chunk for its lane's row;
    // the next chunk's values are loaded while the current one is computed
    float xn[16];
    auto fetch = [&](int c0) {
        if (my_row < L && c0 + warp * 16 < d) {
            load16<T>(x + (size_t)my_row * d + c0 + warp * 16, xn);
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i) xn[i] = 0.0f;
        }
    };
    fetch(0);
    for (int c0 = 0; c0 < d; c0 += HEAD_CH) {
        const int n = d - c0 < HEAD_CH ? d - c0 : HEAD_CH;      // multiple of 16
        const int k16 = warp * 16;
        if (k16 < n) {
            float t[16];
            if (my_row < L) {
                float sc[16], sh[16];
                load16<float>(scale + c0 + k16, sc);
                load16<float>(shift + c0 + k16, sh);
#pragma unroll
                for (int i = 0; i < 16; ++i)
                    t[i] = round_to<T>((xn[i] - my_st.x) * my_st.y * (1.0f + sc[i]) + sh[i]);
            } else {
#pragma unroll
                for (int i = 0; i < 16; ++i) t[i] = 0.0f;
            }
#pragma unroll
            for (int i = 0; i < 16; ++i) hT[(k16 + i) * HEAD_LD + lane] = t[i];
        }
        for (int i = threadIdx.x; i < n * 4; i += blockDim.x)
            reinterpret_cast<float4 *>(ws)[i] = reinterpret_cast<const float4 *>(w + (size_t)c0 * 16)[i];
        __syncthreads();
        if (c0 + HEAD_CH < d) fetch(c0 + HEAD_CH);
        const int k_end = 16 * warp + 16 < n ? 16 * warp + 16 : n;
#pragma unroll 4
        for (int k = 16 * warp; k < k_end; ++k) {
            const float4 hv = *reinterpret_cast<const float4 *>(hT + k * HEAD_LD + 4 * r4);
            const float4 wv = *reinterpret_cast<const float4 *>(ws + k * 16 + 4 * c4);
            fma4(acc[0], hv.x, wv);
            fma4(acc[1], hv.y, wv);
            fma4(acc[2], hv.z, wv);
            fma4(acc[3], hv.w, wv);
        }
        __syncthreads();
    }
    // partial sums of the 8 warps -> shared memory (reuses hT), then add
    float *red = hT;                                          // [8][32][16] = 4096 floats
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        float *dst = red + (warp * HEAD_ROWS + 4 * r4 + i) * 16 + 4 * c4;
        dst[0] = acc[i][0].x;
        dst[1] = acc[i][0].y;
        dst[2] = acc[i][1].x;
        dst[3] = acc[i][1].y;
    }
    __syncthreads();
    for (int o = threadIdx.x; o < HEAD_ROWS * 16; o += blockDim.x) {
        const int r = o >> 4, c = o & 15;
        float sum = b[c];
#pragma unroll
        for (int ww = 0; ww < 8; ++ww) sum += red[(ww * HEAD_ROWS + r) * 16 + c];
        if (row0 + r < L) v[(size_t)(row0 + r) * 16 + c] = sum;
    }
}

template <typename T>
cudaError_t head(const T *x, const float *hm, const float *w, const float *b, float *v, int L, int d, float eps,
                 cudaStream_t st) {
    if (d % 16 != 0) return cudaErrorInvalidValue;
    return launch_pdl(head_kernel<T>, dim3((L + HEAD_ROWS - 1) / HEAD_ROWS), dim3(256), 0, st, x, hm, w, b, v, L, d, eps);
}
template cudaError_t head<float>(const float *, const float *, const float *, const float *, float *, int, int, float,
                                 cudaStream_t);
template cudaError_t head<bf16>(const bf16 *, const float *, const float *, const float *, float *, int, int, float,
                                cudaStream_t);

// --------------------------------------------------------- weight layout
// Wt[n][k] = convert(W[k][n]) for one [K][N] float32 matrix (32x32 tiles).
// fp32 -> storage type, elementwise (condition tokens of the cross-attention).
template <typename T>
__global__ void __launch_bounds__(256) convert_f32_kernel(const float *__restrict__ in, T *__restrict__ out, long n) {
    pdl_wait();
    pdl_release();
    for (long i = (long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (long)gridDim.x * blockDim.x) {
        if constexpr (sizeof(T) == 2)
            out[i] = __float2bfloat16_rn(in[i]);
        else
            out[i] = in[i];
    }
}
template <typename T>
cudaError_t convert_f32(const float *in, T *out, long n, int n_sm, cudaStream_t st) {
    const long want = (n + 255) / 256, cap = 4L * n_sm;
    convert_f32_kernel<T><<<(int)(want < cap ? (want > 0 ? want : 1) : cap), 256, 0, st>>>(in, out, n);
    return cudaGetLastError();
}
template cudaError_t convert_f32<bf16>(const float *, bf16 *, long, int, cudaStream_t);

template <typename T>
__global__ void transpose_convert_kernel(const float *__restrict__ W, T *__restrict__ Wt, int K, int N) {
    __shared__ float tile[32][33];
    const int n0 = blockIdx.x * 32, k0 = blockIdx.y * 32;
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int k = k0 + i, n = n0 + threadIdx.x;
        tile[i][threadIdx.x] = (k < K && n < N) ? W[(size_t)k * N + n] : 0.0f;
    }
    __syncthreads();
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int n = n0 + i, k = k0 + threadIdx.x;
        if (n < N && k < K) Wt[(size_t)n * K + k] = from_f<T>(tile[threadIdx.x][i]);
    }
}
template <typename T>
cudaError_t transpose_convert(const float *W, T *Wt, int K, int N, cudaStream_t st) {
    dim3 grid((N + 31) / 32, (K + 31) / 32), block(32, 8);
    transpose_convert_kernel<T><<<grid, block, 0, st>>>(W, Wt, K, N);
    return cudaGetLastError();
}
template cudaError_t transpose_convert<float>(const float *, float *, int, int, cudaStream_t);
template cudaError_t transpose_convert<bf16>(const float *, bf16 *, int, int, cudaStream_t);

}  // namespace xc
