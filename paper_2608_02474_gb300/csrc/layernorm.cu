// Layer norm without affine, eps 1e-6, biased variance (the block's LN), with
// an optional row gather: out[j] = LN(in[rows[j]]), or, for every row of a bf16
// input, a second copy of the rows a map selects (the "select active latents"
// step of Sec. 3.3 fused with the LN over all latents that the K/V path needs).
//
// A row lives in registers: for bf16 input one warp per row holds it packed (up
// to 32 16-byte chunks per lane); for fp32 input up to 8 chunks of 8 values per
// thread, one warp per row for D <= 1024, four warps per row up to D = 8192.
// Mean first, then the centred variance, both fp32 tree reductions; one HBM
// read, one write.
#include "common.cuh"
#include "internal.h"

namespace {

constexpr int kThreads = 256;
constexpr int kMaxChunks = 8;

template <typename T>
ECHO_DEV void ld8(const T *p, float *f);
template <>
ECHO_DEV void ld8<__nv_bfloat16>(const __nv_bfloat16 *p, float *f) {
    unpack8_bf16(__ldg(reinterpret_cast<const uint4 *>(p)), f);
}
template <>
ECHO_DEV void ld8<float>(const float *p, float *f) {
    const float4 a = __ldg(reinterpret_cast<const float4 *>(p));
    const float4 b = __ldg(reinterpret_cast<const float4 *>(p) + 1);
    f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
    f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
}

template <int TPR>
ECHO_DEV float row_sum(float v, float *red) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (TPR == 32) return v;
    constexpr int W = TPR / 32;
    const int warp = threadIdx.x >> 5;
    const int row_in_block = threadIdx.x / TPR;
    __syncthreads();
    if ((threadIdx.x & 31) == 0) red[warp] = v;
    __syncthreads();
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < W; ++w) s += red[row_in_block * W + w];
    return s;
}

template <typename T, int TPR>
__global__ void __launch_bounds__(kThreads)
layernorm_kernel(const T *__restrict__ in, const int32_t *__restrict__ rows, int n_rows, int D,
                 __nv_bfloat16 *__restrict__ out) {
    __shared__ float red[kThreads / 32];
    constexpr int RPB = kThreads / TPR;
    const int t = threadIdx.x % TPR;
    const int C = D >> 3;
    const float invD = 1.f / (float)D;
    for (int base = blockIdx.x * RPB; base < n_rows; base += gridDim.x * RPB) {
        const int j = base + threadIdx.x / TPR;
        const bool live = j < n_rows;
        const int r = live ? (rows ? rows[j] : j) : 0;
        const T *src = in + (int64_t)r * D;
        float v[kMaxChunks][8];
        float s = 0.f;
#pragma unroll
        for (int k = 0; k < kMaxChunks; ++k) {
            const int c = t + k * TPR;
            if (live && c < C) {
                ld8<T>(src + 8 * c, v[k]);
#pragma unroll
                for (int e = 0; e < 8; ++e) s += v[k][e];
            } else {
#pragma unroll
                for (int e = 0; e < 8; ++e) v[k][e] = 0.f;
            }
        }
        const float mean = row_sum<TPR>(s, red) * invD;
        float ss = 0.f;
#pragma unroll
        for (int k = 0; k < kMaxChunks; ++k) {
            const int c = t + k * TPR;
            if (live && c < C) {
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const float dlt = v[k][e] - mean;
                    ss += dlt * dlt;
                }
            }
        }
        const float var = row_sum<TPR>(ss, red) * invD;
        const float rstd = rsqrtf(var + 1e-6f);
        if (live) {
            __nv_bfloat16 *dst = out + (int64_t)j * D;
#pragma unroll
            for (int k = 0; k < kMaxChunks; ++k) {
                const int c = t + k * TPR;
                if (c < C) {
                    float o[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) o[e] = (v[k][e] - mean) * rstd;
                    *reinterpret_cast<uint4 *>(dst + 8 * c) = pack8_bf16(o);
                }
            }
        }
    }
}

// bf16 input: one warp per row, the row held packed in registers (CPL 16-byte
// chunks per lane), so each row is read from HBM once and no block barrier is
// needed.
template <int CPL>
__global__ void __launch_bounds__(kThreads)
layernorm_warp_bf16(const __nv_bfloat16 *__restrict__ in, const int32_t *__restrict__ rows,
                    int n_rows, int D, __nv_bfloat16 *__restrict__ out) {
    const int lane = threadIdx.x & 31;
    const int warps = kThreads / 32;
    const int C = D >> 3;
    const float invD = 1.f / (float)D;
    for (int j = blockIdx.x * warps + (threadIdx.x >> 5); j < n_rows; j += gridDim.x * warps) {
        const int r = rows ? rows[j] : j;
        const uint4 *src = reinterpret_cast<const uint4 *>(in + (int64_t)r * D);
        uint4 v[CPL];
#pragma unroll
        for (int k = 0; k < CPL; ++k) {
            const int c = lane + 32 * k;
            v[k] = c < C ? __ldcs(src + c) : make_uint4(0, 0, 0, 0);
        }
        float s = 0.f;
#pragma unroll
        for (int k = 0; k < CPL; ++k) {
            float f[8];
            unpack8_bf16(v[k], f);
#pragma unroll
            for (int e = 0; e < 8; ++e) s += f[e];
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        const float mean = s * invD;
        float ss = 0.f;
#pragma unroll
        for (int k = 0; k < CPL; ++k) {
            if (lane + 32 * k < C) {
                float f[8];
                unpack8_bf16(v[k], f);
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const float dlt = f[e] - mean;
                    ss += dlt * dlt;
                }
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        const float rstd = rsqrtf(ss * invD + 1e-6f);
        uint4 *dst = reinterpret_cast<uint4 *>(out + (int64_t)j * D);
#pragma unroll
        for (int k = 0; k < CPL; ++k) {
            const int c = lane + 32 * k;
            if (c < C) {
                float f[8];
                unpack8_bf16(v[k], f);
#pragma unroll
                for (int e = 0; e < 8; ++e) f[e] = (f[e] - mean) * rstd;
                dst[c] = pack8_bf16(f);
            }
        }
    }
}

// All rows of a bf16 input (no gather), for D <= 8192: one warp per row as in
// layernorm_warp_bf16, but each warp streams its rows through two shared-memory
// buffers filled by 1-D bulk copies, the next row's copy in flight while the
// current row is normalised and written.  Same arithmetic, same bits.  With
// scatter_map, row j is also written to out2[scatter_map[j]] when that is
// >= 0: the LN of every latent (for K and V) then also yields the gathered LN
// of the active ones (for Q') without reading them a second time.
constexpr int kBulkWarps = 4;

template <int CPL>
__global__ void __launch_bounds__(kBulkWarps * 32)
layernorm_bulk_bf16(const __nv_bfloat16 *__restrict__ in, int n_rows, int D,
                    __nv_bfloat16 *__restrict__ out, const int32_t *__restrict__ scatter_map,
                    __nv_bfloat16 *__restrict__ out2, int *err) {
    extern __shared__ __align__(128) uint8_t smem_rows[];
    __shared__ __align__(8) uint64_t bar[kBulkWarps][2];
    __shared__ int abort_flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t row_bytes = (uint32_t)D * 2u;
    uint8_t *buf = smem_rows + (size_t)warp * 2 * row_bytes;
    if (lane == 0) {
        mbar_init(&bar[warp][0], 1);
        mbar_init(&bar[warp][1], 1);
    }
    if (threadIdx.x == 0) abort_flag = 0;
    fence_barrier_init();
    __syncthreads();
    volatile int *abort_v = &abort_flag;
    const int C = D >> 3;
    const float invD = 1.f / (float)D;
    const int nw = gridDim.x * kBulkWarps;
    int j = blockIdx.x * kBulkWarps + warp;
    if (j < n_rows && lane == 0) {
        mbar_arrive_expect_tx(&bar[warp][0], row_bytes);
        bulk_load_1d(buf, in + (int64_t)j * D, row_bytes, &bar[warp][0]);
    }
    bool pending_next = false;
    for (int it = 0; j < n_rows; ++it, j += nw) {
        const int b = it & 1;
        const int jn = j + nw;
        __syncwarp();   // every lane is done with buffer b ^ 1 (read in the last iteration)
        pending_next = jn < n_rows;
        if (pending_next && lane == 0) {
            fence_proxy_async_smem();
            mbar_arrive_expect_tx(&bar[warp][b ^ 1], row_bytes);
            bulk_load_1d(buf + (b ^ 1) * row_bytes, in + (int64_t)jn * D, row_bytes,
                         &bar[warp][b ^ 1]);
        }
        if (!__all_sync(0xffffffffu, mbar_wait(&bar[warp][b], (it >> 1) & 1, abort_v, err))) {
            pending_next = false;   // the CTA gives up; let the next copy land first
            if (jn < n_rows)
                mbar_wait(&bar[warp][b ^ 1], ((it + 1) >> 1) & 1, abort_v, nullptr, 100000000ull);
            break;
        }
        const uint4 *src = reinterpret_cast<const uint4 *>(buf + b * row_bytes);
        uint4 v[CPL];
#pragma unroll
        for (int k = 0; k < CPL; ++k) {
            const int c = lane + 32 * k;
            v[k] = c < C ? src[c] : make_uint4(0, 0, 0, 0);
        }
        float s = 0.f;
#pragma unroll
        for (int k = 0; k < CPL; ++k) {
            float f[8];
            unpack8_bf16(v[k], f);
#pragma unroll
            for (int e = 0; e < 8; ++e) s += f[e];
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        const float mean = s * invD;
        float ss = 0.f;
#pragma unroll
        for (int k = 0; k < CPL; ++k) {
            if (lane + 32 * k < C) {
                float f[8];
                unpack8_bf16(v[k], f);
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const float dlt = f[e] - mean;
                    ss += dlt * dlt;
                }
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        const float rstd = rsqrtf(ss * invD + 1e-6f);
        uint4 *dst = reinterpret_cast<uint4 *>(out + (int64_t)j * D);
        const int j2 = scatter_map ? scatter_map[j] : -1;
        uint4 *dst2 = j2 >= 0 ? reinterpret_cast<uint4 *>(out2 + (int64_t)j2 * D) : nullptr;
#pragma unroll
        for (int k = 0; k < CPL; ++k) {
            const int c = lane + 32 * k;
            if (c < C) {
                float f[8];
                unpack8_bf16(v[k], f);
#pragma unroll
                for (int e = 0; e < 8; ++e) f[e] = (f[e] - mean) * rstd;
                const uint4 o = pack8_bf16(f);
                dst[c] = o;
                if (dst2) dst2[c] = o;
            }
        }
    }
    (void)pending_next;
}

template <int CPL>
void launch_bulk_bf16(const __nv_bfloat16 *in, int n_rows, int D, __nv_bfloat16 *out,
                      const int32_t *scatter_map, __nv_bfloat16 *out2, cudaStream_t st) {
    const size_t smem = (size_t)kBulkWarps * 2 * D * sizeof(__nv_bfloat16);
    static int attr_done[64] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_done[dev]) {
        cudaFuncSetAttribute(layernorm_bulk_bf16<CPL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)(kBulkWarps * 2 * 8192 * sizeof(__nv_bfloat16)));
        attr_done[dev] = 1;
    }
    int grid = (n_rows + kBulkWarps - 1) / kBulkWarps;
    if (grid > 152 * 2) grid = 152 * 2;
    layernorm_bulk_bf16<CPL><<<grid, kBulkWarps * 32, smem, st>>>(in, n_rows, D, out, scatter_map,
                                                                  out2, echo::device_error_ptr());
}

template <int CPL>
void launch_warp_bf16(const __nv_bfloat16 *in, const int32_t *rows, int n_rows, int D,
                      __nv_bfloat16 *out, cudaStream_t st) {
    constexpr int RPB = kThreads / 32;
    int grid = (n_rows + RPB - 1) / RPB;
    if (grid > 152 * 8) grid = 152 * 8;
    layernorm_warp_bf16<CPL><<<grid, kThreads, 0, st>>>(in, rows, n_rows, D, out);
}

// gathered rows of a bf16 input: the row packed in registers
void launch_gather_bf16(const __nv_bfloat16 *in, const int32_t *rows, int n_rows, int D,
                        __nv_bfloat16 *out, cudaStream_t st) {
    const int cpl = (D / 8 + 31) / 32;   // 16-byte chunks per lane
    if (cpl <= 4) return launch_warp_bf16<4>(in, rows, n_rows, D, out, st);
    if (cpl <= 8) return launch_warp_bf16<8>(in, rows, n_rows, D, out, st);
    if (cpl <= 16) return launch_warp_bf16<16>(in, rows, n_rows, D, out, st);
    if (cpl <= 20) return launch_warp_bf16<20>(in, rows, n_rows, D, out, st);
    if (cpl <= 24) return launch_warp_bf16<24>(in, rows, n_rows, D, out, st);
    return launch_warp_bf16<32>(in, rows, n_rows, D, out, st);
}

// fp32 rows of up to 8192 values: one CTA of 128 threads per row, the row in
// registers (thread t holds 16-byte chunks t, t + 128, ...), every load in
// flight before the first sum.  Sums: each thread's chunks in order, a xor
// butterfly per warp, then the four warp partials in order.
constexpr int kRowThreads = 128, kRowChunks = 16;

__global__ void __launch_bounds__(kRowThreads)
layernorm_row_f32(const float *__restrict__ in, int D, __nv_bfloat16 *__restrict__ out) {
    __shared__ float red[2][kRowThreads / 32];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int C4 = D >> 2;
    const float4 *row = reinterpret_cast<const float4 *>(in + (int64_t)blockIdx.x * D);
    float4 v[kRowChunks];
#pragma unroll
    for (int k = 0; k < kRowChunks; ++k) {
        const int c = threadIdx.x + k * kRowThreads;
        v[k] = c < C4 ? __ldcs(row + c) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < kRowChunks; ++k) {
        s += v[k].x; s += v[k].y; s += v[k].z; s += v[k].w;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) red[0][warp] = s;
    __syncthreads();
    const float invD = 1.f / (float)D;
    const float mean = (((red[0][0] + red[0][1]) + red[0][2]) + red[0][3]) * invD;
    float ss = 0.f;
#pragma unroll
    for (int k = 0; k < kRowChunks; ++k) {
        if (threadIdx.x + k * kRowThreads < C4) {
            const float a = v[k].x - mean, b = v[k].y - mean, c = v[k].z - mean, d = v[k].w - mean;
            ss += a * a; ss += b * b; ss += c * c; ss += d * d;
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if (lane == 0) red[1][warp] = ss;
    __syncthreads();
    const float rstd = rsqrtf((((red[1][0] + red[1][1]) + red[1][2]) + red[1][3]) * invD + 1e-6f);
    uint2 *dst = reinterpret_cast<uint2 *>(out + (int64_t)blockIdx.x * D);
#pragma unroll
    for (int k = 0; k < kRowChunks; ++k) {
        const int c = threadIdx.x + k * kRowThreads;
        if (c < C4)
            dst[c] = make_uint2(pack_bf16((v[k].x - mean) * rstd, (v[k].y - mean) * rstd),
                                pack_bf16((v[k].z - mean) * rstd, (v[k].w - mean) * rstd));
    }
}

// every row of an fp32 input (D <= 8192: echo_layernorm and the block step
// reject wider rows)
void launch_all_f32(const float *in, int n_rows, int D, __nv_bfloat16 *out, cudaStream_t st) {
    if (n_rows <= 0) return;
    layernorm_row_f32<<<n_rows, kRowThreads, 0, st>>>(in, D, out);
}

// every row of a bf16 input, optionally also scattered through a map: the
// bulk-copy kernel (the same arithmetic as layernorm_warp_bf16)
void launch_all_bf16(const __nv_bfloat16 *in, int n_rows, int D, __nv_bfloat16 *out,
                     const int32_t *scatter_map, __nv_bfloat16 *out2, cudaStream_t st) {
    const int cpl = (D / 8 + 31) / 32;
    if (cpl <= 16) return launch_bulk_bf16<16>(in, n_rows, D, out, scatter_map, out2, st);
    if (cpl <= 20) return launch_bulk_bf16<20>(in, n_rows, D, out, scatter_map, out2, st);
    if (cpl <= 24) return launch_bulk_bf16<24>(in, n_rows, D, out, scatter_map, out2, st);
    return launch_bulk_bf16<32>(in, n_rows, D, out, scatter_map, out2, st);
}

template <typename T>
void launch_t(const T *in, const int32_t *rows, int n_rows, int D, __nv_bfloat16 *out,
              cudaStream_t st) {
    const int C = D / 8;
    echo::LaunchScope ls(ECHO_K_LAYERNORM, n_rows, D, (int64_t)sizeof(T), st);
    if constexpr (sizeof(T) == 2) {
        if (!rows) return launch_all_bf16(in, n_rows, D, out, nullptr, nullptr, st);
        return launch_gather_bf16(in, rows, n_rows, D, out, st);
    } else {
        if (!rows) return launch_all_f32(in, n_rows, D, out, st);
    }
    if (C <= 32 * kMaxChunks / 2) {   // D <= 1024: a warp per row
        constexpr int RPB = kThreads / 32;
        int grid = (n_rows + RPB - 1) / RPB;
        if (grid > 152 * 16) grid = 152 * 16;
        layernorm_kernel<T, 32><<<grid, kThreads, 0, st>>>(in, rows, n_rows, D, out);
    } else {
        constexpr int RPB = kThreads / 128;
        int grid = (n_rows + RPB - 1) / RPB;
        if (grid > 152 * 16) grid = 152 * 16;
        layernorm_kernel<T, 128><<<grid, kThreads, 0, st>>>(in, rows, n_rows, D, out);
    }
}

}  // namespace

namespace echo {

void launch_layernorm_scatter(const void *in, int32_t n_rows, int32_t D, void *out,
                              const int32_t *scatter_map, void *out2, cudaStream_t st) {
    if (n_rows <= 0) return;
    LaunchScope ls(ECHO_K_LAYERNORM, n_rows, D, 2, st);
    launch_all_bf16(static_cast<const __nv_bfloat16 *>(in), n_rows, D,
                    static_cast<__nv_bfloat16 *>(out), scatter_map,
                    static_cast<__nv_bfloat16 *>(out2), st);
}

void launch_layernorm(const void *in, echo_dtype in_t, const int32_t *rows, int32_t n_rows,
                      int32_t D, void *out, cudaStream_t st) {
    if (n_rows <= 0) return;
    __nv_bfloat16 *o = static_cast<__nv_bfloat16 *>(out);
    if (in_t == ECHO_BF16)
        launch_t(static_cast<const __nv_bfloat16 *>(in), rows, n_rows, D, o, st);
    else
        launch_t(static_cast<const float *>(in), rows, n_rows, D, o, st);
}

}  // namespace echo

extern "C" echo_status echo_layernorm(const void *in, echo_dtype in_t, const int32_t *rows,
                                      int32_t n_rows, int32_t D, void *out, echo_stream_t stream) {
    using namespace echo;
    if (n_rows < 0 || D < 8 || D % 8 || D > 8192) return ECHO_ERR_SHAPE;
    if (n_rows == 0) return ECHO_OK;
    if (!in || !out) return ECHO_ERR_INVALID_ARG;
    if (in_t != ECHO_BF16 && in_t != ECHO_F32) return ECHO_ERR_INVALID_ARG;
    if (!aligned16(in) || !aligned16(out) || (rows && !aligned16(rows))) return ECHO_ERR_INVALID_ARG;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    launch_layernorm(in, in_t, rows, n_rows, D, out, reinterpret_cast<cudaStream_t>(stream));
    return last_launch_status();
}
