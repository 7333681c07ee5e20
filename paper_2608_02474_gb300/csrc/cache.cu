// int8 per-token cache (Sec. 3.4): quantise-and-scatter, gather-and-reconstruct,
// and the mask fusion of Sec. 3.3 (active rows take the fresh block output,
// every other row is reconstructed from the cache).
//
// quant_kernel: one warp per source row; pass 1 finds amax, pass 2 (served from
//   L1/L2) writes the codes.  s = amax/127, inv = 127/amax, q = rint(v*inv)
//   clamped to [-127, 127], all fp32 round-to-nearest: bit-exact by construction.
// dequant kernels: one thread per 16 elements, 128-bit loads and stores.
#include "common.cuh"
#include "internal.h"

namespace {

constexpr int kQuantThreads = 256;
constexpr int kVecThreads = 256;

template <typename ST>
ECHO_DEV void load8(const ST *p, float *f);

template <>
ECHO_DEV void load8<__nv_bfloat16>(const __nv_bfloat16 *p, float *f) {
    unpack8_bf16(*reinterpret_cast<const uint4 *>(p), f);
}

template <>
ECHO_DEV void load8<float>(const float *p, float *f) {
    const float4 a = reinterpret_cast<const float4 *>(p)[0];
    const float4 b = reinterpret_cast<const float4 *>(p)[1];
    f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
    f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
}

template <typename ST>
__global__ void __launch_bounds__(kQuantThreads)
quant_kernel(const ST *__restrict__ src, const int32_t *__restrict__ rows, int n_rows, int D,
             int8_t *__restrict__ q, float *__restrict__ scale, int *err) {
    const int lane = threadIdx.x & 31;
    const int warps = blockDim.x >> 5;
    const int C = D >> 3;
    for (int j = blockIdx.x * warps + (threadIdx.x >> 5); j < n_rows; j += gridDim.x * warps) {
        const ST *s = src + (int64_t)j * D;
        float amax = 0.f;
        bool nan = false, inf = false;
        for (int c = lane; c < C; c += 32) {
            float f[8];
            load8<ST>(s + 8 * c, f);
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const float a = fabsf(f[k]);
                nan |= a != a;
                inf |= a == INFINITY;
                amax = fmaxf(amax, a);
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
        nan = __any_sync(0xffffffffu, nan);
        inf = __any_sync(0xffffffffu, inf);
        const int r = rows ? rows[j] : j;
        int8_t *qr = q + (int64_t)r * D;
        if (nan || inf) {
            for (int c = lane; c < C; c += 32) *reinterpret_cast<uint2 *>(qr + 8 * c) = make_uint2(0, 0);
            if (lane == 0) {
                scale[r] = nan ? __int_as_float(0x7fc00000) : INFINITY;
                echo_flag_error(err, ECHO_ERR_NONFINITE);
            }
            continue;
        }
        float sc = 0.f, inv = 0.f;
        if (amax > 0.f) {
            sc = __fdiv_rn(amax, 127.f);
            inv = __fdiv_rn(127.f, amax);
        }
        for (int c = lane; c < C; c += 32) {
            float f[8];
            load8<ST>(s + 8 * c, f);
            uint32_t w[2] = {0u, 0u};
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                float t = rintf(__fmul_rn(f[k], inv));
                t = fminf(fmaxf(t, -127.f), 127.f);
                const uint32_t b = (uint32_t)(uint8_t)(int8_t)(int)t;
                w[k >> 2] |= b << (8 * (k & 3));
            }
            *reinterpret_cast<uint2 *>(qr + 8 * c) = make_uint2(w[0], w[1]);
        }
        if (lane == 0) scale[r] = sc;
    }
}

ECHO_DEV void dequant16(const int4 &qv, float s, float *f) {
    const int8_t *b = reinterpret_cast<const int8_t *>(&qv);
#pragma unroll
    for (int k = 0; k < 16; ++k) f[k] = __fmul_rn((float)b[k], s);
}

template <typename DT>
ECHO_DEV void store16(DT *p, const float *f);

template <>
ECHO_DEV void store16<__nv_bfloat16>(__nv_bfloat16 *p, const float *f) {
    uint4 *o = reinterpret_cast<uint4 *>(p);
    o[0] = pack8_bf16(f);
    o[1] = pack8_bf16(f + 8);
}

template <>
ECHO_DEV void store16<float>(float *p, const float *f) {
    float4 *o = reinterpret_cast<float4 *>(p);
#pragma unroll
    for (int k = 0; k < 4; ++k) o[k] = make_float4(f[4 * k], f[4 * k + 1], f[4 * k + 2], f[4 * k + 3]);
}

template <typename DT>
__global__ void __launch_bounds__(kVecThreads)
dequant_kernel(const int8_t *__restrict__ q, const float *__restrict__ scale,
               const int32_t *__restrict__ rows, int n_rows, int D, DT *__restrict__ dst) {
    const int C = D >> 4;
    const int64_t total = (int64_t)n_rows * C;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int j = (int)(t / C), c = (int)(t % C);
        const int r = rows ? rows[j] : j;
        const int4 qv = __ldcs(reinterpret_cast<const int4 *>(q + (int64_t)r * D + 16 * c));
        float f[16];
        dequant16(qv, scale[r], f);
        store16<DT>(dst + (int64_t)j * D + 16 * c, f);
    }
}

// rowmap[i] = j where idx[j] == i, else -1: idx is ascending and distinct, so
// each row binary-searches it (idx stays in L1/L2).  The first n_zero words of
// `zero` are cleared in the same pass.
__global__ void rowmap_kernel(const int32_t *__restrict__ idx, int K, int NT,
                              int32_t *__restrict__ rowmap, uint32_t *__restrict__ zero,
                              int n_zero) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n_zero) zero[i] = 0u;
    if (i >= NT) return;
    int lo = 0, hi = K;   // the first j with idx[j] >= i
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (__ldg(idx + mid) < i) lo = mid + 1;
        else hi = mid;
    }
    rowmap[i] = (lo < K && __ldg(idx + lo) == i) ? lo : -1;
}

// y[i] = y_act[rowmap[i]] if rowmap[i] >= 0 else bf16(q[i] * s[i]); without
// y_act the active rows of y are already in place and are left alone
__global__ void __launch_bounds__(kVecThreads)
dequant_merge_kernel(const int8_t *__restrict__ q, const float *__restrict__ scale,
                     const int32_t *__restrict__ rowmap, const __nv_bfloat16 *__restrict__ y_act,
                     int NT, int D, __nv_bfloat16 *__restrict__ y) {
    const int C = D >> 4;
    const int64_t total = (int64_t)NT * C;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int i = (int)(t / C), c = (int)(t % C);
        const int pos = rowmap[i];
        uint4 *o = reinterpret_cast<uint4 *>(y + (int64_t)i * D + 16 * c);
        if (pos >= 0) {
            if (y_act) {
                const uint4 *a = reinterpret_cast<const uint4 *>(y_act + (int64_t)pos * D + 16 * c);
                const uint4 v0 = __ldcs(a), v1 = __ldcs(a + 1);
                __stcs(o, v0);
                __stcs(o + 1, v1);
            }
        } else {
            const int4 qv = __ldcs(reinterpret_cast<const int4 *>(q + (int64_t)i * D + 16 * c));
            float f[16];
            dequant16(qv, scale[i], f);
            __stcs(o, pack8_bf16(f));
            __stcs(o + 1, pack8_bf16(f + 8));
        }
    }
}

// The merge and the int8 write of the active rows in one pass over every row
// (Sec. 3.3 mask fusion, Sec. 3.4 cache write): 16 elements per thread.  A row
// with rowmap[i] < 0 is reconstructed from the cache into y (bf16(q s)); an
// active row, which the FFN-down epilogue already stored in y together with
// its max |v| (amax_bits[rowmap[i]], fp32 bits), is quantised into the cache
// with the rules and bits of quant_kernel (the thread of the row's first 16
// elements writes its scale).  Both kinds move 3 bytes per element.
__global__ void __launch_bounds__(kVecThreads)
merge_quant_kernel(int8_t *__restrict__ q, float *__restrict__ scale,
                   const int32_t *__restrict__ rowmap, const uint32_t *__restrict__ amax_bits,
                   int NT, int D, __nv_bfloat16 *__restrict__ y, int *err) {
    const int C = D >> 4;
    const int64_t total = (int64_t)NT * C;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int i = (int)(t / C), c = (int)(t % C);
        const int pos = rowmap[i];
        uint4 *o = reinterpret_cast<uint4 *>(y + (int64_t)i * D + 16 * c);
        int4 *qr = reinterpret_cast<int4 *>(q + (int64_t)i * D + 16 * c);
        if (pos < 0) {
            const int4 qv = __ldcs(qr);
            float f[16];
            dequant16(qv, scale[i], f);
            __stcs(o, pack8_bf16(f));
            __stcs(o + 1, pack8_bf16(f + 8));
            continue;
        }
        const uint32_t ab = amax_bits[pos];
        if (ab >= 0x7F800000u) {   // NaN or infinity in the row
            __stcs(qr, make_int4(0, 0, 0, 0));
            if (c == 0) {
                scale[i] = ab > 0x7F800000u ? __int_as_float(0x7fc00000) : INFINITY;
                echo_flag_error(err, ECHO_ERR_NONFINITE);
            }
            continue;
        }
        const float amax = __uint_as_float(ab);
        float sc = 0.f, inv = 0.f;
        if (amax > 0.f) {
            sc = __fdiv_rn(amax, 127.f);
            inv = __fdiv_rn(127.f, amax);
        }
        const uint4 v0 = __ldcs(o), v1 = __ldcs(o + 1);
        float f[16];
        unpack8_bf16(v0, f);
        unpack8_bf16(v1, f + 8);
        uint32_t w[4] = {0u, 0u, 0u, 0u};
#pragma unroll
        for (int k = 0; k < 16; ++k) {
            float r = rintf(__fmul_rn(f[k], inv));
            r = fminf(fmaxf(r, -127.f), 127.f);
            w[k >> 2] |= (uint32_t)(uint8_t)(int8_t)(int)r << (8 * (k & 3));
        }
        __stcs(qr, make_int4((int)w[0], (int)w[1], (int)w[2], (int)w[3]));
        if (c == 0) scale[i] = sc;
    }
}

int grid_for(int64_t work, int threads) {
    int64_t g = (work + threads - 1) / threads;
    const int64_t cap = 152 * 32;
    if (g > cap) g = cap;
    return (int)(g < 1 ? 1 : g);
}

}  // namespace

namespace echo {

void launch_quant(const void *src, echo_dtype st_t, const int32_t *rows, int32_t n_rows,
                  int32_t D, int8_t *q, float *scale, cudaStream_t st) {
    if (n_rows <= 0) return;
    const int warps = kQuantThreads / 32;
    const int grid = grid_for((int64_t)n_rows * 32, kQuantThreads);
    (void)warps;
    int *err = device_error_ptr();
    LaunchScope ls(ECHO_K_QUANT, n_rows, D, 0, st);
    if (st_t == ECHO_BF16)
        quant_kernel<__nv_bfloat16><<<grid, kQuantThreads, 0, st>>>(
            static_cast<const __nv_bfloat16 *>(src), rows, n_rows, D, q, scale, err);
    else
        quant_kernel<float><<<grid, kQuantThreads, 0, st>>>(static_cast<const float *>(src), rows,
                                                            n_rows, D, q, scale, err);
}

void launch_dequant(const int8_t *q, const float *scale, const int32_t *rows, int32_t n_rows,
                    int32_t D, void *dst, echo_dtype dt, cudaStream_t st) {
    if (n_rows <= 0) return;
    const int grid = grid_for((int64_t)n_rows * (D / 16), kVecThreads);
    LaunchScope ls(ECHO_K_DEQUANT, n_rows, D, 0, st);
    if (dt == ECHO_BF16)
        dequant_kernel<__nv_bfloat16><<<grid, kVecThreads, 0, st>>>(
            q, scale, rows, n_rows, D, static_cast<__nv_bfloat16 *>(dst));
    else
        dequant_kernel<float><<<grid, kVecThreads, 0, st>>>(q, scale, rows, n_rows, D,
                                                            static_cast<float *>(dst));
}

void launch_rowmap(const int32_t *idx, int32_t K, int32_t NT, int32_t *rowmap, uint32_t *zero,
                   int32_t n_zero, cudaStream_t st) {
    const int n = NT > n_zero ? NT : n_zero;
    if (n <= 0) return;
    LaunchScope ls(ECHO_K_ROWMAP, K, NT, 0, st);
    rowmap_kernel<<<(n + 255) / 256, 256, 0, st>>>(idx, K, NT, rowmap, zero, n_zero);
}

void launch_dequant_merge(const int8_t *q, const float *scale, const int32_t *rowmap,
                          const void *y_act, int32_t NT, int32_t D, void *y, cudaStream_t st) {
    const int grid = grid_for((int64_t)NT * (D / 16), kVecThreads);
    LaunchScope ls(ECHO_K_MERGE, NT, D, 0, st);
    dequant_merge_kernel<<<grid, kVecThreads, 0, st>>>(
        q, scale, rowmap, static_cast<const __nv_bfloat16 *>(y_act), NT, D,
        static_cast<__nv_bfloat16 *>(y));
}

void launch_merge_quant(int8_t *q, float *scale, const int32_t *rowmap, const uint32_t *amax,
                        int32_t NT, int32_t D, int32_t K, void *y, cudaStream_t st) {
    const int grid = grid_for((int64_t)NT * (D / 16), kVecThreads);
    LaunchScope ls(ECHO_K_MERGE_QUANT, NT, D, K, st);
    merge_quant_kernel<<<grid, kVecThreads, 0, st>>>(q, scale, rowmap, amax, NT, D,
                                                     static_cast<__nv_bfloat16 *>(y),
                                                     device_error_ptr());
}

}  // namespace echo

extern "C" echo_status echo_cache_quant(const void *src, echo_dtype st_t, const int32_t *rows,
                                        int32_t n_rows, int32_t D, int8_t *q, float *scale,
                                        echo_stream_t stream) {
    using namespace echo;
    if (n_rows < 0 || D < 8 || D % 8) return ECHO_ERR_SHAPE;
    if (n_rows == 0) return ECHO_OK;
    if (!src || !q || !scale) return ECHO_ERR_INVALID_ARG;
    if (st_t != ECHO_BF16 && st_t != ECHO_F32) return ECHO_ERR_INVALID_ARG;
    if (!aligned16(src) || !aligned16(q) || !aligned16(scale) || (rows && !aligned16(rows)))
        return ECHO_ERR_INVALID_ARG;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    launch_quant(src, st_t, rows, n_rows, D, q, scale, reinterpret_cast<cudaStream_t>(stream));
    return last_launch_status();
}

extern "C" echo_status echo_cache_dequant(const int8_t *q, const float *scale, const int32_t *rows,
                                          int32_t n_rows, int32_t D, void *dst, echo_dtype dt,
                                          echo_stream_t stream) {
    using namespace echo;
    if (n_rows < 0 || D < 16 || D % 16) return ECHO_ERR_SHAPE;
    if (n_rows == 0) return ECHO_OK;
    if (!q || !scale || !dst) return ECHO_ERR_INVALID_ARG;
    if (dt != ECHO_BF16 && dt != ECHO_F32) return ECHO_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(scale) || !aligned16(dst) || (rows && !aligned16(rows)))
        return ECHO_ERR_INVALID_ARG;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    launch_dequant(q, scale, rows, n_rows, D, dst, dt, reinterpret_cast<cudaStream_t>(stream));
    return last_launch_status();
}
