// Step-level adaptive update rate (Sec. 3.3): Eq. 1 on two consecutive step
// outputs, reduced over every element, and the clip rule that turns the
// normalised change into the step's refresh budget.
//
// step_delta_partial: grid-stride over 16-byte chunks of both outputs with a
//   fixed grid (independent of the device), so the summation order depends on
//   n only.  Per chunk the |h_prev - h_cur| and |h_cur| values are summed
//   pairwise in fp32, chunk sums go into a compensated (Neumaier) fp32 sum per
//   thread, and the threads of a block are combined in fp64 in a fixed order.
// step_delta_final: one warp adds the block partials in fp64 in a fixed order
//   and writes {Delta, sum|h_prev - h_cur|, sum|h_cur|}.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace {

constexpr int kDeltaThreads = 512;
// 4 x 152 blocks of 512 threads fill a 152-SM GPU in one wave (32 registers a
// thread); fixed, so results do not depend on the device
constexpr int kDeltaBlocks = 608;
constexpr int kDeltaUnroll = 2;

// Neumaier compensated sum of non-negative fp32 terms.
struct CompSum {
    float s = 0.f, c = 0.f;
    ECHO_DEV void add(float x) {
        const float t = __fadd_rn(s, x);
        const float big = s >= x ? s : x;
        const float small = s >= x ? x : s;
        c = __fadd_rn(c, __fadd_rn(__fsub_rn(big, t), small));
        s = t;
    }
    ECHO_DEV double value() const { return (double)s + (double)c; }
};

template <typename T>
struct Chunk;

template <>
struct Chunk<__nv_bfloat16> {
    static constexpr int kVals = 8;
    ECHO_DEV static void get(const uint4 &u, float *f) { unpack8_bf16(u, f); }
    ECHO_DEV static float scalar(const __nv_bfloat16 *p, int64_t i) { return __bfloat162float(p[i]); }
};

template <>
struct Chunk<float> {
    static constexpr int kVals = 4;
    ECHO_DEV static void get(const uint4 &u, float *f) {
        f[0] = __uint_as_float(u.x); f[1] = __uint_as_float(u.y);
        f[2] = __uint_as_float(u.z); f[3] = __uint_as_float(u.w);
    }
    ECHO_DEV static float scalar(const float *p, int64_t i) { return p[i]; }
};

// pairwise fp32 sum of kVals terms (8 or 4)
template <int V>
ECHO_DEV float tree_sum(const float *v) {
    if constexpr (V == 8)
        return __fadd_rn(__fadd_rn(__fadd_rn(v[0], v[1]), __fadd_rn(v[2], v[3])),
                         __fadd_rn(__fadd_rn(v[4], v[5]), __fadd_rn(v[6], v[7])));
    else
        return __fadd_rn(__fadd_rn(v[0], v[1]), __fadd_rn(v[2], v[3]));
}

ECHO_DEV double warp_sum_f64(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

template <typename T>
__global__ void __launch_bounds__(kDeltaThreads, 4)
step_delta_partial(const T *__restrict__ hp, const T *__restrict__ hc, int64_t n,
                   double *__restrict__ partial) {
    using C = Chunk<T>;
    constexpr int V = C::kVals;
    const int64_t chunks = n / V;
    const int64_t stride = (int64_t)gridDim.x * kDeltaThreads;
    const uint4 *pa = reinterpret_cast<const uint4 *>(hp);
    const uint4 *pb = reinterpret_cast<const uint4 *>(hc);
    CompSum sd, sc;
    for (int64_t base = (int64_t)blockIdx.x * kDeltaThreads + threadIdx.x; base < chunks;
         base += kDeltaUnroll * stride) {
        uint4 ua[kDeltaUnroll], ub[kDeltaUnroll];
#pragma unroll
        for (int u = 0; u < kDeltaUnroll; ++u) {
            const int64_t i = base + u * stride;
            if (i < chunks) {
                ua[u] = __ldcs(pa + i);
                ub[u] = __ldcs(pb + i);
            } else {
                ua[u] = make_uint4(0, 0, 0, 0);
                ub[u] = make_uint4(0, 0, 0, 0);
            }
        }
#pragma unroll
        for (int u = 0; u < kDeltaUnroll; ++u) {
            float a[V], b[V], d[V];
            C::get(ua[u], a);
            C::get(ub[u], b);
#pragma unroll
            for (int e = 0; e < V; ++e) {
                d[e] = fabsf(__fsub_rn(a[e], b[e]));
                b[e] = fabsf(b[e]);
            }
            sd.add(tree_sum<V>(d));
            sc.add(tree_sum<V>(b));
        }
    }
    // the last n % V elements: one each for the first threads of block 0
    const int64_t tail = n - chunks * V;
    if (blockIdx.x == 0 && threadIdx.x < tail) {
        const int64_t i = chunks * V + threadIdx.x;
        const float a = C::scalar(hp, i), b = C::scalar(hc, i);
        sd.add(fabsf(__fsub_rn(a, b)));
        sc.add(fabsf(b));
    }

    __shared__ double red[2][kDeltaThreads / 32];
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const double wd = warp_sum_f64(sd.value());
    const double wc = warp_sum_f64(sc.value());
    if (lane == 0) {
        red[0][warp] = wd;
        red[1][warp] = wc;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        double bd = 0.0, bc = 0.0;
        for (int w = 0; w < kDeltaThreads / 32; ++w) {
            bd += red[0][w];
            bc += red[1][w];
        }
        partial[2 * blockIdx.x] = bd;
        partial[2 * blockIdx.x + 1] = bc;
    }
}

__global__ void step_delta_final(const double *__restrict__ partial, int blocks, double xi,
                                 double *__restrict__ out, int *err) {
    double d = 0.0, c = 0.0;
    for (int j = threadIdx.x; j < blocks; j += 32) {
        d += partial[2 * j];
        c += partial[2 * j + 1];
    }
    d = warp_sum_f64(d);
    c = warp_sum_f64(c);
    if (threadIdx.x == 0) {
        const double delta = d / (c + xi);
        out[0] = delta;
        out[1] = d;
        out[2] = c;
        if (!isfinite(delta)) echo_flag_error(err, ECHO_ERR_NONFINITE);
    }
}

int delta_blocks(int64_t n, int vals) {
    const int64_t chunks = n / vals;
    const int64_t want = (chunks + kDeltaThreads - 1) / kDeltaThreads;
    return (int)(want < 1 ? 1 : (want > kDeltaBlocks ? kDeltaBlocks : want));
}

}  // namespace

extern "C" size_t echo_step_delta_workspace_size(int64_t n) {
    if (n < 0) return 0;
    return (size_t)kDeltaBlocks * 2 * sizeof(double);
}

extern "C" echo_status echo_step_delta(const void *h_prev, const void *h_cur, echo_dtype ht,
                                       int64_t n, double xi, double *out, void *workspace,
                                       size_t ws_bytes, echo_stream_t stream) {
    using namespace echo;
    if ((n > 0 && (!h_prev || !h_cur)) || !out || !workspace) return ECHO_ERR_INVALID_ARG;
    if (ht != ECHO_BF16 && ht != ECHO_F32) return ECHO_ERR_INVALID_ARG;
    if (!aligned16(h_prev) || !aligned16(h_cur) || !aligned16(workspace) ||
        (reinterpret_cast<uintptr_t>(out) & 7u))
        return ECHO_ERR_INVALID_ARG;
    if (!(xi > 0.0) || !isfinite(xi)) return ECHO_ERR_INVALID_ARG;
    if (n < 0) return ECHO_ERR_SHAPE;
    if (ws_bytes < echo_step_delta_workspace_size(n)) return ECHO_ERR_WORKSPACE;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    double *partial = static_cast<double *>(workspace);
    const int vals = ht == ECHO_BF16 ? 8 : 4;
    const int grid = delta_blocks(n, vals);
    {
        LaunchScope ls(ECHO_K_STEP_DELTA, n, ht == ECHO_BF16 ? 2 : 4, 0, st);
        if (ht == ECHO_BF16)
            step_delta_partial<__nv_bfloat16><<<grid, kDeltaThreads, 0, st>>>(
                static_cast<const __nv_bfloat16 *>(h_prev), static_cast<const __nv_bfloat16 *>(h_cur),
                n, partial);
        else
            step_delta_partial<float><<<grid, kDeltaThreads, 0, st>>>(
                static_cast<const float *>(h_prev), static_cast<const float *>(h_cur), n, partial);
    }
    if (last_launch_status() != ECHO_OK) return ECHO_ERR_CUDA;
    {
        LaunchScope ls(ECHO_K_STEP_DELTA, 0, 0, grid, st);
        step_delta_final<<<1, 32, 0, st>>>(partial, grid, xi, out, device_error_ptr());
    }
    return last_launch_status();
}

// Host arithmetic in fp64, one rounding per operation in this order (the
// library is built with floating-point contraction off):
//   dh = delta_ref > 0 ? delta / delta_ref : 0
//   r  = min(max(r_min + alpha * dh, r_min), r_max)
//   K  = min(max(ceil(r * NT), 0), NT)
extern "C" echo_status echo_update_rate(double delta, double delta_ref, const echo_rate_params *p,
                                        int32_t NT, double *rate, int32_t *K) {
    if (!p || !K) return ECHO_ERR_INVALID_ARG;
    if (NT < 0) return ECHO_ERR_SHAPE;
    if (!(p->r_min >= 0.0) || !(p->r_max <= 1.0) || !(p->r_min <= p->r_max) || !(p->alpha >= 0.0) ||
        !isfinite(p->alpha))
        return ECHO_ERR_INVALID_ARG;
    if (!isfinite(delta) || !isfinite(delta_ref) || delta < 0.0 || delta_ref < 0.0)
        return ECHO_ERR_NONFINITE;
    const double dh = delta_ref > 0.0 ? delta / delta_ref : 0.0;
    const double prod = p->alpha * dh;
    double r = p->r_min + prod;
    if (!(r >= p->r_min)) r = p->r_min;
    if (r > p->r_max) r = p->r_max;
    double k = ceil(r * (double)NT);
    if (k < 0.0) k = 0.0;
    if (k > (double)NT) k = (double)NT;
    if (rate) *rate = r;
    *K = (int32_t)k;
    return ECHO_OK;
}
