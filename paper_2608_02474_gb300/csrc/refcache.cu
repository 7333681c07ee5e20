// Cache forms of Sec. 3.4 beyond the plain int8 cache: the reference plus
// int8 residual manager (ECHO_CACHE_REF) and the full-precision ablation form
// (ECHO_CACHE_BF16).
//
// A REF write is four stream-ordered kernels:
//   ref_release  every written token drops its old reference (atomic
//                decrement of the slot's count) and the bounds of each scan
//                segment's written rows are recorded;
//   ref_scan     one CTA per scan segment walks its written rows in token
//                order, 8 rows a round: the rows are staged in shared memory,
//                the 16 warps compute every fp32 cosine the walk can need (each
//                row against the entering reference and against each earlier
//                row of the round, canonical order), then one thread walks the
//                8 rows and the last new reference carries into the next round;
//   ref_alloc    one CTA ranks the new references in token order and hands
//                them the free slots in slot order (block scans);
//   ref_store    one warp per written row: a reference copies its row into its
//                slot, a residual quantises x - r by the int8 rule, a run
//                without a slot quantises x itself.
// Reconstruction (read, merge) is one thread per 16 values: bf16(r + q s).
#include "common.cuh"
#include "internal.h"

namespace {

constexpr int kScanWarps = 16;
constexpr int kAllocThreads = 1024;
constexpr int kStoreThreads = 256;
constexpr int kVec = 256;

size_t al256(size_t b) { return (b + 255) & ~(size_t)255; }

int grid_for(int64_t work, int threads) {
    int64_t g = (work + threads - 1) / threads;
    const int64_t cap = 152 * 32;
    if (g > cap) g = cap;
    return (int)(g < 1 ? 1 : g);
}

ECHO_DEV bool bf16_nonfinite(uint32_t two) {
    return ((two & 0x7F80u) == 0x7F80u) || ((two & 0x7F800000u) == 0x7F800000u);
}

// ---------------------------------------------------------------- release
// every written token drops its reference (when a pool exists); the written
// rows of scan segment s are positions [seg_lo[s], seg_hi[s]) of rows (seg_lo
// stays -1 for a segment with none; rows ascending)
__global__ void ref_release_kernel(const int32_t *__restrict__ rows, int n, int seg_len,
                                   const int32_t *__restrict__ ref, int32_t *refcount,
                                   int32_t *__restrict__ seg_lo, int32_t *__restrict__ seg_hi) {
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j < n) {
        const int i = rows[j];
        if (refcount) {
            const int old = ref[i];
            if (old >= 0) atomicSub(&refcount[old], 1);
        }
        const int sg = i / seg_len;
        if (j == 0 || rows[j - 1] / seg_len != sg) seg_lo[sg] = j;
        if (j == n - 1 || rows[j + 1] / seg_len != sg) seg_hi[sg] = j + 1;
    }
}

// ---------------------------------------------------------------- scan
// The canonical-order fp32 sums <a, b> (and <a, a> when `norm`) of two bf16
// rows in shared memory: lane l owns 8-element chunks l, l+32, ..., adds each
// chunk's sum left to right into its accumulator in chunk order, then an xor
// butterfly 16..1.  Every lane returns the same sums.
ECHO_DEV void warp_dot(const uint4 *a, const uint4 *b, int C, int lane, bool norm, float &dot,
                       float &na) {
    dot = 0.f;
    na = 0.f;
    for (int c = lane; c < C; c += 32) {
        float fa[8], fb[8];
        unpack8_bf16(a[c], fa);
        unpack8_bf16(b[c], fb);
        float cd = __fmul_rn(fa[0], fb[0]);
        float cn = __fmul_rn(fa[0], fa[0]);
#pragma unroll
        for (int k = 1; k < 8; ++k) {
            cd = __fadd_rn(cd, __fmul_rn(fa[k], fb[k]));
            if (norm) cn = __fadd_rn(cn, __fmul_rn(fa[k], fa[k]));
        }
        dot = __fadd_rn(dot, cd);
        if (norm) na = __fadd_rn(na, cn);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        dot = __fadd_rn(dot, __shfl_xor_sync(0xffffffffu, dot, o));
        na = __fadd_rn(na, __shfl_xor_sync(0xffffffffu, na, o));
    }
}

// src_pos[j] = position (in rows) of row j's reference; j itself for a reference.
//
// One CTA per scan segment.  The segment's written rows are taken kWin at a
// time: the window's rows are staged in shared memory, then the CTA computes
// every similarity the walk over the window can need (each row against the
// reference it entered with and against every earlier row of the window), and
// one thread walks the window in order.  A window is resolved in one round
// whatever the data.  Dynamic shared memory: kWin window rows, then the
// current reference row (bf16, D each).
constexpr int kWin = 8;
constexpr int kPairs = kWin * (kWin + 1) / 2;

__global__ void __launch_bounds__(kScanWarps * 32)
ref_scan_kernel(const __nv_bfloat16 *__restrict__ src, const int32_t *__restrict__ seg_lo,
                const int32_t *__restrict__ seg_hi, float tau, int D,
                int32_t *__restrict__ src_pos) {
    extern __shared__ uint4 s_buf[];
    __shared__ float s_dot[kWin][kWin + 1];  // [w][t + 1], t = -1: the entering reference
    __shared__ float s_nv[kWin];
    __shared__ float s_nr;
    __shared__ int s_jr, s_newref;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int C = D >> 3;
    uint4 *ref = s_buf + (size_t)kWin * C;
    const int lo = seg_lo[blockIdx.x];
    if (lo < 0) return;
    const int hi = seg_hi[blockIdx.x];
    if (threadIdx.x == 0) {
        src_pos[lo] = lo;
        s_jr = lo;
    }
    // the segment's first written row is its first reference
    {
        const uint4 *v = reinterpret_cast<const uint4 *>(src + (int64_t)lo * D);
        for (int c = threadIdx.x; c < C; c += blockDim.x) ref[c] = __ldg(v + c);
    }
    __syncthreads();
    if (warp == 0) {
        float d, nr;
        warp_dot(ref, ref, C, lane, true, d, nr);
        if (lane == 0) s_nr = nr;
    }
    __syncthreads();
    for (int j = lo + 1; j < hi; j += kWin) {
        const int nvalid = hi - j < kWin ? hi - j : kWin;
        // stage the window's rows, four 16-byte loads in flight per thread
        const int total = nvalid * C;
        for (int b = threadIdx.x; b < total; b += 4 * (int)blockDim.x) {
            uint4 u[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int e = b + k * blockDim.x;
                if (e < total) {
                    const int w = e / C, c = e - w * C;
                    u[k] = __ldg(reinterpret_cast<const uint4 *>(src + (int64_t)(j + w) * D) + c);
                }
            }
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int e = b + k * blockDim.x;
                if (e < total) s_buf[e] = u[k];
            }
        }
        __syncthreads();
        // pair p = (w, t): row w of the window against t = -1 (the entering
        // reference) or the earlier window row t; pairs of row w start at w(w+1)/2
        for (int p = warp; p < kPairs; p += kScanWarps) {
            int w = 0;
            while ((w + 1) * (w + 2) / 2 <= p) ++w;
            const int t = p - w * (w + 1) / 2 - 1;
            if (w >= nvalid) continue;
            float dot, nv;
            warp_dot(s_buf + (size_t)w * C, t < 0 ? ref : s_buf + (size_t)t * C, C, lane, t < 0,
                     dot, nv);
            if (lane == 0) {
                s_dot[w][t + 1] = dot;
                if (t < 0) s_nv[w] = nv;
            }
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            int cur = -1;
            float ncur = s_nr;
            const int jr = s_jr;
            for (int w = 0; w < nvalid; ++w) {
                const float nv = s_nv[w];
                float sim = 0.f;
                if (nv > 0.f && ncur > 0.f)
                    sim = __fdiv_rn(s_dot[w][cur + 1], __fmul_rn(__fsqrt_rn(nv), __fsqrt_rn(ncur)));
                if (sim > tau) {
                    src_pos[j + w] = cur < 0 ? jr : j + cur;
                } else {
                    src_pos[j + w] = j + w;
                    cur = w;
                    ncur = nv;
                }
            }
            s_newref = cur;
            if (cur >= 0) {
                s_jr = j + cur;
                s_nr = ncur;
            }
        }
        __syncthreads();
        const int nr = s_newref;
        if (nr >= 0)
            for (int c = threadIdx.x; c < C; c += blockDim.x) ref[c] = s_buf[(size_t)nr * C + c];
        __syncthreads();
    }
}

// ---------------------------------------------------------------- alloc
// exclusive block scan of one value per thread; *total gets the block sum
ECHO_DEV int block_scan(int v, int *warp_sums, int *total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += t;
    }
    if (lane == 31) warp_sums[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        const int w = lane < (int)(blockDim.x >> 5) ? warp_sums[lane] : 0;
        int wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int t = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += t;
        }
        warp_sums[lane] = wi - w;
        if (lane == 31) warp_sums[32] = wi;
    }
    __syncthreads();
    const int r = warp_sums[warp] + inc - v;
    *total = warp_sums[32];
    __syncthreads();
    return r;
}

// slot_of[j] = pool slot of the reference at position j (-1: none or not a reference)
__global__ void __launch_bounds__(kAllocThreads)
ref_alloc_kernel(const int32_t *__restrict__ src_pos, int n, const int32_t *__restrict__ refcount,
                 int R_cap, int32_t *__restrict__ free_list, int32_t *__restrict__ slot_of) {
    __shared__ int warp_sums[33];
    // rank the references in token order
    int run = 0;
    for (int base = 0; base < n; base += kAllocThreads) {
        const int j = base + threadIdx.x;
        const int is_ref = j < n && src_pos[j] == j;
        int tot;
        const int r = run + block_scan(is_ref, warp_sums, &tot);
        if (j < n) slot_of[j] = is_ref ? r : -1;
        run += tot;
    }
    const int n_new = run;
    // the first n_new free slots in slot order
    int nfree = 0;
    for (int base = 0; base < R_cap && nfree < n_new; base += kAllocThreads) {
        const int sl = base + threadIdx.x;
        const int fr = sl < R_cap && refcount[sl] == 0;
        int tot;
        const int m = nfree + block_scan(fr, warp_sums, &tot);
        if (fr && m < n_new) free_list[m] = sl;
        nfree += tot;
    }
    const int avail = nfree < n_new ? nfree : n_new;
    __syncthreads();
    for (int j = threadIdx.x; j < n; j += kAllocThreads) {
        const int r = slot_of[j];
        if (r >= 0) slot_of[j] = r < avail ? free_list[r] : -1;
    }
}

// ---------------------------------------------------------------- store
__global__ void __launch_bounds__(kStoreThreads)
ref_store_kernel(const __nv_bfloat16 *__restrict__ src, const int32_t *__restrict__ rows, int n,
                 int D, const int32_t *__restrict__ src_pos, const int32_t *__restrict__ slot_of,
                 int8_t *__restrict__ q, float *__restrict__ scale, int32_t *__restrict__ ref,
                 int32_t *refcount, __nv_bfloat16 *__restrict__ pool, int *err) {
    const int lane = threadIdx.x & 31;
    const int warps = blockDim.x >> 5;
    const int C = D >> 3;
    for (int j = blockIdx.x * warps + (threadIdx.x >> 5); j < n; j += gridDim.x * warps) {
        const int i = rows[j];
        const int jr = src_pos[j];
        const int sl = slot_of[jr];
        const __nv_bfloat16 *v = src + (int64_t)j * D;
        int8_t *qr = q + (int64_t)i * D;
        if (sl >= 0 && jr == j) {  // a new reference: the row itself into its slot
            bool bad = false;
            __nv_bfloat16 *pr = pool + (int64_t)sl * D;
            for (int c = lane; c < C; c += 32) {
                const uint4 u = *reinterpret_cast<const uint4 *>(v + 8 * c);
                bad |= bf16_nonfinite(u.x) || bf16_nonfinite(u.y) || bf16_nonfinite(u.z) ||
                       bf16_nonfinite(u.w);
                *reinterpret_cast<uint4 *>(pr + 8 * c) = u;
                *reinterpret_cast<uint2 *>(qr + 8 * c) = make_uint2(0, 0);
            }
            bad = __any_sync(0xffffffffu, bad);
            if (lane == 0) {
                scale[i] = 0.f;
                ref[i] = sl;
                atomicAdd(&refcount[sl], 1);
                if (bad) echo_flag_error(err, ECHO_ERR_NONFINITE);
            }
            continue;
        }
        // residual against the reference row, or the row itself without one
        const __nv_bfloat16 *r = sl >= 0 ? src + (int64_t)jr * D : nullptr;
        float amax = 0.f;
        bool nan = false, inf = false;
        for (int c = lane; c < C; c += 32) {
            float f[8], g[8];
            unpack8_bf16(*reinterpret_cast<const uint4 *>(v + 8 * c), f);
            if (r) unpack8_bf16(*reinterpret_cast<const uint4 *>(r + 8 * c), g);
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const float a = fabsf(r ? __fsub_rn(f[k], g[k]) : f[k]);
                nan |= a != a;
                inf |= a == INFINITY;
                amax = fmaxf(amax, a);
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
        nan = __any_sync(0xffffffffu, nan);
        inf = __any_sync(0xffffffffu, inf);
        if (lane == 0) {
            ref[i] = sl >= 0 ? sl : -1;
            if (sl >= 0) atomicAdd(&refcount[sl], 1);
        }
        if (nan || inf) {
            for (int c = lane; c < C; c += 32) *reinterpret_cast<uint2 *>(qr + 8 * c) = make_uint2(0, 0);
            if (lane == 0) {
                scale[i] = nan ? __int_as_float(0x7fc00000) : INFINITY;
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
            float f[8], g[8];
            unpack8_bf16(*reinterpret_cast<const uint4 *>(v + 8 * c), f);
            if (r) unpack8_bf16(*reinterpret_cast<const uint4 *>(r + 8 * c), g);
            uint32_t w[2] = {0u, 0u};
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const float dv = r ? __fsub_rn(f[k], g[k]) : f[k];
                float t = rintf(__fmul_rn(dv, inv));
                t = fminf(fmaxf(t, -127.f), 127.f);
                const uint32_t b = (uint32_t)(uint8_t)(int8_t)(int)t;
                w[k >> 2] |= b << (8 * (k & 3));
            }
            *reinterpret_cast<uint2 *>(qr + 8 * c) = make_uint2(w[0], w[1]);
        }
        if (lane == 0) scale[i] = sc;
    }
}

// ---------------------------------------------------------------- reconstruction
// 16 values of token i: bf16(r + float(q) s), r = 0 without a reference
ECHO_DEV void ref_reconstruct16(const echo_cache &c, int i, int col, uint4 *out) {
    const int rs = c.ref[i];
    const float s = c.scale[i];
    const int4 qv = __ldcs(reinterpret_cast<const int4 *>(c.q + (int64_t)i * c.D + col));
    const int8_t *qb = reinterpret_cast<const int8_t *>(&qv);
    float r[16];
    if (rs >= 0) {
        const uint4 *p = reinterpret_cast<const uint4 *>(
            static_cast<const __nv_bfloat16 *>(c.pool) + (int64_t)rs * c.D + col);
        unpack8_bf16(p[0], r);
        unpack8_bf16(p[1], r + 8);
    } else {
#pragma unroll
        for (int k = 0; k < 16; ++k) r[k] = 0.f;
    }
    float f[16];
#pragma unroll
    for (int k = 0; k < 16; ++k) f[k] = __fadd_rn(r[k], __fmul_rn((float)qb[k], s));
    out[0] = pack8_bf16(f);
    out[1] = pack8_bf16(f + 8);
}

template <int KIND>
ECHO_DEV void reconstruct16(const echo_cache &c, int i, int col, uint4 *out) {
    if constexpr (KIND == ECHO_CACHE_BF16) {
        const uint4 *p = reinterpret_cast<const uint4 *>(
            static_cast<const __nv_bfloat16 *>(c.full) + (int64_t)i * c.D + col);
        out[0] = __ldcs(p);
        out[1] = __ldcs(p + 1);
    } else {
        ref_reconstruct16(c, i, col, out);
    }
}

template <int KIND>
__global__ void __launch_bounds__(kVec)
cache_read_kernel(echo_cache c, const int32_t *__restrict__ rows, int n,
                  __nv_bfloat16 *__restrict__ dst) {
    const int C = c.D >> 4;
    const int64_t total = (int64_t)n * C;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int j = (int)(t / C), col = 16 * (int)(t % C);
        const int i = rows ? rows[j] : j;
        uint4 o[2];
        reconstruct16<KIND>(c, i, col, o);
        uint4 *d = reinterpret_cast<uint4 *>(dst + (int64_t)j * c.D + col);
        d[0] = o[0];
        d[1] = o[1];
    }
}

// y[i] = y_act[rowmap[i]] if rowmap[i] >= 0 else the reconstruction of token i
template <int KIND>
__global__ void __launch_bounds__(kVec)
cache_merge_kernel(echo_cache c, const int32_t *__restrict__ rowmap,
                   const __nv_bfloat16 *__restrict__ y_act, __nv_bfloat16 *__restrict__ y) {
    const int C = c.D >> 4;
    const int64_t total = (int64_t)c.NT * C;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int i = (int)(t / C), col = 16 * (int)(t % C);
        const int pos = rowmap[i];
        uint4 *o = reinterpret_cast<uint4 *>(y + (int64_t)i * c.D + col);
        uint4 v[2];
        if (pos >= 0) {
            const uint4 *a = reinterpret_cast<const uint4 *>(y_act + (int64_t)pos * c.D + col);
            v[0] = __ldcs(a);
            v[1] = __ldcs(a + 1);
        } else {
            reconstruct16<KIND>(c, i, col, v);
        }
        __stcs(o, v[0]);
        __stcs(o + 1, v[1]);
    }
}

// full[rows[j]] = src[j] (BF16 form)
__global__ void __launch_bounds__(kVec)
cache_copy_kernel(const __nv_bfloat16 *__restrict__ src, const int32_t *__restrict__ rows, int n,
                  int D, __nv_bfloat16 *__restrict__ full, int *err) {
    const int C = D >> 3;
    const int64_t total = (int64_t)n * C;
    bool bad = false;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int j = (int)(t / C), c = (int)(t % C);
        const uint4 u = __ldcs(reinterpret_cast<const uint4 *>(src + (int64_t)j * D + 8 * c));
        bad |= bf16_nonfinite(u.x) || bf16_nonfinite(u.y) || bf16_nonfinite(u.z) ||
               bf16_nonfinite(u.w);
        *reinterpret_cast<uint4 *>(full + (int64_t)rows[j] * D + 8 * c) = u;
    }
    if (bad) echo_flag_error(err, ECHO_ERR_NONFINITE);
}

__global__ void cache_stats_kernel(const int32_t *__restrict__ refcount, int R_cap,
                                   int32_t *__restrict__ out) {
    __shared__ int s_live, s_top;
    if (threadIdx.x == 0) {
        s_live = 0;
        s_top = 0;
    }
    __syncthreads();
    int live = 0, top = 0;
    for (int sl = threadIdx.x; sl < R_cap; sl += blockDim.x)
        if (refcount[sl] > 0) {
            ++live;
            top = sl + 1;
        }
    atomicAdd(&s_live, live);
    atomicMax(&s_top, top);
    __syncthreads();
    if (threadIdx.x == 0) {
        out[0] = s_live;
        out[1] = s_top;
    }
}

struct RefWs {
    int32_t *src_pos, *slot_of, *free_list, *seg_lo, *seg_hi;
};

int n_segments(const echo_cache &c) {
    return (int)((c.NT + (int64_t)c.seg_len - 1) / c.seg_len);
}

size_t ref_ws_bytes(const echo_cache &c, int32_t n) {
    const size_t a = al256(sizeof(int32_t) * (size_t)(n > 0 ? n : 1));
    const size_t b = al256(sizeof(int32_t) * (size_t)n_segments(c));
    return 3 * a + 2 * b;
}

RefWs ref_ws(const echo_cache &c, void *ws, int32_t n) {
    const size_t a = al256(sizeof(int32_t) * (size_t)(n > 0 ? n : 1));
    const size_t b = al256(sizeof(int32_t) * (size_t)n_segments(c));
    uint8_t *p = static_cast<uint8_t *>(ws);
    return {reinterpret_cast<int32_t *>(p), reinterpret_cast<int32_t *>(p + a),
            reinterpret_cast<int32_t *>(p + 2 * a), reinterpret_cast<int32_t *>(p + 3 * a),
            reinterpret_cast<int32_t *>(p + 3 * a + b)};
}

}  // namespace

namespace echo {

echo_status cache_check(const echo_cache *c) {
    if (!c) return ECHO_ERR_INVALID_ARG;
    if (c->NT < 1 || c->D < 16 || c->D % 16) return ECHO_ERR_SHAPE;
    if ((int64_t)c->NT > (int64_t)INT32_MAX / 2) return ECHO_ERR_SHAPE;
    switch (c->kind) {
    case ECHO_CACHE_INT8:
        if (!c->q || !c->scale || !aligned16(c->q) || !aligned16(c->scale)) return ECHO_ERR_INVALID_ARG;
        return ECHO_OK;
    case ECHO_CACHE_BF16:
        if (!c->full || !aligned16(c->full)) return ECHO_ERR_INVALID_ARG;
        return ECHO_OK;
    case ECHO_CACHE_REF:
        if (!c->q || !c->scale || !c->ref || !aligned16(c->q) || !aligned16(c->scale) ||
            !aligned16(c->ref))
            return ECHO_ERR_INVALID_ARG;
        if (c->R_cap < 0 || c->seg_len < 1 || !(c->tau == c->tau)) return ECHO_ERR_INVALID_ARG;
        if (c->R_cap > 0 && (!c->pool || !c->refcount || !aligned16(c->pool) ||
                             !aligned16(c->refcount)))
            return ECHO_ERR_INVALID_ARG;
        return ECHO_OK;
    default:
        return ECHO_ERR_INVALID_ARG;
    }
}

size_t cache_write_ws(const echo_cache &c, int32_t n) {
    return c.kind == ECHO_CACHE_REF ? ref_ws_bytes(c, n) : 0;
}

echo_status launch_cache_write(const echo_cache &c, const void *src, const int32_t *rows,
                               int32_t n, void *ws, cudaStream_t st) {
    if (n <= 0) return ECHO_OK;
    int *err = device_error_ptr();
    const __nv_bfloat16 *s = static_cast<const __nv_bfloat16 *>(src);
    if (c.kind == ECHO_CACHE_INT8) {
        launch_quant(src, ECHO_BF16, rows, n, c.D, c.q, c.scale, st);
        return last_launch_status();
    }
    if (c.kind == ECHO_CACHE_BF16) {
        LaunchScope ls(ECHO_K_CACHE_COPY, n, c.D, 0, st);
        cache_copy_kernel<<<grid_for((int64_t)n * (c.D / 8), kVec), kVec, 0, st>>>(
            s, rows, n, c.D, static_cast<__nv_bfloat16 *>(c.full), err);
        return last_launch_status();
    }
    const RefWs w = ref_ws(c, ws, n);
    const int nseg = n_segments(c);
    if (cudaMemsetAsync(w.seg_lo, 0xFF, sizeof(int32_t) * (size_t)nseg, st) != cudaSuccess)
        return ECHO_ERR_CUDA;
    {
        LaunchScope ls(ECHO_K_REF_ALLOC, n, c.D, 0, st);
        ref_release_kernel<<<(n + 255) / 256, 256, 0, st>>>(
            rows, n, c.seg_len, c.ref, c.R_cap > 0 ? c.refcount : nullptr, w.seg_lo, w.seg_hi);
    }
    if (last_launch_status() != ECHO_OK) return ECHO_ERR_CUDA;
    {
        const size_t smem = (size_t)(kWin + 1) * c.D * sizeof(__nv_bfloat16);
        if (smem > 48 * 1024 &&
            cudaFuncSetAttribute(ref_scan_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem) != cudaSuccess)
            return ECHO_ERR_CUDA;
        LaunchScope ls(ECHO_K_REF_SCAN, n, c.D, 0, st);
        ref_scan_kernel<<<nseg, kScanWarps * 32, smem, st>>>(s, w.seg_lo, w.seg_hi, c.tau, c.D,
                                                             w.src_pos);
    }
    if (last_launch_status() != ECHO_OK) return ECHO_ERR_CUDA;
    {
        LaunchScope ls(ECHO_K_REF_ALLOC, n, c.D, 0, st);
        ref_alloc_kernel<<<1, kAllocThreads, 0, st>>>(w.src_pos, n, c.refcount, c.R_cap,
                                                       w.free_list, w.slot_of);
    }
    if (last_launch_status() != ECHO_OK) return ECHO_ERR_CUDA;
    {
        LaunchScope ls(ECHO_K_REF_STORE, n, c.D, 0, st);
        ref_store_kernel<<<grid_for((int64_t)n * 32, kStoreThreads), kStoreThreads, 0, st>>>(
            s, rows, n, c.D, w.src_pos, w.slot_of, c.q, c.scale, c.ref, c.refcount,
            static_cast<__nv_bfloat16 *>(c.pool), err);
    }
    return last_launch_status();
}

void launch_cache_merge(const echo_cache &c, const int32_t *rowmap, const void *y_act, void *y,
                        cudaStream_t st) {
    if (c.kind == ECHO_CACHE_INT8) {
        launch_dequant_merge(c.q, c.scale, rowmap, y_act, c.NT, c.D, y, st);
        return;
    }
    const int grid = grid_for((int64_t)c.NT * (c.D / 16), kVec);
    LaunchScope ls(ECHO_K_MERGE, c.NT, c.D, 0, st);
    const __nv_bfloat16 *ya = static_cast<const __nv_bfloat16 *>(y_act);
    __nv_bfloat16 *yo = static_cast<__nv_bfloat16 *>(y);
    if (c.kind == ECHO_CACHE_BF16)
        cache_merge_kernel<ECHO_CACHE_BF16><<<grid, kVec, 0, st>>>(c, rowmap, ya, yo);
    else
        cache_merge_kernel<ECHO_CACHE_REF><<<grid, kVec, 0, st>>>(c, rowmap, ya, yo);
}

}  // namespace echo

extern "C" echo_status echo_cache_reset(const echo_cache *c, echo_stream_t stream) {
    using namespace echo;
    const echo_status v = cache_check(c);
    if (v != ECHO_OK) return v;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const size_t NT = c->NT, D = c->D;
    bool ok = true;
    if (c->kind != ECHO_CACHE_BF16) {
        ok &= cudaMemsetAsync(c->q, 0, NT * D, st) == cudaSuccess;
        ok &= cudaMemsetAsync(c->scale, 0, NT * sizeof(float), st) == cudaSuccess;
    }
    if (c->kind == ECHO_CACHE_BF16) ok &= cudaMemsetAsync(c->full, 0, NT * D * 2, st) == cudaSuccess;
    if (c->kind == ECHO_CACHE_REF) {
        ok &= cudaMemsetAsync(c->ref, 0xFF, NT * sizeof(int32_t), st) == cudaSuccess;
        if (c->R_cap > 0)
            ok &= cudaMemsetAsync(c->refcount, 0, (size_t)c->R_cap * sizeof(int32_t), st) ==
                  cudaSuccess;
    }
    return ok ? ECHO_OK : ECHO_ERR_CUDA;
}

extern "C" size_t echo_cache_write_workspace_size(const echo_cache *c, int32_t n_rows) {
    if (echo::cache_check(c) != ECHO_OK || n_rows < 0) return 0;
    return echo::cache_write_ws(*c, n_rows);
}

extern "C" echo_status echo_cache_write(const echo_cache *c, const void *src, const int32_t *rows,
                                        int32_t n_rows, void *workspace, size_t ws_bytes,
                                        echo_stream_t stream) {
    using namespace echo;
    const echo_status v = cache_check(c);
    if (v != ECHO_OK) return v;
    if (n_rows < 0 || n_rows > c->NT) return ECHO_ERR_SHAPE;
    if (n_rows == 0) return ECHO_OK;
    if (!src || !rows || !aligned16(src) || !aligned16(rows)) return ECHO_ERR_INVALID_ARG;
    const size_t need = cache_write_ws(*c, n_rows);
    if (need && (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u)))
        return ECHO_ERR_INVALID_ARG;
    if (ws_bytes < need) return ECHO_ERR_WORKSPACE;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    return launch_cache_write(*c, src, rows, n_rows, workspace,
                              reinterpret_cast<cudaStream_t>(stream));
}

extern "C" echo_status echo_cache_read(const echo_cache *c, const int32_t *rows, int32_t n_rows,
                                       void *dst, echo_stream_t stream) {
    using namespace echo;
    const echo_status v = cache_check(c);
    if (v != ECHO_OK) return v;
    if (n_rows < 0) return ECHO_ERR_SHAPE;
    if (n_rows == 0) return ECHO_OK;
    if (!dst || !aligned16(dst) || (rows && !aligned16(rows))) return ECHO_ERR_INVALID_ARG;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (c->kind == ECHO_CACHE_INT8) {
        launch_dequant(c->q, c->scale, rows, n_rows, c->D, dst, ECHO_BF16, st);
        return last_launch_status();
    }
    const int grid = grid_for((int64_t)n_rows * (c->D / 16), kVec);
    LaunchScope ls(ECHO_K_DEQUANT, n_rows, c->D, 0, st);
    __nv_bfloat16 *d = static_cast<__nv_bfloat16 *>(dst);
    if (c->kind == ECHO_CACHE_BF16)
        cache_read_kernel<ECHO_CACHE_BF16><<<grid, kVec, 0, st>>>(*c, rows, n_rows, d);
    else
        cache_read_kernel<ECHO_CACHE_REF><<<grid, kVec, 0, st>>>(*c, rows, n_rows, d);
    return last_launch_status();
}

extern "C" echo_status echo_cache_stats(const echo_cache *c, int32_t *out, echo_stream_t stream) {
    using namespace echo;
    const echo_status v = cache_check(c);
    if (v != ECHO_OK) return v;
    if (c->kind != ECHO_CACHE_REF || !out) return ECHO_ERR_INVALID_ARG;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (c->R_cap == 0) return cudaMemsetAsync(out, 0, 2 * sizeof(int32_t), st) == cudaSuccess
                                  ? ECHO_OK : ECHO_ERR_CUDA;
    {
        LaunchScope ls(ECHO_K_REF_ALLOC, c->R_cap, 0, 0, st);
        cache_stats_kernel<<<1, 1024, 0, st>>>(c->refcount, c->R_cap, out);
    }
    return last_launch_status();
}
