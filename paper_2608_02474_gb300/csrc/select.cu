// Token selection (Sec. 3.3): per-token drift (Eq. 1 applied per token against
// the int8 cache), weighted by the token's segment energy, then top-K by
// (score descending, index ascending) returned as an ascending index list.
//
// drift_kernel: one warp per token row, 128-bit loads of x and 64-bit loads of
//   the int8 cache; the two L1 sums are fp32 in the canonical order (lane l owns
//   8-element chunks l, l+32, ...; chunk sums left to right; xor butterfly
//   16..1), with explicit round-to-nearest intrinsics so nothing is contracted.
// topk_kernel: one CTA radix-selects the K-th largest 32-bit key (11/11/10-bit
//   digits), then compacts in index order, taking keys equal to the threshold
//   from the lowest index up.  Keys are read four at a time (16-byte loads,
//   several in flight per thread): the kernel is bound by load latency.
// topk_cluster_kernel: the same selection with the keys split over a cluster
//   of 8 CTAs, the histograms summed through distributed shared memory; used
//   from 10240 keys up (28.7 -> 18.3 us at 32760 keys, 53 -> 20 us at 63960).
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace {

constexpr int kDriftThreads = 256;
constexpr int kDriftUnroll = 4;
constexpr int kTopkThreads = 1024;
constexpr int kTopkItems = 4;

ECHO_DEV float segment_weight(float e, float emax, float lam) {
    if (!(emax > 0.f)) return 1.f;
    const float t = __fdiv_rn(e, emax);
    return __fadd_rn(lam, __fmul_rn(__fsub_rn(1.f, lam), t));
}

template <typename XT>
struct XChunk;

template <>
struct XChunk<__nv_bfloat16> {
    uint4 v;
    ECHO_DEV void load(const __nv_bfloat16 *p) { v = __ldcs(reinterpret_cast<const uint4 *>(p)); }
    ECHO_DEV void get(float *f) const { unpack8_bf16(v, f); }
};

template <>
struct XChunk<float> {
    float4 a, b;
    ECHO_DEV void load(const float *p) {
        a = __ldcs(reinterpret_cast<const float4 *>(p));
        b = __ldcs(reinterpret_cast<const float4 *>(p) + 1);
    }
    ECHO_DEV void get(float *f) const {
        f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
        f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
    }
};

// Where the drift reads the cached feature c_i from (Sec. 3.4 forms):
//   kCacheInt8  c = float(q) * s
//   kCacheBf16  c = the stored bf16 row (full-precision ablation)
//   kCacheRef   c = r + float(q) * s, r the token's reference row (0 if none)
struct CacheView {
    const int8_t *q;
    const float *scale;
    const __nv_bfloat16 *full;
    const int32_t *ref;
    const __nv_bfloat16 *pool;
};
constexpr int kCacheInt8 = 0, kCacheBf16 = 1, kCacheRef = 2;

template <typename XT, int CK>
__global__ void __launch_bounds__(kDriftThreads)
drift_kernel(const XT *__restrict__ x, CacheView cv, const float *__restrict__ seg_energy, int T,
             int N, int NT, int D, float lam, float xi, int mode, float *__restrict__ scores,
             int *err) {
    __shared__ float s_emax;
    if (threadIdx.x < 32) {
        float m = 0.f;
        for (int i = threadIdx.x; i < T; i += 32) m = fmaxf(m, seg_energy[i]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        if (threadIdx.x == 0) s_emax = m;
    }
    __syncthreads();
    const float emax = s_emax;
    const int lane = threadIdx.x & 31;
    const int warps = blockDim.x >> 5;
    const int C = D >> 3;
    for (int row = blockIdx.x * warps + (threadIdx.x >> 5); row < NT; row += gridDim.x * warps) {
        const int seg = row / N;
        const float e = seg_energy[seg];
        float w;
        if (mode == ECHO_MODE_SEGMENT) w = segment_weight(e, emax, 0.f);
        else if (mode == ECHO_MODE_DRIFT_ONLY) w = 1.f;
        else w = segment_weight(e, emax, lam);

        float d = 1.f;
        if (mode != ECHO_MODE_SEGMENT) {
            const float sc = CK == kCacheBf16 ? 0.f : cv.scale[row];
            const XT *xr = x + (int64_t)row * D;
            const int8_t *qr = CK == kCacheBf16 ? nullptr : cv.q + (int64_t)row * D;
            const __nv_bfloat16 *fr = nullptr;
            if constexpr (CK == kCacheBf16) fr = cv.full + (int64_t)row * D;
            if constexpr (CK == kCacheRef) {
                const int rs = cv.ref[row];
                fr = rs >= 0 ? cv.pool + (int64_t)rs * D : nullptr;
            }
            float num = 0.f, den = 0.f;
            for (int c0 = lane; c0 < C; c0 += 32 * kDriftUnroll) {
                XChunk<XT> xv[kDriftUnroll];
                uint2 qv[kDriftUnroll];
                uint4 fv[kDriftUnroll];
#pragma unroll
                for (int u = 0; u < kDriftUnroll; ++u) {
                    const int c = c0 + 32 * u;
                    if (c < C) {
                        xv[u].load(xr + 8 * c);
                        if constexpr (CK != kCacheBf16)
                            qv[u] = __ldcs(reinterpret_cast<const uint2 *>(qr + 8 * c));
                        if constexpr (CK != kCacheInt8)
                            fv[u] = fr ? __ldcs(reinterpret_cast<const uint4 *>(fr + 8 * c))
                                       : make_uint4(0, 0, 0, 0);
                    }
                }
#pragma unroll
                for (int u = 0; u < kDriftUnroll; ++u) {
                    const int c = c0 + 32 * u;
                    if (c < C) {
                        float xf[8], rf[8];
                        xv[u].get(xf);
                        if constexpr (CK != kCacheInt8) unpack8_bf16(fv[u], rf);
                        const int8_t *qb = reinterpret_cast<const int8_t *>(&qv[u]);
                        float cn = 0.f, cd = 0.f;
#pragma unroll
                        for (int k = 0; k < 8; ++k) {
                            float ch;
                            if constexpr (CK == kCacheInt8) ch = __fmul_rn((float)qb[k], sc);
                            else if constexpr (CK == kCacheBf16) ch = rf[k];
                            else ch = __fadd_rn(rf[k], __fmul_rn((float)qb[k], sc));
                            const float an = fabsf(__fsub_rn(xf[k], ch));
                            const float ad = fabsf(ch);
                            cn = k ? __fadd_rn(cn, an) : an;
                            cd = k ? __fadd_rn(cd, ad) : ad;
                        }
                        num = __fadd_rn(num, cn);
                        den = __fadd_rn(den, cd);
                    }
                }
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                num = __fadd_rn(num, __shfl_xor_sync(0xffffffffu, num, o));
                den = __fadd_rn(den, __shfl_xor_sync(0xffffffffu, den, o));
            }
            d = __fdiv_rn(num, __fadd_rn(den, xi));
        }
        const float score = __fmul_rn(w, d);
        if (lane == 0) {
            scores[row] = score;
            if (!isfinite(score)) echo_flag_error(err, ECHO_ERR_NONFINITE);
        }
    }
}

ECHO_DEV uint32_t order_key(float f) {
    const uint32_t b = __float_as_uint(f);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Exclusive block scan of one value per thread (blockDim == kTopkThreads).
// Returns the exclusive prefix; *total gets the block sum.
ECHO_DEV int block_exclusive_scan(int v, int *warp_sums, int *total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += n;
    }
    if (lane == 31) warp_sums[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        int w = warp_sums[lane];
        int wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int n = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += n;
        }
        warp_sums[lane] = wi - w;           // exclusive prefix of warp totals
        if (lane == 31) warp_sums[32] = wi; // block total
    }
    __syncthreads();
    const int r = warp_sums[warp] + inc - v;
    *total = warp_sums[32];
    __syncthreads();
    return r;
}

// Radix digits (bits [sh, sh + log2 nb)) of the n keys whose higher bits
// equal `prefix` under `pmask`, counted into hist (zeroed by the caller).
// keys4(i) returns keys i .. i + 3 (i a multiple of 4; keys at or past n are
// ignored whatever they hold).
template <typename KeyFn>
ECHO_DEV void count_digits(KeyFn keys4, int n, int sh, int nb, uint32_t prefix, uint32_t pmask,
                           int *hist) {
    const int stride4 = blockDim.x * 4;
    for (int b = threadIdx.x * 4; b < n; b += stride4 * 4) {
        uint4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int i = b + u * stride4;
            v[u] = i < n ? keys4(i) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int i = b + u * stride4;
            const uint32_t k[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
            for (int c = 0; c < 4; ++c)
                if (i + c < n && (k[c] & pmask) == prefix)
                    atomicAdd(&hist[(k[c] >> sh) & (nb - 1)], 1);
        }
    }
}

// The digit that holds the krem-th largest counted key, the bins taken from
// the highest down (thread t covers hi = nb-1-2t and hi-1); krem becomes that
// key's rank within its bin.  Every thread returns the same digit.
ECHO_DEV int pick_digit(const int *hist, int nb, int &krem, int *warp_sums, int *s_digit,
                        int *s_krem) {
    const int hi = nb - 1 - 2 * (int)threadIdx.x;
    const int c_hi = hi >= 0 ? hist[hi] : 0;
    const int c_lo = hi - 1 >= 0 ? hist[hi - 1] : 0;
    int total;
    const int above = block_exclusive_scan(c_hi + c_lo, warp_sums, &total);
    if (hi >= 0 && above < krem && above + c_hi >= krem) {
        *s_digit = hi;
        *s_krem = krem - above;
    }
    if (hi - 1 >= 0 && above + c_hi < krem && above + c_hi + c_lo >= krem) {
        *s_digit = hi - 1;
        *s_krem = krem - above - c_hi;
    }
    __syncthreads();
    const int digit = *s_digit;
    krem = *s_krem;
    __syncthreads();
    return digit;
}

// Writes, in index order, the indices (first + i) of the n keys above thr and
// of the keys equal to thr while fewer than need_eq of those have been taken.
// eq_run and sel_run: keys equal to thr and keys taken before key 0 (by
// lower-ranked slices); the first index written goes to idx[sel_run].
template <typename KeyFn>
ECHO_DEV void compact_in_index_order(KeyFn keys4, int n, int first, uint32_t thr, int need_eq,
                                     int eq_run, int sel_run, int32_t *__restrict__ idx,
                                     int *warp_sums) {
    const int tile = kTopkThreads * kTopkItems;
    for (int base = 0; base < n; base += tile) {
        bool gt[kTopkItems], eq[kTopkItems];
        int neq = 0;
        const int i0 = base + (int)threadIdx.x * kTopkItems;
        const uint4 kv4 = i0 < n ? keys4(i0) : make_uint4(0, 0, 0, 0);
        const uint32_t kk[4] = {kv4.x, kv4.y, kv4.z, kv4.w};
#pragma unroll
        for (int j = 0; j < kTopkItems; ++j) {
            const int i = i0 + j;
            gt[j] = eq[j] = false;
            if (i < n) {
                gt[j] = kk[j] > thr;
                eq[j] = kk[j] == thr;
            }
            neq += eq[j];
        }
        int eq_total;
        int eq_before = eq_run + block_exclusive_scan(neq, warp_sums, &eq_total);
        bool sel[kTopkItems];
        int nsel = 0;
#pragma unroll
        for (int j = 0; j < kTopkItems; ++j) {
            sel[j] = gt[j];
            if (eq[j]) {
                sel[j] = eq_before < need_eq;
                ++eq_before;
            }
            nsel += sel[j];
        }
        int sel_total;
        int pos = sel_run + block_exclusive_scan(nsel, warp_sums, &sel_total);
#pragma unroll
        for (int j = 0; j < kTopkItems; ++j)
            if (sel[j]) idx[pos++] = first + i0 + j;
        eq_run += eq_total;
        sel_run += sel_total;
    }
}

__global__ void __launch_bounds__(kTopkThreads)
topk_kernel(const float *__restrict__ scores, int NT, int K, int keys_in_smem,
            int32_t *__restrict__ idx) {
    extern __shared__ uint32_t skeys[];
    __shared__ int hist[2048];
    __shared__ int warp_sums[33];
    __shared__ int s_digit, s_krem;
    const int tid = threadIdx.x;

    if (K >= NT) {
        for (int i = tid; i < NT; i += blockDim.x) idx[i] = i;
        return;
    }
    if (K <= 0) return;

    // keys of elements i .. i + 3 (i a multiple of 4); those at or past NT are
    // 0, below every key of a finite score
    auto gkeys4 = [&](int i) -> uint4 {
        if (i + 3 < NT) {
            const float4 v = __ldg(reinterpret_cast<const float4 *>(scores + i));
            return make_uint4(order_key(v.x), order_key(v.y), order_key(v.z), order_key(v.w));
        }
        uint32_t k[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) k[c] = i + c < NT ? order_key(scores[i + c]) : 0u;
        return make_uint4(k[0], k[1], k[2], k[3]);
    };
    const int stride4 = blockDim.x * 4;
    if (keys_in_smem) {
        // eight 16-byte loads in flight per thread
        for (int b = tid * 4; b < NT; b += stride4 * 8) {
            uint4 v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int i = b + u * stride4;
                if (i < NT) v[u] = gkeys4(i);
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int i = b + u * stride4;
                if (i < NT) *reinterpret_cast<uint4 *>(skeys + i) = v[u];
            }
        }
    }
    __syncthreads();
    auto keys4 = [&](int i) -> uint4 {
        return keys_in_smem ? *reinterpret_cast<const uint4 *>(skeys + i) : gkeys4(i);
    };

    uint32_t prefix = 0, pmask = 0;
    int krem = K;
    const int shifts[3] = {21, 10, 0};
    const int widths[3] = {11, 11, 10};
    for (int pass = 0; pass < 3; ++pass) {
        const int sh = shifts[pass];
        const int nb = 1 << widths[pass];
        for (int b = tid; b < 2048; b += blockDim.x) hist[b] = 0;
        __syncthreads();
        count_digits(keys4, NT, sh, nb, prefix, pmask, hist);
        __syncthreads();
        prefix |= (uint32_t)pick_digit(hist, nb, krem, warp_sums, &s_digit, &s_krem) << sh;
        pmask |= (uint32_t)(nb - 1) << sh;
    }
    // prefix is the K-th largest key; take every larger key and the first
    // `krem` keys equal to it in index order.
    compact_in_index_order(keys4, NT, 0, prefix, krem, 0, 0, idx, warp_sums);
}

constexpr int kTopkClusterCtas = 8;
constexpr int kBinsPerRank = 2048 / kTopkClusterCtas;

// red.add of v into a 32-bit word given by its shared::cluster address
ECHO_DEV void red_add_shared_cluster(uint32_t cluster_addr, int v) {
    asm volatile("red.shared::cluster.add.s32 [%0], %1;" ::"r"(cluster_addr), "r"(v) : "memory");
}

ECHO_DEV int4 ld_shared_cluster_v4(uint32_t cluster_addr) {
    int4 v;
    asm volatile("ld.shared::cluster.v4.s32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(cluster_addr)
                 : "memory");
    return v;
}

// The same selection on a cluster of kTopkClusterCtas CTAs (one per SM), each
// holding one contiguous slice of `slice` keys (a multiple of 4) in shared
// memory.  In every radix pass each CTA counts its slice into a local
// histogram and adds its non-zero bins, through distributed shared memory, to
// the CTA that owns them (CTA r owns bins [256 r, 256 r + 256)); after a
// cluster barrier every CTA reads the summed histogram back from the owners
// with 16-byte loads and takes the same digit.  Each pass sums into its own
// buffer, zeroed before the first barrier, so no buffer is reused.  For the
// compaction each CTA publishes how many of its keys are above and how many
// are equal to the threshold; the counts of the lower-ranked CTAs (lower
// indices) give the slice's first output position and its share of the equal
// keys.
__global__ void __launch_bounds__(kTopkThreads)
topk_cluster_kernel(const float *__restrict__ scores, int NT, int K, int slice,
                    int32_t *__restrict__ idx) {
    extern __shared__ uint4 skeys4[];
    __shared__ __align__(16) int hist[2048];                  // this CTA's counts
    __shared__ __align__(16) int red[3][kBinsPerRank];        // owned bins, one buffer a pass
    __shared__ __align__(16) int full[2048];                  // the cluster's counts
    __shared__ int warp_sums[33];
    __shared__ int s_digit, s_krem;
    __shared__ int s_counts[2];   // keys of this slice above / equal to the threshold
    const int tid = threadIdx.x;
    const int rank = (int)cluster_ctarank();

    if (K >= NT) {
        for (int i = rank * blockDim.x + tid; i < NT; i += kTopkClusterCtas * blockDim.x) idx[i] = i;
        return;
    }
    if (K <= 0) return;
    const int lo = min(rank * slice, NT);
    const int n = min(slice, NT - lo);   // keys of this slice (0 for a CTA past the end)
    const float *src = scores + lo;

    for (int b = tid; b < 3 * kBinsPerRank; b += blockDim.x) (&red[0][0])[b] = 0;
    // stage the slice: eight 16-byte loads in flight per thread
    const int stride4 = blockDim.x * 4;
    for (int b = tid * 4; b < n; b += stride4 * 8) {
        uint4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int i = b + u * stride4;
            if (i + 3 < n) {
                const float4 f = __ldg(reinterpret_cast<const float4 *>(src + i));
                v[u] = make_uint4(order_key(f.x), order_key(f.y), order_key(f.z), order_key(f.w));
            } else if (i < n) {
                uint32_t k[4];
#pragma unroll
                for (int c = 0; c < 4; ++c) k[c] = i + c < n ? order_key(src[i + c]) : 0u;
                v[u] = make_uint4(k[0], k[1], k[2], k[3]);
            }
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int i = b + u * stride4;
            if (i < n) skeys4[i >> 2] = v[u];
        }
    }
    cluster_sync_all();   // every owner's buffers are zero before any CTA adds to them

    auto keys4 = [&](int i) -> uint4 { return skeys4[i >> 2]; };
    uint32_t prefix = 0, pmask = 0;
    int krem = K;
    const int shifts[3] = {21, 10, 0};
    const int widths[3] = {11, 11, 10};
    for (int pass = 0; pass < 3; ++pass) {
        const int sh = shifts[pass];
        const int nb = 1 << widths[pass];
        for (int b = tid; b < 2048; b += blockDim.x) hist[b] = 0;
        __syncthreads();
        count_digits(keys4, n, sh, nb, prefix, pmask, hist);
        __syncthreads();
        for (int b = tid; b < nb; b += blockDim.x) {
            const int v = hist[b];
            if (v)
                red_add_shared_cluster(
                    mapa_shared(smem_u32(&red[pass][b % kBinsPerRank]), (uint32_t)(b / kBinsPerRank)),
                    v);
        }
        cluster_sync_all();   // every CTA's counts of this pass are in the owners' buffers
        if (tid * 4 < nb) {
            const int b0 = tid * 4;
            const int4 v = ld_shared_cluster_v4(
                mapa_shared(smem_u32(&red[pass][b0 % kBinsPerRank]), (uint32_t)(b0 / kBinsPerRank)));
            *reinterpret_cast<int4 *>(&full[b0]) = v;
        }
        __syncthreads();
        prefix |= (uint32_t)pick_digit(full, nb, krem, warp_sums, &s_digit, &s_krem) << sh;
        pmask |= (uint32_t)(nb - 1) << sh;
    }
    const uint32_t thr = prefix;
    const int need_eq = krem;

    // this slice's counts above / equal to the threshold
    int n_gt = 0, n_eq = 0;
    for (int b = tid * 4; b < n; b += stride4) {
        const uint4 v = skeys4[b >> 2];
        const uint32_t k[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int c = 0; c < 4; ++c)
            if (b + c < n) {
                n_gt += k[c] > thr;
                n_eq += k[c] == thr;
            }
    }
    int gt_total, eq_total_slice;
    block_exclusive_scan(n_gt, warp_sums, &gt_total);
    block_exclusive_scan(n_eq, warp_sums, &eq_total_slice);
    if (tid == 0) {
        s_counts[0] = gt_total;
        s_counts[1] = eq_total_slice;
    }
    cluster_sync_all();
    int gt_before = 0, eq_before = 0;
    for (int r = 0; r < rank; ++r) {
        gt_before += ld_shared_cluster_s32(mapa_shared(smem_u32(&s_counts[0]), (uint32_t)r));
        eq_before += ld_shared_cluster_s32(mapa_shared(smem_u32(&s_counts[1]), (uint32_t)r));
    }
    compact_in_index_order(keys4, n, lo, thr, need_eq, eq_before,
                           gt_before + min(eq_before, need_eq), idx, warp_sums);
    cluster_sync_all();   // no CTA leaves while another may still read its counts
}

constexpr int kTopkKeyBytesMax = 200 * 1024;   // keys of one CTA in shared memory
constexpr int kTopkSliceMax = kTopkKeyBytesMax / 4;
constexpr int kTopkClusterMinKeys = 10240;   // below: the one-CTA kernel is faster

// Both top-K kernels may take up to kTopkKeyBytesMax of dynamic shared memory
// (on top of their static buffers, which alone leave less than the default
// 48 KB for it).  The cap is raised once per device, before the first launch
// there, whatever the size of that first launch.
bool topk_smem_cap_raised() {
    static int raised[64] = {};
    static std::mutex mu;
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
    std::lock_guard<std::mutex> lk(mu);
    if (!raised[dev]) {
        if (cudaFuncSetAttribute(topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kTopkKeyBytesMax) != cudaSuccess ||
            cudaFuncSetAttribute(topk_cluster_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kTopkKeyBytesMax) != cudaSuccess)
            return false;
        raised[dev] = 1;
    }
    return true;
}

// top-K of NT keys into idx[0..K): the cluster kernel when every slice fits in
// shared memory, else the one-CTA kernel (keys in shared memory when they fit).
// `keys` is 16-byte aligned.
echo_status launch_topk(const float *keys, int NT, int K, int32_t *idx, cudaStream_t st) {
    using namespace echo;
    if (!topk_smem_cap_raised()) return ECHO_ERR_CUDA;
    const int slice = ((NT + kTopkClusterCtas - 1) / kTopkClusterCtas + 3) & ~3;
    if (NT >= kTopkClusterMinKeys && slice <= kTopkSliceMax) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(kTopkClusterCtas, 1, 1);
        cfg.blockDim = dim3(kTopkThreads, 1, 1);
        cfg.dynamicSmemBytes = (size_t)slice * sizeof(uint32_t);
        cfg.stream = st;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = kTopkClusterCtas;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        LaunchScope ls(ECHO_K_TOPK, NT, K, 0, st);
        if (cudaLaunchKernelEx(&cfg, topk_cluster_kernel, keys, NT, K, slice, idx) != cudaSuccess)
            return ECHO_ERR_CUDA;
        return last_launch_status();
    }
    const size_t key_bytes = (size_t)NT * sizeof(uint32_t);
    const int in_smem = key_bytes <= (size_t)kTopkKeyBytesMax ? 1 : 0;
    LaunchScope ls(ECHO_K_TOPK, NT, K, 0, st);
    topk_kernel<<<1, kTopkThreads, in_smem ? key_bytes : 0, st>>>(keys, NT, K, in_smem, idx);
    return last_launch_status();
}

size_t align256(size_t b) { return (b + 255) & ~(size_t)255; }

// idx[j] = floor(j NT / K): K evenly spaced tokens, ascending and distinct
__global__ void uniform_kernel(int NT, int K, int32_t *__restrict__ idx) {
    for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < K; j += gridDim.x * blockDim.x)
        idx[j] = (int32_t)(((int64_t)j * NT) / K);
}

}  // namespace

extern "C" size_t echo_select_workspace_size(int32_t T, int32_t N) {
    if (T < 1 || N < 1) return 0;
    return align256((size_t)T * N * sizeof(float));
}

extern "C" echo_status echo_select(const void *x, echo_dtype xt, const int8_t *cache_q,
                                   const float *cache_scale, const float *seg_energy, int32_t T,
                                   int32_t N, int32_t D, int32_t ratio_num, int32_t ratio_den,
                                   const echo_select_params *p, int32_t *idx, int32_t *K_out,
                                   float *scores, void *workspace, size_t ws_bytes,
                                   echo_stream_t stream) {
    using namespace echo;
    if (!x || !cache_q || !cache_scale || !seg_energy || !idx || !K_out) return ECHO_ERR_INVALID_ARG;
    if (xt != ECHO_BF16 && xt != ECHO_F32) return ECHO_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(cache_q) || !aligned16(cache_scale) || !aligned16(seg_energy) ||
        !aligned16(idx) || (scores && !aligned16(scores)))
        return ECHO_ERR_INVALID_ARG;
    echo_select_params prm = {0.1f, 1e-6f, ECHO_MODE_ENERGY_DRIFT};
    if (p) prm = *p;
    if (prm.mode < 0 || prm.mode > 2 || !(prm.xi > 0.f) || !(prm.lambda >= 0.f) ||
        !(prm.lambda <= 1.f))
        return ECHO_ERR_INVALID_ARG;
    if (T < 1 || N < 1 || D < 8 || D % 8 || ratio_den < 1 || ratio_num < 0 || ratio_num > ratio_den)
        return ECHO_ERR_SHAPE;
    const int64_t NT64 = (int64_t)T * N;
    if (NT64 > (int64_t)INT32_MAX / 2) return ECHO_ERR_SHAPE;
    const int NT = (int)NT64;
    const int K = (int)(((int64_t)ratio_num * NT + ratio_den - 1) / ratio_den);
    float *sc = scores;
    if (!sc) {
        if (!workspace || !aligned16(workspace)) return ECHO_ERR_INVALID_ARG;
        if (ws_bytes < echo_select_workspace_size(T, N)) return ECHO_ERR_WORKSPACE;
        sc = static_cast<float *>(workspace);
    }
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    *K_out = K;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    int *err = device_error_ptr();

    const int warps = kDriftThreads / 32;
    int grid = (NT + warps - 1) / warps;
    {
    LaunchScope ls(ECHO_K_DRIFT, NT, D, 0, st);
    if (xt == ECHO_BF16)
        drift_kernel<__nv_bfloat16, kCacheInt8><<<grid, kDriftThreads, 0, st>>>(
            static_cast<const __nv_bfloat16 *>(x), CacheView{cache_q, cache_scale, nullptr, nullptr,
            nullptr}, seg_energy, T, N, NT, D, prm.lambda, prm.xi, prm.mode, sc, err);
    else
        drift_kernel<float, kCacheInt8><<<grid, kDriftThreads, 0, st>>>(
            static_cast<const float *>(x), CacheView{cache_q, cache_scale, nullptr, nullptr,
            nullptr}, seg_energy, T, N, NT, D, prm.lambda, prm.xi, prm.mode, sc, err);
    }
    if (last_launch_status() != ECHO_OK) return ECHO_ERR_CUDA;

    return launch_topk(sc, NT, K, idx, st);
}

// ---------------------------------------------------------------------------
// echo_select_static: the same selection for callers that cannot allocate.
// The scores live in this file-scope device array instead of a workspace.
// Host code must not pass `g_select_scratch` itself to a kernel (on the host
// it is only a stand-in symbol); the device address is looked up once per
// device with cudaGetSymbolAddress and cached.
// ---------------------------------------------------------------------------
static __device__ __align__(256) float g_select_scratch[ECHO_SELECT_STATIC_MAX_TOKENS];

namespace {

constexpr int kScratchDevices = 64;
float *g_scratch_ptr[kScratchDevices] = {};
std::mutex g_scratch_mu;

// Address of this device's scratch array (the current device), or nullptr.
float *select_scratch_for_current_device() {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kScratchDevices) return nullptr;
    std::lock_guard<std::mutex> lk(g_scratch_mu);
    if (!g_scratch_ptr[dev]) {
        float *ptr = nullptr;
        if (cudaGetSymbolAddress(reinterpret_cast<void **>(&ptr), g_select_scratch) != cudaSuccess ||
            !ptr)
            return nullptr;
        g_scratch_ptr[dev] = ptr;
    }
    return g_scratch_ptr[dev];
}

}  // namespace

extern "C" echo_status echo_select_static(const void *x, echo_dtype xt, const int8_t *cache_q,
                                          const float *cache_scale, const float *seg_energy,
                                          int32_t T, int32_t N, int32_t D, int32_t ratio_num,
                                          int32_t ratio_den, const echo_select_params *p,
                                          int32_t *idx, int32_t *K_out, echo_stream_t stream) {
    using namespace echo;
    if (!x || !cache_q || !cache_scale || !seg_energy || !idx || !K_out) return ECHO_ERR_INVALID_ARG;
    if (xt != ECHO_BF16 && xt != ECHO_F32) return ECHO_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(cache_q) || !aligned16(cache_scale) || !aligned16(seg_energy) ||
        !aligned16(idx))
        return ECHO_ERR_INVALID_ARG;
    echo_select_params prm = {0.1f, 1e-6f, ECHO_MODE_ENERGY_DRIFT};
    if (p) prm = *p;
    if (prm.mode < 0 || prm.mode > 2 || !(prm.xi > 0.f) || !(prm.lambda >= 0.f) ||
        !(prm.lambda <= 1.f))
        return ECHO_ERR_INVALID_ARG;
    if (T < 1 || N < 1 || D < 8 || D % 8 || ratio_den < 1 || ratio_num < 0 || ratio_num > ratio_den)
        return ECHO_ERR_SHAPE;
    const int64_t NT64 = (int64_t)T * N;
    if (NT64 > ECHO_SELECT_STATIC_MAX_TOKENS) return ECHO_ERR_WORKSPACE;
    const int NT = (int)NT64;
    const int K = (int)(((int64_t)ratio_num * NT + ratio_den - 1) / ratio_den);
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    float *sc = select_scratch_for_current_device();
    if (!sc) return ECHO_ERR_CUDA;
    *K_out = K;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    int *err = device_error_ptr();

    const int warps = kDriftThreads / 32;
    const int grid = (NT + warps - 1) / warps;
    {
        LaunchScope ls(ECHO_K_DRIFT, NT, D, 0, st);
        if (xt == ECHO_BF16)
            drift_kernel<__nv_bfloat16, kCacheInt8><<<grid, kDriftThreads, 0, st>>>(
                static_cast<const __nv_bfloat16 *>(x), CacheView{cache_q, cache_scale, nullptr,
                nullptr, nullptr}, seg_energy, T, N, NT, D, prm.lambda, prm.xi, prm.mode, sc, err);
        else
            drift_kernel<float, kCacheInt8><<<grid, kDriftThreads, 0, st>>>(
                static_cast<const float *>(x), CacheView{cache_q, cache_scale, nullptr, nullptr,
                nullptr}, seg_energy, T, N, NT, D, prm.lambda, prm.xi, prm.mode, sc, err);
    }
    if (last_launch_status() != ECHO_OK) return ECHO_ERR_CUDA;
    return launch_topk(sc, NT, K, idx, st);
}

namespace {

// shared argument checks of the ablation selections; returns K or -1
int ablation_budget(int32_t T, int32_t N, int32_t ratio_num, int32_t ratio_den) {
    if (T < 1 || N < 1 || ratio_den < 1 || ratio_num < 0 || ratio_num > ratio_den) return -1;
    const int64_t NT64 = (int64_t)T * N;
    if (NT64 > (int64_t)INT32_MAX / 2) return -1;
    return (int)(((int64_t)ratio_num * NT64 + ratio_den - 1) / ratio_den);
}

}  // namespace

extern "C" echo_status echo_select_uniform(int32_t T, int32_t N, int32_t ratio_num,
                                           int32_t ratio_den, int32_t *idx, int32_t *K_out,
                                           echo_stream_t stream) {
    using namespace echo;
    if (!idx || !K_out || !aligned16(idx)) return ECHO_ERR_INVALID_ARG;
    const int K = ablation_budget(T, N, ratio_num, ratio_den);
    if (K < 0) return ECHO_ERR_SHAPE;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    *K_out = K;
    if (K == 0) return ECHO_OK;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const int grid = (K + 255) / 256;
    {
        LaunchScope ls(ECHO_K_UNIFORM, T * N, K, 0, st);
        uniform_kernel<<<grid, 256, 0, st>>>(T * N, K, idx);
    }
    return last_launch_status();
}

extern "C" echo_status echo_select_random(const float *keys, int32_t T, int32_t N,
                                          int32_t ratio_num, int32_t ratio_den, int32_t *idx,
                                          int32_t *K_out, echo_stream_t stream) {
    using namespace echo;
    if (!keys || !idx || !K_out || !aligned16(keys) || !aligned16(idx)) return ECHO_ERR_INVALID_ARG;
    const int K = ablation_budget(T, N, ratio_num, ratio_den);
    if (K < 0) return ECHO_ERR_SHAPE;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    *K_out = K;
    const int NT = T * N;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    return launch_topk(keys, NT, K, idx, st);
}

extern "C" echo_status echo_select_cache(const void *x, echo_dtype xt, const echo_cache *c,
                                         const float *seg_energy, int32_t T, int32_t N,
                                         int32_t ratio_num, int32_t ratio_den,
                                         const echo_select_params *p, int32_t *idx,
                                         int32_t *K_out, float *scores, void *workspace,
                                         size_t ws_bytes, echo_stream_t stream) {
    using namespace echo;
    const echo_status v = cache_check(c);
    if (v != ECHO_OK) return v;
    if (c->kind == ECHO_CACHE_INT8)
        return echo_select(x, xt, c->q, c->scale, seg_energy, T, N, c->D, ratio_num, ratio_den, p,
                           idx, K_out, scores, workspace, ws_bytes, stream);
    if (!x || !seg_energy || !idx || !K_out) return ECHO_ERR_INVALID_ARG;
    if (xt != ECHO_BF16 && xt != ECHO_F32) return ECHO_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(seg_energy) || !aligned16(idx) || (scores && !aligned16(scores)))
        return ECHO_ERR_INVALID_ARG;
    echo_select_params prm = {0.1f, 1e-6f, ECHO_MODE_ENERGY_DRIFT};
    if (p) prm = *p;
    if (prm.mode < 0 || prm.mode > 2 || !(prm.xi > 0.f) || !(prm.lambda >= 0.f) ||
        !(prm.lambda <= 1.f))
        return ECHO_ERR_INVALID_ARG;
    if (T < 1 || N < 1 || ratio_den < 1 || ratio_num < 0 || ratio_num > ratio_den)
        return ECHO_ERR_SHAPE;
    if ((int64_t)T * N != c->NT) return ECHO_ERR_SHAPE;
    const int NT = c->NT, D = c->D;
    const int K = (int)(((int64_t)ratio_num * NT + ratio_den - 1) / ratio_den);
    float *sc = scores;
    if (!sc) {
        if (!workspace || !aligned16(workspace)) return ECHO_ERR_INVALID_ARG;
        if (ws_bytes < echo_select_workspace_size(T, N)) return ECHO_ERR_WORKSPACE;
        sc = static_cast<float *>(workspace);
    }
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    *K_out = K;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    int *err = device_error_ptr();
    const CacheView cv{c->q, c->scale, static_cast<const __nv_bfloat16 *>(c->full), c->ref,
                       static_cast<const __nv_bfloat16 *>(c->pool)};
    const int warps = kDriftThreads / 32;
    const int grid = (NT + warps - 1) / warps;
    {
        LaunchScope ls(ECHO_K_DRIFT, NT, D, 0, st);
        const bool bf = xt == ECHO_BF16;
        const __nv_bfloat16 *xb = static_cast<const __nv_bfloat16 *>(x);
        const float *xf = static_cast<const float *>(x);
        if (c->kind == ECHO_CACHE_BF16) {
            if (bf)
                drift_kernel<__nv_bfloat16, kCacheBf16><<<grid, kDriftThreads, 0, st>>>(
                    xb, cv, seg_energy, T, N, NT, D, prm.lambda, prm.xi, prm.mode, sc, err);
            else
                drift_kernel<float, kCacheBf16><<<grid, kDriftThreads, 0, st>>>(
                    xf, cv, seg_energy, T, N, NT, D, prm.lambda, prm.xi, prm.mode, sc, err);
        } else {
            if (bf)
                drift_kernel<__nv_bfloat16, kCacheRef><<<grid, kDriftThreads, 0, st>>>(
                    xb, cv, seg_energy, T, N, NT, D, prm.lambda, prm.xi, prm.mode, sc, err);
            else
                drift_kernel<float, kCacheRef><<<grid, kDriftThreads, 0, st>>>(
                    xf, cv, seg_energy, T, N, NT, D, prm.lambda, prm.xi, prm.mode, sc, err);
        }
    }
    if (last_launch_status() != ECHO_OK) return ECHO_ERR_CUDA;
    return launch_topk(sc, NT, K, idx, st);
}
