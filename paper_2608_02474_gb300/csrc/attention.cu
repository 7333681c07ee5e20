// Multi-head attention on (Q', K, V) (Sec. 3.3): queries only for the active
// latents, keys and values over the complete latent set (self-attention) or the
// audio condition tokens (cross-attention).
//
// Flash-style forward on the 5th-generation tensor cores.  One CTA per
// (128-query tile, head), 8 warps:
//   warp 0      TMA producer: the Q tile once, then 128-key blocks of K and V
//               (128-byte swizzle, 64-column boxes) into two-stage rings;
//   warp 1      one thread issues S_j = Q K_j^T (M 128, N 128, K d) into one of
//               two TMEM S buffers, and O += P_j V_j (M 128, N d, K 128; V is
//               read MN-major straight from its row-major tile) into a TMEM O
//               accumulator, one block behind;
//   warp 2      allocates / frees 512 TMEM columns (S0, S1, O);
//   warps 4..7  softmax, one query row per thread (its TMEM lane): tcgen05.ld of
//               the S row, online max, P = 2^(s*scale - m) rounded to bf16 into a
//               swizzled shared-memory tile (the A operand of P V), row sum of the
//               rounded P; O is rescaled in TMEM only when the running max grows
//               by more than 2^8 (otherwise the stale max is kept, which is exact
//               after the final division by the row sum); final O / l to bf16.
// Keys beyond L are masked to P = 0; queries beyond M run on zero rows and are
// not stored.  Every mbarrier wait is bounded (ECHO_ERR_TIMEOUT).
#include "common.cuh"
#include "internal.h"

namespace {

constexpr int BM = 128;        // queries per CTA
constexpr int BN = 128;        // keys per block
constexpr int KST = 2;         // K ring stages
constexpr int VST = 2;         // V ring stages
constexpr int THREADS = 256;
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t O_COL = 256;
constexpr int ATOM_BYTES = 128 * 128;   // one [128 rows x 64 bf16] 128B-swizzled box
constexpr float RESCALE_LOG2 = 8.f;

template <int DH>
struct Cfg {
    static constexpr int ATOMS = DH / 64;
    static constexpr int Q_BYTES = BM * DH * 2;
    static constexpr int K_BYTES = BN * DH * 2;
    static constexpr int V_BYTES = BN * DH * 2;
    static constexpr int P_BYTES = BM * BN * 2;
    static constexpr int SMEM = Q_BYTES + KST * K_BYTES + VST * V_BYTES + P_BYTES + 1024;
    static constexpr uint32_t IDESC_S = idesc_bf16_f32(BM, BN);
    static constexpr uint32_t IDESC_PV = idesc_bf16_f32(BM, DH) | (1u << 16);  // B MN-major
};

struct AttnParams {
    int M, L;
    float scale_log2;
    __nv_bfloat16 *O;
    int64_t ldo;
    int *err;
};

template <int DH>
__global__ void __launch_bounds__(THREADS, 1)
attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
               const __grid_constant__ CUtensorMap tmV, const AttnParams p) {
    using C = Cfg<DH>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    uint8_t *Qs = smem;
    uint8_t *Ks = Qs + C::Q_BYTES;
    uint8_t *Vs = Ks + KST * C::K_BYTES;
    uint8_t *Ps = Vs + VST * C::V_BYTES;

    __shared__ __align__(8) uint64_t q_full, k_full[KST], k_empty[KST], v_full[VST], v_empty[VST];
    __shared__ __align__(8) uint64_t s_full[2], s_free[2], p_full, pv_done, drain;
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_flag;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int h = blockIdx.y;
    const int q0 = blockIdx.x * BM;
    const int nb = (p.L + BN - 1) / BN;

    if (threadIdx.x == 0) {
        mbar_init(&q_full, 1);
        for (int i = 0; i < KST; ++i) { mbar_init(&k_full[i], 1); mbar_init(&k_empty[i], 1); }
        for (int i = 0; i < VST; ++i) { mbar_init(&v_full[i], 1); mbar_init(&v_empty[i], 1); }
        for (int i = 0; i < 2; ++i) { mbar_init(&s_full[i], 1); mbar_init(&s_free[i], 128); }
        mbar_init(&p_full, 128);
        mbar_init(&pv_done, 1);
        mbar_init(&drain, 1);
        abort_flag = 0;
        fence_barrier_init();
        tma_prefetch_desc(&tmQ);
        tma_prefetch_desc(&tmK);
        tma_prefetch_desc(&tmV);
    }
    if (warp == 2) tmem_alloc(&tmem_slot, TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    volatile int *abort_v = &abort_flag;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer ----------------
        const int x0 = h * DH;
        mbar_arrive_expect_tx(&q_full, C::Q_BYTES);
        for (int a = 0; a < C::ATOMS; ++a) tma_load_2d(Qs + a * ATOM_BYTES, &tmQ, &q_full, x0 + 64 * a, q0);
        int k_issued = 0, v_issued = 0;
        for (int j = 0; j < nb; ++j) {
            const int ks = j % KST;
            if (!mbar_wait(&k_empty[ks], ((j / KST) & 1) ^ 1, abort_v, p.err)) break;
            mbar_arrive_expect_tx(&k_full[ks], C::K_BYTES);
            for (int a = 0; a < C::ATOMS; ++a)
                tma_load_2d(Ks + ks * C::K_BYTES + a * ATOM_BYTES, &tmK, &k_full[ks], x0 + 64 * a, j * BN);
            k_issued = j + 1;
            const int vs = j % VST;
            if (!mbar_wait(&v_empty[vs], ((j / VST) & 1) ^ 1, abort_v, p.err)) break;
            mbar_arrive_expect_tx(&v_full[vs], C::V_BYTES);
            for (int a = 0; a < C::ATOMS; ++a)
                tma_load_2d(Vs + vs * C::V_BYTES + a * ATOM_BYTES, &tmV, &v_full[vs], x0 + 64 * a, j * BN);
            v_issued = j + 1;
        }
        if (*abort_v) {  // let this CTA's copies land before it exits
            mbar_wait(&q_full, 0, abort_v, nullptr, 100000000ull);
            for (int j = k_issued - KST < 0 ? 0 : k_issued - KST; j < k_issued; ++j)
                mbar_wait(&k_full[j % KST], (j / KST) & 1, abort_v, nullptr, 100000000ull);
            for (int j = v_issued - VST < 0 ? 0 : v_issued - VST; j < v_issued; ++j)
                mbar_wait(&v_full[j % VST], (j / VST) & 1, abort_v, nullptr, 100000000ull);
        }
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer ----------------
        bool ok = mbar_wait(&q_full, 0, abort_v, p.err);
        for (int j = 0; ok && j <= nb; ++j) {
            if (j < nb) {
                const int b = j & 1;
                if (j >= 2 && !mbar_wait(&s_free[b], ((j >> 1) - 1) & 1, abort_v, p.err)) { ok = false; break; }
                const int ks = j % KST;
                if (!mbar_wait(&k_full[ks], (j / KST) & 1, abort_v, p.err)) { ok = false; break; }
                tc_fence_after();
                const uint8_t *kt = Ks + ks * C::K_BYTES;
#pragma unroll
                for (int kk = 0; kk < DH / 16; ++kk) {
                    const int a = kk >> 2, off = (kk & 3) * 32;
                    tc_mma_f16(tmem + (uint32_t)(b * BN), smem_desc_sw128(Qs + a * ATOM_BYTES + off),
                               smem_desc_sw128(kt + a * ATOM_BYTES + off), C::IDESC_S, kk > 0);
                }
                tc_commit(&s_full[b]);
                tc_commit(&k_empty[ks]);
            }
            if (j >= 1) {
                const int jj = j - 1;
                if (!mbar_wait(&p_full, jj & 1, abort_v, p.err)) { ok = false; break; }
                const int vs = jj % VST;
                if (!mbar_wait(&v_full[vs], (jj / VST) & 1, abort_v, p.err)) { ok = false; break; }
                tc_fence_after();
                const uint8_t *vt = Vs + vs * C::V_BYTES;
#pragma unroll
                for (int kk = 0; kk < BN / 16; ++kk) {
                    const int a = kk >> 2, off = (kk & 3) * 32;
                    tc_mma_f16(tmem + O_COL, smem_desc_sw128(Ps + a * ATOM_BYTES + off),
                               smem_desc_sw128_mn(vt + kk * 2048, ATOM_BYTES, 1024), C::IDESC_PV,
                               (jj > 0 || kk > 0) ? 1u : 0u);
                }
                tc_commit(&pv_done);
                tc_commit(&v_empty[vs]);
            }
        }
        if (!ok) {  // wait for the MMAs already issued before tensor memory is freed
            tc_commit(&drain);
            mbar_wait(&drain, 0, abort_v, nullptr, 100000000ull);
        }
    } else if (warp >= 4) {
        // ---------------- softmax / correction / epilogue ----------------
        const int r = (warp - 4) * 32 + lane;          // row of the tile = TMEM lane
        const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
        const float sl2 = p.scale_log2;
        float m_used = -INFINITY, l = 0.f;
        bool ok = true;
        uint8_t *prow = Ps + r * 128;
        const int sw = r & 7;
        for (int j = 0; j < nb; ++j) {
            const int b = j & 1;
            ok = __all_sync(0xffffffffu, mbar_wait(&s_full[b], (j >> 1) & 1, abort_v, p.err));
            if (!ok) break;
            tc_fence_after();
            uint32_t sraw[BN];
#pragma unroll
            for (int c = 0; c < BN / 32; ++c)
                tmem_ld32(tmem + lane_base + (uint32_t)(b * BN + 32 * c), sraw + 32 * c);
            tmem_ld_wait();
            float s[BN];
#pragma unroll
            for (int i = 0; i < BN; ++i) s[i] = __uint_as_float(sraw[i]);
            tc_fence_before();
            mbar_arrive(&s_free[b]);
            const int kvalid = p.L - j * BN;                 // keys of this block that exist
            if (kvalid < BN) {
#pragma unroll
                for (int i = 0; i < BN; ++i)
                    if (i >= kvalid) s[i] = -INFINITY;
            }
            float mx = s[0];
#pragma unroll
            for (int i = 1; i < BN; ++i) mx = fmaxf(mx, s[i]);
            const float m_new = fmaxf(m_used, mx * sl2);
            const bool need = m_new > m_used + RESCALE_LOG2;
            float alpha = 1.f;
            if (need) {
                alpha = ex2_approx(m_used - m_new);
                l *= alpha;
                m_used = m_new;
            }
            const bool warp_rescale = __any_sync(0xffffffffu, need) && j > 0;
            uint32_t pk[BN / 2];
            float rs = 0.f;
#pragma unroll
            for (int i = 0; i < BN / 2; ++i) {
                const float p0 = ex2_approx(fmaf(s[2 * i], sl2, -m_used));
                const float p1 = ex2_approx(fmaf(s[2 * i + 1], sl2, -m_used));
                pk[i] = pack_bf16(p0, p1);
                rs += bf16lo(pk[i]) + bf16hi(pk[i]);
            }
            l += rs;
            if (j >= 1) {   // P_{j-1} and O are in use by P V_{j-1} until it completes
                ok = __all_sync(0xffffffffu, mbar_wait(&pv_done, (j - 1) & 1, abort_v, p.err));
                if (!ok) break;
                tc_fence_after();
            }
#pragma unroll
            for (int a = 0; a < 2; ++a)
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    const uint32_t *src = pk + a * 32 + c * 4;
                    *reinterpret_cast<uint4 *>(prow + a * ATOM_BYTES + ((c ^ sw) << 4)) =
                        make_uint4(src[0], src[1], src[2], src[3]);
                }
            if (warp_rescale) {
#pragma unroll
                for (int c = 0; c < DH / 32; ++c) {
                    uint32_t o[32];
                    tmem_ld32(tmem + lane_base + O_COL + 32 * c, o);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
                    tmem_st32(tmem + lane_base + O_COL + 32 * c, o);
                }
                tmem_st_wait();
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(&p_full);
        }
        if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&pv_done, (nb - 1) & 1, abort_v, p.err));
        if (ok) {
            tc_fence_after();
            const int row = q0 + r;
            const float inv = 1.f / l;
            __nv_bfloat16 *dst = p.O + (int64_t)row * p.ldo + h * DH;
#pragma unroll
            for (int c = 0; c < DH / 32; ++c) {
                uint32_t o[32];
                tmem_ld32(tmem + lane_base + O_COL + 32 * c, o);
                tmem_ld_wait();
                if (row < p.M) {
                    float f[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) f[i] = __uint_as_float(o[i]) * inv;
                    uint4 *op = reinterpret_cast<uint4 *>(dst + 32 * c);
#pragma unroll
                    for (int i = 0; i < 4; ++i) op[i] = pack8_bf16(f + 8 * i);
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 2) {
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
    }
}

template <int DH>
echo_status launch_dh(const void *Q, int64_t ldq, const void *K, const void *V, int64_t ldkv, int M,
                      int L, int H, void *O, int64_t ldo, cudaStream_t st) {
    static int attr_done[64] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_done[dev]) {
        cudaFuncSetAttribute(attn_tc_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             Cfg<DH>::SMEM);
        attr_done[dev] = 1;
    }
    CUtensorMap tq, tk, tv;
    const uint64_t cols = (uint64_t)H * DH;
    if (!echo::make_tmap_bf16(&tq, Q, (uint64_t)M, cols, (uint64_t)ldq, BM) ||
        !echo::make_tmap_bf16(&tk, K, (uint64_t)L, cols, (uint64_t)ldkv, BN) ||
        !echo::make_tmap_bf16(&tv, V, (uint64_t)L, cols, (uint64_t)ldkv, BN))
        return ECHO_ERR_CUDA;
    AttnParams p;
    p.M = M;
    p.L = L;
    p.scale_log2 = 1.4426950408889634f / sqrtf((float)DH);
    p.O = static_cast<__nv_bfloat16 *>(O);
    p.ldo = ldo;
    p.err = echo::device_error_ptr();
    dim3 grid((M + BM - 1) / BM, H);
    echo::LaunchScope ls(ECHO_K_ATTENTION, M, L, (int64_t)H * DH, st);
    attn_tc_kernel<DH><<<grid, THREADS, Cfg<DH>::SMEM, st>>>(tq, tk, tv, p);
    return echo::last_launch_status();
}

}  // namespace

namespace echo {

echo_status launch_attention(const void *Q, int64_t ldq, const void *K, const void *V, int64_t ldkv,
                             int32_t M, int32_t L, int32_t H, int32_t d, void *O, int64_t ldo,
                             cudaStream_t st) {
    if (M <= 0) return ECHO_OK;
    if (d == 64) return launch_dh<64>(Q, ldq, K, V, ldkv, M, L, H, O, ldo, st);
    return launch_dh<128>(Q, ldq, K, V, ldkv, M, L, H, O, ldo, st);
}

}  // namespace echo

extern "C" echo_status echo_attention(const void *Q, int64_t ldq, const void *K, const void *V,
                                      int64_t ldkv, int32_t M, int32_t L, int32_t H, int32_t d,
                                      void *O, int64_t ldo, echo_stream_t stream) {
    using namespace echo;
    if (M < 0 || L < 1 || H < 1 || (d != 64 && d != 128)) return ECHO_ERR_SHAPE;
    if (ldq < (int64_t)H * d || ldkv < (int64_t)H * d || ldo < (int64_t)H * d || ldq % 8 ||
        ldkv % 8 || ldo % 8)
        return ECHO_ERR_SHAPE;
    if (M == 0) return ECHO_OK;
    if (!Q || !K || !V || !O) return ECHO_ERR_INVALID_ARG;
    if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O)) return ECHO_ERR_INVALID_ARG;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    return launch_attention(Q, ldq, K, V, ldkv, M, L, H, d, O, ldo,
                            reinterpret_cast<cudaStream_t>(stream));
}
