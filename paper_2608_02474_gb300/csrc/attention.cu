// Multi-head attention on (Q', K, V) (Sec. 3.3): queries only for the active
// latents, keys and values over the complete latent set (self-attention) or the
// audio condition tokens (cross-attention).
//
// Flash-style forward: one CTA per (128-query tile, head), 8 warps of 16 query
// rows; K/V blocks of 64 keys double-buffered in swizzled shared memory by
// cp.async; S = Q K^T and O += P V on bf16 mma.sync with fp32 accumulators;
// online softmax in registers (exp2 with the 1/sqrt(d) scale folded in); P is
// rounded to bf16 for the second product.  Keys beyond L are masked, queries
// beyond M are computed on zeros and not stored.
#include "common.cuh"
#include "internal.h"

namespace {

constexpr int BR = 128;       // queries per CTA
constexpr int BC = 64;        // keys per block
constexpr int THREADS = 256;  // 8 warps x 16 query rows

ECHO_DEV void cp_async16(void *dst, const void *src, bool valid) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src),
                 "r"(valid ? 16 : 0)
                 : "memory");
}
ECHO_DEV void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
ECHO_DEV void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

ECHO_DEV void ldsm_x4(uint32_t *r, const void *p) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(smem_u32(p)));
}
ECHO_DEV void ldsm_x4_t(uint32_t *r, const void *p) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(smem_u32(p)));
}
ECHO_DEV void mma_bf16(float *c, const uint32_t *a, uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// byte offset of (row, 16-byte chunk) in a tile with rows of DH bf16, chunk
// index xor-swizzled by the row's low 3 bits
template <int DH>
ECHO_DEV uint32_t sw(int row, int chunk) {
    return (uint32_t)(row * (DH * 2) + ((chunk ^ (row & 7)) << 4));
}

template <int DH>
ECHO_DEV void load_rows(uint8_t *tile, const __nv_bfloat16 *base, int64_t ld, int row0, int nrows,
                        int limit) {
    constexpr int CPR = DH / 8;  // 16-byte chunks per row
    for (int i = threadIdx.x; i < nrows * CPR; i += THREADS) {
        const int r = i / CPR, c = i % CPR;
        const int g = row0 + r;
        const bool ok = g < limit;
        const __nv_bfloat16 *src = base + (int64_t)(ok ? g : 0) * ld + c * 8;
        cp_async16(tile + sw<DH>(r, c), src, ok);
    }
}

template <int DH>
__global__ void __launch_bounds__(THREADS)
attn_kernel(const __nv_bfloat16 *__restrict__ Q, int64_t ldq, const __nv_bfloat16 *__restrict__ K,
            const __nv_bfloat16 *__restrict__ V, int64_t ldkv, int M, int L,
            __nv_bfloat16 *__restrict__ O, int64_t ldo, float scale_log2) {
    extern __shared__ __align__(128) uint8_t sm[];
    uint8_t *Qs = sm;
    uint8_t *Ks = Qs + BR * DH * 2;           // [2][BC][DH]
    uint8_t *Vs = Ks + 2 * BC * DH * 2;       // [2][BC][DH]
    constexpr int KV_TILE = BC * DH * 2;

    const int h = blockIdx.y;
    const int q0 = blockIdx.x * BR;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const __nv_bfloat16 *Qh = Q + h * DH;
    const __nv_bfloat16 *Kh = K + h * DH;
    const __nv_bfloat16 *Vh = V + h * DH;
    const int nkb = (L + BC - 1) / BC;

    load_rows<DH>(Qs, Qh, ldq, q0, BR, M);
    load_rows<DH>(Ks, Kh, ldkv, 0, BC, L);
    load_rows<DH>(Vs, Vh, ldkv, 0, BC, L);
    cp_async_commit();
    cp_async_wait_all();
    __syncthreads();

    // Q fragments of this warp's 16 rows, all DH columns
    uint32_t qf[DH / 16][4];
    {
        const int r = warp * 16 + (lane & 7) + 8 * ((lane >> 3) & 1);
#pragma unroll
        for (int ks = 0; ks < DH / 16; ++ks) {
            const int c = ks * 2 + (lane >> 4);
            ldsm_x4(qf[ks], Qs + sw<DH>(r, c));
        }
    }

    float o[DH / 8][4];
#pragma unroll
    for (int i = 0; i < DH / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
    float m_r[2] = {-INFINITY, -INFINITY}, l_r[2] = {0.f, 0.f};

    for (int kb = 0; kb < nkb; ++kb) {
        const int buf = kb & 1;
        if (kb + 1 < nkb) {
            load_rows<DH>(Ks + (buf ^ 1) * KV_TILE, Kh, ldkv, (kb + 1) * BC, BC, L);
            load_rows<DH>(Vs + (buf ^ 1) * KV_TILE, Vh, ldkv, (kb + 1) * BC, BC, L);
        }
        cp_async_commit();
        const uint8_t *Kt = Ks + buf * KV_TILE;
        const uint8_t *Vt = Vs + buf * KV_TILE;

        float s[BC / 8][4];
#pragma unroll
        for (int nt = 0; nt < BC / 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
        for (int np = 0; np < BC / 16; ++np) {        // pairs of 8-key tiles
            const int kr = np * 16 + (lane & 7) + 8 * (lane >> 4);
#pragma unroll
            for (int ks = 0; ks < DH / 16; ++ks) {
                uint32_t b[4];
                ldsm_x4(b, Kt + sw<DH>(kr, ks * 2 + ((lane >> 3) & 1)));
                mma_bf16(s[2 * np], qf[ks], b[0], b[1]);
                mma_bf16(s[2 * np + 1], qf[ks], b[2], b[3]);
            }
        }
        const int key0 = kb * BC;
        if (key0 + BC > L) {
#pragma unroll
            for (int nt = 0; nt < BC / 8; ++nt) {
                const int j = key0 + nt * 8 + 2 * (lane & 3);
                if (j >= L) s[nt][0] = s[nt][2] = -INFINITY;
                if (j + 1 >= L) s[nt][1] = s[nt][3] = -INFINITY;
            }
        }
        // online softmax over the two rows this thread holds (g and g + 8)
#pragma unroll
        for (int hr = 0; hr < 2; ++hr) {
            float mx = -INFINITY;
#pragma unroll
            for (int nt = 0; nt < BC / 8; ++nt)
                mx = fmaxf(mx, fmaxf(s[nt][2 * hr], s[nt][2 * hr + 1]));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
            const float m_new = fmaxf(m_r[hr], mx * scale_log2);
            const float alpha = exp2f(m_r[hr] - m_new);
            float rs = 0.f;
#pragma unroll
            for (int nt = 0; nt < BC / 8; ++nt) {
                const float p0 = exp2f(s[nt][2 * hr] * scale_log2 - m_new);
                const float p1 = exp2f(s[nt][2 * hr + 1] * scale_log2 - m_new);
                s[nt][2 * hr] = p0;
                s[nt][2 * hr + 1] = p1;
                rs += p0 + p1;
            }
            rs += __shfl_xor_sync(0xffffffffu, rs, 1);
            rs += __shfl_xor_sync(0xffffffffu, rs, 2);
            l_r[hr] = l_r[hr] * alpha + rs;
            m_r[hr] = m_new;
#pragma unroll
            for (int dt = 0; dt < DH / 8; ++dt) {
                o[dt][2 * hr] *= alpha;
                o[dt][2 * hr + 1] *= alpha;
            }
        }
        // O += P V
#pragma unroll
        for (int ks = 0; ks < BC / 16; ++ks) {
            uint32_t a[4];
            a[0] = pack_bf16(s[2 * ks][0], s[2 * ks][1]);
            a[1] = pack_bf16(s[2 * ks][2], s[2 * ks][3]);
            a[2] = pack_bf16(s[2 * ks + 1][0], s[2 * ks + 1][1]);
            a[3] = pack_bf16(s[2 * ks + 1][2], s[2 * ks + 1][3]);
            const int vr = ks * 16 + (lane & 7) + 8 * ((lane >> 3) & 1);
#pragma unroll
            for (int dp = 0; dp < DH / 16; ++dp) {
                uint32_t b[4];
                ldsm_x4_t(b, Vt + sw<DH>(vr, dp * 2 + (lane >> 4)));
                mma_bf16(o[2 * dp], a, b[0], b[1]);
                mma_bf16(o[2 * dp + 1], a, b[2], b[3]);
            }
        }
        cp_async_wait_all();
        __syncthreads();
    }

    // normalise and store
    const int g = lane >> 2, t = lane & 3;
#pragma unroll
    for (int hr = 0; hr < 2; ++hr) {
        const int row = q0 + warp * 16 + g + 8 * hr;
        if (row >= M) continue;
        const float inv = 1.f / l_r[hr];
        __nv_bfloat16 *dst = O + (int64_t)row * ldo + h * DH;
#pragma unroll
        for (int dt = 0; dt < DH / 8; ++dt) {
            const uint32_t v = pack_bf16(o[dt][2 * hr] * inv, o[dt][2 * hr + 1] * inv);
            *reinterpret_cast<uint32_t *>(dst + dt * 8 + 2 * t) = v;
        }
    }
}

template <int DH>
void launch_dh(const void *Q, int64_t ldq, const void *K, const void *V, int64_t ldkv, int M, int L,
               int H, void *O, int64_t ldo, cudaStream_t st) {
    const size_t smem = (size_t)(BR + 4 * BC) * DH * 2;
    static int attr_done[64] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_done[dev]) {
        cudaFuncSetAttribute(attn_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        attr_done[dev] = 1;
    }
    dim3 grid((M + BR - 1) / BR, H);
    const float scale_log2 = 1.4426950408889634f / sqrtf((float)DH);
    echo::LaunchScope ls(ECHO_K_ATTENTION, M, L, (int64_t)H * DH, st);
    attn_kernel<DH><<<grid, THREADS, smem, st>>>(
        static_cast<const __nv_bfloat16 *>(Q), ldq, static_cast<const __nv_bfloat16 *>(K),
        static_cast<const __nv_bfloat16 *>(V), ldkv, M, L, static_cast<__nv_bfloat16 *>(O), ldo,
        scale_log2);
}

}  // namespace

namespace echo {

void launch_attention(const void *Q, int64_t ldq, const void *K, const void *V, int64_t ldkv,
                      int32_t M, int32_t L, int32_t H, int32_t d, void *O, int64_t ldo,
                      cudaStream_t st) {
    if (M <= 0) return;
    if (d == 64)
        launch_dh<64>(Q, ldq, K, V, ldkv, M, L, H, O, ldo, st);
    else
        launch_dh<128>(Q, ldq, K, V, ldkv, M, L, H, O, ldo, st);
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
    launch_attention(Q, ldq, K, V, ldkv, M, L, H, d, O, ldo, reinterpret_cast<cudaStream_t>(stream));
    return last_launch_status();
}
