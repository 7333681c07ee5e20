// Dense bf16 projections of the block (Q', K/V over all latents, output
// projections, FFN on the active latents; Sec. 3.3) on the 5th-generation
// tensor cores:  out = act(A W^T + bias) + resid.
//
// Persistent CTA pairs: a cluster of two CTAs on two SMs walks 256 x 256 output
// tiles in a banded order and computes each with tcgen05.mma.cta_group::2
// (M 256, N 256, K 16): the even CTA holds rows 0..127 of the tile, the odd CTA
// rows 128..255, and each holds one 128-row half of the W tile, so each SM loads
// 32 KB per 64-deep k-block instead of the 48 KB of a one-SM 128 x 256 tile.
// 8 warps per CTA:
//   warp 0      TMA producer: the CTA's A [128 x 64] and W-half [128 x 64] bf16
//               tiles, 128-byte swizzle, into a 6-stage ring (32 KB per stage);
//               both CTAs' copies complete their bytes on the even CTA's barrier;
//   warp 1      (even CTA) one elected lane issues the pair MMAs into one of two
//               256-column fp32 accumulators (the same columns in both CTAs) and
//               commits each stage back to both producers, so the epilogue of one
//               tile overlaps the main loop of the next;
//   warp 2      allocates / frees the 512 tensor-memory columns of the pair;
//   warps 4..7  epilogue, in each CTA: tcgen05.ld 32 columns at a time (warp w
//               reads TMEM lanes 32 (w mod 4) ..), adds bias, GELU, residual, stores.
// Every mbarrier wait is bounded (ECHO_ERR_TIMEOUT); a CTA that gives up lets its
// copies land and drains its MMAs before it frees tensor memory, and a cluster
// barrier keeps either CTA from leaving while the other may still reach it.
#include "common.cuh"
#include "internal.h"

namespace {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 6;   // BM: rows per CTA of a pair tile
constexpr int A_BYTES = BM * BK * 2;         // 16 KB
constexpr int HB_BYTES = (BN / 2) * BK * 2;  // half of a W tile: 16 KB
constexpr int STAGE_BYTES = A_BYTES + HB_BYTES;
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024;  // + alignment slack
constexpr int THREADS = 256;
constexpr uint32_t TMEM_COLS = 512;   // two 256-column accumulators
constexpr int GROUP_N = 16;            // N tiles per raster band
constexpr uint32_t IDESC = idesc_bf16_f32(2 * BM, BN);

// EPI_ROWAMAX: also fold max |v| of each bf16 output row into row_amax (fp32
// bits, atomic max over the row's column tiles; a NaN beats every number)
enum : int { EPI_GELU = 1, EPI_RES_BF16 = 2, EPI_RES_F32 = 4, EPI_OUT_F32 = 8, EPI_ROWAMAX = 16 };

struct GemmParams {
    int M, N, Kd;
    const __nv_bfloat16 *bias;
    const void *resid;
    const int32_t *resid_rows;
    void *out;
    int64_t ldo;
    const int32_t *out_rows;   // output row m goes to row out_rows[m] (NULL: m)
    uint32_t *row_amax;
    int *err;
};

ECHO_DEV float gelu_tanh(float x) {
    const float k0 = 0.7978845608028654f;  // sqrt(2 / pi)
    const float u = k0 * (x + 0.044715f * x * x * x);
    return 0.5f * x * (1.f + tanhf(u));
}

// Tile order: bands of GROUP_N N-tiles; inside a band M is swept with the band's
// N-tiles adjacent, so the CTAs in flight share a few A row blocks and one band
// of W, which stay in L2 while the band is processed.
ECHO_DEV void tile_coords(int t, int num_m, int num_n, int &mt, int &nt) {
    const int band = t / (GROUP_N * num_m);
    const int first_n = band * GROUP_N;
    const int gn = min(GROUP_N, num_n - first_n);
    const int r = t - band * GROUP_N * num_m;
    mt = r / gn;
    nt = first_n + r % gn;
}

// One accumulator row of a tile (thread = TMEM lane): tcgen05.ld 32 columns at a
// time from `tacc`, bias, GELU, residual, store; EPI_ROWAMAX folds the row max.
template <int EPI>
ECHO_DEV void epilogue_row(const GemmParams &p, uint32_t tacc, int row, int n0) {
    const bool row_ok = row < p.M;
    int rrow = row;
    if ((EPI & EPI_RES_BF16) && p.resid_rows && row_ok) rrow = p.resid_rows[row];
    const int64_t orow = (p.out_rows && row_ok) ? p.out_rows[row] : row;
    uint32_t rmax = 0;   // EPI_ROWAMAX: max |v| of this row's stored values, as bits
    for (int c = 0; c < BN; c += 32) {
        const int col = n0 + c;
        if (col >= p.N) break;                       // warp-uniform
        uint32_t r[32];
        tmem_ld32(tacc + (uint32_t)c, r);
        tmem_ld_wait();
        if (!row_ok) continue;
        float v[32];
        if (p.bias) {
            const uint4 *bp = reinterpret_cast<const uint4 *>(p.bias + col);
#pragma unroll
            for (int i = 0; i < 4; ++i) unpack8_bf16(__ldg(bp + i), v + 8 * i);
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] += __uint_as_float(r[i]);
        } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
        }
        if (EPI & EPI_GELU) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = gelu_tanh(v[i]);
        }
        if (EPI & EPI_RES_BF16) {
            const uint4 *rp = reinterpret_cast<const uint4 *>(
                static_cast<const __nv_bfloat16 *>(p.resid) + (int64_t)rrow * p.N + col);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                float tt[8];
                unpack8_bf16(__ldg(rp + i), tt);
#pragma unroll
                for (int e = 0; e < 8; ++e) v[8 * i + e] += tt[e];
            }
        }
        if (EPI & EPI_RES_F32) {
            const float4 *rp = reinterpret_cast<const float4 *>(
                static_cast<const float *>(p.resid) + (int64_t)row * p.N + col);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const float4 tt = __ldg(rp + i);
                v[4 * i] += tt.x; v[4 * i + 1] += tt.y; v[4 * i + 2] += tt.z; v[4 * i + 3] += tt.w;
            }
        }
        if (EPI & EPI_OUT_F32) {
            float4 *op = reinterpret_cast<float4 *>(static_cast<float *>(p.out) +
                                                    orow * p.ldo + col);
#pragma unroll
            for (int i = 0; i < 8; ++i)
                op[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
        } else {
            uint4 *op = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(p.out) +
                                                  orow * p.ldo + col);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const uint4 pk = pack8_bf16(v + 8 * i);
                op[i] = pk;
                if (EPI & EPI_ROWAMAX) {
                    const uint32_t w[4] = {pk.x, pk.y, pk.z, pk.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        rmax = max(rmax, max((w[e] & 0x7FFFu) << 16, w[e] & 0x7FFF0000u));
                }
            }
        }
    }
    if ((EPI & EPI_ROWAMAX) && row_ok) atomicMax(&p.row_amax[row], rmax);
}

template <int EPI>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(THREADS, 1)
gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
            const GemmParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    __shared__ __align__(8) uint64_t full_bar[STAGES], empty_bar[STAGES];
    __shared__ __align__(8) uint64_t acc_full[2], acc_empty[2], drain_bar;
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_flag;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const int pair = blockIdx.x >> 1, num_pairs = gridDim.x >> 1;
    const int num_kb = p.Kd / BK;
    const int num_m = (p.M + 2 * BM - 1) / (2 * BM), num_n = (p.N + BN - 1) / BN;
    const int num_tiles = num_m * num_n;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full_bar[s], 1);    // used in the even CTA
            mbar_init(&empty_bar[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], 8);   // lane 0 of the 4 epilogue warps of both CTAs
        }
        mbar_init(&drain_bar, 1);
        abort_flag = 0;
        fence_barrier_init();
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
    }
    cluster_sync_all();   // both CTAs' barriers exist before any arrival from the other CTA
    if (warp == 2) tmem_alloc_pair(&tmem_slot, TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    volatile int *abort_v = &abort_flag;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer (both CTAs) ----------------
        // A stage is refilled only after the pair's MMAs of its previous use are
        // done (both producers see the same commit), so the bytes of one use
        // never mix with the next on the even CTA's barrier.
        const uint32_t full0 = mapa_shared(smem_u32(&full_bar[0]), 0);
        int it = 0;
        bool ok = true;
        for (int t = pair; ok && t < num_tiles; t += num_pairs) {
            int mt, nt;
            tile_coords(t, num_m, num_n, mt, nt);
            for (int kb = 0; kb < num_kb; ++kb, ++it) {
                const int s = it % STAGES;
                if (!mbar_wait_cluster(&empty_bar[s], ((it / STAGES) & 1) ^ 1, abort_v, p.err)) {
                    ok = false;
                    break;
                }
                uint8_t *a = smem + s * STAGE_BYTES;
                const uint32_t bar = full0 + (uint32_t)(s * sizeof(uint64_t));
                if (rank == 0) mbar_arrive_expect_tx(&full_bar[s], 2 * STAGE_BYTES);
                tma_load_2d_pair(a, &tmA, bar, kb * BK, mt * 2 * BM + (int)rank * BM);
                tma_load_2d_pair(a + A_BYTES, &tmB, bar, kb * BK, nt * BN + (int)rank * (BN / 2));
            }
        }
        if (*abort_v) {  // let this CTA's copies land before it exits
            if (rank == 0) {
                for (int k = it - STAGES < 0 ? 0 : it - STAGES; k < it; ++k)
                    mbar_wait(&full_bar[k % STAGES], (k / STAGES) & 1, abort_v, nullptr, 100000000ull);
            } else {   // its copies complete on the other CTA's barrier: give them time
                const uint64_t t0 = globaltimer_ns();
                while (globaltimer_ns() - t0 < 200000ull) {
                }
            }
        }
    } else if (warp == 1 && rank == 0) {
        // ---------------- MMA issuer (even CTA) ----------------
        // The whole warp runs the loop (stage arithmetic and descriptors stay
        // warp-uniform) and one elected lane issues the MMAs and commits.
        // Descriptor words: the low word holds the start address in 16-byte
        // units (leading byte offset unused for K-major), the high word the
        // 1024-byte stride of eight 128-byte rows, the version and the 128-byte
        // swizzle; a K step of 16 adds 32 bytes to the start address.  The same
        // offsets address the odd CTA's halves.
        const bool leader = elect_one_sync();
        constexpr uint32_t DESC_HI = (1024u >> 4) | (1u << 14) | (2u << 29);
        const uint32_t smem_lo = ((smem_u32(smem) & 0x3FFFFu) >> 4) | (1u << 16);
        auto desc = [](uint32_t lo) -> uint64_t { return ((uint64_t)DESC_HI << 32) | lo; };
        bool ok = true;
        int it = 0, local = 0;
        for (int t = pair; ok && t < num_tiles; t += num_pairs, ++local) {
            const int buf = local & 1;
            if (!__all_sync(0xffffffffu, mbar_wait_cluster(&acc_empty[buf], ((local >> 1) & 1) ^ 1,
                                                           abort_v, p.err))) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t d_tmem = tmem + (uint32_t)(buf * BN);
            for (int kb = 0; kb < num_kb; ++kb, ++it) {
                const int s = it % STAGES;
                if (!__all_sync(0xffffffffu,
                                mbar_wait_cluster(&full_bar[s], (it / STAGES) & 1, abort_v, p.err))) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t a_lo = smem_lo + (uint32_t)(s * (STAGE_BYTES >> 4));
                const uint32_t b_lo = a_lo + (uint32_t)(A_BYTES >> 4);
                if (leader) {
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k)
                        tc_mma_pair_f16(d_tmem, desc(a_lo + 2 * k), desc(b_lo + 2 * k), IDESC,
                                        (kb | k) != 0);
                    tc_commit_pair(&empty_bar[s], 0x3);   // the stage is free in both CTAs
                }
                __syncwarp();
            }
            if (ok && leader) tc_commit_pair(&acc_full[buf], 0x3);
            __syncwarp();
        }
        if (!ok && leader) {  // wait for the MMAs already issued before tensor memory is freed
            tc_commit_pair(&drain_bar, 0x1);
            mbar_wait(&drain_bar, 0, abort_v, nullptr, 100000000ull);
        }
    } else if (warp >= 4) {
        // ---------------- epilogue (both CTAs) ----------------
        const int q = warp & 3;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        const uint32_t empty_even[2] = {mapa_shared(smem_u32(&acc_empty[0]), 0),
                                        mapa_shared(smem_u32(&acc_empty[1]), 0)};
        int local = 0;
        for (int t = pair; t < num_tiles; t += num_pairs, ++local) {
            const int buf = local & 1;
            const bool ok = __all_sync(0xffffffffu, mbar_wait_cluster(&acc_full[buf], (local >> 1) & 1,
                                                                      abort_v, p.err, 4000000000ull));
            if (!ok) break;
            tc_fence_after();
            int mt, nt;
            tile_coords(t, num_m, num_n, mt, nt);
            epilogue_row<EPI>(p, tmem + lane_base + (uint32_t)(buf * BN),
                              mt * 2 * BM + (int)rank * BM + q * 32 + lane, nt * BN);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_remote(empty_even[buf]);
        }
    }
    tc_fence_before();
    __syncwarp();
    cluster_sync_all();   // neither CTA leaves while the other may still reach its memory
    if (warp == 2) {
        tc_fence_after();
        tmem_dealloc_pair(tmem, TMEM_COLS);
    }
}

int num_sms() {
    static int cached[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
    if (!cached[dev]) {
        int n = 0;
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        cached[dev] = n > 0 ? n : 1;
    }
    return cached[dev];
}

template <int EPI>
echo_status run(const CUtensorMap &ta, const CUtensorMap &tb, const GemmParams &p, cudaStream_t st) {
    static int pairs_max[64] = {};   // per device: co-resident CTA pairs (0: not set up yet)
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return ECHO_ERR_CUDA;
    if (!pairs_max[dev]) {   // a benign race computes the same value twice
        if (cudaFuncSetAttribute(gemm_kernel<EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 SMEM_BYTES) != cudaSuccess)
            return ECHO_ERR_CUDA;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(2 * num_sms(), 1, 1);
        cfg.blockDim = dim3(THREADS, 1, 1);
        cfg.dynamicSmemBytes = SMEM_BYTES;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, gemm_kernel<EPI>, &cfg) != cudaSuccess || n < 1)
            return ECHO_ERR_CUDA;
        pairs_max[dev] = n;
    }
    const int tiles = ((p.M + 2 * BM - 1) / (2 * BM)) * ((p.N + BN - 1) / BN);
    const int pairs = tiles < pairs_max[dev] ? tiles : pairs_max[dev];
    echo::LaunchScope ls(ECHO_K_GEMM, p.M, p.N, p.Kd, st);
    gemm_kernel<EPI><<<2 * pairs, THREADS, SMEM_BYTES, st>>>(ta, tb, p);
    return echo::last_launch_status();
}

}  // namespace

namespace echo {

echo_status launch_linear(const LinearArgs &a, cudaStream_t st) {
    if (a.M <= 0) return ECHO_OK;
    CUtensorMap ta, tb;
    if (!make_tmap_bf16(&ta, a.A, (uint64_t)a.M, (uint64_t)a.Kd, (uint64_t)a.lda, BM) ||
        !make_tmap_bf16(&tb, a.W, (uint64_t)a.N, (uint64_t)a.Kd, (uint64_t)a.Kd, BN / 2))
        return ECHO_ERR_CUDA;
    GemmParams p;
    p.M = a.M; p.N = a.N; p.Kd = a.Kd;
    p.bias = static_cast<const __nv_bfloat16 *>(a.bias);
    p.resid = a.resid;
    p.resid_rows = a.resid_rows;
    p.out = a.out;
    p.ldo = a.ldo;
    p.out_rows = a.out_rows;
    p.row_amax = a.row_amax;
    p.err = device_error_ptr();
    int epi = 0;
    if (a.act == 1) epi |= EPI_GELU;
    if (a.resid) epi |= (a.resid_t == ECHO_BF16) ? EPI_RES_BF16 : EPI_RES_F32;
    if (a.out_t == ECHO_F32) epi |= EPI_OUT_F32;
    if (a.row_amax) {
        if (epi != EPI_RES_F32) return ECHO_ERR_INVALID_ARG;   // bf16 out, fp32 residual only
        return run<EPI_RES_F32 | EPI_ROWAMAX>(ta, tb, p, st);
    }
    switch (epi) {
        case 0: return run<0>(ta, tb, p, st);
        case EPI_GELU: return run<EPI_GELU>(ta, tb, p, st);
        case EPI_RES_BF16: return run<EPI_RES_BF16>(ta, tb, p, st);
        case EPI_RES_F32: return run<EPI_RES_F32>(ta, tb, p, st);
        case EPI_GELU | EPI_RES_BF16: return run<EPI_GELU | EPI_RES_BF16>(ta, tb, p, st);
        case EPI_GELU | EPI_RES_F32: return run<EPI_GELU | EPI_RES_F32>(ta, tb, p, st);
        case EPI_OUT_F32: return run<EPI_OUT_F32>(ta, tb, p, st);
        case EPI_GELU | EPI_OUT_F32: return run<EPI_GELU | EPI_OUT_F32>(ta, tb, p, st);
        case EPI_RES_BF16 | EPI_OUT_F32: return run<EPI_RES_BF16 | EPI_OUT_F32>(ta, tb, p, st);
        case EPI_RES_F32 | EPI_OUT_F32: return run<EPI_RES_F32 | EPI_OUT_F32>(ta, tb, p, st);
        case EPI_GELU | EPI_RES_BF16 | EPI_OUT_F32:
            return run<EPI_GELU | EPI_RES_BF16 | EPI_OUT_F32>(ta, tb, p, st);
        case EPI_GELU | EPI_RES_F32 | EPI_OUT_F32:
            return run<EPI_GELU | EPI_RES_F32 | EPI_OUT_F32>(ta, tb, p, st);
    }
    return ECHO_ERR_INVALID_ARG;
}

}  // namespace echo

extern "C" echo_status echo_linear(const void *A, int64_t lda, int32_t M, int32_t Kd, const void *W,
                                   const void *bias, int32_t N, int32_t act, const void *resid,
                                   echo_dtype resid_t, const int32_t *resid_rows, void *out,
                                   int64_t ldo, echo_dtype out_t, echo_stream_t stream) {
    using namespace echo;
    if (M < 0 || Kd < 64 || Kd % 64 || N < 64 || N % 64) return ECHO_ERR_SHAPE;
    if (lda < Kd || lda % 8 || ldo < N || ldo % 8) return ECHO_ERR_SHAPE;
    if (M == 0) return ECHO_OK;
    if (!A || !W || !out) return ECHO_ERR_INVALID_ARG;
    if (act != 0 && act != 1) return ECHO_ERR_INVALID_ARG;
    if ((resid && resid_t != ECHO_BF16 && resid_t != ECHO_F32) ||
        (out_t != ECHO_BF16 && out_t != ECHO_F32))
        return ECHO_ERR_INVALID_ARG;
    if (resid_rows && (!resid || resid_t != ECHO_BF16)) return ECHO_ERR_INVALID_ARG;
    if (!aligned16(A) || !aligned16(W) || !aligned16(out) || (bias && !aligned16(bias)) ||
        (resid && !aligned16(resid)) || (resid_rows && !aligned16(resid_rows)))
        return ECHO_ERR_INVALID_ARG;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    LinearArgs a{A, lda, M, Kd, W, bias, N, act, resid, resid_t, resid_rows, out, ldo, out_t};
    return launch_linear(a, reinterpret_cast<cudaStream_t>(stream));
}
