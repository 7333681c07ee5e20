// Multi-head attention on (Q', K, V) (Sec. 3.3): queries only for the active
// latents, keys and values over the complete latent set (self-attention) or the
// audio condition tokens (cross-attention).
//
// Flash-style forward on the 5th-generation tensor cores.  One CTA per
// (two 128-query tiles, head), 12 warps, with the two tiles in ping-pong so
// that one tile's softmax runs while the tensor cores work on the other:
//   warp 0      TMA producer: both Q tiles once, then 128-key blocks K_0, V_0,
//               K_1, V_1, ... (128-byte swizzle, 64-column boxes) into a ring
//               shared by K and V (5 slots for d = 128);
//   warp 1      one elected lane issues S_t = Q_t K_j^T (M 128, N 128, K d) into the
//               tile's TMEM S columns and O_t += P_t V_j (M 128, N d, K 128; P
//               read from TMEM, V read MN-major straight from its row-major
//               tile) into the tile's TMEM O accumulator, in the order
//               PV0_j S0_{j+1} PV1_j S1_{j+1};
//   warp 2      allocates / frees 512 TMEM columns (S0, S1, O0, O1);
//   warps 4..7  softmax of tile 0, warps 8..11 softmax of tile 1, one query row
//               per thread (its TMEM lane, 224 registers after setmaxnreg): the
//               S row is loaded once, its max taken, P = 2^(s*scale - m) formed
//               on fp32 pairs, rounded to bf16 and stored back into the first 64
//               columns of S_t.  The running max comes from the first block;
//               later blocks reuse it (exact after the final division by the row
//               sum) and redo themselves with a fresh max, rescaling O in TMEM,
//               only when their row sum shows P above 2^64; final O / l to bf16.
// Keys beyond L are masked to P = 0; queries beyond M run on zero rows and are
// not stored.  Every mbarrier wait is bounded (ECHO_ERR_TIMEOUT).
#include "common.cuh"
#include "internal.h"

namespace {

constexpr int BM = 128;        // queries per tile; two tiles per CTA
constexpr int TILES = 2;
constexpr int BN = 128;        // keys per block
constexpr int RING_MAX = 8;    // K/V ring slots (K_j and V_j alternate)
constexpr int THREADS = 384;   // 4 control warps + 2 softmax warpgroups
constexpr uint32_t TMEM_COLS = 512;   // S0, S1, O0, O1
constexpr uint32_t O_COL = 256;
constexpr int ATOM_BYTES = 128 * 128;   // one [128 rows x 64 bf16] 128B-swizzled box
// up to this many keys: the persistent kernel below (measured at 6552 queries,
// 40 heads of 128: faster by 8% at 1280 keys, slower by 3% at 2560 and by 7% at
// 4096, where the one-shot kernel's waves already hide its fixed costs)
constexpr int kItemsMaxKeys = 2048;

template <int DH>
struct Cfg {
    static constexpr int ATOMS = DH / 64;
    static constexpr int Q_BYTES = BM * DH * 2;
    static constexpr int SLOT_BYTES = BN * DH * 2;
    static constexpr int RING = DH == 128 ? 5 : RING_MAX;
    static constexpr int SMEM = TILES * Q_BYTES + RING * SLOT_BYTES + 1024;
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
    constexpr int RING = C::RING;
    uint8_t *Qs = smem;                                  // [TILES][Q_BYTES]
    uint8_t *Ring = Qs + TILES * C::Q_BYTES;             // [RING][SLOT_BYTES]

    // Every barrier is reused only after its previous phase has been observed
    // by its waiter, so no waiter can fall two phases behind.
    __shared__ __align__(8) uint64_t q_full, ring_full[RING_MAX], ring_empty[RING_MAX];
    __shared__ __align__(8) uint64_t s_full[TILES], p_full[TILES], pv_done[TILES];
    __shared__ __align__(8) uint64_t drain;
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_flag;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int h = blockIdx.y;
    const int q0 = blockIdx.x * (TILES * BM);
    const int nb = (p.L + BN - 1) / BN;

    if (threadIdx.x == 0) {
        mbar_init(&q_full, 1);
        for (int i = 0; i < RING; ++i) { mbar_init(&ring_full[i], 1); mbar_init(&ring_empty[i], 1); }
        for (int t = 0; t < TILES; ++t) {
            mbar_init(&s_full[t], 1);
            mbar_init(&p_full[t], 4);    // one arrival per softmax warp
            mbar_init(&pv_done[t], 1);
        }
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
    // Register split (launch: 384 x 168 = 64512): the control warpgroup keeps
    // 48 per thread, the two softmax warpgroups take 224 (128*48 + 256*224 = 63488).
    if (warp < 4) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 48;" ::: "memory");
    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer: Q0, Q1, then K_0, V_0, K_1, V_1, ... ----------------
        const int x0 = h * DH;
        mbar_arrive_expect_tx(&q_full, TILES * C::Q_BYTES);
        for (int t = 0; t < TILES; ++t)
            for (int a = 0; a < C::ATOMS; ++a)
                tma_load_2d(Qs + t * C::Q_BYTES + a * ATOM_BYTES, &tmQ, &q_full, x0 + 64 * a,
                            q0 + t * BM);
        int issued = 0;
        for (int li = 0; li < 2 * nb; ++li) {
            const int slot = li % RING;
            if (!mbar_wait(&ring_empty[slot], ((li / RING) & 1) ^ 1, abort_v, p.err)) break;
            mbar_arrive_expect_tx(&ring_full[slot], C::SLOT_BYTES);
            const CUtensorMap *m = (li & 1) ? &tmV : &tmK;
            for (int a = 0; a < C::ATOMS; ++a)
                tma_load_2d(Ring + slot * C::SLOT_BYTES + a * ATOM_BYTES, m, &ring_full[slot],
                            x0 + 64 * a, (li >> 1) * BN);
            issued = li + 1;
        }
        if (*abort_v) {  // let this CTA's copies land before it exits
            mbar_wait(&q_full, 0, abort_v, nullptr, 100000000ull);
            for (int li = issued - RING < 0 ? 0 : issued - RING; li < issued; ++li)
                mbar_wait(&ring_full[li % RING], (li / RING) & 1, abort_v, nullptr, 100000000ull);
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        // order: S0_0 S1_0 | PV0_0 S0_1 PV1_0 S1_1 | PV0_1 S0_2 PV1_1 S1_2 | ...
        // The whole warp runs this loop and one elected lane issues the MMAs and
        // commits: the ring arithmetic and the descriptors then stay warp-uniform
        // and feed tcgen05.mma directly.  Issued from a single diverged lane, the
        // same loop ran the tensor cores about a quarter slower.
        // Every wait and fence sits on the path that feeds the tensor cores:
        // K_{j+1} is waited for before S0_{j+1}, V_{j+1} after S1_{j+1}.
        // P_t lives in the first 64 columns of S_t; S_t of the next block is
        // issued after P V of this block, and tcgen05.mma from one thread run in
        // order, so the S write cannot overtake the P read.  The commit of S_t
        // (s_full) therefore also tells the softmax that P V_{t, j-1} is done.
        const bool leader = elect_one_sync();
        // Shared-memory descriptors as two words: the low word holds the start
        // address in 16-byte units and the leading byte offset, the high word the
        // 1024-byte stride of eight 128-byte rows, the descriptor version and the
        // 128-byte swizzle.  A K step only adds a constant to the low word.
        constexpr uint32_t DESC_HI = (1024u >> 4) | (1u << 14) | (2u << 29);
        constexpr uint32_t LO_K = 1u << 16;                            // K-major: LBO unused
        constexpr uint32_t LO_MN = (uint32_t)(ATOM_BYTES >> 4) << 16;  // MN-major: LBO = one atom
        const uint32_t q_lo = ((smem_u32(Qs) & 0x3FFFFu) >> 4) | LO_K;
        const uint32_t ring_lo = (smem_u32(Ring) & 0x3FFFFu) >> 4;
        auto desc = [](uint32_t lo) -> uint64_t { return ((uint64_t)DESC_HI << 32) | lo; };
        auto wait_all = [&](uint64_t *bar, uint32_t parity) -> bool {
            return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort_v, p.err));
        };
        bool ok = wait_all(&q_full, 0);
        auto mma_s = [&](int t, int slot) {
            const uint32_t a_lo = q_lo + (uint32_t)t * (C::Q_BYTES >> 4);
            const uint32_t b_lo = (ring_lo + (uint32_t)slot * (C::SLOT_BYTES >> 4)) | LO_K;
            const uint32_t d = tmem + (uint32_t)(t * BN);
#pragma unroll
            for (int kk = 0; kk < DH / 16; ++kk) {
                const uint32_t off = (uint32_t)(((kk >> 2) * ATOM_BYTES + (kk & 3) * 32) >> 4);
                tc_mma_f16(d, desc(a_lo + off), desc(b_lo + off), C::IDESC_S, kk > 0);
            }
        };
        auto mma_pv = [&](int t, int slot, uint32_t acc0) {
            const uint32_t b_lo = (ring_lo + (uint32_t)slot * (C::SLOT_BYTES >> 4)) | LO_MN;
            const uint32_t d = tmem + O_COL + (uint32_t)(t * DH);
            const uint32_t a = tmem + (uint32_t)(t * BN);
            tc_mma_f16_tmem_a(d, a, desc(b_lo), C::IDESC_PV, acc0);
#pragma unroll
            for (int kk = 1; kk < BN / 16; ++kk)
                tc_mma_f16_tmem_a(d, a + 8 * kk, desc(b_lo + (uint32_t)(kk * 2048 >> 4)), C::IDESC_PV, 1u);
        };
        // ring position (slot, phase parity) of K_j; V_j is the next position
        int ks = 0;
        uint32_t kph = 0;
        auto next = [&](int &slot, uint32_t &ph) { if (++slot == RING) { slot = 0; ph ^= 1u; } };
        {   // K_0 and V_0, then S_0 of both tiles
            int vs = ks; uint32_t vph = kph; next(vs, vph);
            ok = ok && wait_all(&ring_full[ks], kph) && wait_all(&ring_full[vs], vph);
        }
        if (ok) {
            tc_fence_after();
            if (leader) {
                mma_s(0, ks);
                tc_commit(&s_full[0]);
                mma_s(1, ks);
                tc_commit(&s_full[1]);
                tc_commit(&ring_empty[ks]);
            }
            __syncwarp();
        }
        for (int j = 0; ok && j < nb; ++j) {
            int vs = ks; uint32_t vph = kph; next(vs, vph);       // V_j
            int ns = vs; uint32_t nph = vph; next(ns, nph);       // K_{j+1}
            int ws = ns; uint32_t wph = nph; next(ws, wph);       // V_{j+1}
            const bool more = j + 1 < nb;
            const uint32_t acc0 = j > 0 ? 1u : 0u;
            // tile 0: P V_j, then S_{j+1} once K_{j+1} has landed
            if (!wait_all(&p_full[0], j & 1)) { ok = false; break; }
            tc_fence_after();
            if (leader) {
                mma_pv(0, vs, acc0);
                if (!more) tc_commit(&pv_done[0]);
            }
            __syncwarp();
            if (more) {
                if (!wait_all(&ring_full[ns], nph)) { ok = false; break; }
                tc_fence_after();
                if (leader) {
                    mma_s(0, ns);
                    tc_commit(&s_full[0]);
                }
                __syncwarp();
            }
            // tile 1
            if (!wait_all(&p_full[1], j & 1)) { ok = false; break; }
            tc_fence_after();
            if (leader) {
                mma_pv(1, vs, acc0);
                if (!more) tc_commit(&pv_done[1]);
                tc_commit(&ring_empty[vs]);                      // V_j no longer needed
                if (more) {
                    mma_s(1, ns);
                    tc_commit(&s_full[1]);
                    tc_commit(&ring_empty[ns]);                  // K_{j+1} no longer needed
                }
            }
            __syncwarp();
            // V_{j+1} is read by the next block's P V only.  Waiting for it here
            // rather than beside K_{j+1} puts the wait in the window in which
            // tile 0's softmax forms P_{j+1}, and lets S0_{j+1} start sooner.
            if (more && !wait_all(&ring_full[ws], wph)) { ok = false; break; }
            ks = ns;
            kph = nph;
        }
        if (!ok && leader) {  // wait for the MMAs already issued before tensor memory is freed
            tc_commit(&drain);
            mbar_wait(&drain, 0, abort_v, nullptr, 100000000ull);
        }
    }
    } else {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 224;" ::: "memory");
        // ---------------- softmax / correction / epilogue of tile t ----------------
        const int t = (warp - 4) >> 2;
        const int quad = warp & 3;
        const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
        const uint32_t s_col = (uint32_t)(t * BN);
        const uint32_t o_col = O_COL + (uint32_t)(t * DH);
        const float sl2 = p.scale_log2;
        float m_used = -INFINITY, l = 0.f;
        bool ok = true;
        for (int j = 0; j < nb; ++j) {
            ok = __all_sync(0xffffffffu, mbar_wait(&s_full[t], j & 1, abort_v, p.err));
            if (!ok) break;
            tc_fence_after();
            // the whole S row of this block in registers (one TMEM round trip)
            const int kvalid = p.L - j * BN;                 // keys of this block that exist
            float sv[BN];
#pragma unroll
            for (int c = 0; c < BN / 32; ++c)
                tmem_ld32(tmem + lane_base + s_col + 32 * c, reinterpret_cast<uint32_t *>(sv + 32 * c));
            tmem_ld_wait();
            if (kvalid < BN) {                               // tail block only
#pragma unroll
                for (int i = 0; i < BN; ++i)
                    if (i >= kvalid) sv[i] = -INFINITY;
            }
            // The running max m_used is taken from the first block only.  Later
            // blocks form P with it directly: the result is exact after the final
            // division by the row sum, and fp32 / bf16 keep their precision at any
            // exponent, so a rescale is needed only when P could overflow.  The
            // block's row sum bounds its largest P; when it exceeds 2^64 (or is
            // not finite) the block is redone with a fresh max and O, l rescaled.
            auto block_max = [&]() -> float {
                float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
                for (int i = 0; i < BN; i += 8) {
                    m4[0] = fmax3(m4[0], sv[i], sv[i + 1]);
                    m4[1] = fmax3(m4[1], sv[i + 2], sv[i + 3]);
                    m4[2] = fmax3(m4[2], sv[i + 4], sv[i + 5]);
                    m4[3] = fmax3(m4[3], sv[i + 6], sv[i + 7]);
                }
                return fmaxf(fmax3(m4[0], m4[1], m4[2]), m4[3]);
            };
            // P = 2^(s*scale - m) on fp32 pairs, rounded to bf16 pairs; returns
            // the row sum of this block
            uint32_t pk[BN / 2];
            auto exp_pass = [&]() -> float {
                const uint64_t scale2 = f2_pack(sl2, sl2);
                const uint64_t negm2 = f2_pack(-m_used, -m_used);
                uint64_t acc2[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
                for (int i = 0; i < BN / 2; ++i) {
                    float x0, x1;
                    f2_unpack(f2_fma(f2_pack(sv[2 * i], sv[2 * i + 1]), scale2, negm2), x0, x1);
                    const float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
                    pk[i] = pack_bf16(p0, p1);
                    acc2[i & 3] = f2_add(acc2[i & 3], f2_pack(p0, p1));
                }
                float a0, a1;
                f2_unpack(f2_add(f2_add(acc2[0], acc2[1]), f2_add(acc2[2], acc2[3])), a0, a1);
                return a0 + a1;
            };
            if (j == 0) m_used = block_max() * sl2;
            float bsum = exp_pass();
            const bool redo = !(bsum <= 1.8446744e19f);     // > 2^64, inf or NaN
            if (__any_sync(0xffffffffu, redo)) {              // rare: warp-uniform slow path
                float alpha = 1.f;
                if (redo) {
                    const float m_new = fmaxf(m_used, block_max() * sl2);
                    alpha = ex2_approx(m_used - m_new);
                    l *= alpha;
                    m_used = m_new;
                }
                if (j > 0) {   // S_t of this block completed after P V_{t, j-1}: O_t is settled
#pragma unroll
                    for (int c = 0; c < DH / 32; ++c) {
                        uint32_t o[32];
                        tmem_ld32(tmem + lane_base + o_col + 32 * c, o);
                        tmem_ld_wait();
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
                        tmem_st32(tmem + lane_base + o_col + 32 * c, o);
                    }
                    tmem_st_wait();
                }
                bsum = exp_pass();
            }
            l += bsum;
            // P into TMEM columns [0, 64) of S_t (S is already in registers)
            tmem_st32(tmem + lane_base + s_col, pk);
            tmem_st32(tmem + lane_base + s_col + 32, pk + 32);
            tmem_st_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&p_full[t]);
        }
        if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&pv_done[t], 0, abort_v, p.err));
        if (ok) {
            tc_fence_after();
            const float inv = 1.f / l;
            // The warp's 32 rows of O go through its quarter of Q_t (free now:
            // every MMA that read Q_t is done) and leave in whole row segments,
            // CH lanes per row, instead of one row per lane.  The 16-byte chunks
            // of a staged row are XOR-swizzled by the row so that both the
            // row-per-lane writes and the chunk-per-lane reads spread over the
            // shared-memory banks.
            constexpr int RB = DH * 2, CH = RB / 16;          // bytes and 16-byte chunks per row
            uint8_t *stage = Qs + t * C::Q_BYTES + quad * 32 * RB;
#pragma unroll
            for (int c = 0; c < DH / 32; ++c) {
                uint32_t o[32];
                tmem_ld32(tmem + lane_base + o_col + 32 * c, o);
                tmem_ld_wait();
                float f[32];
#pragma unroll
                for (int i = 0; i < 32; ++i) f[i] = __uint_as_float(o[i]) * inv;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int cc = 4 * c + i;
                    *reinterpret_cast<uint4 *>(stage + lane * RB + ((cc ^ (lane & (CH - 1))) * 16)) =
                        pack8_bf16(f + 8 * i);
                }
            }
            __syncwarp();
            constexpr int RPI = 32 / CH;                        // rows per warp-wide store
#pragma unroll
            for (int k = 0; k < 32 / RPI; ++k) {
                const int rr = k * RPI + lane / CH, cc = lane % CH;
                const uint4 v =
                    *reinterpret_cast<const uint4 *>(stage + rr * RB + ((cc ^ (rr & (CH - 1))) * 16));
                const int grow = q0 + t * BM + quad * 32 + rr;
                if (grow < p.M)
                    *reinterpret_cast<uint4 *>(p.O + (int64_t)grow * p.ldo + h * DH + 8 * cc) = v;
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

// ---------------------------------------------------------------------------
// Short key sets (the cross-attention to the audio tokens): a persistent form
// of the kernel above.  With a few hundred keys a CTA of the one-shot kernel
// spends about as long on its fixed costs (barrier and tensor-memory set-up,
// the first Q copy, the pipeline fill and the epilogue) as on tensor work.
// Here one CTA per SM walks the work items (two 128-query tiles, head) in
// order item = blockIdx.x + k * gridDim.x, allocates tensor memory once, and
// chains the items through the MMA pipeline: S of the next item's first key
// block is issued right after the last P V of the current one, so the tensor
// cores keep working while the softmax warps run the epilogue.  Q is double
// buffered: warp 3 (idle in the kernel above) copies the Q tiles of item k + 2
// as soon as item k's epilogue has released its buffer.  The epilogue stages O
// in that item's finished Q buffer as above, and its global stores go out a few
// at a time after each of the next item's first four softmax blocks.  The key block BN (96 for the
// 672 audio tokens: 7 blocks, no padding) is chosen per launch to waste few
// keys.  Ring positions, S/P/PV barrier phases and block counters run on
// across items.
// ---------------------------------------------------------------------------
constexpr int kMaxDynSmem = 232448 - 2048;   // 227 KB per CTA, less static shared memory

template <int DH, int BN>
struct ItemCfg {
    static constexpr int ATOMS = DH / 64;
    static constexpr int Q_ATOM = BM * 128;           // [128 rows x 64 bf16]
    static constexpr int KV_ATOM = BN * 128;          // [BN rows x 64 bf16]
    static constexpr int Q_BYTES = BM * DH * 2;
    static constexpr int QBUF_BYTES = TILES * Q_BYTES;
    static constexpr int SLOT_BYTES = BN * DH * 2;
    static constexpr int RING_FIT = (kMaxDynSmem - 1024 - 2 * QBUF_BYTES) / SLOT_BYTES;
    static constexpr int RING = RING_FIT < RING_MAX ? RING_FIT : RING_MAX;
    static_assert(RING >= 3, "K_j, V_j and K_{j+1} must fit in the ring at once");
    static constexpr int SMEM = 2 * QBUF_BYTES + RING * SLOT_BYTES + 1024;
    static constexpr uint32_t IDESC_S = idesc_bf16_f32(BM, BN);
    static constexpr uint32_t IDESC_PV = idesc_bf16_f32(BM, DH) | (1u << 16);  // B MN-major
};

struct ItemParams {
    int M, L, H, ntp, items;   // ntp = query-tile pairs per head; items = ntp * H
    float scale_log2;
    __nv_bfloat16 *O;
    int64_t ldo;
    int *err;
};

template <int DH, int BN>
__global__ void __launch_bounds__(THREADS, 1)
attn_items_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                  const __grid_constant__ CUtensorMap tmV, const ItemParams p) {
    using C = ItemCfg<DH, BN>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    constexpr int RING = C::RING;
    uint8_t *Qs = smem;                                  // [2 buffers][TILES][Q_BYTES]
    uint8_t *Ring = Qs + 2 * C::QBUF_BYTES;              // [RING][SLOT_BYTES]

    // As above, no barrier is reused before its waiter has seen the previous
    // phase: q_full[b] / q_empty[b] alternate per item between the Q producer
    // and the MMA warp / the 8 epilogue warps; s_full, p_full, pv_done and the
    // ring keep their one-phase-per-block (per-item for pv_done) rhythm.
    __shared__ __align__(8) uint64_t q_full[2], q_empty[2], ring_full[RING_MAX], ring_empty[RING_MAX];
    __shared__ __align__(8) uint64_t s_full[TILES], p_full[TILES], pv_done[TILES];
    __shared__ __align__(8) uint64_t drain;
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_flag;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nb = (p.L + BN - 1) / BN;
    const int n_items = (p.items - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x;
    auto item_tp = [&](int k) { return ((int)blockIdx.x + k * (int)gridDim.x) % p.ntp; };
    auto item_h = [&](int k) { return ((int)blockIdx.x + k * (int)gridDim.x) / p.ntp; };

    if (threadIdx.x == 0) {
        for (int b = 0; b < 2; ++b) { mbar_init(&q_full[b], 1); mbar_init(&q_empty[b], 8); }
        for (int i = 0; i < RING; ++i) { mbar_init(&ring_full[i], 1); mbar_init(&ring_empty[i], 1); }
        for (int t = 0; t < TILES; ++t) {
            mbar_init(&s_full[t], 1);
            mbar_init(&p_full[t], 4);    // one arrival per softmax warp
            mbar_init(&pv_done[t], 1);
        }
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
    // Register split as in the kernel above (launch: 384 x 168).
    if (warp < 4) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 48;" ::: "memory");
    if (warp == 3 && lane == 0) {
        // ---------------- Q producer: item k's two tiles into buffer k & 1 ----------------
        int issued = 0;
        for (int k = 0; k < n_items; ++k) {
            const int b = k & 1, u = k >> 1;
            if (u > 0) {
                if (!mbar_wait(&q_empty[b], (u - 1) & 1, abort_v, p.err)) break;
                fence_proxy_async_smem();   // the epilogue's generic accesses before the copy
            }
            const int x0 = item_h(k) * DH, y0 = item_tp(k) * (TILES * BM);
            mbar_arrive_expect_tx(&q_full[b], C::QBUF_BYTES);
            for (int t = 0; t < TILES; ++t)
                for (int a = 0; a < C::ATOMS; ++a)
                    tma_load_2d(Qs + b * C::QBUF_BYTES + t * C::Q_BYTES + a * C::Q_ATOM, &tmQ,
                                &q_full[b], x0 + 64 * a, y0 + t * BM);
            issued = k + 1;
        }
        if (*abort_v)   // let this CTA's copies land before it exits
            for (int k = issued - 2 < 0 ? 0 : issued - 2; k < issued; ++k)
                mbar_wait(&q_full[k & 1], (k >> 1) & 1, abort_v, nullptr, 100000000ull);
    } else if (warp == 0 && lane == 0) {
        // ---------------- K/V producer: K_0, V_0, K_1, V_1, ... of every item ----------------
        int g = 0;
        bool ok = true;
        for (int k = 0; ok && k < n_items; ++k) {
            const int x0 = item_h(k) * DH;
            for (int li = 0; li < 2 * nb; ++li, ++g) {
                const int slot = g % RING;
                if (!mbar_wait(&ring_empty[slot], ((g / RING) & 1) ^ 1, abort_v, p.err)) {
                    ok = false;
                    break;
                }
                mbar_arrive_expect_tx(&ring_full[slot], C::SLOT_BYTES);
                const CUtensorMap *m = (li & 1) ? &tmV : &tmK;
                for (int a = 0; a < C::ATOMS; ++a)
                    tma_load_2d(Ring + slot * C::SLOT_BYTES + a * C::KV_ATOM, m, &ring_full[slot],
                                x0 + 64 * a, (li >> 1) * BN);
            }
        }
        if (*abort_v)
            for (int gi = g - RING < 0 ? 0 : g - RING; gi < g; ++gi)
                mbar_wait(&ring_full[gi % RING], (gi / RING) & 1, abort_v, nullptr, 100000000ull);
    } else if (warp == 1) {
        // ---------------- MMA issuer over the flattened block sequence ----------------
        // Block f = k * nb + j of this CTA (item k, key block j).  Order:
        //   S0_0 S1_0 | PV0_f S0_{f+1} PV1_f S1_{f+1} | ...
        // across item boundaries too: S of an item's first block reads the
        // item's Q buffer (waited for on q_full) and P V of its first block
        // overwrites O (no accumulate).
        const bool leader = elect_one_sync();
        constexpr uint32_t DESC_HI = (1024u >> 4) | (1u << 14) | (2u << 29);
        constexpr uint32_t LO_K = 1u << 16;
        constexpr uint32_t LO_MN = (uint32_t)(C::KV_ATOM >> 4) << 16;   // LBO = one 64-column atom
        const uint32_t q_lo = ((smem_u32(Qs) & 0x3FFFFu) >> 4) | LO_K;
        const uint32_t ring_lo = (smem_u32(Ring) & 0x3FFFFu) >> 4;
        auto desc = [](uint32_t lo) -> uint64_t { return ((uint64_t)DESC_HI << 32) | lo; };
        auto wait_all = [&](uint64_t *bar, uint32_t parity) -> bool {
            return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort_v, p.err));
        };
        auto mma_s = [&](int b, int t, int slot) {
            const uint32_t a_lo = q_lo + (uint32_t)((b * C::QBUF_BYTES + t * C::Q_BYTES) >> 4);
            const uint32_t b_lo = (ring_lo + (uint32_t)slot * (C::SLOT_BYTES >> 4)) | LO_K;
            const uint32_t d = tmem + (uint32_t)(t * 128);
#pragma unroll
            for (int kk = 0; kk < DH / 16; ++kk) {
                const uint32_t a_off = (uint32_t)(((kk >> 2) * C::Q_ATOM + (kk & 3) * 32) >> 4);
                const uint32_t b_off = (uint32_t)(((kk >> 2) * C::KV_ATOM + (kk & 3) * 32) >> 4);
                tc_mma_f16(d, desc(a_lo + a_off), desc(b_lo + b_off), C::IDESC_S, kk > 0);
            }
        };
        auto mma_pv = [&](int t, int slot, uint32_t acc0) {
            const uint32_t b_lo = (ring_lo + (uint32_t)slot * (C::SLOT_BYTES >> 4)) | LO_MN;
            const uint32_t d = tmem + O_COL + (uint32_t)(t * DH);
            const uint32_t a = tmem + (uint32_t)(t * 128);
            tc_mma_f16_tmem_a(d, a, desc(b_lo), C::IDESC_PV, acc0);
#pragma unroll
            for (int kk = 1; kk < BN / 16; ++kk)
                tc_mma_f16_tmem_a(d, a + 8 * kk, desc(b_lo + (uint32_t)(kk * 2048 >> 4)), C::IDESC_PV, 1u);
        };
        int ks = 0;
        uint32_t kph = 0;
        auto next = [&](int &slot, uint32_t &ph) { if (++slot == RING) { slot = 0; ph ^= 1u; } };
        const int total = n_items * nb;
        bool ok = wait_all(&q_full[0], 0);
        {
            int vs = ks; uint32_t vph = kph; next(vs, vph);
            ok = ok && wait_all(&ring_full[ks], kph) && wait_all(&ring_full[vs], vph);
        }
        if (ok) {
            tc_fence_after();
            if (leader) {
                mma_s(0, 0, ks);
                tc_commit(&s_full[0]);
                mma_s(0, 1, ks);
                tc_commit(&s_full[1]);
                tc_commit(&ring_empty[ks]);
            }
            __syncwarp();
        }
        for (int f = 0, k = 0, j = 0; ok && f < total; ++f) {
            int vs = ks; uint32_t vph = kph; next(vs, vph);       // V of block f
            int ns = vs; uint32_t nph = vph; next(ns, nph);       // K of block f + 1
            int ws = ns; uint32_t wph = nph; next(ws, wph);       // V of block f + 1
            const bool more = f + 1 < total;
            const bool last_j = j == nb - 1;
            const int kn = last_j ? k + 1 : k;                    // item of block f + 1
            const uint32_t acc0 = j > 0 ? 1u : 0u;
            if (!wait_all(&p_full[0], f & 1)) { ok = false; break; }
            tc_fence_after();
            if (leader) {
                mma_pv(0, vs, acc0);
                if (last_j) tc_commit(&pv_done[0]);
            }
            __syncwarp();
            if (more) {
                if (last_j && !wait_all(&q_full[kn & 1], (kn >> 1) & 1)) { ok = false; break; }
                if (!wait_all(&ring_full[ns], nph)) { ok = false; break; }
                tc_fence_after();
                if (leader) {
                    mma_s(kn & 1, 0, ns);
                    tc_commit(&s_full[0]);
                }
                __syncwarp();
            }
            if (!wait_all(&p_full[1], f & 1)) { ok = false; break; }
            tc_fence_after();
            if (leader) {
                mma_pv(1, vs, acc0);
                if (last_j) tc_commit(&pv_done[1]);
                tc_commit(&ring_empty[vs]);
                if (more) {
                    mma_s(kn & 1, 1, ns);
                    tc_commit(&s_full[1]);
                    tc_commit(&ring_empty[ns]);
                }
            }
            __syncwarp();
            if (more && !wait_all(&ring_full[ws], wph)) { ok = false; break; }
            ks = ns;
            kph = nph;
            k = kn;
            j = last_j ? 0 : j + 1;
        }
        if (!ok && leader) {
            tc_commit(&drain);
            mbar_wait(&drain, 0, abort_v, nullptr, 100000000ull);
        }
    }
    } else {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 224;" ::: "memory");
        // ---------------- softmax / epilogue of tile t, item after item ----------------
        const int t = (warp - 4) >> 2;
        const int quad = warp & 3;
        const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
        const uint32_t s_col = (uint32_t)(t * 128);
        const uint32_t o_col = O_COL + (uint32_t)(t * DH);
        const float sl2 = p.scale_log2;
        constexpr int RB = DH * 2, CH = RB / 16;               // bytes and 16-byte chunks per row
        constexpr int RPI = 32 / CH;                           // rows per warp-wide store
        constexpr int N_ST = 32 / RPI;                         // warp-wide stores per item
        // spread over the next item's first min(nb, 4) blocks, so that the
        // buffer is released before the next item's last block: the Q of the
        // item after next, which the MMA warp waits for there, needs it
        const int spread = nb < 4 ? nb : 4;
        const int st_per_block = (N_ST + spread - 1) / spread;
        auto stage_of = [&](int k) {
            return Qs + (k & 1) * C::QBUF_BYTES + t * C::Q_BYTES + quad * 32 * RB;
        };
        // Item k's O leaves its staging buffer in parts, a few warp-wide stores
        // after each of the next item's first softmax blocks, so that the
        // stores overlap that work instead of holding the warp at the item
        // boundary; the buffer then goes back to the Q producer.
        int pend_k = -1, pend_i = 0;
        auto store_part = [&](int n) {
            const uint8_t *stage = stage_of(pend_k);
            const int row0 = item_tp(pend_k) * (TILES * BM) + t * BM + quad * 32;
            const int col0 = item_h(pend_k) * DH;
            const int end = pend_i + n < N_ST ? pend_i + n : N_ST;
            for (; pend_i < end; ++pend_i) {
                const int rr = pend_i * RPI + lane / CH, cc = lane % CH;
                const uint4 v =
                    *reinterpret_cast<const uint4 *>(stage + rr * RB + ((cc ^ (rr & (CH - 1))) * 16));
                const int grow = row0 + rr;
                if (grow < p.M)
                    *reinterpret_cast<uint4 *>(p.O + (int64_t)grow * p.ldo + col0 + 8 * cc) = v;
            }
            if (pend_i == N_ST) {
                __syncwarp();
                if (lane == 0) mbar_arrive(&q_empty[pend_k & 1]);   // done with the buffer
                pend_k = -1;
            }
        };
        bool ok = true;
        for (int k = 0, f = 0; ok && k < n_items; ++k) {
            float m_used = -INFINITY, l = 0.f;
            for (int j = 0; j < nb; ++j, ++f) {
                ok = __all_sync(0xffffffffu, mbar_wait(&s_full[t], f & 1, abort_v, p.err));
                if (!ok) break;
                tc_fence_after();
                const int kvalid = p.L - j * BN;
                float sv[BN];
#pragma unroll
                for (int c = 0; c < BN / 32; ++c)
                    tmem_ld32(tmem + lane_base + s_col + 32 * c, reinterpret_cast<uint32_t *>(sv + 32 * c));
                tmem_ld_wait();
                if (kvalid < BN) {
#pragma unroll
                    for (int i = 0; i < BN; ++i)
                        if (i >= kvalid) sv[i] = -INFINITY;
                }
                auto block_max = [&]() -> float {
                    float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
                    for (int i = 0; i < BN; i += 8) {
                        m4[0] = fmax3(m4[0], sv[i], sv[i + 1]);
                        m4[1] = fmax3(m4[1], sv[i + 2], sv[i + 3]);
                        m4[2] = fmax3(m4[2], sv[i + 4], sv[i + 5]);
                        m4[3] = fmax3(m4[3], sv[i + 6], sv[i + 7]);
                    }
                    return fmaxf(fmax3(m4[0], m4[1], m4[2]), m4[3]);
                };
                uint32_t pk[BN / 2];
                auto exp_pass = [&]() -> float {
                    const uint64_t scale2 = f2_pack(sl2, sl2);
                    const uint64_t negm2 = f2_pack(-m_used, -m_used);
                    uint64_t acc2[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
                    for (int i = 0; i < BN / 2; ++i) {
                        float x0, x1;
                        f2_unpack(f2_fma(f2_pack(sv[2 * i], sv[2 * i + 1]), scale2, negm2), x0, x1);
                        const float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
                        pk[i] = pack_bf16(p0, p1);
                        acc2[i & 3] = f2_add(acc2[i & 3], f2_pack(p0, p1));
                    }
                    float a0, a1;
                    f2_unpack(f2_add(f2_add(acc2[0], acc2[1]), f2_add(acc2[2], acc2[3])), a0, a1);
                    return a0 + a1;
                };
                if (j == 0) m_used = block_max() * sl2;
                float bsum = exp_pass();
                const bool redo = !(bsum <= 1.8446744e19f);
                if (__any_sync(0xffffffffu, redo)) {
                    float alpha = 1.f;
                    if (redo) {
                        const float m_new = fmaxf(m_used, block_max() * sl2);
                        alpha = ex2_approx(m_used - m_new);
                        l *= alpha;
                        m_used = m_new;
                    }
                    if (j > 0) {   // S of this block completed after the item's P V_{j-1}
#pragma unroll
                        for (int c = 0; c < DH / 32; ++c) {
                            uint32_t o[32];
                            tmem_ld32(tmem + lane_base + o_col + 32 * c, o);
                            tmem_ld_wait();
#pragma unroll
                            for (int i = 0; i < 32; ++i)
                                o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
                            tmem_st32(tmem + lane_base + o_col + 32 * c, o);
                        }
                        tmem_st_wait();
                    }
                    bsum = exp_pass();
                }
                l += bsum;
#pragma unroll
                for (int c = 0; c + 32 <= BN / 2; c += 32) tmem_st32(tmem + lane_base + s_col + c, pk + c);
                if constexpr ((BN / 2) % 32 != 0)
                    tmem_st16(tmem + lane_base + s_col + (BN / 2 - 16), pk + (BN / 2 - 16));
                tmem_st_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&p_full[t]);
                if (pend_k >= 0) store_part(st_per_block);   // the previous item's O, in parts
            }
            if (!ok) break;
            ok = __all_sync(0xffffffffu, mbar_wait(&pv_done[t], k & 1, abort_v, p.err));
            if (!ok) break;
            tc_fence_after();
            const float inv = 1.f / l;
            // every load of the row's O in flight before one wait
            uint32_t o[DH / 32][32];
#pragma unroll
            for (int c = 0; c < DH / 32; ++c) tmem_ld32(tmem + lane_base + o_col + 32 * c, o[c]);
            tmem_ld_wait();
            // O of this item is out of tensor memory: the next item's first
            // P V may overwrite it once this warp arrives on p_full next time
            tc_fence_before();
            uint8_t *stage = stage_of(k);
#pragma unroll
            for (int c = 0; c < DH / 32; ++c) {
                float fo[32];
#pragma unroll
                for (int i = 0; i < 32; ++i) fo[i] = __uint_as_float(o[c][i]) * inv;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int cc = 4 * c + i;
                    *reinterpret_cast<uint4 *>(stage + lane * RB + ((cc ^ (lane & (CH - 1))) * 16)) =
                        pack8_bf16(fo + 8 * i);
                }
            }
            __syncwarp();
            pend_k = k;
            pend_i = 0;
        }
        if (ok && pend_k >= 0) store_part(N_ST);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 2) {
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
    }
}

// key block for the persistent kernel: the fewest keys computed, counting a
// fixed cost of 32 key-columns per block; ties go to the larger block
int items_block(int L) {
    const int cand[4] = {128, 96, 64, 32};
    int best = 128;
    int64_t best_cost = INT64_MAX;
    for (int bn : cand) {
        const int64_t cost = (int64_t)((L + bn - 1) / bn) * (bn + 32);
        if (cost < best_cost) { best_cost = cost; best = bn; }
    }
    return best;
}

int num_sms() {
    static int sms[64] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64) return 152;
    if (!sms[dev]) {
        int v = 0;
        if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v < 1)
            v = 152;
        sms[dev] = v;
    }
    return sms[dev];
}

template <int DH, int BN>
echo_status launch_items(const void *Q, int64_t ldq, const void *K, const void *V, int64_t ldkv,
                         int M, int L, int H, void *O, int64_t ldo, cudaStream_t st) {
    using C = ItemCfg<DH, BN>;
    static int attr_done[64] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_done[dev]) {
        cudaFuncSetAttribute(attn_items_kernel<DH, BN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             C::SMEM);
        attr_done[dev] = 1;
    }
    CUtensorMap tq, tk, tv;
    const uint64_t cols = (uint64_t)H * DH;
    if (!echo::make_tmap_bf16(&tq, Q, (uint64_t)M, cols, (uint64_t)ldq, BM) ||
        !echo::make_tmap_bf16(&tk, K, (uint64_t)L, cols, (uint64_t)ldkv, BN) ||
        !echo::make_tmap_bf16(&tv, V, (uint64_t)L, cols, (uint64_t)ldkv, BN))
        return ECHO_ERR_CUDA;
    ItemParams p;
    p.M = M;
    p.L = L;
    p.H = H;
    p.ntp = (M + TILES * BM - 1) / (TILES * BM);
    p.items = p.ntp * H;
    p.scale_log2 = 1.4426950408889634f / sqrtf((float)DH);
    p.O = static_cast<__nv_bfloat16 *>(O);
    p.ldo = ldo;
    p.err = echo::device_error_ptr();
    const int grid = p.items < num_sms() ? p.items : num_sms();
    echo::LaunchScope ls(ECHO_K_ATTENTION, M, L, (int64_t)H * DH, st);
    attn_items_kernel<DH, BN><<<grid, THREADS, C::SMEM, st>>>(tq, tk, tv, p);
    return echo::last_launch_status();
}

template <int DH>
echo_status launch_items_dh(const void *Q, int64_t ldq, const void *K, const void *V, int64_t ldkv,
                            int M, int L, int H, void *O, int64_t ldo, cudaStream_t st) {
    switch (items_block(L)) {
        case 32: return launch_items<DH, 32>(Q, ldq, K, V, ldkv, M, L, H, O, ldo, st);
        case 64: return launch_items<DH, 64>(Q, ldq, K, V, ldkv, M, L, H, O, ldo, st);
        case 96: return launch_items<DH, 96>(Q, ldq, K, V, ldkv, M, L, H, O, ldo, st);
        default: return launch_items<DH, 128>(Q, ldq, K, V, ldkv, M, L, H, O, ldo, st);
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
    dim3 grid((M + TILES * BM - 1) / (TILES * BM), H);
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
    if (L <= kItemsMaxKeys) {   // short key sets: the persistent kernel
        if (d == 64) return launch_items_dh<64>(Q, ldq, K, V, ldkv, M, L, H, O, ldo, st);
        return launch_items_dh<128>(Q, ldq, K, V, ldkv, M, L, H, O, ldo, st);
    }
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
