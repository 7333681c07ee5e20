/*
 * echocache.h - C ABI of the energy-guided cached DiT step (EchoCache,
 * arXiv 2608.02474), GB300 (sm_103a) build.
 *
 * One cached step of one DiT layer, in the paper's order:
 *   echo_audio_energy  - audio -> per-segment time-frequency energy
 *                        (Sec. 3.3 "Cross-modal Saliency Anchors")
 *   echo_select        - per-token drift (Eq. 1, per token) weighted by segment
 *                        energy, top-K -> ascending active index list
 *                        (Sec. 3.3, budget k_t = ceil(N r_t) read globally)
 *   echo_block_step    - the block on the active latents: Q' on active, K/V on
 *                        all latents, cross-attention, FFN on active, merge with
 *                        the cache, write the active rows back to the cache
 *                        (Sec. 3.3 "Fine-grained latent-level caching",
 *                        Sec. 3.4 for the int8 cache)
 *   echo_cache_quant / echo_cache_dequant - the int8 per-token cache (Sec. 3.4)
 *
 * Conventions (every entry point):
 *   - All tensor pointers are DEVICE pointers unless stated; all tensors are
 *     row-major and contiguous, batch 1.  bf16 is IEEE bfloat16 (2 bytes).
 *   - The caller allocates and owns every buffer, workspace and the stream.
 *     The library never allocates device memory and never synchronises the
 *     host, except echo_get_device_error.
 *   - Work is enqueued on `stream` (NULL = legacy default stream) and is
 *     stream-ordered; buffers must stay valid until the stream has run it.
 *   - Arguments are checked before anything is enqueued: a bad argument
 *     returns an error and enqueues nothing.  Device pointers must be 16-byte
 *     aligned.  A launch failure returns ECHO_ERR_CUDA.
 *   - Data-dependent errors (a non-finite amax or score, a bounded device wait
 *     that gave up) set a device-side flag; echo_get_device_error reports and
 *     clears it.  No kernel traps.
 *   - Thread safety: calls may come from several host threads; calls on one
 *     stream run in order.
 */
#ifndef ECHOCACHE_H
#define ECHOCACHE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same object as cudaStream_t. */
typedef struct CUstream_st *echo_stream_t;

typedef enum {
    ECHO_OK = 0,
    ECHO_ERR_INVALID_ARG = 1,  /* null pointer, misaligned pointer, bad enum */
    ECHO_ERR_SHAPE = 2,        /* unsupported or inconsistent sizes */
    ECHO_ERR_WORKSPACE = 3,    /* workspace smaller than the size query */
    ECHO_ERR_CUDA = 4,         /* a CUDA call or launch failed */
    ECHO_ERR_NONFINITE = 5,    /* device flag: NaN/Inf met in a score or amax */
    ECHO_ERR_TIMEOUT = 6,      /* device flag: a bounded device wait gave up */
    ECHO_ERR_UNSUPPORTED = 7   /* no sm_103a device */
} echo_status;

typedef enum { ECHO_BF16 = 0, ECHO_F32 = 1 } echo_dtype;

/* Selection rule (Sec. 3.3).  ENERGY_DRIFT: score_i = w_seg(i) * d_i with
 * w = lambda + (1 - lambda) energy / max energy.  SEGMENT: the paper-literal
 * anchor, d_i = 1 and lambda = 0 (whole loudest segments first).  DRIFT_ONLY:
 * w = 1 (no audio guidance). */
typedef enum {
    ECHO_MODE_ENERGY_DRIFT = 0,
    ECHO_MODE_SEGMENT = 1,
    ECHO_MODE_DRIFT_ONLY = 2
} echo_select_mode;

typedef struct {
    float lambda;   /* weight floor of silent segments, in [0, 1]; default 0.1 */
    float xi;       /* Eq. 1 stabiliser, > 0; default 1e-6 */
    int32_t mode;   /* echo_select_mode */
} echo_select_params;

typedef struct {
    int32_t T;    /* latent frames = temporal segments */
    int32_t N;    /* spatial latents per frame; NT = T * N tokens */
    int32_t D;    /* hidden size, multiple of 64 */
    int32_t H;    /* heads */
    int32_t d;    /* head size, 64 or 128, H * d == D */
    int32_t F;    /* FFN width, multiple of 64 */
    int32_t Lc;   /* audio condition tokens, >= 1 */
} echo_block_dims;

/* Device pointers to one block's bf16 parameters, nn.Linear convention
 * (y = x W^T + b, W row-major [out, in]).  Wkv stacks W_k over W_v ([2D, D]),
 * bkv stacks b_k over b_v.  KVc is the block's cross-attention key|value
 * table [Lc, 2D] (columns 0..D-1 keys, D..2D-1 values) from
 * echo_precompute_cross_kv. */
typedef struct {
    const void *Wq, *bq;     /* [D, D], [D] */
    const void *Wkv, *bkv;   /* [2D, D], [2D] */
    const void *Wo, *bo;     /* [D, D], [D] */
    const void *Wqc, *bqc;   /* [D, D], [D] */
    const void *Woc, *boc;   /* [D, D], [D] */
    const void *W1, *b1;     /* [F, D], [F] */
    const void *W2, *b2;     /* [D, F], [D] */
    const void *KVc;         /* [Lc, 2D] */
} echo_block_weights;

/* Human-readable name of a status.  Never NULL. */
const char *echo_status_str(echo_status s);

/* Synchronises `stream`, then reads and clears the device error flag shared by
 * every kernel of this library on the current device.  Returns ECHO_OK, the
 * flagged error (ECHO_ERR_NONFINITE, ECHO_ERR_TIMEOUT) or ECHO_ERR_CUDA if the
 * synchronisation itself failed. */
echo_status echo_get_device_error(echo_stream_t stream);

/* Sec. 3.3 "Cross-modal Saliency Anchors": split the audio evenly into T
 * segments, STFT each, energy = L2 norm of the segment's time-frequency matrix.
 *   audio        f32 [n_samples], mono.  Segment length L_s = n_samples / T
 *                (floor; the remainder is dropped).
 *   n_fft        FFT size, power of two in [64, 4096]; hop >= 1; frames start
 *                at 0, hop, ... while start + n_fft <= L_s (one zero-padded
 *                frame if L_s < n_fft).  Periodic Hann window.
 *   band_energy  f32 [T, n_bands] out: sum over frames of one-sided power
 *                P_k = c_k |X_k|^2 / n_fft (c_0 = c_{n/2} = 1, else 2) over the
 *                linear band [floor(B b / n_bands), floor(B (b+1) / n_bands)),
 *                B = n_fft/2 + 1;  1 <= n_bands <= B.
 *   seg_energy   f32 [T] out: sqrt(sum_b band_energy[tau, b]).
 * Errors: INVALID_ARG (null/misaligned), SHAPE (T < 1, T > n_samples, bad
 * n_fft/hop/n_bands), CUDA. */
echo_status echo_audio_energy(const float *audio, int64_t n_samples, int32_t T,
                              int32_t n_fft, int32_t hop, int32_t n_bands,
                              float *band_energy, float *seg_energy,
                              echo_stream_t stream);

/* Bytes of workspace echo_select needs for NT = T * N tokens. */
size_t echo_select_workspace_size(int32_t T, int32_t N);

/* Sec. 3.3 (selection) with Eq. 1 applied per token against the cache.
 *   x            [NT, D] layer input, dtype xt (ECHO_BF16 or ECHO_F32).
 *   cache_q      int8 [NT, D], cache_scale f32 [NT]: the cached features
 *                c_ij = float(q_ij) * s_i.
 *   seg_energy   f32 [T] (echo_audio_energy output or any non-negative values).
 *   ratio        refresh ratio ratio_num / ratio_den in [0, 1];
 *                K = ceil(ratio_num * NT / ratio_den) computed in integers.
 *   p            selection parameters (host pointer; NULL = defaults).
 *   idx          int32 [>= K] out: the K active tokens, ascending.  The K
 *                largest keys (score descending, index ascending) win.
 *   K_out        host int32 out: K.
 *   scores       f32 [NT] out (may be NULL): score_i = w_{i / N} * d_i with
 *                d_i = sum_j |x_ij - c_ij| / (sum_j |c_ij| + xi), both sums
 *                fp32 in a fixed order (8-element chunks left to right, chunk
 *                c on lane c mod 32 in chunk order, then a xor butterfly
 *                16, 8, 4, 2, 1), so that the result is reproducible bit for bit.
 *   workspace    >= echo_select_workspace_size(T, N) bytes, 16-byte aligned.
 * D must be a multiple of 8.  Errors: INVALID_ARG, SHAPE, WORKSPACE, CUDA;
 * a non-finite score sets the NONFINITE device flag. */
echo_status echo_select(const void *x, echo_dtype xt, const int8_t *cache_q,
                        const float *cache_scale, const float *seg_energy,
                        int32_t T, int32_t N, int32_t D, int32_t ratio_num,
                        int32_t ratio_den, const echo_select_params *p,
                        int32_t *idx, int32_t *K_out, float *scores,
                        void *workspace, size_t ws_bytes, echo_stream_t stream);

/* No counterpart in the paper: a variant of echo_select for callers that
 * cannot allocate device memory.  Some callers own no allocator at all: code
 * running inside a host application that reserves all device memory up front
 * and forbids cudaMalloc after start-up, or code on a latency-critical thread
 * where cudaMalloc/cudaFree would synchronise the whole device.  This entry
 * point takes no workspace and allocates nothing: the drift scores live in a
 * library-owned static device array of ECHO_SELECT_STATIC_MAX_TOKENS floats
 * (256 KiB), which every GPU that loads the library holds until the process
 * exits.
 *   Arguments and results are those of echo_select, without scores and
 *   workspace; T * N must not exceed ECHO_SELECT_STATIC_MAX_TOKENS, otherwise
 *   ECHO_ERR_WORKSPACE is returned and nothing is enqueued.
 *   The first call on a device looks up that device's address of the array
 *   (once, with the device current) and keeps it for the life of the
 *   process; make that first call before any CUDA stream capture.  A device
 *   reset (cudaDeviceReset, or anything else that destroys the primary
 *   context) is not supported: the kept address would then be stale.
 *   All calls on a device share the one array and it keeps the last call's
 *   scores; nothing in it needs to start at zero, because every score the
 *   top-K reads is written first by the same call.  Calls whose work overlaps
 *   on the GPU (different streams, or different host threads without
 *   ordering) race on the array: order them on one stream. */
#define ECHO_SELECT_STATIC_MAX_TOKENS 65536
echo_status echo_select_static(const void *x, echo_dtype xt, const int8_t *cache_q,
                               const float *cache_scale, const float *seg_energy,
                               int32_t T, int32_t N, int32_t D, int32_t ratio_num,
                               int32_t ratio_den, const echo_select_params *p,
                               int32_t *idx, int32_t *K_out, echo_stream_t stream);

/* ---- cache forms (Sec. 3.4 and the quantisation ablation of Sec. 4, Table 2) ----
 *
 * One layer's cache of NT token rows of D values in one of three forms:
 *   ECHO_CACHE_INT8  plain int8 per token ("Naive INT8"): c = bf16(float(q) s),
 *                    the form echo_select / echo_block_step use.
 *   ECHO_CACHE_BF16  the rows kept in the compute precision (the "FP16"
 *                    ablation; compute precision here is bf16): c = full row.
 *   ECHO_CACHE_REF   the paper's manager (Sec. 3.4): a row written to the cache
 *                    is stored either as a reference (in full precision, in a
 *                    pool slot) or as an int8 residual against the current
 *                    reference: c = bf16(r + float(q) s), r = pool[ref] (0 when
 *                    ref = -1).  Writing rows (ascending token order):
 *                    1. release: every row about to be written drops its
 *                       reference; a slot that no token refers to is free;
 *                    2. scan: within each scan segment of seg_len consecutive
 *                       tokens (segment floor(i / seg_len)) the first written
 *                       row becomes the reference; a later row becomes the new
 *                       reference when sim(x, r) <= tau, else it is stored as
 *                       the int8 residual x - r.  sim = <x,r> / (sqrt(<x,x>)
 *                       sqrt(<r,r>)) in fp32, the sums in the canonical order of
 *                       the drift score, 0 when a norm is 0;
 *                    3. allocation: new references in ascending token order
 *                       take the free slots in ascending slot order; a
 *                       reference that finds no free slot is not created and
 *                       its whole run is stored as plain int8 (ref = -1);
 *                    4. store: a reference copies its row into its slot with
 *                       q = 0, s = 0; a residual is quantised by the int8 rule
 *                       of echo_cache_quant; refcount[slot] counts the tokens
 *                       whose entry names the slot.
 *                    The paper gives neither tau, the scan order nor the pool
 *                    size; seg_len = W' makes a segment one spatial row of a
 *                    latent frame ("adjacent latents").
 * All buffers are device memory owned by the caller, 16-byte aligned. */
typedef enum { ECHO_CACHE_INT8 = 0, ECHO_CACHE_BF16 = 1, ECHO_CACHE_REF = 2 } echo_cache_kind;

typedef struct {
    int32_t kind;       /* echo_cache_kind */
    int32_t NT;         /* tokens */
    int32_t D;          /* values per token, multiple of 16 */
    int8_t *q;          /* INT8, REF: int8 [NT, D] codes (REF: of the residual) */
    float *scale;       /* INT8, REF: f32 [NT] */
    void *full;         /* BF16: bf16 [NT, D] */
    int32_t *ref;       /* REF: int32 [NT] pool slot of each token's reference, -1 = none */
    void *pool;         /* REF: bf16 [R_cap, D] reference rows */
    int32_t *refcount;  /* REF: int32 [R_cap], 0 = free slot */
    int32_t R_cap;      /* REF: pool slots, >= 0 (0: every row plain int8) */
    int32_t seg_len;    /* REF: tokens per scan segment, >= 1 */
    float tau;          /* REF: similarity threshold */
} echo_cache;

/* Sets every entry of c to the empty state (q = 0, scale = 0, full = 0,
 * ref = -1, refcount = 0): every token then reconstructs to 0.
 * Errors: INVALID_ARG (descriptor), CUDA. */
echo_status echo_cache_reset(const echo_cache *c, echo_stream_t stream);

/* Bytes of device workspace echo_cache_write needs for n_rows rows (0 for
 * INT8 and BF16). */
size_t echo_cache_write_workspace_size(const echo_cache *c, int32_t n_rows);

/* Writes src (bf16 [n_rows, D], device) into the cache at rows (int32
 * [n_rows], device, ascending and distinct), by the rules of c's form.
 * Errors: INVALID_ARG, SHAPE, WORKSPACE, CUDA; a non-finite row sets the
 * NONFINITE device flag (INT8, REF: as echo_cache_quant). */
echo_status echo_cache_write(const echo_cache *c, const void *src, const int32_t *rows,
                             int32_t n_rows, void *workspace, size_t ws_bytes,
                             echo_stream_t stream);

/* dst[j] = the bf16 reconstruction c of token rows[j] (rows NULL: j), dst bf16
 * [n_rows, D] device.  Errors: INVALID_ARG, SHAPE, CUDA. */
echo_status echo_cache_read(const echo_cache *c, const int32_t *rows, int32_t n_rows, void *dst,
                            echo_stream_t stream);

/* REF only: out[0] = live references (slots with refcount > 0), out[1] = 1 +
 * the highest live slot (the pool rows a caller needs to keep); out int32[2]
 * device.  Errors: INVALID_ARG, CUDA. */
echo_status echo_cache_stats(const echo_cache *c, int32_t *out, echo_stream_t stream);

/* echo_select with the drift taken against the fp32 reconstruction of any
 * cache form: INT8 float(q) s, BF16 the row, REF r + float(q) s (no bf16
 * rounding).  Every other argument as echo_select. */
echo_status echo_select_cache(const void *x, echo_dtype xt, const echo_cache *c,
                              const float *seg_energy, int32_t T, int32_t N, int32_t ratio_num,
                              int32_t ratio_den, const echo_select_params *p, int32_t *idx,
                              int32_t *K_out, float *scores, void *workspace, size_t ws_bytes,
                              echo_stream_t stream);

/* Workspace of echo_block_step_cache: echo_workspace_size(dims, K_max) plus
 * the cache write's. */
size_t echo_block_step_cache_workspace_size(const echo_block_dims *dims, int32_t K_max,
                                            const echo_cache *c);

/* echo_block_step with any cache form: inactive rows take the bf16
 * reconstruction of the cache as it was on entry, and the active rows are
 * written with echo_cache_write's rules.  c->NT = T N and c->D = D. */
echo_status echo_block_step_cache(const echo_block_weights *w, const echo_block_dims *dims,
                                  const void *x, const int32_t *idx, int32_t K,
                                  const echo_cache *c, void *y, void *workspace, size_t ws_bytes,
                                  echo_stream_t stream);

/* ---- ablation selections (Sec. 4, Table 2: "Uniform" and "Random" in place
 *      of the energy-guided anchor selection); no energy and no drift ---- */

/* K = ceil(ratio_num T N / ratio_den) tokens evenly spaced over the token
 * order: idx[j] = floor(j T N / K), ascending and distinct.  idx int32 [K]
 * device, 16-byte aligned; *K_out (host) = K.  Errors: INVALID_ARG, SHAPE, CUDA. */
echo_status echo_select_uniform(int32_t T, int32_t N, int32_t ratio_num, int32_t ratio_den,
                                int32_t *idx, int32_t *K_out, echo_stream_t stream);

/* The K = ceil(ratio_num T N / ratio_den) tokens with the largest keys (key
 * descending, index ascending), as an ascending index list.  keys f32 [T N]
 * device, drawn by the caller (independent uniform keys give a uniformly
 * random K-subset); finite values.  idx int32 [K] device.  *K_out (host) = K.
 * Errors: INVALID_ARG, SHAPE, CUDA. */
echo_status echo_select_random(const float *keys, int32_t T, int32_t N, int32_t ratio_num,
                               int32_t ratio_den, int32_t *idx, int32_t *K_out,
                               echo_stream_t stream);

/* ---- step-level adaptive update rate (Sec. 3.3, with Eq. 1 of Sec. 3.1) ---- */

/* Parameters of r_t = clip(r_min + alpha * Delta-hat_t, r_min, r_max); the
 * paper gives none of the values (0 <= r_min <= r_max <= 1, alpha >= 0). */
typedef struct {
    double r_min;
    double r_max;
    double alpha;
} echo_rate_params;

/* Bytes of device workspace echo_step_delta needs (a fixed 9.5 KiB). */
size_t echo_step_delta_workspace_size(int64_t n);

/* Eq. 1 on two consecutive step outputs h_prev = h_t, h_cur = h_{t+1}:
 *   out[1] = sum_i |h_prev[i] - h_cur[i]|,  out[2] = sum_i |h_cur[i]|,
 *   out[0] = Delta = out[1] / (out[2] + xi),  all fp64.
 *   h_prev, h_cur: n elements of dtype ht (bf16 or f32), device, 16-byte
 *   aligned (may be NULL when n = 0); n >= 0 (n = 0 gives 0).  out: device double[3], written on the
 *   stream.  workspace >= echo_step_delta_workspace_size(n) bytes, 16-byte
 *   aligned, device, contents ignored.  Each element's difference and absolute
 *   value are taken in fp32; the sums are compensated, so their relative error
 *   is a few units of 2^-24; the order of summation depends on n only, so equal
 *   inputs give equal bits on every run.
 * Errors: INVALID_ARG (null, misaligned, xi <= 0), SHAPE (n < 0), WORKSPACE,
 * CUDA; a non-finite Delta sets the NONFINITE device flag. */
echo_status echo_step_delta(const void *h_prev, const void *h_cur, echo_dtype ht, int64_t n,
                            double xi, double *out, void *workspace, size_t ws_bytes,
                            echo_stream_t stream);

/* Host function (no GPU work): the step's update rate and budget from Eq. 1's
 * step-level change, Delta-hat = delta / delta_ref (0 when delta_ref == 0):
 *   *rate = min(max(r_min + alpha * Delta-hat, r_min), r_max)
 *   *K    = min(max(ceil(*rate * NT), 0), NT)   (k_t = ceil(N r_t), one global budget)
 * every operation in fp64 with one rounding each, in the order written.
 * rate may be NULL.  Errors: INVALID_ARG (parameters), SHAPE (NT < 0),
 * NONFINITE (delta or delta_ref negative or not finite). */
echo_status echo_update_rate(double delta, double delta_ref, const echo_rate_params *p,
                             int32_t NT, double *rate, int32_t *K);

/* Bytes of workspace echo_block_step needs for dims and up to K_max active
 * tokens (also enough for echo_precompute_cross_kv). */
size_t echo_workspace_size(const echo_block_dims *dims, int32_t K_max);

/* Cross-attention keys and values of the audio condition tokens, once per
 * block and generation (the condition does not change across steps):
 *   KVc[:, 0:D] = cond Wkc^T + bkc,  KVc[:, D:2D] = cond Wvc^T + bvc.
 *   cond bf16 [Lc, D]; Wkvc bf16 [2D, D] (W_kc over W_vc); bkvc bf16 [2D];
 *   KVc bf16 [Lc, 2D] out.  Errors: INVALID_ARG, SHAPE, CUDA. */
echo_status echo_precompute_cross_kv(const void *cond, const void *Wkvc,
                                     const void *bkvc, int32_t Lc, int32_t D,
                                     void *KVc, echo_stream_t stream);

/* Sec. 3.3 "Fine-grained latent-level caching" for one layer and one step:
 *   n1 = LN(x) (all NT rows; LN: zero mean, unit variance, eps 1e-6, no affine)
 *   K, V = n1 Wk^T + bk, n1 Wv^T + bv        (all latents)
 *   Q'   = n1[idx] Wq^T + bq                  (active latents only)
 *   h1   = x[idx] + MHA(Q', K, V) Wo^T + bo
 *   h2   = h1 + MHA(LN(h1) Wqc^T + bqc, Kc, Vc) Woc^T + boc
 *   y_act = h2 + GELU_tanh(LN(h2) W1^T + b1) W2^T + b2
 *   cache[idx[j]] = int8 quantisation of bf16(y_act[j])   (Sec. 3.4)
 *   y[i] = bf16(y_act[j]) if i == idx[j], else bf16(float(q_i) * s_i) from
 *   the cache as it was on entry (mask fusion, Sec. 3.3).
 *   x        bf16 [NT, D]; idx int32 [K] ascending, distinct, < NT (as from
 *            echo_select); 0 <= K <= NT (K = 0 returns the reconstructed cache,
 *            K = NT is the full step).
 *   cache_q  int8 [NT, D], cache_scale f32 [NT], updated in place at idx.
 *   y        bf16 [NT, D] out; may alias x.
 *   workspace >= echo_workspace_size(dims, K) bytes, 256-byte aligned.
 * Errors: INVALID_ARG, SHAPE, WORKSPACE, CUDA; NONFINITE/TIMEOUT device flags. */
echo_status echo_block_step(const echo_block_weights *w, const echo_block_dims *dims,
                            const void *x, const int32_t *idx, int32_t K,
                            int8_t *cache_q, float *cache_scale, void *y,
                            void *workspace, size_t ws_bytes, echo_stream_t stream);

/* echo_block_step with the K/V of every token kept in a caller-owned buffer
 * across steps, recomputed only for the tokens whose layer input changed.
 * Sec. 3.3 takes K and V from the complete latent set at every step; a token's
 * K/V row is a function of that token's layer input alone (row-wise layer norm
 * and a GEMM whose reduction order per output row is fixed), so a row whose
 * input did not change since it was computed is reused bit for bit.  In a
 * stack, a token's input to layer l >= 1 changes between two steps only if the
 * token was refreshed at layer l - 1 in either of them (fresh value one step,
 * the reconstruction from the int8 cache the next); layer 0's input changes
 * everywhere.  The results equal echo_block_step's on the same x, bit for bit,
 * as long as the rows passed cover every row of x that differs from the input
 * kv was computed from.
 *   kv       bf16 [NT, 2D], device, 16-byte aligned: row i holds K_i | V_i.
 *   kv_valid 0: kv's contents are ignored; K/V of every row are computed from x
 *            (as echo_block_step does) and left in kv.  Non-zero: kv holds K/V
 *            of an earlier input of this layer that differs from x at most at
 *            the rows rows_a[0..n_a) and rows_b[0..n_b); only those are
 *            recomputed (a row in both lists, or twice in one, is computed
 *            again, to the same bits).  rows_a, rows_b int32 device arrays,
 *            16-byte aligned, entries < NT; NULL when empty.
 *   With K = 0 the block is skipped (y = reconstructed cache) but kv is still
 *   brought up to date.  Other arguments as for echo_block_step.
 *   workspace >= echo_workspace_size_kv(dims, K, n_a + n_b) bytes, 256-byte
 *   aligned.
 * The caller owns kv (NT x 2D x 2 bytes per layer: 671 MB for the
 * 32760-token, D 5120 block) and decides which rows changed.
 * Errors: INVALID_ARG, SHAPE, WORKSPACE, CUDA; NONFINITE/TIMEOUT device flags. */
echo_status echo_block_step_kv(const echo_block_weights *w, const echo_block_dims *dims,
                               const void *x, const int32_t *idx, int32_t K, void *kv,
                               int32_t kv_valid, const int32_t *rows_a, int32_t n_a,
                               const int32_t *rows_b, int32_t n_b, int8_t *cache_q,
                               float *cache_scale, void *y, void *workspace, size_t ws_bytes,
                               echo_stream_t stream);

/* Bytes of workspace echo_block_step_kv needs for up to K_max active tokens and
 * up to n_rows_max recomputed rows (n_a + n_b); also enough with kv_valid = 0. */
size_t echo_workspace_size_kv(const echo_block_dims *dims, int32_t K_max, int32_t n_rows_max);

/* Sec. 3.4, int8 per-token symmetric quantisation:
 *   q[rows[j]], scale[rows[j]] = Q(src[j]) for j < n_rows (rows NULL: j),
 *   Q(v): a = max|v|; a == 0 -> s = 0, q = 0; else s = a / 127,
 *   inv = 127 / a, q = clamp(round_half_even(v * inv), -127, 127), fp32.
 *   src [n_rows, D] of dtype st; rows int32 [n_rows] distinct or NULL.
 * D multiple of 8.  A non-finite amax writes q = 0, s = amax and sets the
 * NONFINITE device flag.  Errors: INVALID_ARG, SHAPE, CUDA. */
echo_status echo_cache_quant(const void *src, echo_dtype st, const int32_t *rows,
                             int32_t n_rows, int32_t D, int8_t *q, float *scale,
                             echo_stream_t stream);

/* Sec. 3.4 reconstruction converted back to the compute precision:
 *   dst[j] = cast(float(q[r]) * scale[r]), r = rows ? rows[j] : j, the product
 *   in fp32 and the cast round-to-nearest-even (dt ECHO_BF16) or exact (ECHO_F32).
 *   dst [n_rows, D].  D multiple of 16.  Errors: INVALID_ARG, SHAPE, CUDA. */
echo_status echo_cache_dequant(const int8_t *q, const float *scale, const int32_t *rows,
                               int32_t n_rows, int32_t D, void *dst, echo_dtype dt,
                               echo_stream_t stream);

/* ---- single kernels of echo_block_step, exported so that each can be
 *      checked and timed on its own ---- */

/* out = act(A W^T + bias) + resid: one tcgen05 bf16 GEMM (fp32 accumulate).
 *   A bf16 [M, Kd] (row stride lda elements), W bf16 [N, Kd], bias bf16 [N]
 *   or NULL; act 0 = none, 1 = GELU (tanh form).
 *   resid: NULL, bf16 [*, N] read at row resid_rows[m] (or m if resid_rows is
 *   NULL) when resid_t == ECHO_BF16, or f32 [M, N] when ECHO_F32.
 *   out [M, N] (row stride ldo elements) of dtype out_t.
 * Kd, N multiples of 64; lda, ldo multiples of 8.  Errors: INVALID_ARG, SHAPE, CUDA. */
echo_status echo_linear(const void *A, int64_t lda, int32_t M, int32_t Kd,
                        const void *W, const void *bias, int32_t N, int32_t act,
                        const void *resid, echo_dtype resid_t, const int32_t *resid_rows,
                        void *out, int64_t ldo, echo_dtype out_t, echo_stream_t stream);

/* O[m, h d + e] = sum_j softmax_j(Q_h[m] . K_h[j] / sqrt(d)) V_h[j, e]:
 *   Q bf16 [M, ldq], K and V bf16 [L, ldkv] (head h at columns h d .. h d + d - 1),
 *   O bf16 [M, ldo].  d in {64, 128}; strides multiples of 8.
 * Errors: INVALID_ARG, SHAPE, CUDA. */
echo_status echo_attention(const void *Q, int64_t ldq, const void *K, const void *V,
                           int64_t ldkv, int32_t M, int32_t L, int32_t H, int32_t d,
                           void *O, int64_t ldo, echo_stream_t stream);

/* out[j] = LN(in[rows ? rows[j] : j]) over D columns, eps 1e-6, no affine.
 *   in [*, D] of dtype in_t, out bf16 [n_rows, D].  D multiple of 8.
 * Errors: INVALID_ARG, SHAPE, CUDA. */
echo_status echo_layernorm(const void *in, echo_dtype in_t, const int32_t *rows,
                           int32_t n_rows, int32_t D, void *out, echo_stream_t stream);

/* ---- failure detection (no counterpart in the paper) ---- */

/* Runs the bounded-wait path every library kernel uses on one barrier that
 * nothing completes: one thread waits limit_ns (1 us .. 2 s), gives up, sets
 * the device flag ECHO_ERR_TIMEOUT and returns, leaving the context usable.
 * The next echo_get_device_error reports (and clears) it.  For tests of the
 * timeout handling.  Errors: INVALID_ARG (limit), CUDA. */
echo_status echo_check_timeout_path(int64_t limit_ns, echo_stream_t stream);

/* ---- instrumentation (no counterpart in the paper: measurement only) ---- */

/* Kernel kinds reported by the profiler. */
typedef enum {
    ECHO_K_ENERGY = 0, ECHO_K_DRIFT = 1, ECHO_K_TOPK = 2, ECHO_K_ROWMAP = 3,
    ECHO_K_LAYERNORM = 4, ECHO_K_GEMM = 5, ECHO_K_ATTENTION = 6, ECHO_K_QUANT = 7,
    ECHO_K_DEQUANT = 8, ECHO_K_MERGE = 9, ECHO_K_STEP_DELTA = 10, ECHO_K_UNIFORM = 11,
    ECHO_K_REF_SCAN = 12, ECHO_K_REF_ALLOC = 13, ECHO_K_REF_STORE = 14, ECHO_K_CACHE_COPY = 15,
    ECHO_K_MERGE_QUANT = 16, ECHO_K_COUNT = 17
} echo_kernel_kind;

/* Number of kernels this library has launched in this process (all devices). */
uint64_t echo_launch_count(void);

/* on != 0: from now on bracket every kernel launch with a pair of CUDA events
 * recorded on the launch's own stream (up to 65536 launches are kept).
 * on == 0: stop recording.  Recorded launches stay until read. */
echo_status echo_profile_enable(int32_t on);

/* Synchronises every recorded launch, copies up to `max` records (kind, the
 * launch's shape m, n, k as described below, and its device time in ms) into
 * the host arrays, clears the record list and returns the number copied (or
 * -1 on a CUDA error).  Shapes: GEMM (M, N, Kd); ATTENTION (M queries, L keys,
 * H * d); DRIFT (NT, D, 0); TOPK (NT, K, 0); LAYERNORM (rows, D, input element
 * bytes); QUANT, DEQUANT, MERGE (rows, D, 0); ENERGY (T, frames, n_fft); STEP_DELTA (n, element bytes, 0)
 * for the reduction and (0, 0, blocks) for its final combine; UNIFORM (NT, K, 0);
 * REF_SCAN, REF_ALLOC, REF_STORE, CACHE_COPY (rows, D, 0); MERGE_QUANT (NT, D, K active
 * rows). */
int32_t echo_profile_read(int32_t max, int32_t *kinds, int64_t *m, int64_t *n, int64_t *k,
                          float *ms);

/* Name of a kernel kind ("gemm_tcgen05", ...).  Never NULL. */
const char *echo_kernel_name(int32_t kind);

#ifdef __cplusplus
}
#endif

#endif /* ECHOCACHE_H */
