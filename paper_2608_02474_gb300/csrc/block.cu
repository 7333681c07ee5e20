// One cached layer step on the active latents (Sec. 3.3 "Fine-grained
// latent-level caching", Sec. 3.4 for the cache write), as a fixed sequence of
// stream-ordered kernels over a caller-owned workspace:
//
//   rowmap      token -> position in idx (or -1)
//   LN          n1 = LN(x), all NT rows; the active rows are also written to
//               na = LN(x[idx]) through the row map  ("select active latents")
//   GEMM        KV = n1 [Wk; Wv]^T + [bk; bv]          (K, V over all latents)
//   GEMM        Q' = na Wq^T + bq
//   attention   att = MHA(Q', K, V)
//   GEMM        h1 = att Wo^T + bo + x[idx]             (fp32)
//   LN, GEMM    Qc = LN(h1) Wqc^T + bqc
//   attention   att = MHA(Qc, Kc, Vc)
//   GEMM        h2 = att Woc^T + boc + h1               (fp32)
//   LN, GEMM    u = GELU(LN(h2) W1^T + b1)
//   GEMM        y[idx] = u W2^T + b2 + h2               (bf16, stored at the
//               active tokens' rows of y; the epilogue also folds max |y| per
//               row for the quantiser)
//   merge+quant y = reconstructed cache at every other row, and
//               cache[idx] = Q(y[idx]), in one pass over the rows
#include "common.cuh"
#include "internal.h"

namespace {

size_t al(size_t b) { return (b + 255) & ~(size_t)255; }

struct Layout {
    size_t rowmap, rows, n1, kv, na, qa, att, h1, h2, u, yact, amax, total;
};

// n_ln: rows whose layer norm and K/V are computed (-1: every row); n_rows:
// entries of the list of those rows; kv_in_ws: K/V of every row live in the
// workspace (else in the caller's buffer)
Layout layout(const echo_block_dims &d, int64_t K, int64_t n_ln = -1, int64_t n_rows = 0,
              bool kv_in_ws = true) {
    const int64_t NT = (int64_t)d.T * d.N;
    if (n_ln < 0) n_ln = NT;
    Layout L;
    size_t o = 0;
    L.rowmap = o; o += al(sizeof(int32_t) * NT);
    L.rows = o;   o += al(sizeof(int32_t) * n_rows);
    L.n1 = o;     o += al(2 * (size_t)n_ln * d.D);
    L.kv = o;     o += kv_in_ws ? al(2 * (size_t)NT * 2 * d.D) : 0;
    L.na = o;     o += al(2 * (size_t)K * d.D);
    L.qa = o;     o += al(2 * (size_t)K * d.D);
    L.att = o;    o += al(2 * (size_t)K * d.D);
    L.h1 = o;     o += al(4 * (size_t)K * d.D);
    L.h2 = o;     o += al(4 * (size_t)K * d.D);
    L.u = o;      o += al(2 * (size_t)K * d.F);
    L.yact = o;   o += al(2 * (size_t)K * d.D);
    L.amax = o;   o += al(4 * (size_t)K);
    L.total = o;
    return L;
}

bool dims_ok(const echo_block_dims *d) {
    if (!d) return false;
    if (d->T < 1 || d->N < 1 || d->D < 64 || d->D % 64 || d->F < 64 || d->F % 64 || d->Lc < 1)
        return false;
    if ((d->d != 64 && d->d != 128) || d->H < 1 || (int64_t)d->H * d->d != d->D) return false;
    if (d->D > 8192) return false;
    if ((int64_t)d->T * d->N > (int64_t)INT32_MAX / 2) return false;
    return true;
}

}  // namespace

extern "C" size_t echo_workspace_size(const echo_block_dims *dims, int32_t K_max) {
    if (!dims_ok(dims) || K_max < 0) return 0;
    return layout(*dims, K_max).total;
}

extern "C" echo_status echo_precompute_cross_kv(const void *cond, const void *Wkvc,
                                                const void *bkvc, int32_t Lc, int32_t D,
                                                void *KVc, echo_stream_t stream) {
    return echo_linear(cond, D, Lc, D, Wkvc, bkvc, 2 * D, 0, nullptr, ECHO_BF16, nullptr, KVc,
                       2 * (int64_t)D, ECHO_BF16, stream);
}

namespace {

// argument checks shared by echo_block_step and echo_block_step_cache
echo_status check_block(const echo_block_weights *w, const echo_block_dims *dims, const void *x,
                        const int32_t *idx, int32_t K, const void *y, const void *workspace) {
    using namespace echo;
    if (!w || !dims || !x || !y || !workspace) return ECHO_ERR_INVALID_ARG;
    if (!dims_ok(dims)) return ECHO_ERR_SHAPE;
    const int NT = dims->T * dims->N;
    if (K < 0 || K > NT) return ECHO_ERR_SHAPE;
    if (K > 0 && !idx) return ECHO_ERR_INVALID_ARG;
    const void *ptrs[] = {w->Wq, w->bq, w->Wkv, w->bkv, w->Wo, w->bo, w->Wqc, w->bqc,
                          w->Woc, w->boc, w->W1, w->b1, w->W2, w->b2, w->KVc};
    for (const void *p : ptrs)
        if (!p || !aligned16(p)) return ECHO_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(y) || (idx && !aligned16(idx)) ||
        (reinterpret_cast<uintptr_t>(workspace) & 255u))
        return ECHO_ERR_INVALID_ARG;
    return ECHO_OK;
}

// K/V of the rows listed in rows_a and rows_b (either may be empty; a row in
// both is computed twice, to the same bits): the list [rows_a; rows_b] at
// ws + L.rows, the rows' layer norm into ws + L.n1 (compact, in that order),
// their K/V scattered into kv.
echo_status refresh_kv_rows(const echo_block_weights *w, const echo_block_dims &d,
                            const void *x, const int32_t *rows_a, int32_t n_a,
                            const int32_t *rows_b, int32_t n_b, void *kv, uint8_t *ws,
                            const Layout &L, cudaStream_t st) {
    using namespace echo;
    const int D = d.D;
    int32_t *rows = reinterpret_cast<int32_t *>(ws + L.rows);
    const int n = n_a + n_b;
    if (n == 0) return ECHO_OK;
    if (n_a > 0 && cudaMemcpyAsync(rows, rows_a, sizeof(int32_t) * (size_t)n_a,
                                   cudaMemcpyDeviceToDevice, st) != cudaSuccess)
        return ECHO_ERR_CUDA;
    if (n_b > 0 && cudaMemcpyAsync(rows + n_a, rows_b, sizeof(int32_t) * (size_t)n_b,
                                   cudaMemcpyDeviceToDevice, st) != cudaSuccess)
        return ECHO_ERR_CUDA;
    launch_layernorm(x, ECHO_BF16, rows, n, D, ws + L.n1, st);
    LinearArgs a{ws + L.n1, D, n, D, w->Wkv, w->bkv, 2 * D, 0, nullptr, ECHO_BF16, nullptr, kv,
                 2 * (int64_t)D, ECHO_BF16};
    a.out_rows = rows;
    return launch_linear(a, st);
}

// K/V of every row into kv (layer norm of every row through ws + L.n1)
echo_status refresh_kv_all(const echo_block_weights *w, const echo_block_dims &d, const void *x,
                           void *kv, uint8_t *ws, const Layout &L, cudaStream_t st) {
    using namespace echo;
    const int D = d.D, NT = d.T * d.N;
    launch_layernorm(x, ECHO_BF16, nullptr, NT, D, ws + L.n1, st);
    return launch_linear({ws + L.n1, D, NT, D, w->Wkv, w->bkv, 2 * D, 0, nullptr, ECHO_BF16,
                          nullptr, kv, 2 * (int64_t)D, ECHO_BF16}, st);
}

// rowmap and the block on the K active rows: y_act (bf16 [K, D]) at ws + L.yact,
// or, with y_scatter, straight into rows idx[j] of y_scatter.  With kv_ext the
// K/V of every row come from (and, unless kv_ready, go to) the caller's buffer;
// kv_ready: it is already up to date, and only the active rows are normalised
// (gathered into na) for Q'.
echo_status run_active(const echo_block_weights *w, const echo_block_dims &d, const void *x,
                       const int32_t *idx, int32_t K, uint8_t *ws, const Layout &L,
                       cudaStream_t st, void *y_scatter = nullptr, void *kv_ext = nullptr,
                       bool kv_ready = false) {
    using namespace echo;
    const int NT = d.T * d.N;
    int32_t *rowmap = reinterpret_cast<int32_t *>(ws + L.rowmap);
    void *n1 = ws + L.n1, *kv = kv_ext ? kv_ext : ws + L.kv, *na = ws + L.na, *qa = ws + L.qa;
    void *att = ws + L.att;
    void *h1 = ws + L.h1, *h2 = ws + L.h2, *u = ws + L.u, *yact = ws + L.yact;
    const int D = d.D;
    const __nv_bfloat16 *kvb = static_cast<const __nv_bfloat16 *>(kv);
    const __nv_bfloat16 *kvc = static_cast<const __nv_bfloat16 *>(w->KVc);
    echo_status s = ECHO_OK;
    // the row map, and max |y_act| per row cleared for the FFN-down epilogue
    uint32_t *amax = reinterpret_cast<uint32_t *>(ws + L.amax);
    launch_rowmap(idx, K, NT, rowmap, amax, K, st);
    if (K > 0) {
        if (kv_ready) {
            launch_layernorm(x, ECHO_BF16, idx, K, D, na, st);   // the active rows only
        } else {
            // LN over every latent; the active rows also land in na, gathered
            launch_layernorm_scatter(x, NT, D, n1, rowmap, na, st);
            s = launch_linear({n1, D, NT, D, w->Wkv, w->bkv, 2 * D, 0, nullptr, ECHO_BF16, nullptr,
                               kv, 2 * (int64_t)D, ECHO_BF16}, st);
            if (s != ECHO_OK) return s;
        }
        s = launch_linear({na, D, K, D, w->Wq, w->bq, D, 0, nullptr, ECHO_BF16, nullptr, qa, D,
                           ECHO_BF16}, st);
        if (s != ECHO_OK) return s;
        s = launch_attention(qa, D, kvb, kvb + D, 2 * (int64_t)D, K, NT, d.H, d.d, att, D, st);
        if (s != ECHO_OK) return s;
        s = launch_linear({att, D, K, D, w->Wo, w->bo, D, 0, x, ECHO_BF16, idx, h1, D, ECHO_F32}, st);
        if (s != ECHO_OK) return s;
        launch_layernorm(h1, ECHO_F32, nullptr, K, D, na, st);
        s = launch_linear({na, D, K, D, w->Wqc, w->bqc, D, 0, nullptr, ECHO_BF16, nullptr, qa, D,
                           ECHO_BF16}, st);
        if (s != ECHO_OK) return s;
        s = launch_attention(qa, D, kvc, kvc + D, 2 * (int64_t)D, K, d.Lc, d.H, d.d, att, D, st);
        if (s != ECHO_OK) return s;
        s = launch_linear({att, D, K, D, w->Woc, w->boc, D, 0, h1, ECHO_F32, nullptr, h2, D,
                           ECHO_F32}, st);
        if (s != ECHO_OK) return s;
        launch_layernorm(h2, ECHO_F32, nullptr, K, D, na, st);
        s = launch_linear({na, D, K, D, w->W1, w->b1, d.F, 1, nullptr, ECHO_BF16, nullptr, u, d.F,
                           ECHO_BF16}, st);
        if (s != ECHO_OK) return s;
        // the FFN-down epilogue also records max |y_act| per row for the cache write
        LinearArgs down{u, d.F, K, d.F, w->W2, w->b2, D, 0, h2, ECHO_F32, nullptr,
                        y_scatter ? y_scatter : yact, D, ECHO_BF16};
        down.row_amax = amax;
        if (y_scatter) down.out_rows = idx;
        s = launch_linear(down, st);
        if (s != ECHO_OK) return s;
    }
    return last_launch_status();
}

}  // namespace

extern "C" echo_status echo_block_step(const echo_block_weights *w, const echo_block_dims *dims,
                                       const void *x, const int32_t *idx, int32_t K,
                                       int8_t *cache_q, float *cache_scale, void *y,
                                       void *workspace, size_t ws_bytes, echo_stream_t stream) {
    using namespace echo;
    echo_status s = check_block(w, dims, x, idx, K, y, workspace);
    if (s != ECHO_OK) return s;
    if (!cache_q || !cache_scale) return ECHO_ERR_INVALID_ARG;
    if (!aligned16(cache_q) || !aligned16(cache_scale)) return ECHO_ERR_INVALID_ARG;
    const echo_block_dims d = *dims;
    const int NT = d.T * d.N;
    const Layout L = layout(d, K);
    if (ws_bytes < L.total) return ECHO_ERR_WORKSPACE;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    // the FFN-down epilogue stores the active rows at their token positions in
    // y (every read of x is done by then, so y may alias x)
    s = run_active(w, d, x, idx, K, ws, L, st, y);
    if (s != ECHO_OK) return s;
    const int32_t *rowmap = reinterpret_cast<const int32_t *>(ws + L.rowmap);
    // one pass over every row: an inactive row is reconstructed from the cache
    // into y, an active row of y is quantised into the cache (disjoint rows)
    launch_merge_quant(cache_q, cache_scale, rowmap, reinterpret_cast<const uint32_t *>(ws + L.amax),
                       NT, d.D, K, y, st);
    return last_launch_status();
}

extern "C" size_t echo_workspace_size_kv(const echo_block_dims *dims, int32_t K_max,
                                         int32_t n_rows_max) {
    if (!dims_ok(dims) || K_max < 0 || n_rows_max < 0) return 0;
    const size_t full = layout(*dims, K_max, -1, 0, false).total;
    const size_t part = layout(*dims, K_max, n_rows_max, n_rows_max, false).total;
    return full > part ? full : part;
}

extern "C" echo_status echo_block_step_kv(const echo_block_weights *w, const echo_block_dims *dims,
                                          const void *x, const int32_t *idx, int32_t K, void *kv,
                                          int32_t kv_valid, const int32_t *rows_a, int32_t n_a,
                                          const int32_t *rows_b, int32_t n_b, int8_t *cache_q,
                                          float *cache_scale, void *y, void *workspace,
                                          size_t ws_bytes, echo_stream_t stream) {
    using namespace echo;
    echo_status s = check_block(w, dims, x, idx, K, y, workspace);
    if (s != ECHO_OK) return s;
    if (!cache_q || !cache_scale || !kv) return ECHO_ERR_INVALID_ARG;
    if (!aligned16(cache_q) || !aligned16(cache_scale) || !aligned16(kv)) return ECHO_ERR_INVALID_ARG;
    const echo_block_dims d = *dims;
    const int NT = d.T * d.N;
    if (kv_valid) {
        if (n_a < 0 || n_b < 0 || (int64_t)n_a + n_b > (int64_t)INT32_MAX / 2) return ECHO_ERR_SHAPE;
        if ((n_a > 0 && (!rows_a || !aligned16(rows_a))) || (n_b > 0 && (!rows_b || !aligned16(rows_b))))
            return ECHO_ERR_INVALID_ARG;
    }
    const Layout L = kv_valid ? layout(d, K, n_a + n_b, n_a + n_b, false)
                              : layout(d, K, -1, 0, false);
    if (ws_bytes < L.total) return ECHO_ERR_WORKSPACE;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    if (kv_valid) {
        s = refresh_kv_rows(w, d, x, rows_a, n_a, rows_b, n_b, kv, ws, L, st);
        if (s == ECHO_OK) s = run_active(w, d, x, idx, K, ws, L, st, y, kv, true);
    } else if (K > 0) {
        s = run_active(w, d, x, idx, K, ws, L, st, y, kv, false);
    } else {
        s = refresh_kv_all(w, d, x, kv, ws, L, st);
        if (s == ECHO_OK) s = run_active(w, d, x, idx, K, ws, L, st, y, kv, true);
    }
    if (s != ECHO_OK) return s;
    const int32_t *rowmap = reinterpret_cast<const int32_t *>(ws + L.rowmap);
    launch_merge_quant(cache_q, cache_scale, rowmap, reinterpret_cast<const uint32_t *>(ws + L.amax),
                       NT, d.D, K, y, st);
    return last_launch_status();
}

extern "C" size_t echo_block_step_cache_workspace_size(const echo_block_dims *dims, int32_t K_max,
                                                       const echo_cache *c) {
    if (!dims_ok(dims) || K_max < 0 || echo::cache_check(c) != ECHO_OK) return 0;
    return layout(*dims, K_max).total + echo::cache_write_ws(*c, K_max);
}

extern "C" echo_status echo_block_step_cache(const echo_block_weights *w,
                                             const echo_block_dims *dims, const void *x,
                                             const int32_t *idx, int32_t K, const echo_cache *c,
                                             void *y, void *workspace, size_t ws_bytes,
                                             echo_stream_t stream) {
    using namespace echo;
    echo_status s = check_block(w, dims, x, idx, K, y, workspace);
    if (s != ECHO_OK) return s;
    s = cache_check(c);
    if (s != ECHO_OK) return s;
    const echo_block_dims d = *dims;
    if (c->NT != d.T * d.N || c->D != d.D) return ECHO_ERR_SHAPE;
    const Layout L = layout(d, K);
    const size_t wbytes = cache_write_ws(*c, K);
    if (ws_bytes < L.total + wbytes) return ECHO_ERR_WORKSPACE;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    s = run_active(w, d, x, idx, K, ws, L, st);
    if (s != ECHO_OK) return s;
    const int32_t *rowmap = reinterpret_cast<const int32_t *>(ws + L.rowmap);
    // the merge reads the cache as it was on entry (the inactive rows and the
    // references they name, which the write neither releases nor reuses);
    // then the active rows are written
    launch_cache_merge(*c, rowmap, ws + L.yact, y, st);
    if (last_launch_status() != ECHO_OK) return ECHO_ERR_CUDA;
    if (K > 0) return launch_cache_write(*c, ws + L.yact, idx, K, ws + L.total, st);
    return ECHO_OK;
}
