// Host-side launchers shared between the translation units of the library.
// Every launcher assumes its arguments were validated by the public entry
// point that calls it and only enqueues work on `st`.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/echocache.h"

namespace echo {

// device error flag of the current device (api.cu)
int *device_error_ptr();
// true when the current device is sm_103 (checked once per device)
bool device_supported();
echo_status last_launch_status();

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Counts every kernel launch and, while profiling is on, brackets it with a
// pair of CUDA events on its stream (api.cu).  Construct right before the
// launch, destroy right after it.
class LaunchScope {
  public:
    LaunchScope(int kind, int64_t m, int64_t n, int64_t k, cudaStream_t st);
    ~LaunchScope();
    LaunchScope(const LaunchScope &) = delete;
    LaunchScope &operator=(const LaunchScope &) = delete;

  private:
    int slot_;
    cudaStream_t st_;
};

// tensor maps (api.cu): 2D bf16, row-major [rows, cols] with row stride ld
// (elements), box [box_rows, 64 columns], 128-byte swizzle.
bool make_tmap_bf16(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint64_t ld,
                    uint32_t box_rows);

// layernorm.cu
void launch_layernorm(const void *in, echo_dtype in_t, const int32_t *rows, int32_t n_rows,
                      int32_t D, void *out, cudaStream_t st);
// out = LN(in) for all n_rows bf16 rows; row i also goes to out2[map[i]] when map[i] >= 0
void launch_layernorm_scatter(const void *in, int32_t n_rows, int32_t D, void *out,
                              const int32_t *scatter_map, void *out2, cudaStream_t st);

// gemm.cu: out = act(A W^T + bias) + resid
struct LinearArgs {
    const void *A; int64_t lda; int32_t M; int32_t Kd;
    const void *W; const void *bias; int32_t N; int32_t act;
    const void *resid; echo_dtype resid_t; const int32_t *resid_rows;
    void *out; int64_t ldo; echo_dtype out_t;
    uint32_t *row_amax = nullptr;   // bf16 out with an fp32 residual only: max |out| per row
    const int32_t *out_rows = nullptr;   // output row m is stored at row out_rows[m]
};
echo_status launch_linear(const LinearArgs &a, cudaStream_t st);

// attention.cu
echo_status launch_attention(const void *Q, int64_t ldq, const void *K, const void *V, int64_t ldkv,
                             int32_t M, int32_t L, int32_t H, int32_t d, void *O, int64_t ldo,
                             cudaStream_t st);

// cache.cu
void launch_quant(const void *src, echo_dtype st_t, const int32_t *rows, int32_t n_rows,
                  int32_t D, int8_t *q, float *scale, cudaStream_t st);
void launch_dequant(const int8_t *q, const float *scale, const int32_t *rows, int32_t n_rows,
                    int32_t D, void *dst, echo_dtype dt, cudaStream_t st);
// rowmap[i] = position of token i in idx (ascending, distinct), else -1; also
// clears zero[0 .. n_zero)
void launch_rowmap(const int32_t *idx, int32_t K, int32_t NT, int32_t *rowmap, uint32_t *zero,
                   int32_t n_zero, cudaStream_t st);
void launch_dequant_merge(const int8_t *q, const float *scale, const int32_t *rowmap,
                          const void *y_act, int32_t NT, int32_t D, void *y, cudaStream_t st);
// y[i] = bf16(q[i] s[i]) for rowmap[i] < 0; every other row of y (already the
// fresh block output, max |y| per row in amax[rowmap[i]]) is quantised into
// q[i], s[i]: the merge and the int8 write of the block step in one pass
void launch_merge_quant(int8_t *q, float *scale, const int32_t *rowmap, const uint32_t *amax,
                        int32_t NT, int32_t D, int32_t K, void *y, cudaStream_t st);

// refcache.cu: cache forms other than plain int8 (and int8 through the same calls)
echo_status cache_check(const echo_cache *c);
size_t cache_write_ws(const echo_cache &c, int32_t n);
echo_status launch_cache_write(const echo_cache &c, const void *src, const int32_t *rows,
                               int32_t n, void *ws, cudaStream_t st);
void launch_cache_merge(const echo_cache &c, const int32_t *rowmap, const void *y_act, void *y,
                        cudaStream_t st);

}  // namespace echo
