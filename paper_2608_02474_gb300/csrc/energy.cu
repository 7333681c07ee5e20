// Audio segment energy (Sec. 3.3 "Cross-modal Saliency Anchors"): the audio is
// split evenly into T segments; each segment's frames (periodic Hann window,
// no centring) go through a radix-2 FFT in shared memory; the one-sided power
// P_k = c_k |X_k|^2 / n_fft is summed over the segment's frames per bin and then
// per linear band; energy = sqrt(sum of the bands).
//
// One CTA per segment, eight frame groups of 128 threads.  Each thread keeps
// the frame-summed power of its bins in registers, so the result does not
// depend on scheduling: groups are combined in a fixed order and bands are
// reduced by warps in a fixed order.
#include "common.cuh"
#include "internal.h"

namespace {

constexpr int kGroup = 128;           // threads per frame group
constexpr int kGroups = 8;            // frame groups per CTA
constexpr int kMaxBinsPerThread = 17; // (4096/2 + 1) / 128 rounded up

__global__ void __launch_bounds__(kGroup *kGroups)
segment_energy_kernel(const float *__restrict__ audio, int seg_len, int n_fft, int log2n, int hop,
                      int n_frames, int n_bands, float *__restrict__ band_out,
                      float *__restrict__ seg_out) {
    extern __shared__ float2 sm[];
    const int half = n_fft >> 1;
    const int n_bins = half + 1;
    float2 *tw = sm;                             // [half] twiddles exp(-2 pi i j / n)
    float2 *buf = sm + half;                     // [kGroups][n_fft]
    float *binsum = reinterpret_cast<float *>(buf + kGroups * n_fft);  // [kGroups][n_bins]

    const int tau = blockIdx.x;
    const int g = threadIdx.x / kGroup;
    const int t = threadIdx.x % kGroup;
    const float *seg = audio + (int64_t)tau * seg_len;
    float2 *a = buf + g * n_fft;

    for (int j = threadIdx.x; j < half; j += blockDim.x) {
        float s, c;
        sincospif((2.0f * j) / n_fft, &s, &c);
        tw[j] = make_float2(c, -s);
    }

    float acc[kMaxBinsPerThread];
#pragma unroll
    for (int i = 0; i < kMaxBinsPerThread; ++i) acc[i] = 0.f;

    const int rounds = (n_frames + kGroups - 1) / kGroups;
    for (int r = 0; r < rounds; ++r) {
        const int f = r * kGroups + g;
        const bool live = f < n_frames;
        const int off = f * hop;
        for (int n = t; n < n_fft; n += kGroup) {
            float v = 0.f;
            if (live && off + n < seg_len) {
                const float w = 0.5f - 0.5f * cospif((2.0f * n) / n_fft);
                v = seg[off + n] * w;
            }
            const int rev = __brev((unsigned)n) >> (32 - log2n);
            a[rev] = make_float2(v, 0.f);
        }
        __syncthreads();
        for (int s = 1; s <= log2n; ++s) {
            const int hs = 1 << (s - 1);
            const int tstep = n_fft >> s;
            for (int b = t; b < half; b += kGroup) {
                const int j = b & (hs - 1);
                const int i0 = ((b >> (s - 1)) << s) + j;
                const int i1 = i0 + hs;
                const float2 w = tw[j * tstep];
                const float2 u = a[i0], x = a[i1];
                const float2 v = make_float2(w.x * x.x - w.y * x.y, w.x * x.y + w.y * x.x);
                a[i0] = make_float2(u.x + v.x, u.y + v.y);
                a[i1] = make_float2(u.x - v.x, u.y - v.y);
            }
            __syncthreads();
        }
        if (live) {
#pragma unroll
            for (int i = 0; i < kMaxBinsPerThread; ++i) {
                const int k = t + i * kGroup;
                if (k < n_bins) {
                    const float2 X = a[k];
                    const float c = (k == 0 || k == half) ? 1.f : 2.f;
                    acc[i] += c * (X.x * X.x + X.y * X.y) / (float)n_fft;
                }
            }
        }
        __syncthreads();
    }

#pragma unroll
    for (int i = 0; i < kMaxBinsPerThread; ++i) {
        const int k = t + i * kGroup;
        if (k < n_bins) binsum[g * n_bins + k] = acc[i];
    }
    __syncthreads();
    for (int k = threadIdx.x; k < n_bins; k += blockDim.x) {
        float s = binsum[k];
        for (int gg = 1; gg < kGroups; ++gg) s += binsum[gg * n_bins + k];
        binsum[k] = s;
    }
    __syncthreads();
    float *bands = binsum + n_bins;  // reuse group 1's slot: [n_bands]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int b = warp; b < n_bands; b += blockDim.x >> 5) {
        const int lo = (n_bins * b) / n_bands, hi = (n_bins * (b + 1)) / n_bands;
        float s = 0.f;
        for (int k = lo + lane; k < hi; k += 32) s += binsum[k];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) {
            bands[b] = s;
            band_out[(int64_t)tau * n_bands + b] = s;
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        float e = 0.f;
        for (int b = 0; b < n_bands; ++b) e += bands[b];
        seg_out[tau] = sqrtf(e);
    }
}

}  // namespace

extern "C" echo_status echo_audio_energy(const float *audio, int64_t n_samples, int32_t T,
                                         int32_t n_fft, int32_t hop, int32_t n_bands,
                                         float *band_energy, float *seg_energy,
                                         echo_stream_t stream) {
    using namespace echo;
    if (!audio || !band_energy || !seg_energy) return ECHO_ERR_INVALID_ARG;
    if (!aligned16(audio) || !aligned16(band_energy) || !aligned16(seg_energy))
        return ECHO_ERR_INVALID_ARG;
    if (T < 1 || n_samples < T || hop < 1) return ECHO_ERR_SHAPE;
    if (n_fft < 64 || n_fft > 4096 || (n_fft & (n_fft - 1))) return ECHO_ERR_SHAPE;
    const int n_bins = n_fft / 2 + 1;
    if (n_bands < 1 || n_bands > n_bins) return ECHO_ERR_SHAPE;
    if (n_samples / T > (int64_t)INT32_MAX) return ECHO_ERR_SHAPE;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;

    const int seg_len = (int)(n_samples / T);
    const int n_frames = seg_len < n_fft ? 1 : (seg_len - n_fft) / hop + 1;
    int log2n = 0;
    while ((1 << log2n) < n_fft) ++log2n;
    const size_t smem = sizeof(float2) * (size_t)(n_fft / 2 + kGroups * n_fft) +
                        sizeof(float) * (size_t)kGroups * n_bins;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(segment_energy_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem) != cudaSuccess)
        return ECHO_ERR_CUDA;
    {
        LaunchScope ls(ECHO_K_ENERGY, T, n_frames, n_fft, st);
        segment_energy_kernel<<<T, kGroup * kGroups, smem, st>>>(
            audio, seg_len, n_fft, log2n, hop, n_frames, n_bands, band_energy, seg_energy);
    }
    return last_launch_status();
}
