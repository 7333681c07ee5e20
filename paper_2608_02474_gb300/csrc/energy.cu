// Audio segment energy (Sec. 3.3 "Cross-modal Saliency Anchors"): the audio is
// split evenly into T segments; each segment's frames (periodic Hann window,
// no centring) go through a radix-2 FFT in shared memory; the one-sided power
// P_k = c_k |X_k|^2 / n_fft is summed over the segment's frames per bin and then
// per linear band; energy = sqrt(sum of the bands).
//
// n_fft <= 512 takes the warp kernel below (two frames per complex FFT, the
// transform in registers and warp shuffles).  Larger transforms take the
// shared-memory kernel: one CTA per segment, eight frame groups of 128
// threads.  Each thread keeps
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

// ---------------------------------------------------------------------------
// n_fft = 32 R <= 512: one warp transforms two frames at once, no block-wide
// barrier inside the transform.  The two windowed real frames a and b of a
// segment are packed as z = a + i b and one complex N-point FFT is taken,
// N = R x 32 (Cooley-Tukey with N1 = R, N2 = 32): lane n2 holds z[32 n1 + n2]
// for n1 < R in registers (coalesced loads), takes the R-point DFT over n1 in
// registers (radix-2, decimation in frequency), multiplies by W_N^(n2 k1), and
// the 32-point DFT over n2 runs across the lanes (five xor-shuffle radix-2
// stages).  Lane l then holds Z[k1 + R k2] with k2 = bitrev5(l), k1 = bitrev_R(i)
// for its register i.  Because a and b are real, |A_k|^2 + |B_k|^2 =
// (|Z_k|^2 + |Z_{N-k}|^2) / 2, so the summed one-sided power of the two frames
// at bin k is (|Z_k|^2 + |Z_{N-k}|^2) / N for 0 < k < N/2 and |Z_k|^2 / N at
// k = 0 and N/2: every Z_k adds |Z_k|^2 / N to bin min(k, N - k), and no value
// has to meet its mirror image inside the transform.  A lone last frame takes
// b = 0 (then |Z_{N-k}| = |Z_k|).  Each lane sums |Z|^2 over the pairs its warp
// takes (pair p goes to warp p mod warps); the warps are combined, the mirror
// bins folded and the bands reduced in a fixed order.
// ---------------------------------------------------------------------------
constexpr int kWarpEnergyWarps = 8;

// W_16^m = exp(-2 pi i m / 16) for m = 0..7: cos(m pi / 8) - i sin(m pi / 8)
// (cos(pi/8) = sqrt(2 + sqrt 2) / 2, cos(pi/4) = sqrt(2) / 2, cos(3 pi/8) =
// sqrt(2 - sqrt 2) / 2); folded to immediates in the unrolled loops
__host__ __device__ constexpr float w16_cos(int m) {
    return m == 0 ? 1.f : m == 1 ? 0.92387953251128674f : m == 2 ? 0.70710678118654752f
         : m == 3 ? 0.38268343236508977f : m == 4 ? 0.f : m == 5 ? -0.38268343236508977f
         : m == 6 ? -0.70710678118654752f : -0.92387953251128674f;
}
__host__ __device__ constexpr float w16_sin(int m) { return w16_cos(m >= 4 ? m - 4 : 4 - m); }

ECHO_DEV float2 cmul(float2 a, float2 b) {
    return make_float2(a.x * b.x - a.y * b.y, a.x * b.y + a.y * b.x);
}

template <int R>
__global__ void __launch_bounds__(kWarpEnergyWarps * 32)
segment_energy_warp_kernel(const float *__restrict__ audio, int seg_len, int hop, int n_frames,
                           int n_bands, float *__restrict__ band_out, float *__restrict__ seg_out) {
    constexpr int N = 32 * R, HALF = N / 2;
    constexpr int LOG2R = R == 2 ? 1 : R == 4 ? 2 : R == 8 ? 3 : 4;
    static_assert(R == 2 || R == 4 || R == 8 || R == 16, "R-point DFT in registers: R <= 16");
    __shared__ float win[N];                          // periodic Hann window
    __shared__ float2 tw2[R][32];                     // W_N^(n2 bitrev_R(i)) for lane n2, register i
    __shared__ float acc_sh[kWarpEnergyWarps][N];     // per warp, by full-spectrum index
    __shared__ float bins[HALF + 1];
    __shared__ float bands[64];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tau = blockIdx.x;
    const float *seg = audio + (int64_t)tau * seg_len;

    for (int n = threadIdx.x; n < N; n += blockDim.x) win[n] = 0.5f - 0.5f * cospif((2.0f * n) / N);
    for (int e = threadIdx.x; e < R * 32; e += blockDim.x) {
        const int i = e / 32, n2 = e % 32;
        const int k1 = (int)(__brev((unsigned)i) >> (32 - LOG2R));
        float sn, cs;
        sincospif((2.0f * (float)(n2 * k1)) / N, &sn, &cs);
        tw2[i][n2] = make_float2(cs, -sn);
    }
    // cross-lane stage st (half size h = 16 >> st): the upper lane of a pair
    // multiplies by W_{2h}^(lane mod h); the lower lane by 1
    float2 twl[5];
#pragma unroll
    for (int st = 0; st < 5; ++st) {
        const int h = 16 >> st;
        if (lane & h) {
            float sn, cs;
            sincospif((float)(lane & (h - 1)) / (float)h, &sn, &cs);
            twl[st] = make_float2(cs, -sn);
        } else {
            twl[st] = make_float2(1.f, 0.f);
        }
    }
    __syncthreads();

    float acc[R];
#pragma unroll
    for (int i = 0; i < R; ++i) acc[i] = 0.f;
    const int n_pairs = (n_frames + 1) >> 1;
    for (int pr = warp; pr < n_pairs; pr += kWarpEnergyWarps) {
        const int off_a = 2 * pr * hop, off_b = off_a + hop;
        const bool has_b = 2 * pr + 1 < n_frames;
        float2 v[R];
#pragma unroll
        for (int n1 = 0; n1 < R; ++n1) {
            const int n = 32 * n1 + lane;
            const float w = win[n];
            const float xa = off_a + n < seg_len ? seg[off_a + n] : 0.f;
            const float xb = has_b && off_b + n < seg_len ? seg[off_b + n] : 0.f;
            v[n1] = make_float2(xa * w, xb * w);
        }
        // R-point DFT over n1 in registers (output in bit-reversed order)
#pragma unroll
        for (int h = R / 2; h >= 1; h >>= 1) {
#pragma unroll
            for (int s0 = 0; s0 < R; s0 += 2 * h) {
#pragma unroll
                for (int j = 0; j < h; ++j) {
                    const float2 u = v[s0 + j], x = v[s0 + j + h];
                    v[s0 + j] = make_float2(u.x + x.x, u.y + x.y);
                    const int m = j * (16 / (2 * h));          // W_{2h}^j = W_16^(j 16 / 2h)
                    v[s0 + j + h] = cmul(make_float2(u.x - x.x, u.y - x.y),
                                         make_float2(w16_cos(m), -w16_sin(m)));
                }
            }
        }
#pragma unroll
        for (int i = 0; i < R; ++i) v[i] = cmul(v[i], tw2[i][lane]);
        // 32-point DFT over n2 across the lanes (output lane = bitrev5(k2))
#pragma unroll
        for (int st = 0; st < 5; ++st) {
            const int h = 16 >> st;
            const bool upper = (lane & h) != 0;
#pragma unroll
            for (int i = 0; i < R; ++i) {
                const float px = __shfl_xor_sync(0xffffffffu, v[i].x, h);
                const float py = __shfl_xor_sync(0xffffffffu, v[i].y, h);
                const float2 d = upper ? make_float2(px - v[i].x, py - v[i].y)
                                       : make_float2(v[i].x + px, v[i].y + py);
                v[i] = cmul(d, twl[st]);
            }
        }
#pragma unroll
        for (int i = 0; i < R; ++i) acc[i] += v[i].x * v[i].x + v[i].y * v[i].y;
    }
    const int k2 = (int)(__brev((unsigned)lane) >> 27);
#pragma unroll
    for (int i = 0; i < R; ++i) {
        const int k1 = (int)(__brev((unsigned)i) >> (32 - LOG2R));
        acc_sh[warp][k1 + R * k2] = acc[i];
    }
    __syncthreads();
    constexpr float invN = 1.0f / (float)N;             // a power of two: exact
    for (int b = threadIdx.x; b <= HALF; b += blockDim.x) {
        float s = 0.f;
        for (int w = 0; w < kWarpEnergyWarps; ++w) s += acc_sh[w][b];
        if (b > 0 && b < HALF) {
            float m = 0.f;
            for (int w = 0; w < kWarpEnergyWarps; ++w) m += acc_sh[w][N - b];
            s += m;
        }
        bins[b] = s * invN;
    }
    __syncthreads();
    const int n_bins = HALF + 1;
    for (int b = warp; b < n_bands; b += kWarpEnergyWarps) {
        const int lo = (n_bins * b) / n_bands, hi = (n_bins * (b + 1)) / n_bands;
        float s = 0.f;
        for (int k = lo + lane; k < hi; k += 32) s += bins[k];
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
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (n_fft <= 512 && n_bands <= 64) {   // the warp-per-frame-pair kernel
        LaunchScope ls(ECHO_K_ENERGY, T, n_frames, n_fft, st);
        const int R = n_fft / 32;
        if (R == 2)
            segment_energy_warp_kernel<2><<<T, kWarpEnergyWarps * 32, 0, st>>>(
                audio, seg_len, hop, n_frames, n_bands, band_energy, seg_energy);
        else if (R == 4)
            segment_energy_warp_kernel<4><<<T, kWarpEnergyWarps * 32, 0, st>>>(
                audio, seg_len, hop, n_frames, n_bands, band_energy, seg_energy);
        else if (R == 8)
            segment_energy_warp_kernel<8><<<T, kWarpEnergyWarps * 32, 0, st>>>(
                audio, seg_len, hop, n_frames, n_bands, band_energy, seg_energy);
        else
            segment_energy_warp_kernel<16><<<T, kWarpEnergyWarps * 32, 0, st>>>(
                audio, seg_len, hop, n_frames, n_bands, band_energy, seg_energy);
        return last_launch_status();
    }
    int log2n = 0;
    while ((1 << log2n) < n_fft) ++log2n;
    const size_t smem = sizeof(float2) * (size_t)(n_fft / 2 + kGroups * n_fft) +
                        sizeof(float) * (size_t)kGroups * n_bins;
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
