// Status strings, the per-device error flag and tensor-map construction.
#include <atomic>
#include <mutex>
#include <vector>

#include "common.cuh"
#include "internal.h"

// One error word per device that loads the library; kernels get its address.
static __device__ int g_echo_error;

namespace echo {

namespace {
constexpr int kMaxDevices = 64;
int *g_err_ptr[kMaxDevices] = {};
int g_supported[kMaxDevices] = {};  // 0 unknown, 1 yes, -1 no
std::mutex g_mu;

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn g_encode = nullptr;

int current_device() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return -1;
    return dev;
}
}  // namespace

int *device_error_ptr() {
    int dev = current_device();
    if (dev < 0 || dev >= kMaxDevices) return nullptr;
    if (g_err_ptr[dev]) return g_err_ptr[dev];
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_err_ptr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_echo_error) != cudaSuccess) return nullptr;
        g_err_ptr[dev] = static_cast<int *>(p);
    }
    return g_err_ptr[dev];
}

bool device_supported() {
    int dev = current_device();
    if (dev < 0 || dev >= kMaxDevices) return false;
    if (g_supported[dev] == 0) {
        cudaDeviceProp prop;
        bool ok = cudaGetDeviceProperties(&prop, dev) == cudaSuccess && prop.major == 10 &&
                  prop.minor == 3;
        g_supported[dev] = ok ? 1 : -1;
    }
    return g_supported[dev] == 1;
}

echo_status last_launch_status() {
    return cudaGetLastError() == cudaSuccess ? ECHO_OK : ECHO_ERR_CUDA;
}

bool make_tmap_bf16(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint64_t ld,
                    uint32_t box_rows) {
    if (!g_encode) {
        std::lock_guard<std::mutex> lk(g_mu);
        if (!g_encode) {
            void *fn = nullptr;
            cudaDriverEntryPointQueryResult q;
            if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                 cudaEnableDefault, &q) != cudaSuccess ||
                q != cudaDriverEntryPointSuccess || !fn)
                return false;
            g_encode = reinterpret_cast<EncodeTiledFn>(fn);
        }
    }
    cuuint64_t gdim[2] = {cols, rows};
    cuuint64_t gstride[1] = {ld * 2};
    cuuint32_t box[2] = {64, box_rows};
    cuuint32_t estride[2] = {1, 1};
    CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), gdim,
                          gstride, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// ---------------------------------------------------------------------------
// launch counter and event profiler
// ---------------------------------------------------------------------------
namespace {
std::atomic<uint64_t> g_launches{0};
std::atomic<int> g_prof_on{0};
struct ProfRecord {
    int kind;
    int64_t m, n, k;
    cudaEvent_t start, stop;
};
constexpr size_t kMaxRecords = 65536;
std::vector<ProfRecord> g_records;
std::vector<cudaEvent_t> g_event_pool;
std::mutex g_prof_mu;

cudaEvent_t take_event() {
    if (!g_event_pool.empty()) {
        cudaEvent_t e = g_event_pool.back();
        g_event_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
}
}  // namespace

LaunchScope::LaunchScope(int kind, int64_t m, int64_t n, int64_t k, cudaStream_t st)
    : slot_(-1), st_(st) {
    g_launches.fetch_add(1, std::memory_order_relaxed);
    if (!g_prof_on.load(std::memory_order_relaxed)) return;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (g_records.size() >= kMaxRecords) return;
    ProfRecord r{kind, m, n, k, take_event(), take_event()};
    if (!r.start || !r.stop) return;
    if (cudaEventRecord(r.start, st) != cudaSuccess) return;
    slot_ = (int)g_records.size();
    g_records.push_back(r);
}

LaunchScope::~LaunchScope() {
    if (slot_ < 0) return;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (slot_ < (int)g_records.size()) cudaEventRecord(g_records[slot_].stop, st_);
}

}  // namespace echo

extern "C" uint64_t echo_launch_count(void) { return echo::g_launches.load(); }

extern "C" echo_status echo_profile_enable(int32_t on) {
    echo::g_prof_on.store(on ? 1 : 0);
    return ECHO_OK;
}

extern "C" int32_t echo_profile_read(int32_t max, int32_t *kinds, int64_t *m, int64_t *n,
                                     int64_t *k, float *ms) {
    using namespace echo;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    int32_t out = 0;
    bool ok = true;
    for (auto &r : g_records) {
        if (out < max) {
            float t = 0.f;
            if (cudaEventSynchronize(r.stop) != cudaSuccess ||
                cudaEventElapsedTime(&t, r.start, r.stop) != cudaSuccess)
                ok = false;
            if (kinds) kinds[out] = r.kind;
            if (m) m[out] = r.m;
            if (n) n[out] = r.n;
            if (k) k[out] = r.k;
            if (ms) ms[out] = t;
            ++out;
        }
        g_event_pool.push_back(r.start);
        g_event_pool.push_back(r.stop);
    }
    g_records.clear();
    return ok ? out : -1;
}

extern "C" const char *echo_kernel_name(int32_t kind) {
    static const char *names[ECHO_K_COUNT] = {
        "segment_energy_fft", "drift_score",  "topk_select",  "rowmap",
        "layernorm_gather",   "gemm_tcgen05", "attention",    "quant_scatter",
        "dequant_gather",     "dequant_merge", "step_delta",   "uniform_select",
        "ref_scan",           "ref_alloc",     "ref_store",    "cache_copy",
        "merge_quant"};
    if (kind < 0 || kind >= ECHO_K_COUNT) return "unknown";
    return names[kind];
}

extern "C" const char *echo_status_str(echo_status s) {
    switch (s) {
        case ECHO_OK: return "ECHO_OK";
        case ECHO_ERR_INVALID_ARG: return "ECHO_ERR_INVALID_ARG";
        case ECHO_ERR_SHAPE: return "ECHO_ERR_SHAPE";
        case ECHO_ERR_WORKSPACE: return "ECHO_ERR_WORKSPACE";
        case ECHO_ERR_CUDA: return "ECHO_ERR_CUDA";
        case ECHO_ERR_NONFINITE: return "ECHO_ERR_NONFINITE";
        case ECHO_ERR_TIMEOUT: return "ECHO_ERR_TIMEOUT";
        case ECHO_ERR_UNSUPPORTED: return "ECHO_ERR_UNSUPPORTED";
    }
    return "ECHO_ERR_UNKNOWN";
}

extern "C" echo_status echo_get_device_error(echo_stream_t stream) {
    if (cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
        return ECHO_ERR_CUDA;
    int *p = echo::device_error_ptr();
    if (!p) return ECHO_ERR_CUDA;
    int v = 0;
    if (cudaMemcpy(&v, p, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return ECHO_ERR_CUDA;
    if (v != 0) {
        int zero = 0;
        if (cudaMemcpy(p, &zero, sizeof(int), cudaMemcpyHostToDevice) != cudaSuccess)
            return ECHO_ERR_CUDA;
    }
    return static_cast<echo_status>(v);
}

namespace {

// One thread waits for the first phase of a shared-memory barrier that no one
// arrives at, with the library's bounded wait: after limit_ns it gives up and
// sets ECHO_ERR_TIMEOUT, as every wait in the library does.
__global__ void timeout_probe_kernel(uint64_t limit_ns, int *err) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_barrier_init();
    mbar_wait(&bar, 0, &abort_flag, err, limit_ns);
}

}  // namespace

extern "C" echo_status echo_check_timeout_path(int64_t limit_ns, echo_stream_t stream) {
    using namespace echo;
    if (limit_ns < 1000 || limit_ns > 2000000000ll) return ECHO_ERR_INVALID_ARG;
    if (!device_supported()) return ECHO_ERR_UNSUPPORTED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    timeout_probe_kernel<<<1, 1, 0, st>>>((uint64_t)limit_ns, device_error_ptr());
    return last_launch_status();
}
