// lb_noalloc.cu -- littlebit_linear_forward_noalloc: the two-launch forward
// (lb_generic.cu) run on a fixed scratch array compiled into the library, for
// callers that may not allocate device memory themselves.
//
// Scratch: kNoAllocFloats fp32 words (256 KiB) in a file-scope __device__
// array.  Every GPU that loads the library holds it until the process exits.
// Host code cannot use the array's name as a device address, so the first
// call in each CUDA context looks the address up with cudaGetSymbolAddress
// (with that context's device current) and caches it with the context
// handle; later calls in the same context reuse it.  A new context on the
// device (after cudaDeviceReset, or another context made current) reloads
// the module, so the address is looked up again rather than reused.
#include <mutex>

#include "lb_common.cuh"
#include "lb_kernels.h"

namespace {

constexpr size_t kNoAllocFloats = 65536;  // 256 KiB of fp32 stage-1 sums
constexpr int kMaxDevices = 64;

__device__ __align__(256) float g_noalloc_scratch[kNoAllocFloats];

std::mutex g_mu;
float *g_scratch_ptr[kMaxDevices];
void *g_scratch_ctx[kMaxDevices];  // the context the cached address belongs to

// cuCtxGetCurrent through the runtime's driver entry point (no link to libcuda).
using CtxGetCurrentFn = int (*)(void **);
CtxGetCurrentFn ctx_get_current() {
    static CtxGetCurrentFn fn = [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault,
                                             &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            f = nullptr;
        return reinterpret_cast<CtxGetCurrentFn>(f);
    }();
    return fn;
}

// Device address of g_noalloc_scratch in the current context (looked up on
// the first call in each context).
lb_status scratch_on_current_device(float **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return LB_ERR_CUDA;
    const CtxGetCurrentFn get = ctx_get_current();
    void *ctx = nullptr;
    if (!get || get(&ctx) != 0) return LB_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!ctx || !g_scratch_ptr[dev] || g_scratch_ctx[dev] != ctx) {
        // (also makes the device's primary context current when none was)
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return LB_ERR_CUDA;
        if (get(&ctx) != 0 || !ctx) return LB_ERR_CUDA;
        g_scratch_ptr[dev] = static_cast<float *>(p);
        g_scratch_ctx[dev] = ctx;
    }
    *out = g_scratch_ptr[dev];
    return LB_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" lb_status littlebit_linear_forward_noalloc(const lb_linear *L, const uint16_t *x,
                                                      int64_t T, void *y, int32_t y_dtype,
                                                      lb_stream_t stream) {
    lb_status st = lb::validate_linear(L);
    if (st != LB_OK) return st;
    if (T < 0 || (y_dtype != LB_OUT_BF16 && y_dtype != LB_OUT_FP32)) return LB_ERR_INVALID_ARG;
    if (T == 0) return LB_OK;
    if (!x || !y || !aligned16(x) || !aligned16(y)) return LB_ERR_INVALID_ARG;
    // stage-1 sums of every path and token must fit the fixed scratch
    if (T > (int64_t)kNoAllocFloats || lb::generic_ws_floats(*L, T) > kNoAllocFloats)
        return LB_ERR_WORKSPACE;
    float *scratch = nullptr;
    if ((st = scratch_on_current_device(&scratch)) != LB_OK) return st;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return LB_ERR_CUDA;
    // launch_generic clears the sums it uses before adding into them
    const cudaError_t e = lb::launch_generic(*L, x, T, y, y_dtype == LB_OUT_FP32, scratch, sms,
                                             (cudaStream_t)stream);
    return e == cudaSuccess ? LB_OK : LB_ERR_CUDA;
}
