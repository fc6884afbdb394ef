// noalloc.cu -- per-replica gradient sum of squares without any allocation.
//
// mtdao_grad_sqnorm needs a handle, and creating a handle allocates the state
// arena and the norm workspace.  Some callers cannot allocate device memory
// at the point where they want the norm: a serving or training process whose
// device memory is reserved up front by another allocator (a caching
// allocator owns all of it, so a cudaMalloc from a library fails), a
// latency-critical loop in which a cudaMalloc/cudaFree pair would
// synchronise the device, or a monitoring hook that only sees a gradient
// buffer and has no handle.  mtdao_grad_sqnorm_static serves them: its
// scratch (the per-block partial sums) is a fixed file-scope device array
// that exists for as long as the library is loaded on a device.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdio>
#include <mutex>

#include "mtdao.h"
#include "mtdao_internal.h"

namespace {

// Partial sums of one call: M * blocks_per_replica doubles, each written by
// its block before the finalising kernel reads it, so no slot has to start
// at zero.  Shared by every call on a device; it keeps the last call's
// values.
static __device__ __align__(256) double g_sqnorm_scratch[MTDAO_STATIC_SCRATCH_DOUBLES];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;

// Per device: the array's device address and the unique id of the context
// it was looked up in.  A device reset (cudaDeviceReset) destroys the
// primary context and a later call runs in a new one, where the module is
// loaded again and the array may sit elsewhere; the id tells the two apart
// (context ids are never reused within a process).
struct ScratchAddr {
    void *ptr = nullptr;
    unsigned long long ctx_id = 0;
};
ScratchAddr g_scratch[kMaxDevices];

// cuCtxGetId from the driver, found once through the runtime (so the
// library needs no link-time dependency on libcuda).  nullptr if the
// driver does not offer it; the cache is then kept per device only.
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long *);
CtxGetIdFn ctx_get_id() {
    static CtxGetIdFn fn = [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess) {
            cudaGetLastError();
            p = nullptr;
        }
        return reinterpret_cast<CtxGetIdFn>(p);
    }();
    return fn;
}

// Id of the context current on this thread, or 0 if there is none yet (a
// thread whose first runtime call this is) or it cannot be told.
unsigned long long current_ctx_id() {
    CtxGetIdFn fn = ctx_get_id();
    unsigned long long id = 0;
    if (fn == nullptr || fn(nullptr, &id) != CUDA_SUCCESS) return 0;
    return id;
}

// Device address of g_sqnorm_scratch on the current device.  In host code
// the array's name is only a host-side stand-in, so the address is looked up
// with cudaGetSymbolAddress (the first call on a device, and the first call
// after its context changed, does this; the lookup also makes the device's
// primary context current on this thread) and cached.
int scratch_on_current_device(int dev, void **out) {
    if (dev < 0 || dev >= kMaxDevices)
        return mtdao::set_thread_error(MTDAO_ERR_INVALID, "device index beyond the supported 64");
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    ScratchAddr &slot = g_scratch[dev];
    const unsigned long long id = current_ctx_id();
    if (slot.ptr == nullptr || (id != 0 && id != slot.ctx_id)) {
        void *p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_sqnorm_scratch);
        if (e != cudaSuccess || p == nullptr) {
            char msg[256];
            snprintf(msg, sizeof msg, "cudaGetSymbolAddress of the static scratch: %s",
                     cudaGetErrorString(e));
            return mtdao::set_thread_error(MTDAO_ERR_CUDA, msg);
        }
        slot.ptr = p;
        slot.ctx_id = current_ctx_id();
    }
    *out = slot.ptr;
    return MTDAO_OK;
}

}  // namespace

extern "C" int mtdao_grad_sqnorm_static(const void *grads_dev, int32_t grad_dtype, int32_t M,
                                        int64_t n_padded, double *out_dev, void *cuda_stream) {
    if (grads_dev == nullptr || out_dev == nullptr)
        return mtdao::set_thread_error(MTDAO_ERR_INVALID, "grads or out is NULL");
    if ((reinterpret_cast<uintptr_t>(grads_dev) & 15u) != 0)
        return mtdao::set_thread_error(MTDAO_ERR_ALIGN, "grads not 16-byte aligned");
    if ((reinterpret_cast<uintptr_t>(out_dev) & 7u) != 0)
        return mtdao::set_thread_error(MTDAO_ERR_ALIGN, "out not 8-byte aligned");
    if (grad_dtype != MTDAO_F32 && grad_dtype != MTDAO_BF16)
        return mtdao::set_thread_error(MTDAO_ERR_INVALID, "unknown gradient dtype");
    if (M < 1 || M > MTDAO_MAX_REPLICAS)
        return mtdao::set_thread_error(MTDAO_ERR_INVALID, "M outside 1..MTDAO_MAX_REPLICAS");
    if (n_padded < 1 || n_padded % 256 != 0)
        return mtdao::set_thread_error(MTDAO_ERR_INVALID, "n_padded must be a positive multiple of 256");

    int dev = 0, sms = 1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) {
        char msg[256];
        snprintf(msg, sizeof msg, "no usable CUDA device: %s", cudaGetErrorString(e));
        return mtdao::set_thread_error(MTDAO_ERR_CUDA, msg);
    }
    // Same grid as mtdao_grad_sqnorm, so both give identical bits.
    const int blocks = mtdao::norm_blocks_per_replica(sms, M);
    const long long need = static_cast<long long>(M) * blocks;
    if (need > MTDAO_STATIC_SCRATCH_DOUBLES) {
        char msg[256];
        snprintf(msg, sizeof msg, "needs %lld partial sums; the static scratch holds %d", need,
                 MTDAO_STATIC_SCRATCH_DOUBLES);
        return mtdao::set_thread_error(MTDAO_ERR_INVALID, msg);
    }
    void *scratch = nullptr;
    if (int rc = scratch_on_current_device(dev, &scratch)) return rc;
    e = mtdao::launch_grad_sqnorm(grads_dev, grad_dtype, M, n_padded, blocks,
                                  static_cast<double *>(scratch), out_dev, nullptr, 0.0,
                                  static_cast<cudaStream_t>(cuda_stream));
    if (e != cudaSuccess) {
        char msg[256];
        snprintf(msg, sizeof msg, "gradient norm launch: %s", cudaGetErrorString(e));
        return mtdao::set_thread_error(MTDAO_ERR_CUDA, msg);
    }
    return MTDAO_OK;
}
