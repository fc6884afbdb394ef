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
void *g_scratch_addr[kMaxDevices] = {};

// Device address of g_sqnorm_scratch on the current device.  In host code
// the array's name is only a host-side stand-in, so the address is looked up
// once per device (the first call on a device does this) and cached.
int scratch_on_current_device(int dev, void **out) {
    if (dev < 0 || dev >= kMaxDevices)
        return mtdao::set_thread_error(MTDAO_ERR_INVALID, "device index beyond the supported 64");
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (g_scratch_addr[dev] == nullptr) {
        void *p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_sqnorm_scratch);
        if (e != cudaSuccess || p == nullptr) {
            char msg[256];
            snprintf(msg, sizeof msg, "cudaGetSymbolAddress of the static scratch: %s",
                     cudaGetErrorString(e));
            return mtdao::set_thread_error(MTDAO_ERR_CUDA, msg);
        }
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return MTDAO_OK;
}

}  // namespace

extern "C" int mtdao_grad_sqnorm_static(const void *grads_dev, int32_t grad_dtype, int32_t M,
                                        int64_t n_padded, double *out_dev, void *cuda_stream) {
    if (grads_dev == nullptr || out_dev == nullptr)
        return mtdao::set_thread_error(MTDAO_ERR_INVALID, "grads or out is NULL");
    if ((reinterpret_cast<uintptr_t>(grads_dev) & 15u) != 0)
        return mtdao::set_thread_error(MTDAO_ERR_ALIGN, "grads not 16-byte aligned");
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
