// step_adopt.cu -- instantiates the local-step kernels of Algorithm 2 (MT-DAO-ADOPT).
// One translation unit per base so that the instantiations compile in parallel.
#include "step_kernels.cuh"
#include "step_sync_kernels.cuh"

namespace mtdao {

template cudaError_t launch_step_base<MTDAO_BASE_ADOPT>(int, int, bool, const StepArgs &, int,
                                                cudaStream_t);
template cudaError_t launch_step_sync_base<MTDAO_BASE_ADOPT>(int, int, bool, const StepArgs &, int,
                                                     cudaStream_t);

namespace {

// Step 0 in the original ADOPT order: the second moment is initialised from
// the first gradient, v = g_0^2, and nothing else is read or written (the
// momenta and the parameters make their first move at step 1).  A separate
// kernel rather than the step kernel with zero rates: a zero rate would
// still multiply a non-finite normalised gradient (0 * Inf = NaN) into u
// and x.
template <int GDT>
__global__ void __launch_bounds__(kThreads) adopt_init_v_kernel(float *v, const void *grads, int64_t n4) {
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const float4 g = ld_grad<GDT>(grads, 4 * i);
        st_state(v + 4 * i, make_float4(__fmul_rn(g.x, g.x), __fmul_rn(g.y, g.y), __fmul_rn(g.z, g.z),
                                        __fmul_rn(g.w, g.w)));
    }
}

}  // namespace

cudaError_t launch_adopt_init_v(float *v, const void *grads, int grad_dtype, int64_t count, cudaStream_t stream) {
    const int64_t n4 = count / 4;
    const int grid = stream_grid((n4 + 31) / 32);
    if (grad_dtype == MTDAO_F32)
        adopt_init_v_kernel<MTDAO_F32><<<grid, kThreads, 0, stream>>>(v, grads, n4);
    else
        adopt_init_v_kernel<MTDAO_BF16><<<grid, kThreads, 0, stream>>>(v, grads, n4);
    return cudaGetLastError();
}

}  // namespace mtdao
