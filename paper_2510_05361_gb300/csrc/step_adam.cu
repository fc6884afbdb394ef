// step_adam.cu -- instantiates the local-step kernels of Algorithm 1 (MT-DAO-Adam).
// One translation unit per base so that the instantiations compile in parallel.
#include "step_kernels.cuh"
#include "step_sync_kernels.cuh"

namespace mtdao {

template cudaError_t launch_step_base<MTDAO_BASE_ADAM>(int, int, bool, const StepArgs &, int,
                                                cudaStream_t);
template cudaError_t launch_step_sync_base<MTDAO_BASE_ADAM>(int, int, bool, const StepArgs &, int,
                                                     cudaStream_t);

}  // namespace mtdao
