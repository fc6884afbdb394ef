// kahan.cuh -- the accumulators of the diagnostics and norm reductions.
#pragma once

#include <cuda_runtime.h>

namespace mtdao {

// fp32 accumulator with Kahan compensation; value() folds the compensation
// in at double precision.
struct Kahan {
    float s = 0.0f, c = 0.0f;
    __device__ __forceinline__ void add(float y) {
        y -= c;
        const float t = s + y;
        c = (t - s) - y;
        s = t;
    }
    __device__ __forceinline__ double value() const {
        return static_cast<double>(s) - static_cast<double>(c);
    }
};

// Sum of one double per lane over a warp, valid in lane 0 (fixed order).
__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_down_sync(0xffffffffu, v, off);
    return v;
}

}  // namespace mtdao
