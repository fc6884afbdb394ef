// replica_mean.cuh -- the worker average E_m[s] of one element, shared by
// every kernel that averages (fused step + sync, sync, sync + diagnostics),
// so that all of them produce the same bits.
//
// mean = s_0 + S / M, where S is the Kahan-compensated sum of (s_m - s_0)
// over m = 1..M-1 in replica order.  Summing differences keeps the operands
// small when the replicas are close (the usual case between syncs); the
// compensation keeps the error of S near one rounding instead of growing
// with M (a plain fp32 running sum loses about M ulps relative to a mean that
// is small against the replicas, e.g. 1e-4 at M = 1024).  When S is zero --
// in particular when all replicas agree -- the result is s_0 itself, bit for
// bit (sign of zero included).
#pragma once

#include <cuda_runtime.h>

namespace mtdao {

struct ReplicaMean {
    float s0, sum, comp;

    __device__ __forceinline__ explicit ReplicaMean(float first) : s0(first), sum(0.0f), comp(0.0f) {}

    __device__ __forceinline__ void add(float sm) {
        const float y = (sm - s0) - comp;
        const float t = sum + y;
        comp = (t - sum) - y;
        sum = t;
    }

    __device__ __forceinline__ float value(float M) const {
        const float q = (sum - comp) / M;
        return q == 0.0f ? s0 : s0 + q;
    }
};

}  // namespace mtdao
