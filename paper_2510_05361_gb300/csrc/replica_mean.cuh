// replica_mean.cuh -- the worker average E_m[s] of one element, shared by
// every kernel that averages (fused step + sync, sync, sync + diagnostics),
// so that all of them produce the same bits.
//
// With h = floor(M / 2):
//   A = Kahan-compensated sum of (s_m - s_0), m = 1 .. h-1, in replica order
//   B = Kahan-compensated sum of (s_m - s_0), m = h .. M-1, in replica order
//   mean = s_0 + (A + B) / M      (s_0 itself, bit for bit, when A + B = 0)
// Summing differences keeps the operands small when the replicas are close
// (the usual case between syncs); the compensation keeps the error near one
// rounding instead of growing with M (a plain fp32 running sum loses about M
// ulps relative to a mean that is small against the replicas, 1e-4 at
// M = 1024).  The two parts let a kernel hold the replicas of one element
// in two lanes (replicas 0 .. h-1 and h .. M-1) and still produce exactly
// the value a single thread computes.
//
// Non-finite values: the compensated sum turns one infinite replica value
// into NaN (inf - inf inside the compensation), where the mean of the
// method, sum_m s_m / M, is +-inf when the values hold infinities of one
// sign only.  So a NaN result is replaced by the plain fp32 sum of the M
// values divided by M: NaN when a value is NaN or both infinities occur,
// the infinity otherwise (the outcome does not depend on the order of the
// sum).  Finite values reach this path only if a difference s_m - s_0
// overflows (|s| near 3.4e38); the plain sum is then the fallback as well.
#pragma once

#include <cuda_runtime.h>

namespace mtdao {

// Kahan-compensated sum of differences to a reference value s0.
struct DiffSum {
    float s0, sum, comp;

    __device__ __forceinline__ explicit DiffSum(float ref) : s0(ref), sum(0.0f), comp(0.0f) {}

    __device__ __forceinline__ void add(float sm) {
        const float y = (sm - s0) - comp;
        const float t = sum + y;
        comp = (t - sum) - y;
        sum = t;
    }

    __device__ __forceinline__ float partial() const { return sum - comp; }
};

__device__ __forceinline__ float replica_mean_from_parts(float s0, float part_a, float part_b, float M) {
    const float q = (part_a + part_b) / M;
    return q == 0.0f ? s0 : s0 + q;
}

// The compensated mean, or the plain one where it is NaN (see above).
__device__ __forceinline__ float mean_or_plain(float mean, float plain_sum, float M) {
    return mean != mean ? plain_sum / M : mean;
}

// The mean of M values held by one thread; get(m) returns replica m's value.
template <int M, typename Get>
__device__ __forceinline__ float replica_mean(Get get) {
    constexpr int h = M / 2;
    const float s0 = get(0);
    DiffSum a(s0), b(s0);
#pragma unroll
    for (int m = 1; m < h; ++m) a.add(get(m));
#pragma unroll
    for (int m = (h > 1 ? h : 1); m < M; ++m) b.add(get(m));
    const float mean = replica_mean_from_parts(s0, a.partial(), b.partial(), static_cast<float>(M));
    if (mean == mean) return mean;
    float plain = s0;
#pragma unroll
    for (int m = 1; m < M; ++m) plain += get(m);
    return plain / static_cast<float>(M);
}

// Same, for a replica count known only at run time.
template <typename Get>
__device__ __forceinline__ float replica_mean_rt(int M, Get get) {
    const int h = M / 2;
    const float s0 = get(0);
    DiffSum a(s0), b(s0);
    for (int m = 1; m < h; ++m) a.add(get(m));
    for (int m = (h > 1 ? h : 1); m < M; ++m) b.add(get(m));
    const float mean = replica_mean_from_parts(s0, a.partial(), b.partial(), static_cast<float>(M));
    if (mean == mean) return mean;
    float plain = s0;
    for (int m = 1; m < M; ++m) plain += get(m);
    return plain / static_cast<float>(M);
}

}  // namespace mtdao
