// reduce_kernels.cu -- replica averaging (outer synchronisation) and the
// per-replica gradient norm used by clip(g, rho).
//
// Averaging (Algorithms 1-3, E_m[.] with averaging as OuterOpt): for every
// selected state and element, the M replica values are read once and the
// mean (replica_mean.cuh) is written back to all M replicas.  Algorithmic traffic: 8 * M bytes
// per element per state.  HBM-bound; grid-stride over float4 vectors, one
// grid row (blockIdx.y) per selected state.
//
// Norm: sum_i g[m][i]^2 per replica with a fixed grid and fixed reduction
// order, so the result is bit-reproducible.  Each thread accumulates its
// strided share in fp32 with Kahan compensation, warps and blocks combine in
// fp64, and a second small kernel adds the per-block partials in order.
#include <cuda_runtime.h>
#include <cmath>
#include <cstdint>
#include <type_traits>

#include "mtdao_internal.h"
#include "replica_mean.cuh"
#include "step_kernels.cuh"

namespace mtdao {

namespace {

template <int MT>
__global__ void __launch_bounds__(kThreads) sync_kernel(const SyncArgs a) {
    const int M = MT > 0 ? MT : a.M;
    float *base = a.arena + static_cast<int64_t>(a.sel[blockIdx.y]) * a.stride;
    const int64_t n = a.n_padded;
    const int64_t nv = n / 4;
    const float Mf = static_cast<float>(M);
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nv;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t e = 4 * i;
        float mean[4];
        if constexpr (MT > 0) {
            float r[MT][4];
#pragma unroll
            for (int m = 0; m < MT; ++m) to_array(ld_state(base + m * n + e), r[m]);
#pragma unroll
            for (int k = 0; k < 4; ++k) mean[k] = replica_mean<MT>([&](int m) { return r[m][k]; });
        } else {
            // streamed: replicas 1 .. h-1 feed part A, h .. M-1 part B (replica_mean.cuh)
            float s0[4];
            to_array(ld_state(base + e), s0);
            DiffSum pa[4] = {DiffSum(s0[0]), DiffSum(s0[1]), DiffSum(s0[2]), DiffSum(s0[3])};
            DiffSum pb[4] = {DiffSum(s0[0]), DiffSum(s0[1]), DiffSum(s0[2]), DiffSum(s0[3])};
            const int h = M / 2;
            for (int m = 1; m < M; ++m) {
                float r[4];
                to_array(ld_state(base + m * n + e), r);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    if (m < h) pa[k].add(r[k]);
                    else pb[k].add(r[k]);
                }
            }
#pragma unroll
            for (int k = 0; k < 4; ++k) mean[k] = replica_mean_from_parts(s0[k], pa[k].partial(), pb[k].partial(), Mf);
        }
        const float4 mv = from_array(mean);
        for (int m = 0; m < M; ++m) st_state(base + m * n + e, mv);
    }
}

template <int MT>
cudaError_t launch_sync_t(const SyncArgs &a, int num_sms, cudaStream_t stream) {
    static const int per_sm = blocks_per_sm(sync_kernel<MT>);
    const int64_t nv = a.n_padded / 4;
    int64_t gx = static_cast<int64_t>(per_sm) * num_sms / (a.n_sel > 0 ? a.n_sel : 1);
    const int64_t need = (nv + kThreads - 1) / kThreads;
    if (gx > need) gx = need;
    if (gx < 1) gx = 1;
    dim3 grid(static_cast<unsigned>(gx), static_cast<unsigned>(a.n_sel));
    sync_kernel<MT><<<grid, kThreads, 0, stream>>>(a);
    return cudaGetLastError();
}

__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_down_sync(0xffffffffu, v, off);
    return v;
}

// Deterministic block sum of one double per thread; result valid in thread 0.
__device__ double block_sum(double v) {
    __shared__ double part[kNormThreads / 32];
    v = warp_sum(v);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    if (l == 0) part[w] = v;
    __syncthreads();
    double total = 0.0;
    if (threadIdx.x == 0)
        for (int i = 0; i < static_cast<int>(blockDim.x >> 5); ++i) total += part[i];
    return total;
}

// Positions (groups of 4 elements) a thread of the norm kernels loads
// before it accumulates them: i, i + T, ..., i + (U - 1) T with T the
// replica's thread count, the same order as a plain grid-stride loop, so
// the sums do not depend on the unrolling.  64 bytes per thread in flight:
// 4 positions of f32, 8 of bf16.
template <int GDT>
constexpr int kNormUnroll = GDT == MTDAO_F32 ? 4 : 8;

// Four gradient values as loaded (f32: float4; bf16: two packed words, 2
// registers instead of 4 until they are widened) and their fp32 values.
template <int GDT>
using GradWords = typename std::conditional<GDT == MTDAO_F32, float4, uint2>::type;

template <int GDT>
__device__ __forceinline__ GradWords<GDT> ld_grad_words(const void *g, int64_t e) {
    if constexpr (GDT == MTDAO_F32)
        return __ldcs(reinterpret_cast<const float4 *>(static_cast<const float *>(g) + e));
    else
        return __ldcs(reinterpret_cast<const uint2 *>(static_cast<const uint16_t *>(g) + e));
}

template <int GDT>
__device__ __forceinline__ float4 widen(GradWords<GDT> w) {
    if constexpr (GDT == MTDAO_F32)
        return w;
    else
        return make_float4(__uint_as_float(w.x << 16), __uint_as_float(w.x & 0xffff0000u),
                           __uint_as_float(w.y << 16), __uint_as_float(w.y & 0xffff0000u));
}

template <int GDT>
__global__ void __launch_bounds__(kNormThreads, 4) sqnorm_partial_kernel(const void *g, int64_t n,
                                                                      double *partial) {
    const int m = blockIdx.y;
    const int nb = gridDim.x;
    const int64_t nv = n / 4;
    const int64_t T = static_cast<int64_t>(nb) * blockDim.x;
    float sum = 0.0f, comp = 0.0f;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nv;
         i += kNormUnroll<GDT> * T) {
        GradWords<GDT> w[kNormUnroll<GDT>];
#pragma unroll
        for (int u = 0; u < kNormUnroll<GDT>; ++u)
            if (i + u * T < nv) w[u] = ld_grad_words<GDT>(g, m * n + 4 * (i + u * T));
#pragma unroll
        for (int u = 0; u < kNormUnroll<GDT>; ++u) {
            if (i + u * T >= nv) break;
            const float4 q = widen<GDT>(w[u]);
            const float y = fmaf(q.x, q.x, fmaf(q.y, q.y, fmaf(q.z, q.z, __fmul_rn(q.w, q.w)))) - comp;
            const float t = sum + y;
            comp = (t - sum) - y;
            sum = t;
        }
    }
    const double total = block_sum(static_cast<double>(sum) - static_cast<double>(comp));
    if (threadIdx.x == 0) partial[static_cast<int64_t>(m) * nb + blockIdx.x] = total;
}

// Number of NaN or +-Inf values (all exponent bits set) per replica, with
// the same fixed grid and reduction order as the sum of squares; counts are
// integers well below 2^53, so the double partials are exact.
template <int GDT>
__global__ void __launch_bounds__(kNormThreads, 4) nonfinite_partial_kernel(const void *g, int64_t n,
                                                                         double *partial) {
    const int m = blockIdx.y;
    const int nb = gridDim.x;
    const int64_t nv = n / 4;
    const int64_t T = static_cast<int64_t>(nb) * blockDim.x;
    const uint32_t e = 0x7f800000u;
    uint32_t count = 0;                // at most 4 nv / T per thread
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nv;
         i += kNormUnroll<GDT> * T) {
        GradWords<GDT> w[kNormUnroll<GDT>];
#pragma unroll
        for (int u = 0; u < kNormUnroll<GDT>; ++u)
            if (i + u * T < nv) w[u] = ld_grad_words<GDT>(g, m * n + 4 * (i + u * T));
#pragma unroll
        for (int u = 0; u < kNormUnroll<GDT>; ++u) {
            if (i + u * T >= nv) break;
            const float4 q = widen<GDT>(w[u]);
            count += ((__float_as_uint(q.x) & e) == e) + ((__float_as_uint(q.y) & e) == e) +
                     ((__float_as_uint(q.z) & e) == e) + ((__float_as_uint(q.w) & e) == e);
        }
    }
    const double total = block_sum(static_cast<double>(count));
    if (threadIdx.x == 0) partial[static_cast<int64_t>(m) * nb + blockIdx.x] = total;
}

__global__ void __launch_bounds__(kNormThreads) sqnorm_finalize_kernel(const double *partial, int nb,
                                                                       double *out, float *clip_scale,
                                                                       double rho) {
    const int m = blockIdx.x;
    double acc = 0.0;
    for (int i = threadIdx.x; i < nb; i += blockDim.x) acc += partial[static_cast<int64_t>(m) * nb + i];
    const double total = block_sum(acc);
    if (threadIdx.x == 0) {
        out[m] = total;
        if (clip_scale != nullptr) {
            const double f = rho / (sqrt(total) + 1e-6);
            clip_scale[m] = static_cast<float>(f < 1.0 ? f : 1.0);
        }
    }
}

// ---------------------------------------------------------------- sync + diagnostics

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

// Replica average of the selected states (exactly as sync_kernel) plus, in
// the same pass over the M replicas, per state and block the partial sums of
//   q = 0          sum_m (s_m - s_bar)^2        (cross-worker variance * M)
//   q = 1          s_bar^2
//   q = 2 + m      s_m^2
//   q = 2 + M + m  s_m * s_bar
// written to partial[(sel * gridDim.x + block) * Q + q], Q = 2 + 2M.  s_bar
// is the fp32 mean that is stored.  With M = 1 nothing is stored (there is
// nothing to average) but the sums are still formed.
template <int M>
__global__ void __launch_bounds__(kThreads) sync_stats_kernel(const SyncArgs a, double *partial) {
    constexpr int Q = 2 + 2 * M;
    float *base = a.arena + static_cast<int64_t>(a.sel[blockIdx.y]) * a.stride;
    const int64_t n = a.n_padded;
    const int64_t nv = n / 4;
    Kahan acc[Q];
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nv;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t e = 4 * i;
        float r[M][4];
#pragma unroll
        for (int m = 0; m < M; ++m) to_array(ld_state(base + m * n + e), r[m]);
        float mean[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) mean[k] = replica_mean<M>([&](int m) { return r[m][k]; });
        float q[Q];
#pragma unroll
        for (int j = 0; j < Q; ++j) q[j] = 0.0f;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            q[1] = fmaf(mean[k], mean[k], q[1]);
#pragma unroll
            for (int m = 0; m < M; ++m) {
                const float dv = r[m][k] - mean[k];
                q[0] = fmaf(dv, dv, q[0]);
                q[2 + m] = fmaf(r[m][k], r[m][k], q[2 + m]);
                q[2 + M + m] = fmaf(r[m][k], mean[k], q[2 + M + m]);
            }
        }
#pragma unroll
        for (int j = 0; j < Q; ++j) acc[j].add(q[j]);
        if constexpr (M > 1) {
            const float4 mv = from_array(mean);
#pragma unroll
            for (int m = 0; m < M; ++m) st_state(base + m * n + e, mv);
        }
    }
    __shared__ double part[Q][kThreads / 32];
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
#pragma unroll
    for (int j = 0; j < Q; ++j) {
        const double v = warp_sum(acc[j].value());
        if (l == 0) part[j][w] = v;
    }
    __syncthreads();
    if (threadIdx.x < Q) {
        double total = 0.0;
        for (int i = 0; i < static_cast<int>(blockDim.x >> 5); ++i) total += part[threadIdx.x][i];
        partial[(static_cast<int64_t>(blockIdx.y) * gridDim.x + blockIdx.x) * Q + threadIdx.x] = total;
    }
}

// stats[sel * Q + q] = sum over blocks of partial (in block order); q = 0 is
// divided by divide_first (M for the variance, a mean over workers)
// (divide_first = 0 leaves q = 0 undivided)
__global__ void sync_stats_finalize_kernel(const double *partial, int blocks, int Q, int divide_first,
                                           double *stats) {
    const int sel = blockIdx.x, q = threadIdx.x;
    if (q >= Q) return;
    double total = 0.0;
    for (int b = 0; b < blocks; ++b) total += partial[(static_cast<int64_t>(sel) * blocks + b) * Q + q];
    stats[sel * Q + q] = (q == 0 && divide_first > 0) ? total / divide_first : total;
}

template <int M>
cudaError_t launch_sync_stats_t(const SyncArgs &a, int num_sms, double *partial, size_t partial_cap,
                                double *stats, cudaStream_t stream) {
    constexpr int Q = 2 + 2 * M;
    static const int per_sm = blocks_per_sm(sync_stats_kernel<M>);
    const int64_t nv = a.n_padded / 4;
    int64_t gx = static_cast<int64_t>(per_sm) * num_sms / a.n_sel;
    const int64_t need = (nv + kThreads - 1) / kThreads;
    if (gx > need) gx = need;
    if (gx < 1) gx = 1;
    if (static_cast<size_t>(gx) * a.n_sel * Q > partial_cap) return cudaErrorInvalidValue;
    dim3 grid(static_cast<unsigned>(gx), static_cast<unsigned>(a.n_sel));
    sync_stats_kernel<M><<<grid, kThreads, 0, stream>>>(a, partial);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    sync_stats_finalize_kernel<<<a.n_sel, 32, 0, stream>>>(partial, static_cast<int>(gx), Q, M, stats);
    return cudaGetLastError();
}

// Pseudo-gradient diagnostics of the parameters x[M][n] against the anchor
// a[n] (the parameters at the last average), read-only, with fixed-order
// sums into partial[block * Q + q], Q = 2M + 2:
//   q = m          (x_m - a)^2
//   q = M + m      (x_m - a) * (x_bar - a)
//   q = 2M         (x_bar - a)^2
//   q = 2M + 1     a^2
// x_bar is the replica mean of replica_mean.cuh (the value an average would
// store now).
template <int M>
__global__ void __launch_bounds__(kThreads) pseudo_grad_stats_kernel(const float *x, const float *anchor,
                                                                     int64_t n, double *partial) {
    constexpr int Q = 2 * M + 2;
    const int64_t nv = n / 4;
    Kahan acc[Q];
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nv;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t e = 4 * i;
        float r[M][4], av[4];
#pragma unroll
        for (int m = 0; m < M; ++m) to_array(ld_state(x + m * n + e), r[m]);
        to_array(__ldcs(reinterpret_cast<const float4 *>(anchor + e)), av);
        float q[Q];
#pragma unroll
        for (int j = 0; j < Q; ++j) q[j] = 0.0f;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float mean = replica_mean<M>([&](int m) { return r[m][k]; });
            const float glob = mean - av[k];
            q[2 * M] = fmaf(glob, glob, q[2 * M]);
            q[2 * M + 1] = fmaf(av[k], av[k], q[2 * M + 1]);
#pragma unroll
            for (int m = 0; m < M; ++m) {
                const float loc = r[m][k] - av[k];
                q[m] = fmaf(loc, loc, q[m]);
                q[M + m] = fmaf(loc, glob, q[M + m]);
            }
        }
#pragma unroll
        for (int j = 0; j < Q; ++j) acc[j].add(q[j]);
    }
    __shared__ double part[Q][kThreads / 32];
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
#pragma unroll
    for (int j = 0; j < Q; ++j) {
        const double v = warp_sum(acc[j].value());
        if (l == 0) part[j][w] = v;
    }
    __syncthreads();
    if (threadIdx.x < Q) {
        double total = 0.0;
        for (int i = 0; i < static_cast<int>(blockDim.x >> 5); ++i) total += part[threadIdx.x][i];
        partial[static_cast<int64_t>(blockIdx.x) * Q + threadIdx.x] = total;
    }
}

template <int M>
cudaError_t launch_pseudo_grad_stats_t(const float *x, const float *anchor, int64_t n, int num_sms,
                                       double *partial, size_t partial_cap, double *stats,
                                       cudaStream_t stream) {
    constexpr int Q = 2 * M + 2;
    static const int per_sm = blocks_per_sm(pseudo_grad_stats_kernel<M>);
    int64_t gx = static_cast<int64_t>(per_sm) * num_sms;
    const int64_t need = (n / 4 + kThreads - 1) / kThreads;
    if (gx > need) gx = need;
    if (gx < 1) gx = 1;
    if (static_cast<size_t>(gx) * Q > partial_cap) return cudaErrorInvalidValue;
    pseudo_grad_stats_kernel<M><<<static_cast<unsigned>(gx), kThreads, 0, stream>>>(x, anchor, n, partial);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    // same fixed-order finalisation as the sync diagnostics, with no division
    sync_stats_finalize_kernel<<<1, 32, 0, stream>>>(partial, static_cast<int>(gx), Q, 0, stats);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_pseudo_grad_stats(const float *x, const float *anchor, int64_t n, int M, int num_sms,
                                     double *partial, size_t partial_cap, double *stats,
                                     cudaStream_t stream) {
    switch (M) {
        case 1: return launch_pseudo_grad_stats_t<1>(x, anchor, n, num_sms, partial, partial_cap, stats, stream);
        case 2: return launch_pseudo_grad_stats_t<2>(x, anchor, n, num_sms, partial, partial_cap, stats, stream);
        case 3: return launch_pseudo_grad_stats_t<3>(x, anchor, n, num_sms, partial, partial_cap, stats, stream);
        case 4: return launch_pseudo_grad_stats_t<4>(x, anchor, n, num_sms, partial, partial_cap, stats, stream);
        case 5: return launch_pseudo_grad_stats_t<5>(x, anchor, n, num_sms, partial, partial_cap, stats, stream);
        case 6: return launch_pseudo_grad_stats_t<6>(x, anchor, n, num_sms, partial, partial_cap, stats, stream);
        case 7: return launch_pseudo_grad_stats_t<7>(x, anchor, n, num_sms, partial, partial_cap, stats, stream);
        case 8: return launch_pseudo_grad_stats_t<8>(x, anchor, n, num_sms, partial, partial_cap, stats, stream);
        default: return cudaErrorNotSupported;
    }
}

size_t sync_stats_partial_capacity(int num_sms, int n_states, int M) {
    // at most 16 resident blocks per SM of 256 threads, split over the states
    return static_cast<size_t>(16 * num_sms + n_states) * (2 + 2 * M);
}

cudaError_t launch_sync_stats(const SyncArgs &a, int num_sms, double *partial, size_t partial_cap,
                              double *stats, cudaStream_t stream) {
    if (a.n_sel <= 0) return cudaSuccess;
    switch (a.M) {
        case 1: return launch_sync_stats_t<1>(a, num_sms, partial, partial_cap, stats, stream);
        case 2: return launch_sync_stats_t<2>(a, num_sms, partial, partial_cap, stats, stream);
        case 3: return launch_sync_stats_t<3>(a, num_sms, partial, partial_cap, stats, stream);
        case 4: return launch_sync_stats_t<4>(a, num_sms, partial, partial_cap, stats, stream);
        case 5: return launch_sync_stats_t<5>(a, num_sms, partial, partial_cap, stats, stream);
        case 6: return launch_sync_stats_t<6>(a, num_sms, partial, partial_cap, stats, stream);
        case 7: return launch_sync_stats_t<7>(a, num_sms, partial, partial_cap, stats, stream);
        case 8: return launch_sync_stats_t<8>(a, num_sms, partial, partial_cap, stats, stream);
        default: return cudaErrorNotSupported;
    }
}

cudaError_t launch_sync(const SyncArgs &a, int num_sms, cudaStream_t stream) {
    if (a.n_sel <= 0 || a.M <= 1) return cudaSuccess;
    switch (a.M) {
        case 2: return launch_sync_t<2>(a, num_sms, stream);
        case 4: return launch_sync_t<4>(a, num_sms, stream);
        case 8: return launch_sync_t<8>(a, num_sms, stream);
        default: return launch_sync_t<0>(a, num_sms, stream);
    }
}

int norm_blocks_per_replica(int num_sms, int M) {
    int b = (4 * num_sms) / (M > 0 ? M : 1);
    return b < 1 ? 1 : b;
}

cudaError_t launch_grad_nonfinite(const void *grads, int grad_dtype, int32_t M, int64_t n_padded,
                                  int blocks_per_replica, double *partial, double *out, cudaStream_t stream) {
    dim3 grid(static_cast<unsigned>(blocks_per_replica), static_cast<unsigned>(M));
    if (grad_dtype == MTDAO_F32)
        nonfinite_partial_kernel<MTDAO_F32><<<grid, kNormThreads, 0, stream>>>(grads, n_padded, partial);
    else
        nonfinite_partial_kernel<MTDAO_BF16><<<grid, kNormThreads, 0, stream>>>(grads, n_padded, partial);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    sqnorm_finalize_kernel<<<M, kNormThreads, 0, stream>>>(partial, blocks_per_replica, out, nullptr, 0.0);
    return cudaGetLastError();
}

cudaError_t launch_grad_sqnorm(const void *grads, int grad_dtype, int32_t M, int64_t n_padded,
                               int blocks_per_replica, double *partial, double *out,
                               float *clip_scale, double rho, cudaStream_t stream) {
    dim3 grid(static_cast<unsigned>(blocks_per_replica), static_cast<unsigned>(M));
    if (grad_dtype == MTDAO_F32)
        sqnorm_partial_kernel<MTDAO_F32><<<grid, kNormThreads, 0, stream>>>(grads, n_padded, partial);
    else
        sqnorm_partial_kernel<MTDAO_BF16><<<grid, kNormThreads, 0, stream>>>(grads, n_padded, partial);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    sqnorm_finalize_kernel<<<M, kNormThreads, 0, stream>>>(partial, blocks_per_replica, out, clip_scale,
                                                          rho);
    return cudaGetLastError();
}

}  // namespace mtdao
