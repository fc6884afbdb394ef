// stats_wide.cu -- the cross-worker diagnostics of section 4.1 in one pass
// for 9 <= M <= kWideMaxM replicas (the register-resident kernels of
// reduce_kernels.cu hold up to 8).
//
// Same block layout as the wide fused step (step_sync_wide.cuh): a block
// owns spans of S consecutive elements of all M replicas, thread (r, f)
// loads elements [4f, 4f + 4) of replica r into a shared M x S tile, the
// span's replica means are formed from the tile by tile_means (the bits of
// the standalone average), and each thread then forms its own replica's
// sums against the mean.  Every replica value is read from HBM once; the
// sync diagnostics write the mean over it (the average itself), so a sync
// with diagnostics moves the bytes of a plain sync.
//
// Sums are bit-reproducible: a position's four elements are summed in fp32,
// each thread accumulates its positions with Kahan compensation, the P
// threads of a replica combine in fp64 by a fixed shuffle pattern, the
// block writes one partial row, and a finalize kernel adds the rows in
// block order.  The grid is persistent (spans strided by the grid), so the
// partial rows stay few.
#include <cuda_runtime.h>
#include <cstdint>

#include "kahan.cuh"
#include "mtdao_internal.h"
#include "replica_mean.cuh"
#include "step_kernels.cuh"
#include "step_sync_wide.cuh"

namespace mtdao {

namespace {

// Sum over the P lanes of one replica (aligned groups of P lanes, P a power
// of two dividing 32): every lane of the group ends with the same value.
__device__ __forceinline__ double replica_lanes_sum(double v, int P) {
    for (int off = P >> 1; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    return v;
}

// Sync diagnostics of the selected state blockIdx.y, partial row per block:
//   q = 0          sum_m sum_i (s_m - s_bar)^2
//   q = 1          sum_i s_bar^2
//   q = 2 + m      sum_i s_m^2
//   q = 2 + M + m  sum_i s_m * s_bar
// at partial[(blockIdx.y * gridDim.x + blockIdx.x) * Q + q], Q = 2 + 2M;
// s_bar (the fp32 mean) is written over every replica.
__global__ void __launch_bounds__(kWideMaxThreads) sync_stats_wide_kernel(const SyncArgs a, int log2_p,
                                                                          double *partial) {
    extern __shared__ float smem[];
    const int M = a.M;
    const int P = 1 << log2_p;
    const int S = 4 * P;
    const int Q = 2 + 2 * M;
    const int t = threadIdx.x;
    const int r = t >> log2_p;
    const int f = t & (P - 1);
    const bool live = r < M;
    float *base = a.arena + static_cast<int64_t>(a.sel[blockIdx.y]) * a.stride;
    const int64_t n = a.n_padded;
    const int64_t n_spans = n / S;
    float *tile = smem;                          // [M][S]
    float *mean = smem + M * S;                  // [S]
    Kahan dev, sq, cross, msq;

    for (int64_t span = blockIdx.x; span < n_spans; span += gridDim.x) {
        const int64_t e = span * S + 4 * f;
        float x[4] = {0.0f, 0.0f, 0.0f, 0.0f};
        if (live) {
            const float4 v = ld_state(base + r * n + e);
            to_array(v, x);
            *reinterpret_cast<float4 *>(tile + r * S + 4 * f) = v;
        }
        __syncthreads();
        tile_means(tile, M, S, S, mean);
        __syncthreads();
        if (live) {
            const float4 mv = *reinterpret_cast<const float4 *>(mean + 4 * f);
            float mb[4];
            to_array(mv, mb);
            float p0 = 0.0f, p1 = 0.0f, p2 = 0.0f, p3 = 0.0f;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float dv = x[k] - mb[k];
                p0 = fmaf(dv, dv, p0);
                p1 = fmaf(x[k], x[k], p1);
                p2 = fmaf(x[k], mb[k], p2);
                p3 = fmaf(mb[k], mb[k], p3);
            }
            dev.add(p0);
            sq.add(p1);
            cross.add(p2);
            if (r == 0) msq.add(p3);
            st_state(base + r * n + e, mv);
        }
        __syncthreads();                         // the tile is reused by the next span
    }

    // Per replica: its P lanes' sums; then one row of Q values.
    const double d = replica_lanes_sum(dev.value(), P);
    const double s2 = replica_lanes_sum(sq.value(), P);
    const double c2 = replica_lanes_sum(cross.value(), P);
    const double m2 = replica_lanes_sum(msq.value(), P);   // replica 0's lanes hold sum s_bar^2
    double *red = reinterpret_cast<double *>(smem);        // [3][M] + 1, over the (now idle) tile
    if (live && f == 0) {
        red[r] = d;
        red[M + r] = s2;
        red[2 * M + r] = c2;
        if (r == 0) red[3 * M] = m2;
    }
    __syncthreads();
    double *row = partial + (static_cast<int64_t>(blockIdx.y) * gridDim.x + blockIdx.x) * Q;
    for (int q = t; q < Q; q += blockDim.x) {
        double v;
        if (q == 0) {
            v = 0.0;
            for (int m = 0; m < M; ++m) v += red[m];
        } else if (q == 1) {
            v = red[3 * M];
        } else if (q < 2 + M) {
            v = red[M + (q - 2)];
        } else {
            v = red[2 * M + (q - 2 - M)];
        }
        row[q] = v;
    }
}

// Pseudo-gradient diagnostics of x[M][n] against the anchor a[n], read-only;
// partial row per block (Q = 2M + 2):
//   q = m          sum_i (x_m - a)^2
//   q = M + m      sum_i (x_m - a) * (x_bar - a)
//   q = 2M         sum_i (x_bar - a)^2
//   q = 2M + 1     sum_i a^2
__global__ void __launch_bounds__(kWideMaxThreads) pseudo_grad_stats_wide_kernel(const float *x,
                                                                                 const float *anchor,
                                                                                 int64_t n, int M, int log2_p,
                                                                                 double *partial) {
    extern __shared__ float smem[];
    const int P = 1 << log2_p;
    const int S = 4 * P;
    const int Q = 2 * M + 2;
    const int t = threadIdx.x;
    const int r = t >> log2_p;
    const int f = t & (P - 1);
    const bool live = r < M;
    const int64_t n_spans = n / S;
    float *tile = smem;                          // [M][S]
    float *mean = smem + M * S;                  // [S]
    float *anc = mean + S;                       // [S]
    Kahan loc2, cross, glob2, a2;

    for (int64_t span = blockIdx.x; span < n_spans; span += gridDim.x) {
        const int64_t e = span * S + 4 * f;
        float xv[4] = {0.0f, 0.0f, 0.0f, 0.0f};
        if (live) {
            const float4 v = ld_state(x + r * n + e);
            to_array(v, xv);
            *reinterpret_cast<float4 *>(tile + r * S + 4 * f) = v;
            if (r == 0)
                *reinterpret_cast<float4 *>(anc + 4 * f) = __ldcs(reinterpret_cast<const float4 *>(anchor + e));
        }
        __syncthreads();
        tile_means(tile, M, S, S, mean);
        __syncthreads();
        if (live) {
            float mb[4], av[4];
            to_array(*reinterpret_cast<const float4 *>(mean + 4 * f), mb);
            to_array(*reinterpret_cast<const float4 *>(anc + 4 * f), av);
            float p0 = 0.0f, p1 = 0.0f, p2 = 0.0f, p3 = 0.0f;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float loc = xv[k] - av[k];
                const float glob = mb[k] - av[k];
                p0 = fmaf(loc, loc, p0);
                p1 = fmaf(loc, glob, p1);
                p2 = fmaf(glob, glob, p2);
                p3 = fmaf(av[k], av[k], p3);
            }
            loc2.add(p0);
            cross.add(p1);
            if (r == 0) {
                glob2.add(p2);
                a2.add(p3);
            }
        }
        __syncthreads();
    }

    const double l2 = replica_lanes_sum(loc2.value(), P);
    const double c2 = replica_lanes_sum(cross.value(), P);
    const double g2 = replica_lanes_sum(glob2.value(), P);
    const double aa = replica_lanes_sum(a2.value(), P);
    double *red = reinterpret_cast<double *>(smem);        // [2][M] + 2
    if (live && f == 0) {
        red[r] = l2;
        red[M + r] = c2;
        if (r == 0) {
            red[2 * M] = g2;
            red[2 * M + 1] = aa;
        }
    }
    __syncthreads();
    double *row = partial + static_cast<int64_t>(blockIdx.x) * Q;
    for (int q = t; q < Q; q += blockDim.x) row[q] = red[q];
}

// out[row * Q + q] = sum over blocks b (in order) of partial[(row * blocks + b) * Q + q];
// q = 0 divided by divide_first when that is > 0.
__global__ void wide_stats_finalize_kernel(const double *partial, int blocks, int Q, int divide_first,
                                           double *out) {
    const int row = blockIdx.y;
    const int q = blockIdx.x * blockDim.x + threadIdx.x;
    if (q >= Q) return;
    double total = 0.0;
    for (int b = 0; b < blocks; ++b) total += partial[(static_cast<int64_t>(row) * blocks + b) * Q + q];
    out[static_cast<int64_t>(row) * Q + q] = (q == 0 && divide_first > 0) ? total / divide_first : total;
}

struct WideShape {
    int log2_p, S, threads;
    size_t smem;
};

WideShape wide_shape(int M, int extra_floats) {
    WideShape w;
    const int P = wide_positions(M);
    w.log2_p = 0;
    while ((1 << w.log2_p) < P) ++w.log2_p;
    w.S = 4 * P;
    w.threads = (M * P + 31) / 32 * 32;
    // the tile and the extra per-span vectors; the final reduction reuses it
    size_t floats = static_cast<size_t>(M) * w.S + extra_floats * w.S;
    const size_t red = 2 * (3 * static_cast<size_t>(M) + 2);   // doubles -> floats
    w.smem = (floats > red ? floats : red) * sizeof(float);
    return w;
}

template <typename Kernel>
int wide_blocks_per_sm(Kernel kernel, const WideShape &w) {
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, w.threads, w.smem) != cudaSuccess ||
        per_sm < 1) {
        cudaGetLastError();
        per_sm = 1;
    }
    return per_sm;
}

// Blocks per selected state: the device's resident blocks shared over the
// states, at most one per span, within the workspace.
int wide_grid(int per_sm, int num_sms, int n_sel, int64_t n_spans, int Q, size_t partial_cap) {
    int64_t g = static_cast<int64_t>(per_sm) * num_sms / (n_sel > 0 ? n_sel : 1);
    if (g > n_spans) g = n_spans;
    const int64_t fit = static_cast<int64_t>(partial_cap / (static_cast<size_t>(Q) * (n_sel > 0 ? n_sel : 1)));
    if (g > fit) g = fit;
    return static_cast<int>(g < 1 ? 1 : g);
}

}  // namespace

size_t wide_stats_partial_capacity(int num_sms, int n_states, int M) {
    // at most 32 resident blocks per SM, shared over the states
    return static_cast<size_t>(32 * num_sms + n_states) * (2 + 2 * static_cast<size_t>(M));
}

cudaError_t launch_sync_stats_wide(const SyncArgs &a, int num_sms, double *partial, size_t partial_cap,
                                   double *stats, cudaStream_t stream) {
    if (a.n_sel <= 0) return cudaSuccess;
    if (a.M < 2 || a.M > kWideMaxM) return cudaErrorNotSupported;
    const int Q = 2 + 2 * a.M;
    const WideShape w = wide_shape(a.M, 1);
    const int per_sm = wide_blocks_per_sm(sync_stats_wide_kernel, w);
    if (static_cast<size_t>(Q) * a.n_sel > partial_cap) return cudaErrorInvalidValue;
    const int g = wide_grid(per_sm, num_sms, a.n_sel, a.n_padded / w.S, Q, partial_cap);
    if (w.smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(sync_stats_wide_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(w.smem));
        if (e != cudaSuccess) return e;
    }
    sync_stats_wide_kernel<<<dim3(g, a.n_sel), w.threads, w.smem, stream>>>(a, w.log2_p, partial);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    wide_stats_finalize_kernel<<<dim3((Q + 255) / 256, a.n_sel), 256, 0, stream>>>(partial, g, Q, a.M, stats);
    return cudaGetLastError();
}

cudaError_t launch_pseudo_grad_stats_wide(const float *x, const float *anchor, int64_t n, int M, int num_sms,
                                          double *partial, size_t partial_cap, double *stats,
                                          cudaStream_t stream) {
    if (M < 2 || M > kWideMaxM) return cudaErrorNotSupported;
    const int Q = 2 * M + 2;
    const WideShape w = wide_shape(M, 2);
    const int per_sm = wide_blocks_per_sm(pseudo_grad_stats_wide_kernel, w);
    if (static_cast<size_t>(Q) > partial_cap) return cudaErrorInvalidValue;
    const int g = wide_grid(per_sm, num_sms, 1, n / w.S, Q, partial_cap);
    if (w.smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(pseudo_grad_stats_wide_kernel,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(w.smem));
        if (e != cudaSuccess) return e;
    }
    pseudo_grad_stats_wide_kernel<<<g, w.threads, w.smem, stream>>>(x, anchor, n, M, w.log2_p, partial);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    wide_stats_finalize_kernel<<<dim3((Q + 255) / 256, 1), 256, 0, stream>>>(partial, g, Q, 0, stats);
    return cudaGetLastError();
}

}  // namespace mtdao
