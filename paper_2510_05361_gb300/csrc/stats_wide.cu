// stats_wide.cu -- the cross-worker diagnostics of section 4.1 in one pass
// for 9 <= M <= 64 replicas (the kernels take up to kWideMaxM = 256; above
// 64 the library uses the two-pass form of reduce_kernels.cu, whose
// register-resident kernels cover M <= 8).
//
// Same block layout as the wide fused step (step_sync_wide.cuh): a block
// owns spans of S consecutive elements of all M replicas, thread (r, f)
// copies 16 elements of replica r (four float4 positions f, f + P, ...) into
// a shared M x S tile (double-buffered with cp.async), the
// span's replica means are formed from the tile by tile_means (the bits of
// the standalone average), and each thread then forms its own replica's
// sums against the mean.  Every replica value is read from HBM once; the
// sync diagnostics write the mean over it (the average itself), so a sync
// with diagnostics moves the bytes of a plain sync.
//
// Sums are bit-reproducible: a thread's 16 elements of a span are summed in
// fp32, each thread accumulates its spans with Kahan compensation, the P
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

// float4 positions per thread and span: the span is S = 4 * P * kStatsVec
// elements (rows of 128 bytes or more for every M up to 256).
constexpr int kStatsVec = 4;
constexpr int kStatsVecLog2 = 2;

// Copies this thread's kStatsVec float4 positions of replica r of a span
// (src: the replica's first element of the span) into its tile row, then
// commits the group (an empty one when the span is past the end).
__device__ __forceinline__ void fetch_row(bool live, float *dst, const float *src, int P) {
    if (live) {
#pragma unroll
        for (int j = 0; j < kStatsVec; ++j) cp_async16(dst + 4 * P * j, src + 4 * P * j);
    }
    cp_async_commit();
}

// Sync diagnostics of the selected state blockIdx.y, partial row per block:
//   q = 0          sum_m sum_i (s_m - s_bar)^2
//   q = 1          sum_i s_bar^2
//   q = 2 + m      sum_i s_m^2
//   q = 2 + M + m  sum_i s_m * s_bar
// at partial[(blockIdx.y * gridDim.x + blockIdx.x) * Q + q], Q = 2 + 2M;
// s_bar (the fp32 mean) is written over every replica.
template <bool FOUR>
__global__ void __launch_bounds__(kWideMaxThreads) sync_stats_wide_kernel(const SyncArgs a, int log2_p,
                                                                          double *partial) {
    extern __shared__ __align__(16) float smem[];
    constexpr int NV = kStatsVec;
    const int M = a.M;
    const int P = 1 << log2_p;
    const int log2_s = log2_p + 2 + kStatsVecLog2;
    const int S = 1 << log2_s;
    const int Q = 2 + 2 * M;
    const int t = threadIdx.x;
    const int r = t >> log2_p;
    const int f = t & (P - 1);
    const bool live = r < M;
    float *base = a.arena + static_cast<int64_t>(a.sel[blockIdx.y]) * a.stride;
    const int64_t n = a.n_padded;
    const int64_t n_spans = n / S;
    float *tiles = smem;                         // [2][M][S]
    float *mean = smem + 2 * M * S;              // [S]
    Kahan dev, sq, cross, msq;

    const int64_t first = blockIdx.x;
    fetch_row(live && first < n_spans, tiles + r * S + 4 * f, base + r * n + first * S + 4 * f, P);
    int buf = 0;
    for (int64_t span = first; span < n_spans; span += gridDim.x, buf ^= 1) {
        const int64_t next = span + gridDim.x;
        fetch_row(live && next < n_spans, tiles + ((buf ^ 1) * M + r) * S + 4 * f,
                  base + r * n + next * S + 4 * f, P);
        cp_async_wait<1>();                      // this thread's copies of `span` have landed
        __syncthreads();                         // ... and every thread's
        const float *tile = tiles + buf * M * S;
        tile_means<FOUR>(tile, M, log2_s, S, mean);
        __syncthreads();
        if (live) {
            float p0 = 0.0f, p1 = 0.0f, p2 = 0.0f, p3 = 0.0f;   // this thread's 4 * NV elements
#pragma unroll
            for (int j = 0; j < NV; ++j) {
                const int c = 4 * f + 4 * P * j;
                float x[4], mb[4];
                to_array(*reinterpret_cast<const float4 *>(tile + r * S + c), x);
                const float4 mv = *reinterpret_cast<const float4 *>(mean + c);
                to_array(mv, mb);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const float dv = x[k] - mb[k];
                    p0 = fmaf(dv, dv, p0);
                    p1 = fmaf(x[k], x[k], p1);
                    p2 = fmaf(x[k], mb[k], p2);
                    p3 = fmaf(mb[k], mb[k], p3);
                }
                st_state(base + r * n + span * S + c, mv);
            }
            dev.add(p0);
            sq.add(p1);
            cross.add(p2);
            if (r == 0) msq.add(p3);
        }
        __syncthreads();                         // this tile and the means are rewritten next
    }
    cp_async_wait<0>();

    // Per replica: its P lanes' sums; then one row of Q values.
    const double d = replica_lanes_sum(dev.value(), P);
    const double s2 = replica_lanes_sum(sq.value(), P);
    const double c2 = replica_lanes_sum(cross.value(), P);
    const double m2 = replica_lanes_sum(msq.value(), P);   // replica 0's lanes hold sum s_bar^2
    double *red = reinterpret_cast<double *>(smem);        // [3][M] + 1, over the (now idle) tiles
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
// The anchor's span travels with replica 0's row (one more tile row).
template <bool FOUR>
__global__ void __launch_bounds__(kWideMaxThreads) pseudo_grad_stats_wide_kernel(const float *x,
                                                                                 const float *anchor,
                                                                                 int64_t n, int M, int log2_p,
                                                                                 double *partial) {
    extern __shared__ __align__(16) float smem[];
    constexpr int NV = kStatsVec;
    const int P = 1 << log2_p;
    const int log2_s = log2_p + 2 + kStatsVecLog2;
    const int S = 1 << log2_s;
    const int Q = 2 * M + 2;
    const int t = threadIdx.x;
    const int r = t >> log2_p;
    const int f = t & (P - 1);
    const bool live = r < M;
    const int64_t n_spans = n / S;
    const int R = M + 1;                         // tile rows: the replicas, then the anchor
    float *tiles = smem;                         // [2][M + 1][S]
    float *mean = smem + 2 * R * S;              // [S]
    Kahan loc2, cross, glob2, a2;

    auto fetch = [&](int64_t span, int b) {
        const bool ok = live && span < n_spans;
        if (ok && r == 0) {
#pragma unroll
            for (int j = 0; j < NV; ++j)
                cp_async16(tiles + (b * R + M) * S + 4 * f + 4 * P * j, anchor + span * S + 4 * f + 4 * P * j);
        }
        fetch_row(ok, tiles + (b * R + r) * S + 4 * f, x + r * n + span * S + 4 * f, P);
    };
    fetch(blockIdx.x, 0);
    int buf = 0;
    for (int64_t span = blockIdx.x; span < n_spans; span += gridDim.x, buf ^= 1) {
        fetch(span + gridDim.x, buf ^ 1);
        cp_async_wait<1>();
        __syncthreads();
        const float *tile = tiles + buf * R * S;
        const float *anc = tile + M * S;
        tile_means<FOUR>(tile, M, log2_s, S, mean);
        __syncthreads();
        if (live) {
            float p0 = 0.0f, p1 = 0.0f, p2 = 0.0f, p3 = 0.0f;   // this thread's 4 * NV elements
#pragma unroll
            for (int j = 0; j < NV; ++j) {
                const int c = 4 * f + 4 * P * j;
                float xv[4], mb[4], aj[4];
                to_array(*reinterpret_cast<const float4 *>(tile + r * S + c), xv);
                to_array(*reinterpret_cast<const float4 *>(mean + c), mb);
                to_array(*reinterpret_cast<const float4 *>(anc + c), aj);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const float loc = xv[k] - aj[k];
                    const float glob = mb[k] - aj[k];
                    p0 = fmaf(loc, loc, p0);
                    p1 = fmaf(loc, glob, p1);
                    p2 = fmaf(glob, glob, p2);
                    p3 = fmaf(aj[k], aj[k], p3);
                }
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
    cp_async_wait<0>();

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

WideShape wide_shape(int M, int extra_rows) {
    WideShape w;
    const int P = wide_positions(M);
    w.log2_p = 0;
    while ((1 << w.log2_p) < P) ++w.log2_p;
    w.S = 4 * P * kStatsVec;
    w.threads = (M * P + 31) / 32 * 32;
    // two tiles of M (+ extra) rows and the span's means; the final
    // reduction reuses the tiles
    const size_t floats = 2 * static_cast<size_t>(M + extra_rows) * w.S + w.S;
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

namespace {

template <bool FOUR>
cudaError_t launch_sync_stats_wide_t(const SyncArgs &a, int num_sms, double *partial, size_t partial_cap,
                                     double *stats, cudaStream_t stream) {
    if (a.n_sel <= 0) return cudaSuccess;
    if (a.M < 2 || a.M > kWideMaxM) return cudaErrorNotSupported;
    const int Q = 2 + 2 * a.M;
    const WideShape w = wide_shape(a.M, 0);
    if (w.smem > 48 * 1024) {        // before the occupancy query, which depends on it
        cudaError_t e = cudaFuncSetAttribute(sync_stats_wide_kernel<FOUR>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(w.smem));
        if (e != cudaSuccess) return e;
    }
    const int per_sm = wide_blocks_per_sm(sync_stats_wide_kernel<FOUR>, w);
    if (static_cast<size_t>(Q) * a.n_sel > partial_cap) return cudaErrorInvalidValue;
    const int g = wide_grid(per_sm, num_sms, a.n_sel, a.n_padded / w.S, Q, partial_cap);
    sync_stats_wide_kernel<FOUR><<<dim3(g, a.n_sel), w.threads, w.smem, stream>>>(a, w.log2_p, partial);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    wide_stats_finalize_kernel<<<dim3((Q + 255) / 256, a.n_sel), 256, 0, stream>>>(partial, g, Q, a.M, stats);
    return cudaGetLastError();
}

template <bool FOUR>
cudaError_t launch_pseudo_grad_stats_wide_t(const float *x, const float *anchor, int64_t n, int M, int num_sms,
                                            double *partial, size_t partial_cap, double *stats,
                                            cudaStream_t stream) {
    if (M < 2 || M > kWideMaxM) return cudaErrorNotSupported;
    const int Q = 2 * M + 2;
    const WideShape w = wide_shape(M, 1);
    if (w.smem > 48 * 1024) {        // before the occupancy query, which depends on it
        cudaError_t e = cudaFuncSetAttribute(pseudo_grad_stats_wide_kernel<FOUR>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(w.smem));
        if (e != cudaSuccess) return e;
    }
    const int per_sm = wide_blocks_per_sm(pseudo_grad_stats_wide_kernel<FOUR>, w);
    if (static_cast<size_t>(Q) > partial_cap) return cudaErrorInvalidValue;
    const int g = wide_grid(per_sm, num_sms, 1, n / w.S, Q, partial_cap);
    pseudo_grad_stats_wide_kernel<FOUR><<<g, w.threads, w.smem, stream>>>(x, anchor, n, M, w.log2_p, partial);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    wide_stats_finalize_kernel<<<dim3((Q + 255) / 256, 1), 256, 0, stream>>>(partial, g, Q, 0, stats);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_sync_stats_wide(const SyncArgs &a, int num_sms, double *partial, size_t partial_cap,
                                   double *stats, cudaStream_t stream) {
    return wide_four_columns(a.M) ? launch_sync_stats_wide_t<true>(a, num_sms, partial, partial_cap, stats, stream)
                                  : launch_sync_stats_wide_t<false>(a, num_sms, partial, partial_cap, stats, stream);
}

cudaError_t launch_pseudo_grad_stats_wide(const float *x, const float *anchor, int64_t n, int M, int num_sms,
                                          double *partial, size_t partial_cap, double *stats,
                                          cudaStream_t stream) {
    return wide_four_columns(M)
               ? launch_pseudo_grad_stats_wide_t<true>(x, anchor, n, M, num_sms, partial, partial_cap, stats, stream)
               : launch_pseudo_grad_stats_wide_t<false>(x, anchor, n, M, num_sms, partial, partial_cap, stats, stream);
}

}  // namespace mtdao
