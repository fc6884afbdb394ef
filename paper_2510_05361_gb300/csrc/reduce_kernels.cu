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
#include "kahan.cuh"
#include "replica_mean.cuh"
#include "step_kernels.cuh"

namespace mtdao {

namespace {

// Mean of the M replicas at float4 position e of state s, M known at run
// time (the standalone average above 8 replicas and the two-pass
// diagnostics): replica_mean.cuh's operations in its order, four replicas'
// loads in flight (one at a time, the average of M = 9-64 ran at 5.5-5.8
// TB/s).
__device__ __forceinline__ float4 replica_mean4(const float *s, int64_t n, int M, int64_t e) {
    float s0[4];
    to_array(ld_state(s + e), s0);
    DiffSum pa[4] = {DiffSum(s0[0]), DiffSum(s0[1]), DiffSum(s0[2]), DiffSum(s0[3])};
    DiffSum pb[4] = {DiffSum(s0[0]), DiffSum(s0[1]), DiffSum(s0[2]), DiffSum(s0[3])};
    float plain[4] = {s0[0], s0[1], s0[2], s0[3]};
    const int h = M / 2;
    for (int m = 1; m < M; m += 4) {          // four replicas' loads in flight, added in order
        float r[4][4];
#pragma unroll
        for (int u = 0; u < 4; ++u)
            if (m + u < M) to_array(ld_state(s + (m + u) * n + e), r[u]);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            if (m + u >= M) break;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                if (m + u < h) pa[k].add(r[u][k]);
                else pb[k].add(r[u][k]);
                plain[k] += r[u][k];
            }
        }
    }
    float mean[4];
#pragma unroll
    for (int k = 0; k < 4; ++k)
        mean[k] = mean_or_plain(
            replica_mean_from_parts(s0[k], pa[k].partial(), pb[k].partial(), static_cast<float>(M)), plain[k],
            static_cast<float>(M));
    return from_array(mean);
}

template <int MT>
__global__ void __launch_bounds__(kThreads) sync_kernel(const SyncArgs a) {
    const int M = MT > 0 ? MT : a.M;
    float *base = a.arena + static_cast<int64_t>(a.sel[blockIdx.y]) * a.stride;
    const int64_t n = a.n_padded;
    const int64_t nv = n / 4;
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
            to_array(replica_mean4(base, n, M, e), mean);
        }
        const float4 mv = from_array(mean);
        for (int m = 0; m < M; ++m) st_state(base + m * n + e, mv);
    }
}

template <int MT>
cudaError_t launch_sync_t(const SyncArgs &a, int num_sms, cudaStream_t stream) {
    // M = 2 .. 14 (replicas held in registers): one float4 position per
    // thread, like the local step's stream_grid (flat 2^27, all states, GB/s
    // against the persistent grid: M = 2 6342 -> 7098, M = 4 6447 -> 7025,
    // M = 8 6546 -> 6941; flat 2^30 replica-elements against the streamed
    // loop: M = 3 4588 -> 6336, 5-7 5069 -> 6609-6658, 9-14 5564 -> 6343-6784).
    // At 15 and 16 the replicas take 151-176 registers (M = 16: 5086 against
    // 5796 streamed).  The streamed runtime-M loop (M > 14) keeps the
    // persistent grid (one position per thread: 3-7 % slower at M = 9-64).
    const int64_t nv = a.n_padded / 4;
    const int64_t need = (nv + kThreads - 1) / kThreads;
    int64_t gx;
    if constexpr (MT > 0) {
        gx = need > 0x7fffffff ? 0x7fffffff : need;
    } else {
        static const int per_sm = blocks_per_sm(sync_kernel<MT>);
        gx = static_cast<int64_t>(per_sm) * num_sms / (a.n_sel > 0 ? a.n_sel : 1);
        if (gx > need) gx = need;
    }
    if (gx < 1) gx = 1;
    dim3 grid(static_cast<unsigned>(gx), static_cast<unsigned>(a.n_sel));
    sync_kernel<MT><<<grid, kThreads, 0, stream>>>(a);
    return cudaGetLastError();
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

// A position of the norm kernels is one 16-byte load of the gradient: 4 f32
// or 8 bf16 values (8-byte bf16 loads, half the bytes per load instruction,
// read the ~350M workload's gradients at 5.56 TB/s).  A thread loads
// kNormUnroll positions before it accumulates them: i, i + T, ...,
// i + (U - 1) T with T the replica's thread count, the same order as a
// plain grid-stride loop, so the sums do not depend on the unrolling.
// 64 bytes per thread in flight.
constexpr int kNormUnroll = 4;

template <int GDT>
struct NormPos;
template <>
struct NormPos<MTDAO_F32> {
    static constexpr int E = 4;
    using W = float4;
};
template <>
struct NormPos<MTDAO_BF16> {
    static constexpr int E = 8;
    using W = uint4;
};

template <int GDT>
__device__ __forceinline__ typename NormPos<GDT>::W ld_grad_words(const void *g, int64_t e) {
    if constexpr (GDT == MTDAO_F32)
        return __ldcs(reinterpret_cast<const float4 *>(static_cast<const float *>(g) + e));
    else
        return __ldcs(reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(g) + e));
}

// The position's values in fp32 (bf16 -> fp32 is exact: the bits move up by 16).
template <int GDT>
__device__ __forceinline__ void widen(const typename NormPos<GDT>::W &w, float (&q)[NormPos<GDT>::E]) {
    if constexpr (GDT == MTDAO_F32) {
        q[0] = w.x; q[1] = w.y; q[2] = w.z; q[3] = w.w;
    } else {
        const uint32_t u[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            q[2 * k] = __uint_as_float(u[k] << 16);
            q[2 * k + 1] = __uint_as_float(u[k] & 0xffff0000u);
        }
    }
}

// fp32 range of a position's sum of four squares that the Kahan sum takes:
// above kSqHi a square or the sum may overflow (|g| above ~1.8e19 squares to
// Inf in fp32), below kSqLo a square may have lost bits to underflow (|g|
// below ~1e-19).  Positions outside it (and NaN / Inf) are summed in fp64
// instead, where every finite fp32 value squares exactly enough; the all-zero
// positions of padding and unused rows stay on the fp32 path.  A replica has
// at least 256 threads and, to fit in device memory, fewer than 2^34
// elements, so a thread adds fewer than 2^24 positions of at most 2^100:
// the fp32 sum stays finite.
constexpr float kSqHi = 0x1p100f;
constexpr float kSqLo = 0x1p-100f;

template <int GDT>
__global__ void __launch_bounds__(kNormThreads, 4) sqnorm_partial_kernel(const void *g, int64_t n,
                                                                      double *partial) {
    constexpr int E = NormPos<GDT>::E;
    const int m = blockIdx.y;
    const int nb = gridDim.x;
    const int64_t np = n / E;
    const int64_t T = static_cast<int64_t>(nb) * blockDim.x;
    float sum = 0.0f, comp = 0.0f;
    double wide = 0.0;                 // positions outside [kSqLo, kSqHi]
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < np;
         i += kNormUnroll * T) {
        typename NormPos<GDT>::W w[kNormUnroll];
#pragma unroll
        for (int u = 0; u < kNormUnroll; ++u)
            if (i + u * T < np) w[u] = ld_grad_words<GDT>(g, m * n + E * (i + u * T));
#pragma unroll
        for (int u = 0; u < kNormUnroll; ++u) {
            if (i + u * T >= np) break;
            float q[E];
            widen<GDT>(w[u], q);
            float p = __fmul_rn(q[E - 1], q[E - 1]);
            uint32_t bits = __float_as_uint(q[E - 1]);
#pragma unroll
            for (int k = E - 2; k >= 0; --k) {
                p = fmaf(q[k], q[k], p);
                bits |= __float_as_uint(q[k]);
            }
            const bool tiny = p < kSqLo && (bits & 0x7fffffffu) != 0u;
            if (!(p <= kSqHi) || tiny) {
                double d = static_cast<double>(q[E - 1]) * q[E - 1];
#pragma unroll
                for (int k = E - 2; k >= 0; --k) d = fma(static_cast<double>(q[k]), static_cast<double>(q[k]), d);
                wide += d;
                continue;
            }
            const float y = p - comp;
            const float t = sum + y;
            comp = (t - sum) - y;
            sum = t;
        }
    }
    const double total = block_sum((static_cast<double>(sum) - static_cast<double>(comp)) + wide);
    if (threadIdx.x == 0) partial[static_cast<int64_t>(m) * nb + blockIdx.x] = total;
}

// Number of NaN or +-Inf values (all exponent bits set) per replica, with
// the same fixed grid and reduction order as the sum of squares; counts are
// integers well below 2^53, so the double partials are exact.
template <int GDT>
__global__ void __launch_bounds__(kNormThreads, 4) nonfinite_partial_kernel(const void *g, int64_t n,
                                                                         double *partial) {
    constexpr int E = NormPos<GDT>::E;
    const int m = blockIdx.y;
    const int nb = gridDim.x;
    const int64_t np = n / E;
    const int64_t T = static_cast<int64_t>(nb) * blockDim.x;
    const uint32_t ex = 0x7f800000u;
    uint32_t count = 0;                // at most E np / T per thread
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < np;
         i += kNormUnroll * T) {
        typename NormPos<GDT>::W w[kNormUnroll];
#pragma unroll
        for (int u = 0; u < kNormUnroll; ++u)
            if (i + u * T < np) w[u] = ld_grad_words<GDT>(g, m * n + E * (i + u * T));
#pragma unroll
        for (int u = 0; u < kNormUnroll; ++u) {
            if (i + u * T >= np) break;
            float q[E];
            widen<GDT>(w[u], q);
#pragma unroll
            for (int k = 0; k < E; ++k) count += (__float_as_uint(q[k]) & ex) == ex;
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

// Float4 positions a thread of sync_stats_kernel takes, consecutive for its
// block: block b covers positions [b * tile * 256, (b + 1) * tile * 256).
// One block per tile, started in index order as earlier blocks retire;
// every block leaves one row of sums for stats_finalize_kernel, so the sums
// do not depend on the SM count.  A block's fixed cost is that row (2M + 2
// warp and block reductions in fp64), so the tile must be long.  On the ~1B
// and ~350M workloads this launch took the sync with diagnostics from
// 6426 / 6335 GB/s (persistent grid: occupancy x SMs blocks, grid-stride)
// to 6712 / 6696.  On flat 2^30-element sets (GB/s at M = 4 / 8):
// persistent 5943 / 6139; tiles of 2: 1621 / 1795, 8: 5638 / 4590,
// 32: 6152 / 6275, 128: 6121 / 6308, 512: 6051 / 6173.  The read-only
// pseudo-gradient pass keeps the persistent grid: with tiles of 512 it ran
// 6212 / 5908 GB/s on the two workloads against 7153 / 6237.
constexpr int kSyncStatsTile = 128;

// Replica average of the selected states (exactly as sync_kernel) plus, in
// the same pass over the M replicas, per state and block the partial sums of
//   q = 0          sum_m (s_m - s_bar)^2        (cross-worker variance * M)
//   q = 1          s_bar^2
//   q = 2 + m      s_m^2
//   q = 2 + M + m  s_m * s_bar
// written to partial[(sel * Q + q) * gridDim.x + block], Q = 2 + 2M.  s_bar
// is the fp32 mean that is stored.  With M = 1 nothing is stored (there is
// nothing to average) but the sums are still formed.
template <int M>
__global__ void __launch_bounds__(kThreads) sync_stats_kernel(const SyncArgs a, double *partial) {
    constexpr int Q = 2 + 2 * M;
    float *base = a.arena + static_cast<int64_t>(a.sel[blockIdx.y]) * a.stride;
    const int64_t n = a.n_padded;
    const int64_t nv = n / 4;
    Kahan acc[Q];
    const int64_t first = static_cast<int64_t>(blockIdx.x) * kSyncStatsTile * blockDim.x + threadIdx.x;
    for (int k = 0; k < kSyncStatsTile; ++k) {
        const int64_t i = first + static_cast<int64_t>(k) * blockDim.x;
        if (i >= nv) break;
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
        partial[(static_cast<int64_t>(blockIdx.y) * Q + threadIdx.x) * gridDim.x + blockIdx.x] = total;
    }
}

// stats[row * Q + q] = the sum over blocks of partial[(row * Q + q) * blocks + b]:
// thread t of block (q, row) adds a contiguous run of blocks in order, then
// block_sum adds the threads' sums in a fixed order.  q = 0 is divided by
// divide_first (M for the variance, a mean over workers; 0 leaves it).
__global__ void __launch_bounds__(kNormThreads) stats_finalize_kernel(const double *partial, int64_t blocks,
                                                                      int Q, int divide_first, double *stats) {
    const int q = blockIdx.x, row = blockIdx.y;
    const double *p = partial + (static_cast<int64_t>(row) * Q + q) * blocks;
    const int64_t per = (blocks + blockDim.x - 1) / blockDim.x;
    const int64_t lo = threadIdx.x * per;
    const int64_t hi = lo + per < blocks ? lo + per : blocks;
    double acc = 0.0;
    for (int64_t b = lo; b < hi; ++b) acc += p[b];
    const double total = block_sum(acc);
    if (threadIdx.x == 0) stats[row * Q + q] = (q == 0 && divide_first > 0) ? total / divide_first : total;
}

// Blocks of a register-resident diagnostics kernel per state: each covers
// `tile` consecutive float4 positions per thread.
int64_t stats_blocks(int64_t n_padded, int tile) {
    const int64_t nv = n_padded / 4;
    const int64_t per_block = static_cast<int64_t>(tile) * kThreads;
    const int64_t b = (nv + per_block - 1) / per_block;
    return b < 1 ? 1 : b;
}

template <int M>
cudaError_t launch_sync_stats_t(const SyncArgs &a, double *partial, size_t partial_cap, double *stats,
                                cudaStream_t stream) {
    constexpr int Q = 2 + 2 * M;
    const int64_t gx = stats_blocks(a.n_padded, kSyncStatsTile);
    if (static_cast<size_t>(gx) * a.n_sel * Q > partial_cap || gx > 0x7fffffff) return cudaErrorInvalidValue;
    dim3 grid(static_cast<unsigned>(gx), static_cast<unsigned>(a.n_sel));
    sync_stats_kernel<M><<<grid, kThreads, 0, stream>>>(a, partial);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    stats_finalize_kernel<<<dim3(Q, a.n_sel), kNormThreads, 0, stream>>>(partial, gx, Q, M, stats);
    return cudaGetLastError();
}

// Pseudo-gradient diagnostics of the parameters x[M][n] against the anchor
// a[n] (the parameters at the last average), read-only, on a persistent
// grid, with fixed-order sums into partial[q * gridDim.x + block], Q = 2M + 2:
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
        partial[static_cast<int64_t>(threadIdx.x) * gridDim.x + blockIdx.x] = total;
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
    // the same fixed-order finalisation as the sync diagnostics, with no division
    stats_finalize_kernel<<<dim3(Q, 1), kNormThreads, 0, stream>>>(partial, gx, Q, 0, stats);
    return cudaGetLastError();
}

// ---------------------------------------------------------------- diagnostics for any M

// For M above the register-resident kernels' limit the diagnostics take two
// passes over one state (a [n] fp32 scratch holds the mean between them):
//   pass 1 (grid-stride over float4 positions): the replica mean of
//     replica_mean.cuh (the bits mtdao_sync stores), written to the
//     scratch, and the sums that need only the mean (and the anchor);
//   pass 2 (grid (blocks, M)): per replica the sums against the scratch
//     mean and, for an average, the mean written over the replica.
// As in the one-pass kernels, each position's four elements are summed in
// fp32, each thread accumulates its positions with Kahan compensation, and
// warps, blocks and a finalize kernel reduce in fp64 in fixed order:
// bit-reproducible.  (GB300's fp64 rate is far below its fp32 rate, so the
// per-element work stays in fp32.)

// Deterministic block reduction of K doubles per thread into out[0..K)
// (written by thread 0).
template <int K>
__device__ void block_sum_k(const double (&v)[K], double *out) {
    __shared__ double part[K][kNormThreads / 32];
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
#pragma unroll
    for (int k = 0; k < K; ++k) {
        const double x = warp_sum(v[k]);
        if (l == 0) part[k][w] = x;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
#pragma unroll
        for (int k = 0; k < K; ++k) {
            double t = 0.0;
            for (int i = 0; i < static_cast<int>(blockDim.x >> 5); ++i) t += part[k][i];
            out[k] = t;
        }
    }
}

// Positions a pass-2 thread loads before it accumulates them (i, i + T,
// i + 2T, ...: the order of a plain grid-stride loop): four for the sync
// diagnostics (two float4 loads per position), two for the change
// diagnostics (three per position, within 64 registers).
constexpr int kPass2Unroll = 4;
constexpr int kPass2UnrollChange = 2;

// Pass 1 of the sync diagnostics: mean -> scratch; per block sum s_bar^2.
__global__ void __launch_bounds__(kNormThreads, 4) sync_stats_pass1_kernel(const float *s, int64_t n, int M,
                                                                       float *mean_out, double *partial) {
    const int64_t nv = n / 4;
    Kahan q;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nv;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t e = 4 * i;
        const float4 mv = replica_mean4(s, n, M, e);
        *reinterpret_cast<float4 *>(mean_out + e) = mv;
        q.add(fmaf(mv.x, mv.x, fmaf(mv.y, mv.y, fmaf(mv.z, mv.z, __fmul_rn(mv.w, mv.w)))));
    }
    const double v[1] = {q.value()};
    block_sum_k<1>(v, partial + blockIdx.x);
}

// Pass 2 of the sync diagnostics, replica m = blockIdx.y: per block
// (sum (s_m - s_bar)^2, sum s_m^2, sum s_m * s_bar); with write_mean the
// replica is overwritten by the mean (the average itself).
__global__ void __launch_bounds__(kNormThreads, 4) sync_stats_pass2_kernel(float *s, int64_t n, const float *mean,
                                                                       int write_mean, double *partial) {
    const int m = blockIdx.y;
    const int64_t nv = n / 4;
    const int64_t T = static_cast<int64_t>(gridDim.x) * blockDim.x;
    float *rep = s + m * n;
    Kahan q0, q1, q2;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nv; i += kPass2Unroll * T) {
        float4 rv[kPass2Unroll], mv[kPass2Unroll];
#pragma unroll
        for (int u = 0; u < kPass2Unroll; ++u)
            if (i + u * T < nv) {
                rv[u] = ld_state(rep + 4 * (i + u * T));
                mv[u] = *reinterpret_cast<const float4 *>(mean + 4 * (i + u * T));
            }
#pragma unroll
        for (int u = 0; u < kPass2Unroll; ++u) {
            if (i + u * T >= nv) break;
            float r[4], mb[4];
            to_array(rv[u], r);
            to_array(mv[u], mb);
            float p0 = 0.0f, p1 = 0.0f, p2 = 0.0f;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float dv = r[k] - mb[k];
                p0 = fmaf(dv, dv, p0);
                p1 = fmaf(r[k], r[k], p1);
                p2 = fmaf(r[k], mb[k], p2);
            }
            q0.add(p0);
            q1.add(p1);
            q2.add(p2);
            if (write_mean) st_state(rep + 4 * (i + u * T), mv[u]);
        }
    }
    const double v[3] = {q0.value(), q1.value(), q2.value()};
    block_sum_k<3>(v, partial + 3 * (static_cast<int64_t>(m) * gridDim.x + blockIdx.x));
}

// Pass 1 of the change diagnostics: x_bar -> scratch; per block
// (sum (x_bar - a)^2, sum a^2).
__global__ void __launch_bounds__(kNormThreads, 4) pseudo_grad_pass1_kernel(const float *x, const float *anchor,
                                                                        int64_t n, int M, float *mean_out,
                                                                        double *partial) {
    const int64_t nv = n / 4;
    Kahan q0, q1;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nv;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t e = 4 * i;
        const float4 mv = replica_mean4(x, n, M, e);
        *reinterpret_cast<float4 *>(mean_out + e) = mv;
        float mean[4], a[4];
        to_array(mv, mean);
        to_array(__ldcs(reinterpret_cast<const float4 *>(anchor + e)), a);
        float p0 = 0.0f, p1 = 0.0f;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float glob = mean[k] - a[k];
            p0 = fmaf(glob, glob, p0);
            p1 = fmaf(a[k], a[k], p1);
        }
        q0.add(p0);
        q1.add(p1);
    }
    const double v[2] = {q0.value(), q1.value()};
    block_sum_k<2>(v, partial + 2 * static_cast<int64_t>(blockIdx.x));
}

// Pass 2 of the change diagnostics, replica m = blockIdx.y: per block
// (sum (x_m - a)^2, sum (x_m - a)(x_bar - a)).  Read-only.
__global__ void __launch_bounds__(kNormThreads, 4) pseudo_grad_pass2_kernel(const float *x, const float *anchor,
                                                                        int64_t n, const float *mean,
                                                                        double *partial) {
    const int m = blockIdx.y;
    const int64_t nv = n / 4;
    const int64_t T = static_cast<int64_t>(gridDim.x) * blockDim.x;
    const float *rep = x + m * n;
    Kahan q0, q1;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nv; i += kPass2UnrollChange * T) {
        float4 rv[kPass2UnrollChange], mv[kPass2UnrollChange], av[kPass2UnrollChange];
#pragma unroll
        for (int u = 0; u < kPass2UnrollChange; ++u)
            if (i + u * T < nv) {
                const int64_t e = 4 * (i + u * T);
                rv[u] = ld_state(rep + e);
                mv[u] = *reinterpret_cast<const float4 *>(mean + e);
                av[u] = *reinterpret_cast<const float4 *>(anchor + e);
            }
#pragma unroll
        for (int u = 0; u < kPass2UnrollChange; ++u) {
            if (i + u * T >= nv) break;
            float r[4], mb[4], a[4];
            to_array(rv[u], r);
            to_array(mv[u], mb);
            to_array(av[u], a);
            float p0 = 0.0f, p1 = 0.0f;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float loc = r[k] - a[k];
                const float glob = mb[k] - a[k];
                p0 = fmaf(loc, loc, p0);
                p1 = fmaf(loc, glob, p1);
            }
            q0.add(p0);
            q1.add(p1);
        }
    }
    const double v[2] = {q0.value(), q1.value()};
    block_sum_k<2>(v, partial + 2 * (static_cast<int64_t>(m) * gridDim.x + blockIdx.x));
}

// Adds block partials in block order.  p1 holds K1 values per pass-1
// block, p2 K2 values per (replica, pass-2 block).  For t < K1:
// out[g[t]] = sum_b p1[b][t]; for t < K2 and each replica m:
// out[r[t] + m] = sum_b p2[m][b][t], except that t_sum (if >= 0) is
// summed over the replicas too and divided by M into out[sum_to]
// instead.
struct FinalizeMap {
    int K1, K2;
    int g[2];
    int r[3];
    int t_sum, sum_to;
};

__global__ void general_stats_finalize_kernel(const double *p1, int b1, const double *p2, int b2, int M,
                                              FinalizeMap f, double *out) {
    if (threadIdx.x == 0) {
        for (int t = 0; t < f.K1; ++t) {
            double acc = 0.0;
            for (int b = 0; b < b1; ++b) acc += p1[b * f.K1 + t];
            out[f.g[t]] = acc;
        }
        if (f.t_sum >= 0) {
            double acc = 0.0;
            for (int m = 0; m < M; ++m)
                for (int b = 0; b < b2; ++b) acc += p2[(static_cast<int64_t>(m) * b2 + b) * f.K2 + f.t_sum];
            out[f.sum_to] = acc / M;
        }
    }
    for (int m = threadIdx.x; m < M; m += blockDim.x) {
        for (int t = 0; t < f.K2; ++t) {
            if (t == f.t_sum) continue;
            double acc = 0.0;
            for (int b = 0; b < b2; ++b) acc += p2[(static_cast<int64_t>(m) * b2 + b) * f.K2 + t];
            out[f.r[t] + m] = acc;
        }
    }
}

struct GeneralGrid {
    int b1, b2;
};

GeneralGrid general_grid(int num_sms, int M, int64_t n) {
    const int64_t need = (n / 4 + kNormThreads - 1) / kNormThreads;
    int64_t b1 = 4 * static_cast<int64_t>(num_sms), b2 = b1 / M;
    if (b1 > need) b1 = need;
    if (b2 > need) b2 = need;
    return {static_cast<int>(b1 < 1 ? 1 : b1), static_cast<int>(b2 < 1 ? 1 : b2)};
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

size_t sync_stats_partial_capacity(int num_sms, int64_t n_padded, int n_states, int M) {
    // one row of 2 + 2M sums per block and state, or per persistent block
    // of the pseudo-gradient pass (at most 16 resident blocks per SM)
    const size_t sync = static_cast<size_t>(stats_blocks(n_padded, kSyncStatsTile)) * n_states;
    const size_t change = static_cast<size_t>(16) * num_sms;
    return (sync > change ? sync : change) * (2 + 2 * static_cast<size_t>(M));
}

cudaError_t launch_sync_stats(const SyncArgs &a, int num_sms, double *partial, size_t partial_cap,
                              double *stats, cudaStream_t stream) {
    if (a.n_sel <= 0) return cudaSuccess;
    switch (a.M) {
        case 1: return launch_sync_stats_t<1>(a, partial, partial_cap, stats, stream);
        case 2: return launch_sync_stats_t<2>(a, partial, partial_cap, stats, stream);
        case 3: return launch_sync_stats_t<3>(a, partial, partial_cap, stats, stream);
        case 4: return launch_sync_stats_t<4>(a, partial, partial_cap, stats, stream);
        case 5: return launch_sync_stats_t<5>(a, partial, partial_cap, stats, stream);
        case 6: return launch_sync_stats_t<6>(a, partial, partial_cap, stats, stream);
        case 7: return launch_sync_stats_t<7>(a, partial, partial_cap, stats, stream);
        case 8: return launch_sync_stats_t<8>(a, partial, partial_cap, stats, stream);
        default: return cudaErrorNotSupported;
    }
}

cudaError_t launch_sync(const SyncArgs &a, int num_sms, cudaStream_t stream) {
    if (a.n_sel <= 0 || a.M <= 1) return cudaSuccess;
    switch (a.M) {
        case 2: return launch_sync_t<2>(a, num_sms, stream);
        case 3: return launch_sync_t<3>(a, num_sms, stream);
        case 4: return launch_sync_t<4>(a, num_sms, stream);
        case 5: return launch_sync_t<5>(a, num_sms, stream);
        case 6: return launch_sync_t<6>(a, num_sms, stream);
        case 7: return launch_sync_t<7>(a, num_sms, stream);
        case 8: return launch_sync_t<8>(a, num_sms, stream);
        case 9: return launch_sync_t<9>(a, num_sms, stream);
        case 10: return launch_sync_t<10>(a, num_sms, stream);
        case 11: return launch_sync_t<11>(a, num_sms, stream);
        case 12: return launch_sync_t<12>(a, num_sms, stream);
        case 13: return launch_sync_t<13>(a, num_sms, stream);
        case 14: return launch_sync_t<14>(a, num_sms, stream);
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


size_t general_stats_partial_capacity(int num_sms, int M) {
    const size_t b1 = 4 * static_cast<size_t>(num_sms);
    const size_t b2 = b1 / static_cast<size_t>(M > 0 ? M : 1) + 1;
    return 2 * b1 + 3 * b2 * static_cast<size_t>(M);
}

cudaError_t launch_sync_stats_general(const SyncArgs &a, int num_sms, float *mean_scratch, double *partial,
                                      size_t partial_cap, double *stats, cudaStream_t stream) {
    const int M = a.M;
    const int Q = 2 + 2 * M;
    const GeneralGrid g = general_grid(num_sms, M, a.n_padded);
    if (static_cast<size_t>(g.b1) + 3 * static_cast<size_t>(g.b2) * M > partial_cap) return cudaErrorInvalidValue;
    double *p1 = partial, *p2 = partial + g.b1;
    // stats row: [0] variance (sum over replicas / M), [1] s_bar^2, [2 + m] s_m^2, [2 + M + m] s_m s_bar
    FinalizeMap f = {1, 3, {1, 0}, {0, 2, 2 + M}, 0, 0};
    for (int k = 0; k < a.n_sel; ++k) {
        float *s = a.arena + static_cast<int64_t>(a.sel[k]) * a.stride;
        sync_stats_pass1_kernel<<<g.b1, kNormThreads, 0, stream>>>(s, a.n_padded, M, mean_scratch, p1);
        sync_stats_pass2_kernel<<<dim3(g.b2, M), kNormThreads, 0, stream>>>(s, a.n_padded, mean_scratch,
                                                                            M > 1 ? 1 : 0, p2);
        general_stats_finalize_kernel<<<1, 256, 0, stream>>>(p1, g.b1, p2, g.b2, M, f,
                                                             stats + static_cast<int64_t>(k) * Q);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

cudaError_t launch_pseudo_grad_stats_general(const float *x, const float *anchor, int64_t n, int M, int num_sms,
                                             float *mean_scratch, double *partial, size_t partial_cap,
                                             double *stats, cudaStream_t stream) {
    const GeneralGrid g = general_grid(num_sms, M, n);
    if (2 * static_cast<size_t>(g.b1) + 2 * static_cast<size_t>(g.b2) * M > partial_cap)
        return cudaErrorInvalidValue;
    double *p1 = partial, *p2 = partial + 2 * g.b1;
    // out: [m] (x_m - a)^2, [M + m] (x_m - a)(x_bar - a), [2M] (x_bar - a)^2, [2M + 1] a^2
    FinalizeMap f = {2, 2, {2 * M, 2 * M + 1}, {0, M, 0}, -1, 0};
    pseudo_grad_pass1_kernel<<<g.b1, kNormThreads, 0, stream>>>(x, anchor, n, M, mean_scratch, p1);
    pseudo_grad_pass2_kernel<<<dim3(g.b2, M), kNormThreads, 0, stream>>>(x, anchor, n, mean_scratch, p2);
    general_stats_finalize_kernel<<<1, 256, 0, stream>>>(p1, g.b1, p2, g.b2, M, f, stats);
    return cudaGetLastError();
}

}  // namespace mtdao
