// step_sync_wide.cuh -- the local step with the replica average fused in,
// for replica counts from 9 to 64 (kWideFusedMaxM), and the span layout
// that the one-pass diagnostics of stats_wide.cu share (up to kWideMaxM).
//
// A block owns a span of S consecutive elements of all M replicas.  Thread
// (r, f) of the block updates kWideVec float4 positions of the span in
// replica r (f, f + P, ...) with update_state, issuing every state's loads
// before any arithmetic.  A state that is not due is stored at once.  A due
// state goes to shared memory instead; after one barrier the replica mean
// of every (due state, element) pair is formed by two threads, each running
// one of the two compensated parts of replica_mean.cuh over the replicas in
// order, joined by one shuffle; after a second barrier every thread stores
// the means to its own replica.  The parts are the ones the standalone
// average forms (sync_kernel's streamed loop), in the same order, so fused
// and separate averaging give identical bits for every M.
//
// Rows of the span are 32 bytes or longer: P = 16 (M <= 16), 8 (M <= 64),
// 4 (M <= 128), 2 (M <= 256) float4 positions per thread row, so a block
// has M * P <= 512 threads (rounded up to whole warps; threads beyond M * P
// only take part in the mean).  Shared memory: one M x S tile and S means
// per due state.
#pragma once

#include "replica_mean.cuh"
#include "step_kernels.cuh"

namespace mtdao {

constexpr int kWideMaxM = 256;            // largest M of the span layout (diagnostics)
constexpr int kWideFusedMaxM = 64;        // largest M of the fused step (above: step + average)
constexpr int kWideMaxThreads = 512;      // largest block of the span layout
constexpr int kWideVec = 1;               // float4 positions per thread and state in the fused step
constexpr int kWideVecLog2 = kWideVec == 1 ? 0 : kWideVec == 2 ? 1 : 2;

// Threads per replica row of the span (a power of two).
constexpr int wide_positions(int M) { return M <= 16 ? 16 : M <= 64 ? 8 : M <= 128 ? 4 : 2; }

// Elements of the fused step's span, and its floats of shared memory per
// due state: the M x S tile and S means.
constexpr int wide_span(int M) { return 4 * kWideVec * wide_positions(M); }
constexpr int wide_floats_per_state(int M) { return (M + 1) * wide_span(M); }

// Replica means of the n_cols columns of a block's tile into mean[p]
// (column p: tile + (p / S) * M * S + p % S, the replicas at stride
// S = 2^log2_s; shifts, not a division by a run-time S).
// Lanes 2i and 2i + 1 form the two compensated parts of replica_mean.cuh
// for one column, replicas 1 .. h-1 and h .. M-1 in order (h = M / 2), and
// join them with a shuffle: the bits of replica_mean_rt (with its plain
// mean where the compensated one is NaN).  Every thread of
// the block calls it (the shuffles take whole warps: blockDim.x is a
// multiple of 32 and the loop count is the same for all threads).
__device__ __forceinline__ void tile_means(const float *tile, int M, int log2_s, int n_cols, float *mean) {
    const int t = threadIdx.x;
    const int h = M / 2;
    const int S = 1 << log2_s;
    for (int p0 = 0; p0 < n_cols; p0 += static_cast<int>(blockDim.x >> 1)) {
        const int p = p0 + (t >> 1);
        const int part = t & 1;
        float s0 = 0.0f, mine = 0.0f;
        if (p < n_cols) {
            const float *col = tile + (p >> log2_s) * M * S + (p & (S - 1));
            s0 = col[0];
            DiffSum sum(s0);
            const int lo = part ? h : 1, hi = part ? M : h;
#pragma unroll 4
            for (int m = lo; m < hi; ++m) sum.add(col[m * S]);   // unrolled: the loads run ahead
            mine = sum.partial();
        }
        const float other = __shfl_xor_sync(0xffffffffu, mine, 1);
        if (p < n_cols && part == 0) {
            float v = replica_mean_from_parts(s0, mine, other, static_cast<float>(M));
            if (v != v) {                        // non-finite values: the plain mean (replica_mean.cuh)
                const float *col = tile + (p >> log2_s) * M * S + (p & (S - 1));
                float plain = col[0];
                for (int m = 1; m < M; ++m) plain += col[m * S];
                v = plain / static_cast<float>(M);
            }
            mean[p] = v;
        }
    }
}

template <int BASE, int N, int GDT, bool CLIP>
__global__ void __launch_bounds__(kWideMaxThreads) step_sync_wide_kernel(const StepArgs a, int log2_p) {
    extern __shared__ float smem[];
    constexpr int kStates = kNumStates<BASE, N>;
    constexpr int NV = kWideVec;
    const int M = a.M;
    const int P = 1 << log2_p;
    const int S = 4 * P * NV;                    // elements of the span
    const int t = threadIdx.x;
    const int r = t >> log2_p;                   // replica of this thread
    const int f = t & (P - 1);                   // its first float4 position in the span
    const bool live = r < M;
    const int64_t n = a.n_padded;
    const int64_t n_spans = n / S;
    const uint32_t mask = a.sync_mask;
    const int n_due = __popc(mask);
    float *tile = smem;                          // [n_due][M][S]
    float *mean = smem + n_due * M * S;          // [n_due][S]
    const float s = (CLIP && live) ? __ldg(a.clip_scale + r) : 1.0f;

    for (int64_t span = blockIdx.x; span < n_spans; span += gridDim.x) {
        const int64_t e = span * S + 4 * f;      // element index within a replica (position j: + 4 P j)
        if (live) {
            float g[NV][4], buf[kStates][NV][4], gt[NV][4], acc[NV][4];
#pragma unroll
            for (int j = 0; j < NV; ++j) to_array(ld_grad<GDT>(a.grads, r * n + e + 4 * P * j), g[j]);
#pragma unroll
            for (int i = 0; i < kStates; ++i)
#pragma unroll
                for (int j = 0; j < NV; ++j)
                    to_array(ld_state(a.arena + state_order<BASE, N>(i) * a.stride + r * n + e + 4 * P * j),
                             buf[i][j]);
#pragma unroll
            for (int j = 0; j < NV; ++j)
#pragma unroll
                for (int k = 0; k < 4; ++k) acc[j][k] = step_acc_init<BASE>(a.sc, g[j][k], s);
#pragma unroll
            for (int i = 0; i < kStates; ++i) {
                const int st = state_order<BASE, N>(i);
                const bool due = (mask >> st) & 1u;
                const int slot = __popc(mask & ((1u << st) - 1u));
#pragma unroll
                for (int j = 0; j < NV; ++j) {
                    float *cur = buf[i][j];
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        update_state<BASE, N>(a.sc, st, g[j][k], s, gt[j][k], acc[j][k], cur[k]);
                    if (due)
                        *reinterpret_cast<float4 *>(tile + (slot * M + r) * S + 4 * f + 4 * P * j) = from_array(cur);
                    else
                        st_state(a.arena + st * a.stride + r * n + e + 4 * P * j, from_array(cur));
                }
            }
        }
        __syncthreads();
        tile_means(tile, M, log2_p + 2 + kWideVecLog2, n_due * S, mean);
        __syncthreads();
        if (live) {
#pragma unroll
            for (int st = 0; st < kStates; ++st)
                if ((mask >> st) & 1u) {
                    const int slot = __popc(mask & ((1u << st) - 1u));
#pragma unroll
                    for (int j = 0; j < NV; ++j)
                        st_state(a.arena + st * a.stride + r * n + e + 4 * P * j,
                                 *reinterpret_cast<const float4 *>(mean + slot * S + 4 * f + 4 * P * j));
                }
        }
        __syncthreads();                         // the tile and the means are reused by the next span
    }
}

template <int BASE, int N, int GDT, bool CLIP>
cudaError_t launch_step_sync_wide(const StepArgs &a, cudaStream_t stream) {
    if (a.M < 2 || a.M > kWideFusedMaxM) return cudaErrorNotSupported;
    const int P = wide_positions(a.M);
    int log2_p = 0;
    while ((1 << log2_p) < P) ++log2_p;
    const int S = wide_span(a.M);
    const int threads = (a.M * P + 31) / 32 * 32;
    const int n_due = __builtin_popcount(a.sync_mask);
    const size_t smem = static_cast<size_t>(n_due) * wide_floats_per_state(a.M) * sizeof(float);
    auto kernel = step_sync_wide_kernel<BASE, N, GDT, CLIP>;
    if (smem > 48 * 1024) {       // above the default limit (M >= 33 with most states due)
        const cudaError_t e =
            cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    int64_t grid = a.n_padded / S;
    if (grid > 0x7fffffff) grid = 0x7fffffff;
    kernel<<<static_cast<unsigned>(grid < 1 ? 1 : grid), threads, smem, stream>>>(a, log2_p);
    return cudaGetLastError();
}

}  // namespace mtdao
