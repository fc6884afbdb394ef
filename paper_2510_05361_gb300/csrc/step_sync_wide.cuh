// step_sync_wide.cuh -- the local step with the replica average fused in,
// for replica counts from 9 to 64 (kWideFusedMaxM), and the span layout
// that the one-pass diagnostics of stats_wide.cu share (up to kWideMaxM).
//
// A block owns a span of S consecutive elements of all M replicas; thread
// (r, f) updates elements [4f, 4f + 4) and [4(f + P), 4(f + P) + 4) of
// replica r (one position above M = 32, see wide_fused_vec) with
// update_state.  The
// blocks are persistent and double-buffer their spans in shared memory: the
// next span of every state and of the gradient is copied in with cp.async
// while the current one is updated, so HBM traffic continues through the
// barriers.  A state that is not due is stored from registers at once; a
// due state's new values go back over its tile in shared memory; after one
// barrier the replica mean of every (due state, element) pair is formed by
// two threads, each running one of the two compensated parts of
// replica_mean.cuh over the replicas in order, joined by one shuffle; after
// a second barrier every thread stores the means to its own replica.  The
// parts are the ones the standalone average forms (sync_kernel's streamed
// loop), in the same order, so fused and separate averaging give identical
// bits for every M.
//
// A replica's row of a span is handled by P threads: P = 16 (M <= 16), 8
// (M <= 64), 4 (M <= 128), 2 (M <= 256), so a block has M * P <= 512
// threads (rounded up to whole warps; threads beyond M * P only take part
// in the mean).  The fused step's rows are 128 elements (512 bytes) up to
// M = 16, 64 up to 32 and 32 above; the one-pass diagnostics' rows are 16 P
// elements.
// Shared memory of the fused step: two span buffers (a tile per state and
// the gradient tile) and S means per due state.
#pragma once

#include "replica_mean.cuh"
#include "step_kernels.cuh"

namespace mtdao {

constexpr int kWideMaxM = 256;            // largest M of the span layout (diagnostics)
constexpr int kWideFusedMaxM = 64;        // largest M of the fused step (above: step + average)
constexpr int kWideMaxThreads = 512;      // largest block of the span layout

// Threads per replica row of the span (a power of two).
constexpr int wide_positions(int M) { return M <= 16 ? 16 : M <= 64 ? 8 : M <= 128 ? 4 : 2; }


// Replica means of the n_cols columns of a block's tile into mean[p]
// (column p: tile + (p / S) * M * S + p % S, the replicas at stride
// S = 2^log2_s; shifts, not a division by a run-time S).  Columns go in
// groups of four (n_cols and S are multiples of 4): lanes 2i and 2i + 1
// take one group and form its two compensated parts of replica_mean.cuh,
// replicas 1 .. h-1 and h .. M-1 in order (h = M / 2), four columns at a
// time from one 16-byte shared load per replica, and join them with
// shuffles: the bits of replica_mean_rt (with its plain mean where the
// compensated one is NaN).  Every thread of the block calls it (the
// shuffles take whole warps: blockDim.x is a multiple of 32 and the loop
// count is the same for all threads).
__device__ __forceinline__ void tile_means4(const float *tile, int M, int log2_s, int n_cols, float *mean) {
    const int t = threadIdx.x;
    const int h = M / 2;
    const int S = 1 << log2_s;
    const int n_tasks = n_cols / 2;              // (group of four columns, part) pairs
    for (int q0 = 0; q0 < n_tasks; q0 += static_cast<int>(blockDim.x)) {
        const int q = q0 + t;
        const int part = q & 1;
        const int p = 4 * (q >> 1);              // first column of the group
        const float *base = tile + (p >> log2_s) * M * S + (p & (S - 1));
        float s0[4] = {0.0f, 0.0f, 0.0f, 0.0f}, mine[4] = {0.0f, 0.0f, 0.0f, 0.0f};
        if (q < n_tasks) {
            to_array(*reinterpret_cast<const float4 *>(base), s0);
            DiffSum sum[4] = {DiffSum(s0[0]), DiffSum(s0[1]), DiffSum(s0[2]), DiffSum(s0[3])};
            const int lo = part ? h : 1, hi = part ? M : h;
#pragma unroll 2
            for (int m = lo; m < hi; ++m) {
                float v[4];
                to_array(*reinterpret_cast<const float4 *>(base + m * S), v);
#pragma unroll
                for (int k = 0; k < 4; ++k) sum[k].add(v[k]);
            }
#pragma unroll
            for (int k = 0; k < 4; ++k) mine[k] = sum[k].partial();
        }
        float other[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) other[k] = __shfl_xor_sync(0xffffffffu, mine[k], 1);
        if (q < n_tasks && part == 0) {
            float v[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                v[k] = replica_mean_from_parts(s0[k], mine[k], other[k], static_cast<float>(M));
                if (v[k] != v[k]) {              // non-finite values: the plain mean (replica_mean.cuh)
                    float plain = s0[k];
                    for (int m = 1; m < M; ++m) plain += base[m * S + k];
                    v[k] = plain / static_cast<float>(M);
                }
            }
            *reinterpret_cast<float4 *>(mean + p) = from_array(v);
        }
    }
}

// The same means one column per lane pair (lanes 2i and 2i + 1 run the two
// parts of column i with 4-byte shared loads): more lanes at work on fewer
// columns each, which is the better trade for M above 32.
__device__ __forceinline__ void tile_means1(const float *tile, int M, int log2_s, int n_cols, float *mean) {
    const int t = threadIdx.x;
    const int h = M / 2;
    const int S = 1 << log2_s;
    for (int p0 = 0; p0 < n_cols; p0 += static_cast<int>(blockDim.x >> 1)) {
        const int p = p0 + (t >> 1);
        const int part = t & 1;
        float s0 = 0.0f, mine = 0.0f;
        const float *col = tile + (p >> log2_s) * M * S + (p & (S - 1));
        if (p < n_cols) {
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
                float plain = s0;
                for (int m = 1; m < M; ++m) plain += col[m * S];
                v = plain / static_cast<float>(M);
            }
            mean[p] = v;
        }
    }
}

// The per-span means of the wide kernels: four columns per lane pair up to
// M = 32 (flat sweep, fused step, N = 3: M = 9 4861 -> 5825 GB/s, 24-32
// 5397-5458 -> 5908-5915), one above (M = 64: 4998 against 4887 with four,
// where only n_cols / 2 of up to 512 threads have work).  A compile-time
// choice: with both forms in one kernel the fused step took 101-108
// registers instead of 50-64 and lost occupancy.
constexpr bool wide_four_columns(int M) { return M <= 32; }

template <bool FOUR>
__device__ __forceinline__ void tile_means(const float *tile, int M, int log2_s, int n_cols, float *mean) {
    if constexpr (FOUR)
        tile_means4(tile, M, log2_s, n_cols, mean);
    else
        tile_means1(tile, M, log2_s, n_cols, mean);
}

// 16- and 8-byte asynchronous global -> shared copies (cp.async) and their
// groups: a block copies its next span while it works on the current one.
__device__ __forceinline__ void cp_async16(void *smem_dst, const void *gmem_src) {
    const unsigned dst = static_cast<unsigned>(__cvta_generic_to_shared(smem_dst));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(gmem_src) : "memory");
}
__device__ __forceinline__ void cp_async8(void *smem_dst, const void *gmem_src) {
    const unsigned dst = static_cast<unsigned>(__cvta_generic_to_shared(smem_dst));
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(dst), "l"(gmem_src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

// Floats of one span buffer: a tile of M x S floats per state and the
// gradient tile (M x S f32, or bf16 in half the floats).
template <int BASE, int N, int GDT>
__host__ __device__ constexpr int wide_buffer_floats(int M, int S) {
    return kNumStates<BASE, N> * M * S + (GDT == MTDAO_F32 ? M * S : M * S / 2);
}

// Float4 positions per thread and row of the fused step's span (the
// positions f and f + P): rows of 512 bytes up to M = 16 (S = 128) and 256
// bytes for 17-32 (S = 64).  The row length sets the DRAM efficiency: with
// one position, M = 24 and 32 (rows of 128 bytes) ran at 4.8-4.9 TB/s
// (Adam, N = 3), with two at 5.4; M = 12 and 16 ran 3-10 % faster with
// rows of 512 bytes than of 256.  Above 32 two positions made a span buffer
// so large (up to 96 KB) that one block fitted per SM: M = 48 and 64 fell
// from 4.9-5.0 to 3.9-4.2 TB/s.
constexpr int wide_fused_vec(int M) { return M <= 32 ? 2 : 1; }

// The fused step on spans of all replicas, persistent, double-buffered:
// while a block updates span i from shared memory, span i + gridDim.x of
// every state and of the gradient is on its way in (cp.async).  In a
// buffer the due states' tiles come first (in state index order), so the
// means read them as one [n_due][M][S] array; a due state's updated values
// are written back over its own tile, a state that is not due goes
// straight to HBM.
template <int BASE, int N, int GDT, bool CLIP, bool FOUR>
__global__ void __launch_bounds__(kWideMaxThreads) step_sync_wide_kernel(const StepArgs a, int log2_p,
                                                                         int log2_v) {
    extern __shared__ __align__(16) float smem[];
    constexpr int kStates = kNumStates<BASE, N>;
    constexpr int kMaxVec = 2;
    const int M = a.M;
    const int P = 1 << log2_p;
    const int NV = 1 << log2_v;                  // float4 positions per thread (1 or 2)
    const int log2_s = log2_p + 2 + log2_v;
    const int S = 1 << log2_s;                   // elements of the span
    const int t = threadIdx.x;
    const int r = t >> log2_p;                   // replica of this thread
    const int f = t & (P - 1);                   // its first float4 position in the span
    const bool live = r < M;
    const int64_t n = a.n_padded;
    const int64_t n_spans = n / S;
    const uint32_t mask = a.sync_mask;
    const int n_due = __popc(mask);
    const int tile = M * S;
    const int buf_floats = wide_buffer_floats<BASE, N, GDT>(M, S);
    float *mean = smem + 2 * buf_floats;         // [n_due][S]
    const float s = (CLIP && live) ? __ldg(a.clip_scale + r) : 1.0f;
    const int own = r * S + 4 * f;               // this thread's offset in a tile
    // tile of state st in a buffer: the due states first
    auto slot = [&](int st) {
        const uint32_t below = (1u << st) - 1u;
        return ((mask >> st) & 1u) ? __popc(mask & below) : n_due + __popc(~mask & below);
    };
    auto fetch = [&](int64_t span, float *buf) {
        if (live && span < n_spans) {
#pragma unroll
            for (int j = 0; j < kMaxVec; ++j) {
                if (j >= NV) break;
                const int64_t src = r * n + span * S + 4 * f + 4 * P * j;
                const int dst = own + 4 * P * j;
#pragma unroll
                for (int st = 0; st < kStates; ++st)
                    cp_async16(buf + slot(st) * tile + dst, a.arena + st * a.stride + src);
                if constexpr (GDT == MTDAO_F32)
                    cp_async16(buf + kStates * tile + dst, static_cast<const float *>(a.grads) + src);
                else
                    cp_async8(reinterpret_cast<uint16_t *>(buf + kStates * tile) + dst,
                              static_cast<const uint16_t *>(a.grads) + src);
            }
        }
        cp_async_commit();
    };

    // one span ahead: span k of this block lives in buffer k % 2 (a third
    // buffer, two spans ahead, measured the same or 5-10 % slower: fewer
    // blocks fit per SM)
    int b = 0;
    fetch(blockIdx.x, smem);
    for (int64_t span = blockIdx.x; span < n_spans; span += gridDim.x, b ^= 1) {
        float *buf = smem + b * buf_floats;
        fetch(span + gridDim.x, smem + (b ^ 1) * buf_floats);
        cp_async_wait<1>();                      // this thread's copies of `span` have landed
        __syncthreads();                         // ... and every thread's
        const int64_t e = span * S + 4 * f;      // element index within a replica (position j: + 4 P j)
        if (live) {
#pragma unroll
            for (int j = 0; j < kMaxVec; ++j) {
                if (j >= NV) break;
                const int at = own + 4 * P * j;
                float g[4], gt[4], acc[4];
                if constexpr (GDT == MTDAO_F32) {
                    to_array(*reinterpret_cast<const float4 *>(buf + kStates * tile + at), g);
                } else {
                    const uint2 w =
                        *reinterpret_cast<const uint2 *>(reinterpret_cast<const uint16_t *>(buf + kStates * tile) + at);
                    g[0] = __uint_as_float(w.x << 16);
                    g[1] = __uint_as_float(w.x & 0xffff0000u);
                    g[2] = __uint_as_float(w.y << 16);
                    g[3] = __uint_as_float(w.y & 0xffff0000u);
                }
#pragma unroll
                for (int k = 0; k < 4; ++k) acc[k] = step_acc_init<BASE>(a.sc, g[k], s);
#pragma unroll
                for (int i = 0; i < kStates; ++i) {
                    const int st = state_order<BASE, N>(i);
                    float *cell = buf + slot(st) * tile + at;
                    float cur[4];
                    to_array(*reinterpret_cast<const float4 *>(cell), cur);
#pragma unroll
                    for (int k = 0; k < 4; ++k) update_state<BASE, N>(a.sc, st, g[k], s, gt[k], acc[k], cur[k]);
                    if ((mask >> st) & 1u)
                        *reinterpret_cast<float4 *>(cell) = from_array(cur);
                    else
                        st_state(a.arena + st * a.stride + r * n + e + 4 * P * j, from_array(cur));
                }
            }
        }
        __syncthreads();
        tile_means<FOUR>(buf, M, log2_s, n_due * S, mean);
        __syncthreads();
        if (live) {
#pragma unroll
            for (int st = 0; st < kStates; ++st)
                if ((mask >> st) & 1u) {
#pragma unroll
                    for (int j = 0; j < kMaxVec; ++j) {
                        if (j >= NV) break;
                        st_state(a.arena + st * a.stride + r * n + e + 4 * P * j,
                                 *reinterpret_cast<const float4 *>(mean + slot(st) * S + 4 * f + 4 * P * j));
                    }
                }
        }
        __syncthreads();                         // this buffer and the means are rewritten next
    }
    cp_async_wait<0>();
}

template <int BASE, int N, int GDT, bool CLIP, bool FOUR>
cudaError_t launch_step_sync_wide_t(const StepArgs &a, int num_sms, cudaStream_t stream) {
    if (a.M < 2 || a.M > kWideFusedMaxM) return cudaErrorNotSupported;
    const int P = wide_positions(a.M);
    int log2_p = 0;
    while ((1 << log2_p) < P) ++log2_p;
    const int log2_v = wide_fused_vec(a.M) == 2 ? 1 : 0;
    const int S = 4 * P << log2_v;
    const int threads = (a.M * P + 31) / 32 * 32;
    const int n_due = __builtin_popcount(a.sync_mask);
    const size_t smem = (2 * static_cast<size_t>(wide_buffer_floats<BASE, N, GDT>(a.M, S)) +
                         static_cast<size_t>(n_due) * S) * sizeof(float);
    auto kernel = step_sync_wide_kernel<BASE, N, GDT, CLIP, FOUR>;
    if (smem > 48 * 1024) {       // above the default limit; before the occupancy query
        const cudaError_t e =
            cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, threads, smem) != cudaSuccess ||
        per_sm < 1) {
        cudaGetLastError();
        per_sm = 1;
    }
    int64_t grid = static_cast<int64_t>(per_sm) * num_sms;
    const int64_t n_spans = a.n_padded / S;
    if (grid > n_spans) grid = n_spans;
    kernel<<<static_cast<unsigned>(grid < 1 ? 1 : grid), threads, smem, stream>>>(a, log2_p, log2_v);
    return cudaGetLastError();
}

template <int BASE, int N, int GDT, bool CLIP>
cudaError_t launch_step_sync_wide(const StepArgs &a, int num_sms, cudaStream_t stream) {
    return wide_four_columns(a.M) ? launch_step_sync_wide_t<BASE, N, GDT, CLIP, true>(a, num_sms, stream)
                                  : launch_step_sync_wide_t<BASE, N, GDT, CLIP, false>(a, num_sms, stream);
}

}  // namespace mtdao
