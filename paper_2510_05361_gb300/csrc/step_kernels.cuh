// step_kernels.cuh -- the MT-DAO local step (Algorithms 1-3) for sm_103a.
//
// The step is elementwise and HBM-bound (about 0.3 flop per byte), so it is
// written as a grid-stride streaming kernel launched with one chunk per
// warp (stream_grid): every state of every replica is read once and written
// once per step with 128-bit accesses, the gradient is read once.  A warp
// owns a chunk of 256 consecutive elements; lane l handles elements [4l, 4l+4) and [128+4l, 128+4l+4)
// of the chunk, so every warp-wide load or store instruction covers 512
// contiguous bytes of fp32 (256 bytes of bf16 gradient).
//
// The states of a chunk are visited one after another (state_order): the
// next state's loads are issued before the current state is updated and
// stored, so two states' loads are in flight per lane and the writes of one
// state overlap the reads of the next.
//
// This header holds the per-state update (update_state, in state_order),
// which the fused step + average kernel of step_sync_kernels.cuh writes out
// with the same expressions, and step_kernel, which is replica-major: the
// flat index runs over all M replicas (M * n_padded elements); it serves
// every step with no average.
//
// Measured against the previous form of step_kernel (every load of the
// chunk issued before any arithmetic, then every store): 6437 -> 6512 GB/s
// on the ~1B workload's step, and +1-2% at every flat-vector point.
#pragma once

#include <cuda_runtime.h>
#include <cstdint>

#include "mtdao_internal.h"

namespace mtdao {

// ---------------------------------------------------------------- memory access

// States are read once and overwritten once per step: stream them past the
// caches (evict-first) so that they do not displace anything useful.
__device__ __forceinline__ float4 ld_state(const float *p) {
    return __ldcs(reinterpret_cast<const float4 *>(p));
}
__device__ __forceinline__ void st_state(float *p, float4 v) {
    __stcs(reinterpret_cast<float4 *>(p), v);
}

// Four consecutive gradient elements starting at flat element index e,
// upcast to fp32 (bf16 -> fp32 is exact: the bits move up by 16).
template <int GDT>
__device__ __forceinline__ float4 ld_grad(const void *g, int64_t e) {
    if constexpr (GDT == MTDAO_F32) {
        return __ldcs(reinterpret_cast<const float4 *>(static_cast<const float *>(g) + e));
    } else {
        const uint2 w = __ldcs(reinterpret_cast<const uint2 *>(static_cast<const uint16_t *>(g) + e));
        return make_float4(__uint_as_float(w.x << 16), __uint_as_float(w.x & 0xffff0000u),
                           __uint_as_float(w.y << 16), __uint_as_float(w.y & 0xffff0000u));
    }
}

__device__ __forceinline__ void to_array(float4 v, float *a) {
    a[0] = v.x; a[1] = v.y; a[2] = v.z; a[3] = v.w;
}
__device__ __forceinline__ float4 from_array(const float *a) {
    return make_float4(a[0], a[1], a[2], a[3]);
}

// ---------------------------------------------------------------- the update

// Number of state vectors per replica: x, u_1..u_N and (Adam, ADOPT) v.
template <int BASE, int N>
constexpr int kNumStates = BASE == MTDAO_BASE_SGDM ? N + 1 : N + 2;

// Order in which the kernels visit the states of an element (arena index
// 0 = x, 1 + j = u_j, 1 + N = v): ADOPT takes v first (it normalises the
// gradient), Adam takes v after the momenta (it divides their combination),
// x comes last.
template <int BASE, int N>
__host__ __device__ constexpr int state_order(int i) {
    return BASE == MTDAO_BASE_ADOPT
               ? (i == 0 ? 1 + N : (i <= N ? i : 0))
               : (i < N ? 1 + i : (BASE == MTDAO_BASE_ADAM && i == N ? 1 + N : 0));
}

// Per-element carry of one step across the state visits:
//   gt  : ADOPT's normalised, clamped gradient (set when v is visited)
//   acc : Delta's numerator (Adam), Delta (SGDM, ADOPT)
// Adam/SGDM start acc with the gradient term (1 - sum omega) * clip(g).
template <int BASE>
__device__ __forceinline__ float step_acc_init(const StepScalars &sc, float g, float s) {
    return BASE == MTDAO_BASE_ADOPT ? 0.0f : sc.cg * __fmul_rn(g, s);   // never contracted into an FMA
}

// beta * s for beta = 1 - c, rounded once: s - c * s in one fma, which keeps
// beta's precision however close it is to 1.  For an infinite s the fma
// would form inf - inf = NaN where beta * s is s itself (beta > 0), so an
// infinite state stays infinite from one step to the next, as it does in
// exact arithmetic; c = 1 (beta = 0) keeps the fma's NaN, which is 0 * inf.
__device__ __forceinline__ float ema_decay(float c, float s) {
    const float d = fmaf(-c, s, s);
    return (fabsf(s) == __int_as_float(0x7f800000) && c < 1.0f) ? s : d;
}

// Update state `st` of one element of one replica for step t.
//   g : raw gradient g_t^m          s : clip(g, rho) factor (1 when not clipping)
//   cur : the state's value, updated in place
// With st visited in state_order this is Algorithm 1 (Adam), 2 (ADOPT) or
// 3 (SGDM) for the element; every EMA is beta * s + (1 - beta) * target in
// the fma form described with StepScalars.
template <int BASE, int N>
__device__ __forceinline__ void update_state(const StepScalars &sc, int st, float g, float s, float &gt,
                                             float &acc, float &cur) {
    if (st == 1 + N && BASE == MTDAO_BASE_ADOPT) {
        // Algorithm 2: second moment of the raw gradient first, then the
        // normalised, clamped gradient that every momentum follows.  In the
        // original ADOPT order (uniform flag) v is updated after use.
        float gn;
        if (sc.prev_v) {
            gn = g / (sqrtf(cur) + sc.eps);
            cur = fmaf(__fmul_rn(sc.c2, g), g, ema_decay(sc.c2, cur));
        } else {
            cur = fmaf(__fmul_rn(sc.c2, g), g, ema_decay(sc.c2, cur));
            gn = g / (sqrtf(cur) + sc.eps);
        }
        gn = gn > sc.clip_c ? sc.clip_c : (gn < -sc.clip_c ? -sc.clip_c : gn);  // keeps NaN
        gt = gn;
        acc = sc.cg * gn;
    } else if (st == 1 + N) {
        // Algorithm 1: v of the raw gradient, then the denominator
        // sqrt(v / b_v) + eps of the momenta's combination.
        cur = fmaf(__fmul_rn(sc.c2, g), g, ema_decay(sc.c2, cur));
        acc = acc / fmaf(sqrtf(cur), sc.sv, sc.eps);
    } else if (st == 0) {
        cur = fmaf(sc.neg_lr, acc, cur);                     // x - eta_t Delta
    } else {
        // momentum u_j of clip(g) (Adam, SGDM) or of ADOPT's clamped g
        const int j = st - 1;
        const float target = BASE == MTDAO_BASE_ADOPT ? gt : __fmul_rn(g, s);
        cur = fmaf(sc.c1[j], target, ema_decay(sc.c1[j], cur));
        acc = fmaf(sc.k[j], cur, acc);
    }
}

// ---------------------------------------------------------------- local step

// States whose loads are in flight ahead of the one being updated.  Two
// measured the same as one (within 0.5% on the ~1B and ~350M workloads and
// the flat sweep points) with more registers, so one it is.
constexpr int kStepLookahead = 1;

template <int BASE, int N, int GDT, bool CLIP>
__global__ void __launch_bounds__(kThreads) step_kernel(const StepArgs a) {
    constexpr int kStates = kNumStates<BASE, N>;
    constexpr int kBufs = kStepLookahead + 1;
    const int lane = threadIdx.x & 31;
    const int64_t n_chunks = a.stride / kChunk;
    const int64_t warp = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int64_t n_warps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;

    for (int64_t c = warp; c < n_chunks; c += n_warps) {
        const int64_t e0 = c * kChunk + 4 * lane;
        const int64_t e1 = e0 + 128;
        float g[8];
        to_array(ld_grad<GDT>(a.grads, e0), g);
        to_array(ld_grad<GDT>(a.grads, e1), g + 4);
        float s = 1.0f;
        if constexpr (CLIP) s = __ldg(a.clip_scale + (c * kChunk) / a.n_padded);

        float gt[8], acc[8], buf[kBufs][8];
        auto load = [&](int i) {
            const float *p = a.arena + state_order<BASE, N>(i) * a.stride;
            to_array(ld_state(p + e0), buf[i % kBufs]);
            to_array(ld_state(p + e1), buf[i % kBufs] + 4);
        };
#pragma unroll
        for (int k = 0; k < 8; ++k) acc[k] = step_acc_init<BASE>(a.sc, g[k], s);
#pragma unroll
        for (int i = 0; i < kStepLookahead && i < kStates; ++i) load(i);
#pragma unroll
        for (int i = 0; i < kStates; ++i) {
            if (i + kStepLookahead < kStates) load(i + kStepLookahead);   // before this state's work
            const int st = state_order<BASE, N>(i);
            float *cur = buf[i % kBufs];
#pragma unroll
            for (int k = 0; k < 8; ++k) update_state<BASE, N>(a.sc, st, g[k], s, gt[k], acc[k], cur[k]);
            float *p = a.arena + st * a.stride;
            st_state(p + e0, from_array(cur));
            st_state(p + e1, from_array(cur + 4));
        }
    }
}

// ---------------------------------------------------------------- launch helpers

// Persistent grid: as many blocks as fit on the device at once, but never
// more warps than there are chunks of work.
template <typename Kernel>
inline int blocks_per_sm(Kernel kernel) {
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kThreads, 0) != cudaSuccess ||
        per_sm < 1)
        per_sm = 1;
    return per_sm;
}

inline int persistent_grid(int per_sm, int num_sms, int64_t n_warp_items) {
    const int64_t warps_per_block = kThreads / 32;
    int64_t need = (n_warp_items + warps_per_block - 1) / warps_per_block;
    int64_t grid = static_cast<int64_t>(per_sm) * num_sms;
    if (need < grid) grid = need;
    return static_cast<int>(grid < 1 ? 1 : grid);
}

// Streaming grid: one warp chunk per warp, so the loop of the kernel runs
// once (it stays a grid-stride loop, so any grid is correct).  The block
// scheduler starts blocks in index order as earlier ones retire, which
// keeps the addresses in flight within a narrow window of every slab; a
// persistent grid's warps drift apart over the whole slab.  On the ~1B
// and ~350M workloads the local step ran 10-12% faster this way (7158 vs
// 6484 GB/s, 7128 vs 6375 GB/s on one box).
inline int stream_grid(int64_t n_warp_items) {
    const int64_t warps_per_block = kThreads / 32;
    int64_t grid = (n_warp_items + warps_per_block - 1) / warps_per_block;
    if (grid > 0x7fffffff) grid = 0x7fffffff;
    return static_cast<int>(grid < 1 ? 1 : grid);
}

template <int BASE, int N, int GDT, bool CLIP>
cudaError_t launch_step_t(const StepArgs &a, int num_sms, cudaStream_t stream) {
    auto kernel = step_kernel<BASE, N, GDT, CLIP>;
    (void)num_sms;
    const int grid = stream_grid(a.stride / kChunk);
    kernel<<<grid, kThreads, 0, stream>>>(a);
    return cudaGetLastError();
}

// Dispatch over N, gradient dtype and clipping for one base.
template <int BASE>
cudaError_t launch_step_base(int n_mom, int gdt, bool clip, const StepArgs &a, int num_sms,
                             cudaStream_t st) {
#define MTDAO_STEP_CASE(NN)                                                               \
    case NN:                                                                              \
        if (gdt == MTDAO_F32)                                                             \
            return clip ? launch_step_t<BASE, NN, MTDAO_F32, true>(a, num_sms, st)        \
                        : launch_step_t<BASE, NN, MTDAO_F32, false>(a, num_sms, st);      \
        return clip ? launch_step_t<BASE, NN, MTDAO_BF16, true>(a, num_sms, st)           \
                    : launch_step_t<BASE, NN, MTDAO_BF16, false>(a, num_sms, st);
    if constexpr (BASE == MTDAO_BASE_ADOPT) clip = false;
    switch (n_mom) {
        MTDAO_STEP_CASE(1)
        MTDAO_STEP_CASE(2)
        MTDAO_STEP_CASE(3)
        MTDAO_STEP_CASE(4)
        default:
            return cudaErrorInvalidValue;
    }
#undef MTDAO_STEP_CASE
}

}  // namespace mtdao
