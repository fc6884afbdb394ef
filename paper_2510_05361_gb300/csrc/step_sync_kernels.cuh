// step_sync_kernels.cuh -- the local step with the replica average fused in.
//
// step_sync_kernel is element-major: a lane updates the same few elements
// of all M replicas (M <= 7) or of half of them while the other half-warp
// holds the rest (M = 8; see FusedShape), with the update of
// step_kernels.cuh; then it writes each state due for averaging as the
// replica mean (E_m[.] of Algorithms 1-3) instead of the local values.  The
// average costs no HBM traffic beyond the step's own.
#pragma once

#include "replica_mean.cuh"
#include "step_kernels.cuh"
#include "step_sync_wide.cuh"

namespace mtdao {

// ---------------------------------------------------------------- fused step + sync

// Layout of the fused kernel's work.  A lane holds V consecutive elements
// of R replicas; the G lane groups of a warp hold the same elements of
// different replicas (group k: replicas k*R .. k*R + R-1):
//   M = 2, 3, 4 : one group, R = M, V = 4 (128-bit accesses);
//   M = 5, 6, 7 : one group, R = M, V = 2 (four elements spill registers);
//   M = 8       : two groups (half-warps) of R = 4, V = 4: replicas 0..3 and
//                 4..7 are the two parts of the compensated mean of
//                 replica_mean.cuh, combined by shuffles.
// M from 9 to 64 take the block-staged kernel of step_sync_wide.cuh (lane
// groups went further before: M = 16 as four groups of four replicas, the
// compensated sums handed from group to group by shuffles, ran at 4.9-5.3
// TB/s against 5.2 for the block-staged kernel with every state due and 5.7
// against 6.8 with x alone; M = 32 as eight groups loaded 64-byte pieces of
// eight replica slabs and ran slower than the separate average); above 64,
// the plain step followed by the standalone average.
// The states are visited one after another (state_order); the next
// state's loads are issued before the current state is updated and stored,
// so two states' loads are in flight per lane within the 128-register cap.
// Holding all replicas in one lane doubled the bytes a warp of M = 5..7
// has in flight: as two half-warp groups of V = 2 they ran the fused step
// at 3.7-5.8 TB/s on the flat 2^27 sweep, as one group at 5.8-6.7.  The
// lookahead lifted M = 8 from 6030-6065 GB/s to 6485-6727 and M = 4 from
// 6413-6556 (2 elements per lane, every load of the chunk first, as in
// step_kernel) to 6582-6718; M = 2 is the same with or without it.
template <int M>
struct FusedShape {
    static_assert(M >= 2 && M <= 8, "no fused shape for this M");
    static constexpr int G = M == 8 ? 2 : 1;                  // lane groups per warp
    static constexpr int R = M / G;                          // replicas per lane
    static constexpr int V = (M >= 5 && M <= 7) ? 2 : 4;     // elements per lane
    static constexpr int kLanes = 32 / G;                    // lanes per group
    static constexpr int kChunk = kLanes * V;                // elements per warp iteration
};

template <int V>
__device__ __forceinline__ void ld_v(const float *p, float *a) {
    if constexpr (V == 4) {
        to_array(ld_state(p), a);
    } else {
        const float2 t = __ldcs(reinterpret_cast<const float2 *>(p));
        a[0] = t.x;
        a[1] = t.y;
    }
}
template <int V>
__device__ __forceinline__ void st_v(float *p, const float *a) {
    if constexpr (V == 4)
        st_state(p, from_array(a));
    else
        __stcs(reinterpret_cast<float2 *>(p), make_float2(a[0], a[1]));
}

// V consecutive gradient values starting at flat element index e, in fp32.
template <int GDT, int V>
__device__ __forceinline__ void ld_grad_v(const void *g, int64_t e, float *a) {
    if constexpr (V == 4) {
        to_array(ld_grad<GDT>(g, e), a);
    } else if constexpr (GDT == MTDAO_F32) {
        const float2 t = __ldcs(reinterpret_cast<const float2 *>(static_cast<const float *>(g) + e));
        a[0] = t.x;
        a[1] = t.y;
    } else {
        const unsigned int w =
            __ldcs(reinterpret_cast<const unsigned int *>(static_cast<const uint16_t *>(g) + e));
        a[0] = __uint_as_float(w << 16);
        a[1] = __uint_as_float(w & 0xffff0000u);
    }
}

// Writes one state's R local values (for V elements) to the lane's replicas:
// as they are, or -- when the state is due -- all replaced by the replica
// mean of replica_mean.cuh.  With two lane groups each group forms its part
// of the compensated sum (replicas 1..R-1 and R..M-1 against replica 0's
// value; R = M / 2 is where replica_mean.cuh splits its two parts)
// and the parts are exchanged, so both groups store exactly the value a
// single thread would compute.  The standalone averaging kernels use the
// same routine, so fused and separate averaging give identical bits.
template <int M>
__device__ __forceinline__ void store_replicas(float *state, int64_t n_padded, int64_t e, int grp,
                                               float (&val)[FusedShape<M>::R][FusedShape<M>::V],
                                               bool average) {
    using S = FusedShape<M>;
    if (average) {
        float mean[S::V];
#pragma unroll
        for (int k = 0; k < S::V; ++k) {
            if constexpr (S::G == 1) {
                mean[k] = replica_mean<M>([&](int m) { return val[m][k]; });
            } else {
                // replica 0 lives in group 0: its value is the reference of both parts
                const float s0 = __shfl_sync(0xffffffffu, val[0][k], threadIdx.x & (S::kLanes - 1));
                DiffSum part(s0);
#pragma unroll
                for (int r = 0; r < S::R; ++r)      // constant indices: val stays in registers
                    if (r > 0 || grp != 0) part.add(val[r][k]);
                const float mine = part.partial();
                const float other = __shfl_xor_sync(0xffffffffu, mine, S::kLanes);
                const float a = grp == 0 ? mine : other;          // replicas 1 .. R-1
                const float b = grp == 0 ? other : mine;          // replicas R .. M-1
                float plain = val[0][k];                          // for the non-finite case
#pragma unroll
                for (int r = 1; r < S::R; ++r) plain += val[r][k];
                plain += __shfl_xor_sync(0xffffffffu, plain, S::kLanes);
                mean[k] = mean_or_plain(replica_mean_from_parts(s0, a, b, static_cast<float>(M)), plain,
                                        static_cast<float>(M));
            }
        }
#pragma unroll
        for (int r = 0; r < S::R; ++r)
            st_v<S::V>(state + (grp * S::R + r) * n_padded + e, mean);
    } else {
#pragma unroll
        for (int r = 0; r < S::R; ++r)
            st_v<S::V>(state + (grp * S::R + r) * n_padded + e, val[r]);
    }
}

template <int M>
__device__ __forceinline__ void load_replicas(const float *state, int64_t n_padded, int64_t e, int grp,
                                              float (&val)[FusedShape<M>::R][FusedShape<M>::V]) {
    using S = FusedShape<M>;
#pragma unroll
    for (int r = 0; r < S::R; ++r) ld_v<S::V>(state + (grp * S::R + r) * n_padded + e, val[r]);
}

template <int BASE, int N, int GDT, bool CLIP, int M>
__global__ void __launch_bounds__(kThreads, 2) step_sync_kernel(const StepArgs a) {
    using S = FusedShape<M>;
    constexpr int R = S::R;
    constexpr int V = S::V;
    const int lane = threadIdx.x & 31;
    const int q = lane & (S::kLanes - 1);
    const int grp = lane / S::kLanes;
    const int64_t n = a.n_padded;
    const int64_t n_chunks = n / S::kChunk;
    const int64_t warp = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int64_t n_warps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
    const uint32_t mask = a.sync_mask;

    float s[R];
#pragma unroll
    for (int r = 0; r < R; ++r)
        s[r] = CLIP ? __ldg(a.clip_scale + grp * R + r) : 1.0f;

    for (int64_t c = warp; c < n_chunks; c += n_warps) {
        const int64_t e = c * S::kChunk + V * q;
        // Left to itself ptxas keeps the address of every (state, replica)
        // slab in registers across the loop and, with bf16 gradients or
        // V = 2, spills (M = 8, ADOPT, N = 2, bf16: 128 registers and an
        // 8-byte spill).  Passing the two strides through an empty asm
        // statement each iteration makes it recompute the addresses
        // instead (120 registers, no spill; the fused step of that case
        // from 6063 to 6563 GB/s on a flat 2^27).  The f32 instances
        // fit without it and run as fast.
        int64_t nn = n, stride = a.stride;
        if constexpr (GDT == MTDAO_BF16 || V == 2) asm volatile("" : "+l"(nn), "+l"(stride));
        float g[R][V];
#pragma unroll
        for (int r = 0; r < R; ++r) ld_grad_v<GDT, V>(a.grads, (grp * R + r) * nn + e, g[r]);

        // State by state in state_order; the next state's loads are issued
        // before the current state is updated and stored (different states
        // are different slabs, so the reordering is safe).  The arithmetic
        // is update_state's, written out per state (the same expressions,
        // so the same bits; the written-out form keeps the M = 8 ADOPT
        // instance within its registers).
        constexpr int kStates = kNumStates<BASE, N>;
        float gt[R][V];                   // ADOPT: the normalised, clamped gradient
        float buf[2][R][V];
        float acc[R][V];                  // Delta's numerator (Adam, SGDM) or Delta (ADOPT)
        if constexpr (BASE != MTDAO_BASE_ADOPT) {
#pragma unroll
            for (int r = 0; r < R; ++r)
#pragma unroll
                for (int k = 0; k < V; ++k) acc[r][k] = a.sc.cg * __fmul_rn(g[r][k], s[r]);
        }
#pragma unroll
        for (int i = 0; i < kStates; ++i) {
            const int st = state_order<BASE, N>(i);
            if (i == 0)
                load_replicas<M>(a.arena + st * stride, nn, e, grp, buf[0]);
            if (i + 1 < kStates)
                load_replicas<M>(a.arena + state_order<BASE, N>(i + 1) * stride, nn, e, grp,
                                 buf[(i + 1) & 1]);
            float (&cur)[R][V] = buf[i & 1];
            if (st == 1 + N && BASE == MTDAO_BASE_ADOPT) {
                // v first; gt receives the normalised, clamped gradient.
#pragma unroll
                for (int r = 0; r < R; ++r)
#pragma unroll
                    for (int k = 0; k < V; ++k) {
                        const float gr = g[r][k];
                        float gn;
                        if (a.sc.prev_v) {
                            gn = gr / (sqrtf(cur[r][k]) + a.sc.eps);
                            cur[r][k] = fmaf(__fmul_rn(a.sc.c2, gr), gr, ema_decay(a.sc.c2, cur[r][k]));
                        } else {
                            cur[r][k] = fmaf(__fmul_rn(a.sc.c2, gr), gr, ema_decay(a.sc.c2, cur[r][k]));
                            gn = gr / (sqrtf(cur[r][k]) + a.sc.eps);
                        }
                        gn = gn > a.sc.clip_c ? a.sc.clip_c : (gn < -a.sc.clip_c ? -a.sc.clip_c : gn);
                        gt[r][k] = gn;
                        acc[r][k] = a.sc.cg * gn;
                    }
            } else if (st == 1 + N) {
                // Adam: v of the raw gradient, then the denominator.
#pragma unroll
                for (int r = 0; r < R; ++r)
#pragma unroll
                    for (int k = 0; k < V; ++k) {
                        const float gr = g[r][k];
                        cur[r][k] = fmaf(__fmul_rn(a.sc.c2, gr), gr, ema_decay(a.sc.c2, cur[r][k]));
                        acc[r][k] = acc[r][k] / fmaf(sqrtf(cur[r][k]), a.sc.sv, a.sc.eps);
                    }
            } else if (st == 0) {
#pragma unroll
                for (int r = 0; r < R; ++r)
#pragma unroll
                    for (int k = 0; k < V; ++k) cur[r][k] = fmaf(a.sc.neg_lr, acc[r][k], cur[r][k]);
            } else {
                const int j = st - 1;             // momentum u_j
#pragma unroll
                for (int r = 0; r < R; ++r)
#pragma unroll
                    for (int k = 0; k < V; ++k) {
                        const float target =
                            BASE == MTDAO_BASE_ADOPT ? gt[r][k] : __fmul_rn(g[r][k], s[r]);
                        cur[r][k] = fmaf(a.sc.c1[j], target, ema_decay(a.sc.c1[j], cur[r][k]));
                        acc[r][k] = fmaf(a.sc.k[j], cur[r][k], acc[r][k]);
                    }
            }
            store_replicas<M>(a.arena + st * stride, nn, e, grp, cur, (mask >> st) & 1u);
        }
    }
}

// ---------------------------------------------------------------- launch helpers

template <int BASE, int N, int GDT, bool CLIP, int M>
cudaError_t launch_step_sync_t(const StepArgs &a, int num_sms, cudaStream_t stream) {
    // One chunk per warp (stream_grid) where a warp's chunk spans 128
    // elements or more (M <= 4), except for Adam and ADOPT with a single
    // momentum.  Measured on flat 2^27 cases (GB/s, persistent -> one chunk
    // per warp): the ~1B workload's fused step (M = 4, N = 3) 6510 -> 6964,
    // M = 4 N = 2..4 6.6 -> 6.9-7.0 TB/s, SGDM N = 1 6487 -> 7061, but Adam
    // N = 1 6713 -> 6460 (M = 2), 6725 -> 6120 (M = 4), 6108 -> 5346 (M = 3)
    // and ADOPT N = 1 6447 -> 6248.  The 64-element chunks of M >= 5 keep
    // the persistent grid (M = 8, ~350M workload: 6504 -> 6409).
    auto kernel = step_sync_kernel<BASE, N, GDT, CLIP, M>;
    int grid;
    if constexpr (FusedShape<M>::kChunk >= 128 && (N >= 2 || BASE == MTDAO_BASE_SGDM)) {
        grid = stream_grid(a.n_padded / FusedShape<M>::kChunk);
    } else {
        static const int per_sm = blocks_per_sm(kernel);
        grid = persistent_grid(per_sm, num_sms, a.n_padded / FusedShape<M>::kChunk);
    }
    kernel<<<grid, kThreads, 0, stream>>>(a);
    return cudaGetLastError();
}

template <int BASE, int N, int GDT, bool CLIP>
cudaError_t launch_step_sync_m(const StepArgs &a, int num_sms, cudaStream_t st) {
    switch (a.M) {
        case 2: return launch_step_sync_t<BASE, N, GDT, CLIP, 2>(a, num_sms, st);
        case 3: return launch_step_sync_t<BASE, N, GDT, CLIP, 3>(a, num_sms, st);
        case 4: return launch_step_sync_t<BASE, N, GDT, CLIP, 4>(a, num_sms, st);
        case 5: return launch_step_sync_t<BASE, N, GDT, CLIP, 5>(a, num_sms, st);
        case 6: return launch_step_sync_t<BASE, N, GDT, CLIP, 6>(a, num_sms, st);
        case 7: return launch_step_sync_t<BASE, N, GDT, CLIP, 7>(a, num_sms, st);
        case 8: return launch_step_sync_t<BASE, N, GDT, CLIP, 8>(a, num_sms, st);
        default: return launch_step_sync_wide<BASE, N, GDT, CLIP>(a, num_sms, st);
    }
}

template <int BASE>
cudaError_t launch_step_sync_base(int n_mom, int gdt, bool clip, const StepArgs &a, int num_sms,
                                  cudaStream_t st) {
#define MTDAO_SYNC_CASE(NN)                                                                  \
    case NN:                                                                                 \
        if (gdt == MTDAO_F32)                                                                \
            return clip ? launch_step_sync_m<BASE, NN, MTDAO_F32, true>(a, num_sms, st)      \
                        : launch_step_sync_m<BASE, NN, MTDAO_F32, false>(a, num_sms, st);    \
        return clip ? launch_step_sync_m<BASE, NN, MTDAO_BF16, true>(a, num_sms, st)         \
                    : launch_step_sync_m<BASE, NN, MTDAO_BF16, false>(a, num_sms, st);
    if constexpr (BASE == MTDAO_BASE_ADOPT) clip = false;
    switch (n_mom) {
        MTDAO_SYNC_CASE(1)
        MTDAO_SYNC_CASE(2)
        MTDAO_SYNC_CASE(3)
        MTDAO_SYNC_CASE(4)
        default:
            return cudaErrorInvalidValue;
    }
#undef MTDAO_SYNC_CASE
}

}  // namespace mtdao
