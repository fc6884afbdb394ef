// step_sync_kernels.cuh -- the local step with the replica average fused in.
//
// step_sync_kernel is element-major: a lane updates the same V elements
// (V = 4 for M <= 4, V = 2 for M = 8) of all M replicas with the update of
// step_kernels.cuh, then writes each state due for averaging as the replica
// mean (E_m[.] of Algorithms 1-3) instead of the M local values.  The
// average costs no HBM traffic beyond the step's own.
#pragma once

#include "replica_mean.cuh"
#include "step_kernels.cuh"

namespace mtdao {

// ---------------------------------------------------------------- fused step + sync

// V consecutive fp32 states (V = 4: one 128-bit access, V = 2: one 64-bit
// access) and V gradient elements, upcast to fp32.
template <int V>
__device__ __forceinline__ void ld_state_v(const float *p, float *a) {
    if constexpr (V == 4) {
        to_array(ld_state(p), a);
    } else {
        const float2 v = __ldcs(reinterpret_cast<const float2 *>(p));
        a[0] = v.x; a[1] = v.y;
    }
}
template <int V>
__device__ __forceinline__ void st_state_v(float *p, const float *a) {
    if constexpr (V == 4) {
        st_state(p, from_array(a));
    } else {
        __stcs(reinterpret_cast<float2 *>(p), make_float2(a[0], a[1]));
    }
}
template <int GDT, int V>
__device__ __forceinline__ void ld_grad_v(const void *g, int64_t e, float *a) {
    if constexpr (V == 4) {
        to_array(ld_grad<GDT>(g, e), a);
    } else if constexpr (GDT == MTDAO_F32) {
        const float2 v = __ldcs(reinterpret_cast<const float2 *>(static_cast<const float *>(g) + e));
        a[0] = v.x; a[1] = v.y;
    } else {
        const unsigned int w =
            __ldcs(reinterpret_cast<const unsigned int *>(static_cast<const uint16_t *>(g) + e));
        a[0] = __uint_as_float(w << 16); a[1] = __uint_as_float(w & 0xffff0000u);
    }
}

// Elements per lane in the fused step+sync kernel: a lane holds its
// elements of all M replicas for every state it touches, so wide lanes cost
// registers in proportion to M.  Four elements (128-bit accesses) up to M = 4,
// two (64-bit accesses, still whole 32-byte sectors per warp) beyond.
template <int M>
__host__ __device__ constexpr int sync_lane_width() { return M <= 4 ? 4 : 2; }

// Writes the M replicas' values of one state for V elements: either as they
// are, or (when the state is due) all M replaced by the replica mean of
// replica_mean.cuh.  The standalone averaging kernels use the same routine,
// so fused and separate averaging give identical bits.
template <int M, int V>
__device__ __forceinline__ void store_replicas(float *state, int64_t n_padded, int64_t e,
                                               float (&val)[M][V], bool average) {
    if (average) {
        float mean[V];
#pragma unroll
        for (int k = 0; k < V; ++k) {
            ReplicaMean acc(val[0][k]);
#pragma unroll
            for (int m = 1; m < M; ++m) acc.add(val[m][k]);
            mean[k] = acc.value(static_cast<float>(M));
        }
#pragma unroll
        for (int m = 0; m < M; ++m) st_state_v<V>(state + m * n_padded + e, mean);
    } else {
#pragma unroll
        for (int m = 0; m < M; ++m) st_state_v<V>(state + m * n_padded + e, val[m]);
    }
}

template <int M, int V>
__device__ __forceinline__ void load_replicas(const float *state, int64_t n_padded, int64_t e,
                                              float (&val)[M][V]) {
#pragma unroll
    for (int m = 0; m < M; ++m) ld_state_v<V>(state + m * n_padded + e, val[m]);
}

template <int BASE, int N, int GDT, bool CLIP, int M>
__global__ void __launch_bounds__(kThreads, 2) step_sync_kernel(const StepArgs a) {
    constexpr int V = sync_lane_width<M>();
    constexpr int kLaneChunk = 32 * V;              // elements per warp iteration
    const int lane = threadIdx.x & 31;
    const int64_t n = a.n_padded;
    const int64_t n_chunks = n / kLaneChunk;
    const int64_t warp = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int64_t n_warps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
    const uint32_t mask = a.sync_mask;

    float s[M];
#pragma unroll
    for (int m = 0; m < M; ++m) s[m] = CLIP ? __ldg(a.clip_scale + m) : 1.0f;

    for (int64_t c = warp; c < n_chunks; c += n_warps) {
        const int64_t e = c * kLaneChunk + V * lane;
        float g[M][V];
#pragma unroll
        for (int m = 0; m < M; ++m) ld_grad_v<GDT, V>(a.grads, m * n + e, g[m]);

        if constexpr (BASE == MTDAO_BASE_ADOPT) {
            // v first; g becomes the normalised, clamped gradient.
            {
                float v[M][V];
                float *p = a.arena + (1 + N) * a.stride;
                load_replicas<M, V>(p, n, e, v);
#pragma unroll
                for (int m = 0; m < M; ++m)
#pragma unroll
                    for (int k = 0; k < V; ++k) {
                        const float gr = g[m][k];
                        float gn;
                        if (a.sc.prev_v) {
                            gn = gr / (sqrtf(v[m][k]) + a.sc.eps);
                            v[m][k] = fmaf(a.sc.c2, fmaf(gr, gr, -v[m][k]), v[m][k]);
                        } else {
                            v[m][k] = fmaf(a.sc.c2, fmaf(gr, gr, -v[m][k]), v[m][k]);
                            gn = gr / (sqrtf(v[m][k]) + a.sc.eps);
                        }
                        gn = gn > a.sc.clip_c ? a.sc.clip_c : (gn < -a.sc.clip_c ? -a.sc.clip_c : gn);
                        g[m][k] = gn;
                    }
                store_replicas<M, V>(p, n, e, v, (mask >> (1 + N)) & 1u);
            }
            float d[M][V];
#pragma unroll
            for (int m = 0; m < M; ++m)
#pragma unroll
                for (int k = 0; k < V; ++k) d[m][k] = a.sc.cg * g[m][k];
#pragma unroll
            for (int j = 0; j < N; ++j) {
                float u[M][V];
                float *p = a.arena + (1 + j) * a.stride;
                load_replicas<M, V>(p, n, e, u);
#pragma unroll
                for (int m = 0; m < M; ++m)
#pragma unroll
                    for (int k = 0; k < V; ++k) {
                        u[m][k] = fmaf(a.sc.c1[j], g[m][k] - u[m][k], u[m][k]);
                        d[m][k] = fmaf(a.sc.k[j], u[m][k], d[m][k]);
                    }
                store_replicas<M, V>(p, n, e, u, (mask >> (1 + j)) & 1u);
            }
            float x[M][V];
            load_replicas<M, V>(a.arena, n, e, x);
#pragma unroll
            for (int m = 0; m < M; ++m)
#pragma unroll
                for (int k = 0; k < V; ++k) x[m][k] = fmaf(a.sc.neg_lr, d[m][k], x[m][k]);
            store_replicas<M, V>(a.arena, n, e, x, mask & 1u);
        } else {
            // Adam / SGDM: momenta of the clipped gradient g * s[m], then
            // (Adam) v of the raw gradient and the denominator, then x.
            float num[M][V];
#pragma unroll
            for (int m = 0; m < M; ++m)
#pragma unroll
                for (int k = 0; k < V; ++k) num[m][k] = a.sc.cg * __fmul_rn(g[m][k], s[m]);
#pragma unroll
            for (int j = 0; j < N; ++j) {
                float u[M][V];
                float *p = a.arena + (1 + j) * a.stride;
                load_replicas<M, V>(p, n, e, u);
#pragma unroll
                for (int m = 0; m < M; ++m)
#pragma unroll
                    for (int k = 0; k < V; ++k) {
                        u[m][k] = fmaf(a.sc.c1[j], __fmul_rn(g[m][k], s[m]) - u[m][k], u[m][k]);
                        num[m][k] = fmaf(a.sc.k[j], u[m][k], num[m][k]);
                    }
                store_replicas<M, V>(p, n, e, u, (mask >> (1 + j)) & 1u);
            }
            if constexpr (BASE == MTDAO_BASE_ADAM) {
                float v[M][V];
                float *p = a.arena + (1 + N) * a.stride;
                load_replicas<M, V>(p, n, e, v);
#pragma unroll
                for (int m = 0; m < M; ++m)
#pragma unroll
                    for (int k = 0; k < V; ++k) {
                        const float gr = g[m][k];
                        v[m][k] = fmaf(a.sc.c2, fmaf(gr, gr, -v[m][k]), v[m][k]);
                        num[m][k] = num[m][k] / fmaf(sqrtf(v[m][k]), a.sc.sv, a.sc.eps);
                    }
                store_replicas<M, V>(p, n, e, v, (mask >> (1 + N)) & 1u);
            }
            float x[M][V];
            load_replicas<M, V>(a.arena, n, e, x);
#pragma unroll
            for (int m = 0; m < M; ++m)
#pragma unroll
                for (int k = 0; k < V; ++k) x[m][k] = fmaf(a.sc.neg_lr, num[m][k], x[m][k]);
            store_replicas<M, V>(a.arena, n, e, x, mask & 1u);
        }
    }
}

// ---------------------------------------------------------------- launch helpers

template <int BASE, int N, int GDT, bool CLIP, int M>
cudaError_t launch_step_sync_t(const StepArgs &a, int num_sms, cudaStream_t stream) {
    auto kernel = step_sync_kernel<BASE, N, GDT, CLIP, M>;
    static const int per_sm = blocks_per_sm(kernel);
    const int grid = persistent_grid(per_sm, num_sms, a.n_padded / (32 * sync_lane_width<M>()));
    kernel<<<grid, kThreads, 0, stream>>>(a);
    return cudaGetLastError();
}

template <int BASE, int N, int GDT, bool CLIP>
cudaError_t launch_step_sync_m(const StepArgs &a, int num_sms, cudaStream_t st) {
    switch (a.M) {
        case 2: return launch_step_sync_t<BASE, N, GDT, CLIP, 2>(a, num_sms, st);
        case 4: return launch_step_sync_t<BASE, N, GDT, CLIP, 4>(a, num_sms, st);
        case 8: return launch_step_sync_t<BASE, N, GDT, CLIP, 8>(a, num_sms, st);
        default: return cudaErrorNotSupported;
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
