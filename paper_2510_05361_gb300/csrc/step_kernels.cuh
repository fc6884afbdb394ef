// step_kernels.cuh -- the MT-DAO local step (Algorithms 1-3) for sm_103a.
//
// The step is elementwise and HBM-bound (about 0.3 flop per byte), so it is
// written as a persistent grid-stride streaming kernel: every state of every
// replica is read once and written once per step with 128-bit accesses, the
// gradient is read once.  A warp owns a chunk of 256 consecutive elements
// per iteration; lane l handles elements [4l, 4l+4) and [128+4l, 128+4l+4)
// of the chunk, so every warp-wide load or store instruction covers 512
// contiguous bytes of fp32 (256 bytes of bf16 gradient).
//
// This header holds the per-element update shared by both step kernels and
// step_kernel, which is replica-major: the flat index runs over all M
// replicas (M * n_padded elements); it serves every step with no average.
// The fused step + average kernel is in step_sync_kernels.cuh.
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

// One element of one replica for one step.
//   g : raw gradient g_t^m
//   s : clip(g, rho) factor of the replica (1 when not clipping)
//   x, u[0..N-1], v : the element's states, updated in place
template <int BASE, int N>
__device__ __forceinline__ void update_element(const StepScalars &sc, float g, float s,
                                               float &x, float *u, float &v) {
    if constexpr (BASE == MTDAO_BASE_ADOPT) {
        // Algorithm 2: second moment from the raw gradient first, then the
        // normalised and clamped gradient drives every first momentum.  In
        // the original ADOPT order (uniform flag) v is updated after use.
        float gn;
        if (sc.prev_v) {
            gn = g / (sqrtf(v) + sc.eps);
            v = fmaf(sc.c2, fmaf(g, g, -v), v);
        } else {
            v = fmaf(sc.c2, fmaf(g, g, -v), v);
            gn = g / (sqrtf(v) + sc.eps);
        }
        gn = gn > sc.clip_c ? sc.clip_c : (gn < -sc.clip_c ? -sc.clip_c : gn);  // keeps NaN
        float delta = sc.cg * gn;
#pragma unroll
        for (int j = 0; j < N; ++j) {
            u[j] = fmaf(sc.c1[j], gn - u[j], u[j]);
            delta = fmaf(sc.k[j], u[j], delta);
        }
        x = fmaf(sc.neg_lr, delta, x);
    } else {
        // Algorithm 1 (Adam) and Algorithm 3 (SGDM): momenta of the clipped
        // gradient, combined with the gradient term.
        const float gh = __fmul_rn(g, s);   // never contracted into an FMA
        float num = sc.cg * gh;
#pragma unroll
        for (int j = 0; j < N; ++j) {
            u[j] = fmaf(sc.c1[j], gh - u[j], u[j]);
            num = fmaf(sc.k[j], u[j], num);
        }
        if constexpr (BASE == MTDAO_BASE_ADAM) {
            v = fmaf(sc.c2, fmaf(g, g, -v), v);          // raw gradient
            num = num / fmaf(sqrtf(v), sc.sv, sc.eps);    // sqrt(v / b_v) + eps
        }
        x = fmaf(sc.neg_lr, num, x);
    }
}

// ---------------------------------------------------------------- local step

template <int BASE, int N, int GDT, bool CLIP>
__global__ void __launch_bounds__(kThreads) step_kernel(const StepArgs a) {
    constexpr bool kHasV = BASE != MTDAO_BASE_SGDM;
    const int lane = threadIdx.x & 31;
    const int64_t n_chunks = a.stride / kChunk;
    const int64_t warp = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int64_t n_warps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;

    for (int64_t c = warp; c < n_chunks; c += n_warps) {
        const int64_t e0 = c * kChunk + 4 * lane;
        const int64_t e1 = e0 + 128;
        float g[8], x[8], u[N][8], v[8];
        to_array(ld_grad<GDT>(a.grads, e0), g);
        to_array(ld_grad<GDT>(a.grads, e1), g + 4);
        to_array(ld_state(a.arena + e0), x);
        to_array(ld_state(a.arena + e1), x + 4);
#pragma unroll
        for (int j = 0; j < N; ++j) {
            const float *p = a.arena + (1 + j) * a.stride;
            to_array(ld_state(p + e0), u[j]);
            to_array(ld_state(p + e1), u[j] + 4);
        }
        if constexpr (kHasV) {
            const float *p = a.arena + (1 + N) * a.stride;
            to_array(ld_state(p + e0), v);
            to_array(ld_state(p + e1), v + 4);
        }
        float s = 1.0f;
        if constexpr (CLIP) s = __ldg(a.clip_scale + (c * kChunk) / a.n_padded);

#pragma unroll
        for (int k = 0; k < 8; ++k) {
            float uk[N];
#pragma unroll
            for (int j = 0; j < N; ++j) uk[j] = u[j][k];
            float vk = kHasV ? v[k] : 0.0f;
            update_element<BASE, N>(a.sc, g[k], s, x[k], uk, vk);
#pragma unroll
            for (int j = 0; j < N; ++j) u[j][k] = uk[j];
            if constexpr (kHasV) v[k] = vk;
        }

        st_state(a.arena + e0, from_array(x));
        st_state(a.arena + e1, from_array(x + 4));
#pragma unroll
        for (int j = 0; j < N; ++j) {
            float *p = a.arena + (1 + j) * a.stride;
            st_state(p + e0, from_array(u[j]));
            st_state(p + e1, from_array(u[j] + 4));
        }
        if constexpr (kHasV) {
            float *p = a.arena + (1 + N) * a.stride;
            st_state(p + e0, from_array(v));
            st_state(p + e1, from_array(v + 4));
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

template <int BASE, int N, int GDT, bool CLIP>
cudaError_t launch_step_t(const StepArgs &a, int num_sms, cudaStream_t stream) {
    auto kernel = step_kernel<BASE, N, GDT, CLIP>;
    static const int per_sm = blocks_per_sm(kernel);
    const int grid = persistent_grid(per_sm, num_sms, a.stride / kChunk);
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
