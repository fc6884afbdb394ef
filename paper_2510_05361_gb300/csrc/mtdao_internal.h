// mtdao_internal.h -- shared between the C-ABI host code and the kernels.
//
// The per-step scalars are computed on the host in double precision from the
// configuration and the step counter, rounded once to fp32 and passed to the
// kernels by value (they live in the kernel parameter bank, not in memory).
#pragma once

#include <cuda_runtime.h>
#include <cstdint>

#include "mtdao.h"

namespace mtdao {

constexpr int kThreads = 256;        // threads per block of every streaming kernel
constexpr int kChunk = 256;          // elements per warp iteration of the local step
constexpr int kNormThreads = 256;    // threads per block of the norm reduction

// Scalars of one local step t (Algorithms 1-3).  The decay rates enter as
// c = 1 - beta rounded to fp32, which keeps beta's precision when beta is
// close to 1 (the float nearest 0.9999 is 1.7e-8 away from it, the float
// nearest 1e-4 only 2.5e-12).  A first momentum is evaluated as
// fma(c, target, fma(-c, s, s)): beta * s is formed exactly inside the
// inner fma and rounded once, so beta = 0 gives the target exactly however
// large s was.  The second moment is fma(c * g, g, fma(-c, s, s)) in the
// same way, so beta_2 = 0 gives g^2.  An infinite s skips the inner fma
// (ema_decay): beta * s is then s, not the fma's inf - inf.
struct StepScalars {
    float neg_lr;                    // -eta_t
    float c1[MTDAO_MAX_MOM];         // 1 - beta_{1,j}
    float k[MTDAO_MAX_MOM];          // weight of u^j in Delta: omega_j / b_j (Adam), omega_j
    float cg;                        // weight of the gradient term: 1 - sum omega
    float c2;                        // 1 - beta_2
    float sv;                        // Adam: 1 / sqrt(1 - beta_2^(t+1)), or 1
    float eps;                       // epsilon
    float clip_c;                    // ADOPT clamp bound c_t (+inf when not clipping)
    int prev_v;                      // ADOPT: normalise with the previous v (original order);
                                     // its step 0 runs launch_adopt_init_v instead
};

struct StepArgs {
    float *arena;                    // state-major arena, see mtdao.h "Layout"
    const void *grads;               // [M][n_padded] f32 or bf16
    const float *clip_scale;         // [M] global-norm clip factors, or nullptr
    int64_t n_padded;                // elements per replica (multiple of 256)
    int64_t stride;                  // M * n_padded: distance between two states
    int32_t M;
    uint32_t sync_mask;              // fused step+sync only
    StepScalars sc;
};

struct SyncArgs {
    float *arena;
    int64_t n_padded;
    int64_t stride;
    int32_t M;
    int32_t n_sel;                   // number of states to average
    int32_t sel[2 + MTDAO_MAX_MOM];  // their indices
};

// Local step over all replicas (one pass).  Returns the launch error.
cudaError_t launch_step(int base, int n_mom, int grad_dtype, bool clip, const StepArgs &a,
                        int num_sms, cudaStream_t stream);

// Local step with the replica average of the states in a.sync_mask fused
// into the same pass.  For 2 <= M <= 256; returns cudaErrorNotSupported
// otherwise (the caller then runs launch_step followed by launch_sync).
cudaError_t launch_step_sync(int base, int n_mom, int grad_dtype, bool clip, const StepArgs &a,
                             int num_sms, cudaStream_t stream);

// Step 0 of the original ADOPT order: v = g^2 over count elements (all
// replicas' v slabs, contiguous), nothing else touched.
cudaError_t launch_adopt_init_v(float *v, const void *grads, int grad_dtype, int64_t count,
                                cudaStream_t stream);

// Replace each selected state by its mean over the M replicas.
cudaError_t launch_sync(const SyncArgs &a, int num_sms, cudaStream_t stream);

// launch_sync plus the cross-worker diagnostics of every selected state:
// stats[sel * (2 + 2M) + q], q as documented for mtdao_sync_stats.  Needs a
// workspace of sync_stats_partial_capacity() doubles; M must be 1..8
// (cudaErrorNotSupported otherwise).
size_t sync_stats_partial_capacity(int num_sms, int64_t n_padded, int n_states, int M);
cudaError_t launch_sync_stats(const SyncArgs &a, int num_sms, double *partial, size_t partial_cap,
                              double *stats, cudaStream_t stream);

// One-pass diagnostics for 2 <= M <= 256 (the wide layout of the fused
// step): same outputs as launch_sync_stats / launch_pseudo_grad_stats, the
// averaged states bit-identical to launch_sync's.  Workspace: partial needs
// wide_stats_partial_capacity() doubles.
size_t wide_stats_partial_capacity(int num_sms, int n_states, int M);
cudaError_t launch_sync_stats_wide(const SyncArgs &a, int num_sms, double *partial, size_t partial_cap,
                                   double *stats, cudaStream_t stream);
cudaError_t launch_pseudo_grad_stats_wide(const float *x, const float *anchor, int64_t n, int M, int num_sms,
                                          double *partial, size_t partial_cap, double *stats,
                                          cudaStream_t stream);

// Per-replica sum of squares of the gradient: partial sums into
// partial[M][blocks_per_replica], then out[m] (double) and, when
// clip_scale != nullptr, clip_scale[m] = min(1, rho / (sqrt(out[m]) + 1e-6)).
int norm_blocks_per_replica(int num_sms, int M);
cudaError_t launch_grad_sqnorm(const void *grads, int grad_dtype, int32_t M, int64_t n_padded,
                               int blocks_per_replica, double *partial, double *out,
                               float *clip_scale, double rho, cudaStream_t stream);

// Diagnostics for any M, used above 256 (two passes per state through a
// [n_padded] fp32 scratch that holds the replica mean; see reduce_kernels.cu).  Same
// outputs as launch_sync_stats / launch_pseudo_grad_stats; the averaged
// states are bit-identical to launch_sync's.  Workspace: partial needs
// general_stats_partial_capacity() doubles.
size_t general_stats_partial_capacity(int num_sms, int M);
cudaError_t launch_sync_stats_general(const SyncArgs &a, int num_sms, float *mean_scratch, double *partial,
                                      size_t partial_cap, double *stats, cudaStream_t stream);
cudaError_t launch_pseudo_grad_stats_general(const float *x, const float *anchor, int64_t n, int M, int num_sms,
                                             float *mean_scratch, double *partial, size_t partial_cap,
                                             double *stats, cudaStream_t stream);

// Number of NaN / +-Inf gradient values per replica into out[m] (double,
// exact), with the grid and workspace of launch_grad_sqnorm.
cudaError_t launch_grad_nonfinite(const void *grads, int grad_dtype, int32_t M, int64_t n_padded,
                                  int blocks_per_replica, double *partial, double *out, cudaStream_t stream);

// Pseudo-gradient diagnostics of x[M][n] against anchor[n] into stats[2M+2]
// (as documented for mtdao_pseudo_grad_stats); M must be 1..8.  Uses the
// sync-diagnostics workspace.
cudaError_t launch_pseudo_grad_stats(const float *x, const float *anchor, int64_t n, int M, int num_sms,
                                     double *partial, size_t partial_cap, double *stats,
                                     cudaStream_t stream);

// Record a message for mtdao_last_error(NULL) in the calling thread and
// return code (for entry points that have no handle).
int set_thread_error(int code, const char *msg);

}  // namespace mtdao
