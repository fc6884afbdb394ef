// mtdao_api.cu -- host side of the C ABI declared in include/mtdao.h.
//
// Validation, the flattened layout, the sync schedule, the per-step scalars
// (computed in double from the configuration and the step counter), device
// memory ownership and kernel launches.  No call waits on the device except
// where mtdao.h says it synchronises.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "mtdao.h"
#include "mtdao_internal.h"

namespace mtdao {
template <int BASE>
cudaError_t launch_step_base(int, int, bool, const StepArgs &, int, cudaStream_t);
template <int BASE>
cudaError_t launch_step_sync_base(int, int, bool, const StepArgs &, int, cudaStream_t);
extern template cudaError_t launch_step_base<MTDAO_BASE_ADAM>(int, int, bool, const StepArgs &, int,
                                                              cudaStream_t);
extern template cudaError_t launch_step_base<MTDAO_BASE_ADOPT>(int, int, bool, const StepArgs &, int,
                                                               cudaStream_t);
extern template cudaError_t launch_step_base<MTDAO_BASE_SGDM>(int, int, bool, const StepArgs &, int,
                                                              cudaStream_t);
extern template cudaError_t launch_step_sync_base<MTDAO_BASE_ADAM>(int, int, bool, const StepArgs &,
                                                                   int, cudaStream_t);
extern template cudaError_t launch_step_sync_base<MTDAO_BASE_ADOPT>(int, int, bool, const StepArgs &,
                                                                    int, cudaStream_t);
extern template cudaError_t launch_step_sync_base<MTDAO_BASE_SGDM>(int, int, bool, const StepArgs &,
                                                                   int, cudaStream_t);

cudaError_t launch_step(int base, int n_mom, int gdt, bool clip, const StepArgs &a, int sms,
                        cudaStream_t st) {
    switch (base) {
        case MTDAO_BASE_ADAM: return launch_step_base<MTDAO_BASE_ADAM>(n_mom, gdt, clip, a, sms, st);
        case MTDAO_BASE_ADOPT: return launch_step_base<MTDAO_BASE_ADOPT>(n_mom, gdt, clip, a, sms, st);
        case MTDAO_BASE_SGDM: return launch_step_base<MTDAO_BASE_SGDM>(n_mom, gdt, clip, a, sms, st);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_step_sync(int base, int n_mom, int gdt, bool clip, const StepArgs &a, int sms,
                             cudaStream_t st) {
    switch (base) {
        case MTDAO_BASE_ADAM:
            return launch_step_sync_base<MTDAO_BASE_ADAM>(n_mom, gdt, clip, a, sms, st);
        case MTDAO_BASE_ADOPT:
            return launch_step_sync_base<MTDAO_BASE_ADOPT>(n_mom, gdt, clip, a, sms, st);
        case MTDAO_BASE_SGDM:
            return launch_step_sync_base<MTDAO_BASE_SGDM>(n_mom, gdt, clip, a, sms, st);
        default: return cudaErrorInvalidValue;
    }
}
}  // namespace mtdao

using namespace mtdao;

struct mtdao_ctx {
    mtdao_config cfg;
    int32_t M = 0;
    int32_t n_states = 0;
    int32_t n_tensors = 0;
    int64_t n_padded = 0;
    std::vector<int64_t> offsets;
    int device = 0;
    int num_sms = 1;
    cudaStream_t stream = nullptr;
    float *arena = nullptr;
    float *clip_scale = nullptr;      // [M]
    double *norm_out = nullptr;       // [M]
    double *norm_partial = nullptr;   // [M][norm_blocks]
    int norm_blocks = 1;
    double *stats_partial = nullptr;  // diagnostics workspace (allocated on first use)
    size_t stats_cap = 0;
    float *stats_mean = nullptr;      // M > 8 diagnostics: [n_padded] replica mean (first use)
    float *anchor[2 + MTDAO_MAX_MOM] = {};  // per state: its value at the last average
    // host-gradient staging (mtdao_step_host)
    void *staging[2] = {nullptr, nullptr};
    size_t staging_bytes = 0;
    int staging_next = 0;
    cudaStream_t copy_stream = nullptr;
    cudaEvent_t copy_done[2] = {nullptr, nullptr};
    cudaEvent_t staging_free[2] = {nullptr, nullptr};
    int64_t step = 0;
    std::string err;
};

namespace {

// A named range around each entry point that enqueues GPU work, for Nsight
// tools (ncu --nvtx --nvtx-include "mtdao_step/"); without a tool attached
// a push/pop costs a few nanoseconds.
struct Range {
    explicit Range(const char *name) { nvtxRangePushA(name); }
    ~Range() { nvtxRangePop(); }
    Range(const Range &) = delete;
    Range &operator=(const Range &) = delete;
};

thread_local std::string g_err;

int set_error(mtdao_ctx *h, int code, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (h)
        h->err = buf;
    else
        g_err = buf;
    return code;
}

int cuda_fail(mtdao_ctx *h, cudaError_t e, const char *what) {
    return set_error(h, MTDAO_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool finite_in(double v, double lo, double hi, bool hi_open) {
    if (!std::isfinite(v)) return false;
    return v >= lo && (hi_open ? v < hi : v <= hi);
}

int validate(const mtdao_config *c, int32_t M) {
    if (c == nullptr) return set_error(nullptr, MTDAO_ERR_INVALID, "config is NULL");
    if (c->base < MTDAO_BASE_ADAM || c->base > MTDAO_BASE_SGDM)
        return set_error(nullptr, MTDAO_ERR_INVALID, "unknown base %d", c->base);
    if (c->n_mom < 1 || c->n_mom > MTDAO_MAX_MOM)
        return set_error(nullptr, MTDAO_ERR_INVALID, "n_mom %d outside 1..%d", c->n_mom, MTDAO_MAX_MOM);
    if (M < 1 || M > MTDAO_MAX_REPLICAS)
        return set_error(nullptr, MTDAO_ERR_INVALID, "M %d outside 1..%d", M, MTDAO_MAX_REPLICAS);
    double sum_omega = 0.0;
    for (int j = 0; j < c->n_mom; ++j) {
        if (!finite_in(c->beta1[j], 0.0, 1.0, true))
            return set_error(nullptr, MTDAO_ERR_INVALID, "beta1[%d]=%g outside [0,1)", j, c->beta1[j]);
        if (!finite_in(c->omega[j], 0.0, 1.0, false))
            return set_error(nullptr, MTDAO_ERR_INVALID, "omega[%d]=%g outside [0,1]", j, c->omega[j]);
        if (c->period_u[j] < 0)
            return set_error(nullptr, MTDAO_ERR_INVALID, "period_u[%d] negative", j);
        sum_omega += c->omega[j];
    }
    if (sum_omega > 1.0 + 1e-6)
        return set_error(nullptr, MTDAO_ERR_INVALID, "sum of omega %.9g exceeds 1", sum_omega);
    if (c->base != MTDAO_BASE_SGDM) {
        if (!finite_in(c->beta2, 0.0, 1.0, true))
            return set_error(nullptr, MTDAO_ERR_INVALID, "beta2=%g outside [0,1)", c->beta2);
        if (!(std::isfinite(c->eps) && c->eps > 0.0))
            return set_error(nullptr, MTDAO_ERR_INVALID, "eps=%g must be positive", c->eps);
        if (c->period_v < 0) return set_error(nullptr, MTDAO_ERR_INVALID, "period_v negative");
    }
    if (c->bias_correction != 0 && c->bias_correction != 1)
        return set_error(nullptr, MTDAO_ERR_INVALID, "bias_correction must be 0 or 1");
    if (c->bias_correction && c->base != MTDAO_BASE_ADAM)
        return set_error(nullptr, MTDAO_ERR_INVALID, "bias correction applies to the Adam base only");
    switch (c->clip_mode) {
        case MTDAO_CLIP_NONE: break;
        case MTDAO_CLIP_GLOBAL_NORM:
            if (c->base == MTDAO_BASE_ADOPT)
                return set_error(nullptr, MTDAO_ERR_INVALID, "ADOPT clips elementwise, not by norm");
            if (!(std::isfinite(c->clip_rho) && c->clip_rho > 0.0))
                return set_error(nullptr, MTDAO_ERR_INVALID, "clip_rho=%g must be positive", c->clip_rho);
            break;
        case MTDAO_CLIP_ELEMENTWISE:
            if (c->base != MTDAO_BASE_ADOPT)
                return set_error(nullptr, MTDAO_ERR_INVALID, "elementwise clipping is ADOPT's");
            break;
        default: return set_error(nullptr, MTDAO_ERR_INVALID, "unknown clip mode %d", c->clip_mode);
    }
    if (c->adopt_prev_v != 0 && c->adopt_prev_v != 1)
        return set_error(nullptr, MTDAO_ERR_INVALID, "adopt_prev_v must be 0 or 1");
    if (c->adopt_prev_v && c->base != MTDAO_BASE_ADOPT)
        return set_error(nullptr, MTDAO_ERR_INVALID, "adopt_prev_v applies to the ADOPT base only");
    if (c->sync_phase != MTDAO_PHASE_ALG1 && c->sync_phase != MTDAO_PHASE_ALG2_LITERAL)
        return set_error(nullptr, MTDAO_ERR_INVALID, "unknown sync phase %d", c->sync_phase);
    if (c->period_x < 0) return set_error(nullptr, MTDAO_ERR_INVALID, "period_x negative");
    return MTDAO_OK;
}

int32_t num_states(const mtdao_config *c) {
    return 1 + c->n_mom + (c->base == MTDAO_BASE_SGDM ? 0 : 1);
}

bool divides(int64_t period, int64_t count) { return period > 0 && count % period == 0; }

uint32_t due_mask(const mtdao_config *c, int64_t t) {
    const bool lit = c->sync_phase == MTDAO_PHASE_ALG2_LITERAL;
    const int64_t cm = lit ? t : t + 1;   // count tested for the momenta and v
    uint32_t mask = 0;
    if (divides(c->period_x, t + 1)) mask |= 1u;
    for (int j = 0; j < c->n_mom; ++j)
        if (divides(c->period_u[j], cm)) mask |= 1u << (1 + j);
    if (c->base != MTDAO_BASE_SGDM && divides(c->period_v, cm)) mask |= 1u << (1 + c->n_mom);
    return mask;
}

// Scalars of local step t (see StepScalars), in double then rounded once.
StepScalars step_scalars(const mtdao_config *c, int64_t t, double lr) {
    StepScalars s;
    std::memset(&s, 0, sizeof s);
    const bool adam_bc = c->base == MTDAO_BASE_ADAM && c->bias_correction;
    double sum_omega = 0.0;
    for (int j = 0; j < c->n_mom; ++j) {
        sum_omega += c->omega[j];
        s.c1[j] = static_cast<float>(1.0 - c->beta1[j]);
        const double b = adam_bc ? 1.0 - std::pow(c->beta1[j], static_cast<double>(t + 1)) : 1.0;
        s.k[j] = static_cast<float>(c->omega[j] / b);
    }
    s.neg_lr = static_cast<float>(-lr);
    s.cg = static_cast<float>(1.0 - sum_omega);
    s.c2 = static_cast<float>(1.0 - c->beta2);
    s.sv = adam_bc ? static_cast<float>(1.0 / std::sqrt(1.0 - std::pow(c->beta2, static_cast<double>(t + 1))))
                   : 1.0f;
    s.eps = static_cast<float>(c->eps);
    // k: 1-based index of the parameter update this step makes
    const bool prev_v = c->base == MTDAO_BASE_ADOPT && c->adopt_prev_v;
    const int64_t k = prev_v ? t : t + 1;
    s.clip_c = (c->base == MTDAO_BASE_ADOPT && c->clip_mode == MTDAO_CLIP_ELEMENTWISE && k >= 1)
                   ? static_cast<float>(std::pow(static_cast<double>(k), 0.25))
                   : INFINITY;
    s.prev_v = prev_v ? 1 : 0;
    return s;
}

// Allocation with optional fault injection: MTDAO_FAULT_ALLOC=k makes the
// k-th device allocation of a create (1-based) report out-of-memory.  The
// counter is per thread, so concurrent creates do not disturb each other.
thread_local int g_alloc_counter = 0;

cudaError_t dev_alloc(void **p, size_t bytes) {
    ++g_alloc_counter;
    const char *f = std::getenv("MTDAO_FAULT_ALLOC");
    if (f != nullptr && std::atoi(f) == g_alloc_counter) {
        *p = nullptr;
        return cudaErrorMemoryAllocation;
    }
    return cudaMalloc(p, bytes);
}

void release(mtdao_ctx *h) {
    if (h->stream) cudaStreamSynchronize(h->stream);
    if (h->copy_stream) {
        cudaStreamSynchronize(h->copy_stream);
        cudaStreamDestroy(h->copy_stream);
    }
    for (int i = 0; i < 2; ++i) {
        if (h->staging[i]) cudaFree(h->staging[i]);
        if (h->copy_done[i]) cudaEventDestroy(h->copy_done[i]);
        if (h->staging_free[i]) cudaEventDestroy(h->staging_free[i]);
    }
    if (h->arena) cudaFree(h->arena);
    if (h->clip_scale) cudaFree(h->clip_scale);
    if (h->norm_out) cudaFree(h->norm_out);
    if (h->norm_partial) cudaFree(h->norm_partial);
    if (h->stats_partial) cudaFree(h->stats_partial);
    if (h->stats_mean) cudaFree(h->stats_mean);
    for (float *a : h->anchor)
        if (a) cudaFree(a);
}

int check_handle(mtdao_ctx *h) {
    if (h == nullptr) return set_error(nullptr, MTDAO_ERR_INVALID, "handle is NULL");
    return MTDAO_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool aligned8(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 7u) == 0; }

int select_device(mtdao_ctx *h) {
    int cur = -1;
    cudaError_t e = cudaGetDevice(&cur);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaGetDevice");
    if (cur != h->device) {
        e = cudaSetDevice(h->device);
        if (e != cudaSuccess) return cuda_fail(h, e, "cudaSetDevice");
    }
    return MTDAO_OK;
}

}  // namespace

int mtdao::set_thread_error(int code, const char *msg) { return set_error(nullptr, code, "%s", msg); }

// ====================================================================== host-only

extern "C" int32_t mtdao_version(void) { return MTDAO_VERSION; }

extern "C" int mtdao_config_default(mtdao_config *cfg, int32_t base, int32_t n_mom) {
    if (cfg == nullptr) return set_error(nullptr, MTDAO_ERR_INVALID, "config is NULL");
    if (base < MTDAO_BASE_ADAM || base > MTDAO_BASE_SGDM || n_mom < 1 || n_mom > MTDAO_MAX_MOM)
        return set_error(nullptr, MTDAO_ERR_INVALID, "base %d / n_mom %d unsupported", base, n_mom);
    static const double betas[MTDAO_MAX_MOM] = {0.9, 0.999, 0.5, 0.99};
    std::memset(cfg, 0, sizeof *cfg);
    cfg->base = base;
    cfg->n_mom = n_mom;
    for (int j = 0; j < n_mom; ++j) {
        cfg->beta1[j] = betas[j];
        cfg->omega[j] = 0.95 / n_mom;
        cfg->period_u[j] = 32;
    }
    cfg->beta2 = base == MTDAO_BASE_ADOPT ? 0.9999 : 0.999;
    cfg->eps = 1e-8;
    cfg->bias_correction = base == MTDAO_BASE_ADAM ? 1 : 0;
    cfg->clip_mode = MTDAO_CLIP_NONE;
    cfg->clip_rho = 1.0;
    cfg->sync_phase = MTDAO_PHASE_ALG1;
    cfg->period_x = 32;
    cfg->period_v = base == MTDAO_BASE_SGDM ? 0 : 32;
    cfg->adopt_prev_v = 0;
    return MTDAO_OK;
}

extern "C" int mtdao_config_validate(const mtdao_config *cfg, int32_t M) { return validate(cfg, M); }

extern "C" int32_t mtdao_num_states(const mtdao_config *cfg) {
    if (cfg == nullptr) return 0;
    return num_states(cfg);
}

extern "C" int mtdao_plan_layout(const int64_t *numel, int32_t n_tensors, int64_t *offsets_out,
                                 int64_t *n_padded_out) {
    if (numel == nullptr || n_tensors < 1 || offsets_out == nullptr || n_padded_out == nullptr)
        return set_error(nullptr, MTDAO_ERR_INVALID, "layout: bad arguments");
    int64_t pos = 0;
    for (int32_t k = 0; k < n_tensors; ++k) {
        if (numel[k] < 0) return set_error(nullptr, MTDAO_ERR_INVALID, "tensor %d has numel %lld", k,
                                           static_cast<long long>(numel[k]));
        offsets_out[k] = pos;
        pos += (numel[k] + 7) / 8 * 8;
    }
    if (pos == 0) return set_error(nullptr, MTDAO_ERR_INVALID, "the tensor list holds no element");
    *n_padded_out = (pos + 255) / 256 * 256;
    return MTDAO_OK;
}

extern "C" int mtdao_due_mask(const mtdao_config *cfg, int64_t step, uint32_t *mask_out) {
    if (cfg == nullptr || mask_out == nullptr || step < 0)
        return set_error(nullptr, MTDAO_ERR_INVALID, "due_mask: bad arguments");
    *mask_out = due_mask(cfg, step);
    return MTDAO_OK;
}

extern "C" int mtdao_half_life(double beta, double *tau_out) {
    if (tau_out == nullptr || !(beta >= 0.0 && beta < 1.0))
        return set_error(nullptr, MTDAO_ERR_INVALID, "half_life: beta must lie in [0, 1)");
    *tau_out = beta == 0.0 ? 0.0 : std::log(0.5) / std::log(beta);
    return MTDAO_OK;
}

extern "C" int mtdao_config_half_life_periods(mtdao_config *cfg, int64_t period_x) {
    if (cfg == nullptr || period_x < 0 || cfg->n_mom < 1 || cfg->n_mom > MTDAO_MAX_MOM)
        return set_error(nullptr, MTDAO_ERR_INVALID, "half_life_periods: bad arguments");
    const bool has_v = cfg->base != MTDAO_BASE_SGDM;
    int64_t k_u[MTDAO_MAX_MOM], k_v = cfg->period_v;
    for (int j = 0; j <= cfg->n_mom; ++j) {
        if (j == cfg->n_mom && !has_v) break;
        const double beta = j < cfg->n_mom ? cfg->beta1[j] : cfg->beta2;
        double tau;
        if (mtdao_half_life(beta, &tau) != MTDAO_OK) return MTDAO_ERR_INVALID;
        const int64_t k = std::max<int64_t>(period_x, std::llround(tau));
        if (j < cfg->n_mom) k_u[j] = k; else k_v = k;
    }
    cfg->period_x = period_x;
    for (int j = 0; j < cfg->n_mom; ++j) cfg->period_u[j] = k_u[j];
    cfg->period_v = k_v;
    return MTDAO_OK;
}

extern "C" int mtdao_comm_reduction(const mtdao_config *cfg, double *factor_out) {
    if (cfg == nullptr || factor_out == nullptr || cfg->n_mom < 1 || cfg->n_mom > MTDAO_MAX_MOM)
        return set_error(nullptr, MTDAO_ERR_INVALID, "comm_reduction: bad arguments");
    const int n = cfg->n_mom + (cfg->base == MTDAO_BASE_SGDM ? 1 : 2);
    double vectors_per_step = 0.0;
    for (int s = 0; s < n; ++s) {
        const int64_t k = s == 0 ? cfg->period_x : (s <= cfg->n_mom ? cfg->period_u[s - 1] : cfg->period_v);
        if (k < 0) return set_error(nullptr, MTDAO_ERR_INVALID, "comm_reduction: negative period");
        if (k > 0) vectors_per_step += 1.0 / static_cast<double>(k);
    }
    *factor_out = vectors_per_step > 0.0 ? 1.0 / vectors_per_step : HUGE_VAL;
    return MTDAO_OK;
}

// ====================================================================== lifecycle

extern "C" int mtdao_create(const mtdao_config *cfg, int32_t M, const int64_t *numel, int32_t n_tensors,
                            void *cuda_stream, mtdao_handle *out) {
    if (out == nullptr) return set_error(nullptr, MTDAO_ERR_INVALID, "out is NULL");
    *out = nullptr;
    int rc = validate(cfg, M);
    if (rc != MTDAO_OK) return rc;
    if (numel == nullptr || n_tensors < 1)
        return set_error(nullptr, MTDAO_ERR_INVALID, "empty tensor list");

    mtdao_ctx *h = new mtdao_ctx();
    h->cfg = *cfg;
    h->M = M;
    h->n_states = num_states(cfg);
    h->n_tensors = n_tensors;
    h->offsets.resize(n_tensors);
    rc = mtdao_plan_layout(numel, n_tensors, h->offsets.data(), &h->n_padded);
    if (rc != MTDAO_OK) {
        delete h;
        return rc;
    }
    h->stream = static_cast<cudaStream_t>(cuda_stream);

    cudaError_t e = cudaGetDevice(&h->device);
    if (e == cudaSuccess)
        e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device);
    if (e != cudaSuccess) {
        rc = set_error(nullptr, MTDAO_ERR_CUDA, "no usable CUDA device: %s", cudaGetErrorString(e));
        delete h;
        return rc;
    }

    g_alloc_counter = 0;
    const size_t arena_elems = static_cast<size_t>(h->n_states) * M * h->n_padded;
    h->norm_blocks = norm_blocks_per_replica(h->num_sms, M);
    struct {
        void **p;
        size_t bytes;
        const char *what;
    } allocs[] = {
        {reinterpret_cast<void **>(&h->arena), arena_elems * sizeof(float), "state arena"},
        {reinterpret_cast<void **>(&h->clip_scale), M * sizeof(float), "clip factors"},
        {reinterpret_cast<void **>(&h->norm_out), M * sizeof(double), "norm output"},
        {reinterpret_cast<void **>(&h->norm_partial),
         static_cast<size_t>(M) * h->norm_blocks * sizeof(double), "norm partials"},
    };
    for (auto &a : allocs) {
        e = dev_alloc(a.p, a.bytes);
        if (e != cudaSuccess) {
            cudaGetLastError();
            rc = set_error(nullptr, MTDAO_ERR_OOM, "cudaMalloc of %s (%zu bytes) failed: %s", a.what,
                           a.bytes, cudaGetErrorString(e));
            release(h);
            delete h;
            return rc;
        }
    }
    e = cudaMemsetAsync(h->arena, 0, arena_elems * sizeof(float), h->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
    if (e != cudaSuccess) {
        rc = set_error(nullptr, MTDAO_ERR_CUDA, "zeroing the state arena: %s", cudaGetErrorString(e));
        release(h);
        delete h;
        return rc;
    }
    *out = h;
    return MTDAO_OK;
}

extern "C" void mtdao_destroy(mtdao_handle h) {
    if (h == nullptr) return;
    int cur = -1;
    if (cudaGetDevice(&cur) == cudaSuccess && cur != h->device) cudaSetDevice(h->device);
    release(h);
    if (cur >= 0 && cur != h->device) cudaSetDevice(cur);
    delete h;
}

extern "C" int mtdao_set_stream(mtdao_handle h, void *cuda_stream) {
    if (int rc = check_handle(h)) return rc;
    h->stream = static_cast<cudaStream_t>(cuda_stream);
    return MTDAO_OK;
}

extern "C" int mtdao_set_params(mtdao_handle h, const float *x0_dev) {
    if (int rc = check_handle(h)) return rc;
    if (x0_dev == nullptr) return set_error(h, MTDAO_ERR_INVALID, "x0 is NULL");
    if (int rc = select_device(h)) return rc;
    const size_t bytes = static_cast<size_t>(h->n_padded) * sizeof(float);
    for (int m = 0; m < h->M; ++m) {
        cudaError_t e = cudaMemcpyAsync(h->arena + static_cast<int64_t>(m) * h->n_padded, x0_dev, bytes,
                                        cudaMemcpyDeviceToDevice, h->stream);
        if (e != cudaSuccess) return cuda_fail(h, e, "copying x0");
    }
    const size_t rest = static_cast<size_t>(h->n_states - 1) * h->M * h->n_padded * sizeof(float);
    cudaError_t e = cudaMemsetAsync(h->arena + static_cast<int64_t>(h->M) * h->n_padded, 0, rest, h->stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "zeroing the optimizer states");
    h->step = 0;
    return MTDAO_OK;
}

// ====================================================================== hot path

// After a step or sync that averaged the states in mask, each tracked
// anchor among them becomes the averaged value (replica 0's copy).
static int refresh_anchor(mtdao_ctx *h, uint32_t mask) {
    for (int s = 0; s < h->n_states; ++s) {
        if (h->anchor[s] == nullptr || ((mask >> s) & 1u) == 0) continue;
        const float *src = h->arena + static_cast<int64_t>(s) * h->M * h->n_padded;
        cudaError_t e = cudaMemcpyAsync(h->anchor[s], src, static_cast<size_t>(h->n_padded) * sizeof(float),
                                        cudaMemcpyDeviceToDevice, h->stream);
        if (e != cudaSuccess) return cuda_fail(h, e, "anchor copy");
    }
    return MTDAO_OK;
}

// Diagnostics kernels hold M replicas in registers up to this M; up to
// kWideStatsM they stage all replicas of a span in shared memory (one
// pass); above it they take two passes through a scratch vector (for
// M = 128 and 256 the one-pass form, whose per-element mean is a chain of
// M / 2 compensated additions, ran 2-4x slower than the plain average; the
// two passes take 1.4x).
constexpr int kStatsRegisterM = 8;
constexpr int kWideStatsM = 64;

enum StatsPath { kStatsRegister, kStatsWide, kStatsGeneral };

static StatsPath stats_path(const mtdao_ctx *h) {
    return h->M <= kStatsRegisterM ? kStatsRegister : (h->M <= kWideStatsM ? kStatsWide : kStatsGeneral);
}

static int ensure_stats_workspace(mtdao_ctx *h) {
    const StatsPath path = stats_path(h);
    const bool general = path == kStatsGeneral;
    if (h->stats_partial != nullptr && (!general || h->stats_mean != nullptr)) return MTDAO_OK;
    if (h->stats_partial == nullptr) {
        const size_t cap = path == kStatsGeneral ? general_stats_partial_capacity(h->num_sms, h->M)
                           : path == kStatsWide  ? wide_stats_partial_capacity(h->num_sms, h->n_states, h->M)
                                                 : sync_stats_partial_capacity(h->num_sms, h->n_padded, h->n_states, h->M);
        cudaError_t e = cudaMalloc(reinterpret_cast<void **>(&h->stats_partial), cap * sizeof(double));
        if (e != cudaSuccess) {
            cudaGetLastError();
            h->stats_partial = nullptr;
            return set_error(h, MTDAO_ERR_OOM, "diagnostics workspace: %s", cudaGetErrorString(e));
        }
        h->stats_cap = cap;
    }
    if (general) {
        cudaError_t e = cudaMalloc(reinterpret_cast<void **>(&h->stats_mean), h->n_padded * sizeof(float));
        if (e != cudaSuccess) {
            cudaGetLastError();
            h->stats_mean = nullptr;
            return set_error(h, MTDAO_ERR_OOM, "diagnostics scratch: %s", cudaGetErrorString(e));
        }
    }
    return MTDAO_OK;
}

static int enqueue_sync(mtdao_ctx *h, uint32_t mask) {
    SyncArgs a;
    std::memset(&a, 0, sizeof a);
    a.arena = h->arena;
    a.n_padded = h->n_padded;
    a.stride = static_cast<int64_t>(h->M) * h->n_padded;
    a.M = h->M;
    for (int s = 0; s < h->n_states; ++s)
        if (mask & (1u << s)) a.sel[a.n_sel++] = s;
    cudaError_t e = launch_sync(a, h->num_sms, h->stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "sync launch");
    return MTDAO_OK;
}

extern "C" int mtdao_step(mtdao_handle h, const void *grads_dev, int32_t grad_dtype, double lr,
                          uint32_t sync_mask) {
    Range range("mtdao_step");
    if (int rc = check_handle(h)) return rc;
    if (grads_dev == nullptr) return set_error(h, MTDAO_ERR_INVALID, "grads is NULL");
    if (!aligned16(grads_dev)) return set_error(h, MTDAO_ERR_ALIGN, "grads not 16-byte aligned");
    if (grad_dtype != MTDAO_F32 && grad_dtype != MTDAO_BF16)
        return set_error(h, MTDAO_ERR_INVALID, "unknown gradient dtype %d", grad_dtype);
    if (!std::isfinite(lr)) return set_error(h, MTDAO_ERR_INVALID, "lr is not finite");
    if (sync_mask >> h->n_states) return set_error(h, MTDAO_ERR_INVALID, "sync mask 0x%x has bits beyond "
                                                   "the %d states", sync_mask, h->n_states);
    if (int rc = select_device(h)) return rc;

    const mtdao_config *c = &h->cfg;
    const uint32_t avg_mask = h->M > 1 ? sync_mask : 0u;
    if (c->base == MTDAO_BASE_ADOPT && c->adopt_prev_v && h->step == 0) {
        // Original ADOPT order, step 0: v = g_0^2 on every replica and
        // nothing else moves; then the averages due at the end of the step.
        float *v = h->arena + static_cast<int64_t>(1 + c->n_mom) * h->M * h->n_padded;
        cudaError_t e = launch_adopt_init_v(v, grads_dev, grad_dtype, static_cast<int64_t>(h->M) * h->n_padded,
                                            h->stream);
        if (e != cudaSuccess) return cuda_fail(h, e, "ADOPT initial second-moment launch");
        if (avg_mask != 0)
            if (int rc = enqueue_sync(h, avg_mask)) return rc;
        if (int rc = refresh_anchor(h, sync_mask)) return rc;
        ++h->step;
        return MTDAO_OK;
    }
    const bool clip = c->clip_mode == MTDAO_CLIP_GLOBAL_NORM;
    if (clip) {
        cudaError_t e = launch_grad_sqnorm(grads_dev, grad_dtype, h->M, h->n_padded, h->norm_blocks,
                                           h->norm_partial, h->norm_out, h->clip_scale, c->clip_rho,
                                           h->stream);
        if (e != cudaSuccess) return cuda_fail(h, e, "gradient norm launch");
    }
    StepArgs a;
    std::memset(&a, 0, sizeof a);
    a.arena = h->arena;
    a.grads = grads_dev;
    a.clip_scale = clip ? h->clip_scale : nullptr;
    a.n_padded = h->n_padded;
    a.stride = static_cast<int64_t>(h->M) * h->n_padded;
    a.M = h->M;
    a.sync_mask = avg_mask;
    a.sc = step_scalars(c, h->step, lr);

    cudaError_t e;
    if (a.sync_mask != 0) {
        e = launch_step_sync(c->base, c->n_mom, grad_dtype, clip, a, h->num_sms, h->stream);
        if (e == cudaErrorNotSupported) {
            cudaGetLastError();
            e = launch_step(c->base, c->n_mom, grad_dtype, clip, a, h->num_sms, h->stream);
            if (e != cudaSuccess) return cuda_fail(h, e, "step launch");
            if (int rc = enqueue_sync(h, a.sync_mask)) return rc;
            e = cudaSuccess;
        }
    } else {
        e = launch_step(c->base, c->n_mom, grad_dtype, clip, a, h->num_sms, h->stream);
    }
    if (e != cudaSuccess) return cuda_fail(h, e, "step launch");
    if (int rc = refresh_anchor(h, sync_mask)) return rc;
    ++h->step;
    return MTDAO_OK;
}

extern "C" int mtdao_run(mtdao_handle h, const void *grads_dev, int64_t grads_stride_bytes,
                         int32_t grad_dtype, const double *lrs, int32_t count) {
    Range range("mtdao_run");
    if (int rc = check_handle(h)) return rc;
    if (count < 0 || (count > 0 && (grads_dev == nullptr || lrs == nullptr)))
        return set_error(h, MTDAO_ERR_INVALID, "run: bad count or NULL arguments");
    if (grads_stride_bytes < 0 || grads_stride_bytes % 16 != 0)
        return set_error(h, MTDAO_ERR_ALIGN, "run: gradient stride must be a non-negative multiple of 16");
    for (int32_t k = 0; k < count; ++k) {
        const void *g = static_cast<const char *>(grads_dev) + static_cast<int64_t>(k) * grads_stride_bytes;
        if (int rc = mtdao_step(h, g, grad_dtype, lrs[k], due_mask(&h->cfg, h->step))) return rc;
    }
    return MTDAO_OK;
}

extern "C" int mtdao_step_host(mtdao_handle h, const void *grads_host, int32_t grad_dtype, double lr,
                               uint32_t sync_mask) {
    Range range("mtdao_step_host");
    if (int rc = check_handle(h)) return rc;
    if (grads_host == nullptr) return set_error(h, MTDAO_ERR_INVALID, "grads is NULL");
    if (grad_dtype != MTDAO_F32 && grad_dtype != MTDAO_BF16)
        return set_error(h, MTDAO_ERR_INVALID, "unknown gradient dtype %d", grad_dtype);
    if (int rc = select_device(h)) return rc;
    // Pinned (page-locked or registered) host memory is directly addressable
    // by the GPU: the step kernel streams the gradients over the host link
    // itself, with no staging copy and no staging memory.
    cudaPointerAttributes attr;
    if (cudaPointerGetAttributes(&attr, grads_host) == cudaSuccess && attr.type == cudaMemoryTypeHost &&
        attr.devicePointer != nullptr)
        return mtdao_step(h, attr.devicePointer, grad_dtype, lr, sync_mask);
    cudaGetLastError();
    const size_t full = static_cast<size_t>(h->M) * h->n_padded * sizeof(float);
    const size_t bytes = static_cast<size_t>(h->M) * h->n_padded * (grad_dtype == MTDAO_BF16 ? 2 : 4);
    cudaError_t e;
    if (h->staging[0] == nullptr) {
        for (int i = 0; i < 2; ++i) {
            e = cudaMalloc(&h->staging[i], full);
            if (e != cudaSuccess) {
                cudaGetLastError();
                return set_error(h, MTDAO_ERR_OOM, "staging buffer (%zu bytes): %s", full,
                                 cudaGetErrorString(e));
            }
            if ((e = cudaEventCreateWithFlags(&h->copy_done[i], cudaEventDisableTiming)) != cudaSuccess ||
                (e = cudaEventCreateWithFlags(&h->staging_free[i], cudaEventDisableTiming)) != cudaSuccess)
                return cuda_fail(h, e, "staging events");
        }
        e = cudaStreamCreateWithFlags(&h->copy_stream, cudaStreamNonBlocking);
        if (e != cudaSuccess) return cuda_fail(h, e, "copy stream");
        h->staging_bytes = full;
    }
    const int k = h->staging_next;
    // The copy into buffer k waits for the step that last read buffer k.
    if ((e = cudaStreamWaitEvent(h->copy_stream, h->staging_free[k], 0)) != cudaSuccess ||
        (e = cudaMemcpyAsync(h->staging[k], grads_host, bytes, cudaMemcpyHostToDevice, h->copy_stream)) !=
            cudaSuccess ||
        (e = cudaEventRecord(h->copy_done[k], h->copy_stream)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(h->stream, h->copy_done[k], 0)) != cudaSuccess)
        return cuda_fail(h, e, "host-to-device gradient copy");
    int rc = mtdao_step(h, h->staging[k], grad_dtype, lr, sync_mask);
    if (rc != MTDAO_OK) return rc;
    if ((e = cudaEventRecord(h->staging_free[k], h->stream)) != cudaSuccess)
        return cuda_fail(h, e, "staging release event");
    h->staging_next ^= 1;
    return MTDAO_OK;
}

extern "C" int mtdao_sync(mtdao_handle h, uint32_t mask) {
    Range range("mtdao_sync");
    if (int rc = check_handle(h)) return rc;
    if (mask >> h->n_states) return set_error(h, MTDAO_ERR_INVALID, "sync mask 0x%x has bits beyond "
                                              "the %d states", mask, h->n_states);
    if (mask == 0) return MTDAO_OK;
    if (int rc = select_device(h)) return rc;
    if (h->M > 1)
        if (int rc = enqueue_sync(h, mask)) return rc;
    return refresh_anchor(h, mask);
}

extern "C" int mtdao_sync_stats(mtdao_handle h, uint32_t mask, double *stats_dev) {
    Range range("mtdao_sync_stats");
    if (int rc = check_handle(h)) return rc;
    if (stats_dev == nullptr) return set_error(h, MTDAO_ERR_INVALID, "stats is NULL");
    if (!aligned8(stats_dev)) return set_error(h, MTDAO_ERR_ALIGN, "stats not 8-byte aligned");
    if (mask >> h->n_states) return set_error(h, MTDAO_ERR_INVALID, "sync mask 0x%x has bits beyond "
                                              "the %d states", mask, h->n_states);
    if (mask == 0) return MTDAO_OK;
    if (int rc = select_device(h)) return rc;
    if (int rc = ensure_stats_workspace(h)) return rc;
    SyncArgs a;
    std::memset(&a, 0, sizeof a);
    a.arena = h->arena;
    a.n_padded = h->n_padded;
    a.stride = static_cast<int64_t>(h->M) * h->n_padded;
    a.M = h->M;
    for (int s = 0; s < h->n_states; ++s)
        if (mask & (1u << s)) a.sel[a.n_sel++] = s;
    const StatsPath path = stats_path(h);
    cudaError_t e =
        path == kStatsGeneral
            ? launch_sync_stats_general(a, h->num_sms, h->stats_mean, h->stats_partial, h->stats_cap, stats_dev,
                                        h->stream)
        : path == kStatsWide ? launch_sync_stats_wide(a, h->num_sms, h->stats_partial, h->stats_cap, stats_dev,
                                                      h->stream)
                             : launch_sync_stats(a, h->num_sms, h->stats_partial, h->stats_cap, stats_dev, h->stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "sync with diagnostics launch");
    return refresh_anchor(h, mask);
}

extern "C" int mtdao_track_anchor(mtdao_handle h, uint32_t state_mask) {
    if (int rc = check_handle(h)) return rc;
    if (state_mask >> h->n_states)
        return set_error(h, MTDAO_ERR_INVALID, "state mask 0x%x has bits beyond the %d states", state_mask,
                         h->n_states);
    if (int rc = select_device(h)) return rc;
    bool synced = false;
    for (int s = 0; s < h->n_states; ++s) {
        const bool want = (state_mask >> s) & 1u;
        if (!want && h->anchor[s] != nullptr) {
            if (!synced) {
                cudaStreamSynchronize(h->stream);
                synced = true;
            }
            cudaFree(h->anchor[s]);
            h->anchor[s] = nullptr;
        } else if (want && h->anchor[s] == nullptr) {
            cudaError_t e = cudaMalloc(reinterpret_cast<void **>(&h->anchor[s]),
                                       static_cast<size_t>(h->n_padded) * sizeof(float));
            if (e != cudaSuccess) {
                cudaGetLastError();
                h->anchor[s] = nullptr;
                return set_error(h, MTDAO_ERR_OOM, "anchor of state %d (%lld floats): %s", s,
                                 static_cast<long long>(h->n_padded), cudaGetErrorString(e));
            }
            if (int rc = refresh_anchor(h, 1u << s)) return rc;
        }
    }
    return MTDAO_OK;
}

extern "C" int mtdao_pseudo_grad_stats(mtdao_handle h, int32_t state, double *out_dev) {
    Range range("mtdao_pseudo_grad_stats");
    if (int rc = check_handle(h)) return rc;
    if (out_dev == nullptr) return set_error(h, MTDAO_ERR_INVALID, "out is NULL");
    if (!aligned8(out_dev)) return set_error(h, MTDAO_ERR_ALIGN, "out not 8-byte aligned");
    if (state < 0 || state >= h->n_states) return set_error(h, MTDAO_ERR_INVALID, "state %d out of range", state);
    if (h->anchor[state] == nullptr)
        return set_error(h, MTDAO_ERR_STATE, "state %d has no anchor: track it with mtdao_track_anchor", state);
    if (int rc = select_device(h)) return rc;
    if (int rc = ensure_stats_workspace(h)) return rc;
    const float *x = h->arena + static_cast<int64_t>(state) * h->M * h->n_padded;
    const StatsPath path = stats_path(h);
    cudaError_t e =
        path == kStatsGeneral
            ? launch_pseudo_grad_stats_general(x, h->anchor[state], h->n_padded, h->M, h->num_sms, h->stats_mean,
                                               h->stats_partial, h->stats_cap, out_dev, h->stream)
        : path == kStatsWide ? launch_pseudo_grad_stats_wide(x, h->anchor[state], h->n_padded, h->M, h->num_sms,
                                                             h->stats_partial, h->stats_cap, out_dev, h->stream)
                             : launch_pseudo_grad_stats(x, h->anchor[state], h->n_padded, h->M, h->num_sms,
                                                        h->stats_partial, h->stats_cap, out_dev, h->stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "change diagnostics launch");
    return MTDAO_OK;
}

extern "C" int mtdao_sync_due(mtdao_handle h, uint32_t *mask_out) {
    if (int rc = check_handle(h)) return rc;
    if (mask_out == nullptr) return set_error(h, MTDAO_ERR_INVALID, "mask_out is NULL");
    *mask_out = due_mask(&h->cfg, h->step);
    return MTDAO_OK;
}

extern "C" int mtdao_grad_nonfinite(mtdao_handle h, const void *grads_dev, int32_t grad_dtype,
                                    double *out_dev) {
    Range range("mtdao_grad_nonfinite");
    if (int rc = check_handle(h)) return rc;
    if (grads_dev == nullptr || out_dev == nullptr)
        return set_error(h, MTDAO_ERR_INVALID, "grads or out is NULL");
    if (!aligned16(grads_dev)) return set_error(h, MTDAO_ERR_ALIGN, "grads not 16-byte aligned");
    if (!aligned8(out_dev)) return set_error(h, MTDAO_ERR_ALIGN, "out not 8-byte aligned");
    if (grad_dtype != MTDAO_F32 && grad_dtype != MTDAO_BF16)
        return set_error(h, MTDAO_ERR_INVALID, "unknown gradient dtype %d", grad_dtype);
    if (int rc = select_device(h)) return rc;
    cudaError_t e = launch_grad_nonfinite(grads_dev, grad_dtype, h->M, h->n_padded, h->norm_blocks,
                                          h->norm_partial, out_dev, h->stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "non-finite count launch");
    return MTDAO_OK;
}

extern "C" int mtdao_grad_sqnorm(mtdao_handle h, const void *grads_dev, int32_t grad_dtype,
                                 double *out_dev) {
    Range range("mtdao_grad_sqnorm");
    if (int rc = check_handle(h)) return rc;
    if (grads_dev == nullptr || out_dev == nullptr)
        return set_error(h, MTDAO_ERR_INVALID, "grads or out is NULL");
    if (!aligned16(grads_dev)) return set_error(h, MTDAO_ERR_ALIGN, "grads not 16-byte aligned");
    if (!aligned8(out_dev)) return set_error(h, MTDAO_ERR_ALIGN, "out not 8-byte aligned");
    if (grad_dtype != MTDAO_F32 && grad_dtype != MTDAO_BF16)
        return set_error(h, MTDAO_ERR_INVALID, "unknown gradient dtype %d", grad_dtype);
    if (int rc = select_device(h)) return rc;
    cudaError_t e = launch_grad_sqnorm(grads_dev, grad_dtype, h->M, h->n_padded, h->norm_blocks,
                                       h->norm_partial, out_dev, nullptr, 0.0, h->stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "gradient norm launch");
    return MTDAO_OK;
}

// ====================================================================== state access

static int state_slot(mtdao_ctx *h, int32_t state, int32_t replica, float **p) {
    if (state < 0 || state >= h->n_states || replica < 0 || replica >= h->M)
        return set_error(h, MTDAO_ERR_INVALID, "state %d / replica %d out of range", state, replica);
    *p = h->arena + (static_cast<int64_t>(state) * h->M + replica) * h->n_padded;
    return MTDAO_OK;
}

extern "C" int mtdao_get_state_ptr(mtdao_handle h, int32_t state, int32_t replica, float **dev_ptr) {
    if (int rc = check_handle(h)) return rc;
    if (dev_ptr == nullptr) return set_error(h, MTDAO_ERR_INVALID, "dev_ptr is NULL");
    return state_slot(h, state, replica, dev_ptr);
}

extern "C" int mtdao_copy_state_to_host(mtdao_handle h, int32_t state, int32_t replica, float *host_out) {
    if (int rc = check_handle(h)) return rc;
    if (host_out == nullptr) return set_error(h, MTDAO_ERR_INVALID, "host_out is NULL");
    float *p = nullptr;
    if (int rc = state_slot(h, state, replica, &p)) return rc;
    if (int rc = select_device(h)) return rc;
    cudaError_t e = cudaMemcpyAsync(host_out, p, static_cast<size_t>(h->n_padded) * sizeof(float),
                                    cudaMemcpyDeviceToHost, h->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "device-to-host state copy");
    return MTDAO_OK;
}

extern "C" int mtdao_copy_state_from_host(mtdao_handle h, int32_t state, int32_t replica,
                                          const float *host_in) {
    if (int rc = check_handle(h)) return rc;
    if (host_in == nullptr) return set_error(h, MTDAO_ERR_INVALID, "host_in is NULL");
    float *p = nullptr;
    if (int rc = state_slot(h, state, replica, &p)) return rc;
    if (int rc = select_device(h)) return rc;
    cudaError_t e = cudaMemcpyAsync(p, host_in, static_cast<size_t>(h->n_padded) * sizeof(float),
                                    cudaMemcpyHostToDevice, h->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "host-to-device state copy");
    return MTDAO_OK;
}

extern "C" int mtdao_layout(mtdao_handle h, int64_t *n_padded, int32_t *n_tensors, int32_t *M,
                            int32_t *n_states, const int64_t **tensor_offsets) {
    if (int rc = check_handle(h)) return rc;
    if (n_padded) *n_padded = h->n_padded;
    if (n_tensors) *n_tensors = h->n_tensors;
    if (M) *M = h->M;
    if (n_states) *n_states = h->n_states;
    if (tensor_offsets) *tensor_offsets = h->offsets.data();
    return MTDAO_OK;
}

extern "C" int64_t mtdao_get_step(mtdao_handle h) { return h ? h->step : -1; }

extern "C" int mtdao_set_step(mtdao_handle h, int64_t step) {
    if (int rc = check_handle(h)) return rc;
    if (step < 0) return set_error(h, MTDAO_ERR_INVALID, "step must be >= 0");
    h->step = step;
    return MTDAO_OK;
}

extern "C" const char *mtdao_last_error(mtdao_handle h) {
    return h ? h->err.c_str() : g_err.c_str();
}
