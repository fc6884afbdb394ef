/*
 * mtdao_oracle.c -- plain, slow CPU oracle for the MT-DAO hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the correctness reference that the
 * CUDA library is checked against.  Only the test suite, the smoke check and
 * the CPU-baseline leg of the benchmark may load or run it; the product path
 * never does.  It shares no code, header, table or constant with the CUDA
 * library: it is written from the paper (MT-DAO, arXiv 2510.05361) alone.
 *
 * Precision: every state is held and updated in IEEE double (fp64); per-step
 * scalars (beta^(t+1), c_t) are computed in double too.  Inputs (gradients,
 * initial states) arrive as doubles.  Nothing is blocked, fused or reordered:
 * each worker m and element i is visited in index order, the states in the
 * order the algorithms list them.
 *
 * What it computes (one call = one iteration t of the outer loop):
 *   Algorithm 1 (MT-DAO-Adam), Algorithm 2 (MT-DAO-ADOPT) and Algorithm 3
 *   (MT-DAO-SGDM) for M workers held side by side, with the periodic
 *   averaging E_m[.] of x, each u^j and v (Algorithms 1-3, the "sync every
 *   K steps" rows) on each state's own period.
 *
 * Readings of points the paper leaves open (each one is a config field):
 *   - Sync phase.  Algorithm 1 averages a state just before step t reads it
 *     when t mod K_s == 0 (u-bar_{t-1}, v-bar_{t-1}, x-bar_t).  Algorithm 2
 *     instead averages u and v right after step t when t mod K == 0 and x
 *     after step t when (t+1) mod K_x == 0.  Default (phase 0) is Algorithm
 *     1's rule for every base; phase 1 is Algorithm 2's literal rule.
 *   - Bias correction.  Algorithm 1's caption says local bias correction is
 *     omitted for space.  With bias_correction=1 each first momentum u^j is
 *     divided by 1-beta_{1,j}^(t+1) and v by 1-beta_2^(t+1) (t 0-based, the
 *     global step, identical on all workers) before they form the update.
 *     Algorithms 2 and 3 are used as printed (no correction).
 *   - eps sits outside the square root (Algorithm 1 update-direction row).
 *   - clip(g, rho) for Adam/SGDM is norm clipping of the worker's whole
 *     flattened gradient: g-hat = g * min(1, rho / (||g||_2 + 1e-6)).  The
 *     second moment v keeps the raw gradient, as Algorithm 1 writes it.
 *   - clip(g-hat, c_t) for ADOPT is an elementwise clamp to [-c_t, c_t] with
 *     c_t = (t+1)^(1/4), or no clamp at all.
 *   - ADOPT normalises with the freshly updated v_t (Algorithm 2 order).
 *     adopt_prev_v=1 selects the ordering of the original ADOPT method
 *     instead: step 0 only sets v = g_0^2 (no momentum or parameter update),
 *     and every later step normalises with the previous v before updating
 *     it; the clamp bound is then c = t^(1/4), t being the 1-based index of
 *     the parameter update in both orders.
 */
#include <math.h>
#include <stddef.h>
#include <string.h>

#define MTO_MAX_MOM 8

enum { MTO_ADAM = 0, MTO_ADOPT = 1, MTO_SGDM = 2 };
enum { MTO_CLIP_NONE = 0, MTO_CLIP_GLOBAL_NORM = 1, MTO_CLIP_ELEMENTWISE = 2 };
enum { MTO_PHASE_ALG1 = 0, MTO_PHASE_ALG2_LITERAL = 1 };

typedef struct {
    int base;                       /* MTO_ADAM / MTO_ADOPT / MTO_SGDM        */
    int n_mom;                      /* N, number of first momenta             */
    double beta1[MTO_MAX_MOM];      /* beta_{1,j}                             */
    double omega[MTO_MAX_MOM];      /* omega_j, sum <= 1                      */
    double beta2;                   /* beta_2 (Adam/ADOPT)                    */
    double eps;                     /* epsilon                                */
    int bias_correction;            /* Adam only                              */
    int clip_mode;                  /* MTO_CLIP_*                             */
    double clip_rho;                /* rho for global-norm clipping           */
    long long period_x;             /* K_x  (0 = never average)               */
    long long period_u[MTO_MAX_MOM];/* K_j                                    */
    long long period_v;             /* K_v                                    */
    int sync_phase;                 /* MTO_PHASE_*                            */
    int adopt_prev_v;               /* ADOPT: original ordering (see above)   */
} mto_cfg;

/* Number of state vectors per worker: x, u^1..u^N and (Adam/ADOPT) v. */
int mto_num_states(const mto_cfg *c)
{
    return 1 + c->n_mom + (c->base == MTO_SGDM ? 0 : 1);
}

/* Bit of state s in a sync mask: bit 0 = x, bit j = u^j, bit N+1 = v. */
static unsigned bit_x(void) { return 1u; }
static unsigned bit_u(int j) { return 1u << (1 + j); }           /* j 0-based */
static unsigned bit_v(const mto_cfg *c) { return 1u << (1 + c->n_mom); }

static int divides(long long period, long long count)
{
    return period > 0 && count % period == 0;
}

/*
 * Algorithm 1 rule: the states that step t reads in averaged ("barred")
 * form, i.e. those whose period divides t.
 */
unsigned mto_due_before_step(const mto_cfg *c, long long t)
{
    unsigned mask = 0;
    if (divides(c->period_x, t)) mask |= bit_x();
    for (int j = 0; j < c->n_mom; ++j)
        if (divides(c->period_u[j], t)) mask |= bit_u(j);
    if (c->base != MTO_SGDM && divides(c->period_v, t)) mask |= bit_v(c);
    return mask;
}

/*
 * Algorithm 2 literal rule: states averaged right after step t.
 * u^j and v when t mod K == 0, x when (t+1) mod K_x == 0.
 */
unsigned mto_due_after_step(const mto_cfg *c, long long t)
{
    unsigned mask = 0;
    if (divides(c->period_x, t + 1)) mask |= bit_x();
    for (int j = 0; j < c->n_mom; ++j)
        if (divides(c->period_u[j], t)) mask |= bit_u(j);
    if (c->base != MTO_SGDM && divides(c->period_v, t)) mask |= bit_v(c);
    return mask;
}

/*
 * Half-life of the EMA u = beta u + (1 - beta) g (section 2.1): the number
 * of steps after which a past value's weight beta^k has fallen to 1/2,
 * tau = ln(0.5) / ln(beta).  A rate of 0 remembers nothing: 0.
 */
double mto_half_life(double beta)
{
    if (beta == 0.0)
        return 0.0;
    return log(0.5) / log(beta);
}

/*
 * The half-life sync strategy of the wall-clock appendix (its table of the
 * modelled configurations): parameters every K_x steps; each momentum and
 * the second moment every round(half-life of its rate) steps, but not more
 * often than the parameters.  The caption mentions powers of two, yet the
 * printed periods are the rounded half-lives; those are what this follows.
 */
static long long half_life_period(double beta, long long period_x)
{
    long long k = (long long)floor(mto_half_life(beta) + 0.5);
    return k < period_x ? period_x : k;
}

void mto_half_life_periods(mto_cfg *c, long long period_x)
{
    c->period_x = period_x;
    for (int j = 0; j < c->n_mom; ++j)
        c->period_u[j] = half_life_period(c->beta1[j], period_x);
    if (c->base != MTO_SGDM)
        c->period_v = half_life_period(c->beta2, period_x);
}

/*
 * Communication relative to DDP (section 2.3): DDP averages one
 * d-vector per step; here state s is averaged once per K_s steps, so the
 * saving is 1 / (1/K_x + sum_j 1/K_j + 1/K_v).  Periods of 0 (never) add
 * nothing; if no state is ever averaged the saving is infinite.
 */
double mto_comm_reduction(const mto_cfg *c)
{
    double per_step = 0.0;
    if (c->period_x > 0) per_step += 1.0 / (double)c->period_x;
    for (int j = 0; j < c->n_mom; ++j)
        if (c->period_u[j] > 0) per_step += 1.0 / (double)c->period_u[j];
    if (c->base != MTO_SGDM && c->period_v > 0) per_step += 1.0 / (double)c->period_v;
    return per_step > 0.0 ? 1.0 / per_step : INFINITY;
}

/* E_m[s]: replace s^m by the equal-weight mean over the M workers. */
void mto_mean_over_workers(int M, long long n, double *s)
{
    for (long long i = 0; i < n; ++i) {
        double sum = 0.0;
        for (int m = 0; m < M; ++m)
            sum += s[(long long)m * n + i];
        double mean = sum / (double)M;
        for (int m = 0; m < M; ++m)
            s[(long long)m * n + i] = mean;
    }
}

/*
 * Average the states selected by mask.  Layout: x[M][n], u[N][M][n], v[M][n].
 */
void mto_sync(const mto_cfg *c, int M, long long n, unsigned mask,
              double *x, double *u, double *v)
{
    if (mask & bit_x()) mto_mean_over_workers(M, n, x);
    for (int j = 0; j < c->n_mom; ++j)
        if (mask & bit_u(j))
            mto_mean_over_workers(M, n, u + (long long)j * M * n);
    if (c->base != MTO_SGDM && (mask & bit_v(c)))
        mto_mean_over_workers(M, n, v);
}

/*
 * Cross-worker diagnostics of one state s[M][n] (section 4.1, "Other
 * Metrics"), from the definitions, before any averaging:
 *   out[0]           (1/M) sum_m ||s_m - s_bar||^2   (cross-worker variance)
 *   out[1]           ||s_bar||^2
 *   out[2 + m]       ||s_m||^2
 *   out[2 + M + m]   <s_m, s_bar>   (with the norms: cosine similarity)
 * where s_bar = E_m[s] is the worker mean.
 */
void mto_state_stats(int M, long long n, const double *s, double *out)
{
    for (int k = 0; k < 2 + 2 * M; ++k) out[k] = 0.0;
    for (long long i = 0; i < n; ++i) {
        double sum = 0.0;
        for (int m = 0; m < M; ++m) sum += s[(long long)m * n + i];
        double mean = sum / (double)M;
        out[1] += mean * mean;
        for (int m = 0; m < M; ++m) {
            double v = s[(long long)m * n + i];
            out[0] += (v - mean) * (v - mean) / (double)M;
            out[2 + m] += v * v;
            out[2 + M + m] += v * mean;
        }
    }
}

/*
 * Pseudo-gradient diagnostics (section 4.1 "Other Metrics"; section 5.4 uses
 * the worker update over a round, Delta^m = x^m_{t+K} - x^m_t, and its mean,
 * the global pseudo-gradient).  a = the parameters at the start of the round
 * (the last average), x[M][n] the workers' parameters now, x_bar = E_m[x]:
 *   out[m]           ||x_m - a||^2                         m = 0..M-1
 *   out[M + m]       <x_m - a, x_bar - a>
 *   out[2M]          ||x_bar - a||^2
 *   out[2M + 1]      ||a||^2
 * so cos(local, global pseudo-gradient) = out[M+m] / sqrt(out[m] out[2M]) and
 * the relative change of the averaged model = sqrt(out[2M] / out[2M+1]).
 */
void mto_pseudo_grad_stats(int M, long long n, const double *x, const double *a, double *out)
{
    for (int k = 0; k < 2 * M + 2; ++k) out[k] = 0.0;
    for (long long i = 0; i < n; ++i) {
        double sum = 0.0;
        for (int m = 0; m < M; ++m) sum += x[(long long)m * n + i];
        double global = sum / (double)M - a[i];
        out[2 * M] += global * global;
        out[2 * M + 1] += a[i] * a[i];
        for (int m = 0; m < M; ++m) {
            double local = x[(long long)m * n + i] - a[i];
            out[m] += local * local;
            out[M + m] += local * global;
        }
    }
}

/* ||g^m||_2 of one worker's flattened gradient, summed in index order. */
double mto_grad_norm(long long n, const double *g)
{
    double ss = 0.0;
    for (long long i = 0; i < n; ++i)
        ss += g[i] * g[i];
    return sqrt(ss);
}

/* Factor that clip(g, rho) applies to worker m's gradient. */
double mto_clip_factor(const mto_cfg *c, long long n, const double *g)
{
    if (c->clip_mode != MTO_CLIP_GLOBAL_NORM)
        return 1.0;
    double norm = mto_grad_norm(n, g);
    double f = c->clip_rho / (norm + 1e-6);
    return f < 1.0 ? f : 1.0;
}

/* c_t of the ADOPT clip schedule (t 0-based). */
double mto_adopt_clip_bound(long long t)
{
    return pow((double)(t + 1), 0.25);
}

/* Algorithm 1, one worker, one element: returns the new x. */
static double adam_element(const mto_cfg *c, long long t, double lr,
                           double g, double g_hat,
                           double *x, double *u_j[], long long k, double *v)
{
    double sum_omega = 0.0;
    for (int j = 0; j < c->n_mom; ++j) sum_omega += c->omega[j];

    /* N first momenta on the clipped gradient. */
    double combo = (1.0 - sum_omega) * g_hat;
    for (int j = 0; j < c->n_mom; ++j) {
        double b = c->beta1[j];
        double u_new = b * u_j[j][k] + (1.0 - b) * g_hat;
        u_j[j][k] = u_new;
        double corr = c->bias_correction ? 1.0 - pow(b, (double)(t + 1)) : 1.0;
        combo += c->omega[j] * (u_new / corr);
    }
    /* Second momentum on the raw gradient. */
    double v_new = c->beta2 * v[k] + (1.0 - c->beta2) * g * g;
    v[k] = v_new;
    double corr_v = c->bias_correction ? 1.0 - pow(c->beta2, (double)(t + 1)) : 1.0;
    double delta = combo / (sqrt(v_new / corr_v) + c->eps);
    x[k] = x[k] - lr * delta;
    return x[k];
}

/* Algorithm 2, one worker, one element. */
static double adopt_element(const mto_cfg *c, long long t, double lr, double g,
                            double *x, double *u_j[], long long k, double *v)
{
    double sum_omega = 0.0;
    for (int j = 0; j < c->n_mom; ++j) sum_omega += c->omega[j];

    double g_hat;
    long long update_index = t;           /* 0-based index of this x update */
    if (c->adopt_prev_v) {
        if (t == 0) {                     /* v_0 = g_0^2; nothing else moves */
            v[k] = g * g;
            return x[k];
        }
        g_hat = g / (sqrt(v[k]) + c->eps);
        v[k] = c->beta2 * v[k] + (1.0 - c->beta2) * g * g;
        update_index = t - 1;
    } else {
        double v_new = c->beta2 * v[k] + (1.0 - c->beta2) * g * g;
        v[k] = v_new;
        g_hat = g / (sqrt(v_new) + c->eps);
    }
    double g_tilde = g_hat;
    if (c->clip_mode == MTO_CLIP_ELEMENTWISE) {
        double ct = mto_adopt_clip_bound(update_index);
        if (g_tilde > ct) g_tilde = ct;
        if (g_tilde < -ct) g_tilde = -ct;
    }
    double delta = (1.0 - sum_omega) * g_tilde;
    for (int j = 0; j < c->n_mom; ++j) {
        double b = c->beta1[j];
        double u_new = b * u_j[j][k] + (1.0 - b) * g_tilde;
        u_j[j][k] = u_new;
        delta += c->omega[j] * u_new;
    }
    x[k] = x[k] - lr * delta;
    return x[k];
}

/* Algorithm 3, one worker, one element. */
static double sgdm_element(const mto_cfg *c, double lr, double g_hat,
                           double *x, double *u_j[], long long k)
{
    double sum_omega = 0.0;
    for (int j = 0; j < c->n_mom; ++j) sum_omega += c->omega[j];

    double delta = (1.0 - sum_omega) * g_hat;
    for (int j = 0; j < c->n_mom; ++j) {
        double b = c->beta1[j];
        double u_new = b * u_j[j][k] + (1.0 - b) * g_hat;
        u_j[j][k] = u_new;
        delta += c->omega[j] * u_new;
    }
    x[k] = x[k] - lr * delta;
    return x[k];
}

/*
 * One iteration t of the outer loop for all M workers.
 *   g : [M][n]        stochastic gradients g_t^m (input)
 *   x : [M][n]        parameters x_t^m        -> x_{t+1}^m
 *   u : [N][M][n]     first momenta u_{t-1}   -> u_t
 *   v : [M][n]        second momentum v_{t-1} -> v_t  (ignored for SGDM)
 * Returns 0, or -1 for an unusable configuration.
 */
int mto_step(const mto_cfg *c, int M, long long n, long long t, double lr,
             const double *g, double *x, double *u, double *v)
{
    if (c->n_mom < 0 || c->n_mom > MTO_MAX_MOM || M < 1 || n < 0 || t < 0)
        return -1;
    /* ADOPT clips the normalised gradient elementwise; Adam and SGDM clip
     * the raw gradient by its norm.  Any other pairing is not an algorithm
     * of the paper. */
    if (c->base == MTO_ADOPT && c->clip_mode == MTO_CLIP_GLOBAL_NORM) return -1;
    if (c->base != MTO_ADOPT && c->clip_mode == MTO_CLIP_ELEMENTWISE) return -1;
    if (c->base != MTO_ADOPT && c->adopt_prev_v) return -1;

    if (c->sync_phase == MTO_PHASE_ALG1)
        mto_sync(c, M, n, mto_due_before_step(c, t), x, u, v);

    for (int m = 0; m < M; ++m) {
        const double *gm = g + (long long)m * n;
        double *xm = x + (long long)m * n;
        double *vm = v ? v + (long long)m * n : NULL;
        double *um[MTO_MAX_MOM];
        for (int j = 0; j < c->n_mom; ++j)
            um[j] = u + ((long long)j * M + m) * n;

        double f = (c->base == MTO_ADOPT) ? 1.0 : mto_clip_factor(c, n, gm);
        for (long long i = 0; i < n; ++i) {
            if (c->base == MTO_ADAM)
                adam_element(c, t, lr, gm[i], f * gm[i], xm, um, i, vm);
            else if (c->base == MTO_ADOPT)
                adopt_element(c, t, lr, gm[i], xm, um, i, vm);
            else
                sgdm_element(c, lr, f * gm[i], xm, um, i);
        }
    }

    if (c->sync_phase == MTO_PHASE_ALG2_LITERAL)
        mto_sync(c, M, n, mto_due_after_step(c, t), x, u, v);
    return 0;
}

/*
 * The states as the next iteration t would read them: under Algorithm 1's
 * rule, average those whose period divides t (the barred values of step t).
 * Under the literal Algorithm 2 rule nothing is pending.  Lets a caller
 * compare the oracle's states after T steps with an implementation that
 * performs each average at the end of the step that completes a period.
 */
void mto_settle(const mto_cfg *c, int M, long long n, long long t,
                double *x, double *u, double *v)
{
    if (c->sync_phase == MTO_PHASE_ALG1)
        mto_sync(c, M, n, mto_due_before_step(c, t), x, u, v);
}

/*
 * Run T consecutive iterations t0 .. t0+T-1 with gradients g[T][M][n] and a
 * learning rate per iteration, then settle.  Used to time the oracle.
 */
int mto_run(const mto_cfg *c, int M, long long n, long long t0, long long T,
            const double *lr, const double *g, double *x, double *u, double *v)
{
    for (long long s = 0; s < T; ++s) {
        int rc = mto_step(c, M, n, t0 + s, lr[s], g + s * (long long)M * n, x, u, v);
        if (rc) return rc;
    }
    mto_settle(c, M, n, t0 + T, x, u, v);
    return 0;
}
