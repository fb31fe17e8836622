/*
 * CPU oracle for the AGS optimizer step (Tula, arXiv 2603.18112).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is a plain, slow restatement of what
 * the optimizer step computes, written from the paper (single-threaded; the
 * step's per-tensor parts can also run on several threads, for the CPU
 * baseline on all host cores, with the same result):
 * the data-parallel mean of Eq. 1c, the gradient-variability metric of Eq. 5,
 * the scaled/unscaled branch and UpdateGradScale of Algorithm 1, the static
 * scaling function of Eq. 8, and the momentum-SGD + weight-decay update that
 * the paper's TulaOptimizer wraps (Sec. IV-A, IV-B).  Only the test-suite,
 * the smoke check and the benchmark's CPU-baseline leg may load it.  It shares
 * no code, header or constant with the CUDA library.
 *
 * Precision (a reading; the paper names none): parameters, gradients and
 * momentum are fp32 tensors, so every element-wise operation is one IEEE fp32
 * operation, in the order the equations write it, with no fused multiply-add
 * (build with -ffp-contract=off).  Squared norms are accumulated in fp64,
 * element 0 first, with compensated summation (the square of an fp32 value is
 * exact in fp64); the global norm and the variability metric are fp64.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* rule: how the per-tensor coefficient c_p is chosen */
#define OR_RULE_AGS 0    /* Algorithm 1: c = gradscale[p] when Delta < delta, else 1 */
#define OR_RULE_NONE 1   /* vanilla large batch (LBT): c = 1 */
#define OR_RULE_LARS 2   /* prior art (Sec. V-B): c = trust * ||w|| / ||g|| */
#define OR_RULE_STATIC 3 /* Eq. 8: c = s when Delta < delta, else 1 */

#define OR_GRAN_TENSOR 0  /* one gradscale value per tensor */
#define OR_GRAN_ELEMENT 1 /* one gradscale value per element */

#define OR_BRANCH_AUTO 0
#define OR_BRANCH_SCALED 1
#define OR_BRANCH_UNSCALED 2

#define OR_STATS_LEN 8
#define OR_STATE_LEN 4

typedef struct {
    int K;             /* replica gradient buffers */
    int rule;          /* OR_RULE_* */
    int granularity;   /* OR_GRAN_* */
    int force_branch;  /* OR_BRANCH_* */
    int refresh_scale; /* 1: UpdateGradScale from replica 0 vs the mean after the update */
    int has_momentum;  /* 0: no momentum buffer, w -= lr * d */
    float delta;       /* threshold on Delta(G) */
    float eps;         /* stability term of UpdateGradScale */
    float s_max;       /* bound on every scale factor */
    float static_s;    /* s of Eq. 8 */
    float lars_trust;  /* trust coefficient of the LARS rule */
} oracle_hp;

/* Eq. 1c: the synchronous data-parallel gradient is the mean of the K replica
 * gradients.  fp32: summed k = 0, 1, ..., K-1 in that order, then divided by K. */
void oracle_replica_mean(const float *const *g, int K, int64_t n, float *out)
{
    for (int64_t j = 0; j < n; ++j) {
        float s = g[0][j];
        for (int k = 1; k < K; ++k)
            s = s + g[k][j];
        out[j] = s / (float)K;
    }
}

/* Squared L2 norm |x|^2 (the quantity |G|^2 of Eq. 5 is the sum of these over
 * all tensors).  Each square is exact in fp64; the squares are added in order,
 * element 0 first, with Neumaier's compensated summation, so the result is the
 * exact sum to within about two fp64 roundings whatever n is.  (A per-tensor
 * scale or trust ratio rounds a ratio of these to fp32; an accurate sum keeps
 * that rounding a property of the data, not of the summation order.) */
double oracle_sqnorm(const float *x, int64_t n)
{
    double s = 0.0, c = 0.0;
    for (int64_t j = 0; j < n; ++j) {
        double v = (double)x[j];
        double t = v * v;
        double u = s + t;
        if (fabs(s) >= fabs(t))
            c = c + ((s - u) + t);
        else
            c = c + ((t - u) + s);
        s = u;
    }
    return s + c;
}

/* Eq. 5: Delta(G^(i)) = | (|G^(i)|^2 - |G^(i-1)|^2) / |G^(i-1)|^2 |.
 * Reading: with no previous step there is no |G^(i-1)|^2, so Delta = +inf
 * (sensitive).  A zero previous norm gives inf or NaN by IEEE division, and
 * neither is below any threshold. */
double oracle_grad_variability(double g2, double g2_prev, int64_t steps_done)
{
    if (steps_done == 0)
        return INFINITY;
    return fabs((g2 - g2_prev) / g2_prev);
}

/* Algorithm 1: the update is scaled when Delta < delta (strict), unscaled
 * (sensitive phase) otherwise; Sec. III-C, Eq. 8 uses the same test. */
int oracle_is_scaled(double delta_value, float delta, int force_branch)
{
    if (force_branch == OR_BRANCH_SCALED)
        return 1;
    if (force_branch == OR_BRANCH_UNSCALED)
        return 0;
    return delta_value < (double)delta;
}

/* LARS trust ratio ||w|| / ||g|| (Sec. V-B, prior art); 0 when ||g|| = 0. */
double oracle_trust_ratio(double sw, double sg)
{
    double nw = sqrt(sw), ng = sqrt(sg);
    return ng > 0.0 ? nw / ng : 0.0;
}

/* Per-tensor coefficient on the gradient.  AGS (Algorithm 1): gradscale[p]
 * when scaled, 1 otherwise.  STATIC (Eq. 8): U(s).  NONE: 1.  LARS: the trust
 * ratio times the trust coefficient, every step; 1 when either norm is 0. */
float oracle_coefficient(int rule, int scaled, float scale_p, float static_s,
                         float lars_trust, double sw, double sg)
{
    switch (rule) {
    case OR_RULE_AGS:
        return scaled ? scale_p : 1.0f;
    case OR_RULE_STATIC:
        return scaled ? static_s : 1.0f;
    case OR_RULE_LARS:
        if (sw > 0.0 && sg > 0.0)
            return (float)((double)lars_trust * (sqrt(sw) / sqrt(sg)));
        return 1.0f;
    default:
        return 1.0f;
    }
}

/* Eq. 7b with the wrapped SGD (momentum mu, weight decay wd, dampening 0):
 *   G~ = c * g                (c from Algorithm 1, per tensor or per element)
 *   d  = G~ + wd * w
 *   m  = mu * m + d           (zero-initialised m reproduces buf = d at step 1)
 *   w  = w - lr * m
 * Without a momentum buffer: w = w - lr * d, which with wd = 0 is the update
 * line of Algorithm 1 verbatim.  c_elem (per element) overrides c when given. */
void oracle_sgd_update(float *w, float *m, const float *gbar, int64_t n, float c,
                       const float *c_elem, float lr, float mu, float wd)
{
    for (int64_t j = 0; j < n; ++j) {
        float cj = c_elem ? c_elem[j] : c;
        float gt = cj * gbar[j];
        float d = gt + wd * w[j];
        if (m) {
            float mj = mu * m[j] + d;
            m[j] = mj;
            w[j] = w[j] - lr * mj;
        } else {
            w[j] = w[j] - lr * d;
        }
    }
}

/* UpdateGradScale of Algorithm 1, element-wise (the literal statement):
 *   s = min(|g_small / (g_large + eps)|, s_max).
 * fmin returns s_max when the quotient is NaN. */
void oracle_scale_elementwise(const float *gs, const float *gl, int64_t n, float eps,
                              float s_max, float *s_out)
{
    for (int64_t j = 0; j < n; ++j) {
        float den = gl[j] + eps;
        float q = gs[j] / den;
        s_out[j] = fminf(fabsf(q), s_max);
    }
}

/* UpdateGradScale per tensor (per-layer reading): the same rule on the
 * tensor norms, s = min(||g_small|| / (||g_large|| + eps), s_max), in fp64,
 * rounded once to fp32. */
float oracle_scale_tensor(double s_small, double s_large, float eps, float s_max)
{
    double q = sqrt(s_small) / (sqrt(s_large) + (double)eps);
    return (float)fmin(q, (double)s_max);
}

/* Steps 1-2 for tensor p: the norm of replica 0 (UpdateGradScale's small-batch gradient), the
 * mean written over replica 0, and the norms of the mean and of w. */
static void step_norms(float *const *w, float *const *g, const int64_t *numel, int n, int K, int p,
                       const float **gp, double *sg, double *ss, double *sw)
{
    ss[p] = oracle_sqnorm(g[p], numel[p]);
    for (int k = 0; k < K; ++k)
        gp[k] = g[(int64_t)k * n + p];
    oracle_replica_mean(gp, K, numel[p], g[p]);
    sg[p] = oracle_sqnorm(g[p], numel[p]);
    sw[p] = oracle_sqnorm(w[p], numel[p]);
}

/* Steps 4-5 for tensor p, once the branch is known: the coefficient, the update, the statistics
 * row and UpdateGradScale. */
static void step_update(float *const *w, float *const *m, float *const *g, const int64_t *numel,
                        int p, float lr, float mu, float wd, const oracle_hp *hp, float *scale,
                        float *const *scale_elem, int scaled, const double *sg, const double *ss,
                        const double *sw, double *stats)
{
    int per_elem = hp->rule == OR_RULE_AGS && hp->granularity == OR_GRAN_ELEMENT;
    float c = oracle_coefficient(hp->rule, scaled, scale ? scale[p] : 1.0f, hp->static_s,
                                 hp->lars_trust, sw[p], sg[p]);
    const float *ce = (per_elem && scaled) ? scale_elem[p] : NULL;
    oracle_sgd_update(w[p], hp->has_momentum ? m[p] : NULL, g[p], numel[p], c, ce, lr, mu, wd);
    if (per_elem)
        c = scaled ? NAN : 1.0f; /* no single coefficient: reported as NaN when scaled */
    float s_after = scale ? scale[p] : 0.0f;
    if (hp->refresh_scale && hp->granularity == OR_GRAN_TENSOR && scale) {
        s_after = oracle_scale_tensor(ss[p], sg[p], hp->eps, hp->s_max);
        scale[p] = s_after;
    }
    if (stats) {
        double *row = stats + (int64_t)p * OR_STATS_LEN;
        row[0] = sw[p];
        row[1] = sg[p];
        row[2] = ss[p];
        row[3] = sqrt(sw[p]);
        row[4] = sqrt(sg[p]);
        row[5] = oracle_trust_ratio(sw[p], sg[p]);
        row[6] = (double)c;
        row[7] = (double)s_after;
    }
}

/* The step; threads > 1 runs the per-tensor parts of steps 1-2 and 4-5 on that many threads
 * (OpenMP, when built with it).  Every tensor's arithmetic is the same whichever thread does
 * it, and step 3 adds the norms in tensor order on one thread, so the result does not depend
 * on the thread count. */
static int ags_step(float *const *w, float *const *m, float *const *g, const int64_t *numel, int n,
                    float lr, float mu, float wd, const oracle_hp *hp, float *scale,
                    float *const *scale_elem, double *state, double *stats, int threads)
{
    int K = hp->K;
    double *sg = calloc((size_t)n + 1, sizeof(double));
    double *ss = calloc((size_t)n + 1, sizeof(double));
    double *sw = calloc((size_t)n + 1, sizeof(double));
    if (!sg || !ss || !sw) {
        free(sg); free(ss); free(sw);
        return -1;
    }
    int failed = 0;

#pragma omp parallel for schedule(dynamic, 1) num_threads(threads > 0 ? threads : 1) reduction(|:failed)
    for (int p = 0; p < n; ++p) {
        const float **gp = malloc(sizeof(float *) * (size_t)(K > 0 ? K : 1));
        if (!gp) {
            failed = 1;
            continue;
        }
        step_norms(w, g, numel, n, K, p, gp, sg, ss, sw);
        free(gp);
    }
    if (failed) {
        free(sg); free(ss); free(sw);
        return -1;
    }

    /* step 3: |G|^2 in tensor order, Delta (Eq. 5), the branch (Algorithm 1) */
    double g2 = 0.0;
    for (int p = 0; p < n; ++p)
        g2 = g2 + sg[p];
    int64_t steps_done = (int64_t)state[1];
    double dv = oracle_grad_variability(g2, state[0], steps_done);
    int scaled = oracle_is_scaled(dv, hp->delta, hp->force_branch);

#pragma omp parallel for schedule(dynamic, 1) num_threads(threads > 0 ? threads : 1)
    for (int p = 0; p < n; ++p)
        step_update(w, m, g, numel, p, lr, mu, wd, hp, scale, scale_elem, scaled, sg, ss, sw,
                    stats);

    state[0] = g2;
    state[1] = (double)(steps_done + 1);
    state[2] = dv;
    state[3] = (double)scaled;

    free(sg); free(ss); free(sw);
    return 0;
}

/* One full optimizer step over n tensors, in the paper's order:
 *   1. mean of the K replicas (Eq. 1c), written over replica 0 when K > 1;
 *      |g_0|^2 is taken before it is overwritten
 *   2. per-tensor squared norms of the mean and of w (pre-update)
 *   3. |G|^2 = sum over tensors (ascending), Delta (Eq. 5), branch (Alg. 1)
 *   4. per-tensor coefficient, then the scaled momentum-SGD update
 *   5. statistics, state, and (optionally) UpdateGradScale from replica 0
 *
 * w[p], m[p] (NULL when hp->has_momentum is 0): fp32 tensors, updated in place.
 * g[k * n + p]: replica k of tensor p.  scale[p]: gradscale (per tensor).
 * scale_elem[p]: gradscale per element (granularity ELEMENT).
 * state[4]: |G^(i-1)|^2, steps done, last Delta, last branch (1 = scaled).
 * stats[p * 8 + c], optional: |w|^2, |gbar|^2, |g_0|^2, |w|, |gbar|,
 *   |w|/|gbar|, coefficient applied, gradscale after the step. */
int oracle_ags_step(float *const *w, float *const *m, float *const *g, const int64_t *numel,
                    int n, float lr, float mu, float wd, const oracle_hp *hp, float *scale,
                    float *const *scale_elem, double *state, double *stats)
{
    return ags_step(w, m, g, numel, n, lr, mu, wd, hp, scale, scale_elem, state, stats, 1);
}

/* The same step with its per-tensor parts on `threads` threads (the CPU baseline on all host
 * cores); bitwise equal to oracle_ags_step. */
int oracle_ags_step_threads(float *const *w, float *const *m, float *const *g, const int64_t *numel,
                            int n, float lr, float mu, float wd, const oracle_hp *hp, float *scale,
                            float *const *scale_elem, double *state, double *stats, int threads)
{
    return ags_step(w, m, g, numel, n, lr, mu, wd, hp, scale, scale_elem, state, stats, threads);
}

/* The number of threads oracle_ags_step_threads can use (1 when built without OpenMP). */
int oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Per-layer statistics without an update: the mean of the K replicas is formed
 * in a scratch buffer (replica buffers are not modified).  Row layout as in
 * oracle_ags_step; columns 6 and 7 are 0. */
int oracle_layer_stats(const float *const *w, const float *const *g, int K, const int64_t *numel,
                       int n, double *stats)
{
    const float **gp = malloc(sizeof(float *) * (size_t)K);
    if (!gp)
        return -1;
    for (int p = 0; p < n; ++p) {
        float *tmp = malloc(sizeof(float) * (size_t)(numel[p] > 0 ? numel[p] : 1));
        if (!tmp) {
            free(gp);
            return -1;
        }
        for (int k = 0; k < K; ++k)
            gp[k] = g[(int64_t)k * n + p];
        oracle_replica_mean(gp, K, numel[p], tmp);
        double sw = oracle_sqnorm(w[p], numel[p]);
        double sg = oracle_sqnorm(tmp, numel[p]);
        double ss = oracle_sqnorm(g[p], numel[p]);
        double *row = stats + (int64_t)p * OR_STATS_LEN;
        row[0] = sw;
        row[1] = sg;
        row[2] = ss;
        row[3] = sqrt(sw);
        row[4] = sqrt(sg);
        row[5] = oracle_trust_ratio(sw, sg);
        row[6] = 0.0;
        row[7] = 0.0;
        free(tmp);
    }
    free(gp);
    return 0;
}

/* UpdateGradScale over n tensors with explicit small- and large-batch
 * gradients: per tensor (scale[p]) or per element (scale_elem[p][j]). */
int oracle_update_scale(const float *const *gs, const float *const *gl, const int64_t *numel,
                        int n, float eps, float s_max, int granularity, float *scale,
                        float *const *scale_elem)
{
    for (int p = 0; p < n; ++p) {
        if (granularity == OR_GRAN_ELEMENT)
            oracle_scale_elementwise(gs[p], gl[p], numel[p], eps, s_max, scale_elem[p]);
        else
            scale[p] = oracle_scale_tensor(oracle_sqnorm(gs[p], numel[p]),
                                           oracle_sqnorm(gl[p], numel[p]), eps, s_max);
    }
    return 0;
}
