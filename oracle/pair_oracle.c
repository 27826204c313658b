/*
 * fp64 CPU oracle for the Pair estimator: TEST INFRASTRUCTURE ONLY.
 *
 * Only tests, the smoke check and the benchmark's CPU-baseline leg use this
 * file. The CUDA library shares no code with it. Everything here is written
 * straight from the paper's definitions, in double precision, with plain
 * loops and no blocking or reordering:
 *
 *   Sec. 3.2, Eq. (pair-kernel): h_ij = 1/2 (r_i - r_j)(s_i - s_j).
 *   Sec. 3.3: J_i completion indicators, rho_ij = P(J_i = J_j = 1) > 0.
 *   Sec. 4.5, Eq. (pair-ht): g = (1/M) sum_{i<j} J_i J_j h_ij / rho_ij.
 *   Sec. 4.5, Eq. (pair-advantage): A_i = 1/(2M) sum_{j != i} J_i J_j
 *                                          (r_i - r_j) / rho_ij.
 *   Algorithm 1, pair-corrected update: every observed edge (i, j)
 *     contributes to the coefficients of both endpoints.
 *   App. C, numerical stability: optional centring of the coefficients over
 *     the observed endpoints.
 *
 * The normalisation 1/M is passed in as `scale` (scale = 1/M gives the
 * paper's A_i; scale = 1 gives the plain completed-edge sum).
 * rho is read only at i < j (rho_ij = rho_ji by definition).
 */
#include <math.h>
#include <pthread.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>

#define ORACLE_OK 0
#define ORACLE_ERR_NONPOSITIVE_INCLUSION 1
#define ORACLE_ERR_FORMS_DISAGREE 2
#define ORACLE_ERR_ALLOC 3

static double rho_at(const double *rho_g, int G, int i, int j)
{
    int lo = i < j ? i : j, hi = i < j ? j : i;
    return rho_g[(size_t)lo * G + hi];
}

/* One group. Returns an ORACLE_* code. */
static int coeffs_group(int G, const double *r, const uint8_t *J,
                        const double *rho_g, double scale, int center,
                        double *a, double *a_mag, uint8_t *active,
                        int32_t *edges, int32_t *contrast)
{
    double *a_edge = (double *)calloc((size_t)G, sizeof(double));
    if (!a_edge) return ORACLE_ERR_ALLOC;
    int n_edges = 0, n_contrast = 0, err = ORACLE_OK;

    /* Edge-sum form (Algorithm 1): enumerate each observed edge i < j once
     * and add its contribution to both endpoints. */
    for (int i = 0; i < G; ++i) {
        for (int j = i + 1; j < G; ++j) {
            if (!(J[i] && J[j])) continue;
            double rij = rho_g[(size_t)i * G + j];
            if (!(rij > 0.0)) { err = ORACLE_ERR_NONPOSITIVE_INCLUSION; continue; }
            ++n_edges;
            if (r[i] != r[j]) ++n_contrast;
            double t = (r[i] - r[j]) / rij;
            a_edge[i] += 0.5 * t;
            a_edge[j] -= 0.5 * t;
        }
    }

    /* Direct row form (Eq. pair-advantage without 1/M): for every vertex sum
     * over its partners. Must agree with the edge-sum form. */
    for (int i = 0; i < G; ++i) {
        double s = 0.0, mag = 0.0;
        int has_contrast = 0;
        for (int j = 0; j < G; ++j) {
            if (j == i || !(J[i] && J[j])) continue;
            double rij = rho_at(rho_g, G, i, j);
            if (!(rij > 0.0)) continue;
            double t = (r[i] - r[j]) / rij;
            s += t;
            mag += fabs(t);
            if (r[i] != r[j]) has_contrast = 1;
        }
        s *= 0.5;
        mag *= 0.5;
        double diff = fabs(s - a_edge[i]);
        if (diff > 1e-13 * mag + 1e-300) err = err ? err : ORACLE_ERR_FORMS_DISAGREE;
        a[i] = s;
        a_mag[i] = mag;
        active[i] = (uint8_t)(J[i] && has_contrast);
    }

    if (center) {
        /* App. C: centre across the observed endpoints (J_i = 1). */
        int K = 0;
        double sum = 0.0;
        for (int i = 0; i < G; ++i) if (J[i]) { ++K; sum += a[i]; }
        if (K > 0) {
            double mean = sum / K;
            for (int i = 0; i < G; ++i) if (J[i]) a[i] -= mean;
        }
    }
    for (int i = 0; i < G; ++i) {
        a[i] *= scale;
        a_mag[i] *= fabs(scale);
    }
    *edges = n_edges;
    *contrast = n_contrast;
    free(a_edge);
    return err;
}

/*
 * Edge weights of the estimator variants (App. "Estimated and stabilized
 * propensities" and the ablation table of Sec. 5): for a completed edge e =
 * (i, j) the coefficient term is 1/2 (r_i - r_j) w_e with
 *   ORACLE_W_HT          w_e = 1 / rho_ij                (Eq. pair-ht)
 *   ORACLE_W_UNWEIGHTED  w_e = 1                         (no pair correction)
 *   ORACLE_W_MARGINAL    w_e = 1 / (pi_i pi_j), pi_i = rho_ii (marginal-only)
 *   ORACLE_W_CLIPPED     w_e = min(1 / rho_ij, w_max)
 *   ORACLE_W_HAJEK       w_e = 1 / rho_ij, and the group's coefficients are
 *                        divided by sum_e w_e (self-normalised ratio form)
 * Diagnostics per group over its completed edges: ESS = (sum w)^2 / sum w^2
 * (Sec. 5 metrics) and the largest weight; both 0 without completed edges.
 * `center` holds flags: bit 0 centres over the completed vertices (App. C),
 * bit 1 divides by the completed rewards' sample standard deviation.
 */
#define ORACLE_W_HT 0
#define ORACLE_W_UNWEIGHTED 1
#define ORACLE_W_MARGINAL 2
#define ORACLE_W_CLIPPED 3
#define ORACLE_W_HAJEK 4

/* One group, weighting variant `wmode`. Returns an ORACLE_* code. */
static int coeffs_group_w(int G, const double *r, const uint8_t *J,
                          const double *rho_g, double scale, int center,
                          int wmode, double w_max, double *a, double *a_mag,
                          uint8_t *active, int32_t *edges, int32_t *contrast,
                          double *ess, double *max_w)
{
    int n_edges = 0, n_contrast = 0, err = ORACLE_OK;
    double sum_w = 0.0, sum_w2 = 0.0, mw = 0.0;
    for (int i = 0; i < G; ++i) { a[i] = 0.0; a_mag[i] = 0.0; active[i] = 0; }
    /* Every completed edge i < j once; its term goes to both endpoints. */
    for (int i = 0; i < G; ++i) {
        for (int j = i + 1; j < G; ++j) {
            if (!(J[i] && J[j])) continue;
            double w;
            if (wmode == ORACLE_W_UNWEIGHTED) {
                w = 1.0;
            } else if (wmode == ORACLE_W_MARGINAL) {
                double pi = rho_g[(size_t)i * G + i], pj = rho_g[(size_t)j * G + j];
                if (!(pi > 0.0) || !(pj > 0.0)) { err = ORACLE_ERR_NONPOSITIVE_INCLUSION; continue; }
                w = 1.0 / (pi * pj);
            } else {
                double rij = rho_g[(size_t)i * G + j];
                if (!(rij > 0.0)) { err = ORACLE_ERR_NONPOSITIVE_INCLUSION; continue; }
                w = 1.0 / rij;
                if (wmode == ORACLE_W_CLIPPED && w > w_max) w = w_max;
            }
            ++n_edges;
            if (r[i] != r[j]) {
                ++n_contrast;
                active[i] = 1;
                active[j] = 1;
            }
            double t = 0.5 * (r[i] - r[j]) * w;
            a[i] += t;
            a[j] -= t;
            a_mag[i] += fabs(t);
            a_mag[j] += fabs(t);
            sum_w += w;
            sum_w2 += w * w;
            if (w > mw) mw = w;
        }
    }
    if (wmode == ORACLE_W_HAJEK) {
        for (int i = 0; i < G; ++i) {
            a[i] = sum_w > 0.0 ? a[i] / sum_w : 0.0;
            a_mag[i] = sum_w > 0.0 ? a_mag[i] / sum_w : 0.0;
        }
    }
    if (center & 2) {
        /* Reward standardisation (App. "Practical departures"): divide by the
         * sample standard deviation (n - 1) of the completed rewards; a group
         * with fewer than two completed vertices or equal rewards has no
         * contrast edge, so its coefficients are already 0 and stay 0. */
        int K = 0;
        double mean = 0.0;
        for (int i = 0; i < G; ++i) if (J[i]) { ++K; mean += r[i]; }
        if (K >= 2) {
            mean /= K;
            double ss = 0.0;
            for (int i = 0; i < G; ++i) if (J[i]) ss += (r[i] - mean) * (r[i] - mean);
            double sd = sqrt(ss / (K - 1));
            for (int i = 0; i < G; ++i) {
                a[i] = sd > 0.0 ? a[i] / sd : 0.0;
                a_mag[i] = sd > 0.0 ? a_mag[i] / sd : 0.0;
            }
        }
    }
    if (center & 1) {
        int K = 0;
        double sum = 0.0;
        for (int i = 0; i < G; ++i) if (J[i]) { ++K; sum += a[i]; }
        if (K > 0) {
            double mean = sum / K;
            for (int i = 0; i < G; ++i) if (J[i]) a[i] -= mean;
        }
    }
    for (int i = 0; i < G; ++i) {
        a[i] *= scale;
        a_mag[i] *= fabs(scale);
    }
    *edges = n_edges;
    *contrast = n_contrast;
    *ess = sum_w2 > 0.0 ? sum_w * sum_w / sum_w2 : 0.0;
    *max_w = mw;
    return err;
}

typedef struct {
    int B, G, D, center, nthreads, tid;
    const double *r, *rho;
    const uint8_t *J;
    const float *S32;
    const double *S64;
    double scale;
    double *a, *a_mag, *g;
    uint8_t *active;
    int32_t *edges, *contrast;
    int wmode;
    double w_max;
    const double *p;       /* product design: marginals [B][G] */
    double *ess, *max_w;
    int err;
} job_t;

static void *coeffs_worker(void *p)
{
    job_t *jb = (job_t *)p;
    int G = jb->G;
    for (int b = jb->tid; b < jb->B; b += jb->nthreads) {
        size_t o = (size_t)b * G;
        int e = coeffs_group(G, jb->r + o, jb->J + o, jb->rho + o * G,
                             jb->scale, jb->center, jb->a + o, jb->a_mag + o,
                             jb->active + o, jb->edges + b, jb->contrast + b);
        if (e && !jb->err) jb->err = e;
    }
    return NULL;
}

static void *coeffs_w_worker(void *p)
{
    job_t *jb = (job_t *)p;
    int G = jb->G;
    double *rho_tmp = NULL;
    if (jb->p) {
        rho_tmp = (double *)malloc(sizeof(double) * (size_t)G * G);
        if (!rho_tmp) { jb->err = ORACLE_ERR_ALLOC; return NULL; }
    }
    for (int b = jb->tid; b < jb->B; b += jb->nthreads) {
        size_t o = (size_t)b * G;
        const double *rho_g;
        if (jb->p) {
            /* Independent Bernoulli design: rho_ij = p_i p_j (Sec. 4, the
             * product design), rho_ii = p_i. */
            for (int i = 0; i < G; ++i)
                for (int j = 0; j < G; ++j)
                    rho_tmp[(size_t)i * G + j] = i == j ? jb->p[o + i] : jb->p[o + i] * jb->p[o + j];
            rho_g = rho_tmp;
        } else {
            rho_g = jb->rho + o * G;
        }
        int e = coeffs_group_w(G, jb->r + o, jb->J + o, rho_g, jb->scale, jb->center,
                               jb->wmode, jb->w_max, jb->a + o, jb->a_mag + o,
                               jb->active + o, jb->edges + b, jb->contrast + b,
                               jb->ess + b, jb->max_w + b);
        if (e && !jb->err) jb->err = e;
    }
    free(rho_tmp);
    return NULL;
}

static double s_at(const job_t *jb, size_t idx)
{
    return jb->S64 ? jb->S64[idx] : (double)jb->S32[idx];
}

/* Dense estimator by explicit enumeration of the observed edges with the
 * pair kernel formed for every coordinate (Eq. pair-ht). */
static void *dense_worker(void *p)
{
    job_t *jb = (job_t *)p;
    int G = jb->G, D = jb->D;
    for (int b = jb->tid; b < jb->B; b += jb->nthreads) {
        const double *r = jb->r + (size_t)b * G;
        const uint8_t *J = jb->J + (size_t)b * G;
        const double *rho = jb->rho + (size_t)b * G * G;
        double *g = jb->g + (size_t)b * D;
        for (int k = 0; k < D; ++k) g[k] = 0.0;
        for (int i = 0; i < G; ++i) {
            for (int j = i + 1; j < G; ++j) {
                if (!(J[i] && J[j])) continue;
                double rij = rho[(size_t)i * G + j];
                if (!(rij > 0.0)) { jb->err = ORACLE_ERR_NONPOSITIVE_INCLUSION; continue; }
                size_t si = ((size_t)b * G + i) * D, sj = ((size_t)b * G + j) * D;
                for (int k = 0; k < D; ++k) {
                    double h = 0.5 * (r[i] - r[j]) * (s_at(jb, si + k) - s_at(jb, sj + k));
                    g[k] += h / rij;
                }
            }
        }
        for (int k = 0; k < D; ++k) g[k] *= jb->scale;
    }
    return NULL;
}

static int run_jobs(job_t *base, int nthreads, void *(*fn)(void *))
{
    if (nthreads < 1) nthreads = 1;
    job_t *jobs = (job_t *)malloc(sizeof(job_t) * (size_t)nthreads);
    pthread_t *th = (pthread_t *)malloc(sizeof(pthread_t) * (size_t)nthreads);
    if (!jobs || !th) { free(jobs); free(th); return ORACLE_ERR_ALLOC; }
    for (int t = 0; t < nthreads; ++t) {
        jobs[t] = *base;
        jobs[t].tid = t;
        jobs[t].nthreads = nthreads;
        jobs[t].err = 0;
        pthread_create(&th[t], NULL, fn, &jobs[t]);
    }
    int err = 0;
    for (int t = 0; t < nthreads; ++t) {
        pthread_join(th[t], NULL);
        if (jobs[t].err && !err) err = jobs[t].err;
    }
    free(jobs);
    free(th);
    return err;
}

/*
 * Per-rollout coefficients a[B][G] (scale * 1/2 sum_{j != i} J_i J_j
 * (r_i - r_j)/rho_ij), their magnitudes a_mag (same sum over |terms|, used
 * for error bounds), the active mask (J_i = 1 and some completed partner
 * with a different reward), observed edge counts and contrast edge counts.
 */
int oracle_pair_coeffs(int B, int G, const double *r, const uint8_t *J,
                       const double *rho, double scale, int center,
                       double *a, double *a_mag, uint8_t *active,
                       int32_t *edges, int32_t *contrast, int nthreads)
{
    job_t jb = {0};
    jb.B = B; jb.G = G; jb.center = center; jb.r = r; jb.J = J; jb.rho = rho;
    jb.scale = scale; jb.a = a; jb.a_mag = a_mag; jb.active = active;
    jb.edges = edges; jb.contrast = contrast;
    return run_jobs(&jb, nthreads, coeffs_worker);
}

/*
 * Dense estimator g[B][D] = scale * sum_{i<j} J_i J_j h_ij / rho_ij with
 * h_ij formed explicitly per coordinate. Scores come from exactly one of
 * S32 (float, upcast exactly) or S64, both laid out [B][G][D].
 */
int oracle_pair_estimate_dense(int B, int G, int D, const double *r,
                               const uint8_t *J, const double *rho,
                               const float *S32, const double *S64,
                               double scale, double *g, int nthreads)
{
    job_t jb = {0};
    jb.B = B; jb.G = G; jb.D = D; jb.r = r; jb.J = J; jb.rho = rho;
    jb.S32 = S32; jb.S64 = S64; jb.scale = scale; jb.g = g;
    return run_jobs(&jb, nthreads, dense_worker);
}

/*
 * Coefficients under a weighting variant (ORACLE_W_*, see coeffs_group_w),
 * with the per-group ESS and largest weight of the completed edges.
 */
int oracle_pair_coeffs_w(int B, int G, const double *r, const uint8_t *J,
                         const double *rho, double scale, int center, int wmode,
                         double w_max, double *a, double *a_mag, uint8_t *active,
                         int32_t *edges, int32_t *contrast, double *ess,
                         double *max_w, int nthreads)
{
    job_t jb = {0};
    jb.B = B; jb.G = G; jb.center = center; jb.r = r; jb.J = J; jb.rho = rho;
    jb.scale = scale; jb.a = a; jb.a_mag = a_mag; jb.active = active;
    jb.edges = edges; jb.contrast = contrast; jb.wmode = wmode; jb.w_max = w_max;
    jb.ess = ess; jb.max_w = max_w;
    return run_jobs(&jb, nthreads, coeffs_w_worker);
}

/*
 * Inverse-probability coefficients of the independent (product) design:
 * rho_ij = p_i p_j, i.e. ORACLE_W_HT on the joint probabilities formed from
 * the marginals p[B][G].
 */
int oracle_pair_coeffs_product(int B, int G, const double *r, const uint8_t *J,
                               const double *p, double scale, int center,
                               double *a, double *a_mag, uint8_t *active,
                               int32_t *edges, int32_t *contrast, double *ess,
                               double *max_w, int nthreads)
{
    job_t jb = {0};
    jb.B = B; jb.G = G; jb.center = center; jb.r = r; jb.J = J; jb.p = p;
    jb.scale = scale; jb.a = a; jb.a_mag = a_mag; jb.active = active;
    jb.edges = edges; jb.contrast = contrast; jb.wmode = ORACLE_W_HT;
    jb.ess = ess; jb.max_w = max_w;
    return run_jobs(&jb, nthreads, coeffs_w_worker);
}
