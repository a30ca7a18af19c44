/*
 * GNMR oracle: a plain, slow, double-precision CPU restatement of the GNMR
 * per-step monitor (GNMR: Runtime Stability Control for Low-Precision LLM
 * Training).
 *
 * TEST INFRASTRUCTURE ONLY.  The tests, the smoke check and the benchmark's
 * CPU baseline may load this file's library; the product (the CUDA path in
 * the package) never does, and shares no code, header or table with it.
 *
 * What it computes, in the paper's order and notation:
 *   - n_{b,t} = ||g_{b,t}||_2 for every monitored unit b      (Sec. 2, Eq. local_gradient)
 *   - Algorithm 1: GNMR_{b,t}, Delta-GNMR_{b,t}, A_{b,t}, Q_b   (Sec. 3.1-3.2, Alg. 1)
 *   - Algorithm 2: R_{b,t}, C_t, A_t = Top_maxO(C_t; R), Lock_b (Sec. 3.3, Alg. 2)
 *
 * Readings taken where the paper is silent (each one is listed with its
 * reason in the design notes):
 *   - "t = 1" in Algorithm 1 is read per unit: k_b, the number of steps at
 *     which unit b was observed, plays the role of t (equal to the global t
 *     whenever every step is observed).
 *   - A non-finite norm (NaN or Inf) gives GNMR = Delta-GNMR = R = +Inf and
 *     leaves A_b, Q_b and k_b untouched.
 *   - mean(Q_b) + eps == 0 gives Delta-GNMR = +Inf if GNMR > 0, else 1.
 *   - Top_maxO orders by R descending, then by unit index ascending, and
 *     selects min(maxO, |C_t|) units.
 *   - alpha_t, beta_t: the *_init values for t <= warmup_steps, the *_main
 *     values after, unless the caller overrides them for the step.
 *
 *   - The recovery actuator's fake quantization (App. E.2, the low-cost
 *     activation path of the stress bench in Sec. 5.1): per token row, scale
 *     into the format's range, round to the nearest representable value,
 *     rescale.  The paper fixes no precision for this arithmetic; the reading
 *     taken is fp32 throughout (inv = fmax / amax, v = x * inv, y = q * (amax /
 *     fmax)), ties to the even code, saturation at fmax, rows whose max is 0
 *     or that hold a NaN or Inf left unchanged, and so are rows whose scale
 *     factor fmax / amax overflows fp32 (amax below fmax / FLT_MAX).
 *
 * Build: gcc -O2 -std=c11 -ffp-contract=off -shared -fPIC -o liboracle_gnmr.so
 * gnmr_oracle.c -lm (no fast-math, no fused multiply-add: every operation
 * below rounds as written).
 */
#include <float.h>
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_DTYPE_F32 0
#define ORACLE_DTYPE_BF16 1

/* A bfloat16 value is the upper 16 bits of an IEEE-754 binary32 value, so
 * shifting it into place gives the exact binary32 (and then binary64) value. */
static double bf16_to_double(uint16_t h)
{
    uint32_t bits = ((uint32_t)h) << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

/* Eq. local_gradient: n_b = ||g_b||_2, the square root of the sum of squares
 * of every element of unit b's segment, summed sequentially in double. */
int oracle_unit_norms(const void *arena, int dtype, const int64_t *offsets,
                      const int64_t *lengths, int32_t num_units, double *norms)
{
    if (dtype != ORACLE_DTYPE_F32 && dtype != ORACLE_DTYPE_BF16)
        return 1;
    for (int32_t b = 0; b < num_units; ++b) {
        double sum = 0.0;
        if (dtype == ORACLE_DTYPE_F32) {
            const float *g = (const float *)arena + offsets[b];
            for (int64_t i = 0; i < lengths[b]; ++i) {
                double x = (double)g[i];
                sum += x * x;
            }
        } else {
            const uint16_t *g = (const uint16_t *)arena + offsets[b];
            for (int64_t i = 0; i < lengths[b]; ++i) {
                double x = bf16_to_double(g[i]);
                sum += x * x;
            }
        }
        norms[b] = sqrt(sum);
    }
    return 0;
}

/* Eq. local_gradient for units made of several segments (Sec. 3.4: a whole
 * transformer block as one unit): n_b = sqrt of the sum of squares over
 * every element of every segment of b, one running sum per unit, segments in
 * the order given.  A unit with no segment has n_b = 0. */
int oracle_unit_norms_segmented(const void *arena, int dtype, const int64_t *offsets,
                                const int64_t *lengths, const int32_t *segment_unit,
                                int64_t num_segments, int32_t num_units, double *norms)
{
    if (dtype != ORACLE_DTYPE_F32 && dtype != ORACLE_DTYPE_BF16)
        return 1;
    for (int32_t b = 0; b < num_units; ++b)
        norms[b] = 0.0;                      /* running sums of squares */
    for (int64_t g = 0; g < num_segments; ++g) {
        const int32_t b = segment_unit[g];
        if (b < 0 || b >= num_units)
            return 2;
        double sum = norms[b];
        if (dtype == ORACLE_DTYPE_F32) {
            const float *x = (const float *)arena + offsets[g];
            for (int64_t i = 0; i < lengths[g]; ++i) {
                double v = (double)x[i];
                sum += v * v;
            }
        } else {
            const uint16_t *x = (const uint16_t *)arena + offsets[g];
            for (int64_t i = 0; i < lengths[g]; ++i) {
                double v = bf16_to_double(x[i]);
                sum += v * v;
            }
        }
        norms[b] = sum;
    }
    for (int32_t b = 0; b < num_units; ++b)
        norms[b] = sqrt(norms[b]);
    return 0;
}

/* Per-unit controller state: A_b (historical mean), Q_b (the last <= delta
 * GNMR values, oldest first), k_b (observation count), Lock_b. */
typedef struct {
    int32_t num_units;
    int32_t window;      /* delta */
    int32_t max_o;       /* maxO */
    int32_t lock_len;    /* T_lock */
    int64_t warmup_steps;
    double alpha_init, alpha_main, beta_init, beta_main, eps;
    int64_t t;           /* completed steps */
    uint8_t *recoverable;
    double *A;
    int64_t *k;
    double *Q;           /* num_units * window, oldest first */
    int32_t *qlen;
    int32_t *lock;
    int32_t *cand;       /* scratch for Algorithm 2 */
    /* policy variants (see oracle_ctl_set_policy) */
    int32_t policy;
    int64_t forced_steps;
    int64_t static_warmup;
    double static_fraction;
    uint8_t *active;     /* A_{t-1}: on the recovery path at the previous step */
    double *gsum;        /* sum of GNMR over the static policy's warm-up */
} oracle_ctl;

#define ORACLE_POLICY_ACTIVE_CAP 0
#define ORACLE_POLICY_ADMISSION_CAP 1
#define ORACLE_POLICY_STATIC_TOP 2

void oracle_ctl_destroy(oracle_ctl *c)
{
    if (!c)
        return;
    free(c->recoverable);
    free(c->A);
    free(c->k);
    free(c->Q);
    free(c->qlen);
    free(c->lock);
    free(c->cand);
    free(c->active);
    free(c->gsum);
    free(c);
}

oracle_ctl *oracle_ctl_create(int32_t num_units, int32_t window, int32_t max_o,
                              int32_t lock_len, int64_t warmup_steps,
                              double alpha_init, double alpha_main,
                              double beta_init, double beta_main, double eps,
                              const uint8_t *recoverable)
{
    if (num_units < 1 || window < 1 || max_o < 0 || lock_len < 0)
        return NULL;
    oracle_ctl *c = (oracle_ctl *)calloc(1, sizeof *c);
    if (!c)
        return NULL;
    c->num_units = num_units;
    c->window = window;
    c->max_o = max_o;
    c->lock_len = lock_len;
    c->warmup_steps = warmup_steps;
    c->alpha_init = alpha_init;
    c->alpha_main = alpha_main;
    c->beta_init = beta_init;
    c->beta_main = beta_main;
    c->eps = eps;
    size_t u = (size_t)num_units;
    c->recoverable = (uint8_t *)calloc(u, 1);
    c->A = (double *)calloc(u, sizeof(double));
    c->k = (int64_t *)calloc(u, sizeof(int64_t));
    c->Q = (double *)calloc(u * (size_t)window, sizeof(double));
    c->qlen = (int32_t *)calloc(u, sizeof(int32_t));
    c->lock = (int32_t *)calloc(u, sizeof(int32_t));
    c->cand = (int32_t *)calloc(u, sizeof(int32_t));
    c->active = (uint8_t *)calloc(u, 1);
    c->gsum = (double *)calloc(u, sizeof(double));
    c->static_fraction = 0.25;
    if (!c->recoverable || !c->A || !c->k || !c->Q || !c->qlen || !c->lock || !c->cand ||
        !c->active || !c->gsum) {
        oracle_ctl_destroy(c);
        return NULL;
    }
    for (size_t b = 0; b < u; ++b)
        c->recoverable[b] = recoverable ? (recoverable[b] != 0) : 1;
    return c;
}

/* Policy variants (readings of passages the paper states loosely):
 *   ORACLE_POLICY_ACTIVE_CAP (0, Algorithm 2): |A_t| <= maxO.
 *   ORACLE_POLICY_ADMISSION_CAP (1, the Remark on the maxO budget): only newly
 *     admitted units are capped.  Candidates that were active at t-1 stay
 *     active; of the other candidates the maxO with the largest R (ties by
 *     index) are admitted.  |A_t| may exceed maxO.
 *   ORACLE_POLICY_STATIC_TOP (2, the ADAPT-style baseline of App. E.4): for
 *     t <= static_warmup every recoverable unit is on the recovery path and
 *     GNMR is summed per unit; at t = static_warmup + 1 the
 *     ceil(static_fraction * |B_rec|) recoverable units with the largest sum
 *     (ties by index) are fixed on the recovery path for good.
 * forced_steps (App. E.7): for t <= forced_steps every recoverable unit is on
 * the recovery path (statistics still update, locks stay as they are). */
int oracle_ctl_set_policy(oracle_ctl *c, int32_t policy, int64_t forced_steps,
                          int64_t static_warmup, double static_fraction)
{
    if (policy < 0 || policy > 2 || forced_steps < 0 || static_warmup < 0 ||
        !(static_fraction >= 0.0 && static_fraction <= 1.0))
        return 1;
    c->policy = policy;
    c->forced_steps = forced_steps;
    c->static_warmup = static_warmup;
    c->static_fraction = static_fraction;
    return 0;
}

/* Algorithm 1 for one unit: returns GNMR and Delta-GNMR through g and d, and
 * updates A_b, k_b and Q_b. */
static void algorithm1(oracle_ctl *c, int32_t b, double n, double *g, double *d)
{
    double *Qb = c->Q + (size_t)b * (size_t)c->window;
    double gnmr, dgnmr;

    if (!isfinite(n)) {           /* reading: non-finite norm, no state update */
        *g = INFINITY;
        *d = INFINITY;
        return;
    }
    /* GNMR: 1 at the unit's first step or while the historical mean is 0. */
    if (c->k[b] == 0 || c->A[b] == 0.0)
        gnmr = 1.0;
    else
        gnmr = n / (c->A[b] + c->eps);

    /* Delta-GNMR: GNMR over the mean of the last delta GNMR values, once the
     * queue holds delta values; 1 before that. */
    if (c->qlen[b] == c->window) {
        double s = 0.0;
        for (int32_t i = 0; i < c->window; ++i)
            s += Qb[i];
        double denom = s / (double)c->window + c->eps;
        if (denom == 0.0)
            dgnmr = (gnmr > 0.0) ? INFINITY : 1.0;
        else
            dgnmr = gnmr / denom;
    } else {
        dgnmr = 1.0;
    }

    /* Incremental mean A_{b,t} = A_{b,t-1} + (n - A_{b,t-1}) / t. */
    c->k[b] += 1;
    c->A[b] = c->A[b] + (n - c->A[b]) / (double)c->k[b];

    /* Push GNMR into Q_b, keeping only the most recent delta values. */
    if (c->qlen[b] == c->window) {
        for (int32_t i = 0; i + 1 < c->window; ++i)
            Qb[i] = Qb[i + 1];
        Qb[c->window - 1] = gnmr;
    } else {
        Qb[c->qlen[b]] = gnmr;
        c->qlen[b] += 1;
    }
    *g = gnmr;
    *d = dgnmr;
}

/* qsort has no user pointer: the comparator reads R through this
 * thread-local variable. */
static _Thread_local const double *g_sort_r;

static int by_risk_then_index(const void *pa, const void *pb)
{
    int32_t a = *(const int32_t *)pa, b = *(const int32_t *)pb;
    double ra = g_sort_r[a], rb = g_sort_r[b];
    if (ra > rb)
        return -1;
    if (ra < rb)
        return 1;
    return (a < b) ? -1 : (a > b);
}

/* One training step: Algorithm 1 for every monitored unit, then Algorithm 2.
 * alpha_override / beta_override: NaN selects the two-stage schedule.
 * Outputs (each num_units long): gnmr, dgnmr, risk, mask (1 = recovery
 * path), lock_out (Lock_b after the step).  counts[0] = |C_t|,
 * counts[1] = |A_t|. */
int oracle_ctl_step(oracle_ctl *c, const double *norms, double alpha_override,
                    double beta_override, double *gnmr, double *dgnmr,
                    double *risk, uint8_t *mask, int32_t *lock_out,
                    int32_t *counts)
{
    int32_t U = c->num_units;

    for (int32_t b = 0; b < U; ++b)
        algorithm1(c, b, norms[b], &gnmr[b], &dgnmr[b]);

    c->t += 1;
    double alpha = isnan(alpha_override)
                       ? (c->t <= c->warmup_steps ? c->alpha_init : c->alpha_main)
                       : alpha_override;
    double beta = isnan(beta_override)
                      ? (c->t <= c->warmup_steps ? c->beta_init : c->beta_main)
                      : beta_override;

    /* R_{b,t} = max{GNMR / alpha_t, Delta-GNMR / beta_t}. */
    for (int32_t b = 0; b < U; ++b) {
        double x = gnmr[b] / alpha, y = dgnmr[b] / beta;
        risk[b] = (x > y) ? x : y;
    }

    int32_t nrec = 0;
    for (int32_t b = 0; b < U; ++b)
        nrec += c->recoverable[b];

    if (c->policy == ORACLE_POLICY_STATIC_TOP && c->t <= c->static_warmup)
        for (int32_t b = 0; b < U; ++b)
            if (c->recoverable[b])
                c->gsum[b] += gnmr[b];

    /* Every recoverable unit on the recovery path: forced warm-up, or the
     * static policy's warm-up. */
    if (c->t <= c->forced_steps ||
        (c->policy == ORACLE_POLICY_STATIC_TOP && c->t <= c->static_warmup)) {
        for (int32_t b = 0; b < U; ++b) {
            mask[b] = c->recoverable[b];
            c->active[b] = c->recoverable[b];
            lock_out[b] = c->lock[b];
        }
        counts[0] = 0;
        counts[1] = nrec;
        return 0;
    }

    /* Static policy: choose once, then keep. */
    if (c->policy == ORACLE_POLICY_STATIC_TOP) {
        int32_t pool = 0;
        if (c->t == c->static_warmup + 1) {
            for (int32_t b = 0; b < U; ++b)
                if (c->recoverable[b])
                    c->cand[pool++] = b;
            g_sort_r = c->gsum;
            qsort(c->cand, (size_t)pool, sizeof(int32_t), by_risk_then_index);
            int32_t keep = (int32_t)ceil(c->static_fraction * (double)nrec);
            if (keep > pool)
                keep = pool;
            for (int32_t b = 0; b < U; ++b)
                c->active[b] = 0;
            for (int32_t i = 0; i < keep; ++i)
                c->active[c->cand[i]] = 1;
        }
        int32_t nfixed = 0;
        for (int32_t b = 0; b < U; ++b) {
            mask[b] = c->active[b];
            nfixed += c->active[b];
            lock_out[b] = c->lock[b];
        }
        counts[0] = pool;
        counts[1] = nfixed;
        return 0;
    }

    /* C_t = {b : R > 1} U {b : Lock_b > 0}, over recoverable units only. */
    int32_t ncand = 0;
    for (int32_t b = 0; b < U; ++b)
        if (c->recoverable[b] && (risk[b] > 1.0 || c->lock[b] > 0))
            c->cand[ncand++] = b;

    for (int32_t b = 0; b < U; ++b)
        mask[b] = 0;
    int32_t nsel = 0;
    if (c->policy == ORACLE_POLICY_ADMISSION_CAP) {
        /* candidates active at t-1 stay; at most maxO new ones are admitted */
        int32_t nnew = 0;
        for (int32_t i = 0; i < ncand; ++i) {
            int32_t b = c->cand[i];
            if (c->active[b]) {
                mask[b] = 1;
                ++nsel;
            } else {
                c->cand[nnew++] = b;
            }
        }
        g_sort_r = risk;
        qsort(c->cand, (size_t)nnew, sizeof(int32_t), by_risk_then_index);
        int32_t admit = nnew < c->max_o ? nnew : c->max_o;
        for (int32_t i = 0; i < admit; ++i)
            mask[c->cand[i]] = 1;
        nsel += admit;
    } else {
        /* A_t = Top_maxO(C_t; R): sort by R descending, index ascending. */
        g_sort_r = risk;
        qsort(c->cand, (size_t)ncand, sizeof(int32_t), by_risk_then_index);
        nsel = ncand < c->max_o ? ncand : c->max_o;
        for (int32_t i = 0; i < nsel; ++i)
            mask[c->cand[i]] = 1;
    }
    for (int32_t b = 0; b < U; ++b)
        c->active[b] = mask[b];

    /* Lock bookkeeping of Algorithm 2. */
    for (int32_t b = 0; b < U; ++b) {
        if (!c->recoverable[b]) {
            c->lock[b] = 0;
        } else if (mask[b]) {
            if (risk[b] > 1.0)
                c->lock[b] = c->lock_len;
            else
                c->lock[b] = (c->lock[b] - 1 > 0) ? c->lock[b] - 1 : 0;
        } else {
            c->lock[b] = 0;
        }
        lock_out[b] = c->lock[b];
    }
    counts[0] = ncand;
    counts[1] = nsel;
    return 0;
}

/* State access, for checkpoint/resume tests: A[U], k[U], Q[U*window] (oldest
 * first, qlen[b] valid entries), qlen[U], lock[U], t. */
void oracle_ctl_get_state(const oracle_ctl *c, double *A, int64_t *k, double *Q,
                          int32_t *qlen, int32_t *lock, int64_t *t)
{
    size_t u = (size_t)c->num_units;
    memcpy(A, c->A, u * sizeof(double));
    memcpy(k, c->k, u * sizeof(int64_t));
    memcpy(Q, c->Q, u * (size_t)c->window * sizeof(double));
    memcpy(qlen, c->qlen, u * sizeof(int32_t));
    memcpy(lock, c->lock, u * sizeof(int32_t));
    *t = c->t;
}

void oracle_ctl_set_state(oracle_ctl *c, const double *A, const int64_t *k,
                          const double *Q, const int32_t *qlen,
                          const int32_t *lock, int64_t t)
{
    size_t u = (size_t)c->num_units;
    memcpy(c->A, A, u * sizeof(double));
    memcpy(c->k, k, u * sizeof(int64_t));
    memcpy(c->Q, Q, u * (size_t)c->window * sizeof(double));
    memcpy(c->qlen, qlen, u * sizeof(int32_t));
    memcpy(c->lock, lock, u * sizeof(int32_t));
    c->t = t;
}

/* ---- recovery actuator: fake quantization (App. E.2) ------------------- */

/* Minifloat formats: exponent bits, mantissa bits, exponent bias, largest
 * finite value.  1 = E2M1 (FP4), 2 = E3M2 (FP6), 3 = E4M3, 4 = E5M2 (FP8). */
typedef struct {
    int mbits;
    int emin;      /* exponent of the smallest normal value, 1 - bias */
    float fmax;
} fq_format;

static int fq_lookup(int code, fq_format *f)
{
    switch (code) {
    case 1: f->mbits = 1; f->emin = 1 - 1; f->fmax = 6.0f; return 0;
    case 2: f->mbits = 2; f->emin = 1 - 3; f->fmax = 28.0f; return 0;
    case 3: f->mbits = 3; f->emin = 1 - 7; f->fmax = 448.0f; return 0;
    case 4: f->mbits = 2; f->emin = 1 - 15; f->fmax = 57344.0f; return 0;
    default: return 1;
    }
}

/* Nearest representable value of the format to v (ties to the even code),
 * saturating at +-fmax.  Values with exponent e >= emin are spaced
 * 2^(e - mbits); below 2^emin (subnormals) the spacing stays 2^(emin - mbits). */
float oracle_fq_round(float v, int code)
{
    fq_format f;
    if (fq_lookup(code, &f))
        return v;
    float a = fabsf(v);
    float r;
    if (a >= f.fmax) {
        r = f.fmax;
    } else if (a == 0.0f) {
        r = 0.0f;
    } else {
        int e2;
        frexpf(a, &e2);               /* a = m * 2^e2, m in [0.5, 1) */
        int e = e2 - 1;               /* floor(log2 a) */
        if (e < f.emin)
            e = f.emin;
        float quantum = ldexpf(1.0f, e - f.mbits);
        r = rintf(a / quantum) * quantum;
    }
    return copysignf(r, v);
}

static float bf16_to_float_row(const uint16_t *p, int64_t i)
{
    uint32_t bits = ((uint32_t)p[i]) << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return f;
}

/* float -> bfloat16, round to nearest even (NaN kept as a quiet NaN). */
static uint16_t float_to_bf16_bits(float f)
{
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    if ((u & 0x7fffffffu) > 0x7f800000u)
        return (uint16_t)((u >> 16) | 0x40u);
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

/* Fake-quantizes a row-major [rows x cols] tensor, token (row) by token:
 * amax = max |x|; inv = fmax / amax; scale = amax / fmax; y = round(x * inv)
 * * scale.  code 0 copies.  in and out may be the same buffer. */
int oracle_fake_quant(const void *in, void *out, int dtype, int64_t rows, int64_t cols, int code)
{
    fq_format f = {0, 0, 1.0f};
    if (code != 0 && fq_lookup(code, &f))
        return 1;
    if (dtype != ORACLE_DTYPE_F32 && dtype != ORACLE_DTYPE_BF16)
        return 1;
    for (int64_t r = 0; r < rows; ++r) {
        float amax = 0.0f;
        int nonfinite = 0;
        for (int64_t c = 0; c < cols; ++c) {
            float x = dtype == ORACLE_DTYPE_F32 ? ((const float *)in)[r * cols + c]
                                               : bf16_to_float_row((const uint16_t *)in, r * cols + c);
            if (!isfinite(x))
                nonfinite = 1;
            else if (fabsf(x) > amax)
                amax = fabsf(x);
        }
        int keep = code == 0 || amax == 0.0f || nonfinite;
        if (!keep && isinf(f.fmax / amax))
            keep = 1;   /* the row's scale factor overflows fp32: left unchanged, like a zero row */
        float inv = keep ? 1.0f : f.fmax / amax;
        float scale = keep ? 1.0f : amax / f.fmax;
        for (int64_t c = 0; c < cols; ++c) {
            int64_t i = r * cols + c;
            float x = dtype == ORACLE_DTYPE_F32 ? ((const float *)in)[i]
                                               : bf16_to_float_row((const uint16_t *)in, i);
            float y = keep ? x : oracle_fq_round(x * inv, code) * scale;
            if (dtype == ORACLE_DTYPE_F32)
                ((float *)out)[i] = y;
            else
                ((uint16_t *)out)[i] = keep ? ((const uint16_t *)in)[i] : float_to_bf16_bits(y);
        }
    }
    return 0;
}

/* Policy state for checkpoint tests: active[U] (A_{t-1}) and gsum[U]. */
void oracle_ctl_get_policy_state(const oracle_ctl *c, uint8_t *active, double *gsum)
{
    memcpy(active, c->active, (size_t)c->num_units);
    memcpy(gsum, c->gsum, (size_t)c->num_units * sizeof(double));
}

void oracle_ctl_set_policy_state(oracle_ctl *c, const uint8_t *active, const double *gsum)
{
    memcpy(c->active, active, (size_t)c->num_units);
    memcpy(c->gsum, gsum, (size_t)c->num_units * sizeof(double));
}

/* Eq. generic-memory-bound: Delta M_t = sum over b in A_t of c_b, summed in
 * unit order. */
double oracle_delta_mem(const uint8_t *mask, const double *cost, int32_t num_units)
{
    double s = 0.0;
    for (int32_t b = 0; b < num_units; ++b)
        if (mask[b])
            s += cost[b];
    return s;
}
