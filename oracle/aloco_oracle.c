/*
 * aloco_oracle.c -- plain fp64 CPU oracle for the AutoLoCo outer
 * synchronization round (arxiv 2609.36662).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may link, load or
 * call this file: only the test suite, the smoke check and the CPU-baseline
 * leg of the benchmark do.  It shares no code, header, table or helper with
 * the CUDA library; it is written directly from the paper's definitions,
 * slowly and in the paper's order, so that it can be checked by eye.
 *
 * Every quantity is computed in IEEE double precision with no fused
 * multiply-add (built with -ffp-contract=off), in two separate passes over
 * the parameter vector:
 *   pass 1: pseudo-gradients, their average and the two diagnostics
 *           (Sec. 3.1, Eq. adaptive-h-core-diagnostics; Algorithm 1,
 *            "Synchronization" and "Interval evaluation" blocks);
 *   pass 2: the corrected Nesterov outer step and the replica reset
 *           (Sec. 3.3, Eq. autoloco-corrected-nesterov; Algorithm 1).
 * The scalar correction context (Sec. 3.2; App. B.2-B.4,
 * Eqs. app-outer-correction-lr-masses, app-outer-correction-ratios,
 * app-outer-step-scale, app-adjusted-outer-learning-rate) is evaluated by a
 * plain loop over the inner learning-rate schedule.
 *
 * Readings where the paper leaves a choice open (each is also listed in the
 * design notes of the repository):
 *   - schedule: linear warm-up lr(s) = peak*(s+1)/W for s < W, then cosine
 *     from peak to final over [W, T), then final; T counts the warm-up
 *     (Tab. training settings gives "cosine" with a 1,000-step warm-up);
 *   - eta_{t,h} = lr(s_t + h - 1), h = 1..H, s_t the 0-based global index of
 *     the interval's first local step (App. B.2);
 *   - normalisation divides by rho + eps when enabled (App. B.3);
 *   - one eps, passed in, used everywhere the paper writes epsilon;
 *   - bf16 replicas are widened exactly; the replica reset rounds the fp64
 *     result to bf16 with round-to-nearest-even;
 *   - a non-finite element is one whose updated global weight or momentum is
 *     not finite.
 *
 * Parity status: every function here is pinned by the tests under tests/
 * (closed forms, special cases, hand-computed dyadic rounds, brute force).
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

/* ---- inner learning-rate schedule (Tab. training settings; App. B.2) ---- */

enum { ORC_SCHED_COSINE = 0, ORC_SCHED_CONSTANT = 1, ORC_SCHED_LINEAR = 2 };

/* Learning rate of global inner step s (0-based). */
double orc_lr(int kind, double peak, double final_lr, int64_t warmup,
              int64_t total, int64_t s)
{
    const double pi = 3.14159265358979323846;
    if (kind == ORC_SCHED_CONSTANT)
        return peak;
    if (s < warmup)
        return peak * (double)(s + 1) / (double)warmup;
    if (s >= total)
        return final_lr;
    double frac = (double)(s - warmup) / (double)(total - warmup);
    if (kind == ORC_SCHED_COSINE)
        return final_lr + 0.5 * (peak - final_lr) * (1.0 + cos(pi * frac));
    /* ORC_SCHED_LINEAR */
    return peak + (final_lr - peak) * frac;
}

/* Accumulated inner learning rate sum_{h=1..H} eta_{t,h} with
 * eta_{t,h} = lr(t0 + h - 1)  (Eq. app-outer-correction-lr-masses). */
double orc_lr_mass(int kind, double peak, double final_lr, int64_t warmup,
                   int64_t total, int64_t t0, int64_t H)
{
    double sum = 0.0;
    for (int64_t h = 1; h <= H; ++h)
        sum += orc_lr(kind, peak, final_lr, warmup, total, t0 + h - 1);
    return sum;
}

/* ---- correction context (Sec. 3.2; App. B.2, B.4) ----
 * mode 0 = full correction, 1 = momentum only (outer lr kept at its base
 * value), 2 = none (DiLoCo settings); the three rows of Tab. component
 * ablation that run adaptive intervals.  out[] receives, in order:
 *   lam_sel, lam_base, rho_unc, rho, mu_t, kappa_t, eta_out, inv_norm. */
void orc_correction(int kind, double peak, double final_lr, int64_t warmup,
                    int64_t total, int64_t step, int64_t H_sel,
                    int64_t H_base, double outer_lr, double outer_beta,
                    double mu_min, double mu_max, double kappa_max,
                    double eps, int normalize, int mode, double *out)
{
    /* both sums start from the same scheduler position s_t = step */
    double lam_sel = orc_lr_mass(kind, peak, final_lr, warmup, total, step,
                                 H_sel);
    double lam_base = orc_lr_mass(kind, peak, final_lr, warmup, total, step,
                                  H_base);
    /* Eq. app-outer-correction-ratios */
    double rho_unc = lam_sel / (lam_base + eps);
    double rho = rho_unc > 1.0 ? rho_unc : 1.0;

    double mu_t, kappa_t, eta_out;
    if (mode == 2) {
        mu_t = outer_beta;
        kappa_t = 1.0;
        eta_out = outer_lr;
    } else {
        /* mu_t = clip(mu_base^rho, mu_min, mu_max)  (Sec. 3.2) */
        mu_t = pow(outer_beta, rho);
        if (mu_t < mu_min) mu_t = mu_min;
        if (mu_t > mu_max) mu_t = mu_max;
        if (mode == 1) {
            kappa_t = 1.0;
            eta_out = outer_lr;
        } else {
            /* Eq. app-outer-step-scale and Eq. app-adjusted-outer-learning-rate */
            kappa_t = rho < kappa_max ? rho : kappa_max;
            eta_out = outer_lr * kappa_t * (1.0 - mu_t) / (1.0 - outer_beta);
        }
    }
    /* Eq. normalized-pseudo-gradient, with rho + eps as in App. B.3 */
    double inv_norm = normalize ? 1.0 / (rho + eps) : 1.0;

    out[0] = lam_sel;
    out[1] = lam_base;
    out[2] = rho_unc;
    out[3] = rho;
    out[4] = mu_t;
    out[5] = kappa_t;
    out[6] = eta_out;
    out[7] = inv_norm;
}

/* ---- bf16 <-> double ---- */

/* Exact widening of bf16 bits: a bf16 value is the upper half of an fp32. */
static double orc_bf16_to_double(uint16_t b)
{
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Round a double to the nearest bf16 value, ties to even, in one step.
 * bf16 has an 8-bit exponent (same range as fp32) and 8 significant bits.
 * For |x| in [2^e, 2^(e+1)) with e >= -126 the spacing is 2^(e-7); below
 * 2^-126 the spacing is the subnormal quantum 2^-133.  rint() rounds to the
 * nearest integer with ties to even in the default rounding mode, and the
 * scalings by powers of two are exact in double. */
uint16_t orc_double_to_bf16(double x)
{
    uint32_t u;
    float f;
    if (isnan(x)) {
        u = 0x7FC00000u;
        return (uint16_t)(u >> 16);
    }
    if (isinf(x) || x == 0.0) {
        f = (float)x; /* exact: +-inf or +-0 */
        memcpy(&u, &f, sizeof u);
        return (uint16_t)(u >> 16);
    }
    double ax = fabs(x);
    int e;
    frexp(ax, &e);          /* ax = m * 2^e, m in [0.5, 1) => ax in [2^(e-1), 2^e) */
    int expo = e - 1;       /* ax in [2^expo, 2^(expo+1)) */
    if (expo < -126) expo = -126;
    double quantum = ldexp(1.0, expo - 7);
    double r = rint(ax / quantum) * quantum;
    /* largest finite bf16 is (2 - 2^-7) * 2^127; a rounded value of 2^128 or
     * more overflows to infinity */
    if (r >= ldexp(1.0, 128)) {
        f = INFINITY;
    } else {
        f = (float)r; /* exact: r is a bf16 value */
    }
    if (x < 0) f = -f;
    memcpy(&u, &f, sizeof u);
    return (uint16_t)(u >> 16);
}

/* ---- the synchronization round ---- */

static double orc_replica(const void *x, int dtype, int64_t n)
{
    if (dtype == 0)
        return (double)((const float *)x)[n];
    return orc_bf16_to_double(((const uint16_t *)x)[n]);
}

/*
 * Pass 1 (Algorithm 1, synchronization and interval evaluation):
 *   Delta_m[n] = g[n] - x_m[n]                (pseudo-gradient, Alg. 1)
 *   E[m]      += Delta_m[n]^2                  (||Delta_m||^2)
 *   Dbar[n]    = (1/M) sum_m Delta_m[n]       (average, Alg. 1)
 *   B         += Dbar[n]^2                     (||Dbar||^2)
 * E and B are ACCUMULATED into (the caller zeroes them), so that a long
 * vector can be processed in consecutive slices with the same summation
 * order as one call.
 */
void orc_pass1(const float *g, const void *const *x, int dtype, int64_t N,
               int M, double *E, double *B)
{
    for (int64_t n = 0; n < N; ++n) {
        double gn = (double)g[n];
        double sum = 0.0;
        for (int m = 0; m < M; ++m) {
            double delta = gn - orc_replica(x[m], dtype, n);
            E[m] += delta * delta;
            sum += delta;
        }
        double mean = sum / (double)M;
        *B += mean * mean;
    }
}

/*
 * Pass 2 (Eq. normalized-pseudo-gradient and Eq. autoloco-corrected-nesterov;
 * replica reset theta^(i)_{t+1,0} <- theta_{t+1}, Algorithm 1):
 *   Dtil  = Dbar * inv_norm
 *   v'    = mu_t * v + Dtil
 *   d     = Dtil + mu_t * v'
 *   g'    = g - eta_out * d
 *   x_m'  = g' rounded to the replica storage type
 * Outputs: g_out, v_out (double, unrounded), x_out[m] (replica storage type:
 * float, or bf16 bits).  Returns the number of elements whose g' or v' is
 * not finite.
 */
int64_t orc_pass2(const float *g, const float *v, const void *const *x,
                  int dtype, int64_t N, int M, double mu_t, double eta_out,
                  double inv_norm, double *g_out, double *v_out,
                  void *const *x_out)
{
    int64_t nonfinite = 0;
    for (int64_t n = 0; n < N; ++n) {
        double gn = (double)g[n];
        double sum = 0.0;
        for (int m = 0; m < M; ++m)
            sum += gn - orc_replica(x[m], dtype, n);
        double mean = sum / (double)M;
        double dtil = mean * inv_norm;
        double vn = mu_t * (double)v[n] + dtil;
        double dn = dtil + mu_t * vn;
        double gp = gn - eta_out * dn;
        g_out[n] = gp;
        v_out[n] = vn;
        if (!isfinite(gp) || !isfinite(vn))
            ++nonfinite;
        for (int m = 0; m < M; ++m) {
            if (x_out == 0 || x_out[m] == 0)
                continue;
            if (dtype == 0)
                ((float *)x_out[m])[n] = (float)gp;
            else
                ((uint16_t *)x_out[m])[n] = orc_double_to_bf16(gp);
        }
    }
    return nonfinite;
}

/* Interval statistics from the pass-1 sums (Eq. adaptive-h-core-diagnostics):
 *   D = (1/M) sum_m E[m],   C = M * B / (D + eps).
 * out[0] = D, out[1] = C. */
void orc_stats(const double *E, double B, int M, double eps, double *out)
{
    double s = 0.0;
    for (int m = 0; m < M; ++m)
        s += E[m];
    double D = s / (double)M;
    out[0] = D;
    out[1] = (double)M * B / (D + eps);
}

/* ---- INT8 pseudo-gradient communication (App. G.1) ----
 *
 * Blocks: each tensor part (a contiguous range of the flattened vector,
 * parts given by their sizes) is cut into consecutive blocks of at most 4096
 * elements starting at the part's first element.
 *
 * Codec, in FP32 as the appendix states: scale = max|y| / 127 (1 for an
 * all-zero block; kept within [FLT_MIN, FLT_MAX / 127] so that it neither
 * underflows to zero nor overflows on reconstruction); q = y / scale rounded
 * to the nearest integer, ties to even, clipped to [-127, 127] (a NaN
 * quotient gives q = 0 and the NaN stays in the scale); decode = q * scale.
 * Aggregation: decoded worker contributions are added in FP32 in worker
 * order and divided by M; the mean is encoded and decoded once.
 */
#include <float.h>

#define ORC_INT8_BLOCK 4096

int64_t orc_int8_blocks(const int64_t *parts, int n_parts)
{
    int64_t nb = 0;
    for (int p = 0; p < n_parts; ++p)
        nb += (parts[p] + ORC_INT8_BLOCK - 1) / ORC_INT8_BLOCK;
    return nb;
}

static float orc_int8_scale(const float *y, int64_t n)
{
    float amax = 0.0f;
    for (int64_t i = 0; i < n; ++i) {
        float a = fabsf(y[i]);
        if (isnan(a)) return a;           /* NaN propagates through the scale */
        if (a > amax) amax = a;
    }
    if (amax == 0.0f) return 1.0f;
    float s = amax / 127.0f;
    if (s < FLT_MIN) s = FLT_MIN;
    if (s > FLT_MAX / 127.0f) s = FLT_MAX / 127.0f;
    return s;
}

static int8_t orc_int8_code(float y, float s)
{
    float t = rintf(y / s);
    if (isnan(t)) return 0;
    if (t > 127.0f) t = 127.0f;
    if (t < -127.0f) t = -127.0f;
    return (int8_t)t;
}

/* Encode a vector blockwise: codes[N], scales[n_blocks], decoded[N]. */
void orc_int8_encode(const float *y, const int64_t *parts, int n_parts,
                     int8_t *codes, float *scales, float *decoded)
{
    int64_t off = 0, b = 0;
    for (int p = 0; p < n_parts; ++p) {
        for (int64_t s0 = 0; s0 < parts[p]; s0 += ORC_INT8_BLOCK, ++b) {
            int64_t n = parts[p] - s0 < ORC_INT8_BLOCK ? parts[p] - s0
                                                       : ORC_INT8_BLOCK;
            const float *yb = y + off + s0;
            float s = orc_int8_scale(yb, n);
            scales[b] = s;
            for (int64_t i = 0; i < n; ++i) {
                int8_t q = orc_int8_code(yb[i], s);
                codes[off + s0 + i] = q;
                decoded[off + s0 + i] = (float)q * s;
            }
        }
        off += parts[p];
    }
}

/* One outer round with INT8-communicated pseudo-gradients over the whole
 * vector (length = sum of parts).  Per block:
 *   Delta_m = fl32(g - x_m)               (the FP32 pseudo-gradient sent)
 *   E[m]   += (g - x_m)^2 in double       (D from the pre-quantisation Delta)
 *   mean    = fl32(sum_m decode(encode(Delta_m))) / M       (FP32, in order)
 *   Dq      = decode(encode(mean))        (the aggregate every worker gets)
 *   B      += Dq^2 in double              (C from the decoded aggregate)
 *   v' = mu v + Dq inv ; d = Dq inv + mu v' ; g' = g - eta d   (double)
 * Outputs as orc_pass2 (g_out, v_out double; x_out in storage type, may be
 * NULL).  E, B accumulate.  Returns the number of non-finite elements. */
int64_t orc_int8_round(const float *g, const float *v, const void *const *x,
                       int dtype, const int64_t *parts, int n_parts, int M,
                       double mu_t, double eta_out, double inv_norm,
                       double *g_out, double *v_out, void *const *x_out,
                       double *E, double *B)
{
    float delta[ORC_INT8_BLOCK], dec[ORC_INT8_BLOCK], sum[ORC_INT8_BLOCK];
    int8_t q[ORC_INT8_BLOCK];
    int64_t nonfinite = 0, off = 0;
    for (int p = 0; p < n_parts; ++p) {
        for (int64_t s0 = 0; s0 < parts[p]; s0 += ORC_INT8_BLOCK) {
            int64_t n = parts[p] - s0 < ORC_INT8_BLOCK ? parts[p] - s0
                                                       : ORC_INT8_BLOCK;
            int64_t base = off + s0;
            for (int64_t i = 0; i < n; ++i) sum[i] = 0.0f;
            for (int m = 0; m < M; ++m) {
                for (int64_t i = 0; i < n; ++i) {
                    double xd = orc_replica(x[m], dtype, base + i);
                    double dd = (double)g[base + i] - xd;
                    E[m] += dd * dd;
                    delta[i] = g[base + i] - (float)xd;
                }
                float s = orc_int8_scale(delta, n);
                for (int64_t i = 0; i < n; ++i) {
                    float d = (float)orc_int8_code(delta[i], s) * s;
                    sum[i] = m == 0 ? d : sum[i] + d;
                }
            }
            for (int64_t i = 0; i < n; ++i) sum[i] = sum[i] / (float)M;
            float s = orc_int8_scale(sum, n);
            for (int64_t i = 0; i < n; ++i) {
                q[i] = orc_int8_code(sum[i], s);
                dec[i] = (float)q[i] * s;
            }
            for (int64_t i = 0; i < n; ++i) {
                int64_t e = base + i;
                double dq = (double)dec[i];
                *B += dq * dq;
                double dtil = dq * inv_norm;
                double vn = mu_t * (double)v[e] + dtil;
                double dn = dtil + mu_t * vn;
                double gp = (double)g[e] - eta_out * dn;
                g_out[e] = gp;
                v_out[e] = vn;
                if (!isfinite(gp) || !isfinite(vn)) ++nonfinite;
                for (int m = 0; m < M; ++m) {
                    if (x_out == 0 || x_out[m] == 0) continue;
                    if (dtype == 0)
                        ((float *)x_out[m])[e] = (float)gp;
                    else
                        ((uint16_t *)x_out[m])[e] = orc_double_to_bf16(gp);
                }
            }
        }
        off += parts[p];
    }
    return nonfinite;
}

/* ---- inner optimizer: AdamW on every worker (Sec. 2, Eq.
 * diloco-local-trajectory: each worker takes H local AdamW steps;
 * Tab. training settings: AdamW coefficients, weight decay, gradient-norm
 * clipping 1.0, FP32 master parameters and optimizer states) ----
 *
 * One step on each of M replicas, written from the definition of AdamW
 * with decoupled weight decay:
 *   c      = min(1, max_norm / (||g|| + 1e-6))   (per replica; 1 if max_norm <= 0)
 *   g~     = c g
 *   m'     = beta1 m + (1 - beta1) g~
 *   v'     = beta2 v + (1 - beta2) g~^2
 *   x'     = x - lr wd x - lr (m' / (1 - beta1^t)) / (sqrt(v' / (1 - beta2^t)) + eps)
 * with t the 1-based step count.  Readings: the norm is over the whole
 * replica, the 1e-6 guard and the clipping-factor form are the common
 * convention (the paper names only the threshold), and the weight decay
 * applies to every parameter.  x and g may be fp32 or bf16 (widened
 * exactly); m, v are fp32.  Outputs are unrounded doubles, plus x' in its
 * storage type (fp32 rounding, or bf16 round-to-nearest-even) when x_store
 * is given; norms[m] = ||g_m|| before clipping.  With norms_in != NULL the
 * norms are taken from it instead of the passed elements (for a slice of a
 * longer replica). */
void orc_adamw_step(const void *const *x, int x_dtype, const void *const *grad,
                    int g_dtype, const float *const *m1, const float *const *m2,
                    int64_t N, int M, double lr, double beta1, double beta2,
                    double eps, double weight_decay, double max_norm,
                    int64_t step, double *const *x_out, double *const *m1_out,
                    double *const *m2_out, void *const *x_store, double *norms,
                    const double *norms_in)
{
    double bc1 = 1.0 - pow(beta1, (double)step);
    double bc2 = 1.0 - pow(beta2, (double)step);
    for (int m = 0; m < M; ++m) {
        double norm;
        if (norms_in) {
            /* the gradient's norm over its whole replica, supplied when only a
             * slice of the replica is passed */
            norm = norms_in[m];
        } else {
            double ss = 0.0;
            for (int64_t i = 0; i < N; ++i) {
                double g = orc_replica(grad[m], g_dtype, i);
                ss += g * g;
            }
            norm = sqrt(ss);
        }
        norms[m] = norm;
        double c = 1.0;
        if (max_norm > 0.0) {
            c = max_norm / (norm + 1e-6);
            if (c > 1.0) c = 1.0;
        }
        for (int64_t i = 0; i < N; ++i) {
            double g = c * orc_replica(grad[m], g_dtype, i);
            double xv = orc_replica(x[m], x_dtype, i);
            double mn = beta1 * (double)m1[m][i] + (1.0 - beta1) * g;
            double vn = beta2 * (double)m2[m][i] + (1.0 - beta2) * g * g;
            double mhat = mn / bc1;
            double vhat = vn / bc2;
            double xn = xv - lr * weight_decay * xv - lr * mhat / (sqrt(vhat) + eps);
            x_out[m][i] = xn;
            m1_out[m][i] = mn;
            m2_out[m][i] = vn;
            if (x_store && x_store[m]) {
                if (x_dtype == 0)
                    ((float *)x_store[m])[i] = (float)xn;
                else
                    ((uint16_t *)x_store[m])[i] = orc_double_to_bf16(xn);
            }
        }
    }
}
