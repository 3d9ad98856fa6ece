// Interval controller of AutoLoCo (Sec. 3.1, App. A.1-A.3): host-only,
// scalar.  After each completed interval it assesses D_t and C_t against the
// accepted-horizon reference profile and chooses the next horizon.
#include <algorithm>
#include <cmath>
#include <cstring>

#include "../../include/aloco.h"
#include "aloco_internal.h"

namespace {

constexpr int32_t kStateVersion = 1;

int bad(const char *why) { return aloco::report_error(ALOCO_ERR_ARG, why); }

int check_cfg(const aloco_ctrl_cfg_t *c) {
    if (!c) return bad("controller cfg is NULL");
    if (c->q_H < 1) return bad("q_H must be >= 1");
    if (c->H_min < c->q_H || c->H_min > c->H_base || c->H_base > c->H_max)
        return bad("need q_H <= H_min <= H_base <= H_max");
    if (c->H_min % c->q_H || c->H_max % c->q_H || c->H_base % c->q_H)
        return bad("H_min, H_base and H_max must be multiples of q_H");
    if (!(c->thr_candidate > 0 && c->thr_candidate <= c->thr_moderate &&
          c->thr_moderate <= c->thr_severe))
        return bad("need 0 < thr_candidate <= thr_moderate <= thr_severe");
    if (!(c->exposure_mult >= 1.0)) return bad("exposure_mult must be >= 1");
    if (!(c->div_moderate > 1.0 && c->div_severe > 1.0))
        return bad("reduction divisors must be > 1");
    if (!(c->retire_frac > 0.0 && c->retire_frac <= 1.0))
        return bad("retire_frac must be in (0, 1]");
    if (!(c->ref_ema >= 0.0 && c->ref_ema <= 1.0)) return bad("ref_ema must be in [0, 1]");
    if (!(c->mad_scale > 0.0 && c->scale_floor > 0.0 && c->eps > 0.0))
        return bad("mad_scale, scale_floor and eps must be > 0");
    if (!(c->beta_tok >= 0.0 && c->beta_tok < 1.0)) return bad("beta_tok must be in [0, 1)");
    if (c->mapper_bootstrap < 1 || c->mapper_bootstrap > 8)
        return bad("mapper_bootstrap must be in [1, 8]");
    if (c->ref_bootstrap < 1 || c->variability_intervals < 1 || c->severe_fallback < 1)
        return bad("bootstrap counts must be >= 1");
    if (c->warmup_steps < 0) return bad("warmup_steps must be >= 0");
    return ALOCO_OK;
}

double median_of(double *v, int n) {
    std::sort(v, v + n);
    return (n % 2) ? v[n / 2] : 0.5 * (v[n / 2 - 1] + v[n / 2]);
}

// Admissible horizon nearest to x with lo < h < hi (0 = no such bound);
// ties take the smaller; 0 if none.
int64_t nearest_admissible(const aloco_ctrl_cfg_t &c, double x, int64_t lo,
                           int64_t hi) {
    int64_t best = 0;
    double best_d = 0.0;
    for (int64_t h = c.H_min; h <= c.H_max; h += c.q_H) {
        if (lo > 0 && h <= lo) continue;
        if (hi > 0 && h >= hi) continue;
        const double d = std::fabs((double)h - x);
        if (best == 0 || d < best_d) {
            best = h;
            best_d = d;
        }
    }
    return best;
}

// Token horizon -> executable steps (Eq. adaptive-h-token-mapping).
int64_t map_steps(const aloco_ctrl_state_t &s, const aloco_ctrl_cfg_t &c,
                  int64_t h_tok) {
    if (!s.calibrated || !(s.n_hat > 0.0)) return h_tok;
    const double x = s.M_base * (double)h_tok / ((double)c.H_base * (s.n_hat + c.eps));
    const double q = (double)c.q_H;
    const double lo = std::floor(x / q) * q;
    const double hi = lo + q;
    double h = (x - lo <= hi - x) ? lo : hi;  // ties take the smaller
    if (h < q) h = q;
    return (int64_t)h;
}

double lr_mass(const aloco_schedule_t *sched, int64_t t0, int64_t H) {
    return aloco_inner_lr_accum(sched, t0, H);
}

double safe_log(double x) { return std::log(std::max(x, 1e-300)); }

bool finite_obs(const aloco_interval_obs_t &o) {
    return std::isfinite(o.D) && std::isfinite(o.C) && std::isfinite(o.lam) &&
           o.D >= 0.0 && o.C >= 0.0 && o.lam >= 0.0;
}

// Residuals of Eq. adaptive-h-core-residuals with xi of Eq. adaptive-h-lr-mass.
void residuals(const aloco_ctrl_state_t &s, const aloco_ctrl_cfg_t &c,
               const aloco_interval_obs_t &o, double *r_D, double *r_C) {
    const double xi = o.lam / (s.lam_ref + c.eps);
    const double sqrt_D_ref = std::exp(0.5 * s.log_D_ref);
    const double C_ref = std::exp(s.log_C_ref);
    *r_D = std::log(std::sqrt(o.D) / (sqrt_D_ref * xi + c.eps) + c.eps);
    *r_C = -std::log(o.C / (C_ref + c.eps) + c.eps);
}

// z_t^max of Eq. adaptive-h-core-deviation: positive parts over robust scales.
double deviation(const aloco_ctrl_state_t &s, const aloco_ctrl_cfg_t &c,
                 double r_D, double r_C) {
    const int n = s.n_hist;
    if (n == 0) return 0.0;
    double zs[2];
    const double *hist[2] = {s.hist_D, s.hist_C};
    const double r[2] = {r_D, r_C};
    for (int f = 0; f < 2; ++f) {
        double v[ALOCO_CTRL_HISTORY], a[ALOCO_CTRL_HISTORY];
        for (int i = 0; i < n; ++i) v[i] = hist[f][i];
        const double centre = median_of(v, n);
        for (int i = 0; i < n; ++i) a[i] = std::fabs(hist[f][i] - centre);
        const double scale = std::max(c.mad_scale * median_of(a, n), c.scale_floor);
        const double excess = std::max(r[f] - centre, 0.0);
        zs[f] = excess > 0.0 ? excess / scale : 0.0;
    }
    return std::max(zs[0], zs[1]);
}

int classify(const aloco_ctrl_cfg_t &c, double z) {
    if (!std::isfinite(z)) return ALOCO_ASSESS_INVALID;
    if (z < c.thr_candidate) return ALOCO_ASSESS_SUPPORTED;
    if (z < c.thr_moderate) return ALOCO_ASSESS_CONSISTENT;
    if (z < c.thr_severe) return ALOCO_ASSESS_MODERATE;
    return ALOCO_ASSESS_SEVERE;
}

void push_residuals(aloco_ctrl_state_t &s, double r_D, double r_C) {
    s.hist_D[s.head] = r_D;
    s.hist_C[s.head] = r_C;
    s.head = (s.head + 1) % ALOCO_CTRL_HISTORY;
    if (s.n_hist < ALOCO_CTRL_HISTORY) ++s.n_hist;
}

// Log-space EMA of the diagnostic references; Lambda_ref follows the latest
// accepted interval, and D_ref is first carried to that exposure (under the
// displacement-proportional-to-Lambda model behind xi, sqrt(D) scales with
// Lambda).
void update_profile(aloco_ctrl_state_t &s, const aloco_ctrl_cfg_t &c,
                    const aloco_interval_obs_t &o) {
    const double a = c.ref_ema;
    const double shift = 2.0 * std::log((o.lam + c.eps) / (s.lam_ref + c.eps));
    s.log_D_ref = (1.0 - a) * (s.log_D_ref + shift) + a * safe_log(o.D);
    s.log_C_ref = (1.0 - a) * s.log_C_ref + a * safe_log(o.C);
    s.lam_ref = o.lam;
}

void start_reference(aloco_ctrl_state_t &s, int needed) {
    s.phase = ALOCO_PHASE_REFERENCE;
    s.phase_count = 0;
    s.ref_needed = needed;
    s.sum_log_D = s.sum_log_C = 0.0;
}

void start_variability(aloco_ctrl_state_t &s) {
    s.phase = ALOCO_PHASE_VARIABILITY;
    s.phase_count = 0;
    s.n_hist = 0;
    s.head = 0;
}

void reduce(aloco_ctrl_state_t &s, const aloco_ctrl_cfg_t &c, double div) {
    int64_t h = nearest_admissible(c, (double)s.H_acc / div, 0, s.H_acc);
    if (h == 0 || s.severe_run >= c.severe_fallback) h = c.H_min;
    s.H_acc = s.H_next = h;
    s.H_cand = 0;
    s.moderate_run = 0;
    start_reference(s, 1);
}

void adopt(aloco_ctrl_state_t &s, const aloco_interval_obs_t &o) {
    s.H_acc = s.H_next = s.H_cand;
    s.H_cand = 0;
    if (s.bound && s.H_acc >= s.bound) s.bound = 0;
    s.log_D_ref = safe_log(o.D);
    s.log_C_ref = safe_log(o.C);
    s.lam_ref = o.lam;
    s.referenced = 1;
    s.moderate_run = s.severe_run = 0;
    start_variability(s);
}

void reject(aloco_ctrl_state_t &s, const aloco_interval_obs_t &o) {
    s.bound = s.H_cand;
    s.bound_lam = o.lam;
    s.H_cand = 0;
    s.H_next = s.H_acc;
    s.moderate_run = 0;
    start_reference(s, 1);
}

// Longer horizon to try next (0: none), previewed from step `pos`.
int64_t propose(aloco_ctrl_state_t &s, const aloco_ctrl_cfg_t &c,
                const aloco_schedule_t *sched, int64_t pos) {
    if (s.bound) {
        const double at_bound = lr_mass(sched, pos, map_steps(s, c, s.bound));
        if (at_bound <= c.retire_frac * s.bound_lam) s.bound = 0;
    }
    const double base = lr_mass(sched, pos, map_steps(s, c, s.H_acc));
    int64_t best = 0;
    for (int64_t h = s.H_acc + c.q_H; h <= c.H_max; h += c.q_H) {
        if (h < c.H_min) continue;
        if (lr_mass(sched, pos, map_steps(s, c, h)) <= c.exposure_mult * base)
            best = h;
        else
            break;  // exposure grows with h
    }
    if (s.bound && best) {
        const double mid = std::sqrt((double)s.H_acc * (double)s.bound);
        const int64_t hm = nearest_admissible(c, mid, s.H_acc, s.bound);
        best = hm ? std::min(best, hm) : 0;
    }
    return best;
}

void fill_decision(const aloco_ctrl_state_t &s, const aloco_ctrl_cfg_t &c,
                   aloco_ctrl_decision_t *d) {
    d->H_tok = s.H_next;
    d->H_step = map_steps(s, c, s.H_next);
    d->H_ref_step = map_steps(s, c, c.H_base);
    d->assessment = s.last_assessment;
    d->phase = s.phase;
    d->z = s.last_z;
    d->r_D = s.last_r_D;
    d->r_C = s.last_r_C;
}

}  // namespace

extern "C" {

void aloco_ctrl_default_cfg(aloco_ctrl_cfg_t *cfg, int64_t H_base,
                            int64_t H_min, int64_t H_max, int64_t q_H,
                            int64_t warmup_steps) {
    if (!cfg) return;
    std::memset(cfg, 0, sizeof *cfg);
    cfg->H_base = H_base;
    cfg->H_min = H_min;
    cfg->H_max = H_max;
    cfg->q_H = q_H;
    cfg->warmup_steps = warmup_steps;
    cfg->beta_tok = 0.9;
    cfg->thr_candidate = 1.5;
    cfg->thr_moderate = 2.5;
    cfg->thr_severe = 4.0;
    cfg->exposure_mult = 1.15;
    cfg->div_moderate = 1.20;
    cfg->div_severe = 1.50;
    cfg->retire_frac = 0.90;
    cfg->ref_ema = 0.1;
    cfg->mad_scale = 1.4826;
    cfg->scale_floor = 1e-3;
    cfg->eps = 1e-8;
    cfg->mapper_bootstrap = 3;
    cfg->ref_bootstrap = 2;
    cfg->variability_intervals = 3;
    cfg->severe_fallback = 2;
}

int aloco_ctrl_init(aloco_ctrl_state_t *state, const aloco_ctrl_cfg_t *cfg,
                    aloco_ctrl_decision_t *first) {
    if (!state) return bad("state is NULL");
    int rc = check_cfg(cfg);
    if (rc != ALOCO_OK) return rc;
    std::memset(state, 0, sizeof *state);
    state->version = kStateVersion;
    state->phase = ALOCO_PHASE_WARMUP;
    state->H_acc = state->H_next = cfg->H_base;
    state->ref_needed = cfg->ref_bootstrap;
    state->last_assessment = ALOCO_ASSESS_NONE;
    if (first) fill_decision(*state, *cfg, first);
    return ALOCO_OK;
}

int aloco_select_interval(aloco_ctrl_state_t *state, const aloco_ctrl_cfg_t *cfg,
                          const aloco_interval_obs_t *obs,
                          const aloco_schedule_t *schedule,
                          aloco_ctrl_decision_t *out) {
    if (!state || !obs || !out) return bad("NULL argument");
    int rc = check_cfg(cfg);
    if (rc != ALOCO_OK) return rc;
    if (state->version != kStateVersion) return bad("controller state not initialised");
    if (obs->H_step < 1 || obs->step_end < obs->H_step)
        return bad("interval needs H_step >= 1 and step_end >= H_step");
    if (!std::isfinite(aloco_inner_lr_accum(schedule, 0, 0)))
        return bad("invalid schedule");
    aloco_ctrl_state_t &s = *state;
    const aloco_ctrl_cfg_t &c = *cfg;
    const aloco_interval_obs_t &o = *obs;
    const int64_t H_ran = s.H_next;
    ++s.intervals;
    s.last_assessment = ALOCO_ASSESS_NONE;
    s.last_z = s.last_r_D = s.last_r_C = 0.0;

    // token mapper (App. A.3): density EMA, then M_base from the first
    // recipe-horizon intervals
    if (std::isfinite(o.tokens) && o.tokens >= 0.0) {
        const double nbar = o.tokens / (double)o.H_step;
        s.n_hat = (s.intervals == 1) ? nbar : c.beta_tok * s.n_hat + (1.0 - c.beta_tok) * nbar;
        if (!s.calibrated && H_ran == c.H_base && s.mapper_n < c.mapper_bootstrap) {
            s.mapper_mass[s.mapper_n++] = o.tokens;
            if (s.mapper_n == c.mapper_bootstrap) {
                double v[8];
                for (int i = 0; i < s.mapper_n; ++i) v[i] = s.mapper_mass[i];
                s.M_base = median_of(v, s.mapper_n);
                s.calibrated = 1;
            }
        }
    }

    const bool ok = finite_obs(o);
    if (s.phase == ALOCO_PHASE_WARMUP) {
        if (o.step_end >= c.warmup_steps)
            start_reference(s, c.ref_bootstrap);  // this interval completes warm-up
    }
    switch (s.phase) {
        case ALOCO_PHASE_WARMUP:
            break;
        case ALOCO_PHASE_REFERENCE:
            if (!ok) {
                s.last_assessment = ALOCO_ASSESS_INVALID;
                if (s.referenced) {  // re-estimation: the reduction path
                    ++s.severe_run;
                    reduce(s, c, c.div_severe);
                }  // first estimate: only finite intervals enter it
                break;
            }
            s.sum_log_D += safe_log(o.D);
            s.sum_log_C += safe_log(o.C);
            s.lam_ref = o.lam;
            if (++s.phase_count == s.ref_needed) {
                s.log_D_ref = s.sum_log_D / s.ref_needed;
                s.log_C_ref = s.sum_log_C / s.ref_needed;
                s.referenced = 1;
                start_variability(s);
            }
            break;
        case ALOCO_PHASE_VARIABILITY: {
            if (!ok) {
                s.last_assessment = ALOCO_ASSESS_INVALID;
                ++s.severe_run;
                reduce(s, c, c.div_severe);
                break;
            }
            double r_D, r_C;
            residuals(s, c, o, &r_D, &r_C);
            s.last_r_D = r_D;
            s.last_r_C = r_C;
            push_residuals(s, r_D, r_C);
            update_profile(s, c, o);
            if (++s.phase_count == c.variability_intervals) {
                s.phase = ALOCO_PHASE_MONITOR;
                s.phase_count = 0;
            }
            break;
        }
        case ALOCO_PHASE_MONITOR:
        case ALOCO_PHASE_CANDIDATE:
        case ALOCO_PHASE_CONFIRM: {
            double r_D = 0.0, r_C = 0.0, z = INFINITY;
            int a = ALOCO_ASSESS_INVALID;
            if (ok) {
                residuals(s, c, o, &r_D, &r_C);
                z = deviation(s, c, r_D, r_C);
                a = classify(c, z);
            }
            s.last_assessment = a;
            s.last_z = std::isfinite(z) ? z : 0.0;
            s.last_r_D = r_D;
            s.last_r_C = r_C;
            const bool good = a == ALOCO_ASSESS_SUPPORTED || a == ALOCO_ASSESS_CONSISTENT;
            if (s.phase == ALOCO_PHASE_MONITOR) {
                if (good) {
                    push_residuals(s, r_D, r_C);
                    update_profile(s, c, o);
                    s.moderate_run = s.severe_run = 0;
                    if (a == ALOCO_ASSESS_SUPPORTED) {
                        const int64_t h = propose(s, c, schedule, o.step_end);
                        if (h > s.H_acc) {
                            s.H_cand = s.H_next = h;
                            s.phase = ALOCO_PHASE_CANDIDATE;
                        }
                    }
                } else if (a == ALOCO_ASSESS_MODERATE) {
                    s.severe_run = 0;
                    if (++s.moderate_run >= 2) reduce(s, c, c.div_moderate);
                } else {
                    ++s.severe_run;
                    reduce(s, c, c.div_severe);
                }
            } else if (s.phase == ALOCO_PHASE_CANDIDATE) {
                if (a == ALOCO_ASSESS_SUPPORTED)
                    adopt(s, o);
                else if (a == ALOCO_ASSESS_CONSISTENT)
                    s.phase = ALOCO_PHASE_CONFIRM;
                else
                    reject(s, o);
            } else {  // CONFIRM
                if (good)
                    adopt(s, o);
                else
                    reject(s, o);
            }
            break;
        }
        default:
            return bad("corrupt controller phase");
    }
    fill_decision(s, c, out);
    return ALOCO_OK;
}

size_t aloco_ctrl_state_bytes(void) { return sizeof(aloco_ctrl_state_t); }

int aloco_ctrl_save(const aloco_ctrl_state_t *state, void *buf, size_t len) {
    if (!state || !buf) return bad("NULL argument");
    if (len < sizeof *state) return bad("buffer smaller than aloco_ctrl_state_bytes()");
    std::memcpy(buf, state, sizeof *state);
    return ALOCO_OK;
}

int aloco_ctrl_load(aloco_ctrl_state_t *state, const void *buf, size_t len) {
    if (!state || !buf) return bad("NULL argument");
    if (len < sizeof *state) return bad("buffer smaller than aloco_ctrl_state_bytes()");
    aloco_ctrl_state_t tmp;
    std::memcpy(&tmp, buf, sizeof tmp);
    if (tmp.version != kStateVersion) return bad("controller state version mismatch");
    if (tmp.phase < ALOCO_PHASE_WARMUP || tmp.phase > ALOCO_PHASE_CONFIRM ||
        tmp.n_hist < 0 || tmp.n_hist > ALOCO_CTRL_HISTORY || tmp.head < 0 ||
        tmp.head >= ALOCO_CTRL_HISTORY || tmp.mapper_n < 0 || tmp.mapper_n > 8)
        return bad("corrupt controller state");
    *state = tmp;
    return ALOCO_OK;
}

}  // extern "C"
