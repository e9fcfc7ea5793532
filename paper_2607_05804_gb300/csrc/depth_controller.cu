// Adaptive rollout-depth controller and turn-level loss-allocation
// diagnostics (host code; it reads the small per-turn tables that
// turnopd_turn_stats produces, copied to the host by the caller).
//
//   efficiency mass   m_t = [K_t]_+ n_t / n_0, q_t = m_t / (sum_j m_j + eps),
//                     Hbar_eff = sum_t t q_t, H_eff = round(Hbar_eff)   (Sec. 4.1)
//   coverage bound    F(H) = 1 - n_{H+1} / n_1 over the successful probe
//                     trajectories (or all of them), H_cov = min{H : F(H) >= p},
//                     refreshed when >= min_cov_traj successes were probed (Sec. 4.1)
//   update            H_ctrl = max(H_eff, H_cov), Hbar_k = (1 - a) Hbar_{k-1} + a H_ctrl
//                     on probe steps (Sec. 4.1 "Dynamic Update", Algorithm 1)
//   schedule          Hhat_k = clip(round(Hbar_{k-1}) + 1, H_min, H_max), probe_k =
//                     (k <= K_warm) or (k mod r_probe == 0), H_roll = H_max on probe
//                     steps, Hhat_k otherwise; Hbar_0 = H_max, H_cov = 0 (Algorithm 1)
//   diagnostics       b_t = n_t / N, s_t = sum_i l_{t,i} / sum l, and the deep third of
//                     the reliable turn prefix (Sec. 3, loss-allocation diagnostics)
// round() is round-half-to-even.  The arithmetic is plain IEEE double in a fixed
// order (host code is built with -ffp-contract=off).

#include <cmath>
#include <cstdint>

#include "turnopd.h"

namespace {

inline int32_t round_even(double x) { return (int32_t)std::nearbyint(x); }

bool params_ok(const turnopd_depth_params *p)
{
    return p && p->h_min >= 1 && p->h_max >= p->h_min && p->ema_alpha >= 0.0 && p->ema_alpha <= 1.0 &&
           p->coverage_p > 0.0 && p->coverage_p <= 1.0 && p->min_cov_traj >= 0 && p->warmup_steps >= 0 &&
           p->probe_interval >= 0 && p->eps >= 0.0;
}

bool probe_step(const turnopd_depth_params *p, int64_t k)
{
    return k <= p->warmup_steps || (p->probe_interval > 0 && k % p->probe_interval == 0);
}

}  // namespace

extern "C" {

void turnopd_depth_default_params(turnopd_depth_params *p)
{
    if (!p)
        return;
    p->h_min = 2;
    p->h_max = 50;
    p->ema_alpha = 0.30;
    p->coverage_p = 0.80;
    p->min_cov_traj = 8;
    p->use_success = 1;
    p->warmup_steps = 3;
    p->probe_interval = 8;
    p->eps = 1e-8;
}

turnopd_status turnopd_depth_init(const turnopd_depth_params *p, turnopd_depth_state *s)
{
    if (!p || !s)
        return TURNOPD_ERR_NULL;
    if (!params_ok(p))
        return TURNOPD_ERR_SHAPE;
    s->h_bar = (double)p->h_max;
    s->h_eff_bar = 0.0;
    s->h_eff = 0;
    s->h_cov = 0;
    s->h_ctrl = 0;
    return TURNOPD_OK;
}

turnopd_status turnopd_depth_plan(const turnopd_depth_params *p, const turnopd_depth_state *s, int64_t k,
                                  int32_t *h_hat, int32_t *is_probe, int32_t *h_roll)
{
    if (!p || !s || !h_hat || !is_probe || !h_roll)
        return TURNOPD_ERR_NULL;
    if (!params_ok(p) || k < 1)
        return TURNOPD_ERR_SHAPE;
    int32_t h = round_even(s->h_bar) + 1;
    h = h < p->h_min ? p->h_min : (h > p->h_max ? p->h_max : h);
    *h_hat = h;
    *is_probe = probe_step(p, k) ? 1 : 0;
    *h_roll = *is_probe ? p->h_max : h;
    return TURNOPD_OK;
}

turnopd_status turnopd_depth_efficiency(const double *turn_sum, const int64_t *turn_cnt, const int32_t *turn_surv,
                                        int32_t max_turns, double eps, double *m_out, double *q_out,
                                        double *h_eff_bar, int32_t *h_eff)
{
    if (!turn_sum || !turn_cnt || !turn_surv || !h_eff_bar || !h_eff)
        return TURNOPD_ERR_NULL;
    if (max_turns < 1 || eps < 0.0)
        return TURNOPD_ERR_SHAPE;
    const double n0 = (double)turn_surv[0];
    double total = 0.0;
    for (int32_t t = 0; t < max_turns; ++t) {
        double m = 0.0;
        if (n0 > 0.0) {
            const double K = turn_cnt[t] > 0 ? turn_sum[t] / (double)turn_cnt[t] : 0.0;
            m = (K > 0.0 ? K : 0.0) * (double)turn_surv[t] / n0;
        }
        if (m_out)
            m_out[t] = m;
        total += m;
    }
    double hbar = 0.0;
    for (int32_t t = 0; t < max_turns; ++t) {
        double m;
        if (n0 > 0.0) {
            const double K = turn_cnt[t] > 0 ? turn_sum[t] / (double)turn_cnt[t] : 0.0;
            m = (K > 0.0 ? K : 0.0) * (double)turn_surv[t] / n0;
        } else {
            m = 0.0;
        }
        const double q = m / (total + eps);
        if (q_out)
            q_out[t] = q;
        hbar += (double)t * q;
    }
    *h_eff_bar = hbar;
    *h_eff = round_even(hbar);
    return TURNOPD_OK;
}

turnopd_status turnopd_depth_coverage(const int32_t *traj_len, const uint8_t *traj_success, int32_t num_traj,
                                      double p, int32_t min_cov_traj, int32_t use_success, int32_t previous,
                                      int32_t *h_cov)
{
    if (!h_cov || (num_traj > 0 && (!traj_len || !traj_success)))
        return TURNOPD_ERR_NULL;
    if (num_traj < 0 || p <= 0.0 || p > 1.0 || min_cov_traj < 0)
        return TURNOPD_ERR_SHAPE;
    int64_t n_succ = 0, n1 = 0, max_len = 0;
    for (int32_t b = 0; b < num_traj; ++b) {
        n_succ += traj_success[b] ? 1 : 0;
        const bool in_pool = use_success ? traj_success[b] != 0 : true;
        if (in_pool && traj_len[b] >= 1) {
            ++n1;
            if (traj_len[b] > max_len)
                max_len = traj_len[b];
        }
    }
    *h_cov = previous;
    if (n_succ < min_cov_traj || n1 == 0)
        return TURNOPD_OK;
    for (int64_t H = 0; H <= max_len; ++H) {
        int64_t reach = 0;  // pool trajectories that reach turn H + 1
        for (int32_t b = 0; b < num_traj; ++b) {
            const bool in_pool = use_success ? traj_success[b] != 0 : true;
            reach += (in_pool && traj_len[b] >= H + 1) ? 1 : 0;
        }
        if (1.0 - (double)reach / (double)n1 >= p) {
            *h_cov = (int32_t)H;
            return TURNOPD_OK;
        }
    }
    *h_cov = (int32_t)max_len;
    return TURNOPD_OK;
}

turnopd_status turnopd_depth_update(const turnopd_depth_params *p, turnopd_depth_state *s, int64_t k,
                                    const double *turn_sum, const int64_t *turn_cnt, const int32_t *turn_surv,
                                    int32_t max_turns, const int32_t *traj_len, const uint8_t *traj_success,
                                    int32_t num_traj, double *m_out, double *q_out)
{
    if (!p || !s)
        return TURNOPD_ERR_NULL;
    if (!params_ok(p) || k < 1)
        return TURNOPD_ERR_SHAPE;
    if (!probe_step(p, k))
        return TURNOPD_OK;  // routine (capped) steps leave the depth statistics alone
    double hbar_eff = 0.0;
    int32_t h_eff = 0, h_cov = s->h_cov;
    turnopd_status st =
        turnopd_depth_efficiency(turn_sum, turn_cnt, turn_surv, max_turns, p->eps, m_out, q_out, &hbar_eff, &h_eff);
    if (st != TURNOPD_OK)
        return st;
    st = turnopd_depth_coverage(traj_len, traj_success, num_traj, p->coverage_p, p->min_cov_traj, p->use_success,
                                s->h_cov, &h_cov);
    if (st != TURNOPD_OK)
        return st;
    s->h_eff_bar = hbar_eff;
    s->h_eff = h_eff;
    s->h_cov = h_cov;
    s->h_ctrl = h_eff > h_cov ? h_eff : h_cov;
    s->h_bar = (1.0 - p->ema_alpha) * s->h_bar + p->ema_alpha * (double)s->h_ctrl;
    return TURNOPD_OK;
}

turnopd_status turnopd_turn_diagnostics(const double *turn_sum, const int64_t *turn_cnt, const int32_t *turn_surv,
                                        int32_t max_turns, int32_t n_min, double *b_out, double *s_out,
                                        double *deep_out)
{
    if (!turn_sum || !turn_cnt || !turn_surv || !b_out || !s_out || !deep_out)
        return TURNOPD_ERR_NULL;
    if (max_turns < 1)
        return TURNOPD_ERR_SHAPE;
    double N = 0.0, L = 0.0;
    for (int32_t t = 0; t < max_turns; ++t) {
        N += (double)turn_cnt[t];
        L += turn_sum[t];
    }
    for (int32_t t = 0; t < max_turns; ++t) {
        b_out[t] = N > 0.0 ? (double)turn_cnt[t] / N : 0.0;
        s_out[t] = L != 0.0 ? turn_sum[t] / L : 0.0;
    }
    int32_t P = 0;
    while (P < max_turns && turn_surv[P] >= n_min && turn_surv[P] > 0)
        ++P;
    deep_out[0] = (double)P;
    deep_out[1] = deep_out[2] = deep_out[3] = NAN;
    const int32_t third = P / 3;
    if (third >= 1) {
        auto K = [&](int32_t t) { return turn_cnt[t] > 0 ? turn_sum[t] / (double)turn_cnt[t] : 0.0; };
        double ks = 0.0, kd = 0.0, sup = 0.0, bud = 0.0;
        for (int32_t t = 0; t < third; ++t)
            ks += K(t);
        for (int32_t t = P - third; t < P; ++t) {
            kd += K(t);
            sup += (double)turn_surv[t];
            bud += s_out[t];
        }
        ks /= third;
        kd /= third;
        deep_out[1] = ks != 0.0 ? kd / ks : NAN;
        deep_out[2] = sup / third / (double)turn_surv[0];
        deep_out[3] = bud;
    }
    return TURNOPD_OK;
}

}  // extern "C"
