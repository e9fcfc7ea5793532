/*
 * turnopd_oracle.c -- plain, slow, fp64 CPU oracle for the turn-aware
 * on-policy-distillation (OPD) loss of TurnOPD.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path links, loads or
 * calls this file: only the test-suite, the smoke check and the benchmark's
 * CPU-baseline leg do.  It shares no source, header, table or helper with the
 * CUDA library; the two meet only through seeded inputs.
 *
 * Every quantity is computed in IEEE double precision, straight from its
 * definition, with no blocking, fusion or reordering beyond what the
 * definition states.  Inputs in bf16 or fp32 are widened exactly to double.
 *
 * What each function follows (sections, equations and the algorithm of the
 * TurnOPD paper, arXiv 2607.05804):
 *   oracle_turn_counts   -- multi-turn trace model (Sec. 3, "Multi-turn agent
 *                           interaction"): supervised tokens per (trajectory,
 *                           turn), survivors per turn index (Sec. 4.1 "only
 *                           trajectories that reach each turn", Sec. 5.1 n_t).
 *   oracle_weights       -- Sec. 5.2 (q_t^traj, q_t^turn, q_t^blend) and the
 *                           weight step of Algorithm 1 (w_traj, w_turn, w_blend),
 *                           with the per-trajectory token mean of Eq. (opd-rkl)
 *                           and the seq-mean-token-mean aggregation of the
 *                           hyper-parameter table; turn floor n_min from the same
 *                           table.
 *   oracle_row           -- Eq. (opd-rkl): reverse KL(pi_s || pi_T) per token,
 *                           its gradient w.r.t. the student logits, and the
 *                           single-sample estimator log pi_s(y) - log pi_T(y).
 *   oracle_loss_fwd_bwd  -- L_k = sum_i w_blend,i * l_i (Algorithm 1).
 *   oracle_turn_stats    -- K_t (Eq. observed-turn-kl) as sums and counts per
 *                           (trajectory, turn) and per turn index, plus survivor
 *                           counts n_t (Sec. 5.1; kl_per_turn/num_traj keys).
 *   oracle_fused_lmhead  -- logits z = h W^T from the two LM heads, then the
 *                           row oracle, then dL/dh_s = g W_s and
 *                           dL/dW_s = sum_i g_i^T h_s,i.
 *   oracle_topk_row /    -- the paper's practical loss, the teacher top-K
 *   oracle_topk_loss        reverse KL (loss_mode topk_reverse_kl with support
 *                           size K_top = distill_topk = 50 in the full
 *                           configuration table; Algorithm 1 "top-K reverse-KL
 *                           token losses"): Eq. (opd-rkl) restricted to the K
 *                           vocabulary ids of largest teacher logit.
 *   oracle_alpha_schedule-- alpha = clip((k/K - s)/(e - s), 0, 1) (Sec. 5.2,
 *                           Algorithm 1).
 *
 * Readings where the paper is silent (each also listed in the design notes):
 *   natural log; T counts the turns of a trajectory that hold >= 1 supervised
 *   token; a turn's mass q_t is shared equally by its n_t tokens; the batch
 *   expectation is a mean over the trajectories that hold >= 1 supervised
 *   token; a turn index is reliable iff it is reached by >= n_min trajectories,
 *   tokens of unreliable turns keep the token-level weight and the reliable
 *   turns share the rest equally; the sampled-token gradient is the
 *   score-function form w * l * (e_y - p_s); the top-K support is the K ids of
 *   largest teacher logit, the lower id first among equal logits, and both
 *   distributions are renormalised over that support.
 *
 * Status codes returned (same meaning as the library's public codes):
 *   0 ok, 2 bad shape, 3 bad offsets, 4 turn id out of range,
 *   5 token/row/sampled id out of range, 9 non-finite value.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define OR_OK 0
#define OR_SHAPE 2
#define OR_OFFSETS 3
#define OR_TURN_RANGE 4
#define OR_TOKEN_RANGE 5
#define OR_NONFINITE 9

#define OR_F32 0
#define OR_BF16 1

#define OR_FULL_VOCAB 0
#define OR_SAMPLED_TOKEN 1

#define OR_SCOPE_TRAJ 0
#define OR_SCOPE_BATCH 1

/* ---- exact widening ---------------------------------------------------- */

static double widen_bf16(uint16_t bits)
{
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

static double elem(const void *base, int dtype, int64_t idx)
{
    if (dtype == OR_BF16)
        return widen_bf16(((const uint16_t *)base)[idx]);
    return (double)((const float *)base)[idx];
}

/* Neumaier-compensated running sum. */
typedef struct { double s, c; } kahan_t;
static void kadd(kahan_t *k, double x)
{
    double t = k->s + x;
    if (fabs(k->s) >= fabs(x))
        k->c += (k->s - t) + x;
    else
        k->c += (x - t) + k->s;
    k->s = t;
}
static double kval(const kahan_t *k) { return k->s + k->c; }

/* ---- trajectory / turn bookkeeping ------------------------------------- */

static int check_offsets(const int64_t *off, int32_t B, int64_t T)
{
    if (off[0] != 0 || off[B] != T)
        return OR_OFFSETS;
    for (int32_t b = 0; b < B; ++b)
        if (off[b + 1] < off[b])
            return OR_OFFSETS;
    return OR_OK;
}

/*
 * n_bt[b*Tmax + t] = number of supervised tokens (mask = 1) of trajectory b
 *                    whose turn id is t.
 * counts[0 .. Tmax)        S_t: trajectories with n_bt > 0 (survivors of t)
 * counts[Tmax .. 2 Tmax)   C_t: supervised tokens at turn index t (sum over b)
 * counts[2 Tmax]           B': trajectories holding >= 1 supervised token
 * A supervised token whose turn id lies outside [0, Tmax) is an error.
 */
int oracle_turn_counts(const int32_t *turn_id, const uint8_t *mask,
                       const int64_t *off, int32_t B, int64_t T, int32_t Tmax,
                       int32_t *n_bt, int64_t *counts)
{
    if (B < 0 || T < 0 || Tmax < 1)
        return OR_SHAPE;
    int st = check_offsets(off, B, T);
    if (st)
        return st;
    memset(n_bt, 0, sizeof(int32_t) * (size_t)B * (size_t)Tmax);
    memset(counts, 0, sizeof(int64_t) * (size_t)(2 * Tmax + 1));
    for (int32_t b = 0; b < B; ++b) {
        for (int64_t i = off[b]; i < off[b + 1]; ++i) {
            if (!mask[i])
                continue;
            int32_t t = turn_id[i];
            if (t < 0 || t >= Tmax)
                return OR_TURN_RANGE;
            n_bt[(int64_t)b * Tmax + t] += 1;
        }
    }
    for (int32_t b = 0; b < B; ++b) {
        int64_t Nb = 0;
        for (int32_t t = 0; t < Tmax; ++t) {
            int32_t n = n_bt[(int64_t)b * Tmax + t];
            if (n > 0)
                counts[t] += 1;
            counts[Tmax + t] += n;
            Nb += n;
        }
        if (Nb > 0)
            counts[2 * Tmax] += 1;
    }
    return OR_OK;
}

/*
 * Per-token blend weights w_blend,i = (1 - alpha) w_traj,i + alpha w_turn,i.
 *
 * SCOPE_TRAJ (Eq. opd-rkl: 1/sum_i m_i inside the expectation over
 * trajectories; seq-mean-token-mean):
 *   w_traj,i = 1/N_b                                  (N_b supervised tokens of b)
 *   w_turn,i = q_t^turn / n_bt = 1/(T_b n_bt)         (T_b non-empty turns of b)
 *   w_i      = [(1-alpha) w_traj,i + alpha w_turn,i] / B'
 * With a turn floor n_min > 0, turn index t is reliable iff S_t >= n_min.
 * Tokens of unreliable turns keep w_turn,i = 1/N_b; the R_b reliable
 * non-empty turns of b share the remaining mass 1 - U_b/N_b equally
 * (U_b = unreliable tokens of b); with R_b = 0, w_turn = w_traj.  n_min <= 0
 * makes every turn reliable and reduces exactly to the unfloored form.
 *
 * SCOPE_BATCH (one token mean over the whole batch):
 *   w_traj,i = 1/N, w_turn,i = 1/(S n_bt), N = sum_t C_t, S = sum_t S_t
 *   (floor as above with U, R taken over the batch), no 1/B' factor.
 *
 * global_counts (nullable) replaces the locally derived S_t, C_t, B' by
 * values summed over data-parallel ranks; n_bt, N_b, T_b stay local.
 * Masked tokens get w = 0.
 */
int oracle_weights(const int32_t *turn_id, const uint8_t *mask,
                   const int64_t *off, int32_t B, int64_t T, int32_t Tmax,
                   double alpha, int32_t scope, int32_t n_min,
                   const int64_t *global_counts, double *w)
{
    if (scope != OR_SCOPE_TRAJ && scope != OR_SCOPE_BATCH)
        return OR_SHAPE;
    int32_t *n_bt = (int32_t *)malloc(sizeof(int32_t) * ((size_t)B * Tmax + 1));
    int64_t *counts = (int64_t *)malloc(sizeof(int64_t) * (size_t)(2 * Tmax + 1));
    int st = oracle_turn_counts(turn_id, mask, off, B, T, Tmax, n_bt, counts);
    if (st) {
        free(n_bt);
        free(counts);
        return st;
    }
    const int64_t *g = global_counts ? global_counts : counts;
    const int64_t *S = g;            /* survivors per turn index */
    const int64_t *C = g + Tmax;     /* tokens per turn index    */
    const int64_t Bp = g[2 * Tmax];  /* non-empty trajectories   */

    for (int64_t i = 0; i < T; ++i)
        w[i] = 0.0;

    if (scope == OR_SCOPE_TRAJ) {
        for (int32_t b = 0; b < B; ++b) {
            const int32_t *nb = n_bt + (int64_t)b * Tmax;
            int64_t Nb = 0, Ub = 0, Rb = 0;
            for (int32_t t = 0; t < Tmax; ++t) {
                Nb += nb[t];
                int reliable = (n_min <= 0) || (S[t] >= n_min);
                if (!reliable)
                    Ub += nb[t];
                else if (nb[t] > 0)
                    Rb += 1;
            }
            if (Nb == 0 || Bp == 0)
                continue;
            for (int64_t i = off[b]; i < off[b + 1]; ++i) {
                if (!mask[i])
                    continue;
                int32_t t = turn_id[i];
                int reliable = (n_min <= 0) || (S[t] >= n_min);
                double w_traj = 1.0 / (double)Nb;
                double w_turn;
                if (!reliable || Rb == 0)
                    w_turn = 1.0 / (double)Nb;
                else
                    w_turn = (1.0 - (double)Ub / (double)Nb) / ((double)Rb * (double)nb[t]);
                w[i] = ((1.0 - alpha) * w_traj + alpha * w_turn) / (double)Bp;
            }
        }
    } else {
        int64_t N = 0, U = 0, R = 0;
        for (int32_t t = 0; t < Tmax; ++t) {
            N += C[t];
            int reliable = (n_min <= 0) || (S[t] >= n_min);
            if (!reliable)
                U += C[t];
            else
                R += S[t];
        }
        if (N > 0) {
            for (int32_t b = 0; b < B; ++b) {
                const int32_t *nb = n_bt + (int64_t)b * Tmax;
                for (int64_t i = off[b]; i < off[b + 1]; ++i) {
                    if (!mask[i])
                        continue;
                    int32_t t = turn_id[i];
                    int reliable = (n_min <= 0) || (S[t] >= n_min);
                    double w_traj = 1.0 / (double)N;
                    double w_turn;
                    if (!reliable || R == 0)
                        w_turn = 1.0 / (double)N;
                    else
                        w_turn = (1.0 - (double)U / (double)N) / ((double)R * (double)nb[t]);
                    w[i] = (1.0 - alpha) * w_traj + alpha * w_turn;
                }
            }
        }
    }
    free(n_bt);
    free(counts);
    return OR_OK;
}

/* ---- one logit row ------------------------------------------------------ */

/*
 * For one token with student logits zs[0..V) and teacher logits zt[0..V),
 * both already in double:
 *   LSE = m + log sum_v exp(z_v - m),  m = max_v z_v      (each model)
 *   ls_v = zs_v - LSE_s,  lt_v = zt_v - LSE_t,  p_v = exp(ls_v)
 * full vocabulary:  l = KL(p_s || p_t) = sum_v p_v (ls_v - lt_v)
 *                   g_v = w p_v (ls_v - lt_v - l)          (= w dKL/dzs_v)
 * sampled token y:  l = ls_y - lt_y
 *                   g_v = w l (delta_{v,y} - p_v)          (score function),
 *                   with 1 - p_y taken as sum_{v != y} p_v (equal, as the p_v sum
 *                   to 1, and free of the cancellation of 1 - p_y near p_y = 1)
 * out[0] = LSE_s, out[1] = LSE_t, out[2] = l, out[3] = full-vocab KL.
 * g (nullable) receives V doubles.
 */
static int row_core(const double *zs, const double *zt, int64_t V, int32_t mode,
                    int32_t y, double w, double *out, double *g)
{
    if (mode == OR_SAMPLED_TOKEN && (y < 0 || y >= V))
        return OR_TOKEN_RANGE;
    double ms = -INFINITY, mt = -INFINITY;
    for (int64_t v = 0; v < V; ++v) {
        if (!isfinite(zs[v]) || !isfinite(zt[v]))
            return OR_NONFINITE;
        if (zs[v] > ms)
            ms = zs[v];
        if (zt[v] > mt)
            mt = zt[v];
    }
    kahan_t ss = {0, 0}, st = {0, 0};
    for (int64_t v = 0; v < V; ++v) {
        kadd(&ss, exp(zs[v] - ms));
        kadd(&st, exp(zt[v] - mt));
    }
    double lse_s = ms + log(kval(&ss));
    double lse_t = mt + log(kval(&st));
    kahan_t kl = {0, 0};
    for (int64_t v = 0; v < V; ++v) {
        double ls = zs[v] - lse_s;
        double lt = zt[v] - lse_t;
        kadd(&kl, exp(ls) * (ls - lt));
    }
    double KL = kval(&kl);
    double ell;
    if (mode == OR_FULL_VOCAB)
        ell = KL;
    else
        ell = (zs[y] - lse_s) - (zt[y] - lse_t);
    if (g) {
        kahan_t rest = {0, 0};  /* sampled token: 1 - p_y = sum_{v != y} p_v */
        if (mode == OR_SAMPLED_TOKEN)
            for (int64_t v = 0; v < V; ++v)
                if (v != y)
                    kadd(&rest, exp(zs[v] - lse_s));
        for (int64_t v = 0; v < V; ++v) {
            double ls = zs[v] - lse_s;
            double lt = zt[v] - lse_t;
            double p = exp(ls);
            if (mode == OR_FULL_VOCAB)
                g[v] = w * p * (ls - lt - KL);
            else
                g[v] = v == y ? w * ell * kval(&rest) : -w * ell * p;
        }
    }
    out[0] = lse_s;
    out[1] = lse_t;
    out[2] = ell;
    out[3] = KL;
    return OR_OK;
}

/* The same row, from fp32 or bf16 logits widened exactly to double. */
int oracle_row(const void *zs, const void *zt, int32_t dtype, int64_t V,
               int32_t mode, int32_t y, double w, double *out, double *g)
{
    if (V < 1)
        return OR_SHAPE;
    double *a = (double *)malloc(sizeof(double) * (size_t)V);
    double *b = (double *)malloc(sizeof(double) * (size_t)V);
    for (int64_t v = 0; v < V; ++v) {
        a[v] = elem(zs, dtype, v);
        b[v] = elem(zt, dtype, v);
    }
    int st = row_core(a, b, V, mode, y, w, out, g);
    free(a);
    free(b);
    return st;
}

/* ---- the loss over a packed batch --------------------------------------- */

/*
 * Token i is supervised iff mask[i] = 1.  Its logit row is row_of_token[i]
 * (or i when row_of_token is NULL), rows are ld elements apart.
 * token_loss[i] = l_i (0 for masked tokens); *loss = sum_i w_i l_i summed in
 * token order with compensation.  grad (nullable) is a dense [num_rows, V]
 * double array, zero-filled first; rows of supervised tokens receive g.
 * rows_done (nullable) lists the token indices to evaluate; when it is given,
 * only those tokens are computed and *loss covers only them.
 */
int oracle_loss_fwd_bwd(const void *zs, const void *zt, int32_t dtype, int64_t ld,
                        int64_t V, const int32_t *row_of_token, int64_t num_rows,
                        const int32_t *sampled_ids, const uint8_t *mask,
                        const float *w, int64_t T, int32_t mode,
                        double *grad, double *token_loss, double *loss,
                        const int64_t *subset, int64_t n_subset)
{
    if (V < 1 || ld < V || T < 0)
        return OR_SHAPE;
    if (mode == OR_SAMPLED_TOKEN && !sampled_ids)
        return OR_SHAPE;
    if (grad)
        memset(grad, 0, sizeof(double) * (size_t)num_rows * (size_t)V);
    int64_t n = subset ? n_subset : T;
    /* validate first, in token order, so the reported error is deterministic */
    for (int64_t k = 0; k < n; ++k) {
        int64_t i = subset ? subset[k] : k;
        if (i < 0 || i >= T)
            return OR_SHAPE;
        token_loss[i] = 0.0;
        if (!mask[i])
            continue;
        int64_t r = row_of_token ? row_of_token[i] : i;
        if (r < 0 || r >= num_rows)
            return OR_TOKEN_RANGE;
        if (mode == OR_SAMPLED_TOKEN && (sampled_ids[i] < 0 || sampled_ids[i] >= V))
            return OR_TOKEN_RANGE;
    }
    int err = OR_OK;
    size_t esz = dtype == OR_BF16 ? 2 : 4;
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t k = 0; k < n; ++k) {
        int64_t i = subset ? subset[k] : k;
        if (!mask[i])
            continue;
        int64_t r = row_of_token ? row_of_token[i] : i;
        const char *ps = (const char *)zs + (size_t)r * (size_t)ld * esz;
        const char *pt = (const char *)zt + (size_t)r * (size_t)ld * esz;
        double out[4];
        int st = oracle_row(ps, pt, dtype, V, mode,
                            mode == OR_SAMPLED_TOKEN ? sampled_ids[i] : 0,
                            (double)w[i], out, grad ? grad + (size_t)r * (size_t)V : NULL);
        if (st) {
#pragma omp critical
            err = st;
        } else {
            token_loss[i] = out[2];
        }
    }
    if (err)
        return err;
    kahan_t L = {0, 0};
    for (int64_t k = 0; k < n; ++k) {
        int64_t i = subset ? subset[k] : k;
        if (mask[i])
            kadd(&L, (double)w[i] * token_loss[i]);
    }
    *loss = kval(&L);
    return OR_OK;
}

/* ---- per-turn statistics ------------------------------------------------ */

/*
 * traj_turn_sum[b,t] = sum of l_i over supervised tokens of b at turn t,
 * traj_turn_cnt[b,t] = their number n_bt,
 * turn_sum[t] = sum_b traj_turn_sum[b,t], turn_cnt[t] = sum_b n_bt,
 * turn_surv[t] = #{b : n_bt > 0}.
 * K_t of Eq. (observed-turn-kl) is turn_sum[t] / turn_cnt[t].
 */
int oracle_turn_stats(const double *token_loss, const int32_t *turn_id,
                      const uint8_t *mask, const int64_t *off, int32_t B,
                      int64_t T, int32_t Tmax, double *traj_turn_sum,
                      int32_t *traj_turn_cnt, double *turn_sum, int64_t *turn_cnt,
                      int32_t *turn_surv)
{
    if (B < 0 || T < 0 || Tmax < 1)
        return OR_SHAPE;
    int st = check_offsets(off, B, T);
    if (st)
        return st;
    kahan_t *acc = (kahan_t *)calloc((size_t)B * Tmax + 1, sizeof(kahan_t));
    memset(traj_turn_cnt, 0, sizeof(int32_t) * (size_t)B * Tmax);
    for (int32_t b = 0; b < B; ++b) {
        for (int64_t i = off[b]; i < off[b + 1]; ++i) {
            if (!mask[i])
                continue;
            int32_t t = turn_id[i];
            if (t < 0 || t >= Tmax) {
                free(acc);
                return OR_TURN_RANGE;
            }
            kadd(&acc[(int64_t)b * Tmax + t], token_loss[i]);
            traj_turn_cnt[(int64_t)b * Tmax + t] += 1;
        }
    }
    for (int64_t k = 0; k < (int64_t)B * Tmax; ++k)
        traj_turn_sum[k] = kval(&acc[k]);
    for (int32_t t = 0; t < Tmax; ++t) {
        kahan_t s = {0, 0};
        int64_t c = 0;
        int32_t surv = 0;
        for (int32_t b = 0; b < B; ++b) {
            kadd(&s, traj_turn_sum[(int64_t)b * Tmax + t]);
            c += traj_turn_cnt[(int64_t)b * Tmax + t];
            if (traj_turn_cnt[(int64_t)b * Tmax + t] > 0)
                surv += 1;
        }
        turn_sum[t] = kval(&s);
        turn_cnt[t] = c;
        turn_surv[t] = surv;
    }
    free(acc);
    return OR_OK;
}

/* ---- fused LM heads ------------------------------------------------------ */

/*
 * Student logits z_s[v] = sum_k h_s[i,k] W_s[v,k] (d_s terms) and teacher
 * logits z_t[v] = sum_k h_t[i,k] W_t[v,k] (d_t terms), in double from the
 * bf16 inputs, then the row oracle above, then
 *   dh_s[i,k] = sum_v g_v W_s[v,k]            (chain rule through z_s = h_s W_s^T)
 * dh_s rows of masked tokens are 0.  subset (nullable) restricts the tokens
 * that are computed, as in oracle_loss_fwd_bwd.
 */
/*
 * dh_s [T, d_s] receives dL/dh_s (rows of unsupervised tokens 0); dW_s
 * (nullable) [V, d_s] receives dL/dW_s = sum_i g_i^T h_s,i over the evaluated
 * supervised tokens (the chain rule through z_s = h_s W_s^T), each sum taken
 * in increasing token order.
 */
int oracle_fused_lmhead(const uint16_t *h_s, const uint16_t *W_s, int64_t d_s,
                        const uint16_t *h_t, const uint16_t *W_t, int64_t d_t,
                        int64_t V, const uint8_t *mask, const float *w, int64_t T,
                        int32_t mode, const int32_t *sampled_ids, double *dh_s,
                        double *dW_s, double *token_loss, double *loss,
                        const int64_t *subset, int64_t n_subset)
{
    if (V < 1 || d_s < 1 || d_t < 1 || T < 0)
        return OR_SHAPE;
    if (mode == OR_SAMPLED_TOKEN && !sampled_ids)
        return OR_SHAPE;
    int64_t n = subset ? n_subset : T;
    for (int64_t k = 0; k < n; ++k) {
        int64_t i = subset ? subset[k] : k;
        if (i < 0 || i >= T)
            return OR_SHAPE;
        token_loss[i] = 0.0;
        for (int64_t c = 0; c < d_s; ++c)
            dh_s[i * d_s + c] = 0.0;
        if (mask[i] && mode == OR_SAMPLED_TOKEN && (sampled_ids[i] < 0 || sampled_ids[i] >= V))
            return OR_TOKEN_RANGE;
    }
    int err = OR_OK;
    /* per evaluated token, its logit gradient row (kept for dW_s) */
    double *gall = dW_s ? (double *)calloc((size_t)(n > 0 ? n : 1) * (size_t)V, sizeof(double)) : NULL;
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t k = 0; k < n; ++k) {
        int64_t i = subset ? subset[k] : k;
        if (!mask[i])
            continue;
        double *zs = (double *)malloc(sizeof(double) * (size_t)V);
        double *zt = (double *)malloc(sizeof(double) * (size_t)V);
        double *g = gall ? gall + (size_t)k * (size_t)V : (double *)malloc(sizeof(double) * (size_t)V);
        for (int64_t v = 0; v < V; ++v) {
            double a = 0.0, b = 0.0;
            for (int64_t c = 0; c < d_s; ++c)
                a += widen_bf16(h_s[i * d_s + c]) * widen_bf16(W_s[v * d_s + c]);
            for (int64_t c = 0; c < d_t; ++c)
                b += widen_bf16(h_t[i * d_t + c]) * widen_bf16(W_t[v * d_t + c]);
            zs[v] = a;
            zt[v] = b;
        }
        double out[4];
        int st = row_core(zs, zt, V, mode, mode == OR_SAMPLED_TOKEN ? sampled_ids[i] : 0,
                          (double)w[i], out, g);
        if (st) {
#pragma omp critical
            err = st;
            free(zs);
            free(zt);
            if (!gall)
                free(g);
            continue;
        }
        double ell = out[2];
        /* dh_s[i,c] = sum_v g_v W_s[v,c], each sum taken in increasing v */
        double *dh = dh_s + i * d_s;
        for (int64_t v = 0; v < V; ++v)
            for (int64_t c = 0; c < d_s; ++c)
                dh[c] += g[v] * widen_bf16(W_s[v * d_s + c]);
        token_loss[i] = ell;
        free(zs);
        free(zt);
        if (!gall)
            free(g);
    }
    if (err) {
        free(gall);
        return err;
    }
    if (dW_s) {
        /* dW_s[v,c] = sum over evaluated supervised tokens (in order) of g_i[v] h_s[i,c] */
#pragma omp parallel for schedule(dynamic, 16)
        for (int64_t v = 0; v < V; ++v) {
            double *row = dW_s + v * d_s;
            for (int64_t c = 0; c < d_s; ++c)
                row[c] = 0.0;
            for (int64_t k = 0; k < n; ++k) {
                int64_t i = subset ? subset[k] : k;
                if (!mask[i])
                    continue;
                double gv = gall[(size_t)k * (size_t)V + (size_t)v];
                if (gv == 0.0)
                    continue;
                for (int64_t c = 0; c < d_s; ++c)
                    row[c] += gv * widen_bf16(h_s[i * d_s + c]);
            }
        }
        free(gall);
    }
    kahan_t L = {0, 0};
    for (int64_t k = 0; k < n; ++k) {
        int64_t i = subset ? subset[k] : k;
        if (mask[i])
            kadd(&L, (double)w[i] * token_loss[i]);
    }
    *loss = kval(&L);
    return OR_OK;
}

/* ---- teacher top-K reverse KL -------------------------------------------- */

/* order of the support: larger teacher logit first, lower id among equals */
typedef struct { double zt; int64_t id; } topk_ent_t;
static int topk_cmp(const void *a, const void *b)
{
    const topk_ent_t *x = (const topk_ent_t *)a, *y = (const topk_ent_t *)b;
    if (x->zt > y->zt) return -1;
    if (x->zt < y->zt) return 1;
    return x->id < y->id ? -1 : (x->id > y->id ? 1 : 0);
}

/*
 * One row.  S = the first K ids in the order above.  On S:
 *   ps_v = exp(zs_v) / sum_{u in S} exp(zs_u),  pt_v likewise from zt,
 *   l    = sum_{v in S} ps_v (log ps_v - log pt_v)
 *   g_v  = w ps_v (log ps_v - log pt_v - l)        (= w dl/dzs_v; 0 off S)
 * ids[K] receives S in order, gk[K] the g of those ids (both nullable);
 * g (nullable) receives all V entries (0 off S).
 */
static int topk_core(const double *zs, const double *zt, int64_t V, int32_t K, double w,
                     int32_t *ids, double *gk, double *g, double *ell)
{
    if (K < 1 || K > V)
        return OR_SHAPE;
    topk_ent_t *e = (topk_ent_t *)malloc(sizeof(topk_ent_t) * (size_t)V);
    for (int64_t v = 0; v < V; ++v) {
        if (!isfinite(zs[v]) || !isfinite(zt[v])) {
            free(e);
            return OR_NONFINITE;
        }
        e[v].zt = zt[v];
        e[v].id = v;
    }
    qsort(e, (size_t)V, sizeof(topk_ent_t), topk_cmp);
    double ms = -INFINITY, mt = -INFINITY;
    for (int32_t r = 0; r < K; ++r) {
        int64_t v = e[r].id;
        if (zs[v] > ms) ms = zs[v];
        if (zt[v] > mt) mt = zt[v];
    }
    kahan_t ss = {0, 0}, st = {0, 0};
    for (int32_t r = 0; r < K; ++r) {
        int64_t v = e[r].id;
        kadd(&ss, exp(zs[v] - ms));
        kadd(&st, exp(zt[v] - mt));
    }
    double lse_s = ms + log(kval(&ss)), lse_t = mt + log(kval(&st));
    kahan_t kl = {0, 0};
    for (int32_t r = 0; r < K; ++r) {
        int64_t v = e[r].id;
        double ls = zs[v] - lse_s, lt = zt[v] - lse_t;
        kadd(&kl, exp(ls) * (ls - lt));
    }
    double l = kval(&kl);
    if (g)
        for (int64_t v = 0; v < V; ++v)
            g[v] = 0.0;
    for (int32_t r = 0; r < K; ++r) {
        int64_t v = e[r].id;
        double ls = zs[v] - lse_s, lt = zt[v] - lse_t;
        double gv = w * exp(ls) * (ls - lt - l);
        if (ids) ids[r] = (int32_t)v;
        if (gk) gk[r] = gv;
        if (g) g[v] = gv;
    }
    *ell = l;
    free(e);
    return OR_OK;
}

int oracle_topk_row(const void *zs, const void *zt, int32_t dtype, int64_t V, int32_t K,
                    double w, int32_t *ids, double *gk, double *g, double *ell)
{
    if (V < 1)
        return OR_SHAPE;
    double *a = (double *)malloc(sizeof(double) * (size_t)V);
    double *b = (double *)malloc(sizeof(double) * (size_t)V);
    for (int64_t v = 0; v < V; ++v) {
        a[v] = elem(zs, dtype, v);
        b[v] = elem(zt, dtype, v);
    }
    int st = topk_core(a, b, V, K, w, ids, gk, g, ell);
    free(a);
    free(b);
    return st;
}

/*
 * The top-K loss over a packed batch (same conventions as
 * oracle_loss_fwd_bwd): token_loss[i] = l_i, *loss = sum_i w_i l_i in token
 * order, topk_ids / topk_g [T, K] (nullable) hold S and its g for supervised
 * tokens (untouched otherwise), grad (nullable) a dense [num_rows, V] array.
 */
int oracle_topk_loss(const void *zs, const void *zt, int32_t dtype, int64_t ld, int64_t V,
                     const int32_t *row_of_token, int64_t num_rows, const uint8_t *mask,
                     const float *w, int64_t T, int32_t K, int32_t *topk_ids, double *topk_g,
                     double *grad, double *token_loss, double *loss,
                     const int64_t *subset, int64_t n_subset)
{
    if (V < 1 || ld < V || T < 0 || K < 1 || K > V)
        return OR_SHAPE;
    if (grad)
        memset(grad, 0, sizeof(double) * (size_t)num_rows * (size_t)V);
    int64_t n = subset ? n_subset : T;
    for (int64_t k = 0; k < n; ++k) {
        int64_t i = subset ? subset[k] : k;
        if (i < 0 || i >= T)
            return OR_SHAPE;
        token_loss[i] = 0.0;
        if (!mask[i])
            continue;
        int64_t r = row_of_token ? row_of_token[i] : i;
        if (r < 0 || r >= num_rows)
            return OR_TOKEN_RANGE;
    }
    int err = OR_OK;
    size_t esz = dtype == OR_BF16 ? 2 : 4;
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t k = 0; k < n; ++k) {
        int64_t i = subset ? subset[k] : k;
        if (!mask[i])
            continue;
        int64_t r = row_of_token ? row_of_token[i] : i;
        const char *ps = (const char *)zs + (size_t)r * (size_t)ld * esz;
        const char *pt = (const char *)zt + (size_t)r * (size_t)ld * esz;
        double l = 0.0;
        int st = oracle_topk_row(ps, pt, dtype, V, K, (double)w[i],
                                 topk_ids ? topk_ids + (size_t)i * (size_t)K : NULL,
                                 topk_g ? topk_g + (size_t)i * (size_t)K : NULL,
                                 grad ? grad + (size_t)r * (size_t)V : NULL, &l);
        if (st) {
#pragma omp critical
            err = st;
        } else {
            token_loss[i] = l;
        }
    }
    if (err)
        return err;
    kahan_t L = {0, 0};
    for (int64_t k = 0; k < n; ++k) {
        int64_t i = subset ? subset[k] : k;
        if (mask[i])
            kadd(&L, (double)w[i] * token_loss[i]);
    }
    *loss = kval(&L);
    return OR_OK;
}

/* ---- blend schedule ------------------------------------------------------ */

/* alpha_k = clip((k/K - s)/(e - s), 0, 1), progress k/K (Sec. 5.2). */
double oracle_alpha_schedule(int64_t k, int64_t K, double s, double e)
{
    double progress = (double)k / (double)K;
    double a = (progress - s) / (e - s);
    if (a < 0.0)
        a = 0.0;
    if (a > 1.0)
        a = 1.0;
    return a;
}

/* Threads the OpenMP loops above use (1 when built without OpenMP). */
int oracle_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
