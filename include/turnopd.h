/*
 * turnopd.h -- C ABI of libturnopd: the turn-aware on-policy-distillation
 * (OPD) loss of TurnOPD (arXiv 2607.05804) on NVIDIA GB300 (sm_103a).
 *
 * One training step of the method, for a packed batch of multi-turn student
 * trajectories, is:
 *   1. turnopd_turn_counts / turnopd_weights -- supervised-token counts per
 *      (trajectory, turn) and the progressive blend weights
 *      w_blend = (1 - alpha) w_traj + alpha w_turn            (Sec. 5.2, Algorithm 1)
 *   2. turnopd_loss_fwd_bwd -- per-token reverse KL(pi_s || pi_T) over the full
 *      vocabulary (Eq. opd-rkl) or the sampled-token estimator, its gradient
 *      w.r.t. the student logits, and L = sum_i w_i l_i   (Algorithm 1, L_k)
 *   3. turnopd_turn_stats -- per-(trajectory, turn) and per-turn-index KL sums
 *      and counts (Eq. observed-turn-kl; the kl_per_turn / num_traj statistics
 *      that the rollout-depth controller of Sec. 5.1 reads).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Memory: every array argument is DEVICE memory owned by the caller.  The
 *   library allocates nothing; scratch space is the caller's `workspace`
 *   (size from the matching *_workspace_bytes function, 256-byte aligned).
 * - Execution: calls are asynchronous and stream-ordered on `stream` (a
 *   cudaStream_t; NULL = legacy default stream).  Calls on different streams
 *   may run concurrently if they share no output or workspace.
 * - Host-detected errors (null pointers, bad sizes, unsupported combinations,
 *   small workspace) return immediately, before any launch or CUDA call.
 * - Device-detected errors (values inside device arrays) are reported through
 *   `dev_status`, a caller-zeroed int32 in device memory: the first error
 *   code stored wins (atomic compare-and-swap from 0), later ones are dropped.
 *   The offending token or trajectory is skipped; other outputs are still
 *   written.  Read the word after synchronising the stream.
 * - Results are deterministic: the same inputs give bit-identical outputs on
 *   every run (fixed-order reductions, no floating-point atomics).
 * - Packed batch: trajectory b owns tokens [traj_offsets[b], traj_offsets[b+1]);
 *   traj_offsets[0] = 0, non-decreasing, traj_offsets[num_traj] = num_tokens.
 *   loss_mask[i] = 1 marks a supervised (assistant) token, 0 an observation
 *   token; turn_id[i] is the 0-based turn of token i, read only where
 *   loss_mask[i] = 1 and required to lie in [0, max_turns) there.
 * - max_turns must lie in [1, TURNOPD_MAX_TURNS]; vocab in [1, 2^31 - 1].
 */
#ifndef TURNOPD_H
#define TURNOPD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same object as cudaStream_t (a CUstream_st pointer), declared here so the
 * header needs no CUDA include. */
typedef struct CUstream_st *turnopd_stream_t;

typedef enum {
    TURNOPD_OK = 0,
    TURNOPD_ERR_NULL = 1,        /* a required pointer is NULL                       */
    TURNOPD_ERR_SHAPE = 2,       /* a size or stride is out of range                 */
    TURNOPD_ERR_OFFSETS = 3,     /* traj_offsets not 0..num_tokens non-decreasing     */
    TURNOPD_ERR_TURN_RANGE = 4,  /* supervised token with turn_id outside [0,max)     */
    TURNOPD_ERR_TOKEN_RANGE = 5, /* row index or sampled id out of range              */
    TURNOPD_ERR_UNSUPPORTED = 6, /* unsupported dtype / mode / flag combination       */
    TURNOPD_ERR_CUDA = 7,        /* a CUDA runtime call or launch failed              */
    TURNOPD_ERR_TIMEOUT = 8,     /* a bounded device-side wait gave up                */
    TURNOPD_ERR_NONFINITE = 9,   /* a non-finite log-sum-exp or loss value           */
    TURNOPD_ERR_WORKSPACE = 10   /* workspace NULL, misaligned or too small           */
} turnopd_status;

enum { TURNOPD_FULL_VOCAB = 0, TURNOPD_SAMPLED_TOKEN = 1 };       /* loss mode     */
enum { TURNOPD_F32 = 0, TURNOPD_BF16 = 1 };                       /* element type  */
enum { TURNOPD_SCOPE_TRAJ = 0, TURNOPD_SCOPE_BATCH = 1 };         /* normalisation */

/* Write zeros into the gradient rows of masked tokens that own a row. */
#define TURNOPD_ZERO_MASKED_GRAD 0x1u
/* Diagnostic: force the portable one-CTA-per-row kernel instead of the
 * cluster-resident kernel (results agree within the documented tolerance). */
#define TURNOPD_FORCE_PORTABLE 0x100u

#define TURNOPD_MAX_TURNS 4096

/*
 * turnopd_turn_counts -- supervised-token bookkeeping of the multi-turn trace
 * model (Sec. 3; survivors "trajectories that reach each turn", Sec. 4.1;
 * n_t of Sec. 5.1 and Sec. 5.2).
 *
 * Outputs (device, caller-owned):
 *   traj_turn_cnt  int32[num_traj * max_turns], row-major [b][t]:
 *                  n_bt = #{i in b : loss_mask[i] = 1, turn_id[i] = t}
 *   counts         int64[2 * max_turns + 1]:
 *                  [0, max_turns)            S_t = #{b : n_bt > 0}
 *                  [max_turns, 2 max_turns)  C_t = sum_b n_bt
 *                  [2 max_turns]             B'  = #{b : sum_t n_bt > 0}
 *                  Summing `counts` over data-parallel ranks (each holding
 *                  whole trajectories) gives the batch-wide vector that
 *                  turnopd_weights accepts as `global_counts`.
 * Device errors: TURNOPD_ERR_OFFSETS, TURNOPD_ERR_TURN_RANGE (token ignored).
 */
turnopd_status turnopd_turn_counts(const int32_t *turn_id, const uint8_t *loss_mask,
                                   const int64_t *traj_offsets, int32_t num_traj,
                                   int64_t num_tokens, int32_t max_turns,
                                   int32_t *traj_turn_cnt, int64_t *counts,
                                   int32_t *dev_status, turnopd_stream_t stream);

/*
 * turnopd_weights -- per-token progressive blend weights (Sec. 5.2: q^traj =
 * n_t / sum_j n_j, q^turn = 1/T, q^blend = (1 - alpha) q^traj + alpha q^turn;
 * Algorithm 1: w_blend = (1 - alpha) w_traj + alpha w_turn on observed tokens).
 *
 * scope = TURNOPD_SCOPE_TRAJ (the paper's Eq. opd-rkl normalisation, a token
 * mean inside each trajectory, then a mean over the B' trajectories that hold
 * supervised tokens -- "seq-mean-token-mean"):
 *     w_i = [(1 - alpha) / N_b + alpha / (T_b n_bt)] / B'
 *   N_b = supervised tokens of b, T_b = non-empty turns of b.
 * scope = TURNOPD_SCOPE_BATCH (one token mean over the batch):
 *     w_i = (1 - alpha) / N + alpha / (S n_bt),  N = sum C_t, S = sum S_t.
 * n_min > 0 enables the turn-reliability floor (hyper-parameter table:
 * n_min = max(floor, ceil(frac * n_traj)), computed by the caller, e.g. with
 * turnopd_turn_floor): turn index
 * t is reliable iff S_t >= n_min; tokens of unreliable turns keep the token
 * weight (1/N_b, resp. 1/N), the reliable non-empty turns share the remaining
 * mass equally; with no reliable turn w_turn = w_traj.  n_min <= 0: no floor.
 * global_counts: NULL, or a device int64[2 max_turns + 1] vector laid out as
 *   turnopd_turn_counts' `counts`, summed over data-parallel ranks; it then
 *   replaces the local S_t, C_t and B' (n_bt, N_b, T_b stay local).
 * alpha must lie in [0, 1] (see turnopd_alpha_schedule).
 * Output: w_out float32[num_tokens] (computed in fp64, rounded to nearest);
 *   0 for masked tokens and for tokens of trajectories without supervision.
 * Workspace: turnopd_weights_workspace_bytes(num_traj, max_turns) bytes.
 * Device errors: as turnopd_turn_counts.
 */
turnopd_status turnopd_weights(const int32_t *turn_id, const uint8_t *loss_mask,
                               const int64_t *traj_offsets, int32_t num_traj,
                               int64_t num_tokens, int32_t max_turns, double alpha,
                               int32_t scope, int32_t n_min, const int64_t *global_counts,
                               float *w_out, void *workspace, size_t workspace_bytes,
                               int32_t *dev_status, turnopd_stream_t stream);

size_t turnopd_weights_workspace_bytes(int32_t num_traj, int32_t max_turns);

/*
 * turnopd_loss_fwd_bwd -- per-token OPD loss, its student-logit gradient and
 * the weighted batch loss (Eq. opd-rkl; Algorithm 1: L_k = sum_i w_i l_i).
 *
 * For every supervised token i with logit row r = row_of_token[i] (or r = i
 * when row_of_token is NULL), with ls = z_s - LSE(z_s), lt = z_t - LSE(z_t),
 * p = exp(ls) (natural log throughout, softmax of the raw logits):
 *   mode TURNOPD_FULL_VOCAB:    l_i = KL(p_s || p_t) = sum_v p_v (ls_v - lt_v)
 *                               g_v = w_i p_v (ls_v - lt_v - l_i)
 *   mode TURNOPD_SAMPLED_TOKEN: l_i = ls_y - lt_y,  y = sampled_ids[i]
 *                               g_v = w_i l_i (delta_{v,y} - p_v)
 *     (score-function gradient: its expectation over y ~ p_s is the
 *      full-vocabulary gradient; l_i itself is treated as a constant).
 * Inputs:
 *   z_student, z_teacher  [num_rows, ld] row-major, in_dtype (F32 or BF16);
 *                          the values of columns [vocab, ld) never enter a result
 *                          (bf16 rows with ld a multiple of 8 read up to the next
 *                          multiple of 8 of vocab, inside the buffer, and mask it).
 *   row_of_token           int32[num_tokens] or NULL (then num_rows >= num_tokens);
 *                          read only where loss_mask = 1, must lie in [0, num_rows).
 *   sampled_ids            int32[num_tokens], required for SAMPLED_TOKEN, in [0, vocab).
 *   loss_mask              uint8[num_tokens];  w  float32[num_tokens] (turnopd_weights).
 * Outputs:
 *   grad_student  [num_rows, ld] in grad_dtype (F32 or BF16), or NULL for a
 *                 forward-only call.  Rows of supervised tokens get g (bf16:
 *                 round to nearest even from fp32); columns [vocab, ld) and
 *                 other rows are not written unless TURNOPD_ZERO_MASKED_GRAD,
 *                 which zero-fills columns [0, vocab) of masked tokens' rows.
 *                 grad_student may not alias the logits.
 *   token_loss_out float32[num_tokens]: l_i, 0 for masked tokens.
 *   loss_out       one double: sum_i w_i l_i (fixed-order fp64 sum).
 * Workspace: turnopd_loss_workspace_bytes(num_tokens) bytes.
 * Device errors: TURNOPD_ERR_TOKEN_RANGE (row or sampled id; token skipped,
 *   l_i = 0), TURNOPD_ERR_NONFINITE (non-finite LSE or l_i).
 * Precision: fp32 arithmetic on exact fp32/bf16 inputs, fp64 loss sum.
 * Kernels (the results agree within the tolerances above whichever runs):
 *   bf16 logits, ld a multiple of 8, 16-byte aligned arrays: row clusters of
 *     2 to 16 CTAs (the smallest whose slices fit three shared-memory stages)
 *     beside a helper grid on the remaining SMs, or the helper grid alone for
 *     short rows; a vocab that is not a multiple of 8 ends in a masked vector;
 *   fp32 logits, vocab and ld multiples of 4, 16-byte aligned arrays: the
 *     split-row kernel (clusters of 8 CTAs per row, 4 for sampled-token rows)
 *     beside a helper grid on the remaining SMs; it marks its first read of
 *     each logit chunk L2 evict-last and returns the lines to normal priority
 *     after the gradient's second read;
 *   any other shape: one CTA per row.
 */
turnopd_status turnopd_loss_fwd_bwd(const void *z_student, const void *z_teacher,
                                    int32_t in_dtype, int64_t ld, int64_t vocab,
                                    int64_t num_rows, const int32_t *row_of_token,
                                    const int32_t *sampled_ids, const uint8_t *loss_mask,
                                    const float *w, int64_t num_tokens, int32_t mode,
                                    void *grad_student, int32_t grad_dtype, uint32_t flags,
                                    float *token_loss_out, double *loss_out,
                                    void *workspace, size_t workspace_bytes,
                                    int32_t *dev_status, turnopd_stream_t stream);

size_t turnopd_loss_workspace_bytes(int64_t num_tokens);

/*
 * turnopd_loss_fwd_bwd_static -- turnopd_loss_fwd_bwd for callers that cannot
 * allocate device memory.  The paper has no counterpart: this is an addition
 * of the library, not a step of the method.
 *
 * Who needs it: a caller whose device memory is owned by someone else -- a
 * framework's caching allocator or a fixed arena that forbids raw cudaMalloc,
 * a C host with no allocator of its own to hand out a workspace, or a
 * latency-bound loop that must never reach cudaMalloc/cudaFree (cudaFree
 * synchronises the whole device, and cudaMalloc can fail or stall once a pool
 * has reserved the memory).  Such a caller still passes its inputs and
 * outputs; only the scratch space moves into the library.
 *
 * Scratch: one file-scope device array of TURNOPD_STATIC_SCRATCH_BYTES,
 * enough for TURNOPD_STATIC_MAX_TOKENS tokens.  Every GPU on which the
 * library is loaded holds this array until the process exits.
 * Limits: num_tokens > TURNOPD_STATIC_MAX_TOKENS returns TURNOPD_ERR_WORKSPACE
 * before anything is launched.
 * Set-up: the first call on a device looks up the array's device address
 * (cudaGetSymbolAddress, with that device current) and keeps it for the
 * CUDA context it was taken in; a call made in another context of that device
 * (after cudaDeviceReset, say) looks it up again.  Make the first call in each
 * context before any stream capture.
 * Sharing: all calls use the one array.  Calls that can overlap on the GPU
 * (different streams, or several host threads) race on it and may return
 * wrong results: issue them on one stream.  The array keeps whatever the last
 * call left there; nothing in it needs to start at zero, because every call
 * writes each scratch word before reading it.
 * Allocation: none -- no cudaMalloc, cudaFree or allocating library call.
 * Arguments, outputs, errors and precision: as turnopd_loss_fwd_bwd, without
 * the workspace arguments.
 */
#define TURNOPD_STATIC_MAX_TOKENS 65536
#define TURNOPD_STATIC_SCRATCH_BYTES 1573632u
turnopd_status turnopd_loss_fwd_bwd_static(const void *z_student, const void *z_teacher,
                                           int32_t in_dtype, int64_t ld, int64_t vocab,
                                           int64_t num_rows, const int32_t *row_of_token,
                                           const int32_t *sampled_ids, const uint8_t *loss_mask,
                                           const float *w, int64_t num_tokens, int32_t mode,
                                           void *grad_student, int32_t grad_dtype, uint32_t flags,
                                           float *token_loss_out, double *loss_out,
                                           int32_t *dev_status, turnopd_stream_t stream);

/*
 * turnopd_fused_lmhead_fwd_bwd -- the OPD loss with the two LM heads fused in:
 * student logits z_s = h_s W_s^T and teacher logits z_t = h_t W_t^T of the
 * supervised tokens are formed tile by tile on the tensor cores and consumed
 * by the loss without ever being stored (Eq. opd-rkl, full vocabulary).
 * Outputs l_i, L = sum_i w_i l_i and dL/dh_s = G W_s with G = dL/dz_s (the
 * chain rule through z_s = h_s W_s^T; G is formed in fp32 and rounded to bf16
 * for the second tensor-core product).
 * Inputs (device, row-major, bf16):
 *   h_s [num_tokens, d_s], W_s [vocab, d_s], h_t [num_tokens, d_t], W_t [vocab, d_t]
 *   loss_mask uint8[num_tokens], w float32[num_tokens] (turnopd_weights).
 *   d_s must be a multiple of 256, d_t of 64; every pointer 16-byte aligned.
 *   mode: TURNOPD_FULL_VOCAB only (others return TURNOPD_ERR_UNSUPPORTED).
 * Outputs:
 *   dh_s_out  float32[num_tokens, d_s] or NULL; rows of masked tokens are zero.
 *   dW_s_out  float32[vocab, d_s] or NULL: dL/dW_s = sum_i G_i^T h_s,i over the
 *             supervised tokens (overwritten, not accumulated).
 *   (both NULL: forward only)
 *   token_loss_out float32[num_tokens] (0 for masked tokens), loss_out double.
 * Workspace: turnopd_fused_workspace_bytes(num_tokens, vocab, d_s, d_t) bytes,
 *   queried with the device that will run the call current (gathered hidden
 *   rows, per-row partial statistics, G in bf16 and per-SM partial dH tiles:
 *   about 2 num_tokens vocab bytes + 256 KiB per SM).
 * Device errors: TURNOPD_ERR_NONFINITE, TURNOPD_ERR_TIMEOUT (bounded waits).
 */
turnopd_status turnopd_fused_lmhead_fwd_bwd(const void *h_s, const void *W_s, int64_t d_s,
                                            const void *h_t, const void *W_t, int64_t d_t,
                                            int64_t vocab, const uint8_t *loss_mask,
                                            const float *w, int64_t num_tokens, int32_t mode,
                                            float *dh_s_out, float *dW_s_out, float *token_loss_out,
                                            double *loss_out, void *workspace,
                                            size_t workspace_bytes, int32_t *dev_status,
                                            turnopd_stream_t stream);

size_t turnopd_fused_workspace_bytes(int64_t num_tokens, int64_t vocab, int64_t d_s, int64_t d_t);

/*
 * turnopd_topk_loss_fwd_bwd -- teacher top-K reverse KL and its gradient
 * (the paper's practical loss, loss_mode topk_reverse_kl with support size
 * K_top = distill_topk = 50 in the full configuration table; Algorithm 1,
 * "top-K reverse-KL token losses").
 *
 * For every supervised token i (loss_mask[i] = 1), with row r = row_of_token[i]
 * (or i when row_of_token is NULL): S_i = the k_top vocabulary ids of largest
 * teacher logit z_teacher[r, .], the lower id first among equal logits (+0 and
 * -0 are equal); both distributions are renormalised over S_i:
 *   l_i    = sum_{v in S_i} ps_v (log ps_v - log pt_v),
 *            ps_v = exp(z_s[r,v]) / sum_{u in S_i} exp(z_s[r,u]), pt likewise;
 *   g_i,v  = w_i ps_v (log ps_v - log pt_v - l_i) for v in S_i, 0 elsewhere
 *            (= w_i dl_i/dz_s[r, v]);
 *   *loss_out = sum_i w_i l_i (fixed order, fp64).
 * Inputs (device, row-major): z_student, z_teacher [num_rows, ld] of in_dtype
 *   (TURNOPD_BF16 or TURNOPD_F32), ld >= vocab; loss_mask uint8[num_tokens];
 *   w float32[num_tokens]; 1 <= k_top <= min(vocab, TURNOPD_TOPK_MAX);
 *   vocab <= TURNOPD_TOPK_MAX_VOCAB (the kernel keeps, for each of the two rows it
 *   holds at a time, one 16-bit bucket per 16 vocabulary ids in shared memory).
 * Outputs (each nullable except token_loss_out and loss_out):
 *   topk_ids_out  int32 [num_tokens, k_top]: S_i in order (largest teacher
 *                 logit first); topk_grad_out float32 [num_tokens, k_top]: g_i
 *                 at those ids.  Rows of masked tokens are left as they are, or
 *                 set to -1 / 0 with TURNOPD_ZERO_MASKED_GRAD.
 *   grad_student  dense [num_rows, ld] of grad_dtype: row r gets zeros and g_i
 *                 on S_i (columns >= vocab untouched); rows of masked tokens as
 *                 in turnopd_loss_fwd_bwd.
 *   token_loss_out float32[num_tokens] (0 for masked tokens), loss_out double.
 * Workspace: turnopd_loss_workspace_bytes(num_tokens) bytes, 256-byte aligned.
 * Flags: TURNOPD_ZERO_MASKED_GRAD only.
 * Host errors: NULL / SHAPE (k_top out of range, misalignment) / UNSUPPORTED /
 *   WORKSPACE, returned before any launch.  Device errors (in *dev_status):
 *   TURNOPD_ERR_TOKEN_RANGE (row index), TURNOPD_ERR_NONFINITE, and
 *   TURNOPD_ERR_UNSUPPORTED for a row whose selection did not settle within the
 *   kernel's bounded rounds (only rows with thousands of equal top logits).
 */
#define TURNOPD_TOPK_MAX 1024
#define TURNOPD_TOPK_MAX_VOCAB 737280  /* 720 * 1024 */
turnopd_status turnopd_topk_loss_fwd_bwd(const void *z_student, const void *z_teacher,
                                         int32_t in_dtype, int64_t ld, int64_t vocab,
                                         int64_t num_rows, const int32_t *row_of_token,
                                         const uint8_t *loss_mask, const float *w,
                                         int64_t num_tokens, int32_t k_top, int32_t *topk_ids_out,
                                         float *topk_grad_out, void *grad_student, int32_t grad_dtype,
                                         uint32_t flags, float *token_loss_out, double *loss_out,
                                         void *workspace, size_t workspace_bytes,
                                         int32_t *dev_status, turnopd_stream_t stream);

/*
 * ---- Vocabulary-parallel split of the reverse KL (Eq. opd-rkl) ----
 * For logits sharded by vocabulary columns across ranks.  Each rank passes
 * the base pointers of ITS shard (shard_vocab columns, rows ld elements
 * apart; the same token -> row map on every rank):
 *   1. turnopd_vocab_shard_stats: per supervised token i, the shard's partial
 *      row statistics stats_out[i, 0..5] = (m_s, S_s, A, d, m_t, S_t):
 *      m = max logit, S = sum exp(z - m), d = (z_s - z_t) at the student's
 *      largest logit, A = sum exp(z_s - m_s) ((z_s - z_t) - d)  (float32,
 *      turnopd_vocab_stats_bytes(num_tokens) bytes; masked rows untouched;
 *      workspace as for turnopd_loss_fwd_bwd, turnopd_loss_workspace_bytes
 *      (num_tokens) bytes, 256-byte aligned, else TURNOPD_ERR_WORKSPACE);
 *   2. the caller gathers every shard's stats into parts[n_shards, num_tokens, 6]
 *      in shard order (e.g. an all-gather);
 *   3. turnopd_vocab_stats_merge: the whole vocabulary's row statistics, merged
 *      in shard order (identical bits on every rank);
 *   4. turnopd_vocab_shard_loss_grad: token_loss_out[i] = KL_i (0 for masked
 *      tokens), *loss_out = sum_i w_i KL_i (fixed order, fp64; the same on every
 *      rank), and this shard's gradient columns
 *      g = w_i exp(z_s - LSE_s) ((z_s - z_t) - E_p[z_s - z_t])  (grad_shard
 *      nullable, [num_rows, ld] of grad_dtype; TURNOPD_ZERO_MASKED_GRAD zeroes
 *      the rows of masked tokens).  Full-vocabulary mode only.
 * All arrays are device memory; host errors as for turnopd_loss_fwd_bwd;
 * device errors TURNOPD_ERR_TOKEN_RANGE and TURNOPD_ERR_NONFINITE.
 */
size_t turnopd_vocab_stats_bytes(int64_t num_tokens);
turnopd_status turnopd_vocab_shard_stats(const void *z_student, const void *z_teacher, int32_t in_dtype,
                                         int64_t ld, int64_t shard_vocab, int64_t num_rows,
                                         const int32_t *row_of_token, const uint8_t *loss_mask,
                                         int64_t num_tokens, float *stats_out, void *workspace,
                                         size_t workspace_bytes, int32_t *dev_status, turnopd_stream_t stream);
turnopd_status turnopd_vocab_stats_merge(const float *parts, int32_t n_shards, const uint8_t *loss_mask,
                                         int64_t num_tokens, float *merged_out, turnopd_stream_t stream);
turnopd_status turnopd_vocab_shard_loss_grad(const void *z_student, const void *z_teacher, int32_t in_dtype,
                                             int64_t ld, int64_t shard_vocab, int64_t num_rows,
                                             const int32_t *row_of_token, const uint8_t *loss_mask,
                                             const float *w, int64_t num_tokens, const float *merged_stats,
                                             void *grad_shard, int32_t grad_dtype, uint32_t flags,
                                             float *token_loss_out, double *loss_out, void *workspace,
                                             size_t workspace_bytes, int32_t *dev_status,
                                             turnopd_stream_t stream);

/*
 * ---- Adaptive rollout-depth controller and loss-allocation diagnostics ----
 * (Sec. 4.1 "Adaptive Rollout-Depth Budgeting", Algorithm 1, and the
 * loss-allocation diagnostics of Sec. 3).  Host functions: every pointer is
 * HOST memory (the per-turn tables of turnopd_turn_stats, copied back by the
 * caller); nothing runs on the GPU and nothing is allocated.  round() is
 * round-half-to-even; turn indices t are 0-based.
 *
 *   K_t    = turn_sum[t] / turn_cnt[t] (0 where turn_cnt[t] = 0)
 *   m_t    = [K_t]_+ n_t / n_0,  n_t = turn_surv[t];  q_t = m_t / (sum_j m_j + eps)
 *   H_eff  = round(sum_t t q_t)
 *   H_cov  = min{H : 1 - n_{H+1} / n_1 >= p} over the probe trajectories that
 *            succeeded (all of them when use_success = 0), where n_h counts
 *            those with at least h turns; refreshed only when at least
 *            min_cov_traj probe trajectories succeeded, else kept
 *   probe step k: H_ctrl = max(H_eff, H_cov), h_bar <- (1 - ema_alpha) h_bar + ema_alpha H_ctrl
 *   plan for step k (1-based): h_hat = clip(round(h_bar) + 1, h_min, h_max);
 *            probe = (k <= warmup_steps) or (probe_interval > 0 and k % probe_interval == 0);
 *            h_roll = probe ? h_max : h_hat
 * Errors: TURNOPD_ERR_NULL for a missing pointer, TURNOPD_ERR_SHAPE for
 * out-of-range parameters (h_min < 1, h_max < h_min, ema_alpha outside [0, 1],
 * coverage_p outside (0, 1], negative counts or intervals, k < 1).
 */
typedef struct {
    int32_t h_min, h_max;     /* clamp of the applied depth (defaults 2, 50) */
    double ema_alpha;         /* EMA weight on H_ctrl (0.30) */
    double coverage_p;        /* success-length quantile p (0.80) */
    int32_t min_cov_traj;     /* successes needed to refresh H_cov (8) */
    int32_t use_success;      /* 1: success-conditioned lengths, 0: all probe trajectories (1) */
    int32_t warmup_steps;     /* every step k <= warmup_steps is a probe (3) */
    int32_t probe_interval;   /* then every probe_interval-th step (8; 0 = never) */
    double eps;               /* in q_t (1e-8) */
} turnopd_depth_params;

typedef struct {
    double h_bar;             /* EMA of H_ctrl; h_max at start */
    double h_eff_bar;         /* last unrounded centroid sum_t t q_t */
    int32_t h_eff, h_cov, h_ctrl;  /* last efficiency centroid, coverage bound (0 at start), their max */
} turnopd_depth_state;

void turnopd_depth_default_params(turnopd_depth_params *p);
turnopd_status turnopd_depth_init(const turnopd_depth_params *p, turnopd_depth_state *s);
turnopd_status turnopd_depth_plan(const turnopd_depth_params *p, const turnopd_depth_state *s, int64_t k,
                                  int32_t *h_hat, int32_t *is_probe, int32_t *h_roll);
/* After step k; a no-op unless k is a probe step.  The turn tables are those
 * of the (uncensored) probe batch, max_turns entries each; traj_len[b] = turns
 * of probe trajectory b, traj_success[b] in {0, 1}; m_out / q_out (nullable)
 * receive m_t and q_t. */
turnopd_status turnopd_depth_update(const turnopd_depth_params *p, turnopd_depth_state *s, int64_t k,
                                    const double *turn_sum, const int64_t *turn_cnt,
                                    const int32_t *turn_surv, int32_t max_turns,
                                    const int32_t *traj_len, const uint8_t *traj_success,
                                    int32_t num_traj, double *m_out, double *q_out);
/* The two arms on their own. */
turnopd_status turnopd_depth_efficiency(const double *turn_sum, const int64_t *turn_cnt,
                                        const int32_t *turn_surv, int32_t max_turns, double eps,
                                        double *m_out, double *q_out, double *h_eff_bar,
                                        int32_t *h_eff);
turnopd_status turnopd_depth_coverage(const int32_t *traj_len, const uint8_t *traj_success,
                                      int32_t num_traj, double p, int32_t min_cov_traj,
                                      int32_t use_success, int32_t previous, int32_t *h_cov);
/*
 * Loss-allocation diagnostics of one batch: b_out[t] = turn_cnt[t] / N (token
 * share), s_out[t] = turn_sum[t] / sum turn_sum (KL loss share); over the
 * reliable prefix P (turns 0.. while turn_surv >= n_min and > 0) with
 * third = floor(P / 3): deep_out[0] = P, deep_out[1] = mean K_t over the deepest
 * third / mean K_t over the shallowest third, deep_out[2] = mean turn_surv over
 * the deepest third / turn_surv[0], deep_out[3] = sum of s_t over the deepest
 * third (NaN when P < 3).
 */
turnopd_status turnopd_turn_diagnostics(const double *turn_sum, const int64_t *turn_cnt,
                                        const int32_t *turn_surv, int32_t max_turns, int32_t n_min,
                                        double *b_out, double *s_out, double *deep_out);

/*
 * turnopd_turn_stats -- turn statistics of the per-token losses
 * (Eq. observed-turn-kl: K_t is the mean per-token reverse KL over the
 * supervised tokens at turn t, over trajectories that reach t; the survivor
 * count n_t of Sec. 5.1; the kl_per_turn / num_traj statistics of the
 * hyper-parameter table).  Sums and counts are returned rather than means so
 * that ranks can add them; K_t = turn_sum[t] / turn_cnt[t].
 * Outputs (device, caller-owned):
 *   traj_turn_sum double[num_traj * max_turns]  sum of token_loss over (b, t)
 *   traj_turn_cnt int32 [num_traj * max_turns]  n_bt
 *   turn_sum      double[max_turns]             sum over b of traj_turn_sum
 *   turn_cnt      int64 [max_turns]             sum over b of n_bt
 *   turn_surv     int32 [max_turns]             #{b : n_bt > 0}
 * Device errors: TURNOPD_ERR_OFFSETS, TURNOPD_ERR_TURN_RANGE (token ignored).
 */
turnopd_status turnopd_turn_stats(const float *token_loss, const int32_t *turn_id,
                                  const uint8_t *loss_mask, const int64_t *traj_offsets,
                                  int32_t num_traj, int64_t num_tokens, int32_t max_turns,
                                  double *traj_turn_sum, int32_t *traj_turn_cnt,
                                  double *turn_sum, int64_t *turn_cnt, int32_t *turn_surv,
                                  int32_t *dev_status, turnopd_stream_t stream);

/*
 * turnopd_alpha_schedule -- blend coefficient alpha_k = clip((k/K - s)/(e - s), 0, 1)
 * from training progress k/K (Sec. 5.2; Algorithm 1; s, e = 0, 1 in the
 * paper's runs).  Host function.  Returns NaN if K <= 0 or e <= s.
 */
double turnopd_alpha_schedule(int64_t k, int64_t K, double s, double e);

/*
 * turnopd_turn_floor -- the turn-reliability floor of the internal blend,
 * n_min = max(min_floor, ceil(min_frac * n_traj)) (hyper-parameter table,
 * internal-blend group: min_floor = 8, min_frac = 0.15), to pass as n_min to
 * turnopd_weights.  n_traj is the number of trajectories of the step's batch
 * (all data-parallel ranks together, empty trajectories included), the
 * population over which the survivor counts S_t are taken.  Host function.
 * The ceiling is exact for decimal fractions: 0.07 * 100 gives 7, not 8.
 * Returns -1 if n_traj < 0, min_floor < 0, min_frac is outside [0, 1] (or
 * NaN), or the result exceeds INT32_MAX.
 */
int32_t turnopd_turn_floor(int64_t n_traj, int32_t min_floor, double min_frac);

/*
 * turnopd_selftest_wait_timeout -- diagnostic of the device-side timeout path.
 * Every wait of the library's kernels on an mbarrier or a flag is a bounded poll
 * loop: when the limit runs out the kernel records TURNOPD_ERR_TIMEOUT in
 * *dev_status, stops waiting and returns, so the context stays usable.  This
 * entry launches one CTA that polls, in the same way, a barrier that nothing
 * arrives on, so the path can be exercised without any failure of the GPU.
 * poll_limit: polls before giving up, in [1, 2^24].
 * dev_status: device int32 (caller-zeroed); receives TURNOPD_ERR_TIMEOUT.
 * Errors: TURNOPD_ERR_NULL, TURNOPD_ERR_SHAPE (limit out of range), TURNOPD_ERR_CUDA.
 */
turnopd_status turnopd_selftest_wait_timeout(uint32_t poll_limit, int32_t *dev_status,
                                             turnopd_stream_t stream);

/* Human-readable name of a status code (static string, never NULL). */
const char *turnopd_status_string(turnopd_status status);

#ifdef __cplusplus
}
#endif

#endif /* TURNOPD_H */
