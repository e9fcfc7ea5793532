// C-ABI entry points of libturnopd: host-side validation, workspace carving
// and kernel launches.  Every check that needs no device data happens here,
// before any CUDA call, so argument errors return synchronously.

#include <cmath>
#include <cstring>

#include <nvtx3/nvToolsExt.h>

#include "common.cuh"
#include "kernels.h"

using namespace turnopd;

namespace turnopd {

int device_sm_count()
{
    static int cached[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0)
        return 148;
    if (dev < 64 && cached[dev] > 0)
        return cached[dev];
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
        n = 148;
    if (dev < 64)
        cached[dev] = n;
    return n;
}

}  // namespace turnopd

namespace {

bool misaligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) != 0; }

// An NVTX range around one entry point (shows the library's calls on a profiler
// timeline; without a profiler attached it costs a function-pointer check).
struct NvtxRange {
    explicit NvtxRange(const char *name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
    NvtxRange(const NvtxRange &) = delete;
    NvtxRange &operator=(const NvtxRange &) = delete;
};

turnopd_status cuda_status(cudaError_t e) { return e == cudaSuccess ? TURNOPD_OK : TURNOPD_ERR_CUDA; }

size_t weights_ws(int32_t B, int32_t Tmax)
{
    return align256(sizeof(int32_t) * (size_t)B * (size_t)Tmax) +
           align256(sizeof(int64_t) * (size_t)(2 * Tmax + 1));
}

turnopd_status check_structure(const int32_t *turn_id, const uint8_t *mask, const int64_t *off,
                               int32_t B, int64_t T, int32_t Tmax, const int32_t *dev_status)
{
    if (!off || !dev_status || (T > 0 && (!turn_id || !mask)))
        return TURNOPD_ERR_NULL;
    if (B < 0 || T < 0 || T > INT32_MAX || Tmax < 1 || Tmax > TURNOPD_MAX_TURNS)
        return TURNOPD_ERR_SHAPE;
    if ((int64_t)B * (int64_t)Tmax > INT32_MAX)
        return TURNOPD_ERR_SHAPE;
    return TURNOPD_OK;
}

}  // namespace

extern "C" {

const char *turnopd_status_string(turnopd_status s)
{
    switch (s) {
    case TURNOPD_OK: return "ok";
    case TURNOPD_ERR_NULL: return "a required pointer is NULL";
    case TURNOPD_ERR_SHAPE: return "a size or stride is out of range";
    case TURNOPD_ERR_OFFSETS: return "trajectory offsets are not 0..num_tokens non-decreasing";
    case TURNOPD_ERR_TURN_RANGE: return "supervised token with turn id outside [0, max_turns)";
    case TURNOPD_ERR_TOKEN_RANGE: return "row index or sampled id out of range";
    case TURNOPD_ERR_UNSUPPORTED: return "unsupported dtype, mode or flag combination";
    case TURNOPD_ERR_CUDA: return "CUDA runtime error";
    case TURNOPD_ERR_TIMEOUT: return "bounded device-side wait timed out";
    case TURNOPD_ERR_NONFINITE: return "non-finite log-sum-exp or loss";
    case TURNOPD_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    }
    return "unknown status";
}

double turnopd_alpha_schedule(int64_t k, int64_t K, double s, double e)
{
    if (K <= 0 || !(e > s))
        return NAN;
    double a = ((double)k / (double)K - s) / (e - s);
    return a < 0.0 ? 0.0 : (a > 1.0 ? 1.0 : a);
}

int32_t turnopd_turn_floor(int64_t n_traj, int32_t min_floor, double min_frac)
{
    if (n_traj < 0 || min_floor < 0 || !(min_frac >= 0.0) || !(min_frac <= 1.0))
        return -1;
    // min_frac is usually a short decimal (0.15, 0.07) whose binary value lies a hair
    // off it, so an exact integer product can land one ulp above the integer;
    // the relative guard of 2^-40 keeps ceil() from stepping past it.
    const double x = min_frac * (double)n_traj;
    const double c = ceil(x - x * 0x1p-40);
    const double n = c > (double)min_floor ? c : (double)min_floor;
    return n > 2147483647.0 ? -1 : (int32_t)n;
}

turnopd_status turnopd_selftest_wait_timeout(uint32_t poll_limit, int32_t *dev_status, turnopd_stream_t stream)
{
    if (!dev_status)
        return TURNOPD_ERR_NULL;
    if (poll_limit < 1 || poll_limit > (1u << 24))
        return TURNOPD_ERR_SHAPE;
    return cuda_status(launch_wait_selftest(poll_limit, dev_status, (cudaStream_t)stream));
}

size_t turnopd_weights_workspace_bytes(int32_t num_traj, int32_t max_turns)
{
    if (num_traj < 0 || max_turns < 1)
        return 0;
    return weights_ws(num_traj, max_turns);
}

size_t turnopd_loss_workspace_bytes(int64_t num_tokens)
{
    if (num_tokens < 0)
        return 0;
    return loss_workspace_bytes(num_tokens);
}

turnopd_status turnopd_turn_counts(const int32_t *turn_id, const uint8_t *loss_mask,
                                   const int64_t *traj_offsets, int32_t num_traj,
                                   int64_t num_tokens, int32_t max_turns,
                                   int32_t *traj_turn_cnt, int64_t *counts,
                                   int32_t *dev_status, turnopd_stream_t stream)
{
    NvtxRange nvtx("turnopd_turn_counts");
    turnopd_status st = check_structure(turn_id, loss_mask, traj_offsets, num_traj, num_tokens,
                                        max_turns, dev_status);
    if (st != TURNOPD_OK)
        return st;
    if (!counts || (num_traj > 0 && !traj_turn_cnt))
        return TURNOPD_ERR_NULL;
    return cuda_status(launch_turn_counts(turn_id, loss_mask, traj_offsets, num_traj, num_tokens,
                                          max_turns, traj_turn_cnt, counts, dev_status,
                                          (cudaStream_t)stream));
}

turnopd_status turnopd_weights(const int32_t *turn_id, const uint8_t *loss_mask,
                               const int64_t *traj_offsets, int32_t num_traj,
                               int64_t num_tokens, int32_t max_turns, double alpha,
                               int32_t scope, int32_t n_min, const int64_t *global_counts,
                               float *w_out, void *workspace, size_t workspace_bytes,
                               int32_t *dev_status, turnopd_stream_t stream)
{
    NvtxRange nvtx("turnopd_weights");
    turnopd_status st = check_structure(turn_id, loss_mask, traj_offsets, num_traj, num_tokens,
                                        max_turns, dev_status);
    if (st != TURNOPD_OK)
        return st;
    if (num_tokens > 0 && !w_out)
        return TURNOPD_ERR_NULL;
    if (!(alpha >= 0.0 && alpha <= 1.0))
        return TURNOPD_ERR_SHAPE;
    if (scope != TURNOPD_SCOPE_TRAJ && scope != TURNOPD_SCOPE_BATCH)
        return TURNOPD_ERR_UNSUPPORTED;
    if (!workspace || misaligned(workspace, 256) ||
        workspace_bytes < weights_ws(num_traj, max_turns))
        return TURNOPD_ERR_WORKSPACE;
    char *ws = static_cast<char *>(workspace);
    int32_t *n_bt = reinterpret_cast<int32_t *>(ws);
    int64_t *counts = reinterpret_cast<int64_t *>(
        ws + align256(sizeof(int32_t) * (size_t)num_traj * (size_t)max_turns));
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e = launch_turn_counts(turn_id, loss_mask, traj_offsets, num_traj, num_tokens,
                                       max_turns, n_bt, counts, dev_status, s);
    if (e != cudaSuccess)
        return TURNOPD_ERR_CUDA;
    e = launch_weights(turn_id, loss_mask, traj_offsets, num_traj, num_tokens, max_turns, alpha,
                       scope, n_min, n_bt, global_counts ? global_counts : counts, w_out,
                       dev_status, s);
    return cuda_status(e);
}

turnopd_status turnopd_loss_fwd_bwd(const void *z_student, const void *z_teacher,
                                    int32_t in_dtype, int64_t ld, int64_t vocab,
                                    int64_t num_rows, const int32_t *row_of_token,
                                    const int32_t *sampled_ids, const uint8_t *loss_mask,
                                    const float *w, int64_t num_tokens, int32_t mode,
                                    void *grad_student, int32_t grad_dtype, uint32_t flags,
                                    float *token_loss_out, double *loss_out,
                                    void *workspace, size_t workspace_bytes,
                                    int32_t *dev_status, turnopd_stream_t stream)
{
    NvtxRange nvtx("turnopd_loss_fwd_bwd");
    if (!loss_out || !dev_status)
        return TURNOPD_ERR_NULL;
    if (num_tokens > 0 && (!z_student || !z_teacher || !loss_mask || !w || !token_loss_out))
        return TURNOPD_ERR_NULL;
    if (mode != TURNOPD_FULL_VOCAB && mode != TURNOPD_SAMPLED_TOKEN)
        return TURNOPD_ERR_UNSUPPORTED;
    if (mode == TURNOPD_SAMPLED_TOKEN && num_tokens > 0 && !sampled_ids)
        return TURNOPD_ERR_NULL;
    if ((in_dtype != TURNOPD_F32 && in_dtype != TURNOPD_BF16) ||
        (grad_student && grad_dtype != TURNOPD_F32 && grad_dtype != TURNOPD_BF16))
        return TURNOPD_ERR_UNSUPPORTED;
    if (flags & ~(uint32_t)(TURNOPD_ZERO_MASKED_GRAD | TURNOPD_FORCE_PORTABLE))
        return TURNOPD_ERR_UNSUPPORTED;
    if (num_tokens < 0 || num_tokens > INT32_MAX || vocab < 1 || vocab > INT32_MAX || ld < vocab ||
        num_rows < 0 || (!row_of_token && num_rows < num_tokens))
        return TURNOPD_ERR_SHAPE;
    const size_t esz = in_dtype == TURNOPD_BF16 ? 2 : 4;
    if (misaligned(z_student, esz) || misaligned(z_teacher, esz) ||
        (grad_student && misaligned(grad_student, grad_dtype == TURNOPD_BF16 ? 2 : 4)) ||
        misaligned(loss_out, 8))
        return TURNOPD_ERR_SHAPE;
    if (!workspace || misaligned(workspace, 256) ||
        workspace_bytes < loss_workspace_bytes(num_tokens))
        return TURNOPD_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    if (num_tokens == 0)
        return cuda_status(cudaMemsetAsync(loss_out, 0, sizeof(double), s));

    LossArgs a{z_student, z_teacher, in_dtype, ld, vocab, num_rows, row_of_token, sampled_ids,
               loss_mask, w, num_tokens, mode, grad_student, grad_dtype, flags, token_loss_out,
               loss_out, dev_status};
    return cuda_status(launch_loss(a, loss_workspace_layout(workspace, num_tokens), s));
}

turnopd_status turnopd_topk_loss_fwd_bwd(const void *z_student, const void *z_teacher, int32_t in_dtype,
                                         int64_t ld, int64_t vocab, int64_t num_rows,
                                         const int32_t *row_of_token, const uint8_t *loss_mask,
                                         const float *w, int64_t num_tokens, int32_t k_top,
                                         int32_t *topk_ids_out, float *topk_grad_out, void *grad_student,
                                         int32_t grad_dtype, uint32_t flags, float *token_loss_out,
                                         double *loss_out, void *workspace, size_t workspace_bytes,
                                         int32_t *dev_status, turnopd_stream_t stream)
{
    NvtxRange nvtx("turnopd_topk_loss_fwd_bwd");
    if (!loss_out || !dev_status)
        return TURNOPD_ERR_NULL;
    if (num_tokens > 0 && (!z_student || !z_teacher || !loss_mask || !w || !token_loss_out))
        return TURNOPD_ERR_NULL;
    if ((in_dtype != TURNOPD_F32 && in_dtype != TURNOPD_BF16) ||
        (grad_student && grad_dtype != TURNOPD_F32 && grad_dtype != TURNOPD_BF16))
        return TURNOPD_ERR_UNSUPPORTED;
    if (flags & ~(uint32_t)TURNOPD_ZERO_MASKED_GRAD)
        return TURNOPD_ERR_UNSUPPORTED;
    if (num_tokens < 0 || num_tokens > INT32_MAX || vocab < 1 || vocab > INT32_MAX || ld < vocab ||
        num_rows < 0 || (!row_of_token && num_rows < num_tokens) || k_top < 1 || k_top > TURNOPD_TOPK_MAX ||
        k_top > vocab || vocab > TURNOPD_TOPK_MAX_VOCAB || num_tokens * (int64_t)k_top > INT64_MAX / 8)
        return TURNOPD_ERR_SHAPE;
    const size_t esz = in_dtype == TURNOPD_BF16 ? 2 : 4;
    if (misaligned(z_student, esz) || misaligned(z_teacher, esz) ||
        (grad_student && misaligned(grad_student, grad_dtype == TURNOPD_BF16 ? 2 : 4)) ||
        (topk_ids_out && misaligned(topk_ids_out, 4)) || (topk_grad_out && misaligned(topk_grad_out, 4)) ||
        misaligned(loss_out, 8))
        return TURNOPD_ERR_SHAPE;
    if (!workspace || misaligned(workspace, 256) ||
        workspace_bytes < loss_workspace_bytes(num_tokens))
        return TURNOPD_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    if (num_tokens == 0)
        return cuda_status(cudaMemsetAsync(loss_out, 0, sizeof(double), s));
    TopkCall c;
    c.zs = z_student;
    c.zt = z_teacher;
    c.in_dtype = in_dtype;
    c.ld = ld;
    c.vocab = vocab;
    c.num_rows = num_rows;
    c.row_of_token = row_of_token;
    c.mask = loss_mask;
    c.w = w;
    c.T = num_tokens;
    c.K = k_top;
    c.topk_ids = topk_ids_out;
    c.topk_grad = topk_grad_out;
    c.grad = grad_student;
    c.grad_dtype = grad_dtype;
    c.flags = flags;
    c.token_loss = token_loss_out;
    c.loss = loss_out;
    c.workspace = workspace;
    c.status = dev_status;
    return cuda_status(launch_topk(c, s));
}

size_t turnopd_vocab_stats_bytes(int64_t num_tokens) { return vocab_stats_bytes(num_tokens); }

static turnopd_status vocab_common_checks(const void *z_student, const void *z_teacher, int32_t in_dtype, int64_t ld,
                                          int64_t shard_vocab, int64_t num_rows, const int32_t *row_of_token,
                                          const uint8_t *loss_mask, int64_t num_tokens, int32_t *dev_status)
{
    if (!dev_status || (num_tokens > 0 && (!z_student || !z_teacher || !loss_mask)))
        return TURNOPD_ERR_NULL;
    if (in_dtype != TURNOPD_F32 && in_dtype != TURNOPD_BF16)
        return TURNOPD_ERR_UNSUPPORTED;
    if (num_tokens < 0 || num_tokens > INT32_MAX || shard_vocab < 1 || shard_vocab > INT32_MAX ||
        ld < shard_vocab || num_rows < 0 || (!row_of_token && num_rows < num_tokens))
        return TURNOPD_ERR_SHAPE;
    const size_t esz = in_dtype == TURNOPD_BF16 ? 2 : 4;
    if (misaligned(z_student, esz) || misaligned(z_teacher, esz))
        return TURNOPD_ERR_SHAPE;
    return TURNOPD_OK;
}

turnopd_status turnopd_vocab_shard_stats(const void *z_student, const void *z_teacher, int32_t in_dtype, int64_t ld,
                                         int64_t shard_vocab, int64_t num_rows, const int32_t *row_of_token,
                                         const uint8_t *loss_mask, int64_t num_tokens, float *stats_out,
                                         void *workspace, size_t workspace_bytes, int32_t *dev_status,
                                         turnopd_stream_t stream)
{
    NvtxRange nvtx("turnopd_vocab_shard_stats");
    turnopd_status st = vocab_common_checks(z_student, z_teacher, in_dtype, ld, shard_vocab, num_rows, row_of_token,
                                            loss_mask, num_tokens, dev_status);
    if (st != TURNOPD_OK)
        return st;
    if (num_tokens > 0 && !stats_out)
        return TURNOPD_ERR_NULL;
    if (misaligned(stats_out, 4))
        return TURNOPD_ERR_SHAPE;
    if (!workspace || misaligned(workspace, 256) || workspace_bytes < loss_workspace_bytes(num_tokens))
        return TURNOPD_ERR_WORKSPACE;
    if (num_tokens == 0)
        return TURNOPD_OK;
    VocabShardCall c{z_student, z_teacher, in_dtype, ld, shard_vocab, num_rows, row_of_token, loss_mask, nullptr,
                     num_tokens, nullptr, TURNOPD_F32, 0u, nullptr, nullptr, workspace, dev_status};
    return cuda_status(launch_vocab_shard_stats(c, stats_out, (cudaStream_t)stream));
}

turnopd_status turnopd_vocab_stats_merge(const float *parts, int32_t n_shards, const uint8_t *loss_mask,
                                         int64_t num_tokens, float *merged_out, turnopd_stream_t stream)
{
    NvtxRange nvtx("turnopd_vocab_stats_merge");
    if (num_tokens > 0 && (!parts || !loss_mask || !merged_out))
        return TURNOPD_ERR_NULL;
    if (n_shards < 1 || num_tokens < 0 || num_tokens > INT32_MAX)
        return TURNOPD_ERR_SHAPE;
    if (misaligned(parts, 4) || misaligned(merged_out, 4))
        return TURNOPD_ERR_SHAPE;
    if (num_tokens == 0)
        return TURNOPD_OK;
    return cuda_status(launch_vocab_stats_merge(parts, n_shards, loss_mask, num_tokens, merged_out,
                                                (cudaStream_t)stream));
}

turnopd_status turnopd_vocab_shard_loss_grad(const void *z_student, const void *z_teacher, int32_t in_dtype,
                                             int64_t ld, int64_t shard_vocab, int64_t num_rows,
                                             const int32_t *row_of_token, const uint8_t *loss_mask, const float *w,
                                             int64_t num_tokens, const float *merged_stats, void *grad_shard,
                                             int32_t grad_dtype, uint32_t flags, float *token_loss_out,
                                             double *loss_out, void *workspace, size_t workspace_bytes,
                                             int32_t *dev_status, turnopd_stream_t stream)
{
    NvtxRange nvtx("turnopd_vocab_shard_loss_grad");
    turnopd_status st = vocab_common_checks(z_student, z_teacher, in_dtype, ld, shard_vocab, num_rows, row_of_token,
                                            loss_mask, num_tokens, dev_status);
    if (st != TURNOPD_OK)
        return st;
    if (!loss_out || (num_tokens > 0 && (!w || !merged_stats || !token_loss_out)))
        return TURNOPD_ERR_NULL;
    if (grad_shard && grad_dtype != TURNOPD_F32 && grad_dtype != TURNOPD_BF16)
        return TURNOPD_ERR_UNSUPPORTED;
    if (flags & ~(uint32_t)TURNOPD_ZERO_MASKED_GRAD)
        return TURNOPD_ERR_UNSUPPORTED;
    if ((grad_shard && misaligned(grad_shard, grad_dtype == TURNOPD_BF16 ? 2 : 4)) || misaligned(loss_out, 8) ||
        misaligned(merged_stats, 4))
        return TURNOPD_ERR_SHAPE;
    if (!workspace || misaligned(workspace, 256) || workspace_bytes < loss_workspace_bytes(num_tokens))
        return TURNOPD_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    if (num_tokens == 0)
        return cuda_status(cudaMemsetAsync(loss_out, 0, sizeof(double), s));
    VocabShardCall c{z_student, z_teacher, in_dtype, ld, shard_vocab, num_rows, row_of_token, loss_mask, w,
                     num_tokens, grad_shard, grad_dtype, flags, token_loss_out, loss_out, workspace, dev_status};
    return cuda_status(launch_vocab_shard_grad(c, merged_stats, s));
}

size_t turnopd_fused_workspace_bytes(int64_t num_tokens, int64_t vocab, int64_t d_s, int64_t d_t)
{
    if (num_tokens < 0 || vocab < 1 || d_s < 1 || d_t < 1)
        return 0;
    return fused_workspace_bytes(num_tokens, vocab, d_s, d_t);
}

turnopd_status turnopd_fused_lmhead_fwd_bwd(const void *h_s, const void *W_s, int64_t d_s,
                                            const void *h_t, const void *W_t, int64_t d_t,
                                            int64_t vocab, const uint8_t *loss_mask,
                                            const float *w, int64_t num_tokens, int32_t mode,
                                            float *dh_s_out, float *dW_s_out, float *token_loss_out,
                                            double *loss_out, void *workspace,
                                            size_t workspace_bytes, int32_t *dev_status,
                                            turnopd_stream_t stream)
{
    NvtxRange nvtx("turnopd_fused_lmhead_fwd_bwd");
    if (!loss_out || !dev_status || !W_s || !W_t)
        return TURNOPD_ERR_NULL;
    if (num_tokens > 0 && (!h_s || !h_t || !loss_mask || !w || !token_loss_out))
        return TURNOPD_ERR_NULL;
    if (mode != TURNOPD_FULL_VOCAB)
        return TURNOPD_ERR_UNSUPPORTED;
    if (num_tokens < 0 || num_tokens > INT32_MAX || vocab < 1 || vocab > INT32_MAX || d_s < 256 ||
        d_s % 256 != 0 || d_t < 64 || d_t % 64 != 0 || d_s > 65536 || d_t > 65536)
        return TURNOPD_ERR_SHAPE;
    if (misaligned(h_s, 16) || misaligned(W_s, 16) || misaligned(h_t, 16) || misaligned(W_t, 16) ||
        (dh_s_out && misaligned(dh_s_out, 16)) || (dW_s_out && misaligned(dW_s_out, 16)) ||
        misaligned(loss_out, 8))
        return TURNOPD_ERR_SHAPE;
    if (!workspace || misaligned(workspace, 256) ||
        workspace_bytes < fused_workspace_bytes(num_tokens, vocab, d_s, d_t))
        return TURNOPD_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    if (num_tokens == 0) {
        if (dW_s_out) {
            const cudaError_t e = cudaMemsetAsync(dW_s_out, 0, sizeof(float) * (size_t)vocab * (size_t)d_s, s);
            if (e != cudaSuccess)
                return cuda_status(e);
        }
        return cuda_status(cudaMemsetAsync(loss_out, 0, sizeof(double), s));
    }
    FusedCall c{h_s, W_s, h_t, W_t, d_s, d_t, vocab, num_tokens, loss_mask, w, dh_s_out, dW_s_out,
                token_loss_out, loss_out, workspace, dev_status};
    return cuda_status(launch_fused(c, s));
}

turnopd_status turnopd_turn_stats(const float *token_loss, const int32_t *turn_id,
                                  const uint8_t *loss_mask, const int64_t *traj_offsets,
                                  int32_t num_traj, int64_t num_tokens, int32_t max_turns,
                                  double *traj_turn_sum, int32_t *traj_turn_cnt,
                                  double *turn_sum, int64_t *turn_cnt, int32_t *turn_surv,
                                  int32_t *dev_status, turnopd_stream_t stream)
{
    NvtxRange nvtx("turnopd_turn_stats");
    turnopd_status st = check_structure(turn_id, loss_mask, traj_offsets, num_traj, num_tokens,
                                        max_turns, dev_status);
    if (st != TURNOPD_OK)
        return st;
    if ((num_tokens > 0 && !token_loss) || !turn_sum || !turn_cnt || !turn_surv ||
        (num_traj > 0 && (!traj_turn_sum || !traj_turn_cnt)))
        return TURNOPD_ERR_NULL;
    if (turn_stats_warps(max_turns) < 1)
        return TURNOPD_ERR_UNSUPPORTED;
    return cuda_status(launch_turn_stats(token_loss, turn_id, loss_mask, traj_offsets, num_traj,
                                         num_tokens, max_turns, traj_turn_sum, traj_turn_cnt,
                                         turn_sum, turn_cnt, turn_surv, dev_status,
                                         (cudaStream_t)stream));
}

}  // extern "C"
