// Internal launcher declarations of libturnopd (not part of the public ABI).
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace turnopd {

cudaError_t launch_turn_counts(const int32_t *turn_id, const uint8_t *mask, const int64_t *off,
                               int32_t B, int64_t T, int32_t Tmax, int32_t *n_bt,
                               int64_t *counts, int32_t *status, cudaStream_t stream);

cudaError_t launch_weights(const int32_t *turn_id, const uint8_t *mask, const int64_t *off,
                           int32_t B, int64_t T, int32_t Tmax, double alpha, int32_t scope,
                           int32_t n_min, const int32_t *n_bt, const int64_t *counts,
                           float *w_out, int32_t *status, cudaStream_t stream);

int turn_stats_warps(int32_t Tmax);

cudaError_t launch_turn_stats(const float *token_loss, const int32_t *turn_id,
                              const uint8_t *mask, const int64_t *off, int32_t B, int64_t T,
                              int32_t Tmax, double *traj_turn_sum, int32_t *traj_turn_cnt,
                              double *turn_sum, int64_t *turn_cnt, int32_t *turn_surv,
                              int32_t *status, cudaStream_t stream);

// Loss path.  `ws` points at a workspace laid out by loss_workspace_layout().
struct LossWorkspace {
    int4 *rows;           // [T]  per supervised, in-range token in token order:
                          //      {token i, row r, sampled id y (or -1), bits of w_i}
    int32_t *blk_count;   // [nblk] per-block valid counts (compaction)
    int32_t *nvalid;      // [1]
    double *row_wl;       // [T]  w_i * l_i per compacted row
};

constexpr int kCompactBlock = 4096;  // tokens per compaction block

// The row-count slot of every loss workspace layout is 256 bytes; beside the count it
// holds the loss sum's scratch: a ticket (zeroed by the compaction, reset by the last
// CTA of the sum) and one partial sum per CTA of the sum.
constexpr int kSumCTAs = 24;
static_assert(8 + 8 * kSumCTAs <= 256, "the loss sum's scratch fits the row-count slot");
__host__ __device__ inline uint32_t *sum_ticket(int32_t *nvalid) { return reinterpret_cast<uint32_t *>(nvalid + 1); }
__host__ __device__ inline double *sum_partials(int32_t *nvalid)
{
    return reinterpret_cast<double *>(reinterpret_cast<char *>(nvalid) + 8);
}

size_t loss_workspace_bytes(int64_t T);
LossWorkspace loss_workspace_layout(void *ws, int64_t T);

struct LossArgs {
    const void *zs;
    const void *zt;
    int32_t in_dtype;
    int64_t ld;
    int64_t vocab;
    int64_t num_rows;
    const int32_t *row_of_token;
    const int32_t *sampled_ids;
    const uint8_t *mask;
    const float *w;
    int64_t T;
    int32_t mode;
    void *grad;
    int32_t grad_dtype;
    uint32_t flags;
    float *token_loss;
    double *loss;
    int32_t *status;
};

cudaError_t launch_loss(const LossArgs &a, const LossWorkspace &ws, cudaStream_t stream);

// Row-kernel parameters (compacted supervised rows).
struct RowIn {
    const void *zs;
    const void *zt;
    int64_t ld;
    int64_t vocab;
    const int32_t *row_of_token;
    const int32_t *sampled_ids;
    const float *w;
    int32_t mode;
    void *grad;
    float *token_loss;
    double *row_wl;
    const int4 *rows;
    const int32_t *nvalid;
    int32_t *status;
    // split_den > 0: the cluster kernel takes rows [0, nvalid split_num / split_den) of the
    // row list and the helper kernel the rest (set by launch_row_cluster)
    int32_t split_num, split_den;
};

int device_sm_count();
cudaError_t launch_wait_selftest(uint32_t limit, int32_t *status, cudaStream_t stream);

// Pieces of the loss path reused by the fused LM-head path.
cudaError_t launch_compaction(const LossArgs &a, int4 *rows, int32_t *blk_count, int32_t *nvalid,
                              cudaStream_t stream);
void launch_loss_sum(const double *row_wl, int32_t *nvalid, double *loss, int32_t *status,
                     cudaStream_t stream);
// Zero rows i (of d fp32 values) of out where mask[i] == 0.
void launch_zero_masked_f32(const uint8_t *mask, int64_t T, int64_t d, float *out, cudaStream_t stream);
// Zero the gradient rows (row_of_token[i] or i, ld apart, vocab entries) of masked tokens.
void launch_zero_masked_grad(const uint8_t *mask, const int32_t *row_of_token, int64_t T, int64_t num_rows,
                             int64_t ld, int64_t vocab, void *grad, int32_t grad_dtype, cudaStream_t stream);

// Vocabulary-parallel split.
struct VocabShardCall {
    const void *zs, *zt;
    int32_t in_dtype;
    int64_t ld, vocab, num_rows;
    const int32_t *row_of_token;
    const uint8_t *mask;
    const float *w;
    int64_t T;
    void *grad;
    int32_t grad_dtype;
    uint32_t flags;
    float *token_loss;
    double *loss;
    void *workspace;
    int32_t *status;
};
size_t vocab_stats_bytes(int64_t T);
cudaError_t launch_vocab_shard_stats(const VocabShardCall &c, float *stats, cudaStream_t stream);
cudaError_t launch_vocab_stats_merge(const float *parts, int n_shards, const uint8_t *mask, int64_t T,
                                     float *merged, cudaStream_t stream);
cudaError_t launch_vocab_shard_grad(const VocabShardCall &c, const float *merged, cudaStream_t stream);

// Teacher top-K reverse KL.
constexpr int kTopkMaxK = 1024;
struct TopkCall {
    const void *zs, *zt;
    int32_t in_dtype;
    int64_t ld, vocab, num_rows;
    const int32_t *row_of_token;
    const uint8_t *mask;
    const float *w;
    int64_t T;
    int32_t K;
    int32_t *topk_ids;
    float *topk_grad;
    void *grad;
    int32_t grad_dtype;
    uint32_t flags;
    float *token_loss;
    double *loss;
    void *workspace;
    int32_t *status;
};
cudaError_t launch_topk(const TopkCall &c, cudaStream_t stream);

// Fused LM heads (bf16 hidden states and heads) + loss + dL/dh_s.
struct FusedCall {
    const void *h_s, *W_s, *h_t, *W_t;
    int64_t d_s, d_t, vocab, T;
    const uint8_t *mask;
    const float *w;
    float *dh_s;
    float *dW_s;
    float *token_loss;
    double *loss;
    void *workspace;
    int32_t *status;
};
size_t fused_workspace_bytes(int64_t T, int64_t V, int64_t d_s, int64_t d_t);
cudaError_t launch_fused(const FusedCall &c, cudaStream_t stream);

// Cluster-resident kernel for aligned bf16 rows; sets *used = false (and
// launches nothing) when the shape does not fit it.
cudaError_t launch_row_cluster(const RowIn &p, bool fp32_grad, cudaStream_t stream, bool *used);
// The same for a vocabulary that is not a multiple of 8 (a masked last vector).
cudaError_t launch_row_cluster_tail(const RowIn &p, bool fp32_grad, cudaStream_t stream, bool *used);
// Split-row kernel (clusters of CTAs share each row) for aligned fp32 rows; sets
// *used = false (and launches nothing) when the shape does not fit it.
cudaError_t launch_row_split(const RowIn &p, bool fp32_grad, cudaStream_t stream, bool *used);

}  // namespace turnopd
