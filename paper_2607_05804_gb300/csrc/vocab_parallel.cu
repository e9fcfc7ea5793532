// Vocabulary-parallel split of the reverse-KL loss (Eq. opd-rkl) for logits
// sharded by vocabulary columns across ranks:
//   1. turnopd_vocab_shard_stats    per supervised token, this shard's partial
//      row statistics (m_s, S_s, A, d, m_t, S_t) -- 24 B per token;
//   2. (the caller all-gathers the partials of every shard, in rank order)
//   3. turnopd_vocab_stats_merge    the row statistics of the whole vocabulary,
//      merged in shard order (every rank gets the same bits);
//   4. turnopd_vocab_shard_loss_grad l_i = KL_i, L = sum_i w_i l_i and this
//      shard's gradient columns g = w p_s ((z_s - z_t) - E_p[z_s - z_t]).
// A = sum e^{z_s - m_s} ((z_s - z_t) - d) is kept relative to the reference
// difference d of the shard's largest student logit, as in the single-GPU
// kernels.  One CTA per token row at a time.

#include <cuda_bf16.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.h"
#include "row_math.cuh"

namespace turnopd {
namespace {

constexpr int kVpThreads = 256;
constexpr int kStatWords = 6;  // m_s, S_s, A, d, m_t, S_t

struct ShardIn {
    const void *zs, *zt;
    int64_t ld, vocab, num_rows;
    const int32_t *row_of_token;
    const uint8_t *mask;
    int64_t T;
    int32_t *status;
};

template <typename TIn, bool VEC>
__device__ __forceinline__ void fold_row(const TIn *rs, const TIn *rt, int64_t V, Student &s, Teacher &t)
{
    constexpr int N = Vec<TIn>::N;
    const int64_t nvec = VEC ? V / N : 0;
    if (VEC) {
        for (int64_t q = threadIdx.x; q < nvec; q += kVpThreads) {
            float a[N], b[N];
            Vec<TIn>::load(rs + q * N, a);
            Vec<TIn>::load(rt + q * N, b);
            accumulate<N>(s, t, a, b);
        }
    }
    for (int64_t v = nvec * N + threadIdx.x; v < V; v += kVpThreads) {
        float a = to_float(rs[v]), b = to_float(rt[v]);
        accumulate<1>(s, t, &a, &b);
    }
}

// Block reduction of the per-thread accumulators (result in thread 0).
__device__ __forceinline__ void block_merge(Student &s, Teacher &t, Student *red_s, Teacher *red_t)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    s = warp_merge(s);
    t = warp_merge(t);
    if (lane == 0) {
        red_s[warp] = s;
        red_t[warp] = t;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int k = 1; k < kVpThreads / 32; ++k) {
            red_s[0] = student_merge(red_s[0], red_s[k]);
            red_t[0] = teacher_merge(red_t[0], red_t[k]);
        }
        s = red_s[0];
        t = red_t[0];
    }
}

__device__ __forceinline__ bool token_row(const ShardIn &p, int64_t i, int64_t *r)
{
    if (!p.mask[i])
        return false;
    const int64_t row = p.row_of_token ? (int64_t)p.row_of_token[i] : i;
    if (row < 0 || row >= p.num_rows) {
        if (threadIdx.x == 0)
            set_status(p.status, TURNOPD_ERR_TOKEN_RANGE);
        return false;
    }
    *r = row;
    return true;
}

template <typename TIn, bool VEC>
__global__ void __launch_bounds__(kVpThreads) k_shard_stats(ShardIn p, float *__restrict__ stats)
{
    __shared__ Student red_s[kVpThreads / 32];
    __shared__ Teacher red_t[kVpThreads / 32];
    const TIn *zs = static_cast<const TIn *>(p.zs);
    const TIn *zt = static_cast<const TIn *>(p.zt);
    for (int64_t i = blockIdx.x; i < p.T; i += gridDim.x) {
        int64_t r;
        if (!token_row(p, i, &r))
            continue;
        Student s = student_empty();
        Teacher t = teacher_empty();
        fold_row<TIn, VEC>(zs + r * p.ld, zt + r * p.ld, p.vocab, s, t);
        block_merge(s, t, red_s, red_t);
        if (threadIdx.x == 0) {
            float *o = stats + i * kStatWords;
            o[0] = s.m, o[1] = s.s, o[2] = s.a, o[3] = s.d, o[4] = t.m, o[5] = t.s;
        }
        __syncthreads();
    }
}

__global__ void k_stats_merge(const float *__restrict__ parts, int n_shards, const uint8_t *__restrict__ mask,
                              int64_t T, float *__restrict__ merged)
{
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < T; i += (int64_t)gridDim.x * blockDim.x) {
        if (!mask[i])
            continue;
        Student S = student_empty();
        Teacher U = teacher_empty();
        for (int r = 0; r < n_shards; ++r) {
            const float *q = parts + ((size_t)r * T + i) * kStatWords;
            S = student_merge(S, Student{q[0], q[1], q[2], q[3]});
            U = teacher_merge(U, Teacher{q[4], q[5]});
        }
        float *o = merged + i * kStatWords;
        o[0] = S.m, o[1] = S.s, o[2] = S.a, o[3] = S.d, o[4] = U.m, o[5] = U.s;
    }
}

template <typename TIn, typename TOut, bool VEC>
__global__ void __launch_bounds__(kVpThreads)
k_shard_grad(ShardIn p, const float *__restrict__ merged, const float *__restrict__ w, TOut *grad, float *token_loss,
             double *wl, int32_t *nvalid_slot)
{
    __shared__ float bc[4];
    constexpr int N = Vec<TIn>::N;
    if (blockIdx.x == 0 && threadIdx.x == 0)
        *nvalid_slot = (int32_t)p.T;  // the loss sum runs over every token (0 for masked ones)
    const TIn *zs = static_cast<const TIn *>(p.zs);
    const TIn *zt = static_cast<const TIn *>(p.zt);
    const int64_t V = p.vocab;
    const int64_t nvec = VEC ? V / N : 0;
    for (int64_t i = blockIdx.x; i < p.T; i += gridDim.x) {
        int64_t r;
        if (!token_row(p, i, &r)) {
            if (threadIdx.x == 0) {
                token_loss[i] = 0.f;
                wl[i] = 0.0;
            }
            continue;
        }
        if (threadIdx.x == 0) {
            const float *q = merged + i * kStatWords;
            const RowConst rc = row_const(Student{q[0], q[1], q[2], q[3]}, Teacher{q[4], q[5]});
            if (!isfinite(rc.lse_s) || !isfinite(rc.lse_t) || !isfinite(rc.kl))
                set_status(p.status, TURNOPD_ERR_NONFINITE);
            token_loss[i] = rc.kl;
            wl[i] = (double)w[i] * (double)rc.kl;
            bc[0] = rc.lse_s;
            bc[1] = rc.d;
            bc[2] = rc.cp;
            bc[3] = w[i];
        }
        __syncthreads();
        if (grad) {
            const float nl = -bc[0] * kLog2e, d = bc[1], cp = bc[2], wi = bc[3];
            const TIn *rs = zs + r * p.ld;
            const TIn *rt = zt + r * p.ld;
            TOut *gr = grad + r * p.ld;
            if (VEC) {
                for (int64_t qv = threadIdx.x; qv < nvec; qv += kVpThreads) {
                    float a[N], b[N], g[N];
                    Vec<TIn>::load(rs + qv * N, a);
                    Vec<TIn>::load(rt + qv * N, b);
#pragma unroll
                    for (int k = 0; k < N; ++k)
                        g[k] = wi * ex2(fmaf(a[k], kLog2e, nl)) * (((a[k] - b[k]) - d) - cp);
                    store_vec<TOut, N>(gr + qv * N, g);
                }
            }
            for (int64_t v = nvec * N + threadIdx.x; v < V; v += kVpThreads) {
                const float a = to_float(rs[v]), b = to_float(rt[v]);
                gr[v] = from_float<TOut>(wi * ex2(fmaf(a, kLog2e, nl)) * (((a - b) - d) - cp));
            }
        }
        __syncthreads();
    }
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

size_t vocab_stats_bytes(int64_t T) { return sizeof(float) * kStatWords * (size_t)std::max<int64_t>(T, 0); }

cudaError_t launch_vocab_shard_stats(const VocabShardCall &c, float *stats, cudaStream_t stream)
{
    ShardIn p{c.zs, c.zt, c.ld, c.vocab, c.num_rows, c.row_of_token, c.mask, c.T, c.status};
    const size_t esz = c.in_dtype == TURNOPD_BF16 ? 2 : 4;
    const bool vec = aligned16(c.zs) && aligned16(c.zt) && (c.ld * esz) % 16 == 0;
    const int grid = (int)std::min<int64_t>(std::max<int64_t>(c.T, 1), (int64_t)device_sm_count() * 8);
    if (c.in_dtype == TURNOPD_BF16) {
        if (vec)
            k_shard_stats<__nv_bfloat16, true><<<grid, kVpThreads, 0, stream>>>(p, stats);
        else
            k_shard_stats<__nv_bfloat16, false><<<grid, kVpThreads, 0, stream>>>(p, stats);
    } else {
        if (vec)
            k_shard_stats<float, true><<<grid, kVpThreads, 0, stream>>>(p, stats);
        else
            k_shard_stats<float, false><<<grid, kVpThreads, 0, stream>>>(p, stats);
    }
    return cudaGetLastError();
}

cudaError_t launch_vocab_stats_merge(const float *parts, int n_shards, const uint8_t *mask, int64_t T,
                                     float *merged, cudaStream_t stream)
{
    const int grid = (int)std::min<int64_t>((T + 255) / 256, (int64_t)device_sm_count() * 4);
    k_stats_merge<<<std::max(grid, 1), 256, 0, stream>>>(parts, n_shards, mask, T, merged);
    return cudaGetLastError();
}

template <typename TIn, typename TOut>
static void shard_grad_kernel(const ShardIn &p, bool vec, int grid, const float *merged, const float *w, void *grad,
                              float *tl, double *wl, int32_t *nv, cudaStream_t stream)
{
    if (vec)
        k_shard_grad<TIn, TOut, true><<<grid, kVpThreads, 0, stream>>>(p, merged, w, static_cast<TOut *>(grad), tl,
                                                                      wl, nv);
    else
        k_shard_grad<TIn, TOut, false><<<grid, kVpThreads, 0, stream>>>(p, merged, w, static_cast<TOut *>(grad), tl,
                                                                       wl, nv);
}

cudaError_t launch_vocab_shard_grad(const VocabShardCall &c, const float *merged, cudaStream_t stream)
{
    LossWorkspace ws = loss_workspace_layout(c.workspace, c.T);
    ShardIn p{c.zs, c.zt, c.ld, c.vocab, c.num_rows, c.row_of_token, c.mask, c.T, c.status};
    const size_t esz = c.in_dtype == TURNOPD_BF16 ? 2 : 4;
    const size_t gesz = c.grad_dtype == TURNOPD_BF16 ? 2 : 4;
    const bool vec = aligned16(c.zs) && aligned16(c.zt) && (c.ld * esz) % 16 == 0 &&
                     (!c.grad || (aligned16(c.grad) && (c.ld * gesz) % 16 == 0));
    if (c.grad && (c.flags & TURNOPD_ZERO_MASKED_GRAD))
        launch_zero_masked_grad(c.mask, c.row_of_token, c.T, c.num_rows, c.ld, c.vocab, c.grad, c.grad_dtype, stream);
    const int grid = (int)std::min<int64_t>(std::max<int64_t>(c.T, 1), (int64_t)device_sm_count() * 8);
    const bool bf_in = c.in_dtype == TURNOPD_BF16, bf_out = c.grad_dtype == TURNOPD_BF16;
    if (bf_in && bf_out)
        shard_grad_kernel<__nv_bfloat16, __nv_bfloat16>(p, vec, grid, merged, c.w, c.grad, c.token_loss, ws.row_wl,
                                                        ws.nvalid, stream);
    else if (bf_in)
        shard_grad_kernel<__nv_bfloat16, float>(p, vec, grid, merged, c.w, c.grad, c.token_loss, ws.row_wl, ws.nvalid,
                                                stream);
    else if (bf_out)
        shard_grad_kernel<float, __nv_bfloat16>(p, vec, grid, merged, c.w, c.grad, c.token_loss, ws.row_wl, ws.nvalid,
                                                stream);
    else
        shard_grad_kernel<float, float>(p, vec, grid, merged, c.w, c.grad, c.token_loss, ws.row_wl, ws.nvalid, stream);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess)
        return e;
    launch_loss_sum(ws.row_wl, ws.nvalid, c.loss, c.status, stream);
    return cudaGetLastError();
}

}  // namespace turnopd
