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
#include <type_traits>

#include "kernels.h"
#include "packed.cuh"
#include "row_math.cuh"

namespace turnopd {
namespace {

constexpr int kVpThreads = 128;  // several rows in flight per SM: one row's merge overlaps the others' loads
constexpr int kStatWords = 6;  // m_s, S_s, A, d, m_t, S_t
constexpr int kVpU = 4;        // bf16 rows: vectors of each model in flight per thread

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

// The same statistics for an aligned bf16 row in 16-byte vectors, kVpU vectors of
// each model in flight per thread: a running maximum rescaled once per batch when it
// moves, A kept relative to d at the thread's running student argmax (re-referenced,
// A <- (A + S (d - d')) f, with the maximum), packed f32x2 sums.
__device__ __forceinline__ void fold_row_bf16(const uint4 *vs, const uint4 *vt, int64_t nvec, Student &s,
                                              Teacher &t)
{
    constexpr uint32_t kFill = 0xff7fff7fu;  // lowest finite bf16 pair: adds 0, never the max
    const float2 L2 = splat(kLog2e);
    float ms = -INFINITY, mt = -INFINITY, dd = 0.f;
    float2 S2 = make_float2(0.f, 0.f), A2 = S2, T2 = S2;
    for (int64_t q0 = threadIdx.x; q0 < nvec; q0 += kVpU * kVpThreads) {
        uint4 a[kVpU], b[kVpU];
#pragma unroll
        for (int u = 0; u < kVpU; ++u) {
            const int64_t q = q0 + u * kVpThreads;
            if (q < nvec) {
                a[u] = __ldg(vs + q);
                b[u] = __ldg(vt + q);
            } else {
                a[u] = b[u] = make_uint4(kFill, kFill, kFill, kFill);
            }
        }
        uint32_t bs = hmax4(a[0]), bt = hmax4(b[0]);
#pragma unroll
        for (int u = 1; u < kVpU; ++u) {
            bs = hmax2u(bs, hmax4(a[u]));
            bt = hmax2u(bt, hmax4(b[u]));
        }
        const float nms = fmaxf(ms, fmaxf(bf16lo(bs), bf16hi(bs)));
        const float nmt = fmaxf(mt, fmaxf(bf16lo(bt), bf16hi(bt)));
        if (nms > ms) {
            float xd = 0.f;  // d at the first element of the batch equal to the new maximum
            bool found = false;
#pragma unroll
            for (int u = 0; u < kVpU; ++u)
#pragma unroll
                for (int w = 0; w < 4; ++w) {
                    const float2 x = unpack2(word(a[u], w)), y = unpack2(word(b[u], w));
                    if (!found && x.x == nms) {
                        xd = x.x - y.x;
                        found = true;
                    }
                    if (!found && x.y == nms) {
                        xd = x.y - y.y;
                        found = true;
                    }
                }
            const float2 f = splat(ex2((ms - nms) * kLog2e));
            A2 = fmul2(ffma2(S2, splat(dd - xd), A2), f);
            S2 = fmul2(S2, f);
            dd = xd;
            ms = nms;
        }
        if (nmt > mt) {
            T2 = fmul2(T2, splat(ex2((mt - nmt) * kLog2e)));
            mt = nmt;
        }
        const float2 NS = splat(-ms * kLog2e), NTT = splat(-mt * kLog2e), D = splat(dd);
#pragma unroll
        for (int u = 0; u < kVpU; ++u)
#pragma unroll
            for (int w = 0; w < 4; ++w) {
                const float2 a2 = unpack2(word(a[u], w)), b2 = unpack2(word(b[u], w));
                const float2 es = ex2x2(ffma2(a2, L2, NS));
                S2 = fadd2(S2, es);
                A2 = ffma2(es, fsub2(fsub2(a2, b2), D), A2);
                T2 = fadd2(T2, ex2x2(ffma2(b2, L2, NTT)));
            }
    }
    s = ms == -INFINITY ? student_empty() : Student{ms, S2.x + S2.y, A2.x + A2.y, dd};
    t = mt == -INFINITY ? teacher_empty() : Teacher{mt, T2.x + T2.y};
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

template <typename TIn, bool VEC>
__global__ void __launch_bounds__(kVpThreads) k_shard_stats(ShardIn p, const int4 *__restrict__ rows,
                                                             const int32_t *__restrict__ nvalid, float *__restrict__ stats)
{
    // reduction scratch per row parity: the next row's warps write the other half while
    // thread 0 still reads this one, so no barrier closes the row
    __shared__ Student red_s[2][kVpThreads / 32];
    __shared__ Teacher red_t[2][kVpThreads / 32];
    const TIn *zs = static_cast<const TIn *>(p.zs);
    const TIn *zt = static_cast<const TIn *>(p.zt);
    const int n = *nvalid;
    int4 m_next = (int)blockIdx.x < n ? rows[blockIdx.x] : make_int4(0, 0, 0, 0);
    for (int j = blockIdx.x, par = 0; j < n; j += gridDim.x, par ^= 1) {
        const int4 m = m_next;  // (token, row, -, -), loaded a row ahead
        if (j + (int)gridDim.x < n)
            m_next = rows[j + gridDim.x];
        const int64_t i = m.x, r = m.y;
        Student s = student_empty();
        Teacher t = teacher_empty();
        if constexpr (VEC && std::is_same<TIn, __nv_bfloat16>::value) {
            const int64_t nvec = p.vocab / 8;
            fold_row_bf16(reinterpret_cast<const uint4 *>(zs + r * p.ld), reinterpret_cast<const uint4 *>(zt + r * p.ld),
                          nvec, s, t);
            for (int64_t v = nvec * 8 + threadIdx.x; v < p.vocab; v += kVpThreads) {  // ragged tail
                float a = to_float(zs[r * p.ld + v]), b = to_float(zt[r * p.ld + v]);
                accumulate<1>(s, t, &a, &b);
            }
        } else {
            fold_row<TIn, VEC>(zs + r * p.ld, zt + r * p.ld, p.vocab, s, t);
        }
        block_merge(s, t, red_s[par], red_t[par]);
        if (threadIdx.x == 0) {
            float *o = stats + i * kStatWords;
            o[0] = s.m, o[1] = s.s, o[2] = s.a, o[3] = s.d, o[4] = t.m, o[5] = t.s;
        }
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
k_shard_grad(ShardIn p, const int4 *__restrict__ rows, const int32_t *__restrict__ nvalid,
             const float *__restrict__ merged, TOut *grad, float *token_loss, double *wl)
{
    __shared__ float bc2[2][4];  // per row parity (see k_shard_stats)
    constexpr int N = Vec<TIn>::N;
    const TIn *zs = static_cast<const TIn *>(p.zs);
    const TIn *zt = static_cast<const TIn *>(p.zt);
    const int64_t V = p.vocab;
    const int64_t nvec = VEC ? V / N : 0;
    const int n = *nvalid;
    int4 m_next = (int)blockIdx.x < n ? rows[blockIdx.x] : make_int4(0, 0, 0, 0);
    for (int j = blockIdx.x, par = 0; j < n; j += gridDim.x, par ^= 1) {
        const int4 m = m_next;  // (token, row, -, w bits), loaded a row ahead
        if (j + (int)gridDim.x < n)
            m_next = rows[j + gridDim.x];
        const int64_t i = m.x, r = m.y;
        float *bc = bc2[par];
        if (threadIdx.x == 0) {
            const float wi = __int_as_float(m.w);
            const float *q = merged + i * kStatWords;
            const RowConst rc = row_const(Student{q[0], q[1], q[2], q[3]}, Teacher{q[4], q[5]});
            if (!isfinite(rc.lse_s) || !isfinite(rc.lse_t) || !isfinite(rc.kl))
                set_status(p.status, TURNOPD_ERR_NONFINITE);
            token_loss[i] = rc.kl;
            wl[j] = (double)wi * (double)rc.kl;
            bc[0] = rc.lse_s;
            bc[1] = rc.d;
            bc[2] = rc.cp;
            bc[3] = wi;
        }
        __syncthreads();
        if (grad) {
            const float nl = -bc[0] * kLog2e, d = bc[1], cp = bc[2], wi = bc[3];
            const TIn *rs = zs + r * p.ld;
            const TIn *rt = zt + r * p.ld;
            TOut *gr = grad + r * p.ld;
            if constexpr (VEC && std::is_same<TIn, __nv_bfloat16>::value) {
                // kVpU vector pairs in flight per thread, packed arithmetic
                const uint4 *vs = reinterpret_cast<const uint4 *>(rs), *vt = reinterpret_cast<const uint4 *>(rt);
                const float2 L2 = splat(kLog2e), NL = splat(nl), D = splat(d), CP = splat(cp), WI = splat(wi);
                for (int64_t q0 = threadIdx.x; q0 < nvec; q0 += kVpU * kVpThreads) {
                    uint4 a[kVpU], b[kVpU];
#pragma unroll
                    for (int u = 0; u < kVpU; ++u) {
                        const int64_t q = q0 + u * kVpThreads;
                        if (q < nvec) {
                            a[u] = __ldg(vs + q);
                            b[u] = __ldg(vt + q);
                        }
                    }
#pragma unroll
                    for (int u = 0; u < kVpU; ++u) {
                        const int64_t q = q0 + u * kVpThreads;
                        if (q >= nvec)
                            break;
                        float g[8];
#pragma unroll
                        for (int w = 0; w < 4; ++w) {
                            const float2 a2 = unpack2(word(a[u], w)), b2 = unpack2(word(b[u], w));
                            const float2 x = fsub2(fsub2(fsub2(a2, b2), D), CP);
                            const float2 gg = fmul2(fmul2(ex2x2(ffma2(a2, L2, NL)), WI), x);
                            g[2 * w] = gg.x;
                            g[2 * w + 1] = gg.y;
                        }
                        store_vec<TOut, 8>(gr + q * 8, g);
                    }
                }
            } else if (VEC) {
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
    }
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// The grids are persistent (each CTA strides over the rows), so they are sized to
// the CTAs that are co-resident: a larger grid would run its surplus as a late
// second wave that ends the kernel with a tail.
template <typename K>
int resident_grid(K kern, int64_t rows)
{
    int nb = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, kern, kVpThreads, 0) != cudaSuccess || nb < 1)
        nb = 1;
    return (int)std::min<int64_t>(std::max<int64_t>(rows, 1), (int64_t)device_sm_count() * nb);
}

}  // namespace

size_t vocab_stats_bytes(int64_t T) { return sizeof(float) * kStatWords * (size_t)std::max<int64_t>(T, 0); }

// The supervised rows in token order as (token, row, -, w) records, and their count
// (the loss path's compaction; it also zeroes token_loss of the other tokens), so
// each CTA of a persistent grid takes an equal share of the rows.
static cudaError_t compact_rows(const VocabShardCall &c, const float *w, float *token_loss, const LossWorkspace &ws,
                                cudaStream_t stream)
{
    LossArgs la{};
    la.mask = c.mask;
    la.row_of_token = c.row_of_token;
    la.w = w;
    la.T = c.T;
    la.num_rows = c.num_rows;
    la.vocab = c.vocab;
    la.mode = TURNOPD_FULL_VOCAB;
    la.token_loss = token_loss;
    la.status = c.status;
    return launch_compaction(la, ws.rows, ws.blk_count, ws.nvalid, stream);
}

cudaError_t launch_vocab_shard_stats(const VocabShardCall &c, float *stats, cudaStream_t stream)
{
    LossWorkspace ws = loss_workspace_layout(c.workspace, c.T);
    // The statistics pass needs neither the records' weights nor the zeroed token
    // losses: both point into the row_wl scratch (T doubles), unused by this call.
    float *scratch = reinterpret_cast<float *>(ws.row_wl);
    cudaError_t e = compact_rows(c, scratch, scratch, ws, stream);
    if (e != cudaSuccess)
        return e;
    ShardIn p{c.zs, c.zt, c.ld, c.vocab, c.num_rows, c.row_of_token, c.mask, c.T, c.status};
    const size_t esz = c.in_dtype == TURNOPD_BF16 ? 2 : 4;
    const bool vec = aligned16(c.zs) && aligned16(c.zt) && (c.ld * esz) % 16 == 0;
    auto kern = c.in_dtype == TURNOPD_BF16 ? (vec ? k_shard_stats<__nv_bfloat16, true> : k_shard_stats<__nv_bfloat16, false>)
                                           : (vec ? k_shard_stats<float, true> : k_shard_stats<float, false>);
    kern<<<resident_grid(kern, c.T), kVpThreads, 0, stream>>>(p, ws.rows, ws.nvalid, stats);
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
static void shard_grad_kernel(const ShardIn &p, bool vec, const LossWorkspace &ws, const float *merged, void *grad,
                              float *tl, cudaStream_t stream)
{
    auto kern = vec ? k_shard_grad<TIn, TOut, true> : k_shard_grad<TIn, TOut, false>;
    kern<<<resident_grid(kern, p.T), kVpThreads, 0, stream>>>(p, ws.rows, ws.nvalid, merged,
                                                                  static_cast<TOut *>(grad), tl, ws.row_wl);
}

cudaError_t launch_vocab_shard_grad(const VocabShardCall &c, const float *merged, cudaStream_t stream)
{
    LossWorkspace ws = loss_workspace_layout(c.workspace, c.T);
    ShardIn p{c.zs, c.zt, c.ld, c.vocab, c.num_rows, c.row_of_token, c.mask, c.T, c.status};
    const size_t esz = c.in_dtype == TURNOPD_BF16 ? 2 : 4;
    const size_t gesz = c.grad_dtype == TURNOPD_BF16 ? 2 : 4;
    const bool vec = aligned16(c.zs) && aligned16(c.zt) && (c.ld * esz) % 16 == 0 &&
                     (!c.grad || (aligned16(c.grad) && (c.ld * gesz) % 16 == 0));
    cudaError_t e = compact_rows(c, c.w, c.token_loss, ws, stream);
    if (e != cudaSuccess)
        return e;
    if (c.grad && (c.flags & TURNOPD_ZERO_MASKED_GRAD))
        launch_zero_masked_grad(c.mask, c.row_of_token, c.T, c.num_rows, c.ld, c.vocab, c.grad, c.grad_dtype, stream);
    const bool bf_in = c.in_dtype == TURNOPD_BF16, bf_out = c.grad_dtype == TURNOPD_BF16;
    if (bf_in && bf_out)
        shard_grad_kernel<__nv_bfloat16, __nv_bfloat16>(p, vec, ws, merged, c.grad, c.token_loss, stream);
    else if (bf_in)
        shard_grad_kernel<__nv_bfloat16, float>(p, vec, ws, merged, c.grad, c.token_loss, stream);
    else if (bf_out)
        shard_grad_kernel<float, __nv_bfloat16>(p, vec, ws, merged, c.grad, c.token_loss, stream);
    else
        shard_grad_kernel<float, float>(p, vec, ws, merged, c.grad, c.token_loss, stream);
    e = cudaGetLastError();
    if (e != cudaSuccess)
        return e;
    launch_loss_sum(ws.row_wl, ws.nvalid, c.loss, c.status, stream);
    return cudaGetLastError();
}

}  // namespace turnopd
