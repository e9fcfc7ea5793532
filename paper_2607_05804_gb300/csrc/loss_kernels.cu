// Per-token OPD loss and student-logit gradient: compaction of supervised
// tokens, the portable one-CTA-per-row kernel, masked-row zero fill and the
// fixed-order loss sum (sm_103a).  The cluster-resident row kernel used for
// aligned bf16 rows lives in rowkl_cluster.cu, the split-row kernel for
// aligned fp32 rows in rowkl_split.cu.
//
// Per supervised token (Eq. opd-rkl), from one read of each logit row:
//   m, S = sum exp(z - m) for both models by an online (rescaling) pass,
//   A = sum exp(z_s - m_s) (z_s - z_t)  ->  KL = A/S_s - (LSE_s - LSE_t),
// then the gradient pass g_v = w p_v ((z_s - z_t)_v - (LSE_s - LSE_t) - KL)
// (full vocabulary) or g_v = w l (delta_vy - p_v) (sampled token; g_y = w l (1 - p_y)
// from student statistics without y, merged back at the end, so that it keeps its
// precision when p_y is near 1).

#include <algorithm>
#include <cfloat>

#include "common.cuh"
#include "row_math.cuh"
#include "kernels.h"

namespace turnopd {

size_t loss_workspace_bytes(int64_t T)
{
    const int64_t nblk = (T + kCompactBlock - 1) / kCompactBlock;
    return align256(sizeof(int4) * (size_t)T) + align256(sizeof(int32_t) * (size_t)(nblk + 1)) +
           align256(sizeof(int32_t)) + align256(sizeof(double) * (size_t)T) + 256;
}

LossWorkspace loss_workspace_layout(void *ws, int64_t T)
{
    const int64_t nblk = (T + kCompactBlock - 1) / kCompactBlock;
    char *p = static_cast<char *>(ws);
    LossWorkspace l;
    l.rows = reinterpret_cast<int4 *>(p);
    p += align256(sizeof(int4) * (size_t)T);
    l.blk_count = reinterpret_cast<int32_t *>(p);
    p += align256(sizeof(int32_t) * (size_t)(nblk + 1));
    l.nvalid = reinterpret_cast<int32_t *>(p);
    p += align256(sizeof(int32_t));
    l.row_wl = reinterpret_cast<double *>(p);
    return l;
}

// ---------------------------------------------------------------- compaction

struct CompactIn {
    const uint8_t *mask;
    const int32_t *row_of_token;
    const int32_t *sampled_ids;
    const float *w;
    int64_t num_rows;
    int64_t vocab;
    int64_t T;
    int32_t mode;
    float *token_loss;
    int32_t *status;
};

constexpr int kCompactThreads = 256;
constexpr int kPerThread = kCompactBlock / kCompactThreads;  // 16 contiguous tokens

// The kPerThread tokens i0, i0 + 1, ... of one thread.  Token i enters the row list
// iff it is supervised and its row (and sampled id) are in range; a supervised token
// out of range is "bad" (its loss is 0 and a range error is recorded).  Every array
// read is issued for all the thread's tokens before any is used, so the checks cost
// one memory round trip per array rather than one per token.
struct TokenSlice {
    uint32_t valid, bad;  // bit k: token i0 + k
    int32_t r[kPerThread], y[kPerThread];
};

__device__ __forceinline__ void load_tokens(const CompactIn &c, int64_t i0, TokenSlice &t)
{
    uint32_t sup = 0;
#pragma unroll
    for (int k = 0; k < kPerThread; ++k)
        if (i0 + k < c.T && c.mask[i0 + k])
            sup |= 1u << k;
    const bool sampled = c.mode == TURNOPD_SAMPLED_TOKEN;
#pragma unroll
    for (int k = 0; k < kPerThread; ++k) {
        const bool m = (sup >> k) & 1u;
        t.r[k] = m && c.row_of_token ? c.row_of_token[i0 + k] : (int32_t)(i0 + k);
        t.y[k] = m && sampled ? c.sampled_ids[i0 + k] : -1;
    }
    t.valid = t.bad = 0;
#pragma unroll
    for (int k = 0; k < kPerThread; ++k) {
        if (!((sup >> k) & 1u))
            continue;
        bool ok = t.r[k] >= 0 && (int64_t)t.r[k] < c.num_rows;
        if (ok && sampled)
            ok = t.y[k] >= 0 && (int64_t)t.y[k] < c.vocab;
        if (ok)
            t.valid |= 1u << k;
        else
            t.bad |= 1u << k;
    }
}

__global__ void k_compact_count(CompactIn c, int32_t *__restrict__ blk_count)
{
    // a programmatic dependent of the caller's work; the scatter kernel may start
    // once this has begun: its token loads do not need these counts
    pdl_begin();
    __shared__ int warp_tot[kCompactThreads / 32];
    const int64_t i0 = (int64_t)blockIdx.x * kCompactBlock + (int64_t)threadIdx.x * kPerThread;
    TokenSlice t;
    load_tokens(c, i0, t);
    if (t.bad)
        set_status(c.status, TURNOPD_ERR_TOKEN_RANGE);
#pragma unroll
    for (int k = 0; k < kPerThread; ++k)
        if (i0 + k < c.T && !((t.valid >> k) & 1u))
            c.token_loss[i0 + k] = 0.f;
    int n = warp_sum_i32(__popc(t.valid));
    if ((threadIdx.x & 31) == 0)
        warp_tot[threadIdx.x >> 5] = n;
    __syncthreads();
    if (threadIdx.x == 0) {
        int tot = 0;
        for (int wi = 0; wi < kCompactThreads / 32; ++wi)
            tot += warp_tot[wi];
        blk_count[blockIdx.x] = tot;
    }
}

// Launched as a programmatic dependent of k_compact_count: the thread's tokens are
// loaded before the wait for the block counts.
__global__ void k_compact_scatter(CompactIn c, const int32_t *__restrict__ blk_count,
                                  int4 *__restrict__ rows, int32_t *__restrict__ nvalid)
{
    __shared__ int warp_tot[kCompactThreads / 32];
    __shared__ int warp_off[kCompactThreads / 32];
    __shared__ int64_t base_s;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t i0 = (int64_t)blockIdx.x * kCompactBlock + (int64_t)threadIdx.x * kPerThread;
    TokenSlice t;
    load_tokens(c, i0, t);
    float wv[kPerThread];
#pragma unroll
    for (int k = 0; k < kPerThread; ++k)
        wv[k] = ((t.valid >> k) & 1u) ? c.w[i0 + k] : 0.f;
    asm volatile("griddepcontrol.wait;" ::: "memory");  // every block's count is written
    // exclusive prefix over the preceding blocks
    int64_t pre = 0;
    for (int k = threadIdx.x; k < (int)blockIdx.x; k += kCompactThreads)
        pre += blk_count[k];
    pre = warp_sum_i64(pre);
    if (lane == 0)
        warp_tot[warp] = (int)pre;  // fits: a prefix never exceeds T < 2^31
    __syncthreads();
    if (threadIdx.x == 0) {
        int64_t s = 0;
        for (int wi = 0; wi < kCompactThreads / 32; ++wi)
            s += warp_tot[wi];
        base_s = s;
    }
    __syncthreads();
    const int64_t base = base_s;

    const uint32_t bits = t.valid;
    const int n = __popc(bits);
    // exclusive scan of n across the block (thread order = token order)
    int incl = n;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o)
            incl += y;
    }
    __syncthreads();  // warp_tot reuse
    if (lane == 31)
        warp_tot[warp] = incl;
    __syncthreads();
    if (threadIdx.x == 0) {
        int s = 0;
        for (int wi = 0; wi < kCompactThreads / 32; ++wi) {
            warp_off[wi] = s;
            s += warp_tot[wi];
        }
        if (blockIdx.x == gridDim.x - 1) {
            *nvalid = (int32_t)(base + s);
            *sum_ticket(nvalid) = 0u;  // for the loss sum after the row grids
        }
    }
    __syncthreads();
    int64_t pos = base + warp_off[warp] + (incl - n);
#pragma unroll
    for (int k = 0; k < kPerThread; ++k)
        if ((bits >> k) & 1u)
            rows[pos++] = make_int4((int32_t)(i0 + k), t.r[k], t.y[k], __float_as_int(wv[k]));
}

// ---------------------------------------------------------------- row kernel

constexpr int kRowThreads = 256;

template <typename TIn, typename TOut, bool VEC>
__global__ void __launch_bounds__(kRowThreads)
k_row_portable(RowIn p)
{
    __shared__ Student red_s[kRowThreads / 32];
    __shared__ Teacher red_t[kRowThreads / 32];
    __shared__ float bc[6];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nvalid = *p.nvalid;
    const TIn *zs = static_cast<const TIn *>(p.zs);
    const TIn *zt = static_cast<const TIn *>(p.zt);
    TOut *grad = static_cast<TOut *>(p.grad);
    constexpr int N = Vec<TIn>::N;
    const int64_t V = p.vocab;
    const int64_t nvec = VEC ? V / N : 0;

    for (int j = blockIdx.x; j < nvalid; j += gridDim.x) {
        const int4 meta = p.rows[j];
        const int i = meta.x;
        const int64_t r = meta.y;
        const TIn *rs = zs + r * p.ld;
        const TIn *rt = zt + r * p.ld;
        Student s = student_empty();
        Teacher t = teacher_empty();
        // a sampled-token row leaves y out of the student statistics (add_sampled_term
        // brings its term back at the merge): in a vector its logit reads as the lowest
        // finite value (never the maximum beside the other N - 1, adds 0); read alone
        // it folds into the teacher only
        const int64_t ys = p.mode == TURNOPD_SAMPLED_TOKEN ? (int64_t)meta.z : -1;
        if (VEC) {
            for (int64_t q = threadIdx.x; q < nvec; q += kRowThreads) {
                float a[N], b[N];
                Vec<TIn>::load(rs + q * N, a);
                Vec<TIn>::load(rt + q * N, b);
                if (ys >= 0 && q == ys / N) {
#pragma unroll
                    for (int k = 0; k < N; ++k)
                        if (k == (int)(ys % N))
                            a[k] = -FLT_MAX;
                }
                accumulate<N>(s, t, a, b);
            }
        }
        for (int64_t v = nvec * N + threadIdx.x; v < V; v += kRowThreads) {
            const float a = to_float(rs[v]), b = to_float(rt[v]);
            if (v == ys)
                accumulate_teacher(t, b);
            else
                accumulate<1>(s, t, &a, &b);
        }
        s = warp_merge(s);
        t = warp_merge(t);
        if (lane == 0) {
            red_s[warp] = s;
            red_t[warp] = t;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            Student S = red_s[0];
            Teacher U = red_t[0];
            for (int k = 1; k < kRowThreads / 32; ++k) {
                S = student_merge(S, red_s[k]);
                U = teacher_merge(U, red_t[k]);
            }
            float omp = 0.f;  // 1 - p_y (sampled)
            if (ys >= 0)
                omp = add_sampled_term(S, to_float(rs[ys]));
            const RowConst rc = row_const(S, U);
            float ell = rc.kl;
            if (ys >= 0)
                ell = (to_float(rs[ys]) - to_float(rt[ys])) - rc.dl;
            const float wi = __int_as_float(meta.w);
            if (!isfinite(rc.lse_s) || !isfinite(rc.lse_t) || !isfinite(ell))
                set_status(p.status, TURNOPD_ERR_NONFINITE);
            p.token_loss[i] = ell;
            p.row_wl[j] = (double)wi * (double)ell;
            bc[0] = rc.lse_s;
            bc[1] = rc.d;
            bc[2] = rc.cp;  // g = w p (((z_s - z_t) - d) - cp)
            bc[3] = wi;
            bc[4] = wi * ell;
            bc[5] = wi * ell * omp;  // g_y = w l (1 - p_y)
        }
        __syncthreads();
        if (grad) {
            const float nl = -bc[0] * kLog2e, d = bc[1], cp = bc[2], wi = bc[3], wl = bc[4], gy = bc[5];
            const bool sampled = p.mode == TURNOPD_SAMPLED_TOKEN;
            const int64_t y = sampled ? (int64_t)meta.z : -1;
            TOut *gr = grad + r * p.ld;
            if (VEC) {
                for (int64_t q = threadIdx.x; q < nvec; q += kRowThreads) {
                    float a[N], b[N], g[N];
                    Vec<TIn>::load(rs + q * N, a);
                    Vec<TIn>::load(rt + q * N, b);
#pragma unroll
                    for (int k = 0; k < N; ++k) {
                        const float pv = ex2(fmaf(a[k], kLog2e, nl));
                        g[k] = sampled ? ((q * N + k) == y ? gy : -wl * pv)
                                       : wi * pv * (((a[k] - b[k]) - d) - cp);
                    }
                    store_vec<TOut, N>(gr + q * N, g);
                }
            }
            for (int64_t v = nvec * N + threadIdx.x; v < V; v += kRowThreads) {
                const float a = to_float(rs[v]), b = to_float(rt[v]);
                const float pv = ex2(fmaf(a, kLog2e, nl));
                const float g = sampled ? (v == y ? gy : -wl * pv) : wi * pv * (((a - b) - d) - cp);
                gr[v] = from_float<TOut>(g);
            }
        }
        __syncthreads();  // bc / red reuse by the next row
    }
}

// ---------------------------------------------------------------- zero fill

template <typename TOut>
__global__ void k_zero_masked(const uint8_t *__restrict__ mask, const int32_t *__restrict__ rot,
                              int64_t T, int64_t num_rows, int64_t ld, int64_t vocab, TOut *grad)
{
    for (int64_t i = blockIdx.x; i < T; i += gridDim.x) {
        if (mask[i])
            continue;
        const int64_t r = rot ? (int64_t)rot[i] : i;
        if (r < 0 || r >= num_rows)
            continue;
        // zeros are all-zero bits in both output types: 16-byte stores between an
        // element-wise head (up to the first 16-byte boundary) and tail
        TOut *g = grad + r * ld;
        const int64_t to16 = (int64_t)(((16u - (reinterpret_cast<uintptr_t>(g) & 15u)) & 15u) / sizeof(TOut));
        const int64_t head = to16 < vocab ? to16 : vocab;
        for (int64_t v = threadIdx.x; v < head; v += blockDim.x)
            g[v] = from_float<TOut>(0.f);
        uint4 *body = reinterpret_cast<uint4 *>(g + head);
        const int64_t nvec = (vocab - head) * (int64_t)sizeof(TOut) / 16;
        for (int64_t q = threadIdx.x; q < nvec; q += blockDim.x)
            body[q] = make_uint4(0u, 0u, 0u, 0u);
        for (int64_t v = head + nvec * (int64_t)(16 / sizeof(TOut)) + threadIdx.x; v < vocab; v += blockDim.x)
            g[v] = from_float<TOut>(0.f);
    }
}

// ---------------------------------------------------------------- loss sum

// loss = sum_j row_wl[j] over the compacted rows (= token order), fixed tree.
// sum_i w_i l_i over the row list in a fixed order, on kSumCTAs CTAs: CTA c sums a fixed
// chunk of the rows (threads strided, then the warps' xor trees, then in warp order),
// and the CTA that finishes last adds the partials by a fixed xor tree.  One CTA alone
// was bound by its SM's fp64 rate (a small fraction of the fp32 rate on this part).
// A programmatic dependent of the row grid.
constexpr int kSumThreads = 256;

__global__ void __launch_bounds__(kSumThreads) k_loss_sum(const double *__restrict__ row_wl,
                                                          int32_t *__restrict__ nvalid,
                                                          double *__restrict__ loss, int32_t *status)
{
    __shared__ double part[kSumThreads / 32];
    __shared__ int last;
    // every row's w l is written (and the turn statistics after this may launch)
    pdl_begin();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int n = *nvalid;
    const int chunk = (n + kSumCTAs - 1) / kSumCTAs;
    const int j0 = (int)blockIdx.x * chunk, j1 = min(n, j0 + chunk);
    double s4[4] = {0.0, 0.0, 0.0, 0.0};
    int j = j0 + (int)threadIdx.x;
    for (; j + 3 * kSumThreads < j1; j += 4 * kSumThreads) {
#pragma unroll
        for (int u = 0; u < 4; ++u)
            s4[u] += row_wl[j + u * kSumThreads];
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
        if (j + u * kSumThreads < j1)
            s4[u] += row_wl[j + u * kSumThreads];
    double s = warp_sum_f64((s4[0] + s4[1]) + (s4[2] + s4[3]));
    if (lane == 0)
        part[warp] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < kSumThreads / 32; ++w)
            t += part[w];
        sum_partials(nvalid)[blockIdx.x] = t;
        __threadfence();
        last = atomicAdd(sum_ticket(nvalid), 1u) == (unsigned)(kSumCTAs - 1);
    }
    __syncthreads();
    if (last && warp == 0) {
        __threadfence();
        double v = lane < kSumCTAs ? __ldcg(sum_partials(nvalid) + lane) : 0.0;
        v = warp_sum_f64(v);
        if (lane == 0) {
            if (!isfinite(v))
                set_status(status, TURNOPD_ERR_NONFINITE);
            *loss = v;
            *sum_ticket(nvalid) = 0u;
        }
    }
}

// ---------------------------------------------------------------- launcher


template <typename TIn, typename TOut>
static cudaError_t launch_portable(const RowIn &p, bool vec, int grid, cudaStream_t stream)
{
    if (vec)
        k_row_portable<TIn, TOut, true><<<grid, kRowThreads, 0, stream>>>(p);
    else
        k_row_portable<TIn, TOut, false><<<grid, kRowThreads, 0, stream>>>(p);
    return cudaGetLastError();
}

static bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

cudaError_t launch_compaction(const LossArgs &a, int4 *rows, int32_t *blk_count, int32_t *nvalid,
                              cudaStream_t stream)
{
    const int nblk = (int)((a.T + kCompactBlock - 1) / kCompactBlock);
    CompactIn c{a.mask, a.row_of_token, a.sampled_ids, a.w, a.num_rows, a.vocab, a.T, a.mode,
                a.token_loss, a.status};
    cudaError_t e0 = launch_dependent(k_compact_count, dim3(nblk), dim3(kCompactThreads), 0, stream, c, blk_count);
    if (e0 != cudaSuccess)
        return e0;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.gridDim = dim3(nblk);
    cfg.blockDim = dim3(kCompactThreads);
    cfg.stream = stream;
    const int32_t *cnt = blk_count;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, k_compact_scatter, c, cnt, rows, nvalid);
    return e != cudaSuccess ? e : cudaGetLastError();
}

// A programmatic dependent of the kernel before it: row grids that signal early let it
// take the first SM they free, and it waits for their completion before reading.
void launch_loss_sum(const double *row_wl, int32_t *nvalid, double *loss, int32_t *status,
                     cudaStream_t stream)
{
    launch_dependent(k_loss_sum, dim3(kSumCTAs), dim3(kSumThreads), 0, stream, row_wl, nvalid, loss, status);
}

void launch_zero_masked_f32(const uint8_t *mask, int64_t T, int64_t d, float *out, cudaStream_t stream)
{
    const int grid = (int)std::min<int64_t>(std::max<int64_t>(T, 1), (int64_t)device_sm_count() * 8);
    k_zero_masked<float><<<grid, 256, 0, stream>>>(mask, nullptr, T, T, d, d, out);
}

void launch_zero_masked_grad(const uint8_t *mask, const int32_t *row_of_token, int64_t T, int64_t num_rows,
                             int64_t ld, int64_t vocab, void *grad, int32_t grad_dtype, cudaStream_t stream)
{
    const int grid = (int)std::min<int64_t>(std::max<int64_t>(T, 1), (int64_t)device_sm_count() * 8);
    if (grad_dtype == TURNOPD_BF16)
        k_zero_masked<__nv_bfloat16><<<grid, 256, 0, stream>>>(mask, row_of_token, T, num_rows, ld, vocab,
                                                                static_cast<__nv_bfloat16 *>(grad));
    else
        k_zero_masked<float><<<grid, 256, 0, stream>>>(mask, row_of_token, T, num_rows, ld, vocab,
                                                        static_cast<float *>(grad));
}

cudaError_t launch_loss(const LossArgs &a, const LossWorkspace &ws, cudaStream_t stream)
{
    cudaError_t e = launch_compaction(a, ws.rows, ws.blk_count, ws.nvalid, stream);
    if (e != cudaSuccess)
        return e;

    const int sms = device_sm_count();
    if (a.grad && (a.flags & TURNOPD_ZERO_MASKED_GRAD))
        launch_zero_masked_grad(a.mask, a.row_of_token, a.T, a.num_rows, a.ld, a.vocab, a.grad, a.grad_dtype,
                                stream);

    RowIn p{a.zs, a.zt, a.ld, a.vocab, a.row_of_token, a.sampled_ids, a.w, a.mode, a.grad,
            a.token_loss, ws.row_wl, ws.rows, ws.nvalid, a.status, 0, 0};
    bool done = false;
    if (!(a.flags & TURNOPD_FORCE_PORTABLE)) {
        e = a.in_dtype == TURNOPD_BF16 ? launch_row_cluster(p, a.grad_dtype == TURNOPD_F32, stream, &done)
                                        : launch_row_split(p, a.grad_dtype == TURNOPD_F32, stream, &done);
        if (e != cudaSuccess)
            return e;
    }
    if (!done) {
        const size_t esz = a.in_dtype == TURNOPD_BF16 ? 2 : 4;
        const bool vec = aligned16(a.zs) && aligned16(a.zt) && (!a.grad || aligned16(a.grad)) &&
                         ((size_t)a.ld * esz) % 16 == 0;
        const int grid = (int)std::min<int64_t>(std::max<int64_t>(a.T, 1), (int64_t)sms * 8);
        const bool g32 = a.grad_dtype == TURNOPD_F32;
        if (a.in_dtype == TURNOPD_BF16)
            e = g32 ? launch_portable<__nv_bfloat16, float>(p, vec, grid, stream)
                    : launch_portable<__nv_bfloat16, __nv_bfloat16>(p, vec, grid, stream);
        else
            e = g32 ? launch_portable<float, float>(p, vec, grid, stream)
                    : launch_portable<float, __nv_bfloat16>(p, vec, grid, stream);
        if (e != cudaSuccess)
            return e;
    }
    launch_loss_sum(ws.row_wl, ws.nvalid, a.loss, a.status, stream);
    return cudaGetLastError();
}

}  // namespace turnopd
