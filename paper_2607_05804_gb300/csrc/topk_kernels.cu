// Teacher top-K reverse KL: the paper's practical loss (loss_mode
// topk_reverse_kl, support size K_top = distill_topk; Algorithm 1, "top-K
// reverse-KL token losses").  For a supervised row, S = the K vocabulary ids
// of largest teacher logit (the lower id first among equal logits); both
// distributions are renormalised over S:
//   l   = sum_{v in S} ps_v (log ps_v - log pt_v)
//   g_v = w ps_v (log ps_v - log pt_v - l)  on S, 0 elsewhere (= w dl/dz_s).
//
// One CTA per row at a time (persistent).  Selection with 64-bit keys
// (order-preserving logit bits << 32 | ~id, so larger key = larger logit,
// then lower id):
//   pass A   one read of the teacher row: every thread keeps the 4 largest
//            keys of its elements; a vector of 8 is looked at element by
//            element only when its packed max beats the thread's 4th key;
//   bound    tau = the K-th largest logit among the 4 x 512 held keys: a
//            lower bound of the row's K-th largest (a subset's K-th largest
//            never exceeds the set's);
//   collect  held keys >= tau go to a shared-memory buffer; a thread whose
//            4th held key is >= tau may hold fewer than all of its keys >= tau
//            and rescans its own elements (rare);  a buffer overflow (rows of
//            many equal logits) raises tau to the K-th largest buffered key
//            and collects again (bounded rounds);
//   select   the exact K-th largest buffered key by radix select, then each
//            selected key's rank among the selected gives its position.
// The KL over S is evaluated by one warp in fp32 with
// l = E_p[z_s - z_t] - (LSE_s - LSE_t) and g_v = w p_v ((z_s - z_t)_v - E_p[.]).

#include <cuda_bf16.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace turnopd {
namespace {

constexpr int kTkThreads = 512;
constexpr int kTkHold = 4;        // keys each thread keeps during pass A
constexpr int kTkCap = 4096;      // candidate buffer (keys)
constexpr int kTkRounds = 16;     // bound on overflow rounds

__device__ __forceinline__ uint32_t ord16(uint32_t u)
{
    u &= 0xFFFFu;
    if (u == 0x8000u)
        u = 0;  // -0 and +0 are the same logit
    return (u & 0x8000u) ? (~u & 0xFFFFu) : (u | 0x8000u);
}

__device__ __forceinline__ uint32_t ord32(uint32_t u)
{
    if (u == 0x80000000u)
        u = 0;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ uint64_t mkkey(uint32_t ord, uint32_t id)
{
    return ((uint64_t)ord << 32) | (uint32_t)(~id);
}

__device__ __forceinline__ uint32_t key_id(uint64_t k) { return ~(uint32_t)k; }

template <bool BF16>
__device__ __forceinline__ float key_value(uint64_t k)
{
    const uint32_t o = (uint32_t)(k >> 32);
    if (BF16) {
        const uint32_t bits = (o & 0x8000u) ? (o & 0x7FFFu) : (~o & 0xFFFFu);
        return __uint_as_float(bits << 16);
    }
    const uint32_t bits = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
    return __uint_as_float(bits);
}

__device__ __forceinline__ uint32_t bf16_max8_ord(const uint4 &v)
{
    const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162 *>(&v.x);
    const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162 *>(&v.y);
    const __nv_bfloat162 c = *reinterpret_cast<const __nv_bfloat162 *>(&v.z);
    const __nv_bfloat162 d = *reinterpret_cast<const __nv_bfloat162 *>(&v.w);
    const __nv_bfloat162 m = __hmax2(__hmax2(a, b), __hmax2(c, d));
    const __nv_bfloat16 mm = __hmax(m.x, m.y);
    return ord16(__bfloat16_as_ushort(mm));
}

// Visit this thread's elements of one row in increasing id order, calling
// f(key) for every element whose logit may reach `*thr` (an ordered value;
// elements of smaller ordered value may be skipped).  f may raise *thr.
template <bool BF16, class F>
__device__ __forceinline__ void scan_row(const void *row, int64_t V, bool vec_ok, const uint32_t *thr, F &&f)
{
    constexpr int EPV = BF16 ? 8 : 4;  // elements per 16-byte vector
    const int64_t nvec = vec_ok ? V / EPV : 0;
    const uint4 *rv = static_cast<const uint4 *>(row);
    for (int64_t j0 = threadIdx.x; j0 < nvec; j0 += 4 * kTkThreads) {
        uint4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int64_t j = j0 + (int64_t)u * kTkThreads;
            if (j < nvec)
                v[u] = __ldg(rv + j);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int64_t j = j0 + (int64_t)u * kTkThreads;
            if (j >= nvec)
                break;
            const uint32_t id0 = (uint32_t)(j * EPV);
            if (BF16) {
                if (bf16_max8_ord(v[u]) < *thr)
                    continue;
                const uint32_t w4[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const uint32_t o = ord16(e & 1 ? w4[e >> 1] >> 16 : w4[e >> 1]);
                    if (o >= *thr)
                        f(mkkey(o, id0 + e));
                }
            } else {
                const float x0 = __uint_as_float(v[u].x), x1 = __uint_as_float(v[u].y);
                const float x2 = __uint_as_float(v[u].z), x3 = __uint_as_float(v[u].w);
                if (ord32(__float_as_uint(fmaxf(fmaxf(x0, x1), fmaxf(x2, x3)))) < *thr)
                    continue;
                const uint32_t w4[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const uint32_t o = ord32(w4[e]);
                    if (o >= *thr)
                        f(mkkey(o, id0 + e));
                }
            }
        }
    }
    // elements not covered by whole aligned vectors
    for (int64_t e = nvec * EPV + threadIdx.x; e < V; e += kTkThreads) {
        const uint32_t o = BF16 ? ord16(static_cast<const uint16_t *>(row)[e])
                                : ord32(static_cast<const uint32_t *>(row)[e]);
        if (o >= *thr)
            f(mkkey(o, (uint32_t)e));
    }
}

// Block-wide radix select: the K-th largest of the nonzero keys in keys[0, n)
// (keys are unique; 0 marks an empty slot), deciding bytes hi_byte..lo_byte.
// Returns t such that {keys >= t} holds the K largest keys when lo_byte = 0
// (exactly K), or, when lo_byte > 0, the K-th largest key with its lower bytes
// cleared (every key of equal upper bytes is >= t).  Returns 0 when fewer than
// K keys are present.  Stops early once the chosen bin holds exactly the
// remaining count.  All threads call it; it synchronises the block.
struct SelScratch {
    uint32_t hist[256];
    int bin, need;
};

__device__ uint64_t block_kth_largest(const uint64_t *keys, int n, int K, int hi_byte, int lo_byte,
                                      SelScratch &sc)
{
    const int tid = threadIdx.x, lane = tid & 31;
    uint64_t prefix = 0, mask = 0;
    int need = K;
    for (int byte = hi_byte; byte >= lo_byte; --byte) {
        for (int i = tid; i < 256; i += kTkThreads)
            sc.hist[i] = 0;
        __syncthreads();
        const int sh = 8 * byte;
        for (int i = tid; i < n; i += kTkThreads) {
            const uint64_t k = keys[i];
            if (k != 0 && (k & mask) == prefix)
                atomicAdd(&sc.hist[(k >> sh) & 255u], 1u);
        }
        __syncthreads();
        if (tid < 32) {
            int c[8], tot = 0;
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                c[e] = (int)sc.hist[255 - 8 * lane - e];
                tot += c[e];
            }
            int incl = tot;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int y = __shfl_up_sync(0xffffffffu, incl, off);
                if (lane >= off)
                    incl += y;
            }
            const int excl = incl - tot;
            const unsigned hit = __ballot_sync(0xffffffffu, excl < need && incl >= need);
            if (hit == 0u) {
                if (lane == 0)
                    sc.bin = -1;
            } else if (lane == __ffs(hit) - 1) {
                int cum = excl;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    if (cum + c[e] >= need) {
                        sc.bin = 255 - 8 * lane - e;
                        // remaining count inside the bin; negative marks "the bin is exactly it"
                        sc.need = (cum + c[e] == need) ? -(need - cum) : need - cum;
                        break;
                    }
                    cum += c[e];
                }
            }
        }
        __syncthreads();
        const int bin = sc.bin, nd = sc.need;
        __syncthreads();
        if (bin < 0)
            return 0;
        prefix |= (uint64_t)bin << sh;
        mask |= (uint64_t)255u << sh;
        if (nd < 0)  // every key of this prefix is selected
            return prefix;
        need = nd;
    }
    return prefix;
}

struct TopkArgs {
    const void *zs, *zt;
    int64_t ld, vocab;
    int32_t K;
    const int4 *rows;
    const int32_t *nvalid;
    int32_t *topk_ids;   // [T, K] or null
    float *topk_grad;    // [T, K] or null
    void *grad;          // [R, ld] or null
    int32_t grad_dtype;
    float *token_loss;
    double *row_wl;
    int32_t *status;
};

// Dynamic shared memory: held keys, candidate buffer, the selected keys and
// their gradients.
constexpr size_t kTkSmem = sizeof(uint64_t) * (kTkThreads * kTkHold + kTkCap + kTopkMaxK) +
                           sizeof(float) * kTopkMaxK;

template <bool BF16>
__global__ void __launch_bounds__(kTkThreads, 2) k_topk_rows(TopkArgs a)
{
    extern __shared__ uint64_t tk_smem[];
    uint64_t *s_held = tk_smem;
    uint64_t *s_cand = s_held + kTkThreads * kTkHold;
    uint64_t *s_top = s_cand + kTkCap;
    float *s_g = reinterpret_cast<float *>(s_top + kTopkMaxK);
    __shared__ SelScratch s_sel;
    __shared__ int s_n, s_over;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int K = a.K;
    const int n_rows = *a.nvalid;
    const size_t esz = BF16 ? 2 : 4;
    const int hi_val = BF16 ? 5 : 7;  // top byte of the ordered logit inside a key
    const bool base_ok = ((reinterpret_cast<uintptr_t>(a.zt) | (uintptr_t)(a.ld * esz)) & 15u) == 0;

    for (int j = blockIdx.x; j < n_rows; j += gridDim.x) {
        const int4 m = a.rows[j];
        const int tok = m.x;
        const float w = __int_as_float(m.w);
        const char *zt_row = static_cast<const char *>(a.zt) + (size_t)m.y * (size_t)a.ld * esz;
        const char *zs_row = static_cast<const char *>(a.zs) + (size_t)m.y * (size_t)a.ld * esz;

        // ---- pass A: this thread's 4 largest keys
        uint64_t h0 = 0, h1 = 0, h2 = 0, h3 = 0;
        uint32_t thr = 1;  // admit every finite logit until 4 are held
        scan_row<BF16>(zt_row, a.vocab, base_ok, &thr, [&](uint64_t k) {
            if (k <= h3)
                return;
            h3 = k;
            if (h3 > h2) { const uint64_t t = h2; h2 = h3; h3 = t; }
            if (h2 > h1) { const uint64_t t = h1; h1 = h2; h2 = t; }
            if (h1 > h0) { const uint64_t t = h0; h0 = h1; h1 = t; }
            // a later element (larger id) needs a strictly larger logit than the 4th key
            if (h3 != 0)
                thr = (uint32_t)(h3 >> 32) + 1u;
        });
        s_held[tid * kTkHold + 0] = h0;
        s_held[tid * kTkHold + 1] = h1;
        s_held[tid * kTkHold + 2] = h2;
        s_held[tid * kTkHold + 3] = h3;
        if (tid == 0) {
            s_n = 0;
            s_over = 0;
        }
        __syncthreads();

        // ---- lower bound on the K-th largest logit (value bytes only)
        uint64_t tau = block_kth_largest(s_held, kTkThreads * kTkHold, K, hi_val, 4, s_sel);
        uint32_t tau_ord = (uint32_t)(tau >> 32);
        if (tau_ord == 0)
            tau_ord = 1;

        auto append = [&](uint64_t k) {
            const int p = atomicAdd(&s_n, 1);
            if (p < kTkCap)
                s_cand[p] = k;
            else
                s_over = 1;
        };
        // ---- collect: held keys >= tau, and a rescan where the 4 held may not be all
        const uint64_t hk[4] = {h0, h1, h2, h3};
#pragma unroll
        for (int q = 0; q < 4; ++q)
            if (hk[q] != 0 && hk[q] >= tau)
                append(hk[q]);
        if (h3 != 0 && h3 >= tau) {
            const uint64_t lim = h3;
            scan_row<BF16>(zt_row, a.vocab, base_ok, &tau_ord, [&](uint64_t k) {
                if (k >= tau && k < lim)
                    append(k);
            });
        }
        __syncthreads();
        // ---- overflow: raise tau to the K-th largest buffered key and collect again
        for (int round = 0; s_over && round < kTkRounds; ++round) {
            tau = block_kth_largest(s_cand, kTkCap, K, 7, 0, s_sel);
            tau_ord = (uint32_t)(tau >> 32);
            if (tau_ord == 0)
                tau_ord = 1;
            if (tid == 0) {
                s_n = 0;
                s_over = 0;
            }
            __syncthreads();
            scan_row<BF16>(zt_row, a.vocab, base_ok, &tau_ord, [&](uint64_t k) {
                if (k >= tau)
                    append(k);
            });
            __syncthreads();
        }
        const bool failed = s_over != 0;
        const int nc = min(s_n, kTkCap);
        __syncthreads();
        if (failed) {
            if (tid == 0) {
                set_status(a.status, TURNOPD_ERR_UNSUPPORTED);
                a.token_loss[tok] = 0.f;
                a.row_wl[j] = 0.0;
            }
            continue;
        }
        // ---- the K largest: exact K-th key, then positions by rank
        const uint64_t kth = block_kth_largest(s_cand, nc, K, 7, 0, s_sel);
        for (int i = tid; i < nc; i += kTkThreads) {
            const uint64_t k = s_cand[i];
            if (k < kth)
                continue;
            int rank = 0;
            for (int i2 = 0; i2 < nc; ++i2)
                rank += s_cand[i2] > k;
            if (rank < K)
                s_top[rank] = k;
        }
        __syncthreads();

        // ---- KL over S (one warp, fp32)
        if (warp == 0) {
            float m_s = -INFINITY, m_t = -INFINITY;
            for (int r = lane; r < K; r += 32) {
                const uint32_t id = key_id(s_top[r]);
                const float zt_v = key_value<BF16>(s_top[r]);
                const float zs_v = BF16 ? __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(zs_row)[id])
                                        : reinterpret_cast<const float *>(zs_row)[id];
                s_g[r] = zs_v;  // student logit, kept for the second sweep
                m_s = fmaxf(m_s, zs_v);
                m_t = fmaxf(m_t, zt_v);
            }
            m_s = warp_max_f(m_s);
            m_t = warp_max_f(m_t);
            float s_s = 0.f, s_t = 0.f, a_sd = 0.f;
            for (int r = lane; r < K; r += 32) {
                const float zs_v = s_g[r], zt_v = key_value<BF16>(s_top[r]);
                const float es = expf(zs_v - m_s);
                s_s += es;
                s_t += expf(zt_v - m_t);
                a_sd = fmaf(es, zs_v - zt_v, a_sd);
            }
            s_s = warp_sum_f(s_s);
            s_t = warp_sum_f(s_t);
            a_sd = warp_sum_f(a_sd);
            const float ep = a_sd / s_s;                              // E_p[z_s - z_t]
            const float c = (m_s - m_t) + logf(s_s / s_t);            // LSE_s - LSE_t
            const float ell = ep - c;
            for (int r = lane; r < K; r += 32) {
                const float zs_v = s_g[r], zt_v = key_value<BF16>(s_top[r]);
                const float p = expf(zs_v - m_s) / s_s;
                const float g = w * p * ((zs_v - zt_v) - ep);
                s_g[r] = g;
                if (a.topk_ids)
                    a.topk_ids[(size_t)tok * K + r] = (int32_t)key_id(s_top[r]);
                if (a.topk_grad)
                    a.topk_grad[(size_t)tok * K + r] = g;
            }
            if (lane == 0) {
                if (!isfinite(ell))
                    set_status(a.status, TURNOPD_ERR_NONFINITE);
                a.token_loss[tok] = ell;
                a.row_wl[j] = (double)w * (double)ell;
            }
        }
        // ---- dense gradient row: zeros, then the K entries
        if (a.grad) {
            const size_t gesz = a.grad_dtype == TURNOPD_BF16 ? 2 : 4;
            char *grow = static_cast<char *>(a.grad) + (size_t)m.y * (size_t)a.ld * gesz;
            const int64_t bytes = a.vocab * (int64_t)gesz;
            const bool g_ok = ((reinterpret_cast<uintptr_t>(grow)) & 15u) == 0;
            const int64_t nv16 = g_ok ? bytes / 16 : 0;
            for (int64_t q = tid; q < nv16; q += kTkThreads)
                reinterpret_cast<uint4 *>(grow)[q] = make_uint4(0, 0, 0, 0);
            for (int64_t b = nv16 * 16 + tid; b < bytes; b += kTkThreads)
                grow[b] = 0;
            __syncthreads();
            for (int r = tid; r < K; r += kTkThreads) {
                const uint32_t id = key_id(s_top[r]);
                if (a.grad_dtype == TURNOPD_BF16)
                    reinterpret_cast<__nv_bfloat16 *>(grow)[id] = __float2bfloat16_rn(s_g[r]);
                else
                    reinterpret_cast<float *>(grow)[id] = s_g[r];
            }
        }
        __syncthreads();
    }
}

// Masked tokens' sparse rows: ids -1, gradients 0.
__global__ void k_topk_zero_masked(const uint8_t *mask, int64_t T, int32_t K, int32_t *ids, float *g)
{
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < T * K; i += (int64_t)gridDim.x * blockDim.x) {
        if (mask[i / K])
            continue;
        if (ids)
            ids[i] = -1;
        if (g)
            g[i] = 0.f;
    }
}

}  // namespace

cudaError_t launch_topk(const TopkCall &c, cudaStream_t stream)
{
    LossWorkspace ws = loss_workspace_layout(c.workspace, c.T);
    LossArgs la{};
    la.mask = c.mask;
    la.row_of_token = c.row_of_token;
    la.w = c.w;
    la.T = c.T;
    la.num_rows = c.num_rows;
    la.vocab = c.vocab;
    la.mode = TURNOPD_FULL_VOCAB;
    la.token_loss = c.token_loss;
    la.status = c.status;
    cudaError_t e = launch_compaction(la, ws.rows, ws.blk_count, ws.nvalid, stream);
    if (e != cudaSuccess)
        return e;
    const int sms = device_sm_count();
    if ((c.topk_ids || c.topk_grad) && (c.flags & TURNOPD_ZERO_MASKED_GRAD)) {
        const int grid = (int)std::min<int64_t>((c.T * c.K + 255) / 256, (int64_t)sms * 8);
        k_topk_zero_masked<<<std::max(grid, 1), 256, 0, stream>>>(c.mask, c.T, c.K, c.topk_ids, c.topk_grad);
    }
    if (c.grad && (c.flags & TURNOPD_ZERO_MASKED_GRAD))
        launch_zero_masked_grad(c.mask, c.row_of_token, c.T, c.num_rows, c.ld, c.vocab, c.grad, c.grad_dtype,
                                stream);
    TopkArgs a{c.zs, c.zt, c.ld, c.vocab, c.K, ws.rows, ws.nvalid, c.topk_ids, c.topk_grad, c.grad,
               c.grad_dtype, c.token_loss, ws.row_wl, c.status};
    static int per_sm[64][2] = {};
    int dev = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess)
        return e;
    const int ti = c.in_dtype == TURNOPD_BF16 ? 0 : 1;
    auto kern = c.in_dtype == TURNOPD_BF16 ? k_topk_rows<true> : k_topk_rows<false>;
    if (dev >= 64 || per_sm[dev][ti] == 0) {
        if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kTkSmem)) !=
            cudaSuccess)
            return e;
        int nb = 0;
        if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, kern, kTkThreads, kTkSmem)) != cudaSuccess)
            return e;
        if (nb < 1)
            return cudaErrorInvalidConfiguration;
        if (dev < 64)
            per_sm[dev][ti] = nb;
        else
            per_sm[0][ti] = nb;
    }
    const int grid = sms * per_sm[dev < 64 ? dev : 0][ti];
    kern<<<grid, kTkThreads, kTkSmem, stream>>>(a);
    e = cudaGetLastError();
    if (e != cudaSuccess)
        return e;
    launch_loss_sum(ws.row_wl, ws.nvalid, c.loss, c.status, stream);
    return cudaGetLastError();
}

}  // namespace turnopd
