// Teacher top-K reverse KL: the paper's practical loss (loss_mode
// topk_reverse_kl, support size K_top = distill_topk; Algorithm 1, "top-K
// reverse-KL token losses").  For a supervised row, S = the K vocabulary ids
// of largest teacher logit (the lower id first among equal logits); both
// distributions are renormalised over S:
//   l   = sum_{v in S} ps_v (log ps_v - log pt_v)
//   g_v = w ps_v (log ps_v - log pt_v - l)  on S, 0 elsewhere (= w dl/dz_s).
//
// Persistent CTAs, each with two rows in flight: streaming warps run pass A
// of a row while two selector warps run the later phases of the previous row
// (double-buffered buckets, named barriers).  Selection with 64-bit keys
// (order-preserving logit bits << 32 | ~id, so larger key = larger logit,
// then lower id):
//   pass A   one read of the teacher row, warp-uniform: for every group of 16
//            consecutive ids the largest logit is recorded in shared memory as
//            a 16-bit ordered bucket (the top 16 bits of the order-preserving
//            bits), and every thread keeps the largest logit it saw;
//   bound    tau = the K-th largest of the 8 (or ceil(K/warps)) largest lane
//            maxima of every streaming warp: K-th largest of distinct elements
//            of the row, so a lower bound of the row's K-th largest logit;
//   collect  only the groups whose bucket reaches tau's are read again (a few
//            dozen per row), and their elements >= tau go to a shared-memory
//            candidate buffer; a buffer overflow (rows of many equal logits)
//            raises tau to the K-th largest buffered key and collects again
//            (bounded rounds);
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

#ifndef TURNOPD_TOPK_STREAM_WARPS
#define TURNOPD_TOPK_STREAM_WARPS 8
#endif
#ifndef TURNOPD_TOPK_MINB
#define TURNOPD_TOPK_MINB 3
#endif
constexpr int kTkStreamWarps = TURNOPD_TOPK_STREAM_WARPS;  // pass A, row after row
constexpr int kTkSelThreads = 64;                           // two selector warps
constexpr int kTkStreamThreads = kTkStreamWarps * 32;
constexpr int kTkThreads = kTkStreamThreads + kTkSelThreads;
constexpr int kTkMinBlocks = TURNOPD_TOPK_MINB;  // CTAs (rows in flight) per SM
// named barriers: buffer b full (1 + b), buffer b free (3 + b), selectors only (5),
// streaming warps only (6)
constexpr int kBarFull = 1, kBarFree = 3, kBarSel = 5, kBarStream = 6;
constexpr int kTkGroupCap = 1024;  // candidate groups listed per row by the streaming warps
constexpr int kTkCap = 1024;      // candidate buffer (keys and student logits)
// candidate groups whose loads a thread issues together (bf16 / fp32)
template <bool BF16>
__host__ __device__ constexpr int tk_hits() { return BF16 ? 2 : 1; }
constexpr int kTkRounds = 16;     // bound on overflow rounds
constexpr int kTkGroup = 16;      // ids per recorded bucket

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

// Ordered value of an element (16 significant bits for bf16, 32 for fp32).
template <bool BF16>
__device__ __forceinline__ uint32_t elem_ord(const void *row, int64_t e)
{
    return BF16 ? ord16(static_cast<const uint16_t *>(row)[e]) : ord32(static_cast<const uint32_t *>(row)[e]);
}

// 16-bit bucket of an ordered value: monotone in the value.
template <bool BF16>
__device__ __forceinline__ uint32_t bucket(uint32_t ord)
{
    return BF16 ? ord : ord >> 16;
}

// Largest ordered value of the elements e0 .. e0+15 of a row, clipped to V
// (element by element: the partial last group and misaligned rows).
template <bool BF16>
__device__ __forceinline__ uint32_t group_max_ord_scalar(const void *row, int64_t V, int64_t g)
{
    const int64_t e0 = g * kTkGroup;
    uint32_t m = 0;
    for (int64_t e = e0; e < e0 + kTkGroup && e < V; ++e)
        m = max(m, elem_ord<BF16>(row, e));
    return m;
}

// Ordered values of the 16 elements held in the 16-byte vectors v[0 .. VPG).
template <bool BF16>
__device__ __forceinline__ void unpack_ords(const uint4 *v, uint32_t (&o)[kTkGroup])
{
    if (BF16) {
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const uint32_t w4[4] = {v[q].x, v[q].y, v[q].z, v[q].w};
#pragma unroll
            for (int e = 0; e < 8; ++e)
                o[q * 8 + e] = ord16(e & 1 ? w4[e >> 1] >> 16 : w4[e >> 1]);
        }
    } else {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            o[q * 4 + 0] = ord32(v[q].x);
            o[q * 4 + 1] = ord32(v[q].y);
            o[q * 4 + 2] = ord32(v[q].z);
            o[q * 4 + 3] = ord32(v[q].w);
        }
    }
}

__device__ __forceinline__ void named_sync(int id, int n)
{
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}
__device__ __forceinline__ void named_arrive(int id, int n)
{
    asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(n) : "memory");
}

// Radix select over the selector warps: the K-th largest of the nonzero keys
// in keys[0, n) (keys are unique; 0 marks an empty slot), deciding bytes
// hi_byte..lo_byte.  Returns t such that {keys >= t} holds the K largest keys
// when lo_byte = 0 (exactly K), or, when lo_byte > 0, the K-th largest key
// with its lower bytes cleared (every key of equal upper bytes is >= t).
// Returns 0 when fewer than K keys are present.  Stops early once the chosen
// bin holds exactly the remaining count.  Every selector thread (stid =
// 0 .. kTkSelThreads-1) calls it; it synchronises them on kBarSel.
struct SelScratch {
    uint32_t hist[256];
    int bin, need;
};

__device__ uint64_t sel_kth_largest(const uint64_t *keys, int n, int K, int hi_byte, int lo_byte,
                                    SelScratch &sc, int stid)
{
    const int lane = stid & 31;
    uint64_t prefix = 0, mask = 0;
    int need = K;
    for (int byte = hi_byte; byte >= lo_byte; --byte) {
        for (int i = stid; i < 256; i += kTkSelThreads)
            sc.hist[i] = 0;
        named_sync(kBarSel, kTkSelThreads);
        const int sh = 8 * byte;
        for (int i = stid; i < n; i += kTkSelThreads) {
            const uint64_t k = keys[i];
            if (k != 0 && (k & mask) == prefix)
                atomicAdd(&sc.hist[(k >> sh) & 255u], 1u);
        }
        named_sync(kBarSel, kTkSelThreads);
        if (stid < 32) {
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
        named_sync(kBarSel, kTkSelThreads);
        const int bin = sc.bin, nd = sc.need;
        named_sync(kBarSel, kTkSelThreads);
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

// Dynamic shared memory: candidate keys, the K selected keys, candidate student
// logits, the K selected student logits / gradients, then two buffers of one
// 16-bit bucket per group of 16 ids.
__host__ __device__ __forceinline__ size_t topk_fixed_bytes(int K)
{
    return align256(sizeof(uint64_t) * (kTkCap + (size_t)K) + sizeof(float) * (kTkCap + (size_t)K));
}

__host__ __device__ __forceinline__ int64_t topk_groups(int64_t V) { return (V + kTkGroup - 1) / kTkGroup; }

__host__ __device__ __forceinline__ size_t topk_bucket_bytes(int64_t V)
{
    return align256(sizeof(uint16_t) * (size_t)topk_groups(V));
}

size_t topk_smem_bytes(int64_t V, int K) { return topk_fixed_bytes(K) + 2 * topk_bucket_bytes(V); }

// One CTA holds two rows at a time: its streaming warps run pass A of row
// i + 1 (into bucket buffer (i + 1) % 2) while its two selector warps run
// bound, collect, select and the KL of row i from buffer i % 2, so the SM's
// teacher stream does not pause for the latency-bound phases.
template <bool BF16>
__global__ void __launch_bounds__(kTkThreads, kTkMinBlocks) k_topk_rows(TopkArgs a)
{
    extern __shared__ __align__(128) uint64_t tk_smem[];
    const int K = a.K;
    uint64_t *s_cand = tk_smem;
    uint64_t *s_top = s_cand + kTkCap;
    float *s_cz = reinterpret_cast<float *>(s_top + K);   // student logit of each candidate
    float *s_g = s_cz + kTkCap;                            // selected: student logit, then g
    uint16_t *s_bucket0 = reinterpret_cast<uint16_t *>(reinterpret_cast<unsigned char *>(tk_smem) +
                                                       topk_fixed_bytes(K));
    __shared__ SelScratch s_sel;
    __shared__ int4 s_meta[2];      // per buffer: the row (token, row, -, weight bits)

    __shared__ int s_n, s_over;
    __shared__ uint32_t s_wtop[2][kTkStreamThreads];  // per buffer: the c largest lane maxima of each warp
    __shared__ uint32_t s_tau[2];                     // per buffer: the bound (ordered logit)
    __shared__ int s_ng[2];                           // per buffer: candidate groups found
    __shared__ uint16_t s_glist[2][kTkGroupCap];      // per buffer: their indices

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int n_rows = *a.nvalid;
    const int n_it = n_rows > (int)blockIdx.x ? (n_rows - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x : 0;
    const size_t esz = BF16 ? 2 : 4;
    const bool vec_ok =
        ((reinterpret_cast<uintptr_t>(a.zt) | reinterpret_cast<uintptr_t>(a.zs) | (uintptr_t)(a.ld * esz)) & 15u) == 0;
    const int64_t ng = topk_groups(a.vocab);
    const int ngv = vec_ok ? (int)(a.vocab / kTkGroup) : 0;  // whole groups read as vectors
    const size_t bucket_elems = topk_bucket_bytes(a.vocab) / sizeof(uint16_t);
    constexpr int VPG = BF16 ? 2 : 4;  // 16-byte vectors per group
    // lower bound of the K-th largest logit: every streaming warp contributes the cw largest
    // of its lanes' maxima (cw = max(ceil(K / warps), 8) <= 32); the K-th largest of these
    // distinct elements cannot exceed the row's K-th largest.  No bound (admit everything)
    // when cw would exceed 32.
    const int cw = max((K + kTkStreamWarps - 1) / kTkStreamWarps, 8);

    if (warp < kTkStreamWarps) {
        // ---- streaming warps: pass A, one row after another
        constexpr int U = 8 / VPG;  // groups per batch
        // one batch of whole groups: 8 loads (128 B) in flight per thread
        uint4 v[U * VPG];
        auto load_batch = [&](const uint4 *rv, int g0) {
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int g = g0 + u * kTkStreamThreads;
#pragma unroll
                for (int q = 0; q < VPG; ++q)
                    if (g < ngv)
                        v[u * VPG + q] = __ldg(rv + (size_t)g * VPG + q);
            }
        };
        auto row_vectors = [&](const int4 &mr) {
            return reinterpret_cast<const uint4 *>(static_cast<const char *>(a.zt) + (size_t)mr.y * (size_t)a.ld * esz);
        };
        int4 m_next = n_it > 0 ? a.rows[blockIdx.x] : make_int4(0, 0, -1, 0);
        if (n_it > 0)
            load_batch(row_vectors(m_next), tid);  // the first batch of each row is loaded a row ahead
        for (int it = 0; it < n_it; ++it) {
            const int b = it & 1;
            const int4 m = m_next;  // loaded one row ahead
            if (it + 1 < n_it)
                m_next = a.rows[blockIdx.x + (it + 1) * gridDim.x];
            if (it >= 2)
                named_sync(kBarFree + b, kTkThreads);  // the selectors are done with row it - 2
            if (tid == 0) {
                s_meta[b] = m;
                s_tau[b] = 0;
            }
            const char *zt_row = static_cast<const char *>(a.zt) + (size_t)m.y * (size_t)a.ld * esz;
            uint16_t *s_bucket = s_bucket0 + b * bucket_elems;
            // group buckets and the thread's largest logit; whole groups of a 16-byte
            // aligned row are read as vectors, a batch at a time
            uint32_t tmax = 0;
            const uint4 *rv = reinterpret_cast<const uint4 *>(zt_row);
            for (int g0 = tid; g0 < ngv; g0 += U * kTkStreamThreads) {
                if (g0 != tid)
                    load_batch(rv, g0);
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int g = g0 + u * kTkStreamThreads;
                    if (g >= ngv)
                        break;
                    uint32_t o;
                    if (BF16) {
                        const uint32_t o0 = bf16_max8_ord(v[u * 2]), o1 = bf16_max8_ord(v[u * 2 + 1]);
                        o = max(o0, o1);
                    } else {
                        float mx = -INFINITY;
#pragma unroll
                        for (int q = 0; q < 4; ++q)
                            mx = fmaxf(mx, fmaxf(fmaxf(__uint_as_float(v[u * 4 + q].x), __uint_as_float(v[u * 4 + q].y)),
                                                 fmaxf(__uint_as_float(v[u * 4 + q].z), __uint_as_float(v[u * 4 + q].w))));
                        o = ord32(__float_as_uint(mx));
                    }
                    s_bucket[g] = (uint16_t)bucket<BF16>(o);
                    tmax = max(tmax, o);
                }
            }
            // groups left: the partial last group, or every group of a misaligned row
            for (int g = ngv + tid; g < (int)ng; g += kTkStreamThreads) {
                const uint32_t o = group_max_ord_scalar<BF16>(zt_row, a.vocab, g);
                s_bucket[g] = (uint16_t)bucket<BF16>(o);
                tmax = max(tmax, o);
            }
            if (it + 1 < n_it)
                load_batch(row_vectors(m_next), tid);  // in flight while the row is settled below
            if (cw <= 32) {
                bool taken = false;
                for (int i = 0; i < cw; ++i) {
                    const uint32_t mx = __reduce_max_sync(0xffffffffu, taken ? 0u : tmax);
                    const unsigned who = __ballot_sync(0xffffffffu, !taken && tmax == mx);
                    if (who != 0u && lane == __ffs(who) - 1)
                        taken = true;
                    if (lane == 0)
                        s_wtop[b][warp * cw + i] = mx;
                }
            }
            if (tid == 0)
                s_ng[b] = 0;
            named_sync(kBarStream, kTkStreamThreads);
            if (cw <= 32) {
                const int nw = kTkStreamWarps * cw;
                for (int u0 = tid; u0 < nw; u0 += kTkStreamThreads) {
                    const uint32_t v = s_wtop[b][u0];
                    int gt = 0, ge = 0;
                    for (int u = 0; u < nw; ++u) {
                        const uint32_t x = s_wtop[b][u];
                        gt += x > v;
                        ge += x >= v;
                    }
                    if (v != 0 && gt < K && ge >= K)
                        s_tau[b] = v;  // every such thread writes the same value
                }
            }
            named_sync(kBarStream, kTkStreamThreads);
            // the whole groups that can hold an element >= tau: their bucket reaches tau's
            const uint32_t tb = bucket<BF16>(s_tau[b]);
            for (int g = tid; g < ngv; g += kTkStreamThreads)
                if (s_bucket[g] >= tb) {
                    const int p = atomicAdd(&s_ng[b], 1);
                    if (p < kTkGroupCap)
                        s_glist[b][p] = (uint16_t)g;
                }
            named_arrive(kBarFull + b, kTkThreads);  // row it is in buffer b
        }
        return;
    }

    // ---- selector warps: the phases after pass A, one row behind the stream
    const int stid = tid - kTkStreamThreads, swarp = stid >> 5;
    const int hi_val = BF16 ? 5 : 7;  // top byte of the ordered logit inside a key
    for (int it = 0; it < n_it; ++it) {
        const int b = it & 1;
        const int j = blockIdx.x + it * gridDim.x;
        named_sync(kBarFull + b, kTkThreads);
        const int4 m = s_meta[b];
        const int tok = m.x;
        const float w = __int_as_float(m.w);
        const char *zt_row = static_cast<const char *>(a.zt) + (size_t)m.y * (size_t)a.ld * esz;
        const char *zs_row = static_cast<const char *>(a.zs) + (size_t)m.y * (size_t)a.ld * esz;
        const uint16_t *s_bucket = s_bucket0 + b * bucket_elems;
        if (stid == 0) {
            s_n = 0;
            s_over = 0;
        }
        named_sync(kBarSel, kTkSelThreads);
        uint64_t tau = (uint64_t)s_tau[b] << 32;  // admits every id of logit >= tau's
        const int n_listed = s_ng[b];

        auto append = [&](uint64_t k, float zsv) {
            const int p = atomicAdd(&s_n, 1);
            if (p < kTkCap) {
                s_cand[p] = k;
                s_cz[p] = zsv;
            } else {
                s_over = 1;
            }
        };
        const uint4 *rv = reinterpret_cast<const uint4 *>(zt_row);
        const uint4 *sv = reinterpret_cast<const uint4 *>(zs_row);
        // the candidate elements of up to kTkHits whole groups, teacher and student
        // vectors of all of them loaded before any is used
        constexpr int kTkHits = tk_hits<BF16>();
        // the candidate elements of one whole group: teacher vectors vt, student vectors vs
        auto scan_group = [&](const uint4 *vt, const uint4 *vs, int g) {
            uint32_t o[kTkGroup];
            unpack_ords<BF16>(vt, o);
            const uint32_t e0 = (uint32_t)g * kTkGroup;
#pragma unroll
            for (int e = 0; e < kTkGroup; ++e) {
                const uint64_t k = mkkey(o[e], e0 + e);
                if (k >= tau) {
                    const uint4 &x = vs[e / (16 / (int)esz)];
                    const int wi = (e % (16 / (int)esz)) * (int)esz / 4;
                    const uint32_t word = wi == 0 ? x.x : wi == 1 ? x.y : wi == 2 ? x.z : x.w;
                    const float zsv = BF16 ? __uint_as_float(((e & 1) ? word >> 16 : word & 0xFFFFu) << 16)
                                           : __uint_as_float(word);
                    append(k, zsv);
                }
            }
        };
        // groups read from global memory, kTkHits at a time, all loads before any use
        auto take_groups = [&](const int (&hg)[kTkHits], int nh) {
            uint4 vt[kTkHits * VPG], vs[kTkHits * VPG];
#pragma unroll
            for (int h = 0; h < kTkHits; ++h)
#pragma unroll
                for (int q = 0; q < VPG; ++q)
                    if (h < nh) {
                        vt[h * VPG + q] = __ldg(rv + (size_t)hg[h] * VPG + q);
                        vs[h * VPG + q] = __ldg(sv + (size_t)hg[h] * VPG + q);
                    }
#pragma unroll
            for (int h = 0; h < kTkHits; ++h) {
                if (h >= nh)
                    break;
                scan_group(&vt[h * VPG], &vs[h * VPG], hg[h]);
            }
        };
        // elements >= tau live in groups whose bucket reaches tau's: the groups the
        // streaming warps listed, or (list overflow, raised tau) a scan of the buckets
        auto collect = [&](bool listed) {
            const uint32_t tb = bucket<BF16>((uint32_t)(tau >> 32));
            int hg[kTkHits];
            int nh = 0;
            const int n_scan = listed ? n_listed : ngv;
            for (int i = stid; i < n_scan; i += kTkSelThreads) {
                const int g = listed ? (int)s_glist[b][i] : i;
                if (!listed && s_bucket[g] < tb)
                    continue;

                hg[nh++] = g;
                if (nh == kTkHits) {
                    take_groups(hg, nh);
                    nh = 0;
                }
            }
            if (nh > 0)
                take_groups(hg, nh);
            // the partial last group and misaligned rows, element by element
            for (int g = ngv + stid; g < (int)ng; g += kTkSelThreads) {
                if (s_bucket[g] < tb)
                    continue;
                const int64_t e0 = (int64_t)g * kTkGroup;
                for (int64_t e = e0; e < e0 + kTkGroup && e < a.vocab; ++e) {
                    const uint64_t k = mkkey(elem_ord<BF16>(zt_row, e), (uint32_t)e);
                    if (k >= tau)
                        append(k, BF16 ? __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(zs_row)[e])
                                       : reinterpret_cast<const float *>(zs_row)[e]);
                }
            }
        };
        collect(n_listed <= kTkGroupCap);
        named_sync(kBarSel, kTkSelThreads);
        // ---- overflow: raise tau to the K-th largest buffered key and collect again
        for (int round = 0; s_over && round < kTkRounds; ++round) {
            tau = sel_kth_largest(s_cand, kTkCap, K, 7, 0, s_sel, stid);
            if (stid == 0) {
                s_n = 0;
                s_over = 0;
            }
            named_sync(kBarSel, kTkSelThreads);
            collect(false);
            named_sync(kBarSel, kTkSelThreads);
        }
        const bool failed = s_over != 0;
        const int nc = min(s_n, kTkCap);
        named_sync(kBarSel, kTkSelThreads);
        if (failed) {
            if (stid == 0) {
                set_status(a.status, TURNOPD_ERR_UNSUPPORTED);
                a.token_loss[tok] = 0.f;
                a.row_wl[j] = 0.0;
            }
        } else {
            // ---- the K largest: each candidate's rank among the candidates is its position
            // (keys are unique); a large buffer is first cut to the K largest by radix select
            const uint64_t kth = nc <= kTkSelThreads ? 0 : sel_kth_largest(s_cand, nc, K, hi_val, 0, s_sel, stid);
            for (int i = stid; i < nc; i += kTkSelThreads) {
                const uint64_t k = s_cand[i];
                if (k < kth)
                    continue;
                int rank = 0;
                int i2 = 0;
                for (; i2 + 4 <= nc; i2 += 4)
                    rank += (s_cand[i2] > k) + (s_cand[i2 + 1] > k) + (s_cand[i2 + 2] > k) + (s_cand[i2 + 3] > k);
                for (; i2 < nc; ++i2)
                    rank += s_cand[i2] > k;
                if (rank < K) {
                    s_top[rank] = k;
                    s_g[rank] = s_cz[i];
                }
            }
            named_sync(kBarSel, kTkSelThreads);

            // ---- KL over S (one warp, fp32)
            if (swarp == 0) {
                float m_s = -INFINITY, m_t = -INFINITY;
                for (int r = lane; r < K; r += 32) {
                    const float zt_v = key_value<BF16>(s_top[r]);
                    const float zs_v = s_g[r];  // student logit, carried with the candidate
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
                for (int64_t q = stid; q < nv16; q += kTkSelThreads)
                    reinterpret_cast<uint4 *>(grow)[q] = make_uint4(0, 0, 0, 0);
                for (int64_t q = nv16 * 16 + stid; q < bytes; q += kTkSelThreads)
                    grow[q] = 0;
                named_sync(kBarSel, kTkSelThreads);
                for (int r = stid; r < K; r += kTkSelThreads) {
                    const uint32_t id = key_id(s_top[r]);
                    if (a.grad_dtype == TURNOPD_BF16)
                        reinterpret_cast<__nv_bfloat16 *>(grow)[id] = __float2bfloat16_rn(s_g[r]);
                    else
                        reinterpret_cast<float *>(grow)[id] = s_g[r];
                }
            }
        }
        named_sync(kBarSel, kTkSelThreads);  // buffer b and the candidate arrays are free
        if (it + 2 < n_it)
            named_arrive(kBarFree + b, kTkThreads);
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
    int dev = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess)
        return e;
    const int ti = c.in_dtype == TURNOPD_BF16 ? 0 : 1;
    auto kern = c.in_dtype == TURNOPD_BF16 ? k_topk_rows<true> : k_topk_rows<false>;
    const size_t smem = topk_smem_bytes(c.vocab, c.K);
    static size_t attr_smem[64][2] = {};
    const int di = dev < 64 ? dev : 0;
    if (attr_smem[di][ti] < smem) {
        if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
            cudaSuccess)
            return e;
        attr_smem[di][ti] = smem;
    }
    int nb = 0;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, kern, kTkThreads, smem)) != cudaSuccess)
        return e;
    if (nb < 1)
        return cudaErrorInvalidConfiguration;
    kern<<<sms * nb, kTkThreads, smem, stream>>>(a);
    e = cudaGetLastError();
    if (e != cudaSuccess)
        return e;
    launch_loss_sum(ws.row_wl, ws.nvalid, c.loss, c.status, stream);
    return cudaGetLastError();
}

}  // namespace turnopd
