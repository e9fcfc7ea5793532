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
//   bound    (streaming warps) for K <= 64, tau = the K-th largest of the 8
//            largest lane maxima of every streaming warp: K-th largest of
//            distinct elements of the row, so a lower bound of the row's K-th
//            largest logit; above, the K-th largest group bucket (K groups each
//            hold an element that large), by binary search on its value; then
//            the groups whose bucket reaches tau's are listed;
//   collect  (selector warps) only the listed groups are read again, in step
//            across the lanes (a few dozen per row at K = 50), and their
//            elements >= tau go to a shared-memory candidate buffer (1,024
//            entries, 2,048 above K = 512); when it overflows (rows of many
//            equal logits, sorted rows) a radix select over the row's keys >=
//            tau, one key byte per pass, raises tau until the keys above it fit
//            the buffer, then collects again (at most 6 passes for bf16 keys,
//            8 for fp32);
//   select   up to 256 candidates: the exact K-th largest by radix select, then
//            each selected key's rank among the candidates is its position;
//            more: a bitonic sort of the buffer.
// The KL over S is evaluated by one warp in fp32 with
// l = E_p[z_s - z_t] - (LSE_s - LSE_t) and g_v = w p_v ((z_s - z_t)_v - E_p[.]).

#include <cuda_bf16.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace turnopd {
namespace {

// streaming warps per CTA and CTAs per SM (measured, K = 50, full-size batches, fraction
// of the copy bandwidth packed / household / multihop: 8 x 3: 0.923 / 0.889 / 0.865;
// 12 x 2: 0.942 / 0.910 / 0.874; 10 x 2: 0.926 / 0.895 / 0.864; 14 x 2: 0.921 / 0.884 /
// 0.855; 8 x 2: 0.881 / 0.851 / 0.821; 24 x 1: 0.771 / 0.740 / 0.713)
#ifndef TURNOPD_TOPK_STREAM_WARPS
#define TURNOPD_TOPK_STREAM_WARPS 12
#endif
#ifndef TURNOPD_TOPK_MINB
#define TURNOPD_TOPK_MINB 2
#endif
constexpr int kTkStreamWarps = TURNOPD_TOPK_STREAM_WARPS;  // pass A, row after row
#ifndef TURNOPD_TOPK_SEL_WARPS
#define TURNOPD_TOPK_SEL_WARPS 2
#endif
constexpr int kTkSelWarps = TURNOPD_TOPK_SEL_WARPS;         // the later phases, a row behind
constexpr int kTkSelThreads = kTkSelWarps * 32;
static_assert(kTkSelWarps >= 1 && kTkSelWarps <= 4, "sort_desc needs n >= 2 kTkSelThreads, n >= 256");
constexpr int kTkStreamThreads = kTkStreamWarps * 32;
constexpr int kTkThreads = kTkStreamThreads + kTkSelThreads;
constexpr int kTkMinBlocks = TURNOPD_TOPK_MINB;  // CTAs (rows in flight) per SM
// named barriers: buffer b full (1 + b), buffer b free (3 + b), selectors only (5),
// streaming warps only (6)
constexpr int kBarFull = 1, kBarFree = 3, kBarSel = 5, kBarStream = 6;
constexpr int kTkGroupCap = 2048;  // candidate groups listed per row by the streaming warps
// candidate buffer (keys and student logits): 1,024 entries, 2,048 above K = 512
// (a power of two: the bitonic sort of a large buffer runs in place)
__host__ __device__ constexpr int topk_cap(int K) { return K <= 512 ? 1024 : 2048; }
// K up to which the streaming warps' lane maxima give the bound (the 8 largest
// of each warp's 32); the group buckets give it above
constexpr int kTkLaneTop = 8;
constexpr int kTkLaneBoundMaxK = kTkStreamWarps * kTkLaneTop;
// candidates above which the selection sorts the buffer instead of ranking
constexpr int kTkRankMax = 256;
constexpr uint32_t kTkQueue = 64;  // ring of group indices per selector warp (at most 63 held)
constexpr int kTkGroup = 16;      // ids per recorded bucket
static_assert(kTkQueue >= 64 && (kTkQueue & (kTkQueue - 1)) == 0, "group ring");
static_assert(TURNOPD_TOPK_MAX_VOCAB / kTkGroup <= 65536, "group indices are 16-bit");
static_assert(TURNOPD_TOPK_MAX_VOCAB <= (1 << 20) && topk_cap(TURNOPD_TOPK_MAX) <= 2048,
              "a sorted key holds a 20-bit id and an 11-bit buffer position");

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

// Radix-select scratch of the selector warps: a 256-bin histogram of one key
// byte and the bin chosen from it.
struct SelScratch {
    uint32_t hist[256];
    int bin, need;
};

// The bin of the need-th largest key of a 256-bin histogram sc.hist (bin 255
// holds the largest keys): sc.bin = that bin, or -1 when the histogram holds
// fewer than need keys; sc.need = the count still needed inside the bin,
// negated when the bin holds exactly that many.  Run by one warp (lane 0..31).
__device__ __forceinline__ void pick_bin(SelScratch &sc, int need, int lane)
{
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
                sc.need = (cum + c[e] == need) ? -(need - cum) : need - cum;
                break;
            }
            cum += c[e];
        }
    }
}

// Radix select over the selector warps: the K-th largest of the nonzero keys
// in keys[0, n) (keys are unique; 0 marks an empty slot), deciding bytes
// hi_byte..lo_byte.  Returns t such that {keys >= t} holds the K largest keys
// when lo_byte = 0 (exactly K), or, when lo_byte > 0, the K-th largest key
// with its lower bytes cleared (every key of equal upper bytes is >= t).
// Returns 0 when fewer than K keys are present.  Stops early once the chosen
// bin holds exactly the remaining count.  Every selector thread (stid =
// 0 .. kTkSelThreads-1) calls it; it synchronises them on kBarSel.
__device__ uint64_t sel_kth_largest(const uint64_t *keys, int n, int K, int hi_byte, int lo_byte,
                                    SelScratch &sc, int stid)
{
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
        if (stid < 32)
            pick_bin(sc, need, stid);
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

// Buckets of the 16-bit pair x at or above m.
__device__ __forceinline__ int count_ge2(uint32_t x, uint32_t m)
{
    return (int)((x & 0xFFFFu) >= m) + (int)((x >> 16) >= m);
}

// Sorts keys[0, n) (n a power of two >= 2 kTkSelThreads, distinct keys but for 0
// padding) in descending order: bitonic network over the selector threads, each
// thread loading U pairs before it compares and stores any, synchronised on
// kBarSel after every step.
template <int U>
__device__ void sort_desc(uint64_t *keys, int n, int stid)
{
    const int np = n / 2;  // pairs per step
    for (int k = 2; k <= n; k <<= 1)
        for (int j = k >> 1; j > 0; j >>= 1) {
            for (int i0 = stid; i0 < np; i0 += U * kTkSelThreads) {
                uint64_t x[U], y[U];
                int l[U];
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int i = i0 + u * kTkSelThreads;
                    l[u] = 2 * i - (i & (j - 1));
                    if (i < np) {
                        x[u] = keys[l[u]];
                        y[u] = keys[l[u] + j];
                    }
                }
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    // blocks with (l & k) == 0 descending, the others ascending; the last merge
                    // (k = n) is descending throughout
                    if (i0 + u * kTkSelThreads < np && (x[u] < y[u]) == ((l[u] & k) == 0)) {
                        keys[l[u]] = y[u];
                        keys[l[u] + j] = x[u];
                    }
                }
            }
            named_sync(kBarSel, kTkSelThreads);
        }
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
    return align256((sizeof(uint64_t) + sizeof(float)) * ((size_t)topk_cap(K) + (size_t)K));
}

__host__ __device__ __forceinline__ int64_t topk_groups(int64_t V) { return (V + kTkGroup - 1) / kTkGroup; }

__host__ __device__ __forceinline__ size_t topk_bucket_bytes(int64_t V)
{
    return align256(sizeof(uint16_t) * (size_t)topk_groups(V));
}

size_t topk_smem_bytes(int64_t V, int K) { return topk_fixed_bytes(K) + 2 * topk_bucket_bytes(V); }

// One CTA holds two rows at a time: its streaming warps run pass A and the
// bound of row i + 1 (into bucket buffer (i + 1) % 2) while its two selector
// warps run collect, select and the KL of row i from buffer i % 2, so the SM's
// teacher stream does not pause for the latency-bound phases.
template <bool BF16>
__global__ void __launch_bounds__(kTkThreads, kTkMinBlocks) k_topk_rows(TopkArgs a)
{
    // the loss sum after this grid may take the first SM it frees (it waits for the grid)
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    extern __shared__ __align__(128) uint64_t tk_smem[];
    const int K = a.K;
    uint64_t *s_cand = tk_smem;
    const int cap = topk_cap(K);
    uint64_t *s_top = s_cand + cap;
    float *s_cz = reinterpret_cast<float *>(s_top + K);   // student logit of each candidate
    float *s_g = s_cz + cap;                               // selected: student logit, then g
    uint16_t *s_bucket0 = reinterpret_cast<uint16_t *>(reinterpret_cast<unsigned char *>(tk_smem) +
                                                       topk_fixed_bytes(K));
    __shared__ SelScratch s_sel;
    __shared__ int4 s_meta[2];      // per buffer: the row (token, row, -, weight bits)

    __shared__ int s_n, s_over;
    __shared__ __align__(16) uint32_t s_wtop[2][kTkLaneBoundMaxK];  // per buffer: each warp's 8 largest lane maxima
    __shared__ uint32_t s_tau[2];                     // per buffer: the bound (ordered logit)
    __shared__ int s_ng[2];                           // per buffer: candidate groups found
    __shared__ uint16_t s_glist[2][kTkGroupCap];      // per buffer: their indices
    __shared__ uint16_t s_wq[kTkSelWarps][kTkQueue];  // per selector warp: groups found, not yet read
    __shared__ int s_scnt[2][kTkStreamWarps];         // per streaming warp: a count of buckets
    __shared__ uint32_t s_smax[kTkStreamWarps];       // per streaming warp: its largest bucket

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
    // lower bound of the K-th largest logit: for K <= 64 every streaming warp contributes
    // the 8 largest of its lanes' maxima, and the K-th largest of these distinct elements
    // cannot exceed the row's K-th largest; above, the streaming warps take the K-th
    // largest group bucket.
    const bool lane_bound = K <= kTkLaneBoundMaxK;

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
            if (lane_bound) {
                // the warp's 8 largest lane maxima: a bitonic sort of the 32 in registers,
                // descending, leaves them in lanes 0..7
                uint32_t x = tmax;
#pragma unroll
                for (int k = 2; k <= 32; k <<= 1)
#pragma unroll
                    for (int j = k >> 1; j > 0; j >>= 1) {
                        const uint32_t y = __shfl_xor_sync(0xffffffffu, x, j);
                        x = (((lane & j) == 0) == ((lane & k) == 0)) ? max(x, y) : min(x, y);
                    }
                if (lane < kTkLaneTop)
                    s_wtop[b][warp * kTkLaneTop + lane] = x;
            }
            if (tid == 0)
                s_ng[b] = 0;
            named_sync(kBarStream, kTkStreamThreads);
            if (lane_bound) {
                constexpr int nw = kTkStreamWarps * kTkLaneTop;
                const uint4 *w4 = reinterpret_cast<const uint4 *>(s_wtop[b]);
                for (int u0 = tid; u0 < nw; u0 += kTkStreamThreads) {
                    const uint32_t v = s_wtop[b][u0];
                    int gt = 0, ge = 0;
#pragma unroll
                    for (int q = 0; q < nw / 4; ++q) {
                        const uint4 x = w4[q];
                        gt += (x.x > v) + (x.y > v) + (x.z > v) + (x.w > v);
                        ge += (x.x >= v) + (x.y >= v) + (x.z >= v) + (x.w >= v);
                    }
                    if (v != 0 && gt < K && ge >= K)
                        s_tau[b] = v;  // every such thread writes the same value
                }
            } else if (a.vocab > cap) {
                // the K-th largest group bucket, by binary search on its value with counts of
                // the buckets at or above it: K groups each hold an element that large (no
                // bound, tau = 0, when the row has fewer than K groups)
                const uint4 *b4 = reinterpret_cast<const uint4 *>(s_bucket);
                const int n4 = (int)ng / 8;
                // The answer is at most the row's largest bucket; the first pass probes 255 below
                // it (where the K-th largest bucket of a row with a few hundred large logits lies),
                // and only when fewer than K buckets reach that does the search span the rest.
                const uint32_t wmax = __reduce_max_sync(0xffffffffu, bucket<BF16>(tmax));
                if (lane == 0)
                    s_smax[warp] = wmax;
                named_sync(kBarStream, kTkStreamThreads);
                uint32_t hi = 0;
#pragma unroll
                for (int w = 0; w < kTkStreamWarps; ++w)
                    hi = max(hi, s_smax[w]);
                uint32_t lo = 0;  // count(>= lo) >= K or lo = 0; the answer is in [lo, hi]
                const uint32_t probe = hi > 255u ? hi - 255u : 0u;
                // the warps' counts alternate between two rows of s_scnt, so one barrier a pass
                // suffices: a pass's reads finish before any thread passes the next barrier
                for (int par = 0, first = 1; lo < hi; par ^= 1, first = 0) {
                    const uint32_t mid = first && probe > lo ? probe : (lo + hi + 1) >> 1;
                    int c = 0;
                    for (int i = tid; i < n4; i += kTkStreamThreads) {
                        const uint4 q = b4[i];
                        c += count_ge2(q.x, mid) + count_ge2(q.y, mid) + count_ge2(q.z, mid) + count_ge2(q.w, mid);
                    }
                    for (int g = n4 * 8 + tid; g < (int)ng; g += kTkStreamThreads)
                        c += (uint32_t)s_bucket[g] >= mid;
                    c = __reduce_add_sync(0xffffffffu, c);
                    if (lane == 0)
                        s_scnt[par][warp] = c;
                    named_sync(kBarStream, kTkStreamThreads);
                    int tot = 0;
#pragma unroll
                    for (int w = 0; w < kTkStreamWarps; ++w)
                        tot += s_scnt[par][w];
                    if (tot >= K)
                        lo = mid;
                    else
                        hi = mid - 1;
                }
                if (tid == 0)
                    s_tau[b] = BF16 ? lo : lo << 16;
            }
            named_sync(kBarStream, kTkStreamThreads);
            // the whole groups that can hold an element >= tau: their bucket reaches tau's
            // (eight buckets a load; the list's order does not matter)
            const uint32_t tb = bucket<BF16>(s_tau[b]);
            auto list = [&](int g) {
                const int p = atomicAdd(&s_ng[b], 1);
                if (p < kTkGroupCap)
                    s_glist[b][p] = (uint16_t)g;
            };
            const uint4 *b8 = reinterpret_cast<const uint4 *>(s_bucket);
            const int n8 = ngv / 8;
            for (int i = tid; i < n8; i += kTkStreamThreads) {
                const uint4 q = b8[i];
                const uint32_t w4[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
                for (int e = 0; e < 8; ++e)
                    if (((w4[e >> 1] >> (16 * (e & 1))) & 0xFFFFu) >= tb)
                        list(i * 8 + e);
            }
            for (int g = n8 * 8 + tid; g < ngv; g += kTkStreamThreads)
                if (s_bucket[g] >= tb)
                    list(g);
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
            if (p < cap) {
                s_cand[p] = k;
                s_cz[p] = zsv;
            } else {
                s_over = 1;
            }
        };
        const uint4 *rv = reinterpret_cast<const uint4 *>(zt_row);
        const uint4 *sv = reinterpret_cast<const uint4 *>(zs_row);
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
        // visit(g, ok) for the whole groups (g < ngv) whose bucket reaches tb, one per lane
        // and call, the lanes converged.  Each warp walks its share of the buckets in step,
        // queues the groups that pass (ballot) in its ring in shared memory, and visits 32 at a
        // time, so the lanes' loads are in flight together (a lane that visited its groups
        // alone would hold the warp for one memory round trip per group).
        auto walk_groups = [&](uint32_t tb, auto &&visit) {
            uint16_t *q = s_wq[swarp];
            uint32_t head = 0, tail = 0;  // warp-uniform
            for (int g0 = swarp * 32; g0 < ngv; g0 += kTkSelThreads) {
                const int g = g0 + lane;
                const bool pass = g < ngv && s_bucket[g] >= tb;
                const unsigned hit = __ballot_sync(0xffffffffu, pass);
                if (pass)
                    q[(tail + __popc(hit & ((1u << lane) - 1u))) & (kTkQueue - 1)] = (uint16_t)g;
                tail += __popc(hit);
                __syncwarp();
                if (tail - head >= 32) {
                    const int gq = q[(head + lane) & (kTkQueue - 1)];
                    __syncwarp();
                    head += 32;
                    visit(gq, true);
                }
            }
            if (head != tail) {  // fewer than 32 left
                const bool ok = lane < (int)(tail - head);
                const int gq = ok ? q[(head + lane) & (kTkQueue - 1)] : 0;
                __syncwarp();
                visit(gq, ok);
            }
        };
        // the candidate elements of group g (ok): teacher and student vectors loaded together
        auto take_one = [&](int g, bool ok) {
            if (!ok)
                return;
            uint4 vt[VPG], vs[VPG];
#pragma unroll
            for (int q = 0; q < VPG; ++q) {
                vt[q] = __ldg(rv + (size_t)g * VPG + q);
                vs[q] = __ldg(sv + (size_t)g * VPG + q);
            }
            scan_group(vt, vs, g);
        };
        // elements >= tau live in groups whose bucket reaches tau's: the groups the
        // streaming warps listed, or (list overflow, raised tau) a walk over the buckets
        auto collect = [&](bool listed) {
            const uint32_t tb = bucket<BF16>((uint32_t)(tau >> 32));
            if (listed) {
                for (int i = stid; i < n_listed; i += kTkSelThreads)
                    take_one((int)s_glist[b][i], true);
            } else {
                walk_groups(tb, take_one);
            }
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
        // f(k) for every key >= lo of the row: the whole groups whose bucket reaches
        // lo's are read again (teacher only, a group per lane in step), the partial
        // last group and misaligned rows element by element
        auto each_key = [&](uint64_t lo, auto &&f) {
            const uint32_t tb = bucket<BF16>((uint32_t)(lo >> 32));
            walk_groups(tb, [&](int g, bool ok) {
                if (!ok)
                    return;
                uint4 vt[VPG];
#pragma unroll
                for (int q = 0; q < VPG; ++q)
                    vt[q] = __ldg(rv + (size_t)g * VPG + q);
                uint32_t o[kTkGroup];
                unpack_ords<BF16>(vt, o);
                const uint32_t e0 = (uint32_t)g * kTkGroup;
#pragma unroll
                for (int e = 0; e < kTkGroup; ++e) {
                    const uint64_t k = mkkey(o[e], e0 + e);
                    if (k >= lo)
                        f(k);
                }
            });
            for (int g = ngv + stid; g < (int)ng; g += kTkSelThreads) {
                if (s_bucket[g] < tb)
                    continue;
                const int64_t e0 = (int64_t)g * kTkGroup;
                for (int64_t e = e0; e < e0 + kTkGroup && e < a.vocab; ++e) {
                    const uint64_t k = mkkey(elem_ord<BF16>(zt_row, e), (uint32_t)e);
                    if (k >= lo)
                        f(k);
                }
            }
        };
        collect(n_listed <= kTkGroupCap);
        named_sync(kBarSel, kTkSelThreads);
        if (s_over) {
            // ---- overflow: radix select over the row's keys >= tau, one key byte per
            // pass from the top, until the keys >= the chosen prefix fit the buffer.
            // Keys above the prefix number K - need; those with the prefix, cnt.
            uint64_t prefix = 0, pmask = 0;
            int need = K;
            for (int byte = hi_val; byte >= 0; --byte) {
                const int sh = 8 * byte;
                for (int i = stid; i < 256; i += kTkSelThreads)
                    s_sel.hist[i] = 0;
                named_sync(kBarSel, kTkSelThreads);
                each_key(max(tau, prefix), [&](uint64_t k) {
                    if ((k & pmask) == prefix)
                        atomicAdd(&s_sel.hist[(k >> sh) & 255u], 1u);
                });
                named_sync(kBarSel, kTkSelThreads);
                if (stid < 32)
                    pick_bin(s_sel, need, stid);
                named_sync(kBarSel, kTkSelThreads);
                const int bin = s_sel.bin, nd = s_sel.need;
                const int cnt = bin >= 0 ? (int)s_sel.hist[bin] : 0;
                named_sync(kBarSel, kTkSelThreads);
                if (bin < 0)
                    break;  // fewer than K keys >= tau: not reached, tau is a lower bound
                prefix |= (uint64_t)bin << sh;
                pmask |= (uint64_t)255u << sh;
                if (nd < 0 || K - nd + cnt <= cap)
                    break;
                need = nd;
            }
            tau = max(tau, prefix);
            if (stid == 0) {
                s_n = 0;
                s_over = 0;
            }
            named_sync(kBarSel, kTkSelThreads);
            collect(false);
            named_sync(kBarSel, kTkSelThreads);
        }
        const bool failed = s_over != 0;
        const int nc = min(s_n, cap);
        named_sync(kBarSel, kTkSelThreads);
        if (failed) {
            if (stid == 0) {
                set_status(a.status, TURNOPD_ERR_UNSUPPORTED);
                a.token_loss[tok] = 0.f;
                a.row_wl[j] = 0.0;
            }
        } else {
            if (nc > kTkRankMax) {
                // ---- the K largest of a large buffer: sort it (padded with 0 keys to a power
                // of two, at most the buffer's size) and take the first K
                // Each key carries its buffer position in its low 11 bits, below the id's 20:
                // ids are below 2^20, so ~id's upper 12 bits are ones and the order is kept.
                int n2 = kTkRankMax;
                while (n2 < nc)
                    n2 <<= 1;
                for (int i = stid; i < n2; i += kTkSelThreads) {
                    const uint64_t k = s_cand[i];
                    s_cand[i] = i < nc ? (k & 0xFFFFFFFF00000000ull) | ((k & 0xFFFFFull) << 11) | (uint64_t)i : 0ull;
                }
                named_sync(kBarSel, kTkSelThreads);
                sort_desc<BF16 ? 4 : 2>(s_cand, n2, stid);
                for (int r = stid; r < K; r += kTkSelThreads) {
                    const uint64_t p = s_cand[r];
                    s_top[r] = (p & 0xFFFFFFFF00000000ull) | 0xFFF00000ull | ((p >> 11) & 0xFFFFFull);
                    s_g[r] = s_cz[p & 0x7FFu];
                }
            } else {
                // ---- the K largest: each candidate's rank among the candidates is its position
                // (keys are unique); a buffer larger than the selector threads is first cut to the
                // K largest by radix select
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
