// Split-row kernel for fp32 logit rows (sm_103a).
//
// One fp32 logit row of V = 151,936 values is 607,744 bytes per model, so the
// two rows of a token (1.2 MB) fit no SM, and one row in flight per SM would
// ask 185 MB of the 126 MB L2 for the gradient pass's second read.  A cluster
// of CS CTAs therefore shares every row: CTA c owns the c-th of CS column slices.
// Full-vocabulary rows take clusters of 8 (15 co-resident, 120 SMs, two rows in
// flight each: 36 MB of rows between their first and second reads); sampled-token
// rows, whose second read carries the student only, clusters of 4 (36 co-resident,
// 144 SMs).  The SMs the clusters leave free run k_split_helper on a share of the
// rows.  The gradient's second read of a chunk follows its first within about
// one row's statistics, so it mostly hits L2.
//
// Per CTA (persistent, one per SM, rows cid, cid + nclusters, ...):
//   * a producer warp streams the slice, both models, through a ring of
//     kSStages chunks with bulk asynchronous copies (completion on a "full"
//     mbarrier; a chunk is refilled once every consumer warp has arrived on
//     its "empty" mbarrier).  It does not stop at row boundaries, so HBM stays
//     busy while rows are merged;
//   * two groups of 8 consumer warps take the cluster's rows in turn; each
//     folds its row's chunks into per-thread online accumulators
//     (max, S = sum exp(z - m) for both models, A = sum exp(z_s - m_s)
//     ((z_s - z_t) - d) with d at the running student argmax), merge them
//     across the CTA in a fixed lane order and push the CTA's 32-byte record
//     to every CTA of the cluster (st.async into a record ring, completion on
//     the receiver's mbarrier: no cluster barrier per row);
//   * every CTA merges the CS records in the same fixed order, so all use
//     bit-identical LSE and KL (deterministic), then writes the gradient of its
//     slice, g = w p_s ((z_s - z_t) - LSE_s + LSE_t - KL) (full vocabulary) or
//     g = w l (e_y - p_s) (sampled token), from the slice read again -- from L2,
//     where the stream left it moments before -- by the producer into a second
//     ring.  While one group exchanges records and writes its gradient, the
//     other folds the next row's fresh chunks, so the HBM stream does not pause.
// HBM traffic per row: each logit row read once, the gradient row written once.
// Every wait is bounded: on timeout the kernel records TURNOPD_ERR_TIMEOUT,
// stops waiting, lets its own copies land and returns.

#include <algorithm>
#include <cfloat>

#include "common.cuh"
#include "kernels.h"
#include "packed.cuh"
#include "ptx.cuh"
#include "row_math.cuh"

namespace turnopd {
namespace {

// CTAs per row: full vocabulary / sampled token (measured on the packed 8 x 4096 fp32
// batch with the helper grid at split rate 0.6: full 6.53 ms with clusters of 8, 6.98
// with 4 (6.83 with 4 and no helper); sampled 6.10 with 4, 6.55 with 8)
#ifndef TURNOPD_SPLIT_CS_FULL
#define TURNOPD_SPLIT_CS_FULL 8
#endif
#ifndef TURNOPD_SPLIT_CS_SAMPLED
#define TURNOPD_SPLIT_CS_SAMPLED 4
#endif
constexpr int kCSFull = TURNOPD_SPLIT_CS_FULL;
constexpr int kCSSampled = TURNOPD_SPLIT_CS_SAMPLED;
constexpr int kG = 2;                           // row groups per CTA (alternate rows)
constexpr int kNT = 256;                        // threads per group
constexpr int kNWG = kNT / 32;                  // warps per group
constexpr int kThreads = kG * kNT + 32;         // + the producer warp (17 warps: up to 96 registers)
constexpr int kChunkVec = 4 * kNT;              // float4 vectors per model per chunk (16 KB)
#ifndef TURNOPD_SPLIT_SSTAGES
#define TURNOPD_SPLIT_SSTAGES 3
#endif
#ifndef TURNOPD_SPLIT_KEEP
#define TURNOPD_SPLIT_KEEP 1
#endif
// Seven 32 KB stages in all, split between the fresh chunks and the chunks read
// again.  Measured on the packed 8 x 4096 fp32 batch: 3 fresh + 4 read-again
// stages 7.01 ms, 2 + 5 7.62 ms, 4 + 3 7.88 ms.
constexpr int kSStages = TURNOPD_SPLIT_SSTAGES;  // fresh chunks in flight (from HBM)
constexpr int kGStages = 7 - kSStages;          // chunks read again for the gradient
// The fresh chunks are marked L2 evict-last, so that the gradient's second read
// a few microseconds later finds more of them there; after that read the lines go
// back to normal priority.  Forward-only calls (no second read) leave the
// default priority.
constexpr bool kKeep = TURNOPD_SPLIT_KEEP != 0;
// The helper grid on the SMs the clusters leave free (k_split_helper): vectors per
// model and thread in one batch, threads per CTA, and its rows per second per SM
// against a cluster SM's, which sets the split of the row list.  Measured on the packed
// 8 x 4096 fp32 batch with the helper's statistics fed by its cp.async ring: full
// vocabulary 6.45 / 6.35 / 6.27 / 6.28 / 6.59 ms at 0.7 / 0.8 / 0.9 / 1.0 / 1.1;
// sampled 6.08 / 6.06 / 6.05 / 6.04 / 6.02 ms at 0.6 / 0.7 / 0.8 / 0.9 / 1.0 (with
// register-fed batches the best had been 0.7 and 0.6: 6.41 and 6.07 ms).  Batches of 8
// vectors were no faster than 4.
#ifndef TURNOPD_SPLIT_HELPER
#define TURNOPD_SPLIT_HELPER 1
#endif
#ifndef TURNOPD_SPLIT_RATE_FULL
#define TURNOPD_SPLIT_RATE_FULL 0.9
#endif
#ifndef TURNOPD_SPLIT_RATE_SAMPLED
#define TURNOPD_SPLIT_RATE_SAMPLED 1.0
#endif
#ifndef TURNOPD_SPLIT_HELPER_U
#define TURNOPD_SPLIT_HELPER_U 4
#endif
#ifndef TURNOPD_SPLIT_HELPER_THREADS
#define TURNOPD_SPLIT_HELPER_THREADS 512
#endif
constexpr bool kSplitHelper = TURNOPD_SPLIT_HELPER != 0;
constexpr int kSplitHelpStages = 3;  // cp.async ring of the helper's statistics pass
constexpr size_t split_helper_smem(int u, int nth) { return (size_t)kSplitHelpStages * 2 * u * nth * 16; }
constexpr double kRateFull = TURNOPD_SPLIT_RATE_FULL;
constexpr double kRateSampled = TURNOPD_SPLIT_RATE_SAMPLED;
constexpr int kHelperU = TURNOPD_SPLIT_HELPER_U;
constexpr int kHelperThreads = TURNOPD_SPLIT_HELPER_THREADS;
constexpr int kSlots = 2 * kG;                  // record ring
constexpr uint32_t kWaitLimit = 1u << 22;       // mbarrier polls before giving up
constexpr uint32_t kStageBytes = 2u * kChunkVec * 16u;

constexpr size_t split_smem_bytes(int cs)
{
    return (size_t)(kSStages + kGStages) * kStageBytes  // the two rings
           + kSlots * cs * 8 * sizeof(float)             // records
           + (2 * kSStages + 2 * kGStages + kSlots) * sizeof(uint64_t)
           + (kSStages + kGStages) * sizeof(uint32_t)    // chunk held by each stage
           + kG * kNWG * 8 * sizeof(float)               // per-warp partials
           + kG * 8 * sizeof(float)                      // row constants
           + kG * 2 * sizeof(float);                     // sampled-token logits
}

__device__ __forceinline__ float lane4(const float4 &v, int i)
{
    return i == 0 ? v.x : (i == 1 ? v.y : (i == 2 ? v.z : v.w));
}

// v with lane i replaced by the lowest finite float (never a maximum, adds 0)
__device__ __forceinline__ float4 fill_lane4(float4 v, int i)
{
    v.x = i == 0 ? -FLT_MAX : v.x;
    v.y = i == 1 ? -FLT_MAX : v.y;
    v.z = i == 2 ? -FLT_MAX : v.z;
    v.w = i == 3 ? -FLT_MAX : v.w;
    return v;
}

// Gradient of one vector (4 columns) from the row constants c (set by the
// merge below): g = w p ((z_s - z_t) - d - cp), or -w l p for a sampled-token row
// (SM; its g_y = w l (1 - p_y) is written apart).
template <bool G32, bool SM>
__device__ __forceinline__ float4 grad4(const float4 &a, const float4 &b, const float *c)
{
    const float2 L2 = splat(kLog2e), NLW = splat(c[0]);
    const float2 a01 = make_float2(a.x, a.y), a23 = make_float2(a.z, a.w);
    const float2 p01 = ex2x2(ffma2(a01, L2, NLW)), p23 = ex2x2(ffma2(a23, L2, NLW));
    float2 g01, g23;
    if (!SM) {
        const float2 SG = splat(c[1]);
        const float2 x01 = fsub2(a01, make_float2(b.x, b.y)), x23 = fsub2(a23, make_float2(b.z, b.w));
        if (G32) {
            const float2 ND = splat(c[2]), NCP = splat(c[3]);
            g01 = fmul2(p01, fadd2(ffma2(x01, SG, ND), NCP));
            g23 = fmul2(p23, fadd2(ffma2(x23, SG, ND), NCP));
        } else {
            const float2 NC = splat(c[4]);
            g01 = fmul2(p01, ffma2(x01, SG, NC));
            g23 = fmul2(p23, ffma2(x23, SG, NC));
        }
    } else {
        const float2 SGL = splat(c[5]);
        g01 = fmul2(p01, SGL);
        g23 = fmul2(p23, SGL);
    }
    return make_float4(g01.x, g01.y, g23.x, g23.y);
}

template <int CS, bool G32, bool SM>
__global__ void __launch_bounds__(kThreads, 1) k_row_split(RowIn p, int slice_vec, int nvec)
{
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ int s_dead;
    float4 *sring = reinterpret_cast<float4 *>(smem);                       // [kSStages][2][kChunkVec]
    float4 *gring = sring + (size_t)kSStages * 2 * kChunkVec;              // [kGStages][2][kChunkVec]
    float *rec = reinterpret_cast<float *>(gring + (size_t)kGStages * 2 * kChunkVec);  // [kSlots][CS][8]
    uint64_t *sfull = reinterpret_cast<uint64_t *>(rec + kSlots * CS * 8);  // [kSStages]
    uint64_t *sempty = sfull + kSStages;                                     // [kSStages]
    uint64_t *gfull = sempty + kSStages;                                     // [kGStages]
    uint64_t *gempty = gfull + kGStages;                                     // [kGStages]
    uint64_t *recv = gempty + kGStages;                                      // [kSlots]
    uint32_t *stag = reinterpret_cast<uint32_t *>(recv + kSlots);            // [kSStages]
    uint32_t *gtag = stag + kSStages;                                        // [kGStages]
    float *reds = reinterpret_cast<float *>(gtag + kGStages);                // [kG][kNWG][8]
    float *bcs = reds + kG * kNWG * 8;                                       // [kG][8]
    float *ysvs = bcs + kG * 8;                                              // [kG][2]

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const uint32_t rank = cluster_ctarank();
    const int cid = (int)cluster_id(), ncl = (int)cluster_count();
    const int v0 = (int)rank * slice_vec;  // first vector (4 floats) of my slice
    const int my_vec = max(0, min(slice_vec, nvec - v0));
    const int nchunk = (my_vec + kChunkVec - 1) / kChunkVec;
    const bool do_grad = p.grad != nullptr;

    if (tid == 0) {
        s_dead = 0;
        for (int s = 0; s < kSStages; ++s) {
            mbar_init(&sfull[s], 1);
            mbar_init(&sempty[s], kNWG);
            stag[s] = 0xffffffffu;
        }
        for (int s = 0; s < kGStages; ++s) {
            mbar_init(&gfull[s], 1);
            mbar_init(&gempty[s], kNWG);
            gtag[s] = 0xffffffffu;
        }
        for (int s = 0; s < kSlots; ++s)
            mbar_init(&recv[s], 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        for (int s = 0; s < kSlots; ++s)
            mbar_arrive_expect_tx(&recv[s], CS * 32u);  // first record of each slot
    }
    __syncthreads();
    cluster_sync();  // peers' barriers are initialised before any record is sent
    // Every CTA of this grid is resident: a helper grid launched after this one may
    // start now, on the SMs the clusters left free.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    // split_den > 0: the clusters take rows [0, nvalid split_num / split_den) of the list
    const int nv_all = *p.nvalid;
    const int nv = p.split_den ? (int)((int64_t)nv_all * p.split_num / p.split_den) : nv_all;
    const int n = nv > cid ? (nv - cid + ncl - 1) / ncl : 0;  // same for the whole cluster
    if (n == 0)
        return;

    const float *zs = static_cast<const float *>(p.zs);
    const float *zt = static_cast<const float *>(p.zt);

    auto dead = [&]() { return *(volatile int *)&s_dead != 0; };
    auto give_up = [&]() {
        s_dead = 1;
        set_status(p.status, TURNOPD_ERR_TIMEOUT);
    };
    auto wait_bar = [&](uint64_t *bar, uint32_t parity, bool cluster_scope) {
        if (dead())
            return;
        for (uint32_t it = 0; it < kWaitLimit; ++it)
            if (cluster_scope ? mbar_try_wait_cluster(bar, parity) : mbar_try_wait(bar, parity))
                return;
        give_up();
    };

    if (warp == kG * kNWG) {
        // ---------------------------------------------------------------- producer
        if (lane == 0) {
            const uint64_t keep = evict_last_policy();
            auto issue = [&](float4 *ring, uint64_t *fullb, uint32_t *tag, int stages, uint32_t t, bool fresh) {
                const int k = (int)(t / (uint32_t)nchunk), c = (int)(t % (uint32_t)nchunk);
                const int4 m = p.rows[cid + k * ncl];
                const int s = (int)(t % stages);
                const size_t base = (size_t)m.y * (size_t)p.ld + (size_t)v0 * 4 + (size_t)c * kChunkVec * 4;
                const uint32_t bytes = (uint32_t)min(kChunkVec, my_vec - c * kChunkVec) * 16u;
                const bool teacher = fresh || m.z < 0;  // a sampled-token gradient needs the student only
                float4 *dst = ring + (size_t)s * 2 * kChunkVec;
                *(volatile uint32_t *)&tag[s] = t;     // the stage now belongs to chunk t
                mbar_arrive_expect_tx(&fullb[s], (teacher ? 2u : 1u) * bytes);
                if (kKeep && do_grad && fresh) {
                    bulk_g2s(dst, zs + base, bytes, &fullb[s], keep);
                    bulk_g2s(dst + kChunkVec, zt + base, bytes, &fullb[s], keep);
                } else {
                    bulk_g2s_keep(dst, zs + base, bytes, &fullb[s]);
                    if (teacher)
                        bulk_g2s_keep(dst + kChunkVec, zt + base, bytes, &fullb[s]);
                }
            };
            // fresh chunks in row order; row k's chunks again once all of row k's
            // fresh chunks are issued.  Neither stream waits for the other's ring.
            const uint32_t total = (uint32_t)n * (uint32_t)nchunk;
            const uint32_t total_g = do_grad ? total : 0u;
            uint32_t ts = 0, tg = 0, idle = 0;
            while ((ts < total || tg < total_g) && !dead()) {
                bool moved = false;
                if (ts < total) {
                    const int s = (int)(ts % kSStages);
                    if (ts < (uint32_t)kSStages || mbar_test_wait(&sempty[s], ((ts / kSStages) - 1) & 1)) {
                        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                        issue(sring, sfull, stag, kSStages, ts++, true);
                        moved = true;
                    }
                }
                if (tg < total_g && ts >= (tg / (uint32_t)nchunk + 1u) * (uint32_t)nchunk) {
                    const int s = (int)(tg % kGStages);
                    if (tg < (uint32_t)kGStages || mbar_test_wait(&gempty[s], ((tg / kGStages) - 1) & 1)) {
                        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                        issue(gring, gfull, gtag, kGStages, tg++, false);
                        moved = true;
                    }
                }
                if (moved)
                    idle = 0;
                else if (++idle >= 16 * kWaitLimit)  // test_wait never suspends: more polls
                    give_up();
            }
            // after a timeout, let this CTA's own copies land before it exits
            if (dead()) {
                for (uint32_t u = ts > (uint32_t)kSStages ? ts - kSStages : 0; u < ts; ++u)
                    for (uint32_t it = 0; it < kWaitLimit; ++it)
                        if (mbar_try_wait(&sfull[u % kSStages], (u / kSStages) & 1))
                            break;
                for (uint32_t u = tg > (uint32_t)kGStages ? tg - kGStages : 0; u < tg; ++u)
                    for (uint32_t it = 0; it < kWaitLimit; ++it)
                        if (mbar_try_wait(&gfull[u % kGStages], (u / kGStages) & 1))
                            break;
            }
        }
        cluster_sync();
        return;
    }

    // -------------------------------------------------------------------- row groups
    // Group g takes rows g, g + 2, ... of the cluster's list: the statistics from the
    // fresh chunks, the cluster merge, then the gradient from the chunks read again.
    // While one group exchanges records and writes its gradient, the other folds the
    // next row's fresh chunks, so the HBM stream does not pause for either.
    const int group = warp / kNWG, gwarp = warp % kNWG, gtid = tid % kNT;
    float *red = reds + group * kNWG * 8;
    float *bc = bcs + group * 8;
    float *ysv = ysvs + group * 2;
    auto group_sync = [&]() { asm volatile("bar.sync %0, %1;" ::"r"(1 + group), "r"(kNT) : "memory"); };
    // chunk t of a ring: the stage must first be armed for chunk t (the other group
    // may still hold the stage's previous chunk), then its phase must complete
    auto wait_chunk = [&](uint64_t *fullb, const uint32_t *tag, int stages, uint32_t t) {
        const int s = (int)(t % stages);
        if (dead())
            return;
        uint32_t it = 0;
        while (*(volatile const uint32_t *)&tag[s] != t && ++it < kWaitLimit) {
        }
        if (it >= kWaitLimit) {
            give_up();
            return;
        }
        wait_bar(&fullb[s], (t / stages) & 1, false);
    };

    int4 m = make_int4(0, 0, -1, 0);
    if (group < n)
        m = p.rows[cid + group * ncl];
    for (int k = group; k < n; k += kG) {
        const int4 m_next = k + kG < n ? p.rows[cid + (k + kG) * ncl] : m;  // a row ahead
        const int y = m.z, yq = y >= 0 ? (y >> 2) - v0 : -1;

        // statistics of row k's slice, in packed pairs: per pair of vectors a max
        // pass, one rescale if the maximum moved, then the sums
        float ms = -INFINITY, mt = -INFINITY, dd = 0.f;
        float2 S2 = make_float2(0.f, 0.f), A2 = S2, T2 = S2;
        for (int c = 0; c < nchunk; ++c) {
            const uint32_t t = (uint32_t)k * (uint32_t)nchunk + (uint32_t)c;
            const int s = (int)(t % kSStages);
            wait_chunk(sfull, stag, kSStages, t);
            const float4 *cs = sring + (size_t)s * 2 * kChunkVec;
            const float4 *ct = cs + kChunkVec;
            const int cv = min(kChunkVec, my_vec - c * kChunkVec);
            if (!dead()) {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int q0 = gtid + 2 * h * kNT, q1 = q0 + kNT;
                    if (q0 >= cv)
                        break;
                    const bool v1ok = q1 < cv;
                    // a sampled-token row leaves y out of the student statistics (lowest
                    // finite value in its place; add_sampled_term brings its term back at
                    // the merge)
                    float4 x0 = cs[q0];
                    const float4 z0 = ct[q0];
                    if (SM && c * kChunkVec + q0 == yq) {
                        ysv[0] = lane4(x0, y & 3);
                        ysv[1] = lane4(z0, y & 3);
                        x0 = fill_lane4(x0, y & 3);
                    }
                    float4 x1 = v1ok ? cs[q1] : x0;
                    const float4 z1 = v1ok ? ct[q1] : z0;
                    if (SM && v1ok && c * kChunkVec + q1 == yq) {
                        ysv[0] = lane4(x1, y & 3);
                        ysv[1] = lane4(z1, y & 3);
                        x1 = fill_lane4(x1, y & 3);
                    }
                    // (x1, z1 repeat x0, z0 when the second vector is past the chunk: the
                    // maxima are unchanged and its sums are skipped)
                    const float cm = fmaxf(fmaxf(fmaxf(x0.x, x0.y), fmaxf(x0.z, x0.w)),
                                           fmaxf(fmaxf(x1.x, x1.y), fmaxf(x1.z, x1.w)));
                    const float cmt = fmaxf(fmaxf(fmaxf(z0.x, z0.y), fmaxf(z0.z, z0.w)),
                                            fmaxf(fmaxf(z1.x, z1.y), fmaxf(z1.z, z1.w)));
                    if (cm > ms) {
                        // reference difference at the first element equal to the new maximum
                        float xd = x0.x - z0.x;
                        if (x0.x != cm) {
                            xd = x0.y == cm ? x0.y - z0.y : x0.z == cm ? x0.z - z0.z : x0.w == cm ? x0.w - z0.w
                               : x1.x == cm ? x1.x - z1.x : x1.y == cm ? x1.y - z1.y
                               : x1.z == cm ? x1.z - z1.z : x1.w - z1.w;
                        }
                        const float2 f = splat(ex2((ms - cm) * kLog2e));
                        A2 = fmul2(ffma2(S2, splat(dd - xd), A2), f);
                        S2 = fmul2(S2, f);
                        dd = xd;
                        ms = cm;
                    }
                    if (cmt > mt) {
                        T2 = fmul2(T2, splat(ex2((mt - cmt) * kLog2e)));
                        mt = cmt;
                    }
                    const float2 L2 = splat(kLog2e), NS = splat(-ms * kLog2e), NTT = splat(-mt * kLog2e);
                    const float2 D = splat(dd);
                    const float4 xs[2] = {x0, x1}, zz[2] = {z0, z1};
#pragma unroll
                    for (int u = 0; u < 2; ++u) {
                        if (u == 1 && !v1ok)
                            break;
                        const float2 a01 = make_float2(xs[u].x, xs[u].y), a23 = make_float2(xs[u].z, xs[u].w);
                        const float2 b01 = make_float2(zz[u].x, zz[u].y), b23 = make_float2(zz[u].z, zz[u].w);
                        const float2 e01 = ex2x2(ffma2(a01, L2, NS)), e23 = ex2x2(ffma2(a23, L2, NS));
                        S2 = fadd2(S2, fadd2(e01, e23));
                        A2 = ffma2(e01, fsub2(fsub2(a01, b01), D), A2);
                        A2 = ffma2(e23, fsub2(fsub2(a23, b23), D), A2);
                        T2 = fadd2(T2, fadd2(ex2x2(ffma2(b01, L2, NTT)), ex2x2(ffma2(b23, L2, NTT))));
                    }
                }
            }
            __syncwarp();
            if (lane == 0)
                mbar_arrive(&sempty[s]);
        }

        // row k's partial -> record to every CTA of the cluster
        Student S = ms == -INFINITY ? student_empty() : Student{ms, S2.x + S2.y, A2.x + A2.y, dd};
        Teacher U = mt == -INFINITY ? teacher_empty() : Teacher{mt, T2.x + T2.y};
        lane_merge<32, true>(S, U);
        if (lane == 0) {
            float *rw = red + gwarp * 8;
            rw[0] = S.m, rw[1] = S.s, rw[2] = S.a, rw[3] = S.d, rw[4] = U.m, rw[5] = U.s;
        }
        group_sync();
        const int slot = k % kSlots;
        if (gwarp == 0) {
            Student A = student_empty();
            Teacher B = teacher_empty();
            if (lane < kNWG) {
                const float *r = red + lane * 8;
                A = Student{r[0], r[1], r[2], r[3]};
                B = Teacher{r[4], r[5]};
            }
            lane_merge<kNWG, true>(A, B);
            A.m = __shfl_sync(0xffffffffu, A.m, 0);
            A.s = __shfl_sync(0xffffffffu, A.s, 0);
            A.a = __shfl_sync(0xffffffffu, A.a, 0);
            A.d = __shfl_sync(0xffffffffu, A.d, 0);
            B.m = __shfl_sync(0xffffffffu, B.m, 0);
            B.s = __shfl_sync(0xffffffffu, B.s, 0);
            if (lane < CS) {
                const bool mine = yq >= 0 && yq < my_vec;
                const float ys = mine ? ysv[0] : 0.f, yt = mine ? ysv[1] : 0.f;
                const uint32_t ra = mapa(smem_u32(rec + (slot * CS + (int)rank) * 8), (uint32_t)lane);
                const uint32_t rbar = mapa(smem_u32(&recv[slot]), (uint32_t)lane);
                st_async16(ra, rbar, make_float4(A.m, A.s, A.a, A.d));
                st_async16(ra + 16, rbar, make_float4(B.m, B.s, ys, yt));
            }
            // the row's constants from the CS records, in the same order in every CTA
            wait_bar(&recv[slot], (uint32_t)((k / kSlots) & 1), true);
            const float *r = rec + slot * CS * 8;
            A = student_empty();
            B = teacher_empty();
            if (lane < CS) {
                const float4 x = *reinterpret_cast<const float4 *>(r + lane * 8);
                const float4 z = *reinterpret_cast<const float4 *>(r + lane * 8 + 4);
                A = Student{x.x, x.y, x.z, x.w};
                B = Teacher{z.x, z.y};
            }
            lane_merge<CS, true>(A, B);
            if (lane == 0) {
                const int owner = SM ? (y >> 2) / slice_vec : 0;
                const float omp = SM ? add_sampled_term(A, r[owner * 8 + 6]) : 0.f;  // 1 - p_y
                const RowConst rc = row_const(A, B);
                float e = rc.kl;
                if (SM)
                    e = (r[owner * 8 + 6] - r[owner * 8 + 7]) - rc.dl;
                // p |w| = 2^(z_s log2e - LSE_s log2e + log2 |w|); the sign of w enters
                // through an fma by sg
                const float wi = __int_as_float(m.w), wl = wi * e;
                const float sg = wi < 0.f ? -1.f : 1.f;
                bc[0] = -rc.lse_s * kLog2e + log2f(fabsf(SM ? wl : wi));  // nlw
                bc[1] = sg;
                bc[2] = -sg * rc.d;             // fp32 output: d and cp added separately
                bc[3] = -sg * rc.cp;
                bc[4] = -sg * (rc.d + rc.cp);   // bf16 output: one rounding of d + cp
                bc[5] = wl > 0.f ? -1.f : 1.f;  // sampled: sign of -w l
                bc[6] = wl * omp;               // sampled: g_y = w l (1 - p_y)
                if (rank == 0) {
                    if (!isfinite(rc.lse_s) || !isfinite(rc.lse_t) || !isfinite(e))
                        set_status(p.status, TURNOPD_ERR_NONFINITE);
                    p.token_loss[m.x] = e;
                    p.row_wl[cid + k * ncl] = (double)wi * (double)e;
                }
                mbar_arrive_expect_tx(&recv[slot], CS * 32u);  // re-arm for row k + kSlots
            }
        }
        group_sync();

        // the gradient of my slice from the chunks read again
        if (do_grad) {
            const size_t off = (size_t)m.y * (size_t)p.ld + (size_t)v0 * 4;
            for (int c = 0; c < nchunk; ++c) {
                const uint32_t t = (uint32_t)k * (uint32_t)nchunk + (uint32_t)c;
                const int s = (int)(t % kGStages);
                wait_chunk(gfull, gtag, kGStages, t);
                if (!dead()) {
                    const float4 *ga = gring + (size_t)s * 2 * kChunkVec, *gb = ga + kChunkVec;
                    const int cv = min(kChunkVec, my_vec - c * kChunkVec);
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int ql = gtid + u * kNT;
                        if (ql < cv) {
                            const int q = c * kChunkVec + ql;
                            const float4 a = ga[ql], b = SM ? a : gb[ql];
                            if (kKeep && (ql & 7) == 0) {  // one thread per 128-byte line of each model
                                l2_evict_normal(zs + off + (size_t)q * 4);
                                l2_evict_normal(zt + off + (size_t)q * 4);
                            }
                            const float4 g4 = grad4<G32, SM>(a, b, bc);
                            if (G32) {
                                __stcs(reinterpret_cast<float4 *>(static_cast<float *>(p.grad) + off) + q, g4);
                            } else {
                                uint2 o;
                                o.x = pack_bf16x2(g4.x, g4.y);
                                o.y = pack_bf16x2(g4.z, g4.w);
                                __stcs(reinterpret_cast<uint2 *>(static_cast<__nv_bfloat16 *>(p.grad) + off) + q, o);
                            }
                        }
                    }
                }
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(&gempty[s]);
            }
            // sampled token: g_y = w l (1 - p_y), over the value the vector store wrote
            // (the thread that stored y's vector, so the later store wins)
            if (SM && yq >= 0 && yq < my_vec && yq % kNT == gtid) {
                const size_t yo = (size_t)m.y * (size_t)p.ld + (size_t)y;
                if (G32)
                    static_cast<float *>(p.grad)[yo] = bc[6];
                else
                    static_cast<__nv_bfloat16 *>(p.grad)[yo] = __float2bfloat16_rn(bc[6]);
            }
        }
        m = m_next;
    }
    cluster_sync();  // no CTA leaves while a peer may still address its shared memory
}


// Helper for the SMs the clusters leave free, fp32 logits: one CTA per row at a time,
// rows j0 + blockIdx.x, j0 + blockIdx.x + gridDim.x, ... of the row list (j0 = the
// cluster grid's share).  The statistics pass streams both rows from HBM in batches of
// U vectors per model and thread, staged two batches ahead in a cp.async ring in shared
// memory, with a running maximum per thread (one rescale per batch when it moves) and A
// relative to the reference difference d at the running student argmax, as the cluster
// kernel keeps it; the gradient pass reads the row again from L2.  Launched as a dependent of the cluster grid (it starts once every
// cluster is resident) and completes only after it.
template <bool G32, bool SM, int U, int NTH>
__global__ void __launch_bounds__(NTH, 1) k_split_helper(RowIn p)
{
    constexpr int NW = NTH / 32;
    __shared__ float red[NW][8];
    __shared__ float bc[8];
    extern __shared__ float4 hring4[];  // [kSplitHelpStages][2][U][NTH]: the statistics pass's ring
    // the loss sum after this grid may take the first SM it frees (it waits for the grid)
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nvalid = *p.nvalid;
    const int j0 = p.split_den ? (int)((int64_t)nvalid * p.split_num / p.split_den) : 0;
    const int nvec = (int)(p.vocab / 4);
    const float *zs = static_cast<const float *>(p.zs);
    const float *zt = static_cast<const float *>(p.zt);
    const float2 L2 = splat(kLog2e);
    const float4 kFill4 = make_float4(-FLT_MAX, -FLT_MAX, -FLT_MAX, -FLT_MAX);
    for (int j = j0 + (int)blockIdx.x; j < nvalid; j += gridDim.x) {
        const int4 m = p.rows[j];
        const size_t off = (size_t)m.y * (size_t)p.ld;
        const float4 *vs = reinterpret_cast<const float4 *>(zs + off);
        const float4 *vt = reinterpret_cast<const float4 *>(zt + off);
        const int yvec = SM ? (m.z >> 2) : -1;  // the vector holding the sampled id
        float ms = -INFINITY, mt = -INFINITY, dd = 0.f;
        float2 S2 = make_float2(0.f, 0.f), A2 = S2, T2 = S2;
        // the statistics pass's batches land in a ring in shared memory by cp.async,
        // kSplitHelpStages - 1 batches ahead; each thread copies and reads only its own slots
        const int nbt = nvec > tid ? (nvec - tid + U * NTH - 1) / (U * NTH) : 0;
        auto slot = [&](int s, int mdl, int u) { return ((s * 2 + mdl) * U + u) * NTH + tid; };
        auto issue = [&](int bi) {  // batch bi into the ring (an empty group past the last)
            if (bi < nbt) {
                const int s = bi % kSplitHelpStages, q0 = tid + bi * U * NTH;
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int q = q0 + u * NTH;
                    if (q < nvec) {
                        cp_async16(&hring4[slot(s, 0, u)], vs + q);
                        cp_async16(&hring4[slot(s, 1, u)], vt + q);
                    }
                }
            }
            cp_async_commit();
        };
        for (int bi = 0; bi < kSplitHelpStages - 1; ++bi)
            issue(bi);
        for (int bi = 0; bi < nbt; ++bi) {
            const int q0 = tid + bi * U * NTH;
            float4 a[U], b[U];
            issue(bi + kSplitHelpStages - 1);
            cp_async_wait<kSplitHelpStages - 1>();  // batch bi has landed
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int q = q0 + u * NTH;
                if (q < nvec) {
                    a[u] = hring4[slot(bi % kSplitHelpStages, 0, u)];
                    b[u] = hring4[slot(bi % kSplitHelpStages, 1, u)];
                } else {
                    a[u] = b[u] = kFill4;  // adds 0, never the maximum
                }
            }
            // a sampled-token row leaves y out of the student statistics (lowest finite
            // value in its place; add_sampled_term brings its term back at the merge)
            if (SM && (unsigned)(yvec - q0) < (unsigned)(U * NTH)) {
#pragma unroll
                for (int u = 0; u < U; ++u)
                    if (yvec == q0 + u * NTH)
                        a[u] = fill_lane4(a[u], m.z & 3);
            }
            float cm = fmaxf(fmaxf(a[0].x, a[0].y), fmaxf(a[0].z, a[0].w));
            float cmt = fmaxf(fmaxf(b[0].x, b[0].y), fmaxf(b[0].z, b[0].w));
#pragma unroll
            for (int u = 1; u < U; ++u) {
                cm = fmaxf(cm, fmaxf(fmaxf(a[u].x, a[u].y), fmaxf(a[u].z, a[u].w)));
                cmt = fmaxf(cmt, fmaxf(fmaxf(b[u].x, b[u].y), fmaxf(b[u].z, b[u].w)));
            }
            if (cm > ms) {
                // reference difference at the first element of the batch equal to the new maximum
                float xd = 0.f;
                bool found = false;
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    if (!found && a[u].x == cm) { xd = a[u].x - b[u].x; found = true; }
                    if (!found && a[u].y == cm) { xd = a[u].y - b[u].y; found = true; }
                    if (!found && a[u].z == cm) { xd = a[u].z - b[u].z; found = true; }
                    if (!found && a[u].w == cm) { xd = a[u].w - b[u].w; found = true; }
                }
                const float2 f = splat(ex2((ms - cm) * kLog2e));
                A2 = fmul2(ffma2(S2, splat(dd - xd), A2), f);
                S2 = fmul2(S2, f);
                dd = xd;
                ms = cm;
            }
            if (cmt > mt) {
                T2 = fmul2(T2, splat(ex2((mt - cmt) * kLog2e)));
                mt = cmt;
            }
            const float2 NS = splat(-ms * kLog2e), NTT = splat(-mt * kLog2e), D = splat(dd);
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const float2 a01 = make_float2(a[u].x, a[u].y), a23 = make_float2(a[u].z, a[u].w);
                const float2 b01 = make_float2(b[u].x, b[u].y), b23 = make_float2(b[u].z, b[u].w);
                const float2 e01 = ex2x2(ffma2(a01, L2, NS)), e23 = ex2x2(ffma2(a23, L2, NS));
                S2 = fadd2(S2, fadd2(e01, e23));
                A2 = ffma2(e01, fsub2(fsub2(a01, b01), D), A2);
                A2 = ffma2(e23, fsub2(fsub2(a23, b23), D), A2);
                T2 = fadd2(T2, fadd2(ex2x2(ffma2(b01, L2, NTT)), ex2x2(ffma2(b23, L2, NTT))));
            }
        }
        Student S = ms == -INFINITY ? student_empty() : Student{ms, S2.x + S2.y, A2.x + A2.y, dd};
        Teacher T = mt == -INFINITY ? teacher_empty() : Teacher{mt, T2.x + T2.y};
        lane_merge<32, true>(S, T);
        if (lane == 0) {
            red[warp][0] = S.m, red[warp][1] = S.s, red[warp][2] = S.a, red[warp][3] = S.d;
            red[warp][4] = T.m, red[warp][5] = T.s;
        }
        __syncthreads();
        if (warp == 0) {
            Student A = student_empty();
            Teacher B = teacher_empty();
            if (lane < NW) {
                A = Student{red[lane][0], red[lane][1], red[lane][2], red[lane][3]};
                B = Teacher{red[lane][4], red[lane][5]};
            }
            lane_merge<NW, true>(A, B);
            if (lane == 0) {
                const int y = m.z;  // SM: in [0, V) (the compaction drops ids out of range); else -1
                const float zy = SM ? zs[off + y] : 0.f;
                const float omp = SM ? add_sampled_term(A, zy) : 0.f;  // 1 - p_y
                const RowConst rc = row_const(A, B);
                const float e = SM ? (zy - zt[off + y]) - rc.dl : rc.kl;
                const float wi = __int_as_float(m.w), wl = wi * e;
                const float sg = wi < 0.f ? -1.f : 1.f;
                if (!isfinite(rc.lse_s) || !isfinite(rc.lse_t) || !isfinite(e))
                    set_status(p.status, TURNOPD_ERR_NONFINITE);
                p.token_loss[m.x] = e;
                p.row_wl[j] = (double)wi * (double)e;
                // the row constants of grad4, as the cluster kernel sets them
                bc[0] = -rc.lse_s * kLog2e + log2f(fabsf(SM ? wl : wi));  // nlw
                bc[1] = sg;
                bc[2] = -sg * rc.d;
                bc[3] = -sg * rc.cp;
                bc[4] = -sg * (rc.d + rc.cp);
                bc[5] = wl > 0.f ? -1.f : 1.f;
                bc[6] = wl * omp;  // sampled: g_y = w l (1 - p_y)
            }
        }
        __syncthreads();
        if (p.grad) {
            float c[7];
#pragma unroll
            for (int i = 0; i < 7; ++i)
                c[i] = bc[i];
            for (int q0 = tid; q0 < nvec; q0 += U * NTH) {
                float4 a[U], b[U];
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int q = q0 + u * NTH;
                    if (q < nvec) {
                        a[u] = __ldg(vs + q);
                        b[u] = SM ? a[u] : __ldg(vt + q);
                    }
                }
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int q = q0 + u * NTH;
                    if (q >= nvec)
                        break;
                    const float4 g4 = grad4<G32, SM>(a[u], b[u], c);
                    if (G32) {
                        __stcs(reinterpret_cast<float4 *>(static_cast<float *>(p.grad) + off) + q, g4);
                    } else {
                        uint2 o;
                        o.x = pack_bf16x2(g4.x, g4.y);
                        o.y = pack_bf16x2(g4.z, g4.w);
                        __stcs(reinterpret_cast<uint2 *>(static_cast<__nv_bfloat16 *>(p.grad) + off) + q, o);
                    }
                }
            }
            // sampled token: g_y = w l (1 - p_y), over the value the vector store wrote
            // (same thread, so the later store wins)
            if (SM && yvec % NTH == tid) {
                if (G32)
                    static_cast<float *>(p.grad)[off + m.z] = c[6];
                else
                    static_cast<__nv_bfloat16 *>(p.grad)[off + m.z] = __float2bfloat16_rn(c[6]);
            }
        }
        __syncthreads();  // red and bc are reused by the next row
    }
    asm volatile("griddepcontrol.wait;" ::: "memory");  // complete only after the cluster grid
}

// The cluster grid (as many clusters of CS as are co-resident, cached per device)
// and the helper grid on the SMs the clusters leave free.
template <int CS, bool SM>
cudaError_t launch_split_t(const RowIn &p, bool fp32_grad, int nvec, double rate, cudaStream_t stream)
{
    constexpr size_t kSmem = split_smem_bytes(CS);
    const int slice_vec = (nvec + CS - 1) / CS;
    auto kern = fp32_grad ? k_row_split<CS, true, SM> : k_row_split<CS, false, SM>;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return e;
    if (dev >= 64)
        return cudaErrorInvalidDevice;
    static int grid_cache[64][2];  // per instantiation (cluster size, mode) and gradient type
    const int gi = fp32_grad ? 1 : 0;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmem;
    cfg.stream = stream;
    if (grid_cache[dev][gi] == 0) {
        if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem)) != cudaSuccess)
            return e;
        if (CS > 8 && (e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1)) != cudaSuccess)
            return e;
        cfg.gridDim = dim3(CS);
        int ncl = 0;
        if ((e = cudaOccupancyMaxActiveClusters(&ncl, kern, &cfg)) != cudaSuccess)
            return e;
        if (ncl < 1)
            return cudaErrorInvalidConfiguration;
        grid_cache[dev][gi] = ncl;
    }
    cfg.gridDim = dim3(grid_cache[dev][gi] * CS);
    // the helper grid on the SMs the clusters leave free, with the row list split so
    // that both grids finish together
    RowIn pl = p;
    const int free_sm = kSplitHelper ? device_sm_count() - grid_cache[dev][gi] * CS : 0;
    if (free_sm > 0) {
        const double cl = (double)(grid_cache[dev][gi] * CS);
        pl.split_den = 1 << 20;
        pl.split_num = (int32_t)(pl.split_den * cl / (cl + rate * free_sm) + 0.5);
    }
    e = cudaLaunchKernelEx(&cfg, kern, pl, slice_vec, nvec);
    if (e != cudaSuccess || pl.split_den == 0)
        return e;
    cudaLaunchConfig_t hc = {};
    cudaLaunchAttribute ha[1];
    ha[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    ha[0].val.programmaticStreamSerializationAllowed = 1;
    hc.attrs = ha;
    hc.numAttrs = 1;
    hc.gridDim = dim3(free_sm);
    hc.blockDim = dim3(kHelperThreads);
    hc.dynamicSmemBytes = split_helper_smem(kHelperU, kHelperThreads);
    hc.stream = stream;
    auto helper = fp32_grad ? k_split_helper<true, SM, kHelperU, kHelperThreads>
                            : k_split_helper<false, SM, kHelperU, kHelperThreads>;
    if ((e = cudaFuncSetAttribute(helper, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)split_helper_smem(kHelperU, kHelperThreads))) != cudaSuccess)
        return e;
    return cudaLaunchKernelEx(&hc, helper, pl);
}

}  // namespace

// fp32 logits, 16-byte aligned rows (V and ld multiples of 4): the split-row
// kernel on as many clusters as are co-resident, the helper kernel beside it.
// *used = false leaves the row to the portable kernel.
cudaError_t launch_row_split(const RowIn &p, bool fp32_grad, cudaStream_t stream, bool *used)
{
    *used = false;
    auto al16 = [](const void *q) { return (reinterpret_cast<uintptr_t>(q) & 15u) == 0; };
    if (p.vocab % 4 != 0 || p.ld % 4 != 0 || !al16(p.zs) || !al16(p.zt) || (p.grad && !al16(p.grad)))
        return cudaSuccess;
    if (p.vocab / 4 > (int64_t)0x7fffffff)
        return cudaSuccess;
    const int nvec = (int)(p.vocab / 4);
    *used = true;
    // every listed row of a sampled-token call carries y in [0, V)
    if (p.mode == TURNOPD_SAMPLED_TOKEN)
        return launch_split_t<kCSSampled, true>(p, fp32_grad, nvec, kRateSampled, stream);
    return launch_split_t<kCSFull, false>(p, fp32_grad, nvec, kRateFull, stream);
}

}  // namespace turnopd
