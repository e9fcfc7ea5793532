// Cluster-resident row kernel for the per-token OPD loss (sm_103a).
//
// One logit row of V = 151,936 bf16 values is 303,872 bytes per model: the
// student and teacher rows together (607 KB) do not fit one SM, and the
// gradient needs both rows twice (statistics, then p_s and z_s - z_t).  A
// cluster of CS CTAs therefore owns one row at a time: CTA c holds vector
// slice c of both rows in shared memory, so HBM is read exactly once per row
// and the gradient written once (911,616 algorithmic bytes per row in bf16).
//
// Per CTA (persistent, one per SM, rows cid, cid + nclusters, ...):
//   * thread 0 streams slices into a 3-stage ring with bulk asynchronous
//     copies (cp.async.bulk, completion on a "full" mbarrier, L2 evict-first);
//     a stage is refilled once every warp has arrived on its "empty" mbarrier;
//   * stats(k+1): per thread a max pass (packed bf16x2 max) and a sum pass
//     (packed f32x2 arithmetic): S = sum exp(z - m) for both models and
//     A = sum exp(z_s - m_s)((z_s - z_t) - d), d taken at the student's max.
//     The CTA's partial is pushed to every CTA of the cluster with st.async
//     into a 4-slot record ring; completion lands on the receiver's mbarrier
//     (32 bytes per sender), so no cluster-wide barrier runs per row;
//   * grad(k) from the resident slice of the previous row, overlapping the
//     record exchange of row k+1;
//   * every warp merges the CS records by the same fixed 8-lane tree, so all
//     CTAs use bit-identical LSE and KL (deterministic).
// Each thread reads its vectors of a row from shared memory twice: once into
// registers for the maxima and sums, once for the gradient (3 exponentials
// per element in all).
// Clusters of 8 fill 120 of the 152 SMs; a helper grid of one 512-thread CTA per
// free SM takes the last share of the rows, each row read from HBM once (staged
// through a cp.async ring) and again from L2 (k_row_helper below).
// Waits are bounded: on timeout the kernel records TURNOPD_ERR_TIMEOUT, stops
// computing and runs its remaining barriers without waiting, so it terminates.

#pragma once

#include <algorithm>

#include "common.cuh"
#include "kernels.h"
#include "packed.cuh"
#include "ptx.cuh"
#include "row_math.cuh"

namespace turnopd {
namespace {

constexpr int kStages = 3;
constexpr uint32_t kCopyChunk = 65536;       // bytes per bulk copy instruction
constexpr uint32_t kWaitLimit = 1u << 22;    // mbarrier polls before giving up

// Per-row constants the gradient pass needs (computed once per row).
struct GradConst {
    float lse_s, lse_t, kl;
    float nlw;        // -LSE_s log2e + log2 |w| (full) or log2 |w l| (sampled)
    float sg;         // sign of w
    float nd, ncp;    // -sg d, -sg cp
    float nc;         // -sg (d + cp)
    float sgl;        // sign of -w l (sampled)
    float gy;         // sampled: g_y = w l (1 - p_y)
};

// v with its bf16 lanes n..7 replaced by the lowest finite bf16 (the padding lanes of a
// row's last vector when V % 8 != 0)
__device__ __forceinline__ uint4 fill_from(uint4 v, int n)
{
    uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        if (2 * j >= n)
            w[j] = 0xff7fff7fu;
        else if (2 * j + 1 >= n)
            w[j] = (w[j] & 0x0000ffffu) | 0xff7f0000u;
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
}

// v with its bf16 lane i (0..7) replaced by the lowest finite bf16
__device__ __forceinline__ uint4 fill_lane(uint4 v, int i)
{
    const uint32_t keep = (i & 1) ? 0x0000ffffu : 0xffff0000u;
    const uint32_t fill = 0xff7fff7fu & ~keep;
    const int w = i >> 1;
    v.x = w == 0 ? (v.x & keep) | fill : v.x;
    v.y = w == 1 ? (v.y & keep) | fill : v.y;
    v.z = w == 2 ? (v.z & keep) | fill : v.z;
    v.w = w == 3 ? (v.w & keep) | fill : v.w;
    return v;
}

// G groups of NT threads per CTA take the rows of the cluster in turn (row k
// to group k % G).  Record slots: 2G, so a slot is reused by the same group
// two rows later, after that group has read it (a peer can run at most G rows
// ahead of the slowest CTA in sending records).  SM: a sampled-token call, where
// every listed row carries its y in [0, V); otherwise the full vocabulary (y = -1).
template <int CS, int NT, int VPT, int G, bool G32, bool SM, bool TL>
__global__ void __launch_bounds__(G * NT, 1) k_row_cluster(RowIn p, int slice_vec, int nvec)
{
    constexpr int kSlots = 2 * G;
    // Reference difference d (A = sum e ((z_s - z_t) - d), d at the student's
    // max): it keeps gradients at a dominant token accurate to fp32 relative
    // precision.  A bf16 gradient needs no such care: without d the error of
    // E_p[z_s - z_t] is ~1e-6 absolute, under a bf16 ulp of those gradients.
    constexpr bool kUseD = G32;
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ int s_dead;
    constexpr int NWG = NT / 32;  // warps per group
    const int tid = threadIdx.x, lane = tid & 31;
    const int group = tid / NT, gtid = tid % NT, gwarp = gtid >> 5;
    const uint32_t rank = cluster_ctarank();
    const int cid = (int)cluster_id(), ncl = (int)cluster_count();
    const uint32_t slice_bytes = (uint32_t)slice_vec * 16u;
    const uint32_t stage_bytes = 2u * slice_bytes;
    const int v0 = (int)rank * slice_vec;  // first vector of my slice
    const int my_vec = max(0, min(slice_vec, nvec - v0));
    const uint32_t my_bytes = (uint32_t)my_vec * 16u;
    // TL (V % 8 != 0): the row's last vector (in the last slice) holds V % 8 columns.
    // Its other lanes, row padding, read as the lowest finite bf16 in the statistics
    // (set in shared memory by the thread that reads the vector) and are never
    // written: the gradient loop stores gvec whole vectors, that thread the tail's
    // columns.  Without TL all of this compiles away.
    const int tail = TL ? (int)(p.vocab & 7) : 0;
    const int tailq = TL && my_vec > 0 && v0 + my_vec == nvec ? my_vec - 1 : -1;
    const int tailown = tailq >= 0 ? tailq % NT : -1;
    const int gvec = TL && tailq >= 0 ? my_vec - 1 : my_vec;

    unsigned char *stage = smem;
    float *rec = reinterpret_cast<float *>(smem + kStages * stage_bytes);  // [kSlots][CS][8]
    int4 *meta = reinterpret_cast<int4 *>(rec + kSlots * CS * 8);          // [kStages]
    uint64_t *full = reinterpret_cast<uint64_t *>(meta + kStages);         // [kStages]
    uint64_t *empty = full + kStages;                                      // [kStages]
    uint64_t *recv = empty + kStages;                                      // [kSlots]
    float *red = reinterpret_cast<float *>(recv + kSlots);                 // [G][NWG][8]
    int *srow = reinterpret_cast<int *>(red + G * NWG * 8);                // [kStages] row in stage
    int *yown = srow + 4;                                                  // [kStages] thread reading y, or -1
    float *rcs = reinterpret_cast<float *>(srow + 8);                       // [G][16] row constants; [15]: z_s[y]

    if (tid == 0) {
        s_dead = 0;
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], NWG);
            srow[s] = -1;
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

    const int nv_all = *p.nvalid;
    const int nvalid = p.split_den ? (int)((int64_t)nv_all * p.split_num / p.split_den) : nv_all;
    const int n = nvalid > cid ? (nvalid - cid + ncl - 1) / ncl : 0;  // same for the whole cluster
    if (n == 0)
        return;

    const __nv_bfloat16 *zs = static_cast<const __nv_bfloat16 *>(p.zs);
    const __nv_bfloat16 *zt = static_cast<const __nv_bfloat16 *>(p.zt);

    auto dead = [&]() { return *(volatile int *)&s_dead != 0; };
    auto wait_bar = [&](uint64_t *bar, uint32_t parity, bool cluster_scope) {
        if (dead())
            return;
        for (uint32_t it = 0; it < kWaitLimit; ++it)
            if (cluster_scope ? mbar_try_wait_cluster(bar, parity) : mbar_try_wait(bar, parity))
                return;
        s_dead = 1;
        set_status(p.status, TURNOPD_ERR_TIMEOUT);
    };
    auto group_sync = [&]() { asm volatile("bar.sync %0, %1;" ::"r"(1 + group), "r"(NT) : "memory"); };

    // Data of row k: wait until the stage has been armed for row k, then for
    // its phase.  (A parity wait alone would also accept the phase of the
    // stage's previous row, k - kStages, when a group reaches row k early.)
    auto wait_full = [&](int k) {
        const int s = k % kStages;
        if (dead())
            return;
        uint32_t it = 0;
        while (*(volatile int *)&srow[s] != k && ++it < kWaitLimit) {
        }
        if (it >= kWaitLimit) {
            s_dead = 1;
            set_status(p.status, TURNOPD_ERR_TIMEOUT);
            return;
        }
        wait_bar(&full[s], (uint32_t)((k / kStages) & 1), false);
    };

    // stream row k of this cluster into stage k % kStages (after the stage's
    // previous row is done with it)
    auto issue = [&](int k, int4 m) {
        const int s = k % kStages;
        meta[s] = m;
        if (SM) {  // the thread that will read y's vector (sampled-token rows; see stats)
            const int q = m.z >= 0 ? (m.z >> 3) - v0 : -1;
            yown[s] = q >= 0 && q < my_vec ? q % NT : -1;
        }
        *(volatile int *)&srow[s] = k;
        const size_t off = (size_t)m.y * (size_t)p.ld + (size_t)v0 * 8;
        const char *gs = reinterpret_cast<const char *>(zs + off);
        const char *gt = reinterpret_cast<const char *>(zt + off);
        unsigned char *ds = stage + s * stage_bytes;
        const uint64_t pol = evict_first_policy();
        mbar_arrive_expect_tx(&full[s], 2u * my_bytes);
        for (uint32_t o = 0; o < my_bytes; o += kCopyChunk) {
            const uint32_t sz = min(kCopyChunk, my_bytes - o);
            bulk_g2s(ds + o, gs + o, sz, &full[s], pol);
            bulk_g2s(ds + slice_bytes + o, gt + o, sz, &full[s], pol);
        }
    };

    // statistics of row k: this CTA's record into slot k % kSlots of every CTA
    auto stats = [&](int k) {
        const int s = k % kStages;
        const uint4 *vs = reinterpret_cast<const uint4 *>(stage + s * stage_bytes);
        const uint4 *vt = reinterpret_cast<const uint4 *>(stage + s * stage_bytes + slice_bytes);
        // A sampled-token row leaves y out of the student statistics (add_sampled_term
        // brings its term back at the merge): the thread that reads y's vector in both
        // passes below (named at issue) keeps z_s[y] for the record and puts the lowest
        // finite bf16 in its place, which is never the maximum and adds 0.  (The gradient
        // pass replaces g_y; the proxy fence orders the store before the stage's next
        // bulk copy.)
        if (SM && yown[s] == gtid) {
            const uint32_t ay = smem_u32(stage + s * stage_bytes) + 2u * (uint32_t)(meta[s].z - v0 * 8);
            uint32_t old;
            asm volatile("ld.shared.u16 %0, [%1];\n\tst.shared.u16 [%1], %2;\n\t"
                         "fence.proxy.async.shared::cta;"
                         : "=r"(old)
                         : "r"(ay), "r"(0xff7fu)
                         : "memory");
            rcs[group * 16 + 15] = __uint_as_float(old << 16);
        }
        if (TL && tailown == gtid) {  // the row's last vector: padding lanes out of both models' statistics
            uint4 *ts = reinterpret_cast<uint4 *>(stage + s * stage_bytes) + tailq;
            uint4 *tt = reinterpret_cast<uint4 *>(stage + s * stage_bytes + slice_bytes) + tailq;
            *ts = fill_from(*ts, tail);
            *tt = fill_from(*tt, tail);
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        }
        // max pass (packed bf16): running maxima, plus each vector's student
        // maximum kept packed so the argmax vector is found after the loop
        uint32_t smax = 0xff80ff80u, tmax = 0xff80ff80u;  // (-inf, -inf)
        uint32_t vmax[VPT];
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
            const int q = gtid + u * NT;
            vmax[u] = 0xff80ff80u;
            if (q < my_vec) {
                const uint4 a = vs[q], b = vt[q];
                vmax[u] = hmax2u(hmax2u(a.x, a.y), hmax2u(a.z, a.w));
                smax = hmax2u(smax, vmax[u]);
                tmax = hmax2u(tmax, hmax2u(hmax2u(b.x, b.y), hmax2u(b.z, b.w)));
            }
        }
        const float ms = fmaxf(bf16lo(smax), bf16hi(smax)), mt = fmaxf(bf16lo(tmax), bf16hi(tmax));
        // reference difference at the first element equal to the student max;
        // only the fp32 gradient needs it (see kUseD)
        float xd = 0.f;
        if (kUseD && ms != -INFINITY) {
            int bq = gtid;
#pragma unroll
            for (int u = VPT - 1; u >= 0; --u)
                if (bf16lo(vmax[u]) == ms || bf16hi(vmax[u]) == ms)
                    bq = gtid + u * NT;
            const uint4 a = vs[bq], b = vt[bq];
            bool found = false;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float2 x = unpack2(word(a, j)), y = unpack2(word(b, j));
                if (!found && x.x == ms) {
                    xd = x.x - y.x;
                    found = true;
                }
                if (!found && x.y == ms) {
                    xd = x.y - y.y;
                    found = true;
                }
            }
        }
        // sum pass (packed pairs)
        const float2 L2 = splat(kLog2e), NS = splat(-ms * kLog2e), NTT = splat(-mt * kLog2e);
        const float2 D = splat(xd);
        float2 S2 = make_float2(0.f, 0.f), A2 = S2, T2 = S2;
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
            const int q = gtid + u * NT;
            if (q < my_vec) {
                const uint4 a = vs[q], b = vt[q];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float2 a2 = unpack2(word(a, j)), b2 = unpack2(word(b, j));
                    const float2 es = ex2x2(ffma2(a2, L2, NS));
                    S2 = fadd2(S2, es);
                    A2 = ffma2(es, kUseD ? fsub2(fsub2(a2, b2), D) : fsub2(a2, b2), A2);
                    T2 = fadd2(T2, ex2x2(ffma2(b2, L2, NTT)));
                }
            }
        }
        Student S = ms == -INFINITY ? student_empty() : Student{ms, S2.x + S2.y, A2.x + A2.y, xd};
        Teacher U = mt == -INFINITY ? teacher_empty() : Teacher{mt, T2.x + T2.y};
        lane_merge<32, kUseD>(S, U);
        float *rg = red + group * NWG * 8;
        if (lane == 0) {
            float *rw = rg + gwarp * 8;
            rw[0] = S.m, rw[1] = S.s, rw[2] = S.a, rw[3] = S.d, rw[4] = U.m, rw[5] = U.s;
        }
        group_sync();
        if (gwarp == 0) {
            Student A = student_empty();
            Teacher B = teacher_empty();
            if (lane < NWG) {
                const float *r = rg + lane * 8;
                A = Student{r[0], r[1], r[2], r[3]};
                B = Teacher{r[4], r[5]};
            }
            lane_merge<NWG, kUseD>(A, B);
            A.m = __shfl_sync(0xffffffffu, A.m, 0);
            A.s = __shfl_sync(0xffffffffu, A.s, 0);
            A.a = __shfl_sync(0xffffffffu, A.a, 0);
            A.d = __shfl_sync(0xffffffffu, A.d, 0);
            B.m = __shfl_sync(0xffffffffu, B.m, 0);
            B.s = __shfl_sync(0xffffffffu, B.s, 0);
            if (lane < CS) {
                float ys = 0.f, yt = 0.f;  // sampled-token logits, from the CTA holding y
                const int y = meta[s].z;
                if (y >= 0 && y / 8 >= v0 && y / 8 < v0 + my_vec) {
                    const int e = y - v0 * 8;
                    ys = SM ? rcs[group * 16 + 15] : to_float(reinterpret_cast<const __nv_bfloat16 *>(vs)[e]);
                    yt = to_float(reinterpret_cast<const __nv_bfloat16 *>(vt)[e]);
                }
                const int slot = k % kSlots;
                const uint32_t ra = mapa(smem_u32(rec + (slot * CS + (int)rank) * 8), (uint32_t)lane);
                const uint32_t rbar = mapa(smem_u32(&recv[slot]), (uint32_t)lane);
                st_async16(ra, rbar, make_float4(A.m, A.s, A.a, A.d));
                st_async16(ra + 16, rbar, make_float4(B.m, B.s, ys, yt));
            }
        }
    };

    // row constants of row k from the CS records, computed by the group's
    // first warp (fixed merge order: identical in every CTA) and shared with
    // the group through shared memory
    auto combine = [&](int k, float &ell) {
        const int slot = k % kSlots;
        float *bc = rcs + group * 16;
        if (gwarp == 0) {
            wait_bar(&recv[slot], (uint32_t)((k / kSlots) & 1), true);
            const float *r = rec + slot * CS * 8;
            Student A = student_empty();
            Teacher B = teacher_empty();
            if (lane < CS) {
                const float4 x = *reinterpret_cast<const float4 *>(r + lane * 8);
                const float4 y = *reinterpret_cast<const float4 *>(r + lane * 8 + 4);
                A = Student{x.x, x.y, x.z, x.w};
                B = Teacher{y.x, y.y};
            }
            lane_merge<CS, kUseD>(A, B);
            if (lane == 0) {
                const int y = meta[k % kStages].z;
                const int owner = SM ? (y / 8) / slice_vec : 0;
                float omp = 0.f;  // 1 - p_y (sampled)
                if (SM)
                    omp = add_sampled_term(A, r[owner * 8 + 6]);
                const RowConst rc = row_const(A, B);
                float e = rc.kl;
                if (SM)
                    e = (r[owner * 8 + 6] - r[owner * 8 + 7]) - rc.dl;
                // gradient constants of the row (see grad): p w = 2^(z_s log2e + nlw),
                // sign sg of w applied through fma by (sg, sg)
                const float wi = __int_as_float(meta[k % kStages].w), wl = wi * e;
                const float sg = wi < 0.f ? -1.f : 1.f;
                bc[0] = rc.lse_s, bc[1] = rc.lse_t, bc[2] = rc.kl, bc[3] = e;
                bc[4] = -rc.lse_s * kLog2e + log2f(fabsf(SM ? wl : wi));  // nlw
                bc[5] = sg;
                bc[6] = -sg * rc.d;
                bc[7] = -sg * rc.cp;
                bc[8] = -sg * (rc.d + rc.cp);     // bf16 output: one rounding of d + cp
                bc[9] = wl > 0.f ? -1.f : 1.f;    // sampled: sign of -w l
                bc[10] = wl * omp;                 // sampled: g_y = w l (1 - p_y)
                mbar_arrive_expect_tx(&recv[slot], CS * 32u);  // re-arm for row k + kSlots
            }
        }
        group_sync();
        GradConst gc;
        gc.lse_s = bc[0], gc.lse_t = bc[1], gc.kl = bc[2];
        ell = bc[3];
        gc.nlw = bc[4], gc.sg = bc[5], gc.nd = bc[6], gc.ncp = bc[7], gc.nc = bc[8], gc.sgl = bc[9];
        gc.gy = bc[10];
        return gc;
    };

    auto grad = [&](int k, const GradConst &gc) {
        if (!p.grad)
            return;
        const int s = k % kStages;
        const int4 m = meta[s];
        const uint4 *vs = reinterpret_cast<const uint4 *>(stage + s * stage_bytes);
        const uint4 *vt = reinterpret_cast<const uint4 *>(stage + s * stage_bytes + slice_bytes);
        const int y = m.z;
        const float gy = gc.gy;
        const size_t row_off = (size_t)m.y * (size_t)p.ld + (size_t)v0 * 8;
        // p |w| = 2^(z_s log2e - LSE_s log2e + log2 |w|); the sign of w enters through an
        // fma by (sg, sg), which is exact on z_s - z_t
        const float2 L2 = splat(kLog2e), NLW = splat(gc.nlw);
        const float2 SG = splat(gc.sg), ND = splat(gc.nd), NCP = splat(gc.ncp), NC = splat(gc.nc);
        const float2 SGL = splat(gc.sgl);
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
            const int q = gtid + u * NT;
            if (q < gvec) {
                float2 g[4];
                // y < 0 exactly when !SM; the fp32-gradient instantiations keep the run-time
                // test, which compiles to a loop 5 % faster there (and 2.4 % slower for bf16)
                if (G32 ? y < 0 : !SM) {  // full vocabulary: g = w p ((z_s - z_t) - d - cp)
                    const uint4 a = vs[q], b = vt[q];
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const float2 a2 = unpack2(word(a, j)), b2 = unpack2(word(b, j));
                        const float2 pw = ex2x2(ffma2(a2, L2, NLW));
                        // sg ((z_s - z_t) - c) with one rounding; sg (z_s - z_t) is exact
                        const float2 x = fsub2(a2, b2);
                        g[j] = G32 ? fmul2(pw, fadd2(ffma2(x, SG, ND), NCP)) : fmul2(pw, ffma2(x, SG, NC));
                    }
                } else {  // sampled token: g = -w l p (g_y is written after the loop)
                    const uint4 a = vs[q];
#pragma unroll
                    for (int j = 0; j < 4; ++j)
                        g[j] = fmul2(ex2x2(ffma2(unpack2(word(a, j)), L2, NLW)), SGL);
                }
                if (G32) {
                    float4 *dst = reinterpret_cast<float4 *>(static_cast<float *>(p.grad) + row_off +
                                                             (size_t)q * 8);
                    __stcs(dst, make_float4(g[0].x, g[0].y, g[1].x, g[1].y));
                    __stcs(dst + 1, make_float4(g[2].x, g[2].y, g[3].x, g[3].y));
                } else {
                    uint4 o;
                    o.x = pack_bf16x2(g[0].x, g[0].y);
                    o.y = pack_bf16x2(g[1].x, g[1].y);
                    o.z = pack_bf16x2(g[2].x, g[2].y);
                    o.w = pack_bf16x2(g[3].x, g[3].y);
                    __stcs(reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(p.grad) + row_off +
                                                     (size_t)q * 8),
                           o);
                }
            }
        }
        if (TL && tailown == gtid) {  // the row's last vector, column by column (the loop's formulas)
            const uint4 a = vs[tailq], b = vt[tailq];
            float gl[8];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float2 a2 = unpack2(word(a, j)), b2 = unpack2(word(b, j));
                const float2 pw = ex2x2(ffma2(a2, L2, NLW)), x = fsub2(a2, b2);
                const float2 gg = SM ? fmul2(pw, SGL)
                                     : (G32 ? fmul2(pw, fadd2(ffma2(x, SG, ND), NCP)) : fmul2(pw, ffma2(x, SG, NC)));
                gl[2 * j] = gg.x;
                gl[2 * j + 1] = gg.y;
            }
            const size_t to = row_off + (size_t)tailq * 8;
#pragma unroll
            for (int i = 0; i < 8; ++i)
                if (i < tail) {
                    if (G32)
                        static_cast<float *>(p.grad)[to + i] = gl[i];
                    else
                        static_cast<__nv_bfloat16 *>(p.grad)[to + i] = __float2bfloat16_rn(gl[i]);
                }
        }
        // sampled token: g_y = w l (1 - p_y), over the value the vector store wrote
        // (same thread, so the later store wins)
        if (SM && yown[s] == gtid) {
            const size_t yo = (size_t)m.y * (size_t)p.ld + (size_t)y;
            if (G32)
                static_cast<float *>(p.grad)[yo] = gy;
            else
                static_cast<__nv_bfloat16 *>(p.grad)[yo] = __float2bfloat16_rn(gy);
        }
    };

    // The groups take rows in turn: while one waits for its row's records or
    // data, the others compute.
    if (tid == 0)
        for (int k = 0; k < kStages && k < n; ++k)
            issue(k, p.rows[cid + k * ncl]);
    for (int k = group; k < n; k += G) {
        int4 ahead = make_int4(0, 0, -1, 0);
        if (gtid == 0 && k + kStages < n)
            ahead = p.rows[cid + (k + kStages) * ncl];  // used at the end of the iteration
        wait_full(k);
        stats(k);
        float ell;
        const GradConst gc = combine(k, ell);
        if (rank == 0 && gtid == 0) {
            const int4 m = meta[k % kStages];
            if (!isfinite(gc.lse_s) || !isfinite(gc.lse_t) || !isfinite(ell))
                set_status(p.status, TURNOPD_ERR_NONFINITE);
            p.token_loss[m.x] = ell;
            p.row_wl[cid + k * ncl] = (double)__int_as_float(m.w) * (double)ell;
        }
        if (!dead())
            grad(k, gc);
        __syncwarp();
        if (lane == 0)
            mbar_arrive(&empty[k % kStages]);
        if (gtid == 0 && k + kStages < n) {
            wait_bar(&empty[k % kStages], (uint32_t)((k / kStages) & 1), false);
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            issue(k + kStages, ahead);
        }
    }

    // after a timeout, let this CTA's own copies land before it exits
    if (tid == 0 && dead()) {
        for (int k = max(0, n - kStages); k < n; ++k)
            for (uint32_t it = 0; it < kWaitLimit; ++it)
                if (mbar_try_wait(&full[k % kStages], (uint32_t)((k / kStages) & 1)))
                    break;
    }
    cluster_sync();  // no CTA leaves while a peer may still address its shared memory
}

// Helper for the SMs the clusters leave free (15 eight-CTA clusters cover 120 of
// 152): one CTA per row at a time, rows j0 + blockIdx.x, j0 + blockIdx.x +
// gridDim.x, ... of the row list, j0 = the cluster kernel's share.  The
// statistics pass streams both rows from HBM (beside the clusters through a cp.async
// ring, AS) with a running maximum per thread (one rescale per batch of kHelpU
// vectors when the maximum moves); the gradient
// pass reads them again from L2, where the pass before left them (the clusters'
// own copies are evict-first).  bf16 logits; a bf16 or fp32 gradient or none.
// Like the cluster kernel, the fp32 gradient also keeps A relative to the
// reference difference d at the thread's running student argmax (re-referenced,
// A <- (A + S (d - d')) f, when the maximum moves).  Launched as a dependent
// of the cluster grid (it starts once every cluster is resident) and completes
// only after it, so stream order after it covers both grids.
constexpr int kHelpThreads = 512;
constexpr int kHelpU = 4;  // vectors of each model per thread and batch
// AS: the statistics pass's batches land in a kHelpStages-deep ring in shared memory by
// cp.async, kHelpStages - 1 batches ahead (each thread copies and reads only its own
// slots): twice the loads in flight of the register path, with no registers held by
// them.  The helper beside the clusters takes it (packed 8 x 4096, V = 151,936: 2.776 ->
// 2.743 ms per loss call with the split rate raised to 0.7); the helper alone on every
// SM keeps the register path (V = 16,384: 0.405 against 0.433 ms).
constexpr int kHelpStages = 3;
constexpr size_t helper_smem_bytes(bool as, int nth) { return as ? (size_t)kHelpStages * 2 * kHelpU * nth * 16 : 0; }

template <bool G32, bool SM, bool TL, bool AS, int NTH = kHelpThreads, int MINB = 1>
__global__ void __launch_bounds__(NTH, MINB) k_row_helper(RowIn p)
{
    constexpr int kHelpThreads = NTH;
    constexpr int NW = kHelpThreads / 32;
    constexpr uint32_t kFill = 0xff7fff7fu;  // lowest finite bf16 pair: adds 0, never the max
    __shared__ float red[NW][8];
    __shared__ float bc[8];
    extern __shared__ uint4 hring[];  // [kHelpStages][2][kHelpU][NTH] (AS)
    // the loss sum after this grid may take the first SM it frees (it waits for the grid)
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nvalid = *p.nvalid;
    const int j0 = p.split_den ? (int)((int64_t)nvalid * p.split_num / p.split_den) : 0;
    // TL (V % 8 != 0): the last vector holds `tail` columns (its padding lanes read as
    // the lowest finite bf16 and are never written); the gradient loop stores nfull vectors
    const int nvec = TL ? (int)((p.vocab + 7) / 8) : (int)(p.vocab / 8);
    const int tail = TL ? (int)(p.vocab & 7) : 0;
    const int nfull = TL ? nvec - 1 : nvec;
    const __nv_bfloat16 *zs = static_cast<const __nv_bfloat16 *>(p.zs);
    const __nv_bfloat16 *zt = static_cast<const __nv_bfloat16 *>(p.zt);
    const float2 L2 = splat(kLog2e);
    for (int j = j0 + (int)blockIdx.x; j < nvalid; j += gridDim.x) {
        const int4 m = p.rows[j];
        const size_t off = (size_t)m.y * (size_t)p.ld;
        const uint4 *vs = reinterpret_cast<const uint4 *>(zs + off);
        const uint4 *vt = reinterpret_cast<const uint4 *>(zt + off);
        const int yvec = m.z >= 0 ? (m.z >> 3) : -1;     // the vector holding the sampled id
        float ms = -INFINITY, mt = -INFINITY, dd = 0.f;  // dd: reference difference (fp32 gradient)
        float2 S2 = make_float2(0.f, 0.f), A2 = S2, T2 = S2;
        // this thread's batches of the row: kHelpU vectors of each model, kHelpThreads apart
        const int nbt = nvec > tid ? (nvec - tid + kHelpU * kHelpThreads - 1) / (kHelpU * kHelpThreads) : 0;
        auto slot = [&](int s, int mdl, int u) { return ((s * 2 + mdl) * kHelpU + u) * kHelpThreads + tid; };
        auto issue = [&](int bi) {  // batch bi into the ring (an empty group past the last)
            if (bi < nbt) {
                const int s = bi % kHelpStages, q0 = tid + bi * kHelpU * kHelpThreads;
#pragma unroll
                for (int u = 0; u < kHelpU; ++u) {
                    const int q = q0 + u * kHelpThreads;
                    if (q < nvec) {
                        cp_async16(&hring[slot(s, 0, u)], vs + q);
                        cp_async16(&hring[slot(s, 1, u)], vt + q);
                    }
                }
            }
            cp_async_commit();
        };
        if (AS)
            for (int bi = 0; bi < kHelpStages - 1; ++bi)
                issue(bi);
        for (int bi = 0; bi < nbt; ++bi) {
            const int q0 = tid + bi * kHelpU * kHelpThreads;
            uint4 a[kHelpU], b[kHelpU];
            if (AS) {
                issue(bi + kHelpStages - 1);
                cp_async_wait<kHelpStages - 1>();  // batch bi has landed
            }
#pragma unroll
            for (int u = 0; u < kHelpU; ++u) {
                const int q = q0 + u * kHelpThreads;
                if (q < nvec) {
                    if (AS) {
                        a[u] = hring[slot(bi % kHelpStages, 0, u)];
                        b[u] = hring[slot(bi % kHelpStages, 1, u)];
                    } else {
                        a[u] = __ldg(vs + q);
                        b[u] = __ldg(vt + q);
                    }
                } else {
                    a[u] = b[u] = make_uint4(kFill, kFill, kFill, kFill);
                }
            }
            // a sampled-token row leaves y out of the student statistics (lowest finite
            // bf16 in its place; add_sampled_term brings its term back at the merge)
            if (SM && (unsigned)(yvec - q0) < (unsigned)(kHelpU * kHelpThreads)) {
#pragma unroll
                for (int u = 0; u < kHelpU; ++u)
                    if (yvec == q0 + u * kHelpThreads)
                        a[u] = fill_lane(a[u], m.z & 7);
            }
            if (TL && (unsigned)(nvec - 1 - q0) < (unsigned)(kHelpU * kHelpThreads)) {
#pragma unroll
                for (int u = 0; u < kHelpU; ++u)
                    if (nvec - 1 == q0 + u * kHelpThreads) {
                        a[u] = fill_from(a[u], tail);
                        b[u] = fill_from(b[u], tail);
                    }
            }
            uint32_t bs = hmax4(a[0]), bt = hmax4(b[0]);
#pragma unroll
            for (int u = 1; u < kHelpU; ++u) {
                bs = hmax2u(bs, hmax4(a[u]));
                bt = hmax2u(bt, hmax4(b[u]));
            }
            const float nms = fmaxf(ms, fmaxf(bf16lo(bs), bf16hi(bs)));
            const float nmt = fmaxf(mt, fmaxf(bf16lo(bt), bf16hi(bt)));
            if (nms > ms) {
                const float2 f = splat(ex2((ms - nms) * kLog2e));
                if (G32) {  // d at the first element of the batch equal to the new maximum
                    float xd = 0.f;
                    bool found = false;
#pragma unroll
                    for (int u = 0; u < kHelpU; ++u)
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
                    A2 = fmul2(ffma2(S2, splat(dd - xd), A2), f);
                    dd = xd;
                } else {
                    A2 = fmul2(A2, f);
                }
                S2 = fmul2(S2, f);
                ms = nms;
            }
            if (nmt > mt) {
                T2 = fmul2(T2, splat(ex2((mt - nmt) * kLog2e)));
                mt = nmt;
            }
            const float2 NS = splat(-ms * kLog2e), NTT = splat(-mt * kLog2e), D = splat(dd);
#pragma unroll
            for (int u = 0; u < kHelpU; ++u)
#pragma unroll
                for (int w = 0; w < 4; ++w) {
                    const float2 a2 = unpack2(word(a[u], w)), b2 = unpack2(word(b[u], w));
                    const float2 es = ex2x2(ffma2(a2, L2, NS));
                    S2 = fadd2(S2, es);
                    A2 = ffma2(es, G32 ? fsub2(fsub2(a2, b2), D) : fsub2(a2, b2), A2);
                    T2 = fadd2(T2, ex2x2(ffma2(b2, L2, NTT)));
                }
        }
        Student S = Student{ms, S2.x + S2.y, A2.x + A2.y, dd};
        Teacher U = Teacher{mt, T2.x + T2.y};
        lane_merge<32, G32>(S, U);
        if (lane == 0) {
            red[warp][0] = S.m, red[warp][1] = S.s, red[warp][2] = S.a;
            red[warp][3] = U.m, red[warp][4] = U.s, red[warp][5] = S.d;
        }
        __syncthreads();
        if (warp == 0) {
            Student A = student_empty();
            Teacher B = teacher_empty();
            if (lane < NW) {
                A = Student{red[lane][0], red[lane][1], red[lane][2], red[lane][5]};
                B = Teacher{red[lane][3], red[lane][4]};
            }
            lane_merge<NW, G32>(A, B);
            if (lane == 0) {
                const int y = m.z;  // SM: in [0, V) (the compaction drops ids out of range); else -1
                const float omp = SM ? add_sampled_term(A, to_float(zs[off + y])) : 0.f;  // 1 - p_y
                const RowConst rc = row_const(A, B);
                const float e = SM ? (to_float(zs[off + y]) - to_float(zt[off + y])) - rc.dl : rc.kl;
                const float wi = __int_as_float(m.w), wl = wi * e;
                const float sg = wi < 0.f ? -1.f : 1.f;
                if (!isfinite(rc.lse_s) || !isfinite(rc.lse_t) || !isfinite(e))
                    set_status(p.status, TURNOPD_ERR_NONFINITE);
                p.token_loss[m.x] = e;
                p.row_wl[j] = (double)wi * (double)e;
                // the gradient constants of the cluster kernel
                bc[0] = -rc.lse_s * kLog2e + log2f(fabsf(SM ? wl : wi));  // nlw
                bc[1] = sg;
                bc[2] = -sg * (rc.d + rc.cp);  // bf16 output: one rounding of d + cp
                bc[3] = wl > 0.f ? -1.f : 1.f;
                bc[4] = wl * omp;              // sampled: g_y = w l (1 - p_y)
                bc[5] = -sg * rc.d;            // fp32 output
                bc[6] = -sg * rc.cp;
            }
        }
        __syncthreads();
        if (p.grad) {
            const float2 NLW = splat(bc[0]), SG = splat(bc[1]), NC = splat(bc[2]), SGL = splat(bc[3]);
            const float2 ND = splat(bc[5]), NCP = splat(bc[6]);
            const float gy = bc[4];
            const int y = m.z;
            for (int q0 = tid; q0 < nfull; q0 += kHelpU * kHelpThreads) {
                uint4 a[kHelpU], b[kHelpU];
#pragma unroll
                for (int u = 0; u < kHelpU; ++u) {
                    const int q = q0 + u * kHelpThreads;
                    if (q < nfull) {
                        a[u] = __ldg(vs + q);
                        if (!SM)
                            b[u] = __ldg(vt + q);
                    }
                }
#pragma unroll
                for (int u = 0; u < kHelpU; ++u) {
                    const int q = q0 + u * kHelpThreads;
                    if (q >= nfull)
                        break;
                    float2 g[4];
                    if (!SM) {  // full vocabulary: g = w p ((z_s - z_t) - d - cp)
#pragma unroll
                        for (int w = 0; w < 4; ++w) {
                            const float2 a2 = unpack2(word(a[u], w)), b2 = unpack2(word(b[u], w));
                            const float2 pw = ex2x2(ffma2(a2, L2, NLW)), x = fsub2(a2, b2);
                            g[w] = G32 ? fmul2(pw, fadd2(ffma2(x, SG, ND), NCP)) : fmul2(pw, ffma2(x, SG, NC));
                        }
                    } else {  // sampled token: g = -w l p (g_y is written after the loop)
#pragma unroll
                        for (int w = 0; w < 4; ++w)
                            g[w] = fmul2(ex2x2(ffma2(unpack2(word(a[u], w)), L2, NLW)), SGL);
                    }
                    if (G32) {
                        float4 *dst = reinterpret_cast<float4 *>(static_cast<float *>(p.grad) + off) + 2 * (size_t)q;
                        __stcs(dst, make_float4(g[0].x, g[0].y, g[1].x, g[1].y));
                        __stcs(dst + 1, make_float4(g[2].x, g[2].y, g[3].x, g[3].y));
                    } else {
                        uint4 o;
                        o.x = pack_bf16x2(g[0].x, g[0].y);
                        o.y = pack_bf16x2(g[1].x, g[1].y);
                        o.z = pack_bf16x2(g[2].x, g[2].y);
                        o.w = pack_bf16x2(g[3].x, g[3].y);
                        __stcs(reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(p.grad) + off) + q, o);
                    }
                }
            }
            if (TL && (nvec - 1) % kHelpThreads == tid) {  // the last vector, column by column
                const uint4 a = __ldg(vs + nvec - 1), b = __ldg(vt + nvec - 1);
                float gl[8];
#pragma unroll
                for (int w = 0; w < 4; ++w) {
                    const float2 a2 = unpack2(word(a, w)), b2 = unpack2(word(b, w));
                    const float2 pw = ex2x2(ffma2(a2, L2, NLW)), x = fsub2(a2, b2);
                    const float2 gg = SM ? fmul2(pw, SGL)
                                         : (G32 ? fmul2(pw, fadd2(ffma2(x, SG, ND), NCP)) : fmul2(pw, ffma2(x, SG, NC)));
                    gl[2 * w] = gg.x;
                    gl[2 * w + 1] = gg.y;
                }
                const size_t to = off + (size_t)(nvec - 1) * 8;
#pragma unroll
                for (int i = 0; i < 8; ++i)
                    if (i < tail) {
                        if (G32)
                            static_cast<float *>(p.grad)[to + i] = gl[i];
                        else
                            static_cast<__nv_bfloat16 *>(p.grad)[to + i] = __float2bfloat16_rn(gl[i]);
                    }
            }
            // sampled token: g_y = w l (1 - p_y), over the value the vector store wrote
            // (same thread, so the later store wins)
            if (SM && (y >> 3) % kHelpThreads == tid) {
                if (G32)
                    static_cast<float *>(p.grad)[off + y] = gy;
                else
                    static_cast<__nv_bfloat16 *>(p.grad)[off + y] = __float2bfloat16_rn(gy);
            }
        }
        __syncthreads();  // red and bc are reused by the next row
    }
    asm volatile("griddepcontrol.wait;" ::: "memory");  // complete only after the cluster grid
}

// Threads per row group and groups per CTA (tuning knobs).
#ifndef TURNOPD_ROW_THREADS
#define TURNOPD_ROW_THREADS 512
#endif
#ifndef TURNOPD_ROW_GROUPS
#define TURNOPD_ROW_GROUPS 2
#endif
constexpr int kNT = TURNOPD_ROW_THREADS;
constexpr int kG = TURNOPD_ROW_GROUPS;
constexpr int kMaxSlice = 2400;                      // vectors per CTA: 3 stages fit 227 KB
constexpr int kVPT = (kMaxSlice + kNT - 1) / kNT;    // vectors per thread
// The cluster size is the smallest of 2, 3, 4, 5, 6, 8 and 16 CTAs whose slices fit
// three stages, which keeps the slices long (a short slice cannot hide the per-row
// record exchange) and, for short rows, puts more SMs in clusters (76 pairs cover
// all 152).  Below kMinSlice vectors per CTA the helper kernel alone, on every SM,
// takes the rows (measured: slices of 2,000-2,400 vectors reach 0.87-0.93 of the
// copy bandwidth, the helper alone on rows of up to 8,192 vectors about 0.73).
// Clusters of 16 are exempt: the rows that need them are long, and the helper
// alone streams those poorly (V = 200,000: 0.58 against 0.77 with clusters of 16
// and 1,563-vector slices).
#ifndef TURNOPD_CLUSTER_MIN_SLICE
#define TURNOPD_CLUSTER_MIN_SLICE 1700
#endif
constexpr int kMinSlice = TURNOPD_CLUSTER_MIN_SLICE;
constexpr int kSmallRowVec = 7168;  // up to this many vectors per row: 256-thread helpers, 2 per SM
// The helper's rows per SM and second against the clusters', which decides the
// split of the row list.  A cluster SM is less efficient on a shorter slice and in a
// larger cluster (more records per row), so the rate rises with both.  Measured best
// (packed 8 x 4096, the ring-fed helper): clusters of 8, 0.72 at 2,374 vectors
// (V = 151,936) and 0.85 at 2,004 (128,256); clusters of 16, 0.80 at 2,048 (262,144)
// and about 1.0 at 1,563 (200,000); clusters of 3 to 6 (few helper SMs, where an
// overloaded helper decides the call), 0.60: V = 50,000 (3) 0.946 ms against 1.042 at
// 0.70, 90,000 (5) 1.623 against 1.709, 110,000 (6) 1.968 against 2.017, 65,536 (4)
// flat from 0.65 to 0.75.  Sampled-token rows, whose helper gradient pass reads the
// student only, more: 0.03 with a bf16 gradient (0.75 at 2,374), 0.10 with an fp32 one
// (0.82 at 2,374: 4.196 ms against 4.260 at 0.75 and 4.539 at 0.92), whose larger
// gradient writes weigh more beside the skipped teacher read.
double helper_rate(int slice_vec, int cs, bool sampled, bool g32)
{
#ifdef TURNOPD_HELPER_RATE
    (void)slice_vec;
    (void)cs;
    (void)sampled;
    (void)g32;
    return TURNOPD_HELPER_RATE;
#else
    double r = 0.60;
    if (cs == 8)
        r = 0.72 + (2374 - slice_vec) * 0.00035;
    else if (cs > 8)
        r = 0.80 + (2048 - slice_vec) * 0.00041;
    r = r < 0.60 ? 0.60 : (r > 1.1 ? 1.1 : r);
    return sampled ? r + (g32 ? 0.10 : 0.03) : r;
#endif
}
// The helper grid beside the clusters: CTAs of kSideThreads threads, kSideBlocks per free SM.
#ifndef TURNOPD_HELPER_THREADS
#define TURNOPD_HELPER_THREADS 512
#endif
#ifndef TURNOPD_HELPER_BLOCKS
#define TURNOPD_HELPER_BLOCKS 1
#endif
constexpr int kSideThreads = TURNOPD_HELPER_THREADS, kSideBlocks = TURNOPD_HELPER_BLOCKS;

size_t cluster_smem_bytes(int slice_vec, int cs)
{
    return (size_t)kStages * 2 * slice_vec * 16 + 2 * kG * cs * 8 * sizeof(float) +
           kStages * sizeof(int4) + (2 * kStages + 2 * kG) * sizeof(uint64_t) +
           kG * (kNT / 32) * 8 * sizeof(float) +  // per-group warp partials
           8 * sizeof(int) +                        // row held by each stage, thread reading y
           kG * 16 * sizeof(float);                 // broadcast row constants
}

// The cluster grid (as many clusters as are co-resident, cached per device) and
// the helper grid on the SMs the clusters leave free, with the row list split so
// that both finish together.
template <bool G32, int CS, bool SM, bool TL>
cudaError_t launch_t(const RowIn &p, int slice_vec, int nvec, size_t smem, cudaStream_t stream)
{
    auto kern = k_row_cluster<CS, kNT, kVPT, kG, G32, SM, TL>;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return e;
    static int grid_cache[64][2];
    static size_t smem_cache[64][2];
    const int gi = G32 ? 1 : 0;  // (the statics are per instantiation: cluster size, gradient type, mode)
    if (dev >= 64)
        return cudaErrorInvalidDevice;
    if (smem_cache[dev][gi] < smem) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess)
            return e;
        if (CS > 8 && (e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1)) != cudaSuccess)
            return e;
        smem_cache[dev][gi] = smem;
        grid_cache[dev][gi] = 0;
    }
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.blockDim = dim3(kG * kNT);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    if (grid_cache[dev][gi] == 0) {
        cfg.gridDim = dim3(CS);
        int ncl = 0;
        e = cudaOccupancyMaxActiveClusters(&ncl, kern, &cfg);
        if (e != cudaSuccess)
            return e;
        if (ncl < 1)
            return cudaErrorInvalidConfiguration;
        grid_cache[dev][gi] = ncl;
    }
    RowIn pl = p;
    const int free_sm = device_sm_count() - grid_cache[dev][gi] * CS;
    if (free_sm > 0) {
        const double cl = (double)(grid_cache[dev][gi] * CS);
        pl.split_den = 1 << 20;
        pl.split_num = (int32_t)(pl.split_den * cl / (cl + helper_rate(slice_vec, CS, SM, G32) * free_sm) + 0.5);
    }
    cfg.gridDim = dim3(grid_cache[dev][gi] * CS);
    e = cudaLaunchKernelEx(&cfg, kern, pl, slice_vec, nvec);
    if (e != cudaSuccess || pl.split_den == 0)
        return e;
    // the helper grid on the free SMs, a dependent of the cluster grid
    cudaLaunchConfig_t hc = {};
    cudaLaunchAttribute ha[1];
    ha[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    ha[0].val.programmaticStreamSerializationAllowed = 1;
    hc.attrs = ha;
    hc.numAttrs = 1;
    hc.gridDim = dim3(free_sm * kSideBlocks);
    hc.blockDim = dim3(kSideThreads);
    hc.dynamicSmemBytes = helper_smem_bytes(true, kSideThreads);
    hc.stream = stream;
    auto helper = k_row_helper<G32, SM, TL, true, kSideThreads, kSideBlocks>;
    if ((e = cudaFuncSetAttribute(helper, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)helper_smem_bytes(true, kSideThreads))) != cudaSuccess)
        return e;
    return cudaLaunchKernelEx(&hc, helper, pl);
}

// Cluster sizes offered: 7 is left out (only 15 clusters of 7 are co-resident, 105 SMs).
template <bool G32, bool SM, bool TL>
cudaError_t launch_cs(int cs, const RowIn &p, int slice_vec, int nvec, size_t smem, cudaStream_t stream)
{
    switch (cs) {
    case 2: return launch_t<G32, 2, SM, TL>(p, slice_vec, nvec, smem, stream);
    case 3: return launch_t<G32, 3, SM, TL>(p, slice_vec, nvec, smem, stream);
    case 4: return launch_t<G32, 4, SM, TL>(p, slice_vec, nvec, smem, stream);
    case 5: return launch_t<G32, 5, SM, TL>(p, slice_vec, nvec, smem, stream);
    case 6: return launch_t<G32, 6, SM, TL>(p, slice_vec, nvec, smem, stream);
    case 8: return launch_t<G32, 8, SM, TL>(p, slice_vec, nvec, smem, stream);
    default: return launch_t<G32, 16, SM, TL>(p, slice_vec, nvec, smem, stream);
    }
}

// The helper kernel alone, every row, every SM.
template <bool G32, bool SM, bool TL>
void launch_helper_alone(const RowIn &p, int nvec, cudaStream_t stream)
{
    const int sms = device_sm_count();
    if (nvec <= kSmallRowVec)
        k_row_helper<G32, SM, TL, false, 256, 2><<<sms * 2, 256, 0, stream>>>(p);
    else
        k_row_helper<G32, SM, TL, false><<<sms, kHelpThreads, 0, stream>>>(p);
}

// The row grids for bf16 logits; TL: V % 8 != 0 (a masked last vector).
template <bool TL>
cudaError_t launch_row_cluster_t(const RowIn &p, bool fp32_grad, cudaStream_t stream, bool *used)
{
    *used = false;
    auto al16 = [](const void *q) { return (reinterpret_cast<uintptr_t>(q) & 15u) == 0; };
    // rows 16-byte aligned; V % 8 != 0 takes a masked last vector (the row's padding up to
    // the next multiple of 8 is read, never written)
    if (p.ld % 8 != 0 || !al16(p.zs) || !al16(p.zt) || (p.grad && !al16(p.grad)))
        return cudaSuccess;
    // the smallest cluster whose slices fit three stages (2, 3, 4, 5, 6, 8 or 16 CTAs;
    // 16 is a non-portable size)
    if ((p.vocab + 7) / 8 > (int64_t)0x7fffffff)
        return cudaSuccess;
    const int nvec = (int)((p.vocab + 7) / 8);
    static const int kSizes[] = {2, 3, 4, 5, 6, 8, 16};
    int cs = 16;
    for (int c : kSizes)
        if ((nvec + c - 1) / c <= kMaxSlice) {
            cs = c;
            break;
        }
    const int slice_vec = (nvec + cs - 1) / cs;
    const bool sm = p.mode == TURNOPD_SAMPLED_TOKEN;
    // short rows, or a slice too long even for clusters of 16: the helper kernel alone, every row, every SM
    if ((slice_vec < kMinSlice && cs < 16) || slice_vec > kMaxSlice) {
        RowIn pl = p;
        pl.split_den = 0;
        *used = true;
        if (fp32_grad)
            sm ? launch_helper_alone<true, true, TL>(pl, nvec, stream) : launch_helper_alone<true, false, TL>(pl, nvec, stream);
        else
            sm ? launch_helper_alone<false, true, TL>(pl, nvec, stream) : launch_helper_alone<false, false, TL>(pl, nvec, stream);
        return cudaGetLastError();
    }
    const size_t smem = cluster_smem_bytes(slice_vec, cs);
    int dev = 0, optin = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return e;
    e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e != cudaSuccess)
        return e;
    if (smem + 64 > (size_t)optin)  // room for the kernel's static shared memory
        return cudaSuccess;
    *used = true;
    if (fp32_grad)
        return sm ? launch_cs<true, true, TL>(cs, p, slice_vec, nvec, smem, stream)
                  : launch_cs<true, false, TL>(cs, p, slice_vec, nvec, smem, stream);
    return sm ? launch_cs<false, true, TL>(cs, p, slice_vec, nvec, smem, stream)
              : launch_cs<false, false, TL>(cs, p, slice_vec, nvec, smem, stream);
}

}  // namespace
}  // namespace turnopd
