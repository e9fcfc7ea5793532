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
//     copies (cp.async.bulk, completion on an mbarrier, L2 evict-first);
//   * stats(k+1): each thread takes the max over its vectors, then sums
//     exp(z - m) for both models and A = sum exp(z_s - m_s)((z_s - z_t) - d);
//     the CTA's partial goes to every CTA of the cluster through distributed
//     shared memory (one 32-byte record per CTA per row);
//   * barrier.cluster arrive, grad(k) from the resident slice of the previous
//     row, barrier.cluster wait: the exchange latency of row k+1 hides behind
//     the gradient pass of row k;
//   * every CTA merges the CS records in rank order (identical arithmetic in
//     every CTA, deterministic), so all slices use the same LSE and KL.
// No CTA spins on another CTA's memory; the only waits are the hardware
// cluster barrier (all CTAs of a cluster run the same row count) and
// mbarrier waits on this CTA's own copies, bounded with an error status.

#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace turnopd {
namespace {

constexpr int kStages = 3;
constexpr uint32_t kCopyChunk = 16384;       // bytes per bulk copy instruction
constexpr uint32_t kWaitLimit = 1u << 22;    // mbarrier polls before giving up

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint32_t cluster_ctarank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ uint32_t cluster_id()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
    return r;
}

__device__ __forceinline__ uint32_t cluster_count()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
    return r;
}

__device__ __forceinline__ void cluster_arrive()
{
    asm volatile("barrier.cluster.arrive.release;" ::: "memory");
}

__device__ __forceinline__ void cluster_wait()
{
    asm volatile("barrier.cluster.wait.acquire;" ::: "memory");
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ uint64_t evict_first_policy()
{
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar,
                                         uint64_t pol)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1], %2, [%3], %4;" ::"r"(smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(pol)
        : "memory");
}

// Store 16 bytes into the shared memory of CTA `rank` of this cluster at the
// address that `local` has in this CTA.
__device__ __forceinline__ void st_cluster(const void *local, uint32_t rank, float4 v)
{
    uint32_t raddr;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(raddr) : "r"(smem_u32(local)), "r"(rank));
    asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(raddr), "f"(v.x), "f"(v.y),
                 "f"(v.z), "f"(v.w)
                 : "memory");
}

__device__ __forceinline__ void unpack8(const uint4 u, float *x)
{
    x[0] = bf16lo(u.x), x[1] = bf16hi(u.x), x[2] = bf16lo(u.y), x[3] = bf16hi(u.y);
    x[4] = bf16lo(u.z), x[5] = bf16hi(u.z), x[6] = bf16lo(u.w), x[7] = bf16hi(u.w);
}

struct Smem {
    unsigned char *stage;  // kStages x [zs slice | zt slice]
    float *rec;            // [2 slots][CS][8]
    int4 *meta;            // [kStages] row records
    uint64_t *full;        // [kStages] mbarriers
    float *red;            // [warps][8]
};

template <int CS, int NT, int VPT, bool G32>
__global__ void __launch_bounds__(NT, 1) k_row_cluster(RowIn p, int slice_vec, int nvec)
{
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ int s_dead;
    constexpr int NW = NT / 32;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const uint32_t rank = cluster_ctarank();
    const int cid = (int)cluster_id(), ncl = (int)cluster_count();
    const uint32_t slice_bytes = (uint32_t)slice_vec * 16u;
    const uint32_t stage_bytes = 2u * slice_bytes;
    const int v0 = (int)rank * slice_vec;                       // first vector of my slice
    const int my_vec = max(0, min(slice_vec, nvec - v0));
    const uint32_t my_bytes = (uint32_t)my_vec * 16u;

    Smem sm;
    sm.stage = smem;
    sm.rec = reinterpret_cast<float *>(smem + kStages * stage_bytes);
    sm.meta = reinterpret_cast<int4 *>(sm.rec + 2 * CS * 8);
    sm.full = reinterpret_cast<uint64_t *>(sm.meta + kStages);
    sm.red = reinterpret_cast<float *>(sm.full + kStages);

    if (tid == 0) {
        s_dead = 0;
        for (int s = 0; s < kStages; ++s)
            mbar_init(&sm.full[s], 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    __syncthreads();
    // every CTA of the cluster is resident before any distributed-shared write
    cluster_arrive();
    cluster_wait();

    const int nvalid = *p.nvalid;
    const int n = nvalid > cid ? (nvalid - cid + ncl - 1) / ncl : 0;  // same for the whole cluster
    if (n == 0)
        return;

    const __nv_bfloat16 *zs = static_cast<const __nv_bfloat16 *>(p.zs);
    const __nv_bfloat16 *zt = static_cast<const __nv_bfloat16 *>(p.zt);
    const uint64_t pol = evict_first_policy();

    // thread 0: stream row k of this cluster into stage k % kStages
    auto issue = [&](int k, int4 m) {
        const int s = k % kStages;
        sm.meta[s] = m;
        const size_t off = (size_t)m.y * (size_t)p.ld + (size_t)v0 * 8;
        const char *gs = reinterpret_cast<const char *>(zs + off);
        const char *gt = reinterpret_cast<const char *>(zt + off);
        unsigned char *ds = sm.stage + s * stage_bytes;
        mbar_arrive_expect_tx(&sm.full[s], 2u * my_bytes);
        for (uint32_t o = 0; o < my_bytes; o += kCopyChunk) {
            const uint32_t sz = min(kCopyChunk, my_bytes - o);
            bulk_g2s(ds + o, gs + o, sz, &sm.full[s], pol);
            bulk_g2s(ds + slice_bytes + o, gt + o, sz, &sm.full[s], pol);
        }
    };

    auto wait_full = [&](int k) {
        const int s = k % kStages;
        const uint32_t parity = (uint32_t)((k / kStages) & 1);
        if (*(volatile int *)&s_dead)
            return;
        for (uint32_t it = 0; it < kWaitLimit; ++it)
            if (mbar_try_wait(&sm.full[s], parity))
                return;
        s_dead = 1;
        set_status(p.status, TURNOPD_ERR_TIMEOUT);
    };

    // statistics of the resident slice of row k -> record into every CTA's slot k & 1
    auto stats = [&](int k) {
        const int s = k % kStages;
        const uint4 *vs = reinterpret_cast<const uint4 *>(sm.stage + s * stage_bytes);
        const uint4 *vt = reinterpret_cast<const uint4 *>(sm.stage + s * stage_bytes + slice_bytes);
        float ms = -INFINITY, xd = 0.f, mt = -INFINITY;
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
            const int q = tid + u * NT;
            if (q < my_vec) {
                float a[8], b[8];
                unpack8(vs[q], a);
                unpack8(vt[q], b);
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    if (a[e] > ms) {
                        ms = a[e];
                        xd = a[e] - b[e];
                    }
                    mt = fmaxf(mt, b[e]);
                }
            }
        }
        const float ns = -ms * kLog2e, nt = -mt * kLog2e;
        float ss = 0.f, aa = 0.f, st = 0.f;
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
            const int q = tid + u * NT;
            if (q < my_vec) {
                float a[8], b[8];
                unpack8(vs[q], a);
                unpack8(vt[q], b);
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const float es = ex2(fmaf(a[e], kLog2e, ns));
                    ss += es;
                    aa = fmaf(es, (a[e] - b[e]) - xd, aa);
                    st += ex2(fmaf(b[e], kLog2e, nt));
                }
            }
        }
        Student S = ms == -INFINITY ? student_empty() : Student{ms, ss, aa, xd};
        Teacher U = mt == -INFINITY ? teacher_empty() : Teacher{mt, st};
        S = warp_merge(S);
        U = warp_merge(U);
        if (lane == 0) {
            float *r = sm.red + warp * 8;
            r[0] = S.m, r[1] = S.s, r[2] = S.a, r[3] = S.d, r[4] = U.m, r[5] = U.s;
        }
        __syncthreads();
        if (warp == 0 && lane < CS) {
            Student A = Student{sm.red[0], sm.red[1], sm.red[2], sm.red[3]};
            Teacher B = Teacher{sm.red[4], sm.red[5]};
            for (int w2 = 1; w2 < NW; ++w2) {
                const float *r = sm.red + w2 * 8;
                A = student_merge(A, Student{r[0], r[1], r[2], r[3]});
                B = teacher_merge(B, Teacher{r[4], r[5]});
            }
            // sampled-token logits, from the CTA whose slice holds y
            float ys = 0.f, yt = 0.f;
            const int y = sm.meta[s].z;
            if (y >= 0 && y / 8 >= v0 && y / 8 < v0 + my_vec) {
                const int e = y - v0 * 8;
                ys = to_float(reinterpret_cast<const __nv_bfloat16 *>(vs)[e]);
                yt = to_float(reinterpret_cast<const __nv_bfloat16 *>(vt)[e]);
            }
            float *slot = sm.rec + ((k & 1) * CS + (int)rank) * 8;
            st_cluster(slot, (uint32_t)lane, make_float4(A.m, A.s, A.a, A.d));
            st_cluster(slot + 4, (uint32_t)lane, make_float4(B.m, B.s, ys, yt));
        }
    };

    // row constants of row k from the CS records (same order in every CTA)
    auto combine = [&](int k, float &ell) {
        const float *slot = sm.rec + (k & 1) * CS * 8;
        Student A = Student{slot[0], slot[1], slot[2], slot[3]};
        Teacher B = Teacher{slot[4], slot[5]};
#pragma unroll
        for (int c = 1; c < CS; ++c) {
            const float *r = slot + c * 8;
            A = student_merge(A, Student{r[0], r[1], r[2], r[3]});
            B = teacher_merge(B, Teacher{r[4], r[5]});
        }
        const RowConst rc = row_const(A, B);
        ell = rc.kl;
        const int y = sm.meta[k % kStages].z;
        if (y >= 0) {
            const int owner = (y / 8) / slice_vec;
            ell = (slot[owner * 8 + 6] - slot[owner * 8 + 7]) - rc.dl;
        }
        return rc;
    };

    auto grad = [&](int k, const RowConst &rc, float ell) {
        if (!p.grad)
            return;
        const int s = k % kStages;
        const int4 m = sm.meta[s];
        const uint4 *vs = reinterpret_cast<const uint4 *>(sm.stage + s * stage_bytes);
        const uint4 *vt = reinterpret_cast<const uint4 *>(sm.stage + s * stage_bytes + slice_bytes);
        const float wi = __int_as_float(m.w), wl = wi * ell;
        const float nl = -rc.lse_s * kLog2e, d = rc.d, cp = rc.cp;
        const int y = m.z;
        const size_t row_off = (size_t)m.y * (size_t)p.ld + (size_t)v0 * 8;
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
            const int q = tid + u * NT;
            if (q < my_vec) {
                float a[8], b[8], g[8];
                unpack8(vs[q], a);
                unpack8(vt[q], b);
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const float pv = ex2(fmaf(a[e], kLog2e, nl));
                    if (y < 0)
                        g[e] = wi * pv * (((a[e] - b[e]) - d) - cp);
                    else
                        g[e] = ((v0 + q) * 8 + e == y ? wl : 0.f) - wl * pv;
                }
                if (G32) {
                    float4 *dst = reinterpret_cast<float4 *>(static_cast<float *>(p.grad) + row_off +
                                                             (size_t)q * 8);
                    __stcs(dst, make_float4(g[0], g[1], g[2], g[3]));
                    __stcs(dst + 1, make_float4(g[4], g[5], g[6], g[7]));
                } else {
                    uint4 o;
                    o.x = pack_bf16x2(g[0], g[1]);
                    o.y = pack_bf16x2(g[2], g[3]);
                    o.z = pack_bf16x2(g[4], g[5]);
                    o.w = pack_bf16x2(g[6], g[7]);
                    __stcs(reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(p.grad) + row_off +
                                                     (size_t)q * 8),
                           o);
                }
            }
        }
    };

    // prologue: rows 0..2 in flight, statistics of row 0 exchanged
    if (tid == 0)
        for (int k = 0; k < kStages && k < n; ++k)
            issue(k, p.rows[cid + k * ncl]);
    wait_full(0);
    stats(0);
    cluster_arrive();
    cluster_wait();

    for (int k = 0; k < n; ++k) {
        int4 ahead = make_int4(0, 0, -1, 0);
        if (tid == 0 && k + kStages < n)
            ahead = p.rows[cid + (k + kStages) * ncl];  // consumed at the end of this iteration
        float ell;
        const RowConst rc = combine(k, ell);
        if (rank == 0 && tid == 0) {
            const int4 m = sm.meta[k % kStages];
            if (!isfinite(rc.lse_s) || !isfinite(rc.lse_t) || !isfinite(ell))
                set_status(p.status, TURNOPD_ERR_NONFINITE);
            p.token_loss[m.x] = ell;
            p.row_wl[cid + k * ncl] = (double)__int_as_float(m.w) * (double)ell;
        }
        if (k + 1 < n) {
            wait_full(k + 1);
            stats(k + 1);
        }
        cluster_arrive();
        grad(k, rc, ell);
        cluster_wait();
        __syncthreads();  // every thread is done with stage k % kStages
        if (tid == 0 && k + kStages < n) {
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            issue(k + kStages, ahead);
        }
    }

    // after a timeout, let this CTA's own copies land before the CTA exits
    if (tid == 0 && s_dead) {
        for (int k = max(0, n - kStages); k < n; ++k)
            for (uint32_t it = 0; it < kWaitLimit; ++it)
                if (mbar_try_wait(&sm.full[k % kStages], (uint32_t)((k / kStages) & 1)))
                    break;
    }
}

constexpr int kCS = 8;
constexpr int kNT = 256;
constexpr int kVPT = 10;
constexpr int64_t kMinVocab = 32768;  // below this the portable kernel is faster

size_t cluster_smem_bytes(int slice_vec)
{
    return (size_t)kStages * 2 * slice_vec * 16 + 2 * kCS * 8 * sizeof(float) +
           kStages * sizeof(int4) + kStages * sizeof(uint64_t) + (kNT / 32) * 8 * sizeof(float);
}

template <bool G32>
cudaError_t launch_t(const RowIn &p, int slice_vec, int nvec, size_t smem, cudaStream_t stream)
{
    auto kern = k_row_cluster<kCS, kNT, kVPT, G32>;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return e;
    static int grid_cache[64][2];
    static size_t smem_cache[64][2];
    const int gi = G32 ? 1 : 0;
    if (dev >= 64)
        return cudaErrorInvalidDevice;
    if (smem_cache[dev][gi] < smem) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess)
            return e;
        smem_cache[dev][gi] = smem;
        grid_cache[dev][gi] = 0;
    }
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kCS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.blockDim = dim3(kNT);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    if (grid_cache[dev][gi] == 0) {
        cfg.gridDim = dim3(kCS);
        int ncl = 0;
        e = cudaOccupancyMaxActiveClusters(&ncl, kern, &cfg);
        if (e != cudaSuccess)
            return e;
        if (ncl < 1)
            return cudaErrorInvalidConfiguration;
        grid_cache[dev][gi] = ncl;
    }
    cfg.gridDim = dim3(grid_cache[dev][gi] * kCS);
    return cudaLaunchKernelEx(&cfg, kern, p, slice_vec, nvec);
}

}  // namespace

cudaError_t launch_row_cluster(const RowIn &p, bool fp32_grad, cudaStream_t stream, bool *used)
{
    *used = false;
    auto al16 = [](const void *q) { return (reinterpret_cast<uintptr_t>(q) & 15u) == 0; };
    if (p.vocab < kMinVocab || p.vocab % 8 != 0 || p.ld % 8 != 0 || !al16(p.zs) || !al16(p.zt) ||
        (p.grad && !al16(p.grad)))
        return cudaSuccess;
    const int nvec = (int)(p.vocab / 8);
    const int slice_vec = (nvec + kCS - 1) / kCS;
    if (slice_vec > kVPT * kNT)
        return cudaSuccess;
    const size_t smem = cluster_smem_bytes(slice_vec);
    int dev = 0, optin = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return e;
    e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e != cudaSuccess)
        return e;
    // leave room for the kernel's static shared memory
    if (smem + 64 > (size_t)optin)
        return cudaSuccess;
    *used = true;
    return fp32_grad ? launch_t<true>(p, slice_vec, nvec, smem, stream)
                     : launch_t<false>(p, slice_vec, nvec, smem, stream);
}

}  // namespace turnopd
