// Fused LM heads + OPD loss (sm_103a): the student and teacher logits of the
// supervised tokens are produced tile by tile on the tensor cores and consumed
// in the epilogue, never stored.
//
//   forward   Z_s = H_s W_s^T (K = d_s), Z_t = H_t W_t^T (K = d_t) per 128-row x
//             256-vocab tile, accumulated in tensor memory (512 fp32 columns:
//             Z_s in [0,256), Z_t in [256,512)); the epilogue folds each tile
//             into per-row online statistics (max, sum exp, sum exp (z_s - z_t))
//             for both models over a group of vocabulary tiles;
//   merge     per row: LSE_s, LSE_t, KL = E_p[z_s - z_t] - (LSE_s - LSE_t);
//   backward  the same tiles are recomputed; the epilogue forms
//             G = w p_s ((z_s - z_t) - E_p[z_s - z_t]) = dL/dz_s and stores it in
//             bf16 (the gradient w.r.t. the logits, not the logits);
//   dH_s      = G W_s by a second tensor-core GEMM over the vocabulary.
//
// GEMM structure (persistent, one CTA per SM): warp 0 streams 128x64 A and
// 256x64 B bf16 tiles with TMA (128-byte swizzle) into a 4-stage ring, warp 1
// allocates tensor memory and issues tcgen05.mma (one thread), warps 2..9
// read the accumulator back (tcgen05.ld) for the epilogue.  Stage and
// accumulator hand-offs are mbarriers completed by TMA transaction counts and
// tcgen05.commit.  Every wait is bounded; on timeout the kernel records
// TURNOPD_ERR_TIMEOUT, keeps its hand-off sequence without waiting, and
// releases its tensor memory before it exits.

#include <cudaTypedefs.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.h"
#include "ptx.cuh"

namespace turnopd {
namespace {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2, B_BYTES = BN * BK * 2, STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int kEpiWarps = 8;
constexpr int kThreads = 32 * (2 + kEpiWarps);
constexpr uint32_t kLimit = 1u << 24;
constexpr int kTilesPerGroup = 10;  // vocabulary tiles one work unit folds into one partial

struct FusedArgs {
    int64_t vocab;
    int64_t vpad;          // G row length (vocab rounded up to BK)
    int d_s, d_t;
    const int4 *rows;      // compacted supervised rows {token, row, y, w bits}
    const int32_t *nvalid;
    int n_groups;          // vocabulary groups (units per M tile)
    float *part;           // [n_groups][2 halves][cap rows][8] partial statistics
    int64_t cap;           // row capacity of the gathered buffers
    const float *rowc;     // [cap][4]: lse_s * log2e - log2 |w|, E_p[z_s - z_t], sign w, -
    __nv_bfloat16 *G;      // [cap][vpad] backward output
    int32_t *status;
};

__device__ __forceinline__ bool wait_lim(uint64_t *bar, uint32_t parity, int32_t *status, int *dead)
{
    if (*(volatile int *)dead)
        return false;
    for (uint32_t i = 0; i < kLimit; ++i)
        if (mbar_try_wait(bar, parity))
            return true;
    *(volatile int *)dead = 1;
    set_status(status, TURNOPD_ERR_TIMEOUT);
    return false;
}

// Shared memory: ring of STAGES x (A tile | B tile), then barriers.
struct FusedSmem {
    uint8_t *a, *b;
    uint64_t *full, *empty, *accf, *acce;
    uint32_t *tslot;
};

__device__ __forceinline__ FusedSmem carve(uint8_t *raw)
{
    FusedSmem s;
    uint8_t *base = raw + ((1024 - (smem_u32(raw) & 1023)) & 1023);
    s.a = base;
    s.b = base + STAGES * A_BYTES;
    s.full = reinterpret_cast<uint64_t *>(s.b + STAGES * B_BYTES);
    s.empty = s.full + STAGES;
    s.accf = s.empty + STAGES;
    s.acce = s.accf + 1;
    s.tslot = reinterpret_cast<uint32_t *>(s.acce + 1);
    return s;
}

constexpr size_t kFusedSmem = STAGES * STAGE_BYTES + 1024 + 256;

// ----------------------------------------------------------------------------
// Forward statistics (MODE 0) / backward logit gradient (MODE 1).
// Work unit u: M tile (u % m_tiles), vocabulary group (u / m_tiles) of
// kTilesPerGroup 256-wide tiles.  Units of one group run side by side, so a
// group's W tiles are read from HBM about once and then served from L2.
template <int MODE>
__global__ void __launch_bounds__(kThreads, 1)
k_fused_lm(const __grid_constant__ CUtensorMap tHs, const __grid_constant__ CUtensorMap tWs,
           const __grid_constant__ CUtensorMap tHt, const __grid_constant__ CUtensorMap tWt, FusedArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ int s_dead;
    FusedSmem sm = carve(smem_raw);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int nvalid = *a.nvalid;
    const int m_tiles = (nvalid + BM - 1) / BM;
    const int n_tiles = (int)((a.vocab + BN - 1) / BN);
    const int units = m_tiles * a.n_groups;
    const int kb_s = a.d_s / BK, kb_t = a.d_t / BK, kb_tile = kb_s + kb_t;

    if (threadIdx.x == 0) {
        s_dead = 0;
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&sm.full[s], 1);
            mbar_init(&sm.empty[s], 1);
        }
        mbar_init(sm.accf, 1);
        mbar_init(sm.acce, kEpiWarps);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) {
        tmem_alloc(sm.tslot, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *sm.tslot;

    if (warp == 0 && lane == 0) {
        // ---------------- producer: k-blocks of every tile of every unit
        tma_prefetch_desc(&tHs);
        tma_prefetch_desc(&tWs);
        tma_prefetch_desc(&tHt);
        tma_prefetch_desc(&tWt);
        uint32_t it = 0;
        for (int u = blockIdx.x; u < units; u += gridDim.x) {
            const int mt = u % m_tiles, g = u / m_tiles;
            const int t0 = g * kTilesPerGroup, t1 = min(n_tiles, t0 + kTilesPerGroup);
            for (int nt = t0; nt < t1; ++nt) {
                for (int kb = 0; kb < kb_tile; ++kb, ++it) {
                    const int s = it % STAGES;
                    if (it >= STAGES)
                        wait_lim(&sm.empty[s], ((it / STAGES) - 1) & 1, a.status, &s_dead);
                    mbar_arrive_expect_tx(&sm.full[s], STAGE_BYTES);
                    if (kb < kb_s) {
                        tma_load_2d(sm.a + s * A_BYTES, &tHs, kb * BK, mt * BM, &sm.full[s]);
                        tma_load_2d(sm.b + s * B_BYTES, &tWs, kb * BK, nt * BN, &sm.full[s]);
                    } else {
                        tma_load_2d(sm.a + s * A_BYTES, &tHt, (kb - kb_s) * BK, mt * BM, &sm.full[s]);
                        tma_load_2d(sm.b + s * B_BYTES, &tWt, (kb - kb_s) * BK, nt * BN, &sm.full[s]);
                    }
                }
            }
        }
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer: Z_s into columns [0,256), Z_t into [256,512)
        constexpr uint32_t idesc = idesc_bf16_f32(BM, BN);
        uint32_t it = 0, tile = 0;
        for (int u = blockIdx.x; u < units; u += gridDim.x) {
            const int g = u / m_tiles;
            const int t0 = g * kTilesPerGroup, t1 = min(n_tiles, t0 + kTilesPerGroup);
            for (int nt = t0; nt < t1; ++nt, ++tile) {
                if (tile > 0)  // the epilogue has read the previous tile's accumulators
                    wait_lim(sm.acce, (tile - 1) & 1, a.status, &s_dead);
                tc_fence_after();
                for (int kb = 0; kb < kb_tile; ++kb, ++it) {
                    const int s = it % STAGES;
                    wait_lim(&sm.full[s], (it / STAGES) & 1, a.status, &s_dead);
                    tc_fence_after();
                    const bool teacher = kb >= kb_s;
                    const uint32_t d = tmem + (teacher ? 256u : 0u);
                    const int kk = teacher ? kb - kb_s : kb;
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k) {
                        const uint64_t ad = smem_desc_sw128(smem_u32(sm.a + s * A_BYTES) + k * 32);
                        const uint64_t bd = smem_desc_sw128(smem_u32(sm.b + s * B_BYTES) + k * 32);
                        tc_mma(d, ad, bd, idesc, kk > 0 || k > 0);
                    }
                    tc_commit(&sm.empty[s]);
                }
                tc_commit(sm.accf);
            }
        }
    } else if (warp >= 2) {
        // ---------------- epilogue: warp pair (q, half) owns rows q*32.. and 128 columns
        const int ew = warp - 2;
        const int q = warp % 4;             // tensor-memory lane quarter this warp may read
        const int half = ew / 4;            // columns [half*128, half*128 + 128) of the tile
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        uint32_t tile = 0;
        for (int u = blockIdx.x; u < units; u += gridDim.x) {
            const int mt = u % m_tiles, g = u / m_tiles;
            const int t0 = g * kTilesPerGroup, t1 = min(n_tiles, t0 + kTilesPerGroup);
            const int rloc = q * 32 + lane;
            const int row = mt * BM + rloc;
            const bool valid_row = row < nvalid;
            float ms = -INFINITY, ss = 0.f, sa = 0.f, mt_ = -INFINITY, st = 0.f;
            float nl = 0.f, cp = 0.f, sg = 1.f;
            if (MODE == 1 && valid_row) {
                const float4 c = reinterpret_cast<const float4 *>(a.rowc)[row];
                nl = c.x, cp = c.y, sg = c.z;
            }
            for (int nt = t0; nt < t1; ++nt, ++tile) {
                wait_lim(sm.accf, tile & 1, a.status, &s_dead);
                tc_fence_after();
#pragma unroll 1
                for (int ch = 0; ch < 4; ++ch) {
                    const int c0 = half * 128 + ch * 32;
                    float zs[32], zt[32];
                    tmem_ld32(tmem + lane_off + (uint32_t)c0, zs);
                    tmem_ld32(tmem + lane_off + 256u + (uint32_t)c0, zt);
                    tmem_ld_wait();
                    const int64_t v0 = (int64_t)nt * BN + c0;
                    if (MODE == 0) {
                        // online statistics over the in-vocabulary columns
                        float cmx = -INFINITY, cmt = -INFINITY;
#pragma unroll
                        for (int j = 0; j < 32; ++j) {
                            if (v0 + j < a.vocab) {
                                cmx = fmaxf(cmx, zs[j]);
                                cmt = fmaxf(cmt, zt[j]);
                            }
                        }
                        if (cmx > ms) {
                            const float f = ex2((ms - cmx) * kLog2e);
                            ss *= f;
                            sa *= f;
                            ms = cmx;
                        }
                        if (cmt > mt_) {
                            st *= ex2((mt_ - cmt) * kLog2e);
                            mt_ = cmt;
                        }
                        const float ns = -ms * kLog2e, ntt = -mt_ * kLog2e;
#pragma unroll
                        for (int j = 0; j < 32; ++j) {
                            if (v0 + j < a.vocab) {
                                const float e = ex2(fmaf(zs[j], kLog2e, ns));
                                ss += e;
                                sa = fmaf(e, zs[j] - zt[j], sa);
                                st += ex2(fmaf(zt[j], kLog2e, ntt));
                            }
                        }
                    } else if (valid_row && v0 < a.vpad) {
                        // G = w p ((z_s - z_t) - E_p[z_s - z_t]); zero beyond the vocabulary
                        uint32_t pk[16];
#pragma unroll
                        for (int j = 0; j < 32; j += 2) {
                            float g0 = 0.f, g1 = 0.f;
                            if (v0 + j < a.vocab)
                                g0 = sg * ex2(fmaf(zs[j], kLog2e, -nl)) * ((zs[j] - zt[j]) - cp);
                            if (v0 + j + 1 < a.vocab)
                                g1 = sg * ex2(fmaf(zs[j + 1], kLog2e, -nl)) * ((zs[j + 1] - zt[j + 1]) - cp);
                            pk[j / 2] = pack_bf16x2(g0, g1);
                        }
                        uint4 *dst = reinterpret_cast<uint4 *>(a.G + (size_t)row * a.vpad + v0);
                        // vpad is a multiple of BK = 64, so a 32-column chunk is either
                        // wholly inside [0, vpad) or wholly outside it
#pragma unroll
                        for (int j = 0; j < 4; ++j)
                            dst[j] = make_uint4(pk[4 * j], pk[4 * j + 1], pk[4 * j + 2], pk[4 * j + 3]);
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(sm.acce);
            }
            if (MODE == 0 && valid_row) {
                float *pp = a.part + (((size_t)g * 2 + half) * a.cap + row) * 8;
                reinterpret_cast<float4 *>(pp)[0] = make_float4(ms, ss, sa, mt_);
                reinterpret_cast<float4 *>(pp)[1] = make_float4(st, 0.f, 0.f, 0.f);
            }
        }
    }

    // drain (after a timeout, let in-flight tensor-core work finish) and release
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) {
        if (lane == 0 && *(volatile int *)&s_dead) {
            // one more bounded wait on the accumulator barrier's next phase
            for (uint32_t i = 0; i < kLimit; ++i)
                if (mbar_try_wait(sm.accf, 0) || mbar_try_wait(sm.accf, 1))
                    break;
        }
        __syncwarp();
        tmem_dealloc(tmem, 512);
    }
}

// ----------------------------------------------------------------------------
// dH = G W_s: A = G [rows, vpad] (K-major), B = W_s^T [d_s, vpad] (K-major).
// Output tile 128 x 256 fp32 in tensor memory; rows scattered to their tokens.
__global__ void __launch_bounds__(kThreads, 1)
k_fused_dh(const __grid_constant__ CUtensorMap tG, const __grid_constant__ CUtensorMap tWT, const int4 *rows,
           const int32_t *nvalid_p, int d_s, int64_t vpad, float *dh_out, int32_t *status)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ int s_dead;
    FusedSmem sm = carve(smem_raw);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int nvalid = *nvalid_p;
    const int m_tiles = (nvalid + BM - 1) / BM;
    const int n_tiles = d_s / BN;
    const int tiles = m_tiles * n_tiles;
    const int kbs = (int)(vpad / BK);

    if (threadIdx.x == 0) {
        s_dead = 0;
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&sm.full[s], 1);
            mbar_init(&sm.empty[s], 1);
        }
        mbar_init(sm.accf, 1);
        mbar_init(sm.acce, kEpiWarps);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) {
        tmem_alloc(sm.tslot, 256);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *sm.tslot;

    // tile order: N-tile fastest, so CTAs running together share the G rows (A)
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tG);
        tma_prefetch_desc(&tWT);
        uint32_t it = 0;
        for (int t = blockIdx.x; t < tiles; t += gridDim.x) {
            const int mt = t / n_tiles, nt = t % n_tiles;
            for (int kb = 0; kb < kbs; ++kb, ++it) {
                const int s = it % STAGES;
                if (it >= STAGES)
                    wait_lim(&sm.empty[s], ((it / STAGES) - 1) & 1, status, &s_dead);
                mbar_arrive_expect_tx(&sm.full[s], STAGE_BYTES);
                tma_load_2d(sm.a + s * A_BYTES, &tG, kb * BK, mt * BM, &sm.full[s]);
                tma_load_2d(sm.b + s * B_BYTES, &tWT, kb * BK, nt * BN, &sm.full[s]);
            }
        }
    } else if (warp == 1 && lane == 0) {
        constexpr uint32_t idesc = idesc_bf16_f32(BM, BN);
        uint32_t it = 0, tile = 0;
        for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++tile) {
            if (tile > 0)
                wait_lim(sm.acce, (tile - 1) & 1, status, &s_dead);
            tc_fence_after();
            for (int kb = 0; kb < kbs; ++kb, ++it) {
                const int s = it % STAGES;
                wait_lim(&sm.full[s], (it / STAGES) & 1, status, &s_dead);
                tc_fence_after();
#pragma unroll
                for (int k = 0; k < BK / 16; ++k) {
                    const uint64_t ad = smem_desc_sw128(smem_u32(sm.a + s * A_BYTES) + k * 32);
                    const uint64_t bd = smem_desc_sw128(smem_u32(sm.b + s * B_BYTES) + k * 32);
                    tc_mma(tmem, ad, bd, idesc, kb > 0 || k > 0);
                }
                tc_commit(&sm.empty[s]);
            }
            tc_commit(sm.accf);
        }
    } else if (warp >= 2) {
        const int ew = warp - 2, q = warp % 4, half = ew / 4;
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        uint32_t tile = 0;
        for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++tile) {
            const int mt = t / n_tiles, nt = t % n_tiles;
            const int row = mt * BM + q * 32 + lane;
            wait_lim(sm.accf, tile & 1, status, &s_dead);
            tc_fence_after();
            const bool valid = row < nvalid;
            const int token = valid ? rows[row].x : 0;
#pragma unroll 1
            for (int ch = 0; ch < 4; ++ch) {
                const int c0 = half * 128 + ch * 32;
                float v[32];
                tmem_ld32(tmem + lane_off + (uint32_t)c0, v);
                tmem_ld_wait();
                if (valid) {
                    float4 *dst = reinterpret_cast<float4 *>(dh_out + (size_t)token * d_s + nt * BN + c0);
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        dst[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0)
                mbar_arrive(sm.acce);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) {
        if (lane == 0 && *(volatile int *)&s_dead) {
            for (uint32_t i = 0; i < kLimit; ++i)
                if (mbar_try_wait(sm.accf, 0) || mbar_try_wait(sm.accf, 1))
                    break;
        }
        __syncwarp();
        tmem_dealloc(tmem, 256);
    }
}

// ----------------------------------------------------------------------------
// Gather the supervised hidden rows: out[j] = h[token of row j] (16-byte copies).
__global__ void k_gather_rows(const int4 *__restrict__ rows, const int32_t *__restrict__ nvalid,
                              const uint4 *__restrict__ h, int vec_per_row, uint4 *__restrict__ out)
{
    const int n = *nvalid;
    for (int j = blockIdx.x; j < n; j += gridDim.x) {
        const int64_t tok = rows[j].x;
        const uint4 *src = h + tok * vec_per_row;
        uint4 *dst = out + (int64_t)j * vec_per_row;
        for (int c = threadIdx.x; c < vec_per_row; c += blockDim.x)
            dst[c] = src[c];
    }
}

// W [V, d] -> W^T [d, vpad], zero for columns v >= V (32 x 32 tiles).
__global__ void k_transpose_pad(const __nv_bfloat16 *__restrict__ W, int64_t V, int d, int64_t vpad,
                                __nv_bfloat16 *__restrict__ WT)
{
    __shared__ __nv_bfloat16 tile[32][34];
    const int64_t v0 = (int64_t)blockIdx.x * 32;
    const int c0 = blockIdx.y * 32;
    for (int r = threadIdx.y; r < 32; r += blockDim.y) {
        const int64_t v = v0 + r;
        const int c = c0 + threadIdx.x;
        tile[r][threadIdx.x] = (v < V && c < d) ? W[v * d + c] : __float2bfloat16(0.f);
    }
    __syncthreads();
    for (int r = threadIdx.y; r < 32; r += blockDim.y) {
        const int c = c0 + r;
        const int64_t v = v0 + threadIdx.x;
        if (c < d && v < vpad)
            WT[(int64_t)c * vpad + v] = tile[threadIdx.x][r];
    }
}

// Per supervised row: merge the vocabulary-group partials into LSE_s, LSE_t,
// KL; write l, w*l and the backward constants.
__global__ void k_fused_merge(const int4 *__restrict__ rows, const int32_t *__restrict__ nvalid,
                              const float *__restrict__ part, int n_groups, int64_t cap,
                              float *__restrict__ token_loss, double *__restrict__ row_wl,
                              float *__restrict__ rowc, int32_t *status)
{
    const int n = *nvalid;
    for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < n; j += gridDim.x * blockDim.x) {
        Student S = student_empty();
        Teacher T = teacher_empty();
        for (int gh = 0; gh < 2 * n_groups; ++gh) {
            const float *pp = part + ((size_t)gh * cap + j) * 8;
            const float4 x = reinterpret_cast<const float4 *>(pp)[0];
            const float4 y = reinterpret_cast<const float4 *>(pp)[1];
            if (x.x != -INFINITY)
                S = student_merge(S, Student{x.x, x.y, x.z, 0.f});
            if (x.w != -INFINITY)
                T = teacher_merge(T, Teacher{x.w, y.x});
        }
        const RowConst rc = row_const(S, T);
        const int4 m = rows[j];
        const float w = __int_as_float(m.w);
        const float ell = rc.kl;
        if (!isfinite(rc.lse_s) || !isfinite(rc.lse_t) || !isfinite(ell))
            set_status(status, TURNOPD_ERR_NONFINITE);
        token_loss[m.x] = ell;
        row_wl[j] = (double)w * (double)ell;
        // p |w| = 2^(z_s log2e - nl): nl = LSE_s log2e - log2 |w|
        reinterpret_cast<float4 *>(rowc)[j] =
            make_float4(rc.lse_s * kLog2e - log2f(fabsf(w)), rc.d + rc.cp, w < 0.f ? -1.f : 1.f, 0.f);
    }
}

// ---------------------------------------------------------------- host side

PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        cudaDriverEntryPointQueryResult q;
        void *p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return nullptr;
        fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

bool make_map(CUtensorMap *m, const void *base, int64_t rows, int64_t cols, int box_rows)
{
    auto fn = encode_fn();
    if (!fn)
        return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    cuuint32_t box[2] = {BK, (cuuint32_t)box_rows};
    cuuint32_t es[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct FusedLayout {
    int4 *rows;
    int32_t *blk_count, *nvalid;
    double *row_wl;
    __nv_bfloat16 *hs, *ht, *G, *wsT;
    float *part, *rowc;
    size_t bytes;
};

FusedLayout fused_layout(void *ws, int64_t T, int64_t V, int64_t d_s, int64_t d_t, int n_groups)
{
    const int64_t vpad = (V + BK - 1) / BK * BK;
    const int64_t cap = (T + BM - 1) / BM * BM;
    const int64_t nblk = (T + kCompactBlock - 1) / kCompactBlock;
    char *p = static_cast<char *>(ws);
    size_t off = 0;
    auto take = [&](size_t n) {
        char *q = p ? p + off : nullptr;
        off += align256(n);
        return q;
    };
    FusedLayout L;
    L.rows = reinterpret_cast<int4 *>(take(sizeof(int4) * (size_t)T));
    L.blk_count = reinterpret_cast<int32_t *>(take(sizeof(int32_t) * (size_t)(nblk + 1)));
    L.nvalid = reinterpret_cast<int32_t *>(take(sizeof(int32_t)));
    L.row_wl = reinterpret_cast<double *>(take(sizeof(double) * (size_t)T));
    L.hs = reinterpret_cast<__nv_bfloat16 *>(take(2 * (size_t)cap * d_s));
    L.ht = reinterpret_cast<__nv_bfloat16 *>(take(2 * (size_t)cap * d_t));
    L.part = reinterpret_cast<float *>(take(sizeof(float) * 8 * 2 * (size_t)n_groups * cap));
    L.rowc = reinterpret_cast<float *>(take(sizeof(float) * 4 * (size_t)cap));
    L.G = reinterpret_cast<__nv_bfloat16 *>(take(2 * (size_t)cap * vpad));
    L.wsT = reinterpret_cast<__nv_bfloat16 *>(take(2 * (size_t)d_s * vpad));
    L.bytes = off + 256;
    return L;
}

int groups_for(int64_t V) { return (int)(((V + BN - 1) / BN + kTilesPerGroup - 1) / kTilesPerGroup); }

}  // namespace

size_t fused_workspace_bytes(int64_t T, int64_t V, int64_t d_s, int64_t d_t)
{
    return fused_layout(nullptr, T, V, d_s, d_t, groups_for(V)).bytes;
}

cudaError_t launch_fused(const FusedCall &c, cudaStream_t stream)
{
    const int n_groups = groups_for(c.vocab);
    FusedLayout L = fused_layout(c.workspace, c.T, c.vocab, c.d_s, c.d_t, n_groups);
    const int64_t vpad = (c.vocab + BK - 1) / BK * BK;
    const int64_t cap = (c.T + BM - 1) / BM * BM;
    const int sms = device_sm_count();

    // supervised rows (the compaction of the loss path), then the gathered hidden rows
    LossArgs la{};
    la.mask = c.mask;
    la.w = c.w;
    la.T = c.T;
    la.num_rows = c.T;
    la.vocab = c.vocab;
    la.mode = TURNOPD_FULL_VOCAB;
    la.token_loss = c.token_loss;
    la.status = c.status;
    cudaError_t e = launch_compaction(la, L.rows, L.blk_count, L.nvalid, stream);
    if (e != cudaSuccess)
        return e;
    k_gather_rows<<<sms * 4, 256, 0, stream>>>(L.rows, L.nvalid, static_cast<const uint4 *>(c.h_s), c.d_s / 8,
                                               reinterpret_cast<uint4 *>(L.hs));
    k_gather_rows<<<sms * 4, 256, 0, stream>>>(L.rows, L.nvalid, static_cast<const uint4 *>(c.h_t), c.d_t / 8,
                                               reinterpret_cast<uint4 *>(L.ht));
    {
        dim3 grid((unsigned)((vpad + 31) / 32), (unsigned)((c.d_s + 31) / 32));
        k_transpose_pad<<<grid, dim3(32, 8), 0, stream>>>(static_cast<const __nv_bfloat16 *>(c.W_s), c.vocab,
                                                          (int)c.d_s, vpad, L.wsT);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess)
        return e;

    alignas(64) CUtensorMap tHs, tWs, tHt, tWt, tG, tWT;
    if (!make_map(&tHs, L.hs, cap, c.d_s, BM) || !make_map(&tWs, c.W_s, c.vocab, c.d_s, BN) ||
        !make_map(&tHt, L.ht, cap, c.d_t, BM) || !make_map(&tWt, c.W_t, c.vocab, c.d_t, BN) ||
        !make_map(&tG, L.G, cap, vpad, BM) || !make_map(&tWT, L.wsT, c.d_s, vpad, BN))
        return cudaErrorInvalidValue;

    static bool attr_done = false;
    if (!attr_done) {
        e = cudaFuncSetAttribute(k_fused_lm<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kFusedSmem);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(k_fused_lm<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kFusedSmem);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(k_fused_dh, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kFusedSmem);
        if (e != cudaSuccess)
            return e;
        attr_done = true;
    }

    FusedArgs fa;
    fa.vocab = c.vocab;
    fa.vpad = vpad;
    fa.d_s = (int)c.d_s;
    fa.d_t = (int)c.d_t;
    fa.rows = L.rows;
    fa.nvalid = L.nvalid;
    fa.n_groups = n_groups;
    fa.part = L.part;
    fa.cap = cap;
    fa.rowc = L.rowc;
    fa.G = L.G;
    fa.status = c.status;

    k_fused_lm<0><<<sms, kThreads, kFusedSmem, stream>>>(tHs, tWs, tHt, tWt, fa);
    k_fused_merge<<<(int)((cap + 255) / 256), 256, 0, stream>>>(L.rows, L.nvalid, L.part, n_groups, cap,
                                                               c.token_loss, L.row_wl, L.rowc, c.status);
    e = cudaGetLastError();
    if (e != cudaSuccess)
        return e;
    if (c.dh_s) {
        k_fused_lm<1><<<sms, kThreads, kFusedSmem, stream>>>(tHs, tWs, tHt, tWt, fa);
        launch_zero_masked_f32(c.mask, c.T, (int64_t)c.d_s, c.dh_s, stream);
        k_fused_dh<<<sms, kThreads, kFusedSmem, stream>>>(tG, tWT, L.rows, L.nvalid, (int)c.d_s, vpad, c.dh_s,
                                                         c.status);
    }
    launch_loss_sum(L.row_wl, L.nvalid, c.loss, c.status, stream);
    return cudaGetLastError();
}

}  // namespace turnopd
