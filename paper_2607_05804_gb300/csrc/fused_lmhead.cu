// Fused LM heads + OPD loss (sm_103a): the student and teacher logits of the
// supervised tokens are produced tile by tile on the tensor cores and consumed
// in the epilogue, never stored.
//
//   forward   Z_t = H_t W_t^T (K = d_t), then Z_s = H_s W_s^T (K = d_s), per
//             256-row x 256-vocab tile, accumulated in tensor memory (512 fp32
//             columns per CTA: Z_t in [0,256), Z_s in [256,512)); the epilogue
//             folds each tile into per-row online statistics (max, sum exp,
//             sum exp (z_s - z_t)) for both models over a group of tiles;
//   merge     per row: LSE_s, LSE_t, KL = E_p[z_s - z_t] - (LSE_s - LSE_t);
//   backward  the same tiles are recomputed; the epilogue forms
//             G = w p_s ((z_s - z_t) - E_p[z_s - z_t]) = dL/dz_s and stores it in
//             bf16 (the gradient w.r.t. the logits, not the logits);
//   dH_s      = G W_s by a second tensor-core GEMM over the vocabulary, W_s read
//             in place as an MN-major operand.
//
// GEMM structure: persistent 2-CTA clusters, one CTA per SM.  A tile is
// computed by the pair with cta_group::2 instructions (M = 256, N = 256): each
// CTA stages its own 128 rows of A and 128 rows of B per 64-deep k-block, so a
// pair reads 2/3 of the operand bytes two independent 128 x 256 tiles would.
// In each CTA warp 0 streams the operand tiles with TMA (128-byte swizzle)
// into a 5-stage ring, every copy counted on the even CTA's barrier; warp 1
// allocates tensor memory, and in the even CTA one thread issues tcgen05.mma
// and multicasts its commits to both CTAs; warps 2..17 read this CTA's 128
// accumulator rows back (tcgen05.ld) for the epilogue.  The two halves of the
// accumulator are released separately: the epilogue copies Z_t of tile j into
// registers while Z_s of tile j is computed, and reads Z_s of tile j while Z_t
// of tile j+1 is computed.  The backward epilogue stages each warp's 32 x 64
// block of G in shared memory (128-byte swizzle) and writes it with a TMA
// store, so G leaves the SM in whole 128-byte rows.  Every wait is bounded; on timeout the kernel
// records TURNOPD_ERR_TIMEOUT, keeps its hand-off sequence without waiting,
// drains its in-flight copies and tensor-core work with bounded waits, and
// releases its tensor memory before it exits.

#include <cudaTypedefs.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.h"
#include "ptx.cuh"

namespace turnopd {
namespace {

constexpr int BM = 128;             // accumulator rows per CTA
constexpr int BMP = 2 * BM;         // rows per pair tile
constexpr int BN = 256;             // columns per pair tile
constexpr int BNH = BN / 2;         // B rows staged per CTA
// Operand ring depth: 5 x 32 KB plus the 64 KB G staging buffer fills the
// 227 KB of shared memory a CTA may use (measured: 4 and 6 stages, the
// latter with direct G stores, are both slower).
#ifndef TURNOPD_FUSED_STAGES
#define TURNOPD_FUSED_STAGES 5
#endif
// L2 prefetch distance of the B operand in k-blocks (0: none).  Measured on
// GB300 it slows the GEMMs (the extra tensor requests compete with the ring's
// own copies), so it is off.
#ifndef TURNOPD_FUSED_PF
#define TURNOPD_FUSED_PF 0
#endif
constexpr int BK = 64, STAGES = TURNOPD_FUSED_STAGES;
constexpr int kPrefetch = TURNOPD_FUSED_PF;   // k-blocks of B brought into L2 ahead of the ring
constexpr int A_BYTES = BM * BK * 2, B_BYTES = BNH * BK * 2, STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int kEpiWarps = 16;                    // 4 per tensor-memory lane quarter
constexpr int kColQuarters = kEpiWarps / 4;      // column slices of a tile
constexpr int kEpiCols = BN / kColQuarters;      // 64 columns per epilogue thread
constexpr int kThreads = 32 * (2 + kEpiWarps);
constexpr uint32_t kLimit = 1u << 24;
constexpr int kTilesPerGroup = 10;  // vocabulary tiles one work unit folds into one partial
constexpr uint32_t kColT = 0, kColS = 256;  // tensor-memory columns of Z_t and Z_s
constexpr uint16_t kPairMask = 0x3;

struct FusedArgs {
    int64_t vocab;
    int64_t vpad;          // G row length (vocab rounded up to BK)
    int d_s, d_t;
    const int4 *rows;      // compacted supervised rows {token, row, y, w bits}
    const int32_t *nvalid;
    int n_groups;          // vocabulary groups (units per M tile)
    float *part;           // [n_groups][kColQuarters][cap rows][8] partial statistics
    int64_t cap;           // row capacity of the gathered buffers (multiple of BMP)
    const float *rowc;     // [cap][4]: lse_s * log2e - log2 |w|, E_p[z_s - z_t], sign w, -
    __nv_bfloat16 *G;      // [cap][vpad] backward output
    int32_t *status;
};

// The phase test comes first: the issuing thread's critical path holds no
// other shared-memory access (a load of the timeout flag on every k-block
// costs the tensor pipe about a third of its throughput).
__device__ __forceinline__ bool wait_lim(uint64_t *bar, uint32_t parity, int32_t *status, int *dead,
                                         bool cluster_scope = false)
{
    if (cluster_scope ? mbar_try_wait_cluster(bar, parity) : mbar_try_wait(bar, parity))
        return true;
    if (*(volatile int *)dead)
        return false;
    for (uint32_t i = 0; i < kLimit; ++i)
        if (cluster_scope ? mbar_try_wait_cluster(bar, parity) : mbar_try_wait(bar, parity))
            return true;
    *(volatile int *)dead = 1;
    set_status(status, TURNOPD_ERR_TIMEOUT);
    return false;
}

// Bounded wait used while draining at exit (also after a timeout).
__device__ __forceinline__ void wait_drain(uint64_t *bar, uint32_t parity)
{
    for (uint32_t i = 0; i < kLimit; ++i)
        if (mbar_try_wait_cluster(bar, parity))
            return;
}

// Shared memory: ring of STAGES x (A tile | B half tile), then barriers.  The
// layout is identical in both CTAs of a pair (the tensor-core instructions
// address the peer's operands at the issuing CTA's offsets).
struct FusedSmem {
    uint8_t *a, *b;
    uint8_t *stg;               // backward: per-epilogue-warp 32 x 64 bf16 G staging (4 KB each)
    uint64_t *full, *empty;
    uint64_t *acc_t, *acc_s;    // tensor core -> epilogue: Z_t / Z_s of a tile complete
    uint64_t *free_t, *free_s;  // epilogue (both CTAs) -> tensor core: columns read
    uint64_t *drain;
    uint32_t *tslot;
};

__device__ __forceinline__ FusedSmem carve(uint8_t *raw, int b_region, int stg_bytes)
{
    FusedSmem s;
    uint8_t *base = raw + ((1024 - (smem_u32(raw) & 1023)) & 1023);
    s.a = base;
    s.b = base + STAGES * A_BYTES;
    s.stg = s.b + b_region;
    s.full = reinterpret_cast<uint64_t *>(s.stg + stg_bytes);
    s.empty = s.full + STAGES;
    s.acc_t = s.empty + STAGES;
    s.acc_s = s.acc_t + 1;
    s.free_t = s.acc_s + 1;
    s.free_s = s.free_t + 1;
    s.drain = s.free_s + 1;
    s.tslot = reinterpret_cast<uint32_t *>(s.drain + 1);
    return s;
}

constexpr int kLmBRegion = STAGES * B_BYTES;
constexpr int kStgWarpBytes = 32 * kEpiCols * 2;             // 32 rows x 128 B
constexpr int kStgBytes = kEpiWarps * kStgWarpBytes;          // 64 KB
// The dH kernel reads B as an MN-major operand; 16 KB of slack after the ring
// keeps every address its descriptors can form inside the allocation.
constexpr int kDhBRegion = STAGES * B_BYTES + 16384;
constexpr size_t kFusedSmem = STAGES * A_BYTES + kLmBRegion + kStgBytes + 1024 + 256;
static_assert(kFusedSmem <= 232448, "shared memory per CTA");
constexpr size_t kDhSmem = STAGES * A_BYTES + kDhBRegion + 1024 + 256;
static_assert(kDhSmem <= 232448, "shared memory per CTA");

__device__ __forceinline__ void init_barriers(const FusedSmem &sm)
{
    for (int s = 0; s < STAGES; ++s) {
        mbar_init(&sm.full[s], 1);
        mbar_init(&sm.empty[s], 1);
    }
    mbar_init(sm.acc_t, 1);
    mbar_init(sm.acc_s, 1);
    mbar_init(sm.free_t, 2 * kEpiWarps);
    mbar_init(sm.free_s, 2 * kEpiWarps);
    mbar_init(sm.drain, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Common prologue: barriers, tensor memory for the pair, cluster-wide visibility.
__device__ __forceinline__ uint32_t pair_prologue(const FusedSmem &sm, int *s_dead, uint32_t ncols)
{
    const int warp = threadIdx.x / 32;
    if (threadIdx.x == 0) {
        *s_dead = 0;
        init_barriers(sm);
    }
    if (warp == 1) {
        tmem_alloc_pair(sm.tslot, ncols);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();
    tc_fence_after();
    return *sm.tslot;
}

// Producer exit (both CTAs): wait (bounded) until the tensor core has released
// the last copy of every stage, so no multicast commit is still on its way to
// this CTA's barriers; the even CTA also waits for its full barriers, which
// count the copies of both CTAs.
__device__ __forceinline__ void drain_producer(const FusedSmem &sm, uint32_t issued, uint32_t rank)
{
    const uint32_t first = issued > STAGES ? issued - STAGES : 0;
    for (uint32_t j = first; j < issued; ++j) {
        if (rank == 0)
            wait_drain(&sm.full[j % STAGES], (j / STAGES) & 1);
        wait_drain(&sm.empty[j % STAGES], (j / STAGES) & 1);
    }
}

// Epilogue -> tensor core: this warp has finished reading a half of the accumulator.
__device__ __forceinline__ void release_cols(uint32_t bar_leader, int lane)
{
    tc_fence_before();
    __syncwarp();
    if (lane == 0)
        mbar_arrive_cluster(bar_leader);
}

// Common epilogue of the kernels: every tcgen05 operation of the pair is
// complete (drain barrier in both CTAs) before tensor memory is released.
__device__ __forceinline__ void pair_epilogue(const FusedSmem &sm, uint32_t tmem, uint32_t ncols, uint32_t rank)
{
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    if (warp == 1 && lane == 0) {
        if (rank == 0)
            tc_commit_pair(sm.drain, kPairMask);
        wait_drain(sm.drain, 0);
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();
    tc_fence_after();
    if (warp == 1)
        tmem_dealloc_pair(tmem, ncols);
}

// Work unit u -> (pair M tile, vocabulary group).  The M tiles are cut into
// blocks of at most kMBlock; the units of a block are enumerated group-major,
// so the pairs running side by side share the H rows of one block and the W
// tiles of a few groups: a working set of about (kMBlock + pairs / kMBlock)
// 4.7 MB operand panels, which stays in L2.
constexpr int kMBlock = 16;
__device__ __forceinline__ void unit_coords(int u, int m_tiles, int n_groups, int *mt, int *g)
{
    const int nb = (m_tiles + kMBlock - 1) / kMBlock;
    const int mb = (m_tiles + nb - 1) / nb;          // block height (last block may be shorter)
    const int b = u / (mb * n_groups);
    const int rest = u - b * mb * n_groups;
    const int h = min(mb, m_tiles - b * mb);
    *g = rest / h;
    *mt = b * mb + rest % h;
}

// ----------------------------------------------------------------------------
// Forward statistics (MODE 0) / backward logit gradient (MODE 1).
// Work unit: one pair M tile x one vocabulary group of kTilesPerGroup
// 256-wide tiles, folded into one partial per row.
template <int MODE>
__global__ void __launch_bounds__(kThreads, 1)
k_fused_lm(const __grid_constant__ CUtensorMap tHs, const __grid_constant__ CUtensorMap tWs,
           const __grid_constant__ CUtensorMap tHt, const __grid_constant__ CUtensorMap tWt,
           const __grid_constant__ CUtensorMap tGst, FusedArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ int s_dead;
    FusedSmem sm = carve(smem_raw, kLmBRegion, kStgBytes);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const uint32_t rank = cluster_ctarank();
    const int pair = (int)cluster_id(), n_pairs = (int)cluster_count();
    const int nvalid = *a.nvalid;
    const int m_tiles = (nvalid + BMP - 1) / BMP;
    const int n_tiles = (int)((a.vocab + BN - 1) / BN);
    const int units = m_tiles * a.n_groups;
    const int kb_s = a.d_s / BK, kb_t = a.d_t / BK;
    const uint32_t tmem = pair_prologue(sm, &s_dead, 512);

    if (warp == 0 && lane == 0) {
        // ---------------- producer: per tile the teacher k-blocks, then the student's
        tma_prefetch_desc(&tHs);
        tma_prefetch_desc(&tWs);
        tma_prefetch_desc(&tHt);
        tma_prefetch_desc(&tWt);
        const uint32_t full0 = mapa(smem_u32(sm.full), 0);
        const int kb_tile = kb_t + kb_s;
        uint32_t it = 0;
        for (int u = pair; u < units; u += n_pairs) {
            int mt, g;
            unit_coords(u, m_tiles, a.n_groups, &mt, &g);
            const int t0 = g * kTilesPerGroup, t1 = min(n_tiles, t0 + kTilesPerGroup);
            const int ya = mt * BMP + (int)rank * BM;
            const int n_pos = (t1 - t0) * kb_tile;   // (tile, k-block) positions of this unit
            // L2 prefetch of this CTA's B rows at unit position p
            auto prefetch_b = [&](int p) {
                if (kPrefetch == 0 || p >= n_pos)
                    return;
                const int nt2 = t0 + p / kb_tile, kb2 = p % kb_tile;
                const int yb2 = nt2 * BN + (int)rank * BNH;
                if (kb2 < kb_t)
                    tma_prefetch_l2_2d(&tWt, kb2 * BK, yb2);
                else
                    tma_prefetch_l2_2d(&tWs, (kb2 - kb_t) * BK, yb2);
            };
            for (int p = 0; p < kPrefetch; ++p)
                prefetch_b(p);
            for (int nt = t0; nt < t1; ++nt) {
                const int yb = nt * BN + (int)rank * BNH;
                for (int kb = 0; kb < kb_tile; ++kb, ++it) {
                    prefetch_b((nt - t0) * kb_tile + kb + kPrefetch);
                    const int s = it % STAGES;
                    if (it >= STAGES)
                        wait_lim(&sm.empty[s], ((it / STAGES) - 1) & 1, a.status, &s_dead);
                    if (rank == 0)
                        mbar_arrive_expect_tx(&sm.full[s], 2 * STAGE_BYTES);
                    const uint32_t fb = full0 + (uint32_t)s * 8u;
                    if (kb < kb_t) {
                        tma_load_2d_pair(sm.a + s * A_BYTES, &tHt, kb * BK, ya, fb);
                        tma_load_2d_pair(sm.b + s * B_BYTES, &tWt, kb * BK, yb, fb);
                    } else {
                        tma_load_2d_pair(sm.a + s * A_BYTES, &tHs, (kb - kb_t) * BK, ya, fb);
                        tma_load_2d_pair(sm.b + s * B_BYTES, &tWs, (kb - kb_t) * BK, yb, fb);
                    }
                }
            }
        }
        drain_producer(sm, it, rank);
    } else if (warp == 1 && lane == 0 && rank == 0) {
        // ---------------- MMA issuer (even CTA)
        constexpr uint32_t idesc = idesc_bf16_f32(BMP, BN);
        uint32_t it = 0, tile = 0;
        auto run_k = [&](uint32_t dcol, int nkb) {
            for (int kb = 0; kb < nkb; ++kb, ++it) {
                const int s = it % STAGES;
                // TMA -> tensor core hand-off: the mbarrier completion suffices
                wait_lim(&sm.full[s], (it / STAGES) & 1, a.status, &s_dead);
#pragma unroll
                for (int k = 0; k < BK / 16; ++k) {
                    const uint64_t ad = smem_desc_sw128(smem_u32(sm.a + s * A_BYTES) + k * 32);
                    const uint64_t bd = smem_desc_sw128(smem_u32(sm.b + s * B_BYTES) + k * 32);
                    tc_mma_pair(tmem + dcol, ad, bd, idesc, kb > 0 || k > 0);
                }
                tc_commit_pair(&sm.empty[s], kPairMask);
            }
        };
        for (int u = pair; u < units; u += n_pairs) {
            int mt, g;
            unit_coords(u, m_tiles, a.n_groups, &mt, &g);
            const int t0 = g * kTilesPerGroup, t1 = min(n_tiles, t0 + kTilesPerGroup);
            for (int nt = t0; nt < t1; ++nt, ++tile) {
                if (tile > 0)  // both epilogues hold Z_t of the previous tile in registers
                    wait_lim(sm.free_t, (tile - 1) & 1, a.status, &s_dead, true);
                tc_fence_after();
                run_k(kColT, kb_t);
                tc_commit_pair(sm.acc_t, kPairMask);
                if (tile > 0)  // both epilogues have read Z_s of the previous tile
                    wait_lim(sm.free_s, (tile - 1) & 1, a.status, &s_dead, true);
                tc_fence_after();
                run_k(kColS, kb_s);
                tc_commit_pair(sm.acc_s, kPairMask);
            }
        }
    } else if (warp >= 2) {
        // ---------------- epilogue: warp (q, cq) owns rows q*32.. and columns cq*64..
        const int ew = warp - 2;
        const int q = warp % 4;              // tensor-memory lane quarter this warp may read
        const int cq = ew / 4;               // column slice [cq*64, cq*64 + 64) of the tile
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        const uint32_t col0 = (uint32_t)(cq * kEpiCols);
        const uint32_t free_t0 = mapa(smem_u32(sm.free_t), 0), free_s0 = mapa(smem_u32(sm.free_s), 0);
        uint8_t *stg = sm.stg + ew * kStgWarpBytes;
        uint32_t tile = 0;
        for (int u = pair; u < units; u += n_pairs) {
            int mt, g;
            unit_coords(u, m_tiles, a.n_groups, &mt, &g);
            const int t0 = g * kTilesPerGroup, t1 = min(n_tiles, t0 + kTilesPerGroup);
            const int row = mt * BMP + (int)rank * BM + q * 32 + lane;
            const bool valid_row = row < nvalid;
            float ms = -INFINITY, ss = 0.f, sa = 0.f, mt_ = -INFINITY, st = 0.f;
            float nl = 0.f, cp = 0.f, sg = 1.f;
            if (MODE == 1 && valid_row) {
                const float4 c = reinterpret_cast<const float4 *>(a.rowc)[row];
                nl = c.x, cp = c.y, sg = c.z;
            }
            for (int nt = t0; nt < t1; ++nt, ++tile) {
                const int64_t vbase = (int64_t)nt * BN + col0;   // vocabulary id of column 0 here
                const int64_t left = a.vocab - vbase;
                const int nv = left <= 0 ? 0 : (left >= kEpiCols ? kEpiCols : (int)left);
                // Z_t: 64 columns into registers, then release them to the next tile
                float zt[kEpiCols];
                wait_lim(sm.acc_t, tile & 1, a.status, &s_dead);
                tc_fence_after();
                tmem_ld32(tmem + lane_off + kColT + col0, *reinterpret_cast<float(*)[32]>(&zt[0]));
                tmem_ld32(tmem + lane_off + kColT + col0 + 32, *reinterpret_cast<float(*)[32]>(&zt[32]));
                tmem_ld_wait();
                release_cols(free_t0, lane);
                if (MODE == 0 && nv > 0) {
                    float cmt = -INFINITY;
#pragma unroll
                    for (int j = 0; j < kEpiCols; ++j)
                        if (j < nv)
                            cmt = fmaxf(cmt, zt[j]);
                    if (cmt > mt_) {
                        st *= ex2((mt_ - cmt) * kLog2e);
                        mt_ = cmt;
                    }
                    const float ntt = -mt_ * kLog2e;
#pragma unroll
                    for (int j = 0; j < kEpiCols; ++j)
                        if (j < nv)
                            st += ex2(fmaf(zt[j], kLog2e, ntt));
                }
                // G columns [vbase, vbase + 64) lie wholly inside or outside [0, vpad)
                // (both multiples of 64); the staging buffer is free once the previous
                // tile's store has read it
                const bool in_g = MODE == 1 && vbase < a.vpad;
                if (in_g) {
                    if (lane == 0)
                        bulk_wait_read0();
                    __syncwarp();
                }
                // Z_s: 16 columns at a time
                wait_lim(sm.acc_s, tile & 1, a.status, &s_dead);
                tc_fence_after();
#pragma unroll
                for (int ch = 0; ch < kEpiCols / 16; ++ch) {
                    float zs[16];
                    tmem_ld16(tmem + lane_off + kColS + col0 + ch * 16, zs);
                    tmem_ld_wait();
                    const int c0 = ch * 16;
                    if (MODE == 0) {
                        if (c0 < nv) {
                            float cmx = -INFINITY;
#pragma unroll
                            for (int j = 0; j < 16; ++j)
                                if (c0 + j < nv)
                                    cmx = fmaxf(cmx, zs[j]);
                            if (cmx > ms) {
                                const float f = ex2((ms - cmx) * kLog2e);
                                ss *= f;
                                sa *= f;
                                ms = cmx;
                            }
                            const float ns = -ms * kLog2e;
#pragma unroll
                            for (int j = 0; j < 16; ++j) {
                                if (c0 + j < nv) {
                                    const float e = ex2(fmaf(zs[j], kLog2e, ns));
                                    ss += e;
                                    sa = fmaf(e, zs[j] - zt[c0 + j], sa);
                                }
                            }
                        }
                    } else if (in_g) {
                        // G = w p ((z_s - z_t) - E_p[z_s - z_t]); zero beyond the vocabulary
                        // and on rows past the supervised ones.
                        uint32_t pk[8];
#pragma unroll
                        for (int j = 0; j < 16; j += 2) {
                            float g0 = 0.f, g1 = 0.f;
                            if (valid_row && c0 + j < nv)
                                g0 = sg * ex2(fmaf(zs[j], kLog2e, -nl)) * ((zs[j] - zt[c0 + j]) - cp);
                            if (valid_row && c0 + j + 1 < nv)
                                g1 = sg * ex2(fmaf(zs[j + 1], kLog2e, -nl)) *
                                     ((zs[j + 1] - zt[c0 + j + 1]) - cp);
                            pk[j / 2] = pack_bf16x2(g0, g1);
                        }
                        // this row's two 16-byte pieces 2ch, 2ch+1 of the 128-byte staging row,
                        // placed by the 128-byte swizzle (piece ^ row % 8)
                        uint8_t *srow = stg + lane * 128;
                        const int p0 = (2 * ch) ^ (lane & 7), p1 = (2 * ch + 1) ^ (lane & 7);
                        *reinterpret_cast<uint4 *>(srow + p0 * 16) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                        *reinterpret_cast<uint4 *>(srow + p1 * 16) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
                    }
                }
                release_cols(free_s0, lane);
                if (MODE == 1 && in_g) {
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        tma_store_2d(&tGst, (int)vbase, mt * BMP + (int)rank * BM + q * 32, stg);
                        bulk_commit();
                    }
                }
            }
            if (MODE == 0 && valid_row) {
                float *pp = a.part + (((size_t)g * kColQuarters + cq) * a.cap + row) * 8;
                reinterpret_cast<float4 *>(pp)[0] = make_float4(ms, ss, sa, mt_);
                reinterpret_cast<float4 *>(pp)[1] = make_float4(st, 0.f, 0.f, 0.f);
            }
        }
        if (MODE == 1 && lane == 0)
            bulk_wait0();
    }
    pair_epilogue(sm, tmem, 512, rank);
}

// ----------------------------------------------------------------------------
// dH = G W_s: A = G [rows, vpad] (K-major, K = vocabulary), B = W_s [V, d_s]
// read in place as an MN-major operand (per CTA two 64-column TMA boxes per
// stage).  Output pair tile 256 x 256 fp32 in tensor memory.  Work split, with
// P pairs: the first floor(tiles / P) * P tiles are whole tiles, one per pair
// per wave, written straight to their token rows; the remaining tiles'
// k-blocks are split evenly over all P pairs (each range covers at most two
// tiles) and written as partial tiles, which k_dh_fixup sums in pair order.
// The result is bitwise reproducible for a given number of pairs.
struct DhArgs {
    const int4 *rows;
    const int32_t *nvalid;
    int d_s;
    int kbs;         // vpad / BK
    float *dh;       // [T, d_s]
    float *partial;  // [P][2][BMP][BN]
    int32_t *status;
};

struct DhSeg {
    int tile, k0, k1, slot;  // slot -1: whole tile; 0/1: partial slot of this pair
};

template <class F>
__device__ __forceinline__ void dh_segments(int tiles, int kbs, int P, int c, F &&f)
{
    const int full = tiles / P * P;
    for (int t = c; t < full; t += P)
        f(DhSeg{t, 0, kbs, -1});
    const int rem = tiles - full;
    if (rem > 0) {
        const int64_t total = (int64_t)rem * kbs;
        const int64_t b = total * c / P, e = total * (c + 1) / P;
        int slot = 0;
        for (int64_t it = b; it < e;) {
            const int j = (int)(it / kbs), k0 = (int)(it % kbs);
            const int64_t k1l = k0 + (e - it);
            const int k1 = k1l < kbs ? (int)k1l : kbs;
            f(DhSeg{full + j, k0, k1, slot++});
            it += k1 - k0;
        }
    }
}

__global__ void __launch_bounds__(kThreads, 1)
k_fused_dh(const __grid_constant__ CUtensorMap tG, const __grid_constant__ CUtensorMap tW, DhArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ int s_dead;
    FusedSmem sm = carve(smem_raw, kDhBRegion, 0);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const uint32_t rank = cluster_ctarank();
    const int pair = (int)cluster_id(), n_pairs = (int)cluster_count();
    const int nvalid = *a.nvalid;
    const int m_tiles = (nvalid + BMP - 1) / BMP;
    const int n_tiles = a.d_s / BN;
    const int tiles = m_tiles * n_tiles;
    const uint32_t tmem = pair_prologue(sm, &s_dead, 256);

    // whole tiles: N-tile fastest, so the pairs of one wave share the G rows (A)
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tG);
        tma_prefetch_desc(&tW);
        const uint32_t full0 = mapa(smem_u32(sm.full), 0);
        uint32_t it = 0;
        dh_segments(tiles, a.kbs, n_pairs, pair, [&](const DhSeg &sg) {
            const int mt = sg.tile / n_tiles, nt = sg.tile % n_tiles;
            const int ya = mt * BMP + (int)rank * BM;
            const int xb = nt * BN + (int)rank * BNH;
            auto prefetch = [&](int kb) {
                if (kPrefetch == 0 || kb >= sg.k1)
                    return;
                tma_prefetch_l2_2d(&tG, kb * BK, ya);
#pragma unroll
                for (int j = 0; j < BNH / 64; ++j)
                    tma_prefetch_l2_2d(&tW, xb + j * 64, kb * BK);
            };
            for (int p = 0; p < kPrefetch; ++p)
                prefetch(sg.k0 + p);
            for (int kb = sg.k0; kb < sg.k1; ++kb, ++it) {
                prefetch(kb + kPrefetch);
                const int s = it % STAGES;
                if (it >= STAGES)
                    wait_lim(&sm.empty[s], ((it / STAGES) - 1) & 1, a.status, &s_dead);
                if (rank == 0)
                    mbar_arrive_expect_tx(&sm.full[s], 2 * STAGE_BYTES);
                const uint32_t fb = full0 + (uint32_t)s * 8u;
                tma_load_2d_pair(sm.a + s * A_BYTES, &tG, kb * BK, ya, fb);
#pragma unroll
                for (int j = 0; j < BNH / 64; ++j)
                    tma_load_2d_pair(sm.b + s * B_BYTES + j * (64 * BK * 2), &tW, xb + j * 64, kb * BK, fb);
            }
        });
        drain_producer(sm, it, rank);
    } else if (warp == 1 && lane == 0 && rank == 0) {
        constexpr uint32_t idesc = idesc_bf16_f32(BMP, BN, true);
        uint32_t it = 0, tile = 0;
        dh_segments(tiles, a.kbs, n_pairs, pair, [&](const DhSeg &sg) {
            if (tile > 0)
                wait_lim(sm.free_s, (tile - 1) & 1, a.status, &s_dead, true);
            tc_fence_after();
            for (int kb = sg.k0; kb < sg.k1; ++kb, ++it) {
                const int s = it % STAGES;
                wait_lim(&sm.full[s], (it / STAGES) & 1, a.status, &s_dead);
#pragma unroll
                for (int k = 0; k < BK / 16; ++k) {
                    const uint64_t ad = smem_desc_sw128(smem_u32(sm.a + s * A_BYTES) + k * 32);
                    // 16 K-rows of 128 B per step; 64-wide N blocks 8 KB apart; 8-row atoms 1 KB apart
                    const uint64_t bd =
                        smem_desc_sw128_mn(smem_u32(sm.b + s * B_BYTES) + k * 2048, 64 * BK * 2, 1024);
                    tc_mma_pair(tmem, ad, bd, idesc, kb > sg.k0 || k > 0);
                }
                tc_commit_pair(&sm.empty[s], kPairMask);
            }
            tc_commit_pair(sm.acc_s, kPairMask);
            ++tile;
        });
    } else if (warp >= 2) {
        const int ew = warp - 2, q = warp % 4, cq = ew / 4;
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        const int col0 = cq * kEpiCols;
        const int rloc = (int)rank * BM + q * 32 + lane;   // row within the pair tile
        const uint32_t free_s0 = mapa(smem_u32(sm.free_s), 0);
        uint32_t tile = 0;
        dh_segments(tiles, a.kbs, n_pairs, pair, [&](const DhSeg &sg) {
            const int mt = sg.tile / n_tiles, nt = sg.tile % n_tiles;
            const int row = mt * BMP + rloc;
            wait_lim(sm.acc_s, tile & 1, a.status, &s_dead);
            tc_fence_after();
            const bool valid = row < nvalid;
            float *dst = nullptr;
            if (valid) {
                if (sg.slot < 0)
                    dst = a.dh + (size_t)a.rows[row].x * a.d_s + nt * BN + col0;
                else
                    dst = a.partial + (((size_t)pair * 2 + sg.slot) * BMP + rloc) * BN + col0;
            }
#pragma unroll 1
            for (int ch = 0; ch < kEpiCols / 32; ++ch) {
                float v[32];
                tmem_ld32(tmem + lane_off + (uint32_t)(col0 + ch * 32), v);
                tmem_ld_wait();
                if (valid) {
                    float4 *d4 = reinterpret_cast<float4 *>(dst + ch * 32);
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        d4[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
                }
            }
            release_cols(free_s0, lane);
            ++tile;
        });
    }
    pair_epilogue(sm, tmem, 256, rank);
}

// ----------------------------------------------------------------------------
// dW_s = G^T H_s: [V, d_s] fp32, K = the supervised tokens (padded to the pair
// tile with zero rows of G and H_s).  A = G read as an MN-major operand (its
// columns are vocabulary ids), B = the gathered H_s read MN-major (columns are
// d_s); two 256-column accumulators in tensor memory, so the epilogue's stores
// of tile j overlap the MMAs of tile j+1.  Tiles: 256 vocabulary rows x 256
// columns of d_s, column tile fastest (pairs in flight share the G panel).
struct DwArgs {
    const int32_t *nvalid;
    int64_t vocab;
    int d_s;
    float *dw;       // [vocab, d_s]
    int32_t *status;
};

__global__ void __launch_bounds__(kThreads, 1)
k_fused_dw(const __grid_constant__ CUtensorMap tGmn, const __grid_constant__ CUtensorMap tHmn, DwArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ int s_dead;
    FusedSmem sm = carve(smem_raw, kDhBRegion, 0);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const uint32_t rank = cluster_ctarank();
    const int pair = (int)cluster_id(), n_pairs = (int)cluster_count();
    const int nvalid = *a.nvalid;
    const int kbs = (nvalid + BMP - 1) / BMP * (BMP / BK);
    const int v_tiles = (int)((a.vocab + BMP - 1) / BMP);
    const int d_tiles = a.d_s / BN;
    const int tiles = kbs > 0 ? v_tiles * d_tiles : 0;
    const uint32_t tmem = pair_prologue(sm, &s_dead, 512);
    uint64_t *accf[2] = {sm.acc_t, sm.acc_s};
    uint64_t *acce[2] = {sm.free_t, sm.free_s};

    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tGmn);
        tma_prefetch_desc(&tHmn);
        const uint32_t full0 = mapa(smem_u32(sm.full), 0);
        uint32_t it = 0;
        for (int t = pair; t < tiles; t += n_pairs) {
            const int mv = t / d_tiles, nd = t % d_tiles;
            const int xa = mv * BMP + (int)rank * BM;   // this CTA's 128 vocabulary ids
            const int xb = nd * BN + (int)rank * BNH;   // this CTA's 128 columns of d_s
            for (int kb = 0; kb < kbs; ++kb, ++it) {
                const int s = it % STAGES;
                if (it >= STAGES)
                    wait_lim(&sm.empty[s], ((it / STAGES) - 1) & 1, a.status, &s_dead);
                if (rank == 0)
                    mbar_arrive_expect_tx(&sm.full[s], 2 * STAGE_BYTES);
                const uint32_t fb = full0 + (uint32_t)s * 8u;
#pragma unroll
                for (int j = 0; j < BM / 64; ++j)
                    tma_load_2d_pair(sm.a + s * A_BYTES + j * (64 * BK * 2), &tGmn, xa + j * 64, kb * BK, fb);
#pragma unroll
                for (int j = 0; j < BNH / 64; ++j)
                    tma_load_2d_pair(sm.b + s * B_BYTES + j * (64 * BK * 2), &tHmn, xb + j * 64, kb * BK, fb);
            }
        }
        drain_producer(sm, it, rank);
    } else if (warp == 1 && lane == 0 && rank == 0 && kbs > 0) {
        constexpr uint32_t idesc = idesc_bf16_f32(BMP, BN, true, true);
        uint32_t it = 0, tile = 0;
        for (int t = pair; t < tiles; t += n_pairs, ++tile) {
            const int buf = tile & 1;
            if (tile >= 2)  // both epilogues have read this buffer's previous tile
                wait_lim(acce[buf], ((tile >> 1) - 1) & 1, a.status, &s_dead, true);
            tc_fence_after();
            for (int kb = 0; kb < kbs; ++kb, ++it) {
                const int s = it % STAGES;
                wait_lim(&sm.full[s], (it / STAGES) & 1, a.status, &s_dead);
#pragma unroll
                for (int k = 0; k < BK / 16; ++k) {
                    // 16 K-rows (tokens) of 128 B per step; 64-wide M/N blocks 8 KB apart
                    const uint64_t ad = smem_desc_sw128_mn(smem_u32(sm.a + s * A_BYTES) + k * 2048, 64 * BK * 2, 1024);
                    const uint64_t bd = smem_desc_sw128_mn(smem_u32(sm.b + s * B_BYTES) + k * 2048, 64 * BK * 2, 1024);
                    tc_mma_pair(tmem + (uint32_t)buf * 256u, ad, bd, idesc, kb > 0 || k > 0);
                }
                tc_commit_pair(&sm.empty[s], kPairMask);
            }
            tc_commit_pair(accf[buf], kPairMask);
        }
    } else if (warp >= 2) {
        const int ew = warp - 2, q = warp % 4, cq = ew / 4;
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        const int col0 = cq * kEpiCols;
        const uint32_t acce0[2] = {mapa(smem_u32(acce[0]), 0), mapa(smem_u32(acce[1]), 0)};
        uint32_t tile = 0;
        if (kbs == 0) {  // no supervised token: dW_s = 0
            for (int t = pair; t < v_tiles * d_tiles; t += n_pairs) {
                const int mv = t / d_tiles, nd = t % d_tiles;
                const int64_t v = (int64_t)mv * BMP + (int)rank * BM + q * 32 + lane;
                if (v < a.vocab) {
                    float4 *d4 = reinterpret_cast<float4 *>(a.dw + v * a.d_s + nd * BN + col0);
                    for (int jj = 0; jj < kEpiCols / 4; ++jj)
                        d4[jj] = make_float4(0.f, 0.f, 0.f, 0.f);
                }
            }
        }
        for (int t = pair; t < tiles; t += n_pairs, ++tile) {
            const int mv = t / d_tiles, nd = t % d_tiles, buf = tile & 1;
            const int64_t v = (int64_t)mv * BMP + (int)rank * BM + q * 32 + lane;
            wait_lim(accf[buf], (tile >> 1) & 1, a.status, &s_dead);
            tc_fence_after();
            float *dst = a.dw + v * a.d_s + nd * BN + col0;
#pragma unroll 1
            for (int ch = 0; ch < kEpiCols / 32; ++ch) {
                float x[32];
                tmem_ld32(tmem + lane_off + (uint32_t)buf * 256u + (uint32_t)(col0 + ch * 32), x);
                tmem_ld_wait();
                if (v < a.vocab) {
                    float4 *d4 = reinterpret_cast<float4 *>(dst + ch * 32);
#pragma unroll
                    for (int jj = 0; jj < 8; ++jj)
                        d4[jj] = make_float4(x[4 * jj], x[4 * jj + 1], x[4 * jj + 2], x[4 * jj + 3]);
                }
            }
            release_cols(acce0[buf], lane);
        }
    }
    pair_epilogue(sm, tmem, 512, rank);
}

// Sum the partial tiles of the split part of dH in pair order (P = pairs of
// the dH launch, at most kMaxPairs) and write them to their token rows.  Job =
// (split tile, 8-row block).
constexpr int kMaxPairs = 256;
inline int max_pairs(int sms) { return std::max(1, std::min(kMaxPairs, sms / 2)); }
__global__ void __launch_bounds__(256)
k_dh_fixup(const float *__restrict__ partial, const int4 *__restrict__ rows, const int32_t *__restrict__ nvalid_p,
           int d_s, int kbs, int P, float *__restrict__ dh)
{
    __shared__ int s_src[kMaxPairs + 2];
    __shared__ int s_n;
    const int nvalid = *nvalid_p;
    const int n_tiles = d_s / BN;
    const int tiles = (nvalid + BMP - 1) / BMP * n_tiles;
    const int full = tiles / P * P;
    const int rem = tiles - full;
    const int64_t total = (int64_t)rem * kbs;
    constexpr int kRowsPerJob = 8;
    for (int job = blockIdx.x; job < rem * (BMP / kRowsPerJob); job += gridDim.x) {
        const int j = job / (BMP / kRowsPerJob), rb = job % (BMP / kRowsPerJob);
        __syncthreads();
        if (threadIdx.x == 0) {
            // pairs whose non-empty k-block range meets tile j's [lo, hi), in pair order
            const int64_t lo = (int64_t)j * kbs, hi = lo + kbs;
            int n = 0;
            for (int c = 0; c < P; ++c) {
                const int64_t b = total * c / P, en = total * (c + 1) / P;
                if (b >= en || en <= lo || b >= hi)
                    continue;
                s_src[n++] = c * 2 + ((b / kbs == j) ? 0 : 1);
            }
            s_n = n;
        }
        __syncthreads();
        const int t = full + j, mt = t / n_tiles, nt = t % n_tiles;
        const int n = s_n;
        for (int e = threadIdx.x; e < kRowsPerJob * (BN / 4); e += blockDim.x) {
            const int r = rb * kRowsPerJob + e / (BN / 4), c4 = e % (BN / 4);
            const int row = mt * BMP + r;
            if (row >= nvalid)
                continue;
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
            for (int i = 0; i < n; ++i) {
                const float4 v = reinterpret_cast<const float4 *>(partial)[((size_t)s_src[i] * BMP + r) * (BN / 4) + c4];
                acc.x += v.x;
                acc.y += v.y;
                acc.z += v.z;
                acc.w += v.w;
            }
            reinterpret_cast<float4 *>(dh + (size_t)rows[row].x * d_s + nt * BN)[c4] = acc;
        }
    }
}

// ----------------------------------------------------------------------------
// Gather the supervised hidden rows: out[j] = h[token of row j] (16-byte copies).
// Rows from the supervised count up to the next pair-tile boundary are zeroed
// (the weight-gradient GEMM reads them as zero-weight tokens).
__global__ void k_gather_rows(const int4 *__restrict__ rows, const int32_t *__restrict__ nvalid,
                              const uint4 *__restrict__ h, int vec_per_row, uint4 *__restrict__ out)
{
    const int n = *nvalid;
    const int n_pad = (n + BMP - 1) / BMP * BMP;
    for (int j = blockIdx.x; j < n_pad; j += gridDim.x) {
        uint4 *dst = out + (int64_t)j * vec_per_row;
        if (j < n) {
            const uint4 *src = h + (int64_t)rows[j].x * vec_per_row;
            for (int c = threadIdx.x; c < vec_per_row; c += blockDim.x)
                dst[c] = src[c];
        } else {
            for (int c = threadIdx.x; c < vec_per_row; c += blockDim.x)
                dst[c] = make_uint4(0, 0, 0, 0);
        }
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
        for (int gh = 0; gh < kColQuarters * n_groups; ++gh) {
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

// 2-D bf16 tensor map over a row-major [rows, cols] matrix, 128-byte swizzle,
// box of box_cols (128 B) x box_rows; rows beyond the matrix read as zero.
bool make_map(CUtensorMap *m, const void *base, int64_t rows, int64_t cols, int box_rows, int box_cols)
{
    auto fn = encode_fn();
    if (!fn)
        return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
    cuuint32_t es[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct FusedLayout {
    int4 *rows;
    int32_t *blk_count, *nvalid;
    double *row_wl;
    __nv_bfloat16 *hs, *ht, *G;
    float *part, *rowc, *dh_partial;
    size_t bytes;
};

FusedLayout fused_layout(void *ws, int64_t T, int64_t V, int64_t d_s, int64_t d_t, int n_groups, int sms)
{
    const int64_t vpad = (V + BK - 1) / BK * BK;
    const int64_t cap = (T + BMP - 1) / BMP * BMP;
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
    L.part = reinterpret_cast<float *>(take(sizeof(float) * 8 * kColQuarters * (size_t)n_groups * cap));
    L.rowc = reinterpret_cast<float *>(take(sizeof(float) * 4 * (size_t)cap));
    L.G = reinterpret_cast<__nv_bfloat16 *>(take(2 * (size_t)cap * vpad));
    L.dh_partial = reinterpret_cast<float *>(take(sizeof(float) * (size_t)max_pairs(sms) * 2 * BMP * BN));
    L.bytes = off + 256;
    return L;
}

int groups_for(int64_t V) { return (int)(((V + BN - 1) / BN + kTilesPerGroup - 1) / kTilesPerGroup); }

// Launch `kern` on `pairs` 2-CTA clusters.
template <class... KArgs, class... Args>
cudaError_t launch_pairs(void (*kern)(KArgs...), int pairs, size_t smem, cudaStream_t stream, Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cfg.gridDim = dim3(2 * pairs);
    return cudaLaunchKernelEx(&cfg, kern, args...);
}

// Co-resident 2-CTA clusters of `kern` (cached per device), at most max_pairs.
template <class... KArgs>
cudaError_t pairs_for(void (*kern)(KArgs...), size_t smem, int slot, int *pairs)
{
    static int cache[64][4] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return e;
    if (dev < 64 && cache[dev][slot] > 0) {
        *pairs = cache[dev][slot];
        return cudaSuccess;
    }
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess)
        return e;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.gridDim = dim3(2);
    int ncl = 0;
    e = cudaOccupancyMaxActiveClusters(&ncl, kern, &cfg);
    if (e != cudaSuccess)
        return e;
    if (ncl < 1)
        return cudaErrorInvalidConfiguration;
    ncl = std::min(ncl, max_pairs(device_sm_count()));
    if (dev < 64)
        cache[dev][slot] = ncl;
    *pairs = ncl;
    return cudaSuccess;
}

}  // namespace

size_t fused_workspace_bytes(int64_t T, int64_t V, int64_t d_s, int64_t d_t)
{
    return fused_layout(nullptr, T, V, d_s, d_t, groups_for(V), device_sm_count()).bytes;
}

cudaError_t launch_fused(const FusedCall &c, cudaStream_t stream)
{
    const int n_groups = groups_for(c.vocab);
    const int sms = device_sm_count();
    FusedLayout L = fused_layout(c.workspace, c.T, c.vocab, c.d_s, c.d_t, n_groups, sms);
    const int64_t vpad = (c.vocab + BK - 1) / BK * BK;
    const int64_t cap = (c.T + BMP - 1) / BMP * BMP;

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
    e = cudaGetLastError();
    if (e != cudaSuccess)
        return e;

    alignas(64) CUtensorMap tHs, tWs, tHt, tWt, tG, tGst, tWmn, tGmn, tHmn;
    if (!make_map(&tHs, L.hs, cap, c.d_s, BM, BK) || !make_map(&tWs, c.W_s, c.vocab, c.d_s, BNH, BK) ||
        !make_map(&tHt, L.ht, cap, c.d_t, BM, BK) || !make_map(&tWt, c.W_t, c.vocab, c.d_t, BNH, BK) ||
        !make_map(&tG, L.G, cap, vpad, BM, BK) || !make_map(&tGst, L.G, cap, vpad, 32, kEpiCols) ||
        // W_s as the MN-major B of dH: boxes of 64 d-columns x BK vocabulary rows
        !make_map(&tWmn, c.W_s, c.vocab, c.d_s, BK, 64) ||
        // G and the gathered H_s as the MN-major operands of dW_s: 64 columns x BK token rows
        !make_map(&tGmn, L.G, cap, vpad, BK, 64) || !make_map(&tHmn, L.hs, cap, c.d_s, BK, 64))
        return cudaErrorInvalidValue;

    int p_lm0 = 0, p_lm1 = 0, p_dh = 0, p_dw = 0;
    if ((e = pairs_for(k_fused_dw, kDhSmem, 3, &p_dw)) != cudaSuccess)
        return e;
    if ((e = pairs_for(k_fused_lm<0>, kFusedSmem, 0, &p_lm0)) != cudaSuccess ||
        (e = pairs_for(k_fused_lm<1>, kFusedSmem, 1, &p_lm1)) != cudaSuccess ||
        (e = pairs_for(k_fused_dh, kDhSmem, 2, &p_dh)) != cudaSuccess)
        return e;

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

    if ((e = launch_pairs(k_fused_lm<0>, p_lm0, kFusedSmem, stream, tHs, tWs, tHt, tWt, tGst, fa)) != cudaSuccess)
        return e;
    k_fused_merge<<<(int)((cap + 255) / 256), 256, 0, stream>>>(L.rows, L.nvalid, L.part, n_groups, cap,
                                                               c.token_loss, L.row_wl, L.rowc, c.status);
    e = cudaGetLastError();
    if (e != cudaSuccess)
        return e;
    if (c.dh_s || c.dW_s) {
        if ((e = launch_pairs(k_fused_lm<1>, p_lm1, kFusedSmem, stream, tHs, tWs, tHt, tWt, tGst, fa)) != cudaSuccess)
            return e;
    }
    if (c.dW_s) {
        DwArgs wa;
        wa.nvalid = L.nvalid;
        wa.vocab = c.vocab;
        wa.d_s = (int)c.d_s;
        wa.dw = c.dW_s;
        wa.status = c.status;
        if ((e = launch_pairs(k_fused_dw, p_dw, kDhSmem, stream, tGmn, tHmn, wa)) != cudaSuccess)
            return e;
    }
    if (c.dh_s) {
        launch_zero_masked_f32(c.mask, c.T, (int64_t)c.d_s, c.dh_s, stream);
        DhArgs da;
        da.rows = L.rows;
        da.nvalid = L.nvalid;
        da.d_s = (int)c.d_s;
        da.kbs = (int)(vpad / BK);
        da.dh = c.dh_s;
        da.partial = L.dh_partial;
        da.status = c.status;
        if ((e = launch_pairs(k_fused_dh, p_dh, kDhSmem, stream, tG, tWmn, da)) != cudaSuccess)
            return e;
        k_dh_fixup<<<2 * sms, 256, 0, stream>>>(L.dh_partial, L.rows, L.nvalid, (int)c.d_s, da.kbs, p_dh, c.dh_s);
    }
    launch_loss_sum(L.row_wl, L.nvalid, c.loss, c.status, stream);
    return cudaGetLastError();
}

}  // namespace turnopd
