// Turn bookkeeping, blend weights and turn statistics (sm_103a).
//
// All three are light, latency-bound passes over int32 turn ids, uint8 masks
// and fp32 token losses: ~5-9 bytes per token, far below the logit rows.
// One CTA owns one trajectory, so every reduction over a trajectory's tokens
// happens inside that CTA in a fixed order (integer shared-memory atomics are
// order-free; floating-point sums use fixed per-warp chunks and fixed trees).
// Nothing is accumulated with floating-point global atomics.

#include "common.cuh"
#include "kernels.h"

namespace turnopd {

// ---------------------------------------------------------------- counts

// Validates trajectory b's offsets and returns its token range (clamped to
// [0, T]); on error sets the status and returns an empty range.
__device__ __forceinline__ bool traj_range(const int64_t *off, int32_t B, int64_t T, int b,
                                           int64_t &lo, int64_t &hi, int32_t *status)
{
    lo = off[b];
    hi = off[b + 1];
    bool ok = lo >= 0 && hi >= lo && hi <= T;
    if (b == 0 && lo != 0)
        ok = false;
    if (b == B - 1 && hi != T)
        ok = false;
    if (!ok) {
        if (threadIdx.x == 0)
            set_status(status, TURNOPD_ERR_OFFSETS);
        lo = hi = 0;
    }
    return ok;
}

// n_bt[b][t] = supervised tokens of trajectory b at turn t (grid = B CTAs).
__global__ void k_traj_counts(const int32_t *__restrict__ turn_id,
                              const uint8_t *__restrict__ mask,
                              const int64_t *__restrict__ off, int32_t B, int64_t T,
                              int32_t Tmax, int32_t *__restrict__ n_bt, int32_t *status)
{
    pdl_begin();
    extern __shared__ int32_t hist[];
    const int b = blockIdx.x;
    for (int t = threadIdx.x; t < Tmax; t += blockDim.x)
        hist[t] = 0;
    __syncthreads();
    int64_t lo, hi;
    traj_range(off, B, T, b, lo, hi, status);
    bool bad = false;
    // four tokens per thread in flight; mask and turn id loaded together (a token's turn
    // id is read whether or not it is supervised: the index lies inside the trajectory)
    const int64_t step = blockDim.x;
    for (int64_t i0 = lo + threadIdx.x; i0 < hi; i0 += 4 * step) {
        uint8_t m[4];
        int32_t t[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int64_t i = i0 + u * step;
            m[u] = i < hi ? mask[i] : 0;
            t[u] = i < hi ? turn_id[i] : 0;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            if (!m[u])
                continue;
            if (t[u] < 0 || t[u] >= Tmax) {
                bad = true;
                continue;
            }
            atomicAdd(&hist[t[u]], 1);
        }
    }
    if (bad)
        set_status(status, TURNOPD_ERR_TURN_RANGE);
    __syncthreads();
    for (int t = threadIdx.x; t < Tmax; t += blockDim.x)
        n_bt[(int64_t)b * Tmax + t] = hist[t];
}

// counts = [S_t (Tmax), C_t (Tmax), B'] from the n_bt table (one CTA).
__global__ void k_counts_reduce(const int32_t *__restrict__ n_bt, int32_t B, int32_t Tmax,
                                int64_t *__restrict__ counts)
{
    pdl_begin();
    __shared__ int64_t warp_bp[32];
    // eight table entries loaded at a time (integer sums: any order gives the same result)
    for (int t = threadIdx.x; t < Tmax; t += blockDim.x) {
        int64_t s = 0, c = 0;
        for (int b0 = 0; b0 < B; b0 += 8) {
            int32_t n[8];
#pragma unroll
            for (int u = 0; u < 8; ++u)
                n[u] = b0 + u < B ? n_bt[(int64_t)(b0 + u) * Tmax + t] : 0;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                s += n[u] > 0;
                c += n[u];
            }
        }
        counts[t] = s;
        counts[Tmax + t] = c;
    }
    // B' = trajectories holding at least one supervised token
    int64_t bp = 0;
    for (int b = threadIdx.x; b < B; b += blockDim.x) {
        int64_t nb = 0;
        for (int t0 = 0; t0 < Tmax; t0 += 8) {
            int32_t n[8];
#pragma unroll
            for (int u = 0; u < 8; ++u)
                n[u] = t0 + u < Tmax ? n_bt[(int64_t)b * Tmax + t0 + u] : 0;
#pragma unroll
            for (int u = 0; u < 8; ++u)
                nb += n[u];
        }
        bp += nb > 0;
    }
    bp = warp_sum_i64(bp);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0)
        warp_bp[warp] = bp;
    __syncthreads();
    if (threadIdx.x == 0) {
        int64_t tot = 0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w)
            tot += warp_bp[w];
        counts[2 * Tmax] = tot;
    }
}

// ---------------------------------------------------------------- weights

// One CTA per trajectory: its token weights from n_bt[b][:] and the
// (possibly rank-summed) count vector.  Arithmetic in fp64, once per turn: a
// token's weight depends only on its trajectory and turn, so the CTA fills a
// per-turn table and each token reads its entry (fp64 runs at a small fraction
// of the fp32 rate, and a division per token on one SM per trajectory cost
// more than the rest of the kernel).
__global__ void k_weights(const int32_t *__restrict__ turn_id, const uint8_t *__restrict__ mask,
                          const int64_t *__restrict__ off, int32_t B, int64_t T, int32_t Tmax,
                          double alpha, int32_t scope, int32_t n_min,
                          const int32_t *__restrict__ n_bt, const int64_t *__restrict__ counts,
                          float *__restrict__ w_out, int32_t *status)
{
    pdl_begin();
    __shared__ int64_t red[4][32];
    __shared__ double coef[3];  // token weight 1/N_b (or 1/N), reliable-turn numerator, R
    __shared__ float s_wt[TURNOPD_MAX_TURNS];  // this trajectory's token weight per turn
    const int b = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nw = blockDim.x >> 5;
    const int64_t *S = counts;
    const int64_t *C = counts + Tmax;
    const int64_t Bp = counts[2 * Tmax];
    const int32_t *nb = n_bt + (int64_t)b * Tmax;

    // per-trajectory (traj scope) or batch-wide (batch scope) sums over t:
    //   tokens, unreliable tokens, reliable non-empty turns (or pairs)
    int64_t v_tok = 0, v_unrel = 0, v_rel = 0;
    for (int t = threadIdx.x; t < Tmax; t += blockDim.x) {
        const bool reliable = n_min <= 0 || S[t] >= n_min;
        const int64_t n = scope == TURNOPD_SCOPE_TRAJ ? (int64_t)nb[t] : C[t];
        v_tok += n;
        if (!reliable)
            v_unrel += n;
        else
            v_rel += scope == TURNOPD_SCOPE_TRAJ ? (int64_t)(nb[t] > 0) : S[t];
    }
    v_tok = warp_sum_i64(v_tok);
    v_unrel = warp_sum_i64(v_unrel);
    v_rel = warp_sum_i64(v_rel);
    if (lane == 0) {
        red[0][warp] = v_tok;
        red[1][warp] = v_unrel;
        red[2][warp] = v_rel;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int64_t tok = 0, unrel = 0, rel = 0;
        for (int w = 0; w < nw; ++w) {
            tok += red[0][w];
            unrel += red[1][w];
            rel += red[2][w];
        }
        double base = tok > 0 ? 1.0 / (double)tok : 0.0;           // w_traj
        double share = tok > 0 ? 1.0 - (double)unrel / (double)tok : 0.0;
        coef[0] = base;
        coef[1] = share;
        coef[2] = (double)rel;
    }
    __syncthreads();
    const double w_traj = coef[0], share = coef[1], R = coef[2];
    const double norm = scope == TURNOPD_SCOPE_TRAJ ? (Bp > 0 ? 1.0 / (double)Bp : 0.0) : 1.0;
    for (int t = threadIdx.x; t < Tmax; t += blockDim.x) {
        float wt = 0.f;
        if (w_traj > 0.0) {
            const bool reliable = n_min <= 0 || S[t] >= n_min;
            const double w_turn = (!reliable || R == 0.0) ? w_traj : share / (R * (double)nb[t]);
            wt = (float)(((1.0 - alpha) * w_traj + alpha * w_turn) * norm);
        }
        s_wt[t] = wt;  // turns without tokens here are never read
    }
    __syncthreads();

    int64_t lo, hi;
    traj_range(off, B, T, b, lo, hi, status);
    // four tokens per thread in flight, mask and turn id loaded together
    const int64_t step = blockDim.x;
    for (int64_t i0 = lo + threadIdx.x; i0 < hi; i0 += 4 * step) {
        uint8_t m[4];
        int32_t t[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int64_t i = i0 + u * step;
            m[u] = i < hi ? mask[i] : 0;
            t[u] = i < hi ? turn_id[i] : -1;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int64_t i = i0 + u * step;
            if (i < hi)
                w_out[i] = m[u] && t[u] >= 0 && t[u] < Tmax ? s_wt[t[u]] : 0.f;
        }
    }
    // tokens outside every trajectory range (only with bad offsets) stay untouched
}

// ---------------------------------------------------------------- turn stats

// One CTA per trajectory.  Warp w sums a fixed contiguous chunk of the
// trajectory's tokens into its own shared-memory bins; inside a 32-token
// step, tokens of the same turn are combined by a fixed xor tree.  The warp
// bins are then added in warp order.  Deterministic for fixed launch shape.
__global__ void k_turn_stats_traj(const float *__restrict__ token_loss,
                                  const int32_t *__restrict__ turn_id,
                                  const uint8_t *__restrict__ mask,
                                  const int64_t *__restrict__ off, int32_t B, int64_t T,
                                  int32_t Tmax, double *__restrict__ traj_turn_sum,
                                  int32_t *__restrict__ traj_turn_cnt, int32_t *status)
{
    pdl_begin();
    extern __shared__ unsigned char smem_raw[];
    const int nw = blockDim.x >> 5;
    double *bsum = reinterpret_cast<double *>(smem_raw);                    // [nw][Tmax]
    int32_t *bcnt = reinterpret_cast<int32_t *>(bsum + (size_t)nw * Tmax);  // [nw][Tmax]
    const int b = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int k = threadIdx.x; k < nw * Tmax; k += blockDim.x) {
        bsum[k] = 0.0;
        bcnt[k] = 0;
    }
    __syncthreads();
    int64_t lo, hi;
    traj_range(off, B, T, b, lo, hi, status);
    const int64_t n = hi - lo;
    const int64_t chunk = ((n + nw - 1) / nw + 31) / 32 * 32;
    const int64_t c0 = lo + (int64_t)warp * chunk;
    const int64_t c1 = min(hi, c0 + chunk);
    bool bad = false;
    // four 32-token steps per iteration: every load of the four is issued first (mask,
    // turn id and loss together), then the steps are folded in order as before
    for (int64_t base = c0; base < c1; base += 4 * 32) {
        uint8_t mk[4];
        int32_t tt[4];
        float lv[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int64_t i = base + u * 32 + lane;
            const bool in = i < c1;
            mk[u] = in ? mask[i] : 0;
            tt[u] = in ? turn_id[i] : -1;
            lv[u] = in ? token_loss[i] : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            int32_t key = -1;
            float val = 0.f;
            if (mk[u]) {
                if (tt[u] >= 0 && tt[u] < Tmax) {
                    key = tt[u];
                    val = lv[u];
                } else {
                    bad = true;
                }
            }
            unsigned todo = __ballot_sync(0xffffffffu, key >= 0);
            while (todo) {
                const int leader = __ffs(todo) - 1;
                const int k0 = __shfl_sync(0xffffffffu, key, leader);
                const bool mine = key == k0 && key >= 0;
                const unsigned members = __ballot_sync(0xffffffffu, mine);
                const double s = warp_sum_f64(mine ? (double)val : 0.0);
                if (lane == 0) {
                    bsum[(size_t)warp * Tmax + k0] += s;
                    bcnt[(size_t)warp * Tmax + k0] += __popc(members);
                }
                todo &= ~members;
            }
        }
    }
    if (bad)
        set_status(status, TURNOPD_ERR_TURN_RANGE);
    __syncthreads();
    for (int t = threadIdx.x; t < Tmax; t += blockDim.x) {
        double s = 0.0;
        int32_t c = 0;
        for (int w = 0; w < nw; ++w) {
            s += bsum[(size_t)w * Tmax + t];
            c += bcnt[(size_t)w * Tmax + t];
        }
        traj_turn_sum[(int64_t)b * Tmax + t] = s;
        traj_turn_cnt[(int64_t)b * Tmax + t] = c;
    }
}

// Per turn index: sums over trajectories in trajectory order.
__global__ void k_turn_stats_index(const double *__restrict__ traj_turn_sum,
                                   const int32_t *__restrict__ traj_turn_cnt, int32_t B,
                                   int32_t Tmax, double *__restrict__ turn_sum,
                                   int64_t *__restrict__ turn_cnt, int32_t *__restrict__ turn_surv)
{
    pdl_begin();
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= Tmax)
        return;
    double s = 0.0;
    int64_t c = 0;
    int32_t v = 0;
    // eight trajectories' entries loaded at a time, added in trajectory order
    for (int b0 = 0; b0 < B; b0 += 8) {
        double sv[8];
        int32_t nv[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int b = b0 + u;
            sv[u] = b < B ? traj_turn_sum[(int64_t)b * Tmax + t] : 0.0;
            nv[u] = b < B ? traj_turn_cnt[(int64_t)b * Tmax + t] : 0;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u)
            if (b0 + u < B) {
                s += sv[u];
                c += nv[u];
                v += nv[u] > 0;
            }
    }
    turn_sum[t] = s;
    turn_cnt[t] = c;
    turn_surv[t] = v;
}

// ---------------------------------------------------------------- launchers

// One CTA per trajectory: 32 warps, so a 4096-token trajectory takes 4 load steps per warp.
constexpr int kTrajThreads = 1024;

cudaError_t launch_turn_counts(const int32_t *turn_id, const uint8_t *mask, const int64_t *off,
                               int32_t B, int64_t T, int32_t Tmax, int32_t *n_bt,
                               int64_t *counts, int32_t *status, cudaStream_t stream)
{
    cudaError_t e = cudaSuccess;
    if (B > 0 &&
        (e = launch_dependent(k_traj_counts, dim3(B), dim3(kTrajThreads), sizeof(int32_t) * Tmax, stream,
                              turn_id, mask, off, B, T, Tmax, n_bt, status)) != cudaSuccess)
        return e;
    if ((e = launch_dependent(k_counts_reduce, dim3(1), dim3(256), 0, stream, n_bt, B, Tmax, counts)) != cudaSuccess)
        return e;
    return cudaGetLastError();
}

cudaError_t launch_weights(const int32_t *turn_id, const uint8_t *mask, const int64_t *off,
                           int32_t B, int64_t T, int32_t Tmax, double alpha, int32_t scope,
                           int32_t n_min, const int32_t *n_bt, const int64_t *counts,
                           float *w_out, int32_t *status, cudaStream_t stream)
{
    if (B > 0) {
        const cudaError_t e = launch_dependent(k_weights, dim3(B), dim3(kTrajThreads), 0, stream, turn_id, mask,
                                               off, B, T, Tmax, alpha, scope, n_min, n_bt, counts, w_out, status);
        if (e != cudaSuccess)
            return e;
    }
    return cudaGetLastError();
}

int turn_stats_warps(int32_t Tmax)
{
    // per-warp bins: Tmax * (8 + 4) bytes; keep the block under 160 KB
    const size_t per_warp = (size_t)Tmax * 12;
    int nw = (int)((160u * 1024u) / per_warp);
    return nw > kTrajThreads / 32 ? kTrajThreads / 32 : nw;
}

cudaError_t launch_turn_stats(const float *token_loss, const int32_t *turn_id,
                              const uint8_t *mask, const int64_t *off, int32_t B, int64_t T,
                              int32_t Tmax, double *traj_turn_sum, int32_t *traj_turn_cnt,
                              double *turn_sum, int64_t *turn_cnt, int32_t *turn_surv,
                              int32_t *status, cudaStream_t stream)
{
    const int nw = turn_stats_warps(Tmax);
    const size_t smem = (size_t)nw * Tmax * (sizeof(double) + sizeof(int32_t));
    if (B > 0) {
        if (smem > 48 * 1024) {
            cudaError_t e = cudaFuncSetAttribute(k_turn_stats_traj,
                                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)smem);
            if (e != cudaSuccess)
                return e;
        }
        const cudaError_t e = launch_dependent(k_turn_stats_traj, dim3(B), dim3(nw * 32), smem, stream,
                                               token_loss, turn_id, mask, off, B, T, Tmax, traj_turn_sum,
                                               traj_turn_cnt, status);
        if (e != cudaSuccess)
            return e;
    }
    const cudaError_t e = launch_dependent(k_turn_stats_index, dim3((Tmax + 127) / 128), dim3(128), 0, stream,
                                           traj_turn_sum, traj_turn_cnt, B, Tmax, turn_sum, turn_cnt, turn_surv);
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace turnopd
