// Row-streaming helpers shared by the row kernels and the vocabulary-parallel
// kernels: 16-byte vector loads widened to fp32, vector stores of the
// gradient, the online fold of logits into the student / teacher accumulators
// (max, sum exp, sum exp ((z_s - z_t) - d)), and the fixed-order merge of
// per-lane partials across a warp.
#pragma once

#include "common.cuh"

namespace turnopd {

template <typename TIn> struct Vec;
template <> struct Vec<__nv_bfloat16> {
    static constexpr int N = 8;
    __device__ static void load(const void *p, float *x)
    {
        const uint4 u = __ldg(reinterpret_cast<const uint4 *>(p));
        x[0] = bf16lo(u.x), x[1] = bf16hi(u.x), x[2] = bf16lo(u.y), x[3] = bf16hi(u.y);
        x[4] = bf16lo(u.z), x[5] = bf16hi(u.z), x[6] = bf16lo(u.w), x[7] = bf16hi(u.w);
    }
};
template <> struct Vec<float> {
    static constexpr int N = 4;
    __device__ static void load(const void *p, float *x)
    {
        const float4 u = __ldg(reinterpret_cast<const float4 *>(p));
        x[0] = u.x, x[1] = u.y, x[2] = u.z, x[3] = u.w;
    }
};

template <typename TOut, int N> __device__ __forceinline__ void store_vec(TOut *p, const float *g);
template <> __device__ __forceinline__ void store_vec<__nv_bfloat16, 8>(__nv_bfloat16 *p, const float *g)
{
    uint4 u;
    u.x = pack_bf16x2(g[0], g[1]);
    u.y = pack_bf16x2(g[2], g[3]);
    u.z = pack_bf16x2(g[4], g[5]);
    u.w = pack_bf16x2(g[6], g[7]);
    *reinterpret_cast<uint4 *>(p) = u;
}
template <> __device__ __forceinline__ void store_vec<__nv_bfloat16, 4>(__nv_bfloat16 *p, const float *g)
{
    uint2 u;
    u.x = pack_bf16x2(g[0], g[1]);
    u.y = pack_bf16x2(g[2], g[3]);
    *reinterpret_cast<uint2 *>(p) = u;
}
template <> __device__ __forceinline__ void store_vec<float, 8>(float *p, const float *g)
{
    reinterpret_cast<float4 *>(p)[0] = make_float4(g[0], g[1], g[2], g[3]);
    reinterpret_cast<float4 *>(p)[1] = make_float4(g[4], g[5], g[6], g[7]);
}
template <> __device__ __forceinline__ void store_vec<float, 4>(float *p, const float *g)
{
    *reinterpret_cast<float4 *>(p) = make_float4(g[0], g[1], g[2], g[3]);
}

// Merge per-lane partial statistics across the first `width` lanes of a warp
// (lanes beyond hold empty partials): exact max by butterfly, one rescale
// exponential per lane, then butterfly sums.  Lane 0's result is used; its
// association order is fixed, so every warp and CTA gets the same bits.
template <int WIDTH, bool USE_D = true>
__device__ __forceinline__ void lane_merge(Student &S, Teacher &T)
{
    float m = S.m, mt = T.m;
#pragma unroll
    for (int o = 1; o < WIDTH; o <<= 1) {
        m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, o));
    }
    // reference difference of the lowest lane holding the max
    float d = 0.f;
    if (USE_D) {
        const unsigned own = __ballot_sync(0xffffffffu, S.m == m && m != -INFINITY);
        const int src = own ? __ffs(own) - 1 : 0;
        d = __shfl_sync(0xffffffffu, S.d, src);
    }
    const float f = m == -INFINITY ? 0.f : ex2((S.m - m) * kLog2e);
    const float ft = mt == -INFINITY ? 0.f : ex2((T.m - mt) * kLog2e);
    float s = S.s * f, a = (USE_D ? fmaf(S.s, S.d - d, S.a) : S.a) * f, t = T.s * ft;
    if (S.m == -INFINITY)
        s = 0.f, a = 0.f;
    if (T.m == -INFINITY)
        t = 0.f;
#pragma unroll
    for (int o = 1; o < WIDTH; o <<= 1) {
        s += __shfl_xor_sync(0xffffffffu, s, o);
        a += __shfl_xor_sync(0xffffffffu, a, o);
        t += __shfl_xor_sync(0xffffffffu, t, o);
    }
    S = Student{m, s, a, d};
    T = Teacher{mt, t};
}

// Fold n student/teacher values into the online accumulators.
template <int N>
__device__ __forceinline__ void accumulate(Student &s, Teacher &t, const float *a, const float *b)
{
    float mx = a[0], xd = a[0] - b[0], my = b[0];
#pragma unroll
    for (int k = 1; k < N; ++k) {
        if (a[k] > mx) {
            mx = a[k];
            xd = a[k] - b[k];
        }
        my = fmaxf(my, b[k]);
    }
    if (mx > s.m) {
        const float f = ex2((s.m - mx) * kLog2e);
        s.a = fmaf(s.s, s.d - xd, s.a) * f;
        s.s *= f;
        s.m = mx;
        s.d = xd;
    }
    if (my > t.m) {
        t.s *= ex2((t.m - my) * kLog2e);
        t.m = my;
    }
    const float ns = -s.m * kLog2e, nt = -t.m * kLog2e;
#pragma unroll
    for (int k = 0; k < N; ++k) {
        const float e = ex2(fmaf(a[k], kLog2e, ns));
        s.s += e;
        s.a = fmaf(e, (a[k] - b[k]) - s.d, s.a);
        t.s += ex2(fmaf(b[k], kLog2e, nt));
    }
}

// Fold one teacher value alone, in the steps of accumulate<1>: a sampled-token row's y
// where it is not part of a vector (see add_sampled_term).
__device__ __forceinline__ void accumulate_teacher(Teacher &t, float b)
{
    if (b > t.m) {
        t.s *= ex2((t.m - b) * kLog2e);
        t.m = b;
    }
    t.s += ex2(fmaf(b, kLog2e, -t.m * kLog2e));
}

// Sampled-token row (Eq. opd-rkl's one-token estimator): the student statistics leave y
// out altogether -- within a vector of finite logits its logit is replaced by the
// lowest finite value, which is then never the maximum and adds 0 to every sum; a y
// read alone folds into the teacher only -- so s holds S' = sum_{v != y} exp(z_s - m')
// at the maximum m' of the other logits.  This adds y's own term at M = max(m', z_y):
// S = S' e^{m' - M} + e^{z_y - M}, and returns 1 - p_y = S' e^{m' - M} / S, which
// keeps its relative precision when p_y is close to 1 (1 - p_y formed as 1 - e_y / S,
// or as w l - w l p_y, loses it to cancellation).  A is rescaled with S; y's term of
// A stays out (a sampled-token row does not use A).
__device__ __forceinline__ float add_sampled_term(Student &s, float zy)
{
    const float M = fmaxf(s.m, zy);
    const float f = s.m == -INFINITY ? 0.f : ex2((s.m - M) * kLog2e);
    const float sx = s.s * f;
    s.a *= f;
    s.m = M;
    s.s = sx + ex2((zy - M) * kLog2e);
    return sx / s.s;
}

}  // namespace turnopd
