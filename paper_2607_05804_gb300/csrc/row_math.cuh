// Row-streaming helpers shared by the portable row kernel and the
// vocabulary-parallel kernels: 16-byte vector loads widened to fp32, vector
// stores of the gradient, and the online fold of logits into the student /
// teacher accumulators (max, sum exp, sum exp ((z_s - z_t) - d)).
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

}  // namespace turnopd
