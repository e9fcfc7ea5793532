// Device helpers shared by the libturnopd kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "turnopd.h"

namespace turnopd {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// First device-side error wins; later ones are dropped.
__device__ __forceinline__ void set_status(int32_t *status, int32_t code)
{
    if (status)
        atomicCAS(status, 0, code);
}

// 2^x by the PTX approximate base-2 exponential (flushes subnormal results).
__device__ __forceinline__ float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float to_float(float x) { return x; }
__device__ __forceinline__ float to_float(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T> __device__ __forceinline__ T from_float(float x);
template <> __device__ __forceinline__ float from_float<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_float<__nv_bfloat16>(float x)
{
    return __float2bfloat16_rn(x);
}

// bf16 pair packed in a 32-bit word -> two floats (exact).
__device__ __forceinline__ float bf16lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf16hi(uint32_t u) { return __uint_as_float(u & 0xffff0000u); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&v);
}

// Online accumulators of one logit row.
//
// Student: running max m, S = sum exp(z_s - m), and
//   A = sum exp(z_s - m) ((z_s - z_t) - d),
// taken relative to a reference difference d = (z_s - z_t) at the student's
// running argmax.  E_p[z_s - z_t] = d + A/S; when a few tokens dominate p_s,
// A/S is small and the gradient factor (z_s - z_t) - E_p[z_s - z_t] =
// ((z_s - z_t) - d) - A/S keeps full fp32 relative precision at those tokens
// ((z_s - z_t) - d is exact for bf16 inputs).
// Teacher: running max and S only.
struct Student {
    float m, s, a, d;
};
struct Teacher {
    float m, s;
};

__device__ __forceinline__ Student student_empty() { return Student{-INFINITY, 0.f, 0.f, 0.f}; }
__device__ __forceinline__ Teacher teacher_empty() { return Teacher{-INFINITY, 0.f}; }

// Merge two accumulators: rescale both to the larger max and re-reference A
// to the shift of the side holding that max.
__device__ __forceinline__ Student student_merge(Student x, Student y)
{
    const float m = fmaxf(x.m, y.m);
    if (m == -INFINITY)
        return x;
    const float d = x.m >= y.m ? x.d : y.d;
    const float fx = ex2((x.m - m) * kLog2e);
    const float fy = ex2((y.m - m) * kLog2e);
    Student r;
    r.m = m;
    r.d = d;
    r.s = x.s * fx + y.s * fy;
    r.a = fmaf(x.s, x.d - d, x.a) * fx + fmaf(y.s, y.d - d, y.a) * fy;
    return r;
}

__device__ __forceinline__ Teacher teacher_merge(Teacher x, Teacher y)
{
    const float m = fmaxf(x.m, y.m);
    if (m == -INFINITY)
        return x;
    return Teacher{m, x.s * ex2((x.m - m) * kLog2e) + y.s * ex2((y.m - m) * kLog2e)};
}

__device__ __forceinline__ Student shfl_xor(Student x, int o)
{
    Student y;
    y.m = __shfl_xor_sync(0xffffffffu, x.m, o);
    y.s = __shfl_xor_sync(0xffffffffu, x.s, o);
    y.a = __shfl_xor_sync(0xffffffffu, x.a, o);
    y.d = __shfl_xor_sync(0xffffffffu, x.d, o);
    return y;
}

__device__ __forceinline__ Teacher shfl_xor(Teacher x, int o)
{
    Teacher y;
    y.m = __shfl_xor_sync(0xffffffffu, x.m, o);
    y.s = __shfl_xor_sync(0xffffffffu, x.s, o);
    return y;
}

// Butterfly merges across the warp (the value of lane 0 is the one used).
__device__ __forceinline__ Student warp_merge(Student x)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        x = student_merge(x, shfl_xor(x, o));
    return x;
}

__device__ __forceinline__ Teacher warp_merge(Teacher x)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        x = teacher_merge(x, shfl_xor(x, o));
    return x;
}

// Per-row constants once both distributions are reduced.
struct RowConst {
    float lse_s, lse_t;
    float dl;   // LSE_s - LSE_t, as (m_s - m_t) + log(S_s / S_t): no cancellation of two
                // large LSE values, so l = (z_s - z_t)_y - dl stays accurate near 0
    float d;    // reference difference
    float cp;   // A/S: E_p[z_s - z_t] - d
    float kl;   // full-vocabulary reverse KL
};

__device__ __forceinline__ RowConst row_const(Student s, Teacher t)
{
    RowConst c;
    c.lse_s = s.m + logf(s.s);
    c.lse_t = t.m + logf(t.s);
    c.dl = (s.m - t.m) + logf(s.s / t.s);
    c.d = s.d;
    c.cp = s.a / s.s;
    c.kl = (s.d + c.cp) - c.dl;
    return c;
}

__device__ __forceinline__ double warp_sum_f64(double x)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

__device__ __forceinline__ int64_t warp_sum_i64(int64_t x)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

__device__ __forceinline__ float warp_sum_f(float x)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

__device__ __forceinline__ float warp_max_f(float x)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
    return x;
}

// Programmatic dependent launch.  A kernel launched with launch_dependent may start
// before the work ahead of it in the stream has finished: it must call pdl_begin()
// before its first global memory access.  pdl_begin waits until that work has
// completed and its writes are visible, then lets the next dependent launch.
__device__ __forceinline__ void pdl_begin()
{
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                             cudaStream_t stream, Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

__device__ __forceinline__ int warp_sum_i32(int x)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

// Workspace carving: 256-byte aligned sub-buffers.
__host__ __device__ __forceinline__ size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

}  // namespace turnopd
