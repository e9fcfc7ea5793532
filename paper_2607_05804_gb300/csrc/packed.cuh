// Packed arithmetic on bf16 logit vectors: two fp32 lanes per instruction
// (the sm_100-family paired-fp32 operations) and bf16x2 maxima.
#pragma once

#include <cstdint>

#include "common.cuh"

namespace turnopd {

// Subtraction is an exact fma by -1.
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) { return __ffma2_rn(a, b, c); }
__device__ __forceinline__ float2 fadd2(float2 a, float2 b) { return __fadd2_rn(a, b); }
__device__ __forceinline__ float2 fmul2(float2 a, float2 b) { return __fmul2_rn(a, b); }
__device__ __forceinline__ float2 fsub2(float2 a, float2 b)
{
    return __ffma2_rn(b, make_float2(-1.f, -1.f), a);
}

__device__ __forceinline__ float2 unpack2(uint32_t u) { return make_float2(bf16lo(u), bf16hi(u)); }
__device__ __forceinline__ float2 splat(float x) { return make_float2(x, x); }
__device__ __forceinline__ float2 ex2x2(float2 x) { return make_float2(ex2(x.x), ex2(x.y)); }

__device__ __forceinline__ uint32_t hmax2u(uint32_t a, uint32_t b)
{
    uint32_t d;
    asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}

__device__ __forceinline__ uint32_t word(const uint4 &v, int j)
{
    return j == 0 ? v.x : (j == 1 ? v.y : (j == 2 ? v.z : v.w));
}

// largest of the 8 bf16 values of a vector, as a bf16 pair whose halves are both candidates
__device__ __forceinline__ uint32_t hmax4(const uint4 &v) { return hmax2u(hmax2u(v.x, v.y), hmax2u(v.z, v.w)); }

}  // namespace turnopd
