// Shared-memory staging helpers of the tensor-core kernels: cp.async
// 16-byte copies into 128-byte-swizzled rows (the layout the UMMA
// descriptors of salt_tcgen05.cuh read) and bf16 conversions.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

namespace salt {

__device__ __forceinline__ uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ int swz128(int row, int chunk) { return row * 128 + ((chunk ^ (row & 7)) << 4); }

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, bool valid)
{
    int n = valid ? 16 : 0;  // 0: zero-fill, nothing read
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(n));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }
// wait until at most n groups are pending (n in [0, 7])
__device__ __forceinline__ void cp_async_wait_dyn(int n)
{
    switch (n) {
    case 0: cp_async_wait<0>(); break;
    case 1: cp_async_wait<1>(); break;
    case 2: cp_async_wait<2>(); break;
    case 3: cp_async_wait<3>(); break;
    case 4: cp_async_wait<4>(); break;
    case 5: cp_async_wait<5>(); break;
    case 6: cp_async_wait<6>(); break;
    default: cp_async_wait<7>(); break;
    }
}

__device__ __forceinline__ float bf16_to_f(uint16_t h) { return __uint_as_float(((uint32_t)h) << 16); }
__device__ __forceinline__ uint16_t f_to_bf16(float f)
{
    __nv_bfloat16 b = __float2bfloat16_rn(f);
    return *reinterpret_cast<uint16_t *>(&b);
}

// Two bf16 (low half first) plus two fp32 deltas, each sum rounded once to
// bf16 (round to nearest even), packed the same way.
__device__ __forceinline__ uint32_t add_bf16x2(uint32_t y2, float d_lo, float d_hi)
{
    const float lo = __uint_as_float(y2 << 16) + d_lo;
    const float hi = __uint_as_float(y2 & 0xffff0000u) + d_hi;
    const __nv_bfloat162 r = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t *>(&r);
}

}  // namespace salt
