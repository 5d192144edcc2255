// dbl_act.cuh -- the 16-bit storage format of activations, activation gradients
// and the convolutions' weight copies.  The default build stores bfloat16; the
// build with DBL_ACT_F16 defined (libdbl_f16.so) stores IEEE binary16, the
// format of the paper's mixed-precision ImageNet runs (Sec. 5.2.3).  Everything
// else (fp32 accumulation, master weights, statistics) is the same in both.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#ifdef DBL_ACT_F16
typedef __half act_t;
typedef __half2 act2_t;
#define DBL_ACT_X2 "f16x2"
#else
typedef __nv_bfloat16 act_t;
typedef __nv_bfloat162 act2_t;
#define DBL_ACT_X2 "bf16x2"
#endif

namespace dbl {
namespace act {

#ifdef DBL_ACT_F16
constexpr bool kF16 = true;
constexpr uint32_t kMmaFormat = 0;  // tcgen05 kind::f16 A/B format field: f16
#else
constexpr bool kF16 = false;
constexpr uint32_t kMmaFormat = 1;  // bf16
#endif

#ifdef __CUDACC__
// two fp32 values rounded to nearest even into one 16-bit pair (a in the low half)
__device__ __forceinline__ act2_t pack2(float a, float b)
{
#ifdef DBL_ACT_F16
    return __floats2half2_rn(a, b);
#else
    return __floats2bfloat162_rn(a, b);
#endif
}

__device__ __forceinline__ float2 unpack2(act2_t h)
{
#ifdef DBL_ACT_F16
    return __half22float2(h);
#else
    return __bfloat1622float2(h);
#endif
}

__device__ __forceinline__ act_t from_f(float x)
{
#ifdef DBL_ACT_F16
    return __float2half_rn(x);
#else
    return __float2bfloat16_rn(x);
#endif
}

__device__ __forceinline__ float to_f(act_t h)
{
#ifdef DBL_ACT_F16
    return __half2float(h);
#else
    return __bfloat162float(h);
#endif
}

// the same on the raw 32-bit pattern of a pair
__device__ __forceinline__ uint32_t pack2_u32(float a, float b)
{
    const act2_t h = pack2(a, b);
    return *reinterpret_cast<const uint32_t*>(&h);
}

__device__ __forceinline__ float2 unpack2_u32(uint32_t u)
{
    return unpack2(*reinterpret_cast<const act2_t*>(&u));
}
#endif  // __CUDACC__

}  // namespace act
}  // namespace dbl
