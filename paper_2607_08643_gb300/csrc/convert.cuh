// convert.cuh -- number-format conversions shared by the kernels of the
// method's variants (rows.cu, decoder.cu, formats.cu).  bf16 and fp16 are
// passed as their bit patterns; every widening here is exact.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

namespace bisco {
namespace cvt {

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ float bf16_to_f32(uint16_t b) {
    return __uint_as_float(static_cast<uint32_t>(b) << 16);
}

__device__ __forceinline__ double bf16_to_f64(uint16_t b) { return static_cast<double>(bf16_to_f32(b)); }

__device__ __forceinline__ double f16_to_f64(uint16_t h) {
    return static_cast<double>(__half2float(__ushort_as_half(h)));
}

// binary64 -> binary16 bits, round to nearest even, gradual underflow.
__device__ __forceinline__ uint16_t f64_to_f16_rn(double x) {
    unsigned short r;
    asm("cvt.rn.f16.f64 %0, %1;" : "=h"(r) : "d"(x));
    return r;
}

// fp32 -> an output element type, round to nearest even.
template <typename T>
__device__ __forceinline__ T from_f32(float v);
template <>
__device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }
template <>
__device__ __forceinline__ __half from_f32<__half>(float v) { return __float2half_rn(v); }

}  // namespace cvt
}  // namespace bisco
