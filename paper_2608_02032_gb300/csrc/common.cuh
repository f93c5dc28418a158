// Shared device helpers for the DART CUDA kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace dart {

typedef long long i64;

template <typename T> __device__ __forceinline__ float ld_f32(const T* p);
template <> __device__ __forceinline__ float ld_f32<float>(const float* p) { return *p; }
template <> __device__ __forceinline__ float ld_f32<__nv_bfloat16>(const __nv_bfloat16* p) {
    return __bfloat162float(*p);
}

template <typename T> __device__ __forceinline__ T cvt_from_f32(float v);
template <> __device__ __forceinline__ float cvt_from_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 cvt_from_f32<__nv_bfloat16>(float v) {
    return __float2bfloat16_rn(v);
}

// Value of v after a round trip through storage type T, i.e. the value a
// later kernel reads back from memory written in T.
template <typename T> __device__ __forceinline__ float stored_value(float v);
template <> __device__ __forceinline__ float stored_value<float>(float v) { return v; }
template <> __device__ __forceinline__ float stored_value<__nv_bfloat16>(float v) {
    return __bfloat162float(__float2bfloat16_rn(v));
}

// SiLU(z) = z * sigmoid(z), the SMA residual gate (Sec. 3).
__device__ __forceinline__ float silu_f32(float z) { return z / (1.0f + expf(-z)); }

}  // namespace dart
