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

// 32 consecutive values of a row (16-byte aligned) as vector loads / stores.
__device__ __forceinline__ void load_row32(const float* src, float* v) {
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        const float4 f = reinterpret_cast<const float4*>(src)[q];
        v[4 * q] = f.x; v[4 * q + 1] = f.y; v[4 * q + 2] = f.z; v[4 * q + 3] = f.w;
    }
}
__device__ __forceinline__ void load_row32(const __nv_bfloat16* src, float* v) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const uint4 u = reinterpret_cast<const uint4*>(src)[q];
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[e]));
            v[8 * q + 2 * e] = f.x; v[8 * q + 2 * e + 1] = f.y;
        }
    }
}
__device__ __forceinline__ void store_row32(float* dst, const float* v) {
#pragma unroll
    for (int q = 0; q < 8; ++q)
        reinterpret_cast<float4*>(dst)[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
}
__device__ __forceinline__ void store_row32(__nv_bfloat16* dst, const float* v) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const __nv_bfloat162 p = __floats2bfloat162_rn(v[8 * q + 2 * e], v[8 * q + 2 * e + 1]);
            w[e] = *reinterpret_cast<const uint32_t*>(&p);
        }
        reinterpret_cast<uint4*>(dst)[q] = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

// 16-value variants (half the registers).
__device__ __forceinline__ void load_row16(const float* src, float* v) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const float4 f = reinterpret_cast<const float4*>(src)[q];
        v[4 * q] = f.x; v[4 * q + 1] = f.y; v[4 * q + 2] = f.z; v[4 * q + 3] = f.w;
    }
}
__device__ __forceinline__ void load_row16(const __nv_bfloat16* src, float* v) {
#pragma unroll
    for (int q = 0; q < 2; ++q) {
        const uint4 u = reinterpret_cast<const uint4*>(src)[q];
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[e]));
            v[8 * q + 2 * e] = f.x; v[8 * q + 2 * e + 1] = f.y;
        }
    }
}
__device__ __forceinline__ void store_row16(float* dst, const float* v) {
#pragma unroll
    for (int q = 0; q < 4; ++q)
        reinterpret_cast<float4*>(dst)[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
}
__device__ __forceinline__ void store_row16(__nv_bfloat16* dst, const float* v) {
#pragma unroll
    for (int q = 0; q < 2; ++q) {
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const __nv_bfloat162 p = __floats2bfloat162_rn(v[8 * q + 2 * e], v[8 * q + 2 * e + 1]);
            w[e] = *reinterpret_cast<const uint32_t*>(&p);
        }
        reinterpret_cast<uint4*>(dst)[q] = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

// 8 consecutive bf16 values (16-byte aligned) as floats.
__device__ __forceinline__ void load_row8(const __nv_bfloat16* src, float* v) {
    const uint4 u = *reinterpret_cast<const uint4*>(src);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[e]));
        v[2 * e] = f.x; v[2 * e + 1] = f.y;
    }
}

// 8 floats as bf16 (16-byte aligned destination).
__device__ __forceinline__ void store_row8(__nv_bfloat16* dst, const float* v) {
    uint32_t w[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const __nv_bfloat162 p = __floats2bfloat162_rn(v[2 * e], v[2 * e + 1]);
        w[e] = *reinterpret_cast<const uint32_t*>(&p);
    }
    *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
}

// SiLU(z) = z * sigmoid(z), the SMA residual gate (Sec. 3).
__device__ __forceinline__ float silu_f32(float z) { return z / (1.0f + expf(-z)); }

// Programmatic dependent launch (PTX griddepcontrol). launch_dependents: a kernel
// launched next on the stream with programmatic stream serialization may start
// once every CTA of this grid has executed it or exited. wait: blocks the thread
// until the grid this one was launched after has completed and its memory
// operations are visible; it returns at once in a kernel launched without that
// attribute (the stream order has already done it).
__device__ __forceinline__ void griddep_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
// d SiLU / dz = s (1 + z (1 - s)), s = sigmoid(z)
__device__ __forceinline__ float silu_grad_f32(float z) {
    const float s = 1.0f / (1.0f + expf(-z));
    return s * (1.0f + z * (1.0f - s));
}

}  // namespace dart
