// Per-head slices of (rows x H) arrays: dst[r, k] = src[r, h0 + k] for k < hg.
// The host-buffer prefill uses it to cut one head group's dt and gate logits
// out of the full arrays once they are on the device.
#include "common.cuh"
#include "kernels.h"

namespace dart {
namespace {

template <typename T>
__global__ void gather_heads_kernel(const T* __restrict__ src, T* __restrict__ dst, i64 rows, int H,
                                    int h0, int hg) {
    const i64 n = rows * hg;
    for (i64 i = (i64)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (i64)gridDim.x * blockDim.x) {
        const i64 r = i / hg;
        const int k = (int)(i - r * hg);
        dst[i] = src[r * H + h0 + k];
    }
}

}  // namespace

cudaError_t launch_gather_heads(const void* src, void* dst, int64_t rows, int64_t H, int64_t h0,
                                int64_t hg, int elem_bytes, cudaStream_t stream) {
    const i64 n = rows * hg;
    if (n <= 0) return cudaSuccess;
    const int threads = 256;
    const unsigned blocks = (unsigned)((n + threads - 1) / threads < 4096 ? (n + threads - 1) / threads : 4096);
    if (elem_bytes == 4)
        gather_heads_kernel<float><<<blocks, threads, 0, stream>>>((const float*)src, (float*)dst, rows,
                                                                   (int)H, (int)h0, (int)hg);
    else if (elem_bytes == 2)
        gather_heads_kernel<unsigned short><<<blocks, threads, 0, stream>>>(
            (const unsigned short*)src, (unsigned short*)dst, rows, (int)H, (int)h0, (int)hg);
    else
        return cudaErrorInvalidValue;
    note_launches(1);
    return cudaGetLastError();
}

}  // namespace dart
