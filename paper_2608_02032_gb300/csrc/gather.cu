// Per-head slices of (rows x H) arrays: dst[r, k] = src[r, h0 + k] for k < hg.
// The host-buffer prefill uses it to cut one head group's dt and gate logits
// out of the full arrays once they are on the device.
//
// Strided row copies: dst[r * dst_pitch + i] = src[r * src_pitch + i] for
// i < row_bytes, r < rows (pitches and row length in bytes). The tensor-core
// backward at G > 1 runs once per group on such copies: a group's heads are a
// contiguous slice of every token row (X, dt, dY, dM, ...), its B, C, Q, E one
// column block of every (G x N) or (G x P) row.
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

// Unit-sized words (16, 4 or 2 bytes, whichever divides every pitch, offset and
// the row length), one per thread and iteration.
template <typename W>
__global__ void copy_rows_kernel(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst, i64 rows,
                                 i64 words, i64 src_pitch, i64 dst_pitch) {
    const i64 n = rows * words;
    for (i64 i = (i64)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (i64)gridDim.x * blockDim.x) {
        const i64 r = i / words, k = i - r * words;
        reinterpret_cast<W*>(dst + r * dst_pitch)[k] = reinterpret_cast<const W*>(src + r * src_pitch)[k];
    }
}

}  // namespace

cudaError_t launch_copy_rows(void* dst, int64_t dst_pitch, const void* src, int64_t src_pitch, int64_t row_bytes,
                             int64_t rows, cudaStream_t stream) {
    if (rows <= 0 || row_bytes <= 0) return cudaSuccess;
    const uint64_t all = (uint64_t)(uintptr_t)dst | (uint64_t)(uintptr_t)src | (uint64_t)dst_pitch |
                         (uint64_t)src_pitch | (uint64_t)row_bytes;
    const int unit = (all & 15) == 0 ? 16 : (all & 3) == 0 ? 4 : (all & 1) == 0 ? 2 : 0;
    if (unit == 0) return cudaErrorInvalidValue;
    const i64 words = row_bytes / unit, n = rows * words;
    const int threads = 256;
    const unsigned blocks = (unsigned)((n + threads - 1) / threads < 8192 ? (n + threads - 1) / threads : 8192);
    const uint8_t* s = (const uint8_t*)src;
    uint8_t* d = (uint8_t*)dst;
    if (unit == 16)
        copy_rows_kernel<uint4><<<blocks, threads, 0, stream>>>(s, d, rows, words, src_pitch, dst_pitch);
    else if (unit == 4)
        copy_rows_kernel<uint32_t><<<blocks, threads, 0, stream>>>(s, d, rows, words, src_pitch, dst_pitch);
    else
        copy_rows_kernel<uint16_t><<<blocks, threads, 0, stream>>>(s, d, rows, words, src_pitch, dst_pitch);
    note_launches(1);
    return cudaGetLastError();
}

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
