// The block's projections on the 5th-generation tensor cores: C = A B^T with A
// (M x K) the token rows and B (N x K) a weight in nn.Linear layout, both
// bf16 and row-major (K contiguous), fp32 accumulation in TMEM, C stored as
// bf16 or fp32 with leading dimension ldc. The in-projection U W_in^T and the
// out-projection y W_out^T of the DART block (Sec. 3; the Mamba-2 block the
// paper builds on) are this product.
//
// Persistent: one CTA per SM walks the 128 x 256 tiles of C (N-fastest, so that
// neighbouring CTAs share the A tile in L2). 192 threads:
//   warp 0 lane 0  producer: TMA copies of the A and B tiles of each 64-wide K
//                  step (16 + 32 KiB, 128-byte swizzle = the MMA's K-major
//                  layout) into a 4-stage ring that runs on across tiles
//   warp 1         TMEM allocation (512 columns: two 256-column accumulators);
//                  lane 0 issues four M128 N256 K16 MMAs per stage, releases
//                  the stage with a commit, and commits each finished tile
//   warps 2..5     epilogue: each thread reads its row of a finished
//                  accumulator (warp w owns TMEM lanes 32 (w % 4) ..), hands the
//                  accumulator back and stores the row, while the MMAs of the
//                  next tile run in the other accumulator
#include <cuda_bf16.h>

#include "common.cuh"
#include "kernels.h"
#include "tc_ptx.cuh"
#include "tma.cuh"

namespace dart {
namespace {

__device__ int g_gemm_status;  // first timeout code since the last read (0 = none)

constexpr int kGM = 128, kGN = 256, kGK = 64, kGStages = 4;
constexpr int kGThreads = 192;
constexpr uint32_t kATile = kGM * 128, kBTile = kGN * 128;  // bytes per stage
constexpr uint64_t kGDrainNs = 2000000000ull;

struct GemmSmem {
    uint8_t a[kGStages][kATile];  // 1024-aligned by placement
    uint8_t b[kGStages][kBTile];
    uint64_t full[kGStages];      // the stage's A and B tiles landed (TMA -> MMA)
    uint64_t empty[kGStages];     // the stage's MMAs are done (MMA commit -> producer)
    uint64_t acc_full[2];         // a tile's MMAs into accumulator b are done (-> epilogue)
    uint64_t acc_empty[2];        // the epilogue has read accumulator b (4 warps -> MMA)
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
};

__device__ __forceinline__ void gemm_fail(volatile int* abort, int code) {
    *abort = 1;
    atomicCAS(&g_gemm_status, 0, code);
}

template <typename Tc>
__global__ void __launch_bounds__(kGThreads, 1)
gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
               Tc* __restrict__ C, int M, int N, int K, int ldc, int n_store, unsigned long long wait_limit_ns) {
    extern __shared__ uint8_t smem_raw[];
    GemmSmem& sm = *reinterpret_cast<GemmSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~(uintptr_t)1023);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int ksteps = (K + kGK - 1) / kGK;
    const int tiles_n = (N + kGN - 1) / kGN, tiles = tiles_n * ((M + kGM - 1) / kGM);
    volatile int* abort = &sm.abort;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kGStages; ++s) {
            tc::mbar_init(&sm.full[s], 1);
            tc::mbar_init(&sm.empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            tc::mbar_init(&sm.acc_full[b], 1);
            tc::mbar_init(&sm.acc_empty[b], 4);  // one arrival per epilogue warp
        }
        tc::mbar_init(&sm.drain, 1);
        sm.abort = 0;
        tc::fence_barrier_init();
        tc::tma_prefetch_map(&tmA);
        tc::tma_prefetch_map(&tmB);
    }
    if (warp == 1) {
        tc::tmem_alloc(&sm.tmem_base, 2 * kGN);
        tc::tmem_relinquish();
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = sm.tmem_base;

    if (warp == 0) {
        if (lane == 0) {
            // ------------------------------------------------------- producer
            int g = 0;  // K steps issued over all tiles (ring position)
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < tiles; tile += gridDim.x) {
                const int n0 = (tile % tiles_n) * kGN, m0 = (tile / tiles_n) * kGM;
                for (int ks = 0; ks < ksteps; ++ks, ++g) {
                    const int s = g % kGStages;
                    // the stage was last used by step g - kGStages: wait for its MMAs
                    if (g >= kGStages &&
                        !tc::mbar_wait(&sm.empty[s], (uint32_t)(((g / kGStages) - 1) & 1), wait_limit_ns, abort)) {
                        gemm_fail(abort, 61);
                        ok = false;
                        break;
                    }
                    tc::mbar_arrive_expect_tx(&sm.full[s], kATile + kBTile);
                    tc::tma_load_2d(sm.a[s], &tmA, ks * kGK, m0, &sm.full[s]);
                    tc::tma_load_2d(sm.b[s], &tmB, ks * kGK, n0, &sm.full[s]);
                }
            }
            // never leave a copy in flight behind: wait for the last copy into each stage
            for (int k = g - 1; k >= 0 && k >= g - kGStages; --k)
                if (!tc::mbar_wait(&sm.full[k % kGStages], (uint32_t)((k / kGStages) & 1), kGDrainNs, nullptr))
                    atomicCAS(&g_gemm_status, 0, 62);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ------------------------------------------------------- MMA issuer
            constexpr uint32_t idesc = tc::idesc_f16(1, false, kGM, kGN);  // bf16, A and B K-major
            bool ok = true, issued = false;
            int g = 0, it = 0;
            for (int tile = blockIdx.x; ok && tile < tiles; tile += gridDim.x, ++it) {
                const int ab = it & 1;
                // accumulator ab was last used by tile it - 2: wait until the epilogue read it
                if (it >= 2 && !tc::mbar_wait(&sm.acc_empty[ab], (uint32_t)(((it >> 1) - 1) & 1), wait_limit_ns, abort)) {
                    ok = false;
                    break;
                }
                tc::tc_fence_after();
                const uint32_t d = tmem + (uint32_t)(ab * kGN);
                for (int ks = 0; ks < ksteps; ++ks, ++g) {
                    const int s = g % kGStages;
                    if (!tc::mbar_wait(&sm.full[s], (uint32_t)((g / kGStages) & 1), wait_limit_ns, abort)) {
                        ok = false;
                        break;
                    }
                    tc::tc_fence_after();
                    const uint32_t a0 = tc::smem_u32(sm.a[s]), b0 = tc::smem_u32(sm.b[s]);
#pragma unroll
                    for (int kk = 0; kk < kGK / 16; ++kk)  // +32 bytes per K = 16 step inside the swizzled row
                        tc::mma_f16_ss(d, tc::smem_desc_sw128(a0 + 32u * kk, 16u, 1024u),
                                       tc::smem_desc_sw128(b0 + 32u * kk, 16u, 1024u), idesc,
                                       (ks > 0 || kk > 0) ? 1u : 0u);
                    tc::mma_commit(&sm.empty[s]);
                    issued = true;
                }
                if (ok) tc::mma_commit(&sm.acc_full[ab]);
            }
            if (!ok) gemm_fail(abort, 63);
            if (issued) {  // every MMA issued is done when this arrives, before TMEM is freed
                tc::mma_commit(&sm.drain);
                if (!tc::mbar_wait(&sm.drain, 0, kGDrainNs, nullptr)) atomicCAS(&g_gemm_status, 0, 65);
            }
        }
    } else {
        // ------------------------------------------------------- epilogue
        const int q = warp & 3;  // TMEM lane quarter of this warp
        const int row = 32 * q + lane;
        int it = 0;
        for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x, ++it) {
            const int ab = it & 1;
            const bool got = tc::mbar_wait(&sm.acc_full[ab], (uint32_t)((it >> 1) & 1), wait_limit_ns, abort);
            if (!__all_sync(0xffffffffu, got)) {
                if (lane == 0) gemm_fail(abort, 64);
                break;
            }
            tc::tc_fence_after();
            const int n0 = (tile % tiles_n) * kGN, m0 = (tile / tiles_n) * kGM;
            const int m = m0 + row;
            Tc* crow = C + (i64)m * ldc;
            const uint32_t taddr = tmem + (uint32_t)(ab * kGN) + ((uint32_t)(32 * q) << 16);
#pragma unroll 1
            for (int c0 = 0; c0 < kGN; c0 += 32) {
                uint32_t r[32];
                asm volatile(
                    "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
                    "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
                    "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n\t"
                    "tcgen05.wait::ld.sync.aligned;"
                    : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
                      "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
                      "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
                      "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
                      "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
                    : "r"(taddr + (uint32_t)c0)
                    : "memory");
                if (c0 + 32 == kGN) {  // the whole row is in registers: hand the accumulator back
                    tc::tc_fence_before();
                    __syncwarp();
                    if (lane == 0) tc::mbar_arrive(&sm.acc_empty[ab]);
                }
                if (m < M) {
                    float v[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
                    const int n = n0 + c0;
                    if (n + 32 <= n_store) {
                        store_row32(crow + n, v);
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            if (n + i < n_store) crow[n + i] = cvt_from_f32<Tc>(v[i]);
                    }
                }
            }
        }
    }

    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, 2 * kGN);
    }
}

}  // namespace

template <typename Tc>
cudaError_t launch_gemm_tc(const void* A, const void* B, Tc* C, int64_t M, int64_t N, int64_t K, int64_t ldc,
                           int64_t n_store, unsigned long long wait_limit_ns, cudaStream_t stream) {
    if (M <= 0 || N <= 0 || K <= 0 || K % 8 != 0 || n_store > ldc || M > 0x7fffffff ||
        ((N + kGN - 1) / kGN) * ((M + kGM - 1) / kGM) > 0x7fffffff || (ldc * (int64_t)sizeof(Tc)) % 16 != 0 ||
        (reinterpret_cast<uintptr_t>(C) & 15u) != 0)
        return cudaErrorInvalidValue;
    CUtensorMap ma, mb;
    if (!encode_bf16_rows_map(&ma, A, (uint64_t)M, (uint64_t)K, (uint64_t)K * 2, kGM, kGK) ||
        !encode_bf16_rows_map(&mb, B, (uint64_t)N, (uint64_t)K, (uint64_t)K * 2, kGN, kGK))
        return cudaErrorInvalidValue;
    auto kern = gemm_tc_kernel<Tc>;
    const size_t smem = sizeof(GemmSmem) + 1024;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int dev = 0, nsm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    const int64_t tiles = ((N + kGN - 1) / kGN) * ((M + kGM - 1) / kGM);
    const int grid = (int)(tiles < nsm ? tiles : nsm);  // persistent: one CTA per SM
    kern<<<grid, kGThreads, smem, stream>>>(ma, mb, C, (int)M, (int)N, (int)K, (int)ldc, (int)n_store,
                                            wait_limit_ns);
    note_launches(1);
    return cudaGetLastError();
}
template cudaError_t launch_gemm_tc<float>(const void*, const void*, float*, int64_t, int64_t, int64_t,
                                           int64_t, int64_t, unsigned long long, cudaStream_t);
template cudaError_t launch_gemm_tc<__nv_bfloat16>(const void*, const void*, __nv_bfloat16*, int64_t, int64_t,
                                                   int64_t, int64_t, int64_t, unsigned long long, cudaStream_t);

// Read and clear of the status word in one device-side exchange (see take_tc_status).
__device__ int g_gemm_status_taken;
__global__ void take_gemm_status_kernel() { g_gemm_status_taken = atomicExch(&g_gemm_status, 0); }

int take_gemm_status(cudaStream_t stream) {
    take_gemm_status_kernel<<<1, 1, 0, stream>>>();
    int v = 0;
    if (cudaGetLastError() != cudaSuccess ||
        cudaMemcpyFromSymbolAsync(&v, g_gemm_status_taken, sizeof(int), 0, cudaMemcpyDeviceToHost, stream) !=
            cudaSuccess ||
        cudaStreamSynchronize(stream) != cudaSuccess)
        return -1;
    return v;
}

}  // namespace dart
