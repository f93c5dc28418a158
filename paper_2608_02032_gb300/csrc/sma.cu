// State-memory attention forward with the gated residual merge, FFMA path
// (Sec. 3 value/key readouts, chunk logit, softmax over earlier chunks, R_t
// and Y_t = C_t H_t + G_t R_t; App. B.1 normalised score branch; Alg. 1
// streaming order with the online softmax of App. C).
//
// One block of 256 threads per (64-token tile, h, b). The tile's Qbar^T,
// C^T and Ebar stay in shared memory; memories j are streamed through shared
// memory once per tile. For each memory the block forms, per token t,
//   U_t = Qbar_t (r_j (.) M_j)   (so l_{t,j} = U_t . Ebar_t / sqrt(N))
//   V_t = C_t M_j
// as two 64 x P x N FFMA tiles, then updates the online softmax (m, d, O).
// Only R, lse and Y are written (Alg. 1 keeps keys, values and logits on chip).
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dart {

// r_{j,n} = (mean_p M_j[n,p]^2 + eps)^-1/2 of the stored memory (App. B.1).
// One warp per row of P elements.
template <typename Tmem>
__global__ void memory_rms_kernel(const Tmem* __restrict__ M, float* __restrict__ rM, i64 rows,
                                  int P, float eps) {
    const i64 row = (i64)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
    const int lane = threadIdx.x & 31;
    if (row >= rows) return;
    float ss = 0.0f;
    for (int p = lane; p < P; p += 32) {
        const float v = ld_f32(M + row * P + p);
        ss = fmaf(v, v, ss);
    }
    for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    if (lane == 0) rM[row] = __frsqrt_rn(ss / (float)P + eps);
}

template <typename Tmem>
cudaError_t launch_memory_rms(const void* M, float* rM, int64_t rows, int64_t P, float eps,
                              cudaStream_t stream) {
    const int warps = 8;
    memory_rms_kernel<Tmem><<<(unsigned)((rows + warps - 1) / warps), 32 * warps, 0, stream>>>(
        (const Tmem*)M, rM, rows, (int)P, eps);
    note_launches(1);
    return cudaGetLastError();
}

template cudaError_t launch_memory_rms<float>(const void*, float*, int64_t, int64_t, float,
                                              cudaStream_t);
template cudaError_t launch_memory_rms<__nv_bfloat16>(const void*, float*, int64_t, int64_t,
                                                      float, cudaStream_t);

constexpr int kTT = 64;  // tokens per tile

template <typename Tin, typename Tmem, typename Tout>
__global__ void __launch_bounds__(256)
sma_forward_simt_kernel(const Tmem* __restrict__ Mem, const float* __restrict__ rM,
                        const Tin* __restrict__ Q, const Tin* __restrict__ Cm,
                        const Tin* __restrict__ E, const Tin* __restrict__ z,
                        const Tout* __restrict__ Yssd, Tout* __restrict__ Y, Tout* __restrict__ R,
                        float* __restrict__ lse, int L, int H, int G, int P, int N, int S, int Mc,
                        float eps) {
    extern __shared__ float4 smem4[];
    float* smem = reinterpret_cast<float*>(smem4);
    float* sQt = smem;             // [N][64]  Qbar^T
    float* sCt = sQt + N * kTT;    // [N][64]  C^T
    float* sE = sCt + N * kTT;     // [64][64] Ebar (columns >= P are zero)
    float* sD = sE + kTT * 64;     // [N][64]  M_j (columns >= P are zero)
    float* sW = sD + N * 64;       // [N][64]  r_j (.) M_j

    const int tile = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int g = h / (H / G);
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int lane = tid & 31, warp = tid >> 5;
    const int t0 = tile * kTT;
    const int ntok = min(kTT, L - t0);
    const i64 row0 = (i64)b * L + t0;  // token row of the tile start

    // prologue: normalised query, value-read vector and verifier of the tile
    for (int r = warp; r < kTT; r += 8) {
        const bool ok = r < ntok;
        const Tin* q = Q + ((row0 + r) * G + g) * N;
        const Tin* c = Cm + ((row0 + r) * G + g) * N;
        const Tin* e = E + ((row0 + r) * G + g) * P;
        float ssq = 0.0f, sse = 0.0f;
        for (int n = lane; n < N; n += 32) {
            const float v = ok ? ld_f32(q + n) : 0.0f;
            ssq = fmaf(v, v, ssq);
        }
        for (int p = lane; p < P; p += 32) {
            const float v = ok ? ld_f32(e + p) : 0.0f;
            sse = fmaf(v, v, sse);
        }
        for (int off = 16; off > 0; off >>= 1) {
            ssq += __shfl_xor_sync(0xffffffffu, ssq, off);
            sse += __shfl_xor_sync(0xffffffffu, sse, off);
        }
        const float iq = __frsqrt_rn(ssq / (float)N + eps);
        const float ie = __frsqrt_rn(sse / (float)P + eps);
        for (int n = lane; n < N; n += 32) {
            sQt[n * kTT + r] = ok ? ld_f32(q + n) * iq : 0.0f;
            sCt[n * kTT + r] = ok ? ld_f32(c + n) : 0.0f;
        }
        for (int p = lane; p < 64; p += 32) sE[r * 64 + p] = (ok && p < P) ? ld_f32(e + p) * ie : 0.0f;
    }

    int nh[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) nh[i] = (t0 + ty * 4 + i) / S;  // memories each row attends to
    const int nh_max = (t0 + ntok - 1) / S;
    const float inv_sqrt_n = __frsqrt_rn((float)N);

    float O[4][4] = {}, m[4], d[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) { m[i] = -INFINITY; d[i] = 0.0f; }

    for (int j = 0; j < nh_max; ++j) {
        __syncthreads();
        const i64 mbase = (((i64)b * Mc + j) * H + h);
        const Tmem* Mj = Mem + mbase * N * P;
        const float* rj = rM + mbase * N;
        for (int e = tid; e < N * 64; e += 256) {
            const int n = e >> 6, p = e & 63;
            const float v = p < P ? ld_f32(Mj + (i64)n * P + p) : 0.0f;
            sD[e] = v;
            sW[e] = v * rj[n];
        }
        __syncthreads();
        float U[4][4] = {}, V[4][4] = {};
#pragma unroll 4
        for (int n = 0; n < N; ++n) {
            const float4 q4 = *reinterpret_cast<const float4*>(&sQt[n * kTT + ty * 4]);
            const float4 c4 = *reinterpret_cast<const float4*>(&sCt[n * kTT + ty * 4]);
            const float4 w4 = *reinterpret_cast<const float4*>(&sW[n * 64 + tx * 4]);
            const float4 d4 = *reinterpret_cast<const float4*>(&sD[n * 64 + tx * 4]);
            const float qq[4] = {q4.x, q4.y, q4.z, q4.w}, cc[4] = {c4.x, c4.y, c4.z, c4.w};
            const float ww[4] = {w4.x, w4.y, w4.z, w4.w}, dd[4] = {d4.x, d4.y, d4.z, d4.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    U[i][k] = fmaf(qq[i], ww[k], U[i][k]);
                    V[i][k] = fmaf(cc[i], dd[k], V[i][k]);
                }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float4 e4 = *reinterpret_cast<const float4*>(&sE[(ty * 4 + i) * 64 + tx * 4]);
            float part = U[i][0] * e4.x + U[i][1] * e4.y + U[i][2] * e4.z + U[i][3] * e4.w;
            for (int off = 8; off > 0; off >>= 1) part += __shfl_xor_sync(0xffffffffu, part, off);
            const float l = part * inv_sqrt_n;
            if (j < nh[i]) {
                const float mn = fmaxf(m[i], l);
                const float sc = expf(m[i] - mn);
                const float pe = expf(l - mn);
                d[i] = fmaf(d[i], sc, pe);
#pragma unroll
                for (int k = 0; k < 4; ++k) O[i][k] = fmaf(O[i][k], sc, pe * V[i][k]);
                m[i] = mn;
            }
        }
    }

    // epilogue: R = O / d, lse = m + log d, Y = Y_ssd + SiLU(z) R
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int tl = ty * 4 + i;
        if (tl >= ntok) continue;
        const i64 row = (row0 + tl) * H + h;
        const bool has = nh[i] > 0;
        const float inv_d = has ? 1.0f / d[i] : 0.0f;
        const float gate = silu_f32(ld_f32(z + row));
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int p = tx * 4 + k;
            if (p >= P) continue;
            const float r = has ? O[i][k] * inv_d : 0.0f;
            const float y = ld_f32(Yssd + row * P + p) + gate * r;
            Y[row * P + p] = cvt_from_f32<Tout>(y);
            if (R != nullptr) R[row * P + p] = cvt_from_f32<Tout>(r);
        }
        if (tx == 0 && lse != nullptr) lse[row] = has ? m[i] + logf(d[i]) : -INFINITY;
    }
}

template <typename Tin, typename Tmem, typename Tout>
cudaError_t launch_sma_forward_simt(const SmaArgs& a, cudaStream_t stream) {
    const int N = (int)a.N;
    const size_t smem = (size_t)(4 * N * 64 + 64 * 64) * sizeof(float);
    auto kern = sma_forward_simt_kernel<Tin, Tmem, Tout>;
    cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem);
    if (err != cudaSuccess) return err;
    const int M = (int)(a.L / a.S);
    dim3 grid((unsigned)((a.L + kTT - 1) / kTT), (unsigned)a.H, (unsigned)a.B);
    kern<<<grid, 256, smem, stream>>>((const Tmem*)a.M, a.rM, (const Tin*)a.Q, (const Tin*)a.Cm,
                                      (const Tin*)a.E, (const Tin*)a.z, (const Tout*)a.Yssd,
                                      (Tout*)a.Y, (Tout*)a.R, a.lse, (int)a.L, (int)a.H, (int)a.G,
                                      (int)a.P, N, (int)a.S, M, a.eps);
    note_launches(1);
    return cudaGetLastError();
}

typedef __nv_bfloat16 bf16;
template cudaError_t launch_sma_forward_simt<float, float, float>(const SmaArgs&, cudaStream_t);
template cudaError_t launch_sma_forward_simt<bf16, float, float>(const SmaArgs&, cudaStream_t);
template cudaError_t launch_sma_forward_simt<bf16, bf16, float>(const SmaArgs&, cudaStream_t);
template cudaError_t launch_sma_forward_simt<bf16, bf16, bf16>(const SmaArgs&, cudaStream_t);

}  // namespace dart
