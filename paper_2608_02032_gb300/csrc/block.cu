// The whole DART block around the hot path (Sec. 3: Q, E and the gate from the
// block input, C shared with the SSM branch, Y = C H + G R; for the rest the
// Mamba-2 block the paper builds on, with the sizes of App. D.2):
//   zx  = U W_in^T                                  in-projection (tensor cores, fp32 out)
//   z | x | B | C | dt | Q | E | gate              its column blocks
//   x, B, C = SiLU(causal depthwise conv(x, B, C))  width conv_width, per channel
//   dt = softplus(dt + dt_bias), A = -exp(A_log)
//   Y = scan + state-memory attention + merge       dart_chunk_scan, dart_sma_forward
//   y = Y + D_h x;  yn = RMSNorm(y SiLU(z)) w      over d_inner
//   out = yn W_out^T                                out-projection (tensor cores)
// The gate is one logit per token, broadcast to the heads (App. D.2).
#include <math.h>

#include <cuda_bf16.h>

#include "common.cuh"
#include "dart.h"
#include "kernels.h"

namespace dart {
namespace {

constexpr int kMaxConv = 8;

// One thread per (token, 8 channels) of the in-projection's x, B, C blocks (the
// convolution), then per (token, 8 channels) of Q and E (copies) and per (token,
// head) of dt and the gate. Columns of zx: z [0, di), x [di, 2 di), B, C (GN
// each), dt (H), Q (GN), E (GP), gate (1).
__global__ void __launch_bounds__(128)
block_conv_split_kernel(const float* __restrict__ zx, int ldz, int L, int di, int GN, int GP, int H,
                        int W, const float* __restrict__ conv_w, const float* __restrict__ conv_b,
                        const float* __restrict__ dt_bias, const float* __restrict__ A_log,
                        __nv_bfloat16* __restrict__ X, __nv_bfloat16* __restrict__ Bm,
                        __nv_bfloat16* __restrict__ Cm, float* __restrict__ dt, float* __restrict__ A,
                        __nv_bfloat16* __restrict__ Q, __nv_bfloat16* __restrict__ E,
                        __nv_bfloat16* __restrict__ gate) {
    const i64 tok = blockIdx.x;            // b L + t
    const int t = (int)(tok % L);          // position inside the sequence (the conv is causal per sequence)
    const int conv_groups = (di + 2 * GN) / 8, qe_groups = (GN + GP) / 8;
    const int i = blockIdx.y * blockDim.x + threadIdx.x;
    const float* row = zx + tok * ldz;
    if (tok == 0 && i < H) A[i] = -expf(A_log[i]);
    if (i < conv_groups) {
        const int c0 = 8 * i;  // channel within x | B | C
        float acc[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] = conv_b[c0 + e];
        for (int k = 0; k < W; ++k) {  // tap k reads the token W - 1 - k steps back
            const int back = W - 1 - k;
            if (t - back < 0) continue;
            const float4 u0 = *reinterpret_cast<const float4*>(row - (i64)back * ldz + di + c0);
            const float4 u1 = *reinterpret_cast<const float4*>(row - (i64)back * ldz + di + c0 + 4);
            const float v[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[e] = fmaf(conv_w[(c0 + e) * W + k], v[e], acc[e]);
        }
        uint32_t o[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const __nv_bfloat162 p = __floats2bfloat162_rn(silu_f32(acc[2 * e]), silu_f32(acc[2 * e + 1]));
            o[e] = *reinterpret_cast<const uint32_t*>(&p);
        }
        __nv_bfloat16* dst = c0 < di ? X + tok * di + c0
                           : c0 < di + GN ? Bm + tok * GN + (c0 - di)
                                          : Cm + tok * GN + (c0 - di - GN);
        *reinterpret_cast<uint4*>(dst) = make_uint4(o[0], o[1], o[2], o[3]);
    } else if (i < conv_groups + qe_groups) {
        const int c0 = 8 * (i - conv_groups);  // channel within Q | E
        float v[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = row[2 * di + 2 * GN + H + c0 + e];
        __nv_bfloat16* dst = c0 < GN ? Q + tok * GN + c0 : E + tok * GP + (c0 - GN);
        store_row8(dst, v);
    } else if (i < conv_groups + qe_groups + H) {
        const int h = i - conv_groups - qe_groups;
        const float raw = row[2 * di + 2 * GN + h] + dt_bias[h];
        dt[tok * H + h] = raw > 20.0f ? raw : log1pf(expf(raw));  // softplus
        gate[tok * H + h] = __float2bfloat16_rn(row[2 * di + 2 * GN + H + GN + GP]);  // the token's gate logit
    }
}

// y = Y + D_h x, g = y SiLU(z), yn = g / sqrt(mean(g^2) + eps) w over d_inner, bf16.
// One block of 256 threads per token, 8 consecutive channels per thread and step.
__global__ void __launch_bounds__(256)
block_norm_kernel(const float* __restrict__ Y, const __nv_bfloat16* __restrict__ X,
                  const float* __restrict__ zx, int ldz, const float* __restrict__ D,
                  const float* __restrict__ norm_w, __nv_bfloat16* __restrict__ yn, int di, int P,
                  float eps) {
    const i64 tok = blockIdx.x;
    __shared__ float red[8];
    constexpr int kMaxPer = 4;  // up to 4 x 8 x 256 = 8192 channels
    float g[kMaxPer][8];
    float ss = 0.0f;
#pragma unroll
    for (int s = 0; s < kMaxPer; ++s) {
        const int c0 = 8 * (threadIdx.x + 256 * s);
        if (c0 >= di) continue;
        const float4 y0 = *reinterpret_cast<const float4*>(Y + tok * di + c0);
        const float4 y1 = *reinterpret_cast<const float4*>(Y + tok * di + c0 + 4);
        const float yv[8] = {y0.x, y0.y, y0.z, y0.w, y1.x, y1.y, y1.z, y1.w};
        float xv[8];
        load_row8(X + tok * di + c0, xv);
        const float4 z0 = *reinterpret_cast<const float4*>(zx + tok * ldz + c0);  // z: the first column block
        const float4 z1 = *reinterpret_cast<const float4*>(zx + tok * ldz + c0 + 4);
        const float zv[8] = {z0.x, z0.y, z0.z, z0.w, z1.x, z1.y, z1.z, z1.w};
        const float d = D[c0 / P];  // 8 channels never straddle heads (P % 8 == 0)
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            g[s][e] = fmaf(d, xv[e], yv[e]) * silu_f32(zv[e]);
            ss = fmaf(g[s][e], g[s][e], ss);
        }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.0f;
#pragma unroll
    for (int w = 0; w < 8; ++w) tot += red[w];
    const float inv = rsqrtf(tot / (float)di + eps);
#pragma unroll
    for (int s = 0; s < kMaxPer; ++s) {
        const int c0 = 8 * (threadIdx.x + 256 * s);
        if (c0 >= di) continue;
        uint32_t o[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const __nv_bfloat162 p = __floats2bfloat162_rn(g[s][2 * e] * inv * norm_w[c0 + 2 * e],
                                                           g[s][2 * e + 1] * inv * norm_w[c0 + 2 * e + 1]);
            o[e] = *reinterpret_cast<const uint32_t*>(&p);
        }
        *reinterpret_cast<uint4*>(yn + tok * di + c0) = make_uint4(o[0], o[1], o[2], o[3]);
    }
}

}  // namespace

cudaError_t launch_block_conv_split(const BlockArgs& a, cudaStream_t stream) {
    const int di = (int)(a.H * a.P), GN = (int)(a.G * a.N), GP = (int)(a.G * a.P);
    const int items = (di + 2 * GN) / 8 + (GN + GP) / 8 + (int)a.H;
    const dim3 grid((unsigned)(a.B * a.L), (unsigned)((items + 127) / 128));
    block_conv_split_kernel<<<grid, 128, 0, stream>>>(
        (const float*)a.zx, (int)a.ldz, (int)a.L, di, GN, GP, (int)a.H, (int)a.conv_width, a.conv_w,
        a.conv_b, a.dt_bias, a.A_log, (__nv_bfloat16*)a.X, (__nv_bfloat16*)a.Bm, (__nv_bfloat16*)a.Cm, a.dt,
        a.A, (__nv_bfloat16*)a.Q, (__nv_bfloat16*)a.E, (__nv_bfloat16*)a.gate);
    note_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_block_norm(const BlockArgs& a, cudaStream_t stream) {
    const int di = (int)(a.H * a.P);
    if (di > 8 * 256 * 4) return cudaErrorInvalidValue;
    block_norm_kernel<<<(unsigned)(a.B * a.L), 256, 0, stream>>>(
        a.Y, (const __nv_bfloat16*)a.X, (const float*)a.zx, (int)a.ldz, a.D, a.norm_w,
        (__nv_bfloat16*)a.yn, di, (int)a.P, a.norm_eps);
    note_launches(1);
    return cudaGetLastError();
}

bool block_conv_width_ok(int64_t w) { return w >= 1 && w <= kMaxConv; }

}  // namespace dart
