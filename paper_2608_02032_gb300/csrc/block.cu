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

#include <type_traits>

#include <cuda_bf16.h>

#include "common.cuh"
#include "dart.h"
#include "kernels.h"

namespace dart {
namespace {

constexpr int kMaxConv = 8;

// The convolution of the in-projection's x, B, C blocks (columns di .. di + conv_ch
// of zx). A block of 256 threads covers 128 channels x 128 tokens: warp r takes the
// tokens tok0 + 16 r .. + 15, lane c the channels 4 c .. 4 c + 3 of the block's range
// (a warp's loads of one row are 512 contiguous bytes). Each thread loads the W - 1
// rows before its first token and its 16 rows up front, all in flight at once, and
// keeps its channels' taps in registers. A group of 4 channels never straddles x, B
// and C (di and GN are multiples of 4).
constexpr int kConvTok = 16, kConvWarps = 8, kConvCh = 128;
template <int W>
__global__ void __launch_bounds__(256)
block_conv_kernel(const float* __restrict__ zx, int ldz, int64_t T, int L, int di, int conv_ch,
                  const float* __restrict__ conv_w, const float* __restrict__ conv_b,
                  __nv_bfloat16* __restrict__ X, __nv_bfloat16* __restrict__ Bm, __nv_bfloat16* __restrict__ Cm,
                  int GN) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int c0 = kConvCh * blockIdx.y + 4 * lane;  // channel within x | B | C
    if (c0 >= conv_ch) return;
    const i64 tok0 = ((i64)blockIdx.x * kConvWarps + warp) * kConvTok;
    if (tok0 >= T) return;
    float w[4][W], bias[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        bias[e] = conv_b[c0 + e];
#pragma unroll
        for (int k = 0; k < W; ++k) w[e][k] = conv_w[(c0 + e) * W + k];
    }
    __nv_bfloat16* dst = c0 < di ? X + c0 : c0 < di + GN ? Bm + (c0 - di) : Cm + (c0 - di - GN);
    const int ld_dst = c0 < di ? di : GN;
    // v[r] holds the row of token tok0 - (W - 1) + r (zeros outside 0 .. T - 1)
    constexpr int kR = W - 1 + kConvTok;
    float4 v[kR];
#pragma unroll
    for (int r = 0; r < kR; ++r) {
        const i64 tk = tok0 - (W - 1) + r;
        v[r] = tk >= 0 && tk < T ? *reinterpret_cast<const float4*>(zx + tk * ldz + di + c0)
                                 : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    }
    const int t0 = (int)(tok0 % L);
#pragma unroll
    for (int i = 0; i < kConvTok; ++i) {
        if (tok0 + i >= T) break;
        const int pos = (t0 + i) % L;  // position in its sequence: taps further back read zeros
        float acc[4] = {bias[0], bias[1], bias[2], bias[3]};
#pragma unroll
        for (int k = 0; k < W; ++k) {
            if (W - 1 - k <= pos) {
                const float4 x = v[i + k];
                acc[0] = fmaf(w[0][k], x.x, acc[0]);
                acc[1] = fmaf(w[1][k], x.y, acc[1]);
                acc[2] = fmaf(w[2][k], x.z, acc[2]);
                acc[3] = fmaf(w[3][k], x.w, acc[3]);
            }
        }
        const __nv_bfloat162 lo = __floats2bfloat162_rn(silu_f32(acc[0]), silu_f32(acc[1]));
        const __nv_bfloat162 hi = __floats2bfloat162_rn(silu_f32(acc[2]), silu_f32(acc[3]));
        uint2 o;
        o.x = *reinterpret_cast<const uint32_t*>(&lo);
        o.y = *reinterpret_cast<const uint32_t*>(&hi);
        *reinterpret_cast<uint2*>(dst + (tok0 + i) * ld_dst) = o;
    }
}

// Q and E (copies to bf16), dt = softplus(dt + dt_bias) and the gate logit for every
// head: one warp per token. Columns of zx: z [0, di), x [di, 2 di), B, C (GN each),
// dt (H), Q (GN), E (GP), gate (1).
__global__ void __launch_bounds__(256)
block_split_kernel(const float* __restrict__ zx, int ldz, int64_t T, int di, int GN, int GP, int H,
                   const float* __restrict__ dt_bias, const float* __restrict__ A_log, float* __restrict__ dt,
                   float* __restrict__ A, __nv_bfloat16* __restrict__ Q, __nv_bfloat16* __restrict__ E,
                   __nv_bfloat16* __restrict__ gate) {
    const i64 tok = (i64)blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (tok == 0 && lane < H) A[lane] = -expf(A_log[lane]);
    if (tok == 0 && H > 32)
        for (int h = 32 + lane; h < H; h += 32) A[h] = -expf(A_log[h]);
    if (tok >= T) return;
    const float* row = zx + tok * ldz;
    const int o_dt = 2 * di + 2 * GN, o_q = o_dt + H, o_g = o_q + GN + GP;
    for (int c = lane; c < GN + GP; c += 32) {
        const __nv_bfloat16 v = __float2bfloat16_rn(row[o_q + c]);
        if (c < GN) Q[tok * GN + c] = v;
        else E[tok * GP + (c - GN)] = v;
    }
    const __nv_bfloat16 g = __float2bfloat16_rn(row[o_g]);  // the token's one gate logit
    for (int h = lane; h < H; h += 32) {
        const float raw = row[o_dt + h] + dt_bias[h];
        dt[tok * H + h] = raw > 20.0f ? raw : log1pf(expf(raw));  // softplus
        gate[tok * H + h] = g;
    }
}

// y = Y + D_h x, g = y SiLU(z), yn = g / sqrt(mean(g^2) + eps) w over d_inner, bf16:
// one warp per token (4 per block), lane l taking the 8-channel groups l, l + 32, ...
// (at most kNormGroups per lane, kept in registers between the two passes:
// d_inner <= kNormGroups x 32 x 8).
template <int kNormGroups>
__global__ void __launch_bounds__(128)
block_norm_kernel(const float* __restrict__ Y, const __nv_bfloat16* __restrict__ X,
                  const float* __restrict__ zx, int ldz, const float* __restrict__ D,
                  const float* __restrict__ norm_w, __nv_bfloat16* __restrict__ yn, int64_t T, int di, int P,
                  float eps) {
    const i64 tok = (i64)blockIdx.x * 4 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (tok >= T) return;
    const int groups = di / 8;
    float g[kNormGroups][8];
    float ss = 0.0f;
    // every group of the lane: no early exit, so that all its loads are in flight together
#pragma unroll
    for (int j = 0; j < kNormGroups; ++j) {
        const int q = lane + 32 * j;
        const bool live = q < groups;
        const int c0 = live ? 8 * q : 0;
        const float4 zero = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        const float4 y0 = live ? *reinterpret_cast<const float4*>(Y + tok * di + c0) : zero;
        const float4 y1 = live ? *reinterpret_cast<const float4*>(Y + tok * di + c0 + 4) : zero;
        const float4 z0 = live ? *reinterpret_cast<const float4*>(zx + tok * ldz + c0) : zero;  // z: the first block
        const float4 z1 = live ? *reinterpret_cast<const float4*>(zx + tok * ldz + c0 + 4) : zero;
        const uint4 xr = live ? *reinterpret_cast<const uint4*>(X + tok * di + c0) : make_uint4(0u, 0u, 0u, 0u);
        const uint32_t xw[4] = {xr.x, xr.y, xr.z, xr.w};
        float xv[8];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&xw[e]));
            xv[2 * e] = f.x;
            xv[2 * e + 1] = f.y;
        }
        const float yv[8] = {y0.x, y0.y, y0.z, y0.w, y1.x, y1.y, y1.z, y1.w};
        const float zv[8] = {z0.x, z0.y, z0.z, z0.w, z1.x, z1.y, z1.z, z1.w};
        const float d = live ? D[c0 / P] : 0.0f;  // 8 channels never straddle heads (P % 8 == 0)
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            g[j][e] = fmaf(d, xv[e], yv[e]) * silu_f32(zv[e]);  // 0 for a dead group
            ss = fmaf(g[j][e], g[j][e], ss);
        }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    const float inv = rsqrtf(ss / (float)di + eps);
#pragma unroll
    for (int j = 0; j < kNormGroups; ++j) {
        const int q = lane + 32 * j;
        if (q >= groups) break;
        const int c0 = 8 * q;
        // norm_w is 16-byte aligned (checked by the entry point) and c0 a multiple of 8
        const float4 w0 = *reinterpret_cast<const float4*>(norm_w + c0);
        const float4 w1 = *reinterpret_cast<const float4*>(norm_w + c0 + 4);
        const float wv[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
        float o[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) o[e] = g[j][e] * inv * wv[e];
        store_row8(yn + tok * di + c0, o);
    }
}

}  // namespace

cudaError_t launch_block_conv_split(const BlockArgs& a, cudaStream_t stream) {
    const int di = (int)(a.H * a.P), GN = (int)(a.G * a.N), GP = (int)(a.G * a.P);
    const int64_t T = a.B * a.L;
    const int conv_ch = di + 2 * GN;
    constexpr int kBlockTok = kConvTok * kConvWarps;
    if ((T + kBlockTok - 1) / kBlockTok > 0x7fffffff) return cudaErrorInvalidValue;
    const dim3 grid((unsigned)((T + kBlockTok - 1) / kBlockTok), (unsigned)((conv_ch + kConvCh - 1) / kConvCh));
    auto conv = [&](auto kw) {
        block_conv_kernel<decltype(kw)::value><<<grid, 256, 0, stream>>>(
            (const float*)a.zx, (int)a.ldz, T, (int)a.L, di, conv_ch, a.conv_w, a.conv_b, (__nv_bfloat16*)a.X,
            (__nv_bfloat16*)a.Bm, (__nv_bfloat16*)a.Cm, GN);
    };
    switch (a.conv_width) {  // the taps live in registers: one instantiation per width
        case 1: conv(std::integral_constant<int, 1>{}); break;
        case 2: conv(std::integral_constant<int, 2>{}); break;
        case 3: conv(std::integral_constant<int, 3>{}); break;
        case 4: conv(std::integral_constant<int, 4>{}); break;
        case 5: conv(std::integral_constant<int, 5>{}); break;
        case 6: conv(std::integral_constant<int, 6>{}); break;
        case 7: conv(std::integral_constant<int, 7>{}); break;
        case 8: conv(std::integral_constant<int, 8>{}); break;
        default: return cudaErrorInvalidValue;
    }
    block_split_kernel<<<(unsigned)((T + 7) / 8), 256, 0, stream>>>(
        (const float*)a.zx, (int)a.ldz, T, di, GN, GP, (int)a.H, a.dt_bias, a.A_log, a.dt, a.A,
        (__nv_bfloat16*)a.Q, (__nv_bfloat16*)a.E, (__nv_bfloat16*)a.gate);
    note_launches(2);
    return cudaGetLastError();
}

cudaError_t launch_block_norm(const BlockArgs& a, cudaStream_t stream) {
    const int di = (int)(a.H * a.P);
    const int64_t T = a.B * a.L;
    if (di > 16 * 32 * 8) return cudaErrorInvalidValue;
    auto kern = di <= 8 * 32 * 8 ? block_norm_kernel<8> : block_norm_kernel<16>;
    kern<<<(unsigned)((T + 3) / 4), 128, 0, stream>>>(
        a.Y, (const __nv_bfloat16*)a.X, (const float*)a.zx, (int)a.ldz, a.D, a.norm_w, (__nv_bfloat16*)a.yn, T,
        di, (int)a.P, a.norm_eps);
    note_launches(1);
    return cudaGetLastError();
}

bool block_conv_width_ok(int64_t w) { return w >= 1 && w <= kMaxConv; }

}  // namespace dart
