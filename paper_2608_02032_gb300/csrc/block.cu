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
// of zx). A block of 256 threads covers 256 channels x 64 tokens: warp r takes the
// tokens tok0 + 8 r .. + 7, lane c the channels 8 c .. 8 c + 7 of the block's range
// (a warp's loads of one row are 1 KiB contiguous). Each thread keeps its channels'
// taps and a window of the last W input rows in registers, so every row is loaded
// once per thread: W - 1 rows before its first token, then one per token.
constexpr int kConvTok = 64, kConvCh = 256;
template <int W>
__global__ void __launch_bounds__(256)
block_conv_kernel(const float* __restrict__ zx, int ldz, int64_t T, int L, int di, int conv_ch,
                  const float* __restrict__ conv_w, const float* __restrict__ conv_b,
                  __nv_bfloat16* __restrict__ X, __nv_bfloat16* __restrict__ Bm, __nv_bfloat16* __restrict__ Cm,
                  int GN) {
    const int c0 = kConvCh * blockIdx.y + 8 * (threadIdx.x & 31);  // channel within x | B | C
    if (c0 >= conv_ch) return;
    const i64 tok0 = (i64)kConvTok * blockIdx.x + 8 * (threadIdx.x >> 5);
    if (tok0 >= T) return;
    float w[8][W], bias[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        bias[e] = conv_b[c0 + e];
#pragma unroll
        for (int k = 0; k < W; ++k) w[e][k] = conv_w[(c0 + e) * W + k];
    }
    __nv_bfloat16* dst = c0 < di ? X + c0 : c0 < di + GN ? Bm + (c0 - di) : Cm + (c0 - di - GN);
    const int ld_dst = c0 < di ? di : GN;
    auto load = [&](i64 tok, float (&v)[8]) {
        const float* src = zx + tok * ldz + di + c0;
        const float4 u0 = *reinterpret_cast<const float4*>(src);
        const float4 u1 = *reinterpret_cast<const float4*>(src + 4);
        v[0] = u0.x; v[1] = u0.y; v[2] = u0.z; v[3] = u0.w; v[4] = u1.x; v[5] = u1.y; v[6] = u1.z; v[7] = u1.w;
    };
    // win[k] holds the row of token tok - (W - 1) + k (zeros before the sequence start)
    float win[W][8];
    const int t0 = (int)(tok0 % L);
#pragma unroll
    for (int k = 0; k < W - 1; ++k) {
        const int back = W - 1 - k;
        if (t0 - back >= 0) {
            load(tok0 - back, win[k]);
        } else {
#pragma unroll
            for (int e = 0; e < 8; ++e) win[k][e] = 0.0f;
        }
    }
    const bool full = tok0 + 8 <= T;
    float nxt[4][8];  // the rows of four tokens, loaded together ahead of their arithmetic
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const i64 tok = tok0 + i;
        if ((i & 3) == 0) {
#pragma unroll
            for (int u = 0; u < 4; ++u)
                if (full || tok + u < T) load(tok + u, nxt[u]);
        }
        if (!full && tok >= T) break;
        if (i > 0 && (t0 + i) % L == 0) {  // a new sequence starts: nothing before it
#pragma unroll
            for (int k = 0; k < W - 1; ++k)
#pragma unroll
                for (int e = 0; e < 8; ++e) win[k][e] = 0.0f;
        }
#pragma unroll
        for (int e = 0; e < 8; ++e) win[W - 1][e] = nxt[i & 3][e];
        float acc[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            acc[e] = bias[e];
#pragma unroll
            for (int k = 0; k < W; ++k) acc[e] = fmaf(w[e][k], win[k][e], acc[e]);
            acc[e] = silu_f32(acc[e]);
        }
        store_row8(dst + tok * ld_dst, acc);
#pragma unroll
        for (int k = 0; k < W - 1; ++k)
#pragma unroll
            for (int e = 0; e < 8; ++e) win[k][e] = win[k + 1][e];
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
// one warp per token (8 per block), lane l taking the 8-channel groups l, l + 32, ...
// (at most kNormGroups per lane, kept in registers between the two passes:
// d_inner <= kNormGroups x 32 x 8).
template <int kNormGroups>
__global__ void __launch_bounds__(256)
block_norm_kernel(const float* __restrict__ Y, const __nv_bfloat16* __restrict__ X,
                  const float* __restrict__ zx, int ldz, const float* __restrict__ D,
                  const float* __restrict__ norm_w, __nv_bfloat16* __restrict__ yn, int64_t T, int di, int P,
                  float eps) {
    const i64 tok = (i64)blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (tok >= T) return;
    const int groups = di / 8;
    float g[kNormGroups][8];
    float ss = 0.0f;
#pragma unroll
    for (int j = 0; j < kNormGroups; ++j) {
        const int q = lane + 32 * j;
        if (q >= groups) break;
        const int c0 = 8 * q;
        const float4 y0 = *reinterpret_cast<const float4*>(Y + tok * di + c0);
        const float4 y1 = *reinterpret_cast<const float4*>(Y + tok * di + c0 + 4);
        const float4 z0 = *reinterpret_cast<const float4*>(zx + tok * ldz + c0);  // z: the first column block
        const float4 z1 = *reinterpret_cast<const float4*>(zx + tok * ldz + c0 + 4);
        float xv[8];
        load_row8(X + tok * di + c0, xv);
        const float yv[8] = {y0.x, y0.y, y0.z, y0.w, y1.x, y1.y, y1.z, y1.w};
        const float zv[8] = {z0.x, z0.y, z0.z, z0.w, z1.x, z1.y, z1.z, z1.w};
        const float d = D[c0 / P];  // 8 channels never straddle heads (P % 8 == 0)
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            g[j][e] = fmaf(d, xv[e], yv[e]) * silu_f32(zv[e]);
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
        float o[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) o[e] = g[j][e] * inv * norm_w[c0 + e];
        store_row8(yn + tok * di + c0, o);
    }
}

}  // namespace

cudaError_t launch_block_conv_split(const BlockArgs& a, cudaStream_t stream) {
    const int di = (int)(a.H * a.P), GN = (int)(a.G * a.N), GP = (int)(a.G * a.P);
    const int64_t T = a.B * a.L;
    const int conv_ch = di + 2 * GN;
    if ((T + kConvTok - 1) / kConvTok > 0x7fffffff) return cudaErrorInvalidValue;
    const dim3 grid((unsigned)((T + kConvTok - 1) / kConvTok), (unsigned)((conv_ch + kConvCh - 1) / kConvCh));
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
    kern<<<(unsigned)((T + 7) / 8), 256, 0, stream>>>(
        a.Y, (const __nv_bfloat16*)a.X, (const float*)a.zx, (int)a.ldz, a.D, a.norm_w, (__nv_bfloat16*)a.yn, T,
        di, (int)a.P, a.norm_eps);
    note_launches(1);
    return cudaGetLastError();
}

bool block_conv_width_ok(int64_t w) { return w >= 1 && w <= kMaxConv; }

}  // namespace dart
