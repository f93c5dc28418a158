// Backward of the chunked SSD scan, FFMA path. The paper prints no backward;
// this is the chain rule on the chunked forms of App. A (Sec. 2 selective SSM,
// Sec. 3 chunk memories):
//   L[t,s] = exp(cum_t - cum_s) (s <= t in one chunk), W = L (C B^T) dt_s,
//   Y_t    = sum_s W[t,s] X_s + exp(cum_t) C_t H_[c-1],
//   dH_c   = sum_s exp(cum_end - cum_s) dt_s B_s^T X_s   (the chunk memory M_c),
//   H_c    = exp(cum_end) H_[c-1] + dH_c,   cum = within-chunk cumsum of dt A.
// Kernels:
//   1. scan_bwd_inter_kernel: Z_c = sum_{t in c} exp(cum_t) C_t^T dY_t, the
//      adjoint H_[c-1] receives from chunk c's outputs;
//   2. scan_bwd_passing_kernel: reverse over chunks, adjoint of H_c:
//      A_c = A_{c+1}-side; d(dH_c) = A_c + dM_c; A_{c-1} = Z_c + exp(cum_end) A_c,
//      and d(cum_end_c) gets exp(cum_end) <A_c, H_[c-1]>;
//   3. scan_bwd_chunk_kernel, one block per (c, h, b): pass A over 32-token
//      target blocks gives dC_t (intra + inter) and the row part of d(cum_t);
//      pass B over 32-token source blocks gives dX_s, dB_s, the multiplier part
//      of d(dt_s) and the column part of d(cum); then d(dA) is the reverse
//      cumsum of d(cum) over the chunk, d(dt) += A_h d(dA), dA_h += dt d(dA).
// B and C are shared by the heads of a group: dB and dC are summed with fp32
// atomics (dC on top of what the caller already holds, e.g. the SMA part).
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dart {
namespace {

constexpr int kTB = 32;  // tokens per block

// Z_c[n,p] = sum_{t in c} exp(cum_t) C_t[n] dY_t[p]; one block per (c, h, b),
// thread owns (n, p) pairs e = tid + 256 k.
template <typename Tin>
__global__ void __launch_bounds__(256)
scan_bwd_inter_kernel(const Tin* __restrict__ Cm, const Tin* __restrict__ dY,
                      const float* __restrict__ cum, float* __restrict__ Z, int L, int H, int G,
                      int P, int N, int S, int Mc) {
    __shared__ float sC[kTB][129];
    __shared__ float sY[kTB][65];
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int g = h / (H / G);
    const int tid = threadIdx.x;
    const int NP = N * P;
    const float* cumc = cum + (((i64)b * H + h) * Mc + c) * S;
    float acc[32];
#pragma unroll
    for (int k = 0; k < 32; ++k) acc[k] = 0.0f;
    for (int s0 = 0; s0 < S; s0 += kTB) {
        __syncthreads();
        for (int e = tid; e < kTB * N; e += 256) {
            const int r = e / N, n = e % N;
            const i64 row = (i64)b * L + (i64)c * S + s0 + r;
            sC[r][n] = (s0 + r < S) ? expf(cumc[s0 + r]) * ld_f32(Cm + (row * G + g) * N + n) : 0.0f;
        }
        for (int e = tid; e < kTB * P; e += 256) {
            const int r = e / P, p = e % P;
            const i64 row = (i64)b * L + (i64)c * S + s0 + r;
            sY[r][p] = (s0 + r < S) ? ld_f32(dY + (row * H + h) * P + p) : 0.0f;
        }
        __syncthreads();
        for (int r = 0; r < kTB; ++r) {
#pragma unroll
            for (int k = 0; k < 32; ++k) {
                const int e = tid + 256 * k;
                if (e < NP) acc[k] = fmaf(sC[r][e / P], sY[r][e % P], acc[k]);
            }
        }
    }
    float* Zc = Z + (((i64)b * Mc + c) * H + h) * NP;
#pragma unroll
    for (int k = 0; k < 32; ++k) {
        const int e = tid + 256 * k;
        if (e < NP) Zc[e] = acc[k];
    }
}

// Reverse pass over chunks for each (b, h, element): ZD holds Z on entry and
// d(dH_c) on exit. dcum_end[b,h,c] += exp(cum_end) <A_c, H_[c-1]>. With Dops
// (P = 64), d(dH_c) is also written as bf16 hi | lo tiles in the 128-byte
// swizzled layout of the tensor-core kernels (32 KiB per (b, c, h)).
__global__ void scan_bwd_passing_kernel(float* __restrict__ ZD, const float* __restrict__ dM,
                                        const float* __restrict__ Hprev,
                                        const float* __restrict__ cum,
                                        float* __restrict__ dcum_end, uint8_t* __restrict__ Dops,
                                        int H, int S, int Mc, int NP) {
    const int e = blockIdx.x * blockDim.x + threadIdx.x;
    const int h = blockIdx.y, b = blockIdx.z;
    const float* cumh = cum + ((i64)b * H + h) * Mc * S;
    float adj = 0.0f;  // adjoint of H_c (nothing after the last chunk)
    for (int c = Mc - 1; c >= 0; --c) {
        const i64 idx = (((i64)b * Mc + c) * H + h) * NP + e;
        const float dec = expf(cumh[(i64)c * S + S - 1]);
        float part = 0.0f;
        if (e < NP) {
            const float z = ZD[idx];
            const float dmv = dM != nullptr ? dM[idx] : 0.0f;
            part = dec * adj * Hprev[idx];
            const float dd = adj + dmv;
            ZD[idx] = dd;
            if (Dops != nullptr) {
                const int n = e >> 6, p = e & 63;
                const uint32_t o = ((uint32_t)n * 128u + (uint32_t)p * 2u) ^ (((uint32_t)n & 7u) << 4);
                uint8_t* tile = Dops + (((i64)b * Mc + c) * H + h) * 32768;
                const __nv_bfloat16 hi = __float2bfloat16_rn(dd);
                *reinterpret_cast<__nv_bfloat16*>(tile + o) = hi;
                *reinterpret_cast<__nv_bfloat16*>(tile + 16384 + o) = __float2bfloat16_rn(dd - __bfloat162float(hi));
            }
            adj = fmaf(dec, adj, z);
        }
        for (int off = 16; off > 0; off >>= 1) part += __shfl_xor_sync(0xffffffffu, part, off);
        if ((threadIdx.x & 31) == 0) atomicAdd(dcum_end + ((i64)b * H + h) * Mc + c, part);
    }
}

template <typename Tin>
__global__ void __launch_bounds__(256)
scan_bwd_chunk_kernel(const Tin* __restrict__ X, const float* __restrict__ dt,
                      const float* __restrict__ A, const Tin* __restrict__ Bm,
                      const Tin* __restrict__ Cm, const Tin* __restrict__ dY,
                      const float* __restrict__ cum, const float* __restrict__ Hprev,
                      const float* __restrict__ dDH, const float* __restrict__ dcum_end,
                      float* __restrict__ dX, float* __restrict__ ddt, float* __restrict__ dA,
                      float* __restrict__ dB, float* __restrict__ dC, int L, int H, int G, int P,
                      int N, int S, int Mc) {
    extern __shared__ float4 smem4[];
    float* smem = reinterpret_cast<float*>(smem4);
    float* sHm = smem;                    // [N][65] H_[c-1] (pass A) or d(dH_c) (pass B)
    float* sCt = sHm + N * 65;            // [32][129] C of the target block
    float* sBs = sCt + kTB * 129;         // [32][129] B of the source block
    float* sYt = sBs + kTB * 129;         // [32][65]  dY of the target block
    float* sXs = sYt + kTB * 65;          // [32][65]  X of the source block
    float* sW = sXs + kTB * 65;           // [32][33]  W[t,s]
    float* sDCB = sW + kTB * 33;          // [32][33]  d(CB)[t,s]
    float* sQ = sDCB + kTB * 33;          // [32][33]  q[t,s] = dW W
    float* sCum = sQ + kTB * 33;          // [S]
    float* sDt = sCum + S;                // [S]
    float* sDcum = sDt + S;               // [S] d(cum_t)
    float* sKap = sDcum + S;              // [32] kappa_s of the source block

    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int g = h / (H / G);
    const int tid = threadIdx.x;
    const int NP = N * P;
    const i64 tok0 = (i64)b * L + (i64)c * S;
    const float* cumc = cum + (((i64)b * H + h) * Mc + c) * S;
    const i64 hoff = (((i64)b * Mc + c) * H + h) * NP;
    for (int s = tid; s < S; s += 256) {
        sCum[s] = cumc[s];
        sDt[s] = dt[(tok0 + s) * H + h];
        sDcum[s] = 0.0f;
    }
    const float cum_end = cumc[S - 1];

    // rows of a 32-token block past the chunk end (S < 32) load as zero
    auto load_block = [&](float* dst, int ld, const Tin* src, i64 row_mul, i64 row_add, int width,
                          int blk) {
        for (int e = tid; e < kTB * width; e += 256) {
            const int r = e / width, k = e % width;
            dst[r * ld + k] = blk + r < S ? ld_f32(src + ((tok0 + blk + r) * row_mul + row_add) * width + k)
                                          : 0.0f;
        }
    };
    // W, d(CB), q for the block pair (tb, sb): rows t, cols s
    auto pair_terms = [&](int tb, int sb) {
        for (int e = tid; e < kTB * kTB; e += 256) {
            const int r = e >> 5, k = e & 31;
            const int t = tb + r, s = sb + k;
            float cb = 0.0f, dw = 0.0f;
            const bool live = s <= t && t < S;
            if (live) {
                for (int n = 0; n < N; ++n) cb = fmaf(sCt[r * 129 + n], sBs[k * 129 + n], cb);
                for (int p = 0; p < P; ++p) dw = fmaf(sYt[r * 65 + p], sXs[k * 65 + p], dw);
            }
            const float lts = live ? expf(sCum[t] - sCum[s]) : 0.0f;
            const float dts = live ? sDt[s] : 0.0f;
            const float w = lts * cb * dts;
            sW[r * 33 + k] = w;
            sDCB[r * 33 + k] = dw * lts * dts;
            sQ[r * 33 + k] = dw * w;
        }
    };

    // ---- pass A: target blocks; dC_t (intra + inter), d(cum_t) row part
    for (int i = tid; i < N * 64; i += 256) {
        const int n = i >> 6, p = i & 63;
        sHm[n * 65 + p] = p < P ? Hprev[hoff + (i64)n * P + p] : 0.0f;
    }
    for (int tb = 0; tb < S; tb += kTB) {
        __syncthreads();
        load_block(sCt, 129, Cm, G, g, N, tb);
        load_block(sYt, 65, dY, H, h, P, tb);
        __syncthreads();
        // inter: hd_t = H dY_t; dC_t = exp(cum_t) hd_t; d(cum_t) += exp(cum_t) C_t . hd_t
        float dCa[16];
        const int r = tid >> 3;  // target row of this thread
#pragma unroll
        for (int k = 0; k < 16; ++k) {
            const int n = (tid & 7) + 8 * k;
            float hd = 0.0f;
            if (n < N)
                for (int p = 0; p < P; ++p) hd = fmaf(sHm[n * 65 + p], sYt[r * 65 + p], hd);
            dCa[k] = (c > 0 && tb + r < S) ? expf(sCum[tb + r]) * hd : 0.0f;
        }
        {
            float part = 0.0f;
#pragma unroll
            for (int k = 0; k < 16; ++k) {
                const int n = (tid & 7) + 8 * k;
                if (n < N) part = fmaf(sCt[r * 129 + n], dCa[k], part);
            }
            for (int off = 4; off > 0; off >>= 1) part += __shfl_xor_sync(0xffffffffu, part, off);
            if ((tid & 7) == 0 && tb + r < S) atomicAdd(&sDcum[tb + r], part);
        }
        // intra: source blocks sb <= tb
        for (int sb = 0; sb <= tb; sb += kTB) {
            __syncthreads();
            load_block(sBs, 129, Bm, G, g, N, sb);
            load_block(sXs, 65, X, H, h, P, sb);
            __syncthreads();
            pair_terms(tb, sb);
            __syncthreads();
            // dC_t += sum_s dCB[t,s] B_s ; d(cum_t) += sum_s q[t,s]
#pragma unroll
            for (int k = 0; k < 16; ++k) {
                const int n = (tid & 7) + 8 * k;
                if (n >= N) continue;
                float acc = dCa[k];
                for (int s = 0; s < kTB; ++s) acc = fmaf(sDCB[r * 33 + s], sBs[s * 129 + n], acc);
                dCa[k] = acc;
            }
            if (tid < kTB && tb + tid < S) {
                float qs = 0.0f;
                for (int s = 0; s < kTB; ++s) qs += sQ[tid * 33 + s];
                sDcum[tb + tid] += qs;
            }
        }
        if (tb + r < S) {
#pragma unroll
            for (int k = 0; k < 16; ++k) {
                const int n = (tid & 7) + 8 * k;
                if (n < N) atomicAdd(dC + ((tok0 + tb + r) * G + g) * N + n, dCa[k]);
            }
        }
    }

    // ---- pass B: source blocks; dX_s, dB_s, d(dt_s) multiplier part, d(cum_s) column part
    __syncthreads();
    for (int i = tid; i < N * 64; i += 256) {
        const int n = i >> 6, p = i & 63;
        sHm[n * 65 + p] = p < P ? dDH[hoff + (i64)n * P + p] : 0.0f;
    }
    float kap_sum = 0.0f;
    for (int sb = 0; sb < S; sb += kTB) {
        __syncthreads();
        load_block(sBs, 129, Bm, G, g, N, sb);
        load_block(sXs, 65, X, H, h, P, sb);
        __syncthreads();
        const int r = tid >> 3;  // source row of this thread
        const int s = sb + r;
        const bool srow = s < S;
        const float ws = srow ? expf(cum_end - sCum[s]) * sDt[s] : 0.0f;
        // memory term: dX_s += w_s B_s d(dH); dB_s += w_s d(dH) X_s; kappa_s = w_s B_s d(dH) X_s
        float dXa[8], dBa[16];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int p = (tid & 7) + 8 * k;
            float acc = 0.0f;
            if (p < P)
                for (int n = 0; n < N; ++n) acc = fmaf(sBs[r * 129 + n], sHm[n * 65 + p], acc);
            dXa[k] = ws * acc;
        }
        float kap = 0.0f;
#pragma unroll
        for (int k = 0; k < 16; ++k) {
            const int n = (tid & 7) + 8 * k;
            float acc = 0.0f;
            if (n < N)
                for (int p = 0; p < P; ++p) acc = fmaf(sHm[n * 65 + p], sXs[r * 65 + p], acc);
            dBa[k] = ws * acc;
            if (n < N) kap = fmaf(sBs[r * 129 + n], acc, kap);
        }
        for (int off = 4; off > 0; off >>= 1) kap += __shfl_xor_sync(0xffffffffu, kap, off);
        kap *= ws;  // kappa_s
        const float ddt_mult = ((tid & 7) == 0 && srow && sDt[s] != 0.0f) ? kap / sDt[s] : 0.0f;
        if ((tid & 7) == 0) {
            sKap[r] = kap;
            kap_sum += kap;
        }
        // intra: target blocks tb >= sb
        float qcol = 0.0f, wcb = 0.0f;  // sum_t q[t,s], sum_t dW L CB (on the tid & 7 == 0 lane)
        for (int tb = sb; tb < S; tb += kTB) {
            __syncthreads();
            load_block(sCt, 129, Cm, G, g, N, tb);
            load_block(sYt, 65, dY, H, h, P, tb);
            __syncthreads();
            pair_terms(tb, sb);
            __syncthreads();
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const int p = (tid & 7) + 8 * k;
                if (p >= P) continue;
                float acc = dXa[k];
                for (int t = 0; t < kTB; ++t) acc = fmaf(sW[t * 33 + r], sYt[t * 65 + p], acc);
                dXa[k] = acc;
            }
#pragma unroll
            for (int k = 0; k < 16; ++k) {
                const int n = (tid & 7) + 8 * k;
                if (n >= N) continue;
                float acc = dBa[k];
                for (int t = 0; t < kTB; ++t) acc = fmaf(sDCB[t * 33 + r], sCt[t * 129 + n], acc);
                dBa[k] = acc;
            }
            if ((tid & 7) == 0 && srow) {
                for (int t = 0; t < kTB; ++t) {
                    qcol += sQ[t * 33 + r];
                    // dW L CB = q / dt_s (q = dW W, W = L CB dt_s)
                    wcb += sDt[s] != 0.0f ? sQ[t * 33 + r] / sDt[s] : 0.0f;
                }
            }
        }
        if (!srow) continue;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int p = (tid & 7) + 8 * k;
            if (p < P) dX[((tok0 + s) * H + h) * P + p] = dXa[k];
        }
#pragma unroll
        for (int k = 0; k < 16; ++k) {
            const int n = (tid & 7) + 8 * k;
            if (n < N) atomicAdd(dB + ((tok0 + s) * G + g) * N + n, dBa[k]);
        }
        if ((tid & 7) == 0) {
            ddt[(tok0 + s) * H + h] = ddt_mult + wcb;  // multiplier part; decay part added below
            atomicAdd(&sDcum[s], -(qcol + kap));
        }
    }
    // d(cum_end) += sum_s kappa_s + exp(cum_end) <A_c, H_[c-1]>
    for (int off = 16; off > 0; off >>= 1) kap_sum += __shfl_xor_sync(0xffffffffu, kap_sum, off);
    __syncthreads();
    if ((tid & 31) == 0) atomicAdd(&sDcum[S - 1], kap_sum);
    if (tid == 0) atomicAdd(&sDcum[S - 1], dcum_end[((i64)b * H + h) * Mc + c]);
    __syncthreads();
    // d(dA_u) = sum_{t >= u} d(cum_t); d(dt_u) += A_h d(dA_u); dA_h += dt_u d(dA_u)
    if (tid == 0) {
        float run = 0.0f, da = 0.0f;
        const float Ah = A[h];
        for (int u = S - 1; u >= 0; --u) {
            run += sDcum[u];
            const i64 di = (tok0 + u) * H + h;
            ddt[di] += Ah * run;
            da = fmaf(sDt[u], run, da);
        }
        atomicAdd(dA + h, da);
    }
}

}  // namespace

size_t scan_bwd_workspace(int64_t B, int64_t L, int64_t H, int64_t N, int64_t P, int64_t S) {
    const int64_t M = L / S;
    auto al = [](size_t x) { return (x + 255) & ~(size_t)255; };
    return al((size_t)(B * H * M * S) * sizeof(float))          // cum
           + 2 * al((size_t)(B * M * H * N * P) * sizeof(float)) // H_[c-1]; Z / d(dH)
           + al((size_t)(B * H * M) * sizeof(float));           // d(cum_end)
}

cudaError_t launch_scan_bwd_passing(float* ZD, const float* dM, const float* Hprev, const float* cum,
                                    float* dcum_end, uint8_t* Dops, int B, int H, int S, int Mc,
                                    int NP, cudaStream_t stream) {
    scan_bwd_passing_kernel<<<dim3((NP + 255) / 256, H, B), 256, 0, stream>>>(
        ZD, dM, Hprev, cum, dcum_end, Dops, H, S, Mc, NP);
    note_launches(1);
    return cudaGetLastError();
}

// The backward's output-kernel modes run 128-token tiles inside a chunk: S in {128, 256}.
bool scan_bwd_tc_supported(const ScanArgs& f) { return f.G == 1 && f.S >= 128 && scan_tc_supported(f); }

template <typename Tin>
cudaError_t launch_chunk_scan_backward(const ScanBwdArgs& a, void* ws, unsigned long long wait_limit_ns,
                                       cudaStream_t stream) {
    const ScanArgs& f = a.fwd;
    const int B = (int)f.B, L = (int)f.L, H = (int)f.H, G = (int)f.G, P = (int)f.P,
              N = (int)f.N, S = (int)f.S, Mc = L / S, NP = N * P;
    auto al = [](size_t x) { return (x + 255) & ~(size_t)255; };
    uint8_t* w = (uint8_t*)ws;
    float* cum = (float*)w;
    w += al((size_t)(f.B * f.H * Mc * f.S) * sizeof(float));
    float* Hprev = (float*)w;
    w += al((size_t)(f.B * Mc * f.H) * NP * sizeof(float));
    float* ZD = (float*)w;
    w += al((size_t)(f.B * Mc * f.H) * NP * sizeof(float));
    float* dcum_end = (float*)w;

    // bf16 inputs at the tensor-core shapes with G = 1: the whole backward on the tensor
    // cores; other bf16 inputs at those shapes: the state recompute and Z_c there
    if (sizeof(Tin) == 2 && scan_bwd_tc_supported(f))
        return launch_chunk_scan_backward_tc(a, ws, wait_limit_ns, stream);
    const bool tc = sizeof(Tin) == 2 && scan_tc_supported(f);
    // recompute cum and the state entering every chunk (forward kernels)
    cudaError_t e = tc ? launch_scan_states_tc(a.fwd, cum, Hprev, nullptr, wait_limit_ns, stream)
                       : launch_scan_states<Tin>(a.fwd, cum, Hprev, ZD, stream);
    if (e != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(dcum_end, 0, (size_t)(f.B * f.H * Mc) * sizeof(float), stream)) != cudaSuccess)
        return e;
    if ((e = cudaMemsetAsync(a.dA, 0, (size_t)f.H * sizeof(float), stream)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(a.dB, 0, (size_t)(f.B * f.L * f.G * f.N) * sizeof(float), stream)) != cudaSuccess)
        return e;
    if (!a.accumulate_dC &&
        (e = cudaMemsetAsync(a.dC, 0, (size_t)(f.B * f.L * f.G * f.N) * sizeof(float), stream)) != cudaSuccess)
        return e;
    if (tc) {
        if ((e = launch_scan_bwd_inter_tc(f, cum, a.dY, ZD, wait_limit_ns, stream)) != cudaSuccess) return e;
    } else {
        scan_bwd_inter_kernel<Tin><<<dim3(Mc, H, B), 256, 0, stream>>>(
            (const Tin*)a.fwd.Cm, (const Tin*)a.dY, cum, ZD, L, H, G, P, N, S, Mc);
        note_launches(1);
    }
    scan_bwd_passing_kernel<<<dim3((NP + 255) / 256, H, B), 256, 0, stream>>>(
        ZD, a.dM, Hprev, cum, dcum_end, nullptr, H, S, Mc, NP);
    const size_t smem = (size_t)(N * 65 + 2 * kTB * 129 + 2 * kTB * 65 + 3 * kTB * 33 + 3 * S + kTB) *
                        sizeof(float);
    auto k3 = scan_bwd_chunk_kernel<Tin>;
    if ((e = cudaFuncSetAttribute(k3, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) != cudaSuccess)
        return e;
    k3<<<dim3(Mc, H, B), 256, smem, stream>>>(
        (const Tin*)a.fwd.X, a.fwd.dt, a.fwd.A, (const Tin*)a.fwd.Bm, (const Tin*)a.fwd.Cm,
        (const Tin*)a.dY, cum, Hprev, ZD, dcum_end, a.dX, a.ddt, a.dA, a.dB, a.dC, L, H, G, P, N, S,
        Mc);
    note_launches(2);
    return cudaGetLastError();
}

typedef __nv_bfloat16 bf16;
template cudaError_t launch_chunk_scan_backward<float>(const ScanBwdArgs&, void*, unsigned long long,
                                                       cudaStream_t);
template cudaError_t launch_chunk_scan_backward<bf16>(const ScanBwdArgs&, void*, unsigned long long,
                                                      cudaStream_t);

}  // namespace dart
