// One decode step over the chunk-memory cache (the persistent inference cache
// of Sec. 4 "Inference Cache"; SMA of Sec. 3 / App. B.1 for one token).
//
// One block of 256 threads per (h, b):
//   phase 1  state <- a state + dt b^T x, partial likewise (reset at a chunk
//            start), y_ssd = c state; the completed chunk's partial is
//            appended to the cache when (pos + 1) % S == 0.
//   phase 2  the 8 warps split the i = pos / S completed memories. A warp
//            sweeps one memory with 16-byte loads, LPR lanes per row: each
//            row gives its key entry r_n (M_j Ebar)_n (reduced over the LPR
//            lanes) and adds c_n M_j[n, :] to the value; the warp then folds
//            (l_j, V_j) into its online-softmax state (m, d, O).
//   phase 3  the warps' partial softmaxes are merged; y = y_ssd + SiLU(z) R.
// The sweep is the HBM-bound part: the whole cache of (b, h) is read once.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dart {

constexpr int kDecThreads = 256;
constexpr int kDecWarps = kDecThreads / 32;

template <typename T> struct Vec16;
template <> struct Vec16<__nv_bfloat16> {
    static constexpr int n = 8;
    __device__ static void load(const __nv_bfloat16* p, float* out) {
        const uint4 u = __ldcs(reinterpret_cast<const uint4*>(p));  // streamed once
        const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __bfloat1622float2(h2[i]);
            out[2 * i] = f.x;
            out[2 * i + 1] = f.y;
        }
    }
};
template <> struct Vec16<float> {
    static constexpr int n = 4;
    __device__ static void load(const float* p, float* out) {
        const float4 f = __ldcs(reinterpret_cast<const float4*>(p));
        out[0] = f.x; out[1] = f.y; out[2] = f.z; out[3] = f.w;
    }
};

template <typename Tin, typename Tmem, typename Tout, int P>
__global__ void __launch_bounds__(kDecThreads)
decode_step_kernel(long long pos, int m_cap, Tmem* __restrict__ cache, float* __restrict__ state,
                   float* __restrict__ partial, const Tin* __restrict__ x,
                   const float* __restrict__ dt, const float* __restrict__ A,
                   const Tin* __restrict__ bv, const Tin* __restrict__ cv,
                   const Tin* __restrict__ qv, const Tin* __restrict__ ev,
                   const Tin* __restrict__ z, Tout* __restrict__ y, float* __restrict__ lse, int H,
                   int G, int N, int S, float eps) {
    constexpr int VEC = Vec16<Tmem>::n;
    constexpr int LPR = P / VEC;  // lanes per memory row
    constexpr int RPW = 32 / LPR; // rows per warp step
    static_assert(LPR >= 1 && LPR <= 32 && (32 % LPR) == 0, "unsupported P");

    __shared__ float sx[P], se[P], sb[128], sc[128], sq[128];
    __shared__ float sY[kDecThreads];
    __shared__ float sWm[kDecWarps], sWd[kDecWarps], sWO[kDecWarps][P];
    __shared__ float sRed[2];

    const int h = blockIdx.x, b = blockIdx.y, g = h / (H / G);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const i64 bh = (i64)b * H + h;
    const int NP = N * P;

    // per-token vectors; q and e are RMS-normalised (App. B.1)
    for (int i = tid; i < N; i += kDecThreads) {
        sb[i] = ld_f32(bv + ((i64)b * G + g) * N + i);
        sc[i] = ld_f32(cv + ((i64)b * G + g) * N + i);
        sq[i] = ld_f32(qv + ((i64)b * G + g) * N + i);
    }
    for (int i = tid; i < P; i += kDecThreads) {
        sx[i] = ld_f32(x + bh * P + i);
        se[i] = ld_f32(ev + ((i64)b * G + g) * P + i);
    }
    __syncthreads();
    if (warp < 2) {
        const float* v = warp == 0 ? sq : se;
        const int n = warp == 0 ? N : P;
        float ss = 0.0f;
        for (int i = lane; i < n; i += 32) ss = fmaf(v[i], v[i], ss);
        for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
        if (lane == 0) sRed[warp] = rsqrtf(ss / (float)n + eps);
    }
    __syncthreads();
    for (int i = tid; i < N; i += kDecThreads) sq[i] *= sRed[0];
    for (int i = tid; i < P; i += kDecThreads) se[i] *= sRed[1];
    __syncthreads();

    // phase 1: recurrent state, partial-chunk memory, y_ssd
    const float d = dt[bh];
    const float a = expf(d * A[h]);
    const bool chunk_start = (pos % S) == 0;
    const bool chunk_end = ((pos + 1) % S) == 0;
    const i64 ichunk = pos / S;
    float* St = state + bh * NP;
    float* Pt = partial + bh * NP;
    Tmem* slot = (chunk_end && ichunk < m_cap) ? cache + (((i64)b * m_cap + ichunk) * H + h) * NP
                                               : nullptr;
    // thread owns columns p = tid % P (kDecThreads % P == 0) and rows n = tid / P + k * rstep
    static_assert(kDecThreads % P == 0, "P must divide the block");
    const int p_own = tid % P;
    const int rstep = kDecThreads / P;
    float yp = 0.0f;
    for (int n = tid / P; n < N; n += rstep) {
        const int e = n * P + p_own;
        const float w = d * sb[n] * sx[p_own];
        const float hn = fmaf(a, St[e], w);
        const float pn = chunk_start ? w : fmaf(a, Pt[e], w);
        St[e] = hn;
        Pt[e] = pn;
        if (slot != nullptr) slot[e] = cvt_from_f32<Tmem>(pn);
        yp = fmaf(sc[n], hn, yp);
    }
    sY[tid] = yp;

    // phase 2: sweep the completed memories
    const int nhist = (int)(ichunk < (i64)m_cap ? ichunk : (i64)m_cap);
    const int p0 = (lane % LPR) * VEC;
    const int r0 = lane / LPR;
    float ev_reg[VEC];
#pragma unroll
    for (int v = 0; v < VEC; ++v) ev_reg[v] = se[p0 + v];
    const float inv_sqrt_n = rsqrtf((float)N);
    float m_w = -INFINITY, d_w = 0.0f, O_w[VEC];
#pragma unroll
    for (int v = 0; v < VEC; ++v) O_w[v] = 0.0f;

    for (int j = warp; j < nhist; j += kDecWarps) {
        const Tmem* Mj = cache + (((i64)b * m_cap + j) * H + h) * NP;
        float lacc = 0.0f, vacc[VEC];
#pragma unroll
        for (int v = 0; v < VEC; ++v) vacc[v] = 0.0f;
#pragma unroll 4
        for (int n = r0; n < N; n += RPW) {
            float val[VEC];
            Vec16<Tmem>::load(Mj + (i64)n * P + p0, val);
            float dot = 0.0f, ssq = 0.0f;
#pragma unroll
            for (int v = 0; v < VEC; ++v) {
                dot = fmaf(val[v], ev_reg[v], dot);
                ssq = fmaf(val[v], val[v], ssq);
            }
#pragma unroll
            for (int off = 1; off < LPR; off <<= 1) {
                dot += __shfl_xor_sync(0xffffffffu, dot, off);
                ssq += __shfl_xor_sync(0xffffffffu, ssq, off);
            }
            const float rn = rsqrtf(ssq / (float)P + eps);
            lacc = fmaf(sq[n], rn * dot, lacc);
            const float cn = sc[n];
#pragma unroll
            for (int v = 0; v < VEC; ++v) vacc[v] = fmaf(cn, val[v], vacc[v]);
        }
        // logit: one copy of each row's term lives in the LPR lanes of its group
        float l = (lane % LPR) == 0 ? lacc : 0.0f;
        for (int off = 16; off > 0; off >>= 1) l += __shfl_xor_sync(0xffffffffu, l, off);
        l *= inv_sqrt_n;
        // value: sum the row groups that share the same columns
#pragma unroll
        for (int off = LPR; off < 32; off <<= 1)
#pragma unroll
            for (int v = 0; v < VEC; ++v) vacc[v] += __shfl_xor_sync(0xffffffffu, vacc[v], off);
        const float mn = fmaxf(m_w, l);
        const float sc_old = expf(m_w - mn);
        const float pe = expf(l - mn);
        d_w = fmaf(d_w, sc_old, pe);
#pragma unroll
        for (int v = 0; v < VEC; ++v) O_w[v] = fmaf(O_w[v], sc_old, pe * vacc[v]);
        m_w = mn;
    }
    if (lane < LPR) {
#pragma unroll
        for (int v = 0; v < VEC; ++v) sWO[warp][p0 + v] = O_w[v];
    }
    if (lane == 0) {
        sWm[warp] = m_w;
        sWd[warp] = d_w;
    }
    __syncthreads();

    // phase 3: merge the warps' partial softmaxes, gate, write y
    if (tid < P) {
        float yssd = 0.0f;
        for (int k = tid; k < kDecThreads; k += P) yssd += sY[k];
        float mx = -INFINITY;
        for (int w = 0; w < kDecWarps; ++w) mx = fmaxf(mx, sWm[w]);
        float den = 0.0f, num = 0.0f;
        if (nhist > 0) {
            for (int w = 0; w < kDecWarps; ++w) {
                if (sWm[w] == -INFINITY) continue;
                const float s = expf(sWm[w] - mx);
                den = fmaf(sWd[w], s, den);
                num = fmaf(sWO[w][tid], s, num);
            }
        }
        const float r = nhist > 0 ? num / den : 0.0f;
        const float gate = silu_f32(ld_f32(z + bh));
        y[bh * P + tid] = cvt_from_f32<Tout>(yssd + gate * r);
        if (tid == 0 && lse != nullptr) lse[bh] = nhist > 0 ? mx + logf(den) : -INFINITY;
    }
}

template <typename Tin, typename Tmem, typename Tout>
cudaError_t launch_decode_step(const DecodeArgs& a, cudaStream_t stream) {
    dim3 grid((unsigned)a.H, (unsigned)a.B);
#define DART_DECODE_CASE(PP)                                                                  \
    case PP:                                                                                  \
        decode_step_kernel<Tin, Tmem, Tout, PP><<<grid, kDecThreads, 0, stream>>>(            \
            a.pos, (int)a.m_cap, (Tmem*)a.cache, a.state, a.partial, (const Tin*)a.x, a.dt,  \
            a.A, (const Tin*)a.b, (const Tin*)a.c, (const Tin*)a.q, (const Tin*)a.e,          \
            (const Tin*)a.z, (Tout*)a.y, a.lse, (int)a.H, (int)a.G, (int)a.N, (int)a.S, a.eps); \
        break;
    switch ((int)a.P) {
        DART_DECODE_CASE(16)
        DART_DECODE_CASE(32)
        DART_DECODE_CASE(64)
        default:
            return cudaErrorInvalidValue;
    }
#undef DART_DECODE_CASE
    note_launches(1);
    return cudaGetLastError();
}

typedef __nv_bfloat16 bf16;
template cudaError_t launch_decode_step<float, float, float>(const DecodeArgs&, cudaStream_t);
template cudaError_t launch_decode_step<bf16, float, float>(const DecodeArgs&, cudaStream_t);
template cudaError_t launch_decode_step<bf16, bf16, float>(const DecodeArgs&, cudaStream_t);
template cudaError_t launch_decode_step<bf16, bf16, bf16>(const DecodeArgs&, cudaStream_t);

}  // namespace dart
