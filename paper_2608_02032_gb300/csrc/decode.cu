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
// Three blocks per SM (registers capped at 80; a few spill): measured 427 us
// at decode_b64 against 462 us at two blocks per SM and 476 us at four.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dart {

constexpr int kDecThreads = 256;
constexpr int kDecWarps = kDecThreads / 32;

// 16-byte pieces of a memory row: raw load (streamed once) and unpack to fp32.
template <typename T> struct Vec16;
template <> struct Vec16<__nv_bfloat16> {
    static constexpr int n = 8;
    typedef uint4 raw_t;
    __device__ static raw_t load(const __nv_bfloat16* p) {
        return __ldcs(reinterpret_cast<const uint4*>(p));
    }
    __device__ static void unpack(const raw_t& u, float* out) {
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
    typedef float4 raw_t;
    __device__ static raw_t load(const float* p) { return __ldcs(reinterpret_cast<const float4*>(p)); }
    __device__ static void unpack(const raw_t& f, float* out) {
        out[0] = f.x; out[1] = f.y; out[2] = f.z; out[3] = f.w;
    }
};

constexpr int kBatch = 8;  // row steps whose loads a lane issues before using any

template <typename Tin, typename Tmem, typename Tout, int P>
__global__ void __launch_bounds__(kDecThreads, 3)
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
    __shared__ float sY[4 * kDecThreads];  // per (row group, column) partial y_ssd
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
    // thread owns columns 4 q .. 4 q + 3 (q = tid % (P / 4)) of rows n = tid / (P / 4) + k rstep;
    // the loads of all its rows are issued before any is used
    constexpr int QP = P / 4;
    static_assert(kDecThreads % QP == 0, "P / 4 must divide the block");
    const int q_own = tid % QP;
    const int rstep = kDecThreads / QP;
    constexpr int kRowBatch = 4;  // rows whose loads are issued together
    float yp[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    for (int k0 = 0; tid / QP + k0 * rstep < N; k0 += kRowBatch) {
    float4 s4[kRowBatch], p4[kRowBatch];
#pragma unroll
    for (int k = 0; k < kRowBatch; ++k) {
        const int n = tid / QP + (k0 + k) * rstep;
        if (n < N) {
            s4[k] = reinterpret_cast<const float4*>(St + n * P)[q_own];
            if (!chunk_start) p4[k] = reinterpret_cast<const float4*>(Pt + n * P)[q_own];
        }
    }
#pragma unroll
    for (int k = 0; k < kRowBatch; ++k) {
        const int n = tid / QP + (k0 + k) * rstep;
        if (n >= N) continue;
        const float bd = d * sb[n];
        const float4 xs = make_float4(sx[4 * q_own], sx[4 * q_own + 1], sx[4 * q_own + 2], sx[4 * q_own + 3]);
        const float w[4] = {bd * xs.x, bd * xs.y, bd * xs.z, bd * xs.w};
        const float so[4] = {s4[k].x, s4[k].y, s4[k].z, s4[k].w};
        float hn[4], pn[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) hn[i] = fmaf(a, so[i], w[i]);
        if (chunk_start) {
#pragma unroll
            for (int i = 0; i < 4; ++i) pn[i] = w[i];
        } else {
            const float po[4] = {p4[k].x, p4[k].y, p4[k].z, p4[k].w};
#pragma unroll
            for (int i = 0; i < 4; ++i) pn[i] = fmaf(a, po[i], w[i]);
        }
        reinterpret_cast<float4*>(St + n * P)[q_own] = make_float4(hn[0], hn[1], hn[2], hn[3]);
        reinterpret_cast<float4*>(Pt + n * P)[q_own] = make_float4(pn[0], pn[1], pn[2], pn[3]);
        if (slot != nullptr) {
#pragma unroll
            for (int i = 0; i < 4; ++i) slot[n * P + 4 * q_own + i] = cvt_from_f32<Tmem>(pn[i]);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) yp[i] = fmaf(sc[n], hn[i], yp[i]);
    }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) sY[(tid / QP) * P + 4 * q_own + i] = yp[i];

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
        for (int n0 = r0; n0 < N; n0 += kBatch * RPW) {
            typename Vec16<Tmem>::raw_t raw[kBatch];
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                const int n = n0 + u * RPW;
                if (n < N) raw[u] = Vec16<Tmem>::load(Mj + (i64)n * P + p0);
            }
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                const int n = n0 + u * RPW;
                if (n >= N) break;  // N is a multiple of RPW: every lane leaves at the same u
                float val[VEC];
                Vec16<Tmem>::unpack(raw[u], val);
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
        for (int k = 0; k < kDecThreads / (P / 4); ++k) yssd += sY[k * P + tid];
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
