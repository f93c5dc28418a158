// Chunked SSD scan with chunk state memories (Sec. 2; Sec. 3 "Chunk State
// Memories"; App. A). Four kernels on the caller's stream:
//   1. chunk_cumsum   cum[b,h,c,k] = sum_{u<=k} dt A within chunk c (the
//                     exponent of the decay products A_{u:v}, Sec. 2).
//   2. chunk_state    Delta H_[c] = B_c^T diag(w) X_c with
//                     w_s = exp(cum_end - cum_s) dt_s (App. A eq.
//                     "mamba2_delta_h_chunk"); writes the memory M_j, its
//                     inverse RMS r (App. B.1) and an fp32 copy for step 3.
//   3. state_passing  H_[c] = exp(cum_end_c) H_[c-1] + Delta H_[c] (App. A eq.
//                     "mamba2_chunk_state"), in place: slot c of the fp32
//                     copy becomes the state entering chunk c.
//   4. chunk_output   Y_t = sum_{s<=t in c} exp(cum_t - cum_s)(C_t.B_s) dt_s X_s
//                     + exp(cum_t) C_t H_[c-1] (App. A intra/inter split).
// These are FFMA (fp32 CUDA-core) kernels: exact enough for fp32 inputs and
// the generic path for every supported size.
#include "common.cuh"
#include "kernels.h"

namespace dart {

// ---------------------------------------------------------------- 1. cumsum
// One block per (c, h, b); blockDim.x == S (power of two, <= 1024).
__global__ void chunk_cumsum_kernel(const float* __restrict__ dt, const float* __restrict__ A,
                                    float* __restrict__ cum, int L, int H, int S, int M) {
    extern __shared__ float sh[];
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z, k = threadIdx.x;
    const i64 t = (i64)c * S + k;
    float v = dt[((i64)b * L + t) * H + h] * A[h];
    // inclusive warp scan, then scan of the warp totals
    const int lane = k & 31, warp = k >> 5;
    // S is a power of two; below 32 only the first S lanes of warp 0 exist
    const unsigned mask = S >= 32 ? 0xffffffffu : ((1u << S) - 1u);
    for (int off = 1; off < 32; off <<= 1) {
        float o = __shfl_up_sync(mask, v, off);
        if (lane >= off) v += o;
    }
    if (lane == 31 || k == S - 1) sh[warp] = v;
    __syncthreads();
    if (warp == 0) {
        const int nw = (S + 31) / 32;
        float w = lane < nw ? sh[lane] : 0.0f;
        for (int off = 1; off < 32; off <<= 1) {
            float o = __shfl_up_sync(mask, w, off);
            if (lane >= off) w += o;
        }
        if (lane < nw) sh[32 + lane] = w;
    }
    __syncthreads();
    if (warp > 0) v += sh[32 + warp - 1];
    cum[(((i64)b * H + h) * M + c) * S + k] = v;
}

// ----------------------------------------------------------- 2. chunk state
// One block of 256 threads per (c, h, b). Output tiles of 64 (n) x 64 (p);
// thread (ty, tx) owns rows n = 4 ty + i, columns p = 4 tx + j.
constexpr int kST = 32;  // tokens per staged slice

template <typename Tin, typename Tmem>
__global__ void __launch_bounds__(256)
chunk_state_kernel(const Tin* __restrict__ X, const float* __restrict__ dt,
                   const float* __restrict__ cum, const Tin* __restrict__ Bm,
                   float* __restrict__ dH32, Tmem* __restrict__ Mout, float* __restrict__ rM,
                   int L, int H, int G, int P, int N, int S, int M, float eps) {
    __shared__ float sB[kST][64];
    __shared__ float sX[kST][64];
    __shared__ float sW[kST];
    __shared__ float sSq[128];
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int g = h / (H / G);
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const float* cumc = cum + (((i64)b * H + h) * M + c) * S;
    const float cum_end = cumc[S - 1];
    const i64 t0 = (i64)c * S;
    const i64 mem_base = (((i64)b * M + c) * H + h) * (i64)N * P;

    for (int nt = 0; nt < N; nt += 64) {
        for (int i = tid; i < 64; i += 256) sSq[i] = 0.0f;
        for (int pt = 0; pt < P; pt += 64) {
            float acc[4][4] = {};
            for (int s0 = 0; s0 < S; s0 += kST) {
                __syncthreads();
                if (tid < kST) {
                    const int s = s0 + tid;
                    sW[tid] = s < S ? expf(cum_end - cumc[s]) * dt[((i64)b * L + t0 + s) * H + h] : 0.0f;
                }
                __syncthreads();
                for (int e = tid; e < kST * 64; e += 256) {
                    const int s = e >> 6, col = e & 63;
                    const int n = nt + col, p = pt + col;
                    const bool sv = s0 + s < S;
                    const i64 tok = (i64)b * L + t0 + s0 + s;
                    sB[s][col] = (sv && n < N) ? sW[s] * ld_f32(Bm + (tok * G + g) * N + n) : 0.0f;
                    sX[s][col] = (sv && p < P) ? ld_f32(X + (tok * H + h) * P + p) : 0.0f;
                }
                __syncthreads();
#pragma unroll 8
                for (int s = 0; s < kST; ++s) {
                    const float4 bv = *reinterpret_cast<const float4*>(&sB[s][ty * 4]);
                    const float4 xv = *reinterpret_cast<const float4*>(&sX[s][tx * 4]);
                    const float bb[4] = {bv.x, bv.y, bv.z, bv.w};
                    const float xx[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
                    for (int i = 0; i < 4; ++i)
#pragma unroll
                        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(bb[i], xx[j], acc[i][j]);
                }
            }
            // epilogue: store fp32 copy and the memory, accumulate squares of
            // the stored values for r
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int n = nt + ty * 4 + i;
                float sq = 0.0f;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int p = pt + tx * 4 + j;
                    if (n < N && p < P) {
                        const i64 o = mem_base + (i64)n * P + p;
                        dH32[o] = acc[i][j];
                        Mout[o] = cvt_from_f32<Tmem>(acc[i][j]);
                        const float sv = stored_value<Tmem>(acc[i][j]);
                        sq = fmaf(sv, sv, sq);
                    }
                }
                if (n < N) atomicAdd(&sSq[ty * 4 + i], sq);
            }
        }
        __syncthreads();
        if (rM != nullptr) {
            for (int i = tid; i < 64; i += 256) {
                const int n = nt + i;
                if (n < N)
                    rM[(((i64)b * M + c) * H + h) * N + n] = __frsqrt_rn(sSq[i] / (float)P + eps);
            }
        }
        __syncthreads();
    }
}

// --------------------------------------------------------- 3. state passing
// One thread per state element (n, p) of one (b, h); loops over chunks.
__global__ void state_passing_kernel(float* __restrict__ dH32, const float* __restrict__ cum,
                                     float* __restrict__ final_state, int H, int M, int S, int NP) {
    const int e = blockIdx.x * blockDim.x + threadIdx.x;
    const int h = blockIdx.y, b = blockIdx.z;
    if (e >= NP) return;
    const float* cumh = cum + ((i64)b * H + h) * M * S;
    const i64 stride = (i64)H * NP;  // between chunk slots of the same element
    float* base = dH32 + ((i64)b * M * H + h) * NP + e;
    float st = 0.0f;
    // groups of 16 chunks: issue the independent loads first, then the chain
    for (int c0 = 0; c0 < M; c0 += 16) {
        const int n = min(16, M - c0);
        float d[16], dec[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) {
            if (k < n) {
                d[k] = base[(i64)(c0 + k) * stride];
                dec[k] = expf(cumh[(i64)(c0 + k) * S + S - 1]);
            }
        }
#pragma unroll
        for (int k = 0; k < 16; ++k) {
            if (k < n) {
                base[(i64)(c0 + k) * stride] = st;  // state entering chunk c0 + k
                st = fmaf(dec[k], st, d[k]);
            }
        }
    }
    if (final_state != nullptr) final_state[((i64)b * H + h) * NP + e] = st;
}

// ---------------------------------------------------------- 4. chunk output
// One block of 256 threads per (64-token tile, c * H + h, b). Thread (ty, tx)
// owns tokens 4 ty + i and, per 64-wide p tile, columns 4 tx + j.
constexpr int kNS = 16;  // state rows per staged slice

template <typename Tin, typename Tout>
__global__ void __launch_bounds__(256)
chunk_output_kernel(const Tin* __restrict__ X, const float* __restrict__ dt,
                    const float* __restrict__ cum, const Tin* __restrict__ Bm,
                    const Tin* __restrict__ Cm, const float* __restrict__ Hin,
                    Tout* __restrict__ Y, int L, int H, int G, int P, int N, int S, int M) {
    __shared__ float sCt[kNS][64];  // C^T slice: [n][t]
    __shared__ float sBt[kNS][64];  // B^T slice: [n][s] (also reused for H: [n][p])
    __shared__ float sSc[64][65];  // masked, decayed scores [t][s]
    __shared__ float sXs[64][64];  // dt_s X_s [s][p]
    __shared__ float sCum[64];
    __shared__ float sCumS[64];
    const int tt = blockIdx.x;  // token tile within the chunk
    const int c = blockIdx.y / H, h = blockIdx.y % H, b = blockIdx.z;
    const int g = h / (H / G);
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int tl0 = tt * 64;                 // first chunk-local token of the tile
    const int nt_tok = min(64, S - tl0);     // tokens in this tile
    const i64 tok0 = (i64)b * L + (i64)c * S;  // global token row of chunk start
    const float* cumc = cum + (((i64)b * H + h) * M + c) * S;
    if (tid < 64) sCum[tid] = tid < nt_tok ? cumc[tl0 + tid] : 0.0f;

    for (int pt = 0; pt < P; pt += 64) {
        float acc[4][4] = {};
        // inter-chunk term: C_t H_[c-1]
        const float* Hc = Hin + (((i64)b * M + c) * H + h) * (i64)N * P;
        for (int n0 = 0; n0 < N; n0 += kNS) {
            __syncthreads();
            for (int e = tid; e < kNS * 64; e += 256) {
                const int n = e >> 6, col = e & 63;
                const bool nv = n0 + n < N;
                sCt[n][col] = (nv && col < nt_tok)
                                  ? ld_f32(Cm + ((tok0 + tl0 + col) * G + g) * N + n0 + n) : 0.0f;
                sBt[n][col] = (nv && pt + col < P) ? Hc[(i64)(n0 + n) * P + pt + col] : 0.0f;
            }
            __syncthreads();
#pragma unroll 8
            for (int n = 0; n < kNS; ++n) {
                const float4 cv = *reinterpret_cast<const float4*>(&sCt[n][ty * 4]);
                const float4 hv = *reinterpret_cast<const float4*>(&sBt[n][tx * 4]);
                const float cc[4] = {cv.x, cv.y, cv.z, cv.w};
                const float hh[4] = {hv.x, hv.y, hv.z, hv.w};
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(cc[i], hh[j], acc[i][j]);
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float dec = expf(sCum[ty * 4 + i]);
#pragma unroll
            for (int j = 0; j < 4; ++j) acc[i][j] *= dec;
        }
        // intra-chunk term over source tiles up to this one
        for (int st = 0; st <= tt; ++st) {
            const int sl0 = st * 64;
            const int ns_tok = min(64, S - sl0);
            float sc[4][4] = {};
            for (int n0 = 0; n0 < N; n0 += kNS) {
                __syncthreads();
                for (int e = tid; e < kNS * 64; e += 256) {
                    const int n = e >> 6, col = e & 63;
                    const bool nv = n0 + n < N;
                    sCt[n][col] = (nv && col < nt_tok)
                                      ? ld_f32(Cm + ((tok0 + tl0 + col) * G + g) * N + n0 + n) : 0.0f;
                    sBt[n][col] = (nv && col < ns_tok)
                                      ? ld_f32(Bm + ((tok0 + sl0 + col) * G + g) * N + n0 + n) : 0.0f;
                }
                __syncthreads();
#pragma unroll 8
                for (int n = 0; n < kNS; ++n) {
                    const float4 cv = *reinterpret_cast<const float4*>(&sCt[n][ty * 4]);
                    const float4 bv = *reinterpret_cast<const float4*>(&sBt[n][tx * 4]);
                    const float cc[4] = {cv.x, cv.y, cv.z, cv.w};
                    const float bb[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
                    for (int i = 0; i < 4; ++i)
#pragma unroll
                        for (int j = 0; j < 4; ++j) sc[i][j] = fmaf(cc[i], bb[j], sc[i][j]);
                }
            }
            __syncthreads();
            if (tid < 64) sCumS[tid] = tid < ns_tok ? cumc[sl0 + tid] : 0.0f;
            for (int e = tid; e < 64 * 64; e += 256) {
                const int s = e >> 6, col = e & 63;
                const i64 tok = tok0 + sl0 + s;
                sXs[s][col] = (s < ns_tok && pt + col < P)
                                  ? dt[tok * H + h] * ld_f32(X + (tok * H + h) * P + pt + col) : 0.0f;
            }
            __syncthreads();
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int t = tl0 + ty * 4 + i;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int s = sl0 + tx * 4 + j;
                    const bool ok = s <= t && (ty * 4 + i) < nt_tok && (tx * 4 + j) < ns_tok;
                    sSc[ty * 4 + i][tx * 4 + j] =
                        ok ? sc[i][j] * expf(sCum[ty * 4 + i] - sCumS[tx * 4 + j]) : 0.0f;
                }
            }
            __syncthreads();
#pragma unroll 8
            for (int s = 0; s < 64; ++s) {
                const float4 xv = *reinterpret_cast<const float4*>(&sXs[s][tx * 4]);
                const float xx[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float a = sSc[ty * 4 + i][s];
#pragma unroll
                    for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a, xx[j], acc[i][j]);
                }
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int tl = ty * 4 + i;
            if (tl >= nt_tok) continue;
            const i64 tok = tok0 + tl0 + tl;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int p = pt + tx * 4 + j;
                if (p < P) Y[(tok * H + h) * P + p] = cvt_from_f32<Tout>(acc[i][j]);
            }
        }
    }
}

// ------------------------------------------------------------------ launch
cudaError_t launch_chunk_cumsum(const ScanArgs& a, cudaStream_t stream) {
    const int B = (int)a.B, L = (int)a.L, H = (int)a.H, S = (int)a.S, M = L / S;
    chunk_cumsum_kernel<<<dim3(M, H, B), S, 64 * sizeof(float), stream>>>(a.dt, a.A, a.cum, L, H,
                                                                             S, M);
    note_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_state_passing(const ScanArgs& a, cudaStream_t stream) {
    const int B = (int)a.B, H = (int)a.H, S = (int)a.S, M = (int)(a.L / a.S);
    const int NP = (int)(a.N * a.P);
    state_passing_kernel<<<dim3((NP + 255) / 256, H, B), 256, 0, stream>>>(
        a.dH32, a.cum, a.final_state, H, M, S, NP);
    note_launches(1);
    return cudaGetLastError();
}

template <typename Tin, typename Tmem, typename Tout>
cudaError_t launch_chunk_scan_simt(const ScanArgs& a, cudaStream_t stream) {
    const int B = (int)a.B, L = (int)a.L, H = (int)a.H, G = (int)a.G, P = (int)a.P,
              N = (int)a.N, S = (int)a.S, M = L / S;
    cudaError_t e = launch_chunk_cumsum(a, stream);
    if (e != cudaSuccess) return e;
    chunk_state_kernel<Tin, Tmem><<<dim3(M, H, B), 256, 0, stream>>>(
        (const Tin*)a.X, a.dt, a.cum, (const Tin*)a.Bm, a.dH32, (Tmem*)a.M, a.rM, L, H, G, P, N, S,
        M, a.eps);
    note_launches(1);
    e = launch_state_passing(a, stream);
    if (e != cudaSuccess) return e;
    chunk_output_kernel<Tin, Tout><<<dim3((S + 63) / 64, M * H, B), 256, 0, stream>>>(
        (const Tin*)a.X, a.dt, a.cum, (const Tin*)a.Bm, (const Tin*)a.Cm, a.dH32, (Tout*)a.Y, L, H,
        G, P, N, S, M);
    note_launches(1);
    return cudaGetLastError();
}

template <typename Tin>
cudaError_t launch_scan_states(const ScanArgs& a0, float* cum, float* Hprev, float* scratch,
                               cudaStream_t stream) {
    ScanArgs a = a0;
    a.cum = cum;
    a.dH32 = Hprev;
    a.M = scratch;
    a.rM = nullptr;
    a.final_state = nullptr;
    const int L = (int)a.L, H = (int)a.H, G = (int)a.G, P = (int)a.P, N = (int)a.N,
              S = (int)a.S, M = L / S;
    cudaError_t e = launch_chunk_cumsum(a, stream);
    if (e != cudaSuccess) return e;
    chunk_state_kernel<Tin, float><<<dim3(M, H, (int)a.B), 256, 0, stream>>>(
        (const Tin*)a.X, a.dt, a.cum, (const Tin*)a.Bm, a.dH32, scratch, nullptr, L, H, G, P, N, S,
        M, a.eps);
    note_launches(1);
    return launch_state_passing(a, stream);
}

typedef __nv_bfloat16 bf16;
template cudaError_t launch_scan_states<float>(const ScanArgs&, float*, float*, float*, cudaStream_t);
template cudaError_t launch_scan_states<bf16>(const ScanArgs&, float*, float*, float*, cudaStream_t);
template cudaError_t launch_chunk_scan_simt<float, float, float>(const ScanArgs&, cudaStream_t);
template cudaError_t launch_chunk_scan_simt<bf16, float, float>(const ScanArgs&, cudaStream_t);
template cudaError_t launch_chunk_scan_simt<bf16, bf16, float>(const ScanArgs&, cudaStream_t);
template cudaError_t launch_chunk_scan_simt<bf16, bf16, bf16>(const ScanArgs&, cudaStream_t);

}  // namespace dart
