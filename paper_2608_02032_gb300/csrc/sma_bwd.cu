// Backward of state-memory attention and the gated merge, FFMA path. The
// paper prints no backward (Sec. 3 only says the layer is trained end to
// end); this is the chain rule on the forward of Sec. 3 / App. B.1:
//   per token t (chunk i > 0) and memory j < i, with dR = SiLU(z) dY,
//   g_{t,j} = exp(l_{t,j} - lse_t),  D_t = dR_t . R_t,
//   dl_{t,j} = g_{t,j} (dR_t . V_{t,j} - D_t),  dV_{t,j} = g_{t,j} dR_t,
//   dEbar_t = sum_j dl_{t,j} U_{t,j} / sqrt(N),  U = Qbar (r (.) M_j),
//   dQbar_t = sum_j dl_{t,j} (r_j (.) M_j Ebar_t) / sqrt(N),
//   dC_t    = sum_j g_{t,j} M_j dR_t,
//   dM_j    = sum_t g_{t,j} C_t^T dR_t + r_j (.) G_j - (M_j G_j^T-diag) r_j^3 M_j / P,
//             G_j = sum_t dl_{t,j} Qbar_t^T Ebar_t / sqrt(N)   (the r_j(M_j) term),
//   dz_t    = (dY_t . R_t) SiLU'(z_t),
// and the unit-weight RMSNorm backwards take dQbar, dEbar to dQ, dE.
//
// sma_bwd_rows_kernel, one block of 256 threads per (64-token tile, h, b):
// pass 1 streams the memories to rebuild R_t from the saved lse; pass 2
// streams them again for dl, dEbar, dQbar and dC, and writes g and dl for
// the memory-gradient kernel. sma_bwd_mem_kernel, one block per (j, h, b),
// streams the tokens of later chunks for dM_j. Q, C and E are shared by the
// heads of a group, so their gradients are summed with fp32 atomics into
// outputs the launcher zeroes first.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace dart {
namespace {

constexpr int kBT = 64;  // tokens per tile
constexpr int kPad = 65; // padded row of 64 floats (conflict-free column walks)

// Warp lanes 16 apart hold the same token row of a 16-wide tx group: sums
// over the 16 lanes of a half-warp.
__device__ __forceinline__ float sum16(float v) {
#pragma unroll
    for (int off = 8; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    return v;
}

template <typename Tin, typename Tmem>
__global__ void __launch_bounds__(256)
sma_bwd_rows_kernel(const Tmem* __restrict__ Mem, const float* __restrict__ rM,
                    const Tin* __restrict__ Q, const Tin* __restrict__ Cm,
                    const Tin* __restrict__ E, const Tin* __restrict__ z,
                    const Tin* __restrict__ dY, const float* __restrict__ lse,
                    float* __restrict__ gbuf, float* __restrict__ dlbuf, float* __restrict__ dQ,
                    float* __restrict__ dC, float* __restrict__ dE, float* __restrict__ dz, int L,
                    int H, int G, int P, int N, int S, int Mc, float eps) {
    extern __shared__ float4 smem4[];
    float* smem = reinterpret_cast<float*>(smem4);
    float* sQt = smem;                // [N][64]  Qbar^T
    float* sCt = sQt + N * kBT;       // [N][64]  C^T
    float* sE = sCt + N * kBT;        // [64][65] Ebar (p >= P zero)
    float* sdR = sE + kBT * kPad;     // [64][65] dR = SiLU(z) dY
    float* sD = sdR + kBT * kPad;     // [N][65]  M_j
    float* sW = sD + N * kPad;        // [N][65]  r_j (.) M_j
    float* sG = sW + N * kPad;        // [64] g_{t,j}
    float* sDL = sG + kBT;            // [64] dl_{t,j} / sqrt(N)
    float* sIq = sDL + kBT;           // [64] 1 / rms(Q_t)
    float* sIe = sIq + kBT;           // [64] 1 / rms(E_t)
    float* sLse = sIe + kBT;          // [64]

    const int tile = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int g = h / (H / G);
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int lane = tid & 31, warp = tid >> 5;
    const int t0 = tile * kBT;
    const int ntok = min(kBT, L - t0);
    const i64 row0 = (i64)b * L + t0;
    const float rsn = __frsqrt_rn((float)N);

    for (int r = warp; r < kBT; r += 8) {
        const bool ok = r < ntok;
        const Tin* q = Q + ((row0 + r) * G + g) * N;
        const Tin* c = Cm + ((row0 + r) * G + g) * N;
        const Tin* e = E + ((row0 + r) * G + g) * P;
        const Tin* dy = dY + ((row0 + r) * H + h) * P;
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
        const float gate = ok ? silu_f32(ld_f32(z + (row0 + r) * H + h)) : 0.0f;
        for (int n = lane; n < N; n += 32) {
            sQt[n * kBT + r] = ok ? ld_f32(q + n) * iq : 0.0f;
            sCt[n * kBT + r] = ok ? ld_f32(c + n) : 0.0f;
        }
        for (int p = lane; p < 64; p += 32) {
            sE[r * kPad + p] = (ok && p < P) ? ld_f32(e + p) * ie : 0.0f;
            sdR[r * kPad + p] = (ok && p < P) ? gate * ld_f32(dy + p) : 0.0f;
        }
        if (lane == 0) {
            sIq[r] = iq;
            sIe[r] = ie;
            sLse[r] = ok ? lse[(row0 + r) * H + h] : -INFINITY;
        }
    }

    int nh[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) nh[i] = (t0 + ty * 4 + i) / S;
    const int nh_max = ntok > 0 ? (t0 + ntok - 1) / S : 0;

    // stage memory j as M_j and r_j (.) M_j
    auto stage = [&](int j) {
        __syncthreads();
        const i64 mbase = ((i64)b * Mc + j) * H + h;
        const Tmem* Mj = Mem + mbase * N * P;
        const float* rj = rM + mbase * N;
        for (int e = tid; e < N * 64; e += 256) {
            const int n = e >> 6, p = e & 63;
            const float v = p < P ? ld_f32(Mj + (i64)n * P + p) : 0.0f;
            sD[n * kPad + p] = v;
            sW[n * kPad + p] = v * rj[n];
        }
        __syncthreads();
    };
    // U = Qbar (r (.) M_j), V = C M_j for the thread's 4 tokens x 4 columns
    auto readouts = [&](float (&U)[4][4], float (&V)[4][4]) {
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int k = 0; k < 4; ++k) { U[i][k] = 0.0f; V[i][k] = 0.0f; }
#pragma unroll 4
        for (int n = 0; n < N; ++n) {
            const float4 q4 = *reinterpret_cast<const float4*>(&sQt[n * kBT + ty * 4]);
            const float4 c4 = *reinterpret_cast<const float4*>(&sCt[n * kBT + ty * 4]);
            const float qq[4] = {q4.x, q4.y, q4.z, q4.w}, cc[4] = {c4.x, c4.y, c4.z, c4.w};
            float ww[4], dd[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                ww[k] = sW[n * kPad + tx * 4 + k];
                dd[k] = sD[n * kPad + tx * 4 + k];
            }
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    U[i][k] = fmaf(qq[i], ww[k], U[i][k]);
                    V[i][k] = fmaf(cc[i], dd[k], V[i][k]);
                }
        }
    };

    // ---- pass 1: R_t = sum_j g V, g = exp(l - lse), and G1_t = sum_j g (1 up to rounding)
    float Rr[4][4] = {}, G1[4] = {};
    for (int j = 0; j < nh_max; ++j) {
        stage(j);
        float U[4][4], V[4][4];
        readouts(U, V);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int tl = ty * 4 + i;
            float part = 0.0f;
#pragma unroll
            for (int k = 0; k < 4; ++k) part = fmaf(U[i][k], sE[tl * kPad + tx * 4 + k], part);
            const float l = sum16(part) * rsn;
            const float gw = j < nh[i] ? expf(l - sLse[tl]) : 0.0f;
            G1[i] += gw;
#pragma unroll
            for (int k = 0; k < 4; ++k) Rr[i][k] = fmaf(gw, V[i][k], Rr[i][k]);
        }
    }
    float Dt[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int tl = ty * 4 + i;
        float dr = 0.0f, dyr = 0.0f;
        const i64 row = (row0 + tl) * H + h;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int p = tx * 4 + k;
            dr = fmaf(sdR[tl * kPad + p], Rr[i][k], dr);
            if (tl < ntok && p < P) dyr = fmaf(ld_f32(dY + row * P + p), Rr[i][k], dyr);
        }
        Dt[i] = sum16(dr);
        dyr = sum16(dyr);
        if (tx == 0 && tl < ntok) dz[row] = nh[i] > 0 ? dyr * silu_grad_f32(ld_f32(z + row)) : 0.0f;
    }

    // ---- pass 2: dl, dEbar (t x p layout), dQbar and dC (t x n layout: n = tx + 16 k)
    float dEb[4][4] = {};
    float dQb[4][8] = {}, dCc[4][8] = {};
    for (int j = 0; j < nh_max; ++j) {
        stage(j);
        float U[4][4], V[4][4];
        readouts(U, V);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int tl = ty * 4 + i;
            float part = 0.0f, drv = 0.0f;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                part = fmaf(U[i][k], sE[tl * kPad + tx * 4 + k], part);
                drv = fmaf(sdR[tl * kPad + tx * 4 + k], V[i][k], drv);
            }
            const float l = sum16(part) * rsn;
            drv = sum16(drv);
            const bool use = j < nh[i];
            const float gw = use ? expf(l - sLse[tl]) : 0.0f;
            // dl = g_j sum_k g_k (s_j - s_k) with s = dR . V: with the computed weights'
            // own sum G1 instead of 1, the weights' rounding does not leave a term
            // g_j s_j (1 - G1), which for a peaked softmax is large next to dl itself
            const float dl = use ? gw * fmaf(drv, G1[i], -Dt[i]) : 0.0f;
#pragma unroll
            for (int k = 0; k < 4; ++k) dEb[i][k] = fmaf(dl * rsn, U[i][k], dEb[i][k]);
            if (tx == 0) {
                sG[tl] = gw;
                sDL[tl] = dl * rsn;
                if (use && tl < ntok) {
                    const i64 gi = (((i64)b * H + h) * Mc + j) * L + t0 + tl;
                    gbuf[gi] = gw;
                    dlbuf[gi] = dl;
                }
            }
        }
        __syncthreads();
        // K_t[n] = sum_p W[n,p] Ebar_t[p];  Mr_t[n] = sum_p M[n,p] dR_t[p]
        float Kt[4][8] = {}, Mr[4][8] = {};
        for (int p = 0; p < P; ++p) {
            float ev[4], rv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                ev[i] = sE[(ty * 4 + i) * kPad + p];
                rv[i] = sdR[(ty * 4 + i) * kPad + p];
            }
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const int n = tx + 16 * k;
                const float w = n < N ? sW[n * kPad + p] : 0.0f;
                const float d = n < N ? sD[n * kPad + p] : 0.0f;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    Kt[i][k] = fmaf(w, ev[i], Kt[i][k]);
                    Mr[i][k] = fmaf(d, rv[i], Mr[i][k]);
                }
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float gw = sG[ty * 4 + i], dls = sDL[ty * 4 + i];
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                dQb[i][k] = fmaf(dls, Kt[i][k], dQb[i][k]);
                dCc[i][k] = fmaf(gw, Mr[i][k], dCc[i][k]);
            }
        }
    }

    // ---- RMSNorm backwards and the group-shared gradients
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int tl = ty * 4 + i;
        const bool ok = tl < ntok && nh[i] > 0;
        float dq_dot = 0.0f, de_dot = 0.0f;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int n = tx + 16 * k;
            if (n < N) dq_dot = fmaf(dQb[i][k], sQt[n * kBT + tl], dq_dot);
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) de_dot = fmaf(dEb[i][k], sE[tl * kPad + tx * 4 + k], de_dot);
        dq_dot = sum16(dq_dot);
        de_dot = sum16(de_dot);
        if (!ok) continue;
        const i64 grow = (row0 + tl) * G + g;
        const float iq = sIq[tl], ie = sIe[tl];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int n = tx + 16 * k;
            if (n >= N) continue;
            const float qb = sQt[n * kBT + tl];
            atomicAdd(dQ + grow * N + n, iq * (dQb[i][k] - qb * dq_dot / (float)N));
            atomicAdd(dC + grow * N + n, dCc[i][k]);
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int p = tx * 4 + k;
            if (p >= P) continue;
            atomicAdd(dE + grow * P + p, ie * (dEb[i][k] - sE[tl * kPad + p] * de_dot / (float)P));
        }
    }
}

// dM_j, one block of 256 threads per (j, h, b). Thread (ty, tx) owns rows
// n = ty + 16 a (a < 8) and columns p = 4 tx + k (k < 4).
template <typename Tin, typename Tmem>
__global__ void __launch_bounds__(256)
sma_bwd_mem_kernel(const Tmem* __restrict__ Mem, const float* __restrict__ rM,
                   const Tin* __restrict__ Q, const Tin* __restrict__ Cm,
                   const Tin* __restrict__ E, const Tin* __restrict__ z,
                   const Tin* __restrict__ dY, const float* __restrict__ gbuf,
                   const float* __restrict__ dlbuf, float* __restrict__ dM, int L, int H, int G,
                   int P, int N, int S, int Mc, float eps) {
    extern __shared__ float4 smem4[];
    float* smem = reinterpret_cast<float*>(smem4);
    float* sGC = smem;               // [64][N]   g_{t,j} C_t
    float* sDQ = sGC + kBT * N;      // [64][N]   dl_{t,j} Qbar_t / sqrt(N)
    float* sdR = sDQ + kBT * N;      // [64][64]  dR_t
    float* sE = sdR + kBT * 64;      // [64][64]  Ebar_t

    const int j = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int g = h / (H / G);
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int lane = tid & 31, warp = tid >> 5;
    const float rsn = __frsqrt_rn((float)N);
    const float* gj = gbuf + (((i64)b * H + h) * Mc + j) * L;
    const float* dlj = dlbuf + (((i64)b * H + h) * Mc + j) * L;

    float T1[8][4] = {}, Gp[8][4] = {};
    for (int t0 = (j + 1) * S; t0 < L; t0 += kBT) {
        const int ntok = min(kBT, L - t0);
        __syncthreads();
        for (int r = warp; r < kBT; r += 8) {
            const bool ok = r < ntok;
            const i64 row = (i64)b * L + t0 + r;
            const Tin* q = Q + (row * G + g) * N;
            const Tin* c = Cm + (row * G + g) * N;
            const Tin* e = E + (row * G + g) * P;
            const Tin* dy = dY + (row * H + h) * P;
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
            const float gw = ok ? gj[t0 + r] : 0.0f;
            const float dls = ok ? dlj[t0 + r] * rsn : 0.0f;
            const float gate = ok ? silu_f32(ld_f32(z + row * H + h)) : 0.0f;
            for (int n = lane; n < N; n += 32) {
                sGC[r * N + n] = ok ? gw * ld_f32(c + n) : 0.0f;
                sDQ[r * N + n] = ok ? dls * ld_f32(q + n) * iq : 0.0f;
            }
            for (int p = lane; p < 64; p += 32) {
                sdR[r * 64 + p] = (ok && p < P) ? gate * ld_f32(dy + p) : 0.0f;
                sE[r * 64 + p] = (ok && p < P) ? ld_f32(e + p) * ie : 0.0f;
            }
        }
        __syncthreads();
        // two-level sums (per 64-token tile, then across tiles): the terms have
        // mixed signs and a memory can collect thousands of them
        float T1t[8][4] = {}, Gpt[8][4] = {};
        for (int r = 0; r < ntok; ++r) {
            const float4 d4 = *reinterpret_cast<const float4*>(&sdR[r * 64 + tx * 4]);
            const float4 e4 = *reinterpret_cast<const float4*>(&sE[r * 64 + tx * 4]);
            const float dr[4] = {d4.x, d4.y, d4.z, d4.w}, ev[4] = {e4.x, e4.y, e4.z, e4.w};
#pragma unroll
            for (int a = 0; a < 8; ++a) {
                const int n = ty + 16 * a;
                const float gc = n < N ? sGC[r * N + n] : 0.0f;
                const float dq = n < N ? sDQ[r * N + n] : 0.0f;
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    T1t[a][k] = fmaf(gc, dr[k], T1t[a][k]);
                    Gpt[a][k] = fmaf(dq, ev[k], Gpt[a][k]);
                }
            }
        }
#pragma unroll
        for (int a = 0; a < 8; ++a)
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                T1[a][k] += T1t[a][k];
                Gp[a][k] += Gpt[a][k];
            }
    }
    // dM = T1 + r (.) G' - (sum_q M G')_n r^3 M / P
    const i64 mbase = ((i64)b * Mc + j) * H + h;
    const Tmem* Mj = Mem + mbase * N * P;
    float* dMj = dM + mbase * N * P;
#pragma unroll
    for (int a = 0; a < 8; ++a) {
        const int n = ty + 16 * a;
        float mv[4], dr = 0.0f;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int p = tx * 4 + k;
            mv[k] = (n < N && p < P) ? ld_f32(Mj + (i64)n * P + p) : 0.0f;
            dr = fmaf(mv[k], Gp[a][k], dr);
        }
        dr = sum16(dr);
        if (n >= N) continue;
        const float rn = rM[mbase * N + n];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int p = tx * 4 + k;
            if (p < P) dMj[(i64)n * P + p] = T1[a][k] + rn * Gp[a][k] - dr * rn * rn * rn * mv[k] / (float)P;
        }
    }
}

}  // namespace

size_t sma_bwd_workspace(int64_t B, int64_t L, int64_t H, int64_t Mc, int64_t N) {
    const size_t gl = (size_t)(B * H * Mc * L) * sizeof(float);
    const size_t r = (size_t)(B * Mc * H * N) * sizeof(float);
    return 2 * ((gl + 255) & ~(size_t)255) + ((r + 255) & ~(size_t)255);
}

template <typename Tin, typename Tmem>
cudaError_t launch_sma_backward(const SmaBwdArgs& a, void* ws, cudaStream_t stream) {
    const int B = (int)a.B, L = (int)a.L, H = (int)a.H, G = (int)a.G, P = (int)a.P, N = (int)a.N,
              S = (int)a.S, Mc = L / S;
    const size_t gl = ((size_t)(a.B * a.H * Mc * a.L) * sizeof(float) + 255) & ~(size_t)255;
    float* gbuf = (float*)ws;
    float* dlbuf = (float*)((uint8_t*)ws + gl);
    float* rM = a.rM != nullptr ? (float*)a.rM : (float*)((uint8_t*)ws + 2 * gl);
    cudaError_t e;
    if (a.rM == nullptr) {
        e = launch_memory_rms<Tmem>(a.M, rM, a.B * Mc * a.H * a.N, a.P, a.eps, stream);
        if (e != cudaSuccess) return e;
    }
    const size_t gq = (size_t)(a.B * a.L * a.G);
    if ((e = cudaMemsetAsync(a.dQ, 0, gq * N * sizeof(float), stream)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(a.dC, 0, gq * N * sizeof(float), stream)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(a.dE, 0, gq * P * sizeof(float), stream)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(a.dM, 0, (size_t)(a.B * Mc * a.H) * N * P * sizeof(float), stream)) !=
        cudaSuccess)
        return e;

    const size_t smem1 = (size_t)(2 * N * kBT + 2 * kBT * kPad + 2 * N * kPad + 5 * kBT) * sizeof(float);
    auto k1 = sma_bwd_rows_kernel<Tin, Tmem>;
    if ((e = cudaFuncSetAttribute(k1, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1)) !=
        cudaSuccess)
        return e;
    k1<<<dim3((unsigned)((L + kBT - 1) / kBT), (unsigned)H, (unsigned)B), 256, smem1, stream>>>(
        (const Tmem*)a.M, rM, (const Tin*)a.Q, (const Tin*)a.Cm, (const Tin*)a.E, (const Tin*)a.z,
        (const Tin*)a.dY, a.lse, gbuf, dlbuf, a.dQ, a.dC, a.dE, a.dz, L, H, G, P, N, S, Mc, a.eps);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (Mc > 1) {
        const size_t smem2 = (size_t)(2 * kBT * N + 2 * kBT * 64) * sizeof(float);
        auto k2 = sma_bwd_mem_kernel<Tin, Tmem>;
        if ((e = cudaFuncSetAttribute(k2, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem2)) !=
            cudaSuccess)
            return e;
        k2<<<dim3((unsigned)(Mc - 1), (unsigned)H, (unsigned)B), 256, smem2, stream>>>(
            (const Tmem*)a.M, rM, (const Tin*)a.Q, (const Tin*)a.Cm, (const Tin*)a.E,
            (const Tin*)a.z, (const Tin*)a.dY, gbuf, dlbuf, a.dM, L, H, G, P, N, S, Mc, a.eps);
        note_launches(1);
    }
    return cudaGetLastError();
}

typedef __nv_bfloat16 bf16;
template cudaError_t launch_sma_backward<float, float>(const SmaBwdArgs&, void*, cudaStream_t);
template cudaError_t launch_sma_backward<bf16, float>(const SmaBwdArgs&, void*, cudaStream_t);
template cudaError_t launch_sma_backward<bf16, bf16>(const SmaBwdArgs&, void*, cudaStream_t);

}  // namespace dart
