// Backward of the chunked SSD scan on the tensor cores, for bf16 inputs with
// P = 64, N = 128, G = 1, S in {128, 256} (the chain rule on the chunked
// forms of App. A; the paper prints no backward). With cum the within-chunk
// cumsum of dt A, L[t,s] = exp(cum_t - cum_s) (s <= t in one chunk), the
// chunk-entry states H_[c-1] and the adjoint d(dH_c) of each chunk state:
//   dX_s   = dt_s Y'_s,  Y'_s = sum_{t >= s} L[t,s] (B_s . C_t) dY_t
//                               + exp(cum_end - cum_s) B_s d(dH_c)
//            (the output kernel in reversed time, scan_tc.cu);
//   dC_t  += sum_s Psi[t,s] B_s + sum_h exp(cum_t) dY_t H_[c-1]^T,
//   dB_s   = sum_t Psi[t,s] C_t + sum_h exp(cum_end - cum_s) dt_s X_s d(dH_c)^T,
//            Psi[t,s] = sum_h L[t,s] dt_s (dY_t . X_s): with B and C shared by
//            the heads (G = 1) the intra-chunk terms need only this head sum;
//   d(cum_t) = dY_t . Y_t - dt_t X_t . Y'_t, plus at the chunk end
//            sum_s kappa_s (kappa_s = dt_s X_s . (exp(cum_end - cum_s) B_s d(dH_c)))
//            and exp(cum_end) <adjoint of H_c, H_[c-1]> (passing kernel);
//   d(dt_u) = X_u . Y'_u + A_h sum_{k >= u} d(cum_k),  dA_h = sum_u dt_u sum_{k >= u} d(cum_k).
// Kernels here: psi_kernel (Psi, per chunk and 128-row tile, summed over the
// heads from one tensor-core score tile dY X^T per head), dcdb_kernel (dC and
// dB as MMA chains over K units: Psi blocks against B or C rows, then one unit
// per head for the inter-chunk term), finalize_kernel (the d(cum) reverse sums).
// Operands that are not exact bf16 inputs are split bf16 hi + lo.
#include <math.h>

#include <cuda_bf16.h>

#include "common.cuh"
#include "kernels.h"
#include "tc_ptx.cuh"
#include "tma.cuh"

namespace dart {
namespace {

__device__ int g_sbwd_tc_status;  // first timeout code since the last read (0 = none)

constexpr int kP = 64;
constexpr int kN = 128;
constexpr int kT = 128;
constexpr uint64_t kDrainLimitNs = 2000000000ull;
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ uint32_t sw128(uint32_t row, uint32_t byte_in_row) {
    const uint32_t o = row * 128u + byte_in_row;
    return o ^ ((row & 7u) << 4);
}
__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&v);
}
__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
// Splits 8 floats into bf16 hi and lo words (4 + 4).
__device__ __forceinline__ void split8(const float* v, uint4& hi, uint4& lo) {
    uint32_t h[4], l[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const __nv_bfloat162 hv = __floats2bfloat162_rn(v[2 * e], v[2 * e + 1]);
        const float2 hf = __bfloat1622float2(hv);
        h[e] = *reinterpret_cast<const uint32_t*>(&hv);
        l[e] = pack_bf16(v[2 * e] - hf.x, v[2 * e + 1] - hf.y);
    }
    hi = make_uint4(h[0], h[1], h[2], h[3]);
    lo = make_uint4(l[0], l[1], l[2], l[3]);
}

__host__ __device__ constexpr uint32_t idesc_bf16(bool a_mn, bool b_mn, uint32_t M, uint32_t N) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) |
           ((N >> 3) << 17) | ((M >> 4) << 24);
}
__device__ __forceinline__ void mma_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                       uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
        ::"r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
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
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Bounded wait by every thread of the CTA, then a CTA-wide AND of the outcome.
__device__ __forceinline__ bool cta_wait(uint64_t* bar, uint32_t parity, uint64_t limit_ns, int code) {
    const bool got = tc::mbar_wait(bar, parity, limit_ns, nullptr);
    if (!got) atomicCAS(&g_sbwd_tc_status, 0, code);
    const bool all = __syncthreads_and(got ? 1 : 0) != 0;
    tc::tc_fence_after();
    return all;
}

// Psi layout, per (b, c): two parts (hi, lo) of S / 64 column blocks, each
// block S rows x 128 bytes in the 128-byte swizzle (row t, bytes 2 (s % 64)).
// A block read K-major (rows t, K = s) and one read MN-major (M = s, K = t)
// have this same layout.
__host__ __device__ inline int64_t psi_chunk_bytes(int S) { return 2LL * S * S * 2; }

// ---------------------------------------------------------------- psi / phi
// One CTA of 512 threads (four per row, a quarter of the sources each) per
// (128-token tile, chunk, b), looping over the heads; per head one MMA chain
// gives the score tile dY X^T (rows t, columns s <= t of the chunk).
//   !kPhi: Psi[t,s] = sum_h L[t,s] dt_s (dY_t . X_s), kept in registers, written
//          split hi + lo in the Psi layout;
//   kPhi:  Phi_h[t,s] = L[t,s] dt_s (C_t . B_s)(dY_t . X_s) with C B^T from one
//          more MMA chain (shared by the heads), reduced to its row sums
//          (phi_row, per (t, h)) and column sums (phi_col, per (s, h); two tiles
//          add to the columns of the first, so phi_col is accumulated).
constexpr int kPsiThreads = 512;

struct PsiSmem {
    uint8_t yt[2][kT * 128];      // dY rows of the tile, heads h and h + 1: A (rows t, K = p), K-major
    uint8_t xs[2][256 * 128];     // X rows of the sources: B (rows s, K = p), K-major
    uint8_t ct[2][kT * 128];      // kPhi: C rows of the tile, K-major A (two K blocks)
    uint8_t bs[2][256 * 128];     // kPhi: B rows of the sources, K-major B (two K blocks)
    float c2[2][256];             // cum log2(e) of tokens 0 .. ns - 1 (by head parity)
    float e2[2][256];             // c2 - log2(dt): exp2(c2_t - e2_s) = L[t,s] dt_s
    float bfac[2][256];           // exp2(c2_r - e2_s), r = last token of s's group of 32
    float rowacc[kT];             // kPhi: row sums of the head
    float colacc[256];            // kPhi: column sums of the head
    uint64_t full[2];             // a head's dY and X tiles landed in buffer 0 / 1
    uint64_t mma[2];              // a head's score chain done (heads of parity 0 / 1)
    uint64_t drain;
    uint32_t tmem_base;
};

// Sums v[i] over the 32 lanes for i = 0..31; lane l returns the sum of v[l].
__device__ __forceinline__ float warp_colsum32(float (&v)[32], int lane) {
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) {
        const bool upper = (lane & off) != 0;
#pragma unroll
        for (int i = 0; i < off; ++i) {
            const float send = upper ? v[i] : v[i + off];
            const float keep = upper ? v[i + off] : v[i];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, off);
        }
    }
    return v[0];
}

// The heads' dY and X tiles arrive by TMA two heads ahead (double-buffered); in
// the Psi mode the scores are double-buffered in TMEM too, so head h + 1's MMA
// chain runs under head h's epilogue. cum and dt of head h + 1 are prefetched
// into registers during head h.
template <bool kPhi>
__global__ void __launch_bounds__(kPsiThreads, 1)
psi_kernel(const __grid_constant__ CUtensorMap tm_X, const __grid_constant__ CUtensorMap tm_dY,
           const float* __restrict__ dt, const float* __restrict__ cum,
           const __nv_bfloat16* __restrict__ Bm, const __nv_bfloat16* __restrict__ Cm,
           uint8_t* __restrict__ psi, float* __restrict__ phi_row, float* __restrict__ phi_col,
           int L, int H, int S, int Mc, unsigned long long wait_limit_ns) {
    extern __shared__ uint8_t smem_raw[];
    PsiSmem& sm = *reinterpret_cast<PsiSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                              ~(uintptr_t)1023);
    // the tile in z, the slowest launch index: tiles with the most sources start first
    const int tt = (int)(gridDim.z - 1 - blockIdx.z), c = blockIdx.x, b = blockIdx.y;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int row = tid & (kT - 1), quarter = tid >> 7;
    const int ns = (tt + 1) * kT;
    const i64 tok0 = (i64)b * L + (i64)c * S;
    const uint32_t lane_addr = (uint32_t)(32 * (warp & 3)) << 16;
    const int tl = tt * kT + row;
    const int tl_warp_max = tt * kT + 32 * (warp & 3) + 31;
    const int sq = ns / 4, s_lo = quarter * sq;  // 32 or 64 sources of this thread
    constexpr uint32_t kColCB = 256;
    const uint32_t head_bytes = (uint32_t)(kT + ns) * 128u;

    if (tid == 0) {
        for (int u = 0; u < 2; ++u) {
            tc::mbar_init(&sm.full[u], 1);
            tc::mbar_init(&sm.mma[u], 1);
        }
        tc::mbar_init(&sm.drain, 1);
        tc::fence_barrier_init();
        tc::tma_prefetch_map(&tm_X);
        tc::tma_prefetch_map(&tm_dY);
    }
    if (warp == 0) {
        tc::tmem_alloc(&sm.tmem_base, 512);
        tc::tmem_relinquish();
    }
    if (kPhi) {
        for (int i = tid; i < kT * 16; i += kPsiThreads) {
            const int r = i / 16, q = i % 16;
            *reinterpret_cast<uint4*>(sm.ct[q / 8] + sw128((uint32_t)r, (uint32_t)(q % 8) * 16u)) =
                reinterpret_cast<const uint4*>(Cm + (tok0 + tt * kT + r) * kN)[q];
        }
        for (int i = tid; i < ns * 16; i += kPsiThreads) {
            const int r = i / 16, q = i % 16;
            *reinterpret_cast<uint4*>(sm.bs[q / 8] + sw128((uint32_t)r, (uint32_t)(q % 8) * 16u)) =
                reinterpret_cast<const uint4*>(Bm + (tok0 + r) * kN)[q];
        }
        for (int i = tid; i < kT; i += kPsiThreads) sm.rowacc[i] = 0.0f;
        for (int i = tid; i < 256; i += kPsiThreads) sm.colacc[i] = 0.0f;
        tc::fence_proxy_async_shared();
    }
    // cum and dt of head hh for source tid (tid < ns)
    auto head_c2e2 = [&](int hh, float& c2v, float& e2v) {
        c2v = cum[(((i64)b * H + hh) * Mc + c) * S + tid] * kLog2e;
        e2v = c2v - log2f(dt[(tok0 + tid) * H + hh]);  // dt = 0 gives +inf: a zero weight
    };
    if (tid < ns) head_c2e2(0, sm.c2[0][tid], sm.e2[0][tid]);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = sm.tmem_base;

    // thread 0: the dY rows of the tile and the X rows of the sources of head hh into
    // buffer hh & 1 (boxes of 128 rows x 64 columns at column hh P)
    auto issue_head = [&](int hh) {
        const int hb = hh & 1;
        tc::mbar_arrive_expect_tx(&sm.full[hb], head_bytes);
        tc::tma_load_2d(sm.yt[hb], &tm_dY, hh * kP, (int)(tok0 + tt * kT), &sm.full[hb]);
        for (int r0 = 0; r0 < ns; r0 += kT)
            tc::tma_load_2d(sm.xs[hb] + r0 * 128, &tm_X, hh * kP, (int)(tok0 + r0), &sm.full[hb]);
    };
    // thread 0: scores dY X^T of head hh (its tiles landed) into TMEM, committed on mma[hh & 1]
    auto issue_scores = [&](int hh) {
        const int hb = hh & 1;
        const uint32_t id = idesc_bf16(false, false, kT, (uint32_t)ns);
        const uint32_t dcol = kPhi ? 0u : 256u * (uint32_t)hb;
        for (int ks = 0; ks < kP / 16; ++ks) {
            const uint64_t ad = tc::smem_desc_sw128(tc::smem_u32(sm.yt[hb]) + 32u * ks, 16u, 1024u);
            const uint64_t bd = tc::smem_desc_sw128(tc::smem_u32(sm.xs[hb]) + 32u * ks, 16u, 1024u);
            mma_ss(tmem + dcol, ad, bd, id, ks > 0 ? 1u : 0u);
        }
        tc::mma_commit(&sm.mma[hb]);
    };
    int copies = 0, mmas = 0;  // heads whose tiles / score chains thread 0 issued
    if (tid == 0) {
        for (int hh = 0; hh < H && hh < 2; ++hh) issue_head(hh);
        copies = H < 2 ? H : 2;
        if (kPhi) {  // C B^T of the tile, committed with the first head's scores
            const uint32_t id = idesc_bf16(false, false, kT, (uint32_t)ns);
            for (int ks = 0; ks < kN / 16; ++ks) {
                const uint64_t ad = tc::smem_desc_sw128(tc::smem_u32(sm.ct[ks / 4]) + 32u * (ks % 4), 16u, 1024u);
                const uint64_t bd = tc::smem_desc_sw128(tc::smem_u32(sm.bs[ks / 4]) + 32u * (ks % 4), 16u, 1024u);
                mma_ss(tmem + kColCB, ad, bd, id, ks > 0 ? 1u : 0u);
            }
        }
        if (H > 0) {
            if (tc::mbar_wait(&sm.full[0], 0, wait_limit_ns, nullptr)) {
                tc::tc_fence_after();
                issue_scores(0);
                mmas = 1;
            } else {
                atomicCAS(&g_sbwd_tc_status, 0, 48);  // the wait on mma[0] then runs out
            }
        }
    }
    float acc[kPhi ? 1 : 64];
#pragma unroll
    for (int i = 0; i < (kPhi ? 1 : 64); ++i) acc[i] = 0.0f;
    bool ok = true;
    for (int h = 0; h < H && ok; ++h) {
        const int hb = h & 1;
        if (tid < ns) sm.bfac[hb][tid] = ex2_approx(sm.c2[hb][tid | 31] - sm.e2[hb][tid]);
        float nc2 = 0.0f, ne2 = 0.0f;
        if (h + 1 < H && tid < ns) head_c2e2(h + 1, nc2, ne2);
        ok = cta_wait(&sm.mma[hb], (uint32_t)((h >> 1) & 1), wait_limit_ns, 41);
        if (!ok) break;
        // head h + 1's cum and dt into the other slot (its head h - 1 values were last read
        // before the previous closing barrier)
        if (h + 1 < H && tid < ns) {
            sm.c2[hb ^ 1][tid] = nc2;
            sm.e2[hb ^ 1][tid] = ne2;
        }
        if (tid == 0) {
            // buffer hb's tiles were read by head h's MMAs: head h + 2's go there
            if (h + 2 < H) {
                issue_head(h + 2);
                ++copies;
            }
            // Psi mode: head h + 1's scores into the other TMEM buffer (last read by head
            // h - 1's epilogue, finished at its closing barrier)
            if (!kPhi && h + 1 < H) {
                if (tc::mbar_wait(&sm.full[hb ^ 1], (uint32_t)(((h + 1) >> 1) & 1), wait_limit_ns, nullptr)) {
                    tc::tc_fence_after();
                    issue_scores(h + 1);
                    ++mmas;
                } else {
                    atomicCAS(&g_sbwd_tc_status, 0, 48);
                }
            }
        }
        const uint32_t dcol = kPhi ? 0u : 256u * (uint32_t)hb;
        const float* c2h = sm.c2[hb];
        const float* e2h = sm.e2[hb];
        const float* bfh = sm.bfac[hb];
        const float c2t = c2h[tl];
        float rsum = 0.0f;
#pragma unroll
        for (int g0 = 0; g0 < 64; g0 += 32) {
            const int s0 = s_lo + g0;
            if (g0 >= sq || s0 > tl_warp_max) continue;  // warp-uniform
            float v[32];
            tmem_ld32(tmem + lane_addr + dcol + (uint32_t)s0, v);
            // v <- L[t,s] dt_s scores[t,s] (zero for s > t)
            if (s0 + 31 <= tl) {  // the whole group at or before t: factored decay
                const float a = ex2_approx(c2t - c2h[s0 + 31]);
#pragma unroll
                for (int i = 0; i < 32; ++i) v[i] *= bfh[s0 + i] * a;
            } else {
#pragma unroll
                for (int i = 0; i < 32; ++i) v[i] = s0 + i <= tl ? v[i] * ex2_approx(c2t - e2h[s0 + i]) : 0.0f;
            }
            if constexpr (kPhi) {
                float w[32];
                tmem_ld32(tmem + lane_addr + kColCB + (uint32_t)s0, w);
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    v[i] *= w[i];
                    rsum += v[i];
                }
                const float cs = warp_colsum32(v, lane);  // this warp's rows, column s0 + lane
                atomicAdd(&sm.colacc[s0 + lane], cs);
            } else {
#pragma unroll
                for (int i = 0; i < 32; ++i) acc[g0 + i] += v[i];
            }
        }
        if constexpr (kPhi) {
            atomicAdd(&sm.rowacc[row], rsum);
            __syncthreads();
            for (int i = tid; i < kT; i += kPsiThreads) {
                phi_row[(tok0 + tt * kT + i) * H + h] = sm.rowacc[i];
                sm.rowacc[i] = 0.0f;
            }
            for (int i = tid; i < ns; i += kPsiThreads) {
                atomicAdd(phi_col + (tok0 + i) * H + h, sm.colacc[i]);
                sm.colacc[i] = 0.0f;
            }
        }
        tc::tc_fence_before();
        __syncthreads();  // TMEM reads, slots and sums of head h are done
        if (kPhi && tid == 0 && h + 1 < H) {  // one TMEM score buffer: head h + 1 starts now
            tc::tc_fence_after();
            if (tc::mbar_wait(&sm.full[hb ^ 1], (uint32_t)(((h + 1) >> 1) & 1), wait_limit_ns, nullptr)) {
                issue_scores(h + 1);
                ++mmas;
            } else {
                atomicCAS(&g_sbwd_tc_status, 0, 48);
            }
        }
    }
    if (tid == 0) {
        // never free TMEM under an MMA nor leave a tile copy in flight behind
        if (!ok && mmas > 0) {
            tc::mma_commit(&sm.drain);
            if (!tc::mbar_wait(&sm.drain, 0, kDrainLimitNs, nullptr)) atomicCAS(&g_sbwd_tc_status, 0, 42);
        }
        for (int k = copies - 1; k >= 0 && k >= copies - 2; --k)
            if (!tc::mbar_wait(&sm.full[k & 1], (uint32_t)((k >> 1) & 1), kDrainLimitNs, nullptr))
                atomicCAS(&g_sbwd_tc_status, 0, 49);
    }
    if (!kPhi && ok) {
        uint8_t* base = psi + (i64)(b * Mc + c) * psi_chunk_bytes(S);
        const i64 part = (i64)(S / 64) * S * 128;
#pragma unroll
        for (int g8 = 0; g8 < 64; g8 += 8) {
            if (g8 >= sq) continue;
            const int s = s_lo + g8;
            uint4 hi, lo;
            split8(acc + g8, hi, lo);
            const i64 o = (i64)(s / 64) * S * 128 + sw128((uint32_t)tl, (uint32_t)(s % 64) * 2u);
            *reinterpret_cast<uint4*>(base + o) = hi;
            *reinterpret_cast<uint4*>(base + part + o) = lo;
        }
        // the tile's rows beyond its sources are zero
        const int zc = (S - ns) / 8;  // 16-byte chunks per row
        for (int i = tid; i < kT * zc; i += kPsiThreads) {
            const int r = i / zc, s = ns + 8 * (i % zc);
            const i64 o = (i64)(s / 64) * S * 128 + sw128((uint32_t)(tt * kT + r), (uint32_t)(s % 64) * 2u);
            *reinterpret_cast<uint4*>(base + o) = make_uint4(0, 0, 0, 0);
            *reinterpret_cast<uint4*>(base + part + o) = make_uint4(0, 0, 0, 0);
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        __syncwarp();
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, 512);
    }
}

// ---------------------------------------------------------------- dC / dB
// Warps 0..15 stage each unit's register-formed operand part; warp 16 issues the
// unit's bulk copy and its MMAs. formed[b] (one arrival per staging warp) and
// full[b] (the copy) hand buffer b to the MMA thread, mma_done[b] hands it back,
// so no staging warp waits for the MMA issue.
constexpr int kDcFormThreads = 512;
constexpr int kDcThreads = kDcFormThreads + 32;
constexpr int kUnit = 16384;  // one operand slot

struct DcSmem {
    uint8_t slot[2][4][kUnit];  // per buffer: A hi, A lo, B (or B hi), B lo
    uint64_t full[2];           // the unit's 32 KiB bulk-copied part landed in buffer 0 / 1
    uint64_t formed[2];         // the staging warps' part is in buffer 0 / 1
    uint64_t mma_done[2];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
};

// kind 0: dC rows of a 128-token tile (accumulated into dC); kind 1: dB rows.
__global__ void __launch_bounds__(kDcThreads, 1)
dcdb_kernel(const __nv_bfloat16* __restrict__ X, const float* __restrict__ dt,
            const float* __restrict__ cum, const __nv_bfloat16* __restrict__ Bm,
            const __nv_bfloat16* __restrict__ Cm, const __nv_bfloat16* __restrict__ dY,
            const uint8_t* __restrict__ psi, const uint8_t* __restrict__ Hops,
            const uint8_t* __restrict__ Dops, float* __restrict__ dC, float* __restrict__ dB, int L,
            int H, int S, int Mc, unsigned long long wait_limit_ns) {
    extern __shared__ uint8_t smem_raw[];
    DcSmem& sm = *reinterpret_cast<DcSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                            ~(uintptr_t)1023);
    const int tiles = S / kT;
    const int kind = (int)blockIdx.x / tiles, tt = (int)blockIdx.x % tiles;
    const int c = blockIdx.y, b = blockIdx.z;
    const int tid = threadIdx.x, warp = tid >> 5;
    const i64 tok0 = (i64)b * L + (i64)c * S;
    const uint8_t* pbase = psi + (i64)(b * Mc + c) * psi_chunk_bytes(S);
    const i64 ppart = (i64)(S / 64) * S * 128;
    // K units: intra blocks of 64 tokens, then one per head (dC: only after chunk 0)
    const int nintra = kind == 0 ? (tt + 1) * kT / 64 : (S - tt * kT) / 64;
    const int ninter = (kind == 0 && c == 0) ? 0 : H;
    const int nunits = nintra + ninter;

    if (tid == 0) {
        for (int u = 0; u < 2; ++u) {
            tc::mbar_init(&sm.full[u], 1);
            tc::mbar_init(&sm.formed[u], kDcFormThreads / 32);
            tc::mbar_init(&sm.mma_done[u], 1);
        }
        tc::mbar_init(&sm.drain, 1);
        sm.abort = 0;
        tc::fence_barrier_init();
    }
    if (warp == 0) {
        tc::tmem_alloc(&sm.tmem_base, 128);
        tc::tmem_relinquish();
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = sm.tmem_base;
    const float* cumb = cum + (i64)b * H * Mc * S;  // + (h Mc + c) S + t
    volatile int* abort = &sm.abort;
    auto fail_code = [&](int code) {
        *abort = 1;
        atomicCAS(&g_sbwd_tc_status, 0, code);
    };

    if (tid < kDcFormThreads) {
        // a unit's global inputs for this thread, loaded one unit ahead: intra, w = two
        // pieces of B (dC) or C (dB) rows; per head, w = two pieces of dY (dC) or X (dB)
        // rows, f = cum_t (dC) or dt_s (dB), g = cum_s and e = cum_end (dB)
        struct DcRegs {
            uint4 w[2];
            float f[2], g[2], e;
        };
        auto load_unit = [&](int u, DcRegs& R) {
            if (u < nintra) {
                const int r0 = kind == 0 ? 64 * u : tt * kT + 64 * u;
                const __nv_bfloat16* src = kind == 0 ? Bm : Cm;
#pragma unroll
                for (int k = 0; k < 2; ++k) {
                    const int i = tid + k * kDcFormThreads, r = i / 16, q = i % 16;
                    R.w[k] = reinterpret_cast<const uint4*>(src + (tok0 + r0 + r) * kN)[q];
                }
            } else {
                const int h = u - nintra;
                const float* cumh = cumb + ((i64)h * Mc + c) * S;
                R.e = kind == 0 ? 0.0f : cumh[S - 1];
#pragma unroll
                for (int k = 0; k < 2; ++k) {
                    const int i = tid + k * kDcFormThreads, r = i / 8, q = i % 8;
                    const int t = tt * kT + r;
                    const i64 tok = tok0 + t;
                    if (kind == 0) {
                        R.f[k] = cumh[t];
                        R.w[k] = reinterpret_cast<const uint4*>(dY + (tok * H + h) * kP)[q];
                    } else {
                        R.f[k] = dt[tok * H + h];
                        R.g[k] = cumh[t];
                        R.w[k] = reinterpret_cast<const uint4*>(X + (tok * H + h) * kP)[q];
                    }
                }
            }
        };
        DcRegs cur, nxt;
        if (nunits > 0) load_unit(0, cur);
        for (int u = 0; u < nunits; ++u) {
            const int bi = u & 1;
            if (u + 1 < nunits) load_unit(u + 1, nxt);  // in flight under this unit's wait and stores
            // buffer bi was read by the MMAs of unit u - 2
            if (u >= 2) {
                const bool got = tc::mbar_wait(&sm.mma_done[bi], (uint32_t)(((u - 2) >> 1) & 1), wait_limit_ns, abort);
                if (!__all_sync(0xffffffffu, got)) {
                    if ((tid & 31) == 0) fail_code(43);
                    break;
                }
            }
            uint8_t* a_hi = sm.slot[bi][0];
            uint8_t* a_lo = sm.slot[bi][1];
            uint8_t* b0 = sm.slot[bi][2];
            if (u < nintra) {
                // B: 64 token rows of B (dC) or C (dB), MN-major N = 128: [n block][64 rows][128 bytes]
#pragma unroll
                for (int k = 0; k < 2; ++k) {
                    const int i = tid + k * kDcFormThreads, r = i / 16, q = i % 16;
                    *reinterpret_cast<uint4*>(b0 + (q / 8) * 8192 + sw128((uint32_t)r, (uint32_t)(q % 8) * 16u)) = cur.w[k];
                }
            } else {
                // A: exp(cum_t) dY_t (dC) or exp(cum_end - cum_s) dt_s X_s (dB) of head h, K = p, split
#pragma unroll
                for (int k = 0; k < 2; ++k) {
                    const int i = tid + k * kDcFormThreads, r = i / 8, q = i % 8;
                    const float fk = kind == 0 ? expf(cur.f[k]) : expf(cur.e - cur.g[k]) * cur.f[k];
                    const uint32_t ww[4] = {cur.w[k].x, cur.w[k].y, cur.w[k].z, cur.w[k].w};
                    float v[8];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        v[2 * e] = bf_lo(ww[e]) * fk;
                        v[2 * e + 1] = bf_hi(ww[e]) * fk;
                    }
                    uint4 hi, lo;
                    split8(v, hi, lo);
                    const uint32_t o = sw128((uint32_t)r, (uint32_t)q * 16u);
                    *reinterpret_cast<uint4*>(a_hi + o) = hi;
                    *reinterpret_cast<uint4*>(a_lo + o) = lo;
                }
                // B: H_[c-1] (dC) or d(dH_c) (dB) of head h, [n][p] hi | lo, K-major (rows n,
                // K = p): the MMA thread's bulk copy
            }
            tc::fence_proxy_async_shared();
            __syncwarp();
            if ((tid & 31) == 0) tc::mbar_arrive(&sm.formed[bi]);
            cur = nxt;
        }
        // the last unit's MMAs (and with them every earlier one) are done
        if (!*abort && nunits > 0) {
            const int last = nunits - 1;
            const bool got = tc::mbar_wait(&sm.mma_done[last & 1], (uint32_t)((last >> 1) & 1), wait_limit_ns, abort);
            if (!__all_sync(0xffffffffu, got) && (tid & 31) == 0) fail_code(44);
        }
    } else if (tid == kDcFormThreads) {
        int issued = 0;  // units whose MMAs were issued
        int copied = 0;  // units whose bulk copy was issued
        for (int u = 0; u < nunits; ++u) {
            const int bi = u & 1;
            if (u >= 2 && !tc::mbar_wait(&sm.mma_done[bi], (uint32_t)(((u - 2) >> 1) & 1), wait_limit_ns, abort)) {
                fail_code(43);
                break;
            }
            uint8_t* a_hi = sm.slot[bi][0];
            uint8_t* a_lo = sm.slot[bi][1];
            uint8_t* b0 = sm.slot[bi][2];
            uint8_t* b1 = sm.slot[bi][3];
            const bool intra = u < nintra;
            // Every unit has one 32 KiB part that is already laid out in global memory: the
            // Psi blocks (intra) or the H / d(dH) operand tile (per head); the bulk copy
            // brings it in while the staging warps form the rest.
            tc::mbar_arrive_expect_tx(&sm.full[bi], 32768u);
            if (!intra) {
                const int h = u - nintra;
                const uint8_t* tile = (kind == 0 ? Hops : Dops) + (((i64)b * Mc + c) * H + h) * 32768;
                tc::bulk_g2s(b0, tile, 32768u, &sm.full[bi]);  // into b0 and b1
            } else if (kind == 0) {
                // A: Psi rows of the tile, column block u (K = 64 sources), K-major
                for (int part = 0; part < 2; ++part)
                    tc::bulk_g2s(part ? a_lo : a_hi,
                                 pbase + part * ppart + (i64)u * S * 128 + (i64)tt * kT * 128,
                                 (uint32_t)(kT * 128), &sm.full[bi]);
            } else {
                // A: Psi^T, M = the tile's 128 sources (column blocks 2 tt, 2 tt + 1), K = 64
                // target rows from tt * 128 + 64 u, MN-major: [block][64 rows][128 bytes]
                const int t0u = tt * kT + 64 * u;
                for (int part = 0; part < 2; ++part)
                    for (int blk = 0; blk < 2; ++blk)
                        tc::bulk_g2s((part ? a_lo : a_hi) + blk * 8192,
                                     pbase + part * ppart + (i64)(2 * tt + blk) * S * 128 + (i64)t0u * 128,
                                     8192u, &sm.full[bi]);
            }
            copied = u + 1;
            if (!tc::mbar_wait(&sm.formed[bi], (uint32_t)((u >> 1) & 1), wait_limit_ns, abort)) {
                fail_code(48);
                break;
            }
            if (!tc::mbar_wait(&sm.full[bi], (uint32_t)((u >> 1) & 1), wait_limit_ns, abort)) {
                fail_code(46);
                break;
            }
            tc::tc_fence_after();
            const uint32_t sa_hi = tc::smem_u32(a_hi), sa_lo = tc::smem_u32(a_lo);
            const uint32_t sb0 = tc::smem_u32(b0), sb1 = tc::smem_u32(b1);
            if (intra) {
                const uint32_t id = idesc_bf16(kind == 1, true, kT, kN);
                for (int part = 0; part < 2; ++part) {
                    const uint32_t sa = part ? sa_lo : sa_hi;
                    for (int ks = 0; ks < 4; ++ks) {
                        const uint64_t ad = kind == 0 ? tc::smem_desc_sw128(sa + 32u * ks, 16u, 1024u)
                                                      : tc::smem_desc_sw128(sa + 2048u * ks, 8192u, 1024u);
                        const uint64_t bd = tc::smem_desc_sw128(sb0 + 2048u * ks, 8192u, 1024u);
                        mma_ss(tmem, ad, bd, id, (u > 0 || part > 0 || ks > 0) ? 1u : 0u);
                    }
                }
            } else {
                const uint32_t id = idesc_bf16(false, false, kT, kN);
                for (int term = 0; term < 3; ++term) {  // a_hi b_hi, a_lo b_hi, a_hi b_lo
                    const uint32_t sa = term == 1 ? sa_lo : sa_hi;
                    const uint32_t sb = term == 2 ? sb1 : sb0;
                    for (int ks = 0; ks < 4; ++ks) {
                        const uint64_t ad = tc::smem_desc_sw128(sa + 32u * ks, 16u, 1024u);
                        const uint64_t bd = tc::smem_desc_sw128(sb + 32u * ks, 16u, 1024u);
                        mma_ss(tmem, ad, bd, id, (u > 0 || term > 0 || ks > 0) ? 1u : 0u);
                    }
                }
            }
            tc::mma_commit(&sm.mma_done[bi]);
            issued = u + 1;
        }
        if (*abort && issued > 0) {  // let the MMAs in flight finish before TMEM is freed
            tc::mma_commit(&sm.drain);
            if (!tc::mbar_wait(&sm.drain, 0, kDrainLimitNs, nullptr)) atomicCAS(&g_sbwd_tc_status, 0, 45);
        }
        // never leave a copy in flight behind: the last copy into each buffer
        for (int k = copied - 1; k >= 0 && k >= copied - 2; --k)
            if (!tc::mbar_wait(&sm.full[k & 1], (uint32_t)((k >> 1) & 1), kDrainLimitNs, nullptr))
                atomicCAS(&g_sbwd_tc_status, 0, 47);
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    if (!*abort && tid < kDcFormThreads) {
        // thread (row, quarter): 32 columns of its token row
        const int r = tid & (kT - 1), qc = tid >> 7;
        const uint32_t lane_addr = (uint32_t)(32 * (warp & 3)) << 16;
        const i64 tok = tok0 + tt * kT + r;
        float* dst = (kind == 0 ? dC : dB) + tok * kN + 32 * qc;
        {
            float v[32];
            tmem_ld32(tmem + lane_addr + (uint32_t)(32 * qc), v);
            float4* d4 = reinterpret_cast<float4*>(dst);
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                float4 o = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                if (kind == 0) {
                    const float4 p = d4[q];
                    o.x += p.x; o.y += p.y; o.z += p.z; o.w += p.w;
                }
                d4[q] = o;
            }
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        __syncwarp();
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, 128);
    }
}

// ------------------------------------------------------------- passing
// Reverse pass over the chunks for one (1024-element slab of the N x P state,
// h, b): with adj the adjoint of H_c (zero after the last chunk),
//   d(dH_c) = adj + dM_c   (written as split operand tiles),
//   d(cum_end_c) += exp(cum_end_c) <adj, H_[c-1]>,
//   adj <- exp(cum_end_c) adj + Z_c.
// The slabs of Z, dM and H_[c-1] stream through a ring of shared-memory
// stages filled by 4 KiB bulk copies, chunks in reverse order.
constexpr int kBpThreads = 256;
constexpr int kBpElems = 4;
constexpr int kBpSlab = kBpThreads * kBpElems;  // 1024 elements
constexpr int kBpStages = 6;

struct BpSmem {
    float z[kBpStages][kBpSlab];
    float m[kBpStages][kBpSlab];
    float hp[kBpStages][kBpSlab];
    float red[kBpThreads / 32];
    uint64_t full[kBpStages];
};

__global__ void __launch_bounds__(kBpThreads)
bwd_passing_tc_kernel(const float* __restrict__ Z, const float* __restrict__ dM,
                      const float* __restrict__ Hprev, const float* __restrict__ cum,
                      float* __restrict__ dcum_end, uint8_t* __restrict__ Dops, int H, int S, int Mc,
                      unsigned long long wait_limit_ns, int withhold) {
    extern __shared__ uint8_t smem_raw[];
    BpSmem& sm = *reinterpret_cast<BpSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~(uintptr_t)127);
    constexpr int NP = kN * kP;
    const int slab = blockIdx.x, h = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
    const int lane = tid & 31, warp = tid >> 5;
    const int e0 = slab * kBpSlab + tid * kBpElems;
    const int n = e0 / kP, p = e0 % kP;
    const i64 cstride = (i64)H * NP;
    const i64 base = ((i64)b * Mc * H + h) * NP + (i64)slab * kBpSlab;  // + c cstride
    uint8_t* dop = Dops + ((i64)b * Mc * H + h) * 32768 + sw128((uint32_t)n, (uint32_t)p * 2u);
    const i64 dstride = (i64)H * 32768;
    const float* cumh = cum + ((i64)b * H + h) * (i64)Mc * S;
    const uint32_t bytes = (uint32_t)(kBpSlab * 4) * (dM != nullptr ? 3u : 2u);

    if (tid == 0) {
        for (int k = 0; k < kBpStages; ++k) tc::mbar_init(&sm.full[k], 1);
        tc::fence_barrier_init();
    }
    __syncthreads();
    int issued = 0;  // reverse-order steps whose copies thread 0 issued
    auto issue = [&](int k) {  // step k = chunk Mc - 1 - k
        const int c = Mc - 1 - k, stg = k % kBpStages;
        const i64 off = base + (i64)c * cstride;
        tc::mbar_arrive_expect_tx(&sm.full[stg], bytes);
        tc::bulk_g2s(sm.z[stg], Z + off, (uint32_t)(kBpSlab * 4), &sm.full[stg]);
        tc::bulk_g2s(sm.hp[stg], Hprev + off, (uint32_t)(kBpSlab * 4), &sm.full[stg]);
        if (dM != nullptr) tc::bulk_g2s(sm.m[stg], dM + off, (uint32_t)(kBpSlab * 4), &sm.full[stg]);
        ++issued;
    };
    // (withhold: the failure-path test hook; every wait on the slabs then runs out)
    if (tid == 0 && !withhold)
        for (int k = 0; k < min(kBpStages, Mc); ++k) issue(k);
    float adj[kBpElems] = {0.0f, 0.0f, 0.0f, 0.0f};
    bool ok = true;
    int k = 0;
    for (; k < Mc; ++k) {
        const int c = Mc - 1 - k, stg = k % kBpStages;
        const bool got = tc::mbar_wait(&sm.full[stg], (uint32_t)((k / kBpStages) & 1), wait_limit_ns, nullptr);
        float part = 0.0f;
        if (got) {
            const float dec = expf(cumh[(i64)c * S + S - 1]);
            const float4 zv = *reinterpret_cast<const float4*>(&sm.z[stg][tid * kBpElems]);
            const float4 hv = *reinterpret_cast<const float4*>(&sm.hp[stg][tid * kBpElems]);
            float4 mv = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            if (dM != nullptr) mv = *reinterpret_cast<const float4*>(&sm.m[stg][tid * kBpElems]);
            const float zz[4] = {zv.x, zv.y, zv.z, zv.w}, hh[4] = {hv.x, hv.y, hv.z, hv.w};
            const float mm[4] = {mv.x, mv.y, mv.z, mv.w};
            float dd[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                part = fmaf(dec * adj[i], hh[i], part);
                dd[i] = adj[i] + mm[i];
                adj[i] = fmaf(dec, adj[i], zz[i]);
            }
            uint4 hi, lo;
            {
                uint32_t hw[2], lw[2];
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const __nv_bfloat162 h2 = __floats2bfloat162_rn(dd[2 * e], dd[2 * e + 1]);
                    const float2 hf = __bfloat1622float2(h2);
                    hw[e] = *reinterpret_cast<const uint32_t*>(&h2);
                    lw[e] = pack_bf16(dd[2 * e] - hf.x, dd[2 * e + 1] - hf.y);
                }
                hi = make_uint4(hw[0], hw[1], 0, 0);
                lo = make_uint4(lw[0], lw[1], 0, 0);
            }
            uint8_t* t = dop + (i64)c * dstride;
            *reinterpret_cast<uint2*>(t) = make_uint2(hi.x, hi.y);
            *reinterpret_cast<uint2*>(t + 16384) = make_uint2(lo.x, lo.y);
        } else {
            atomicCAS(&g_sbwd_tc_status, 0, 46);
        }
        for (int off = 16; off > 0; off >>= 1) part += __shfl_xor_sync(0xffffffffu, part, off);
        if (lane == 0) sm.red[warp] = part;
        // every thread has read the stage before it is refilled; the partial sums are in
        ok = __syncthreads_and(got ? 1 : 0) != 0;
        if (!ok) break;
        if (tid == 0) {
            float sum = 0.0f;
            for (int w = 0; w < kBpThreads / 32; ++w) sum += sm.red[w];
            atomicAdd(dcum_end + ((i64)b * H + h) * Mc + c, sum);
            if (!withhold && k + kBpStages < Mc) issue(k + kBpStages);
        }
        __syncthreads();  // red is reused by the next step
    }
    if (!ok && tid == 0) {  // the copies in flight land before the CTA exits
        for (int kk = k; kk < issued; ++kk)
            if (!tc::mbar_wait(&sm.full[kk % kBpStages], (uint32_t)((kk / kBpStages) & 1), kDrainLimitNs, nullptr)) {
                atomicCAS(&g_sbwd_tc_status, 0, 47);
                break;
            }
    }
}

// ------------------------------------------------------------- finalize
// One CTA of S threads per (c, h, b): d(cum) of the chunk,
//   d(cum_t) = phi_row_t + rowI_t - phi_col_t - kappa_t,  kappa_t = dt_t xi_t,
// plus sum_s kappa_s and the passing term at the chunk's last token; then the
// reverse sums, d(dt) and the chunk's share of dA_h.
__global__ void finalize_kernel(const float* __restrict__ dt, const float* __restrict__ A,
                                const float* __restrict__ phi_row, const float* __restrict__ phi_col,
                                const float* __restrict__ rowI, const float* __restrict__ xi,
                                const float* __restrict__ dcum_end, float* __restrict__ ddt,
                                float* __restrict__ dA, int L, int H, int S, int Mc) {
    __shared__ float sv[256];
    __shared__ float red[8];
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const i64 idx = ((i64)b * L + (i64)c * S + t) * H + h;
    const float dtv = dt[idx];
    const float pc = phi_col[idx], xv = xi[idx];
    const float kap = dtv * xv;
    float dcum = phi_row[idx] + rowI[idx] - pc - kap;
    float k = kap;
    for (int off = 16; off > 0; off >>= 1) k += __shfl_xor_sync(0xffffffffu, k, off);
    if (lane == 0) red[warp] = k;
    __syncthreads();
    if (t == S - 1) {
        float ks = 0.0f;
        for (int w = 0; w < S / 32; ++w) ks += red[w];
        dcum += ks + dcum_end[((i64)b * H + h) * Mc + c];
    }
    // reverse inclusive scan: run_t = sum_{k >= t} dcum_k
    sv[t] = dcum;
    __syncthreads();
    for (int off = 1; off < S; off <<= 1) {
        const float add = t + off < S ? sv[t + off] : 0.0f;
        __syncthreads();
        sv[t] += add;
        __syncthreads();
    }
    const float run = sv[t];
    // d(dt) direct part: X_t . Y'_t = phi_col_t / dt_t + xi_t
    ddt[idx] = (dtv != 0.0f ? pc / dtv : 0.0f) + xv + A[h] * run;
    float da = dtv * run;
    for (int off = 16; off > 0; off >>= 1) da += __shfl_xor_sync(0xffffffffu, da, off);
    __syncthreads();
    if (lane == 0) red[warp] = da;
    __syncthreads();
    if (t == 0) {
        float s = 0.0f;
        for (int w = 0; w < S / 32; ++w) s += red[w];
        atomicAdd(dA + h, s);
    }
}

}  // namespace

// Workspace of the tensor-core scan backward.
size_t scan_bwd_tc_workspace(int64_t B, int64_t L, int64_t H, int64_t S) {
    const int64_t M = L / S;
    auto al = [](size_t x) { return (x + 255) & ~(size_t)255; };
    const size_t states = (size_t)(B * M * H) * kN * kP * 4;
    return al((size_t)(B * H * M * S) * 4)        // cum
           + 2 * al(states)                        // H_[c-1] fp32; Z, then d(dH_c)
           + al((size_t)(B * H * M) * 4)           // d(cum_end)
           + 2 * al((size_t)(B * M * H) * 32768)   // Hops, Dops
           + 4 * al((size_t)(B * L * H) * 4)       // rowI, xi, phi_row, phi_col
           + al((size_t)(B * M) * psi_chunk_bytes((int)S));  // Psi
}

cudaError_t launch_chunk_scan_backward_tc(const ScanBwdArgs& a, void* ws,
                                          unsigned long long wait_limit_ns, cudaStream_t stream) {
    const ScanArgs& f = a.fwd;
    const int B = (int)f.B, L = (int)f.L, H = (int)f.H, S = (int)f.S, Mc = L / S, NP = kN * kP;
    auto al = [](size_t x) { return (x + 255) & ~(size_t)255; };
    const size_t states = (size_t)(f.B * Mc * f.H) * NP * 4;
    uint8_t* w = (uint8_t*)ws;
    float* cum = (float*)w;            w += al((size_t)(f.B * f.H * Mc * S) * 4);
    float* Hprev = (float*)w;          w += al(states);
    float* ZD = (float*)w;             w += al(states);
    float* dcum_end = (float*)w;       w += al((size_t)(f.B * f.H * Mc) * 4);
    uint8_t* Hops = w;                 w += al((size_t)(f.B * Mc * f.H) * 32768);
    uint8_t* Dops = w;                 w += al((size_t)(f.B * Mc * f.H) * 32768);
    const size_t tokh = al((size_t)(f.B * f.L * f.H) * 4);
    float* rowI = (float*)w;           w += tokh;
    float* xi = (float*)w;             w += tokh;
    float* phi_row = (float*)w;        w += tokh;
    float* phi_col = (float*)w;        w += tokh;
    uint8_t* psi = w;

    cudaError_t e = launch_scan_states_tc(f, cum, Hprev, Hops, wait_limit_ns, stream);
    if (e != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(dcum_end, 0, (size_t)(f.B * f.H * Mc) * 4, stream)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(a.dA, 0, (size_t)f.H * 4, stream)) != cudaSuccess) return e;
    if (!a.accumulate_dC &&
        (e = cudaMemsetAsync(a.dC, 0, (size_t)(f.B * f.L) * kN * 4, stream)) != cudaSuccess)
        return e;
    if ((e = launch_scan_bwd_inter_tc(f, cum, a.dY, ZD, wait_limit_ns, stream)) != cudaSuccess) return e;
    {
        const size_t smem = sizeof(BpSmem) + 128;
        if ((e = cudaFuncSetAttribute(bwd_passing_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)smem)) != cudaSuccess)
            return e;
        bwd_passing_tc_kernel<<<dim3(NP / kBpSlab, H, B), kBpThreads, smem, stream>>>(
            ZD, a.dM, Hprev, cum, dcum_end, Dops, H, S, Mc, wait_limit_ns, a.fwd.test_withhold);
        note_launches(1);
    }
    if ((e = launch_scan_bwd_output_tc(f, cum, Hops, Dops, a.dY, rowI, a.dX, xi, wait_limit_ns,
                                       stream)) != cudaSuccess)
        return e;
    if ((e = cudaMemsetAsync(phi_col, 0, (size_t)(f.B * f.L * f.H) * 4, stream)) != cudaSuccess) return e;
    // X and dY as (B L) x (H P) bf16 matrices, copied in 128 x 64 boxes (one head's rows)
    CUtensorMap tm_X, tm_dY;
    if (!encode_bf16_rows_map(&tm_X, f.X, (uint64_t)(f.B * f.L), (uint64_t)(H * kP), (uint64_t)H * kP * 2, kT, kP) ||
        !encode_bf16_rows_map(&tm_dY, a.dY, (uint64_t)(f.B * f.L), (uint64_t)(H * kP), (uint64_t)H * kP * 2, kT, kP))
        return cudaErrorNotSupported;
    for (int phi = 0; phi < 2; ++phi) {
        const size_t smem = sizeof(PsiSmem) + 1024;
        auto k = phi ? psi_kernel<true> : psi_kernel<false>;
        if ((e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) != cudaSuccess)
            return e;
        k<<<dim3(Mc, B, S / kT), kPsiThreads, smem, stream>>>(
            tm_X, tm_dY, f.dt, cum, (const __nv_bfloat16*)f.Bm, (const __nv_bfloat16*)f.Cm, psi, phi_row,
            phi_col, L, H, S, Mc, wait_limit_ns);
    }
    {
        const size_t smem = sizeof(DcSmem) + 1024;
        if ((e = cudaFuncSetAttribute(dcdb_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
            cudaSuccess)
            return e;
        dcdb_kernel<<<dim3(2 * (S / kT), Mc, B), kDcThreads, smem, stream>>>(
            (const __nv_bfloat16*)f.X, f.dt, cum, (const __nv_bfloat16*)f.Bm, (const __nv_bfloat16*)f.Cm,
            (const __nv_bfloat16*)a.dY, psi, Hops, Dops, a.dC, a.dB, L, H, S, Mc, wait_limit_ns);
    }
    finalize_kernel<<<dim3(Mc, H, B), S, 0, stream>>>(f.dt, f.A, phi_row, phi_col, rowI, xi, dcum_end,
                                                      a.ddt, a.dA, L, H, S, Mc);
    note_launches(4);
    return cudaGetLastError();
}

// Read and clear of the status word in one device-side exchange: a code that a
// kernel still running on another stream records is either returned now or kept
// for the next read, never lost between a read and a separate clear.
__device__ int g_sbwd_tc_status_taken;
__global__ void take_scan_bwd_tc_status_kernel() { g_sbwd_tc_status_taken = atomicExch(&g_sbwd_tc_status, 0); }

int take_scan_bwd_tc_status(cudaStream_t stream) {
    take_scan_bwd_tc_status_kernel<<<1, 1, 0, stream>>>();
    int v = 0;
    if (cudaGetLastError() != cudaSuccess ||
        cudaMemcpyFromSymbolAsync(&v, g_sbwd_tc_status_taken, sizeof(int), 0, cudaMemcpyDeviceToHost, stream) !=
            cudaSuccess ||
        cudaStreamSynchronize(stream) != cudaSuccess)
        return -1;
    return v;
}

}  // namespace dart
