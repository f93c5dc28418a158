// Backward of state-memory attention and the gated merge on the 5th-generation
// tensor cores, for bf16 token inputs with P = 64, N = 128, G = 1 and S a
// multiple of 128 (the chain rule on Sec. 3 / App. B.1; the paper prints no
// backward). With dR = SiLU(z) dY, g_{t,j} = exp(l_{t,j} - lse_t),
// s_{t,j} = dY_t . V_{t,j}, G1_t = sum_j g, D_t = SiLU(z_t) sum_j g s and
//   dl_{t,j} = g_{t,j} (SiLU(z_t) s_{t,j} G1_t - D_t)
// (the softmax gradient written with the weights' own sum G1, so that their
// rounding cancels), the gradients are
//   dQbar_t = sum_j dl_{t,j} W_j Ebar_t / sqrt(N),      W_j = r_j (.) M_j,
//   dEbar_t = sum_j dl_{t,j} W_j^T Qbar_t / sqrt(N),
//   dC_t    = sum_j g_{t,j} M_j dR_t,
//   dM_j    = T_j + r_j (.) G_j - (rowsum(M_j (.) G_j)) r_j^3 (.) M_j / P,
//   T_j = sum_t g_{t,j} C_t^T dR_t,  G_j = sum_t dl_{t,j} Qbar_t^T Ebar_t / sqrt(N),
// followed by the unit-weight RMSNorm backwards of Qbar and Ebar.
//
// Four kernels, after the operand kernel (sma_tc.cu), which here also writes
// M_j split bf16 hi + lo beside W_hi, W_lo and M16:
//   1. the forward kernel in its statistics mode (sma_tc.cu): g, s per (t, j)
//      and G1, D, dz per t, from the same U and V tiles as the forward;
//   2. sma_bwd_rows_kernel<true>, one CTA per (b, 128-token tile), all heads in
//      pairs: per job (head pair, memory j) U = Q W gives dEbar in registers;
//      the epilogue writes the A operand dl Ebar / sqrt(N) and dQbar += A W^T
//      accumulates in TMEM over every job of the tile, so dQ and dE are
//      written once, without atomics;
//   3. sma_bwd_rows_kernel<false>: the same for dC += (g dR) M^T;
//   4. sma_bwd_mem_kernel, one CTA per (b, j, head pair): over the tokens of
//      the later chunks, T_j += C^T (g dR) and G_j += Q^T (iq dl Ebar / sqrt N)
//      with the token operands staged MN-major, then the r_j chain rule.
// Every operand that is not an exact bf16 input is split bf16 hi + lo.
#include <math.h>

#include <cuda_bf16.h>

#include "common.cuh"
#include "kernels.h"
#include "tc_ptx.cuh"

namespace dart {
namespace {

__device__ int g_bwd_tc_status;  // first timeout code since the last read (0 = none)

constexpr int kRows = 128;
constexpr int kP = 64;
constexpr int kN = 128;
constexpr int kTile = kN * kP * 2;  // one head's 16-bit N x P tile
constexpr int kPart = 2 * kTile;    // a head pair's tiles side by side
constexpr int kJob = 2 * kPart;     // staged per job: two parts
constexpr uint64_t kDrainLimitNs = 2000000000ull;

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

// Instruction descriptor for kind::f16 with bf16 A and B, fp32 D, either
// operand K-major (0) or MN-major (1).
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

// 16 fp32 columns of this thread's lane, waited.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void fail(volatile int* abort, int code) {
    *abort = 1;
    atomicCAS(&g_bwd_tc_status, 0, code);
}

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, uint64_t limit_ns,
                                          volatile int* abort) {
    const bool got = tc::mbar_wait(bar, parity, limit_ns, abort);
    return __all_sync(0xffffffffu, got);
}

// One arrival per warp once every lane's TMEM loads / shared stores are done.
__device__ __forceinline__ void warp_arrive(uint64_t* bar) {
    tc::tc_fence_before();
    __syncwarp();
    if ((threadIdx.x & 31) == 0) tc::mbar_arrive(bar);
}

// Splits 8 floats into bf16 hi and lo words.
__device__ __forceinline__ void split_bf16x8(const float* v, uint4& hi, uint4& lo) {
    uint32_t hw[4], lw[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const __nv_bfloat162 h2 = __floats2bfloat162_rn(v[2 * e], v[2 * e + 1]);
        const float2 hf = __bfloat1622float2(h2);
        hw[e] = *reinterpret_cast<const uint32_t*>(&h2);
        lw[e] = pack_bf16(v[2 * e] - hf.x, v[2 * e + 1] - hf.y);
    }
    hi = make_uint4(hw[0], hw[1], hw[2], hw[3]);
    lo = make_uint4(lw[0], lw[1], lw[2], lw[3]);
}

// AND of v over the 256 threads of named barrier 1 (the epilogue warpgroups).
__device__ __forceinline__ bool epi_and(bool v) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.and.pred q, 1, 256, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)(v ? 1 : 0))
        : "memory");
    return r != 0;
}

// ---------------------------------------------------------------- rows kernels
// One template, two kernels, one CTA per (b, 128-token tile) looping over every
// job (head pair hp, memory j) of the tile; a job's two 32 KiB operand parts
// stream through a two-stage ring. Per job a readout chain R = A0 (part 0 +
// part 1) with a token operand A0 that is exact in bf16 (two chains) feeds the
// epilogue, which builds an A operand that accumulates against the same parts
// in TMEM over all jobs:
//   !kDQ (runs first): A0 = C, parts M_hi, M_lo: R = V_{t,j}, s = dY . V,
//         D = SiLU(z) sum_j g s, dz; dC += c M^T with c = g SiLU(z) dY;
//   kDQ:  A0 = Q, parts W_hi, W_lo: R = U_{t,j}; dl = g (SiLU(z) s G1 - D),
//         dEbar += dl lfac U in registers, dQbar += a W^T with a = dl Ebar / sqrt(N).
// The accumulations split both sides hi + lo (a_hi B_hi + a_lo B_hi + a_hi B_lo).
// The softmax-gradient sums cancel to a small fraction of their terms, so a
// single bf16 rounding of either operand costs several percent of the result;
// the split keeps the operands to ~2^-16.
constexpr int kRowsThreads = 384;
// Launched at 168 registers a thread; warpgroup 0 (producer, MMA, two idle
// warps) drops to 64 and the two epilogue warpgroups rise to 216:
// 128 x 64 + 256 x 216 = 63488 <= 384 x 168 = 64512.
constexpr int kRegsLow = 64, kRegsHigh = 216;
constexpr uint32_t kColU = 0, kColAcc = 256;  // U buffer b at kColU + 128 b (kDQ)
constexpr int kSlotB = 2 * kN + 16;           // one staged 256-byte row, padded
constexpr int kPairB = 5 * kPart;             // W_hi, W_lo, M16, M_hi, M_lo per (memory, head pair)
// Each (b, tile) is split over kRowSplit CTAs by head pairs, so the uneven
// per-tile work (nj memories) balances over more, smaller CTAs; the partial
// dQ, dC, dE (linear in the head sums) are added into zeroed outputs.
constexpr int kRowSplit = 2;

// dst[0..15] += v[0..15] (16-byte aligned), four vector reductions.
__device__ __forceinline__ void red_add16(float* dst, const float* v) {
#pragma unroll
    for (int q = 0; q < 4; ++q)
        asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(dst + 4 * q), "f"(v[4 * q]),
                     "f"(v[4 * q + 1]), "f"(v[4 * q + 2]), "f"(v[4 * q + 3])
                     : "memory");
}

struct RowsSmem {
    uint8_t q[2][kRows * 128];     // Q (raw bf16), K-major A of U: two 64-wide K blocks (kDQ)
    uint8_t stage[2][kJob];        // job operands: two parts [head 0 | head 1]
    uint8_t a[2][2][kRows * 128];  // A operand hi / lo; K block x = head x
    float lq[kRows];               // 1 / (rms(Q_t) sqrt(N))
    float xch[kRows];              // cross-warpgroup partial dot products
    uint64_t full[2];              // job operands landed (producer -> MMA)
    uint64_t uready[2];            // U of a job in buffer b done (MMA -> epilogue)
    uint64_t u_free[2];            // U buffer b read (epilogue -> MMA), 8 warps
    uint64_t stage_free[2];        // stage b's job fully consumed (MMA -> producer)
    uint64_t a_ready;              // prologue done (epilogue -> MMA, producer), 256
    uint64_t a_full;               // A operand of a job written (epilogue -> MMA), 8 warps
    uint64_t a_free;               // A operand consumed (MMA -> epilogue)
    uint64_t done;                 // every accumulation finished (MMA -> epilogue)
    uint32_t tmem_base;
    int abort;
};

template <bool kDQ>
__global__ void __launch_bounds__(kRowsThreads, 1)
sma_bwd_rows_kernel(const uint8_t* __restrict__ ops, const __nv_bfloat16* __restrict__ Q,
                    const __nv_bfloat16* __restrict__ E, const __nv_bfloat16* __restrict__ z,
                    const __nv_bfloat16* __restrict__ dY, const float* __restrict__ gbuf,
                    float* __restrict__ sdl, float2* __restrict__ gd, float2* __restrict__ rs,
                    float* __restrict__ dQC, float* __restrict__ dE, float* __restrict__ dz,
                    const __nv_bfloat16* __restrict__ Cm, int Bsz, int L, int H, int S, int Mc,
                    float eps, unsigned long long wait_limit_ns, int withhold) {
    extern __shared__ uint8_t smem_raw[];
    RowsSmem& sm = *reinterpret_cast<RowsSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~(uintptr_t)1023);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tiles = L / kRows;
    const int split = (int)blockIdx.x % kRowSplit, rest = (int)blockIdx.x / kRowSplit;
    const int tt = tiles - 1 - rest / Bsz;  // heaviest tiles first
    const int b = rest % Bsz;
    const int t0 = tt * kRows;
    const int nj = t0 / S;  // memories seen by every token of the tile
    const int hpairs = H / 2;
    const int hp_lo = split * hpairs / kRowSplit, hp_hi = (split + 1) * hpairs / kRowSplit;
    const int njobs = (hp_hi - hp_lo) * nj;  // job k = (head pair hp_lo + k / nj, memory k % nj)
    volatile int* abort = &sm.abort;

    if (threadIdx.x == 0) {
        for (int u = 0; u < 2; ++u) {
            tc::mbar_init(&sm.full[u], 1);
            tc::mbar_init(&sm.uready[u], 1);
            tc::mbar_init(&sm.u_free[u], 8);
            tc::mbar_init(&sm.stage_free[u], 1);
        }
        tc::mbar_init(&sm.a_ready, 256);
        tc::mbar_init(&sm.a_full, 8);
        tc::mbar_init(&sm.a_free, 1);
        tc::mbar_init(&sm.done, 1);
        sm.abort = 0;
        tc::fence_barrier_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(&sm.tmem_base, 512);
        tc::tmem_relinquish();
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = sm.tmem_base;

    if (warp < 4) {
        asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsLow));
        if (warp == 0 && lane == 0) {
            // ------------------------------------------------------- producer
            bool ok = true;
            int issued = 0;
            const int part0 = kDQ ? 0 : 3;  // W_hi, W_lo or M_hi, M_lo (contiguous)
            // (withhold: the failure-path test hook; every wait on the operands then runs out)
            for (int k = 0; k < (withhold ? 0 : njobs); ++k) {
                const int sb = k & 1, hp = hp_lo + k / nj, j = k % nj;
                const uint32_t par = (uint32_t)((k >> 1) & 1) ^ 1u;
                // stage 1 and the A buffers hold the prologue's row staging until a_ready
                ok = (k != 1 || tc::mbar_wait(&sm.a_ready, 0, wait_limit_ns, abort)) &&
                     tc::mbar_wait(&sm.stage_free[sb], par, wait_limit_ns, abort);
                if (!ok) {
                    fail(abort, 21);
                    break;
                }
                const uint8_t* src = ops + (((i64)b * Mc + j) * hpairs + hp) * (i64)kPairB + part0 * kPart;
                tc::mbar_arrive_expect_tx(&sm.full[sb], (uint32_t)kJob);
                tc::bulk_g2s(sm.stage[sb], src, (uint32_t)kJob, &sm.full[sb]);
                ++issued;
            }
            for (int k = issued - 1; k >= 0 && k >= issued - 2; --k)
                if (!tc::mbar_wait(&sm.full[k & 1], (uint32_t)((k >> 1) & 1), kDrainLimitNs, nullptr))
                    atomicCAS(&g_bwd_tc_status, 0, 22);
        } else if (warp == 1 && lane == 0) {
            // ------------------------------------------------------- MMA issuer
            constexpr uint32_t idU = idesc_bf16(false, true, kRows, 2 * kP);  // B MN-major (K = n)
            constexpr uint32_t idK = idesc_bf16(false, false, kRows, kN);     // B K-major (K = p)
            bool ok = njobs == 0 || tc::mbar_wait(&sm.a_ready, 0, wait_limit_ns, abort);
            if (!ok) fail(abort, 23);
            tc::tc_fence_after();
            bool any = false;
            const uint32_t q0 = tc::smem_u32(sm.q[0]);
            const uint32_t a0 = tc::smem_u32(sm.a[0][0]);  // a[h][x] at a0 + (2 h + x) 16 KiB
            for (int k = 0; ok && k <= njobs; ++k) {
                if (k < njobs) {
                    const int sb = k & 1;
                    const uint32_t par = (uint32_t)((k >> 1) & 1);
                    ok = tc::mbar_wait(&sm.u_free[sb], par ^ 1u, wait_limit_ns, abort) &&
                         tc::mbar_wait(&sm.full[sb], par, wait_limit_ns, abort);
                    if (!ok) break;
                    tc::tc_fence_after();
                    const uint32_t st = tc::smem_u32(sm.stage[sb]);
                    for (int part = 0; part < 2; ++part)
                        for (int ks = 0; ks < kN / 16; ++ks) {
                            const uint64_t ad = tc::smem_desc_sw128(q0 + 16384u * (ks / 4) + 32u * (ks % 4), 16u, 1024u);
                            const uint64_t bd = tc::smem_desc_sw128(st + (uint32_t)(part * kPart) + 2048u * ks,
                                                                    (uint32_t)kTile, 1024u);
                            mma_ss(tmem + kColU + 128u * sb, ad, bd, idU, (part > 0 || ks > 0) ? 1u : 0u);
                        }
                    tc::mma_commit(&sm.uready[sb]);
                    any = true;
                }
                if (k >= 1) {
                    const int kk = k - 1, sb = kk & 1;
                    ok = tc::mbar_wait(&sm.a_full, (uint32_t)(kk & 1), wait_limit_ns, abort);
                    if (!ok) break;
                    tc::tc_fence_after();
                    const uint32_t st = tc::smem_u32(sm.stage[sb]);
                    // a_hi B_hi + a_lo B_hi + a_hi B_lo over both heads of the pair
                    for (int term = 0; term < 3; ++term) {
                        const int ah = term == 1 ? 1 : 0, bh = term == 2 ? 1 : 0;
                        for (int x = 0; x < 2; ++x)
                            for (int ks = 0; ks < kP / 16; ++ks) {
                                const uint32_t acc = (kk > 0 || term > 0 || x > 0 || ks > 0) ? 1u : 0u;
                                const uint64_t ad = tc::smem_desc_sw128(
                                    a0 + (uint32_t)((2 * ah + x) * kRows * 128) + 32u * ks, 16u, 1024u);
                                const uint64_t bd = tc::smem_desc_sw128(
                                    st + (uint32_t)(bh * kPart + x * kTile) + 32u * ks, 16u, 1024u);
                                mma_ss(tmem + kColAcc, ad, bd, idK, acc);
                            }
                    }
                    tc::mma_commit(&sm.a_free);
                    tc::mma_commit(&sm.stage_free[sb]);
                    any = true;
                }
            }
            if (!ok) fail(abort, 24);
            // arrives once every MMA issued so far is done (also the drain after a failure)
            if (any) {
                tc::mma_commit(&sm.done);
                if (!ok && !tc::mbar_wait(&sm.done, 0, kDrainLimitNs, nullptr))
                    atomicCAS(&g_bwd_tc_status, 0, 25);
            }
        }
    } else {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegsHigh));
        // ----------------------------------------------------------- epilogue
        const int x = (warp - 4) >> 2;  // head 2 hp + x of each pair
        const int row = 32 * (warp & 3) + lane;
        const uint32_t lane_addr = (uint32_t)(32 * (warp & 3)) << 16;
        const int t = t0 + row;
        const i64 tok = (i64)b * L + t;
        const i64 tok0 = tok - lane;
        const float rsn = rsqrtf((float)kN);

        // prologue: the token operand (Q or C, warpgroup 0) and, for kDQ, E rows
        // through the slots in stage 1 .. a
        uint8_t* slots = sm.stage[1] + (warp - 4) * 32 * kSlotB;
        uint32_t ew[kDQ ? kP / 2 : 1];  // E row as bf16 pairs
        float ie = 0.0f, lfac = 0.0f;
        if (x == 0) {
            const uint8_t* src = reinterpret_cast<const uint8_t*>((kDQ ? Q : Cm) + tok0 * kN);
            {
#pragma unroll
                for (int i = 0; i < 16; ++i) {  // 2 rows per pass: 16 lanes x 16 bytes each
                    const int r = 2 * i + (lane >> 4), c = lane & 15;
                    *reinterpret_cast<uint4*>(slots + r * kSlotB + c * 16) =
                        *reinterpret_cast<const uint4*>(src + (i64)r * kN * 2 + c * 16);
                }
                __syncwarp();
                float ssq = 0.0f;
#pragma unroll
                for (int c = 0; c < 16; ++c) {
                    const uint4 v = *reinterpret_cast<const uint4*>(slots + lane * kSlotB + c * 16);
                    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) ssq = fmaf(bf_lo(w[e]), bf_lo(w[e]), fmaf(bf_hi(w[e]), bf_hi(w[e]), ssq));
                    *reinterpret_cast<uint4*>(sm.q[c / 8] + sw128((uint32_t)row, (uint32_t)(c % 8) * 16u)) = v;
                }
                sm.lq[row] = rsqrtf(ssq / (float)kN + eps) * rsn;
                __syncwarp();
            }
        }
        tc::fence_proxy_async_shared();  // the token tile visible to the MMAs
        if constexpr (kDQ) {
            const uint8_t* src = reinterpret_cast<const uint8_t*>(E + tok0 * kP);
#pragma unroll
            for (int i = 0; i < 8; ++i) {  // 4 rows per pass: 8 lanes x 16 bytes each
                const int r = 4 * i + (lane >> 3), c = lane & 7;
                *reinterpret_cast<uint4*>(slots + r * kSlotB + c * 16) =
                    *reinterpret_cast<const uint4*>(src + (i64)r * kP * 2 + c * 16);
            }
            __syncwarp();
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                const uint4 v = *reinterpret_cast<const uint4*>(slots + lane * kSlotB + c * 16);
                ew[4 * c] = v.x; ew[4 * c + 1] = v.y; ew[4 * c + 2] = v.z; ew[4 * c + 3] = v.w;
            }
            float sse = 0.0f;
#pragma unroll
            for (int i = 0; i < kP / 2; ++i) sse = fmaf(bf_lo(ew[i]), bf_lo(ew[i]), fmaf(bf_hi(ew[i]), bf_hi(ew[i]), sse));
            ie = rsqrtf(sse / (float)kP + eps);
        }
        tc::mbar_arrive(&sm.a_ready);
        asm volatile("bar.sync 1, 256;" ::: "memory");  // lq visible; slots free for the A tiles
        if constexpr (kDQ) {
            lfac = sm.lq[row];
            if (x == 0 && split == 0) rs[tok] = make_float2(lfac * sqrtf((float)kN), ie);
        }

        float de[kDQ ? kP : 1];  // dEbar partial over this warpgroup's heads
#pragma unroll
        for (int i = 0; i < (kDQ ? kP : 1); ++i) de[i] = 0.0f;
        bool ok = true;
        for (int hp = hp_lo; hp < hp_hi && ok && nj > 0; ++hp) {
            const int h = 2 * hp + x;
            const i64 rowo = tok * H + h;
            const float gate = silu_f32(__bfloat162float(z[rowo]));
            const float2 g1d = gd[rowo];  // (G1, D); !kDQ uses G1 and writes D
            float e1 = 0.0f;               // !kDQ: sum_j g s
            uint32_t dyw[kDQ ? 1 : kP / 2];
            if constexpr (!kDQ) {
                const uint4* dr = reinterpret_cast<const uint4*>(dY + rowo * kP);
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    const uint4 v = dr[c];
                    dyw[4 * c] = v.x; dyw[4 * c + 1] = v.y; dyw[4 * c + 2] = v.z; dyw[4 * c + 3] = v.w;
                }
            }
            const i64 sidx = ((i64)b * H + h) * Mc * L + t;  // + j L
            float g_next = gbuf[sidx], s_next = kDQ ? sdl[sidx] : 0.0f;  // s (!kDQ writes it)
            for (int j = 0; j < nj; ++j) {
                const int k = (hp - hp_lo) * nj + j, ub = k & 1;
                const float gw = g_next, sv = s_next;
                if (j + 1 < nj) {
                    g_next = gbuf[sidx + (i64)(j + 1) * L];
                    if (kDQ) s_next = sdl[sidx + (i64)(j + 1) * L];
                }
                float f;  // the A row's factor
                if constexpr (kDQ) {
                    const float dl = gw * (gate * sv * g1d.x - g1d.y);
                    sdl[sidx + (i64)j * L] = dl;  // for the memory kernel
                    // dEbar += dl lfac U_{t,j}, U of this head: columns 64 x .. 64 x + 63
                    if (!warp_wait(&sm.uready[ub], (uint32_t)((k >> 1) & 1), wait_limit_ns, abort)) {
                        fail(abort, 26);
                        ok = false;
                        break;
                    }
                    tc::tc_fence_after();
                    const float cu = dl * lfac;
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        float v[16];
                        tmem_ld16(tmem + lane_addr + kColU + 128u * ub + (uint32_t)(kP * x + 16 * c), v);
#pragma unroll
                        for (int i = 0; i < 16; ++i) de[16 * c + i] = fmaf(cu, v[i], de[16 * c + i]);
                    }
                    warp_arrive(&sm.u_free[ub]);
                    f = dl * rsn * ie;
                } else {
                    // V_{t,j} of this head: s = dY . V
                    if (!warp_wait(&sm.uready[ub], (uint32_t)((k >> 1) & 1), wait_limit_ns, abort)) {
                        fail(abort, 26);
                        ok = false;
                        break;
                    }
                    tc::tc_fence_after();
                    float sacc = 0.0f;
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        float v[16];
                        tmem_ld16(tmem + lane_addr + kColU + 128u * ub + (uint32_t)(kP * x + 16 * c), v);
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const uint32_t w = dyw[8 * c + i];
                            sacc = fmaf(bf_lo(w), v[2 * i], fmaf(bf_hi(w), v[2 * i + 1], sacc));
                        }
                    }
                    warp_arrive(&sm.u_free[ub]);
                    sdl[sidx + (i64)j * L] = sacc;
                    e1 = fmaf(gw, sacc, e1);
                    f = gw * gate;
                }
                // the A operand of the previous job has been consumed
                if (k > 0 && !warp_wait(&sm.a_free, (uint32_t)((k - 1) & 1), wait_limit_ns, abort)) {
                    fail(abort, 27);
                    ok = false;
                    break;
                }
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    uint32_t ah[4], al[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const uint32_t w = kDQ ? ew[(4 * c + e) % (kDQ ? kP / 2 : 1)] : dyw[(4 * c + e) % (kDQ ? 1 : kP / 2)];
                        const float v0 = f * bf_lo(w), v1 = f * bf_hi(w);
                        const __nv_bfloat162 hv = __floats2bfloat162_rn(v0, v1);
                        const float2 hf = __bfloat1622float2(hv);
                        ah[e] = *reinterpret_cast<const uint32_t*>(&hv);
                        al[e] = pack_bf16(v0 - hf.x, v1 - hf.y);
                    }
                    const uint32_t o = sw128((uint32_t)row, (uint32_t)c * 16u);
                    *reinterpret_cast<uint4*>(sm.a[0][x] + o) = make_uint4(ah[0], ah[1], ah[2], ah[3]);
                    *reinterpret_cast<uint4*>(sm.a[1][x] + o) = make_uint4(al[0], al[1], al[2], al[3]);
                }
                tc::fence_proxy_async_shared();
                warp_arrive(&sm.a_full);
            }
            if (!kDQ && ok) {
                const float zz = __bfloat162float(z[rowo]);
                gd[rowo] = make_float2(g1d.x, gate * e1);
                dz[rowo] = (e1 / g1d.x) * silu_grad_f32(zz);
            }
        }
        if (!kDQ && nj == 0) {  // no history: the gate's gradient is zero
            for (int hp = hp_lo; hp < hp_hi; ++hp) dz[tok * H + 2 * hp + x] = 0.0f;
        }
        if (ok && nj > 0 && !warp_wait(&sm.done, 0, wait_limit_ns, abort)) {
            fail(abort, 28);
            ok = false;
        }
        tc::tc_fence_after();
        ok = epi_and(ok);  // every epilogue thread takes the same branch below (named barriers)
        if (ok && nj > 0) {  // (no history: the zeroed outputs stay zero)
            const i64 grow = tok;  // G = 1: one group row per token
            if constexpr (!kDQ) {
                // dC over this warpgroup's 64 columns
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    float v[16];
                    if (nj > 0) {
                        tmem_ld16(tmem + lane_addr + kColAcc + (uint32_t)(kP * x + 16 * c), v);
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i) v[i] = 0.0f;
                    }
                    red_add16(dQC + grow * kN + kP * x + 16 * c, v);
                }
            } else {
                // dQ = iq (dQbar - Qbar (Qbar . dQbar) / N) over this warpgroup's 64 columns,
                // in two sweeps of 16 columns (the dot product first)
                const float iq = lfac * sqrtf((float)kN);
                auto qbar16 = [&](int c, float (&qb)[16]) {  // Qbar columns 64 x + 16 c ..
#pragma unroll
                    for (int u = 0; u < 2; ++u) {
                        const uint4 v = *reinterpret_cast<const uint4*>(
                            sm.q[x] + sw128((uint32_t)row, (uint32_t)(2 * c + u) * 16u));
                        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            qb[8 * u + 2 * e] = bf_lo(w[e]) * iq;
                            qb[8 * u + 2 * e + 1] = bf_hi(w[e]) * iq;
                        }
                    }
                };
                float pd = 0.0f;
                if (nj > 0) {
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        float v[16], qb[16];
                        tmem_ld16(tmem + lane_addr + kColAcc + (uint32_t)(kP * x + 16 * c), v);
                        qbar16(c, qb);
#pragma unroll
                        for (int i = 0; i < 16; ++i) pd = fmaf(qb[i], v[i], pd);
                    }
                }
                if (x == 1) sm.xch[row] = pd;
                asm volatile("bar.sync 1, 256;" ::: "memory");
                if (x == 0) sm.xch[row] += pd;
                asm volatile("bar.sync 1, 256;" ::: "memory");
                const float qdq = sm.xch[row] / (float)kN;
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    float v[16], qb[16];
                    if (nj > 0) {
                        tmem_ld16(tmem + lane_addr + kColAcc + (uint32_t)(kP * x + 16 * c), v);
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i) v[i] = 0.0f;
                    }
                    qbar16(c, qb);
#pragma unroll
                    for (int i = 0; i < 16; ++i) v[i] = iq * (v[i] - qb[i] * qdq);
                    red_add16(dQC + grow * kN + kP * x + 16 * c, v);
                }
                // dE = ie (dEbar - Ebar (Ebar . dEbar) / P), the two warpgroups' partials
                // summed through the (now idle) stage buffers
                float* part = reinterpret_cast<float*>(sm.stage[0]) + row * (kP + 4);
                if (x == 1) {
#pragma unroll
                    for (int i = 0; i < kP; i += 4)
                        *reinterpret_cast<float4*>(part + i) = make_float4(de[i], de[i + 1], de[i + 2], de[i + 3]);
                }
                asm volatile("bar.sync 1, 256;" ::: "memory");
                if (x == 0) {
#pragma unroll
                    for (int i = 0; i < kP; i += 4) {
                        const float4 o = *reinterpret_cast<const float4*>(part + i);
                        de[i] += o.x; de[i + 1] += o.y; de[i + 2] += o.z; de[i + 3] += o.w;
                    }
                    float ed = 0.0f;
#pragma unroll
                    for (int i = 0; i < kP / 2; ++i) {
                        ed = fmaf(bf_lo(ew[i]) * ie, de[2 * i], ed);
                        ed = fmaf(bf_hi(ew[i]) * ie, de[2 * i + 1], ed);
                    }
                    ed /= (float)kP;
#pragma unroll
                    for (int i = 0; i < kP / 2; ++i) {
                        de[2 * i] = ie * (de[2 * i] - bf_lo(ew[i]) * ie * ed);
                        de[2 * i + 1] = ie * (de[2 * i + 1] - bf_hi(ew[i]) * ie * ed);
                    }
#pragma unroll
                    for (int c = 0; c < 4; ++c) red_add16(dE + grow * kP + 16 * c, de + 16 * c);
                }
            }
        }
    }

    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, 512);
    }
}

// ---------------------------------------------------------- memory kernel
// One CTA per (two memories j, head pair, b), 32-token tiles of the later chunks:
// T += C^T (c_hi + c_lo), G += Q^T (a_hi + a_lo) with C and Q exact (bf16 inputs,
// MN-major A) and the scaled B rows split hi + lo:
// c = g SiLU(z) dY, a = iq dl Ebar / sqrt(N) (Qbar's scale moved onto B).
// A tile's global rows (C, Q in the MMA layout; dY, E, g, dl, z, (iq, ie) as they
// are) land by cp.async in a three-stage ring, two tiles ahead of the one being
// formed, so the loads' latency hides under a whole tile of work; the B operands
// are double-buffered. Warps 0..15 form the B operands; warp 16 issues the MMAs,
// so no forming warp waits for the issue: full[b] (one arrival per forming warp)
// hands a tile's operands to the MMA warp, mma_done[b] hands buffer b back.
constexpr int kMemFormThreads = 512;
constexpr int kMemThreads = kMemFormThreads + 32;
constexpr int kMT = 32;          // tokens per staged tile (K of one MMA chain: 2 steps)
constexpr int kBlk = kMT * 128;  // one 64-column MN block of kMT rows
constexpr int kMemPerCta = 2;    // memories per CTA, sharing the staged C and Q rows
constexpr int kMemStages = 3;    // tiles in flight in the input ring

struct MemSmem {
    uint8_t bc[kMemStages][2 * kBlk];  // C^T, Q^T of a tile (two 64-row blocks of n each)
    uint8_t bq[kMemStages][2 * kBlk];
    // per buffer and memory: c_hi, c_lo, a_hi, a_lo (one 64-column block per head each)
    uint8_t bm[2][kMemPerCta][4][2 * kBlk];
    uint8_t dy[kMemStages][kMT][2][kP * 2];  // dY rows of the two heads, bf16
    uint8_t ee[kMemStages][kMT][kP * 2];     // E rows, bf16
    float gb[kMemStages][kMemPerCta][2][kMT];  // g per (memory, head, token)
    float dl[kMemStages][kMemPerCta][2][kMT];  // dl per (memory, head, token)
    uint32_t zz[kMemStages][kMT];              // z of the two heads (a bf16 pair) per token
    float2 rq[kMemStages][kMT];                // (iq, ie) per token
    uint64_t full[2];
    uint64_t mma_done[2];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
};

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(tc::smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(tc::smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait1() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait0() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

template <typename Tmem>
__global__ void __launch_bounds__(kMemThreads, 1)
sma_bwd_mem_kernel(const Tmem* __restrict__ Mem, const float* __restrict__ rM,
                   const __nv_bfloat16* __restrict__ Q, const __nv_bfloat16* __restrict__ Cm,
                   const __nv_bfloat16* __restrict__ E, const __nv_bfloat16* __restrict__ z,
                   const __nv_bfloat16* __restrict__ dY, const float* __restrict__ gbuf,
                   const float* __restrict__ dlbuf, const float2* __restrict__ rs,
                   float* __restrict__ dM, int L, int H, int S, int Mc,
                   unsigned long long wait_limit_ns) {
    extern __shared__ uint8_t smem_raw[];
    MemSmem& sm = *reinterpret_cast<MemSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                              ~(uintptr_t)1023);
    // memory pairs in z, the slowest launch index: the heaviest (earliest) memories,
    // whose later chunks hold the most tokens, start first
    const int j0 = blockIdx.z * kMemPerCta, hp = blockIdx.x, b = blockIdx.y;
    const int tid = threadIdx.x, warp = tid >> 5;
    const int nm = min(kMemPerCta, Mc - j0);  // memories of this CTA
    const int first = (j0 + 1) * S;           // tokens of the chunks after memory j0
    const int ntiles = (L - first) / kMT;
    const float rsn = rsqrtf((float)kN);

    if (tid == 0) {
        tc::mbar_init(&sm.full[0], kMemFormThreads / 32);
        tc::mbar_init(&sm.full[1], kMemFormThreads / 32);
        tc::mbar_init(&sm.mma_done[0], 1);
        tc::mbar_init(&sm.mma_done[1], 1);
        tc::mbar_init(&sm.drain, 1);
        sm.abort = 0;
        tc::fence_barrier_init();
    }
    if (warp == 0) {
        tc::tmem_alloc(&sm.tmem_base, 512);
        tc::tmem_relinquish();
    }
    const bool former = tid < kMemFormThreads;
    const int cr = tid >> 4, cq = tid & 15;                      // C / Q row, piece
    const int ex = tid >> 8, er = (tid >> 3) & 31, eq = tid & 7;  // head, dY / E row, piece
    const int eh = 2 * hp + ex;
    // the copies of tile `it` into ring stage it % kMemStages (one commit group per
    // tile and thread, empty past the last tile)
    auto issue = [&](int it) {
        if (it < ntiles) {
            const int st = it % kMemStages;
            const i64 tok0 = (i64)b * L + first + it * kMT;
            const uint32_t o = (uint32_t)(cq >> 3) * kBlk + sw128((uint32_t)cr, (uint32_t)(cq & 7) * 16u);
            cp_async16(sm.bc[st] + o, Cm + (tok0 + cr) * kN + 8 * cq);
            cp_async16(sm.bq[st] + o, Q + (tok0 + cr) * kN + 8 * cq);
            cp_async16(&sm.dy[st][er][ex][16 * eq], dY + ((tok0 + er) * H + eh) * kP + 8 * eq);
            if (tid < 256) {
                cp_async16(&sm.ee[st][tid >> 3][16 * (tid & 7)], E + (tok0 + (tid >> 3)) * kP + 8 * (tid & 7));
            } else if (tid < 320) {  // g (256 .. 287) and dl (288 .. 319): 4 tokens a thread
                const int i = tid - 256, which = i >> 5, m = (i >> 4) & 1, x = (i >> 3) & 1, pc = i & 7;
                if (m < nm) {  // the other memory's rows lie past this CTA's last one
                    const i64 sidx = (((i64)b * H + 2 * hp + x) * Mc + j0 + m) * L + first + it * kMT + 4 * pc;
                    cp_async16(which ? &sm.dl[st][m][x][4 * pc] : &sm.gb[st][m][x][4 * pc],
                               (which ? dlbuf : gbuf) + sidx);
                }
            } else if (tid < 352) {  // z of both heads for token tid - 320
                const int r = tid - 320;
                cp_async4(&sm.zz[st][r], z + (tok0 + r) * H + 2 * hp);
            } else if (tid < 368) {  // (iq, ie) of two tokens
                const int r = 2 * (tid - 352);
                cp_async16(&sm.rq[st][r], rs + tok0 + r);
            }
        }
        cp_async_commit();
    };
    if (former) {
        issue(0);
        issue(1);
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = sm.tmem_base;
    volatile int* abort = &sm.abort;

    bool ok = true;
    if (former) {
        for (int it = 0; it < ntiles; ++it) {
            const int bi = it & 1, st = it % kMemStages;
            cp_async_wait1();  // this thread's copies of tile it (tile it + 1's may be in flight)
            // everyone's copies, and one decision for all forming threads: stop if any of
            // them has seen a wait give up (a forming warp's or the MMA thread's)
            const uint32_t seen = *abort != 0 ? 1u : 0u;
            uint32_t stop;
            asm volatile(
                "{\n\t.reg .pred p, q;\n\t"
                "setp.ne.u32 q, %1, 0;\n\t"
                "bar.red.or.pred p, 1, %2, q;\n\t"
                "selp.u32 %0, 1, 0, p;\n\t}"
                : "=r"(stop)
                : "r"(seen), "n"(kMemFormThreads)
                : "memory");
            if (stop) break;
            // c and a rows split hi / lo: memory m, token r, head x, columns p -> block x,
            // row r. Buffer bi was read by the MMAs of tile it - 2, waited at the end of
            // tile it - 1.
            {
                const int t = first + it * kMT + er;  // position in the sequence
                const uint32_t zw = sm.zz[st][er];
                const float gate = silu_f32(ex ? bf_hi(zw) : bf_lo(zw));
                const float2 q = sm.rq[st][er];
                const uint4 dv = *reinterpret_cast<const uint4*>(&sm.dy[st][er][ex][16 * eq]);
                const uint4 ev = *reinterpret_cast<const uint4*>(&sm.ee[st][er][16 * eq]);
                const uint32_t dw[4] = {dv.x, dv.y, dv.z, dv.w};
                const uint32_t ew[4] = {ev.x, ev.y, ev.z, ev.w};
                const uint32_t o = (uint32_t)ex * kBlk + sw128((uint32_t)er, (uint32_t)eq * 16u);
#pragma unroll
                for (int m = 0; m < kMemPerCta; ++m) {
                    // memory j sees tokens of later chunks only (its factors are zero before)
                    const bool live = m < nm && t >= (j0 + m + 1) * S;
                    const float fg = live ? sm.gb[st][m][ex][er] * gate : 0.0f;
                    const float fd = live ? sm.dl[st][m][ex][er] * q.x * q.y * rsn : 0.0f;
                    float gv[8], av[8];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        gv[2 * e] = bf_lo(dw[e]) * fg;
                        gv[2 * e + 1] = bf_hi(dw[e]) * fg;
                        av[2 * e] = bf_lo(ew[e]) * fd;
                        av[2 * e + 1] = bf_hi(ew[e]) * fd;
                    }
                    uint4 hi, lo;
                    split_bf16x8(gv, hi, lo);
                    *reinterpret_cast<uint4*>(sm.bm[bi][m][0] + o) = hi;
                    *reinterpret_cast<uint4*>(sm.bm[bi][m][1] + o) = lo;
                    split_bf16x8(av, hi, lo);
                    *reinterpret_cast<uint4*>(sm.bm[bi][m][2] + o) = hi;
                    *reinterpret_cast<uint4*>(sm.bm[bi][m][3] + o) = lo;
                }
            }
            // the copied C and Q rows and the stored B rows, to the MMA warp
            tc::fence_proxy_async_shared();
            __syncwarp();
            if ((tid & 31) == 0) tc::mbar_arrive(&sm.full[bi]);
            // tile it + 2 goes to the stage of tile it - 1, whose MMAs read its C and Q
            // rows (and leave buffer bi ^ 1 free for tile it + 1)
            if (it >= 1 && !warp_wait(&sm.mma_done[bi ^ 1], (uint32_t)(((it - 1) >> 1) & 1), wait_limit_ns, abort)) {
                fail(abort, 31);
                ok = false;
            }
            if (ok) issue(it + 2);
            else cp_async_commit();  // keeps this thread's group count; the barrier then breaks
        }
        cp_async_wait0();  // also when a wait gave up: no copy outlives the CTA
        // the last tile's MMAs (and with them every earlier one) are done
        if (ok && !*abort && ntiles > 0) {
            const int last = ntiles - 1;
            if (!warp_wait(&sm.mma_done[last & 1], (uint32_t)((last >> 1) & 1), wait_limit_ns, abort)) {
                fail(abort, 32);
            }
        }
    } else if (tid == kMemFormThreads) {
        // the MMA thread: tile it's operands on full[it & 1], its MMAs into mma_done[it & 1]
        constexpr uint32_t idM = idesc_bf16(true, true, kN, 2 * kP);  // A and B MN-major
        int issued = 0;
        for (int it = 0; it < ntiles; ++it) {
            const int bi = it & 1, st = it % kMemStages;
            if (!tc::mbar_wait(&sm.full[bi], (uint32_t)((it >> 1) & 1), wait_limit_ns, abort)) {
                fail(abort, 34);
                break;
            }
            tc::tc_fence_after();
            const int tb = first + it * kMT;
            for (int m = 0; m < nm; ++m) {
                const int jfirst = (j0 + m + 1) * S;  // memory m's first token
                if (tb < jfirst) continue;             // nothing of memory m in this tile
                const bool fresh = tb == jfirst;       // its first tile starts the sums
                const uint32_t d = tmem + 256u * (uint32_t)m;
                for (int part = 0; part < 2; ++part)
                    for (int ks = 0; ks < kMT / 16; ++ks) {
                        const uint32_t acc = (!fresh || part > 0 || ks > 0) ? 1u : 0u;
                        const uint64_t ac = tc::smem_desc_sw128(tc::smem_u32(sm.bc[st]) + 2048u * ks, (uint32_t)kBlk, 1024u);
                        const uint64_t bgd = tc::smem_desc_sw128(tc::smem_u32(sm.bm[bi][m][part]) + 2048u * ks,
                                                                 (uint32_t)kBlk, 1024u);
                        mma_ss(d, ac, bgd, idM, acc);
                        const uint64_t aq = tc::smem_desc_sw128(tc::smem_u32(sm.bq[st]) + 2048u * ks, (uint32_t)kBlk, 1024u);
                        const uint64_t bdd = tc::smem_desc_sw128(tc::smem_u32(sm.bm[bi][m][2 + part]) + 2048u * ks,
                                                                 (uint32_t)kBlk, 1024u);
                        mma_ss(d + 128u, aq, bdd, idM, acc);
                    }
            }
            tc::mma_commit(&sm.mma_done[bi]);
            issued = it + 1;
        }
        if (*abort && issued > 0) {  // let the MMAs in flight finish before TMEM is freed
            tc::mma_commit(&sm.drain);
            if (!tc::mbar_wait(&sm.drain, 0, kDrainLimitNs, nullptr)) atomicCAS(&g_bwd_tc_status, 0, 33);
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    ok = !*abort;
    tc::tc_fence_after();
    const int m = tid >> 8;
    if (ok && m < nm) {
        // thread (n, x, m): row n of T and G for head 2 hp + x of memory j0 + m
        const int n = tid & 127, x = (tid >> 7) & 1;
        const int j = j0 + m, h = 2 * hp + x;
        const bool any = (j + 1) * S < L;  // the memory has later tokens
        const uint32_t lane_addr = (uint32_t)(32 * (warp & 3)) << 16;
        const uint32_t col = 256u * (uint32_t)m + (uint32_t)(kP * x);
        const i64 mbase = ((i64)b * Mc + j) * H + h;
        const Tmem* Mj = Mem + (mbase * kN + n) * kP;
        float* dMj = dM + (mbase * kN + n) * kP;
        const float rn = rM[mbase * kN + n];
        auto sweep = [&](int c, float (&tv)[16], float (&gv)[16], float (&mv)[16]) {
#pragma unroll
            for (int i = 0; i < 16; ++i) mv[i] = ld_f32(Mj + 16 * c + i);
            if (any) {
                tmem_ld16(tmem + lane_addr + col + (uint32_t)(16 * c), tv);
                tmem_ld16(tmem + lane_addr + col + 128u + (uint32_t)(16 * c), gv);
            } else {
#pragma unroll
                for (int i = 0; i < 16; ++i) { tv[i] = 0.0f; gv[i] = 0.0f; }
            }
        };
        float dr = 0.0f;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            float tv[16], gv[16], mv[16];
            sweep(c, tv, gv, mv);
#pragma unroll
            for (int i = 0; i < 16; ++i) dr = fmaf(mv[i], gv[i], dr);
        }
        const float c3 = dr * rn * rn * rn / (float)kP;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            float tv[16], gv[16], mv[16];
            sweep(c, tv, gv, mv);
#pragma unroll
            for (int i = 0; i < 16; ++i) tv[i] = tv[i] + rn * gv[i] - c3 * mv[i];
            store_row16(dMj + 16 * c, tv);
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

}  // namespace

bool sma_bwd_tc_supported(const SmaBwdArgs& a) {
    return a.P == kP && a.N == kN && a.G == 1 && a.S % kRows == 0 && a.L % kRows == 0 &&
           a.H % 2 == 0;
}

// Workspace: operand tiles (five parts per memory and head pair), their
// scales, g and s / dl per (b, h, j, t), (G1, D) per (t, h), (iq, ie) per t,
// and r when the caller passes none.
size_t sma_bwd_tc_workspace(int64_t B, int64_t L, int64_t H, int64_t Mc, int64_t N) {
    auto al = [](size_t v) { return (v + 255) & ~(size_t)255; };
    return al((size_t)(B * Mc * (H / 2)) * kPairB) + al((size_t)(B * Mc * H) * 4) +
           2 * al((size_t)(B * H * Mc * L) * 4) + al((size_t)(B * L * H) * 8) +
           al((size_t)(B * L) * 8) + al((size_t)(B * Mc * H * N) * 4);
}

template <typename Tmem>
cudaError_t launch_sma_backward_tc(const SmaBwdArgs& a, void* ws, unsigned long long wait_limit_ns,
                                   cudaStream_t stream) {
    const int Bsz = (int)a.B, L = (int)a.L, H = (int)a.H, S = (int)a.S, Mc = L / S;
    auto al = [](size_t v) { return (v + 255) & ~(size_t)255; };
    uint8_t* p = (uint8_t*)ws;
    uint8_t* ops = p;                        p += al((size_t)(a.B * Mc * (a.H / 2)) * kPairB);
    float* scale = (float*)p;                p += al((size_t)(a.B * Mc * a.H) * 4);
    float* gbuf = (float*)p;                 p += al((size_t)(a.B * a.H * Mc * a.L) * 4);
    float* sdl = (float*)p;                  p += al((size_t)(a.B * a.H * Mc * a.L) * 4);
    float2* gd = (float2*)p;                 p += al((size_t)(a.B * a.L * a.H) * 8);
    float2* rs = (float2*)p;                 p += al((size_t)(a.B * a.L) * 8);
    float* rM = a.rM != nullptr ? (float*)a.rM : (float*)p;
    cudaError_t e;
    if (a.rM == nullptr) {
        e = launch_memory_rms<Tmem>(a.M, rM, a.B * Mc * a.H * a.N, a.P, a.eps, stream);
        if (e != cudaSuccess) return e;
    }
    e = a.logits != nullptr
            ? launch_sma_bwd_stats_from_logits<Tmem>(a, rM, ops, kPairB, scale, gbuf, gd, stream)
            : launch_sma_bwd_stats_tc<Tmem>(a, rM, ops, kPairB, scale, gbuf, gd, wait_limit_ns, stream);
    if (e != cudaSuccess) return e;
    // the row kernels add their head-pair halves into these
    const size_t rows = (size_t)(a.B * a.L);
    if ((e = cudaMemsetAsync(a.dQ, 0, rows * kN * sizeof(float), stream)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(a.dC, 0, rows * kN * sizeof(float), stream)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(a.dE, 0, rows * kP * sizeof(float), stream)) != cudaSuccess) return e;
    const size_t smem_rows = sizeof(RowsSmem) + 1024;
    for (int pass = 0; pass < 2; ++pass) {  // dC, s, D, dz first; then dQ, dE, dl
        auto k = pass == 0 ? sma_bwd_rows_kernel<false> : sma_bwd_rows_kernel<true>;
        if ((e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_rows)) != cudaSuccess)
            return e;
        k<<<Bsz * (L / kRows) * kRowSplit, kRowsThreads, smem_rows, stream>>>(
            ops, (const __nv_bfloat16*)a.Q, (const __nv_bfloat16*)a.E, (const __nv_bfloat16*)a.z,
            (const __nv_bfloat16*)a.dY, gbuf, sdl, gd, rs, pass == 0 ? a.dC : a.dQ, a.dE, a.dz,
            (const __nv_bfloat16*)a.Cm, Bsz, L, H, S, Mc, a.eps, wait_limit_ns, a.test_withhold);
        note_launches(1);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    {
        const size_t smem = sizeof(MemSmem) + 1024;
        auto k = sma_bwd_mem_kernel<Tmem>;
        if ((e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) != cudaSuccess)
            return e;
        k<<<dim3(H / 2, Bsz, (Mc + kMemPerCta - 1) / kMemPerCta), kMemThreads, smem, stream>>>(
            (const Tmem*)a.M, rM, (const __nv_bfloat16*)a.Q, (const __nv_bfloat16*)a.Cm,
            (const __nv_bfloat16*)a.E, (const __nv_bfloat16*)a.z, (const __nv_bfloat16*)a.dY, gbuf, sdl,
            rs, a.dM, L, H, S, Mc, wait_limit_ns);
        note_launches(1);
    }
    return cudaGetLastError();
}

template cudaError_t launch_sma_backward_tc<float>(const SmaBwdArgs&, void*, unsigned long long, cudaStream_t);
template cudaError_t launch_sma_backward_tc<__nv_bfloat16>(const SmaBwdArgs&, void*, unsigned long long,
                                                           cudaStream_t);

// Read and clear of the status word in one device-side exchange: a code that a
// kernel still running on another stream records is either returned now or kept
// for the next read, never lost between a read and a separate clear.
__device__ int g_bwd_tc_status_taken;
__global__ void take_bwd_tc_status_kernel() { g_bwd_tc_status_taken = atomicExch(&g_bwd_tc_status, 0); }

int take_bwd_tc_status(cudaStream_t stream) {
    take_bwd_tc_status_kernel<<<1, 1, 0, stream>>>();
    int v = 0;
    if (cudaGetLastError() != cudaSuccess ||
        cudaMemcpyFromSymbolAsync(&v, g_bwd_tc_status_taken, sizeof(int), 0, cudaMemcpyDeviceToHost, stream) !=
            cudaSuccess ||
        cudaStreamSynchronize(stream) != cudaSuccess)
        return -1;
    return v;
}

}  // namespace dart
