// State-memory attention forward + gated merge on the 5th-generation tensor
// cores (tcgen05, TMEM, bulk async copies), for bf16 token inputs with
// P = 64, N = 128 and S a multiple of 128 (Sec. 3 value/key readouts, chunk
// logit, softmax over earlier chunks and R_t; App. B.1 normalised score
// branch; Alg. 1 streaming order; Sec. 3 gated merge).
//
// For a tile of 128 tokens (one TMEM lane each) and memory M_j of head h the
// kernel needs, per token t,
//   U_t = Q_t (r_j (.) M_j),   V_t = C_t M_j     (N = 128 -> P = 64 each)
//   l_{t,j} = (U_t . Ebar_t) / (rms(Q_t) sqrt(N))
// U and V are GEMMs whose token operands Q, C stay fixed for the whole tile
// (they sit in TMEM as the A operand) while the memories stream through as
// the B operand.
//
// Precision. Rounding the memory operand to bf16 moves the logits enough to
// break the 2e-2 parity bar, so W = r (.) M is split into bf16 hi + lo parts
// (two MMA chains into one accumulator, ~2^-16 relative) and the value path
// runs in fp16 on M / max|M_j| (scale re-applied in the epilogue). Q and C are
// exact (bf16 inputs; C widened to fp16 exactly); Qbar's RMS scale and Ebar
// stay fp32 in the epilogue.
//
// Shape. A tcgen05.mma with M = 128, K = 16 costs about the same for any
// N <= 128 and only reaches the tensor peak at N >= 192 (measured on GB300:
// ~90-99 cycles at N <= 128, ~137 at N = 256 with A in TMEM). So one job is
// one memory j for the CTA's two heads: U is one N = 256 chain over the tiles
// [W_hi h0 | W_lo h0 | W_hi h1 | W_lo h1] (the epilogue adds hi + lo), V is
// one N = 128 chain over [M16 h0 | M16 h1]. U and V have one TMEM buffer each
// and alternate, so each buffer is read by the epilogue while the other one
// is being computed.
//
// Kernel 1 (sma_operands_kernel) writes per (memory, pair of heads) a 64 KiB
// U part and a 32 KiB V part, already in the 128-byte-swizzled shared-memory
// layout, so each part is one bulk copy.
// Kernel 2 (sma_tc_kernel), one CTA per (batch, 128-token tile, 2 heads),
// heaviest tiles first:
//   warp 0      producer: bulk copies of the parts into a 3-stage ring
//   warp 1      TMEM allocation; one thread issues the MMAs
//   warps 2, 3  idle (they complete warpgroup 0 for the register split)
//   warps 4..7  epilogue warpgroup 0: head 0 of the pair
//   warps 8..11 epilogue warpgroup 1: head 1 of the pair
// An epilogue thread owns one token row of its head: it reads U and V from
// TMEM with wide loads (three waits per job), runs the online softmax, and
// finally writes R = O / d, lse and Y = Y_ssd + SiLU(z) R. Warpgroup 0 also
// stages Q and C into TMEM, warpgroup 1 writes Ebar to shared memory.
// TMEM: [0,64) Q (bf16 pairs), [64,128) C (fp16 pairs), [128,384) U,
// [384,512) V.
#include <math.h>

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "common.cuh"
#include "kernels.h"
#include "tc_ptx.cuh"

namespace dart {
namespace {

__device__ int g_tc_status;  // first timeout code since the last read (0 = none)

constexpr int kRows = 128;   // tokens per tile (TMEM lanes)
constexpr int kP = 64;
constexpr int kN = 128;
constexpr int kHeadsPerCta = 2;
constexpr int kTile = kN * kP * 2;            // bytes of one 16-bit N x P operand tile
constexpr int kPartU = 4 * kTile;             // W_hi h0 | W_lo h0 | W_hi h1 | W_lo h1
constexpr int kPartV = 2 * kTile;             // M16 h0 | M16 h1
constexpr int kPair = kPartU + kPartV;        // operand bytes per (memory, head pair)
constexpr int kStages = 3;                    // ring of kPartU-sized stages
constexpr int kThreads = 384;
// Register split: launched at 168 per thread (384 x 168 = 64512 of the 65536
// of an SM); warpgroup 0 (producer, MMA, two idle warps) drops to 56 and the
// epilogue warpgroups rise to 224: 128 x 56 + 256 x 224 = 64512, within the
// launch pool, and per sub-partition (56 + 2 x 224) x 32 = 16128 <= 16384.
constexpr int kRegsLow = 56, kRegsHigh = 224;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColQ = 0, kColC = 64, kColU = 128, kColV = 384;
// Bound on the final waits for this CTA's own copies and MMAs (never cut short).
constexpr uint64_t kDrainLimitNs = 2000000000ull;

constexpr uint32_t kIdescU = tc::idesc_f16(1, true, kRows, 4 * kP);  // bf16, N = 256
constexpr uint32_t kIdescV = tc::idesc_f16(0, true, kRows, 2 * kP);  // fp16, N = 128

// Byte offset of element (n, p) of a 128-row x 128-byte tile in the
// 128-byte-swizzled layout: the 16-byte chunk index is XORed with n mod 8.
__device__ __forceinline__ uint32_t sw128(int n, int p) {
    const uint32_t o = (uint32_t)n * 128u + (uint32_t)p * 2u;
    return o ^ (((uint32_t)n & 7u) << 4);
}

// ------------------------------------------------------------ kernel 1
// One block of 256 threads per (j, h, b) memory. Warp w owns rows n = w + 8k;
// lane owns columns p = lane, lane + 32. Head h = 2 hp + x writes
//   W_hi to  ops + ((b Mc + j) (H/2) + hp) kPair + 2x kTile,
//   W_lo one tile further, M16 to  ... + kPartU + x kTile.
template <typename Tmem>
__global__ void __launch_bounds__(256)
sma_operands_kernel(const Tmem* __restrict__ M, const float* __restrict__ rM,
                    uint8_t* __restrict__ ops, float* __restrict__ scale, int Mc, int H,
                    float eps) {
    const int j = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const i64 mem = ((i64)b * Mc + j) * H + h;
    const Tmem* src = M + mem * (kN * kP);
    const i64 pair = ((i64)b * Mc + j) * (H / kHeadsPerCta) + h / kHeadsPerCta;
    const int x = h % kHeadsPerCta;
    uint8_t* dst_u = ops + pair * kPair + 2 * x * kTile;
    uint8_t* dst_v = ops + pair * kPair + kPartU + x * kTile;
    __shared__ float s_max[8];

    float v0[16], v1[16], rr[16];
    float amax = 0.0f;
#pragma unroll
    for (int k = 0; k < 16; ++k) {
        const int n = warp + 8 * k;
        v0[k] = ld_f32(src + n * kP + lane);
        v1[k] = ld_f32(src + n * kP + lane + 32);
        amax = fmaxf(amax, fmaxf(fabsf(v0[k]), fabsf(v1[k])));
        float ss = v0[k] * v0[k] + v1[k] * v1[k];
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
        rr[k] = rM != nullptr ? rM[mem * kN + n] : rsqrtf(ss / (float)kP + eps);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
    if (lane == 0) s_max[warp] = amax;
    __syncthreads();
    float s = 0.0f;
#pragma unroll
    for (int w = 0; w < 8; ++w) s = fmaxf(s, s_max[w]);
    const float inv_s = s > 0.0f ? 1.0f / s : 1.0f;
    if (threadIdx.x == 0) scale[mem] = s > 0.0f ? s : 1.0f;
#pragma unroll
    for (int k = 0; k < 16; ++k) {
        const int n = warp + 8 * k;
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const int p = lane + 32 * half;
            const float v = half ? v1[k] : v0[k];
            const float wv = rr[k] * v;
            const __nv_bfloat16 hi = __float2bfloat16_rn(wv);
            const __nv_bfloat16 lo = __float2bfloat16_rn(wv - __bfloat162float(hi));
            const __half m16 = __float2half_rn(v * inv_s);
            const uint32_t o = sw128(n, p);
            *reinterpret_cast<__nv_bfloat16*>(dst_u + o) = hi;
            *reinterpret_cast<__nv_bfloat16*>(dst_u + kTile + o) = lo;
            *reinterpret_cast<__half*>(dst_v + o) = m16;
        }
    }
}

// ------------------------------------------------------------ kernel 2
struct TcSmem {
    uint8_t stage[kStages][kPartU];  // 1024-aligned by placement
    float4 ebar[kRows][kP / 4];      // Ebar rows, 16-byte chunks swizzled by row
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t u_full, u_free, v_full, v_free;
    uint64_t a_ready, drain;
    uint32_t tmem_base;
    int abort;
};

__device__ __forceinline__ void fail(volatile int* abort, int code) {
    *abort = 1;
    atomicCAS(&g_tc_status, 0, code);
}

// tcgen05.ld of 16 consecutive fp32 columns of this thread's lane, waited.
__device__ __forceinline__ void tmem_ld16w(uint32_t taddr, float (&v)[16]) {
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

// Warp-uniform bounded wait (every lane waits; all lanes see the same outcome).
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, uint64_t limit_ns,
                                          volatile int* abort) {
    const bool got = tc::mbar_wait(bar, parity, limit_ns, abort);
    return __all_sync(0xffffffffu, got);
}

// tcgen05.ld of 32 + 32 fp32 columns (two addresses) of this thread's lane, one wait.
__device__ __forceinline__ void tmem_ld32x2(uint32_t ta, uint32_t tb, float (&v)[64]) {
    uint32_t r[64];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%64];\n\t"
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,"
        "%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [%65];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
          "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
          "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
          "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]),
          "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]),
          "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]), "=r"(r[49]),
          "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
          "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]),
          "=r"(r[62]), "=r"(r[63])
        : "r"(ta), "r"(tb)
        : "memory");
#pragma unroll
    for (int i = 0; i < 64; ++i) v[i] = __uint_as_float(r[i]);
}

// Dot product of 16 columns of U with Ebar[p0 .. p0+15] of row `row`.
__device__ __forceinline__ float dot16(const float (&u)[16], const TcSmem& sm, int row, int p0) {
    float acc = 0.0f;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int chunk = (p0 / 4 + q) ^ (row & 15);
        const float4 e = sm.ebar[row][chunk];
        acc = fmaf(u[4 * q], e.x, acc);
        acc = fmaf(u[4 * q + 1], e.y, acc);
        acc = fmaf(u[4 * q + 2], e.z, acc);
        acc = fmaf(u[4 * q + 3], e.w, acc);
    }
    return acc;
}

template <typename Tout>
__global__ void __launch_bounds__(kThreads, 1)
sma_tc_kernel(const uint8_t* __restrict__ ops, const float* __restrict__ scale,
              const __nv_bfloat16* __restrict__ Q, const __nv_bfloat16* __restrict__ Cm,
              const __nv_bfloat16* __restrict__ E, const __nv_bfloat16* __restrict__ z,
              const Tout* __restrict__ Yssd, Tout* __restrict__ Y, Tout* __restrict__ R,
              float* __restrict__ lse, int Bsz, int L, int H, int G, int S, int Mc, float eps,
              unsigned long long wait_limit_ns) {
    extern __shared__ uint8_t smem_raw[];
    TcSmem& sm = *reinterpret_cast<TcSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                            ~(uintptr_t)1023);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // work item: heaviest token tiles first
    const int tiles = L / kRows;
    const int hpairs = H / kHeadsPerCta;
    const int item = blockIdx.x;
    const int tt = tiles - 1 - item / (Bsz * hpairs);
    const int rem = item % (Bsz * hpairs);
    const int b = rem / hpairs;
    const int hp = rem % hpairs;
    const int h0 = hp * kHeadsPerCta;
    const int t0 = tt * kRows;
    const int nj = (t0 + kRows - 1) / S;  // memories the last token of the tile sees
    volatile int* abort = &sm.abort;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(&sm.full[s], 1);
            tc::mbar_init(&sm.empty[s], 1);
        }
        tc::mbar_init(&sm.u_full, 1);
        tc::mbar_init(&sm.u_free, 256);
        tc::mbar_init(&sm.v_full, 1);
        tc::mbar_init(&sm.v_free, 256);
        tc::mbar_init(&sm.a_ready, 256);  // Q from warpgroup 0, C from warpgroup 1
        tc::mbar_init(&sm.drain, 1);
        sm.abort = 0;
        tc::fence_barrier_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(&sm.tmem_base, kTmemCols);
        tc::tmem_relinquish();
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = sm.tmem_base;

    if (warp < 4) {
      asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsLow));
      if (warp == 0) {
        // ------------------------------------------------------- producer
        // parts in order U(0), V(0), U(1), V(1), ...; part k uses stage k % 3
        if (lane == 0) {
            const int nparts = 2 * nj;
            int k = 0;
            for (; k < nparts; ++k) {
                const int st = k % kStages;
                const uint32_t round = (uint32_t)(k / kStages);
                if (!tc::mbar_wait(&sm.empty[st], (round & 1u) ^ 1u, wait_limit_ns, abort)) {
                    fail(abort, 1);
                    break;
                }
                const int j = k >> 1;
                const bool is_v = (k & 1) != 0;
                const uint8_t* src = ops + (((i64)b * Mc + j) * hpairs + hp) * (i64)kPair +
                                     (is_v ? kPartU : 0);
                const uint32_t bytes = is_v ? (uint32_t)kPartV : (uint32_t)kPartU;
                tc::mbar_arrive_expect_tx(&sm.full[st], bytes);
                tc::bulk_g2s(sm.stage[st], src, bytes, &sm.full[st]);
            }
            // never leave a copy in flight behind: wait for the last one of each stage
            for (int kk = k - 1; kk >= 0 && kk >= k - kStages; --kk) {
                if (!tc::mbar_wait(&sm.full[kk % kStages], (uint32_t)((kk / kStages) & 1),
                                   kDrainLimitNs, nullptr))
                    atomicCAS(&g_tc_status, 0, 5);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------- MMA issuer
        if (lane == 0) {
            bool ok = tc::mbar_wait(&sm.a_ready, 0, wait_limit_ns, abort);
            if (!ok) fail(abort, 2);
            tc::tc_fence_after();
            bool issued = false;
            for (int k = 0; ok && k < 2 * nj; ++k) {
                const int j = k >> 1;
                const bool is_v = (k & 1) != 0;
                const int st = k % kStages;
                const uint32_t ph = (uint32_t)(j & 1);
                // the buffer is free once the epilogue has read the previous job's contents
                if (!tc::mbar_wait(is_v ? &sm.v_free : &sm.u_free, ph ^ 1u, wait_limit_ns, abort) ||
                    !tc::mbar_wait(&sm.full[st], (uint32_t)((k / kStages) & 1), wait_limit_ns, abort)) {
                    fail(abort, 3);
                    ok = false;
                    break;
                }
                tc::tc_fence_after();
                const uint32_t sb = tc::smem_u32(sm.stage[st]);
#pragma unroll
                for (int ks = 0; ks < kN / 16; ++ks) {
                    const uint64_t bd = tc::smem_desc_sw128(sb + 2048u * ks, (uint32_t)kTile, 1024u);
                    if (is_v)
                        tc::mma_f16_ts(tmem + kColV, tmem + kColC + 8u * ks, bd, kIdescV, ks > 0 ? 1u : 0u);
                    else
                        tc::mma_f16_ts(tmem + kColU, tmem + kColQ + 8u * ks, bd, kIdescU, ks > 0 ? 1u : 0u);
                }
                issued = true;
                tc::mma_commit(&sm.empty[st]);
                tc::mma_commit(is_v ? &sm.v_full : &sm.u_full);
            }
            if (!ok && issued) {
                // drain: this commit arrives once every MMA issued so far is done
                tc::mma_commit(&sm.drain);
                if (!tc::mbar_wait(&sm.drain, 0, kDrainLimitNs, nullptr))
                    atomicCAS(&g_tc_status, 0, 6);
            }
        }
      }
    } else {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegsHigh));
        // ------------------------------------------------------- epilogue
        const int wg = (warp - 4) >> 2;  // head h0 + wg
        const int h = h0 + wg;
        const int row = 32 * (warp & 3) + lane;
        const uint32_t lane_addr = (uint32_t)(32 * (warp & 3)) << 16;
        const int t = t0 + row;
        const i64 tok = (i64)b * L + t;
        const int g = h0 / (H / G);
        const int nh = t / S;
        float ssq = 0.0f;
        if (wg == 0) {
            // A operand Q (bf16 pairs) into TMEM
            const uint4* qrow = reinterpret_cast<const uint4*>(Q + (tok * G + g) * kN);
            uint4 qv[16];
#pragma unroll
            for (int u = 0; u < 16; ++u) qv[u] = qrow[u];
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                uint32_t qa[16];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const uint32_t qw[4] = {qv[c * 4 + u].x, qv[c * 4 + u].y, qv[c * 4 + u].z, qv[c * 4 + u].w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        qa[u * 4 + e] = qw[e];
                        const float2 qf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&qw[e]));
                        ssq = fmaf(qf.x, qf.x, fmaf(qf.y, qf.y, ssq));
                    }
                }
                tc::tmem_st16(tmem + lane_addr + kColQ + 16u * c, qa);
            }
        } else {
            // A operand C (fp16 pairs) into TMEM, and the Q row's sum of squares
            const uint4* crow = reinterpret_cast<const uint4*>(Cm + (tok * G + g) * kN);
            const uint4* qrow = reinterpret_cast<const uint4*>(Q + (tok * G + g) * kN);
            uint4 cv[16];
#pragma unroll
            for (int u = 0; u < 16; ++u) cv[u] = crow[u];
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                uint32_t ca[16];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const uint32_t cw[4] = {cv[c * 4 + u].x, cv[c * 4 + u].y, cv[c * 4 + u].z, cv[c * 4 + u].w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float2 cf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&cw[e]));
                        const __half2 ch = __floats2half2_rn(cf.x, cf.y);
                        ca[u * 4 + e] = *reinterpret_cast<const uint32_t*>(&ch);
                    }
                }
                tc::tmem_st16(tmem + lane_addr + kColC + 16u * c, ca);
            }
#pragma unroll
            for (int u = 0; u < 16; ++u) cv[u] = qrow[u];
#pragma unroll
            for (int u = 0; u < 16; ++u) {
                const uint32_t qw[4] = {cv[u].x, cv[u].y, cv[u].z, cv[u].w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float2 qf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&qw[e]));
                    ssq = fmaf(qf.x, qf.x, fmaf(qf.y, qf.y, ssq));
                }
            }
            // Ebar row (fp32) into shared memory, 16-byte chunks swizzled by row
            const uint4* erow = reinterpret_cast<const uint4*>(E + (tok * G + g) * kP);
            uint4 ev[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) ev[u] = erow[u];
            float e[kP];
            float sse = 0.0f;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const uint32_t ew[4] = {ev[u].x, ev[u].y, ev[u].z, ev[u].w};
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&ew[q]));
                    e[u * 8 + 2 * q] = f.x;
                    e[u * 8 + 2 * q + 1] = f.y;
                    sse = fmaf(f.x, f.x, fmaf(f.y, f.y, sse));
                }
            }
            const float ie = rsqrtf(sse / (float)kP + eps);
#pragma unroll
            for (int c = 0; c < kP / 4; ++c)
                sm.ebar[row][c ^ (row & 15)] =
                    make_float4(e[4 * c] * ie, e[4 * c + 1] * ie, e[4 * c + 2] * ie, e[4 * c + 3] * ie);
        }
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
        tc::tc_fence_before();
        tc::mbar_arrive(&sm.a_ready);
        asm volatile("bar.sync 1, 256;" ::: "memory");  // Ebar rows visible to both warpgroups
        const float lscale = rsqrtf(ssq / (float)kN + eps) * rsqrtf((float)kN);

        float O[kP];
#pragma unroll
        for (int p = 0; p < kP; ++p) O[p] = 0.0f;
        float m = -INFINITY, dsum = 0.0f;
        bool ok = true;
        const uint32_t ua = tmem + lane_addr + kColU + (uint32_t)(128 * wg);  // hi | lo of head h
        const uint32_t va = tmem + lane_addr + kColV + (uint32_t)(64 * wg);
        for (int j = 0; j < nj; ++j) {
            const uint32_t ph = (uint32_t)(j & 1);
            if (!warp_wait(&sm.u_full, ph, wait_limit_ns, abort)) {
                fail(abort, 4);
                ok = false;
                break;
            }
            tc::tc_fence_after();
            float l = 0.0f;
#pragma unroll
            for (int half = 0; half < 2; ++half) {  // columns 0..31 then 32..63, hi and lo
                float v[64];
                tmem_ld32x2(ua + 32u * half, ua + 64u + 32u * half, v);
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const float4 e = sm.ebar[row][(8 * half + q) ^ (row & 15)];
                    l = fmaf(v[4 * q] + v[32 + 4 * q], e.x, l);
                    l = fmaf(v[4 * q + 1] + v[33 + 4 * q], e.y, l);
                    l = fmaf(v[4 * q + 2] + v[34 + 4 * q], e.z, l);
                    l = fmaf(v[4 * q + 3] + v[35 + 4 * q], e.w, l);
                }
            }
            tc::tc_fence_before();
            tc::mbar_arrive(&sm.u_free);
            l *= lscale;
            const bool use = j < nh;
            const float mn = use ? fmaxf(m, l) : m;
            const float sc = use ? expf(m - mn) : 1.0f;
            const float pe = use ? expf(l - mn) : 0.0f;
            const float w = pe * __ldg(scale + ((i64)b * Mc + j) * H + h);
            dsum = fmaf(dsum, sc, pe);
            m = mn;
            if (!warp_wait(&sm.v_full, ph, wait_limit_ns, abort)) {
                fail(abort, 4);
                ok = false;
                break;
            }
            tc::tc_fence_after();
            {
                float v[64];
                tmem_ld32x2(va, va + 32u, v);
                tc::tc_fence_before();
                tc::mbar_arrive(&sm.v_free);
#pragma unroll
                for (int p = 0; p < kP; ++p) O[p] = fmaf(O[p], sc, w * v[p]);
            }
        }
        if (ok) {
            // R = O / d, lse, gated merge (the row's loads issued first)
            const i64 rowo = tok * H + h;
            const bool has = nh > 0;
            const float inv_d = has ? 1.0f / dsum : 0.0f;
            const float gate = silu_f32(__bfloat162float(z[rowo]));
            float ys[kP];
#pragma unroll
            for (int c = 0; c < 4; ++c) load_row16(Yssd + rowo * kP + 16 * c, ys + 16 * c);
#pragma unroll
            for (int p = 0; p < kP; ++p) {
                O[p] = has ? O[p] * inv_d : 0.0f;
                ys[p] = fmaf(gate, O[p], ys[p]);
            }
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                store_row16(Y + rowo * kP + 16 * c, ys + 16 * c);
                if (R != nullptr) store_row16(R + rowo * kP + 16 * c, O + 16 * c);
            }
            if (lse != nullptr) lse[rowo] = has ? m + logf(dsum) : -INFINITY;
        }
    }

    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, kTmemCols);
    }
}

}  // namespace

size_t sma_tc_workspace(int64_t B, int64_t Mc, int64_t H) {
    const size_t ops = (size_t)(B * Mc * (H / kHeadsPerCta)) * kPair;
    const size_t sc = (size_t)(B * Mc * H) * sizeof(float);
    return ops + ((sc + 255) & ~(size_t)255);
}

bool sma_tc_supported(const SmaArgs& a) {
    return a.P == kP && a.N == kN && a.S % kRows == 0 && a.L % kRows == 0 &&
           a.H % kHeadsPerCta == 0 && (a.H / a.G) % kHeadsPerCta == 0;
}

template <typename Tmem, typename Tout>
cudaError_t launch_sma_forward_tc(const SmaArgs& a, void* ws, unsigned long long wait_limit_ns,
                                  cudaStream_t stream) {
    const int Bsz = (int)a.B, L = (int)a.L, H = (int)a.H, Mc = (int)(a.L / a.S);
    uint8_t* ops = (uint8_t*)ws;
    float* scale = (float*)(ops + (size_t)(a.B * Mc * (H / kHeadsPerCta)) * kPair);
    if (Mc > 1) {
        sma_operands_kernel<Tmem><<<dim3(Mc - 1, H, Bsz), 256, 0, stream>>>(
            (const Tmem*)a.M, a.rM, ops, scale, Mc, H, a.eps);
        note_launches(1);
    }
    const size_t smem = sizeof(TcSmem) + 1024;
    auto kern = sma_tc_kernel<Tout>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int items = (L / kRows) * Bsz * (H / kHeadsPerCta);
    kern<<<items, kThreads, smem, stream>>>(ops, scale, (const __nv_bfloat16*)a.Q,
                                            (const __nv_bfloat16*)a.Cm, (const __nv_bfloat16*)a.E,
                                            (const __nv_bfloat16*)a.z, (const Tout*)a.Yssd,
                                            (Tout*)a.Y, (Tout*)a.R, a.lse, Bsz, L, H, (int)a.G,
                                            (int)a.S, Mc, a.eps, wait_limit_ns);
    note_launches(1);
    return cudaGetLastError();
}

typedef __nv_bfloat16 bf16;
template cudaError_t launch_sma_forward_tc<float, float>(const SmaArgs&, void*, unsigned long long,
                                                         cudaStream_t);
template cudaError_t launch_sma_forward_tc<bf16, float>(const SmaArgs&, void*, unsigned long long,
                                                        cudaStream_t);
template cudaError_t launch_sma_forward_tc<bf16, bf16>(const SmaArgs&, void*, unsigned long long,
                                                       cudaStream_t);

int take_tc_status() {
    int v = 0;
    if (cudaMemcpyFromSymbol(&v, g_tc_status, sizeof(int)) != cudaSuccess) return -1;
    if (v != 0) {
        const int zero = 0;
        cudaMemcpyToSymbol(g_tc_status, &zero, sizeof(int));
    }
    return v;
}

}  // namespace dart
