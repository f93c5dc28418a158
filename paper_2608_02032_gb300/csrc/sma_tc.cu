// State-memory attention forward + gated merge on the 5th-generation tensor
// cores (tcgen05, TMEM, bulk async copies), for bf16 token inputs with
// P = 64, N = 128 and L a multiple of 128; for S < 128 a tile spans several
// chunks and each row keeps its own history (Sec. 3 value/key readouts, chunk
// logit, softmax over earlier chunks and R_t; App. B.1 normalised score
// branch; Alg. 1 streaming order; Sec. 3 gated merge).
//
// For a tile of 128 tokens (one TMEM lane each) and memory M_j of head h the
// kernel needs, per token t,
//   U_t = Q_t (r_j (.) M_j),   V_t = C_t M_j     (N = 128 -> P = 64 each)
//   l_{t,j} = (U_t . Ebar_t) / (rms(Q_t) sqrt(N))
// U and V are GEMMs whose token operands Q, C stay fixed for the whole tile
// (they sit in TMEM as the A operand) while the memories stream through as
// the B operand. Heads of one group share Q, C and E, so one job is one
// memory j for two heads of the same group: both heads' tiles side by side
// make an N = 128 B operand.
//
// Precision. Rounding the memory operand to one 16-bit type moves the logits
// enough to break the 2e-2 parity bar (fp16: max|err|/RMS(Y) 1.6e-2 at L = 16K
// in a CPU emulation against the oracle, bf16 far more), so W = r (.) M is
// split into an fp16 part W16 and its residual 2^12 (W - W16) in e4m3: one
// chain of eight fp16 MMAs (K = 16) and one of four e4m3 MMAs (K = 32, the
// kind::f8f6f4 form) into the same accumulator, together ~2^-15 relative.
// Their A operands are Q itself: fp16 after an exact per-row power-of-two
// scale that puts its largest entry in [2^14, 2^15) (in TMEM), and e4m3 of
// the same row scaled 2^-12 further (in shared memory), so both chains
// accumulate Q W at one scale. The value path runs in fp16 on M / max|M_j|
// (scale re-applied in the epilogue); C is widened to fp16 after the same kind
// of row scale (undone on R). Qbar's RMS scale, the row scale and Ebar stay
// fp32 in the epilogue. Emulated against the oracle at L = 16K, R and Y
// carry the same error as a bf16 hi + lo split of W (~3e-3, set by the value
// path); lse's error grows from 5e-6 to 1.6e-5.
//
// Cost model (measured on GB300): a tcgen05.mma with M = 128 takes ~64 cycles
// at N = 128 (K = 16 for 16-bit operands, K = 32 for e4m3), i.e. the full
// 8192 flop/cycle/SM. One job is twenty such MMAs (W16 and residual into U,
// value into V), ~1280 cycles, fed by 80 KiB of operands.
//
// Kernel 1 (sma_operands_kernel) writes per (memory, pair of heads) the
// 32 KiB part [W16 h0 | W16 h1] (MN-major), the 16 KiB residual part (rows
// h * 64 + p, K-major) and the 32 KiB part [M16 h0 | M16 h1], already in the
// 128-byte-swizzled shared-memory layouts, contiguous, so a job's operands
// are one bulk copy.
// Kernel 2 (sma_tc_kernel), one CTA per (batch, 128-token tile, 2 heads),
// grouped by (batch, head pair), heaviest tiles first inside a group:
//   warp 0      producer: one bulk copy per job into two 80 KiB job buffers
//   warp 1      TMEM allocation; one thread issues the MMAs
//   warps 2, 3  idle (they complete warpgroup 0 for the register split)
//   warps 4..7  epilogue warpgroup 0: head 0 of the pair (stages Q)
//   warps 8..11 epilogue warpgroup 1: head 1 of the pair (stages C)
// An epilogue thread owns one token row of its head: it reads its 64 columns
// of U and of V from TMEM, runs the online softmax (the running sum is only
// rescaled when the maximum moves), and finally writes R = O / d, lse and
// Y = Y_ssd + SiLU(z) R.
// TMEM: [0,64) Q (fp16 pairs), [64,128) C (fp16 pairs), [128,256) U,
// [256,384) and [384,512) V (two buffers, jobs alternate). Shared memory
// (192 KiB): two 80 KiB job buffers, the 16 KiB e4m3 Q tile and a 16 KiB tail
// where the prologue stages the E rows; the prologue's Q / C rows and the
// merge's Y_ssd, Y and R rows pass through job buffers no copy is using.
//
// Synchronisation, job j, b = j & 1. The MMA thread pays for barrier
// operations with idle tensor cycles, and most for a wait right after a
// commit (measured: ~100 cycles each time), so it does all of a job's waits
// first and commits only between MMA chains: wait u_free (the epilogue has
// read U of job j - 1), v_free[b] (it has read V of job j - 2) and the
// job's parts (full[b], one copy), then W16, residual, commit uready[b], V into buffer
// b, commit vready[b]. The producer refills job buffer b once job j - 2 is done
// with it (uready[b], vready[b]); the epilogue reads U on uready[b] and V on
// vready[b]. Every barrier's waiter is at most one phase behind it, which the
// parity waits need.
#include <math.h>

#include <type_traits>

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_fp8.h>

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
constexpr int kPart = kHeadsPerCta * kTile;   // one N = 128 B operand: both heads' tiles
constexpr int kPartsPerJob = 3;               // backward layout parts: W_hi, W_lo, M16 (+ M_hi, M_lo)
constexpr int kPair = kPartsPerJob * kPart;   // workspace bytes per (memory, head pair)
constexpr int kStages = 6;                    // ring of kPart-sized stages (192 KiB)
// forward layout, per (memory, head pair): [W16 h0 | W16 h1], the e4m3 residual
// (128 rows h * 64 + p of 128 bytes n), [M16 h0 | M16 h1]
constexpr int kLoPart = kHeadsPerCta * kP * kN;
constexpr int kOffLo = kPart, kOffV = kPart + kLoPart;
constexpr int kFwdJob = 2 * kPart + kLoPart;  // 80 KiB
static_assert(kFwdJob == kSmaJob && kOffLo == kSmaOffLo && kOffV == kSmaOffV && kTile == kSmaTile,
              "the forward layout is the one the chunk-state kernel writes");
constexpr int kQ8Off = 2 * kFwdJob;           // the e4m3 Q tile (A of the residual chain) after two jobs
static_assert(kQ8Off + kRows * kN <= kStages * kPart, "two job buffers and the Q tile fit the ring");
static_assert(kFwdJob <= kPair, "the forward layout fits the workspace sized for the backward one");
constexpr int kThreads = 384;
// Register split: launched at 168 per thread (384 x 168 = 64512 of the 65536
// of an SM); warpgroup 0 (producer, MMA, two idle warps) drops to 64 and the
// epilogue warpgroups rise to 216: 128 x 64 + 256 x 216 = 63488, within the
// launch pool, and per sub-partition (64 + 2 x 216) x 32 = 15872 <= 16384.
constexpr int kRegsLow = 64, kRegsHigh = 216;
constexpr uint32_t kTmemCols = 512;
// Row transposes in shared memory: an epilogue warp moves the 32 rows of its
// quadrant between global memory (whole rows per vector load or store,
// coalesced) and row slots padded by 16 bytes (a lane's 16-byte accesses to
// its own row then hit all 32 banks across the warp).
constexpr int kSlots = 32 * (256 + 16);  // one warp's slots for rows of up to 256 bytes
static_assert(kFwdJob + 8 * kSlots <= kQ8Off, "prologue slots fit job buffer 1");
static_assert(16 * kSlots <= kStages * kPart, "merge slots fit the ring");
static_assert(8 * kSlots <= kFwdJob, "one job buffer holds every epilogue warp's merge slots");
// E rows of the prologue: 32 rows of 128 bytes per quadrant, 16-byte chunks XORed with
// the row, in the ring's tail after the e4m3 Q tile (untouched by copies and the merge)
constexpr int kEOff = kQ8Off + kRows * kN;
static_assert(kEOff + 4 * 32 * 2 * kP <= kStages * kPart, "the E rows fit the ring's tail");
constexpr uint32_t kColQ = 0, kColC = 64, kColU = 128, kColV = 256;  // V buffer b at kColV + 128 b
// Bound on the final waits for this CTA's own copies and MMAs (never cut short).
constexpr uint64_t kDrainLimitNs = 2000000000ull;

constexpr uint32_t kIdescU = tc::idesc_f16(0, true, kRows, kHeadsPerCta * kP);  // fp16 W16, N = 128
constexpr uint32_t kIdescLo = tc::idesc_e4m3(kRows, kHeadsPerCta * kP);         // e4m3 residual, N = 128
constexpr uint32_t kIdescV = tc::idesc_f16(0, true, kRows, kHeadsPerCta * kP);  // fp16, N = 128

// Byte offset of element (n, p) of a 128-row x 128-byte tile in the
// 128-byte-swizzled layout: the 16-byte chunk index is XORed with n mod 8.
__device__ __forceinline__ uint32_t sw128(int n, int p) {
    const uint32_t o = (uint32_t)n * 128u + (uint32_t)p * 2u;
    return o ^ (((uint32_t)n & 7u) << 4);
}

// ------------------------------------------------------------ kernel 1
// One block of 256 threads per (j, h, b) memory. Warp w owns rows n = w + 8k;
// lane owns columns p = lane, lane + 32. Head h = 2 hp + x writes its share of
// the operands of memory j for the head pair hp:
//   pair_bytes == 0 (forward and statistics pass): at ops + ((b Mc + j) (H/2) + hp) kFwdJob
//     W16 tile x of [W16 h0 | W16 h1], rows x 64 .. x 64 + 63 of the e4m3 residual
//     part (transposed through shared memory: K-major, the reduction index n along
//     a row), and tile x of [M16 h0 | M16 h1];
//   otherwise (the backward's layout, pair_bytes bytes per pair): tile x of each
//     part W_hi, W_lo, M16 and, when pair_bytes holds five parts, M split bf16 hi + lo.
template <typename Tmem>
__global__ void __launch_bounds__(256)
sma_operands_kernel(const Tmem* __restrict__ M, const float* __restrict__ rM,
                    uint8_t* __restrict__ ops, float* __restrict__ scale, int Mc, int H,
                    float eps, int pair_bytes) {
    const int j = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const i64 mem = ((i64)b * Mc + j) * H + h;
    const Tmem* src = M + mem * (kN * kP);
    const i64 pair = ((i64)b * Mc + j) * (H / kHeadsPerCta) + h / kHeadsPerCta;
    const int x = h % kHeadsPerCta;
    const bool fwd = pair_bytes == 0;
    uint8_t* base = ops + pair * (fwd ? (i64)kFwdJob : (i64)pair_bytes);
    uint8_t* dst_hi = base + x * kTile;                        // W16 or W_hi
    uint8_t* dst_lo = fwd ? nullptr : dst_hi + kPart;          // W_lo (backward layout)
    uint8_t* dst_v = fwd ? base + kOffV + x * kTile : dst_hi + 2 * kPart;
    uint8_t* dst_mb = pair_bytes > kPair ? dst_hi + 3 * kPart : nullptr;  // then + kPart: lo
    __shared__ float s_max[8];
    __shared__ __align__(16) uint8_t s_res[kP][kN + 16];  // forward: e4m3 residual rows p, bytes n

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
            const uint32_t o = sw128(n, p);
            *reinterpret_cast<__half*>(dst_v + o) = __float2half_rn(v * inv_s);
            if (fwd) {
                // |W| <= sqrt(P) (r normalises the row), so W16 needs no scale; the
                // residual is at most 2^-11 |W| <= 2^-8, and 2^12 times it stays
                // inside e4m3's range
                const __half w16 = __float2half_rn(wv);
                *reinterpret_cast<__half*>(dst_hi + o) = w16;
                const __nv_fp8_e4m3 r8(4096.0f * (wv - __half2float(w16)));
                s_res[p][n] = r8.__x;
            } else {
                const __nv_bfloat16 hi = __float2bfloat16_rn(wv);
                *reinterpret_cast<__nv_bfloat16*>(dst_hi + o) = hi;
                *reinterpret_cast<__nv_bfloat16*>(dst_lo + o) = __float2bfloat16_rn(wv - __bfloat162float(hi));
                if (dst_mb != nullptr) {
                    const __nv_bfloat16 mh = __float2bfloat16_rn(v);
                    *reinterpret_cast<__nv_bfloat16*>(dst_mb + o) = mh;
                    *reinterpret_cast<__nv_bfloat16*>(dst_mb + kPart + o) = __float2bfloat16_rn(v - __bfloat162float(mh));
                }
            }
        }
    }
    if (fwd) {
        // the residual rows x 64 + p, 128 bytes each, in the 128-byte swizzle: 512 chunks of 16 bytes
        __syncthreads();
        uint8_t* dres = base + kOffLo;
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const int c = threadIdx.x + 256 * i, p = c >> 3, q = c & 7;
            const uint32_t row = (uint32_t)(x * kP + p);
            *reinterpret_cast<uint4*>(dres + row * 128u + (((uint32_t)q ^ (row & 7u)) << 4)) =
                *reinterpret_cast<const uint4*>(&s_res[p][q * 16]);
        }
    }
}

// ------------------------------------------------------------ kernel 2
struct TcSmem {
    uint8_t ring[kStages * kPart];  // job buffers, the e4m3 Q tile, row staging; 1024-aligned by placement
    float lq[kRows];                // per-row logit factor 1 / (rms(Q_t) sqrt(N))
    float cdown[kRows];             // per-row power of two undoing C's scale
    uint64_t full[2];        // job j's three parts landed in stages 3b .. 3b+2 (producer -> MMA)
    uint64_t uready[2];      // U of job j done, i.e. its hi and lo stages consumed (MMA -> epilogue, producer)
    uint64_t vready[2];      // V of job j done, its value stage consumed (MMA -> epilogue, producer)
    uint64_t u_free;         // epilogue read U of job j (MMA waits before job j + 1); 8 warps
    uint64_t v_free[2];      // epilogue read V of job j from buffer j & 1 (MMA waits before job j + 2)
    uint64_t a_ready, drain;
    uint32_t tmem_base;
    int abort;
};

__device__ __forceinline__ void fail(volatile int* abort, int code) {
    *abort = 1;
    atomicCAS(&g_tc_status, 0, code);
}

// Warp-uniform bounded wait (every lane waits; all lanes see the same outcome).
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, uint64_t limit_ns,
                                          volatile int* abort) {
    const bool got = tc::mbar_wait(bar, parity, limit_ns, abort);
    return __all_sync(0xffffffffu, got);
}

// The warp's TMEM loads are complete (each lane waited on them): one arrival
// for the whole warp (the barrier counts warps, keeping its traffic low).
__device__ __forceinline__ void warp_release(uint64_t* bar) {
    tc::tc_fence_before();
    __syncwarp();
    if ((threadIdx.x & 31) == 0) tc::mbar_arrive(bar);
}

// tcgen05.ld of 32 consecutive fp32 columns of this thread's lane, waited; the
// values come back as 16 packed pairs (column 2i in the low half).
__device__ __forceinline__ void tmem_ld32p(uint32_t taddr, uint64_t (&v)[16]) {
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
    for (int i = 0; i < 16; ++i)
        asm("mov.b64 %0, {%1, %2};" : "=l"(v[i]) : "r"(r[2 * i]), "r"(r[2 * i + 1]));
}

// Packed fp32 pairs (x in the low half). The epilogue's multiply-adds run as
// fma.rn.f32x2, two lanes of fp32 per instruction: same rounding as two
// scalar fmaf, half the issue slots, which matters here because the MMA warp
// shares each sub-partition's issue slots with two epilogue warps.
__device__ __forceinline__ uint64_t f2_pack(float x, float y) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(x), "f"(y));
    return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t v, float& x, float& y) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(x), "=f"(y) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}
__device__ __forceinline__ uint64_t f2_mul(uint64_t a, uint64_t b) {
    uint64_t d;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}

// The two bf16 values packed in a 32-bit word, as floats (low half first).
__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Warp-cooperative row transposes. Rows r = 0..31 of a warp start at
// base + r * stride (16-byte aligned) and hold RB bytes; slot r is at
// slots + r * (RB + 16). Each vector access of the warp covers 512 bytes of
// whole rows on the global side.
template <int RB>
__device__ __forceinline__ void rows_to_slots(uint8_t* slots, const uint8_t* base, i64 stride, int lane) {
    constexpr int kCpr = RB / 16, kRpi = 32 / kCpr;  // 16-byte chunks per row, rows per access
    uint4 v[kCpr];
#pragma unroll
    for (int i = 0; i < kCpr; ++i)
        v[i] = *reinterpret_cast<const uint4*>(base + (i64)(i * kRpi + lane / kCpr) * stride + (lane % kCpr) * 16);
#pragma unroll
    for (int i = 0; i < kCpr; ++i)
        *reinterpret_cast<uint4*>(slots + (i * kRpi + lane / kCpr) * (RB + 16) + (lane % kCpr) * 16) = v[i];
}
template <int RB>
__device__ __forceinline__ void slots_to_rows(uint8_t* base, i64 stride, const uint8_t* slots, int lane) {
    constexpr int kCpr = RB / 16, kRpi = 32 / kCpr;
#pragma unroll
    for (int i = 0; i < kCpr; ++i)
        *reinterpret_cast<uint4*>(base + (i64)(i * kRpi + lane / kCpr) * stride + (lane % kCpr) * 16) =
            *reinterpret_cast<const uint4*>(slots + (i * kRpi + lane / kCpr) * (RB + 16) + (lane % kCpr) * 16);
}

// rows_to_slots without the registers: cp.async copies straight into the slots
// (completed by cp_async_wait_all).
template <int RB>
__device__ __forceinline__ void rows_to_slots_async(uint8_t* slots, const uint8_t* base, i64 stride, int lane) {
    constexpr int kCpr = RB / 16, kRpi = 32 / kCpr;
#pragma unroll
    for (int i = 0; i < kCpr; ++i) {
        const uint32_t dst = tc::smem_u32(slots + (i * kRpi + lane / kCpr) * (RB + 16) + (lane % kCpr) * 16);
        const uint8_t* src = base + (i64)(i * kRpi + lane / kCpr) * stride + (lane % kCpr) * 16;
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// Prefetches an RB-byte row and one gate value into L2.
template <int RB, typename T>
__device__ __forceinline__ void prefetch_row(const T* row, const __nv_bfloat16* zv) {
#pragma unroll
    for (int o = 0; o < RB; o += 128)
        asm volatile("prefetch.global.L2 [%0];" ::"l"(reinterpret_cast<const uint8_t*>(row) + o));
    asm volatile("prefetch.global.L2 [%0];" ::"l"(zv));
}

// Issues the eight K = 16 MMAs of one N = 128 part: D (+)= A[tmem] * B[stage].
// `first_acc` is 0 when the first MMA starts a fresh accumulator.
template <uint32_t kIdesc, uint32_t first_acc>
__device__ __forceinline__ void issue_part(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc) {
#pragma unroll
    for (uint32_t ks = 0; ks < kN / 16; ++ks)  // +2048 bytes (+128 in the address field) per K step
        tc::mma_f16_ts(d_tmem, a_tmem + 8u * ks, b_desc + 128u * ks, kIdesc, ks > 0 ? 1u : first_acc);
}

// What the backward-statistics variant (kStats) writes instead of the merge:
// the softmax weights g_{t,j} = exp(l_{t,j} - lse_t) (lse from the forward)
// and their sum G1_t. It runs the U half of each job only (the W16 part and
// the e4m3 residual of the forward layout; no value chain). The forward variant, when g is given, writes the logits
// l_{t,j} there instead, for a backward that then needs no statistics pass.
struct SmaStats {
    float* g;    // B x H x Mc x L
    float2* gd;  // B x L x H: (G1, -) -- the second field is written later
};

template <typename Tout, bool kStats, bool kLogits = false>
__global__ void __launch_bounds__(kThreads, 1)
sma_tc_kernel(const uint8_t* __restrict__ ops, const float* __restrict__ scale,
              const __nv_bfloat16* __restrict__ Q, const __nv_bfloat16* __restrict__ Cm,
              const __nv_bfloat16* __restrict__ E, const __nv_bfloat16* __restrict__ z,
              const Tout* __restrict__ Yssd, Tout* __restrict__ Y, Tout* __restrict__ R,
              float* __restrict__ lse, int Bsz, int L, int H, int G, int S, int Mc, float eps,
              unsigned long long wait_limit_ns, int withhold, SmaStats st) {
    extern __shared__ uint8_t smem_raw[];
    TcSmem& sm = *reinterpret_cast<TcSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                            ~(uintptr_t)1023);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // work item: (batch, head pair) major, heaviest token tiles first inside it, so the
    // CTAs resident at one time stream the operands of one or two head pairs (a few MB
    // that stay in L2) rather than of all of them
    const int tiles = L / kRows;
    const int hpairs = H / kHeadsPerCta;
    const int item = blockIdx.x;
    const int grp = item / tiles;
    const int tt = tiles - 1 - item % tiles;
    const int b = grp / hpairs;
    const int hp = grp % hpairs;
    const int h0 = hp * kHeadsPerCta;
    const int t0 = tt * kRows;
    // The tile runs the jobs of its last token, j < (t0 + 127) / S; each token keeps
    // those of its own history, j < t / S (all of them when S is a multiple of the
    // tile height: the tile then lies in one chunk).
    const int nj = (t0 + kRows - 1) / S;
    volatile int* abort = &sm.abort;

    if (threadIdx.x == 0) {
        tc::mbar_init(&sm.full[0], 1);
        tc::mbar_init(&sm.full[1], 1);
        for (int u = 0; u < 2; ++u) {
            tc::mbar_init(&sm.uready[u], 1);
            tc::mbar_init(&sm.vready[u], 1);
        }
        tc::mbar_init(&sm.u_free, 8);  // one arrival per epilogue warp
        tc::mbar_init(&sm.v_free[0], 8);
        tc::mbar_init(&sm.v_free[1], 8);
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
        // one copy per job (80 KiB; the statistics pass takes only W16 and the
        // residual): job j lands in job buffer j & 1
        if (lane == 0) {
            const uint8_t* src = ops + ((i64)b * Mc * hpairs + hp) * (i64)kFwdJob;
            const i64 job_stride = (i64)hpairs * kFwdJob;
            bool ok = true;
            int njobs = 0;  // jobs whose copy was issued
            // (withhold: the failure-path test hook; every wait on the operands then runs out)
            for (int j = 0; j < (withhold ? 0 : nj); ++j) {
                const int ub = j & 1;
                // job buffer 1 holds the epilogue's row staging until the operands are in TMEM;
                // buffer j & 1 was last used by job j - 2: wait for its U and V
                const uint32_t par = (uint32_t)((j >> 1) & 1) ^ 1u;
                ok = (j != 1 || tc::mbar_wait(&sm.a_ready, 0, wait_limit_ns, abort)) &&
                     tc::mbar_wait(&sm.uready[ub], par, wait_limit_ns, abort) &&
                     (kStats || tc::mbar_wait(&sm.vready[ub], par, wait_limit_ns, abort));
                if (!ok) {
                    fail(abort, 1);
                    break;
                }
                // the job's parts are contiguous in global and in the ring
                constexpr uint32_t bytes = kStats ? kOffV : kFwdJob;
                tc::mbar_arrive_expect_tx(&sm.full[ub], bytes);
                tc::bulk_g2s(sm.ring + ub * kFwdJob, src + j * job_stride, bytes, &sm.full[ub]);
                ++njobs;
            }
            // never leave a copy in flight behind: wait for the last copy into each half
            for (int j = njobs - 1; j >= 0 && j >= njobs - 2; --j)
                if (!tc::mbar_wait(&sm.full[j & 1], (uint32_t)((j >> 1) & 1), kDrainLimitNs, nullptr))
                    atomicCAS(&g_tc_status, 0, 5);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------- MMA issuer
        if (lane == 0) {
            bool ok = tc::mbar_wait(&sm.a_ready, 0, wait_limit_ns, abort);
            if (!ok) fail(abort, 2);
            tc::tc_fence_after();
            bool issued = false;
            // descriptors of job buffer 0 (MN-major W16 / M16, K-major residual) and of the
            // e4m3 Q tile; buffer 1 is kFwdJob bytes further (>> 4 in the address field)
            const uint64_t desc0 = tc::smem_desc_sw128(tc::smem_u32(sm.ring), (uint32_t)kTile, 1024u);
            const uint64_t rdesc0 = tc::smem_desc_sw128(tc::smem_u32(sm.ring + kOffLo), 16u, 1024u);
            const uint64_t qdesc = tc::smem_desc_sw128(tc::smem_u32(sm.ring + kQ8Off), 16u, 1024u);
            for (int j = 0; ok && j < nj; ++j) {
                const int ub = j & 1;
                const uint32_t par = (uint32_t)((j >> 1) & 1);
                const uint64_t boff = (uint64_t)((ub * kFwdJob) >> 4);
                const uint64_t bd = desc0 + boff;
                ok = tc::mbar_wait(&sm.u_free, (uint32_t)ub ^ 1u, wait_limit_ns, abort) &&
                     (kStats || tc::mbar_wait(&sm.v_free[ub], par ^ 1u, wait_limit_ns, abort));
                tc::tc_fence_after();
                ok = ok && tc::mbar_wait(&sm.full[ub], par, wait_limit_ns, abort);
                if (!ok) break;
                issue_part<kIdescU, 0u>(tmem + kColU, tmem + kColQ, bd);
#pragma unroll
                for (uint32_t ks = 0; ks < kN / 32; ++ks)  // residual chain: +32 bytes per K = 32 step
                    tc::mma_e4m3_ss(tmem + kColU, qdesc + 2u * ks, rdesc0 + boff + 2u * ks, kIdescLo, 1u);
                tc::mma_commit(&sm.uready[ub]);
                if (!kStats) {
                    issue_part<kIdescV, 0u>(tmem + kColV + 128u * (uint32_t)ub, tmem + kColC,
                                            bd + (uint64_t)(kOffV >> 4));
                    tc::mma_commit(&sm.vready[ub]);
                }
                issued = true;
            }
            if (!ok) fail(abort, 3);
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

        // Rows in through shared memory, 32 rows per warp, in one round trip: Q (warpgroup 0)
        // or C (warpgroup 1) into padded slots in job buffer 1 (not needed before job 1),
        // and E, which warpgroup 0 loads for both into the ring's tail (kEOff).
        uint8_t* slots = sm.ring + kFwdJob + (warp - 4) * kSlots;
        uint8_t* eslots = sm.ring + kEOff + (warp & 3) * (32 * 2 * kP);  // rows of the quadrant
        const i64 tok0 = tok - lane;  // first token of this warp's rows
        uint4 av[16];
        uint32_t e2[kP / 2];  // the E row as bf16 pairs; Ebar = E * ie
        {
            const uint8_t* qc = reinterpret_cast<const uint8_t*>((wg == 0 ? Q : Cm) + (tok0 * G + g) * kN);
            const uint8_t* er = reinterpret_cast<const uint8_t*>(E + (tok0 * G + g) * kP);
            const i64 qs = (i64)G * kN * 2, es = (i64)G * kP * 2;
            uint4 v[16], ev[8];  // whole rows per warp access: 2 rows of Q or C, 4 of E
#pragma unroll
            for (int i = 0; i < 16; ++i)
                v[i] = *reinterpret_cast<const uint4*>(qc + (i64)(2 * i + lane / 16) * qs + (lane % 16) * 16);
            if (wg == 0) {
#pragma unroll
                for (int i = 0; i < 8; ++i)
                    ev[i] = *reinterpret_cast<const uint4*>(er + (i64)(4 * i + lane / 8) * es + (lane % 8) * 16);
            }
#pragma unroll
            for (int i = 0; i < 16; ++i)
                *reinterpret_cast<uint4*>(slots + (2 * i + lane / 16) * (2 * kN + 16) + (lane % 16) * 16) = v[i];
            if (wg == 0) {
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const int r = 4 * i + lane / 8, c = lane % 8;
                    *reinterpret_cast<uint4*>(eslots + r * 128 + ((c ^ (r & 7)) << 4)) = ev[i];
                }
            }
        }
        __syncwarp();
#pragma unroll
        for (int u = 0; u < 16; ++u) av[u] = reinterpret_cast<const uint4*>(slots + lane * (2 * kN + 16))[u];
        asm volatile("bar.sync 2, 256;" ::: "memory");  // warpgroup 0's E rows are staged
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const uint4 w = *reinterpret_cast<const uint4*>(eslots + lane * 128 + ((u ^ (lane & 7)) << 4));
            e2[4 * u] = w.x; e2[4 * u + 1] = w.y; e2[4 * u + 2] = w.z; e2[4 * u + 3] = w.w;
        }
        // The A operands: the row (Q for warpgroup 0, C for warpgroup 1) as fp16 after an
        // exact power-of-two scale 2^k that puts its largest entry in [2^14, 2^15)
        // (cmax = 1.f * 2^(ebits - 127), so k = 141 - ebits), into TMEM
        float cmax = 0.0f, ssq = 0.0f;
#pragma unroll
        for (int u = 0; u < 16; ++u) {
            const uint32_t cw[4] = {av[u].x, av[u].y, av[u].z, av[u].w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float a = bf_lo(cw[e]), d = bf_hi(cw[e]);
                cmax = fmaxf(cmax, fmaxf(fabsf(a), fabsf(d)));
                ssq = fmaf(a, a, fmaf(d, d, ssq));
            }
        }
        const int ebits = (__float_as_int(cmax) >> 23) & 0xff;
        const int k = cmax > 0.0f ? min(max(141 - ebits, -60), 60) : 0;
        const float up = __int_as_float((127 + k) << 23);
        const float down = __int_as_float((127 - k) << 23);
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            uint32_t ca[16];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const uint32_t cw[4] = {av[c * 4 + u].x, av[c * 4 + u].y, av[c * 4 + u].z, av[c * 4 + u].w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const __half2 ch = __floats2half2_rn(bf_lo(cw[e]) * up, bf_hi(cw[e]) * up);
                    ca[u * 4 + e] = *reinterpret_cast<const uint32_t*>(&ch);
                }
            }
            tc::tmem_st16(tmem + lane_addr + (wg == 0 ? kColQ : kColC) + 16u * c, ca);
        }
        if (wg == 0) {
            // Q also as e4m3 at scale 2^(k - 12) (largest entry in [4, 8)): row `row` of the
            // residual chain's K-major A tile, 128 bytes in the 128-byte swizzle
            const float up8 = __int_as_float((127 + k - 12) << 23);
            uint8_t* qrow = sm.ring + kQ8Off + row * 128;
#pragma unroll
            for (int q = 0; q < 8; ++q) {  // 16 entries n = 16 q .. 16 q + 15 per chunk
                uint32_t w4[4];  // bytes in n order (the low half of a bf16 or e4m3 pair first)
                const uint32_t wds[8] = {av[2 * q].x, av[2 * q].y, av[2 * q].z, av[2 * q].w,
                                         av[2 * q + 1].x, av[2 * q + 1].y, av[2 * q + 1].z, av[2 * q + 1].w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const uint32_t p0 = (uint32_t)__nv_cvt_float2_to_fp8x2(
                        make_float2(bf_lo(wds[2 * e]) * up8, bf_hi(wds[2 * e]) * up8), __NV_SATFINITE, __NV_E4M3);
                    const uint32_t p1 = (uint32_t)__nv_cvt_float2_to_fp8x2(
                        make_float2(bf_lo(wds[2 * e + 1]) * up8, bf_hi(wds[2 * e + 1]) * up8), __NV_SATFINITE,
                        __NV_E4M3);
                    w4[e] = (p0 & 0xffffu) | (p1 << 16);
                }
                *reinterpret_cast<uint4*>(qrow + (((uint32_t)q ^ ((uint32_t)row & 7u)) << 4)) =
                    make_uint4(w4[0], w4[1], w4[2], w4[3]);
            }
            tc::fence_proxy_async_shared();  // the MMAs read the tile through the async proxy
            // logit factor: 1 / (rms(Q_t) sqrt(N)), and the row scale undone
            sm.lq[row] = rsqrtf(ssq / (float)kN + eps) * rsqrtf((float)kN) * down;
        } else {
            sm.cdown[row] = down;
        }
        float sse = 0.0f;
#pragma unroll
        for (int i = 0; i < kP / 2; ++i) {
            const float a = bf_lo(e2[i]), c = bf_hi(e2[i]);
            sse = fmaf(a, a, fmaf(c, c, sse));
        }
        const float ie = rsqrtf(sse / (float)kP + eps);
        uint64_t eb[kP / 2];  // Ebar row as fp32 pairs
#pragma unroll
        for (int i = 0; i < kP / 2; ++i) eb[i] = f2_pack(bf_lo(e2[i]) * ie, bf_hi(e2[i]) * ie);
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
        tc::tc_fence_before();
        tc::mbar_arrive(&sm.a_ready);
        // lq and cdown visible to both warpgroups; all staging reads done before
        // the merge reuses the ring
        asm volatile("bar.sync 1, 256;" ::: "memory");
        const float lfac = sm.lq[row];
        const float cdown = sm.cdown[row];

        if constexpr (kStats) {
            // backward statistics: g_{t,j} = exp(l_{t,j} - lse_t) and G1_t = sum_j g
            const i64 rowo = tok * H + h;
            const float lse_t = lse[rowo];
            float G1 = 0.0f;
            bool ok = true;
            const uint32_t ua = tmem + lane_addr + kColU + (uint32_t)(kP * wg);
            float* gp = st.g + ((i64)b * H + h) * Mc * L + t;  // + j L
            const int njr = t / S;  // this row's memories
            for (int j = 0; j < nj; ++j) {
                const int ub = j & 1;
                if (!warp_wait(&sm.uready[ub], (uint32_t)((j >> 1) & 1), wait_limit_ns, abort)) {
                    fail(abort, 4);
                    ok = false;
                    break;
                }
                tc::tc_fence_after();
                float l;
                {
                    uint64_t acc = 0ull, v[16];
                    tmem_ld32p(ua, v);
#pragma unroll
                    for (int i = 0; i < 16; ++i) acc = f2_fma(v[i], eb[i], acc);
                    tmem_ld32p(ua + 32u, v);
                    warp_release(&sm.u_free);
#pragma unroll
                    for (int i = 0; i < 16; ++i) acc = f2_fma(v[i], eb[16 + i], acc);
                    float lx, ly;
                    f2_unpack(acc, lx, ly);
                    l = __fmul_rn(lx + ly, lfac);  // rounded: the stored and the recomputed logits agree
                }
                if (j < njr) {
                    const float gw = expf(l - lse_t);
                    G1 += gw;
                    gp[(i64)j * L] = gw;
                }
            }
            if (ok) st.gd[rowo] = make_float2(G1, 0.0f);
        } else {
            uint64_t O[kP / 2];  // running sum of w_j V_j as fp32 pairs
    #pragma unroll
            for (int i = 0; i < kP / 2; ++i) O[i] = 0ull;
            float m = -INFINITY, dsum = 0.0f;
            bool ok = true;
            const int njr = t / S;  // this row's memories (the tile's jobs beyond them are skipped)
            const float* scl = scale + (i64)b * Mc * H + h;  // scale of memory j at scl[j H]
            float s_next = nj > 0 ? __ldg(scl) : 0.0f;
            const uint32_t ua = tmem + lane_addr + kColU + (uint32_t)(kP * wg);
            const uint32_t va = tmem + lane_addr + kColV + (uint32_t)(kP * wg);  // + 128 per V buffer
            // training variant: the logits l_{t,j} for the backward (st.g: B x H x Mc x L)
            float* lgp = kLogits ? st.g + ((i64)b * H + h) * Mc * L + t : nullptr;
            // the merge's Y_ssd row and gate come from L2 if fetched a few jobs ahead
            const i64 rowo_pf = tok * H + h;
            const int pf_job = nj > 4 ? nj - 4 : 0;
            if (nj == 0) prefetch_row<kP * (int)sizeof(Tout)>(Yssd + rowo_pf * kP, z + rowo_pf);
            // one job: U -> logit -> online softmax, V -> weighted sum. kMasked: some lanes
            // of the warp may be past their history (j >= njr) and skip the softmax update
            // The merge's Y_ssd rows land in the job buffer of job nj - 2 (done) while the last
            // job runs: cp.async straight into this warp's slots there.
            uint8_t* yslots_last = sm.ring + (nj & 1) * kFwdJob + (warp - 4) * kSlots;
            float zlast = 0.0f;
            auto job = [&](int j, auto masked) -> bool {
                constexpr bool kMasked = decltype(masked)::value;
                const int ub = j & 1;
                const float s_j = s_next;
                if (j == pf_job) prefetch_row<kP * (int)sizeof(Tout)>(Yssd + rowo_pf * kP, z + rowo_pf);
                if (j == nj - 1) {
                    griddep_wait();  // Y_ssd: the kernel launched before this one is done
                    rows_to_slots_async<kP * (int)sizeof(Tout)>(
                        yslots_last, reinterpret_cast<const uint8_t*>(Yssd + (tok0 * H + h) * kP),
                        (i64)H * kP * (i64)sizeof(Tout), lane);
                    zlast = __bfloat162float(z[rowo_pf]);
                }
                if (j + 1 < nj) s_next = __ldg(scl + (i64)(j + 1) * H);  // one job ahead
                if (!warp_wait(&sm.uready[ub], (uint32_t)((j >> 1) & 1), wait_limit_ns, abort)) {
                    fail(abort, 4);
                    return false;
                }
                tc::tc_fence_after();
                float l;
                {
                    uint64_t acc = 0ull, v[16];
                    tmem_ld32p(ua, v);
#pragma unroll
                    for (int i = 0; i < 16; ++i) acc = f2_fma(v[i], eb[i], acc);
                    tmem_ld32p(ua + 32u, v);
                    warp_release(&sm.u_free);
#pragma unroll
                    for (int i = 0; i < 16; ++i) acc = f2_fma(v[i], eb[16 + i], acc);
                    float lx, ly;
                    f2_unpack(acc, lx, ly);
                    l = __fmul_rn(lx + ly, lfac);  // rounded: the stored and the recomputed logits agree
                }
                float w = 0.0f;
                if (!kMasked || j < njr) {
                    if constexpr (kLogits) lgp[(i64)j * L] = l;
                    // online softmax; the running sums are rescaled only when the maximum moves
                    if (l > m) {
                        const float sc = expf(m - l);
                        const uint64_t sc2 = f2_pack(sc, sc);
#pragma unroll
                        for (int i = 0; i < kP / 2; ++i) O[i] = f2_mul(O[i], sc2);
                        dsum *= sc;
                        m = l;
                    }
                    const float pe = expf(l - m);
                    dsum += pe;
                    w = pe * s_j;
                }
                const uint64_t w2 = f2_pack(w, w);
                if (!warp_wait(&sm.vready[ub], (uint32_t)((j >> 1) & 1), wait_limit_ns, abort)) {
                    fail(abort, 4);
                    return false;
                }
                tc::tc_fence_after();
                {
                    uint64_t v[16];
                    tmem_ld32p(va + 128u * ub, v);
#pragma unroll
                    for (int i = 0; i < 16; ++i) O[i] = f2_fma(w2, v[i], O[i]);
                    tmem_ld32p(va + 128u * ub + 32u, v);
                    warp_release(&sm.v_free[ub]);
#pragma unroll
                    for (int i = 0; i < 16; ++i) O[16 + i] = f2_fma(w2, v[i], O[16 + i]);
                }
                return true;
            };
            // jobs every row of the warp keeps (all of them when S >= 128), then the tail
            const int njw = min(nj, (t0 + 32 * (warp & 3)) / S);
            int j = 0;
            for (; ok && j < njw; ++j) ok = job(j, std::false_type{});
            for (; ok && j < nj; ++j) ok = job(j, std::true_type{});
            if (nj > 0) cp_async_wait_all();  // also when a wait gave up: no copy outlives the CTA
            if (ok) {
                // R = O / d (C's row scale undone), lse, gated merge. Every MMA is done
                // (the last job's V was read, or there were no jobs), so the ring is free
                // for the row transposes: Y_ssd in (already there when there were jobs),
                // Y and R out.
                constexpr int kRowB = kP * (int)sizeof(Tout);
                const i64 rowo = tok * H + h;
                const i64 row0 = tok0 * H + h;  // this warp's first output row
                uint8_t* yslots = nj > 0 ? yslots_last : sm.ring + (warp - 4) * 2 * kSlots;
                uint8_t* rslots = nj > 0 ? sm.ring + ((nj - 1) & 1) * kFwdJob + (warp - 4) * kSlots
                                         : yslots + kSlots;
                const i64 rstride = (i64)H * kRowB;
                const bool has = njr > 0;
                const float inv_d = has ? cdown / dsum : 0.0f;
                const float gate = silu_f32(nj > 0 ? zlast : __bfloat162float(z[rowo]));
                if (nj == 0) {
                    griddep_wait();
                    rows_to_slots<kRowB>(yslots, reinterpret_cast<const uint8_t*>(Yssd + row0 * kP), rstride, lane);
                }
                float r[kP];
    #pragma unroll
                for (int i = 0; i < kP / 2; ++i) {
                    f2_unpack(O[i], r[2 * i], r[2 * i + 1]);
                    r[2 * i] *= inv_d;
                    r[2 * i + 1] *= inv_d;
                }
                Tout* rs = reinterpret_cast<Tout*>(rslots + lane * (kRowB + 16));
                Tout* ys = reinterpret_cast<Tout*>(yslots + lane * (kRowB + 16));
    #pragma unroll
                for (int c = 0; c < 4; ++c) store_row16(rs + 16 * c, r + 16 * c);
                if (lse != nullptr) lse[rowo] = has ? m + logf(dsum) : -INFINITY;
                __syncwarp();
    #pragma unroll
                for (int c = 0; c < 4; ++c) {
                    float y[16];
                    load_row16(ys + 16 * c, y);
    #pragma unroll
                    for (int i = 0; i < 16; ++i) y[i] = fmaf(gate, r[16 * c + i], y[i]);
                    store_row16(ys + 16 * c, y);
                }
                __syncwarp();
                slots_to_rows<kRowB>(reinterpret_cast<uint8_t*>(Y + row0 * kP), rstride, yslots, lane);
                if (R != nullptr) slots_to_rows<kRowB>(reinterpret_cast<uint8_t*>(R + row0 * kP), rstride, rslots, lane);
            }
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

size_t sma_tiles_scale_offset(int64_t B, int64_t Mc, int64_t H) {
    return ((size_t)(B * Mc * (H / kHeadsPerCta)) * kFwdJob + 255) & ~(size_t)255;
}
size_t sma_tiles_bytes(int64_t B, int64_t Mc, int64_t H) {
    return sma_tiles_scale_offset(B, Mc, H) + (((size_t)(B * Mc * H) * sizeof(float) + 255) & ~(size_t)255);
}

size_t sma_tc_workspace(int64_t B, int64_t Mc, int64_t H) {
    const size_t ops = (size_t)(B * Mc * (H / kHeadsPerCta)) * kPair;
    const size_t sc = (size_t)(B * Mc * H) * sizeof(float);
    return ops + ((sc + 255) & ~(size_t)255);
}

bool sma_tc_supported(const SmaArgs& a) {
    return a.P == kP && a.N == kN && a.L % kRows == 0 &&
           a.H % kHeadsPerCta == 0 && (a.H / a.G) % kHeadsPerCta == 0;
}

template <typename Tmem, typename Tout>
cudaError_t launch_sma_forward_tc(const SmaArgs& a, void* ws, unsigned long long wait_limit_ns,
                                  cudaStream_t stream) {
    const int Bsz = (int)a.B, L = (int)a.L, H = (int)a.H, Mc = (int)(a.L / a.S);
    const uint8_t* ops;
    const float* scale;
    if (a.tiles != nullptr) {  // built by the chunk-state kernel
        ops = a.tiles;
        scale = (const float*)(a.tiles + sma_tiles_scale_offset(a.B, Mc, a.H));
    } else {
        uint8_t* w = (uint8_t*)ws;
        float* sc = (float*)(w + (size_t)(a.B * Mc * (H / kHeadsPerCta)) * kPair);
        if (Mc > 1) {
            sma_operands_kernel<Tmem><<<dim3(Mc - 1, H, Bsz), 256, 0, stream>>>(
                (const Tmem*)a.M, a.rM, w, sc, Mc, H, a.eps, 0);  // the forward layout
            note_launches(1);
        }
        ops = w;
        scale = sc;
    }
    const size_t smem = sizeof(TcSmem) + 1024;
    auto kern = a.logits != nullptr ? sma_tc_kernel<Tout, false, true> : sma_tc_kernel<Tout, false>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int items = (L / kRows) * Bsz * (H / kHeadsPerCta);
    // Programmatic stream serialization: after the scan's output kernel (which lets
    // its dependents start once all its CTAs run), this grid's CTAs take the SMs that
    // kernel's last wave leaves idle. Only Y_ssd comes from that kernel, and every
    // thread reads it after griddep_wait. After any other kernel the launch waits for
    // it to finish, as a plain launch does.
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)items);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, kern, ops, scale, (const __nv_bfloat16*)a.Q, (const __nv_bfloat16*)a.Cm,
                           (const __nv_bfloat16*)a.E, (const __nv_bfloat16*)a.z, (const Tout*)a.Yssd, (Tout*)a.Y,
                           (Tout*)a.R, a.lse, Bsz, L, H, (int)a.G, (int)a.S, Mc, a.eps, wait_limit_ns,
                           a.test_withhold, SmaStats{a.logits, nullptr});
    if (e != cudaSuccess) return e;
    note_launches(1);
    return cudaGetLastError();
}

template <typename Tmem>
cudaError_t launch_sma_bwd_stats_tc(const SmaBwdArgs& a, const float* rM, uint8_t* ops,
                                    int pair_bytes, float* scale, float* g, float2* gd,
                                    unsigned long long wait_limit_ns, cudaStream_t stream) {
    const int Bsz = (int)a.B, L = (int)a.L, H = (int)a.H, Mc = (int)(a.L / a.S);
    // the statistics pass recomputes the logits exactly as the forward did, from the
    // forward's operand layout; the backward's own layout (pair_bytes per pair) then
    // overwrites it for the kernels that follow
    if (Mc > 1) {
        sma_operands_kernel<Tmem><<<dim3(Mc - 1, H, Bsz), 256, 0, stream>>>(
            (const Tmem*)a.M, rM, ops, scale, Mc, H, a.eps, 0);
        note_launches(1);
    }
    const size_t smem = sizeof(TcSmem) + 1024;
    auto kern = sma_tc_kernel<float, true>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int items = (L / kRows) * Bsz * (H / kHeadsPerCta);
    SmaStats st{g, gd};
    kern<<<items, kThreads, smem, stream>>>(ops, scale, (const __nv_bfloat16*)a.Q,
                                            (const __nv_bfloat16*)a.Cm, (const __nv_bfloat16*)a.E,
                                            (const __nv_bfloat16*)a.z, nullptr, nullptr, nullptr,
                                            const_cast<float*>(a.lse), Bsz, L, H, (int)a.G,
                                            (int)a.S, Mc, a.eps, wait_limit_ns, 0, st);
    note_launches(1);
    if (Mc > 1) {
        sma_operands_kernel<Tmem><<<dim3(Mc - 1, H, Bsz), 256, 0, stream>>>(
            (const Tmem*)a.M, rM, ops, scale, Mc, H, a.eps, pair_bytes);
        note_launches(1);
    }
    return cudaGetLastError();
}
template cudaError_t launch_sma_bwd_stats_tc<float>(const SmaBwdArgs&, const float*, uint8_t*, int,
                                                    float*, float*, float2*, unsigned long long,
                                                    cudaStream_t);
template cudaError_t launch_sma_bwd_stats_tc<__nv_bfloat16>(const SmaBwdArgs&, const float*, uint8_t*,
                                                            int, float*, float*, float2*,
                                                            unsigned long long, cudaStream_t);

// g_{t,j} = exp(l_{t,j} - lse_t) for j < t / S and G1_t = sum_j g from the
// logits the forward saved: the statistics pass's arithmetic in its order,
// without recomputing the logit chains. One thread per (b, h, t).
__global__ void sma_g_from_logits_kernel(const float* __restrict__ logits, const float* __restrict__ lse,
                                         float* __restrict__ g, float2* __restrict__ gd, int L, int H,
                                         int S, int Mc) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x, h = blockIdx.y, b = blockIdx.z;
    if (t >= L) return;
    const int nj = t / S;
    const i64 rowo = ((i64)b * L + t) * H + h;
    const float lse_t = lse[rowo];
    const i64 base = ((i64)b * H + h) * Mc * L + t;
    float G1 = 0.0f;
    for (int j = 0; j < nj; ++j) {
        const float gw = expf(logits[base + (i64)j * L] - lse_t);
        G1 += gw;
        g[base + (i64)j * L] = gw;
    }
    gd[rowo] = make_float2(G1, 0.0f);
}

template <typename Tmem>
cudaError_t launch_sma_bwd_stats_from_logits(const SmaBwdArgs& a, const float* rM, uint8_t* ops,
                                             int pair_bytes, float* scale, float* g, float2* gd,
                                             cudaStream_t stream) {
    const int Bsz = (int)a.B, L = (int)a.L, H = (int)a.H, Mc = (int)(a.L / a.S);
    if (Mc > 1) {  // the backward's operand tiles, as in the statistics pass
        sma_operands_kernel<Tmem><<<dim3(Mc - 1, H, Bsz), 256, 0, stream>>>(
            (const Tmem*)a.M, rM, ops, scale, Mc, H, a.eps, pair_bytes);
        note_launches(1);
    }
    sma_g_from_logits_kernel<<<dim3((L + 255) / 256, H, Bsz), 256, 0, stream>>>(a.logits, a.lse, g, gd, L, H,
                                                                                 (int)a.S, Mc);
    note_launches(1);
    return cudaGetLastError();
}
template cudaError_t launch_sma_bwd_stats_from_logits<float>(const SmaBwdArgs&, const float*, uint8_t*, int,
                                                             float*, float*, float2*, cudaStream_t);
template cudaError_t launch_sma_bwd_stats_from_logits<__nv_bfloat16>(const SmaBwdArgs&, const float*,
                                                                     uint8_t*, int, float*, float*, float2*,
                                                                     cudaStream_t);

typedef __nv_bfloat16 bf16;
template cudaError_t launch_sma_forward_tc<float, float>(const SmaArgs&, void*, unsigned long long,
                                                         cudaStream_t);
template cudaError_t launch_sma_forward_tc<bf16, float>(const SmaArgs&, void*, unsigned long long,
                                                        cudaStream_t);
template cudaError_t launch_sma_forward_tc<bf16, bf16>(const SmaArgs&, void*, unsigned long long,
                                                       cudaStream_t);

// Read and clear of the status word in one device-side exchange: a code that a
// kernel still running on another stream records is either returned now or kept
// for the next read, never lost between a read and a separate clear.
__device__ int g_tc_status_taken;
__global__ void take_tc_status_kernel() { g_tc_status_taken = atomicExch(&g_tc_status, 0); }

int take_tc_status(cudaStream_t stream) {
    take_tc_status_kernel<<<1, 1, 0, stream>>>();
    int v = 0;
    if (cudaGetLastError() != cudaSuccess ||
        cudaMemcpyFromSymbolAsync(&v, g_tc_status_taken, sizeof(int), 0, cudaMemcpyDeviceToHost, stream) !=
            cudaSuccess ||
        cudaStreamSynchronize(stream) != cudaSuccess)
        return -1;
    return v;
}

}  // namespace dart
