// Chunked SSD scan on the 5th-generation tensor cores for bf16 token inputs,
// P = 64, N = 128, S in {64, 128, 256} (Sec. 2; Sec. 3 "Chunk State Memories";
// App. A chunked scan). The chunk-state and chunk-output kernels run on the
// tensor cores, the state passing streams the chunk states through shared
// memory with bulk copies; the within-chunk cumsum is shared with the FFMA
// path (scan.cu).
//
// chunk_state_tc_kernel, one CTA (256 threads) per (chunk c, head group, b):
//   M_c = B_c^T (w (.) X_c),  w_s = exp(cum_end - cum_s) dt_s      (App. A)
//   A = B_c^T sits in TMEM (lane n, K = s); the B operand w (.) X_c is staged
//   per head as bf16 hi + lo (two MMAs, ~2^-16 relative) in the 128-byte
//   swizzled MN-major layout, from X rows prefetched into registers while the
//   previous head computes. The epilogue (two threads per row n) writes the
//   memory, its inverse RMS r (App. B.1) and, for bf16 memories, an fp32 copy
//   for the state passing (fp32 memories are read by it directly).
// chunk_output_tc_kernel, one CTA (512 threads) per (128-token tile, chunk, head group, b):
//   scores = C_tile B_src^T                  (once, shared by the heads: G = 1)
//   W_h[t,s] = scores[t,s] exp(cum_t - cum_s) dt_s  for s <= t, else 0
//   Y_t = W_h X_h + exp(cum_t) C_t H_[c-1]   (App. A intra + inter terms)
//   W_h is scaled per row by 1 / (|C_t| max_s |B_s| dt_s), a bound on
//   max_s |W_h[t,s]| (the decay is at most 1), and stored fp16 in TMEM as the
//   A operand (fp16 keeps 11 bits; the row scale keeps small decayed weights
//   out of the subnormal range, and the bound needs no pass over the row);
//   H_[c-1] arrives split bf16 hi + lo, already swizzled by the state passing
//   (one 32 KiB bulk copy per head, double-buffered). A CPU emulation against the oracle gives
//   max|err|/RMS(Y) = 2.1e-3 with the exact row maximum as the scale (5.4e-3
//   without a row scale, 4.2e-2 with plain bf16).
//   With S = 64 the tile holds one chunk: rows 64 .. 127 are idle (zero C rows,
//   nothing stored) and the 64 sources are two groups of 32 per row.
// TMEM of the output kernel: scores [0, 256), W [256, 384), intra accumulator
// [384, 448), inter accumulator [448, 512).
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

__device__ int g_scan_tc_status;  // first timeout code since the last read (0 = none)

constexpr int kP = 64;
constexpr int kN = 128;
constexpr int kT = 128;  // tokens per output tile
// The tensor-core scan's backward wants H and H / G to be multiples of 8, its
// forward multiples of kStateHeads (4, the chunk-state kernel's heads per CTA).
// The output kernel takes a runtime number of heads per CTA (a divisor of H / G,
// at most kMaxOutHeads) chosen on the host so that its CTAs fill the SMs in few
// waves.
constexpr int kHeadsPerCta = 8;
constexpr int kMaxOutHeads = 16;
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
// Packed fp32 pairs (low half first) for the two-wide FMUL.
__device__ __forceinline__ uint64_t f2_pack(float x, float y) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(x), "f"(y));
    return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t v, float& x, float& y) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(x), "=f"(y) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_mul(uint64_t a, uint64_t b) {
    uint64_t d;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ uint32_t pack_f16(float a, float b) {
    const __half2 v = __floats2half2_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&v);
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

// The x16 load without the wait, so that several can be in flight; the caller
// issues tcgen05.wait::ld before reading any of the registers.
__device__ __forceinline__ void tmem_ld16_nowait(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
}
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

[[maybe_unused]] __device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
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

// D[tmem] (+)= A[smem] * B[smem]
__device__ __forceinline__ void mma_f16_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                           uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
        ::"r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Commit the MMAs issued by thread 0 and wait (all threads) for them; on a
// timeout set the status and return false (the caller stops; the final drain
// waits for the MMAs in flight with the long bound).
__device__ __forceinline__ bool commit_and_wait(uint64_t* bar, uint32_t parity,
                                                unsigned long long limit_ns, int code,
                                                bool pre_ok = true) {
    if (threadIdx.x == 0) tc::mma_commit(bar);
    const bool ok = tc::mbar_wait(bar, parity, limit_ns, nullptr) && pre_ok;
    if (!ok) atomicCAS(&g_scan_tc_status, 0, code);
    const bool all_ok = __syncthreads_and(ok ? 1 : 0) != 0;
    tc::tc_fence_after();
    return all_ok;
}

// ------------------------------------------------------------ chunk state
constexpr int kStateThreads = 256;  // two threads per chunk row s and per memory row n
// Heads per CTA of the chunk-state kernel (B^T in TMEM is shared by them): four,
// so that batches of many chunks fill the SMs in more, shorter waves.
constexpr int kStateHeads = 4;

struct StateSmem {
    union {
        uint8_t wx[2][256 * 128];        // (w (.) X) hi | lo: S rows x 128 bytes, swizzled
        __nv_bfloat16 b_rows[256 * kN];  // the chunk's B rows (only while building A)
    };
    float w[256];
    float ssq[2][kN];  // sum of squares of each half of each memory row
    float smax[8];     // per warp: max |M| of its rows and half (SMA tiles)
    uint8_t s_res[kP][kN + 16];  // SMA tiles: e4m3 residual rows p, bytes n
    uint64_t bar;
    uint32_t tmem_base;
};

// Next head's inputs, loaded into registers while the current head computes.
struct StateRegs {
    uint4 xv[8];           // X pieces i = tid + 256 k: row i / 8, 16-byte piece i % 8
    float cumv, cend, dtv;  // cum of source tid and of the chunk's last token, dt of tid
};

// kZ: the backward's inter-chunk term Z_c = sum_{t in c} exp(cum_t) C_t^T dY_t
// with the same kernel: Bm <- C, X <- dY, w_t = exp(cum_t), only the fp32 output.
template <typename Tmem, bool kZ = false>
__global__ void __launch_bounds__(kStateThreads, 2)
chunk_state_tc_kernel(const __nv_bfloat16* __restrict__ X, const float* __restrict__ dt,
                      const float* __restrict__ cum, const __nv_bfloat16* __restrict__ Bm,
                      float* __restrict__ dH32, Tmem* __restrict__ Mout, float* __restrict__ rM,
                      int L, int H, int G, int S, int Mc, float eps,
                      unsigned long long wait_limit_ns, uint8_t* __restrict__ tiles,
                      float* __restrict__ tile_scale) {
    extern __shared__ uint8_t smem_raw[];
    StateSmem& sm = *reinterpret_cast<StateSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                  ~(uintptr_t)1023);
    const int c = blockIdx.x, hg = blockIdx.y, b = blockIdx.z;
    const int tid = threadIdx.x, warp = tid >> 5;
    const int n = tid & (kN - 1), half = tid >> 7;  // memory row (TMEM lane) and column half
    const int h0 = hg * kStateHeads;
    const int g = h0 / (H / G);
    const i64 tok0 = (i64)b * L + (i64)c * S;
    const uint32_t lane_addr = (uint32_t)(32 * (warp & 3)) << 16;

    if (tid == 0) {
        tc::mbar_init(&sm.bar, 1);
        tc::fence_barrier_init();
    }
    if (warp == 0) {
        tc::tmem_alloc(&sm.tmem_base, 256);
        tc::tmem_relinquish();
    }
    // register prefetch of a head's sources
    const int xiters = S * 8 / kStateThreads;  // 4 or 8 pieces of 16 bytes
    StateRegs nx;
    auto load_head = [&](int h) {
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            if (k < xiters) {
                const int i = tid + k * kStateThreads, s = i / 8, q = i % 8;
                nx.xv[k] = reinterpret_cast<const uint4*>(X + ((tok0 + s) * H + h) * kP)[q];
            }
        }
        if (tid < S) {
            const float* cumc = cum + (((i64)b * H + h) * Mc + c) * S;
            nx.cumv = cumc[tid];
            nx.cend = cumc[S - 1];
            nx.dtv = dt[(tok0 + tid) * H + h];
        }
    };
    load_head(h0);
    // the chunk's B rows into shared memory (16-byte loads)
    {
        uint4* dst = reinterpret_cast<uint4*>(sm.b_rows);
        const int per_row = kN * 2 / 16;  // 16
        for (int i = tid; i < S * per_row; i += kStateThreads) {
            const int s = i / per_row, q = i % per_row;
            dst[i] = reinterpret_cast<const uint4*>(Bm + ((tok0 + s) * G + g) * kN)[q];
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = sm.tmem_base;
    // A = B^T into TMEM: lane n, columns s / 2 (bf16 pairs); each half of the threads
    // writes half of the columns
    {
        const int cw = S / 4;  // 64 or 32 columns per half
        for (int c0 = half * cw; c0 < (half + 1) * cw; c0 += 16) {
            uint32_t r[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const int s = 2 * (c0 + i);
                __nv_bfloat162 p;
                p.x = sm.b_rows[s * kN + n];
                p.y = sm.b_rows[(s + 1) * kN + n];
                r[i] = *reinterpret_cast<const uint32_t*>(&p);
            }
            tc::tmem_st16(tmem + lane_addr + (uint32_t)c0, r);
        }
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
    }
    __syncthreads();  // b_rows is overwritten by the staging buffers below
    // two accumulators after the A operand (64 columns each): head hh's MMAs run into
    // buffer hh & 1 while the epilogue of head hh - 1 reads the other
    const uint32_t d_col = (uint32_t)(S / 2);
    constexpr uint32_t idesc = tc::idesc_f16(1, true, kN, kP);
    uint32_t phase = 0;
    bool ok = true;
    // epilogue of head hh from its accumulator: row n of the memory, columns 32 half ..
    // 32 half + 31
    // With `tiles`, the epilogue also writes the SMA forward's operands of the memory
    // (the layout of sma_operands_kernel, the same arithmetic): W16 = fp16(r M), the
    // e4m3 residual of 2^12 (W - W16) transposed through shared memory, M16 =
    // fp16(M / max|M|) and the scale max|M|. The last memory has no later token to read it.
    const bool tiled = !kZ && tiles != nullptr && c < Mc - 1;
    auto epilogue = [&](int hh) {
        const int h = h0 + hh;
        const i64 mrow = ((((i64)b * Mc + c) * H + h) * kN + n);
        float ss = 0.0f, am = 0.0f;
        float v[32];
        tmem_ld32(tmem + lane_addr + d_col + 64u * (uint32_t)(hh & 1) + 32u * half, v);
        if (dH32 != nullptr) {
            float4* d32 = reinterpret_cast<float4*>(dH32 + mrow * kP + 32 * half);
#pragma unroll
            for (int q = 0; q < 8; ++q)
                d32[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        }
        if (!kZ) {
            store_row32(Mout + mrow * kP + 32 * half, v);
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                v[i] = stored_value<Tmem>(v[i]);  // the memory as stored (bf16-rounded for bf16 memories)
                ss = fmaf(v[i], v[i], ss);
                am = fmaxf(am, fabsf(v[i]));
            }
        }
        sm.ssq[half][n] = ss;
        if (tiled) {
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, o));
            if ((tid & 31) == 0) sm.smax[warp] = am;
        }
        tc::tc_fence_before();
        __syncthreads();  // ssq, smax; the accumulator is free for head hh + 2
        const float r = rsqrtf((sm.ssq[0][n] + sm.ssq[1][n]) / (float)kP + eps);
        if (!kZ && half == 0 && rM != nullptr) rM[mrow] = r;
        if (tiled) {
            float smx = 0.0f;
#pragma unroll
            for (int w = 0; w < 8; ++w) smx = fmaxf(smx, sm.smax[w]);
            const float inv_s = smx > 0.0f ? 1.0f / smx : 1.0f;
            const int x = h & 1;
            uint8_t* job = tiles + (((i64)b * Mc + c) * (H / 2) + h / 2) * (i64)kSmaJob;
            if (tid == 0) tile_scale[((i64)b * Mc + c) * H + h] = smx > 0.0f ? smx : 1.0f;
            // row n, columns p = 32 half .. 32 half + 31: four 16-byte chunks of 8 fp16
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                uint32_t wq[4], mq[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int i = 8 * q + 2 * e;
                    const float w0 = r * v[i], w1 = r * v[i + 1];
                    const __half h0w = __float2half_rn(w0), h1w = __float2half_rn(w1);
                    // |W| <= sqrt(P) (r normalises the row): W16 needs no scale, and 2^12 times
                    // the residual (at most 2^-11 |W|) stays inside e4m3's range
                    const __nv_fp8_e4m3 r0(4096.0f * (w0 - __half2float(h0w)));
                    const __nv_fp8_e4m3 r1(4096.0f * (w1 - __half2float(h1w)));
                    sm.s_res[32 * half + i][n] = r0.__x;
                    sm.s_res[32 * half + i + 1][n] = r1.__x;
                    wq[e] = (uint32_t)__half_as_ushort(h0w) | ((uint32_t)__half_as_ushort(h1w) << 16);
                    const __half m0 = __float2half_rn(v[i] * inv_s), m1 = __float2half_rn(v[i + 1] * inv_s);
                    mq[e] = (uint32_t)__half_as_ushort(m0) | ((uint32_t)__half_as_ushort(m1) << 16);
                }
                const uint32_t o = sw128((uint32_t)n, (uint32_t)(64 * half + 16 * q));
                *reinterpret_cast<uint4*>(job + x * kSmaTile + o) = make_uint4(wq[0], wq[1], wq[2], wq[3]);
                *reinterpret_cast<uint4*>(job + kSmaOffV + x * kSmaTile + o) = make_uint4(mq[0], mq[1], mq[2], mq[3]);
            }
            __syncthreads();  // the residual rows are complete
            // rows x 64 + p, 128 bytes each, in the 128-byte swizzle: 512 chunks of 16 bytes
#pragma unroll
            for (int k2 = 0; k2 < 2; ++k2) {
                const int ci = tid + kStateThreads * k2, p = ci >> 3, q = ci & 7;
                const uint32_t row = (uint32_t)(x * kP + p);
                *reinterpret_cast<uint4*>(job + kSmaOffLo + row * 128u + (((uint32_t)q ^ (row & 7u)) << 4)) =
                    *reinterpret_cast<const uint4*>(&sm.s_res[p][q * 16]);
            }
        }
    };
    for (int hh = 0; hh < kStateHeads && ok; ++hh) {
        const int h = h0 + hh;
        if (tid < S) sm.w[tid] = kZ ? expf(nx.cumv) : expf(nx.cend - nx.cumv) * nx.dtv;
        __syncthreads();  // also: ssq of head hh - 2 read
        // stage (w (.) X_h) as bf16 hi / lo, rows s, 128-byte swizzle (the MMAs of head
        // hh - 1, the last to read these buffers, were waited for)
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            if (k < xiters) {
                const int i = tid + k * kStateThreads, s = i / 8, q = i % 8;
                const float ws = sm.w[s];
                const uint32_t xw[4] = {nx.xv[k].x, nx.xv[k].y, nx.xv[k].z, nx.xv[k].w};
                uint32_t hi[4], lo[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&xw[e]));
                    const float a0 = ws * f.x, a1 = ws * f.y;
                    const __nv_bfloat162 hv = __floats2bfloat162_rn(a0, a1);
                    const float2 hf = __bfloat1622float2(hv);
                    hi[e] = *reinterpret_cast<const uint32_t*>(&hv);
                    lo[e] = pack_bf16(a0 - hf.x, a1 - hf.y);
                }
                const uint32_t o = sw128((uint32_t)s, (uint32_t)q * 16u);
                *reinterpret_cast<uint4*>(sm.wx[0] + o) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                *reinterpret_cast<uint4*>(sm.wx[1] + o) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
            }
        }
        if (hh + 1 < kStateHeads) load_head(h + 1);  // lands while this head computes
        tc::fence_proxy_async_shared();
        tc::tc_fence_before();
        __syncthreads();
        if (tid == 0) {
            tc::tc_fence_after();
            const uint32_t dcur = tmem + d_col + 64u * (uint32_t)(hh & 1);
            for (int part = 0; part < 2; ++part) {
                const uint32_t base = tc::smem_u32(sm.wx[part]);
                for (int ks = 0; ks < S / 16; ++ks) {
                    const uint64_t bd = tc::smem_desc_sw128(base + 2048u * ks, 1024u, 1024u);
                    tc::mma_f16_ts(dcur, tmem + 8u * ks, bd, idesc, (part > 0 || ks > 0) ? 1u : 0u);
                }
            }
            tc::mma_commit(&sm.bar);
        }
        if (hh > 0) epilogue(hh - 1);  // under this head's MMAs
        // this head's MMAs done: its accumulator is complete and the staging buffers free
        {
            const bool got = tc::mbar_wait(&sm.bar, phase, wait_limit_ns, nullptr);
            if (!got) atomicCAS(&g_scan_tc_status, 0, 1);
            ok = __syncthreads_and(got ? 1 : 0) != 0;
            tc::tc_fence_after();
        }
        phase ^= 1u;
    }
    if (ok) epilogue(kStateHeads - 1);
    if (!ok) {  // a wait ran out: let the MMAs in flight finish before freeing TMEM
        if (!tc::mbar_wait(&sm.bar, phase ^ 1u, kDrainLimitNs, nullptr))
            atomicCAS(&g_scan_tc_status, 0, 9);
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        __syncwarp();
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, 256);
    }
}

// ----------------------------------------------------------- state passing
// H_[c] = exp(cum_end_c) H_[c-1] + dH_c over the chunks (App. A), written as the
// output kernel's operand tiles: for each (b, c, h) the state entering chunk c
// as bf16 hi | lo, 128-byte swizzled, 32 KiB. One CTA per (1024-element slab
// of the N x P state, h, b); the slabs of successive chunks stream through a
// ring of shared-memory stages filled by 4 KiB bulk copies, so the loads stay
// in flight independently of the per-thread recurrence.
constexpr int kSpThreads = 256;
constexpr int kSpElems = 4;                     // consecutive (n, p) elements per thread
constexpr int kSpSlab = kSpThreads * kSpElems;  // 1024 elements, 4 KiB per chunk
constexpr int kSpStages = 8;
constexpr int kSpDec = 1024;                    // chunk decays staged per block of chunks

struct SpSmem {
    float slab[kSpStages][kSpSlab];
    float dec[kSpDec];
    uint64_t full[kSpStages];
};

__global__ void __launch_bounds__(kSpThreads)
state_passing_tc_kernel(const float* dH, const float* __restrict__ cum,
                        float* __restrict__ final_state, uint8_t* __restrict__ Hops,
                        float* Hout, int H, int M, int S,  // Hout may be dH (in place)
                        unsigned long long wait_limit_ns, int withhold) {
    __shared__ __align__(128) SpSmem sm;
    constexpr int NP = kN * kP;
    const int slab = blockIdx.x, h = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
    const int e0 = slab * kSpSlab + tid * kSpElems;  // this thread's first element (n, p)
    const int n = e0 / kP, p = e0 % kP;
    const i64 cstride = (i64)H * NP;  // floats between the chunk slots of one (b, h)
    const float* src = dH + ((i64)b * M * H + h) * NP + (i64)slab * kSpSlab;
    uint8_t* hop = Hops == nullptr ? nullptr : Hops + ((i64)b * M * H + h) * 32768 + sw128((uint32_t)n, (uint32_t)p * 2u);
    const i64 hstride = (i64)H * 32768;
    const float* cumh = cum + ((i64)b * H + h) * (i64)M * S;

    if (tid == 0) {
        for (int k = 0; k < kSpStages; ++k) tc::mbar_init(&sm.full[k], 1);
        tc::fence_barrier_init();
    }
    __syncthreads();
    int issued = 0;  // chunks whose copy thread 0 has issued
    auto issue = [&](int c) {
        const int stg = c % kSpStages;
        tc::mbar_arrive_expect_tx(&sm.full[stg], (uint32_t)(kSpSlab * 4));
        tc::bulk_g2s(sm.slab[stg], src + (i64)c * cstride, (uint32_t)(kSpSlab * 4), &sm.full[stg]);
        ++issued;
    };
    // (withhold: the failure-path test hook; every wait on the slabs then runs out)
    if (tid == 0 && !withhold)
        for (int c = 0; c < min(kSpStages, M); ++c) issue(c);
    float st[kSpElems] = {0.0f, 0.0f, 0.0f, 0.0f};
    bool ok = true;
    int c = 0;
    for (; c < M; ++c) {
        if (c % kSpDec == 0) {
            for (int i = tid; i < min(kSpDec, M - c); i += kSpThreads)
                sm.dec[i] = expf(cumh[(i64)(c + i) * S + S - 1]);
            __syncthreads();
        }
        const int stg = c % kSpStages;
        const bool got = tc::mbar_wait(&sm.full[stg], (uint32_t)((c / kSpStages) & 1), wait_limit_ns, nullptr);
        if (got) {
            const float4 d = *reinterpret_cast<const float4*>(&sm.slab[stg][tid * kSpElems]);
            // the state entering chunk c, as the split operand
            uint32_t hi[2], lo[2];
#pragma unroll
            for (int k = 0; k < 2; ++k) {
                const __nv_bfloat162 hv = __floats2bfloat162_rn(st[2 * k], st[2 * k + 1]);
                const float2 hf = __bfloat1622float2(hv);
                hi[k] = *reinterpret_cast<const uint32_t*>(&hv);
                lo[k] = pack_bf16(st[2 * k] - hf.x, st[2 * k + 1] - hf.y);
            }
            if (hop != nullptr) {
                uint8_t* t = hop + (i64)c * hstride;
                *reinterpret_cast<uint2*>(t) = make_uint2(hi[0], hi[1]);
                *reinterpret_cast<uint2*>(t + 16384) = make_uint2(lo[0], lo[1]);
            }
            if (Hout != nullptr)  // also fp32 (may be dH itself: chunk c's slab is already read)
                *reinterpret_cast<float4*>(Hout + ((i64)b * M * H + h) * NP + (i64)slab * kSpSlab +
                                           (i64)c * cstride + tid * kSpElems) =
                    make_float4(st[0], st[1], st[2], st[3]);
            const float a = sm.dec[c % kSpDec];
            st[0] = fmaf(a, st[0], d.x);
            st[1] = fmaf(a, st[1], d.y);
            st[2] = fmaf(a, st[2], d.z);
            st[3] = fmaf(a, st[3], d.w);
        } else {
            atomicCAS(&g_scan_tc_status, 0, 13);
        }
        // every thread has read the stage (and the decays) before it is refilled
        ok = __syncthreads_and(got ? 1 : 0) != 0;
        if (!ok) break;
        if (tid == 0 && !withhold && c + kSpStages < M) issue(c + kSpStages);
    }
    if (!ok && tid == 0) {  // let the copies in flight land before the CTA exits
        for (int k = c; k < issued; ++k)
            if (!tc::mbar_wait(&sm.full[k % kSpStages], (uint32_t)((k / kSpStages) & 1), kDrainLimitNs, nullptr)) {
                atomicCAS(&g_scan_tc_status, 0, 14);
                break;
            }
    }
    if (ok && final_state != nullptr)
        *reinterpret_cast<float4*>(final_state + ((i64)b * H + h) * NP + e0) =
            make_float4(st[0], st[1], st[2], st[3]);
}

// ----------------------------------------------------------- chunk output
struct OutSmem {
    uint8_t c_tile[2][kT * 128];   // C of the tile, K-major, two 64-wide K blocks
    uint8_t b_src[2][256 * 128];   // B of the sources, K-major (rows s), two K blocks
    uint8_t x_src[256 * 128];      // X_h of the sources as fp16, MN-major (rows s)
    uint8_t h_prev[2][kN * 128];   // H_[c-1] of a head, bf16 hi | lo, MN-major (rows n); the
                                   // second buffer of the pair is b_src, free after the scores
    float c2[256];                 // cum * log2(e) of the sources
    float e2[256];                 // c2 - log2(dt): exp2(c2_t - e2_s) = exp(cum_t - cum_s) dt_s
    float bfac[256];               // exp2(c2_r - e2_s), r = last source of s's group of 32
    float bnorm[256];              // |B_s| of the sources
    float cnorm[kT];               // |C_t| of the tile's rows
    uint32_t bdmax[2];             // max_s |B_s| dt_s of a head (float bits), by head parity
    float dacc[kMaxOutHeads][kT][2];  // backward modes: per (head, row) dot product
    uint64_t bar;
    uint64_t hbar[2];              // H_[c-1] tile copy into buffer 0 / 1 landed
    uint32_t tmem_base;
};

constexpr int kOutThreads = 512;  // four threads per token row

// Modes of the output kernel. kOutY: the forward, Y. kOutDot: for the
// backward, only the inter-chunk part of the forward (no intra work), writing
// dY_t . exp(cum_t) C_t H_[c-1] per (t, h). kOutRev: the backward's dX as the
// same computation in reversed time inside each chunk (target s, sources
// t >= s; C <- B, B <- C, X <- dY, dt <- 1, cum' = cum_end - cum,
// H_[c-1] <- d(dH_c)):
//   Y'_s = sum_{t >= s} e^{cum_t - cum_s} (B_s . C_t) dY_t + e^{cum_end - cum_s} B_s d(dH_c),
// writing dX_s = dt_s Y'_s and per (s, h) X_s . (its inter-chunk part).
constexpr int kOutY = 0, kOutDot = 1, kOutRev = 2;

__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Next head's inputs, loaded into registers while the current head computes.
struct HeadRegs {
    uint4 xv[4];    // X rows of the sources (bf16), 16-byte pieces i = tid + 512 k
    float c2, dtv;  // source tid (tid < ns)
};

template <typename Tout, int kMode = kOutY>
__global__ void __launch_bounds__(kOutThreads, 1)
chunk_output_tc_kernel(const __nv_bfloat16* __restrict__ X, const float* __restrict__ dt,
                       const float* __restrict__ cum, const __nv_bfloat16* __restrict__ Bm,
                       const __nv_bfloat16* __restrict__ Cm, const uint8_t* __restrict__ Hops,
                       Tout* __restrict__ Y, int L, int H, int G, int S, int Mc, int hpc,
                       unsigned long long wait_limit_ns,
                       const __nv_bfloat16* __restrict__ Zd = nullptr, float* __restrict__ dots = nullptr) {
    extern __shared__ uint8_t smem_raw[];
    OutSmem& sm = *reinterpret_cast<OutSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                              ~(uintptr_t)1023);
    // the SMA kernel that follows may take the SMs this grid's last wave leaves idle: it
    // reads nothing this kernel writes before its own griddep_wait
    griddep_launch_dependents();
    const int tt = blockIdx.x;  // tile inside the chunk
    const int c = blockIdx.y / (H / hpc);
    const int hg = blockIdx.y % (H / hpc);
    const int b = blockIdx.z;
    const int tid = threadIdx.x, warp = tid >> 5;
    const int row = tid & (kT - 1), quarter = tid >> 7;  // token row, quarter of the sources / columns
    const int h0 = hg * hpc;
    const int g = h0 / (H / G);
    // sources 0 .. ns-1 of the chunk; with S = 64 the 128-row tile holds one chunk and
    // its rows S .. 127 are idle (zero C rows, nothing stored)
    const int ns = min((tt + 1) * kT, S);
    const i64 tok0 = (i64)b * L + (i64)c * S;
    const uint32_t lane_addr = (uint32_t)(32 * (warp & 3)) << 16;
    const bool has_prev = kMode == kOutRev || c > 0;
    constexpr uint32_t kColSc = 0, kColW = 256, kColIn = 384, kColEx = 448;
    // chunk position of the kernel's token k (reversed inside the chunk for kOutRev)
    auto pos = [&](int k) { return kMode == kOutRev ? S - 1 - k : k; };
    constexpr bool kIntra = kMode != kOutDot;
    if (kMode != kOutY)
        for (int i = tid; i < hpc * kT * 2; i += kOutThreads) (&sm.dacc[0][0][0])[i] = 0.0f;

    if (tid == 0) {
        tc::mbar_init(&sm.bar, 1);
        tc::mbar_init(&sm.hbar[0], 1);
        tc::mbar_init(&sm.hbar[1], 1);
        tc::fence_barrier_init();
    }
    if (warp == 0) {
        tc::tmem_alloc(&sm.tmem_base, 512);
        tc::tmem_relinquish();
    }
    // H_[c-1] tiles (bf16 hi | lo, 32 KiB per head, written swizzled by the state passing):
    // head hh's copy goes to buffer hh & 1; only thread 0 issues, waits and drains them
    auto hbuf = [&](int bi) -> uint8_t* { return bi ? sm.b_src[0] : sm.h_prev[0]; };
    int hissued = 0;  // copies issued (thread 0)
    auto issue_h = [&](int hh) {
        const int bi = hh & 1;
        const uint8_t* src = Hops + (((i64)b * Mc + c) * H + h0 + hh) * 32768;
        tc::mbar_arrive_expect_tx(&sm.hbar[bi], 32768u);
        tc::bulk_g2s(hbuf(bi), src, 32768u, &sm.hbar[bi]);
        ++hissued;
    };
    __syncthreads();  // barriers initialised before any copy
    if (tid == 0 && has_prev) issue_h(0);
    // C of the tile and B of the sources, K-major (row t or s, two K blocks of 64, 16-byte
    // chunks, swizzled). Every load of a thread is issued before any store; the 16 lanes
    // of a half-warp hold one row, and their squares give its norm for the W scale bound
    // (|C_t|, |B_s|) without a second pass over the rows.
    constexpr int kCIt = kT * 16 / kOutThreads;    // 4 pieces of C per thread
    constexpr int kBItMax = 256 * 16 / kOutThreads;  // up to 8 pieces of B
    const int bit = kIntra ? ns * 16 / kOutThreads : 0;  // 2, 4 or 8 (ns = 64, 128, 256)
    auto sumsq8 = [](const uint4 v) {
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
        float ss = 0.0f;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[e]));
            ss = fmaf(f.x, f.x, fmaf(f.y, f.y, ss));
        }
        return ss;
    };
    auto half_sum = [](float ss) {  // over the 16 lanes of a half-warp
#pragma unroll
        for (int o = 8; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        return ss;
    };
    {
        uint4 cv[kCIt], bv[kBItMax];
#pragma unroll
        for (int k = 0; k < kCIt; ++k) {
            const int i = tid + k * kOutThreads, t = i / 16, q = i % 16;
            cv[k] = tt * kT + t < S ? reinterpret_cast<const uint4*>(Cm + ((tok0 + pos(tt * kT + t)) * G + g) * kN)[q]
                                    : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int k = 0; k < kBItMax; ++k) {
            if (k < bit) {
                const int i = tid + k * kOutThreads, sidx = i / 16, q = i % 16;
                bv[k] = reinterpret_cast<const uint4*>(Bm + ((tok0 + pos(sidx)) * G + g) * kN)[q];
            }
        }
#pragma unroll
        for (int k = 0; k < kCIt; ++k) {
            const int i = tid + k * kOutThreads, t = i / 16, q = i % 16;
            *reinterpret_cast<uint4*>(sm.c_tile[q / 8] + sw128((uint32_t)t, (uint32_t)(q % 8) * 16u)) = cv[k];
            const float ss = half_sum(sumsq8(cv[k]));
            if (q == 0) sm.cnorm[t] = sqrtf(ss);
        }
#pragma unroll
        for (int k = 0; k < kBItMax; ++k) {
            if (k < bit) {  // uniform over the block
                const int i = tid + k * kOutThreads, sidx = i / 16, q = i % 16;
                *reinterpret_cast<uint4*>(sm.b_src[q / 8] + sw128((uint32_t)sidx, (uint32_t)(q % 8) * 16u)) = bv[k];
                const float ss = half_sum(sumsq8(bv[k]));
                if (q == 0) sm.bnorm[sidx] = sqrtf(ss);
            }
        }
    }
    if (tid < 2) sm.bdmax[tid] = 0u;
    tc::fence_proxy_async_shared();
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = sm.tmem_base;
    uint32_t phase = 0;
    // scores = C_tile B_src^T (M 128, N ns, K 128), shared by the CTA's heads
    if (kIntra && tid == 0) {
        const uint32_t idesc = tc::idesc_f16(1, false, kT, (uint32_t)ns);
        for (int ks = 0; ks < kN / 16; ++ks) {
            const uint64_t ad = tc::smem_desc_sw128(tc::smem_u32(sm.c_tile[ks / 4]) + 32u * (ks % 4), 16u, 1024u);
            const uint64_t bd = tc::smem_desc_sw128(tc::smem_u32(sm.b_src[ks / 4]) + 32u * (ks % 4), 16u, 1024u);
            mma_f16_ss(tmem + kColSc, ad, bd, idesc, ks > 0 ? 1u : 0u);
        }
    }

    // register prefetch of a head's sources (X rows, H_[c-1], cum, dt)
    const int xiters = ns * 8 / kOutThreads;  // 2 or 4 pieces of 16 bytes
    HeadRegs nx;
    auto load_head = [&](int h) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            if (kIntra && k < xiters) {
                const int i = tid + k * kOutThreads, sidx = i / 8, q = i % 8;
                nx.xv[k] = reinterpret_cast<const uint4*>(X + ((tok0 + pos(sidx)) * H + h) * kP)[q];
            }
        }
        if (tid < ns) {
            const float* cumc = cum + (((i64)b * H + h) * Mc + c) * S;
            if (kMode == kOutRev) {  // cum' = cum_end - cum (reversed), dt' = 1
                nx.c2 = (cumc[S - 1] - cumc[pos(tid)]) * kLog2e;
                nx.dtv = 1.0f;
            } else {
                nx.c2 = cumc[tid] * kLog2e;
                nx.dtv = dt[(tok0 + tid) * H + h];
            }
        }
    };
    load_head(h0);
    bool ok = commit_and_wait(&sm.bar, phase, wait_limit_ns, 2);
    phase ^= 1u;

    const int tl = tt * kT + row;  // this thread's token inside the chunk (kernel order)
    const i64 tok = tok0 + pos(tl);
    const int tl_warp_max = tt * kT + 32 * (warp & 3) + 31;
    // this thread's sources: a quarter of them (32 or 64) for ns >= 128, else 32 per
    // thread for the first two quarters (ns = 64) and none for the others
    const int per_q = ns >= 128 ? ns / 4 : 32;
    const int s_lo = quarter * per_q, s_hi = min(s_lo + per_q, ns);
    for (int hh = 0; hh < hpc && ok; ++hh) {
        const int h = h0 + hh;
        // the inter-chunk chain C H_[c-1] needs no W: issued first, it runs under the W pass
        bool hok = true;
        if (tid == 0 && has_prev) {
            tc::tc_fence_after();
            hok = tc::mbar_wait(&sm.hbar[hh & 1], (uint32_t)((hh >> 1) & 1), wait_limit_ns, nullptr);
            if (hok) {
                const uint32_t idb = tc::idesc_f16(1, true, kT, kP);
                for (int part = 0; part < 2; ++part) {
                    for (int ks = 0; ks < kN / 16; ++ks) {
                        const uint64_t ad = tc::smem_desc_sw128(
                            tc::smem_u32(sm.c_tile[ks / 4]) + 32u * (ks % 4), 16u, 1024u);
                        const uint64_t bd = tc::smem_desc_sw128(
                            tc::smem_u32(hbuf(hh & 1) + 16384 * part) + 2048u * ks, 1024u, 1024u);
                        mma_f16_ss(tmem + kColEx, ad, bd, idb, (part > 0 || ks > 0) ? 1u : 0u);
                    }
                }
            } else {
                atomicCAS(&g_scan_tc_status, 0, 11);
            }
        }
        // prefetched sources into shared memory (the previous head's MMAs are done)
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            if (kIntra && k < xiters) {
                const int i = tid + k * kOutThreads, sidx = i / 8, q = i % 8;
                const uint32_t xw[4] = {nx.xv[k].x, nx.xv[k].y, nx.xv[k].z, nx.xv[k].w};
                uint32_t f[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float2 v = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&xw[e]));
                    f[e] = pack_f16(v.x, v.y);
                }
                *reinterpret_cast<uint4*>(sm.x_src + sw128((uint32_t)sidx, (uint32_t)q * 16u)) =
                    make_uint4(f[0], f[1], f[2], f[3]);
            }
        }
        if (tid < ns) {
            sm.c2[tid] = nx.c2;
            sm.e2[tid] = nx.c2 - log2f(nx.dtv);  // dt = 0 gives +inf: a zero weight
            // non-negative floats order like their bit patterns
            atomicMax(&sm.bdmax[hh & 1], __float_as_uint(sm.bnorm[tid] * fabsf(nx.dtv)));
        }
        if (tid == 0) sm.bdmax[(hh + 1) & 1] = 0u;  // last read by head hh - 1's W pass
        __syncthreads();
        // exp(cum_t - cum_s) dt_s = exp2(c2_t - c2_r) exp2(c2_r - e2_s) for the group of 32
        // sources ending at r; both factors are at most 1 (cum never rises) when r <= t
        if (tid < ns) sm.bfac[tid] = ex2_approx(sm.c2[tid | 31] - sm.e2[tid]);
        __syncthreads();
        if (hh + 1 < hpc) {  // lands while this head computes
            load_head(h + 1);
            // buffer (hh + 1) & 1 was last read by head hh - 1's MMAs (or the scores), both
            // done: their commit was waited for before head hh began
            if (tid == 0 && has_prev) issue_h(hh + 1);
        }

        // W row of this thread over its quarter of the sources, scaled by the bound
        // 1 / (|C_t| max_s |B_s| dt_s) and stored fp16 in one pass
        const float c2t = sm.c2[min(tl, ns - 1)];  // an idle row (tl >= S) reads a live entry
        const float bound = sm.cnorm[row] * __uint_as_float(sm.bdmax[hh & 1]);
        const float wmax = bound > 0.0f ? bound : 1.0f;  // undone on the intra accumulator
        const float rscale = 1.0f / wmax;
        auto w_group = [&](int s0, const float (&v)[32], bool live) {
            uint32_t pk[16];
            if (!live) {  // every row of the warp is before these sources
#pragma unroll
                for (int i = 0; i < 16; ++i) pk[i] = 0u;
            } else if (s0 + 31 <= tl) {  // the whole group is at or before t: factored decay
                const float a = ex2_approx(c2t - sm.c2[s0 + 31]) * rscale;
                const uint64_t a2 = f2_pack(a, a);
#pragma unroll
                for (int i = 0; i < 16; ++i) {  // packed pairs: (v bfac) a
                    const uint64_t bf = *reinterpret_cast<const uint64_t*>(&sm.bfac[s0 + 2 * i]);
                    float w0, w1;
                    f2_unpack(f2_mul(f2_mul(f2_pack(v[2 * i], v[2 * i + 1]), bf), a2), w0, w1);
                    pk[i] = pack_f16(w0, w1);
                }
            } else {  // the group holding t: masked, one exp per element
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const int sidx = s0 + 2 * i;
                    const float w0 = sidx <= tl ? v[2 * i] * ex2_approx(c2t - sm.e2[sidx]) : 0.0f;
                    const float w1 = sidx + 1 <= tl ? v[2 * i + 1] * ex2_approx(c2t - sm.e2[sidx + 1]) : 0.0f;
                    pk[i] = pack_f16(w0 * rscale, w1 * rscale);
                }
            }
            tc::tmem_st16(tmem + lane_addr + kColW + (uint32_t)(s0 / 2), pk);
        };
        for (int s0 = s_lo; kIntra && s0 < s_hi; s0 += 32) {  // s_hi - s_lo is 0, 32 or 64
            const bool live = s0 <= tl_warp_max;
            float v[32];
            if (live) tmem_ld32(tmem + lane_addr + kColSc + (uint32_t)s0, v);
            w_group(s0, v, live);
        }
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
        tc::fence_proxy_async_shared();
        tc::tc_fence_before();
        __syncthreads();
        if (tid == 0) {
            tc::tc_fence_after();
            const uint32_t id16 = tc::idesc_f16(0, true, kT, kP);
            for (int ks = 0; kIntra && ks < ns / 16; ++ks) {
                const uint64_t bd = tc::smem_desc_sw128(tc::smem_u32(sm.x_src) + 2048u * ks, 1024u, 1024u);
                tc::mma_f16_ts(tmem + kColIn, tmem + kColW + 8u * ks, bd, id16, ks > 0 ? 1u : 0u);
            }
        }
        // the commit tracks both chains
        ok = commit_and_wait(&sm.bar, phase, wait_limit_ns, 3, hok);
        phase ^= 1u;
        if (!ok) break;
        // Y_t = wmax * (W~ X)_t + exp(cum_t) (C H)_t, columns 16 quarter .. 16 quarter + 15
        {
            const float dec = exp2f(c2t);
            float vi[16], ve[16];
            {
                uint32_t ri[16], re[16];
                if (kIntra) tmem_ld16_nowait(tmem + lane_addr + kColIn + 16u * quarter, ri);
                if (has_prev) tmem_ld16_nowait(tmem + lane_addr + kColEx + 16u * quarter, re);
                if (kIntra || has_prev) tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    vi[i] = kIntra ? __uint_as_float(ri[i]) : 0.0f;
                    ve[i] = has_prev ? __uint_as_float(re[i]) : 0.0f;
                }
            }
            if (kMode == kOutRev) {
                // dX = dt Y', and X . (inter part of Y')
                const float dts = dt[tok * H + h];
                float zv[16];
                load_row16(Zd + (tok * H + h) * kP + 16 * quarter, zv);
                float d2 = 0.0f;
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const float inter = dec * ve[i];
                    vi[i] = fmaf(wmax, vi[i], inter) * dts;
                    d2 = fmaf(zv[i], inter, d2);
                }
                store_row16(Y + (tok * H + h) * kP + 16 * quarter, vi);
                atomicAdd(&sm.dacc[hh][row][0], d2);
            } else {
#pragma unroll
                for (int i = 0; i < 16; ++i) vi[i] = fmaf(wmax, vi[i], dec * ve[i]);
                if (kMode == kOutY) {
                    if (tl < S) store_row16(Y + (tok * H + h) * kP + 16 * quarter, vi);
                } else {  // dY . (inter part of Y); vi holds only that part here
                    float zv[16];
                    load_row16(Zd + (tok * H + h) * kP + 16 * quarter, zv);
                    float d1 = 0.0f;
#pragma unroll
                    for (int i = 0; i < 16; ++i) d1 = fmaf(zv[i], vi[i], d1);
                    atomicAdd(&sm.dacc[hh][row][0], d1);
                }
            }
        }
        tc::tc_fence_before();
        __syncthreads();  // shared staging and TMEM are reused by the next head
    }
    if (!ok) {
        if (!tc::mbar_wait(&sm.bar, phase ^ 1u, kDrainLimitNs, nullptr))
            atomicCAS(&g_scan_tc_status, 0, 10);
    }
    // never leave an H copy in flight behind: wait for the last one into each buffer
    if (tid == 0) {
        for (int k = hissued - 1; k >= 0 && k >= hissued - 2; --k)
            if (!tc::mbar_wait(&sm.hbar[k & 1], (uint32_t)((k >> 1) & 1), kDrainLimitNs, nullptr))
                atomicCAS(&g_scan_tc_status, 0, 12);
    }
    tc::tc_fence_before();
    __syncthreads();
    if (kMode != kOutY && ok) {  // the per (token, head) dots
        for (int i = tid; i < hpc * kT; i += kOutThreads) {
            const int hh = i / kT, r = i % kT;
            const i64 tk = tok0 + pos(tt * kT + r);
            dots[tk * H + h0 + hh] = sm.dacc[hh][r][0];
        }
    }
    if (warp == 0) {
        __syncwarp();
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, 512);
    }
}

}  // namespace

// Heads per CTA of the output kernel: the divisor d of H / G (d <= kMaxOutHeads)
// with the least modelled time, waves x (prologue + d heads). The prologue
// (scores, tile and source staging) costs about two heads' work.
int out_heads_per_cta(int units, int H, int G) {
    int dev = 0, nsm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || nsm <= 0)
        nsm = 1;
    const int hg = H / G;
    int best = kHeadsPerCta;
    long long best_cost = -1;
    for (int d = 1; d <= kMaxOutHeads && d <= hg; ++d) {
        if (hg % d) continue;
        const long long ctas = (long long)units * (H / d);
        const long long cost = (ctas + nsm - 1) / nsm * (2 + d);
        if (best_cost < 0 || cost < best_cost || (cost == best_cost && d > best)) {
            best = d;
            best_cost = cost;
        }
    }
    return best;
}

bool scan_tc_supported(const ScanArgs& a) {
    return a.P == kP && a.N == kN && (a.S == 64 || a.S == 128 || a.S == 256) &&
           a.H % kHeadsPerCta == 0 && (a.H / a.G) % kHeadsPerCta == 0;
}

bool scan_fwd_tc_supported(const ScanArgs& a) {
    return a.P == kP && a.N == kN && (a.S == 64 || a.S == 128 || a.S == 256) &&
           a.H % kStateHeads == 0 && (a.H / a.G) % kStateHeads == 0;
}

template <typename Tmem, typename Tout>
cudaError_t launch_chunk_scan_tc(const ScanArgs& a, unsigned long long wait_limit_ns,
                                 cudaStream_t stream) {
    const int B = (int)a.B, L = (int)a.L, H = (int)a.H, G = (int)a.G, S = (int)a.S, M = L / S;
    constexpr bool mem_is_f32 = std::is_same<Tmem, float>::value;
    if (a.Hops == nullptr) return cudaErrorInvalidValue;  // the output kernel's H_[c-1] tiles
    cudaError_t e0 = launch_chunk_cumsum(a, stream);
    if (e0 != cudaSuccess) return e0;
    {
        auto kern = chunk_state_tc_kernel<Tmem>;
        const size_t smem = sizeof(StateSmem) + 1024;
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        uint8_t* tiles = a.sma_tiles;
        float* tile_scale = tiles != nullptr ? (float*)(tiles + sma_tiles_scale_offset(a.B, M, a.H)) : nullptr;
        kern<<<dim3(M, H / kStateHeads, B), kStateThreads, smem, stream>>>(
            (const __nv_bfloat16*)a.X, a.dt, a.cum, (const __nv_bfloat16*)a.Bm,
            mem_is_f32 ? nullptr : a.dH32, (Tmem*)a.M, a.rM, L, H, G, S, M, a.eps, wait_limit_ns, tiles,
            tile_scale);
    }
    // fp32 memories are the chunk states themselves: the state passing reads them
    state_passing_tc_kernel<<<dim3(kN * kP / kSpSlab, H, B), kSpThreads, 0, stream>>>(
        mem_is_f32 ? (const float*)a.M : a.dH32, a.cum, a.final_state, a.Hops, nullptr, H, M, S,
        wait_limit_ns, a.test_withhold);
    {
        auto kern = chunk_output_tc_kernel<Tout>;
        const size_t smem = sizeof(OutSmem) + 1024;
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        const int tiles = S >= kT ? S / kT : 1;  // S = 64: one tile, half of its rows idle
        const int hpc = out_heads_per_cta(tiles * M * B, H, G);
        kern<<<dim3(tiles, M * (H / hpc), B), kOutThreads, smem, stream>>>(
            (const __nv_bfloat16*)a.X, a.dt, a.cum, (const __nv_bfloat16*)a.Bm,
            (const __nv_bfloat16*)a.Cm, a.Hops, (Tout*)a.Y, L, H, G, S, M, hpc, wait_limit_ns,
            nullptr, nullptr);
    }
    note_launches(3);
    return cudaGetLastError();
}

// Backward helpers on the tensor-core path (bf16 inputs, the same shapes).
// States: cum and the state entering every chunk, fp32 (in Hprev) and as the
// split operand tiles (Hops), i.e. the forward's chunk states followed by the
// state passing.
cudaError_t launch_scan_states_tc(const ScanArgs& a0, float* cum, float* Hprev, uint8_t* Hops,
                                  unsigned long long wait_limit_ns, cudaStream_t stream) {
    ScanArgs a = a0;
    a.cum = cum;
    const int B = (int)a.B, L = (int)a.L, H = (int)a.H, G = (int)a.G, S = (int)a.S, M = L / S;
    cudaError_t e = launch_chunk_cumsum(a, stream);
    if (e != cudaSuccess) return e;
    auto kern = chunk_state_tc_kernel<float, false>;
    const size_t smem = sizeof(StateSmem) + 1024;
    if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) != cudaSuccess)
        return e;
    kern<<<dim3(M, H / kStateHeads, B), kStateThreads, smem, stream>>>(
        (const __nv_bfloat16*)a.X, a.dt, a.cum, (const __nv_bfloat16*)a.Bm, nullptr, Hprev, nullptr,
        L, H, G, S, M, a.eps, wait_limit_ns, nullptr, nullptr);
    state_passing_tc_kernel<<<dim3(kN * kP / kSpSlab, H, B), kSpThreads, 0, stream>>>(
        Hprev, a.cum, nullptr, Hops, Hprev, H, M, S, wait_limit_ns, 0);
    note_launches(2);
    return cudaGetLastError();
}

// Z_c = sum_{t in c} exp(cum_t) C_t^T dY_t for every chunk (fp32, B x Mc x H x N x P).
cudaError_t launch_scan_bwd_inter_tc(const ScanArgs& a, const float* cum, const void* dY, float* Z,
                                     unsigned long long wait_limit_ns, cudaStream_t stream) {
    const int B = (int)a.B, L = (int)a.L, H = (int)a.H, G = (int)a.G, S = (int)a.S, M = L / S;
    auto kern = chunk_state_tc_kernel<float, true>;
    const size_t smem = sizeof(StateSmem) + 1024;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    kern<<<dim3(M, H / kStateHeads, B), kStateThreads, smem, stream>>>(
        (const __nv_bfloat16*)dY, a.dt, cum, (const __nv_bfloat16*)a.Cm, Z, nullptr, nullptr, L, H, G,
        S, M, a.eps, wait_limit_ns, nullptr, nullptr);
    note_launches(1);
    return cudaGetLastError();
}

// The output kernel's backward modes. rowI (B x L x H): dY_t . exp(cum_t) C_t
// H_[c-1], from the forward operand tiles Hops. dX (B x L x H x P, fp32) and
// xi (B x L x H): X_s . exp(cum_end - cum_s) B_s d(dH_c), from the reversed
// computation with Dops (d(dH_c)) as the state operand.
cudaError_t launch_scan_bwd_output_tc(const ScanArgs& a, const float* cum, const uint8_t* Hops,
                                      const uint8_t* Dops, const void* dY, float* rowI,
                                      float* dX, float* xi, unsigned long long wait_limit_ns,
                                      cudaStream_t stream) {
    const int B = (int)a.B, L = (int)a.L, H = (int)a.H, G = (int)a.G, S = (int)a.S, M = L / S;
    typedef __nv_bfloat16 bf;
    const size_t smem = sizeof(OutSmem) + 1024;
    const int hpc = out_heads_per_cta(S / kT * M * B, H, G);
    const dim3 grid(S / kT, M * (H / hpc), B);
    {
        auto kern = chunk_output_tc_kernel<float, kOutDot>;
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        kern<<<grid, kOutThreads, smem, stream>>>((const bf*)a.X, a.dt, cum, (const bf*)a.Bm,
                                                  (const bf*)a.Cm, Hops, nullptr, L, H, G, S, M,
                                                  hpc, wait_limit_ns, (const bf*)dY, rowI);
    }
    {
        auto kern = chunk_output_tc_kernel<float, kOutRev>;
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        // sources X <- dY, B <- C, C <- B; the dots take X
        kern<<<grid, kOutThreads, smem, stream>>>((const bf*)dY, a.dt, cum, (const bf*)a.Cm,
                                                  (const bf*)a.Bm, Dops, dX, L, H, G, S, M,
                                                  hpc, wait_limit_ns, (const bf*)a.X, xi);
    }
    note_launches(2);
    return cudaGetLastError();
}

typedef __nv_bfloat16 bf16;
template cudaError_t launch_chunk_scan_tc<float, float>(const ScanArgs&, unsigned long long, cudaStream_t);
template cudaError_t launch_chunk_scan_tc<bf16, float>(const ScanArgs&, unsigned long long, cudaStream_t);
template cudaError_t launch_chunk_scan_tc<bf16, bf16>(const ScanArgs&, unsigned long long, cudaStream_t);

// Read and clear of the status word in one device-side exchange: a code that a
// kernel still running on another stream records is either returned now or kept
// for the next read, never lost between a read and a separate clear.
__device__ int g_scan_tc_status_taken;
__global__ void take_scan_tc_status_kernel() { g_scan_tc_status_taken = atomicExch(&g_scan_tc_status, 0); }

int take_scan_tc_status(cudaStream_t stream) {
    take_scan_tc_status_kernel<<<1, 1, 0, stream>>>();
    int v = 0;
    if (cudaGetLastError() != cudaSuccess ||
        cudaMemcpyFromSymbolAsync(&v, g_scan_tc_status_taken, sizeof(int), 0, cudaMemcpyDeviceToHost, stream) !=
            cudaSuccess ||
        cudaStreamSynchronize(stream) != cudaSuccess)
        return -1;
    return v;
}

}  // namespace dart
