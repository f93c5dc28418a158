// Internal launch interface between the C ABI (dart_api.cu) and the kernels.
// Not installed; the public interface is include/dart.h.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "dart.h"

namespace dart {

// Validation of dims shared by the entry points (dart_api.cu).
dart_status validate_dims(const dart_dims* d, bool need_seqlen);
// Records e for dart_last_cuda_error() and returns DART_ERR_CUDA.
dart_status record_cuda_error(cudaError_t e);

struct ScanArgs {
    int64_t B, L, H, G, P, N, S;
    float eps;
    const void* X;
    const float* dt;
    const float* A;
    const void* Bm;
    const void* Cm;
    void* Y;
    void* M;
    float* rM;
    float* final_state;
    // workspace
    float* cum;   // B x H x M x S
    float* dH32;  // B x M x H x N x P (fp32 memories, then states entering each chunk)
    // optional (tensor-core path): the states entering each chunk as bf16 hi | lo
    // tiles in the 128-byte-swizzled shared-memory layout, 32 KiB per (b, c, h)
    uint8_t* Hops;
    int test_withhold = 0;  // tensor-core path: the state passing issues no copies (failure-path test hook)
    // optional (tensor-core path): the SMA forward's operand tiles and scales, written by
    // the chunk-state epilogue (layout of sma_tiles_bytes), or null
    uint8_t* sma_tiles = nullptr;
};

struct SmaArgs {
    int64_t B, L, H, G, P, N, S;
    float eps;
    const void* M;
    const float* rM;
    const void* Q;
    const void* Cm;
    const void* E;
    const void* z;
    const void* Yssd;
    void* Y;
    void* R;
    float* lse;
    int test_withhold;  // tensor-core path: issue no operand copies (failure-path test hook)
    float* logits = nullptr;  // tensor-core path: B x H x Mc x L logits for the backward, or null
    // tensor-core path: operand tiles already built (by the chunk-state kernel), or null;
    // M and rM are then not read
    const uint8_t* tiles = nullptr;
};

struct DecodeArgs {
    int64_t B, H, G, P, N, S, pos, m_cap;
    float eps;
    void* cache;
    float* state;
    float* partial;
    const void* x;
    const float* dt;
    const float* A;
    const void* b;
    const void* c;
    const void* q;
    const void* e;
    const void* z;
    void* y;
    float* lse;
};

// Backward of SMA + merge (sma_bwd.cu). Gradients are fp32.
struct SmaBwdArgs {
    int64_t B, L, H, G, P, N, S;
    float eps;
    const void* M;
    const float* rM;  // nullptr: recomputed into the workspace
    const void* Q;
    const void* Cm;
    const void* E;
    const void* z;
    const float* lse;
    const void* dY;
    float* dM;  // B x Mc x H x N x P (overwritten)
    float* dQ;  // B x L x G x N (overwritten)
    float* dC;  // B x L x G x N (overwritten)
    float* dE;  // B x L x G x P (overwritten)
    float* dz;  // B x L x H (overwritten)
    const float* logits = nullptr;  // the forward's logits (B x H x Mc x L) or null: recomputed
    int test_withhold = 0;  // tensor-core path: the row kernels issue no operand copies (test hook)
};

// Backward of the chunked scan (scan_bwd.cu). Gradients are fp32.
struct ScanBwdArgs {
    ScanArgs fwd;      // sizes and the forward inputs X, dt, A, Bm, Cm
    const void* dY;    // gradient w.r.t. Y_ssd, input dtype
    const float* dM;   // gradient w.r.t. the chunk memories (fp32) or nullptr
    float* dX;         // B x L x H x P (overwritten)
    float* ddt;        // B x L x H (overwritten)
    float* dA;         // H (overwritten)
    float* dB;         // B x L x G x N (overwritten)
    float* dC;         // B x L x G x N (accumulated into when accumulate_dC)
    bool accumulate_dC;
};

size_t sma_bwd_workspace(int64_t B, int64_t L, int64_t H, int64_t Mc, int64_t N);
template <typename Tin, typename Tmem>
cudaError_t launch_sma_backward(const SmaBwdArgs& a, void* ws, cudaStream_t stream);

size_t scan_bwd_workspace(int64_t B, int64_t L, int64_t H, int64_t N, int64_t P, int64_t S);
template <typename Tin>
cudaError_t launch_chunk_scan_backward(const ScanBwdArgs& a, void* ws, unsigned long long wait_limit_ns,
                                       cudaStream_t stream);
// Forward steps 1-3 of the scan (cumsum, chunk states, state passing) for the
// backward: cum and the states entering each chunk, with scratch (fp32, the
// size of the memories) for the chunk-state kernel's memory output.
template <typename Tin>
cudaError_t launch_scan_states(const ScanArgs& a, float* cum, float* Hprev, float* scratch,
                               cudaStream_t stream);

// The whole block (block.cu, gemm_tc.cu): sizes, weights and the workspace buffers.
struct BlockArgs {
    int64_t B, L, H, G, P, N, d_model, conv_width;
    float norm_eps;
    const float* conv_w;  // (d_inner + 2 G N) x conv_width
    const float* conv_b;
    const float* dt_bias;  // H
    const float* A_log;    // H
    const float* D;        // H
    const float* norm_w;   // d_inner
    // workspace
    void* zx;     // B L x ldz fp32: the in-projection output
    int64_t ldz;
    void* X;      // B L x H P bf16 (after the convolution)
    void* Bm;     // B L x G N bf16
    void* Cm;     // B L x G N bf16
    float* dt;    // B L x H
    float* A;     // H
    void* Q;      // B L x G N bf16
    void* E;      // B L x G P bf16
    void* gate;   // B L x H bf16 (the token's gate logit for every head)
    float* Y;     // B L x H P: the hot path's merged output
    void* yn;     // B L x H P bf16: the normalised, gated output
};
cudaError_t launch_block_conv_split(const BlockArgs& a, cudaStream_t stream);
cudaError_t launch_block_norm(const BlockArgs& a, cudaStream_t stream);
bool block_conv_width_ok(int64_t w);
// C (M x ldc, n_store columns written) = A (M x K) B (N x K)^T, bf16 inputs, fp32 accumulation.
template <typename Tc>
cudaError_t launch_gemm_tc(const void* A, const void* B, Tc* C, int64_t M, int64_t N, int64_t K, int64_t ldc,
                           int64_t n_store, unsigned long long wait_limit_ns, cudaStream_t stream);
int take_gemm_status(cudaStream_t stream);

// Kernels launched by the library (read by dart_launch_count()).
void note_launches(int n);

template <typename Tin, typename Tmem, typename Tout>
cudaError_t launch_chunk_scan_simt(const ScanArgs& a, cudaStream_t stream);
// Steps 1 and 3 of the scan (scan.cu), shared by both scan paths.
cudaError_t launch_chunk_cumsum(const ScanArgs& a, cudaStream_t stream);
cudaError_t launch_state_passing(const ScanArgs& a, cudaStream_t stream);

// Tensor-core scan (scan_tc.cu): bf16 inputs, P = 64, N = 128, S in {64, 128, 256}
// (the backward helpers: S in {128, 256}). The forward (launch_chunk_scan_tc) takes
// H and H / G multiples of 4; the backward helpers multiples of 8.
bool scan_tc_supported(const ScanArgs& a);
bool scan_fwd_tc_supported(const ScanArgs& a);
template <typename Tmem, typename Tout>
cudaError_t launch_chunk_scan_tc(const ScanArgs& a, unsigned long long wait_limit_ns,
                                 cudaStream_t stream);
int take_scan_tc_status(cudaStream_t stream);
cudaError_t launch_scan_states_tc(const ScanArgs& a, float* cum, float* Hprev, uint8_t* Hops,
                                  unsigned long long wait_limit_ns, cudaStream_t stream);
cudaError_t launch_scan_bwd_inter_tc(const ScanArgs& a, const float* cum, const void* dY, float* Z,
                                     unsigned long long wait_limit_ns, cudaStream_t stream);
cudaError_t launch_scan_bwd_output_tc(const ScanArgs& a, const float* cum, const uint8_t* Hops,
                                      const uint8_t* Dops, const void* dY, float* rowI,
                                      float* dX, float* xi, unsigned long long wait_limit_ns,
                                      cudaStream_t stream);
size_t scan_bwd_tc_workspace(int64_t B, int64_t L, int64_t H, int64_t S);
cudaError_t launch_chunk_scan_backward_tc(const ScanBwdArgs& a, void* ws,
                                          unsigned long long wait_limit_ns, cudaStream_t stream);
int take_scan_bwd_tc_status(cudaStream_t stream);
cudaError_t launch_scan_bwd_passing(float* ZD, const float* dM, const float* Hprev, const float* cum,
                                    float* dcum_end, uint8_t* Dops, int B, int H, int S, int Mc,
                                    int NP, cudaStream_t stream);
bool scan_bwd_tc_supported(const ScanArgs& f);

template <typename Tmem>
cudaError_t launch_memory_rms(const void* M, float* rM, int64_t rows, int64_t P, float eps,
                              cudaStream_t stream);

template <typename Tin, typename Tmem, typename Tout>
cudaError_t launch_sma_forward_simt(const SmaArgs& a, cudaStream_t stream);

template <typename Tin, typename Tmem, typename Tout>
cudaError_t launch_decode_step(const DecodeArgs& a, cudaStream_t stream);

// dst[r * dst_pitch + i] = src[r * src_pitch + i], i < row_bytes, r < rows (bytes).
cudaError_t launch_copy_rows(void* dst, int64_t dst_pitch, const void* src, int64_t src_pitch, int64_t row_bytes,
                             int64_t rows, cudaStream_t stream);
// dst[r, k] = src[r, h0 + k] for r < rows, k < hg (elements of elem_bytes = 2 or 4;
// src rows of H elements, dst rows of hg).
cudaError_t launch_gather_heads(const void* src, void* dst, int64_t rows, int64_t H, int64_t h0,
                                int64_t hg, int elem_bytes, cudaStream_t stream);

// The SMA forward's operand tiles (P = 64, N = 128): per (b, memory, head pair) an
// 80 KiB job (fp16 W = r M, its e4m3 residual, fp16 M / max|M|) at
// ((b Mc + j) (H / 2) + hp) * 80 KiB, then one fp32 scale max|M| per (b, j, h) at
// sma_tiles_scale_offset. Written by the tensor-core chunk-state kernel or by the
// SMA's own operand kernel; read by the SMA kernel.
size_t sma_tiles_bytes(int64_t B, int64_t Mc, int64_t H);
// Byte layout of one job: [W16 h0 | W16 h1] (MN-major, 128-byte swizzle, rows n),
// the e4m3 residual 2^12 (W - W16) (K-major: rows x 64 + p of 128 bytes over n, the
// same swizzle), [M16 h0 | M16 h1] (as W16).
constexpr int kSmaTile = 128 * 64 * 2;
constexpr int kSmaOffLo = 2 * kSmaTile;
constexpr int kSmaOffV = kSmaOffLo + 2 * 64 * 128;
constexpr int kSmaJob = kSmaOffV + 2 * kSmaTile;
size_t sma_tiles_scale_offset(int64_t B, int64_t Mc, int64_t H);
// Tensor-core SMA (sma_tc.cu): bf16 token inputs, P = 64, N = 128, L % 128 == 0, any S.
bool sma_tc_supported(const SmaArgs& a);
size_t sma_tc_workspace(int64_t B, int64_t Mc, int64_t H);
template <typename Tmem, typename Tout>
cudaError_t launch_sma_forward_tc(const SmaArgs& a, void* ws, unsigned long long wait_limit_ns,
                                  cudaStream_t stream);
// Reads and clears the tensor-core kernels' timeout code (0 = none, -1 = read failed).
int take_tc_status(cudaStream_t stream);

// Tensor-core SMA backward (sma_bwd_tc.cu; statistics pass in sma_tc.cu).
template <typename Tmem>
cudaError_t launch_sma_bwd_stats_tc(const SmaBwdArgs& a, const float* rM, uint8_t* ops,
                                    int pair_bytes, float* scale, float* g, float2* gd,
                                    unsigned long long wait_limit_ns, cudaStream_t stream);
// The same outputs from a.logits (saved by the forward) instead of the logit chains.
template <typename Tmem>
cudaError_t launch_sma_bwd_stats_from_logits(const SmaBwdArgs& a, const float* rM, uint8_t* ops,
                                             int pair_bytes, float* scale, float* g, float2* gd,
                                             cudaStream_t stream);
bool sma_bwd_tc_supported(const SmaBwdArgs& a);
size_t sma_bwd_tc_workspace(int64_t B, int64_t L, int64_t H, int64_t Mc, int64_t N);
template <typename Tmem>
cudaError_t launch_sma_backward_tc(const SmaBwdArgs& a, void* ws, unsigned long long wait_limit_ns,
                                   cudaStream_t stream);
int take_bwd_tc_status(cudaStream_t stream);

}  // namespace dart
