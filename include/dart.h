/*
 * dart.h -- C ABI of the GB300 (sm_103a) hot path of DART, "Decoded Attention
 * over Recurrent sTates" (arXiv 2608.02032).
 *
 * The hot path of one DART block, from the precomputed token projections to
 * the block output (the same boundary as the paper's kernel benchmark,
 * Sec. 5.3 "Kernel Forward Time and Inference Cache"):
 *   dart_chunk_scan   Mamba-2 chunked SSD scan (Sec. 2; App. A) that also
 *                     keeps every chunk state contribution as a chunk state
 *                     memory M_j = Delta H_[j] (Sec. 3).
 *   dart_sma_forward  token-conditioned key/value decoding from the memories,
 *                     causal state-memory attention over chunks (Sec. 3;
 *                     App. B.1; Alg. 1) and the gated residual merge
 *                     Y = Y_ssd + SiLU(z) R (Sec. 3).
 *   dart_decode_step  one autoregressive token over the chunk-memory cache
 *                     and the running state (Sec. 4 "Inference Cache").
 *   dart_sma_backward, dart_chunk_scan_backward
 *                     gradients of the two prefill calls for training (the
 *                     paper trains the layer end to end but prints no
 *                     backward; these are the chain rule on the forms above).
 *   dart_sma_forward_with_logits, dart_sma_backward_with_logits
 *                     the SMA pair for training that keeps the forward's
 *                     logits so the backward need not recompute them.
 *   dart_prefill_host the two prefill calls from host buffers to a host
 *                     buffer, copies overlapped with the kernels.
 *
 * Conventions shared by every entry point
 *   - Every tensor pointer is a DEVICE pointer owned by the caller, 16-byte
 *     aligned, contiguous and row-major in the shapes given below (the
 *     paper's table of compact tensor shapes, App. B.2), except the host
 *     buffers of dart_prefill_host. The library keeps no reference to any
 *     pointer after the call returns.
 *   - The library never allocates device memory. Scratch comes from the
 *     caller's `workspace` (device memory of at least
 *     dart_workspace_size(dims, op) bytes, 256-byte aligned).
 *   - Every call is asynchronous on `stream` (a cudaStream_t; NULL is the
 *     legacy default stream) and does not synchronise the host.
 *     dart_prefill_host also works on streams of its own (created once per
 *     device); calls from several host threads share them and run in turn.
 *   - Stream order holds as for plain launches, with one overlap inside it:
 *     the tensor-core SMA kernel (dart_sma_forward, _with_tiles and
 *     _with_logits on their tensor-core shapes) is launched with programmatic
 *     stream serialization. When the kernel just before it on the stream is
 *     the scan's output kernel, which writes only Y_ssd, its CTAs may start
 *     while that kernel's last CTAs still run, and they read Y_ssd only after
 *     it has completed. After any other kernel, copy or event it starts once
 *     that work is done.
 *   - Arguments are validated on the host before anything is launched; a
 *     call that returns an error has written nothing.
 *   - Token and chunk indices are 0-based: token t lies in chunk t / S, the
 *     paper's 1-based c(t) = ceil(t / S) (Sec. 3).
 *   - Head h reads projection group h / (H / G) (G = 1 in the paper).
 *
 * Numerical readings where the paper is silent
 *   - a_t = exp(dt_t * A_h) and the write term is dt_t * B_t^T X_t; dt is the
 *     post-softplus step size.
 *   - RMSNorm (Qbar, Ebar) and the memory inverse RMS r use unit weight and
 *     dims.eps (App. B.1 names eps without a value).
 *   - The state before the first token is zero (App. A).
 *   - All accumulation is fp32. With mem_dtype = DART_BF16 the memories are
 *     stored in bf16 and r is computed from the stored values.
 */
#ifndef DART_H_
#define DART_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    DART_OK = 0,
    DART_ERR_INVALID_ARG = 1,  /* NULL or misaligned pointer, bad dims, H % G != 0, eps <= 0 */
    DART_ERR_UNSUPPORTED = 2,  /* valid but not built: P/N/S outside the set below, L % S != 0 where required */
    DART_ERR_WORKSPACE = 3,    /* workspace NULL/misaligned or smaller than dart_workspace_size */
    DART_ERR_CUDA = 4,         /* a CUDA call failed; see dart_last_cuda_error() */
    DART_ERR_TIMEOUT = 5,      /* a device-side wait gave up (see dart_get_device_status) */
    DART_ERR_TOO_LARGE = 6     /* beyond the fixed scratch of dart_sma_forward_noalloc */
} dart_status;

typedef enum { DART_F32 = 0, DART_BF16 = 1 } dart_dtype;

/* Problem sizes in the paper's notation (App. B.2). */
typedef struct {
    int64_t batch;     /* Bsz */
    int64_t seqlen;    /* L (ignored by dart_decode_step) */
    int64_t nheads;    /* H */
    int64_t ngroups;   /* G, must divide H */
    int64_t headdim;   /* P, value axis of a memory */
    int64_t dstate;    /* N, key axis of a memory (SSD state size) */
    int64_t chunk;     /* S, chunk size; M = ceil(L / S) memories per (b, h) */
    int32_t in_dtype;  /* dart_dtype of the token inputs X, B, C, Q, E, z and x, b, c, q, e, z */
    int32_t mem_dtype; /* dart_dtype of the chunk memories M and the decode cache */
    int32_t out_dtype; /* dart_dtype of the outputs Y_ssd, Y, R and the decode output y */
    float eps;         /* RMSNorm / inverse-RMS epsilon, > 0 */
} dart_dims;

/* Supported sizes: P in {16, 32, 64}, N in {16, 32, 64, 128},
 * S in {16, 32, 64, 128, 256}. L need not be a multiple of S for
 * dart_chunk_scan, dart_sma_forward and dart_prefill_host (M = ceil(L / S)
 * memories; the last holds the partial chunk, e(c) = L - 1, which is the
 * running partial memory a decode continues from); the backward calls,
 * dart_sma_forward_with_logits and dart_sma_forward_noalloc need L % S == 0
 * (DART_ERR_UNSUPPORTED otherwise). Supported dtype triples
 * (in, mem, out): (F32, F32, F32), (BF16, F32, F32), (BF16, BF16, F32) and
 * (BF16, BF16, BF16). Accumulation is fp32 in every case. Outputs and
 * memories heavy-tailed enough that rounding them to bf16 costs several
 * percent of their RMS, so fp32 outputs are the default for bf16 inputs.
 * Size limits: (L / S) H <= 65535 * 64 and Bsz, H <= 65535 (refused with
 * DART_ERR_UNSUPPORTED); on the tensor-core scan the output kernel's grid also
 * needs (L / S) H / d <= 65535, d its heads per CTA (8 to 16), so past about
 * a million (chunk, head) pairs dart_chunk_scan returns DART_ERR_CUDA. */

typedef enum {
    DART_OP_CHUNK_SCAN = 0,
    DART_OP_SMA_FORWARD = 1,
    DART_OP_DECODE_STEP = 2,
    DART_OP_SMA_BACKWARD = 3,
    DART_OP_SCAN_BACKWARD = 4,
    DART_OP_PREFILL_HOST = 5
} dart_op;

/* Human-readable name of a status code (static storage, never NULL). */
const char* dart_status_string(dart_status status);

/* The cudaError_t of the most recent DART_ERR_CUDA on this thread (0 if none). */
int dart_last_cuda_error(void);

/* Bytes of workspace `op` needs for `dims` (0 if none). Returns 0 for
 * invalid dims too; the entry point then reports the error. */
size_t dart_workspace_size(const dart_dims* dims, int op);

/*
 * Chunked SSD scan with chunk state memories (Sec. 2 SSD recurrence;
 * App. A eqs. "mamba2_chunk_state" and "mamba2_delta_h_chunk"; Sec. 3
 * equation for Delta H_[c]):
 *   Y_ssd_t = C_t H_t with H_t = exp(dt_t A_h) H_{t-1} + dt_t B_t^T X_t,
 *   M[b, c, h] = sum_{s in chunk c} exp(sum_{k=s+1}^{e(c)} dt_k A_h) dt_s B_s^T X_s.
 * Inputs:  X  (Bsz, L, H, P) in_dtype;  dt (Bsz, L, H) fp32 (post-softplus);
 *          A  (H) fp32;  Bm, Cm (Bsz, L, G, N) in_dtype.
 * Outputs: Y_ssd (Bsz, L, H, P) out_dtype;  M (Bsz, M, H, N, P) mem_dtype;
 *          rM (Bsz, M, H, N) fp32 or NULL: r[n] = (mean_p M[n, p]^2 + eps)^-1/2
 *          of the stored memory (App. B.1);
 *          final_state (Bsz, H, N, P) fp32 or NULL: H_{L-1}.
 * Ragged L (L % S != 0): the kernels run on copies of the inputs zero-padded to
 * ceil(L / S) S tokens inside the workspace (a padded token has dt = 0: decay 1,
 * no write, so states and memories are exactly the L-token ones) and the first L
 * rows of Y_ssd are copied out; dart_workspace_size includes the copies.
 * The tensor-core kernels serve bf16 inputs with P = 64, N = 128, S in
 * {64, 128, 256} and H, H / G multiples of 4; every other shape runs on the
 * CUDA-core kernels.
 */
dart_status dart_chunk_scan(const dart_dims* dims, const void* X, const float* dt,
                            const float* A, const void* Bm, const void* Cm, void* Y_ssd,
                            void* M, float* rM, float* final_state, void* workspace,
                            size_t workspace_bytes, void* stream);

/*
 * State-memory attention and gated merge (Sec. 3 value/key readouts, chunk
 * logit, softmax over earlier chunks and R_t; App. B.1 normalised score
 * branch; Alg. 1 streaming form; Sec. 3 "Gated Residual Integration"):
 *   Qbar = RMSNorm(Q_t), Ebar = RMSNorm(E_t),
 *   l_{t,j} = Qbar (r_j (.) (M_j Ebar)) / sqrt(N),  V_{t,j} = C_t M_j,
 *   g = softmax over j < t / S,  R_t = sum_j g_j V_{t,j},
 *   lse_t = log sum_j exp(l_{t,j}),  Y = Y_ssd + SiLU(z) R.
 * Tokens of chunk 0 have R = 0, lse = -inf and Y = Y_ssd.
 * Inputs:  M (Bsz, M, H, N, P) mem_dtype;  rM (Bsz, M, H, N) fp32 or NULL
 *          (NULL: computed from M into the workspace);
 *          Q, Cm (Bsz, L, G, N) in_dtype;  E (Bsz, L, G, P) in_dtype;
 *          z (Bsz, L, H) in_dtype gate logits;  Y_ssd (Bsz, L, H, P) out_dtype.
 * Outputs: Y (Bsz, L, H, P) out_dtype;  R (Bsz, L, H, P) out_dtype or NULL;
 *          lse (Bsz, L, H) fp32 or NULL.
 * Workspace: dart_workspace_size(dims, DART_OP_SMA_FORWARD) bytes. Always
 *          needed on the tensor-core path (bf16 inputs, P = 64, N = 128,
 *          L a multiple of 128 after padding to whole chunks, H / G even; any S:
 *          a 128-token tile spanning several chunks runs the memories of its
 *          last token and each token keeps its own), where it holds each memory's MMA
 *          operands (48 KiB per memory and head); elsewhere only when rM is
 *          NULL (for r).
 */
dart_status dart_sma_forward(const dart_dims* dims, const void* M, const float* rM,
                             const void* Q, const void* Cm, const void* E, const void* z,
                             const void* Y_ssd, void* Y, void* R, float* lse, void* workspace,
                             size_t workspace_bytes, void* stream);

/*
 * The prefill of one block (dart_chunk_scan then dart_sma_forward) from
 * host buffers to a host buffer, with the copies overlapped with the kernels.
 * The heads are taken in groups of 4 when G = 1 and H is a larger multiple of
 * 4 with at most 64 groups (one group otherwise): per group the X rows go to
 * the device (a pitched copy), the scan and SMA kernels run on them, and the
 * group's Y rows come back, on five streams of the library's own (copy in,
 * three for the kernels taking the groups in turn, copy out), so that the
 * copies run under the kernels and neighbouring groups' kernels share the SMs. The shared inputs
 * (B, C, Q, E, dt, A, z) go first; the gather of a group's dt and gate logits
 * runs on the device. Per head the result is that of the device entry points.
 * Inputs:  X (Bsz, L, H, P), Bm, Cm, Q (Bsz, L, G, N), E (Bsz, L, G, P),
 *          z (Bsz, L, H) in_dtype; dt (Bsz, L, H), A (H) fp32: HOST memory,
 *          page-locked for the copies to overlap.
 * Output:  Y (Bsz, L, H, P) out_dtype, HOST memory (page-locked), complete
 *          once `stream` reaches the point where the call left it.
 * Workspace: dart_workspace_size(dims, DART_OP_PREFILL_HOST) bytes of device
 *          memory, 256-byte aligned: device copies of the inputs, each group's
 *          Y_ssd, Y, memories and their r, and the scan and SMA workspaces. On
 *          the shapes of dart_chunk_scan_with_tiles each group's scan writes
 *          the SMA's operand tiles, which take the SMA workspace's place.
 * The call orders itself after the work already on `stream` and leaves
 * `stream` waiting for its last copy (also when it fails part way, for what
 * it had enqueued). The four streams are created on the
 * first call for the current device and kept for the process.
 */
dart_status dart_prefill_host(const dart_dims* dims, const void* X, const float* dt, const float* A,
                              const void* Bm, const void* Cm, const void* Q, const void* E,
                              const void* z, void* Y, void* workspace, size_t workspace_bytes,
                              void* stream);

/*
 * One decode step over the chunk-memory cache (the persistent inference
 * cache of Sec. 4 "Inference Cache" and Sec. 5.3; the paper gives no decode
 * algorithm, this is the reading that makes prefill followed by decode equal
 * a longer prefill). For the token at index pos (pos tokens absorbed before
 * it) and i = pos / S completed chunks:
 *   a = exp(dt A_h);  state <- a state + dt b^T x;
 *   partial <- dt b^T x if pos % S == 0, else a partial + dt b^T x;
 *   y = c state + SiLU(z) R, R = SMA over cache memories j < i (as above);
 *   if (pos + 1) % S == 0: cache[b, i, h] <- partial (and i < m_cap).
 * In/out:  cache (Bsz, m_cap, H, N, P) mem_dtype; memories j < i are read,
 *          slot i is written when its chunk completes;
 *          state, partial (Bsz, H, N, P) fp32, updated in place.
 * Inputs:  x (Bsz, H, P) in_dtype; dt (Bsz, H) fp32; A (H) fp32;
 *          b, c, q (Bsz, G, N) in_dtype; e (Bsz, G, P) in_dtype; z (Bsz, H) in_dtype.
 * Outputs: y (Bsz, H, P) out_dtype; lse (Bsz, H) fp32 or NULL.
 * Requires pos >= 0 and pos / S <= m_cap; dims.seqlen is ignored.
 */
dart_status dart_decode_step(const dart_dims* dims, int64_t pos, int64_t m_cap, void* cache,
                             float* state, float* partial, const void* x, const float* dt,
                             const float* A, const void* b, const void* c, const void* q,
                             const void* e, const void* z, void* y, float* lse,
                             void* workspace, size_t workspace_bytes, void* stream);

/*
 * Backward of dart_sma_forward (training). Chain rule on the forward above,
 * with the saved lse as the softmax normaliser: per token t with history and
 * memory j,
 *   dR_t = SiLU(z_t) dY_t,  g_{t,j} = exp(l_{t,j} - lse_t),
 *   dl_{t,j} = g_{t,j} (dR_t . V_{t,j} - dR_t . R_t),  dV_{t,j} = g_{t,j} dR_t,
 * then through V = C M_j, l = Qbar (r_j (.) M_j Ebar) / sqrt(N), r_j(M_j) and
 * the unit-weight RMSNorms to dM, dQ, dC, dE; dz_t = (dY_t . R_t) SiLU'(z_t).
 * The gradient w.r.t. Y_ssd is dY itself and is not written.
 * Inputs:  M, rM (or NULL), Q, Cm, E, z as for dart_sma_forward (rM, when
 *          given, must be the one the forward used); lse (Bsz, L, H) fp32 as
 *          written by dart_sma_forward; dY (Bsz, L, H, P) in_dtype.
 * Outputs: fp32, overwritten: dM (Bsz, M, H, N, P); dQ, dC (Bsz, L, G, N);
 *          dE (Bsz, L, G, P); dz (Bsz, L, H). dQ, dC and dE are summed over
 *          the heads of a group with fp32 atomics, so their low bits vary from
 *          run to run.
 * Workspace: dart_workspace_size(dims, DART_OP_SMA_BACKWARD): the weights g and
 *          logit gradients dl of every (memory, token) pair, 2 x Bsz x H x M x L
 *          fp32, plus r when rM is NULL.
 * Groups: the tensor-core backward (bf16 inputs, P = 64, N = 128, S % 128 == 0,
 *          L % 128 == 0) sums dQ, dC, dE over all heads of a launch. At G > 1
 *          with H/G even it runs once per group, on the group's heads and its
 *          Q, C, E column block copied into contiguous buffers in the workspace,
 *          and copies the group's gradients back; other G > 1 shapes take the
 *          CUDA-core kernels.
 */
dart_status dart_sma_backward(const dart_dims* dims, const void* M, const float* rM,
                              const void* Q, const void* Cm, const void* E, const void* z,
                              const float* lse, const void* dY, float* dM, float* dQ, float* dC,
                              float* dE, float* dz, void* workspace, size_t workspace_bytes,
                              void* stream);

/*
 * Training pair that saves the logits. dart_sma_forward_with_logits is
 * dart_sma_forward that also writes logits (Bsz, H, M, L) fp32, the entry
 * (b, h, j, t) holding l_{t,j} for j < t / S (other entries unwritten); lse
 * is required. It needs the tensor-core path (bf16 inputs, P = 64, N = 128,
 * L % 128 == 0, H/G even) and gives DART_ERR_UNSUPPORTED elsewhere.
 * dart_sma_backward_with_logits is dart_sma_backward with those logits: on
 * the tensor-core path the weights g come from them (the same values as the
 * recomputation, which it skips); the CUDA-core path recomputes them.
 */
dart_status dart_sma_forward_with_logits(const dart_dims* dims, const void* M, const float* rM,
                                         const void* Q, const void* Cm, const void* E, const void* z,
                                         const void* Y_ssd, void* Y, void* R, float* lse, float* logits,
                                         void* workspace, size_t workspace_bytes, void* stream);
dart_status dart_sma_backward_with_logits(const dart_dims* dims, const void* M, const float* rM,
                                          const void* Q, const void* Cm, const void* E, const void* z,
                                          const float* lse, const float* logits, const void* dY, float* dM,
                                          float* dQ, float* dC, float* dE, float* dz, void* workspace,
                                          size_t workspace_bytes, void* stream);

/*
 * Prefill pair that hands the SMA its operands from the scan (no counterpart in
 * the paper: a fusion of data movement). The tensor-core SMA forward reads each
 * memory M_j as operand tiles per memory and pair of heads:
 *   W = r_j (.) M_j as fp16 and the e4m3 residual 2^12 (W - fp16(W));
 *   M_j / max|M_j| as fp16, with the scale max|M_j|.
 * dart_sma_forward builds them from M and rM in a pass of its own.
 * dart_chunk_scan_with_tiles is dart_chunk_scan that also writes those tiles from
 * the chunk-state kernel, which holds each memory in registers as it computes it,
 * into `tiles`. dart_sma_forward_with_tiles is dart_sma_forward that reads them
 * instead of M and rM. The results equal the two regular calls' bit for bit; the
 * tile-building pass and its re-read of M are saved.
 * tiles:   caller-owned device buffer of dart_sma_tiles_size(dims) bytes, 256-byte
 *          aligned, an opaque layout; valid for the dims and the memories of the
 *          dart_chunk_scan_with_tiles call that wrote it.
 * Other arguments, outputs and the scan's workspace as for dart_chunk_scan and
 * dart_sma_forward; dart_sma_forward_with_tiles takes no workspace.
 * Requires the tensor-core paths of both calls: bf16 inputs, P = 64, N = 128,
 * S in {64, 128, 256}, H and H/G multiples of 4, L a multiple of 128 and of S.
 * dart_sma_tiles_size returns 0 elsewhere, and the calls DART_ERR_UNSUPPORTED.
 */
size_t dart_sma_tiles_size(const dart_dims* dims);
dart_status dart_chunk_scan_with_tiles(const dart_dims* dims, const void* X, const float* dt,
                                       const float* A, const void* Bm, const void* Cm, void* Y_ssd,
                                       void* M, float* rM, float* final_state, void* tiles,
                                       void* workspace, size_t workspace_bytes, void* stream);
dart_status dart_sma_forward_with_tiles(const dart_dims* dims, const void* tiles, const void* Q,
                                        const void* Cm, const void* E, const void* z, const void* Y_ssd,
                                        void* Y, void* R, float* lse, void* stream);

/*
 * Backward of dart_chunk_scan (training): gradients of a loss that depends on
 * Y_ssd (through dY) and on the chunk memories (through dM, e.g. the output of
 * dart_sma_backward). Chain rule on the chunked forms of App. A: the states
 * entering each chunk are recomputed, the adjoint of the inter-chunk state runs
 * backwards over the chunks, and each chunk's intra-chunk, inter-chunk and
 * memory terms give dX, dB, dC and the gradient of the within-chunk decay,
 * which a reverse cumulative sum turns into d(dt) and dA.
 * Inputs:  X, dt, A, Bm, Cm as for dart_chunk_scan; dY (Bsz, L, H, P) in_dtype;
 *          dM (Bsz, M, H, N, P) fp32 or NULL (no memory gradient).
 * Outputs: fp32. Overwritten: dX (Bsz, L, H, P), ddt (Bsz, L, H), dA (H),
 *          dB (Bsz, L, G, N). ACCUMULATED: dC (Bsz, L, G, N) gets the scan's
 *          part added, so the SMA part from dart_sma_backward can be passed in
 *          (zero it first otherwise). dA, dB and dC are sums over heads or
 *          tokens taken with fp32 atomics.
 * Workspace: dart_workspace_size(dims, DART_OP_SCAN_BACKWARD): the within-chunk
 *          cumulative decay, the state entering each chunk and the memory
 *          adjoints (2 x Bsz x M x H x N x P fp32).
 * Groups: the tensor-core backward (bf16 inputs, P = 64, N = 128, S in {128,
 *          256}) sums its intra-chunk dB, dC over all heads of a launch. At
 *          G > 1 with H/G a multiple of 8 it runs once per group on copies of
 *          the group's slices in the workspace (dC's block is copied in, added
 *          to and copied back); other G > 1 shapes take the CUDA-core kernels.
 */
dart_status dart_chunk_scan_backward(const dart_dims* dims, const void* X, const float* dt,
                                     const float* A, const void* Bm, const void* Cm,
                                     const void* dY, const float* dM, float* dX, float* ddt,
                                     float* dA, float* dB, float* dC, void* workspace,
                                     size_t workspace_bytes, void* stream);

/*
 * The whole DART block around the hot path, for a prefill (Sec. 3: Q, E and the
 * gate are projections of the block input U_t, C is shared with the SSM branch
 * and Y_t = C_t H_t + G_t R_t; for the rest the Mamba-2 block the paper builds
 * on, with the sizes of App. D.2: head dimension 64, one B, C group,
 * convolution width 4, RMSNorm):
 *   zx = U W_in^T, cut into z (d_inner), x (d_inner), B (G N), C (G N), dt (H),
 *        Q (G N), E (G P), gate (1) in this column order, d_inner = H P;
 *   x, B, C <- SiLU(causal depthwise convolution, per channel c:
 *        b[c] + sum_k conv_w[c, k] v[t - width + 1 + k, c], zero before t = 0);
 *   dt <- softplus(dt + dt_bias), A = -exp(A_log), the gate logit of token t for
 *        every head (one scalar per token, App. D.2);
 *   Y = the hot path (dart_chunk_scan, dart_sma_forward) on X, dt, A, B, C, Q, E, gate;
 *   y = Y + D_h x;  yn = RMSNorm(y * SiLU(z)) * norm_w over d_inner (norm_eps);
 *   out = yn W_out^T.
 * Precision: U and the weights W_in, W_out are bf16; the in-projection output, the
 * memories and Y are fp32; the hot path's token inputs (x, B, C, Q, E, the gate
 * logit) and yn are rounded to bf16; every accumulation is fp32.
 * Inputs:  U (Bsz, L, d_model) bf16; W_in (D_in, d_model) bf16 with D_in = 2 d_inner
 *          + 3 G N + H + G P + 1; conv_w (d_inner + 2 G N, conv_width), conv_b
 *          (d_inner + 2 G N), dt_bias, A_log, D (H), norm_w (d_inner) fp32;
 *          W_out (d_model, d_inner) bf16 (nn.Linear layouts).
 * Output:  out (Bsz, L, d_model) in core.out_dtype (DART_F32 or DART_BF16).
 * Requires core.in_dtype == DART_BF16, d_model % 8 == 0, H % 8 == 0, H P <= 4096;
 * L need not be a multiple of S. Workspace: dart_block_workspace_size(dims): zx,
 * the hot path's inputs and outputs, yn, the scan's workspace and either the SMA's
 * workspace or, on the shapes of dart_chunk_scan_with_tiles, the SMA's operand tiles
 * (written by the scan).
 */
typedef struct {
    dart_dims core;      /* Bsz, L, H, G, P, N, S, eps of the hot path; in_dtype (DART_BF16) and
                            out_dtype (of the block output); mem_dtype is ignored (fp32 memories) */
    int64_t d_model;     /* width of U and of the output */
    int64_t conv_width;  /* 1 .. 8 (4 in the paper) */
    float norm_eps;      /* epsilon of the output RMSNorm, > 0 */
} dart_block_dims;

size_t dart_block_workspace_size(const dart_block_dims* dims);
dart_status dart_block_forward(const dart_block_dims* dims, const void* U, const void* W_in,
                               const float* conv_w, const float* conv_b, const float* dt_bias,
                               const float* A_log, const float* D, const float* norm_w,
                               const void* W_out, void* out, void* workspace, size_t workspace_bytes,
                               void* stream);

/*
 * dart_sma_forward_noalloc: dart_sma_forward with rM = NULL, for callers that
 * cannot allocate device memory and cannot pass a workspace. The paper has no
 * counterpart; this entry point exists for integration. Typical callers: a
 * host framework that hands a plugin only its input and output buffers and
 * owns all other device memory; a latency-critical service that forbids
 * allocation after start-up (cudaMalloc and cudaFree can synchronise the
 * device); a process under a fixed device-memory budget.
 * It computes what dart_sma_forward computes when rM is NULL, with the same
 * definitions, but always on the CUDA-core (FFMA) SMA kernel: there is no
 * tensor-core path here. Its results therefore equal dart_sma_forward's bit for
 * bit only on shapes that take the CUDA-core kernel there too; on the
 * tensor-core shapes (bf16 inputs, P = 64, N = 128, L % 128 == 0, H/G even)
 * they agree within the bf16-input tolerance (max|err| / RMS <= 2e-2), and the
 * call is several times slower at long L. Its only scratch, the inverse RMS of
 * every memory row, lives in a fixed device array of 2^20 fp32 values (4 MiB)
 * inside the library, which every GPU that loads the library holds until the
 * process exits. It calls no cudaMalloc, no cudaFree and no allocating library
 * routine.
 * Arguments: as dart_sma_forward, without rM and the workspace. The caller
 * still passes (and owns) every input and output.
 * Limit: Bsz * (L / S) * H * N <= 2^20 memory rows (e.g. B1 H32 L16384 N128
 * S256 uses 2^18); larger problems return DART_ERR_TOO_LARGE before anything
 * is launched.
 * Set-up: the first call on a device looks up the array's device address on
 * that device (with that device current) and caches it; make that first call
 * before any stream capture. The cached address assumes the device context
 * lives as long as the process: the library does not support cudaDeviceReset
 * (or a primary-context release) between its calls. All calls share the array and it keeps the last
 * call's contents (every entry read is first written by the same call, so
 * nothing needs clearing). Calls that overlap on the GPU, on any streams,
 * race on the array: serialise them.
 */
dart_status dart_sma_forward_noalloc(const dart_dims* dims, const void* M, const void* Q,
                                     const void* Cm, const void* E, const void* z,
                                     const void* Y_ssd, void* Y, void* R, float* lse,
                                     void* stream);

/* Number of kernels this library has launched in this process since it was
 * loaded (all entry points, all threads). A diagnostic for benchmarks. */
uint64_t dart_launch_count(void);

/*
 * Bound on every device-side wait of the tensor-core kernels, in nanoseconds
 * of wall-clock time per wait (default 2 s; 0 restores the default). A wait
 * that runs out makes the kernel stop its pipeline, finish its own copies and
 * MMAs in flight, free its tensor memory and record DART_ERR_TIMEOUT for
 * dart_get_device_status(); the outputs of that call are then undefined.
 * Tests set a tiny bound to exercise that path without faulting the GPU.
 * Process-wide; takes effect for launches after the call.
 */
void dart_set_wait_limit_ns(uint64_t limit_ns);

/*
 * Test hook for the failure path of the tensor-core kernels (no counterpart in
 * the paper): while on, one ring-fed kernel of each tensor-core call issues
 * none of its copies (dart_sma_forward: the SMA kernel's operands;
 * dart_chunk_scan: the state passing's chunk slabs; dart_sma_backward: the row
 * kernels' operands; dart_chunk_scan_backward: the reverse passing's slabs),
 * so its pipeline waits can only run out (each bounded by
 * dart_set_wait_limit_ns); the call then reports DART_ERR_TIMEOUT through
 * dart_get_device_status and its outputs are undefined. Process-wide; 0 (the
 * default) turns it off. For tests only.
 */
void dart_test_withhold_copies(int on);

/*
 * Synchronises `stream`, then reports and clears the device status word that
 * kernels set when a bounded device-side wait gives up: DART_ERR_TIMEOUT if
 * one did since the last call, DART_ERR_CUDA if the synchronisation failed,
 * else DART_OK.
 */
dart_status dart_get_device_status(void* stream);

#ifdef __cplusplus
}
#endif

#endif /* DART_H_ */
