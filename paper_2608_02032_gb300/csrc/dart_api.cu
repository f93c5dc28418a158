// C ABI of the DART hot path: host-side validation, workspace layout and
// kernel dispatch. Declarations and the contract are in include/dart.h.
#include <algorithm>
#include <atomic>
#include <mutex>

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "dart.h"
#include "kernels.h"

namespace {

thread_local int t_last_cuda_error = 0;

typedef long long i64;

dart_status cuda_fail(cudaError_t e) {
    t_last_cuda_error = (int)e;
    return DART_ERR_CUDA;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }
bool is_pow2(int64_t v) { return v > 0 && (v & (v - 1)) == 0; }

size_t align256(size_t v) { return (v + 255) & ~(size_t)255; }

// Supported (in, mem, out) dtype triples.
enum class Combo { kFFF, kBFF, kBBF, kBBB, kNone };

Combo combo_of(const dart_dims* d) {
    const int i = d->in_dtype, m = d->mem_dtype, o = d->out_dtype;
    if (i == DART_F32 && m == DART_F32 && o == DART_F32) return Combo::kFFF;
    if (i == DART_BF16 && m == DART_F32 && o == DART_F32) return Combo::kBFF;
    if (i == DART_BF16 && m == DART_BF16 && o == DART_F32) return Combo::kBBF;
    if (i == DART_BF16 && m == DART_BF16 && o == DART_BF16) return Combo::kBBB;
    return Combo::kNone;
}

// Calls L<Tin, Tmem, Tout>::run(args...) for the dtype triple of d.
template <template <typename, typename, typename> class L, typename... Args>
cudaError_t dispatch(const dart_dims* d, Args&&... args) {
    typedef __nv_bfloat16 bf;
    switch (combo_of(d)) {
        case Combo::kFFF: return L<float, float, float>::run(args...);
        case Combo::kBFF: return L<bf, float, float>::run(args...);
        case Combo::kBBF: return L<bf, bf, float>::run(args...);
        case Combo::kBBB: return L<bf, bf, bf>::run(args...);
        default: return cudaErrorInvalidValue;
    }
}

template <typename I, typename M, typename O> struct ScanL {
    static cudaError_t run(const dart::ScanArgs& a, cudaStream_t s) {
        return dart::launch_chunk_scan_simt<I, M, O>(a, s);
    }
};
template <typename I, typename M, typename O> struct SmaL {
    static cudaError_t run(const dart::SmaArgs& a, cudaStream_t s) {
        return dart::launch_sma_forward_simt<I, M, O>(a, s);
    }
};
template <typename I, typename M, typename O> struct DecodeL {
    static cudaError_t run(const dart::DecodeArgs& a, cudaStream_t s) {
        return dart::launch_decode_step<I, M, O>(a, s);
    }
};

// Shared validation of the sizes in dims (without the op-specific parts).
dart_status check_dims(const dart_dims* d, bool need_seqlen, bool ragged_ok = false) {
    if (d == nullptr) return DART_ERR_INVALID_ARG;
    if (d->batch <= 0 || d->nheads <= 0 || d->ngroups <= 0 || d->headdim <= 0 || d->dstate <= 0 ||
        d->chunk <= 0)
        return DART_ERR_INVALID_ARG;
    if (need_seqlen && d->seqlen <= 0) return DART_ERR_INVALID_ARG;
    if (d->nheads % d->ngroups != 0) return DART_ERR_INVALID_ARG;
    if (!(d->eps > 0.0f)) return DART_ERR_INVALID_ARG;
    if (d->in_dtype != DART_F32 && d->in_dtype != DART_BF16) return DART_ERR_INVALID_ARG;
    if (d->mem_dtype != DART_F32 && d->mem_dtype != DART_BF16) return DART_ERR_INVALID_ARG;
    if (d->out_dtype != DART_F32 && d->out_dtype != DART_BF16) return DART_ERR_INVALID_ARG;
    if (combo_of(d) == Combo::kNone) return DART_ERR_UNSUPPORTED;
    const int64_t P = d->headdim, N = d->dstate, S = d->chunk;
    if (!(P == 16 || P == 32 || P == 64)) return DART_ERR_UNSUPPORTED;
    if (!(N == 16 || N == 32 || N == 64 || N == 128)) return DART_ERR_UNSUPPORTED;
    if (!(is_pow2(S) && S >= 16 && S <= 256)) return DART_ERR_UNSUPPORTED;
    if (need_seqlen && d->seqlen % S != 0 && !ragged_ok) return DART_ERR_UNSUPPORTED;
    // every offset below is computed in 64-bit, but grid dimensions are 32-bit
    if (need_seqlen && (d->seqlen + S - 1) / S * d->nheads > 65535 * 64) return DART_ERR_UNSUPPORTED;
    if (d->batch > 65535 || d->nheads > 65535) return DART_ERR_UNSUPPORTED;
    return DART_OK;
}

struct ScanWs {
    size_t cum_off, dh_off, hops_off, total;
};

bool scan_uses_tc(const dart_dims* d) {
    dart::ScanArgs a{};
    a.B = d->batch; a.L = d->seqlen; a.H = d->nheads; a.G = d->ngroups;
    a.P = d->headdim; a.N = d->dstate; a.S = d->chunk;
    return d->in_dtype == DART_BF16 && dart::scan_fwd_tc_supported(a);
}

// Workspace of the scan for L % S == 0.
ScanWs scan_ws(const dart_dims* d) {
    const i64 M = d->seqlen / d->chunk;
    const size_t states = align256((size_t)(d->batch * M * d->nheads * d->dstate * d->headdim) *
                                   sizeof(float));
    ScanWs w;
    w.cum_off = 0;
    w.dh_off = align256((size_t)(d->batch * d->nheads * M * d->chunk) * sizeof(float));
    w.hops_off = w.dh_off + states;
    // tensor-core path: the chunk-entry states also as bf16 hi | lo operand tiles (same bytes)
    w.total = w.hops_off + (scan_uses_tc(d) ? states : 0);
    return w;
}

dart::SmaArgs sma_args(const dart_dims* d) {
    dart::SmaArgs a{};
    a.B = d->batch; a.L = d->seqlen; a.H = d->nheads; a.G = d->ngroups;
    a.P = d->headdim; a.N = d->dstate; a.S = d->chunk; a.eps = d->eps;
    return a;
}

// The tensor-core SMA serves bf16 token inputs at its tile shape; everything
// else runs on the FFMA kernel.
bool sma_uses_tc(const dart_dims* d) {
    return d->in_dtype == DART_BF16 && dart::sma_tc_supported(sma_args(d));
}

// The tensor-core SMA backward serves bf16 token inputs at its tile shape with G = 1.
dart::SmaBwdArgs sma_bwd_args(const dart_dims* d) {
    dart::SmaBwdArgs a{};
    a.B = d->batch; a.L = d->seqlen; a.H = d->nheads; a.G = d->ngroups;
    a.P = d->headdim; a.N = d->dstate; a.S = d->chunk; a.eps = d->eps;
    return a;
}
bool sma_bwd_uses_tc(const dart_dims* d) {
    return d->in_dtype == DART_BF16 && dart::sma_bwd_tc_supported(sma_bwd_args(d));
}

// ---- G > 1 on the tensor-core backward. The backward kernels sum over all heads
// of a call (the SMA row kernels' dQ, dC over head pairs; the scan's intra-chunk
// dB, dC through the head-summed Psi), so they serve G = 1. A group g is itself
// a G = 1 problem over its H/G heads: a contiguous slice of every token row (X,
// dt, z, lse, dY and the per-head gradients), one column block of every B, C, Q,
// E row, and a slice of every (b, chunk) block of the memories. The grouped path
// copies a group's inputs into contiguous buffers, runs the G = 1 tensor-core
// backward on them and copies its gradients back, group after group on the
// caller's stream (the groups share the buffers).
dart_dims group_dims(const dart_dims* d) {
    dart_dims g = *d;
    g.nheads = d->nheads / d->ngroups;
    g.ngroups = 1;
    return g;
}
bool sma_bwd_grouped(const dart_dims* d) {
    if (d->ngroups <= 1 || d->in_dtype != DART_BF16) return false;
    const dart_dims g = group_dims(d);
    return sma_bwd_uses_tc(&g);
}
bool scan_bwd_grouped(const dart_dims* d) {
    if (d->ngroups <= 1 || d->in_dtype != DART_BF16) return false;
    dart::ScanArgs a{};
    a.B = d->batch; a.L = d->seqlen; a.H = d->nheads / d->ngroups; a.G = 1;
    a.P = d->headdim; a.N = d->dstate; a.S = d->chunk;
    return dart::scan_bwd_tc_supported(a);
}

struct SmaBwdGroupWs {  // byte offsets into the workspace
    size_t tc, M, rM, Q, C, E, z, lse, dY, logits, dM, dQ, dC, dE, dz, total;
};
SmaBwdGroupWs sma_bwd_group_ws(const dart_dims* d) {
    const size_t B = d->batch, L = d->seqlen, Hg = d->nheads / d->ngroups, P = d->headdim, N = d->dstate,
                 Mc = d->seqlen / d->chunk;
    const size_t em = d->mem_dtype == DART_F32 ? 4 : 2, ei = 2;
    SmaBwdGroupWs w{};
    size_t o = 0;
    auto take = [&](size_t bytes) { const size_t at = o; o += align256(bytes); return at; };
    w.tc = take(dart::sma_bwd_tc_workspace(B, L, Hg, Mc, N));
    w.M = take(B * Mc * Hg * N * P * em);
    w.rM = take(B * Mc * Hg * N * 4);
    w.Q = take(B * L * N * ei);
    w.C = take(B * L * N * ei);
    w.E = take(B * L * P * ei);
    w.z = take(B * L * Hg * ei);
    w.lse = take(B * L * Hg * 4);
    w.dY = take(B * L * Hg * P * ei);
    w.logits = take(B * Hg * Mc * L * 4);
    w.dM = take(B * Mc * Hg * N * P * 4);
    w.dQ = take(B * L * N * 4);
    w.dC = take(B * L * N * 4);
    w.dE = take(B * L * P * 4);
    w.dz = take(B * L * Hg * 4);
    w.total = o;
    return w;
}

struct ScanBwdGroupWs {
    size_t tc, X, dt, Bm, Cm, dY, dM, dX, ddt, dB, dC, total;
};
ScanBwdGroupWs scan_bwd_group_ws(const dart_dims* d) {
    const size_t B = d->batch, L = d->seqlen, Hg = d->nheads / d->ngroups, P = d->headdim, N = d->dstate,
                 Mc = d->seqlen / d->chunk;
    ScanBwdGroupWs w{};
    size_t o = 0;
    auto take = [&](size_t bytes) { const size_t at = o; o += align256(bytes); return at; };
    w.tc = take(dart::scan_bwd_tc_workspace(B, L, Hg, d->chunk));
    w.X = take(B * L * Hg * P * 2);
    w.dt = take(B * L * Hg * 4);
    w.Bm = take(B * L * N * 2);
    w.Cm = take(B * L * N * 2);
    w.dY = take(B * L * Hg * P * 2);
    w.dM = take(B * Mc * Hg * N * P * 4);
    w.dX = take(B * L * Hg * P * 4);
    w.ddt = take(B * L * Hg * 4);
    w.dB = take(B * L * N * 4);
    w.dC = take(B * L * N * 4);
    w.total = o;
    return w;
}

// One group's slice of rows: `rows` rows of `row` bytes, `pitch` bytes apart in the
// full array, starting `off` bytes in; packed (pitch = row) in the group buffer.
struct Slice {
    i64 rows, row, pitch, off;
};
cudaError_t gather(void* dst, const void* src, Slice s, cudaStream_t st) {
    return dart::launch_copy_rows(dst, s.row, (const uint8_t*)src + s.off, s.pitch, s.row, s.rows, st);
}
cudaError_t scatter(void* dst, const void* src, Slice s, cudaStream_t st) {
    return dart::launch_copy_rows((uint8_t*)dst + s.off, s.pitch, src, s.row, s.row, s.rows, st);
}

cudaError_t sma_backward_grouped(const dart_dims* d, const dart::SmaBwdArgs& f, void* ws,
                                 unsigned long long lim, cudaStream_t st) {
    const i64 B = d->batch, L = d->seqlen, H = d->nheads, G = d->ngroups, Hg = H / G, P = d->headdim,
              N = d->dstate, Mc = d->seqlen / d->chunk;
    const i64 em = d->mem_dtype == DART_F32 ? 4 : 2, ei = 2;
    const SmaBwdGroupWs w = sma_bwd_group_ws(d);
    uint8_t* b = (uint8_t*)ws;
    const dart_dims gd = group_dims(d);
    dart::SmaBwdArgs a = sma_bwd_args(&gd);
    a.test_withhold = f.test_withhold;
    a.M = b + w.M; a.rM = f.rM != nullptr ? (const float*)(b + w.rM) : nullptr;
    a.Q = b + w.Q; a.Cm = b + w.C; a.E = b + w.E; a.z = b + w.z; a.lse = (const float*)(b + w.lse);
    a.dY = b + w.dY; a.logits = f.logits != nullptr ? (const float*)(b + w.logits) : nullptr;
    a.dM = (float*)(b + w.dM); a.dQ = (float*)(b + w.dQ); a.dC = (float*)(b + w.dC);
    a.dE = (float*)(b + w.dE); a.dz = (float*)(b + w.dz);
    cudaError_t e = cudaSuccess;
    for (i64 g = 0; g < G && e == cudaSuccess; ++g) {
        const i64 h0 = g * Hg;
        const Slice mem{B * Mc, Hg * N * P * em, H * N * P * em, h0 * N * P * em};
        const Slice rms{B * Mc, Hg * N * 4, H * N * 4, h0 * N * 4};
        const Slice key{B * L, N * ei, G * N * ei, g * N * ei};
        const Slice val{B * L, P * ei, G * P * ei, g * P * ei};
        const Slice head_in{B * L, Hg * ei, H * ei, h0 * ei};
        const Slice head_f32{B * L, Hg * 4, H * 4, h0 * 4};
        const Slice row_in{B * L, Hg * P * ei, H * P * ei, h0 * P * ei};
        const Slice lgt{B, Hg * Mc * L * 4, H * Mc * L * 4, h0 * Mc * L * 4};
        const Slice dmem{B * Mc, Hg * N * P * 4, H * N * P * 4, h0 * N * P * 4};
        const Slice dkey{B * L, N * 4, G * N * 4, g * N * 4};
        const Slice dval{B * L, P * 4, G * P * 4, g * P * 4};
        if ((e = gather((void*)a.M, f.M, mem, st)) != cudaSuccess ||
            (f.rM != nullptr && (e = gather((void*)a.rM, f.rM, rms, st)) != cudaSuccess) ||
            (e = gather((void*)a.Q, f.Q, key, st)) != cudaSuccess ||
            (e = gather((void*)a.Cm, f.Cm, key, st)) != cudaSuccess ||
            (e = gather((void*)a.E, f.E, val, st)) != cudaSuccess ||
            (e = gather((void*)a.z, f.z, head_in, st)) != cudaSuccess ||
            (e = gather((void*)a.lse, f.lse, head_f32, st)) != cudaSuccess ||
            (e = gather((void*)a.dY, f.dY, row_in, st)) != cudaSuccess ||
            (f.logits != nullptr && (e = gather((void*)a.logits, f.logits, lgt, st)) != cudaSuccess))
            break;
        e = d->mem_dtype == DART_F32 ? dart::launch_sma_backward_tc<float>(a, b + w.tc, lim, st)
                                     : dart::launch_sma_backward_tc<__nv_bfloat16>(a, b + w.tc, lim, st);
        if (e != cudaSuccess) break;
        if ((e = scatter(f.dM, a.dM, dmem, st)) != cudaSuccess || (e = scatter(f.dQ, a.dQ, dkey, st)) != cudaSuccess ||
            (e = scatter(f.dC, a.dC, dkey, st)) != cudaSuccess || (e = scatter(f.dE, a.dE, dval, st)) != cudaSuccess ||
            (e = scatter(f.dz, a.dz, head_f32, st)) != cudaSuccess)
            break;
    }
    return e;
}

cudaError_t scan_backward_grouped(const dart_dims* d, const dart::ScanBwdArgs& f, void* ws,
                                  unsigned long long lim, cudaStream_t st) {
    const i64 B = d->batch, L = d->seqlen, H = d->nheads, G = d->ngroups, Hg = H / G, P = d->headdim,
              N = d->dstate, Mc = d->seqlen / d->chunk;
    const ScanBwdGroupWs w = scan_bwd_group_ws(d);
    uint8_t* b = (uint8_t*)ws;
    dart::ScanBwdArgs a{};
    dart::ScanArgs& g1 = a.fwd;
    g1 = f.fwd;
    g1.H = Hg; g1.G = 1;
    g1.X = b + w.X; g1.dt = (const float*)(b + w.dt); g1.Bm = b + w.Bm; g1.Cm = b + w.Cm;
    a.dY = b + w.dY; a.dM = f.dM != nullptr ? (const float*)(b + w.dM) : nullptr;
    a.dX = (float*)(b + w.dX); a.ddt = (float*)(b + w.ddt); a.dB = (float*)(b + w.dB); a.dC = (float*)(b + w.dC);
    a.accumulate_dC = true;  // onto the caller's dC block, copied in below
    cudaError_t e = cudaSuccess;
    for (i64 g = 0; g < G && e == cudaSuccess; ++g) {
        const i64 h0 = g * Hg;
        const Slice row_in{B * L, Hg * P * 2, H * P * 2, h0 * P * 2};
        const Slice row_f32{B * L, Hg * P * 4, H * P * 4, h0 * P * 4};
        const Slice head_f32{B * L, Hg * 4, H * 4, h0 * 4};
        const Slice key{B * L, N * 2, G * N * 2, g * N * 2};
        const Slice dkey{B * L, N * 4, G * N * 4, g * N * 4};
        const Slice dmem{B * Mc, Hg * N * P * 4, H * N * P * 4, h0 * N * P * 4};
        g1.A = f.fwd.A + h0;
        a.dA = f.dA + h0;
        if ((e = gather((void*)g1.X, f.fwd.X, row_in, st)) != cudaSuccess ||
            (e = gather((void*)g1.dt, f.fwd.dt, head_f32, st)) != cudaSuccess ||
            (e = gather((void*)g1.Bm, f.fwd.Bm, key, st)) != cudaSuccess ||
            (e = gather((void*)g1.Cm, f.fwd.Cm, key, st)) != cudaSuccess ||
            (e = gather((void*)a.dY, f.dY, row_in, st)) != cudaSuccess ||
            (f.dM != nullptr && (e = gather((void*)a.dM, f.dM, dmem, st)) != cudaSuccess) ||
            (e = gather(a.dC, f.dC, dkey, st)) != cudaSuccess)
            break;
        if ((e = dart::launch_chunk_scan_backward<__nv_bfloat16>(a, b + w.tc, lim, st)) != cudaSuccess) break;
        if ((e = scatter(f.dX, a.dX, row_f32, st)) != cudaSuccess ||
            (e = scatter(f.ddt, a.ddt, head_f32, st)) != cudaSuccess ||
            (e = scatter(f.dB, a.dB, dkey, st)) != cudaSuccess || (e = scatter(f.dC, a.dC, dkey, st)) != cudaSuccess)
            break;
    }
    return e;
}

// Workspace of the SMA forward for L % S == 0.
size_t sma_ws_aligned(const dart_dims* d) {
    const i64 M = d->seqlen / d->chunk;
    if (sma_uses_tc(d)) return align256(dart::sma_tc_workspace(d->batch, M, d->nheads));
    return align256((size_t)(d->batch * M * d->nheads * d->dstate) * sizeof(float));
}

// Ragged sequences (L % S != 0). The scan and SMA run unchanged on copies of their
// token inputs zero-padded to Lp = ceil(L / S) S tokens. A padded token has dt = 0, so
// its decay is exp(0 A) = 1 and its write term dt B^T X is zero: every state, the
// final state and every memory are those of the L-token sequence (the last memory
// holds the partial chunk, whose last token is L - 1), and the first L rows of each
// output are the outputs. A padded token reads the memories of the chunks before it
// like any other, but its outputs are dropped.
bool is_ragged(const dart_dims* d) { return d->seqlen % d->chunk != 0; }
dart_dims padded_dims(const dart_dims* d) {
    dart_dims p = *d;
    p.seqlen = (d->seqlen + d->chunk - 1) / d->chunk * d->chunk;
    return p;
}
size_t dtype_size(int t) { return t == DART_F32 ? 4 : 2; }

// Padded copies of the scan's inputs and output, then the aligned scan workspace.
struct RaggedScanWs {
    size_t x, dt, b, c, y, inner, inner_bytes, total;
};
RaggedScanWs ragged_scan_ws(const dart_dims* d) {
    const dart_dims p = padded_dims(d);
    const size_t rows = (size_t)(p.batch * p.seqlen), ei = dtype_size(d->in_dtype), eo = dtype_size(d->out_dtype);
    RaggedScanWs w{};
    size_t o = 0;
    auto take = [&o](size_t bytes) { const size_t at = o; o += align256(bytes); return at; };
    w.x = take(rows * d->nheads * d->headdim * ei);
    w.dt = take(rows * d->nheads * 4);
    w.b = take(rows * d->ngroups * d->dstate * ei);
    w.c = take(rows * d->ngroups * d->dstate * ei);
    w.y = take(rows * d->nheads * d->headdim * eo);
    w.inner_bytes = scan_ws(&p).total;
    w.inner = take(w.inner_bytes);
    w.total = o;
    return w;
}
size_t scan_ws_bytes(const dart_dims* d) { return is_ragged(d) ? ragged_scan_ws(d).total : scan_ws(d).total; }

// Padded copies of the SMA forward's token inputs and outputs, then its aligned workspace.
struct RaggedSmaWs {
    size_t q, c, e, z, yssd, y, r, lse, inner, inner_bytes, total;
};
RaggedSmaWs ragged_sma_ws(const dart_dims* d) {
    const dart_dims p = padded_dims(d);
    const size_t rows = (size_t)(p.batch * p.seqlen), ei = dtype_size(d->in_dtype), eo = dtype_size(d->out_dtype);
    RaggedSmaWs w{};
    size_t o = 0;
    auto take = [&o](size_t bytes) { const size_t at = o; o += align256(bytes); return at; };
    w.q = take(rows * d->ngroups * d->dstate * ei);
    w.c = take(rows * d->ngroups * d->dstate * ei);
    w.e = take(rows * d->ngroups * d->headdim * ei);
    w.z = take(rows * d->nheads * ei);
    w.yssd = take(rows * d->nheads * d->headdim * eo);
    w.y = take(rows * d->nheads * d->headdim * eo);
    w.r = take(rows * d->nheads * d->headdim * eo);
    w.lse = take(rows * d->nheads * 4);
    w.inner_bytes = sma_ws_aligned(&p);
    w.inner = take(w.inner_bytes);
    w.total = o;
    return w;
}
size_t sma_ws(const dart_dims* d) { return is_ragged(d) ? ragged_sma_ws(d).total : sma_ws_aligned(d); }

// dst: Bsz blocks of rows_dst rows; src: Bsz blocks of rows_src <= rows_dst rows of row_bytes
// each. Copies the rows and zeroes the rest of each block (pad) or copies the first
// rows_dst rows of each source block (unpad, rows_dst <= rows_src).
cudaError_t pad_rows(void* dst, const void* src, int64_t bsz, int64_t rows_src, int64_t rows_dst,
                     size_t row_bytes, cudaStream_t s) {
    cudaError_t e = cudaMemcpy2DAsync(dst, rows_dst * row_bytes, src, rows_src * row_bytes, rows_src * row_bytes,
                                      (size_t)bsz, cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess || rows_dst == rows_src) return e;
    return cudaMemset2DAsync((uint8_t*)dst + rows_src * row_bytes, rows_dst * row_bytes, 0,
                             (rows_dst - rows_src) * row_bytes, (size_t)bsz, s);
}
cudaError_t unpad_rows(void* dst, const void* src, int64_t bsz, int64_t rows_src, int64_t rows_dst,
                       size_t row_bytes, cudaStream_t s) {
    return cudaMemcpy2DAsync(dst, rows_dst * row_bytes, src, rows_src * row_bytes, rows_dst * row_bytes,
                             (size_t)bsz, cudaMemcpyDeviceToDevice, s);
}

std::atomic<unsigned long long> g_wait_limit_ns{2000000000ull};
std::atomic<int> g_test_withhold{0};

std::atomic<uint64_t> g_launches{0};

// ------------------------------------------------ host-buffer prefill layout
constexpr int kMaxHostGroups = 64;
constexpr int kHostComp = 3;  // compute streams of dart_prefill_host (groups take them in turn)

size_t dtype_bytes(int t) { return t == DART_F32 ? 4 : 2; }

// Heads of each copy/compute group of dart_prefill_host: groups of 4 heads for
// G = 1 with H a multiple of 4 above 4 (at most 64 groups), else one group of all
// heads. Small groups start the first kernels after a short copy-in and leave a
// short copy-out after the last; three compute streams run neighbouring groups'
// kernels side by side, which makes up for the small grids of 4-head kernels.
// Returns the group count.
int host_groups(const dart_dims* d, int64_t* gh) {
    const int64_t H = d->nheads;
    if (d->ngroups != 1 || H <= 4 || H % 4 != 0 || H / 4 > kMaxHostGroups) {
        gh[0] = H;
        return 1;
    }
    for (int64_t g = 0; g < H / 4; ++g) gh[g] = 4;
    return (int)(H / 4);
}

// Device workspace of dart_prefill_host: the shared inputs, then per group its X,
// dt, z, Y_ssd, Y, memories and r (every group sized for the largest), then one
// scan workspace and one set of SMA tiles (or SMA workspace) per compute stream
// (groups take the compute streams in turn).
struct HostLayout {
    int64_t groups, hmax;
    int nc;  // compute streams in use
    int64_t gh[kMaxHostGroups], gfirst[kMaxHostGroups];  // heads of each group, its first head
    size_t bm, cm, q, e, dt, z, a;          // shared inputs
    size_t g0, stride;                      // first group, bytes per group
    size_t x, dtg, zg, yssd, y, m, rm;      // offsets inside a group
    size_t scan_ws[kHostComp], scan_bytes, sma_ws[kHostComp], sma_bytes;
    size_t tiles[kHostComp], tiles_bytes;  // the SMA's operand tiles from the scan (0: not on this shape)
    size_t total;
};

HostLayout host_layout(const dart_dims* d) {
    HostLayout h{};
    const int64_t B = d->batch, L = d->seqlen, H = d->nheads, G = d->ngroups, P = d->headdim;
    const int64_t N = d->dstate, M = (L + d->chunk - 1) / d->chunk;
    h.groups = host_groups(d, h.gh);
    for (int64_t g = 0, h0 = 0; g < h.groups; h0 += h.gh[g], ++g) {
        h.gfirst[g] = h0;
        h.hmax = std::max(h.hmax, h.gh[g]);
    }
    const size_t ei = dtype_bytes(d->in_dtype), em = dtype_bytes(d->mem_dtype);
    const size_t eo = dtype_bytes(d->out_dtype);
    const size_t rows = (size_t)(B * L);
    size_t o = 0;
    auto take = [&o](size_t bytes) {
        const size_t at = o;
        o += align256(bytes);
        return at;
    };
    h.bm = take(rows * G * N * ei);
    h.cm = take(rows * G * N * ei);
    h.q = take(rows * G * N * ei);
    h.e = take(rows * G * P * ei);
    h.dt = take(rows * H * 4);
    h.z = take(rows * H * ei);
    h.a = take((size_t)H * 4);
    h.g0 = o;
    const size_t hg = (size_t)h.hmax;
    h.x = take(rows * hg * P * ei) - h.g0;
    h.dtg = take(rows * hg * 4) - h.g0;
    h.zg = take(rows * hg * ei) - h.g0;
    h.yssd = take(rows * hg * P * eo) - h.g0;
    h.y = take(rows * hg * P * eo) - h.g0;
    h.m = take((size_t)(B * M) * hg * N * P * em) - h.g0;
    h.rm = take((size_t)(B * M) * hg * N * 4) - h.g0;
    h.stride = o - h.g0;
    o = h.g0 + (size_t)h.groups * h.stride;
    // workspaces for the largest group (their sizes grow with the heads); the tiles
    // only where every group's shape takes them
    dart_dims dg = *d;
    dg.nheads = h.hmax;
    h.scan_bytes = scan_ws_bytes(&dg);
    h.tiles_bytes = dart_sma_tiles_size(&dg);
    for (int64_t g = 0; g < h.groups && h.tiles_bytes > 0; ++g) {
        dart_dims dk = *d;
        dk.nheads = h.gh[g];
        if (dart_sma_tiles_size(&dk) == 0) h.tiles_bytes = 0;
    }
    h.sma_bytes = h.tiles_bytes > 0 ? 0 : sma_ws(&dg);  // the tiles replace the SMA's workspace
    h.nc = (int)std::min<int64_t>(kHostComp, h.groups);
    for (int k = 0; k < h.nc; ++k) {
        h.scan_ws[k] = take(h.scan_bytes);
        h.sma_ws[k] = take(h.sma_bytes);
        h.tiles[k] = take(h.tiles_bytes);
    }
    h.total = o;
    return h;
}

// The streams of dart_prefill_host (copy in, kHostComp for the kernels, copy out)
// for the current device, created on first use and kept.
struct HostStreams {
    cudaStream_t in = nullptr, comp[kHostComp] = {}, out = nullptr;
};
std::mutex g_host_mu;
HostStreams g_host_streams[64];

cudaError_t host_streams(HostStreams** hs) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_host_mu);
    HostStreams& s = g_host_streams[dev];
    if (s.in == nullptr) {
        cudaStream_t t[kHostComp + 2];
        for (int i = 0; i < kHostComp + 2; ++i)
            if ((e = cudaStreamCreateWithFlags(&t[i], cudaStreamNonBlocking)) != cudaSuccess) return e;
        s.in = t[0];
        for (int k = 0; k < kHostComp; ++k) s.comp[k] = t[1 + k];
        s.out = t[kHostComp + 1];
    }
    *hs = &s;
    return cudaSuccess;
}

// Workspace of dart_block_forward: the in-projection output, the hot path's inputs
// and outputs, the normalised output, then the scan and SMA workspaces.
struct BlockWs {
    int64_t ldz, d_in;
    size_t zx, x, bm, cm, dt, a, q, e, gate, yssd, y, mem, rm, yn, scan, scan_bytes, sma, sma_bytes;
    size_t tiles, tiles_bytes;  // the SMA's operand tiles from the scan (0: not on this shape)
    size_t total;
};
dart_dims block_core(const dart_block_dims* b) {
    dart_dims c = b->core;
    c.in_dtype = DART_BF16;
    c.mem_dtype = DART_F32;
    c.out_dtype = DART_F32;
    return c;
}
BlockWs block_ws(const dart_block_dims* b) {
    const dart_dims c = block_core(b);
    const int64_t T = c.batch * c.seqlen, H = c.nheads, di = H * c.headdim, GN = c.ngroups * c.dstate;
    const int64_t GP = c.ngroups * c.headdim, Mc = (c.seqlen + c.chunk - 1) / c.chunk;
    BlockWs w{};
    w.d_in = 2 * di + 3 * GN + H + GP + 1;
    w.ldz = (w.d_in + 7) / 8 * 8;
    size_t o = 0;
    auto take = [&o](size_t bytes) { const size_t at = o; o += align256(bytes); return at; };
    w.zx = take((size_t)(T * w.ldz) * 4);
    w.x = take((size_t)(T * di) * 2);
    w.bm = take((size_t)(T * GN) * 2);
    w.cm = take((size_t)(T * GN) * 2);
    w.dt = take((size_t)(T * H) * 4);
    w.a = take((size_t)H * 4);
    w.q = take((size_t)(T * GN) * 2);
    w.e = take((size_t)(T * GP) * 2);
    w.gate = take((size_t)(T * H) * 2);
    w.yssd = take((size_t)(T * di) * 4);
    w.y = take((size_t)(T * di) * 4);
    w.mem = take((size_t)(c.batch * Mc * H * c.dstate * c.headdim) * 4);
    w.rm = take((size_t)(c.batch * Mc * H * c.dstate) * 4);
    w.yn = take((size_t)(T * di) * 2);
    w.scan_bytes = scan_ws_bytes(&c);
    w.scan = take(w.scan_bytes);
    w.tiles_bytes = dart_sma_tiles_size(&c);
    w.sma_bytes = w.tiles_bytes > 0 ? 0 : sma_ws(&c);  // the tiles replace the SMA's workspace
    w.sma = take(w.sma_bytes);
    w.tiles = take(w.tiles_bytes);
    w.total = o;
    return w;
}
dart_status check_block(const dart_block_dims* b) {
    if (b == nullptr) return DART_ERR_INVALID_ARG;
    if (b->core.in_dtype != DART_BF16) return DART_ERR_UNSUPPORTED;
    if (b->core.out_dtype != DART_F32 && b->core.out_dtype != DART_BF16) return DART_ERR_INVALID_ARG;
    const dart_dims c = block_core(b);
    const dart_status st = check_dims(&c, true, true);
    if (st != DART_OK) return st;
    if (b->d_model <= 0 || !(b->norm_eps > 0.0f) || !dart::block_conv_width_ok(b->conv_width))
        return DART_ERR_INVALID_ARG;
    if (b->d_model % 8 != 0 || c.nheads % 8 != 0 || c.nheads * c.headdim > 4096) return DART_ERR_UNSUPPORTED;
    return DART_OK;
}

}  // namespace

namespace dart {
void note_launches(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }
dart_status validate_dims(const dart_dims* d, bool need_seqlen) { return check_dims(d, need_seqlen); }
dart_status record_cuda_error(cudaError_t e) { return cuda_fail(e); }
}  // namespace dart

extern "C" {

uint64_t dart_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }


const char* dart_status_string(dart_status s) {
    switch (s) {
        case DART_OK: return "DART_OK";
        case DART_ERR_INVALID_ARG: return "DART_ERR_INVALID_ARG: invalid argument";
        case DART_ERR_UNSUPPORTED: return "DART_ERR_UNSUPPORTED: valid but unsupported sizes or dtypes";
        case DART_ERR_WORKSPACE: return "DART_ERR_WORKSPACE: workspace missing, misaligned or too small";
        case DART_ERR_CUDA: return "DART_ERR_CUDA: a CUDA call failed (see dart_last_cuda_error)";
        case DART_ERR_TIMEOUT: return "DART_ERR_TIMEOUT: a device-side wait gave up";
        case DART_ERR_TOO_LARGE:
            return "DART_ERR_TOO_LARGE: problem exceeds the fixed scratch of dart_sma_forward_noalloc";
    }
    return "unknown dart_status";
}

int dart_last_cuda_error(void) { return t_last_cuda_error; }

size_t dart_workspace_size(const dart_dims* d, int op) {
    switch (op) {
        case DART_OP_CHUNK_SCAN:
            if (check_dims(d, true, true) != DART_OK) return 0;
            return scan_ws_bytes(d);
        case DART_OP_SMA_FORWARD:
            if (check_dims(d, true, true) != DART_OK) return 0;
            return sma_ws(d);
        case DART_OP_DECODE_STEP:
            return 0;
        case DART_OP_PREFILL_HOST:
            if (check_dims(d, true, true) != DART_OK) return 0;
            return host_layout(d).total;
        case DART_OP_SMA_BACKWARD:
            if (check_dims(d, true) != DART_OK) return 0;
            if (sma_bwd_uses_tc(d))
                return align256(dart::sma_bwd_tc_workspace(d->batch, d->seqlen, d->nheads,
                                                           d->seqlen / d->chunk, d->dstate));
            if (sma_bwd_grouped(d)) return sma_bwd_group_ws(d).total;
            return align256(dart::sma_bwd_workspace(d->batch, d->seqlen, d->nheads,
                                                    d->seqlen / d->chunk, d->dstate));
        case DART_OP_SCAN_BACKWARD: {
            if (check_dims(d, true) != DART_OK) return 0;
            dart::ScanArgs a{};
            a.B = d->batch; a.L = d->seqlen; a.H = d->nheads; a.G = d->ngroups;
            a.P = d->headdim; a.N = d->dstate; a.S = d->chunk;
            if (d->in_dtype == DART_BF16 && dart::scan_bwd_tc_supported(a))
                return align256(dart::scan_bwd_tc_workspace(d->batch, d->seqlen, d->nheads, d->chunk));
            if (scan_bwd_grouped(d)) return scan_bwd_group_ws(d).total;
            return align256(dart::scan_bwd_workspace(d->batch, d->seqlen, d->nheads, d->dstate,
                                                     d->headdim, d->chunk));
        }
    }
    return 0;
}

static dart_status chunk_scan_impl(const dart_dims* d, const void* X, const float* dt, const float* A,
                                   const void* Bm, const void* Cm, void* Y_ssd, void* M, float* rM,
                                   float* final_state, uint8_t* tiles, void* ws, size_t ws_bytes,
                                   void* stream) {
    dart_status st = check_dims(d, true, true);
    if (st != DART_OK) return st;
    const void* req[] = {X, dt, A, Bm, Cm, Y_ssd, M};
    for (const void* p : req)
        if (p == nullptr || !aligned16(p)) return DART_ERR_INVALID_ARG;
    if ((rM && !aligned16(rM)) || (final_state && !aligned16(final_state)))
        return DART_ERR_INVALID_ARG;
    if (is_ragged(d)) {  // zero-padded copies, the aligned scan, the first L rows of Y_ssd
        const RaggedScanWs w = ragged_scan_ws(d);
        if (ws == nullptr || ((uintptr_t)ws & 255u) != 0 || ws_bytes < w.total) return DART_ERR_WORKSPACE;
        const dart_dims p = padded_dims(d);
        uint8_t* b = (uint8_t*)ws;
        cudaStream_t s = (cudaStream_t)stream;
        const size_t ei = dtype_size(d->in_dtype), eo = dtype_size(d->out_dtype);
        const int64_t L = d->seqlen, Lp = p.seqlen, H = d->nheads, P = d->headdim, GN = d->ngroups * d->dstate;
        cudaError_t e;
        if ((e = pad_rows(b + w.x, X, d->batch, L, Lp, H * P * ei, s)) != cudaSuccess ||
            (e = pad_rows(b + w.dt, dt, d->batch, L, Lp, H * 4, s)) != cudaSuccess ||
            (e = pad_rows(b + w.b, Bm, d->batch, L, Lp, GN * ei, s)) != cudaSuccess ||
            (e = pad_rows(b + w.c, Cm, d->batch, L, Lp, GN * ei, s)) != cudaSuccess)
            return cuda_fail(e);
        st = dart_chunk_scan(&p, b + w.x, (const float*)(b + w.dt), A, b + w.b, b + w.c, b + w.y, M, rM,
                             final_state, b + w.inner, w.inner_bytes, stream);
        if (st != DART_OK) return st;
        e = unpad_rows(Y_ssd, b + w.y, d->batch, Lp, L, H * P * eo, s);
        return e == cudaSuccess ? DART_OK : cuda_fail(e);
    }
    const ScanWs w = scan_ws(d);
    if (ws == nullptr || ((uintptr_t)ws & 255u) != 0 || ws_bytes < w.total)
        return DART_ERR_WORKSPACE;

    dart::ScanArgs a{};
    a.B = d->batch; a.L = d->seqlen; a.H = d->nheads; a.G = d->ngroups;
    a.P = d->headdim; a.N = d->dstate; a.S = d->chunk; a.eps = d->eps;
    a.X = X; a.dt = dt; a.A = A; a.Bm = Bm; a.Cm = Cm; a.Y = Y_ssd; a.M = M; a.rM = rM;
    a.final_state = final_state;
    a.test_withhold = g_test_withhold.load();
    a.cum = (float*)((char*)ws + w.cum_off);
    a.dH32 = (float*)((char*)ws + w.dh_off);
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e;
    if (scan_uses_tc(d)) {
        a.Hops = (uint8_t*)ws + w.hops_off;
        a.sma_tiles = tiles;
        typedef __nv_bfloat16 bf;
        const unsigned long long lim = g_wait_limit_ns.load();
        if (d->mem_dtype == DART_F32)
            e = dart::launch_chunk_scan_tc<float, float>(a, lim, s);
        else if (d->out_dtype == DART_F32)
            e = dart::launch_chunk_scan_tc<bf, float>(a, lim, s);
        else
            e = dart::launch_chunk_scan_tc<bf, bf>(a, lim, s);
    } else {
        e = dispatch<ScanL>(d, a, s);
    }
    return e == cudaSuccess ? DART_OK : cuda_fail(e);
}

dart_status dart_chunk_scan(const dart_dims* d, const void* X, const float* dt, const float* A,
                            const void* Bm, const void* Cm, void* Y_ssd, void* M, float* rM,
                            float* final_state, void* ws, size_t ws_bytes, void* stream) {
    return chunk_scan_impl(d, X, dt, A, Bm, Cm, Y_ssd, M, rM, final_state, nullptr, ws, ws_bytes, stream);
}

// The SMA operand tiles built by the scan: both calls on their tensor-core paths,
// whole chunks.
static bool tiles_supported(const dart_dims* d) {
    return check_dims(d, true) == DART_OK && scan_uses_tc(d) && sma_uses_tc(d);
}

size_t dart_sma_tiles_size(const dart_dims* d) {
    if (!tiles_supported(d)) return 0;
    return dart::sma_tiles_bytes(d->batch, d->seqlen / d->chunk, d->nheads);
}

dart_status dart_chunk_scan_with_tiles(const dart_dims* d, const void* X, const float* dt, const float* A,
                                       const void* Bm, const void* Cm, void* Y_ssd, void* M, float* rM,
                                       float* final_state, void* tiles, void* ws, size_t ws_bytes,
                                       void* stream) {
    dart_status st = check_dims(d, true);
    if (st != DART_OK) return st;
    if (!tiles_supported(d)) return DART_ERR_UNSUPPORTED;
    if (tiles == nullptr || ((uintptr_t)tiles & 255u) != 0) return DART_ERR_INVALID_ARG;
    return chunk_scan_impl(d, X, dt, A, Bm, Cm, Y_ssd, M, rM, final_state, (uint8_t*)tiles, ws, ws_bytes,
                           stream);
}

dart_status dart_sma_forward_with_tiles(const dart_dims* d, const void* tiles, const void* Q, const void* Cm,
                                        const void* E, const void* z, const void* Y_ssd, void* Y, void* R,
                                        float* lse, void* stream) {
    dart_status st = check_dims(d, true);
    if (st != DART_OK) return st;
    if (!tiles_supported(d)) return DART_ERR_UNSUPPORTED;
    if (tiles == nullptr || ((uintptr_t)tiles & 255u) != 0) return DART_ERR_INVALID_ARG;
    const void* req[] = {Q, Cm, E, z, Y_ssd, Y};
    for (const void* p : req)
        if (p == nullptr || !aligned16(p)) return DART_ERR_INVALID_ARG;
    if ((R && !aligned16(R)) || (lse && !aligned16(lse))) return DART_ERR_INVALID_ARG;
    dart::SmaArgs a = sma_args(d);
    a.M = nullptr; a.rM = nullptr; a.Q = Q; a.Cm = Cm; a.E = E; a.z = z; a.Yssd = Y_ssd; a.Y = Y;
    a.R = R; a.lse = lse; a.tiles = (const uint8_t*)tiles;
    a.test_withhold = g_test_withhold.load();
    const unsigned long long lim = g_wait_limit_ns.load();
    cudaStream_t s = (cudaStream_t)stream;
    typedef __nv_bfloat16 bf;
    cudaError_t e;
    if (d->mem_dtype == DART_F32)
        e = dart::launch_sma_forward_tc<float, float>(a, nullptr, lim, s);
    else if (d->out_dtype == DART_F32)
        e = dart::launch_sma_forward_tc<bf, float>(a, nullptr, lim, s);
    else
        e = dart::launch_sma_forward_tc<bf, bf>(a, nullptr, lim, s);
    return e == cudaSuccess ? DART_OK : cuda_fail(e);
}

static dart_status sma_forward_impl(const dart_dims* d, const void* M, const float* rM, const void* Q,
                                    const void* Cm, const void* E, const void* z, const void* Y_ssd,
                                    void* Y, void* R, float* lse, float* logits, void* ws,
                                    size_t ws_bytes, void* stream) {
    dart_status st = check_dims(d, true, logits == nullptr);
    if (st != DART_OK) return st;
    const void* req[] = {M, Q, Cm, E, z, Y_ssd, Y};
    for (const void* p : req)
        if (p == nullptr || !aligned16(p)) return DART_ERR_INVALID_ARG;
    if ((rM && !aligned16(rM)) || (R && !aligned16(R)) || (lse && !aligned16(lse)) ||
        (logits && !aligned16(logits)))
        return DART_ERR_INVALID_ARG;
    if (is_ragged(d)) {  // zero-padded copies, the aligned call, the first L rows of each output
        const RaggedSmaWs w = ragged_sma_ws(d);
        if (ws == nullptr || ((uintptr_t)ws & 255u) != 0 || ws_bytes < w.total) return DART_ERR_WORKSPACE;
        const dart_dims p = padded_dims(d);
        uint8_t* b = (uint8_t*)ws;
        cudaStream_t s = (cudaStream_t)stream;
        const size_t ei = dtype_size(d->in_dtype), eo = dtype_size(d->out_dtype);
        const int64_t L = d->seqlen, Lp = p.seqlen, H = d->nheads, P = d->headdim, G = d->ngroups;
        const size_t nrow = (size_t)(G * d->dstate) * ei, erow = (size_t)(G * P) * ei, yrow = (size_t)(H * P) * eo;
        cudaError_t e;
        if ((e = pad_rows(b + w.q, Q, d->batch, L, Lp, nrow, s)) != cudaSuccess ||
            (e = pad_rows(b + w.c, Cm, d->batch, L, Lp, nrow, s)) != cudaSuccess ||
            (e = pad_rows(b + w.e, E, d->batch, L, Lp, erow, s)) != cudaSuccess ||
            (e = pad_rows(b + w.z, z, d->batch, L, Lp, (size_t)H * ei, s)) != cudaSuccess ||
            (e = pad_rows(b + w.yssd, Y_ssd, d->batch, L, Lp, yrow, s)) != cudaSuccess)
            return cuda_fail(e);
        st = sma_forward_impl(&p, M, rM, b + w.q, b + w.c, b + w.e, b + w.z, b + w.yssd, b + w.y,
                              R ? b + w.r : nullptr, lse ? (float*)(b + w.lse) : nullptr, nullptr, b + w.inner,
                              w.inner_bytes, stream);
        if (st != DART_OK) return st;
        if ((e = unpad_rows(Y, b + w.y, d->batch, Lp, L, yrow, s)) != cudaSuccess ||
            (R && (e = unpad_rows(R, b + w.r, d->batch, Lp, L, yrow, s)) != cudaSuccess) ||
            (lse && (e = unpad_rows(lse, b + w.lse, d->batch, Lp, L, (size_t)H * 4, s)) != cudaSuccess))
            return cuda_fail(e);
        return DART_OK;
    }
    const bool tc = sma_uses_tc(d);
    if (logits != nullptr && !tc) return DART_ERR_UNSUPPORTED;  // saved by the tensor-core kernel only
    const size_t need = (tc || rM == nullptr) ? sma_ws_aligned(d) : 0;
    if (need > 0 && (ws == nullptr || ((uintptr_t)ws & 255u) != 0 || ws_bytes < need))
        return DART_ERR_WORKSPACE;

    cudaStream_t s = (cudaStream_t)stream;
    if (tc) {
        dart::SmaArgs a = sma_args(d);
        a.M = M; a.rM = rM; a.Q = Q; a.Cm = Cm; a.E = E; a.z = z; a.Yssd = Y_ssd; a.Y = Y;
        a.R = R; a.lse = lse; a.logits = logits;
        a.test_withhold = g_test_withhold.load();
        const unsigned long long lim = g_wait_limit_ns.load();
        typedef __nv_bfloat16 bf;
        cudaError_t e;
        if (d->mem_dtype == DART_F32)
            e = dart::launch_sma_forward_tc<float, float>(a, ws, lim, s);
        else if (d->out_dtype == DART_F32)
            e = dart::launch_sma_forward_tc<bf, float>(a, ws, lim, s);
        else
            e = dart::launch_sma_forward_tc<bf, bf>(a, ws, lim, s);
        return e == cudaSuccess ? DART_OK : cuda_fail(e);
    }
    const float* r = rM;
    if (r == nullptr) {
        const i64 rows = d->batch * (d->seqlen / d->chunk) * d->nheads * d->dstate;
        float* rws = (float*)ws;
        cudaError_t e = d->mem_dtype == DART_F32
                            ? dart::launch_memory_rms<float>(M, rws, rows, d->headdim, d->eps, s)
                            : dart::launch_memory_rms<__nv_bfloat16>(M, rws, rows, d->headdim,
                                                                      d->eps, s);
        if (e != cudaSuccess) return cuda_fail(e);
        r = rws;
    }
    dart::SmaArgs a;
    a.B = d->batch; a.L = d->seqlen; a.H = d->nheads; a.G = d->ngroups;
    a.P = d->headdim; a.N = d->dstate; a.S = d->chunk; a.eps = d->eps;
    a.M = M; a.rM = r; a.Q = Q; a.Cm = Cm; a.E = E; a.z = z; a.Yssd = Y_ssd; a.Y = Y; a.R = R;
    a.lse = lse;
    cudaError_t e = dispatch<SmaL>(d, a, s);
    return e == cudaSuccess ? DART_OK : cuda_fail(e);
}

dart_status dart_sma_forward(const dart_dims* d, const void* M, const float* rM, const void* Q,
                             const void* Cm, const void* E, const void* z, const void* Y_ssd,
                             void* Y, void* R, float* lse, void* ws, size_t ws_bytes,
                             void* stream) {
    return sma_forward_impl(d, M, rM, Q, Cm, E, z, Y_ssd, Y, R, lse, nullptr, ws, ws_bytes, stream);
}

dart_status dart_sma_forward_with_logits(const dart_dims* d, const void* M, const float* rM,
                                         const void* Q, const void* Cm, const void* E, const void* z,
                                         const void* Y_ssd, void* Y, void* R, float* lse, float* logits,
                                         void* ws, size_t ws_bytes, void* stream) {
    if (logits == nullptr || lse == nullptr) return DART_ERR_INVALID_ARG;
    return sma_forward_impl(d, M, rM, Q, Cm, E, z, Y_ssd, Y, R, lse, logits, ws, ws_bytes, stream);
}

dart_status dart_prefill_host(const dart_dims* d, const void* X, const float* dt, const float* A,
                              const void* Bm, const void* Cm, const void* Q, const void* E,
                              const void* z, void* Y, void* ws, size_t ws_bytes, void* stream) {
    dart_status st = check_dims(d, true, true);
    if (st != DART_OK) return st;
    const void* req[] = {X, dt, A, Bm, Cm, Q, E, z, Y};
    for (const void* p : req)
        if (p == nullptr) return DART_ERR_INVALID_ARG;
    const HostLayout h = host_layout(d);
    if (ws == nullptr || ((uintptr_t)ws & 255u) != 0 || ws_bytes < h.total) return DART_ERR_WORKSPACE;
    HostStreams* hs = nullptr;
    cudaError_t e = host_streams(&hs);
    if (e != cudaSuccess) return cuda_fail(e);

    const int64_t B = d->batch, L = d->seqlen, H = d->nheads, G = d->ngroups, P = d->headdim;
    const int64_t N = d->dstate;
    const size_t ei = dtype_bytes(d->in_dtype), eo = dtype_bytes(d->out_dtype);
    const size_t rows = (size_t)(B * L);
    uint8_t* w = (uint8_t*)ws;
    cudaStream_t s = (cudaStream_t)stream;
    const int ng = (int)h.groups;
    // events: the start on the caller's stream, per group copy-in and kernels done, the end
    cudaEvent_t start = nullptr, done = nullptr, sma_ev = nullptr, in_ev[kMaxHostGroups] = {},
                comp_ev[kMaxHostGroups] = {};
    // events are released once recorded (the driver frees each when its work is done)
    auto release = [&]() {
        if (start != nullptr) cudaEventDestroy(start);
        if (done != nullptr) cudaEventDestroy(done);
        if (sma_ev != nullptr) cudaEventDestroy(sma_ev);
        for (int g = 0; g < ng; ++g) {
            if (in_ev[g] != nullptr) cudaEventDestroy(in_ev[g]);
            if (comp_ev[g] != nullptr) cudaEventDestroy(comp_ev[g]);
        }
    };
    // on an error after the start: the caller's stream still waits for whatever was
    // enqueued on the library's streams, so that no copy outlives the caller's buffers
    bool started = false;
    auto join = [&]() {
        if (!started) return;
        cudaStream_t own[kHostComp + 2] = {hs->in, hs->out};
        for (int k = 0; k < kHostComp; ++k) own[2 + k] = hs->comp[k];
        for (cudaStream_t x : own) {
            cudaEvent_t ev = nullptr;
            if (cudaEventCreateWithFlags(&ev, cudaEventDisableTiming) == cudaSuccess) {
                if (cudaEventRecord(ev, x) == cudaSuccess) cudaStreamWaitEvent(s, ev, 0);
                cudaEventDestroy(ev);
            } else {
                cudaStreamSynchronize(x);  // no event to be had: wait here instead
            }
        }
    };
    auto fail = [&](cudaError_t err) {
        join();
        release();
        return cuda_fail(err);
    };
    const unsigned fl = cudaEventDisableTiming;
    if ((e = cudaEventCreateWithFlags(&start, fl)) != cudaSuccess) return fail(e);
    if ((e = cudaEventCreateWithFlags(&done, fl)) != cudaSuccess) return fail(e);
    if ((e = cudaEventCreateWithFlags(&sma_ev, fl)) != cudaSuccess) return fail(e);
    for (int g = 0; g < ng; ++g)
        if ((e = cudaEventCreateWithFlags(&in_ev[g], fl)) != cudaSuccess ||
            (e = cudaEventCreateWithFlags(&comp_ev[g], fl)) != cudaSuccess)
            return fail(e);
    // after the caller's earlier work on `stream`
    if ((e = cudaEventRecord(start, s)) != cudaSuccess) return fail(e);
    started = true;
    if ((e = cudaStreamWaitEvent(hs->in, start, 0)) != cudaSuccess) return fail(e);
    for (int k = 0; k < h.nc; ++k)
        if ((e = cudaStreamWaitEvent(hs->comp[k], start, 0)) != cudaSuccess) return fail(e);
    if ((e = cudaStreamWaitEvent(hs->out, start, 0)) != cudaSuccess) return fail(e);
    // shared inputs, one copy each: the scan's first (B, C, dt, A), then, after the
    // first group's X, the SMA's (Q, E, z), which land under the first group's scan
    struct Copy {
        size_t off;
        const void* src;
        size_t bytes;
    };
    const Copy scan_in[] = {{h.bm, Bm, rows * G * N * ei}, {h.cm, Cm, rows * G * N * ei},
                            {h.dt, dt, rows * H * 4}, {h.a, A, (size_t)H * 4}};
    const Copy sma_in[] = {{h.q, Q, rows * G * N * ei}, {h.e, E, rows * G * P * ei}, {h.z, z, rows * H * ei}};
    for (const auto& c : scan_in)
        if ((e = cudaMemcpyAsync(w + c.off, c.src, c.bytes, cudaMemcpyHostToDevice, hs->in)) != cudaSuccess)
            return fail(e);
    for (int g = 0; g < ng; ++g) {
        const int64_t h0 = h.gfirst[g], hg = h.gh[g];
        dart_dims dg = *d;
        dg.nheads = hg;
        const size_t xrow = (size_t)hg * P * ei, yrow = (size_t)hg * P * eo;
        uint8_t* gb = w + h.g0 + (size_t)g * h.stride;
        // copy in: the group's X rows (pitched)
        e = cudaMemcpy2DAsync(gb + h.x, xrow, (const uint8_t*)X + (size_t)h0 * P * ei, (size_t)H * P * ei,
                              xrow, rows, cudaMemcpyHostToDevice, hs->in);
        if (e != cudaSuccess) return fail(e);
        if ((e = cudaEventRecord(in_ev[g], hs->in)) != cudaSuccess) return fail(e);
        if (g == 0) {  // the SMA's shared inputs follow the first group's X
            for (const auto& c : sma_in)
                if ((e = cudaMemcpyAsync(w + c.off, c.src, c.bytes, cudaMemcpyHostToDevice, hs->in)) !=
                    cudaSuccess)
                    return fail(e);
            if ((e = cudaEventRecord(sma_ev, hs->in)) != cudaSuccess) return fail(e);
        }
        // kernels, groups taking the compute streams in turn (so that the kernels
        // of neighbouring groups share the SMs): the group's dt and z
        // columns, the scan, the SMA and merge
        const int k = g % h.nc;
        cudaStream_t cs = hs->comp[k];
        if ((e = cudaStreamWaitEvent(cs, in_ev[g], 0)) != cudaSuccess) return fail(e);
        const float* dtg = (const float*)(w + h.dt);
        const void* zg = w + h.z;
        if (ng > 1) {
            if ((e = dart::launch_gather_heads(w + h.dt, gb + h.dtg, (int64_t)rows, H, h0, hg, 4, cs)) !=
                cudaSuccess)
                return fail(e);
            dtg = (const float*)(gb + h.dtg);
        }
        // the SMA's shared inputs (Q, E, z), then the group's z columns: for the first
        // group after its scan (they land under it), for the others before it (long
        // there by then), so that their SMA kernel directly follows the scan's last
        // kernel and may start under its last wave
        auto sma_inputs = [&]() -> cudaError_t {
            cudaError_t err = cudaStreamWaitEvent(cs, sma_ev, 0);
            if (err == cudaSuccess && ng > 1) {
                err = dart::launch_gather_heads(w + h.z, gb + h.zg, (int64_t)rows, H, h0, hg, (int)ei, cs);
                zg = gb + h.zg;
            }
            return err;
        };
        if (g > 0 && (e = sma_inputs()) != cudaSuccess) return fail(e);
        // the scan writes the SMA's operand tiles where both run on the tensor cores
        uint8_t* tiles = h.tiles_bytes > 0 ? w + h.tiles[k] : nullptr;
        st = chunk_scan_impl(&dg, gb + h.x, dtg, (const float*)(w + h.a) + h0, w + h.bm, w + h.cm,
                             gb + h.yssd, gb + h.m, (float*)(gb + h.rm), nullptr, tiles, w + h.scan_ws[k],
                             h.scan_bytes, cs);
        if (st == DART_OK && g == 0 && (e = sma_inputs()) != cudaSuccess) return fail(e);
        if (st == DART_OK && tiles != nullptr)
            st = dart_sma_forward_with_tiles(&dg, tiles, w + h.q, w + h.cm, w + h.e, zg, gb + h.yssd, gb + h.y,
                                             nullptr, nullptr, cs);
        else if (st == DART_OK)
            st = dart_sma_forward(&dg, gb + h.m, (const float*)(gb + h.rm), w + h.q, w + h.cm, w + h.e, zg,
                                  gb + h.yssd, gb + h.y, nullptr, nullptr, w + h.sma_ws[k], h.sma_bytes, cs);
        if (st != DART_OK) {
            join();
            release();
            return st;
        }
        if ((e = cudaEventRecord(comp_ev[g], cs)) != cudaSuccess) return fail(e);
        // copy out: the group's Y rows (pitched)
        if ((e = cudaStreamWaitEvent(hs->out, comp_ev[g], 0)) != cudaSuccess) return fail(e);
        e = cudaMemcpy2DAsync((uint8_t*)Y + (size_t)h0 * P * eo, (size_t)H * P * eo, gb + h.y, yrow, yrow, rows,
                              cudaMemcpyDeviceToHost, hs->out);
        if (e != cudaSuccess) return fail(e);
    }
    // the caller's stream continues after the last copy out (which follows every kernel)
    if ((e = cudaEventRecord(done, hs->out)) != cudaSuccess) return fail(e);
    if ((e = cudaStreamWaitEvent(s, done, 0)) != cudaSuccess) return fail(e);
    release();
    return DART_OK;
}

dart_status dart_decode_step(const dart_dims* d, int64_t pos, int64_t m_cap, void* cache,
                             float* state, float* partial, const void* x, const float* dt,
                             const float* A, const void* b, const void* c, const void* q,
                             const void* e, const void* z, void* y, float* lse, void* ws,
                             size_t ws_bytes, void* stream) {
    (void)ws;
    (void)ws_bytes;
    dart_status st = check_dims(d, false);
    if (st != DART_OK) return st;
    if (pos < 0 || m_cap < 0 || pos / d->chunk > m_cap) return DART_ERR_INVALID_ARG;
    if (m_cap > 0 && cache == nullptr) return DART_ERR_INVALID_ARG;
    const void* req[] = {state, partial, x, dt, A, b, c, q, e, z, y};
    for (const void* p : req)
        if (p == nullptr || !aligned16(p)) return DART_ERR_INVALID_ARG;
    if ((cache && !aligned16(cache)) || (lse && !aligned16(lse))) return DART_ERR_INVALID_ARG;

    dart::DecodeArgs a;
    a.B = d->batch; a.H = d->nheads; a.G = d->ngroups; a.P = d->headdim; a.N = d->dstate;
    a.S = d->chunk; a.pos = pos; a.m_cap = m_cap; a.eps = d->eps;
    a.cache = cache; a.state = state; a.partial = partial; a.x = x; a.dt = dt; a.A = A;
    a.b = b; a.c = c; a.q = q; a.e = e; a.z = z; a.y = y; a.lse = lse;
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t err = dispatch<DecodeL>(d, a, s);
    return err == cudaSuccess ? DART_OK : cuda_fail(err);
}

static dart_status sma_backward_impl(const dart_dims* d, const void* M, const float* rM, const void* Q,
                                     const void* Cm, const void* E, const void* z, const float* lse,
                                     const float* logits, const void* dY, float* dM, float* dQ, float* dC,
                                     float* dE, float* dz, void* ws, size_t ws_bytes, void* stream) {
    dart_status st = check_dims(d, true);
    if (st != DART_OK) return st;
    const void* req[] = {M, Q, Cm, E, z, lse, dY, dM, dQ, dC, dE, dz};
    for (const void* p : req)
        if (p == nullptr || !aligned16(p)) return DART_ERR_INVALID_ARG;
    if ((rM != nullptr && !aligned16(rM)) || (logits != nullptr && !aligned16(logits)))
        return DART_ERR_INVALID_ARG;
    const size_t need = dart_workspace_size(d, DART_OP_SMA_BACKWARD);
    if (ws == nullptr || ((uintptr_t)ws & 255u) != 0 || ws_bytes < need) return DART_ERR_WORKSPACE;
    dart::SmaBwdArgs a = sma_bwd_args(d);
    a.M = M; a.rM = rM; a.Q = Q; a.Cm = Cm; a.E = E; a.z = z; a.lse = lse; a.dY = dY;
    a.dM = dM; a.dQ = dQ; a.dC = dC; a.dE = dE; a.dz = dz;
    a.logits = logits;  // the CUDA-core path recomputes the logits and ignores them
    a.test_withhold = g_test_withhold.load();
    cudaStream_t s = (cudaStream_t)stream;
    typedef __nv_bfloat16 bf;
    cudaError_t e;
    if (sma_bwd_uses_tc(d)) {
        const unsigned long long lim = g_wait_limit_ns.load();
        if (d->mem_dtype == DART_F32)
            e = dart::launch_sma_backward_tc<float>(a, ws, lim, s);
        else
            e = dart::launch_sma_backward_tc<bf>(a, ws, lim, s);
    } else if (sma_bwd_grouped(d)) {
        e = sma_backward_grouped(d, a, ws, g_wait_limit_ns.load(), s);
    } else if (d->in_dtype == DART_F32 && d->mem_dtype == DART_F32)
        e = dart::launch_sma_backward<float, float>(a, ws, s);
    else if (d->in_dtype == DART_BF16 && d->mem_dtype == DART_F32)
        e = dart::launch_sma_backward<bf, float>(a, ws, s);
    else if (d->in_dtype == DART_BF16 && d->mem_dtype == DART_BF16)
        e = dart::launch_sma_backward<bf, bf>(a, ws, s);
    else
        return DART_ERR_UNSUPPORTED;
    return e == cudaSuccess ? DART_OK : cuda_fail(e);
}

dart_status dart_sma_backward(const dart_dims* d, const void* M, const float* rM, const void* Q,
                              const void* Cm, const void* E, const void* z, const float* lse,
                              const void* dY, float* dM, float* dQ, float* dC, float* dE,
                              float* dz, void* ws, size_t ws_bytes, void* stream) {
    return sma_backward_impl(d, M, rM, Q, Cm, E, z, lse, nullptr, dY, dM, dQ, dC, dE, dz, ws, ws_bytes,
                             stream);
}

dart_status dart_sma_backward_with_logits(const dart_dims* d, const void* M, const float* rM,
                                          const void* Q, const void* Cm, const void* E, const void* z,
                                          const float* lse, const float* logits, const void* dY, float* dM,
                                          float* dQ, float* dC, float* dE, float* dz, void* ws,
                                          size_t ws_bytes, void* stream) {
    if (logits == nullptr) return DART_ERR_INVALID_ARG;
    return sma_backward_impl(d, M, rM, Q, Cm, E, z, lse, logits, dY, dM, dQ, dC, dE, dz, ws, ws_bytes,
                             stream);
}

dart_status dart_chunk_scan_backward(const dart_dims* d, const void* X, const float* dt,
                                     const float* A, const void* Bm, const void* Cm,
                                     const void* dY, const float* dM, float* dX, float* ddt,
                                     float* dA, float* dB, float* dC, void* ws, size_t ws_bytes,
                                     void* stream) {
    dart_status st = check_dims(d, true);
    if (st != DART_OK) return st;
    const void* req[] = {X, dt, A, Bm, Cm, dY, dX, ddt, dA, dB, dC};
    for (const void* p : req)
        if (p == nullptr || !aligned16(p)) return DART_ERR_INVALID_ARG;
    if (dM != nullptr && !aligned16(dM)) return DART_ERR_INVALID_ARG;
    const size_t need = dart_workspace_size(d, DART_OP_SCAN_BACKWARD);
    if (ws == nullptr || ((uintptr_t)ws & 255u) != 0 || ws_bytes < need) return DART_ERR_WORKSPACE;
    dart::ScanBwdArgs a{};
    dart::ScanArgs& f = a.fwd;
    f.B = d->batch; f.L = d->seqlen; f.H = d->nheads; f.G = d->ngroups;
    f.P = d->headdim; f.N = d->dstate; f.S = d->chunk; f.eps = d->eps;
    f.X = X; f.dt = dt; f.A = A; f.Bm = Bm; f.Cm = Cm;
    a.dY = dY; a.dM = dM; a.dX = dX; a.ddt = ddt; a.dA = dA; a.dB = dB; a.dC = dC;
    a.accumulate_dC = true;
    f.test_withhold = g_test_withhold.load();
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e;
    if (scan_bwd_grouped(d))
        e = scan_backward_grouped(d, a, ws, g_wait_limit_ns.load(), s);
    else if (d->in_dtype == DART_F32)
        e = dart::launch_chunk_scan_backward<float>(a, ws, g_wait_limit_ns.load(), s);
    else if (d->in_dtype == DART_BF16)
        e = dart::launch_chunk_scan_backward<__nv_bfloat16>(a, ws, g_wait_limit_ns.load(), s);
    else
        return DART_ERR_UNSUPPORTED;
    return e == cudaSuccess ? DART_OK : cuda_fail(e);
}

size_t dart_block_workspace_size(const dart_block_dims* b) {
    if (check_block(b) != DART_OK) return 0;
    return block_ws(b).total;
}

dart_status dart_block_forward(const dart_block_dims* b, const void* U, const void* W_in, const float* conv_w,
                               const float* conv_b, const float* dt_bias, const float* A_log, const float* D,
                               const float* norm_w, const void* W_out, void* out, void* ws, size_t ws_bytes,
                               void* stream) {
    dart_status st = check_block(b);
    if (st != DART_OK) return st;
    const void* req[] = {U, W_in, conv_w, conv_b, dt_bias, A_log, D, norm_w, W_out, out};
    for (const void* p : req)
        if (p == nullptr || !aligned16(p)) return DART_ERR_INVALID_ARG;
    const BlockWs w = block_ws(b);
    if (ws == nullptr || ((uintptr_t)ws & 255u) != 0 || ws_bytes < w.total) return DART_ERR_WORKSPACE;
    const dart_dims c = block_core(b);
    uint8_t* p = (uint8_t*)ws;
    cudaStream_t s = (cudaStream_t)stream;
    const unsigned long long lim = g_wait_limit_ns.load();
    const int64_t T = c.batch * c.seqlen, di = c.nheads * c.headdim;
    dart::BlockArgs a{};
    a.B = c.batch; a.L = c.seqlen; a.H = c.nheads; a.G = c.ngroups; a.P = c.headdim; a.N = c.dstate;
    a.d_model = b->d_model; a.conv_width = b->conv_width; a.norm_eps = b->norm_eps;
    a.conv_w = conv_w; a.conv_b = conv_b; a.dt_bias = dt_bias; a.A_log = A_log; a.D = D; a.norm_w = norm_w;
    a.zx = p + w.zx; a.ldz = w.ldz; a.X = p + w.x; a.Bm = p + w.bm; a.Cm = p + w.cm;
    a.dt = (float*)(p + w.dt); a.A = (float*)(p + w.a); a.Q = p + w.q; a.E = p + w.e; a.gate = p + w.gate;
    a.Y = (float*)(p + w.y); a.yn = p + w.yn;
    typedef __nv_bfloat16 bf;
    cudaError_t e = dart::launch_gemm_tc<float>(U, W_in, (float*)a.zx, T, w.d_in, b->d_model, w.ldz, w.ldz, lim, s);
    if (e == cudaSuccess) e = dart::launch_block_conv_split(a, s);
    if (e != cudaSuccess) return cuda_fail(e);
    // the scan writes the SMA's operand tiles where both run on the tensor cores
    uint8_t* tiles = w.tiles_bytes > 0 ? p + w.tiles : nullptr;
    st = chunk_scan_impl(&c, a.X, a.dt, a.A, a.Bm, a.Cm, p + w.yssd, p + w.mem, (float*)(p + w.rm), nullptr,
                         tiles, p + w.scan, w.scan_bytes, stream);
    if (st != DART_OK) return st;
    st = tiles != nullptr
             ? dart_sma_forward_with_tiles(&c, tiles, a.Q, a.Cm, a.E, a.gate, p + w.yssd, a.Y, nullptr, nullptr,
                                           stream)
             : dart_sma_forward(&c, p + w.mem, (const float*)(p + w.rm), a.Q, a.Cm, a.E, a.gate, p + w.yssd,
                                a.Y, nullptr, nullptr, p + w.sma, w.sma_bytes, stream);
    if (st != DART_OK) return st;
    e = dart::launch_block_norm(a, s);
    if (e == cudaSuccess)
        e = b->core.out_dtype == DART_F32
                ? dart::launch_gemm_tc<float>(a.yn, W_out, (float*)out, T, b->d_model, di, b->d_model,
                                              b->d_model, lim, s)
                : dart::launch_gemm_tc<bf>(a.yn, W_out, (bf*)out, T, b->d_model, di, b->d_model, b->d_model,
                                           lim, s);
    return e == cudaSuccess ? DART_OK : cuda_fail(e);
}

dart_status dart_get_device_status(void* stream) {
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e);
    cudaStream_t s = (cudaStream_t)stream;
    const int code = dart::take_tc_status(s);
    const int code2 = dart::take_scan_tc_status(s);
    const int code3 = dart::take_bwd_tc_status(s);
    const int code4 = dart::take_scan_bwd_tc_status(s);
    const int code5 = dart::take_gemm_status(s);
    if (code < 0 || code2 < 0 || code3 < 0 || code4 < 0 || code5 < 0) return cuda_fail(cudaGetLastError());
    return (code != 0 || code2 != 0 || code3 != 0 || code4 != 0 || code5 != 0) ? DART_ERR_TIMEOUT : DART_OK;
}

void dart_test_withhold_copies(int on) { g_test_withhold.store(on != 0 ? 1 : 0); }

void dart_set_wait_limit_ns(uint64_t limit_ns) {
    g_wait_limit_ns.store(limit_ns == 0 ? 2000000000ull : (unsigned long long)limit_ns);
}

}  // extern "C"
