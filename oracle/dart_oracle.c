/*
 * dart_oracle.c -- plain, slow, fp64 CPU oracle for the DART hot path
 * (arXiv 2608.02032, "Decoded Attention over Recurrent sTates").
 *
 * TEST INFRASTRUCTURE. This file exists only to check the CUDA path. The test
 * suite, the smoke check and the CPU-baseline leg of the benchmark load it;
 * the product library never does, and the two share no code, header, table
 * or helper. Every quantity is computed straight from the paper's
 * definitions, with no blocking, fusion or reordering, in double precision.
 *
 * Tensor layouts follow the paper's table of compact tensor shapes
 * (App. B.2, Table "mva_tensor_shapes"), all row-major:
 *   X   : Bsz x L x H x P          dt : Bsz x L x H        A : H
 *   Bm, Cm, Q : Bsz x L x G x N    E  : Bsz x L x G x P
 *   dH (chunk state memories)      : Bsz x M x H x N x P,   M = ceil(L / S)
 * Head h reads projection group h / (H / G).
 *
 * Indices are 0-based. Token t lies in chunk floor(t / S), which is the
 * paper's 1-based c(t) = ceil(t / S) (Sec. 3, "Chunk State Memories").
 *
 * Readings taken where the paper is silent (each is also listed in the
 * design notes of the repository):
 *   - a_t = exp(dt_t * A_h) and the write term is dt_t * B_t^T X_t (the
 *     Mamba-2 discretisation; Sec. 2 leaves a_t and B_t abstract). dt is
 *     taken after softplus.
 *   - RMSNorm has unit weight; one eps serves Qbar, Ebar and r (App. B.1
 *     names eps without a value).
 *   - The state before the first token is zero (App. A, "zero-initial-state").
 *   - Decode: token pos attends to the completed chunks j < floor(pos / S);
 *     the running partial-chunk memory is appended when its chunk completes.
 *
 * Parity status of each function is stated above it; all are pinned by the
 * tests in tests/test_oracle_pins.py (brute-force cross-formulations, closed
 * forms, invariants and special cases).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef int64_t i64;

int oracle_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

static i64 group_of(i64 h, i64 H, i64 G) { return h / (H / G); }

/* SiLU(z) = z * sigmoid(z) (Sec. 3, "Gated Residual Integration"). */
static double silu(double z) { return z / (1.0 + exp(-z)); }

/* RMSNorm with unit weight (App. B.1): out = x / sqrt(mean(x^2) + eps). */
static void rmsnorm(const double* x, i64 n, double eps, double* out)
{
    double ss = 0.0;
    for (i64 i = 0; i < n; ++i) ss += x[i] * x[i];
    double inv = 1.0 / sqrt(ss / (double)n + eps);
    for (i64 i = 0; i < n; ++i) out[i] = x[i] * inv;
}

/*
 * Token recurrence of the selective SSM (Sec. 2, "State Space Duality";
 * App. A): H_t = A_t H_{t-1} + B_t^T X_t and Y_t = C_t H_t, with
 * A_t = a_t I_N, a_t = exp(dt_t A_h) and the write term scaled by dt_t.
 * H_{-1} = 0. Writes Y (Bsz x L x H x P) and, when Hlast is not NULL, the
 * state after the last token (Bsz x H x N x P).
 * Pinned: causal linear attention when a_t = 1, dt = 1 (Sec. 2, SSD form
 * with L_SSD = all-ones lower triangle); agreement with the chunked scan of
 * App. A written independently in the tests.
 */
void oracle_ssd_recurrence(i64 Bsz, i64 L, i64 H, i64 G, i64 P, i64 N,
                           const double* X, const double* dt, const double* A,
                           const double* Bm, const double* Cm,
                           double* Y, double* Hlast)
{
#pragma omp parallel for collapse(2) schedule(static)
    for (i64 b = 0; b < Bsz; ++b) {
        for (i64 h = 0; h < H; ++h) {
            double* St = (double*)calloc((size_t)(N * P), sizeof(double));
            i64 g = group_of(h, H, G);
            for (i64 t = 0; t < L; ++t) {
                double d = dt[(b * L + t) * H + h];
                double a = exp(d * A[h]);
                const double* Bt = Bm + ((b * L + t) * G + g) * N;
                const double* Ct = Cm + ((b * L + t) * G + g) * N;
                const double* Xt = X + ((b * L + t) * H + h) * P;
                for (i64 n = 0; n < N; ++n)
                    for (i64 p = 0; p < P; ++p)
                        St[n * P + p] = a * St[n * P + p] + d * Bt[n] * Xt[p];
                double* Yt = Y + ((b * L + t) * H + h) * P;
                for (i64 p = 0; p < P; ++p) {
                    double acc = 0.0;
                    for (i64 n = 0; n < N; ++n) acc += Ct[n] * St[n * P + p];
                    Yt[p] = acc;
                }
            }
            if (Hlast) memcpy(Hlast + (b * H + h) * N * P, St, (size_t)(N * P) * sizeof(double));
            free(St);
        }
    }
}

/*
 * Chunk state memories (Sec. 3, equation for Delta H_[c]; App. A,
 * eq. "mamba2_delta_h_chunk"):
 *   dH_[c] = sum_{s in chunk c} A_{s+1:e(c)} B_s^T X_s,
 * with A_{s+1:e(c)} = prod_{k=s+1}^{e(c)} a_k taken literally as a product
 * (empty product = 1) and the write term dt_s B_s^T X_s. The last chunk may
 * be ragged: e(c) = min((c+1) S, L) - 1.
 * Pinned: the decayed sum of the memories equals the recurrent state at every
 * chunk boundary (App. A, eq. "mamba2_chunk_state" unrolled); S = L gives
 * the final state itself.
 */
void oracle_chunk_memories(i64 Bsz, i64 L, i64 H, i64 G, i64 P, i64 N, i64 S,
                           const double* X, const double* dt, const double* A,
                           const double* Bm, double* dH)
{
    i64 M = (L + S - 1) / S;
#pragma omp parallel for collapse(2) schedule(static)
    for (i64 b = 0; b < Bsz; ++b) {
        for (i64 h = 0; h < H; ++h) {
            i64 g = group_of(h, H, G);
            for (i64 c = 0; c < M; ++c) {
                i64 first = c * S;
                i64 last = (c + 1) * S < L ? (c + 1) * S - 1 : L - 1;
                double* D = dH + ((b * M + c) * H + h) * N * P;
                for (i64 i = 0; i < N * P; ++i) D[i] = 0.0;
                for (i64 s = first; s <= last; ++s) {
                    double decay = 1.0;
                    for (i64 k = s + 1; k <= last; ++k)
                        decay *= exp(dt[(b * L + k) * H + h] * A[h]);
                    double w = decay * dt[(b * L + s) * H + h];
                    const double* Bs = Bm + ((b * L + s) * G + g) * N;
                    const double* Xs = X + ((b * L + s) * H + h) * P;
                    for (i64 n = 0; n < N; ++n)
                        for (i64 p = 0; p < P; ++p)
                            D[n * P + p] += w * Bs[n] * Xs[p];
                }
            }
        }
    }
}

/*
 * State-memory attention for one token over its first `nhist` memories
 * (Sec. 3, value/key readouts, chunk logit, softmax over c < c(t) and R_t;
 * App. B.1, normalised score branch):
 *   Qbar = RMSNorm(q), Ebar = RMSNorm(e)
 *   r_{j,n} = (mean_p dH_j[n,p]^2 + eps)^(-1/2)
 *   K_j = r_j (.) (dH_j Ebar),  l_j = Qbar K_j / sqrt(N),  V_j = c dH_j
 *   g = softmax_j(l),  R = sum_j g_j V_j,  lse = log sum_j exp(l_j)
 * The softmax is the exact two-pass form (maximum, then sum). With no
 * history R = 0 and lse = -inf (Sec. 3: empty historical set).
 * Memory j starts at mem0 + j * mem_stride and is N x P row-major.
 */
static void sma_token(i64 N, i64 P, double eps, i64 nhist,
                      const double* mem0, i64 mem_stride,
                      const double* q, const double* c, const double* e,
                      double* R, double* lse, double* g_out)
{
    for (i64 p = 0; p < P; ++p) R[p] = 0.0;
    if (nhist <= 0) {
        *lse = -INFINITY;
        return;
    }
    double* qbar = (double*)malloc((size_t)N * sizeof(double));
    double* ebar = (double*)malloc((size_t)P * sizeof(double));
    double* ell = (double*)malloc((size_t)nhist * sizeof(double));
    double* K = (double*)malloc((size_t)N * sizeof(double));
    double* V = (double*)malloc((size_t)P * sizeof(double));
    rmsnorm(q, N, eps, qbar);
    rmsnorm(e, P, eps, ebar);

    for (i64 j = 0; j < nhist; ++j) {
        const double* D = mem0 + j * mem_stride;
        for (i64 n = 0; n < N; ++n) {
            double ss = 0.0, ke = 0.0;
            for (i64 p = 0; p < P; ++p) {
                ss += D[n * P + p] * D[n * P + p];
                ke += D[n * P + p] * ebar[p];
            }
            double r = 1.0 / sqrt(ss / (double)P + eps);
            K[n] = r * ke;
        }
        double l = 0.0;
        for (i64 n = 0; n < N; ++n) l += qbar[n] * K[n];
        ell[j] = l / sqrt((double)N);
    }

    double m = ell[0];
    for (i64 j = 1; j < nhist; ++j) if (ell[j] > m) m = ell[j];
    double sum = 0.0;
    for (i64 j = 0; j < nhist; ++j) sum += exp(ell[j] - m);

    for (i64 j = 0; j < nhist; ++j) {
        const double* D = mem0 + j * mem_stride;
        double gj = exp(ell[j] - m) / sum;
        if (g_out) g_out[j] = gj;
        for (i64 p = 0; p < P; ++p) {
            double v = 0.0;
            for (i64 n = 0; n < N; ++n) v += c[n] * D[n * P + p];
            V[p] = v;
        }
        for (i64 p = 0; p < P; ++p) R[p] += gj * V[p];
    }
    *lse = m + log(sum);
    free(qbar); free(ebar); free(ell); free(K); free(V);
}

/*
 * State-memory attention over chunk memories for a list of (b, t, h) tokens
 * (Sec. 3; App. B.1). Token t attends to memories j < floor(t / S).
 * tok: ntok x 3 int64 triples (b, t, h); NULL means every token in b, t, h
 * order (ntok must then be Bsz * L * H, and R is Bsz x L x H x P).
 * R: ntok x P. lse: ntok. g: ntok x M softmax weights (entries j >= the
 * token's history are set to 0), or NULL.
 * Pinned: closed forms for a token with one memory (R = C dH_0), for Q = 0
 * (uniform weights) and for rank-1 memories; weights sum to 1; S = L gives
 * R = 0, lse = -inf.
 */
void oracle_sma(i64 Bsz, i64 L, i64 H, i64 G, i64 P, i64 N, i64 S, double eps,
                const double* dH, const double* Q, const double* Cm, const double* E,
                i64 ntok, const i64* tok, double* R, double* lse, double* g)
{
    i64 M = (L + S - 1) / S;
#pragma omp parallel for schedule(dynamic, 16)
    for (i64 i = 0; i < ntok; ++i) {
        i64 b, t, h;
        if (tok) {
            b = tok[3 * i]; t = tok[3 * i + 1]; h = tok[3 * i + 2];
        } else {
            b = i / (L * H); t = (i / H) % L; h = i % H;
        }
        i64 grp = group_of(h, H, G);
        const double* q = Q + ((b * L + t) * G + grp) * N;
        const double* c = Cm + ((b * L + t) * G + grp) * N;
        const double* e = E + ((b * L + t) * G + grp) * P;
        const double* mem0 = dH + ((b * M + 0) * H + h) * N * P;
        i64 nhist = t / S;
        double* gi = g ? g + i * M : NULL;
        if (gi) for (i64 j = 0; j < M; ++j) gi[j] = 0.0;
        sma_token(N, P, eps, nhist, mem0, H * N * P, q, c, e, R + i * P, lse + i, gi);
    }
}

/*
 * Inverse RMS of every memory row along the value axis (App. B.1):
 *   r_{j,n} = (mean_p dH_j[n,p]^2 + eps)^(-1/2),  rows = Bsz * M * H * N.
 * Pinned: closed forms for constant and two-valued rows.
 */
void oracle_memory_inverse_rms(i64 rows, i64 P, double eps, const double* dH, double* r)
{
    for (i64 i = 0; i < rows; ++i) {
        double ss = 0.0;
        for (i64 p = 0; p < P; ++p) ss += dH[i * P + p] * dH[i * P + p];
        r[i] = 1.0 / sqrt(ss / (double)P + eps);
    }
}

/*
 * Gated residual merge (Sec. 3, "Gated Residual Integration"):
 *   Y = Y_ssd + SiLU(z) R,  one gate logit z per (b, t, h) row.
 * Pinned: z = 0 reproduces Y_ssd exactly (the SMA-removal special case).
 */
void oracle_merge(i64 rows, i64 P, const double* Yssd, const double* z,
                  const double* R, double* Y)
{
    for (i64 i = 0; i < rows; ++i) {
        double gate = silu(z[i]);
        for (i64 p = 0; p < P; ++p) Y[i * P + p] = Yssd[i * P + p] + gate * R[i * P + p];
    }
}

/*
 * One decode step over the chunk-memory cache (the paper's persistent
 * inference cache, Sec. 4 "Inference Cache" and Sec. 5.3; the step itself is
 * this oracle's reading, since the paper prints no decode algorithm):
 *   token index pos (pos tokens were absorbed before it), chunk i = pos / S
 *   a = exp(dt A_h);  state <- a state + dt b^T x
 *   partial <- dt b^T x            if pos % S == 0 (first token of a chunk)
 *   partial <- a partial + dt b^T x otherwise
 *   y = c state + SiLU(z) R, R = SMA over the i completed memories
 *   if (pos + 1) % S == 0: cache[b, i, h] <- partial (the memory of chunk i)
 * cache: Bsz x m_cap x H x N x P; state, partial: Bsz x H x N x P;
 * x: Bsz x H x P; dt, z: Bsz x H; b, c, q: Bsz x G x N; e: Bsz x G x P;
 * y: Bsz x H x P; lse (optional): Bsz x H.
 * Pinned: prefill of L tokens followed by k decode steps reproduces the
 * prefill of L + k tokens, and the appended memories equal the prefill's.
 */
void oracle_decode_step(i64 Bsz, i64 H, i64 G, i64 P, i64 N, i64 S, double eps,
                        i64 pos, i64 m_cap, double* cache, double* state, double* partial,
                        const double* x, const double* dt, const double* A,
                        const double* bv, const double* cv, const double* qv,
                        const double* ev, const double* z, double* y, double* lse)
{
    i64 chunk = pos / S;
#pragma omp parallel for collapse(2) schedule(static)
    for (i64 b = 0; b < Bsz; ++b) {
        for (i64 h = 0; h < H; ++h) {
            i64 grp = group_of(h, H, G);
            double d = dt[b * H + h];
            double a = exp(d * A[h]);
            const double* bt = bv + (b * G + grp) * N;
            const double* ct = cv + (b * G + grp) * N;
            const double* qt = qv + (b * G + grp) * N;
            const double* et = ev + (b * G + grp) * P;
            const double* xt = x + (b * H + h) * P;
            double* St = state + (b * H + h) * N * P;
            double* Pt = partial + (b * H + h) * N * P;
            for (i64 n = 0; n < N; ++n) {
                for (i64 p = 0; p < P; ++p) {
                    double w = d * bt[n] * xt[p];
                    St[n * P + p] = a * St[n * P + p] + w;
                    Pt[n * P + p] = (pos % S == 0) ? w : a * Pt[n * P + p] + w;
                }
            }
            double* R = (double*)malloc((size_t)P * sizeof(double));
            double l;
            const double* mem0 = cache + ((b * m_cap + 0) * H + h) * N * P;
            sma_token(N, P, eps, chunk, mem0, H * N * P, qt, ct, et, R, &l, NULL);
            double gate = silu(z[b * H + h]);
            double* yt = y + (b * H + h) * P;
            for (i64 p = 0; p < P; ++p) {
                double acc = 0.0;
                for (i64 n = 0; n < N; ++n) acc += ct[n] * St[n * P + p];
                yt[p] = acc + gate * R[p];
            }
            if (lse) lse[b * H + h] = l;
            free(R);
            if ((pos + 1) % S == 0 && chunk < m_cap)
                memcpy(cache + ((b * m_cap + chunk) * H + h) * N * P, Pt,
                       (size_t)(N * P) * sizeof(double));
        }
    }
}

/*
 * Backward of the SSD scan (gradients of the paper's selective-SSM forms,
 * Sec. 2 and App. A; the paper prints no backward, so this is the chain rule
 * on the token recurrence, written out by hand).
 * Outputs of the forward that a loss can depend on: Y_ssd (through dY, the
 * same layout as Y) and the chunk memories dH_[c] (through dMem, the layout of
 * oracle_chunk_memories; NULL means zero).
 * Forward, per (b, h):  H_t = a_t H_{t-1} + u_t,  u_t = dt_t B_t^T X_t,
 * a_t = exp(dt_t A_h), Y_t = C_t H_t; the memory of chunk c is the state of
 * the same recurrence restarted from zero at the chunk's first token and
 * read at its last token.
 * Adjoints (reverse order over t): dH_t = C_t^T dY_t + a_{t+1} dH_{t+1};
 * the chunk-local adjoint starts from dMem_[c] at the chunk's last token and
 * dies at its first; du_t = dH_t + dHloc_t gives dX_t = dt_t B_t du_t,
 * dB_t = dt_t du_t X_t, d(dt_t) = B_t du_t X_t; dC_t = H_t dY_t; the decay
 * gives da_t = <dH_t, H_{t-1}> + <dHloc_t, Hloc_{t-1}>, d(dt_t) += A_h a_t
 * da_t and dA_h += dt_t a_t da_t.
 * dX (Bsz x L x H x P), ddt (Bsz x L x H), dA (H), dB, dC (Bsz x L x G x N,
 * summed over the heads of a group). All outputs are overwritten.
 * Pinned: central finite differences of a weighted sum of Y_ssd and the
 * memories (tests/test_oracle_backward.py).
 */
void oracle_ssd_backward(i64 Bsz, i64 L, i64 H, i64 G, i64 P, i64 N, i64 S,
                         const double* X, const double* dt, const double* A,
                         const double* Bm, const double* Cm, const double* dY,
                         const double* dMem, double* dX, double* ddt, double* dA,
                         double* dB, double* dC)
{
    i64 M = (L + S - 1) / S;
    i64 NP = N * P;
    memset(dX, 0, (size_t)(Bsz * L * H * P) * sizeof(double));
    memset(ddt, 0, (size_t)(Bsz * L * H) * sizeof(double));
    memset(dA, 0, (size_t)H * sizeof(double));
    memset(dB, 0, (size_t)(Bsz * L * G * N) * sizeof(double));
    memset(dC, 0, (size_t)(Bsz * L * G * N) * sizeof(double));
    /* heads of one group write the same dB, dC rows: parallel over b only */
#pragma omp parallel for schedule(static)
    for (i64 b = 0; b < Bsz; ++b) {
        double* ckpt = (double*)calloc((size_t)(M * NP), sizeof(double));
        double* Hg = (double*)malloc((size_t)(S * NP) * sizeof(double));
        double* Hl = (double*)malloc((size_t)(S * NP) * sizeof(double));
        double* dHg = (double*)malloc((size_t)NP * sizeof(double));
        double* dHl = (double*)malloc((size_t)NP * sizeof(double));
        for (i64 h = 0; h < H; ++h) {
            i64 g = group_of(h, H, G);
            /* forward once: the global state entering every chunk */
            double* St = (double*)calloc((size_t)NP, sizeof(double));
            for (i64 t = 0; t < L; ++t) {
                if (t % S == 0) memcpy(ckpt + (t / S) * NP, St, (size_t)NP * sizeof(double));
                double d = dt[(b * L + t) * H + h], a = exp(d * A[h]);
                const double* Bt = Bm + ((b * L + t) * G + g) * N;
                const double* Xt = X + ((b * L + t) * H + h) * P;
                for (i64 n = 0; n < N; ++n)
                    for (i64 p = 0; p < P; ++p)
                        St[n * P + p] = a * St[n * P + p] + d * Bt[n] * Xt[p];
            }
            free(St);
            double dAh = 0.0;
            for (i64 i = 0; i < NP; ++i) dHg[i] = 0.0;
            for (i64 c = M - 1; c >= 0; --c) {
                i64 first = c * S, last = (c + 1) * S < L ? (c + 1) * S - 1 : L - 1;
                /* recompute the chunk's global and local states */
                for (i64 t = first; t <= last; ++t) {
                    i64 k = t - first;
                    double d = dt[(b * L + t) * H + h], a = exp(d * A[h]);
                    const double* Bt = Bm + ((b * L + t) * G + g) * N;
                    const double* Xt = X + ((b * L + t) * H + h) * P;
                    const double* gprev = k > 0 ? Hg + (k - 1) * NP : ckpt + c * NP;
                    for (i64 n = 0; n < N; ++n) {
                        for (i64 p = 0; p < P; ++p) {
                            double u = d * Bt[n] * Xt[p];
                            Hg[k * NP + n * P + p] = a * gprev[n * P + p] + u;
                            Hl[k * NP + n * P + p] = (k > 0 ? a * Hl[(k - 1) * NP + n * P + p] : 0.0) + u;
                        }
                    }
                }
                const double* dm = dMem ? dMem + ((b * M + c) * H + h) * NP : NULL;
                for (i64 i = 0; i < NP; ++i) dHl[i] = dm ? dm[i] : 0.0;
                for (i64 t = last; t >= first; --t) {
                    i64 k = t - first;
                    double d = dt[(b * L + t) * H + h], a = exp(d * A[h]);
                    const double* Bt = Bm + ((b * L + t) * G + g) * N;
                    const double* Ct = Cm + ((b * L + t) * G + g) * N;
                    const double* Xt = X + ((b * L + t) * H + h) * P;
                    const double* dYt = dY + ((b * L + t) * H + h) * P;
                    double* dXt = dX + ((b * L + t) * H + h) * P;
                    double* dBt = dB + ((b * L + t) * G + g) * N;
                    double* dCt = dC + ((b * L + t) * G + g) * N;
                    /* Y_t = C_t H_t */
                    for (i64 n = 0; n < N; ++n) {
                        double acc = 0.0;
                        for (i64 p = 0; p < P; ++p) {
                            dHg[n * P + p] += Ct[n] * dYt[p];
                            acc += Hg[k * NP + n * P + p] * dYt[p];
                        }
                        dCt[n] += acc;
                    }
                    /* u_t = dt_t B_t^T X_t */
                    double dd = 0.0;
                    for (i64 n = 0; n < N; ++n) {
                        double acc = 0.0;
                        for (i64 p = 0; p < P; ++p) {
                            double du = dHg[n * P + p] + dHl[n * P + p];
                            acc += du * Xt[p];
                            dXt[p] += d * Bt[n] * du;
                        }
                        dBt[n] += d * acc;
                        dd += Bt[n] * acc;
                    }
                    /* a_t = exp(dt_t A_h) */
                    const double* gprev = k > 0 ? Hg + (k - 1) * NP : ckpt + c * NP;
                    double da = 0.0;
                    for (i64 i = 0; i < NP; ++i) {
                        da += dHg[i] * gprev[i];
                        if (k > 0) da += dHl[i] * Hl[(k - 1) * NP + i];
                    }
                    ddt[(b * L + t) * H + h] = dd + A[h] * a * da;
                    dAh += d * a * da;
                    for (i64 i = 0; i < NP; ++i) {
                        dHg[i] *= a;
                        dHl[i] *= a;
                    }
                }
            }
#pragma omp atomic
            dA[h] += dAh;
        }
        free(ckpt); free(Hg); free(Hl); free(dHg); free(dHl);
    }
}

/*
 * Backward of state-memory attention and the gated merge (Sec. 3 readouts,
 * logit, softmax over earlier chunks, R_t and Y = Y_ssd + SiLU(z) R; App. B.1
 * normalisations). The paper prints no backward; this is the chain rule on
 * the plain per-token forms of oracle_sma, with the exact softmax Jacobian.
 * For each (b, t, h) with history: dR = SiLU(z) dY, dz = (dY . R) SiLU'(z),
 * dV_j = g_j dR, dl_j = g_j (dR . V_j - dR . R); through V_j = c dH_j and
 * l_j = Qbar (r_j (.) dH_j Ebar) / sqrt(N) into dMem, dQbar, dEbar, dc, and
 * through r_{j,n} = (mean_p dH_j[n,p]^2 + eps)^(-1/2) into dMem; the unit-
 * weight RMSNorms take dQbar, dEbar back to dQ, dE. dY_ssd = dY and is not
 * written here.
 * dMem: Bsz x M x H x N x P; dQ, dC: Bsz x L x G x N; dE: Bsz x L x G x P
 * (summed over the heads of a group); dz: Bsz x L x H. All overwritten.
 * Pinned: central finite differences of a weighted sum of Y
 * (tests/test_oracle_backward.py), and the closed form dz = dY . R / 2 at z = 0.
 */
void oracle_sma_backward(i64 Bsz, i64 L, i64 H, i64 G, i64 P, i64 N, i64 S, double eps,
                         const double* dHm, const double* Q, const double* Cm, const double* E,
                         const double* z, const double* dY, double* dMem, double* dQ,
                         double* dC, double* dE, double* dz)
{
    i64 M = (L + S - 1) / S;
    i64 NP = N * P;
    memset(dMem, 0, (size_t)(Bsz * M * H * NP) * sizeof(double));
    memset(dQ, 0, (size_t)(Bsz * L * G * N) * sizeof(double));
    memset(dC, 0, (size_t)(Bsz * L * G * N) * sizeof(double));
    memset(dE, 0, (size_t)(Bsz * L * G * P) * sizeof(double));
    memset(dz, 0, (size_t)(Bsz * L * H) * sizeof(double));
    double rsn = 1.0 / sqrt((double)N);
#pragma omp parallel for schedule(static)
    for (i64 b = 0; b < Bsz; ++b) {
        double* qbar = (double*)malloc((size_t)N * sizeof(double));
        double* ebar = (double*)malloc((size_t)P * sizeof(double));
        double* r = (double*)malloc((size_t)(M * N) * sizeof(double));
        double* Kraw = (double*)malloc((size_t)(M * N) * sizeof(double));
        double* V = (double*)malloc((size_t)(M * P) * sizeof(double));
        double* ell = (double*)malloc((size_t)M * sizeof(double));
        double* gw = (double*)malloc((size_t)M * sizeof(double));
        double* R = (double*)malloc((size_t)P * sizeof(double));
        double* dqbar = (double*)malloc((size_t)N * sizeof(double));
        double* debar = (double*)malloc((size_t)P * sizeof(double));
        for (i64 h = 0; h < H; ++h) {
            i64 g = group_of(h, H, G);
            const double* mem0 = dHm + ((b * M) * H + h) * NP;
            double* dmem0 = dMem + ((b * M) * H + h) * NP;
            for (i64 j = 0; j < M; ++j) {
                const double* D = mem0 + j * H * NP;
                for (i64 n = 0; n < N; ++n) {
                    double ss = 0.0;
                    for (i64 p = 0; p < P; ++p) ss += D[n * P + p] * D[n * P + p];
                    r[j * N + n] = 1.0 / sqrt(ss / (double)P + eps);
                }
            }
            for (i64 t = 0; t < L; ++t) {
                i64 nh = t / S;
                if (nh == 0) continue;  /* R = 0: no gradient reaches this token's inputs */
                const double* q = Q + ((b * L + t) * G + g) * N;
                const double* c = Cm + ((b * L + t) * G + g) * N;
                const double* e = E + ((b * L + t) * G + g) * P;
                const double* dYt = dY + ((b * L + t) * H + h) * P;
                rmsnorm(q, N, eps, qbar);
                rmsnorm(e, P, eps, ebar);
                /* forward: Kraw, l, V, two-pass softmax, R */
                for (i64 j = 0; j < nh; ++j) {
                    const double* D = mem0 + j * H * NP;
                    double l = 0.0;
                    for (i64 n = 0; n < N; ++n) {
                        double ke = 0.0;
                        for (i64 p = 0; p < P; ++p) ke += D[n * P + p] * ebar[p];
                        Kraw[j * N + n] = ke;
                        l += qbar[n] * r[j * N + n] * ke;
                    }
                    ell[j] = l * rsn;
                    for (i64 p = 0; p < P; ++p) {
                        double v = 0.0;
                        for (i64 n = 0; n < N; ++n) v += c[n] * D[n * P + p];
                        V[j * P + p] = v;
                    }
                }
                double m = ell[0];
                for (i64 j = 1; j < nh; ++j) if (ell[j] > m) m = ell[j];
                double sum = 0.0;
                for (i64 j = 0; j < nh; ++j) sum += exp(ell[j] - m);
                for (i64 p = 0; p < P; ++p) R[p] = 0.0;
                for (i64 j = 0; j < nh; ++j) {
                    gw[j] = exp(ell[j] - m) / sum;
                    for (i64 p = 0; p < P; ++p) R[p] += gw[j] * V[j * P + p];
                }
                /* merge: Y = Y_ssd + SiLU(z) R */
                double zz = z[(b * L + t) * H + h];
                double sg = 1.0 / (1.0 + exp(-zz));
                double gate = zz * sg;
                double dyr = 0.0;
                for (i64 p = 0; p < P; ++p) dyr += dYt[p] * R[p];
                dz[(b * L + t) * H + h] = dyr * sg * (1.0 + zz * (1.0 - sg));
                /* softmax and readouts */
                double Dt = gate * dyr;  /* dR . R */
                for (i64 n = 0; n < N; ++n) dqbar[n] = 0.0;
                for (i64 p = 0; p < P; ++p) debar[p] = 0.0;
                double* dCt = dC + ((b * L + t) * G + g) * N;
                for (i64 j = 0; j < nh; ++j) {
                    const double* D = mem0 + j * H * NP;
                    double* dD = dmem0 + j * H * NP;
                    double drv = 0.0;
                    for (i64 p = 0; p < P; ++p) drv += gate * dYt[p] * V[j * P + p];
                    double dl = gw[j] * (drv - Dt);
                    for (i64 n = 0; n < N; ++n) {
                        double rn = r[j * N + n];
                        double dkr = rsn * dl * qbar[n] * rn;          /* d Kraw[n] */
                        double dr = rsn * dl * qbar[n] * Kraw[j * N + n]; /* d r[n] */
                        dqbar[n] += rsn * dl * rn * Kraw[j * N + n];
                        double acc = 0.0;
                        for (i64 p = 0; p < P; ++p) {
                            double dv = gw[j] * gate * dYt[p];
                            acc += D[n * P + p] * dv;
                            dD[n * P + p] += c[n] * dv + dkr * ebar[p]
                                             - dr * rn * rn * rn * D[n * P + p] / (double)P;
                            debar[p] += D[n * P + p] * dkr;
                        }
                        dCt[n] += acc;
                    }
                }
                /* unit-weight RMSNorm backward: dx = s (dxbar - xbar (dxbar . xbar) / n) */
                double sq = 0.0, se = 0.0, dq_dot = 0.0, de_dot = 0.0;
                for (i64 n = 0; n < N; ++n) { sq += q[n] * q[n]; dq_dot += dqbar[n] * qbar[n]; }
                for (i64 p = 0; p < P; ++p) { se += e[p] * e[p]; de_dot += debar[p] * ebar[p]; }
                double s_q = 1.0 / sqrt(sq / (double)N + eps), s_e = 1.0 / sqrt(se / (double)P + eps);
                double* dQt = dQ + ((b * L + t) * G + g) * N;
                double* dEt = dE + ((b * L + t) * G + g) * P;
                for (i64 n = 0; n < N; ++n) dQt[n] += s_q * (dqbar[n] - qbar[n] * dq_dot / (double)N);
                for (i64 p = 0; p < P; ++p) dEt[p] += s_e * (debar[p] - ebar[p] * de_dot / (double)P);
            }
        }
        free(qbar); free(ebar); free(r); free(Kraw); free(V); free(ell); free(gw); free(R);
        free(dqbar); free(debar);
    }
}
