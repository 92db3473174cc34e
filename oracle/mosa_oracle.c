/*
 * Plain CPU oracle for the Mixture-of-Sparse-Attention (MoSA) layer.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call, link or
 * load this file; only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg do.  It shares no code, header, table or helper with the
 * CUDA library: it is written directly from the paper's definitions, in fp64,
 * with explicit loops, in the paper's order of operations, so that a reader
 * can check each line against the text.
 *
 * Paper: "Mixture of Sparse Attention: Content-Based Learnable Sparse
 * Attention via Expert-Choice Routing" (arXiv 2505.00315).
 *   Sec. 2.1, Eq. (attention): Attention(Q,K,V,M) = softmax((QK^T + M)/sqrt(h')) V
 *   Sec. 2.1, Eq. (mha):       X_out = sum_i Attention(Q_i,K_i,V_i,M) W^O_i
 *   Sec. 2.2 (MoSA head):      r = sigma(X W^r);  r^topk, I = TopK(r, k);
 *                              X^s = (X_{I_1}, ..., X_{I_k});  Q = X^s W^Q, K = X^s W^K,
 *                              V = X^s W^V;  M_ij = 0 iff I_i >= I_j, else -inf;
 *                              A = Attention(Q,K,V,M);  X^o = diag(r^topk) A W^o;
 *                              Y_j = X^o_i if j = I_i, else 0.
 *   Sec. 2.2, Eq. (mosa_mha):  MoSA(X) = sum_i MoSA_head(X; theta_i)
 *   Sec. 3.2 (IsoFLOP models): the first token is always in every head's set
 *   Sec. 2.2 (positional encodings): RoPE rotates Q and K after the mapping by
 *                              angles of the tokens' original positions I,
 *                              half of the dimensions rotated, half unchanged
 *   Sec. 2.2 (last paragraph of the output definition): the router receives
 *                              its gradient only through the diag(r) scaling;
 *                              TopK itself is not differentiated.
 *
 * Readings of points the paper leaves open:
 *   - TopK ranks the sigmoid scores r; ties go to the lower token index.
 *   - I is returned in ascending token order (the mask uses the indices
 *     themselves, so the layer output does not depend on the order).
 *   - diag(r) in the output definition is diag(r^topk): it has size k.
 *   - The mask is applied inside the 1/sqrt(h') scaling; -inf stays -inf.
 *     The diagonal I_i >= I_i is always allowed, so no row is empty.
 *   - No router noise, no biases, no dropout.
 *   - RoPE (optional): base 10000 and adjacent pairs (the RoFormer form) in
 *     the first h'/2 dimensions: pair p = 0 .. h'/4-1 of position t turns by
 *     t * 10000^(-2p / (h'/2)); dimensions h'/2 .. h'-1 are left unchanged.
 *   - Sec. 3.2 (IsoFLOP models) keeps the first token in every head and
 *     selects the other k-1 by router score: read as token 0 plus TopK(k-1)
 *     over tokens 1..T-1 (same tie rule), token 0 scaled by its own score.
 *   - Hybrid layers (Sec. 2.2, hybridization) add dense heads (Sec. 2.1,
 *     Eq. mha, causal M, no router and no scaling) or, for long sequences
 *     (Sec. 3.4), local heads.  The paper does not define its local
 *     attention; read as the block pattern of the cited fixed sparse
 *     attention: token i sees token j iff j <= i and floor(j/w) = floor(i/w)
 *     for a window of w tokens (the last block may be shorter).  The layer
 *     output is the sum over all heads, sparse and dense.
 *
 * Layouts (row-major, all fp64 here):
 *   X [B,T,d]; W_r [d,H]; W_q, W_k, W_v [H,d,h']; W_o [H,h',d];
 *   Y, dY, dX [B,T,d]; I [B,H,k] (int32); r_sel [B,H,k]; r_full [B,H,T].
 *
 * Sampling: every batch/head loop can be restricted with a byte mask
 * (bsel[B], hsel[H]; NULL = all).  Units (b,h) outside the masks contribute
 * nothing, so Y[b] and dX[b] are exact for a batch whose every head is
 * selected, and the weight gradients of head h are exact when every batch is
 * selected.  Parallelism is plain OpenMP over independent loops.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define IDX2(a, b, nb) ((size_t)(a) * (size_t)(nb) + (size_t)(b))
#define IDX3(a, b, c, nb, nc) (((size_t)(a) * (size_t)(nb) + (size_t)(b)) * (size_t)(nc) + (size_t)(c))

int oracle_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void oracle_set_num_threads(int n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* Sec. 2.2: sigma(x) = 1 / (1 + e^{-x}), the non-competitive sigmoid. */
static double sigmoid(double x) { return 1.0 / (1.0 + exp(-x)); }

/* Sec. 2.2: r = sigma(X W^r) for every head; r_full[b,h,t]. */
void oracle_router(int B, int T, int d, int H, const double *X, const double *Wr,
                   double *r_full) {
    #pragma omp parallel for collapse(2) schedule(static)
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < H; ++h)
            for (int t = 0; t < T; ++t) {
                double logit = 0.0;
                for (int c = 0; c < d; ++c)
                    logit += X[IDX3(b, t, c, T, d)] * Wr[IDX2(c, h, H)];
                r_full[IDX3(b, h, t, H, T)] = sigmoid(logit);
            }
}

/* Sort key for TopK: larger score first; equal scores -> lower token first. */
typedef struct { double score; int t; } scored_token;

static int by_score_then_index(const void *pa, const void *pb) {
    const scored_token *a = (const scored_token *)pa, *b = (const scored_token *)pb;
    if (a->score > b->score) return -1;
    if (a->score < b->score) return 1;
    return (a->t < b->t) ? -1 : (a->t > b->t);
}

static int ascending_int(const void *pa, const void *pb) {
    int a = *(const int *)pa, b = *(const int *)pb;
    return (a < b) ? -1 : (a > b);
}

/* Sec. 2.2: r^topk, I = TopK(r, k), by a full sort of all T scores.
 * Returns 0, or -1 on bad arguments.  I is written in ascending order and
 * r_sel[i] = r[I[i]]. */
int oracle_topk(int T, int k, const double *r, int32_t *I, double *r_sel) {
    if (T <= 0 || k <= 0 || k > T) return -1;
    scored_token *all = (scored_token *)malloc(sizeof(scored_token) * (size_t)T);
    int *chosen = (int *)malloc(sizeof(int) * (size_t)k);
    if (!all || !chosen) { free(all); free(chosen); return -1; }
    for (int t = 0; t < T; ++t) { all[t].score = r[t]; all[t].t = t; }
    qsort(all, (size_t)T, sizeof(scored_token), by_score_then_index);
    for (int i = 0; i < k; ++i) chosen[i] = all[i].t;
    qsort(chosen, (size_t)k, sizeof(int), ascending_int);
    for (int i = 0; i < k; ++i) { I[i] = chosen[i]; r_sel[i] = r[chosen[i]]; }
    free(all);
    free(chosen);
    return 0;
}

/* Sec. 3.2 (IsoFLOP models): every head always includes the first token; it
 * selects the other k-1 tokens by router score.  Token 0 plus the k-1 largest
 * of r[1..T-1] by a full sort of those T-1 scores (ties: lower index), I in
 * ascending order, r_sel[i] = r[I[i]] (token 0 keeps its own score).
 * Returns 0, or -1 on bad arguments. */
int oracle_topk_first(int T, int k, const double *r, int32_t *I, double *r_sel) {
    if (T <= 0 || k <= 0 || k > T) return -1;
    I[0] = 0;
    r_sel[0] = r[0];
    if (k == 1) return 0;
    /* the rest: TopK(k-1) over tokens 1..T-1, shifted back to token indices */
    if (oracle_topk(T - 1, k - 1, r + 1, I + 1, r_sel + 1) != 0) return -1;
    for (int i = 1; i < k; ++i) I[i] += 1;
    return 0;
}

/* Per-head intermediate state of the forward pass of one (b,h) unit. */
typedef struct {
    int k, d, hp;
    double *Xs;   /* [k,d]   X^s = rows I of X[b]                */
    double *Q;    /* [k,h']  X^s W^Q                             */
    double *K;    /* [k,h']  X^s W^K                             */
    double *V;    /* [k,h']  X^s W^V                             */
    double *P;    /* [k,k]   softmax((QK^T + M)/sqrt(h'))        */
    double *A;    /* [k,h']  P V                                 */
    double *AWo;  /* [k,d]   A W^o (before the diag(r) scaling)  */
} head_state;

static int head_state_alloc(head_state *s, int k, int d, int hp) {
    s->k = k; s->d = d; s->hp = hp;
    s->Xs = (double *)calloc((size_t)k * d, sizeof(double));
    s->Q = (double *)calloc((size_t)k * hp, sizeof(double));
    s->K = (double *)calloc((size_t)k * hp, sizeof(double));
    s->V = (double *)calloc((size_t)k * hp, sizeof(double));
    s->P = (double *)calloc((size_t)k * k, sizeof(double));
    s->A = (double *)calloc((size_t)k * hp, sizeof(double));
    s->AWo = (double *)calloc((size_t)k * d, sizeof(double));
    return (s->Xs && s->Q && s->K && s->V && s->P && s->A && s->AWo) ? 0 : -1;
}

static void head_state_free(head_state *s) {
    free(s->Xs); free(s->Q); free(s->K); free(s->V); free(s->P); free(s->A); free(s->AWo);
}

/* Sec. 2.2 (positional encodings): rotate the first h'/2 entries of v, a
 * query or key row of the token at original position t, by +t theta_p
 * (dir = +1) or back by -t theta_p (dir = -1, the transpose, for gradients);
 * pair p = (2p, 2p+1), theta_p = 10000^(-2p / (h'/2)). */
static void rope_rotate(double *v, int hp, int t, int dir) {
    const int half = hp / 2;
    for (int p = 0; p < half / 2; ++p) {
        const double theta = pow(10000.0, -2.0 * p / (double)half);
        const double ang = dir * (double)t * theta;
        const double c = cos(ang), sn = sin(ang);
        const double x0 = v[2 * p], x1 = v[2 * p + 1];
        v[2 * p] = x0 * c - x1 * sn;
        v[2 * p + 1] = x0 * sn + x1 * c;
    }
}

/* The attention mask M of Sec. 2.2: query i may attend to key j iff
 * I_i >= I_j; with a window w > 0 (local heads, Sec. 3.4) also only within
 * the same block of w original positions. */
static int visible(const int32_t *I, int i, int j, int window) {
    if (I[i] < I[j]) return 0;
    return window <= 0 || I[i] / window == I[j] / window;
}

/* Sec. 2.2, steps gather -> projections (-> RoPE at the original positions
 * I when `rope`) -> masked attention -> A W^o for one head on one sequence.
 * Xb is X[b] ([T,d]); the weights are this head's. */
static void head_forward(const head_state *s, int T, const double *Xb, const int32_t *I,
                         const double *Wq, const double *Wk, const double *Wv,
                         const double *Wo, int rope, int window) {
    const int k = s->k, d = s->d, hp = s->hp;
    (void)T;
    /* X^s = (X_{I_1}, ..., X_{I_k}) */
    for (int i = 0; i < k; ++i)
        for (int c = 0; c < d; ++c) s->Xs[IDX2(i, c, d)] = Xb[IDX2(I[i], c, d)];
    /* Q = X^s W^Q, K = X^s W^K, V = X^s W^V */
    for (int i = 0; i < k; ++i)
        for (int p = 0; p < hp; ++p) {
            double q = 0.0, kk = 0.0, v = 0.0;
            for (int c = 0; c < d; ++c) {
                double x = s->Xs[IDX2(i, c, d)];
                q += x * Wq[IDX2(c, p, hp)];
                kk += x * Wk[IDX2(c, p, hp)];
                v += x * Wv[IDX2(c, p, hp)];
            }
            s->Q[IDX2(i, p, hp)] = q;
            s->K[IDX2(i, p, hp)] = kk;
            s->V[IDX2(i, p, hp)] = v;
        }
    if (rope)
        for (int i = 0; i < k; ++i) {
            rope_rotate(s->Q + IDX2(i, 0, hp), hp, I[i], +1);
            rope_rotate(s->K + IDX2(i, 0, hp), hp, I[i], +1);
        }
    /* P = softmax((QK^T + M) / sqrt(h')), M_ij = 0 iff visible(i, j) (I_i >= I_j,
     * and the same block of a local head) else -inf.  Masked entries get
     * probability exactly 0. */
    const double scale = 1.0 / sqrt((double)hp);
    for (int i = 0; i < k; ++i) {
        double row_max = -INFINITY;
        for (int j = 0; j < k; ++j) {
            if (visible(I, i, j, window)) {
                double dot = 0.0;
                for (int p = 0; p < hp; ++p) dot += s->Q[IDX2(i, p, hp)] * s->K[IDX2(j, p, hp)];
                double sij = dot * scale;
                s->P[IDX2(i, j, k)] = sij;
                if (sij > row_max) row_max = sij;
            }
        }
        double denom = 0.0;
        for (int j = 0; j < k; ++j) {
            if (visible(I, i, j, window)) {
                double e = exp(s->P[IDX2(i, j, k)] - row_max);
                s->P[IDX2(i, j, k)] = e;
                denom += e;
            } else {
                s->P[IDX2(i, j, k)] = 0.0;
            }
        }
        for (int j = 0; j < k; ++j) s->P[IDX2(i, j, k)] /= denom;
    }
    /* A = P V */
    for (int i = 0; i < k; ++i)
        for (int p = 0; p < hp; ++p) {
            double a = 0.0;
            for (int j = 0; j < k; ++j) a += s->P[IDX2(i, j, k)] * s->V[IDX2(j, p, hp)];
            s->A[IDX2(i, p, hp)] = a;
        }
    /* A W^o */
    for (int i = 0; i < k; ++i)
        for (int c = 0; c < d; ++c) {
            double o = 0.0;
            for (int p = 0; p < hp; ++p) o += s->A[IDX2(i, p, hp)] * Wo[IDX2(p, c, d)];
            s->AWo[IDX2(i, c, d)] = o;
        }
}

static int selected(const unsigned char *mask, int i) { return mask == NULL || mask[i] != 0; }

/* Heads on fixed token sets: Y[b] = sum_h scatter(diag(r) A W^o) with the
 * mask window of head_forward.  r is r_sel_in if non-NULL, else
 * sigma(X W^r)[I].  Y [B,T,d] is overwritten. */
static int forward_units(int B, int T, int d, int H, int hp, int k, const double *X,
                         const double *Wr, const double *Wq, const double *Wk,
                         const double *Wv, const double *Wo, const int32_t *I,
                         const double *r_sel_in, double *Y, const unsigned char *bsel,
                         const unsigned char *hsel, int rope, int window) {
    if (B <= 0 || T <= 0 || d <= 0 || H <= 0 || hp <= 0 || k <= 0 || k > T) return -1;
    memset(Y, 0, sizeof(double) * (size_t)B * T * d);
    int failed = 0;
    /* Units (b,h) run in parallel; rows of Y shared between heads are
     * updated atomically. */
    #pragma omp parallel for collapse(2) schedule(dynamic, 1) reduction(| : failed)
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < H; ++h) {
            if (!selected(bsel, b) || !selected(hsel, h)) continue;
            head_state s;
            double *rs = (double *)malloc(sizeof(double) * (size_t)k);
            if (head_state_alloc(&s, k, d, hp) != 0 || !rs) {
                head_state_free(&s); free(rs); failed |= 1; continue;
            }
            const double *Xb = X + IDX3(b, 0, 0, T, d);
            double *Yb = Y + IDX3(b, 0, 0, T, d);
            const int32_t *Ibh = I + IDX3(b, h, 0, H, k);
            for (int i = 0; i < k; ++i) {
                if (r_sel_in) {
                    rs[i] = r_sel_in[IDX3(b, h, i, H, k)];
                } else {
                    double logit = 0.0;
                    for (int c = 0; c < d; ++c) logit += Xb[IDX2(Ibh[i], c, d)] * Wr[IDX2(c, h, H)];
                    rs[i] = sigmoid(logit);
                }
            }
            head_forward(&s, T, Xb, Ibh, Wq + IDX3(h, 0, 0, d, hp), Wk + IDX3(h, 0, 0, d, hp),
                         Wv + IDX3(h, 0, 0, d, hp), Wo + IDX3(h, 0, 0, hp, d), rope, window);
            /* X^o = diag(r^topk) A W^o;  Y_{I_i} += X^o_i  (Eq. mosa_mha sums the heads) */
            for (int i = 0; i < k; ++i)
                for (int c = 0; c < d; ++c) {
                    #pragma omp atomic
                    Yb[IDX2(Ibh[i], c, d)] += rs[i] * s.AWo[IDX2(i, c, d)];
                }
            free(rs);
            head_state_free(&s);
        }
    return failed ? -1 : 0;
}

/* Forward of the layer with the token sets fixed by the caller.
 * I [B,H,k]; if r_sel_in is non-NULL it is used as r^topk (the fixed-sparse
 * special case of Sec. 3.1 passes ones), otherwise r^topk = sigma(X W^r)[I]
 * is computed, which keeps W^r differentiable with TopK held constant.
 * Y [B,T,d] is overwritten: Y[b] = sum_h scatter(diag(r^topk) A W^o).
 * Returns 0 or -1. */
int oracle_forward_indices(int B, int T, int d, int H, int hp, int k, const double *X,
                           const double *Wr, const double *Wq, const double *Wk,
                           const double *Wv, const double *Wo, const int32_t *I,
                           const double *r_sel_in, double *Y, const unsigned char *bsel,
                           const unsigned char *hsel, int rope) {
    return forward_units(B, T, d, H, hp, k, X, Wr, Wq, Wk, Wv, Wo, I, r_sel_in, Y, bsel, hsel,
                         rope, 0);
}

/* Full forward: router -> TopK -> heads -> sum (Sec. 2.2, Eq. mosa_mha).
 * Writes Y [B,T,d], I [B,H,k], r_sel [B,H,k] and, if non-NULL, r_full [B,H,T].
 * With masks, I / r_sel / r_full are written for the selected units only. */
int oracle_forward(int B, int T, int d, int H, int hp, int k, const double *X,
                   const double *Wr, const double *Wq, const double *Wk, const double *Wv,
                   const double *Wo, double *Y, int32_t *I, double *r_sel, double *r_full,
                   const unsigned char *bsel, const unsigned char *hsel, int first_token,
                   int rope) {
    if (B <= 0 || T <= 0 || d <= 0 || H <= 0 || hp <= 0 || k <= 0 || k > T) return -1;
    int failed = 0;
    #pragma omp parallel for collapse(2) schedule(dynamic, 1) reduction(| : failed)
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < H; ++h) {
            if (!selected(bsel, b) || !selected(hsel, h)) continue;
            double *r = (double *)malloc(sizeof(double) * (size_t)T);
            if (!r) { failed |= 1; continue; }
            for (int t = 0; t < T; ++t) {
                double logit = 0.0;
                for (int c = 0; c < d; ++c) logit += X[IDX3(b, t, c, T, d)] * Wr[IDX2(c, h, H)];
                r[t] = sigmoid(logit);
            }
            if (r_full)
                for (int t = 0; t < T; ++t) r_full[IDX3(b, h, t, H, T)] = r[t];
            int32_t *Ib = I + IDX3(b, h, 0, H, k);
            double *rb = r_sel + IDX3(b, h, 0, H, k);
            if ((first_token ? oracle_topk_first(T, k, r, Ib, rb) : oracle_topk(T, k, r, Ib, rb)) != 0)
                failed |= 1;
            free(r);
        }
    if (failed) return -1;
    return oracle_forward_indices(B, T, d, H, hp, k, X, Wr, Wq, Wk, Wv, Wo, I, r_sel, Y, bsel,
                                  hsel, rope);
}

/* Backward of the layer for the token sets I (TopK held constant, Sec. 2.2):
 * the gradient reaches W^r and X through r^topk = sigma(X W^r)[I] only.
 * All outputs are overwritten.  The chain rule, step by step, for one head:
 *   dX^o      = dY[I]                               (scatter is a copy)
 *   dr_i      = <dX^o_i, (A W^o)_i>                 (X^o = diag(r) A W^o)
 *   dW^o     += (diag(r) A)^T dX^o
 *   dA        = diag(r) dX^o (W^o)^T
 *   dV        = P^T dA,   dP = dA V^T
 *   dS_ij     = P_ij (dP_ij - sum_l P_il dP_il)     (softmax; masked P = 0)
 *   dQ        = dS K / sqrt(h'),   dK = dS^T Q / sqrt(h')   (Q, K after RoPE)
 *   with RoPE: dQ, dK rotated back to the projections' outputs (transpose)
 *   dW^{Q,K,V}+= X^s^T d{Q,K,V}
 *   dlogit_i  = dr_i r_i (1 - r_i)                  (sigma' = sigma (1 - sigma))
 *   dW^r     += X^s^T dlogit
 *   dX[I]    += dQ W^Q^T + dK W^K^T + dV W^V^T + dlogit W^r^T
 * Returns 0 or -1. */
/* The chain rule above for heads on fixed token sets.  With `unit_scores`
 * the heads have no router (r = 1, Sec. 2.1): the dr, dlogit and W^r terms
 * are absent and dWr / Wr are not touched (may be NULL).  `window` as in
 * head_forward. */
static int backward_units(int B, int T, int d, int H, int hp, int k, const double *X,
                          const double *Wr, const double *Wq, const double *Wk,
                          const double *Wv, const double *Wo, const int32_t *I,
                          const double *dY, double *dX, double *dWr, double *dWq, double *dWk,
                          double *dWv, double *dWo, const unsigned char *bsel,
                          const unsigned char *hsel, int rope, int unit_scores, int window) {
    if (B <= 0 || T <= 0 || d <= 0 || H <= 0 || hp <= 0 || k <= 0 || k > T) return -1;
    memset(dX, 0, sizeof(double) * (size_t)B * T * d);
    if (!unit_scores) memset(dWr, 0, sizeof(double) * (size_t)d * H);
    memset(dWq, 0, sizeof(double) * (size_t)H * d * hp);
    memset(dWk, 0, sizeof(double) * (size_t)H * d * hp);
    memset(dWv, 0, sizeof(double) * (size_t)H * d * hp);
    memset(dWo, 0, sizeof(double) * (size_t)H * hp * d);
    const double scale = 1.0 / sqrt((double)hp);
    int failed = 0;
    /* Units (h,b) run in parallel; every shared accumulation (rows of dX,
     * weight gradients) is an atomic add. */
    #pragma omp parallel for collapse(2) schedule(dynamic, 1) reduction(| : failed)
    for (int h = 0; h < H; ++h)
    for (int b = 0; b < B; ++b) {
        if (!selected(hsel, h) || !selected(bsel, b)) continue;
        head_state s;
        if (head_state_alloc(&s, k, d, hp) != 0) { head_state_free(&s); failed |= 1; continue; }
        double *rs = (double *)malloc(sizeof(double) * (size_t)k);
        double *dXo = (double *)malloc(sizeof(double) * (size_t)k * d);
        double *dr = (double *)malloc(sizeof(double) * (size_t)k);
        double *dA = (double *)malloc(sizeof(double) * (size_t)k * hp);
        double *dV = (double *)malloc(sizeof(double) * (size_t)k * hp);
        double *dS = (double *)malloc(sizeof(double) * (size_t)k * k);
        double *dQ = (double *)malloc(sizeof(double) * (size_t)k * hp);
        double *dK = (double *)malloc(sizeof(double) * (size_t)k * hp);
        double *dlogit = (double *)malloc(sizeof(double) * (size_t)k);
        if (!rs || !dXo || !dr || !dA || !dV || !dS || !dQ || !dK || !dlogit) failed |= 1;
        const double *Wq_h = Wq + IDX3(h, 0, 0, d, hp), *Wk_h = Wk + IDX3(h, 0, 0, d, hp);
        const double *Wv_h = Wv + IDX3(h, 0, 0, d, hp), *Wo_h = Wo + IDX3(h, 0, 0, hp, d);
        double *dWq_h = dWq + IDX3(h, 0, 0, d, hp), *dWk_h = dWk + IDX3(h, 0, 0, d, hp);
        double *dWv_h = dWv + IDX3(h, 0, 0, d, hp), *dWo_h = dWo + IDX3(h, 0, 0, hp, d);
        if (!failed) {
            const double *Xb = X + IDX3(b, 0, 0, T, d);
            const double *dYb = dY + IDX3(b, 0, 0, T, d);
            double *dXb = dX + IDX3(b, 0, 0, T, d);
            const int32_t *Ibh = I + IDX3(b, h, 0, H, k);
            for (int i = 0; i < k; ++i) {
                if (unit_scores) { rs[i] = 1.0; continue; }
                double logit = 0.0;
                for (int c = 0; c < d; ++c) logit += Xb[IDX2(Ibh[i], c, d)] * Wr[IDX2(c, h, H)];
                rs[i] = sigmoid(logit);
            }
            head_forward(&s, T, Xb, Ibh, Wq_h, Wk_h, Wv_h, Wo_h, rope, window);
            /* dX^o = dY[I] */
            for (int i = 0; i < k; ++i)
                for (int c = 0; c < d; ++c) dXo[IDX2(i, c, d)] = dYb[IDX2(Ibh[i], c, d)];
            /* dr_i = <dX^o_i, (A W^o)_i> */
            for (int i = 0; i < k; ++i) {
                double acc = 0.0;
                for (int c = 0; c < d; ++c) acc += dXo[IDX2(i, c, d)] * s.AWo[IDX2(i, c, d)];
                dr[i] = acc;
            }
            /* dW^o += (diag(r) A)^T dX^o */
            for (int p = 0; p < hp; ++p)
                for (int c = 0; c < d; ++c) {
                    double acc = 0.0;
                    for (int i = 0; i < k; ++i)
                        acc += rs[i] * s.A[IDX2(i, p, hp)] * dXo[IDX2(i, c, d)];
                    #pragma omp atomic
                    dWo_h[IDX2(p, c, d)] += acc;
                }
            /* dA = diag(r) dX^o W^o^T */
            for (int i = 0; i < k; ++i)
                for (int p = 0; p < hp; ++p) {
                    double acc = 0.0;
                    for (int c = 0; c < d; ++c) acc += dXo[IDX2(i, c, d)] * Wo_h[IDX2(p, c, d)];
                    dA[IDX2(i, p, hp)] = rs[i] * acc;
                }
            /* dV = P^T dA */
            for (int j = 0; j < k; ++j)
                for (int p = 0; p < hp; ++p) {
                    double acc = 0.0;
                    for (int i = 0; i < k; ++i) acc += s.P[IDX2(i, j, k)] * dA[IDX2(i, p, hp)];
                    dV[IDX2(j, p, hp)] = acc;
                }
            /* dP = dA V^T;  dS = P o (dP - rowsum(P o dP)) */
            for (int i = 0; i < k; ++i) {
                double rowsum = 0.0;
                for (int j = 0; j < k; ++j) {
                    double dp = 0.0;
                    for (int p = 0; p < hp; ++p) dp += dA[IDX2(i, p, hp)] * s.V[IDX2(j, p, hp)];
                    dS[IDX2(i, j, k)] = dp;
                    rowsum += s.P[IDX2(i, j, k)] * dp;
                }
                for (int j = 0; j < k; ++j)
                    dS[IDX2(i, j, k)] = s.P[IDX2(i, j, k)] * (dS[IDX2(i, j, k)] - rowsum);
            }
            /* dQ = dS K / sqrt(h'),  dK = dS^T Q / sqrt(h') */
            for (int i = 0; i < k; ++i)
                for (int p = 0; p < hp; ++p) {
                    double aq = 0.0, ak = 0.0;
                    for (int j = 0; j < k; ++j) {
                        aq += dS[IDX2(i, j, k)] * s.K[IDX2(j, p, hp)];
                        ak += dS[IDX2(j, i, k)] * s.Q[IDX2(j, p, hp)];
                    }
                    dQ[IDX2(i, p, hp)] = aq * scale;
                    dK[IDX2(i, p, hp)] = ak * scale;
                }
            if (rope)
                for (int i = 0; i < k; ++i) {
                    rope_rotate(dQ + IDX2(i, 0, hp), hp, Ibh[i], -1);
                    rope_rotate(dK + IDX2(i, 0, hp), hp, Ibh[i], -1);
                }
            /* dlogit = dr o r o (1 - r); no router term for heads without one */
            for (int i = 0; i < k; ++i)
                dlogit[i] = unit_scores ? 0.0 : dr[i] * rs[i] * (1.0 - rs[i]);
            /* dW^{Q,K,V} += X^s^T d{Q,K,V};  dW^r[:,h] += X^s^T dlogit */
            for (int c = 0; c < d; ++c) {
                for (int p = 0; p < hp; ++p) {
                    double aq = 0.0, ak = 0.0, av = 0.0;
                    for (int i = 0; i < k; ++i) {
                        double x = s.Xs[IDX2(i, c, d)];
                        aq += x * dQ[IDX2(i, p, hp)];
                        ak += x * dK[IDX2(i, p, hp)];
                        av += x * dV[IDX2(i, p, hp)];
                    }
                    #pragma omp atomic
                    dWq_h[IDX2(c, p, hp)] += aq;
                    #pragma omp atomic
                    dWk_h[IDX2(c, p, hp)] += ak;
                    #pragma omp atomic
                    dWv_h[IDX2(c, p, hp)] += av;
                }
                if (unit_scores) continue;
                double ar = 0.0;
                for (int i = 0; i < k; ++i) ar += s.Xs[IDX2(i, c, d)] * dlogit[i];
                #pragma omp atomic
                dWr[IDX2(c, h, H)] += ar;
            }
            /* dX[I] += dQ W^Q^T + dK W^K^T + dV W^V^T + dlogit W^r[:,h]^T */
            for (int i = 0; i < k; ++i)
                for (int c = 0; c < d; ++c) {
                    double acc = unit_scores ? 0.0 : dlogit[i] * Wr[IDX2(c, h, H)];
                    for (int p = 0; p < hp; ++p)
                        acc += dQ[IDX2(i, p, hp)] * Wq_h[IDX2(c, p, hp)] +
                               dK[IDX2(i, p, hp)] * Wk_h[IDX2(c, p, hp)] +
                               dV[IDX2(i, p, hp)] * Wv_h[IDX2(c, p, hp)];
                    #pragma omp atomic
                    dXb[IDX2(Ibh[i], c, d)] += acc;
                }
        }
        free(rs); free(dXo); free(dr); free(dA); free(dV); free(dS); free(dQ); free(dK);
        free(dlogit);
        head_state_free(&s);
    }
    return failed ? -1 : 0;
}

/* Backward of the layer for the token sets I: the chain rule above with
 * r^topk = sigma(X W^r)[I].  All outputs are overwritten.  Returns 0 or -1. */
int oracle_backward(int B, int T, int d, int H, int hp, int k, const double *X,
                    const double *Wr, const double *Wq, const double *Wk, const double *Wv,
                    const double *Wo, const int32_t *I, const double *dY, double *dX,
                    double *dWr, double *dWq, double *dWk, double *dWv, double *dWo,
                    const unsigned char *bsel, const unsigned char *hsel, int rope) {
    return backward_units(B, T, d, H, hp, k, X, Wr, Wq, Wk, Wv, Wo, I, dY, dX, dWr, dWq, dWk,
                          dWv, dWo, bsel, hsel, rope, 0, 0);
}

/* I [B,H,T] = 0..T-1 for every (b,h): a dense head sees every token. */
static int32_t *all_tokens(int B, int H, int T) {
    int32_t *I = (int32_t *)malloc(sizeof(int32_t) * (size_t)B * H * T);
    if (!I) return NULL;
    for (size_t u = 0; u < (size_t)B * H; ++u)
        for (int t = 0; t < T; ++t) I[u * T + t] = t;
    return I;
}

/* Dense heads of a hybrid layer (Sec. 2.2, hybridization): multi-head
 * attention of Sec. 2.1, Eq. (mha), Y[b] = sum_h Attention(X W^Q_h, X W^K_h,
 * X W^V_h, M) W^O_h over all T tokens, causal M, no router; window > 0 makes
 * them the local heads of Sec. 3.4 (same block of `window` positions only).
 * RoPE, if on, at the positions 0..T-1.  Y is overwritten.  Returns 0 or -1. */
int oracle_dense_forward(int B, int T, int d, int H, int hp, int window, const double *X,
                         const double *Wq, const double *Wk, const double *Wv,
                         const double *Wo, double *Y, const unsigned char *bsel,
                         const unsigned char *hsel, int rope) {
    if (B <= 0 || T <= 0 || H <= 0 || window < 0) return -1;
    int32_t *I = all_tokens(B, H, T);
    double *ones = (double *)malloc(sizeof(double) * (size_t)B * H * T);
    int rc = -1;
    if (I && ones) {
        for (size_t i = 0; i < (size_t)B * H * T; ++i) ones[i] = 1.0;
        rc = forward_units(B, T, d, H, hp, T, X, NULL, Wq, Wk, Wv, Wo, I, ones, Y, bsel, hsel,
                           rope, window);
    }
    free(I);
    free(ones);
    return rc;
}

/* Gradients of sum(Y * dY) for the dense (or local) heads above: dX, dW^Q,
 * dW^K, dW^V, dW^O (overwritten), by the chain rule of oracle_backward with
 * r = 1 and no router terms.  Returns 0 or -1. */
int oracle_dense_backward(int B, int T, int d, int H, int hp, int window, const double *X,
                          const double *Wq, const double *Wk, const double *Wv,
                          const double *Wo, const double *dY, double *dX, double *dWq,
                          double *dWk, double *dWv, double *dWo, const unsigned char *bsel,
                          const unsigned char *hsel, int rope) {
    if (B <= 0 || T <= 0 || H <= 0 || window < 0) return -1;
    int32_t *I = all_tokens(B, H, T);
    int rc = -1;
    if (I)
        rc = backward_units(B, T, d, H, hp, T, X, NULL, Wq, Wk, Wv, Wo, I, dY, dX, NULL, dWq, dWk,
                            dWv, dWo, bsel, hsel, rope, 1, window);
    free(I);
    return rc;
}
