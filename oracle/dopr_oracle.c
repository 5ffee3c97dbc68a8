/*
 * dopr_oracle.c -- plain fp64 CPU oracle for the DoPR online scoring pass.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, obviously-correct
 * restatement of what the GPU library computes.  Only the test suite, the
 * package smoke check and the CPU-baseline leg of the benchmark may load it;
 * the product path never does, and this file shares no code, header, table
 * or constant with the CUDA library.
 *
 * What it computes (DoPR, Sec. 3.1 "Problem Formulation" and Sec. 3.4
 * "Online Reranking"): for a query q and a document d whose compressed prefix
 * states C~_d (per-layer key/value states of m_d prefix positions) were
 * stored offline, run the decoder over the online input [q ; t_score] only,
 * with every attention layer also attending to the stored prefix keys/values,
 * and read the relevance score at the score token.  The decoder is a
 * Qwen3-style block stack (the paper's backbone, Sec. 4.1): pre-RMSNorm,
 * grouped-query attention with per-head RMSNorm on q and k, rotary position
 * embedding, SwiGLU feed-forward, residual connections.  The score is the
 * difference of two output-row logits (yes minus no) after the final norm.
 *
 * Readings where the paper is silent (each one listed in the design notes):
 *   - positions: prefix slot i sits at position i (0..m-1); online token j of
 *     [q ; t_score] sits at position m + j;
 *   - stored prefix K is the post-QK-norm, post-RoPE key; stored V is the raw
 *     value projection; neither is re-normalised nor re-rotated here;
 *   - RoPE is the rotate-half form on pairs (i, i + D/2) with angular
 *     frequency theta^(-2i/D);
 *   - q head h reads kv head floor(h / G), G = Hq / Hkv;
 *   - RMSNorm(x) = x / sqrt(mean(x^2) + eps) * g;
 *   - score = <W_s[0], RMSNorm(h_last) * g_final> - <W_s[1], ...> (or, with the
 *     optional MLP head, one hidden layer over the same normed state).
 *
 * Also here: the attention-based key token selection of Sec. 3.2.1 (the
 * last layer's head-averaged attention weights from oracle_forward, the
 * column top-p salience, the top-K positions), which the offline prefix
 * construction feeds from.  The paper leaves p open; ties in the ranking go to
 * the lower position and the selected positions come out in ascending order.
 *
 * Everything is fp64.  Weights and stored states arrive as bf16 bit
 * patterns (uint16) or fp64 and are widened exactly; no intermediate value
 * is rounded.  Parallelism (OpenMP) is only over independent outputs (one
 * output feature or one head per iteration); every individual sum runs in
 * index order, so results do not depend on the thread count.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef struct {
    int32_t n_layers, hidden, n_q_heads, n_kv_heads, head_dim, ffn, vocab;
    int32_t score_token_id;
    double rope_theta, rms_eps;
    /* bf16 bit patterns; matrices are [out][in] row-major (y = W x). */
    const uint16_t *embed;               /* [vocab][hidden]               */
    const uint16_t *const *attn_norm;    /* [L] -> [hidden]               */
    const uint16_t *const *wq;           /* [L] -> [Hq*D][hidden]         */
    const uint16_t *const *wk;           /* [L] -> [Hkv*D][hidden]        */
    const uint16_t *const *wv;           /* [L] -> [Hkv*D][hidden]        */
    const uint16_t *const *q_norm;       /* [L] -> [D]                    */
    const uint16_t *const *k_norm;       /* [L] -> [D]                    */
    const uint16_t *const *wo;           /* [L] -> [hidden][Hq*D]         */
    const uint16_t *const *mlp_norm;     /* [L] -> [hidden]               */
    const uint16_t *const *w_gate;       /* [L] -> [ffn][hidden]          */
    const uint16_t *const *w_up;         /* [L] -> [ffn][hidden]          */
    const uint16_t *const *w_down;       /* [L] -> [hidden][ffn]          */
    const uint16_t *final_norm;          /* [hidden]                      */
    const uint16_t *score_head;          /* [2][hidden]: row 0 yes, 1 no  */
} oracle_model;

enum { ORACLE_OK = 0, ORACLE_ERR_ARG = 1, ORACLE_ERR_NOMEM = 2 };

/* Exact widening of a bf16 bit pattern. */
double oracle_bf16_to_f64(uint16_t b)
{
    union { uint32_t u; float f; } c;
    c.u = (uint32_t)b << 16;
    return (double)c.f;
}

int oracle_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* RMSNorm of one vector: y = x / sqrt(mean(x^2) + eps) * g. */
void oracle_rmsnorm(const double *x, const double *g, int n, double eps, double *y)
{
    double ss = 0.0;
    for (int i = 0; i < n; ++i) ss += x[i] * x[i];
    double inv = 1.0 / sqrt(ss / (double)n + eps);
    for (int i = 0; i < n; ++i) y[i] = x[i] * inv * g[i];
}

/* Rotary position embedding, rotate-half form, in place on one head
 * vector of even length D at position pos. */
void oracle_rope(double *x, int D, double pos, double theta)
{
    int half = D / 2;
    for (int i = 0; i < half; ++i) {
        double freq = pow(theta, -2.0 * (double)i / (double)D);
        double a = pos * freq;
        double c = cos(a), s = sin(a);
        double x1 = x[i], x2 = x[i + half];
        x[i] = x1 * c - x2 * s;
        x[i + half] = x2 * c + x1 * s;
    }
}

/* Softmax attention of one query over n keys: out = sum_i p_i v_i with
 * p = softmax(<q, k_i> * scale).  K and V are [n][D] row-major. */
void oracle_attend(const double *q, const double *K, const double *V, int n, int D,
                   double scale, double *out)
{
    for (int d = 0; d < D; ++d) out[d] = 0.0;
    if (n <= 0) return;
    double *s = (double *)malloc(sizeof(double) * (size_t)n);
    if (!s) return;
    double mx = -INFINITY;
    for (int i = 0; i < n; ++i) {
        double acc = 0.0;
        for (int d = 0; d < D; ++d) acc += q[d] * K[(size_t)i * D + d];
        s[i] = acc * scale;
        if (s[i] > mx) mx = s[i];
    }
    double z = 0.0;
    for (int i = 0; i < n; ++i) { s[i] = exp(s[i] - mx); z += s[i]; }
    for (int i = 0; i < n; ++i) {
        double p = s[i] / z;
        for (int d = 0; d < D; ++d) out[d] += p * V[(size_t)i * D + d];
    }
    free(s);
}

/* The softmax weights themselves: p[i] = exp(s_i - max) / sum_j exp(s_j - max),
 * s_i = <q, K_i> * scale, i < n (the weights oracle_attend applies to V). */
void oracle_attn_probs(const double *q, const double *K, int n, int D, double scale, double *p)
{
    if (n <= 0) return;
    double mx = -INFINITY;
    for (int i = 0; i < n; ++i) {
        double acc = 0.0;
        for (int d = 0; d < D; ++d) acc += q[d] * K[(size_t)i * D + d];
        p[i] = acc * scale;
        if (p[i] > mx) mx = p[i];
    }
    double z = 0.0;
    for (int i = 0; i < n; ++i) { p[i] = exp(p[i] - mx); z += p[i]; }
    for (int i = 0; i < n; ++i) p[i] /= z;
}

double oracle_silu(double x) { return x / (1.0 + exp(-x)); }

/* Y[t][o] = sum_i X[t][i] * W[o][i] for t < T, o < out; W is bf16. */
static void linear_bf16(const double *X, int T, int in, const uint16_t *W, int out, double *Y)
{
    #pragma omp parallel
    {
        double *wrow = (double *)malloc(sizeof(double) * (size_t)in);
        #pragma omp for schedule(static)
        for (int o = 0; o < out; ++o) {
            const uint16_t *w = W + (size_t)o * in;
            for (int i = 0; i < in; ++i) wrow[i] = oracle_bf16_to_f64(w[i]);
            for (int t = 0; t < T; ++t) {
                const double *x = X + (size_t)t * in;
                double acc = 0.0;
                for (int i = 0; i < in; ++i) acc += x[i] * wrow[i];
                Y[(size_t)t * out + o] = acc;
            }
        }
        free(wrow);
    }
}

static void widen(const uint16_t *src, int n, double *dst)
{
    for (int i = 0; i < n; ++i) dst[i] = oracle_bf16_to_f64(src[i]);
}

/*
 * One causal decoder pass over T online input vectors x0[T][H] at positions
 * pos0 .. pos0+T-1, each layer attending to m stored prefix positions
 * (pk/pv: [L][m][Hkv][D] fp64, may be NULL when m == 0) followed by the
 * online keys up to and including its own position.
 *
 * Outputs (any may be NULL except h_out):
 *   h_out   [T][H]            residual stream after the last layer
 *   k_out   [L][T][Hkv][D]    keys the online tokens produced (post norm+RoPE)
 *   v_out   [L][T][Hkv][D]    values the online tokens produced
 *   attn_out[L][T][Hq*D]      attention outputs before the output projection
 *   probs_out[T][m+T]         the last layer's attention weights averaged over
 *                             the q heads (row = attending token, column = key:
 *                             prefix slots, then online tokens; 0 where masked) --
 *                             the matrix A-bar of Sec. 3.2.1 when m == 0
 */
int oracle_forward(const oracle_model *M, int T, const double *x0, int pos0, int m,
                   const double *pk, const double *pv, double *h_out, double *k_out,
                   double *v_out, double *attn_out, double *probs_out)
{
    if (!M || T < 0 || m < 0 || !h_out || (T > 0 && !x0) || (m > 0 && (!pk || !pv)))
        return ORACLE_ERR_ARG;
    const int H = M->hidden, Hq = M->n_q_heads, Hkv = M->n_kv_heads, D = M->head_dim;
    const int F = M->ffn, L = M->n_layers;
    if (Hkv <= 0 || Hq % Hkv != 0 || D % 2 != 0) return ORACLE_ERR_ARG;
    const int G = Hq / Hkv;
    const int S = m + T; /* keys visible to the last online token */
    const double scale = 1.0 / sqrt((double)D);

    double *r = (double *)malloc(sizeof(double) * (size_t)T * H);
    double *xn = (double *)malloc(sizeof(double) * (size_t)T * H);
    double *q = (double *)malloc(sizeof(double) * (size_t)T * Hq * D);
    double *k = (double *)malloc(sizeof(double) * (size_t)T * Hkv * D);
    double *v = (double *)malloc(sizeof(double) * (size_t)T * Hkv * D);
    double *att = (double *)malloc(sizeof(double) * (size_t)T * Hq * D);
    double *Kall = (double *)malloc(sizeof(double) * (size_t)Hkv * S * D);
    double *Vall = (double *)malloc(sizeof(double) * (size_t)Hkv * S * D);
    double *gbuf = (double *)malloc(sizeof(double) * (size_t)T * F);
    double *ubuf = (double *)malloc(sizeof(double) * (size_t)T * F);
    double *dlt = (double *)malloc(sizeof(double) * (size_t)T * H);
    double *gw = (double *)malloc(sizeof(double) * (size_t)(H > D ? H : D));
    int rc = ORACLE_OK;
    if (!r || !xn || !q || !k || !v || !att || !Kall || !Vall || !gbuf || !ubuf || !dlt || !gw) {
        rc = ORACLE_ERR_NOMEM;
        goto done;
    }
    memcpy(r, x0, sizeof(double) * (size_t)T * H);

    for (int l = 0; l < L; ++l) {
        /* input RMSNorm */
        widen(M->attn_norm[l], H, gw);
        for (int t = 0; t < T; ++t) oracle_rmsnorm(r + (size_t)t * H, gw, H, M->rms_eps, xn + (size_t)t * H);
        /* projections */
        linear_bf16(xn, T, H, M->wq[l], Hq * D, q);
        linear_bf16(xn, T, H, M->wk[l], Hkv * D, k);
        linear_bf16(xn, T, H, M->wv[l], Hkv * D, v);
        /* per-head RMSNorm on q and k, then RoPE at position pos0 + t */
        widen(M->q_norm[l], D, gw);
        for (int t = 0; t < T; ++t)
            for (int h = 0; h < Hq; ++h) {
                double *qh = q + ((size_t)t * Hq + h) * D;
                oracle_rmsnorm(qh, gw, D, M->rms_eps, qh);
                oracle_rope(qh, D, (double)(pos0 + t), M->rope_theta);
            }
        widen(M->k_norm[l], D, gw);
        for (int t = 0; t < T; ++t)
            for (int h = 0; h < Hkv; ++h) {
                double *kh = k + ((size_t)t * Hkv + h) * D;
                oracle_rmsnorm(kh, gw, D, M->rms_eps, kh);
                oracle_rope(kh, D, (double)(pos0 + t), M->rope_theta);
            }
        /* key/value sequence per kv head: stored prefix first, then online */
        for (int g = 0; g < Hkv; ++g) {
            for (int i = 0; i < m; ++i) {
                const double *sk = pk + (((size_t)l * m + i) * Hkv + g) * D;
                const double *sv = pv + (((size_t)l * m + i) * Hkv + g) * D;
                memcpy(Kall + ((size_t)g * S + i) * D, sk, sizeof(double) * D);
                memcpy(Vall + ((size_t)g * S + i) * D, sv, sizeof(double) * D);
            }
            for (int t = 0; t < T; ++t) {
                memcpy(Kall + ((size_t)g * S + m + t) * D, k + ((size_t)t * Hkv + g) * D, sizeof(double) * D);
                memcpy(Vall + ((size_t)g * S + m + t) * D, v + ((size_t)t * Hkv + g) * D, sizeof(double) * D);
            }
        }
        if (k_out) memcpy(k_out + (size_t)l * T * Hkv * D, k, sizeof(double) * (size_t)T * Hkv * D);
        if (v_out) memcpy(v_out + (size_t)l * T * Hkv * D, v, sizeof(double) * (size_t)T * Hkv * D);
        /* attention: online token t sees all m prefix keys and online keys 0..t */
        #pragma omp parallel for collapse(2) schedule(static)
        for (int t = 0; t < T; ++t)
            for (int h = 0; h < Hq; ++h) {
                int g = h / G;
                oracle_attend(q + ((size_t)t * Hq + h) * D, Kall + (size_t)g * S * D,
                              Vall + (size_t)g * S * D, m + t + 1, D, scale,
                              att + ((size_t)t * Hq + h) * D);
            }
        if (attn_out) memcpy(attn_out + (size_t)l * T * Hq * D, att, sizeof(double) * (size_t)T * Hq * D);
        if (probs_out && l == L - 1) {
            /* head average of the last layer's weights, heads added in index order */
            #pragma omp parallel
            {
                double *pw = (double *)malloc(sizeof(double) * (size_t)S);
                #pragma omp for schedule(static)
                for (int t = 0; t < T; ++t) {
                    double *row = probs_out + (size_t)t * S;
                    for (int i = 0; i < S; ++i) row[i] = 0.0;
                    for (int h = 0; h < Hq; ++h) {
                        const int kvh = h / G;
                        oracle_attn_probs(q + ((size_t)t * Hq + h) * D, Kall + (size_t)kvh * S * D, m + t + 1, D,
                                          scale, pw);
                        for (int i = 0; i <= m + t; ++i) row[i] += pw[i] / (double)Hq;
                    }
                }
                free(pw);
            }
        }
        /* output projection + residual */
        linear_bf16(att, T, Hq * D, M->wo[l], H, dlt);
        for (size_t i = 0; i < (size_t)T * H; ++i) r[i] += dlt[i];
        /* post-attention RMSNorm, SwiGLU feed-forward, residual */
        widen(M->mlp_norm[l], H, gw);
        for (int t = 0; t < T; ++t) oracle_rmsnorm(r + (size_t)t * H, gw, H, M->rms_eps, xn + (size_t)t * H);
        linear_bf16(xn, T, H, M->w_gate[l], F, gbuf);
        linear_bf16(xn, T, H, M->w_up[l], F, ubuf);
        for (size_t i = 0; i < (size_t)T * F; ++i) gbuf[i] = oracle_silu(gbuf[i]) * ubuf[i];
        linear_bf16(gbuf, T, F, M->w_down[l], H, dlt);
        for (size_t i = 0; i < (size_t)T * H; ++i) r[i] += dlt[i];
    }
    memcpy(h_out, r, sizeof(double) * (size_t)T * H);

done:
    free(r); free(xn); free(q); free(k); free(v); free(att); free(Kall); free(Vall);
    free(gbuf); free(ubuf); free(dlt); free(gw);
    return rc;
}

/* Score head: yes-minus-no logit of the final-normed hidden state h[H]. */
double oracle_score_head(const oracle_model *M, const double *h)
{
    const int H = M->hidden;
    double *g = (double *)malloc(sizeof(double) * (size_t)H);
    double *hn = (double *)malloc(sizeof(double) * (size_t)H);
    if (!g || !hn) { free(g); free(hn); return NAN; }
    widen(M->final_norm, H, g);
    oracle_rmsnorm(h, g, H, M->rms_eps, hn);
    double yes = 0.0, no = 0.0;
    for (int i = 0; i < H; ++i) yes += hn[i] * oracle_bf16_to_f64(M->score_head[i]);
    for (int i = 0; i < H; ++i) no += hn[i] * oracle_bf16_to_f64(M->score_head[(size_t)H + i]);
    free(g); free(hn);
    return yes - no;
}

/*
 * The lightweight MLP scoring head of Sec. 3.2.3, s = MLP(h_score), whose
 * shape the paper does not give: here one hidden layer of width d,
 *   s = sum_j w2[j] * act(sum_i W1[j][i] * hn[i] + b1[j]) + b2,
 * hn = RMSNorm(h) * g_final (the score token's final state), W1 [d][H],
 * b1 [d] and w2 [d] bf16, b2 fp64; act: 0 ReLU, 1 GELU (erf form), 2 SiLU,
 * 3 tanh.
 */
double oracle_mlp_head(const oracle_model *M, const double *h, int d, const uint16_t *W1, const uint16_t *b1,
                       const uint16_t *w2, double b2, int act)
{
    const int H = M->hidden;
    double *g = (double *)malloc(sizeof(double) * (size_t)H);
    double *xs = (double *)malloc(sizeof(double) * (size_t)H);
    if (!g || !xs || d < 1 || act < 0 || act > 3) { free(g); free(xs); return NAN; }
    widen(M->final_norm, H, g);
    oracle_rmsnorm(h, g, H, M->rms_eps, xs);
    double s = b2;
    for (int j = 0; j < d; ++j) {
        double z = oracle_bf16_to_f64(b1[j]);
        for (int i = 0; i < H; ++i) z += oracle_bf16_to_f64(W1[(size_t)j * H + i]) * xs[i];
        double a;
        switch (act) {
            case 0: a = z > 0.0 ? z : 0.0; break;
            case 1: a = 0.5 * z * (1.0 + erf(z / sqrt(2.0))); break;
            case 2: a = oracle_silu(z); break;
            default: a = tanh(z); break;
        }
        s += oracle_bf16_to_f64(w2[j]) * a;
    }
    free(g); free(xs);
    return s;
}

/* Embedding lookup of n token ids into x[n][H]. */
int oracle_embed(const oracle_model *M, int n, const int32_t *ids, double *x)
{
    const int H = M->hidden;
    for (int t = 0; t < n; ++t) {
        if (ids[t] < 0 || ids[t] >= M->vocab) return ORACLE_ERR_ARG;
        widen(M->embed + (size_t)ids[t] * H, H, x + (size_t)t * H);
    }
    return ORACLE_OK;
}

/*
 * Score n_pairs (query, document) pairs.  Query p is
 * q_tokens[q_offsets[p] .. q_offsets[p+1]); the score token is appended
 * here.  pair_doc[p] indexes the document arrays: doc_m[d] prefix length,
 * doc_k[d] / doc_v[d] -> [L][m][Hkv][D] fp64 (NULL allowed when m == 0).
 * Pairs are independent; each is computed alone, in input order.
 */
int oracle_score_pairs(const oracle_model *M, int n_pairs, const int32_t *q_offsets,
                       const int32_t *q_tokens, const int32_t *pair_doc, const int32_t *doc_m,
                       const double *const *doc_k, const double *const *doc_v, double *scores)
{
    if (!M || n_pairs < 0 || (n_pairs > 0 && (!q_offsets || !pair_doc || !doc_m || !scores)))
        return ORACLE_ERR_ARG;
    const int H = M->hidden;
    for (int p = 0; p < n_pairs; ++p) {
        int L = q_offsets[p + 1] - q_offsets[p];
        if (L < 0) return ORACLE_ERR_ARG;
        int T = L + 1;
        int d = pair_doc[p];
        int m = doc_m[d];
        int32_t *ids = (int32_t *)malloc(sizeof(int32_t) * (size_t)T);
        double *x = (double *)malloc(sizeof(double) * (size_t)T * H);
        double *h = (double *)malloc(sizeof(double) * (size_t)T * H);
        int rc = (ids && x && h) ? ORACLE_OK : ORACLE_ERR_NOMEM;
        if (rc == ORACLE_OK) {
            for (int j = 0; j < L; ++j) ids[j] = q_tokens[q_offsets[p] + j];
            ids[L] = M->score_token_id;
            rc = oracle_embed(M, T, ids, x);
        }
        if (rc == ORACLE_OK)
            rc = oracle_forward(M, T, x, m, m, m > 0 ? doc_k[d] : NULL, m > 0 ? doc_v[d] : NULL,
                                h, NULL, NULL, NULL, NULL);
        if (rc == ORACLE_OK) scores[p] = oracle_score_head(M, h + (size_t)(T - 1) * H);
        free(ids); free(x); free(h);
        if (rc != ORACLE_OK) return rc;
    }
    return ORACLE_OK;
}

/* ------------------------------------------------------------------ */
/* Attention-based key token selection (Sec. 3.2.1)                   */

static int cmp_desc(const void *a, const void *b)
{
    const double x = *(const double *)a, y = *(const double *)b;
    return (x < y) - (x > y);
}

/*
 * Salience of each document token from the head-averaged final-layer
 * attention matrix A[n][n] (row = attending token, causal: A[t][i] = 0 for
 * i > t): u_i = the mean of the top_p largest values of column i among its
 * n - i causal entries A[i..n-1][i], i.e. of min(top_p, n - i) values
 * (0-based i; the paper's 1-based min(p, n - i + 1)).
 */
int oracle_salience(int n, const double *A, int top_p, double *u)
{
    if (n < 0 || top_p < 1 || (n > 0 && (!A || !u))) return ORACLE_ERR_ARG;
    double *col = (double *)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    if (!col) return ORACLE_ERR_NOMEM;
    for (int i = 0; i < n; ++i) {
        const int cnt = n - i;
        for (int t = i; t < n; ++t) col[t - i] = A[(size_t)t * n + i];
        qsort(col, (size_t)cnt, sizeof(double), cmp_desc);
        const int k = top_p < cnt ? top_p : cnt;
        double acc = 0.0;
        for (int j = 0; j < k; ++j) acc += col[j];
        u[i] = acc / (double)k;
    }
    free(col);
    return ORACLE_OK;
}

typedef struct { double u; int32_t idx; } sal_key;

static int cmp_sal(const void *a, const void *b)
{
    const sal_key *x = (const sal_key *)a, *y = (const sal_key *)b;
    if (x->u != y->u) return (x->u < y->u) - (x->u > y->u); /* larger salience first */
    return (x->idx > y->idx) - (x->idx < y->idx);          /* then the lower index  */
}

static int cmp_i32(const void *a, const void *b)
{
    const int32_t x = *(const int32_t *)a, y = *(const int32_t *)b;
    return (x > y) - (x < y);
}

/* The positions of the k most salient tokens (k = min(K, n)), equal salience
 * going to the lower position, written in ascending position order; returns k. */
int oracle_select_topk(int n, const double *u, int K, int32_t *idx)
{
    if (n < 0 || K < 0 || (n > 0 && (!u || !idx))) return -1;
    const int k = K < n ? K : n;
    sal_key *keys = (sal_key *)malloc(sizeof(sal_key) * (size_t)(n > 0 ? n : 1));
    if (!keys) return -1;
    for (int i = 0; i < n; ++i) { keys[i].u = u[i]; keys[i].idx = i; }
    qsort(keys, (size_t)n, sizeof(sal_key), cmp_sal);
    for (int j = 0; j < k; ++j) idx[j] = keys[j].idx;
    qsort(idx, (size_t)k, sizeof(int32_t), cmp_i32);
    free(keys);
    return k;
}

/* ------------------------------------------------------------------ */
/* Batch plan: group pairs by document, keep input order inside a group */

typedef struct { int64_t doc; int32_t idx; } pack_key;

static int cmp_pack_key(const void *a, const void *b)
{
    const pack_key *x = (const pack_key *)a, *y = (const pack_key *)b;
    if (x->doc != y->doc) return x->doc < y->doc ? -1 : 1;
    return x->idx < y->idx ? -1 : (x->idx > y->idx ? 1 : 0);
}

/*
 * Packing plan of a batch: pairs ordered by (doc_id, input index), so all
 * pairs of one document are adjacent (the cross-query prefix reuse of
 * Sec. 3.4) and ties keep input order; each pair contributes its query
 * tokens plus the score token, laid end to end in that order.
 *   perm[s]       input index of the pair in sorted slot s        [n]
 *   tok_off[s]    first packed token of sorted pair s             [n+1]
 *   tok_pos[t]    position of packed token t: m_doc + j           [T]
 *   tok_id[t]     token id of packed token t (score id last)      [T]
 *   tok_pair[t]   sorted pair index of packed token t             [T]
 * pair_m[p] is the prefix length of pair p's document.
 */
int oracle_pack_plan(int n, const int32_t *q_offsets, const int32_t *q_tokens,
                     const int64_t *doc_ids, const int32_t *pair_m, int32_t score_token_id,
                     int32_t *perm, int32_t *tok_off, int32_t *tok_pos, int32_t *tok_id,
                     int32_t *tok_pair)
{
    if (n < 0) return ORACLE_ERR_ARG;
    pack_key *keys = (pack_key *)malloc(sizeof(pack_key) * (size_t)(n > 0 ? n : 1));
    if (!keys) return ORACLE_ERR_NOMEM;
    for (int p = 0; p < n; ++p) { keys[p].doc = doc_ids[p]; keys[p].idx = p; }
    qsort(keys, (size_t)n, sizeof(pack_key), cmp_pack_key);
    int32_t off = 0;
    for (int s = 0; s < n; ++s) {
        int p = keys[s].idx;
        perm[s] = p;
        tok_off[s] = off;
        int L = q_offsets[p + 1] - q_offsets[p];
        for (int j = 0; j <= L; ++j) {
            tok_pos[off + j] = pair_m[p] + j;
            tok_id[off + j] = (j < L) ? q_tokens[q_offsets[p] + j] : score_token_id;
            tok_pair[off + j] = s;
        }
        off += L + 1;
    }
    tok_off[n] = off;
    free(keys);
    return ORACLE_OK;
}
