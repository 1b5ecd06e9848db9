/*
 * oracle.c -- plain, slow CPU oracle of the confidence-gated early-exit
 * decode step of a frozen decoder-only transformer.
 *
 * TEST INFRASTRUCTURE.  Only the test suite, the smoke check and the CPU
 * baseline leg of the benchmark load this code; the product path never does.
 * It shares no code, header, table or constant generator with the CUDA
 * library.  Everything is written from the paper's statement of the method:
 *
 *   - Section 2 (definitions): a readout is a square matrix plus an offset
 *     applied to the residual stream at an intermediate layer, whose result
 *     goes through the model's own final normalisation and unembedding
 *     unchanged; the confidence gate accepts the readout's best token when
 *     its probability exceeds a threshold; later tokens consult a key-value
 *     cache that early tokens leave incomplete at skipped layers.
 *   - Section 4, step five: each token runs the layers up to the exit depth;
 *     if the readout's confidence exceeds the threshold the token is emitted,
 *     otherwise the remaining layers run and the full model's token is used;
 *     the skipped layers' cache entries are supplied by projecting the
 *     exit-layer state through those layers' key and value matrices.
 *   - Section 4, step three: more than one exit point is possible.
 *   - Appendix B: greedy decoding (the emitted token is the top-scoring one).
 *   - Section 10: the probability of the best token, the margin between the
 *     best and second-best probabilities, and the negative entropy of the
 *     readout's distribution are interchangeable softmax confidences; the
 *     gate can use any of them (orc_set_confidence).
 *   - Section 2 (nucleus, acceptance) and Section 4, step four: an early
 *     answer is acceptable when it lies in the full model's nucleus (the
 *     most probable tokens holding 90 percent of the probability); the
 *     threshold is the lowest one at which the required share of early
 *     answers is acceptable (orc_select_tau).
 *   - Section 11: a periodic full-depth pass over the most recent tokens
 *     recomputes their cache entries exactly (orc_repass): each token that
 *     exited runs its skipped layers from the residual it exited with.
 *   - Section 4, step five, deferred (orc_set_lazy_fill): a skipped entry is
 *     only read by a later token that runs its layer, so its fill may wait
 *     until the first such token; it is the same projection of the same
 *     exit-layer residual.
 *   - Appendix C: the layer is four attention projections with grouped-query
 *     attention (A query heads, K key-value heads of size D) and a gated
 *     feed-forward block of three matrices of width F.
 *
 * The model family's unstated details (RMSNorm, rotary position embedding in
 * the rotate-half pairing, SwiGLU) follow the standard decoder that the
 * paper's Qwen2.5 models use.  Readings where the paper is silent:
 *   affine readout first, then the final RMSNorm with the model's own gain,
 *   then the unembedding; the KV fill source is the raw exit-layer residual
 *   passed through each skipped layer's own input RMSNorm; the fill happens
 *   in the exit step itself; the gate is strict (p > tau); argmax ties go to
 *   the lowest token id; prefill runs at full depth with no gate; with
 *   several readouts the shallowest passing one exits.
 *
 * Long prompts (prefill_gemm): when the caller supplies a BLAS dgemm, the
 * prompt runs layer by layer over blocks of positions and each matrix-vector
 * product of a block becomes one library matrix product (double sums in the
 * library's order); every other step is the same code in the same order.
 * The pins compare it with the position-by-position prefill.
 *
 * Numerics contract: weights are bf16 values held exactly; activations (the
 * residual stream, RMSNorm outputs, q, scores, softmax, attention output, FFN
 * product, readout output, logits) are float; products accumulate in double;
 * the KV cache holds bf16 values (round to nearest even).  The option
 * bf16_activations additionally rounds every matmul input activation to
 * bf16, the half-precision activations the paper's own runs used.
 *
 * Parity pins (tests/test_oracle_pins.py, tests/test_oracle_model.py): every
 * exported op is checked against closed forms, library routines or brute
 * force; the model against the paper's invariants (tau > 1 reproduces the
 * plain model, tau = 0 always exits and never touches upper-layer query,
 * output or FFN weights, a readout at layer L equal to identity reproduces
 * the final logits) and against special weight settings with closed-form
 * results.  End-to-end logits of a random model have no published value:
 * parity unpinned beyond those checks.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_MAX_READOUTS 8
#define ORC_CONF_PMAX 0    /* p1: probability of the best token           */
#define ORC_CONF_MARGIN 1  /* p1 - p2: margin to the second-best token     */
#define ORC_CONF_NEGENT 2  /* sum_v p_v log p_v: negative entropy (<= 0)   */
#define ORC_FORCE_FREE 0
#define ORC_FORCE_FULL 1
#define ORC_FORCE_EXIT_AT(r) (2 + (r))

typedef struct {
    int32_t n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn_dim, vocab, max_ctx;
    double rms_eps, rope_base;
    int32_t qkv_bias, bf16_activations;
} orc_config;

/* Per-layer tensors are arrays of n_layers pointers to bf16 [out, in]. */
typedef struct {
    const uint16_t* embed;      /* [V, d] */
    const uint16_t* lm_head;    /* [V, d]; NULL means tied to embed */
    const uint16_t* final_norm; /* [d] */
    const uint16_t* const* attn_norm;
    const uint16_t* const* wq; /* [A*D, d] */
    const uint16_t* const* wk; /* [K*D, d] */
    const uint16_t* const* wv; /* [K*D, d] */
    const uint16_t* const* bq; /* [A*D] or NULL array */
    const uint16_t* const* bk;
    const uint16_t* const* bv;
    const uint16_t* const* wo; /* [d, A*D] */
    const uint16_t* const* mlp_norm;
    const uint16_t* const* wg; /* [F, d] */
    const uint16_t* const* wu; /* [F, d] */
    const uint16_t* const* wd; /* [d, F] */
} orc_weights;

typedef struct {
    float p1;        /* top-1 probability */
    float p2;        /* second-best probability */
    float gap;       /* p1 - p2 */
    float max_logit;
    int32_t argmax;  /* lowest index attaining the maximum */
    float neg_entropy; /* sum_v p_v log p_v */
} orc_conf;

typedef struct {
    int32_t token, exited, exit_readout, exit_layer, n_evaluated, full_token;
    int32_t gate_pass[ORC_MAX_READOUTS];
    int32_t readout_token[ORC_MAX_READOUTS];
    float confidence[ORC_MAX_READOUTS];
    float gap[ORC_MAX_READOUTS];
    float full_confidence, full_gap;
    /* Full steps with a readout: whether readout 0's token lies in the full
     * model's nucleus (1/0; -1 when not computed) and the full-model
     * probability of the tokens strictly more probable than it. */
    int32_t nucleus_member;
    float nucleus_mass;
} orc_step_result;

/* A BLAS double-precision matrix product (Fortran dgemm calling convention,
 * column-major): C = alpha op(A) op(B) + beta C. */
typedef void (*orc_dgemm_fn)(const char* transa, const char* transb, const int* m, const int* n, const int* k,
                             const double* alpha, const double* a, const int* lda, const double* b, const int* ldb,
                             const double* beta, double* c, const int* ldc);

/* Optional captures of one step; any pointer may be NULL. */
typedef struct {
    float* h_readout;      /* [n_readouts][d]: residual at each evaluated readout */
    float* y_readout;      /* [n_readouts][d]: readout affine output */
    float* readout_logits; /* [n_readouts][V] */
    float* h_final;        /* [d]: residual after layer L (full steps) */
    float* final_logits;   /* [V] */
    float* layer_trace;    /* [L][trace_stride] per-layer internals */
} orc_capture;

typedef struct {
    orc_config c;
    orc_weights w;
    const uint16_t** ptrs; /* owned copies of the per-layer pointer arrays */
    int n_readouts;
    int readout_layer[ORC_MAX_READOUTS];
    const uint16_t* readout_w[ORC_MAX_READOUTS];
    const uint16_t* readout_b[ORC_MAX_READOUTS];
    float* kc;       /* [L][K][max_ctx][D], bf16 values */
    float* vc;
    int8_t* kv_src;  /* [L][max_ctx]: 0 empty (or a deferred fill), 1 computed by the layer, 2 filled */
    float* h_exit;   /* [max_ctx][d]: the residual a position exited with */
    int16_t* exit_at; /* [max_ctx]: layer a position exited after (0: ran every layer) */
    int pos;
    int conf_kind; /* ORC_CONF_*: the signal the gate compares with tau */
    double nucleus_p; /* share of probability the nucleus holds */
    int lazy_fill;    /* 1: exit steps leave their skipped entries empty (flush_layer fills them) */
    orc_dgemm_fn gemm; /* if set, long prompts take their products as BLAS calls (prefill_gemm) */
    int64_t steps, full_steps, exits[ORC_MAX_READOUTS];
    float *h, *u, *q, *kk, *vv, *o, *g, *up, *a, *y, *z, *logits, *tmp;
} orc_model;

/* ------------------------------------------------------------------ */
/* scalar helpers                                                      */
/* ------------------------------------------------------------------ */

static inline float bf16_bits_to_f32(uint16_t b) {
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, 4);
    return f;
}

/* Round a float to the nearest bf16 value, ties to even (NaN stays NaN). */
static inline float round_bf16(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    if ((u & 0x7f800000u) == 0x7f800000u) {
        if (u & 0x007fffffu) u |= 0x00400000u;
        u &= 0xffff0000u;
    } else {
        u += 0x7fffu + ((u >> 16) & 1u);
        u &= 0xffff0000u;
    }
    memcpy(&f, &u, 4);
    return f;
}

static inline float act_round(const orc_model* m, float f) {
    return m->c.bf16_activations ? round_bf16(f) : f;
}

/* ------------------------------------------------------------------ */
/* exported ops (each pinned on its own by the tests)                  */
/* ------------------------------------------------------------------ */

void orc_op_bf16_round(const float* x, int64_t n, float* out) {
    for (int64_t i = 0; i < n; ++i) out[i] = round_bf16(x[i]);
}

/* RMSNorm: out_i = h_i / sqrt(mean(h^2) + eps) * g_i, in double, stored as float. */
void orc_op_rmsnorm(const float* h, const uint16_t* g, int d, double eps, float* out) {
    double ss = 0.0;
    for (int i = 0; i < d; ++i) ss += (double)h[i] * (double)h[i];
    const double inv = 1.0 / sqrt(ss / (double)d + eps);
    for (int i = 0; i < d; ++i) out[i] = (float)((double)h[i] * inv * (double)bf16_bits_to_f32(g[i]));
}

/* out_i = sum_j W[i, j] * x_j (+ b_i), W bf16 row-major [rows, cols], double sums. */
void orc_op_matvec(const uint16_t* W, const uint16_t* b, int64_t rows, int64_t cols,
                   const float* x, float* out) {
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < rows; ++i) {
        const uint16_t* wr = W + i * cols;
        double acc = 0.0;
#pragma omp simd reduction(+ : acc)
        for (int64_t j = 0; j < cols; ++j) acc += (double)bf16_bits_to_f32(wr[j]) * (double)x[j];
        if (b) acc += (double)bf16_bits_to_f32(b[i]);
        out[i] = (float)acc;
    }
}

/* Rotary position embedding of one head vector of size D at position pos:
 * pairs (i, i + D/2) for i < D/2 rotate by angle pos * base^(-2i/D); the
 * angle is formed in double and its cosine and sine rounded to float. */
void orc_op_rope(float* x, int D, int64_t pos, double base) {
    const int half = D / 2;
    for (int i = 0; i < half; ++i) {
        const double theta = pow(base, -2.0 * (double)i / (double)D);
        const double ang = (double)pos * theta;
        const float c = (float)cos(ang), s = (float)sin(ang);
        const double a = x[i], bb = x[i + half];
        x[i] = (float)(a * (double)c - bb * (double)s);
        x[i + half] = (float)(a * (double)s + bb * (double)c);
    }
}

/* Single-query attention of one head over T cached positions:
 * out = softmax(q . K^T / sqrt(D)) V, everything in double. */
void orc_op_attention(const float* q, const float* K, const float* V, int T, int D, float* out) {
    double* s = (double*)malloc(sizeof(double) * (size_t)(T > 0 ? T : 1));
    const double scale = 1.0 / sqrt((double)D);
    double mx = -INFINITY;
    for (int t = 0; t < T; ++t) {
        double acc = 0.0;
#pragma omp simd reduction(+ : acc)
        for (int e = 0; e < D; ++e) acc += (double)q[e] * (double)K[(size_t)t * D + e];
        s[t] = acc * scale;
        if (s[t] > mx) mx = s[t];
    }
    double sum = 0.0;
    for (int t = 0; t < T; ++t) {
        s[t] = exp(s[t] - mx);
        sum += s[t];
    }
    /* out_e = sum_t P_t V[t, e], each dimension's sum taken in position order */
    double* acc = (double*)calloc((size_t)D, sizeof(double));
    for (int t = 0; t < T; ++t) {
        const double p = s[t] / sum;
        const float* vr = V + (size_t)t * D;
        for (int e = 0; e < D; ++e) acc[e] += p * (double)vr[e];
    }
    for (int e = 0; e < D; ++e) out[e] = (float)acc[e];
    free(acc);
    free(s);
}

/* SiLU(x) = x / (1 + exp(-x)). */
double orc_op_silu(double x) { return x / (1.0 + exp(-x)); }

void orc_op_silu_array(const double* x, int64_t n, double* out) {
    for (int64_t i = 0; i < n; ++i) out[i] = orc_op_silu(x[i]);
}

/* Softmax statistics of a logit vector: top-1 probability
 * p1 = 1 / sum_v exp(l_v - max l), the second-best probability and the
 * lowest index attaining the maximum. */
void orc_op_confidence(const float* l, int64_t V, orc_conf* out) {
    float mx = l[0];
    int64_t arg = 0;
    for (int64_t v = 1; v < V; ++v)
        if (l[v] > mx) {
            mx = l[v];
            arg = v;
        }
    float second = -INFINITY;
    for (int64_t v = 0; v < V; ++v)
        if (v != arg && l[v] > second) second = l[v];
    double sum = 0.0;
    for (int64_t v = 0; v < V; ++v) sum += exp((double)l[v] - (double)mx);
    out->p1 = (float)(1.0 / sum);
    out->p2 = V > 1 ? (float)(exp((double)second - (double)mx) / sum) : 0.0f;
    out->gap = out->p1 - out->p2;
    out->max_logit = mx;
    out->argmax = (int32_t)arg;
    /* negative entropy straight from its definition, p log p with 0 log 0 = 0 */
    double ne = 0.0;
    for (int64_t v = 0; v < V; ++v) {
        const double p = exp((double)l[v] - (double)mx) / sum;
        if (p > 0.0) ne += p * log(p);
    }
    out->neg_entropy = (float)ne;
}

/* The gate's signal under the model's confidence kind (Section 10). */
static float conf_signal(const orc_model* m, const orc_conf* cf) {
    switch (m->conf_kind) {
        case ORC_CONF_MARGIN: return cf->gap;
        case ORC_CONF_NEGENT: return cf->neg_entropy;
        default: return cf->p1;
    }
}

/* Nucleus membership (Section 2): token x belongs to the nucleus of share
 * p_nuc when the tokens strictly more probable than x hold less than p_nuc
 * of the probability (the smallest top set reaching p_nuc then includes x,
 * a tied group at the boundary included).  Returns that mass in *mass. */
int orc_op_nucleus_member(const float* l, int64_t V, int32_t x, double p_nuc, double* mass) {
    float mx = l[0];
    for (int64_t v = 1; v < V; ++v)
        if (l[v] > mx) mx = l[v];
    double sum = 0.0, above = 0.0;
    for (int64_t v = 0; v < V; ++v) {
        const double e = exp((double)l[v] - (double)mx);
        sum += e;
        if (l[v] > l[x]) above += e;
    }
    const double mabove = above / sum;
    if (mass) *mass = mabove;
    return mabove < p_nuc ? 1 : 0;
}

int orc_set_nucleus(orc_model* m, double p_nuc) {
    if (!m || !(p_nuc > 0.0 && p_nuc <= 1.0)) return -1;
    m->nucleus_p = p_nuc;
    return 0;
}

/* Section 4, step four: given the readout's confidence conf[i] and whether
 * its answer was acceptable (member[i]) at n held-out positions, the lowest
 * threshold tau at which at least `target` of the early answers (the
 * positions with conf > tau) are acceptable.  Candidates are -inf (every
 * position exits) and each observed confidence; a candidate with no early
 * answer does not count.  *tau = +inf when none meets the target. */
int orc_select_tau(const float* conf, const int32_t* member, int n, double target, float* tau) {
    if (!conf || !member || !tau || n < 0) return -1;
    *tau = INFINITY;
    for (int c = -1; c < n; ++c) {
        const float cand = c < 0 ? -INFINITY : conf[c];
        if (c >= 0 && !(cand < *tau)) continue; /* only lower candidates can improve */
        int early = 0, good = 0;
        for (int i = 0; i < n; ++i)
            if (conf[i] > cand) {
                ++early;
                good += member[i] != 0;
            }
        if (early > 0 && (double)good >= target * (double)early && cand < *tau) *tau = cand;
    }
    return 0;
}

int orc_set_confidence(orc_model* m, int kind) {
    if (!m || kind < ORC_CONF_PMAX || kind > ORC_CONF_NEGENT) return -1;
    m->conf_kind = kind;
    return 0;
}

/* ------------------------------------------------------------------ */
/* model                                                               */
/* ------------------------------------------------------------------ */

/* Floats per layer in a layer trace, and the offsets of its parts:
 * h_in, u_attn, q, k, v, o, h_mid, u_mlp, gate, up, a, h_out. */
int64_t orc_trace_layout(const orc_config* c, int64_t* off) {
    const int64_t d = c->d_model, qd = (int64_t)c->n_heads * c->head_dim,
                  kd = (int64_t)c->n_kv_heads * c->head_dim, F = c->ffn_dim;
    const int64_t sizes[12] = {d, d, qd, kd, kd, qd, d, d, F, F, F, d};
    int64_t acc = 0;
    for (int i = 0; i < 12; ++i) {
        if (off) off[i] = acc;
        acc += sizes[i];
    }
    return acc;
}

static size_t kv_index(const orc_model* m, int j, int g, int t) {
    const orc_config* c = &m->c;
    return (((size_t)j * c->n_kv_heads + g) * (size_t)c->max_ctx + (size_t)t) * (size_t)c->head_dim;
}

void orc_free(orc_model* m) {
    if (!m) return;
    free(m->ptrs);
    free(m->kc);
    free(m->vc);
    free(m->kv_src);
    free(m->h_exit);
    free(m->exit_at);
    free(m->h); free(m->u); free(m->q); free(m->kk); free(m->vv); free(m->o);
    free(m->g); free(m->up); free(m->a); free(m->y); free(m->z); free(m->logits); free(m->tmp);
    free(m);
}

orc_model* orc_create(const orc_config* c, const orc_weights* w) {
    if (!c || !w || c->n_layers <= 0 || c->d_model <= 0 || c->n_heads <= 0 || c->n_kv_heads <= 0 ||
        c->head_dim <= 0 || (c->head_dim % 2) || (c->n_heads % c->n_kv_heads) || c->ffn_dim <= 0 ||
        c->vocab <= 0 || c->max_ctx <= 0)
        return NULL;
    orc_model* m = (orc_model*)calloc(1, sizeof(orc_model));
    if (!m) return NULL;
    m->c = *c;
    m->nucleus_p = 0.9;
    const int L = c->n_layers;
    m->ptrs = (const uint16_t**)calloc((size_t)L * 13, sizeof(uint16_t*));
    const uint16_t* const* src[13] = {w->attn_norm, w->wq, w->wk, w->wv, w->bq, w->bk, w->bv,
                                      w->wo, w->mlp_norm, w->wg, w->wu, w->wd, NULL};
    for (int t = 0; t < 12; ++t)
        for (int j = 0; j < L; ++j) m->ptrs[(size_t)t * L + j] = src[t] ? src[t][j] : NULL;
    m->w = *w;
    m->w.attn_norm = m->ptrs + 0 * L;
    m->w.wq = m->ptrs + 1 * L;
    m->w.wk = m->ptrs + 2 * L;
    m->w.wv = m->ptrs + 3 * L;
    m->w.bq = m->ptrs + 4 * L;
    m->w.bk = m->ptrs + 5 * L;
    m->w.bv = m->ptrs + 6 * L;
    m->w.wo = m->ptrs + 7 * L;
    m->w.mlp_norm = m->ptrs + 8 * L;
    m->w.wg = m->ptrs + 9 * L;
    m->w.wu = m->ptrs + 10 * L;
    m->w.wd = m->ptrs + 11 * L;
    if (!m->w.lm_head) m->w.lm_head = m->w.embed;
    const size_t kvn = (size_t)L * c->n_kv_heads * (size_t)c->max_ctx * c->head_dim;
    m->kc = (float*)calloc(kvn, sizeof(float));
    m->vc = (float*)calloc(kvn, sizeof(float));
    m->kv_src = (int8_t*)calloc((size_t)L * c->max_ctx, 1);
    m->h_exit = (float*)calloc((size_t)c->max_ctx * c->d_model, 4);
    m->exit_at = (int16_t*)calloc((size_t)c->max_ctx, 2);
    const size_t d = (size_t)c->d_model, qd = (size_t)c->n_heads * c->head_dim,
                 kd = (size_t)c->n_kv_heads * c->head_dim, F = (size_t)c->ffn_dim;
    const size_t big = d > qd ? d : qd;
    m->h = (float*)calloc(d, 4);
    m->u = (float*)calloc(d, 4);
    m->q = (float*)calloc(qd, 4);
    m->kk = (float*)calloc(kd, 4);
    m->vv = (float*)calloc(kd, 4);
    m->o = (float*)calloc(qd, 4);
    m->g = (float*)calloc(F, 4);
    m->up = (float*)calloc(F, 4);
    m->a = (float*)calloc(F, 4);
    m->y = (float*)calloc(d, 4);
    m->z = (float*)calloc(d, 4);
    m->logits = (float*)calloc((size_t)c->vocab, 4);
    m->tmp = (float*)calloc(big > F ? big : F, 4);
    if (!m->kc || !m->vc || !m->kv_src || !m->h_exit || !m->exit_at || !m->logits || !m->tmp) {
        orc_free(m);
        return NULL;
    }
    return m;
}

/* Readouts must be added in increasing layer order; layer in [1, L]. */
int orc_add_readout(orc_model* m, int layer, const uint16_t* W, const uint16_t* b) {
    if (!m || m->n_readouts >= ORC_MAX_READOUTS || layer < 1 || layer > m->c.n_layers || !W || !b)
        return -1;
    if (m->n_readouts > 0 && layer <= m->readout_layer[m->n_readouts - 1]) return -1;
    m->readout_layer[m->n_readouts] = layer;
    m->readout_w[m->n_readouts] = W;
    m->readout_b[m->n_readouts] = b;
    return m->n_readouts++;
}

void orc_reset(orc_model* m) {
    const orc_config* c = &m->c;
    const size_t kvn = (size_t)c->n_layers * c->n_kv_heads * (size_t)c->max_ctx * c->head_dim;
    memset(m->kc, 0, kvn * sizeof(float));
    memset(m->vc, 0, kvn * sizeof(float));
    memset(m->kv_src, 0, (size_t)c->n_layers * c->max_ctx);
    memset(m->exit_at, 0, (size_t)c->max_ctx * 2);
    m->pos = 0;
    m->steps = m->full_steps = 0;
    memset(m->exits, 0, sizeof(m->exits));
}

/* Write one position's K and V (already projected; K rotated) as bf16. */
static void store_kv(orc_model* m, int j, int t, const float* k, const float* v, int8_t src) {
    const orc_config* c = &m->c;
    for (int g = 0; g < c->n_kv_heads; ++g) {
        float* kd = m->kc + kv_index(m, j, g, t);
        float* vd = m->vc + kv_index(m, j, g, t);
        for (int e = 0; e < c->head_dim; ++e) {
            kd[e] = round_bf16(k[(size_t)g * c->head_dim + e]);
            vd[e] = round_bf16(v[(size_t)g * c->head_dim + e]);
        }
    }
    m->kv_src[(size_t)j * c->max_ctx + t] = src;
}

/* One decoder layer (0-based index j) at position t, updating h in place. */
static void layer_forward(orc_model* m, int j, int t, float* h, float* tr) {
    const orc_config* c = &m->c;
    const int d = c->d_model, A = c->n_heads, KH = c->n_kv_heads, D = c->head_dim, F = c->ffn_dim;
    const int group = A / KH;
    int64_t off[12];
    orc_trace_layout(c, off);
    if (tr) memcpy(tr + off[0], h, sizeof(float) * d);

    /* attention input: u = bf16(RMSNorm(h) * g_attn) */
    orc_op_rmsnorm(h, m->w.attn_norm[j], d, c->rms_eps, m->u);
    for (int i = 0; i < d; ++i) m->u[i] = act_round(m, m->u[i]);
    /* q, k, v projections (grouped-query: K*D rows for k and v) */
    orc_op_matvec(m->w.wq[j], c->qkv_bias ? m->w.bq[j] : NULL, (int64_t)A * D, d, m->u, m->q);
    orc_op_matvec(m->w.wk[j], c->qkv_bias ? m->w.bk[j] : NULL, (int64_t)KH * D, d, m->u, m->kk);
    orc_op_matvec(m->w.wv[j], c->qkv_bias ? m->w.bv[j] : NULL, (int64_t)KH * D, d, m->u, m->vv);
    for (int hh = 0; hh < A; ++hh) orc_op_rope(m->q + (size_t)hh * D, D, t, c->rope_base);
    for (int g = 0; g < KH; ++g) orc_op_rope(m->kk + (size_t)g * D, D, t, c->rope_base);
    store_kv(m, j, t, m->kk, m->vv, 1);
    if (tr) {
        memcpy(tr + off[1], m->u, sizeof(float) * d);
        memcpy(tr + off[2], m->q, sizeof(float) * A * D);
        for (int g = 0; g < KH; ++g)
            for (int e = 0; e < D; ++e) {
                tr[off[3] + g * D + e] = m->kc[kv_index(m, j, g, t) + e];
                tr[off[4] + g * D + e] = m->vc[kv_index(m, j, g, t) + e];
            }
    }
    /* attention of each query head over its key-value group, positions 0..t
     * (the heads are independent and run on separate host threads) */
#pragma omp parallel for schedule(static)
    for (int hh = 0; hh < A; ++hh) {
        const int g = hh / group;
        orc_op_attention(m->q + (size_t)hh * D, m->kc + kv_index(m, j, g, 0), m->vc + kv_index(m, j, g, 0),
                         t + 1, D, m->o + (size_t)hh * D);
    }
    for (int i = 0; i < A * D; ++i) m->o[i] = act_round(m, m->o[i]);
    /* output projection and residual add */
    orc_op_matvec(m->w.wo[j], NULL, d, (int64_t)A * D, m->o, m->tmp);
    for (int i = 0; i < d; ++i) h[i] = h[i] + m->tmp[i];
    if (tr) {
        memcpy(tr + off[5], m->o, sizeof(float) * A * D);
        memcpy(tr + off[6], h, sizeof(float) * d);
    }
    /* gated feed-forward: a = bf16(SiLU(W_g u) * (W_u u)), h += W_d a */
    orc_op_rmsnorm(h, m->w.mlp_norm[j], d, c->rms_eps, m->u);
    for (int i = 0; i < d; ++i) m->u[i] = act_round(m, m->u[i]);
    orc_op_matvec(m->w.wg[j], NULL, F, d, m->u, m->g);
    orc_op_matvec(m->w.wu[j], NULL, F, d, m->u, m->up);
    for (int i = 0; i < F; ++i) m->a[i] = act_round(m, (float)(orc_op_silu(m->g[i]) * (double)m->up[i]));
    orc_op_matvec(m->w.wd[j], NULL, d, F, m->a, m->tmp);
    for (int i = 0; i < d; ++i) h[i] = h[i] + m->tmp[i];
    if (tr) {
        memcpy(tr + off[7], m->u, sizeof(float) * d);
        memcpy(tr + off[8], m->g, sizeof(float) * F);
        memcpy(tr + off[9], m->up, sizeof(float) * F);
        memcpy(tr + off[10], m->a, sizeof(float) * F);
        memcpy(tr + off[11], h, sizeof(float) * d);
    }
}

/* KV repair for a skipped layer j at position t: project the exit-layer
 * residual hk through layer j's input RMSNorm and its key and value
 * matrices; the key is rotated at position t. */
static void kv_fill(orc_model* m, int j, int t, const float* hk) {
    const orc_config* c = &m->c;
    const int d = c->d_model, KH = c->n_kv_heads, D = c->head_dim;
    orc_op_rmsnorm(hk, m->w.attn_norm[j], d, c->rms_eps, m->u);
    for (int i = 0; i < d; ++i) m->u[i] = act_round(m, m->u[i]);
    orc_op_matvec(m->w.wk[j], c->qkv_bias ? m->w.bk[j] : NULL, (int64_t)KH * D, d, m->u, m->kk);
    orc_op_matvec(m->w.wv[j], c->qkv_bias ? m->w.bv[j] : NULL, (int64_t)KH * D, d, m->u, m->vv);
    for (int g = 0; g < KH; ++g) orc_op_rope(m->kk + (size_t)g * D, D, t, c->rope_base);
    store_kv(m, j, t, m->kk, m->vv, 2);
}

/* Deferred fills of layer j (0-based) needed before position t reads it:
 * every position p < t that exited after layer k <= j and whose entry at
 * layer j is still empty gets the fill kv_fill would have written in its
 * exit step, from the residual it exited with.  Nothing to do unless the
 * lazy fill is on. */
static void flush_layer(orc_model* m, int j, int t) {
    if (!m->lazy_fill) return;
    const orc_config* c = &m->c;
    for (int p = 0; p < t; ++p) {
        const int k = m->exit_at[p];
        if (k > 0 && k <= j && m->kv_src[(size_t)j * c->max_ctx + p] == 0)
            kv_fill(m, j, p, m->h_exit + (size_t)p * c->d_model);
    }
}

/* Every deferred fill at positions before the current one. */
int orc_flush_fills(orc_model* m) {
    if (!m) return -1;
    const int lazy = m->lazy_fill;
    m->lazy_fill = 1;
    for (int j = 0; j < m->c.n_layers; ++j) flush_layer(m, j, m->pos);
    m->lazy_fill = lazy;
    return 0;
}

/* on = 1: exit steps defer their fills; on = 0 fills every deferred entry
 * first, then fills in the exit step again. */
int orc_set_lazy_fill(orc_model* m, int on) {
    if (!m || (on != 0 && on != 1)) return -1;
    if (!on) orc_flush_fills(m);
    m->lazy_fill = on;
    return 0;
}

/* Final normalisation + unembedding of a residual-space vector x:
 * logits = U bf16(RMSNorm(x) * g_final). */
static void unembed(orc_model* m, const float* x, float* logits) {
    const orc_config* c = &m->c;
    orc_op_rmsnorm(x, m->w.final_norm, c->d_model, c->rms_eps, m->z);
    for (int i = 0; i < c->d_model; ++i) m->z[i] = act_round(m, m->z[i]);
    orc_op_matvec(m->w.lm_head, NULL, c->vocab, c->d_model, m->z, logits);
}

/* Readout r applied to the residual h: y = W_r bf16(h) + b_r, then the
 * model's own final normalisation and unembedding. */
static void readout(orc_model* m, int r, const float* h, float* y, float* logits) {
    const orc_config* c = &m->c;
    for (int i = 0; i < c->d_model; ++i) m->tmp[i] = act_round(m, h[i]);
    orc_op_matvec(m->readout_w[r], m->readout_b[r], c->d_model, c->d_model, m->tmp, y);
    unembed(m, y, logits);
}

static int check_step(const orc_model* m, int32_t tok) {
    if (tok < 0 || tok >= m->c.vocab) return -1;
    if (m->pos >= m->c.max_ctx) return -2;
    return 0;
}

int orc_set_gemm(orc_model* m, orc_dgemm_fn gemm) {
    if (!m) return -1;
    m->gemm = gemm;
    return 0;
}

/* Prompts at least this long take the matrix-product form of the prefill
 * when a BLAS product is set. */
#define ORC_GEMM_MIN_PROMPT 64
/* Positions per block of the matrix-product prefill. */
#define ORC_GEMM_BLOCK 512

/* out[p][i] = (float)(sum_j W[i][j] X[p][j] + b_i) for the n rows of X: the
 * orc_op_matvec of every row of X, its double sums taken by one BLAS product
 * (Wd: W as doubles; xb, ob: n * cols and n * rows doubles of scratch). */
static void project_rows(orc_dgemm_fn gemm, const double* Wd, const uint16_t* b, int rows, int cols,
                         const float* X, int n, float* out, double* xb, double* ob) {
    for (int64_t i = 0; i < (int64_t)n * cols; ++i) xb[i] = (double)X[i];
    /* column-major view: W is cols x rows, X is cols x n, OUT is rows x n */
    const char tA = 'T', tB = 'N';
    const double one = 1.0, zero = 0.0;
    gemm(&tA, &tB, &rows, &n, &cols, &one, Wd, &cols, xb, &cols, &zero, ob, &rows);
#pragma omp parallel for schedule(static)
    for (int p = 0; p < n; ++p)
        for (int i = 0; i < rows; ++i) {
            double acc = ob[(int64_t)p * rows + i];
            if (b) acc += (double)bf16_bits_to_f32(b[i]);
            out[(int64_t)p * rows + i] = (float)acc;
        }
}

/* orc_op_attention for the block of positions tb..tb+nb-1 (rotated queries
 * in Qb, [nb][A*D]) over the cache of layer j: for each query head, the
 * scores q.k of every position of the block against keys 0..tb+nb-1 are one
 * BLAS product, each position then takes the softmax of its scores at
 * positions <= t (the rest weigh 0), and the weighted sums of the values are
 * a second product.  Scratch: kd, vd (T * D), qb (nb * D), sd (nb * T),
 * od (nb * D) doubles, T = tb + nb. */
static void attend_rows(orc_model* m, int j, int tb, int nb, const float* Qb, float* Ob, double* kd, double* vd,
                        double* qb, double* sd, double* od) {
    const orc_config* c = &m->c;
    const int A = c->n_heads, KH = c->n_kv_heads, D = c->head_dim, group = A / KH, qdim = A * D;
    const int T = tb + nb;
    const double scale = 1.0 / sqrt((double)D), one = 1.0, zero = 0.0;
    const char tT = 'T', tN = 'N';
    for (int g = 0; g < KH; ++g) {
        const float* Kg = m->kc + kv_index(m, j, g, 0);
        const float* Vg = m->vc + kv_index(m, j, g, 0);
#pragma omp parallel for schedule(static)
        for (int64_t i = 0; i < (int64_t)T * D; ++i) {
            kd[i] = (double)Kg[i];
            vd[i] = (double)Vg[i];
        }
        for (int hh = g * group; hh < (g + 1) * group; ++hh) {
            for (int p = 0; p < nb; ++p)
                for (int e = 0; e < D; ++e) qb[(int64_t)p * D + e] = (double)Qb[(int64_t)p * qdim + (int64_t)hh * D + e];
            /* column-major: S (T x nb) = K^T-view (T x D) * Q-view (D x nb) */
            m->gemm(&tT, &tN, &T, &nb, &D, &one, kd, &D, qb, &D, &zero, sd, &T);
#pragma omp parallel for schedule(static)
            for (int p = 0; p < nb; ++p) {
                double* sr = sd + (int64_t)p * T;
                const int tp = tb + p;
                double mx = -INFINITY;
                for (int t = 0; t <= tp; ++t) {
                    sr[t] *= scale;
                    if (sr[t] > mx) mx = sr[t];
                }
                double sum = 0.0;
                for (int t = 0; t <= tp; ++t) {
                    sr[t] = exp(sr[t] - mx);
                    sum += sr[t];
                }
                for (int t = 0; t <= tp; ++t) sr[t] = sr[t] / sum;
                for (int t = tp + 1; t < T; ++t) sr[t] = 0.0;
            }
            /* column-major: O (D x nb) = V-view (D x T) * P-view (T x nb) */
            m->gemm(&tN, &tN, &D, &nb, &T, &one, vd, &D, sd, &T, &zero, od, &D);
            for (int p = 0; p < nb; ++p)
                for (int e = 0; e < D; ++e) Ob[(int64_t)p * qdim + (int64_t)hh * D + e] = (float)od[(int64_t)p * D + e];
        }
    }
}

static void to_double(const uint16_t* W, int64_t n, double* out) {
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) out[i] = (double)bf16_bits_to_f32(W[i]);
}

/* The prompt layer by layer, in blocks of positions: each step of the
 * layer (the same steps as layer_forward, in the same order, rounded to
 * float at the same points) runs for every position of the block, and each
 * matrix-vector product of those positions becomes one matrix product.  At
 * layer j a block's cache entries are stored before its attention, which
 * reads positions <= t of layer j only: the entries of earlier blocks and of
 * the block itself.  The products' double sums run in the library's order,
 * so results may differ from the position-by-position prefill in the last
 * bit of a float.  Returns 0, or -3 if memory runs out. */
static int prefill_gemm(orc_model* m, const int32_t* ids, int n) {
    const orc_config* c = &m->c;
    const int d = c->d_model, L = c->n_layers, A = c->n_heads, KH = c->n_kv_heads, D = c->head_dim;
    const int F = c->ffn_dim, t0 = m->pos;
    const int qd = A * D, kd = KH * D, B = n < ORC_GEMM_BLOCK ? n : ORC_GEMM_BLOCK;
    const int wide = F > qd ? (F > d ? F : d) : (qd > d ? qd : d);
    const int64_t wq = (int64_t)qd * d, wk = (int64_t)kd * d, wo = (int64_t)d * qd, wf = (int64_t)F * d;
    double* Wd = (double*)malloc(sizeof(double) * (size_t)(wq + 2 * wk + wo + 3 * wf));
    double* xb = (double*)malloc(sizeof(double) * (size_t)B * wide);
    double* ob = (double*)malloc(sizeof(double) * (size_t)B * wide);
    float* H = (float*)malloc(sizeof(float) * (size_t)n * d);
    float* U = (float*)malloc(sizeof(float) * (size_t)B * d);
    float* Q = (float*)malloc(sizeof(float) * (size_t)B * qd);
    float* Kb = (float*)malloc(sizeof(float) * (size_t)B * kd);
    float* Vb = (float*)malloc(sizeof(float) * (size_t)B * kd);
    float* O = (float*)malloc(sizeof(float) * (size_t)B * qd);
    float* G = (float*)malloc(sizeof(float) * (size_t)B * F);
    float* UP = (float*)malloc(sizeof(float) * (size_t)B * F);
    float* T = (float*)malloc(sizeof(float) * (size_t)B * d);
    const size_t Tmax = (size_t)t0 + n;
    double* kdb = (double*)malloc(sizeof(double) * Tmax * D);
    double* vdb = (double*)malloc(sizeof(double) * Tmax * D);
    double* qb = (double*)malloc(sizeof(double) * (size_t)B * D);
    double* sb = (double*)malloc(sizeof(double) * (size_t)B * Tmax);
    double* odb = (double*)malloc(sizeof(double) * (size_t)B * D);
    int rc = 0;
    if (!Wd || !xb || !ob || !H || !U || !Q || !Kb || !Vb || !O || !G || !UP || !T || !kdb || !vdb || !qb || !sb ||
        !odb) {
        rc = -3;
        goto done;
    }
    for (int i = 0; i < n; ++i) {
        const uint16_t* e = m->w.embed + (size_t)ids[i] * d;
        for (int x = 0; x < d; ++x) H[(size_t)i * d + x] = bf16_bits_to_f32(e[x]);
    }
    for (int j = 0; j < L; ++j) {
        double *Wq = Wd, *Wk = Wq + wq, *Wv = Wk + wk, *Wo = Wv + wk, *Wg = Wo + wo, *Wu = Wg + wf, *Wdn = Wu + wf;
        to_double(m->w.wq[j], wq, Wq);
        to_double(m->w.wk[j], wk, Wk);
        to_double(m->w.wv[j], wk, Wv);
        to_double(m->w.wo[j], wo, Wo);
        to_double(m->w.wg[j], wf, Wg);
        to_double(m->w.wu[j], wf, Wu);
        to_double(m->w.wd[j], wf, Wdn);
        for (int p0 = 0; p0 < n; p0 += B) {
            const int nb = n - p0 < B ? n - p0 : B;
            float* Hb = H + (size_t)p0 * d;
            /* attention input, q, k, v; RoPE; the block's cache entries */
#pragma omp parallel for schedule(static)
            for (int p = 0; p < nb; ++p) {
                orc_op_rmsnorm(Hb + (size_t)p * d, m->w.attn_norm[j], d, c->rms_eps, U + (size_t)p * d);
                for (int i = 0; i < d; ++i) U[(size_t)p * d + i] = act_round(m, U[(size_t)p * d + i]);
            }
            project_rows(m->gemm, Wq, c->qkv_bias ? m->w.bq[j] : NULL, qd, d, U, nb, Q, xb, ob);
            project_rows(m->gemm, Wk, c->qkv_bias ? m->w.bk[j] : NULL, kd, d, U, nb, Kb, xb, ob);
            project_rows(m->gemm, Wv, c->qkv_bias ? m->w.bv[j] : NULL, kd, d, U, nb, Vb, xb, ob);
#pragma omp parallel for schedule(static)
            for (int p = 0; p < nb; ++p) {
                const int t = t0 + p0 + p;
                for (int hh = 0; hh < A; ++hh) orc_op_rope(Q + (size_t)p * qd + (size_t)hh * D, D, t, c->rope_base);
                for (int g = 0; g < KH; ++g) orc_op_rope(Kb + (size_t)p * kd + (size_t)g * D, D, t, c->rope_base);
                store_kv(m, j, t, Kb + (size_t)p * kd, Vb + (size_t)p * kd, 1);
            }
            /* attention of every position and head over positions 0..t */
            attend_rows(m, j, t0 + p0, nb, Q, O, kdb, vdb, qb, sb, odb);
            for (int64_t i = 0; i < (int64_t)nb * qd; ++i) O[i] = act_round(m, O[i]);
            /* output projection and residual add */
            project_rows(m->gemm, Wo, NULL, d, qd, O, nb, T, xb, ob);
            for (int64_t i = 0; i < (int64_t)nb * d; ++i) Hb[i] = Hb[i] + T[i];
            /* gated feed-forward and residual add */
#pragma omp parallel for schedule(static)
            for (int p = 0; p < nb; ++p) {
                orc_op_rmsnorm(Hb + (size_t)p * d, m->w.mlp_norm[j], d, c->rms_eps, U + (size_t)p * d);
                for (int i = 0; i < d; ++i) U[(size_t)p * d + i] = act_round(m, U[(size_t)p * d + i]);
            }
            project_rows(m->gemm, Wg, NULL, F, d, U, nb, G, xb, ob);
            project_rows(m->gemm, Wu, NULL, F, d, U, nb, UP, xb, ob);
#pragma omp parallel for schedule(static)
            for (int64_t i = 0; i < (int64_t)nb * F; ++i)
                G[i] = act_round(m, (float)(orc_op_silu(G[i]) * (double)UP[i]));
            project_rows(m->gemm, Wdn, NULL, d, F, G, nb, T, xb, ob);
            for (int64_t i = 0; i < (int64_t)nb * d; ++i) Hb[i] = Hb[i] + T[i];
        }
    }
    memcpy(m->h, H + (size_t)(n - 1) * d, sizeof(float) * d);
    m->pos += n;
done:
    free(Wd); free(xb); free(ob); free(H); free(U); free(Q); free(Kb); free(Vb); free(O); free(G); free(UP);
    free(T); free(kdb); free(vdb); free(qb); free(sb); free(odb);
    return rc;
}

/* Prefill: every prompt position runs the full depth, no gate; returns the
 * full model's greedy token after the last position.  With a BLAS product
 * set (orc_set_gemm), prompts of ORC_GEMM_MIN_PROMPT positions or more take
 * the matrix-product form (prefill_gemm). */
int orc_prefill(orc_model* m, const int32_t* ids, int n, int32_t* first_token, orc_capture* cap) {
    if (!m || n <= 0 || m->pos + n > m->c.max_ctx) return -2;
    for (int i = 0; i < n; ++i)
        if (ids[i] < 0 || ids[i] >= m->c.vocab) return -1;
    const int d = m->c.d_model, L = m->c.n_layers;
    if (m->gemm && n >= ORC_GEMM_MIN_PROMPT) {
        const int rc = prefill_gemm(m, ids, n);
        if (rc) return rc;
    } else {
        for (int i = 0; i < n; ++i) {
            const int t = m->pos;
            const uint16_t* e = m->w.embed + (size_t)ids[i] * d;
            for (int x = 0; x < d; ++x) m->h[x] = bf16_bits_to_f32(e[x]);
            for (int j = 0; j < L; ++j) layer_forward(m, j, t, m->h, NULL);
            m->pos++;
        }
    }
    unembed(m, m->h, m->logits);
    orc_conf cf;
    orc_op_confidence(m->logits, m->c.vocab, &cf);
    if (first_token) *first_token = cf.argmax;
    if (cap && cap->h_final) memcpy(cap->h_final, m->h, sizeof(float) * d);
    if (cap && cap->final_logits) memcpy(cap->final_logits, m->logits, sizeof(float) * m->c.vocab);
    return 0;
}

/* One gated decode step (Section 4, step five) at the current position.
 * force: ORC_FORCE_FREE lets the gate decide; ORC_FORCE_FULL never exits;
 * ORC_FORCE_EXIT_AT(r) exits at readout r.  The gate's own verdict at every
 * evaluated readout is reported in gate_pass either way. */
int orc_decode_step(orc_model* m, int32_t in_tok, const float* taus, int force, orc_step_result* res,
                    orc_capture* cap) {
    if (!m || !res) return -1;
    const int rc = check_step(m, in_tok);
    if (rc) return rc;
    if (force >= 2 && force - 2 >= m->n_readouts) return -1;
    const orc_config* c = &m->c;
    const int d = c->d_model, L = c->n_layers, V = c->vocab;
    const int t = m->pos;
    memset(res, 0, sizeof(*res));
    res->nucleus_member = -1;
    res->exit_readout = -1;
    res->full_token = -1;
    res->exit_layer = L;
    int64_t toff[12];
    const int64_t tstride = orc_trace_layout(c, toff);

    const uint16_t* e = m->w.embed + (size_t)in_tok * d;
    for (int x = 0; x < d; ++x) m->h[x] = bf16_bits_to_f32(e[x]);
    int r = 0, exited = 0;
    for (int j = 0; j < L && !exited; ++j) {
        flush_layer(m, j, t);
        layer_forward(m, j, t, m->h, cap && cap->layer_trace ? cap->layer_trace + (size_t)j * tstride : NULL);
        if (r < m->n_readouts && m->readout_layer[r] == j + 1) {
            readout(m, r, m->h, m->y, m->logits);
            orc_conf cf;
            orc_op_confidence(m->logits, V, &cf);
            res->confidence[r] = conf_signal(m, &cf);
            res->gap[r] = cf.gap;
            res->readout_token[r] = cf.argmax;
            res->gate_pass[r] = res->confidence[r] > taus[r];
            res->n_evaluated = r + 1;
            if (cap && cap->h_readout) memcpy(cap->h_readout + (size_t)r * d, m->h, sizeof(float) * d);
            if (cap && cap->y_readout) memcpy(cap->y_readout + (size_t)r * d, m->y, sizeof(float) * d);
            if (cap && cap->readout_logits)
                memcpy(cap->readout_logits + (size_t)r * V, m->logits, sizeof(float) * V);
            const int take = force == ORC_FORCE_FREE ? res->gate_pass[r] : force == ORC_FORCE_EXIT_AT(r);
            if (take) {
                exited = 1;
                res->exited = 1;
                res->exit_readout = r;
                res->exit_layer = j + 1;
                res->token = cf.argmax;
                if (!m->lazy_fill)
                    for (int jj = j + 1; jj < L; ++jj) kv_fill(m, jj, t, m->h);
                memcpy(m->h_exit + (size_t)t * d, m->h, sizeof(float) * d);
                m->exit_at[t] = (int16_t)(j + 1);
            }
            ++r;
        }
    }
    if (!exited) {
        unembed(m, m->h, m->logits);
        orc_conf cf;
        orc_op_confidence(m->logits, V, &cf);
        res->token = cf.argmax;
        res->full_token = cf.argmax;
        res->full_confidence = conf_signal(m, &cf);
        res->full_gap = cf.gap;
        if (m->n_readouts > 0 && res->n_evaluated > 0) {
            double mass = 0.0;
            res->nucleus_member = orc_op_nucleus_member(m->logits, V, res->readout_token[0], m->nucleus_p, &mass);
            res->nucleus_mass = (float)mass;
        }
        if (cap && cap->h_final) memcpy(cap->h_final, m->h, sizeof(float) * d);
        if (cap && cap->final_logits) memcpy(cap->final_logits, m->logits, sizeof(float) * V);
        m->full_steps++;
    } else {
        m->exits[res->exit_readout]++;
    }
    m->steps++;
    m->pos++;
    return 0;
}

int orc_position(const orc_model* m) { return m->pos; }

/* Forget the positions from pos on, so that decoding continues from there
 * as if they had never been decoded: their cache entries, exit records and
 * residuals are cleared, the position moves back to pos and the step counts
 * restart.  Positions below pos are untouched.  -1 unless 0 <= pos <= the
 * current position. */
int orc_truncate(orc_model* m, int pos) {
    if (!m || pos < 0 || pos > m->pos) return -1;
    const orc_config* c = &m->c;
    const int n = c->max_ctx - pos;
    for (int j = 0; j < c->n_layers; ++j) {
        memset(m->kv_src + (size_t)j * c->max_ctx + pos, 0, (size_t)n);
        for (int g = 0; g < c->n_kv_heads; ++g) {
            memset(m->kc + kv_index(m, j, g, pos), 0, sizeof(float) * (size_t)n * c->head_dim);
            memset(m->vc + kv_index(m, j, g, pos), 0, sizeof(float) * (size_t)n * c->head_dim);
        }
    }
    memset(m->exit_at + pos, 0, sizeof(int16_t) * (size_t)n);
    memset(m->h_exit + (size_t)pos * c->d_model, 0, sizeof(float) * (size_t)n * c->d_model);
    m->pos = pos;
    m->steps = m->full_steps = 0;
    memset(m->exits, 0, sizeof(m->exits));
    return 0;
}

/* Section 11's full-depth re-pass: for each position t in [t0, t1), in
 * order, whose upper layers still hold filled (or deferred) entries (it
 * exited after layer k and kv_src[k][t] is not 1), run layers k+1..L from the
 * residual it exited with, storing computed entries in place of the filled
 * ones.  Attention at t sees the cache as it stands (deferred fills of
 * earlier positions done first), including positions re-passed just before.
 * The decode position is unchanged.  Returns the number of positions
 * re-passed (-1 on a bad range). */
int orc_repass(orc_model* m, int t0, int t1) {
    if (!m || t0 < 0 || t1 < t0 || t1 > m->pos) return -1;
    const orc_config* c = &m->c;
    const int d = c->d_model, L = c->n_layers;
    int n = 0;
    for (int t = t0; t < t1; ++t) {
        const int k = m->exit_at[t];
        if (k <= 0 || k >= L || m->kv_src[(size_t)k * c->max_ctx + t] == 1) continue;
        memcpy(m->y, m->h_exit + (size_t)t * d, sizeof(float) * d);
        for (int j = k; j < L; ++j) {
            flush_layer(m, j, t);
            layer_forward(m, j, t, m->y, NULL);
        }
        ++n;
    }
    return n;
}

/* Copy the cached K and V (all key-value heads, [K*D] each) of layer j
 * (0-based) at position t, and the entry's origin (0/1/2). */
int orc_kv(const orc_model* m, int j, int t, float* k, float* v, int8_t* src) {
    const orc_config* c = &m->c;
    if (j < 0 || j >= c->n_layers || t < 0 || t >= c->max_ctx) return -1;
    for (int g = 0; g < c->n_kv_heads; ++g) {
        if (k) memcpy(k + (size_t)g * c->head_dim, m->kc + kv_index(m, j, g, t), sizeof(float) * c->head_dim);
        if (v) memcpy(v + (size_t)g * c->head_dim, m->vc + kv_index(m, j, g, t), sizeof(float) * c->head_dim);
    }
    if (src) *src = m->kv_src[(size_t)j * c->max_ctx + t];
    return 0;
}

/* steps, full_steps, exits[ORC_MAX_READOUTS] */
void orc_stats(const orc_model* m, int64_t* out) {
    out[0] = m->steps;
    out[1] = m->full_steps;
    for (int r = 0; r < ORC_MAX_READOUTS; ++r) out[2 + r] = m->exits[r];
}
