/*
 * pbd_oracle.c -- CPU reference ("oracle") for PEFT-BD speculative decoding.
 *
 * TEST INFRASTRUCTURE.  This file exists only to check the GPU library.  The test
 * suite, the smoke check and the benchmark's CPU-baseline leg are the only code
 * that may build, load or call it; the product path never does, and it shares no
 * code, header or table with the CUDA sources.
 *
 * What it computes (paper: "Accepted Prefixes Are Not All You Need", arXiv 2607.12422):
 *   - one forward pass of a Qwen3-shaped decoder (Section 4.1 names Qwen3-0.6B in bf16)
 *     over a block of rows appended to a KV cache, with the LoRA-like adapter switched
 *     on or off at run time (Section 3, steps 1 and 3; Appendix A.2: rank 16, alpha 32,
 *     all seven block linears; Appendix A.4: adapter on for drafting, off for verifying),
 *   - under either the causal mask (verification, prefill, plain decoding) or the
 *     block-diffusion draft mask (Section 3, steps 1-2; Appendix A.4 notes that the
 *     verify pass uses a different attention mask from the draft pass).
 * The speculative loop itself (accept the longest matching prefix, append, repeat:
 * Section 3, steps 4-5) lives in the Python harness next to this file.
 *
 * Precision: "bf16 precision" (Section 4.1) read as bf16 storage and fp32 arithmetic:
 *   - weights are bf16, used exactly as fp32;
 *   - every activation handed from one step to the next is rounded to bf16 (RNE):
 *     residual stream, norm outputs, q/k after norm+RoPE, v, attention output,
 *     SiLU*up output, LoRA intermediate u = bf16(x A^T);
 *   - dot products accumulate in fp32; a linear's output is bf16(acc_W + s*acc_B(u));
 *   - softmax and logits stay fp32; argmax takes the lowest index on ties.
 * Every dot product uses one fixed summation order (term k goes to partial sum k mod 16,
 * partials combined by a fixed pairwise tree), so a row's result never depends on how
 * many other rows share the pass.  Compile with -ffp-contract=off so every product and
 * sum is a single IEEE fp32 operation on any host.
 *
 * Readings where the paper is silent (all listed in the design notes):
 *   - Qwen3 block: pre-norm RMSNorm, no biases, per-head RMSNorm of q and k before
 *     rotate-half RoPE (theta 1e6), GQA, SwiGLU MLP, final RMSNorm, tied lm_head.
 *   - Draft block = [pending token, D mask rows] at positions L..L+D.  The pending
 *     token's row sees the cache and itself; mask rows see the cache, the pending row
 *     and every mask row (bidirectional inside the mask block).  Row j predicts the
 *     token at position L+j+1.
 *   - The mask rows use one adapter-owned embedding vector (the paper trains
 *     "diffusion special-token embeddings", Appendix A.2).
 *   - Block K/V are written to cache slots L..L+n-1; the caller owns the valid length,
 *     so a pass that is not accepted is rolled back by not advancing it.
 *
 * Parity pins (tests/test_oracle_*.py): spec output == greedy output for any drafts;
 * B=0 with D=1 reduces to greedy with n=1 every round; the anchor row of a draft equals
 * the verify row bitwise when B=0; LoRA equals the merged weight in fp64; attention
 * equals dense softmax with an explicit mask; RoPE relative-position invariance; KV
 * after commits equals a fresh prefill.  The logit values themselves have no printed
 * reference (the paper prints none): parity unpinned beyond those properties.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

typedef struct {
    int32_t n_layers, hidden, n_q_heads, n_kv_heads, head_dim, intermediate, vocab;
    float rms_eps, rope_theta;
    int32_t lora_rank;
    float lora_scale;
} orc_config;

enum { LIN_Q = 0, LIN_K, LIN_V, LIN_O, LIN_GATE, LIN_UP, LIN_DOWN, N_LIN };

typedef struct {
    const uint16_t *embed;      /* [V, H] bf16 bits, tied with the lm_head */
    const uint16_t *final_norm; /* [H] */
    const uint16_t *attn_norm;  /* [nl, H] */
    const uint16_t *mlp_norm;   /* [nl, H] */
    const uint16_t *q_norm;     /* [nl, d] */
    const uint16_t *k_norm;     /* [nl, d] */
    const uint16_t *w[N_LIN];   /* [nl, out, in] */
    const uint16_t *lora_a[N_LIN]; /* [nl, r, in] */
    const uint16_t *lora_b[N_LIN]; /* [nl, out, r] */
    const uint16_t *mask_embed; /* [H] */
} orc_weights;

typedef struct {
    int32_t capacity;  /* token slots */
    float *k, *v;      /* [nl][capacity][n_kv_heads*head_dim], bf16 values held in fp32 */
} orc_cache;

enum { MASK_CAUSAL = 0, MASK_BLOCK_DRAFT = 1 };

/* ------------------------------------------------------------------ numerics */

static inline float bf16_to_f32(uint16_t b) {
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, 4);
    return f;
}

/* IEEE-754 round-to-nearest-even from binary32 to bfloat16, returned widened to fp32. */
static inline float round_bf16(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    if ((u & 0x7f800000u) == 0x7f800000u) {
        if (u & 0x007fffffu) u |= 0x00400000u; /* keep NaN quiet and non-zero */
        u &= 0xffff0000u;
    } else {
        u += 0x7fffu + ((u >> 16) & 1u);
        u &= 0xffff0000u;
    }
    memcpy(&f, &u, 4);
    return f;
}

/* Accumulator of every dot product: fp32 (the reference build).  Built with -DORC_ACC_DOUBLE
 * the same sums run in fp64; the tests use that second build only to measure how far two
 * valid summation orders of the bf16 model drift apart (the floor of any logit tolerance). */
#ifdef ORC_ACC_DOUBLE
typedef double acc_t;
#else
typedef float acc_t;
#endif

/* Fixed-order sums: term k accumulates into partial k % 16, then a pairwise tree. */
static inline float combine16(acc_t s[16]) {
    for (int w = 8; w >= 1; w >>= 1)
        for (int j = 0; j < w; j++) s[j] = s[j] + s[j + w];
    return (float)s[0];
}

static float dot_fw(const float *x, const uint16_t *w, int n) {
    acc_t s[16] = {0};
    int k = 0;
    for (; k + 16 <= n; k += 16)
        for (int j = 0; j < 16; j++) s[j] = s[j] + x[k + j] * bf16_to_f32(w[k + j]);
    for (int j = 0; k + j < n; j++) s[j] = s[j] + x[k + j] * bf16_to_f32(w[k + j]);
    return combine16(s);
}

static float dot_ff(const float *x, const float *y, int n) {
    acc_t s[16] = {0};
    int k = 0;
    for (; k + 16 <= n; k += 16)
        for (int j = 0; j < 16; j++) s[j] = s[j] + x[k + j] * y[k + j];
    for (int j = 0; k + j < n; j++) s[j] = s[j] + x[k + j] * y[k + j];
    return combine16(s);
}

/* ------------------------------------------------------------------ model steps */

/* RMSNorm (Qwen3): y = bf16( g * bf16( x * 1/sqrt(mean(x^2) + eps) ) ). */
static void rmsnorm_rows(int n, int dim, const float *x, const uint16_t *g, float eps, float *y) {
    for (int i = 0; i < n; i++) {
        const float *xi = x + (size_t)i * dim;
        float ss = dot_ff(xi, xi, dim);
        float r = 1.0f / sqrtf(ss / (float)dim + eps);
        for (int j = 0; j < dim; j++) y[(size_t)i * dim + j] = round_bf16(bf16_to_f32(g[j]) * round_bf16(xi[j] * r));
    }
}

/* Linear with optional LoRA delta (Appendix A.2):
 *   u = bf16(x A^T)                 [n, r]
 *   y = bf16(x W^T + s * (u B^T))   [n, out]  -- one rounding of the fp32 sum.
 * W is [out, in], A is [r, in], B is [out, r]. */
static void linear_rows(const orc_config *c, int n, int in, int out, const float *x, const uint16_t *W,
                        const uint16_t *A, const uint16_t *B, int adapter_on, float *y) {
    const int r = c->lora_rank;
    float *u = NULL;
    if (adapter_on) {
        u = (float *)malloc(sizeof(float) * (size_t)n * r);
        for (int i = 0; i < n; i++)
            for (int j = 0; j < r; j++) u[(size_t)i * r + j] = round_bf16(dot_fw(x + (size_t)i * in, A + (size_t)j * in, in));
    }
#pragma omp parallel for schedule(static)
    for (int o = 0; o < out; o++) {
        for (int i = 0; i < n; i++) {
            float acc = dot_fw(x + (size_t)i * in, W + (size_t)o * in, in);
            if (adapter_on) {
                float lb = dot_fw(u + (size_t)i * r, B + (size_t)o * r, r);
                acc = acc + c->lora_scale * lb;
            }
            y[(size_t)i * out + o] = round_bf16(acc);
        }
    }
    free(u);
}

/* Rotate-half RoPE on one head vector at integer position pos (Qwen3 convention):
 *   inv_freq_i = theta^(-2i/d), angle = pos * inv_freq_i (double), cos/sin rounded to fp32,
 *   out[i]       = bf16(x[i] cos - x[i+d/2] sin)
 *   out[i + d/2] = bf16(x[i+d/2] cos + x[i] sin),   i < d/2. */
static void rope_head(float *x, int d, int pos, double theta) {
    int half = d / 2;
    for (int i = 0; i < half; i++) {
        double inv_freq = pow(theta, -2.0 * (double)i / (double)d);
        double ang = (double)pos * inv_freq;
        float cs = (float)cos(ang), sn = (float)sin(ang);
        float a = x[i], b = x[i + half];
        float ya = a * cs - b * sn;
        float yb = b * cs + a * sn;
        x[i] = round_bf16(ya);
        x[i + half] = round_bf16(yb);
    }
}

/* SwiGLU gate: act = bf16( silu(g) * u ), silu(g) = g / (1 + exp(-g)). */
static void swiglu(size_t count, const float *g, const float *u, float *act) {
    for (size_t e = 0; e < count; e++) {
        float sg = g[e] / (1.0f + expf(-g[e]));
        act[e] = round_bf16(sg * u[e]);
    }
}

/* Key visibility for query row i (absolute position L+i) and key position kp.
 * Causal: kp <= L+i.  Block draft: row 0 (the pending token) is causal; a mask row
 * (i >= 1) additionally sees every key of the block above the pending token. */
static inline int key_visible(int mask_mode, int L, int i, int kp) {
    int qp = L + i;
    if (kp <= qp) return 1;
    if (mask_mode == MASK_BLOCK_DRAFT && i >= 1 && kp > L) return 1;
    return 0;
}

/* Attention for n block rows against cache slots [0, L+n): softmax(q k^T / sqrt(d)) v, GQA.
 * Sums run over key positions in increasing order. */
static void attention_rows(const orc_config *c, int layer, const orc_cache *cache, int L, int n, int mask_mode,
                           const float *q, float *out) {
    const int d = c->head_dim, Hq = c->n_q_heads, Hkv = c->n_kv_heads, group = Hq / Hkv;
    const int kvw = Hkv * d, T = L + n;
    const float scale = (float)(1.0 / sqrt((double)d));
    const float *K = cache->k + (size_t)layer * cache->capacity * kvw;
    const float *V = cache->v + (size_t)layer * cache->capacity * kvw;
#pragma omp parallel for schedule(static) collapse(2)
    for (int i = 0; i < n; i++) {
        for (int h = 0; h < Hq; h++) {
            const int g = h / group;
            const float *qv = q + (size_t)i * Hq * d + (size_t)h * d;
            float *s = (float *)malloc(sizeof(float) * (size_t)T);
            float *acc = (float *)calloc((size_t)d, sizeof(float));
            float m = -INFINITY;
            for (int kp = 0; kp < T; kp++) {
                if (!key_visible(mask_mode, L, i, kp)) continue;
                s[kp] = dot_ff(qv, K + (size_t)kp * kvw + (size_t)g * d, d) * scale;
                if (s[kp] > m) m = s[kp];
            }
            float l = 0.0f;
            for (int kp = 0; kp < T; kp++) {
                if (!key_visible(mask_mode, L, i, kp)) continue;
                float p = expf(s[kp] - m);
                l = l + p;
                const float *vv = V + (size_t)kp * kvw + (size_t)g * d;
                for (int j = 0; j < d; j++) acc[j] = acc[j] + p * vv[j];
            }
            for (int j = 0; j < d; j++) out[(size_t)i * Hq * d + (size_t)h * d + j] = round_bf16(acc[j] / l);
            free(s);
            free(acc);
        }
    }
}

/* ------------------------------------------------------------------ public entry points */

orc_cache *orc_cache_new(const orc_config *c, int32_t capacity) {
    orc_cache *cc = (orc_cache *)calloc(1, sizeof(orc_cache));
    size_t n = (size_t)c->n_layers * capacity * c->n_kv_heads * c->head_dim;
    cc->capacity = capacity;
    cc->k = (float *)calloc(n, sizeof(float));
    cc->v = (float *)calloc(n, sizeof(float));
    if (!cc->k || !cc->v) {
        free(cc->k);
        free(cc->v);
        free(cc);
        return NULL;
    }
    return cc;
}

void orc_cache_free(orc_cache *cc) {
    if (!cc) return;
    free(cc->k);
    free(cc->v);
    free(cc);
}

/* Copy the first n slots of one cache into another (the harness's snapshot tool). */
int orc_cache_copy(const orc_config *c, const orc_cache *src, orc_cache *dst, int32_t n) {
    if (n > src->capacity || n > dst->capacity) return 1;
    size_t kvw = (size_t)c->n_kv_heads * c->head_dim;
    for (int l = 0; l < c->n_layers; l++) {
        memcpy(dst->k + (size_t)l * dst->capacity * kvw, src->k + (size_t)l * src->capacity * kvw, sizeof(float) * n * kvw);
        memcpy(dst->v + (size_t)l * dst->capacity * kvw, src->v + (size_t)l * src->capacity * kvw, sizeof(float) * n * kvw);
    }
    return 0;
}

/* Read one layer's K or V slots [0, n) as fp32 (which: 0 = K, 1 = V). */
int orc_cache_read(const orc_config *c, const orc_cache *cc, int32_t layer, int32_t which, int32_t n, float *out) {
    if (n > cc->capacity || layer < 0 || layer >= c->n_layers) return 1;
    size_t kvw = (size_t)c->n_kv_heads * c->head_dim;
    const float *src = (which ? cc->v : cc->k) + (size_t)layer * cc->capacity * kvw;
    memcpy(out, src, sizeof(float) * n * kvw);
    return 0;
}

/* One forward pass over n rows at positions L..L+n-1.
 *   tokens[i] >= 0: embedding row; tokens[i] < 0: the adapter's mask embedding.
 *   adapter_on: LoRA delta on all seven linears of every layer.
 *   mask_mode: MASK_CAUSAL or MASK_BLOCK_DRAFT.
 *   Block K/V are written to slots L..L+n-1 of every layer.
 *   Rows read_first..read_first+n_read-1 get fp32 logits (if logits != NULL) and argmax.
 *   hidden_out (optional): final-norm output of the read rows, [n_read, H].
 * Returns 0, or 1 when the cache is too small. */
int orc_forward(const orc_config *c, const orc_weights *w, orc_cache *cache, int32_t L, int32_t n,
                const int32_t *tokens, int32_t adapter_on, int32_t mask_mode, int32_t read_first, int32_t n_read,
                float *logits, int32_t *argmax, float *hidden_out, uint64_t skip_layers) {
    if (L < 0 || n <= 0 || L + n > cache->capacity) return 1;
    if (read_first < 0 || read_first + n_read > n) return 1;
    for (int i = 0; i < n; i++)
        if (tokens[i] >= c->vocab) return 1;
    const int H = c->hidden, d = c->head_dim, Hq = c->n_q_heads, Hkv = c->n_kv_heads, I = c->intermediate;
    const int qw = Hq * d, kvw = Hkv * d, r = c->lora_rank;
    float *h = (float *)malloc(sizeof(float) * (size_t)n * H);
    float *x = (float *)malloc(sizeof(float) * (size_t)n * H);
    float *q = (float *)malloc(sizeof(float) * (size_t)n * qw);
    float *k = (float *)malloc(sizeof(float) * (size_t)n * kvw);
    float *v = (float *)malloc(sizeof(float) * (size_t)n * kvw);
    float *att = (float *)malloc(sizeof(float) * (size_t)n * qw);
    float *y = (float *)malloc(sizeof(float) * (size_t)n * H);
    float *gt = (float *)malloc(sizeof(float) * (size_t)n * I);
    float *up = (float *)malloc(sizeof(float) * (size_t)n * I);
    float *act = (float *)malloc(sizeof(float) * (size_t)n * I);

    for (int i = 0; i < n; i++) {
        const uint16_t *src = tokens[i] >= 0 ? w->embed + (size_t)tokens[i] * H : w->mask_embed;
        for (int j = 0; j < H; j++) h[(size_t)i * H + j] = bf16_to_f32(src[j]);
    }

    for (int l = 0; l < c->n_layers; l++) {
        /* layer skipping (Section 6 names it beside the early exit as a cheaper draft path):
         * a layer whose bit is set in skip_layers leaves the residual stream untouched and
         * writes no K/V */
        if (l < 64 && ((skip_layers >> l) & 1u)) continue;
        const uint16_t *Wl[N_LIN], *Al[N_LIN], *Bl[N_LIN];
        for (int t = 0; t < N_LIN; t++) {
            int fin, fout;
            switch (t) {
                case LIN_Q: fin = H; fout = qw; break;
                case LIN_K: case LIN_V: fin = H; fout = kvw; break;
                case LIN_O: fin = qw; fout = H; break;
                case LIN_GATE: case LIN_UP: fin = H; fout = I; break;
                default: fin = I; fout = H; break;
            }
            Wl[t] = w->w[t] + (size_t)l * fout * fin;
            Al[t] = adapter_on ? w->lora_a[t] + (size_t)l * r * fin : NULL;
            Bl[t] = adapter_on ? w->lora_b[t] + (size_t)l * fout * r : NULL;
        }
        /* attention block */
        rmsnorm_rows(n, H, h, w->attn_norm + (size_t)l * H, c->rms_eps, x);
        linear_rows(c, n, H, qw, x, Wl[LIN_Q], Al[LIN_Q], Bl[LIN_Q], adapter_on, q);
        linear_rows(c, n, H, kvw, x, Wl[LIN_K], Al[LIN_K], Bl[LIN_K], adapter_on, k);
        linear_rows(c, n, H, kvw, x, Wl[LIN_V], Al[LIN_V], Bl[LIN_V], adapter_on, v);
        for (int i = 0; i < n; i++) {
            for (int hh = 0; hh < Hq; hh++) {
                float *qh = q + (size_t)i * qw + (size_t)hh * d;
                rmsnorm_rows(1, d, qh, w->q_norm + (size_t)l * d, c->rms_eps, qh);
                rope_head(qh, d, L + i, (double)c->rope_theta);
            }
            for (int hh = 0; hh < Hkv; hh++) {
                float *kh = k + (size_t)i * kvw + (size_t)hh * d;
                rmsnorm_rows(1, d, kh, w->k_norm + (size_t)l * d, c->rms_eps, kh);
                rope_head(kh, d, L + i, (double)c->rope_theta);
            }
        }
        float *Kc = cache->k + ((size_t)l * cache->capacity + L) * kvw;
        float *Vc = cache->v + ((size_t)l * cache->capacity + L) * kvw;
        memcpy(Kc, k, sizeof(float) * (size_t)n * kvw);
        memcpy(Vc, v, sizeof(float) * (size_t)n * kvw);
        attention_rows(c, l, cache, L, n, mask_mode, q, att);
        linear_rows(c, n, qw, H, att, Wl[LIN_O], Al[LIN_O], Bl[LIN_O], adapter_on, y);
        for (size_t e = 0; e < (size_t)n * H; e++) h[e] = round_bf16(h[e] + y[e]);
        /* MLP block: down( bf16(silu(gate) * up) ) */
        rmsnorm_rows(n, H, h, w->mlp_norm + (size_t)l * H, c->rms_eps, x);
        linear_rows(c, n, H, I, x, Wl[LIN_GATE], Al[LIN_GATE], Bl[LIN_GATE], adapter_on, gt);
        linear_rows(c, n, H, I, x, Wl[LIN_UP], Al[LIN_UP], Bl[LIN_UP], adapter_on, up);
        swiglu(n * I, gt, up, act);
        linear_rows(c, n, I, H, act, Wl[LIN_DOWN], Al[LIN_DOWN], Bl[LIN_DOWN], adapter_on, y);
        for (size_t e = 0; e < (size_t)n * H; e++) h[e] = round_bf16(h[e] + y[e]);
    }

    /* final norm + tied lm_head over the read-out rows, fp32 logits, lowest-index argmax */
    rmsnorm_rows(n_read, H, h + (size_t)read_first * H, w->final_norm, c->rms_eps, x);
    if (hidden_out) memcpy(hidden_out, x, sizeof(float) * (size_t)n_read * H);
    const int V = c->vocab;
    float *lg = logits ? logits : (float *)malloc(sizeof(float) * (size_t)n_read * V);
#pragma omp parallel for schedule(static)
    for (int t = 0; t < V; t++)
        for (int i = 0; i < n_read; i++) lg[(size_t)i * V + t] = dot_fw(x + (size_t)i * H, w->embed + (size_t)t * H, H);
    for (int i = 0; i < n_read; i++) {
        const float *row = lg + (size_t)i * V;
        int best = 0;
        for (int t = 1; t < V; t++)
            if (row[t] > row[best]) best = t;
        if (argmax) argmax[i] = best;
    }
    if (!logits) free(lg);
    free(h); free(x); free(q); free(k); free(v); free(att); free(y); free(gt); free(up); free(act);
    return 0;
}

/* ---- single steps exposed for the pin tests (same code as the pass uses) ---- */

void orc_op_rmsnorm(int32_t n, int32_t dim, const float *x, const uint16_t *g, float eps, float *y) {
    rmsnorm_rows(n, dim, x, g, eps, y);
}

void orc_op_linear(const orc_config *c, int32_t n, int32_t in, int32_t out, const float *x, const uint16_t *W,
                   const uint16_t *A, const uint16_t *B, int32_t adapter_on, float *y) {
    linear_rows(c, n, in, out, x, W, A, B, adapter_on, y);
}

void orc_op_rope(float *x, int32_t d, int32_t pos, double theta) { rope_head(x, d, pos, theta); }

void orc_op_swiglu(int32_t count, const float *g, const float *u, float *act) { swiglu((size_t)count, g, u, act); }

/* Attention of n block rows of `layer` against a cache whose slots [0, L+n) hold K/V. */
void orc_op_attention(const orc_config *c, int32_t layer, const orc_cache *cache, int32_t L, int32_t n,
                      int32_t mask_mode, const float *q, float *out) {
    attention_rows(c, layer, cache, L, n, mask_mode, q, out);
}

/* Write raw K/V rows into slots [L, L+n) of one layer (pin tests build caches by hand). */
int orc_cache_write(const orc_config *c, orc_cache *cc, int32_t layer, int32_t L, int32_t n, const float *k,
                    const float *v) {
    if (L < 0 || L + n > cc->capacity) return 1;
    size_t kvw = (size_t)c->n_kv_heads * c->head_dim;
    memcpy(cc->k + ((size_t)layer * cc->capacity + L) * kvw, k, sizeof(float) * n * kvw);
    memcpy(cc->v + ((size_t)layer * cc->capacity + L) * kvw, v, sizeof(float) * n * kvw);
    return 0;
}

float orc_round_bf16(float f) { return round_bf16(f); }

int32_t orc_num_threads(void) {
#ifdef _OPENMP
    return (int32_t)omp_get_max_threads();
#else
    return 1;
#endif
}
