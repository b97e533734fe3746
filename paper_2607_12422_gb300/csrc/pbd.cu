// pbd.cu -- host orchestration and C ABI of the PEFT-BD hot path (see include/pbd.h).
//
// One context owns a caller-provided device workspace holding: the weights re-tiled for the
// tensor-core kernels, the adapter's B matrices, a paged bf16 KV cache, the device-resident
// decoding state (cached lengths, pending tokens, outputs, done flags), and the scratch of
// the passes (activations, split-K partial sums, attention partials, lm_head tile maxima).
// A speculative round (draft pass, verify pass, accept/commit) only reads and writes device
// memory, so it is captured once as a CUDA graph and replayed; the host looks at the done
// flags every few rounds.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/pbd.h"
#include "pbd_internal.h"

using namespace pbd;

namespace {

thread_local std::string g_last_error;

constexpr size_t ALIGN = 1024;
constexpr int N_BN = 4;
const int BN_CHOICES[N_BN] = {32, 64, 128, 256};
constexpr int POLL_ROUNDS = 4;

enum Phase { PH_NONE = 0, PH_READY, PH_DRAFTED, PH_VERIFIED };
enum PassKind { PK_DRAFT = 0, PK_VERIFY = 1, PK_DECODE = 2, PK_PREFILL = 3 };
enum ActBuf { AB_X = 0, AB_ATTN = 1, AB_ACT = 2, AB_XRO = 3, N_AB = 4 };

struct Bump {
    uint8_t *base;
    size_t off = 0;
    explicit Bump(void *b) : base(static_cast<uint8_t *>(b)) {}
    void *take(size_t bytes) {
        off = (off + ALIGN - 1) / ALIGN * ALIGN;
        void *p = base ? base + off : nullptr;
        off += bytes;
        return p;
    }
};

int k_splits_for(int K) {
    const int kt = K / KT;
    return (kt % 4 == 0) ? kt / 4 : 1;  // 256-wide K slices per CTA when possible
}

int pick_bn(int M) {
    for (int i = 0; i < N_BN; ++i)
        if (M <= BN_CHOICES[i]) return BN_CHOICES[i];
    return 256;
}

int bn_index(int bn) {
    for (int i = 0; i < N_BN; ++i)
        if (BN_CHOICES[i] == bn) return i;
    return N_BN - 1;
}

}  // namespace

struct pbd_ctx {
    pbd_config cfg;
    Dims dm;
    cudaStream_t st;
    int D, rows_alloc, ro_alloc, out_cap, rope_rows, n_splits, pages_per_seq, n_pages;
    // weights
    std::vector<TiledWeight> w_qkv, w_o, w_gu, w_down;
    TiledWeight w_lm;
    void *lb_qkv, *lb_o, *lb_gu, *lb_down;  // adapter B, fused per layer [nl][out][r]
    void *attn_norm, *mlp_norm, *q_norm, *k_norm, *final_norm, *mask_embed;
    float2 *rope_cs;
    KVCache kv;
    int *page_table;
    // scratch
    void *h, *x, *q, *attn, *act, *x_ro;
    float *part;
    size_t part_floats;
    float *o_part;
    float2 *ml_part;
    float *tile_max;
    int *tile_arg;
    int *ids, *draft_ids, *verify_ids, *first_id, *status;
    SeqState s;
    CUtensorMap maps[N_AB][N_BN];
    // host state
    int batch = 0, max_new = 0;
    Phase phase = PH_NONE;
    std::string err;
    // graphs of pbd_bench_rounds, reused while batch size and forced table are unchanged
    cudaGraphExec_t bench_gx[2][3] = {{nullptr, nullptr, nullptr}, {nullptr, nullptr, nullptr}};
    const int32_t *bench_forced[2] = {nullptr, nullptr};
    int bench_batch[2] = {0, 0};
    size_t bench_nodes[2] = {0, 0};
    void drop_bench_graphs(int mode) {
        for (auto &g : bench_gx[mode])
            if (g) {
                cudaGraphExecDestroy(g);
                g = nullptr;
            }
        bench_batch[mode] = 0;
    }
    ~pbd_ctx() {
        drop_bench_graphs(0);
        drop_bench_graphs(1);
    }
};

namespace {

pbd_status fail(pbd_ctx *c, pbd_status code, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (c) c->err = buf;
    g_last_error = buf;
    return code;
}

#define CK(expr)                                                                                   \
    do {                                                                                           \
        cudaError_t e_ = (expr);                                                                   \
        if (e_ != cudaSuccess) return fail(c, PBD_ERR_CUDA, "%s: %s", #expr, cudaGetErrorString(e_)); \
    } while (0)

bool valid_config(const pbd_config *cfg, std::string *why) {
    char b[256];
    auto bad = [&](const char *m) {
        snprintf(b, sizeof b, "%s", m);
        *why = b;
        return false;
    };
    if (!cfg) return bad("null config");
    const pbd_config &k = *cfg;
    if (k.n_layers < 1 || k.hidden < 128 || k.n_q_heads < 1 || k.n_kv_heads < 1 || k.intermediate < 64 ||
        k.vocab < 128)
        return bad("non-positive model dimension");
    if (k.head_dim != 64 && k.head_dim != 128) return bad("head_dim must be 64 or 128");
    if (k.n_q_heads % k.n_kv_heads) return bad("n_q_heads must be a multiple of n_kv_heads");
    if (k.hidden % 128 || k.hidden > 4096) return bad("hidden must be a multiple of 128, at most 4096");
    if (((k.n_q_heads + 2 * k.n_kv_heads) * k.head_dim) % 128 || (k.n_q_heads * k.head_dim) % 64)
        return bad("q/k/v widths must tile by 128");
    if (k.intermediate % 64 || (2 * k.intermediate) % 128) return bad("intermediate must be a multiple of 64");
    if (k.vocab % 128) return bad("vocab must be a multiple of 128");
    if (k.lora_rank < 1 || k.lora_rank > 32) return bad("lora_rank must be in [1, 32]");
    if (k.page_size != PAGE) return bad("page_size must be 16");
    if (k.block_D < 1 || k.block_D > 64) return bad("block_D must be in [1, 64]");
    if (k.max_batch < 1 || k.max_batch > 64) return bad("max_batch must be in [1, 64]");
    if (k.max_batch * (k.block_D + 1) > 1024) return bad("max_batch * (block_D + 1) must be <= 1024");
    if (k.max_seq_len < 2 || k.max_seq_len > (1 << 20)) return bad("max_seq_len out of range");
    if (!(k.rms_eps > 0.f) || !(k.rope_theta > 0.f)) return bad("rms_eps and rope_theta must be positive");
    return true;
}

// Carves the workspace; with base == nullptr it only measures.  Returns total bytes.
size_t layout(pbd_ctx *c, void *base) {
    const pbd_config &k = c->cfg;
    const int nl = k.n_layers, H = k.hidden, d = k.head_dim, Hq = k.n_q_heads, Hkv = k.n_kv_heads;
    const int I = k.intermediate, V = k.vocab, r = k.lora_rank, D = k.block_D;
    c->D = D;
    c->rows_alloc = std::max(((k.max_batch * (D + 1) + 255) / 256) * 256, PREFILL_ROWS);
    c->ro_alloc = k.max_batch * (D + 1);
    c->out_cap = k.max_seq_len;
    // a truncated last round can leave L up to D past the budget, and every later pass still
    // touches D+1 slots above L: reserve twice the block width beyond max_seq_len
    const int max_tokens = k.max_seq_len + 2 * (D + 1);
    c->rope_rows = max_tokens;
    c->n_splits = (max_tokens + ATT_SPLIT - 1) / ATT_SPLIT;
    c->pages_per_seq = (max_tokens + PAGE - 1) / PAGE;
    c->n_pages = k.max_batch * c->pages_per_seq;
    const int B = k.max_batch, RA = c->rows_alloc;

    Bump bp(base);
    // device state and small buffers
    c->status = (int *)bp.take(64);
    c->s.all_done = c->status + 1;
    c->s.round = c->status + 2;
    c->s.stats = (long long *)bp.take(3 * sizeof(long long));
    c->s.L = (int *)bp.take(sizeof(int) * B);
    c->s.pending = (int *)bp.take(sizeof(int) * B);
    c->s.n_out = (int *)bp.take(sizeof(int) * B);
    c->s.done = (int *)bp.take(sizeof(int) * B);
    c->s.out_tokens = (int *)bp.take(sizeof(int) * (size_t)B * c->out_cap);
    c->ids = (int *)bp.take(sizeof(int) * RA);
    c->draft_ids = (int *)bp.take(sizeof(int) * B * D);
    c->verify_ids = (int *)bp.take(sizeof(int) * B * (D + 1));
    c->first_id = (int *)bp.take(sizeof(int) * 4);
    c->page_table = (int *)bp.take(sizeof(int) * (size_t)B * c->pages_per_seq);
    c->rope_cs = (float2 *)bp.take(sizeof(float2) * (size_t)c->rope_rows * (d / 2));

    // weights
    auto tiled = [&](int n_main, int lora_rows, int K) {
        TiledWeight w;
        w.n_main = n_main;
        w.lora_rows = lora_rows;
        w.K = K;
        const int row_tiles = n_main / TILE_ROWS + (lora_rows > 0 ? 1 : 0);
        w.tiles = bp.take((size_t)row_tiles * (K / KT) * TILE_BYTES);
        return w;
    };
    c->w_qkv.assign(nl, TiledWeight());
    c->w_o.assign(nl, TiledWeight());
    c->w_gu.assign(nl, TiledWeight());
    c->w_down.assign(nl, TiledWeight());
    const int n_qkv = (Hq + 2 * Hkv) * d;
    for (int l = 0; l < nl; ++l) {
        c->w_qkv[l] = tiled(n_qkv, 3 * r, H);
        c->w_o[l] = tiled(H, r, Hq * d);
        c->w_gu[l] = tiled(2 * I, 2 * r, H);
        c->w_down[l] = tiled(H, r, I);
    }
    c->w_lm = tiled(V, 0, H);
    const size_t e2 = 2;
    c->lb_qkv = bp.take(e2 * nl * n_qkv * r);
    c->lb_o = bp.take(e2 * nl * H * r);
    c->lb_gu = bp.take(e2 * nl * 2 * I * r);
    c->lb_down = bp.take(e2 * nl * H * r);
    c->attn_norm = bp.take(e2 * nl * H);
    c->mlp_norm = bp.take(e2 * nl * H);
    c->q_norm = bp.take(e2 * nl * d);
    c->k_norm = bp.take(e2 * nl * d);
    c->final_norm = bp.take(e2 * H);
    c->mask_embed = bp.take(e2 * H);

    // KV cache
    const size_t kv_elems = (size_t)nl * c->n_pages * Hkv * PAGE * d;
    c->kv.k = bp.take(kv_elems * e2);
    c->kv.v = bp.take(kv_elems * e2);
    c->kv.page_table = c->page_table;
    c->kv.pages_per_seq = c->pages_per_seq;
    c->kv.n_pages = c->n_pages;

    // activations and scratch
    c->h = bp.take(e2 * RA * H);
    c->x = bp.take(e2 * RA * H);
    c->q = bp.take(e2 * RA * Hq * d);
    c->attn = bp.take(e2 * RA * Hq * d);
    c->act = bp.take(e2 * RA * I);
    c->x_ro = bp.take(e2 * c->ro_alloc * H);
    size_t pf = 0;
    pf = std::max(pf, (size_t)k_splits_for(H) * RA * (n_qkv + 3 * r));
    pf = std::max(pf, (size_t)k_splits_for(Hq * d) * RA * (H + r));
    pf = std::max(pf, (size_t)k_splits_for(H) * RA * (2 * I + 2 * r));
    pf = std::max(pf, (size_t)k_splits_for(I) * RA * (H + r));
    c->part_floats = pf;
    c->part = (float *)bp.take(sizeof(float) * pf);
    c->o_part = (float *)bp.take(sizeof(float) * (size_t)RA * Hq * c->n_splits * d);
    c->ml_part = (float2 *)bp.take(sizeof(float2) * (size_t)RA * Hq * c->n_splits);
    c->tile_max = (float *)bp.take(sizeof(float) * (size_t)(V / TILE_ROWS) * c->ro_alloc);
    c->tile_arg = (int *)bp.take(sizeof(int) * (size_t)(V / TILE_ROWS) * c->ro_alloc);
    return bp.off + ALIGN;
}

Partials partials_for(pbd_ctx *c, const TiledWeight &w) {
    Partials p;
    p.p = c->part;
    p.k_splits = k_splits_for(w.K);
    p.rows_alloc = c->rows_alloc;
    p.n_total = w.n_main + w.lora_rows;
    return p;
}

pbd_status make_maps(pbd_ctx *c) {
    const pbd_config &k = c->cfg;
    struct {
        void *p;
        int rows, cols;
    } bufs[N_AB] = {{c->x, c->rows_alloc, k.hidden},
                    {c->attn, c->rows_alloc, k.n_q_heads * k.head_dim},
                    {c->act, c->rows_alloc, k.intermediate},
                    {c->x_ro, c->ro_alloc, k.hidden}};
    for (int a = 0; a < N_AB; ++a)
        for (int i = 0; i < N_BN; ++i)
            if (!encode_bf16_map(&c->maps[a][i], bufs[a].p, bufs[a].rows, bufs[a].cols, BN_CHOICES[i]))
                return fail(c, PBD_ERR_CUDA, "tensor map encode failed (buffer %d, box rows %d)", a, BN_CHOICES[i]);
    return PBD_OK;
}

// Copy rows of a layer-stacked source into a tiled weight at a row offset.
pbd_status repack(pbd_ctx *c, const void *src, size_t layer_elems, int l, int rows, int K, const TiledWeight &w,
                  int row0) {
    if (!src) return fail(c, PBD_ERR_INVALID_ARG, "null weight pointer");
    const void *p = static_cast<const uint8_t *>(src) + 2 * layer_elems * l;
    CK(launch_repack_tiled(p, rows, K, const_cast<void *>(w.tiles), row0, c->st));
    return PBD_OK;
}

pbd_status copy_dev(pbd_ctx *c, void *dst, const void *src, size_t bytes) {
    if (!src) return fail(c, PBD_ERR_INVALID_ARG, "null weight pointer");
    CK(cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToDevice, c->st));
    return PBD_OK;
}

#define TRY(expr)                             \
    do {                                      \
        pbd_status s_ = (expr);               \
        if (s_ != PBD_OK) return s_;          \
    } while (0)

pbd_status load_weights(pbd_ctx *c, const pbd_base_weights *bw, const pbd_adapter_weights *aw) {
    const pbd_config &k = c->cfg;
    const int nl = k.n_layers, H = k.hidden, d = k.head_dim, Hq = k.n_q_heads, Hkv = k.n_kv_heads;
    const int I = k.intermediate, r = k.lora_rank;
    const int qw = Hq * d, kvw = Hkv * d, n_qkv = qw + 2 * kvw;
    // zero the tile storage first so the padding rows of the adapter tiles are defined
    for (int l = 0; l < nl; ++l) {
        const TiledWeight *ws[4] = {&c->w_qkv[l], &c->w_o[l], &c->w_gu[l], &c->w_down[l]};
        for (const TiledWeight *w : ws) {
            const int rt = w->n_main / TILE_ROWS + (w->lora_rows > 0 ? 1 : 0);
            CK(cudaMemsetAsync(const_cast<void *>(w->tiles), 0, (size_t)rt * (w->K / KT) * TILE_BYTES, c->st));
        }
    }
    const size_t e2 = 2;
    for (int l = 0; l < nl; ++l) {
        // fused q|k|v rows, then the adapter's A_q, A_k, A_v rows
        TRY(repack(c, bw->w[0], (size_t)qw * H, l, qw, H, c->w_qkv[l], 0));
        TRY(repack(c, bw->w[1], (size_t)kvw * H, l, kvw, H, c->w_qkv[l], qw));
        TRY(repack(c, bw->w[2], (size_t)kvw * H, l, kvw, H, c->w_qkv[l], qw + kvw));
        for (int t = 0; t < 3; ++t) TRY(repack(c, aw->lora_a[t], (size_t)r * H, l, r, H, c->w_qkv[l], n_qkv + t * r));
        TRY(repack(c, bw->w[3], (size_t)H * qw, l, H, qw, c->w_o[l], 0));
        TRY(repack(c, aw->lora_a[3], (size_t)r * qw, l, r, qw, c->w_o[l], H));
        TRY(repack(c, bw->w[4], (size_t)I * H, l, I, H, c->w_gu[l], 0));
        TRY(repack(c, bw->w[5], (size_t)I * H, l, I, H, c->w_gu[l], I));
        TRY(repack(c, aw->lora_a[4], (size_t)r * H, l, r, H, c->w_gu[l], 2 * I));
        TRY(repack(c, aw->lora_a[5], (size_t)r * H, l, r, H, c->w_gu[l], 2 * I + r));
        TRY(repack(c, bw->w[6], (size_t)H * I, l, H, I, c->w_down[l], 0));
        TRY(repack(c, aw->lora_a[6], (size_t)r * I, l, r, I, c->w_down[l], H));
        // adapter B matrices, fused in the same output order as the main rows
        uint8_t *lq = static_cast<uint8_t *>(c->lb_qkv) + e2 * (size_t)l * n_qkv * r;
        const int outs[3] = {qw, kvw, kvw};
        size_t off = 0;
        for (int t = 0; t < 3; ++t) {
            if (!aw->lora_b[t]) return fail(c, PBD_ERR_INVALID_ARG, "null adapter B pointer");
            TRY(copy_dev(c, lq + off, static_cast<const uint8_t *>(aw->lora_b[t]) + e2 * (size_t)l * outs[t] * r,
                         e2 * (size_t)outs[t] * r));
            off += e2 * (size_t)outs[t] * r;
        }
        TRY(copy_dev(c, static_cast<uint8_t *>(c->lb_o) + e2 * (size_t)l * H * r,
                     static_cast<const uint8_t *>(aw->lora_b[3]) + e2 * (size_t)l * H * r, e2 * (size_t)H * r));
        uint8_t *lg = static_cast<uint8_t *>(c->lb_gu) + e2 * (size_t)l * 2 * I * r;
        TRY(copy_dev(c, lg, static_cast<const uint8_t *>(aw->lora_b[4]) + e2 * (size_t)l * I * r, e2 * (size_t)I * r));
        TRY(copy_dev(c, lg + e2 * (size_t)I * r, static_cast<const uint8_t *>(aw->lora_b[5]) + e2 * (size_t)l * I * r,
                     e2 * (size_t)I * r));
        TRY(copy_dev(c, static_cast<uint8_t *>(c->lb_down) + e2 * (size_t)l * H * r,
                     static_cast<const uint8_t *>(aw->lora_b[6]) + e2 * (size_t)l * H * r, e2 * (size_t)H * r));
    }
    TRY(repack(c, bw->embed, 0, 0, k.vocab, H, c->w_lm, 0));
    TRY(copy_dev(c, c->attn_norm, bw->attn_norm, e2 * nl * H));
    TRY(copy_dev(c, c->mlp_norm, bw->mlp_norm, e2 * nl * H));
    TRY(copy_dev(c, c->q_norm, bw->q_norm, e2 * nl * d));
    TRY(copy_dev(c, c->k_norm, bw->k_norm, e2 * nl * d));
    TRY(copy_dev(c, c->final_norm, bw->final_norm, e2 * H));
    TRY(copy_dev(c, c->mask_embed, aw->mask_embed, e2 * H));
    return PBD_OK;
}

pbd_status build_rope(pbd_ctx *c) {
    const int d = c->cfg.head_dim, half = d / 2;
    std::vector<float2> t((size_t)c->rope_rows * half);
    for (int p = 0; p < c->rope_rows; ++p)
        for (int i = 0; i < half; ++i) {
            const double inv = std::pow((double)c->cfg.rope_theta, -2.0 * i / d);
            const double a = (double)p * inv;
            t[(size_t)p * half + i] = make_float2((float)std::cos(a), (float)std::sin(a));
        }
    CK(cudaMemcpyAsync(c->rope_cs, t.data(), t.size() * sizeof(float2), cudaMemcpyHostToDevice, c->st));
    CK(cudaStreamSynchronize(c->st));
    return PBD_OK;
}

// One forward pass of nb sequences x R rows through all layers and the lm_head.
pbd_status run_pass(pbd_ctx *c, const PassDesc &pd, int *ids_out, float *logits) {
    const Dims &dm = c->dm;
    const int nl = dm.nl;
    const int bn = pick_bn(pd.M), bi = bn_index(bn);
    cudaStream_t st = c->st;
    CK(launch_embed_norm(dm, pd, c->ids, c->w_lm.tiles, c->mask_embed, c->attn_norm, c->h, c->x, c->status, st));
    const size_t e2 = 2;
    const int n_qkv = (dm.Hq + 2 * dm.Hkv) * dm.d;
    for (int l = 0; l < nl; ++l) {
        const Partials pq = partials_for(c, c->w_qkv[l]);
        CK(launch_linear_partials(&c->maps[AB_X][bi], bn, c->w_qkv[l], pd.adapter, pd.M, pq, c->status, st));
        CK(launch_qkv_finalize(dm, pd, l, pq, static_cast<uint8_t *>(c->lb_qkv) + e2 * (size_t)l * n_qkv * dm.r,
                               c->q_norm, c->k_norm, c->rope_cs, c->rope_rows, c->s.L, c->kv, c->q, c->status, st));
        CK(launch_attention(dm, pd, l, c->q, c->kv, c->s.L, c->n_splits, c->o_part, c->ml_part, st));
        CK(launch_attn_combine(dm, pd, c->s.L, c->n_splits, c->o_part, c->ml_part, c->attn, st));
        const Partials po = partials_for(c, c->w_o[l]);
        CK(launch_linear_partials(&c->maps[AB_ATTN][bi], bn, c->w_o[l], pd.adapter, pd.M, po, c->status, st));
        CK(launch_residual_norm(dm, pd, po, dm.H, static_cast<uint8_t *>(c->lb_o) + e2 * (size_t)l * dm.H * dm.r,
                                static_cast<uint8_t *>(c->mlp_norm) + e2 * (size_t)l * dm.H, c->h, c->x, nullptr, st));
        const Partials pg = partials_for(c, c->w_gu[l]);
        CK(launch_linear_partials(&c->maps[AB_X][bi], bn, c->w_gu[l], pd.adapter, pd.M, pg, c->status, st));
        CK(launch_act(dm, pd, pg, static_cast<uint8_t *>(c->lb_gu) + e2 * (size_t)l * 2 * dm.I * dm.r, c->act, st));
        const Partials pdn = partials_for(c, c->w_down[l]);
        CK(launch_linear_partials(&c->maps[AB_ACT][bi], bn, c->w_down[l], pd.adapter, pd.M, pdn, c->status, st));
        const void *gain = (l + 1 < nl) ? static_cast<const void *>(static_cast<uint8_t *>(c->attn_norm) +
                                                                    e2 * (size_t)(l + 1) * dm.H)
                                        : c->final_norm;
        CK(launch_residual_norm(dm, pd, pdn, dm.H, static_cast<uint8_t *>(c->lb_down) + e2 * (size_t)l * dm.H * dm.r,
                                gain, c->h, c->x, (l + 1 == nl) ? c->x_ro : nullptr, st));
    }
    const int n_ro = pd.nb * pd.ro_count;
    if (n_ro > 0) {
        const int bro = pick_bn(n_ro);
        CK(launch_lm_head(&c->maps[AB_XRO][bn_index(bro)], bro, c->w_lm, n_ro, c->tile_max, c->tile_arg, logits,
                          c->status, st));
        CK(launch_argmax_reduce(c->tile_max, c->tile_arg, dm.V / TILE_ROWS, n_ro, ids_out, st));
    }
    return PBD_OK;
}

PassDesc block_pass(pbd_ctx *c, int kind) {
    PassDesc pd;
    pd.b0 = 0;
    pd.nb = c->batch;
    pd.R = (kind == PK_DECODE) ? 1 : c->D + 1;
    pd.M = pd.nb * pd.R;
    pd.adapter = kind == PK_DRAFT ? 1 : 0;
    pd.mask_mode = kind == PK_DRAFT ? MASK_BLOCK_DRAFT : MASK_CAUSAL;
    pd.ro_first = 0;
    pd.ro_count = kind == PK_DRAFT ? c->D : pd.R;
    return pd;
}

pbd_status enqueue_draft(pbd_ctx *c, float *logits) {
    const PassDesc pd = block_pass(c, PK_DRAFT);
    CK(launch_build_ids(pd, 0, c->s.pending, nullptr, c->D, c->ids, c->st));
    return run_pass(c, pd, c->draft_ids, logits);
}

pbd_status enqueue_verify(pbd_ctx *c, const int *drafts, float *logits) {
    const PassDesc pd = block_pass(c, PK_VERIFY);
    CK(launch_build_ids(pd, 1, c->s.pending, drafts, c->D, c->ids, c->st));
    return run_pass(c, pd, c->verify_ids, logits);
}

pbd_status enqueue_accept(pbd_ctx *c, const int *forced, int *accepted) {
    CK(launch_accept_commit(c->s, c->batch, c->D, c->draft_ids, c->verify_ids, forced, c->batch, c->max_new,
                            c->out_cap, accepted, c->st));
    return PBD_OK;
}

pbd_status enqueue_decode(pbd_ctx *c, float *logits) {
    const PassDesc pd = block_pass(c, PK_DECODE);
    CK(launch_build_ids(pd, 2, c->s.pending, nullptr, 0, c->ids, c->st));
    TRY(run_pass(c, pd, c->verify_ids, logits));
    CK(launch_accept_commit(c->s, c->batch, 0, c->draft_ids, c->verify_ids, nullptr, c->batch, c->max_new, c->out_cap,
                            nullptr, c->st));
    return PBD_OK;
}

pbd_status check_device(pbd_ctx *c) {
    CK(cudaStreamSynchronize(c->st));
    int code = 0;
    CK(cudaMemcpy(&code, c->status, sizeof(int), cudaMemcpyDeviceToHost));
    if (code != 0) return fail(c, PBD_ERR_DEVICE, "device status %d latched by a kernel", code);
    return PBD_OK;
}

}  // namespace

extern "C" {

size_t pbd_workspace_bytes(const pbd_config *cfg) {
    std::string why;
    if (!valid_config(cfg, &why)) return 0;
    pbd_ctx tmp;
    tmp.cfg = *cfg;
    return layout(&tmp, nullptr);
}

pbd_status pbd_create(const pbd_config *cfg, const pbd_base_weights *base, const pbd_adapter_weights *adapter,
                      void *d_workspace, size_t workspace_bytes, void *d_stream, pbd_ctx **out) {
    pbd_ctx *c = nullptr;
    if (!out) return fail(c, PBD_ERR_INVALID_ARG, "null output pointer");
    *out = nullptr;
    std::string why;
    if (!valid_config(cfg, &why)) return fail(c, PBD_ERR_INVALID_ARG, "invalid config: %s", why.c_str());
    if (!base || !adapter) return fail(c, PBD_ERR_INVALID_ARG, "null weights");
    if (!d_workspace || (reinterpret_cast<uintptr_t>(d_workspace) & 255))
        return fail(c, PBD_ERR_WORKSPACE, "workspace missing or not 256-byte aligned");
    c = new pbd_ctx();
    c->cfg = *cfg;
    const size_t need = layout(c, nullptr);
    if (workspace_bytes < need) {
        delete c;
        return fail(nullptr, PBD_ERR_WORKSPACE, "workspace too small: %zu < %zu bytes", workspace_bytes, need);
    }
    // align the carve base to 1024 bytes inside the workspace
    uint8_t *wb = static_cast<uint8_t *>(d_workspace);
    uint8_t *b1024 = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(wb) + ALIGN - 1) & ~(uintptr_t)(ALIGN - 1));
    layout(c, b1024);
    c->st = static_cast<cudaStream_t>(d_stream);
    c->dm = Dims{cfg->n_layers, cfg->hidden,      cfg->n_q_heads, cfg->n_kv_heads, cfg->head_dim,
                 cfg->intermediate, cfg->vocab, cfg->lora_rank, cfg->rms_eps,     cfg->lora_scale};
    pbd_status s;
    cudaError_t e;
    if ((e = configure_linear_kernels()) != cudaSuccess || (e = configure_attention_kernels()) != cudaSuccess) {
        s = fail(c, PBD_ERR_CUDA, "kernel configuration: %s", cudaGetErrorString(e));
        delete c;
        return s;
    }
    if ((s = load_weights(c, base, adapter)) != PBD_OK || (s = build_rope(c)) != PBD_OK || (s = make_maps(c)) != PBD_OK) {
        delete c;
        return s;
    }
    const size_t kv_bytes = (size_t)cfg->n_layers * c->n_pages * cfg->n_kv_heads * PAGE * cfg->head_dim * 2;
    if ((e = cudaMemsetAsync(c->kv.k, 0, kv_bytes, c->st)) != cudaSuccess ||
        (e = cudaMemsetAsync(c->kv.v, 0, kv_bytes, c->st)) != cudaSuccess ||
        (e = cudaMemsetAsync(c->status, 0, 64, c->st)) != cudaSuccess ||
        (e = cudaMemsetAsync(c->part, 0, sizeof(float) * c->part_floats, c->st)) != cudaSuccess ||
        (e = cudaStreamSynchronize(c->st)) != cudaSuccess) {
        s = fail(c, PBD_ERR_CUDA, "workspace init: %s", cudaGetErrorString(e));
        delete c;
        return s;
    }
    *out = c;
    return PBD_OK;
}

pbd_status pbd_destroy(pbd_ctx *c) {
    if (!c) return PBD_ERR_INVALID_ARG;
    cudaStreamSynchronize(c->st);
    delete c;
    return PBD_OK;
}

pbd_status pbd_prefill(pbd_ctx *c, int32_t batch, const int32_t *d_prompt_ids, const int32_t *h_prompt_lens,
                       int32_t max_new, int32_t *d_first_token) {
    if (!c) return fail(c, PBD_ERR_INVALID_ARG, "null context");
    if (batch < 1 || batch > c->cfg.max_batch) return fail(c, PBD_ERR_CAPACITY, "batch %d outside [1, %d]", batch, c->cfg.max_batch);
    if (!d_prompt_ids || !h_prompt_lens) return fail(c, PBD_ERR_INVALID_ARG, "null prompt");
    if (max_new < 1) return fail(c, PBD_ERR_INVALID_ARG, "max_new must be >= 1");
    for (int b = 0; b < batch; ++b)
        if (h_prompt_lens[b] < 1 || h_prompt_lens[b] + max_new > c->cfg.max_seq_len)
            return fail(c, PBD_ERR_CAPACITY, "sequence %d: prompt %d + max_new %d exceeds max_seq_len %d", b,
                        h_prompt_lens[b], max_new, c->cfg.max_seq_len);
    // pages of sequence b are interleaved across the batch: page (b, j) -> j * batch + b
    std::vector<int> pt((size_t)c->cfg.max_batch * c->pages_per_seq, 0);
    for (int b = 0; b < batch; ++b)
        for (int j = 0; j < c->pages_per_seq; ++j) pt[(size_t)b * c->pages_per_seq + j] = j * batch + b;
    CK(cudaMemcpyAsync(c->page_table, pt.data(), pt.size() * sizeof(int), cudaMemcpyHostToDevice, c->st));
    CK(cudaMemsetAsync(c->s.L, 0, sizeof(int) * c->cfg.max_batch, c->st));
    CK(cudaMemsetAsync(c->s.n_out, 0, sizeof(int) * c->cfg.max_batch, c->st));
    CK(cudaMemsetAsync(c->s.done, 0, sizeof(int) * c->cfg.max_batch, c->st));
    CK(cudaMemsetAsync(c->s.all_done, 0, 2 * sizeof(int), c->st));
    CK(cudaMemsetAsync(c->s.stats, 0, 3 * sizeof(long long), c->st));
    c->batch = batch;
    c->max_new = max_new;
    size_t off = 0;
    for (int b = 0; b < batch; ++b) {
        const int P = h_prompt_lens[b];
        for (int c0 = 0; c0 < P; c0 += PREFILL_ROWS) {
            const int rows = std::min(PREFILL_ROWS, P - c0);
            const bool last = c0 + rows == P;
            PassDesc pd;
            pd.b0 = b;
            pd.nb = 1;
            pd.R = rows;
            pd.M = rows;
            pd.adapter = 0;
            pd.mask_mode = MASK_CAUSAL;
            pd.ro_first = last ? rows - 1 : 0;
            pd.ro_count = last ? 1 : 0;
            CK(launch_set_len(c->s.L, b, c0, c->st));
            CK(cudaMemcpyAsync(c->ids, d_prompt_ids + off + c0, sizeof(int) * rows, cudaMemcpyDeviceToDevice, c->st));
            TRY(run_pass(c, pd, c->first_id, nullptr));
        }
        CK(launch_prefill_finish(c->s, b, P, c->first_id, max_new, c->out_cap, c->st));
        off += P;
    }
    if (d_first_token)
        CK(cudaMemcpyAsync(d_first_token, c->s.pending, sizeof(int) * batch, cudaMemcpyDeviceToDevice, c->st));
    TRY(check_device(c));
    c->phase = PH_READY;
    return PBD_OK;
}

pbd_status pbd_draft_block(pbd_ctx *c, int32_t *d_draft, float *d_logits_opt) {
    if (!c) return fail(c, PBD_ERR_INVALID_ARG, "null context");
    if (c->phase != PH_READY) return fail(c, PBD_ERR_STATE, "draft needs a prefilled or committed state");
    TRY(enqueue_draft(c, d_logits_opt));
    if (d_draft)
        CK(cudaMemcpyAsync(d_draft, c->draft_ids, sizeof(int) * c->batch * c->D, cudaMemcpyDeviceToDevice, c->st));
    c->phase = PH_DRAFTED;
    return PBD_OK;
}

pbd_status pbd_verify_block(pbd_ctx *c, const int32_t *d_draft, int32_t *d_verify, float *d_logits_opt) {
    if (!c) return fail(c, PBD_ERR_INVALID_ARG, "null context");
    if (c->phase == PH_DRAFTED || (c->phase == PH_READY && d_draft != nullptr)) {
        if (d_draft && d_draft != c->draft_ids)
            CK(cudaMemcpyAsync(c->draft_ids, d_draft, sizeof(int) * c->batch * c->D, cudaMemcpyDeviceToDevice, c->st));
        TRY(enqueue_verify(c, c->draft_ids, d_logits_opt));
        if (d_verify)
            CK(cudaMemcpyAsync(d_verify, c->verify_ids, sizeof(int) * c->batch * (c->D + 1), cudaMemcpyDeviceToDevice,
                               c->st));
        c->phase = PH_VERIFIED;
        return PBD_OK;
    }
    return fail(c, PBD_ERR_STATE, "verify needs a draft (or explicit proposals)");
}

pbd_status pbd_accept_commit(pbd_ctx *c, const int32_t *d_forced_n_opt, int32_t *d_accepted_n) {
    if (!c) return fail(c, PBD_ERR_INVALID_ARG, "null context");
    if (c->phase != PH_VERIFIED) return fail(c, PBD_ERR_STATE, "accept/commit needs a verify pass first");
    // a forced length for this call only: index it as round 0 of a one-row table
    if (d_forced_n_opt) {
        CK(cudaMemsetAsync(c->s.round, 0, sizeof(int), c->st));
    }
    TRY(enqueue_accept(c, d_forced_n_opt, d_accepted_n));
    c->phase = PH_READY;
    return PBD_OK;
}

pbd_status pbd_decode_step(pbd_ctx *c, int32_t *d_next_opt, float *d_logits_opt) {
    if (!c) return fail(c, PBD_ERR_INVALID_ARG, "null context");
    if (c->phase != PH_READY) return fail(c, PBD_ERR_STATE, "decode step needs a prefilled or committed state");
    TRY(enqueue_decode(c, d_logits_opt));
    if (d_next_opt) CK(cudaMemcpyAsync(d_next_opt, c->verify_ids, sizeof(int) * c->batch, cudaMemcpyDeviceToDevice, c->st));
    return PBD_OK;
}

pbd_status pbd_generate(pbd_ctx *c, int32_t batch, const int32_t *d_prompt_ids, const int32_t *h_prompt_lens,
                        int32_t max_new, int32_t mode, const int32_t *d_forced_n_seq_opt, int32_t *d_out_tokens,
                        pbd_stats *h_stats_opt) {
    if (!c) return fail(c, PBD_ERR_INVALID_ARG, "null context");
    if (mode != 0 && mode != 1) return fail(c, PBD_ERR_INVALID_ARG, "mode must be 0 (speculative) or 1 (AR)");
    if (!d_out_tokens) return fail(c, PBD_ERR_INVALID_ARG, "null output");
    TRY(pbd_prefill(c, batch, d_prompt_ids, h_prompt_lens, max_new, nullptr));
    CK(cudaMemsetAsync(c->s.round, 0, sizeof(int), c->st));
    // capture one round as a graph (legacy default stream cannot be captured: run eagerly there)
    cudaGraph_t g = nullptr;
    cudaGraphExec_t ge = nullptr;
    const bool use_graph = c->st != nullptr && c->st != cudaStreamLegacy;
    auto enqueue_round = [&]() -> pbd_status {
        if (mode == 0) {
            TRY(enqueue_draft(c, nullptr));
            TRY(enqueue_verify(c, c->draft_ids, nullptr));
            return enqueue_accept(c, d_forced_n_seq_opt, nullptr);
        }
        return enqueue_decode(c, nullptr);
    };
    if (use_graph) {
        CK(cudaStreamBeginCapture(c->st, cudaStreamCaptureModeThreadLocal));
        pbd_status s = enqueue_round();
        cudaError_t e = cudaStreamEndCapture(c->st, &g);
        if (s != PBD_OK) {
            if (g) cudaGraphDestroy(g);
            return s;
        }
        CK(e);
        e = cudaGraphInstantiate(&ge, g, 0);
        cudaGraphDestroy(g);
        CK(e);
    }
    pbd_status result = PBD_OK;
    const int max_rounds = max_new + 1;
    int rounds = 0;
    int flags[2] = {0, 0};
    while (rounds < max_rounds) {
        for (int i = 0; i < POLL_ROUNDS && rounds < max_rounds; ++i, ++rounds) {
            if (use_graph) {
                cudaError_t e = cudaGraphLaunch(ge, c->st);
                if (e != cudaSuccess) {
                    result = fail(c, PBD_ERR_CUDA, "graph launch: %s", cudaGetErrorString(e));
                    break;
                }
            } else if ((result = enqueue_round()) != PBD_OK) {
                break;
            }
        }
        if (result != PBD_OK) break;
        cudaError_t e = cudaMemcpyAsync(flags, c->status, 2 * sizeof(int), cudaMemcpyDeviceToHost, c->st);
        if (e == cudaSuccess) e = cudaStreamSynchronize(c->st);
        if (e != cudaSuccess) {
            result = fail(c, PBD_ERR_CUDA, "poll: %s", cudaGetErrorString(e));
            break;
        }
        if (flags[0] != 0) {
            result = fail(c, PBD_ERR_DEVICE, "device status %d latched by a kernel", flags[0]);
            break;
        }
        if (flags[1]) break;
    }
    if (ge) cudaGraphExecDestroy(ge);
    if (result != PBD_OK) return result;
    if (!flags[1]) return fail(c, PBD_ERR_DEVICE, "generation did not finish within %d rounds", max_rounds);
    CK(cudaMemcpy2DAsync(d_out_tokens, sizeof(int) * max_new, c->s.out_tokens, sizeof(int) * c->out_cap,
                         sizeof(int) * max_new, batch, cudaMemcpyDeviceToDevice, c->st));
    if (h_stats_opt) {
        long long st3[3];
        CK(cudaMemcpyAsync(st3, c->s.stats, sizeof st3, cudaMemcpyDeviceToHost, c->st));
        CK(cudaStreamSynchronize(c->st));
        h_stats_opt->rounds = st3[0];
        h_stats_opt->accepted = st3[1];
        h_stats_opt->emitted = st3[2] + batch;
        h_stats_opt->draft_ms = 0;
        h_stats_opt->verify_ms = 0;
    }
    c->phase = PH_READY;
    return check_device(c);
}

pbd_status pbd_get_state(pbd_ctx *c, int32_t *h_L, int32_t *h_pending, int32_t *h_n_out) {
    if (!c) return fail(c, PBD_ERR_INVALID_ARG, "null context");
    TRY(check_device(c));
    const size_t n = sizeof(int) * std::max(c->batch, 1);
    if (h_L) CK(cudaMemcpy(h_L, c->s.L, n, cudaMemcpyDeviceToHost));
    if (h_pending) CK(cudaMemcpy(h_pending, c->s.pending, n, cudaMemcpyDeviceToHost));
    if (h_n_out) CK(cudaMemcpy(h_n_out, c->s.n_out, n, cudaMemcpyDeviceToHost));
    return PBD_OK;
}

pbd_status pbd_get_tokens(pbd_ctx *c, int32_t *d_out_tokens) {
    if (!c || !d_out_tokens) return fail(c, PBD_ERR_INVALID_ARG, "null argument");
    if (c->batch < 1) return fail(c, PBD_ERR_STATE, "no generation started");
    CK(cudaMemcpy2DAsync(d_out_tokens, sizeof(int) * c->max_new, c->s.out_tokens, sizeof(int) * c->out_cap,
                         sizeof(int) * c->max_new, c->batch, cudaMemcpyDeviceToDevice, c->st));
    return PBD_OK;
}

pbd_status pbd_read_kv(pbd_ctx *c, int32_t layer, int32_t seq, int32_t n, void *d_k_out, void *d_v_out) {
    if (!c || !d_k_out || !d_v_out) return fail(c, PBD_ERR_INVALID_ARG, "null argument");
    if (layer < 0 || layer >= c->cfg.n_layers || seq < 0 || seq >= c->cfg.max_batch || n < 0 ||
        n > c->pages_per_seq * PAGE)
        return fail(c, PBD_ERR_INVALID_ARG, "layer/seq/n out of range");
    CK(launch_read_kv(c->dm, c->kv, layer, seq, n, d_k_out, d_v_out, c->st));
    return PBD_OK;
}

pbd_status pbd_sync(pbd_ctx *c) {
    if (!c) return fail(c, PBD_ERR_INVALID_ARG, "null context");
    return check_device(c);
}

pbd_status pbd_bench_rounds(pbd_ctx *c, int32_t mode, int32_t warmup, int32_t steps, const int32_t *d_forced_n_seq_opt,
                            double *h_ms, int32_t *h_launches) {
    if (!c || !h_ms) return fail(c, PBD_ERR_INVALID_ARG, "null argument");
    if (mode != 0 && mode != 1) return fail(c, PBD_ERR_INVALID_ARG, "mode must be 0 or 1");
    if (steps < 1 || warmup < 0) return fail(c, PBD_ERR_INVALID_ARG, "steps must be >= 1");
    if (c->phase != PH_READY) return fail(c, PBD_ERR_STATE, "bench needs a prefilled or committed state");
    if (c->st == nullptr || c->st == cudaStreamLegacy)
        return fail(c, PBD_ERR_INVALID_ARG, "bench needs a non-default stream (graph capture)");
    CK(cudaMemsetAsync(c->s.round, 0, sizeof(int), c->st));
    const int nph = 3;
    cudaGraphExec_t *gx = c->bench_gx[mode];
    const bool cached = c->bench_batch[mode] == c->batch && c->bench_forced[mode] == d_forced_n_seq_opt &&
                        gx[mode == 0 ? 0 : 1] != nullptr;
    if (!cached) c->drop_bench_graphs(mode);
    size_t nodes = cached ? c->bench_nodes[mode] : 0;
    pbd_status s = PBD_OK;
    for (int ph = 0; ph < nph && s == PBD_OK && !cached; ++ph) {
        if (mode == 1 && ph == 0) continue;  // no draft phase in plain decoding
        cudaGraph_t g = nullptr;
        CK(cudaStreamBeginCapture(c->st, cudaStreamCaptureModeThreadLocal));
        if (mode == 0) {
            if (ph == 0) s = enqueue_draft(c, nullptr);
            if (ph == 1) s = enqueue_verify(c, c->draft_ids, nullptr);
            if (ph == 2) s = enqueue_accept(c, d_forced_n_seq_opt, nullptr);
        } else {
            const PassDesc pd = block_pass(c, PK_DECODE);
            if (ph == 1) {
                cudaError_t e = launch_build_ids(pd, 2, c->s.pending, nullptr, 0, c->ids, c->st);
                s = e == cudaSuccess ? run_pass(c, pd, c->verify_ids, nullptr)
                                     : fail(c, PBD_ERR_CUDA, "build ids: %s", cudaGetErrorString(e));
            }
            if (ph == 2) {
                cudaError_t e = launch_accept_commit(c->s, c->batch, 0, c->draft_ids, c->verify_ids, nullptr,
                                                     c->batch, c->max_new, c->out_cap, nullptr, c->st);
                if (e != cudaSuccess) s = fail(c, PBD_ERR_CUDA, "accept: %s", cudaGetErrorString(e));
            }
        }
        cudaError_t e = cudaStreamEndCapture(c->st, &g);
        if (s == PBD_OK && e != cudaSuccess) s = fail(c, PBD_ERR_CUDA, "capture: %s", cudaGetErrorString(e));
        if (s == PBD_OK) {
            size_t n = 0;
            cudaGraphGetNodes(g, nullptr, &n);
            nodes += n;
            e = cudaGraphInstantiate(&gx[ph], g, 0);
            if (e != cudaSuccess) s = fail(c, PBD_ERR_CUDA, "instantiate: %s", cudaGetErrorString(e));
        }
        if (g) cudaGraphDestroy(g);
    }
    if (s != PBD_OK) {
        c->drop_bench_graphs(mode);
        return s;
    }
    if (!cached) {
        c->bench_batch[mode] = c->batch;
        c->bench_forced[mode] = d_forced_n_seq_opt;
        c->bench_nodes[mode] = nodes;
    }
    std::vector<cudaEvent_t> ev;
    if (s == PBD_OK) {
        ev.resize((size_t)steps * 4, nullptr);
        for (auto &x : ev)
            if (cudaEventCreate(&x) != cudaSuccess) s = fail(c, PBD_ERR_CUDA, "event create");
    }
    for (int i = 0; s == PBD_OK && i < warmup + steps; ++i) {
        const bool timed = i >= warmup;
        cudaEvent_t *e4 = timed ? &ev[(size_t)(i - warmup) * 4] : nullptr;
        for (int ph = 0; ph < nph; ++ph) {
            if (timed) cudaEventRecord(e4[ph], c->st);
            if (gx[ph] && cudaGraphLaunch(gx[ph], c->st) != cudaSuccess) {
                s = fail(c, PBD_ERR_CUDA, "graph launch");
                break;
            }
        }
        if (timed) cudaEventRecord(e4[3], c->st);
    }
    if (s == PBD_OK && cudaStreamSynchronize(c->st) != cudaSuccess) s = fail(c, PBD_ERR_CUDA, "bench sync");
    if (s == PBD_OK) {
        double acc[3] = {0, 0, 0};
        for (int i = 0; i < steps; ++i)
            for (int ph = 0; ph < 3; ++ph) {
                float ms = 0.f;
                cudaEventElapsedTime(&ms, ev[(size_t)i * 4 + ph], ev[(size_t)i * 4 + ph + 1]);
                acc[ph] += ms;
            }
        float tot = 0.f;
        cudaEventElapsedTime(&tot, ev[0], ev[(size_t)(steps - 1) * 4 + 3]);
        h_ms[0] = acc[0];
        h_ms[1] = acc[1];
        h_ms[2] = acc[2];
        h_ms[3] = tot;
        if (h_launches) *h_launches = (int32_t)nodes;
    }
    for (auto &x : ev)
        if (x) cudaEventDestroy(x);
    if (s != PBD_OK) {
        c->drop_bench_graphs(mode);
        return s;
    }
    c->phase = PH_READY;
    return check_device(c);
}

pbd_status pbd_time_linear(pbd_ctx *c, int32_t which, int32_t rows, int32_t adapter, int32_t iters,
                           double *h_ms_per_launch, double *h_weight_bytes) {
    if (!c || !h_ms_per_launch) return fail(c, PBD_ERR_INVALID_ARG, "null argument");
    if (which < 0 || which > 4 || iters < 1) return fail(c, PBD_ERR_INVALID_ARG, "which in [0,4], iters >= 1");
    const int max_rows = which == 4 ? c->ro_alloc : c->rows_alloc;
    if (rows < 1 || rows > max_rows) return fail(c, PBD_ERR_CAPACITY, "rows outside [1, %d]", max_rows);
    const int bn = pick_bn(rows), bi = bn_index(bn);
    const int nl = c->cfg.n_layers;
    const int per_sweep = which == 4 ? 1 : nl;
    auto launch = [&](int l) -> cudaError_t {
        switch (which) {
            case 0: return launch_linear_partials(&c->maps[AB_X][bi], bn, c->w_qkv[l], adapter, rows,
                                                  partials_for(c, c->w_qkv[l]), c->status, c->st);
            case 1: return launch_linear_partials(&c->maps[AB_ATTN][bi], bn, c->w_o[l], adapter, rows,
                                                  partials_for(c, c->w_o[l]), c->status, c->st);
            case 2: return launch_linear_partials(&c->maps[AB_X][bi], bn, c->w_gu[l], adapter, rows,
                                                  partials_for(c, c->w_gu[l]), c->status, c->st);
            case 3: return launch_linear_partials(&c->maps[AB_ACT][bi], bn, c->w_down[l], adapter, rows,
                                                  partials_for(c, c->w_down[l]), c->status, c->st);
            default: return launch_lm_head(&c->maps[AB_XRO][bi], bn, c->w_lm, rows, c->tile_max, c->tile_arg,
                                           nullptr, c->status, c->st);
        }
    };
    for (int l = 0; l < per_sweep; ++l) CK(launch(l));  // warm-up sweep
    cudaEvent_t e0, e1;
    CK(cudaEventCreate(&e0));
    CK(cudaEventCreate(&e1));
    CK(cudaEventRecord(e0, c->st));
    for (int it = 0; it < iters; ++it)
        for (int l = 0; l < per_sweep; ++l) CK(launch(l));
    CK(cudaEventRecord(e1, c->st));
    CK(cudaEventSynchronize(e1));
    float ms = 0.f;
    cudaEventElapsedTime(&ms, e0, e1);
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    *h_ms_per_launch = (double)ms / ((double)iters * per_sweep);
    if (h_weight_bytes) {
        const TiledWeight &w = which == 0 ? c->w_qkv[0] : which == 1 ? c->w_o[0] : which == 2 ? c->w_gu[0]
                               : which == 3 ? c->w_down[0] : c->w_lm;
        *h_weight_bytes = 2.0 * (double)w.K * (w.n_main + (adapter && which < 4 ? w.lora_rows : 0));
    }
    return check_device(c);
}

const char *pbd_last_error(const pbd_ctx *c) { return c ? c->err.c_str() : g_last_error.c_str(); }

const char *pbd_version(void) { return "pbd sm_103a " __DATE__; }

}  // extern "C"
