// pbd.cu -- host orchestration and C ABI of the PEFT-BD hot path (see include/pbd.h).
//
// One context owns a caller-provided device workspace holding: the weights re-tiled for the
// tensor-core kernels, the adapter's B matrices, a paged bf16 KV cache, the device-resident
// decoding state (cached lengths, pending tokens, outputs, done flags), the work schedules of
// the persistent pass kernel, and the pass scratch (activations, split-K partial sums,
// attention partials, completion counters, lm_head tile maxima).
//
// A pass is: zero the pass counters, build the rows' token ids, one persistent pass kernel
// (all decoder layers), the lm_head over the read-out rows, the final argmax.  A speculative
// round (draft pass, verify pass, accept/commit) only reads and writes device memory, so it is
// captured once as a CUDA graph and replayed; the host looks at the done flags every few rounds.
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
enum PassKind { PK_DRAFT = 0, PK_VERIFY = 1, PK_DECODE = 2, PK_PREFILL = 3, N_PK = 4 };

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

struct Sched {
    MKItem *items = nullptr;  // device
    int *off = nullptr;       // device [grid + 1]
    int *nsplit = nullptr;    // device [max_batch]
    bool valid = false;
};

}  // namespace

struct pbd_ctx {
    pbd_config cfg;
    Dims dm;
    cudaStream_t st;
    int D, rows_alloc, ro_alloc, out_cap, rope_rows, n_splits, pages_per_seq, n_pages, grid;
    size_t items_cap;
    // weights
    std::vector<TiledWeight> w[4];  // q|k|v, o, gate|up (interleaved), down
    TiledWeight w_lm;
    void *lb[4];                    // adapter B, fused per layer [nl][out][r]
    void *attn_norm, *mlp_norm, *q_norm, *k_norm, *final_norm, *mask_embed;
    float2 *rope_cs;
    KVCache kv;
    int *page_table;
    // scratch
    void *h, *q, *attn, *act, *x_ro;
    unsigned long long *part[4];  // tagged split-K partials of the pass kernel
    size_t part_bytes[4];
    size_t act_bytes;
    float *ss, *o_part;
    float2 *ml_part;
    float *tile_max;
    int *tile_arg;
    unsigned long long *trace;  // per-item timestamps of pbd_trace_pass
    int *ids, *draft_ids, *verify_ids, *first_id, *status, *cnt;  // cnt[0] = abort flag
    CounterLayout cl;
    Sched sched[N_PK];
    SeqState s;
    CUtensorMap maps[N_BN];  // x_ro, per box height
    CUtensorMap kmap, vmap;  // paged K and V caches
    // host state
    int batch = 0, max_new = 0;
    std::vector<int> prompt_lens;
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

#define TRY(expr)                    \
    do {                             \
        pbd_status s_ = (expr);      \
        if (s_ != PBD_OK) return s_; \
    } while (0)

bool valid_config(const pbd_config *cfg, std::string *why) {
    auto bad = [&](const char *m) {
        *why = m;
        return false;
    };
    if (!cfg) return bad("null config");
    const pbd_config &k = *cfg;
    if (k.n_layers < 1 || k.hidden < 128 || k.n_q_heads < 1 || k.n_kv_heads < 1 || k.intermediate < 64 ||
        k.vocab < 128)
        return bad("non-positive model dimension");
    if (k.head_dim != 64 && k.head_dim != 128) return bad("head_dim must be 64 or 128");
    if (k.n_q_heads % k.n_kv_heads) return bad("n_q_heads must be a multiple of n_kv_heads");
    if (k.hidden % 256 || k.hidden > 4096) return bad("hidden must be a multiple of 256, at most 4096");
    if ((k.n_q_heads * k.head_dim) % 256 || ((k.n_q_heads + 2 * k.n_kv_heads) * k.head_dim) % 128)
        return bad("q/k/v widths must tile by 128 and the attention width by 256");
    if (k.intermediate % 256 || k.intermediate > 16384)
        return bad("intermediate must be a multiple of 256, at most 16384");
    if (k.n_q_heads * k.head_dim > 16384) return bad("n_q_heads * head_dim must be at most 16384");
    if (k.vocab % 128) return bad("vocab must be a multiple of 128");
    if (k.lora_rank != 8 && k.lora_rank != 16) return bad("lora_rank must be 8 or 16");
    if (k.page_size != PAGE) return bad("page_size must be 16");
    if (k.block_D < 1 || k.block_D > 64) return bad("block_D must be in [1, 64]");
    if (k.max_batch < 1 || k.max_batch > 64) return bad("max_batch must be in [1, 64]");
    if (k.max_batch * (k.block_D + 1) > 256) return bad("max_batch * (block_D + 1) must be <= 256");
    if (k.max_seq_len < 2 || k.max_seq_len > (1 << 20)) return bad("max_seq_len out of range");
    if (!(k.rms_eps > 0.f) || !(k.rope_theta > 0.f)) return bad("rms_eps and rope_theta must be positive");
    if (k.draft_layers < 0 || k.draft_layers > k.n_layers) return bad("draft_layers must be in [0, n_layers]");
    if (k.denoise_steps < 0 || k.denoise_steps > 8) return bad("denoise_steps must be in [0, 8]");
    if (k.draft_unanchored != 0 && k.draft_unanchored != 1) return bad("draft_unanchored must be 0 or 1");
    if (k.n_layers < 64 && (k.draft_skip_mask >> k.n_layers) != 0)
        return bad("draft_skip_mask has bits at or above n_layers");
    if (k.max_ctas < 0 || k.max_ctas > 256) return bad("max_ctas must be in [0, 256]");
    {
        const int E = k.draft_layers > 0 ? k.draft_layers : k.n_layers;
        int kept = 0;
        for (int l = 0; l < E; ++l) kept += (l < 64 && ((k.draft_skip_mask >> l) & 1u)) ? 0 : 1;
        if (kept == 0) return bad("the draft must keep at least one layer");
    }
    return true;
}

int lin_K(const pbd_config &k, int lin) {
    return lin == 1 ? k.n_q_heads * k.head_dim : (lin == 3 ? k.intermediate : k.hidden);
}
int lin_main(const pbd_config &k, int lin) {
    return lin == 0 ? (k.n_q_heads + 2 * k.n_kv_heads) * k.head_dim
                    : (lin == 2 ? 2 * k.intermediate : k.hidden);
}
int lin_lora(const pbd_config &k, int lin) {
    return k.lora_rank * (lin == 0 ? 3 : (lin == 2 ? 2 : 1));
}

// Carves the workspace; with base == nullptr it only measures.  Returns total bytes.
size_t layout(pbd_ctx *c, void *base) {
    const pbd_config &k = c->cfg;
    const int nl = k.n_layers, H = k.hidden, d = k.head_dim, Hq = k.n_q_heads, Hkv = k.n_kv_heads;
    const int I = k.intermediate, V = k.vocab, r = k.lora_rank, D = k.block_D;
    c->D = D;
    c->rows_alloc = ((std::max(k.max_batch * (D + 1), PREFILL_ROWS) + 31) / 32) * 32;
    c->ro_alloc = k.max_batch * (D + 1);
    c->out_cap = k.max_seq_len;
    // a truncated last round can leave L up to D past the budget, and every later pass still
    // touches D+1 slots above L: reserve twice the block width beyond max_seq_len
    const int max_tokens = k.max_seq_len + 2 * (D + 1);
    c->rope_rows = max_tokens;
    c->n_splits = (max_tokens + ATT_SPLIT - 1) / ATT_SPLIT;
    c->pages_per_seq = (max_tokens + PAGE - 1) / PAGE;
    c->n_pages = k.max_batch * c->pages_per_seq;
    if (c->grid <= 0) c->grid = 160;  // measuring only; pbd_create uses the device's SM count
    const int B = k.max_batch, RA = c->rows_alloc;
    mk_counter_layout(c->dm, B, &c->cl);
    size_t lin_items = 0;
    for (int lin = 0; lin < 4; ++lin) lin_items += (size_t)(lin_main(k, lin) / TILE_ROWS + 1) * (lin_K(k, lin) / 256);
    c->items_cap = (size_t)RA + (size_t)nl * (lin_items + (size_t)B * Hkv * c->n_splits) + (size_t)c->ro_alloc;

    Bump bp(base);
    c->status = (int *)bp.take(64);
    c->s.all_done = c->status + 1;
    c->s.round = c->status + 2;
    // abort flag, the pass counters, then the pass counter that tags split-K partials
    c->cnt = (int *)bp.take(sizeof(int) * (size_t)(c->cl.total + 2));
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
    for (int p = 0; p < N_PK; ++p) {
        c->sched[p].items = (MKItem *)bp.take(sizeof(MKItem) * c->items_cap);
        c->sched[p].off = (int *)bp.take(sizeof(int) * (size_t)(c->grid + 1));
        c->sched[p].nsplit = (int *)bp.take(sizeof(int) * B);
    }

    // weights
    for (int lin = 0; lin < 4; ++lin) {
        c->w[lin].assign(nl, TiledWeight());
        for (int l = 0; l < nl; ++l) {
            TiledWeight &w = c->w[lin][l];
            w.n_main = lin_main(k, lin);
            w.lora_rows = lin_lora(k, lin);
            w.K = lin_K(k, lin);
            w.tiles = bp.take((size_t)(w.n_main / TILE_ROWS + 1) * (w.K / KT) * TILE_BYTES);
        }
    }
    c->w_lm.n_main = V;
    c->w_lm.lora_rows = 0;
    c->w_lm.K = H;
    c->w_lm.tiles = bp.take((size_t)(V / TILE_ROWS) * (H / KT) * TILE_BYTES);
    const size_t e2 = 2;
    for (int lin = 0; lin < 4; ++lin) c->lb[lin] = bp.take(e2 * nl * (size_t)lin_main(k, lin) * r);
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

    // activations and pass scratch
    c->h = bp.take(e2 * RA * H);
    c->q = bp.take(e2 * RA * Hq * d);
    c->attn = bp.take(e2 * RA * Hq * d);
    c->act_bytes = sizeof(unsigned long long) * RA * (I / 2);  // tagged words of two bf16
    c->act = bp.take(c->act_bytes);
    c->x_ro = bp.take(e2 * c->ro_alloc * H);
    c->ss = (float *)bp.take(sizeof(float) * RA * (H / TILE_ROWS));
    for (int lin = 0; lin < 4; ++lin) {
        c->part_bytes[lin] = sizeof(unsigned long long) * (size_t)(lin_K(k, lin) / 256) * RA *
                             (lin_main(k, lin) + lin_lora(k, lin));
        c->part[lin] = (unsigned long long *)bp.take(c->part_bytes[lin]);
    }
    c->o_part = (float *)bp.take(sizeof(float) * (size_t)RA * Hq * c->n_splits * ATT_SUBS_MAX * d);
    c->ml_part = (float2 *)bp.take(sizeof(float2) * (size_t)RA * Hq * c->n_splits * ATT_SUBS_MAX);
    c->tile_max = (float *)bp.take(sizeof(float) * (size_t)(V / TILE_ROWS) * c->ro_alloc);
    c->tile_arg = (int *)bp.take(sizeof(int) * (size_t)(V / TILE_ROWS) * c->ro_alloc);
    c->trace = (unsigned long long *)bp.take(sizeof(unsigned long long) * MK_STAMPS * c->items_cap);
    return bp.off + ALIGN;
}

pbd_status make_maps(pbd_ctx *c) {
    for (int i = 0; i < N_BN; ++i)
        if (!encode_bf16_map(&c->maps[i], c->x_ro, c->ro_alloc, c->cfg.hidden, BN_CHOICES[i]))
            return fail(c, PBD_ERR_CUDA, "tensor map encode failed (box rows %d)", BN_CHOICES[i]);
    // K and V caches seen as rows of head_dim values: (layer, page, kv head, token) -> one row
    const int kv_rows = c->cfg.n_layers * c->n_pages * c->cfg.n_kv_heads * PAGE;
    if (!encode_bf16_map(&c->kmap, c->kv.k, kv_rows, c->cfg.head_dim, PAGE) ||
        !encode_bf16_map(&c->vmap, c->kv.v, kv_rows, c->cfg.head_dim, PAGE))
        return fail(c, PBD_ERR_CUDA, "KV tensor map encode failed");
    return PBD_OK;
}

pbd_status repack(pbd_ctx *c, const void *src, size_t layer_elems, int l, int rows, int K, const TiledWeight &w,
                  int row0, int group = 0, int stride = 0) {
    if (!src) return fail(c, PBD_ERR_INVALID_ARG, "null weight pointer");
    const void *p = static_cast<const uint8_t *>(src) + 2 * layer_elems * l;
    CK(launch_repack_tiled_map(p, rows, K, const_cast<void *>(w.tiles), row0, group ? group : rows, stride, c->st));
    return PBD_OK;
}

pbd_status copy_dev(pbd_ctx *c, void *dst, const void *src, size_t bytes) {
    if (!src) return fail(c, PBD_ERR_INVALID_ARG, "null weight pointer");
    CK(cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToDevice, c->st));
    return PBD_OK;
}

pbd_status load_weights(pbd_ctx *c, const pbd_base_weights *bw, const pbd_adapter_weights *aw) {
    const pbd_config &k = c->cfg;
    const int nl = k.n_layers, H = k.hidden, d = k.head_dim, Hq = k.n_q_heads, Hkv = k.n_kv_heads;
    const int I = k.intermediate, r = k.lora_rank;
    const int qw = Hq * d, kvw = Hkv * d, n_qkv = qw + 2 * kvw;
    for (int lin = 0; lin < 4; ++lin)
        for (int l = 0; l < nl; ++l) {
            const TiledWeight &w = c->w[lin][l];
            CK(cudaMemsetAsync(const_cast<void *>(w.tiles), 0,
                               (size_t)(w.n_main / TILE_ROWS + 1) * (w.K / KT) * TILE_BYTES, c->st));
        }
    const size_t e2 = 2;
    for (int l = 0; l < nl; ++l) {
        // q|k|v rows, then the adapter's A_q, A_k, A_v rows in the extra tile
        TRY(repack(c, bw->w[0], (size_t)qw * H, l, qw, H, c->w[0][l], 0));
        TRY(repack(c, bw->w[1], (size_t)kvw * H, l, kvw, H, c->w[0][l], qw));
        TRY(repack(c, bw->w[2], (size_t)kvw * H, l, kvw, H, c->w[0][l], qw + kvw));
        for (int t = 0; t < 3; ++t) TRY(repack(c, aw->lora_a[t], (size_t)r * H, l, r, H, c->w[0][l], n_qkv + t * r));
        TRY(repack(c, bw->w[3], (size_t)H * qw, l, H, qw, c->w[1][l], 0));
        TRY(repack(c, aw->lora_a[3], (size_t)r * qw, l, r, qw, c->w[1][l], H));
        // gate and up interleaved in 64-row blocks: tile t = [gate 64t..64t+63 | up 64t..64t+63]
        TRY(repack(c, bw->w[4], (size_t)I * H, l, I, H, c->w[2][l], 0, 64, 128));
        TRY(repack(c, bw->w[5], (size_t)I * H, l, I, H, c->w[2][l], 64, 64, 128));
        TRY(repack(c, aw->lora_a[4], (size_t)r * H, l, r, H, c->w[2][l], 2 * I));
        TRY(repack(c, aw->lora_a[5], (size_t)r * H, l, r, H, c->w[2][l], 2 * I + r));
        TRY(repack(c, bw->w[6], (size_t)H * I, l, H, I, c->w[3][l], 0));
        TRY(repack(c, aw->lora_a[6], (size_t)r * I, l, r, I, c->w[3][l], H));
        // adapter B matrices, fused per layer: q|k|v rows, o rows, gate rows then up rows, down rows
        uint8_t *lq = static_cast<uint8_t *>(c->lb[0]) + e2 * (size_t)l * n_qkv * r;
        const int outs[3] = {qw, kvw, kvw};
        size_t off = 0;
        for (int t = 0; t < 3; ++t) {
            if (!aw->lora_b[t]) return fail(c, PBD_ERR_INVALID_ARG, "null adapter B pointer");
            TRY(copy_dev(c, lq + off, static_cast<const uint8_t *>(aw->lora_b[t]) + e2 * (size_t)l * outs[t] * r,
                         e2 * (size_t)outs[t] * r));
            off += e2 * (size_t)outs[t] * r;
        }
        TRY(copy_dev(c, static_cast<uint8_t *>(c->lb[1]) + e2 * (size_t)l * H * r,
                     static_cast<const uint8_t *>(aw->lora_b[3]) + e2 * (size_t)l * H * r, e2 * (size_t)H * r));
        uint8_t *lg = static_cast<uint8_t *>(c->lb[2]) + e2 * (size_t)l * 2 * I * r;
        TRY(copy_dev(c, lg, static_cast<const uint8_t *>(aw->lora_b[4]) + e2 * (size_t)l * I * r, e2 * (size_t)I * r));
        TRY(copy_dev(c, lg + e2 * (size_t)I * r, static_cast<const uint8_t *>(aw->lora_b[5]) + e2 * (size_t)l * I * r,
                     e2 * (size_t)I * r));
        TRY(copy_dev(c, static_cast<uint8_t *>(c->lb[3]) + e2 * (size_t)l * H * r,
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

// decoder layers a pass of this kind runs: the draft may exit early, every other pass runs all
int draft_pass_layers(const pbd_ctx *c, int kind) {
    return (kind == PK_DRAFT && c->cfg.draft_layers > 0) ? c->cfg.draft_layers : c->cfg.n_layers;
}

// Partial results per attention split, a constant of the context (every pass of every generation
// uses the same key partition, so verify rows stay bitwise equal to decode rows): two 64-key halves
// on separate warps when a full-length pass's split items fit one wave of CTAs; otherwise one warp
// per query tile over all 128 keys, which halves the partials the merge reads.
int att_subs_of(const pbd_ctx *c) {
    return (long)c->cfg.max_batch * c->n_splits * c->cfg.n_kv_heads > c->grid ? 1 : ATT_SUBS_MAX;
}
// 128-key splits per attention item: with one partial per split, an item covers two splits (one
// query tile and split per warp, all six warps busy), halving the items of long contexts; the
// key partition, and with it every result, is the same
int att_span_of(const pbd_ctx *c) { return att_subs_of(c) == 1 ? ATT_SPAN_MAX : 1; }

PassDesc block_pass(pbd_ctx *c, int kind) {
    PassDesc pd;
    pd.b0 = 0;
    pd.nb = c->batch;
    pd.R = (kind == PK_DECODE) ? 1 : c->D + 1;
    pd.M = pd.nb * pd.R;
    pd.adapter = kind == PK_DRAFT ? 1 : 0;
    pd.mask_mode = kind == PK_DRAFT ? MASK_BLOCK_DRAFT : MASK_CAUSAL;
    // the draft reads D rows: rows 0..D-1 (row j-1 proposes position L+j) or, unanchored,
    // the mask rows 1..D (each proposes its own position)
    pd.ro_first = (kind == PK_DRAFT && c->cfg.draft_unanchored) ? 1 : 0;
    pd.ro_count = kind == PK_DRAFT ? c->D : pd.R;
    pd.nl_run = draft_pass_layers(c, kind);
    pd.skip = kind == PK_DRAFT ? c->cfg.draft_skip_mask : 0;
    pd.att_span = att_span_of(c);
    return pd;
}

// Builds a pass schedule on the host and uploads it (synchronously) into slot `kind`.
pbd_status upload_schedule(pbd_ctx *c, int kind, const PassDesc &pd, const std::vector<int> &nsplit) {
    std::vector<MKItem> items;
    std::vector<int> off;
    mk_build_schedule(c->dm, pd, nsplit, c->grid, c->cl, &items, &off);
    if (items.size() > c->items_cap)
        return fail(c, PBD_ERR_CAPACITY, "pass schedule of %zu items exceeds %zu", items.size(), c->items_cap);
    Sched &s = c->sched[kind];
    // ordered on the context's stream (which may not synchronise with the legacy stream), and
    // finished before the host vectors go away
    CK(cudaMemcpyAsync(s.items, items.data(), items.size() * sizeof(MKItem), cudaMemcpyHostToDevice, c->st));
    CK(cudaMemcpyAsync(s.off, off.data(), off.size() * sizeof(int), cudaMemcpyHostToDevice, c->st));
    CK(cudaMemcpyAsync(s.nsplit, nsplit.data(), nsplit.size() * sizeof(int), cudaMemcpyHostToDevice, c->st));
    CK(cudaStreamSynchronize(c->st));
    s.valid = true;
    return PBD_OK;
}

MKLaunch make_launch(pbd_ctx *c, const PassDesc &pd, int kind) {
    MKLaunch L;
    const pbd_config &k = c->cfg;
    L.kmap = &c->kmap;
    L.vmap = &c->vmap;
    L.dm = c->dm;
    L.pd = pd;
    L.grid = c->grid;
    L.items = c->sched[kind].items;
    L.cta_off = c->sched[kind].off;
    L.nsplit = c->sched[kind].nsplit;
    L.cnt = c->cnt + 1;
    L.cl = c->cl;
    for (int lin = 0; lin < 4; ++lin) {
        const TiledWeight &w0 = c->w[lin][0];
        L.wt[lin] = w0.tiles;
        L.wt_stride[lin] = k.n_layers > 1 ? (size_t)(static_cast<const uint8_t *>(c->w[lin][1].tiles) -
                                                     static_cast<const uint8_t *>(w0.tiles))
                                          : 0;
        L.n_main[lin] = w0.n_main;
        L.lora_rows[lin] = w0.lora_rows;
        L.K[lin] = w0.K;
        L.lora_b[lin] = c->lb[lin];
        L.lb_stride[lin] = (size_t)w0.n_main * k.lora_rank;
        L.part[lin] = c->part[lin];
    }
    L.epoch = c->cnt + c->cl.total + 1;
    L.attn_norm = c->attn_norm;
    L.mlp_norm = c->mlp_norm;
    L.q_norm = c->q_norm;
    L.k_norm = c->k_norm;
    L.final_norm = c->final_norm;
    L.mask_embed = c->mask_embed;
    L.embed_tiled = c->w_lm.tiles;
    L.rope_cs = c->rope_cs;
    L.rope_rows = c->rope_rows;
    L.kv = c->kv;
    L.Lbuf = c->s.L;
    L.ids = c->ids;
    L.part_rows = c->rows_alloc;
    L.h = c->h;
    L.q = c->q;
    L.attn = c->attn;
    L.act = c->act;
    L.x_ro = c->x_ro;
    L.ss = c->ss;
    L.o_part = c->o_part;
    L.ml_part = c->ml_part;
    L.att_subs = att_subs_of(c);
    L.att_splits_alloc = c->n_splits * L.att_subs;  // partial results per (row, head)
    L.status = c->status;
    L.abort = c->cnt;
    return L;
}

// Zero the pass counters and launch the persistent kernel for all decoder layers.
pbd_status enqueue_pass_kernel(pbd_ctx *c, const PassDesc &pd, int kind) {
    CK(cudaMemsetAsync(c->cnt, 0, sizeof(int) * (size_t)(c->cl.total + 1), c->st));
    CK(launch_pass_kernel(make_launch(c, pd, kind), c->st));
    return PBD_OK;
}

// lm_head + argmax over the read-out rows written by the pass kernel
pbd_status enqueue_readout(pbd_ctx *c, const PassDesc &pd, int *ids_out, float *logits) {
    const int n_ro = pd.nb * pd.ro_count;
    if (n_ro <= 0) return PBD_OK;
    const int bro = pick_bn(n_ro);
    CK(launch_lm_head(&c->maps[bn_index(bro)], bro, c->w_lm, n_ro, c->tile_max, c->tile_arg, logits, c->status,
                      c->st));
    CK(launch_argmax_reduce(c->tile_max, c->tile_arg, c->cfg.vocab / TILE_ROWS, n_ro, ids_out, c->st));
    return PBD_OK;
}

pbd_status run_pass(pbd_ctx *c, const PassDesc &pd, int kind, int *ids_out, float *logits) {
    if (!c->sched[kind].valid) return fail(c, PBD_ERR_STATE, "no schedule for pass kind %d", kind);
    TRY(enqueue_pass_kernel(c, pd, kind));
    return enqueue_readout(c, pd, ids_out, logits);
}

pbd_status enqueue_draft(pbd_ctx *c, float *logits) {
    const PassDesc pd = block_pass(c, PK_DRAFT);
    const int steps = std::max(1, c->cfg.denoise_steps);
    for (int s = 0; s < steps; ++s) {
        // step 1 runs [p, MASK x D]; each further step refills row j (position L+j) with the
        // previous step's proposal d_j and replaces the proposals with its own
        CK(launch_build_ids(pd, s == 0 ? 0 : 1, c->s.pending, c->draft_ids, c->D, c->ids, c->st));
        TRY(run_pass(c, pd, PK_DRAFT, c->draft_ids, s + 1 == steps ? logits : nullptr));
    }
    return PBD_OK;
}

pbd_status enqueue_verify(pbd_ctx *c, const int *drafts, float *logits) {
    const PassDesc pd = block_pass(c, PK_VERIFY);
    CK(launch_build_ids(pd, 1, c->s.pending, drafts, c->D, c->ids, c->st));
    return run_pass(c, pd, PK_VERIFY, c->verify_ids, logits);
}

pbd_status enqueue_accept(pbd_ctx *c, const int *forced, int *accepted) {
    CK(launch_accept_commit(c->s, c->batch, c->D, c->draft_ids, c->verify_ids, forced, c->batch, c->max_new,
                            c->out_cap, accepted, c->st));
    return PBD_OK;
}

pbd_status enqueue_decode_pass(pbd_ctx *c, float *logits) {
    const PassDesc pd = block_pass(c, PK_DECODE);
    CK(launch_build_ids(pd, 2, c->s.pending, nullptr, 0, c->ids, c->st));
    return run_pass(c, pd, PK_DECODE, c->verify_ids, logits);
}

pbd_status enqueue_decode_commit(pbd_ctx *c) {
    CK(launch_accept_commit(c->s, c->batch, 0, c->draft_ids, c->verify_ids, nullptr, c->batch, c->max_new, c->out_cap,
                            nullptr, c->st));
    return PBD_OK;
}

pbd_status check_device(pbd_ctx *c) {
    CK(cudaStreamSynchronize(c->st));
    int code = 0;
    CK(cudaMemcpy(&code, c->status, sizeof(int), cudaMemcpyDeviceToHost));
    if (code != 0) {
        CK(cudaMemsetAsync(c->status, 0, sizeof(int), c->st));  // reported once; the context stays usable
        CK(cudaStreamSynchronize(c->st));
        return fail(c, PBD_ERR_DEVICE, "device status %d latched by a kernel", code);
    }
    return PBD_OK;
}

// attention split items per sequence over the whole generation (positions up to P + max_new + 2(D+1))
std::vector<int> decode_splits(pbd_ctx *c) {
    std::vector<int> ns(c->batch);
    for (int b = 0; b < c->batch; ++b) {
        const int tmax = std::min(c->prompt_lens[b] + c->max_new + 2 * (c->D + 1), c->pages_per_seq * PAGE);
        ns[b] = std::min(c->n_splits, (tmax + ATT_SPLIT - 1) / ATT_SPLIT);
    }
    return ns;
}

double pass_bytes(pbd_ctx *c, int kind, const std::vector<int> &Ls) {
    const pbd_config &k = c->cfg;
    double w = 0, lora = 0;
    for (int lin = 0; lin < 4; ++lin) {
        w += 2.0 * lin_main(k, lin) * lin_K(k, lin);
        lora += 2.0 * k.lora_rank * (lin_K(k, lin) + lin_main(k, lin));
    }
    int nl = 0;  // decoder layers the pass runs
    for (int l = 0; l < draft_pass_layers(c, kind); ++l)
        nl += (kind == PK_DRAFT && l < 64 && ((k.draft_skip_mask >> l) & 1u)) ? 0 : 1;
    double bytes = nl * (w + (kind == PK_DRAFT ? lora : 0.0));
    bytes += 2.0 * (2.0 * nl * k.hidden + 2.0 * nl * k.head_dim);  // norm gains
    const double kv_tok = 2.0 * 2.0 * nl * k.n_kv_heads * k.head_dim;
    const int rows = kind == PK_DECODE ? 1 : c->D + 1;
    for (int L : Ls) bytes += kv_tok * (L + rows);
    return bytes;
}

}  // namespace

extern "C" {

size_t pbd_workspace_bytes(const pbd_config *cfg) {
    std::string why;
    if (!valid_config(cfg, &why)) return 0;
    pbd_ctx tmp{};
    tmp.cfg = *cfg;
    tmp.dm = Dims{cfg->n_layers, cfg->hidden,      cfg->n_q_heads, cfg->n_kv_heads, cfg->head_dim,
                  cfg->intermediate, cfg->vocab, cfg->lora_rank, cfg->rms_eps,     cfg->lora_scale};
    tmp.grid = 256;  // upper bound of SMs per device for the per-CTA schedule offsets
    return layout(&tmp, nullptr);
}

pbd_status pbd_plan_pass(const pbd_config *cfg, int32_t kind, int32_t batch, const int32_t *h_prompt_lens,
                         int32_t max_new, int32_t grid, int32_t *h_items, int32_t *h_cta_off, int32_t cap, int32_t *h_n) {
    std::string why;
    if (!valid_config(cfg, &why)) return fail(nullptr, PBD_ERR_INVALID_ARG, "%s", why.c_str());
    if (kind < 0 || kind > 2 || batch < 1 || batch > cfg->max_batch || !h_prompt_lens || max_new < 1 || grid < 1 ||
        !h_items || !h_cta_off || !h_n)
        return fail(nullptr, PBD_ERR_INVALID_ARG, "pbd_plan_pass: bad argument");
    for (int b = 0; b < batch; ++b)
        if (h_prompt_lens[b] < 1 || h_prompt_lens[b] + max_new > cfg->max_seq_len)
            return fail(nullptr, PBD_ERR_CAPACITY, "prompt %d of %d tokens + %d exceeds max_seq_len", b,
                        h_prompt_lens[b], max_new);
    pbd_ctx tmp{};  // value-initialised, as pbd_create does
    tmp.cfg = *cfg;
    tmp.dm = Dims{cfg->n_layers, cfg->hidden,      cfg->n_q_heads, cfg->n_kv_heads, cfg->head_dim,
                  cfg->intermediate, cfg->vocab, cfg->lora_rank, cfg->rms_eps,     cfg->lora_scale};
    tmp.grid = grid;
    layout(&tmp, nullptr);
    tmp.batch = batch;
    tmp.max_new = max_new;
    tmp.prompt_lens.assign(h_prompt_lens, h_prompt_lens + batch);
    std::vector<MKItem> items;
    std::vector<int> off;
    mk_build_schedule(tmp.dm, block_pass(&tmp, kind), decode_splits(&tmp), grid, tmp.cl, &items, &off);
    *h_n = (int32_t)items.size();
    if ((int)items.size() > cap) return fail(nullptr, PBD_ERR_CAPACITY, "%zu items exceed cap %d", items.size(), cap);
    for (size_t i = 0; i < items.size(); ++i) {
        int32_t *o = h_items + 8 * i;
        o[0] = items[i].op | (items[i].lin << 8) | (items[i].layer << 16);
        o[1] = items[i].a;
        o[2] = items[i].b;
        o[3] = items[i].c;
        o[4] = items[i].wait_off;
        o[5] = items[i].wait_tgt;
        o[6] = items[i].rel[0];
        o[7] = items[i].rel[1];
    }
    for (int k = 0; k <= grid; ++k) h_cta_off[k] = off[k];
    return PBD_OK;
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
    c->dm = Dims{cfg->n_layers, cfg->hidden,      cfg->n_q_heads, cfg->n_kv_heads, cfg->head_dim,
                 cfg->intermediate, cfg->vocab, cfg->lora_rank, cfg->rms_eps,     cfg->lora_scale};
    c->grid = 256;
    const size_t need = layout(c, nullptr);
    if (workspace_bytes < need) {
        delete c;
        return fail(nullptr, PBD_ERR_WORKSPACE, "workspace too small: %zu < %zu bytes", workspace_bytes, need);
    }
    c->grid = mk_grid_size();
    if (c->grid <= 0 || c->grid > 256) {
        delete c;
        return fail(nullptr, PBD_ERR_CUDA, "cannot query the SM count");
    }
    if (cfg->max_ctas > 0) c->grid = std::min(c->grid, cfg->max_ctas);
    {
        // the K slices of one tile reduce each other's partial sums: one CTA each
        int need = 1;
        for (int lin = 0; lin < 4; ++lin)
            need = std::max(need, lin_K(*cfg, lin) / (mk_slice_atoms(lin, lin_K(*cfg, lin)) * KT));
        if (c->grid < need) {
            const int g = c->grid;
            delete c;
            return fail(nullptr, PBD_ERR_INVALID_ARG, "max_ctas %d below the %d K slices of one linear", g, need);
        }
    }
    uint8_t *wb = static_cast<uint8_t *>(d_workspace);
    uint8_t *b1024 = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(wb) + ALIGN - 1) & ~(uintptr_t)(ALIGN - 1));
    layout(c, b1024);
    c->st = static_cast<cudaStream_t>(d_stream);
    pbd_status s;
    cudaError_t e;
    if ((e = configure_linear_kernels()) != cudaSuccess) {
        s = fail(c, PBD_ERR_CUDA, "kernel configuration: %s", cudaGetErrorString(e));
        delete c;
        return s;
    }
    if ((s = load_weights(c, base, adapter)) != PBD_OK || (s = build_rope(c)) != PBD_OK || (s = make_maps(c)) != PBD_OK) {
        delete c;
        return s;
    }
    const size_t kv_bytes = (size_t)cfg->n_layers * c->n_pages * cfg->n_kv_heads * PAGE * cfg->head_dim * 2;
    // the split-K partials start with tag 0, below every pass's tag (the pass counter starts at 0)
    for (int lin = 0; lin < 4 && e == cudaSuccess; ++lin) e = cudaMemsetAsync(c->part[lin], 0, c->part_bytes[lin], c->st);
    if (e == cudaSuccess) e = cudaMemsetAsync(c->act, 0, c->act_bytes, c->st);
    if (e != cudaSuccess || (e = cudaMemsetAsync(c->cnt, 0, sizeof(int) * (size_t)(c->cl.total + 2), c->st)) != cudaSuccess ||
        (e = cudaMemsetAsync(c->kv.k, 0, kv_bytes, c->st)) != cudaSuccess ||
        (e = cudaMemsetAsync(c->kv.v, 0, kv_bytes, c->st)) != cudaSuccess ||
        (e = cudaMemsetAsync(c->status, 0, 64, c->st)) != cudaSuccess ||
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
    if (batch < 1 || batch > c->cfg.max_batch)
        return fail(c, PBD_ERR_CAPACITY, "batch %d outside [1, %d]", batch, c->cfg.max_batch);
    if (!d_prompt_ids || !h_prompt_lens) return fail(c, PBD_ERR_INVALID_ARG, "null prompt");
    if (max_new < 1) return fail(c, PBD_ERR_INVALID_ARG, "max_new must be >= 1");
    for (int b = 0; b < batch; ++b)
        if (h_prompt_lens[b] < 1 || h_prompt_lens[b] + max_new > c->cfg.max_seq_len)
            return fail(c, PBD_ERR_CAPACITY, "sequence %d: prompt %d + max_new %d exceeds max_seq_len %d", b,
                        h_prompt_lens[b], max_new, c->cfg.max_seq_len);
    c->drop_bench_graphs(0);
    c->drop_bench_graphs(1);
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
    CK(cudaStreamSynchronize(c->st));
    c->batch = batch;
    c->max_new = max_new;
    c->prompt_lens.assign(h_prompt_lens, h_prompt_lens + batch);
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
            pd.att_span = att_span_of(c);
            pd.M = rows;
            pd.adapter = 0;
            pd.mask_mode = MASK_CAUSAL;
            pd.ro_first = last ? rows - 1 : 0;
            pd.ro_count = last ? 1 : 0;
            pd.nl_run = c->cfg.n_layers;
            const std::vector<int> ns(1, (c0 + rows + ATT_SPLIT - 1) / ATT_SPLIT);
            CK(cudaStreamSynchronize(c->st));  // the schedule slot is rewritten per chunk
            TRY(upload_schedule(c, PK_PREFILL, pd, ns));
            CK(launch_set_len(c->s.L, b, c0, c->st));
            CK(cudaMemcpyAsync(c->ids, d_prompt_ids + off + c0, sizeof(int) * rows, cudaMemcpyDeviceToDevice, c->st));
            TRY(run_pass(c, pd, PK_PREFILL, c->first_id, nullptr));
        }
        CK(launch_prefill_finish(c->s, b, P, c->first_id, max_new, c->out_cap, c->st));
        off += P;
    }
    if (d_first_token)
        CK(cudaMemcpyAsync(d_first_token, c->s.pending, sizeof(int) * batch, cudaMemcpyDeviceToDevice, c->st));
    TRY(check_device(c));
    // schedules of the decode passes of this generation
    const std::vector<int> ns = decode_splits(c);
    TRY(upload_schedule(c, PK_DRAFT, block_pass(c, PK_DRAFT), ns));
    TRY(upload_schedule(c, PK_VERIFY, block_pass(c, PK_VERIFY), ns));
    TRY(upload_schedule(c, PK_DECODE, block_pass(c, PK_DECODE), ns));
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
    if (d_forced_n_opt) CK(cudaMemsetAsync(c->s.round, 0, sizeof(int), c->st));
    TRY(enqueue_accept(c, d_forced_n_opt, d_accepted_n));
    c->phase = PH_READY;
    return PBD_OK;
}

pbd_status pbd_decode_step(pbd_ctx *c, int32_t *d_next_opt, float *d_logits_opt) {
    if (!c) return fail(c, PBD_ERR_INVALID_ARG, "null context");
    if (c->phase != PH_READY) return fail(c, PBD_ERR_STATE, "decode step needs a prefilled or committed state");
    TRY(enqueue_decode_pass(c, d_logits_opt));
    TRY(enqueue_decode_commit(c));
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
    cudaGraph_t g = nullptr;
    cudaGraphExec_t ge = nullptr;
    const bool use_graph = c->st != nullptr && c->st != cudaStreamLegacy;
    auto enqueue_round = [&]() -> pbd_status {
        if (mode == 0) {
            TRY(enqueue_draft(c, nullptr));
            TRY(enqueue_verify(c, c->draft_ids, nullptr));
            return enqueue_accept(c, d_forced_n_seq_opt, nullptr);
        }
        TRY(enqueue_decode_pass(c, nullptr));
        return enqueue_decode_commit(c);
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
            result = check_device(c);
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
            if (ph == 1) s = enqueue_decode_pass(c, nullptr);
            if (ph == 2) s = enqueue_decode_commit(c);
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
    std::vector<cudaEvent_t> ev((size_t)steps * 4, nullptr);
    for (auto &x : ev)
        if (s == PBD_OK && cudaEventCreate(&x) != cudaSuccess) s = fail(c, PBD_ERR_CUDA, "event create");
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

pbd_status pbd_time_pass(pbd_ctx *c, int32_t kind, int32_t iters, double *h_ms_per_launch, double *h_bytes_per_launch) {
    if (!c || !h_ms_per_launch) return fail(c, PBD_ERR_INVALID_ARG, "null argument");
    if (kind < 0 || kind > 2 || iters < 1) return fail(c, PBD_ERR_INVALID_ARG, "kind in [0,2], iters >= 1");
    if (c->phase != PH_READY) return fail(c, PBD_ERR_STATE, "timing needs a prefilled or committed state");
    const PassDesc pd = block_pass(c, kind);
    CK(launch_build_ids(pd, kind == PK_DRAFT ? 0 : (kind == PK_VERIFY ? 1 : 2), c->s.pending, c->draft_ids, c->D,
                        c->ids, c->st));
    TRY(enqueue_pass_kernel(c, pd, kind));  // warm-up launch
    std::vector<cudaEvent_t> ev((size_t)iters * 2, nullptr);
    pbd_status s = PBD_OK;
    for (auto &x : ev)
        if (s == PBD_OK && cudaEventCreate(&x) != cudaSuccess) s = fail(c, PBD_ERR_CUDA, "event create");
    for (int i = 0; s == PBD_OK && i < iters; ++i) {
        cudaError_t e = cudaMemsetAsync(c->cnt, 0, sizeof(int) * (size_t)(c->cl.total + 1), c->st);
        if (e == cudaSuccess) e = cudaEventRecord(ev[2 * i], c->st);
        if (e == cudaSuccess) e = launch_pass_kernel(make_launch(c, pd, kind), c->st);
        if (e == cudaSuccess) e = cudaEventRecord(ev[2 * i + 1], c->st);
        if (e != cudaSuccess) s = fail(c, PBD_ERR_CUDA, "timed launch: %s", cudaGetErrorString(e));
    }
    if (s == PBD_OK && cudaStreamSynchronize(c->st) != cudaSuccess) s = fail(c, PBD_ERR_CUDA, "timing sync");
    double tot = 0;
    if (s == PBD_OK)
        for (int i = 0; i < iters; ++i) {
            float ms = 0.f;
            cudaEventElapsedTime(&ms, ev[2 * i], ev[2 * i + 1]);
            tot += ms;
        }
    for (auto &x : ev)
        if (x) cudaEventDestroy(x);
    TRY(s);
    *h_ms_per_launch = tot / iters;
    if (h_bytes_per_launch) {
        std::vector<int> Ls(c->batch);
        CK(cudaMemcpy(Ls.data(), c->s.L, sizeof(int) * c->batch, cudaMemcpyDeviceToHost));
        *h_bytes_per_launch = pass_bytes(c, kind, Ls);
    }
    return check_device(c);
}

pbd_status pbd_check_stalled_pass(pbd_ctx *c, int32_t *h_device_code) {
    if (!c || !h_device_code) return fail(c, PBD_ERR_INVALID_ARG, "null argument");
    if (c->phase != PH_READY) return fail(c, PBD_ERR_STATE, "the check needs a prefilled or committed state");
    const PassDesc pd = block_pass(c, PK_VERIFY);
    const std::vector<int> ns = decode_splits(c);
    std::vector<MKItem> all, items;
    std::vector<int> off;
    mk_build_schedule(c->dm, pd, ns, 1, c->cl, &all, &off);  // one CTA: the items in order
    bool dropped = false;
    for (const MKItem &it : all) {
        if (!dropped && it.op == MK_LINEAR && it.lin == 0 && it.layer == 0) {
            dropped = true;
            continue;
        }
        items.push_back(it);
    }
    // deal the remaining items round-robin, as mk_build_schedule does
    std::vector<int> cta_off(c->grid + 1, 0);
    for (size_t i = 0; i < items.size(); ++i) cta_off[i % c->grid + 1]++;
    for (int k = 0; k < c->grid; ++k) cta_off[k + 1] += cta_off[k];
    std::vector<MKItem> dealt(items.size());
    std::vector<int> fill(cta_off.begin(), cta_off.end() - 1);
    for (size_t i = 0; i < items.size(); ++i) dealt[fill[i % c->grid]++] = items[i];
    Sched &sv = c->sched[PK_VERIFY];
    CK(cudaMemcpyAsync(sv.items, dealt.data(), dealt.size() * sizeof(MKItem), cudaMemcpyHostToDevice, c->st));
    CK(cudaMemcpyAsync(sv.off, cta_off.data(), cta_off.size() * sizeof(int), cudaMemcpyHostToDevice, c->st));
    CK(cudaStreamSynchronize(c->st));
    CK(launch_build_ids(pd, 1, c->s.pending, c->draft_ids, c->D, c->ids, c->st));
    TRY(enqueue_pass_kernel(c, pd, PK_VERIFY));
    CK(cudaStreamSynchronize(c->st));
    int code = 0;
    CK(cudaMemcpy(&code, c->status, sizeof(int), cudaMemcpyDeviceToHost));
    *h_device_code = code;
    // the normal verify schedule again; the device code is reported (and cleared) below
    TRY(upload_schedule(c, PK_VERIFY, pd, ns));
    return check_device(c);
}

pbd_status pbd_trace_pass(pbd_ctx *c, int32_t kind, int32_t *h_items, uint64_t *h_trace, int32_t cap, int32_t *h_n) {
    if (!c || !h_items || !h_trace || !h_n) return fail(c, PBD_ERR_INVALID_ARG, "null argument");
    if (kind < 0 || kind > 2) return fail(c, PBD_ERR_INVALID_ARG, "kind in [0,2]");
    if (c->phase != PH_READY) return fail(c, PBD_ERR_STATE, "tracing needs a prefilled or committed state");
    const PassDesc pd = block_pass(c, kind);
    std::vector<MKItem> items;
    std::vector<int> off;
    mk_build_schedule(c->dm, pd, decode_splits(c), c->grid, c->cl, &items, &off);
    if ((int)items.size() > cap) return fail(c, PBD_ERR_CAPACITY, "%zu items exceed cap %d", items.size(), cap);
    CK(launch_build_ids(pd, kind == PK_DRAFT ? 0 : (kind == PK_VERIFY ? 1 : 2), c->s.pending, c->draft_ids, c->D,
                        c->ids, c->st));
    CK(cudaMemsetAsync(c->trace, 0, sizeof(unsigned long long) * MK_STAMPS * items.size(), c->st));
    CK(cudaMemsetAsync(c->cnt, 0, sizeof(int) * (size_t)(c->cl.total + 1), c->st));
    MKLaunch L = make_launch(c, pd, kind);
    L.trace = c->trace;
    CK(launch_pass_kernel(L, c->st));
    CK(cudaMemcpyAsync(h_trace, c->trace, sizeof(unsigned long long) * MK_STAMPS * items.size(), cudaMemcpyDeviceToHost,
                       c->st));
    CK(cudaStreamSynchronize(c->st));
    for (size_t i = 0; i < items.size(); ++i) {
        h_items[4 * i] = items[i].op | (items[i].lin << 8) | (items[i].layer << 16);
        h_items[4 * i + 1] = items[i].a;
        h_items[4 * i + 2] = items[i].b;
        h_items[4 * i + 3] = items[i].c;
    }
    *h_n = (int32_t)items.size();
    return check_device(c);
}

const char *pbd_last_error(const pbd_ctx *c) { return c ? c->err.c_str() : g_last_error.c_str(); }

const char *pbd_version(void) { return "pbd sm_103a " __DATE__; }

}  // extern "C"
