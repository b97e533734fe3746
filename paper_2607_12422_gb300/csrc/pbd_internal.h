// pbd_internal.h -- host-side interface between the orchestration (pbd.cu) and the kernel
// translation units.  Plain structs of device pointers and sizes; no torch types.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

#include "../../include/pbd.h"

namespace pbd {

constexpr int PAGE = 16;           // KV page length in tokens
constexpr int ATT_SPLIT = 128;     // key positions per attention split (position-aligned)
constexpr int ATT_SUBS_MAX = 2;    // partial results per split at most (its two 64-key halves)
constexpr int ATT_SPAN_MAX = 2;    // 128-key splits per attention item at most
constexpr int PREFILL_ROWS = 64;   // rows per prefill chunk
constexpr int KT = 64;             // K elements per 128-byte swizzle atom row (bf16)
constexpr int TILE_ROWS = 128;     // output features per tensor-core tile
constexpr int TILE_BYTES = TILE_ROWS * KT * 2;  // 16 KiB per pre-tiled weight tile

enum MaskMode : int { MASK_CAUSAL = 0, MASK_BLOCK_DRAFT = 1 };

struct Dims {
    int nl, H, Hq, Hkv, d, I, V, r;
    float eps, lora_scale;
};

// One forward pass over nb sequences x R rows; row m -> sequence b0 + m / R at position L[b] + m % R.
struct PassDesc {
    int b0, nb, R, M;
    int adapter;     // LoRA delta on
    int mask_mode;   // MaskMode
    int ro_first;    // read-out rows per sequence: i in [ro_first, ro_first + ro_count)
    int ro_count;
    int nl_run;      // decoder layers the pass runs before the final norm (the draft's early exit)
    uint64_t skip = 0;  // decoder layers below nl_run the pass skips (the draft's layer skipping)
    int att_span = 1;   // consecutive 128-key splits one attention item covers (a context constant)
};

// Paged KV cache: [layer][page][Hkv][PAGE][d] bf16 for K and for V.
struct KVCache {
    void *k, *v;
    const int *page_table;  // [max_batch][pages_per_seq]
    int pages_per_seq;
    int n_pages;
};

// A weight pre-tiled for the tensor-core kernel: row tiles x k tiles of 128 x 64 bf16 in the
// 128-byte swizzle layout, 16 KiB each.  The adapter's A rows (x A^T, stacked) occupy one
// extra row tile after the main rows.
struct TiledWeight {
    const void *tiles;
    int n_main;      // main output features (multiple of 128)
    int lora_rows;   // rows of the adapter tile (r x number of adapters)
    int K;           // input features (multiple of 64)
};

// Split-K partial sums, fp32 [k_splits][rows_alloc][n_total], n_total = n_main + lora_rows.
struct Partials {
    float *p;
    int k_splits;
    int rows_alloc;
    int n_total;
};

// ---- persistent pass kernel (pass_kernel.cu) ----

enum MKOp : uint8_t { MK_EMBED = 0, MK_LINEAR = 1, MK_ATTN = 2, MK_FINAL = 3 };

// Timestamps per item recorded by a traced pass (%globaltimer ns; 0 = not reached):
//   0 start, 1 inputs ready, 2 work done, 3 end (next item's start);
//   linear items: 4 operand staged, 5 accumulator ready, 6 partials stored, 7 reduced,
//     8 norm scales ready (RMSNorm inputs) or act words valid (down), 9 first reduced row's
//     partial sums present, 10 its outputs computed, 11 reduction's stores issued;
//   attention items: 4 K/V pages landed, 5 V converted, 6 counted (all splits stored), 7 merged,
//     8 block pages requested, 9 q fragments loaded, 10 softmax done, 11 partials stored,
//     12 merge inputs loaded.
constexpr int MK_STAMPS = 16;

// One work item of a pass.  MK_LINEAR: lin (0 q|k|v, 1 o, 2 gate|up, 3 down), a = row tile
// (the adapter tile is the last one), b = K slice.  MK_ATTN: a = sequence in the pass, b = KV
// head, c = item index (splits c * att_span .. c * att_span + att_span - 1 of 128 keys each).
// MK_EMBED: a = row.  MK_FINAL: a = read-out index, b = row.
// Dependencies, worked out on the host: the item waits until counter wait_off (an index into the
// pass's counters, -1: none) reaches wait_tgt, and once its result is stored it adds one to each
// counter rel[k] >= 0 (a reduction, an embedded row, an attention merge).
struct __align__(16) MKItem {
    uint8_t op, lin;
    uint16_t layer;
    int32_t a, b, c;
    int32_t wait_off, wait_tgt;
    int32_t rel[2];
};

// Offsets of the pass's completion counters (ints, zeroed before every pass).
struct CounterLayout {
    int embed;      // rows embedded
    int global;     // first per-layer counter (slots before it: embed, CTAs started)
    int per_layer;  // counters per layer
    int res_o, res_dn;  // residual tiles finished after o / down
    int att;        // per (sequence, KV head): split items done (+1 once merged)
    int att_in;     // per KV head: reduced q|k|v tile slices that its attention reads
    int att_o;      // per K slice of the o projection: attention merges of the heads it reads
    int total;
};

struct MKLaunch {
    const CUtensorMap *kmap, *vmap;  // paged K / V cache, box {64 dims, 16 tokens}
    Dims dm;
    PassDesc pd;
    int grid;
    const MKItem *items;
    const int *cta_off;
    const int *nsplit;
    int *cnt;
    CounterLayout cl;
    const void *wt[4];
    size_t wt_stride[4];
    int n_main[4], lora_rows[4], K[4];
    const void *lora_b[4];
    size_t lb_stride[4];
    const void *attn_norm, *mlp_norm, *q_norm, *k_norm, *final_norm, *mask_embed, *embed_tiled;
    const float2 *rope_cs;
    int rope_rows;
    KVCache kv;
    const int *Lbuf;
    const int *ids;
    unsigned long long *part[4];  // split-K partials, tagged with the pass counter
    int *epoch;                   // pass counter (device)
    int part_rows;
    void *h, *q, *attn, *act, *x_ro;
    float *ss;
    float *o_part;
    float2 *ml_part;
    int att_splits_alloc;
    int att_subs;  // partial results per split: 2 (64-key halves) or 1 (one warp covers the 128 keys)
    int *status, *abort;
    unsigned long long *trace = nullptr;  // optional per-item timestamps
};

int mk_grid_size();
void mk_counter_layout(const Dims &dm, int max_nb, CounterLayout *cl);
void mk_build_schedule(const Dims &dm, const PassDesc &pd, const std::vector<int> &nsplit, int grid,
                       const CounterLayout &cl, std::vector<MKItem> *out, std::vector<int> *off);
size_t mk_union_bytes(int bn, int head_dim, int att_span);
int mk_slice_atoms(int lin, int K);  // 64-wide K atoms per work item of linear `lin`
cudaError_t launch_pass_kernel(const MKLaunch &L, cudaStream_t st);

// ---- launchers (each returns cudaGetLastError()) ----

// Tensor-core linear: part[s][m][f] = sum over split s of x[m,k] * W[f,k], for f in the main
// rows (and the adapter rows when with_lora).  x is read through a TMA map with box {64, BN}.
cudaError_t launch_linear_partials(const CUtensorMap *x_map, int bn, const TiledWeight &w, int with_lora, int M,
                                   const Partials &out, int *status, cudaStream_t st);

// lm_head over the read-out rows: per 128-row vocabulary tile the (max, argmax) of each row,
// and optionally the fp32 logits [rows][V].
cudaError_t launch_lm_head(const CUtensorMap *x_map, int bn, const TiledWeight &w, int M, float *tile_max,
                           int *tile_arg, float *logits, int *status, cudaStream_t st);

cudaError_t launch_argmax_reduce(const float *tile_max, const int *tile_arg, int n_tiles, int rows, int *ids_out,
                                 cudaStream_t st);

// Builds the row token ids of a pass from the device state: draft [pending, -1 x D],
// verify [pending, drafts], decode [pending].
cudaError_t launch_build_ids(const PassDesc &pd, int kind, const int *pending, const int *drafts, int D, int *ids,
                             cudaStream_t st);

struct SeqState {
    int *L;          // [B] committed length
    int *pending;    // [B]
    int *n_out;      // [B]
    int *done;       // [B]
    int *all_done;   // [1]
    int *out_tokens; // [B][max_new_cap]
    int *round;      // [1] rounds executed (index into the forced-n sequence)
    long long *stats;// [3]: rounds, accepted, emitted
};

// Accept/commit for nb sequences: n from drafts vs verify ids (or forced), emit, advance.
cudaError_t launch_accept_commit(const SeqState &s, int nb, int D, const int *drafts, const int *verify,
                                 const int *forced, int forced_stride, int max_new, int out_cap,
                                 int *accepted_out, cudaStream_t st);

// Repack rows [0, rows) of a row-major bf16 matrix [rows, K] into the tiled layout at
// destination row offset dst_row0.
cudaError_t launch_repack_tiled(const void *src, int rows, int K, void *dst_tiles, int dst_row0, cudaStream_t st);
// Same, with source row i placed on tile row dst_row0 + (i / group) * stride + i % group
// (gate and up rows interleaved in 64-row blocks inside each 128-row tile).
cudaError_t launch_repack_tiled_map(const void *src, int rows, int K, void *dst_tiles, int dst_row0, int group,
                                    int stride, cudaStream_t st);

cudaError_t launch_read_kv(const Dims &dm, const KVCache &kv, int layer, int seq, int n, void *k_out, void *v_out,
                           cudaStream_t st);

// L[b] = value (prefill chunks run at L = chunk start).
cudaError_t launch_set_len(int *L, int b, int value, cudaStream_t st);

// After the prompt of sequence b: L = P, pending = first token = output token 0.
cudaError_t launch_prefill_finish(const SeqState &s, int b, int P, const int *first_id, int max_new, int out_cap,
                                  cudaStream_t st);

// y[m, f] = bf16(sum of splits + scale * sum_j bf16(u_j) B[f, j]) for f < N (standalone linear).
cudaError_t launch_linear_finalize(const Partials &P, int M, int N, int r, float scale, const void *lora_b, void *y,
                                   cudaStream_t st);

// 2-D bf16 row-major [rows, cols] tensor map, box {64, box_rows}, 128-byte swizzle.
bool encode_bf16_map(CUtensorMap *map, const void *base, int rows, int cols, int box_rows);

// Per-instantiation kernel attributes (dynamic shared memory), set once before any capture.
cudaError_t configure_linear_kernels();

// Records the message pbd_op_last_error() returns on this thread.
void op_record_error(const char *msg);

// Single-op status words: wait for the stream and read the latched DEV_* code; turn a nonzero
// code into PBD_ERR_DEVICE with its message (pbd_op_last_error()).
pbd_status read_device_code(const int *d_status, cudaStream_t st, int *code, const char *who);
pbd_status device_fail(int code, const char *who);

}  // namespace pbd
