// pbd_internal.h -- host-side interface between the orchestration (pbd.cu) and the kernel
// translation units.  Plain structs of device pointers and sizes; no torch types.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace pbd {

constexpr int PAGE = 16;           // KV page length in tokens
constexpr int ATT_SPLIT = 128;     // key positions per attention split (position-aligned)
constexpr int PREFILL_ROWS = 256;  // rows per prefill chunk
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

cudaError_t launch_embed_norm(const Dims &dm, const PassDesc &pd, const int *ids, const void *embed_tiled,
                              const void *mask_embed, const void *gain, void *h, void *x, int *status,
                              cudaStream_t st);

cudaError_t launch_qkv_finalize(const Dims &dm, const PassDesc &pd, int layer, const Partials &part,
                                const void *lora_b_qkv, const void *q_norm, const void *k_norm,
                                const float2 *rope_cs, int rope_rows, const int *L, const KVCache &kv, void *q_out,
                                int *status, cudaStream_t st);

cudaError_t launch_attention(const Dims &dm, const PassDesc &pd, int layer, const void *q, const KVCache &kv,
                             const int *L, int n_splits, float *o_part, float2 *ml_part, cudaStream_t st);

cudaError_t launch_attn_combine(const Dims &dm, const PassDesc &pd, const int *L, int n_splits, const float *o_part,
                                const float2 *ml_part, void *attn_out, cudaStream_t st);

// h <- bf16(h + bf16(sum partials + s * u B^T)); x <- RMSNorm(h) * gain; read-out rows also to x_ro.
cudaError_t launch_residual_norm(const Dims &dm, const PassDesc &pd, const Partials &part, int n_out,
                                 const void *lora_b, const void *gain, void *h, void *x, void *x_ro,
                                 cudaStream_t st);

// act <- bf16(silu(gate) * up) from the fused gate|up partials (+ adapter delta)
cudaError_t launch_act(const Dims &dm, const PassDesc &pd, const Partials &part, const void *lora_b_gu, void *act,
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
cudaError_t configure_attention_kernels();

}  // namespace pbd
