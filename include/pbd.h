/*
 * pbd.h -- C ABI of the PEFT-BD speculative-decoding hot path on one GB300 (sm_103a).
 *
 * PEFT-BD ("Accepted Prefixes Are Not All You Need", arXiv 2607.12422, Section 3) decodes
 * with one backbone in two modes.  Each speculative round is
 *   1. a draft pass with the LoRA-like adapter ON: the pending token plus D masked
 *      positions are run through the whole decoder in one denoising step (Section 3,
 *      steps 1-2; Appendix A.4: draft width D+1 = 17);
 *   2. a verify pass with the adapter OFF over [pending, d_1..d_D] under the causal mask
 *      (Section 3, step 3; Appendix A.4: "a different attention mask");
 *   3. greedy top-1 matching, acceptance of the longest matching prefix d_1..d_n, and the
 *      verifier's next token v_n appended as well (Section 3, steps 4-5; Appendix A.1);
 *   4. commit of the accepted KV, roll-back of the rest (Appendix A.4: the draft's KV is
 *      scratch and is not interchangeable with the verifier's).
 * The model is a Qwen3-shaped decoder in bf16 (Section 4.1) with the adapter on all
 * seven block linears (Appendix A.2).
 *
 * Conventions for every entry point:
 *   - Pointers prefixed d_ are device memory, h_ host memory.  The library never allocates
 *     device memory: the caller provides one workspace of pbd_workspace_bytes() bytes.
 *   - Calls are asynchronous on the stream given to pbd_create, except where stated.
 *   - Every call returns a pbd_status; no exception crosses the ABI.  pbd_last_error()
 *     returns the message of the last failure on that context.
 *   - Errors detected inside kernels (a bounded wait that ran out, an index out of range)
 *     latch a device status word; the next synchronising call (pbd_get_state, pbd_generate,
 *     pbd_sync) returns PBD_ERR_DEVICE.
 *   - Calls in the wrong order (verify before draft, commit before verify) return
 *     PBD_ERR_STATE and do nothing.
 *   - A context is used from one host thread at a time.
 */
#ifndef PBD_H
#define PBD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    PBD_OK = 0,
    PBD_ERR_INVALID_ARG = 1, /* null pointer, unsupported shape, out-of-range value */
    PBD_ERR_WORKSPACE = 2,   /* workspace missing, misaligned or too small */
    PBD_ERR_CAPACITY = 3,    /* batch, prompt or generation length beyond the configured maximum */
    PBD_ERR_STATE = 4,       /* call out of order */
    PBD_ERR_CUDA = 5,        /* a CUDA runtime call or launch failed */
    PBD_ERR_DEVICE = 6       /* a kernel latched an error (bounded wait expired, bad index) */
} pbd_status;

/* Model and run limits (Qwen3 shape of Section 4.1; adapter of Appendix A.2). */
typedef struct {
    int32_t n_layers, hidden, n_q_heads, n_kv_heads, head_dim, intermediate, vocab;
    float rms_eps;      /* 1e-6 */
    float rope_theta;   /* 1e6 */
    int32_t lora_rank;  /* r */
    float lora_scale;   /* alpha / r */
    int32_t block_D;    /* masked positions per draft block (16 in the paper) */
    int32_t max_batch;  /* sequences decoded together */
    int32_t max_seq_len;/* prompt + generated tokens per sequence (the D+1 scratch slots are added internally) */
    int32_t page_size;  /* KV page length in tokens; must be 16 */
    /* Draft variants; all zero = the method of Section 3 (one adapter-on pass over every layer,
     * row j-1 proposing position L+j).  Fixed for the context's lifetime. */
    int32_t draft_layers;     /* early exit (Section 6): the draft runs only the first draft_layers
                                 decoder layers before the final norm and the head; 0 = all */
    int32_t denoise_steps;    /* adapter-on block passes per draft (the two-step ablation of Sections
                                 4.4 and 5.3): each pass after the first refills the mask rows with the
                                 previous pass's proposals; 0 or 1 = one pass, at most 8 */
    int32_t draft_unanchored; /* 1: mask row j proposes its own position L+j (rows 1..D are read, the
                                 pending token's row is context only; the unanchored ablation of
                                 Sections 4.4 and 5.3); 0: row j-1 proposes position L+j */
    uint64_t draft_skip_mask; /* layer skipping (Section 6): bit l set = the draft skips decoder
                                 layer l (its residual stream passes the layer unchanged and it
                                 writes no K/V there); 0 = none.  Bits at or above n_layers must be
                                 clear, and the draft must keep at least one layer (together with
                                 draft_layers) */
    int32_t max_ctas;         /* CTAs of the persistent pass kernel: 0 = one per SM; otherwise at most
                                 max_ctas (leaving SMs to other work).  It must be at least the largest
                                 number of K slices of one linear, whose reductions wait for one
                                 another and so must sit on distinct CTAs: pbd_create fails with
                                 PBD_ERR_INVALID_ARG below that */
} pbd_config;

/* Backbone weights: bf16, row-major [out, in] per linear, stacked over layers.  They are
 * copied (re-tiled) into the workspace by pbd_create and not read afterwards. */
typedef struct {
    const void *embed;       /* [V, H]      tied with the lm_head */
    const void *final_norm;  /* [H] */
    const void *attn_norm;   /* [nl, H] */
    const void *mlp_norm;    /* [nl, H] */
    const void *q_norm;      /* [nl, d]     per-head RMSNorm gain of q */
    const void *k_norm;      /* [nl, d]     per-head RMSNorm gain of k */
    const void *w[7];        /* q [nl,Hq*d,H], k [nl,Hkv*d,H], v [nl,Hkv*d,H], o [nl,H,Hq*d],
                                gate [nl,I,H], up [nl,I,H], down [nl,H,I] */
} pbd_base_weights;

/* Adapter: for each of the seven linears (same order) A [nl, r, in] and B [nl, out, r], bf16;
 * plus the embedding of the mask token [H] used by the draft's masked rows. */
typedef struct {
    const void *lora_a[7];
    const void *lora_b[7];
    const void *mask_embed;
} pbd_adapter_weights;

typedef struct {
    int64_t rounds;          /* speculative rounds (or AR steps) summed over sequences */
    int64_t accepted;        /* sum of accepted draft lengths n over rounds */
    int64_t emitted;         /* tokens written to the output, prefill token included */
    double  draft_ms;        /* host-timed totals of the graph launches, 0 when not timed */
    double  verify_ms;
} pbd_stats;

typedef struct pbd_ctx pbd_ctx;

/* Bytes of device workspace pbd_create needs for this configuration (0 if the config is invalid). */
size_t pbd_workspace_bytes(const pbd_config *cfg);

/* Validates cfg, carves the workspace (256-byte aligned, >= pbd_workspace_bytes), copies the
 * weights into the kernels' tiled layouts, builds RoPE tables and TMA descriptors.
 * d_stream: a cudaStream_t (NULL = legacy default stream).  Synchronises the stream on return. */
pbd_status pbd_create(const pbd_config *cfg, const pbd_base_weights *base, const pbd_adapter_weights *adapter,
                      void *d_workspace, size_t workspace_bytes, void *d_stream, pbd_ctx **out);
pbd_status pbd_destroy(pbd_ctx *ctx);

/* Starts a generation of `batch` sequences (Appendix A.1: prompts up to the configured length,
 * greedy continuation, budget max_new tokens per sequence, no other stop rule).
 * d_prompt_ids: the prompts' token ids packed back to back; h_prompt_lens[b] their lengths.
 * Runs the causal adapter-off prefill, sets each sequence's cached length L_b = P_b and its
 * pending token to the verifier's argmax after the prompt; that token is output token 0,
 * also written to d_first_token[b] when non-null.  Synchronous on return. */
pbd_status pbd_prefill(pbd_ctx *ctx, int32_t batch, const int32_t *d_prompt_ids, const int32_t *h_prompt_lens,
                       int32_t max_new, int32_t *d_first_token);

/* Draft pass (Section 3, steps 1-2): adapter ON, rows [pending, MASK x D] at positions
 * L_b..L_b+D, pending row causal, mask rows bidirectional among themselves.  Writes the D
 * proposals of each sequence to d_draft [batch, D] (optional) and keeps them internally.
 * d_logits_opt [batch, D, V] fp32 receives the readout rows' logits when non-null. */
pbd_status pbd_draft_block(pbd_ctx *ctx, int32_t *d_draft, float *d_logits_opt);

/* Verify pass (Section 3, step 3): adapter OFF, causal, rows [pending, d_1..d_D].
 * d_draft: proposals to verify [batch, D]; NULL verifies the last draft.  Writes the
 * verifier's greedy tokens v_0..v_D to d_verify [batch, D+1] (optional), the rows' KV into
 * cache slots L_b..L_b+D, and logits to d_logits_opt [batch, D+1, V] when non-null. */
pbd_status pbd_verify_block(pbd_ctx *ctx, const int32_t *d_draft, int32_t *d_verify, float *d_logits_opt);

/* Acceptance and commit (Section 3, steps 4-5), on the device: n_b = longest prefix with
 * d_i == v_{i-1}; appends d_1..d_n and v_n (cut at the budget), L_b += n_b + 1, pending = v_n.
 * d_forced_n_opt [batch]: replaces n_b (timing mode with seeded acceptance).
 * d_accepted_n [batch] (optional) receives n_b (-1 for a sequence already done). */
pbd_status pbd_accept_commit(pbd_ctx *ctx, const int32_t *d_forced_n_opt, int32_t *d_accepted_n);

/* Plain greedy step by the verifier (the baseline the method must reproduce): one causal
 * adapter-off row per sequence, then emit its argmax and advance L_b by one. */
pbd_status pbd_decode_step(pbd_ctx *ctx, int32_t *d_next_opt, float *d_logits_opt);

/* Whole generation: prefill, then speculative rounds (mode 0) or AR steps (mode 1) until every
 * sequence has max_new tokens.  Rounds run as one captured CUDA graph each; the host polls the
 * done flags every few rounds.  d_forced_n_seq_opt [max_rounds, batch] forces the accepted
 * lengths of successive rounds (mode 0 only; max_rounds = max_new).  d_out_tokens [batch, max_new].
 * Synchronous on return. */
pbd_status pbd_generate(pbd_ctx *ctx, int32_t batch, const int32_t *d_prompt_ids, const int32_t *h_prompt_lens,
                        int32_t max_new, int32_t mode, const int32_t *d_forced_n_seq_opt, int32_t *d_out_tokens,
                        pbd_stats *h_stats_opt);

/* Synchronous reads of the decoding state (for tests and reports).
 * h_L [batch]: committed lengths; h_pending [batch]; h_n_out [batch]: tokens emitted. */
pbd_status pbd_get_state(pbd_ctx *ctx, int32_t *h_L, int32_t *h_pending, int32_t *h_n_out);

/* Copies the emitted tokens [batch, max_new] of the current generation to d_out_tokens. */
pbd_status pbd_get_tokens(pbd_ctx *ctx, int32_t *d_out_tokens);

/* Gathers committed K and V of `layer` for sequence `seq`, slots [0, n), from the paged cache into
 * contiguous bf16 [n, Hkv*d] buffers (tests of the commit/roll-back rule). */
pbd_status pbd_read_kv(pbd_ctx *ctx, int32_t layer, int32_t seq, int32_t n, void *d_k_out, void *d_v_out);

/* Waits for the stream and reports a latched device error. */
pbd_status pbd_sync(pbd_ctx *ctx);

/* Timing of the decode loop (the profile of Appendix A.5 measures draft and verify forward
 * latency separately).  On a prefilled context, replays `warmup` untimed and then `steps` timed
 * rounds, each as CUDA graphs on the context's stream: mode 0 = draft pass, verify pass,
 * accept/commit; mode 1 = one plain greedy step (verify-style pass of one row, commit).
 * CUDA events bracket each phase of every timed round.  h_ms[0..3] receive the summed ms of
 * the draft passes, the verify (or AR) passes, the commits, and the whole timed region;
 * h_launches receives the kernels launched per round.  d_forced_n_seq_opt as in pbd_generate
 * (indexed by round from the start of the call).  Synchronous on return. */
pbd_status pbd_bench_rounds(pbd_ctx *ctx, int32_t mode, int32_t warmup, int32_t steps,
                            const int32_t *d_forced_n_seq_opt, double *h_ms, int32_t *h_launches);

/* Times the persistent pass kernel alone (all decoder layers of one pass; the lm_head and the
 * small kernels around it excluded).  On a prefilled context, launches the draft (kind 0),
 * verify (1) or plain-decoding (2) pass kernel `iters` times with CUDA events bracketing each
 * launch; the decoding state is not advanced, so every launch does the same work, and the
 * weights it streams (about 0.9 GB for the 0.6B shape) exceed L2.  *h_ms_per_launch receives the
 * mean duration; *h_bytes_per_launch the algorithmic bytes of one launch: every layer weight once
 * (adapter factors too for the draft), the cached K/V read and the block's K/V written. */
pbd_status pbd_time_pass(pbd_ctx *ctx, int32_t kind, int32_t iters, double *h_ms_per_launch,
                         double *h_bytes_per_launch);

/* Timeline of one pass of the persistent kernel (a profiling aid; the paper's Appendix A.5 profiles
 * draft and verify forward latency).  On a prefilled context, runs one draft (kind 0), verify (1)
 * or plain-decoding (2) pass without advancing the state, recording for every work item sixteen
 * %globaltimer stamps in ns: start, inputs complete, main work done, end, then per item kind
 * (linear: operand staged, accumulator ready, partials stored, reduction done, norm scales or
 * act words ready, first reduced row's partial sums present, its outputs computed, reduction's
 * stores issued; attention: K/V landed, V converted, all splits stored, merge done, block pages
 * requested, q fragments loaded, softmax done, partials stored, merge inputs loaded; 0 when not
 * reached).  h_items receives per item {op | lin << 8 | layer << 16, a, b, c}, h_trace the
 * stamps [n, 16], both in the schedule's order; at most `cap` items; *h_n the item count. */
pbd_status pbd_trace_pass(pbd_ctx *ctx, int32_t kind, int32_t *h_items, uint64_t *h_trace, int32_t cap,
                          int32_t *h_n);

/* Failure-detection check (no GPU fault is involved).  On a prefilled context, runs one verify
 * pass whose schedule lacks the first q|k|v item of layer 0: that item's partial sums never
 * arrive, so the waits polling for them run out after their bound (1 s), latch a device code
 * and end the pass.  Returns PBD_ERR_DEVICE with the latched code in *h_device_code (a
 * DEV_TIMEOUT_* value; 0 would mean the pass ended without noticing).  The cached tokens and
 * the decoding state are untouched (the pass writes scratch slots only) and the context stays
 * usable: the normal schedules are restored before returning.  Synchronous. */
pbd_status pbd_check_stalled_pass(pbd_ctx *ctx, int32_t *h_device_code);

/* The work schedule of one pass, computed on the host with no context and no GPU (for checks
 * of the schedule's properties).  For a generation of `batch` prompts of h_prompt_lens tokens
 * and a budget of max_new tokens under cfg (whose draft variant applies to kind 0), returns the
 * items of a draft (kind 0), verify (1) or plain-decoding (2) pass dealt round-robin over `grid`
 * CTAs: h_items[8 i..8 i+7] = {op | lin << 8 | layer << 16, a, b, c, wait counter, wait target,
 * release counter 0, release counter 1} (op 0 embedding row, 1 linear slice, 2 attention split,
 * 3 final norm; see pbd_trace_pass; the item waits until the pass counter `wait counter` (-1:
 * none) reaches `wait target`, and adds one to each release counter >= 0 once its result is
 * stored), grouped by CTA with CTA
 * k's items at [h_cta_off[k], h_cta_off[k + 1]) (h_cta_off has grid + 1 entries; CTA k takes
 * the topologically ordered list's items k, k + grid, ...).  *h_n is the item count; at most
 * `cap` items are written (PBD_ERR_CAPACITY beyond).  Errors: PBD_ERR_INVALID_ARG (bad config or
 * argument), PBD_ERR_CAPACITY (prompt plus budget beyond max_seq_len, or cap too small). */
pbd_status pbd_plan_pass(const pbd_config *cfg, int32_t kind, int32_t batch, const int32_t *h_prompt_lens,
                         int32_t max_new, int32_t grid, int32_t *h_items, int32_t *h_cta_off, int32_t cap,
                         int32_t *h_n);

const char *pbd_last_error(const pbd_ctx *ctx);

/* Build/version tag of the library ("pbd sm_103a <date>"). */
const char *pbd_version(void);

#ifdef __cplusplus
}
#endif
#endif /* PBD_H */
