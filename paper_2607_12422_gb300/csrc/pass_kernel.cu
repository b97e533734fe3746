// pass_kernel.cu -- one persistent, cooperative kernel per decoder pass (draft, verify, plain
// decoding, prefill chunk) of the PEFT-BD hot path.
//
// Why: at batch 1 and D = 16 a pass moves 1.2 GB of weights (~180 us at full HBM bandwidth)
// through ~500 small dependent steps.  As separate kernel launches, launch gaps and latency
// chains dominated.  Here one CTA per SM walks a static, topologically ordered list of work
// items, and items wait only for the items they read (completion counters or tagged words in
// global memory, with bounded spins), so phases overlap and no kernel boundary separates them.
//
// Roles inside a CTA (256 threads):
//   warp 0      weight producer: walks the CTA's linear items ahead of the others and streams
//               their 128 x 64 weight tiles (16 KiB, pre-tiled in the 128-byte swizzle layout)
//               into a ring of shared-memory slots with 1-D bulk TMA (L2 evict-first).  Weights
//               depend on nothing, so the ring fills across phase boundaries.
//   warp 1      MMA issuer: per linear item, 4 x 4 tcgen05.mma (128 x BN x 16, bf16 -> fp32) into
//               a TMEM accumulator; frees ring slots with tcgen05.commit.
//   warps 2-7   compute group: dependency waits, operand staging (RMSNorm applied in place in
//               the activation tile's swizzle layout), the TMEM epilogue (warps 4-7, one per TMEM
//               lane quarter), attention, split reductions.
//
// A linear is split along K into 256-wide slices (512 for gate|up; fixed per linear, independent
// of the row count).  Each slice item stores its fp32 partial sums as 64-bit words tagged with
// the (pass, layer); the tile's slice items sit on distinct CTAs, and each of them then reduces
// every ks-th row of the tile, adding the slices in slice order as their tagged words arrive
// (no completion counter between the slices), and finishes the step for those rows:
//   q|k|v tile   -> + adapter delta, bf16, per-head RMSNorm, RoPE, q buffer / paged K, V
//   o tile       -> + adapter delta, residual add into h, per-tile sum of squares of h
//   gate|up tile -> + adapter delta, SiLU(gate) * up into the act buffer (gate/up interleaved)
//   down tile    -> + adapter delta, residual add into h, per-tile sum of squares of h
// The adapter's A rows form one extra tile whose partials u = x A^T the reducers above sum
// themselves.  Each reduction then counts once, with release semantics, on the counter its
// consumers poll (attention inputs per KV head, the residual), except gate|up: SiLU(gate) * up
// goes out as tagged words that the down projection's operand staging polls.
// Attention items cover (sequence, KV head, att_span consecutive 128-key splits: one, or two in
// long contexts); when a group's items sit on distinct CTAs they wait for one another and each
// merges a share of the rows, else the last one merges all.  RMSNorm statistics are summed per
// 128-feature tile in one fixed order, so every row's arithmetic is independent of the pass it
// is in.
#include <algorithm>
#include <cmath>
#include <vector>

#include "common.cuh"
#include "pbd_internal.h"

namespace pbd {

constexpr int MK_THREADS = 256;
constexpr int CT = 192;            // compute-group threads (warps 2-7)
constexpr int HALF_ATOMS = 4;      // 64-wide swizzle atoms of one operand staging round (K 256)
constexpr int MAX_ATOMS = 8;       // atoms per linear item at most (K slice 512)
constexpr int MAX_SLOT = 12;
constexpr int MK_STARTED = 1;      // global counter slot: CTAs that have read the pass counter
constexpr int CT_PAGES = 32;       // first compute thread of the warp (warp 3) that requests attention pages
constexpr int RING_SLOTS = 4;      // weight tiles in the ring (64 KiB)
constexpr int MAX_ROWS = 256;

// ------------------------------------------------------------------ device helpers

__device__ __forceinline__ void bar_compute() { asm volatile("bar.sync 1, 192;" ::: "memory"); }

__device__ __forceinline__ int ld_acquire(const int *p) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ int ld_relaxed(const int *p) {
    int v;
    asm volatile("ld.relaxed.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// single-copy-atomic 64-bit accesses of the tagged partials
__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p));
    return v;
}
__device__ __forceinline__ void st_relaxed_u64(unsigned long long *p, unsigned long long v) {
    asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(v));
}
__device__ __forceinline__ bool tag_is(unsigned long long w, uint32_t tag) { return (uint32_t)(w >> 32) == tag; }
// one tagged word (value in the low half, tag in the high half), single-copy atomic
__device__ __forceinline__ void st_tagged(unsigned long long *p, uint32_t v, uint32_t tag) {
    asm volatile("{\n\t.reg .b64 w;\n\tmov.b64 w, {%1, %2};\n\tst.relaxed.gpu.global.b64 [%0], w;\n\t}" ::"l"(p),
                 "r"(v), "r"(tag));
}
// 16-byte load, single-copy atomic per 64-bit element
__device__ __forceinline__ void ld_relaxed_2u64(const unsigned long long *p, unsigned long long &a,
                                                unsigned long long &b) {
    asm volatile("ld.relaxed.gpu.global.v2.b64 {%0, %1}, [%2];" : "=l"(a), "=l"(b) : "l"(p));
}

__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

struct MKParams {
    CUtensorMap kmap, vmap;  // paged K / V cache as [rows of 128 dims] x d, box {64, 16}, 128-byte swizzle
    Dims dm;
    PassDesc pd;
    const MKItem *items;
    const int *cta_off;
    int *cnt;            // counters of this pass (zeroed before launch)
    CounterLayout cl;
    const int *nsplit;   // [nb] 128-key attention splits per sequence (items: ceil(nsplit / att_span))
    // weights
    const uint8_t *wt[4];      // tiled weights of layer 0; layer stride wt_stride[lin] bytes
    size_t wt_stride[4];
    int n_main[4], lora_rows[4], K[4], ks[4];
    int katoms[4];             // 64-wide K atoms per item (the K slice is 64 * katoms wide)
    int b_dbl;                 // the operand area holds a whole MAX_ATOMS item at once
    const bf16 *lora_b[4];     // fused adapter B of layer 0, [n_out][r]
    size_t lb_stride[4];       // elements per layer
    const bf16 *attn_norm, *mlp_norm, *q_norm, *k_norm, *final_norm, *mask_embed, *embed_tiled;
    const float2 *rope_cs;
    int rope_rows;
    KVCache kv;
    const int *L;
    const int *ids;
    // scratch
    unsigned long long *part[4];  // split-K partials: fp32 bits | (pass, layer) tag << 32 (see sum_parts)
    int *epoch;                   // tag counter: layer l of a pass tags its partials *epoch + 1 + l
    int part_rows;
    bf16 *h, *q, *attn, *x_ro;
    unsigned long long *act;   // SiLU(gate) * up: words of two bf16 (features 2j, 2j+1) | tag << 32
    float *ss;                 // [rows][H/128]
    float *o_part;
    float2 *ml_part;
    int att_splits_alloc;
    int att_subs;              // partial results per split (1 or 2)
    float att_scale;           // 1/sqrt(head_dim)
    int *status, *abort;
    unsigned long long *trace;  // optional: MK_STAMPS timestamps per item (see pbd_internal.h)
    // launch geometry
    int bn, nslot, ring_bytes, union_bytes;
    uint32_t tmem_cols;
};

__device__ __forceinline__ bool aborted(const MKParams &P) { return ld_relaxed(P.abort) != 0; }

// sub-step timestamp of a traced pass (st = the item's stamp row, null when not tracing)
__device__ __forceinline__ void stamp_at(unsigned long long *st, int k) {
    if (st) st[k] = globaltimer_ns();
}

// Code size matters here: the compute warps walk every kind of item each layer, and code the
// SM's instruction caches cannot hold streams from L2 at several cycles per instruction.  Wait
// loops, error paths and rarely taken branches are therefore kept out of line and not unrolled.
__device__ __noinline__ void raise_abort(const MKParams &P, int code) {
    latch_error(P.status, code);
    atomicExch(P.abort, 1);
}

// one thread: wait until *c >= target (bounded)
__device__ __noinline__ bool spin_until(const int *c, int target, const MKParams &P) {
    if (ld_acquire(c) >= target) return true;
    const uint64_t t0 = globaltimer_ns();
    for (;;) {
#pragma unroll 1
        for (int i = 0; i < 8; ++i) {
            if (ld_acquire(c) >= target) return true;
            __nanosleep(40);
        }
        if (aborted(P)) return false;
        if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) {
            raise_abort(P, DEV_TIMEOUT_DEP);
            return false;
        }
    }
}

// bounded mbarrier wait that does not give up on abort: the pass is ending and its asynchronous
// copies and MMAs must land before the CTA releases its shared memory and TMEM
__device__ __noinline__ void drain_wait(uint64_t *bar, uint32_t parity) {
    const uint32_t a = smem_u32(bar);
    const uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(a, parity) && globaltimer_ns() - t0 < WAIT_LIMIT_NS) {
    }
}

// bounded mbarrier wait that also gives up when the pass is aborted (slow path out of line)
__device__ __noinline__ bool mbar_wait_slow(uint32_t a, uint32_t parity, const MKParams &P, int code) {
    const uint64_t t0 = globaltimer_ns();
    for (;;) {
#pragma unroll 1
        for (int i = 0; i < 16; ++i)
            if (mbar_try_wait(a, parity)) return true;
        if (aborted(P)) return false;
        if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) {
            raise_abort(P, code);
            return false;
        }
    }
}
__device__ __forceinline__ bool mbar_wait_mk(uint64_t *bar, uint32_t parity, const MKParams &P, int code) {
    const uint32_t a = smem_u32(bar);
    return mbar_try_wait(a, parity) || mbar_wait_slow(a, parity, P, code);
}

__device__ __forceinline__ int *ctr(const MKParams &P, int layer, int off) {
    return P.cnt + P.cl.global + layer * P.cl.per_layer + off;
}

// Sum of squares of one 128-feature tile of a row, in one fixed order: lane l adds elements
// l, l+32, l+64, l+96 in that order, then a butterfly; lane 0's value is the result.
__device__ __forceinline__ float tile_sumsq(const float (&v)[4]) {
    float s = __fmul_rn(v[0], v[0]);
#pragma unroll
    for (int e = 1; e < 4; ++e) s = __fadd_rn(s, __fmul_rn(v[e], v[e]));
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) s = __fadd_rn(s, __shfl_xor_sync(0xffffffffu, s, off));
    return __shfl_sync(0xffffffffu, s, 0);
}

// With one CTA per SM only six compute warps hide memory latency, so every helper below issues
// all of its independent loads before it consumes any; sums still run in one fixed order.
// Data written by other CTAs during the pass is read with L2-only loads (never a stale L1 line).
constexpr int MAX_RANK = 16;   // adapter rank (8 or 16)

__device__ __forceinline__ float ldcg_bf(const bf16 *p) {
    return __ushort_as_bfloat16(__ldcg(reinterpret_cast<const unsigned short *>(p)));
}

// 1/sqrt(mean(h^2) + eps) of row m from its per-tile sums (tiles added in order)
__device__ __forceinline__ float row_rms(const MKParams &P, int m) {
    const int nt = P.dm.H / TILE_ROWS;  // even (H is a multiple of 256)
    const float2 *s = reinterpret_cast<const float2 *>(P.ss + (size_t)m * nt);
    float a = 0.f;
    for (int t0 = 0; t0 < nt; t0 += 8) {
        float2 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) v[u] = t0 + 2 * u < nt ? __ldcg(s + t0 / 2 + u) : make_float2(0.f, 0.f);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            if (t0 + 2 * u >= nt) break;
            a = (t0 + u == 0) ? v[u].x : __fadd_rn(a, v[u].x);
            a = __fadd_rn(a, v[u].y);
        }
    }
    return __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(__fdiv_rn(a, (float)P.dm.H), P.dm.eps)));
}

// one B row (r bf16 values) of the adapter, for lora_dot_w
struct BRow {
    uint4 w[MAX_RANK / 8];
};
// The tile's B rows in shared memory: row j's r / 8 chunks of 16 bytes start at chunk
// j * (r / 8) + j / 4, i.e. 16 bytes of padding after every 4 rows.  Lane l reads rows 4l + e (or
// 2l + e), so without the padding the 8 lanes of a 128-byte load phase would hit the same four
// banks (8-way conflicts, with all six warps contending for the SM's shared-memory pipe: ~1700
// cycles for the four rows' dot products, ~750 padded).
__device__ __forceinline__ int brow_chunk(int j, int r) { return j * (r / 8) + (j >> 2); }
// the B row of local tile row j, from the tile's B rows staged in shared memory
__device__ __forceinline__ BRow smem_brow(const uint4 *brows, int j, int r) {
    BRow b;
#pragma unroll
    for (int q = 0; q < MAX_RANK / 8; ++q) b.w[q] = q * 8 < r ? brows[brow_chunk(j, r) + q] : make_uint4(0, 0, 0, 0);
    return b;
}
__device__ __forceinline__ float lora_dot_w(const float (&u)[MAX_RANK], const BRow &b, int r) {
    float a = 0.f;
#pragma unroll
    for (int q = 0; q < MAX_RANK / 8; ++q) {
        if (q * 8 < r) {
            const bf16 *e = reinterpret_cast<const bf16 *>(&b.w[q]);
#pragma unroll
            for (int j = 0; j < 8; ++j) a = __fadd_rn(a, __fmul_rn(u[q * 8 + j], bf2f(e[j])));
        }
    }
    return a;
}

// the adapter intermediates u[0..r) of one row, from lane j's slice-ordered sum (lane j < r holds u_j
// before rounding), shared by the warp
__device__ __forceinline__ void share_u(float lane_sum, int base, float (&u)[MAX_RANK]) {
    const float a = rbf(lane_sum);
#pragma unroll
    for (int j = 0; j < MAX_RANK; ++j) u[j] = __shfl_sync(0xffffffffu, a, base + j);
}

// Feature offsets (from a lane's first feature f0) of the four partial sums a lane reduces: two
// pairs of adjacent features, the second pair at f0 + OFF2 (2 for four consecutive features,
// 64 for gate|up: a gate pair and the up pair of the same act features).
// Sums of the K-slice partials of row m: out[0..3] for features f0, f0 + 1, f0 + OFF2, f0 + OFF2 + 1
// and, when X, out[4] for feature fx; slices added in order, loads in batches of S slices (every
// load of a batch in flight before the first add).  Each partial is one 64-bit word, the fp32
// value and the tag of the (pass, layer) that stored it, written and read with single-copy-atomic
// accesses: a word carrying this layer's tag holds this layer's value, so the sum polls the words
// themselves instead of a completion counter.  A batch with a word still carrying an older tag is
// read again (bounded; on timeout or abort the pass is lost).  One copy of the load code serves
// the first read and the re-reads, which keeps the function small.
template <int OFF2, bool X, int S>
__device__ __forceinline__ void sum_parts(const MKParams &P, int lin, int m, int f0, int fx, float *out, uint32_t tag) {
    constexpr int EX = 4 + (X ? 1 : 0);
    const int nt = P.n_main[lin] + P.lora_rows[lin];
    const unsigned long long *p = P.part[lin] + (size_t)m * nt;
    const size_t stride = (size_t)P.part_rows * nt;
    const int ks = P.ks[lin];
    const unsigned long long none = (unsigned long long)tag << 32;
#pragma unroll 1
    for (int s0 = 0; s0 < ks; s0 += S) {
        unsigned long long v[EX][S];
        uint64_t t0 = 0;
#pragma unroll 1
        for (int round = 0;; ++round) {
#pragma unroll
            for (int s = 0; s < S; ++s) {
                const unsigned long long *ps = p + (size_t)(s0 + s) * stride;
                if (s0 + s < ks) {
                    ld_relaxed_2u64(ps + f0, v[0][s], v[1][s]);
                    ld_relaxed_2u64(ps + f0 + OFF2, v[2][s], v[3][s]);
                    if (X) v[EX - 1][s] = ld_relaxed_u64(ps + fx);
                } else {
#pragma unroll
                    for (int e = 0; e < EX; ++e) v[e][s] = none;
                }
            }
            bool stale = false;
#pragma unroll
            for (int s = 0; s < S; ++s)
#pragma unroll
                for (int e = 0; e < EX; ++e) stale |= (uint32_t)(v[e][s] >> 32) != tag;
            if (!stale) break;
            // the abort flag and the time limit every 8 rounds (each check is an L2 round trip)
            if (round == 0) t0 = globaltimer_ns();
            __nanosleep(32);
            if ((round & 7) == 7 && (aborted(P) || globaltimer_ns() - t0 > WAIT_LIMIT_NS)) {
                if (!aborted(P)) raise_abort(P, DEV_TIMEOUT_DEP);
                break;
            }
        }
#pragma unroll
        for (int e = 0; e < EX; ++e) {
#pragma unroll
            for (int s = 0; s < S; ++s) {
                if (s0 + s >= ks) break;
                const float x = __uint_as_float((uint32_t)v[e][s]);
                out[e] = (s0 + s == 0) ? x : __fadd_rn(out[e], x);
            }
        }
    }
}

// element (v, k) of a matrix in the 128 x 64 swizzled tile layout
__device__ __forceinline__ const bf16 *tiled_at(const bf16 *tiles, int K, int v, int k) {
    const int t = v >> 7, r = v & 127, kt = k >> 6, c = (k & 63) >> 3, e = k & 7;
    return tiles + ((size_t)t * (K >> 6) + kt) * (TILE_ROWS * KT) + r * KT + ((c ^ (r & 7)) << 3) + e;
}

// ------------------------------------------------------------------ work items

// token / mask-embedding row -> residual h and its per-tile sums of squares.  A mask row is
// id -1 and exists only in adapter-on (draft) passes; any other id outside [0, V) latches
// DEV_BAD_TOKEN and reads row 0 instead of memory outside the embedding.
__device__ __noinline__ void do_embed(const MKParams &P, int m, int cw, int lane) {
    int tok = P.ids[m];
    if (tok >= P.dm.V || tok < -1 || (tok == -1 && !P.pd.adapter)) {
        latch_error(P.status, DEV_BAD_TOKEN);
        tok = 0;
    }
    const int H = P.dm.H, nt = H / TILE_ROWS;
    for (int t = cw; t < nt; t += CT / 32) {
        float v[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int f = t * TILE_ROWS + lane + 32 * e;
            v[e] = tok >= 0 ? bf2f(*tiled_at(P.embed_tiled, H, tok, f)) : bf2f(P.mask_embed[f]);
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) P.h[(size_t)m * H + t * TILE_ROWS + lane + 32 * e] = f2bf(v[e]);
        const float s = tile_sumsq(v);
        if (lane == 0) P.ss[(size_t)m * nt + t] = s;
    }
}

// Activation tile of one linear item in the 128-byte swizzle layout: four atoms (K columns
// 64j..64j+63 of the slice, starting a0 atoms into it) hold row m at m*128 bytes, 16-byte chunk c
// at (c ^ (m & 7)) * 16.  The chunks are copied straight into place with cp.async (one L2 round
// trip whatever the row count).  Rows of the q|k|v and gate|up inputs are then normalised in
// place: bf16(g * bf16(h * rs)), the product with the gain taken in bf16x2 (the exact product of
// two bf16 numbers rounded once to nearest even, as fp32 and then rounding gives).  A row has
// 32 chunks of 8 elements; thread ct handles chunks ct, ct + 192, ..., so its chunk column
// (ct % 32), and with it its gain chunk, is the same for all of them.
__device__ __noinline__ void build_b(const MKParams &P, int lin, int layer, int slice, uint8_t *sb, float *s_rms,
                                     const uint4 *s_gain, int ct, int a0, bool need_rms, unsigned long long *st) {
    const int M = P.pd.M;
    const bool norm = lin != 1;
    const bf16 *src = norm ? P.h : P.attn;  // (the down projection's operand: build_b_act)
    const int ld = norm ? P.dm.H : P.dm.Hq * P.dm.d;
    const int chunks = M * 32, c = ct & 31;
    const size_t col = (size_t)(slice * P.katoms[lin] + a0) * KT + c * 8;
    uint8_t *dst_c = sb + (size_t)(c >> 3) * P.bn * 128 + ((c & 7) << 4);
#pragma unroll 1
    for (int q = ct; q < chunks; q += CT) {
        const int m = q >> 5;
        cp_async16(dst_c + m * 128 - ((c & 7) << 4) + (((c & 7) ^ (m & 7)) << 4), src + (size_t)m * ld + col);
    }
    cp_async_commit();
    if (!norm) {
        cp_async_wait_all();
        return;
    }
    if (need_rms)  // while the copies are in flight
        for (int m = ct; m < M; m += CT) s_rms[m] = row_rms(P, m);
    cp_async_wait_all();
    const uint4 gv = s_gain[a0 * (KT / 8) + c];
    if (need_rms) {
        bar_compute();
        if (ct == 0) stamp_at(st, 8);
    }
    const __nv_bfloat162 *g2 = reinterpret_cast<const __nv_bfloat162 *>(&gv);
#pragma unroll 1
    for (int q = ct; q < chunks; q += CT) {
        const int m = q >> 5;
        uint4 *p = reinterpret_cast<uint4 *>(dst_c + m * 128 - ((c & 7) << 4) + (((c & 7) ^ (m & 7)) << 4));
        uint4 val = *p;
        __nv_bfloat162 *v2 = reinterpret_cast<__nv_bfloat162 *>(&val);
        const float rs = s_rms[m];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 f = __bfloat1622float2(v2[e]);
            v2[e] = __hmul2(g2[e], __floats2bfloat162_rn(__fmul_rn(f.x, rs), __fmul_rn(f.y, rs)));
        }
        *p = val;
    }
}

// The down projection's activation tile from the tagged act words of this layer's gate|up
// reductions (same layout as build_b): every 16-byte chunk of 8 features is four words, read
// again until all carry the tag (bounded).  No completion counter precedes it.
__device__ __noinline__ void build_b_act(const MKParams &P, int slice, uint8_t *sb, int ct, uint32_t tag,
                                         unsigned long long *st) {
    constexpr int U = 4;  // chunks in flight per thread
    const int M = P.pd.M, ld = P.dm.I;
    const int k0 = slice * P.katoms[3] * KT;
    const int cpr = P.katoms[3] * (KT / 8);  // 16-byte chunks per row
    const int chunks = M * cpr;
    for (int q0 = ct; q0 < chunks; q0 += U * CT) {
        unsigned long long tw[U][4];
        const unsigned long long none = (unsigned long long)tag << 32;
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int q = q0 + u * CT;
            if (q < chunks) {
                const unsigned long long *w = P.act + ((size_t)(q / cpr) * ld + k0 + (q % cpr) * 8) / 2;
                ld_relaxed_2u64(w, tw[u][0], tw[u][1]);
                ld_relaxed_2u64(w + 2, tw[u][2], tw[u][3]);
            } else {
                tw[u][0] = tw[u][1] = tw[u][2] = tw[u][3] = none;
            }
        }
        // stale words of all U chunks are read again together; the abort flag and the time
        // limit every 8 rounds
        bool stale = false;
#pragma unroll
        for (int u = 0; u < U; ++u)
#pragma unroll
            for (int k = 0; k < 4; ++k) stale |= !tag_is(tw[u][k], tag);
        const uint64_t t0 = stale ? globaltimer_ns() : 0;
        for (int round = 1; stale; ++round) {
            __nanosleep(32);
            stale = false;
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int q = min(q0 + u * CT, chunks - 1);
                const unsigned long long *w = P.act + ((size_t)(q / cpr) * ld + k0 + (q % cpr) * 8) / 2;
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    if (!tag_is(tw[u][k], tag)) {
                        tw[u][k] = ld_relaxed_u64(w + k);
                        stale |= !tag_is(tw[u][k], tag);
                    }
            }
            if (stale && (round & 7) == 0 && (aborted(P) || globaltimer_ns() - t0 > WAIT_LIMIT_NS)) {
                if (!aborted(P)) raise_abort(P, DEV_TIMEOUT_DEP);
                break;
            }
        }
        if (q0 == ct && ct == 0) stamp_at(st, 8);
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int q = q0 + u * CT;
            if (q >= chunks) break;
            const int m = q / cpr, c = q % cpr;
            const int atom = c >> 3, cc = c & 7;
            *reinterpret_cast<uint4 *>(sb + (size_t)atom * P.bn * 128 + m * 128 + ((cc ^ (m & 7)) << 4)) =
                make_uint4((uint32_t)tw[u][0], (uint32_t)tw[u][1], (uint32_t)tw[u][2], (uint32_t)tw[u][3]);
        }
    }
}

// q|k|v tile: adapter delta, bf16, per-head RMSNorm + RoPE for q and k, store q / paged K, V.
// Lane l reduces the four consecutive features 4l..4l+3 of the 128-feature tile (one head of 128,
// or two heads of 64: lanes 0-15 the first); the RoPE partner of feature i (i + DH/2 within the
// head) sits in lane l ^ (DH/8).  Per pass row m: rowpos[m] its position (-1 beyond the RoPE
// table), rowkv[m] its KV slot (page << 4 | slot in page; -1 beyond the reserved pages), both set
// at kernel start.
template <int DH, bool AD>
__device__ __noinline__ void reduce_qkv(const MKParams &P, int layer, int tile, int cw, int lane, int m0, int mstep,
                                       uint32_t tag, const int *rowpos, const int *rowkv, const uint4 *brows,
                                       unsigned long long *st) {
    constexpr int LPH = DH / 4;  // lanes per head
    const Dims &dm = P.dm;
    const int M = P.pd.M, r = dm.r;
    const int qw = dm.Hq * DH, kvw = dm.Hkv * DH, ft = tile * TILE_ROWS;
    const int kind = ft < qw ? 0 : (ft < qw + kvw ? 1 : 2);
    const int hl = lane / LPH, e0 = 4 * (lane % LPH);  // head within the tile, first element in the head
    const int head = (ft - (kind == 0 ? 0 : (kind == 1 ? qw : qw + kvw))) / DH + hl;
    const int f0 = ft + 4 * lane;
    const bool lo = e0 < DH / 2;  // first half of the head (RoPE: x cos - partner sin)
    float g[4];
    if (kind < 2) {
        const uint2 graw = __ldg(reinterpret_cast<const uint2 *>((kind == 0 ? P.q_norm : P.k_norm) + (size_t)layer * DH + e0));
        const float2 ga = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&graw.x));
        const float2 gb = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&graw.y));
        g[0] = ga.x, g[1] = ga.y, g[2] = gb.x, g[3] = gb.y;
    }
#pragma unroll 1
    for (int m = m0 + cw * mstep; m < M; m += (CT / 32) * mstep) {
        const int pos = rowpos[m];
        // the RoPE factors go out before the partial sums and land while they poll
        float4 cs4[2];
        if (kind < 2 && pos >= 0) {
            const float4 *c4 = reinterpret_cast<const float4 *>(P.rope_cs + (size_t)pos * (DH / 2) + (e0 % (DH / 2)));
            cs4[0] = __ldg(c4);
            cs4[1] = __ldg(c4 + 1);
        }
        float y[5];
        sum_parts<2, AD, AD ? 4 : 8>(P, 0, m, f0, P.n_main[0] + kind * r + (lane < r ? lane : 0), y, tag);
        unsigned long long *sw = (cw == 0 && m == m0 + cw * mstep && lane == 0) ? st : nullptr;  // first row
        stamp_at(sw, 9);
        float u[MAX_RANK];
        if (AD) share_u(y[4], 0, u);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            if (AD) y[j] = __fadd_rn(y[j], __fmul_rn(dm.lora_scale, lora_dot_w(u, smem_brow(brows, 4 * lane + j, r), r)));
            y[j] = rbf(y[j]);
        }
        if (kind < 2) {
            float ss = __fmul_rn(y[0], y[0]);
#pragma unroll
            for (int j = 1; j < 4; ++j) ss = __fadd_rn(ss, __fmul_rn(y[j], y[j]));
#pragma unroll
            for (int off = LPH / 2; off >= 1; off >>= 1) ss = __fadd_rn(ss, __shfl_xor_sync(0xffffffffu, ss, off));
            const float rs = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(__fdiv_rn(ss, (float)DH), dm.eps)));
#pragma unroll
            for (int j = 0; j < 4; ++j) y[j] = rbf(__fmul_rn(g[j], rbf(__fmul_rn(y[j], rs))));
            const float *cs = reinterpret_cast<const float *>(cs4);  // cos, sin of elements e0..e0+3
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float partner = __shfl_xor_sync(0xffffffffu, y[j], LPH / 2);
                const float c = cs[2 * j], sn = cs[2 * j + 1];
                y[j] = lo ? rbf(__fsub_rn(__fmul_rn(y[j], c), __fmul_rn(partner, sn)))
                          : rbf(__fadd_rn(__fmul_rn(y[j], c), __fmul_rn(partner, sn)));
            }
            if (pos < 0) {
                latch_error(P.status, DEV_BAD_POSITION);
                continue;
            }
        }
        stamp_at(sw, 10);
        bf16 *dst;
        if (kind == 0) {
            dst = P.q + ((size_t)m * dm.Hq + head) * DH + e0;
        } else {
            const int rk = rowkv[m];
            if (rk < 0) {
                latch_error(P.status, DEV_BAD_POSITION);
                continue;
            }
            dst = static_cast<bf16 *>(kind == 1 ? P.kv.k : P.kv.v) +
                  ((((size_t)layer * P.kv.n_pages + (rk >> 4)) * dm.Hkv + head) * PAGE + (rk & 15)) * DH + e0;
        }
        uint2 o;
        *reinterpret_cast<__nv_bfloat162 *>(&o.x) = __floats2bfloat162_rn(y[0], y[1]);
        *reinterpret_cast<__nv_bfloat162 *>(&o.y) = __floats2bfloat162_rn(y[2], y[3]);
        *reinterpret_cast<uint2 *>(dst) = o;
        stamp_at(sw, 11);
    }
}

// o or down tile: adapter delta, residual add into h, per-tile sum of squares.  Lane l reduces the
// four consecutive features 4l..4l+3 of the tile; the tile's sum of squares adds them in order,
// then across the lanes by a fixed butterfly.
template <bool AD>
__device__ __noinline__ void reduce_residual(const MKParams &P, int lin, int layer, int tile, int cw, int lane, int m0,
                                             int mstep, uint32_t tag, const uint4 *brows, unsigned long long *st) {
    const Dims &dm = P.dm;
    const int M = P.pd.M, r = dm.r, H = dm.H, nt = H / TILE_ROWS;
    const int f0 = tile * TILE_ROWS + 4 * lane;
#pragma unroll 1
    for (int m = m0 + cw * mstep; m < M; m += (CT / 32) * mstep) {
        uint2 *hp = reinterpret_cast<uint2 *>(P.h + (size_t)m * H + f0);
        const uint2 hraw = __ldcg(hp);
        float acc[5];
        sum_parts<2, AD, AD ? 4 : 12>(P, lin, m, f0, P.n_main[lin] + (lane < r ? lane : 0), acc, tag);
        unsigned long long *sw = (cw == 0 && m == m0 && lane == 0) ? st : nullptr;  // first row's sub-steps
        stamp_at(sw, 9);
        float u[MAX_RANK];
        if (AD) share_u(acc[4], 0, u);
        const __nv_bfloat162 *h2 = reinterpret_cast<const __nv_bfloat162 *>(&hraw);
        const float2 ha = __bfloat1622float2(h2[0]), hb = __bfloat1622float2(h2[1]);
        const float hv[4] = {ha.x, ha.y, hb.x, hb.y};
        float v[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            if (AD) acc[e] = __fadd_rn(acc[e], __fmul_rn(dm.lora_scale, lora_dot_w(u, smem_brow(brows, 4 * lane + e, r), r)));
            v[e] = rbf(__fadd_rn(hv[e], rbf(acc[e])));
        }
        uint2 o;
        *reinterpret_cast<__nv_bfloat162 *>(&o.x) = __floats2bfloat162_rn(v[0], v[1]);
        *reinterpret_cast<__nv_bfloat162 *>(&o.y) = __floats2bfloat162_rn(v[2], v[3]);
        *hp = o;
        stamp_at(sw, 10);
        float sq = __fmul_rn(v[0], v[0]);
#pragma unroll
        for (int e = 1; e < 4; ++e) sq = __fadd_rn(sq, __fmul_rn(v[e], v[e]));
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) sq = __fadd_rn(sq, __shfl_xor_sync(0xffffffffu, sq, off));
        if (lane == 0) P.ss[(size_t)m * nt + tile] = sq;
        stamp_at(sw, 11);
    }
}

// gate|up tile (rows 0-63 gate features 64t.., rows 64-127 up features 64t..): SiLU(gate)*up.
// Lane l produces act features 64t + 2l and 64t + 2l + 1 (tile rows 2l, 2l + 1 and 64 + 2l,
// 64 + 2l + 1) and stores them as one tagged word.
template <bool AD>
__device__ __noinline__ void reduce_gu(const MKParams &P, int layer, int tile, int cw, int lane, int m0, int mstep,
                                      uint32_t tag, const uint4 *brows, unsigned long long *st) {
    const Dims &dm = P.dm;
    const int M = P.pd.M, r = dm.r, I = dm.I;
    const int a0 = tile * 64 + 2 * lane;  // the lane's first act feature
#pragma unroll 1
    for (int m = m0 + cw * mstep; m < M; m += (CT / 32) * mstep) {
        // sums: gate pair, up pair; feature 4: adapter row lane (lanes 0..r-1 sum u_gate, r..2r-1 u_up)
        float ug[MAX_RANK], uu[MAX_RANK], s[5];
        sum_parts<64, AD, 2>(P, 2, m, tile * TILE_ROWS + 2 * lane, P.n_main[2] + (lane < 2 * r ? lane : 0), s, tag);
        unsigned long long *sw = (cw == 0 && m == m0 && lane == 0) ? st : nullptr;  // first row's sub-steps
        stamp_at(sw, 9);
        if (AD) {
            share_u(s[4], 0, ug);
            share_u(s[4], r, uu);
        }
        uint32_t bits[2];
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            float g = s[e], up = s[2 + e];
            if (AD) {
                g = __fadd_rn(g, __fmul_rn(dm.lora_scale, lora_dot_w(ug, smem_brow(brows, 2 * lane + e, r), r)));
                up = __fadd_rn(up, __fmul_rn(dm.lora_scale, lora_dot_w(uu, smem_brow(brows, 64 + 2 * lane + e, r), r)));
            }
            g = rbf(g);
            up = rbf(up);
            const float sg = __fdiv_rn(g, __fadd_rn(1.0f, expf(-g)));
            bits[e] = __bfloat16_as_ushort(f2bf(__fmul_rn(sg, up)));
        }
        st_relaxed_u64(P.act + ((size_t)m * I + a0) / 2, ((unsigned long long)tag << 32) | (bits[1] << 16) | bits[0]);
        stamp_at(sw, 11);
    }
}

// ---- attention

// Attention split staging layout in the union buffer: K then V, each DH/64 sub-tiles of
// [128 keys x 128 bytes] in the 128-byte swizzle layout (16-byte chunk c of key n at
// (c ^ (n & 7)) * 16), exactly as the tiled TMA writes them.
constexpr int ATT_SUB_BYTES = ATT_SPLIT * 128;

__device__ __forceinline__ uint32_t sw128(int row, int colb) {
    return (uint32_t)(row * 128 + ((((colb >> 4) ^ (row & 7)) << 4) | (colb & 15)));
}

// TMA loads of the pages of one attention item (att_span consecutive 128-key splits), issued by
// one warp of the compute group (all lanes call): stage 0 = pages entirely below the cached length
// L (written by earlier passes: requested before the item's inputs are ready); stage 1 = pages
// holding this pass's block rows.  Lane p < 8 * span reads the page-table entry of the item's page
// p (one round trip for all); lane 0 announces the stage's bytes on `bar` (stage 1 with the item's
// one arrival); then the lanes issue the copies (page, K or V, 64-dim half) together, one per lane
// and round.  Split j of the item lands at smem + j * 2 (d/64) ATT_SUB_BYTES: its K halves, then its
// V halves.
__device__ __noinline__ void attn_pages(const MKParams &P, int layer, int bl, int g, int s, int stage, uint8_t *smem,
                                        uint64_t *bar, int lane) {
    constexpr int NP = ATT_SPLIT / PAGE;
    const int span = P.pd.att_span, npg = NP * span;
    const int b = P.pd.b0 + bl;
    const int L = P.L[b], T = L + P.pd.R, k0 = s * span * ATT_SPLIT, pg0 = k0 / PAGE;
    int ph = 0;
    bool ok = false;
    if (lane < npg) {
        const int kp0 = k0 + lane * PAGE;
        ok = kp0 < T && pg0 + lane < P.kv.pages_per_seq && ((kp0 + PAGE <= L) == (stage == 0));
        if (ok) ph = P.kv.page_table[(size_t)b * P.kv.pages_per_seq + pg0 + lane];
    }
    const unsigned mask = __ballot_sync(0xffffffffu, ok);
    const int subs = P.dm.d / 64, tpp = 2 * subs;  // copies per page: K and V, per 64-dim half
    if (lane == 0) {
        const uint32_t bytes = (uint32_t)__popc(mask) * (uint32_t)tpp * PAGE * 128u;
        if (stage == 1)
            mbar_arrive_expect_tx(bar, bytes);
        else if (bytes)
            mbar_expect_tx(bar, bytes);
    }
    __syncwarp();
    // the block's pages were written by this pass's q|k|v reducers (generic stores, acquired
    // before this call): order them before the TMA reads
    if (stage == 1 && mask) fence_proxy_async_global();
#pragma unroll 1
    for (int c0 = 0; c0 < npg * tpp; c0 += 32) {  // uniform over the warp: one or two rounds
        const int cp = c0 + lane, p = min(cp / tpp, 31), r = cp % tpp;
        const int phys = __shfl_sync(0xffffffffu, ph, p);
        if (cp < npg * tpp && ((mask >> p) & 1u)) {
            const int kind = r / subs, sub = r % subs, sp = p / NP;
            const int row0 = ((layer * P.kv.n_pages + phys) * P.dm.Hkv + g) * PAGE;
            tma_load_2d(smem + ((sp * 2 + kind) * subs + sub) * ATT_SUB_BYTES + (p % NP) * PAGE * 128,
                        kind ? &P.vmap : &P.kmap, sub * 64, row0, bar);
        }
    }
}

// One (sequence, KV head, att_span 128-key splits) item on the compute group, after its K/V pages
// landed in `smem` (stages 0 and 1 of attn_pages) and `bar` completed phase `parity`.  Each warp
// takes units of one 16-row query tile against one split's keys, or one 64-key half of them when a
// split has two partial results; every unit is a partial result (m, l, O) that the merge combines
// in key order; the partition of the keys does not depend on the span.  Within a unit the keys go
// in chunks of 32 with a running maximum (online softmax): scores by bf16 mma.sync, the row maximum
// and the weights in fp32, P (weights) rounded to bf16 against the cached bf16 V, O in fp32.  The loop
// over chunks is not unrolled: the code stays small enough for the instruction cache.
template <int DH, bool BLK>
__device__ __noinline__ void attn_split(const MKParams &P, int layer, int bl, int g, int s, uint8_t *smem,
                                        uint64_t *bar, uint32_t parity, int ct, int cw, int lane,
                                        unsigned long long *stamp) {
    constexpr int KS = DH / 16, DT = DH / 8, SUBS = DH / 64;
    constexpr int SPB = 2 * SUBS * ATT_SUB_BYTES;  // staged bytes per split (K, then V)
    const int subs = P.att_subs, HALF = ATT_SPLIT / subs;
    const Dims &dm = P.dm;
    const int b = P.pd.b0 + bl;
    const int L = P.L[b];
    const int R = P.pd.R;
    const int T = L + R;
    const int sp0 = s * P.pd.att_span;  // the item's first split
    const int nsx = min(P.pd.att_span, (T - sp0 * ATT_SPLIT + ATT_SPLIT - 1) / ATT_SPLIT);  // splits holding keys
    const int grp = dm.Hq / dm.Hkv;
    const int QV = R * grp;
    const int n_mt = (QV + 15) / 16;
    const bool landed = mbar_wait_mk(bar, parity, P, DEV_TIMEOUT_LOAD);
    if (stamp && ct == 0) stamp[4] = globaltimer_ns();
    if (stamp && ct == 0) stamp[5] = globaltimer_ns();
    if (!landed) return;
    const int gq = lane >> 2, tq = lane & 3;
    const float scale = P.att_scale;
#pragma unroll 1
    for (int unit = cw; unit < n_mt * nsx * subs; unit += CT / 32) {
        const int mt = unit / (nsx * subs), sp = (unit / subs) % nsx, half = unit % subs, kb = half * HALF;
        const int k0 = (sp0 + sp) * ATT_SPLIT;
        const uint8_t *sK = smem + sp * SPB, *sV = sK + SUBS * ATT_SUB_BYTES;
        const int qv0 = mt * 16 + gq, qv1 = qv0 + 8;
        const bool val0 = qv0 < QV, val1 = qv1 < QV;
        const int i0 = val0 ? qv0 / grp : 0, i1 = val1 ? qv1 / grp : 0;
        const int h0 = g * grp + (val0 ? qv0 % grp : 0), h1 = g * grp + (val1 ? qv1 % grp : 0);
        unsigned long long *sw = (unit == 0 && lane == 0) ? stamp : nullptr;  // first unit's sub-steps
        uint32_t qa[KS][4];
        {
            const bf16 *q0 = P.q + ((size_t)(bl * R + i0) * dm.Hq + h0) * DH + 2 * tq;
            const bf16 *q1 = P.q + ((size_t)(bl * R + i1) * dm.Hq + h1) * DH + 2 * tq;
#pragma unroll
            for (int ks = 0; ks < KS; ++ks) {
                qa[ks][0] = val0 ? __ldcg(reinterpret_cast<const unsigned *>(q0 + ks * 16)) : 0u;
                qa[ks][1] = val1 ? __ldcg(reinterpret_cast<const unsigned *>(q1 + ks * 16)) : 0u;
                qa[ks][2] = val0 ? __ldcg(reinterpret_cast<const unsigned *>(q0 + ks * 16 + 8)) : 0u;
                qa[ks][3] = val1 ? __ldcg(reinterpret_cast<const unsigned *>(q1 + ks * 16 + 8)) : 0u;
            }
        }
        // last visible key of each row: causal rows see up to themselves; in the draft the
        // block's mask rows (i >= 1) also see the rest of the block
        const int lim0 = val0 ? ((BLK && i0 >= 1) ? T - 1 : L + i0) : -1;
        const int lim1 = val1 ? ((BLK && i1 >= 1) ? T - 1 : L + i1) : -1;
        float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
        float oc[DT][4];
#pragma unroll
        for (int dt = 0; dt < DT; ++dt) oc[dt][0] = oc[dt][1] = oc[dt][2] = oc[dt][3] = 0.f;
        const int kend = min(HALF, T - (k0 + kb));  // keys of the half that exist
        constexpr int CN = 4;  // n-tiles of 8 keys per chunk (32 keys)
#pragma unroll 1
        for (int c0 = 0; c0 < kend; c0 += 8 * CN) {
            float sc[CN][4];
#pragma unroll
            for (int nt = 0; nt < CN; ++nt) {
                sc[nt][0] = sc[nt][1] = sc[nt][2] = sc[nt][3] = 0.f;
                // K fragments of two k-steps per ldmatrix.x4: matrix j = keys n0..n0+7, dims 8j..8j+7
                // of the 32-dim chunk; thread t addresses row t % 8 of matrix t / 8
                const int kr = kb + c0 + nt * 8 + (lane & 7);
#pragma unroll
                for (int ks = 0; ks < KS; ks += 2) {
                    const int e = ks * 16 + (lane >> 3) * 8;
                    const uint32_t addr = smem_u32(sK + (e >> 6) * ATT_SUB_BYTES + sw128(kr, (e & 63) * 2));
                    uint32_t b0, b1, b2, b3;
                    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                                 : "=r"(b0), "=r"(b1), "=r"(b2), "=r"(b3)
                                 : "r"(addr));
                    mma_m16n8k16_bf16(sc[nt], qa[ks], b0, b1);
                    mma_m16n8k16_bf16(sc[nt], qa[ks + 1], b2, b3);
                }
            }
            float c0m = -INFINITY, c1m = -INFINITY;
#pragma unroll
            for (int nt = 0; nt < CN; ++nt)
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const int kp = k0 + kb + c0 + nt * 8 + 2 * tq + e;
                    sc[nt][e] = kp <= lim0 ? __fmul_rn(sc[nt][e], scale) : -INFINITY;
                    sc[nt][2 + e] = kp <= lim1 ? __fmul_rn(sc[nt][2 + e], scale) : -INFINITY;
                    c0m = fmaxf(c0m, sc[nt][e]);
                    c1m = fmaxf(c1m, sc[nt][2 + e]);
                }
            c0m = fmaxf(c0m, __shfl_xor_sync(0xffffffffu, c0m, 1));
            c0m = fmaxf(c0m, __shfl_xor_sync(0xffffffffu, c0m, 2));
            c1m = fmaxf(c1m, __shfl_xor_sync(0xffffffffu, c1m, 1));
            c1m = fmaxf(c1m, __shfl_xor_sync(0xffffffffu, c1m, 2));
            const float n0 = fmaxf(m0, c0m), n1 = fmaxf(m1, c1m);
            // rescale what was summed so far to the new maximum (nothing was while it is -inf;
            // skipped by the whole warp when no row's maximum moved)
            if (__any_sync(0xffffffffu, (n0 != m0 && m0 != -INFINITY) || (n1 != m1 && m1 != -INFINITY))) {
                const float a0 = m0 == -INFINITY ? 0.f : __expf(m0 - n0), a1 = m1 == -INFINITY ? 0.f : __expf(m1 - n1);
                l0 = __fmul_rn(l0, a0);
                l1 = __fmul_rn(l1, a1);
#pragma unroll
                for (int dt = 0; dt < DT; ++dt) {
                    oc[dt][0] = __fmul_rn(oc[dt][0], a0);
                    oc[dt][1] = __fmul_rn(oc[dt][1], a0);
                    oc[dt][2] = __fmul_rn(oc[dt][2], a1);
                    oc[dt][3] = __fmul_rn(oc[dt][3], a1);
                }
            }
            const float z0 = n0 == -INFINITY ? 0.f : n0, z1 = n1 == -INFINITY ? 0.f : n1;
            m0 = n0;
            m1 = n1;
#pragma unroll
            for (int nt = 0; nt < CN; ++nt)
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    sc[nt][e] = sc[nt][e] == -INFINITY ? 0.f : __expf(sc[nt][e] - z0);
                    sc[nt][2 + e] = sc[nt][2 + e] == -INFINITY ? 0.f : __expf(sc[nt][2 + e] - z1);
                    l0 += sc[nt][e];
                    l1 += sc[nt][2 + e];
                }
            // P as the bf16 A fragments of two 16-key steps
#pragma unroll
            for (int kstep = 0; kstep < CN / 2; ++kstep) {
                uint32_t pa[4];
                pa[0] = pack_bf162(sc[2 * kstep][0], sc[2 * kstep][1]);
                pa[1] = pack_bf162(sc[2 * kstep][2], sc[2 * kstep][3]);
                pa[2] = pack_bf162(sc[2 * kstep + 1][0], sc[2 * kstep + 1][1]);
                pa[3] = pack_bf162(sc[2 * kstep + 1][2], sc[2 * kstep + 1][3]);
                const int vrow = kb + c0 + kstep * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
                // V of keys at or past T is set to zero in the fragments: their weights are 0, but
                // their rows hold whatever the cache or shared memory held (a page's tail beyond the
                // sequence, or pages not loaded at all), and 0 times an Inf or NaN there would
                // poison the sum.  Fragment registers b0 / b1 hold keys 2 tq, 2 tq + 1 / + 8, + 9 of
                // the 16-key step, the lower key in the low half.
                const int kst = k0 + kb + c0 + kstep * 16;  // first key of the step
                uint32_t ma = 0xFFFFFFFFu, mb = 0xFFFFFFFFu;
                if (kst + 16 > T) {  // warp-uniform: only the steps that reach T
                    const int ka = kst + 2 * tq;
                    ma = (ka < T ? 0x0000FFFFu : 0u) | (ka + 1 < T ? 0xFFFF0000u : 0u);
                    mb = (ka + 8 < T ? 0x0000FFFFu : 0u) | (ka + 9 < T ? 0xFFFF0000u : 0u);
                }
#pragma unroll
                for (int dt = 0; dt < DT; dt += 2) {
                    const int vcol = dt * 8 + (lane >> 4) * 8;
                    const uint32_t addr = smem_u32(sV + (vcol >> 6) * ATT_SUB_BYTES + sw128(vrow, (vcol & 63) * 2));
                    uint32_t r0, r1, r2, r3;
                    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                                 : "r"(addr));
                    mma_m16n8k16_bf16(oc[dt], pa, r0 & ma, r1 & mb);
                    mma_m16n8k16_bf16(oc[dt + 1], pa, r2 & ma, r3 & mb);
                }
            }
        }
        stamp_at(sw, 10);
        l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
        l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
        l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
        l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
        const int nsa = P.att_splits_alloc;
        const int sub = (sp0 + sp) * subs + half;  // index of this partial result
        if (val0) {
            float *dst = P.o_part + (((size_t)(bl * R + i0) * dm.Hq + h0) * nsa + sub) * DH + 2 * tq;
#pragma unroll
            for (int dt = 0; dt < DT; ++dt) *reinterpret_cast<float2 *>(dst + dt * 8) = make_float2(oc[dt][0], oc[dt][1]);
            if (tq == 0) P.ml_part[((size_t)(bl * R + i0) * dm.Hq + h0) * nsa + sub] = make_float2(m0, l0);
        }
        if (val1) {
            float *dst = P.o_part + (((size_t)(bl * R + i1) * dm.Hq + h1) * nsa + sub) * DH + 2 * tq;
#pragma unroll
            for (int dt = 0; dt < DT; ++dt) *reinterpret_cast<float2 *>(dst + dt * 8) = make_float2(oc[dt][2], oc[dt][3]);
            if (tq == 0) P.ml_part[((size_t)(bl * R + i1) * dm.Hq + h1) * nsa + sub] = make_float2(m1, l1);
        }
        stamp_at(sw, 11);
    }
}

// merge the splits of (row, head) in split order; splits where the row saw no key are skipped
template <int DH>
__device__ __noinline__ void attn_combine(const MKParams &P, int bl, int g, int cw, int lane, int p0, int pstep,
                                          unsigned long long *st) {
    const Dims &dm = P.dm;
    const int R = P.pd.R, grp = dm.Hq / dm.Hkv;
    const int b = P.pd.b0 + bl;
    const int T = P.L[b] + R;
    const int nsa = P.att_splits_alloc;
    // partial results computed in this pass: att_subs per split that holds a key
    const int nv = min(P.nsplit[bl], (T + ATT_SPLIT - 1) / ATT_SPLIT) * P.att_subs;
    constexpr int E = DH / 32;
    for (int it = p0 + cw * pstep; it < R * grp; it += (CT / 32) * pstep) {
        const int i = it / grp, h = g * grp + it % grp;
        const int m = bl * R + i;
        const float2 *ml = P.ml_part + ((size_t)m * dm.Hq + h) * nsa;
        const float *ob = P.o_part + ((size_t)m * dm.Hq + h) * nsa * DH + lane;
        // the first 16 partial results' statistics and the first 8 outputs go out together
        constexpr int NB = 16, OB = 8;
        float2 v[NB];
        float o[OB][E];
#pragma unroll
        for (int u = 0; u < NB; ++u) v[u] = u < nv ? __ldcg(ml + u) : make_float2(-INFINITY, 0.f);
#pragma unroll
        for (int u = 0; u < OB; ++u)
#pragma unroll
            for (int e = 0; e < E; ++e) o[u][e] = u < nv ? __ldcg(ob + (size_t)u * DH + 32 * e) : 0.f;
        float mx = -INFINITY;
#pragma unroll
        for (int u = 0; u < NB; ++u)
            if (v[u].y > 0.f) mx = fmaxf(mx, v[u].x);
        if (cw == 0 && it == p0 && lane == 0) stamp_at(st, 12);
        for (int s0 = NB; s0 < nv; s0 += NB) {  // long contexts only: NB statistics per round
            float2 w[NB];
#pragma unroll
            for (int u = 0; u < NB; ++u) w[u] = s0 + u < nv ? __ldcg(ml + s0 + u) : make_float2(-INFINITY, 0.f);
#pragma unroll
            for (int u = 0; u < NB; ++u)
                if (w[u].y > 0.f) mx = fmaxf(mx, w[u].x);
        }
        float num[E];
#pragma unroll
        for (int e = 0; e < E; ++e) num[e] = 0.f;
        float den = 0.f;
        for (int s0 = 0; s0 < nv; s0 += OB) {
            if (s0 > 0)
#pragma unroll
                for (int u = 0; u < OB; ++u)
#pragma unroll
                    for (int e = 0; e < E; ++e) o[u][e] = s0 + u < nv ? __ldcg(ob + (size_t)(s0 + u) * DH + 32 * e) : 0.f;
#pragma unroll
            for (int u = 0; u < OB; ++u) {
                const int sp = s0 + u;
                if (sp >= nv) break;
                const float2 st = sp < NB ? v[sp < NB ? sp : 0] : __ldcg(ml + sp);
                if (!(st.y > 0.f)) continue;  // the row saw no key in this partial result
                const float w = __expf(st.x - mx);
                den = __fadd_rn(den, __fmul_rn(w, st.y));
#pragma unroll
                for (int e = 0; e < E; ++e) num[e] = __fadd_rn(num[e], __fmul_rn(w, o[u][e]));
            }
        }
        bf16 *dst = P.attn + ((size_t)m * dm.Hq + h) * DH;
#pragma unroll
        for (int e = 0; e < E; ++e) dst[lane + 32 * e] = f2bf(__fdiv_rn(num[e], den));
    }
}

// Attention merge mode of a (sequence, head) with nsp items: shared by all items when they sit on
// distinct CTAs (nsp <= grid), else done by the last one.
__device__ __forceinline__ bool att_shared_merge(int nsp) { return nsp <= (int)gridDim.x; }

// the item's inputs are complete (one thread; false on abort)
__device__ __forceinline__ bool wait_deps(const MKParams &P, const MKItem &it) {
    return it.wait_off < 0 || spin_until(P.cnt + it.wait_off, it.wait_tgt, P);
}

// one thread: the item's result is stored (and made visible to it by a barrier): count it
__device__ __forceinline__ void release_item(const MKParams &P, const MKItem &it) {
    if (it.rel[0] >= 0) red_release_add(P.cnt + it.rel[0], 1);
    if (it.rel[1] >= 0) red_release_add(P.cnt + it.rel[1], 1);
}

// ------------------------------------------------------------------ the kernel

// Per-CTA shared state of the pass kernel (static shared memory).
struct CtaState {
    uint64_t full[MAX_SLOT], empty[MAX_SLOT], b_full[2], b_empty, acc_full, att_bar, mma_drain;
    uint32_t tmem_slot;
    // compute-group flags: each is written by thread 0 and read by all after a barrier, and is
    // not written again before every thread has passed at least one more barrier
    int flag, red, ok;
    uint32_t tag;  // this pass's partial-sum tag
    float rms[MAX_ROWS];
    // per pass row: position (-1 beyond the RoPE table) and KV slot (page << 4 | slot; -1 beyond
    // the reserved pages)
    int rowpos[MAX_ROWS], rowkv[MAX_ROWS];
    // the adapter's B rows of the tile a draft's linear item reduces (tile row order: for
    // gate|up rows 0-63 gate, 64-127 up), staged at the item's start
    uint4 brows[TILE_ROWS * MAX_RANK / 8 + TILE_ROWS / 4];
    // the RMSNorm gain of the K slice a q|k|v or gate|up item stages
    uint4 gain[MAX_ATOMS * KT / 8];
};

// ---- warp 0 lane 0: weight producer.  Walks the CTA's linear items ahead of the others and
// streams their 128 x 64 weight tiles into the ring (1-D bulk TMA, L2 evict-first); weights depend
// on nothing, so the ring fills across phase boundaries.
__device__ __noinline__ void run_producer(const MKParams &P, const MKItem *my, int n_my, uint8_t *ring, CtaState &S) {
    const uint64_t pol = l2_policy_evict_first();
    uint32_t kt = 0;
#pragma unroll 1
    for (int i = 0; i < n_my && !aborted(P); ++i) {
        const MKItem it = my[i];
        if (it.op != MK_LINEAR) continue;
        const int lin = it.lin;
        const bool lt = it.a >= P.n_main[lin] / TILE_ROWS;
        const uint32_t bytes = lt ? (uint32_t)P.lora_rows[lin] * 128u : (uint32_t)TILE_BYTES;
        const int kts = P.K[lin] / KT;
        const uint8_t *src =
            P.wt[lin] + P.wt_stride[lin] * it.layer + ((size_t)it.a * kts + (size_t)it.b * P.katoms[lin]) * TILE_BYTES;
        bool ok = true;
#pragma unroll 1
        for (int j = 0; j < P.katoms[lin]; ++j, ++kt) {
            const int slot = kt % P.nslot;
            if (kt >= (uint32_t)P.nslot && !mbar_wait_mk(&S.empty[slot], ((kt / P.nslot) - 1) & 1, P, DEV_TIMEOUT_SLOT)) {
                ok = false;
                break;
            }
            mbar_arrive_expect_tx(&S.full[slot], bytes);
            bulk_g2s(ring + (size_t)slot * TILE_BYTES, src + (size_t)j * TILE_BYTES, bytes, &S.full[slot], pol);
        }
        if (!ok) break;
    }
    if (aborted(P))  // the last nslot tiles issued may still be in flight: let them land
#pragma unroll 1
        for (uint32_t h = kt > (uint32_t)P.nslot ? kt - P.nslot : 0; h < kt; ++h)
            drain_wait(&S.full[h % P.nslot], (h / P.nslot) & 1);
}

// ---- warp 1 lane 0: MMA issuer.  Per linear item, 4 (or 8) x 4 tcgen05.mma (128 x bn x 16,
// bf16 -> fp32) into the TMEM accumulator; frees ring slots with tcgen05.commit.
__device__ __noinline__ void run_mma(const MKParams &P, const MKItem *my, int n_my, uint8_t *ring, uint8_t *uni,
                                     uint32_t tmem, CtaState &S) {
    const uint32_t idesc = idesc_bf16_f32(128, P.bn);
    uint32_t kt = 0, li = 0, l8 = 0;
#pragma unroll 1
    for (int i = 0; i < n_my; ++i) {
        const MKItem it = my[i];
        if (it.op != MK_LINEAR) continue;
        const int na = P.katoms[it.lin];
        if (!mbar_wait_mk(&S.b_full[0], li & 1, P, DEV_TIMEOUT_LOAD)) break;
        tc_fence_after();
        bool ok = true;
#pragma unroll 1
        for (int j = 0; j < na; ++j, ++kt) {
            if (j == HALF_ATOMS) {
                // second half of a wide slice: its operand is staged after the first half's reads
                // completed (same area) or was staged with it
                if (!P.b_dbl) mma_commit(&S.b_empty);
                if (!mbar_wait_mk(&S.b_full[1], l8 & 1, P, DEV_TIMEOUT_LOAD)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
            }
            const int slot = kt % P.nslot;
            if (!mbar_wait_mk(&S.full[slot], (kt / P.nslot) & 1, P, DEV_TIMEOUT_LOAD)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint64_t ad = sw128_kmajor_desc(ring + (size_t)slot * TILE_BYTES);
            const int bj = (P.b_dbl || j < HALF_ATOMS) ? j : j - HALF_ATOMS;
            const uint64_t bd = sw128_kmajor_desc(uni + (size_t)bj * P.bn * 128);
#pragma unroll
            for (int kk = 0; kk < KT / 16; ++kk)
                mma_bf16_ss(tmem, ad + 2ull * kk, bd + 2ull * kk, idesc, (j | kk) != 0 ? 1u : 0u);
            mma_commit(&S.empty[slot]);
        }
        if (!ok) break;
        mma_commit(&S.acc_full);
        ++li;
        if (na > HALF_ATOMS) ++l8;
    }
    if (aborted(P)) {
        // every MMA issued so far completes before TMEM and the operands are released
        mma_commit(&S.mma_drain);
        drain_wait(&S.mma_drain, 0);
    }
}

// ---- compute group: final RMSNorm of one read-out row (the lm_head's input)
__device__ __noinline__ void item_final(const MKParams &P, const MKItem &it, int ct, CtaState &S) {
    const int r = it.a, m = it.b;
    if (ct == 0) S.rms[0] = row_rms(P, m);
    bar_compute();
    const float rs = S.rms[0];
#pragma unroll 1
    for (int c8 = ct; c8 < P.dm.H / 8; c8 += CT) {
        uint4 hv = __ldcg(reinterpret_cast<const uint4 *>(P.h + (size_t)m * P.dm.H) + c8);
        const uint4 gv = __ldg(reinterpret_cast<const uint4 *>(P.final_norm) + c8);
        __nv_bfloat162 *h2 = reinterpret_cast<__nv_bfloat162 *>(&hv);
        const __nv_bfloat162 *g2 = reinterpret_cast<const __nv_bfloat162 *>(&gv);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 f = __bfloat1622float2(h2[e]);
            h2[e] = __hmul2(g2[e], __floats2bfloat162_rn(__fmul_rn(f.x, rs), __fmul_rn(f.y, rs)));
        }
        reinterpret_cast<uint4 *>(P.x_ro + (size_t)r * P.dm.H)[c8] = hv;
    }
}

// ---- compute group: one attention split item (pages, split, merge).  Returns false on abort.
template <bool DRAFT, int DH>
__device__ __noinline__ bool item_attn(const MKParams &P, const MKItem &it, bool active, uint8_t *uni, CtaState &S,
                                       uint32_t &ai, int ct, int cw, int lane, unsigned long long *st) {
    const int bl = it.a, g = it.b, s = it.c;
    if (active) {
        if (cw == 0) {
            attn_pages(P, it.layer, bl, g, s, 1, uni, &S.att_bar, lane);
            if (lane == 0) stamp_at(st, 8);
        }
        attn_split<DH, DRAFT>(P, it.layer, bl, g, s, uni, &S.att_bar, ai & 1, ct, cw, lane, st);
        ++ai;
    }
    bar_compute();
    if (ct == 0) stamp_at(st, 2);
    // merge: when the (sequence, head)'s items fit on distinct CTAs, every item waits for the
    // others and merges pairs s, s + items, ...; otherwise the last one merges all
    int *c = ctr(P, it.layer, P.cl.att + bl * P.dm.Hkv + g);
    const int nsp = (P.nsplit[bl] + P.pd.att_span - 1) / P.pd.att_span;
    const bool shared_merge = att_shared_merge(nsp);
    if (ct == 0) {
        if (shared_merge) {
            red_release_add(c, 1);
            S.ok = spin_until(c, nsp, P) ? 1 : 0;
            S.red = 1;
        } else {
            S.red = (atom_acq_rel_add(c, 1) == nsp - 1) ? 1 : 0;
            S.ok = 1;
        }
        stamp_at(st, 6);
        stamp_at(st, 7);
    }
    bar_compute();
    if (!S.ok) return false;
    if (S.red) {
        const int p0 = shared_merge ? s : 0, pstep = shared_merge ? nsp : 1;
        attn_combine<DH>(P, bl, g, cw, lane, p0, pstep, st);
        bar_compute();
        if (ct == 0) {
            release_item(P, it);  // counts on the o slice that reads the group
            stamp_at(st, 7);
        }
    }
    return true;
}

// ---- compute group: one linear slice item: stage the activation operand (warp 1 then issues the
// MMAs), read the accumulator out as tagged partial sums, and reduce this CTA's share of the tile's
// rows.  The tile's K slices are consecutive items of the round-robin schedule, so they sit on
// distinct CTAs that all reach them: each CTA stores its tagged slice partials, then reduces rows
// s, s + ks, ... of the tile (s = its slice), reading the other slices' partials as they arrive.
// The adapter tile's partials are summed by the main tiles' reducers themselves.  Returns false
// on abort.
template <bool DRAFT, int DH>
__device__ __noinline__ bool item_linear(const MKParams &P, const MKItem &it, uint8_t *uni, uint32_t tmem, CtaState &S,
                                         uint32_t &li, uint32_t &l8, int ct, int cw, int lane, int warp,
                                         unsigned long long *st) {
    const int lin = it.lin, l = it.layer, t = it.a, s = it.b;
    const int na = P.katoms[lin];
    if (na <= HALF_ATOMS) {
        if (lin == 3) {
            build_b_act(P, s, uni, ct, S.tag + l, st);
            if (DRAFT) cp_async_wait_all();  // the B rows (the operand needed no copies)
        } else
            build_b(P, lin, l, s, uni, S.rms, S.gain, ct, 0, true, st);
        fence_proxy_async();
        bar_compute();
        if (ct == 0) mbarrier_arrive_one(&S.b_full[0]);
    } else {
        // wide slice in two halves: when both fit, the first half's MMAs run while the second is
        // staged; else the second goes through the same area after the first half's reads
        build_b(P, lin, l, s, uni, S.rms, S.gain, ct, 0, true, st);
        fence_proxy_async();
        bar_compute();
        if (ct == 0) {
            mbarrier_arrive_one(&S.b_full[0]);
            if (!P.b_dbl) S.ok = mbar_wait_mk(&S.b_empty, l8 & 1, P, DEV_TIMEOUT_MMA) ? 1 : 0;
        }
        if (!P.b_dbl) {
            bar_compute();
            if (!S.ok) return false;
        }
        build_b(P, lin, l, s, uni + (P.b_dbl ? (size_t)HALF_ATOMS * P.bn * 128 : 0), S.rms, S.gain, ct, HALF_ATOMS,
                false, nullptr);
        fence_proxy_async();
        bar_compute();
        if (ct == 0) mbarrier_arrive_one(&S.b_full[1]);
        ++l8;
    }
    if (ct == 0) stamp_at(st, 4);
    const bool lt = t >= P.n_main[lin] / TILE_ROWS;
    const uint32_t tag = S.tag + l;
    if (warp >= 4) {
        // epilogue: warp 4 + q reads TMEM lanes 32q..32q+31 (the tile's weight rows), 32 token
        // columns at a time, and stores them as tagged partial sums
        const int quarter = warp - 4;
        const bool have = mbar_wait_mk(&S.acc_full, li & 1, P, DEV_TIMEOUT_MMA);
        if (warp == 4 && lane == 0) stamp_at(st, 5);
        tc_fence_after();
        const int row = quarter * 32 + lane;
        if (have) {
            // eight token columns per TMEM load (a warp-wide access: every lane takes part)
            const bool mine = row < (lt ? P.lora_rows[lin] : TILE_ROWS);
            const int n_total = P.n_main[lin] + P.lora_rows[lin];
            unsigned long long *d = P.part[lin] + (size_t)s * P.part_rows * n_total + t * TILE_ROWS + row;
            const uint32_t taddr = tmem + ((uint32_t)(quarter * 32) << 16);
            if (P.pd.M <= 32) {  // one load of all token columns
                uint32_t v[32];
                tmem_ld_32cols(taddr, v);
                tmem_ld_wait();
                const int nc = mine ? P.pd.M : 0;
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    if (j < nc) st_tagged(d, v[j], tag);
                    d += n_total;
                }
            } else
#pragma unroll 1
            for (int c0 = 0; c0 < P.pd.M; c0 += 8) {
                uint32_t v[8];
                tmem_ld_8cols(taddr + (uint32_t)c0, v);
                tmem_ld_wait();
                const int nc = mine ? min(8, P.pd.M - c0) : 0;
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    if (j < nc) st_tagged(d, v[j], tag);
                    d += n_total;
                }
            }
        }
        tc_fence_before();
    }
    ++li;
    bar_compute();
    if (ct == 0) {
        stamp_at(st, 2);
        stamp_at(st, 6);
    }
    if (lt) {
        if (ct == 0) stamp_at(st, 7);
        return true;
    }
    const int ks = P.ks[lin];
    if (lin == 0)
        reduce_qkv<DH, DRAFT>(P, l, t, cw, lane, s, ks, tag, S.rowpos, S.rowkv, S.brows, st);
    else if (lin == 2)
        reduce_gu<DRAFT>(P, l, t, cw, lane, s, ks, tag, S.brows, st);
    else
        reduce_residual<DRAFT>(P, lin, l, t, cw, lane, s, ks, tag, S.brows, st);
    bar_compute();
    // one release per reduction, on the counters its consumers poll
    if (ct == 0) {
        release_item(P, it);
        stamp_at(st, 7);
    }
    return true;
}

// ---- compute group: a linear item's constants of the layer, requested before its inputs are
// ready (they depend on nothing computed in the pass): the RMSNorm gain of a normalised operand's
// K slice and, in the draft, the adapter's B rows of the tile, copied to shared memory (each thread
// waits for its own copies before the barrier that follows the input wait, which publishes them to
// the threads that read them); the QK-norm gains of the layer into L2.  The previous item's
// readers of these buffers passed a barrier before this is called.
template <bool DRAFT>
__device__ __forceinline__ void item_consts(const MKParams &P, const MKItem &it, CtaState &S, int ct) {
    const int lin = it.lin, l = it.layer, t = it.a;
    bool any = false;
    if (DRAFT && t < P.n_main[lin] / TILE_ROWS) {
        const int r = P.dm.r, cpr = r / 8;  // 16-byte chunks per B row
        const bf16 *lb = P.lora_b[lin] + (size_t)l * P.lb_stride[lin];
#pragma unroll 1
        for (int q = ct; q < TILE_ROWS * cpr; q += CT) {
            const int j = q / cpr, c = q % cpr;
            const int f = lin == 2 ? (j < 64 ? t * 64 + j : P.dm.I + t * 64 + (j - 64)) : t * TILE_ROWS + j;
            cp_async16(&S.brows[brow_chunk(j, r) + c], lb + (size_t)f * r + c * 8);
        }
        any = true;
    }
    if (lin == 0 || lin == 2) {
        const int n = P.katoms[lin] * (KT / 8);  // 16-byte chunks of the slice's gain
        const bf16 *g = (lin == 0 ? P.attn_norm : P.mlp_norm) + (size_t)l * P.dm.H + (size_t)it.b * n * 8;
        if (ct < n) cp_async16(&S.gain[ct], g + ct * 8);
        any = true;
    }
    if (lin == 0 && ct < 2 * P.dm.d / 64) {  // the q and k gains: 128-byte lines
        const int kind = ct / (P.dm.d / 64), line = ct % (P.dm.d / 64);
        prefetch_l2((kind ? P.k_norm : P.q_norm) + (size_t)l * P.dm.d + line * 64);
    }
    if (any) cp_async_commit();
}

// ---- compute group (warps 2-7): dependency waits, operand staging, epilogues, reductions,
// attention; the attention's cached pages are requested by warp CT_PAGES / 32 while thread 0 polls
// the item's inputs
template <bool DRAFT, int DH>
__device__ __noinline__ void run_compute(const MKParams &P, const MKItem *my, int n_my, uint8_t *uni, uint32_t tmem,
                                         CtaState &S, int tid) {
    const int ct = tid - 64, cw = ct >> 5, lane = tid & 31, warp = tid >> 5;
    uint32_t li = 0, ai = 0, l8 = 0;
    unsigned long long *tr = P.trace ? P.trace + (size_t)MK_STAMPS * P.cta_off[blockIdx.x] : nullptr;
    bool att_pend = false;  // (that warp) pages requested for a split that has not waited
#pragma unroll 1
    for (int i = 0; i < n_my; ++i) {
        const MKItem it = my[i];
        unsigned long long *st = tr ? tr + MK_STAMPS * i : nullptr;
        if (tr && ct == 0) {
            const unsigned long long now = globaltimer_ns();
            if (i > 0) tr[MK_STAMPS * (i - 1) + 3] = now;
            st[0] = now;
        }
        const bool att_active =
            it.op == MK_ATTN && it.c * P.pd.att_span * ATT_SPLIT < P.L[P.pd.b0 + it.a] + P.pd.R;
        if (att_active && cw == CT_PAGES / 32) {
            // pages below the cached length do not depend on this pass: fetch them now (the
            // barrier after the input wait orders this before the split's arrival)
            attn_pages(P, it.layer, it.a, it.b, it.c, 0, uni, &S.att_bar, lane);
            att_pend = true;
        }
        if (it.op == MK_LINEAR) item_consts<DRAFT>(P, it, S, ct);
        if (ct == 0) S.flag = wait_deps(P, it) ? 1 : 0;
        cp_async_wait_all();  // the constants each thread requested, published by the barrier
        bar_compute();
        if (!S.flag) break;
        if (ct == 0 && st) st[1] = st[2] = globaltimer_ns();
        bool ok = true;
        if (it.op == MK_LINEAR) {
            ok = item_linear<DRAFT, DH>(P, it, uni, tmem, S, li, l8, ct, cw, lane, warp, st);
        } else if (it.op == MK_ATTN) {
            ok = item_attn<DRAFT, DH>(P, it, att_active, uni, S, ai, ct, cw, lane, st);
            if (att_active) att_pend = false;
        } else if (it.op == MK_EMBED) {
            do_embed(P, it.a, cw, lane);
            bar_compute();
            if (ct == 0) release_item(P, it);
        } else {
            item_final(P, it, ct, S);
        }
        if (!ok) break;
    }
    cp_async_wait_all();  // an item left on abort may have requested its constants
    if (tr && ct == 0 && n_my > 0) tr[MK_STAMPS * (n_my - 1) + 3] = globaltimer_ns();
    if (ct == CT_PAGES && att_pend) {
        // the pass ended before the split waited for its pages: complete the phase's arrival and
        // let the copies land (bounded) before the shared memory is released
        mbarrier_arrive_one(&S.att_bar);
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(smem_u32(&S.att_bar), ai & 1) && globaltimer_ns() - t0 < WAIT_LIMIT_NS) {
        }
    }
}

// DRAFT: the adapter-on pass with the block-diffusion mask; otherwise adapter off and causal.
// One instantiation per kind keeps each kernel's code and registers to what that pass runs.
template <bool DRAFT, int DH>
__global__ void __launch_bounds__(MK_THREADS, 1) k_pass(const __grid_constant__ MKParams P) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *ring = base;
    uint8_t *uni = base + P.ring_bytes;  // activation tile / attention staging
    __shared__ CtaState S;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const MKItem *my = P.items + P.cta_off[blockIdx.x];
    const int n_my = P.cta_off[blockIdx.x + 1] - P.cta_off[blockIdx.x];

    if (tid == 0) {
        // the previous pass on this stream has finished: its counter advance is visible. Layer l
        // of this pass tags its partials S.tag + l; the buffers are reused by every layer and
        // pass, so a tag identifies both (acquire: read before the arrival below)
        S.tag = (uint32_t)ld_acquire(P.epoch) + 1u;
        atomicAdd(P.cnt + MK_STARTED, 1);
        for (int i = 0; i < P.nslot; ++i) {
            mbar_init(&S.full[i], 1);
            mbar_init(&S.empty[i], 1);
        }
        mbar_init(&S.b_full[0], 1);
        mbar_init(&S.b_full[1], 1);
        mbar_init(&S.b_empty, 1);
        mbar_init(&S.acc_full, 1);
        mbar_init(&S.att_bar, 1);
        mbar_init(&S.mma_drain, 1);
        prefetch_tensormap(&P.kmap);
        prefetch_tensormap(&P.vmap);
        fence_mbarrier_init();
    }
    if (warp == 0) tmem_alloc(&S.tmem_slot, P.tmem_cols);
    for (int m = tid; m < P.pd.M; m += MK_THREADS) {
        const int b = P.pd.b0 + m / P.pd.R, pos = P.L[b] + m % P.pd.R, pg = pos / PAGE;
        S.rowpos[m] = pos < P.rope_rows ? pos : -1;
        S.rowkv[m] = pg < P.kv.pages_per_seq ? (P.kv.page_table[b * P.kv.pages_per_seq + pg] << 4) | (pos % PAGE) : -1;
    }
    // zero the padding rows of the activation tile once (rows >= M are never written)
    for (int q = tid; q < (P.b_dbl ? MAX_ATOMS : HALF_ATOMS) * P.bn * 8; q += MK_THREADS) {
        const int atom = q / (P.bn * 8), rem = q % (P.bn * 8), m = rem / 8;
        if (m >= P.pd.M) *reinterpret_cast<uint4 *>(uni + (size_t)atom * P.bn * 128 + rem * 16) = make_uint4(0, 0, 0, 0);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = S.tmem_slot;
    if (warp == 0) {
        if (lane == 0) run_producer(P, my, n_my, ring, S);
    } else if (warp == 1) {
        if (lane == 0) run_mma(P, my, n_my, ring, uni, tmem, S);
    } else {
        run_compute<DRAFT, DH>(P, my, n_my, uni, tmem, S, tid);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, P.tmem_cols);
    if (blockIdx.x == 0 && tid == 0) {
        // once every CTA has read the pass counter (bounded), advance it for the next pass
        const uint64_t t0 = globaltimer_ns();
        while (ld_relaxed(P.cnt + MK_STARTED) < (int)gridDim.x && globaltimer_ns() - t0 < WAIT_LIMIT_NS) {
        }
        asm volatile("st.relaxed.gpu.global.b32 [%0], %1;" ::"l"(P.epoch), "r"((int)(S.tag + P.dm.nl - 1)) : "memory");
    }
}

// ------------------------------------------------------------------ host side

static int g_num_sms = 0, g_smem_optin = 0;

static cudaError_t device_limits() {
    if (g_num_sms) return cudaSuccess;
    int dev;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    return cudaDeviceGetAttribute(&g_smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
}

int mk_grid_size() {
    return device_limits() == cudaSuccess ? g_num_sms : 0;
}

void mk_counter_layout(const Dims &dm, int max_nb, CounterLayout *cl) {
    cl->embed = 0;
    cl->global = 4;
    cl->res_o = 0;
    cl->res_dn = cl->res_o + 1;
    cl->att = cl->res_dn + 1;
    cl->att_in = cl->att + max_nb * dm.Hkv;
    cl->att_o = cl->att_in + dm.Hkv;
    cl->per_layer = cl->att_o + (dm.Hq * dm.d + 255) / 256;
    cl->total = cl->global + dm.nl * cl->per_layer;
}

// Topologically ordered item list, dealt round-robin over `grid` CTAs (CTA i takes items
// i, i+grid, ...), so each CTA's list is in dependency order.  Returns items sorted by CTA.
// Every item carries the one counter it waits for and the counters it adds to once done:
//   embed row       -> embed counter (target M for layer 0's q|k|v)
//   q|k|v slice     waits for the previous layer run's residual after down (8 tiles x 12 slices at
//                   0.6B) or the embeddings; its reduction counts on att_in of each KV group it feeds
//   attention split waits for att_in of its group (every slice of every q, k, v tile of the
//                   group); the (sequence, group) merge counter orders the split's own merge, and a
//                   finished merge counts on att_o of the o slice that reads the group
//   o slice         waits for att_o (every merge of every sequence's groups in the slice); its
//                   reduction counts on res_o
//   gate|up slice   waits for res_o (every o tile slice); its reduction writes tagged act words
//   down slice      waits for nothing (its staging polls the act words); counts on res_dn
//   final norm row  waits for res_dn of the last layer run.
void mk_build_schedule(const Dims &dm, const PassDesc &pd, const std::vector<int> &nsplit, int grid,
                       const CounterLayout &cl, std::vector<MKItem> *out, std::vector<int> *off) {
    std::vector<MKItem> all;
    auto push = [&](uint8_t op, uint8_t lin, int layer, int a, int b, int c, int wait_off, int wait_tgt, int rel0,
                    int rel1) {
        MKItem it;
        it.op = op;
        it.lin = lin;
        it.layer = (uint16_t)layer;
        it.a = a;
        it.b = b;
        it.c = c;
        it.wait_off = wait_off;
        it.wait_tgt = wait_tgt;
        it.rel[0] = rel0;
        it.rel[1] = rel1;
        all.push_back(it);
    };
    const int nq = (dm.Hq + 2 * dm.Hkv) * dm.d / TILE_ROWS;
    const int n_main[4] = {nq, dm.H / TILE_ROWS, 2 * dm.I / TILE_ROWS, dm.H / TILE_ROWS};
    const int K[4] = {dm.H, dm.Hq * dm.d, dm.H, dm.I};
    int ks[4];
    for (int lin = 0; lin < 4; ++lin) ks[lin] = K[lin] / (mk_slice_atoms(lin, K[lin]) * KT);
    const int grp = dm.Hq / dm.Hkv, qw = dm.Hq * dm.d, kvw = dm.Hkv * dm.d, gw = grp * dm.d;
    auto ctr = [&](int layer, int o) { return cl.global + layer * cl.per_layer + o; };
    // KV groups a q|k|v tile feeds
    auto tile_groups = [&](int t, int *g0, int *g1) {
        const int f0 = t * TILE_ROWS, f1 = f0 + TILE_ROWS - 1;
        if (f0 < qw) {
            *g0 = f0 / gw;
            *g1 = f1 / gw;
        } else {
            const int base = f0 < qw + kvw ? qw : qw + kvw;
            *g0 = (f0 - base) / dm.d;
            *g1 = (f1 - base) / dm.d;
        }
    };
    // reduced slices an attention item of group g waits for
    std::vector<int> att_in_tgt(dm.Hkv, 0);
    for (int t = 0; t < nq; ++t) {
        int g0, g1;
        tile_groups(t, &g0, &g1);
        for (int g = g0; g <= g1; ++g) att_in_tgt[g] += ks[0];
    }
    // attention items per sequence (each covers att_span consecutive 128-key splits) and merges per
    // (sequence, group): every item when the items sit on distinct CTAs, else the last
    const int span = pd.att_span;
    int merges = 0;
    for (int bl = 0; bl < pd.nb; ++bl) {
        const int items = (nsplit[bl] + span - 1) / span;
        merges += items <= grid ? items : 1;
    }
    const int o_w = mk_slice_atoms(1, K[1]) * KT;  // o slice width
    for (int m = 0; m < pd.M; ++m) push(MK_EMBED, 0, 0, m, 0, 0, -1, 0, cl.embed, -1);
    int prev = -1;  // the last layer run so far (skipped layers have no items)
    for (int l = 0; l < pd.nl_run; ++l) {
        if (l < 64 && ((pd.skip >> l) & 1u)) continue;
        auto linear = [&](int lin, int wait_off, int wait_tgt) {
            for (int r = 0; r < (pd.adapter ? 1 : 0) + n_main[lin]; ++r) {
                const int t = pd.adapter ? (r == 0 ? n_main[lin] : r - 1) : r;  // adapter tile first
                int rel0 = -1, rel1 = -1;
                if (t < n_main[lin]) {
                    if (lin == 0) {
                        int g0, g1;
                        tile_groups(t, &g0, &g1);
                        rel0 = ctr(l, cl.att_in + g0);
                        rel1 = g1 != g0 ? ctr(l, cl.att_in + g1) : -1;
                    } else if (lin == 1) {
                        rel0 = ctr(l, cl.res_o);
                    } else if (lin == 3) {
                        rel0 = ctr(l, cl.res_dn);
                    }
                }
                for (int sl = 0; sl < ks[lin]; ++sl) push(MK_LINEAR, lin, l, t, sl, 0, wait_off, wait_tgt, rel0, rel1);
            }
        };
        if (prev < 0)
            linear(0, cl.embed, pd.M);
        else
            linear(0, ctr(prev, cl.res_dn), n_main[3] * ks[3]);
        prev = l;
        for (int bl = 0; bl < pd.nb; ++bl)
            for (int g = 0; g < dm.Hkv; ++g)
                for (int sp = 0; sp < (nsplit[bl] + span - 1) / span; ++sp)
                    push(MK_ATTN, 0, l, bl, g, sp, ctr(l, cl.att_in + g), att_in_tgt[g], ctr(l, cl.att_o + g * gw / o_w),
                         -1);
        // o slice sl reads the heads of the groups g with g * gw / o_w == sl
        for (int r = 0; r < (pd.adapter ? 1 : 0) + n_main[1]; ++r) {
            const int t = pd.adapter ? (r == 0 ? n_main[1] : r - 1) : r;
            for (int sl = 0; sl < ks[1]; ++sl) {
                int groups = 0;
                for (int g = 0; g < dm.Hkv; ++g) groups += (g * gw / o_w == sl) ? 1 : 0;
                push(MK_LINEAR, 1, l, t, sl, 0, ctr(l, cl.att_o + sl), groups * merges,
                     t < n_main[1] ? ctr(l, cl.res_o) : -1, -1);
            }
        }
        linear(2, ctr(l, cl.res_o), n_main[1] * ks[1]);
        linear(3, -1, 0);
    }
    for (int bl = 0; bl < pd.nb; ++bl)
        for (int i = pd.ro_first; i < pd.ro_first + pd.ro_count; ++i)
            push(MK_FINAL, 0, prev, bl * pd.ro_count + (i - pd.ro_first), bl * pd.R + i, 0, ctr(prev, cl.res_dn),
                 n_main[3] * ks[3], -1, -1);
    off->assign(grid + 1, 0);
    for (size_t i = 0; i < all.size(); ++i) (*off)[i % grid + 1]++;
    for (int c = 0; c < grid; ++c) (*off)[c + 1] += (*off)[c];
    out->resize(all.size());
    std::vector<int> fill(off->begin(), off->end() - 1);
    for (size_t i = 0; i < all.size(); ++i) (*out)[fill[i % grid]++] = all[i];
}

// 64-wide K atoms per item of linear `lin`: gate|up takes 512-wide slices (half as many items,
// so that one pass's gate|up items fit one per CTA), the others 256-wide
int mk_slice_atoms(int lin, int K) { return (lin == 2 && K % (MAX_ATOMS * KT) == 0) ? MAX_ATOMS : HALF_ATOMS; }

size_t mk_union_bytes(int bn, int head_dim, int att_span) {
    const size_t b = (size_t)HALF_ATOMS * bn * 128;
    const size_t att = (size_t)att_span * 2 * (head_dim / 64) * ATT_SUB_BYTES;
    return std::max(b, att);
}

cudaError_t launch_pass_kernel(const MKLaunch &L, cudaStream_t st) {
    cudaError_t e = device_limits();
    if (e != cudaSuccess) return e;
    MKParams P;
    P.kmap = *L.kmap;
    P.vmap = *L.vmap;
    P.dm = L.dm;
    P.pd = L.pd;
    if (L.pd.nl_run < 1 || L.pd.nl_run > L.dm.nl) return cudaErrorInvalidValue;
    P.items = L.items;
    P.cta_off = L.cta_off;
    P.cnt = L.cnt;
    P.cl = L.cl;
    P.nsplit = L.nsplit;
    for (int i = 0; i < 4; ++i) {
        P.wt[i] = static_cast<const uint8_t *>(L.wt[i]);
        P.wt_stride[i] = L.wt_stride[i];
        P.n_main[i] = L.n_main[i];
        P.lora_rows[i] = L.lora_rows[i];
        P.K[i] = L.K[i];
        P.katoms[i] = mk_slice_atoms(i, L.K[i]);
        P.ks[i] = L.K[i] / (P.katoms[i] * KT);
        // a tile's K slices wait for one another, so each must sit on its own CTA
        if (P.ks[i] > L.grid) return cudaErrorInvalidConfiguration;
        P.lora_b[i] = static_cast<const bf16 *>(L.lora_b[i]);
        P.lb_stride[i] = L.lb_stride[i];
        P.part[i] = L.part[i];
        P.epoch = L.epoch;
    }
    P.attn_norm = static_cast<const bf16 *>(L.attn_norm);
    P.mlp_norm = static_cast<const bf16 *>(L.mlp_norm);
    P.q_norm = static_cast<const bf16 *>(L.q_norm);
    P.k_norm = static_cast<const bf16 *>(L.k_norm);
    P.final_norm = static_cast<const bf16 *>(L.final_norm);
    P.mask_embed = static_cast<const bf16 *>(L.mask_embed);
    P.embed_tiled = static_cast<const bf16 *>(L.embed_tiled);
    P.rope_cs = L.rope_cs;
    P.rope_rows = L.rope_rows;
    P.kv = L.kv;
    P.L = L.Lbuf;
    P.ids = L.ids;
    P.part_rows = L.part_rows;
    P.h = static_cast<bf16 *>(L.h);
    P.q = static_cast<bf16 *>(L.q);
    P.attn = static_cast<bf16 *>(L.attn);
    P.act = static_cast<unsigned long long *>(L.act);
    P.x_ro = static_cast<bf16 *>(L.x_ro);
    P.ss = L.ss;
    P.o_part = L.o_part;
    P.ml_part = L.ml_part;
    P.att_splits_alloc = L.att_splits_alloc;
    P.att_subs = L.att_subs;
    if (L.att_subs < 1 || L.att_subs > ATT_SUBS_MAX) return cudaErrorInvalidValue;
    P.att_scale = (float)(1.0 / std::sqrt((double)L.dm.d));
    P.status = L.status;
    P.trace = L.trace;
    P.abort = L.abort;
    P.bn = ((L.pd.M + 31) / 32) * 32;
    if (P.bn > MAX_ROWS || L.pd.M > MAX_ROWS) return cudaErrorInvalidValue;
    P.tmem_cols = 32;
    while ((int)P.tmem_cols < P.bn) P.tmem_cols <<= 1;
    if (L.pd.att_span < 1 || L.pd.att_span > ATT_SPAN_MAX) return cudaErrorInvalidValue;
    const size_t uni = mk_union_bytes(P.bn, L.dm.d, L.pd.att_span);
    const size_t static_smem = sizeof(CtaState) + 1024;
    const long avail = (long)g_smem_optin - (long)uni - 1024 - (long)static_smem;
    // a shallow ring: what shared memory does not take stays L1 cache, which the compute warps
    // stack frames, spills and read-only loads need more than the weight stream needs depth
    P.nslot = (int)std::min<long>(RING_SLOTS, avail / TILE_BYTES);
    if (P.nslot < 2) return cudaErrorInvalidValue;
    P.ring_bytes = P.nslot * TILE_BYTES;
    P.union_bytes = (int)uni;
    P.b_dbl = (size_t)MAX_ATOMS * P.bn * 128 <= uni ? 1 : 0;
    const size_t dyn = (size_t)P.ring_bytes + uni + 1024;
    // the two pass kinds the kernel is built for
    const bool draft = L.pd.adapter != 0;
    if (draft != (L.pd.mask_mode == MASK_BLOCK_DRAFT)) return cudaErrorInvalidValue;
    static size_t configured = 0;
    if (dyn > configured) {
        e = cudaFuncSetAttribute(k_pass<true, 128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
        if (e == cudaSuccess) e = cudaFuncSetAttribute(k_pass<false, 128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
        if (e == cudaSuccess) e = cudaFuncSetAttribute(k_pass<true, 64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
        if (e == cudaSuccess) e = cudaFuncSetAttribute(k_pass<false, 64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
        if (e != cudaSuccess) return e;
        configured = dyn;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(L.grid);
    cfg.blockDim = dim3(MK_THREADS);
    cfg.dynamicSmemBytes = dyn;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (L.dm.d == 128)
        return draft ? cudaLaunchKernelEx(&cfg, k_pass<true, 128>, P) : cudaLaunchKernelEx(&cfg, k_pass<false, 128>, P);
    return draft ? cudaLaunchKernelEx(&cfg, k_pass<true, 64>, P) : cudaLaunchKernelEx(&cfg, k_pass<false, 64>, P);
}

}  // namespace pbd
