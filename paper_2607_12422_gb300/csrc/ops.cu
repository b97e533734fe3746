// ops.cu -- the non-contraction steps of a PEFT-BD pass, each fused into the consumer of a
// linear's split-K partial sums:
//   k_embed_norm      token / mask-embedding rows -> residual h, RMSNorm -> x
//   k_qkv_finalize    q|k|v = bf16(sum of splits + s * u B^T); per-head RMSNorm of q and k,
//                     rotate-half RoPE, k and v written to their paged cache slots
//   k_residual_norm   h = bf16(h + bf16(sum + s * u B^T)); x = RMSNorm(h) * gain
//   k_act             act = bf16(silu(gate) * up) from the fused gate|up sums (+ adapter)
//   k_build_ids       row token ids of a draft / verify / decode pass from the device state
//   k_accept_commit   longest accepted prefix, emission, KV commit (Section 3, steps 4-5)
// All elementwise arithmetic uses explicitly rounded fp32 operations (no contraction into
// FMA) and rounds every hand-off to bf16, the precision contract of a bf16 model (Section 4.1).
#include "common.cuh"
#include "pbd_internal.h"

namespace pbd {

// Fixed-order block sum of one float per thread (warp butterflies, then warps in order).
template <int NT>
__device__ __forceinline__ float block_sum(float v, float *red) {
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, off));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) red[warp] = v;
    __syncthreads();
    float t = red[0];
#pragma unroll
    for (int w = 1; w < NT / 32; ++w) t = __fadd_rn(t, red[w]);
    __syncthreads();
    return t;
}

__device__ __forceinline__ float rms_scale(float ss, int dim, float eps) {
    return __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(__fdiv_rn(ss, (float)dim), eps)));
}

// bf16 element (row v, col k) of a matrix stored in the 128 x 64 swizzled tile layout
__device__ __forceinline__ const bf16 *tiled_elem(const bf16 *tiles, int K, int v, int k) {
    const int t = v >> 7, r = v & 127, kt = k >> 6, c = (k & 63) >> 3, e = k & 7;
    return tiles + ((size_t)t * (K >> 6) + kt) * (TILE_ROWS * KT) + r * KT + ((c ^ (r & 7)) << 3) + e;
}

constexpr int ROW_THREADS = 256;
constexpr int MAX_PER_THREAD = 16;  // hidden sizes up to 4096

__global__ void __launch_bounds__(ROW_THREADS)
    k_embed_norm(Dims dm, PassDesc pd, const int *__restrict__ ids, const bf16 *__restrict__ embed_tiled,
                 const bf16 *__restrict__ mask_embed, const bf16 *__restrict__ gain, bf16 *__restrict__ h,
                 bf16 *__restrict__ x, int *status) {
    __shared__ float red[ROW_THREADS / 32];
    const int m = blockIdx.x;
    int tok = ids[m];
    if (tok >= dm.V) {
        latch_error(status, DEV_BAD_TOKEN);
        tok = 0;
    }
    const int H = dm.H;
    float hv[MAX_PER_THREAD];
    float ss = 0.f;
#pragma unroll
    for (int j = 0; j < MAX_PER_THREAD; ++j) {
        const int f = threadIdx.x + j * ROW_THREADS;
        if (f < H) {
            const float v = tok >= 0 ? bf2f(*tiled_elem(embed_tiled, H, tok, f)) : bf2f(mask_embed[f]);
            hv[j] = v;
            h[(size_t)m * H + f] = f2bf(v);
            ss = __fadd_rn(ss, __fmul_rn(v, v));
        }
    }
    ss = block_sum<ROW_THREADS>(ss, red);
    const float r = rms_scale(ss, H, dm.eps);
#pragma unroll
    for (int j = 0; j < MAX_PER_THREAD; ++j) {
        const int f = threadIdx.x + j * ROW_THREADS;
        if (f < H) x[(size_t)m * H + f] = f2bf(__fmul_rn(bf2f(gain[f]), rbf(__fmul_rn(hv[j], r))));
    }
}

cudaError_t launch_embed_norm(const Dims &dm, const PassDesc &pd, const int *ids, const void *embed_tiled,
                              const void *mask_embed, const void *gain, void *h, void *x, int *status,
                              cudaStream_t st) {
    if (dm.H > ROW_THREADS * MAX_PER_THREAD) return cudaErrorInvalidValue;
    k_embed_norm<<<pd.M, ROW_THREADS, 0, st>>>(dm, pd, ids, static_cast<const bf16 *>(embed_tiled),
                                               static_cast<const bf16 *>(mask_embed), static_cast<const bf16 *>(gain),
                                               static_cast<bf16 *>(h), static_cast<bf16 *>(x), status);
    return cudaGetLastError();
}

// Sum of the k_splits partials of (row m, feature f) in split order.
__device__ __forceinline__ float sum_splits(const Partials &P, int m, int f) {
    float a = P.p[(size_t)m * P.n_total + f];
    for (int s = 1; s < P.k_splits; ++s) a = __fadd_rn(a, P.p[((size_t)s * P.rows_alloc + m) * P.n_total + f]);
    return a;
}

// Adapter contribution of one output feature: sum_j u_j * B[f, j] (fp32, j in order).
__device__ __forceinline__ float lora_dot(const float *u, const bf16 *Brow, int r) {
    float a = 0.f;
    for (int j = 0; j < r; ++j) a = __fadd_rn(a, __fmul_rn(u[j], bf2f(Brow[j])));
    return a;
}

constexpr int MAX_R = 64;

// One warp per (row, head item); head items: Hq query heads, Hkv key heads, Hkv value heads.
template <int DH>
__global__ void __launch_bounds__(128)
    k_qkv_finalize(Dims dm, PassDesc pd, int layer, Partials P, const bf16 *__restrict__ lora_b,
                   const bf16 *__restrict__ q_norm, const bf16 *__restrict__ k_norm, const float2 *__restrict__ rope_cs,
                   int rope_rows, const int *__restrict__ Lbuf, KVCache kv, bf16 *__restrict__ q_out, int *status) {
    constexpr int E = DH / 32;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int hi = blockIdx.y * 4 + warp;
    const int Hq = dm.Hq, Hkv = dm.Hkv, r = dm.r;
    if (hi >= Hq + 2 * Hkv) return;
    const int m = blockIdx.x;
    const int b = pd.b0 + m / pd.R;
    const int pos = Lbuf[b] + m % pd.R;
    const int kind = hi < Hq ? 0 : (hi < Hq + Hkv ? 1 : 2);
    const int head = kind == 0 ? hi : (kind == 1 ? hi - Hq : hi - Hq - Hkv);
    const int fbase = kind == 0 ? hi * DH : (kind == 1 ? Hq * DH + head * DH : (Hq + Hkv) * DH + head * DH);
    const int n_main = (Hq + 2 * Hkv) * DH;

    float u[MAX_R];
    if (pd.adapter) {
        const float mine = lane < r ? rbf(sum_splits(P, m, n_main + kind * r + lane)) : 0.f;
        for (int j = 0; j < r; ++j) u[j] = __shfl_sync(0xffffffffu, mine, j & 31);
    }
    float y[E];
#pragma unroll
    for (int j = 0; j < E; ++j) {
        const int f = fbase + lane + 32 * j;
        float acc = sum_splits(P, m, f);
        if (pd.adapter) acc = __fadd_rn(acc, __fmul_rn(dm.lora_scale, lora_dot(u, lora_b + (size_t)f * r, r)));
        y[j] = rbf(acc);
    }
    if (kind < 2) {
        const bf16 *gn = (kind == 0 ? q_norm : k_norm) + (size_t)layer * DH;
        float ss = 0.f;
#pragma unroll
        for (int j = 0; j < E; ++j) ss = __fadd_rn(ss, __fmul_rn(y[j], y[j]));
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) ss = __fadd_rn(ss, __shfl_xor_sync(0xffffffffu, ss, off));
        const float rs = rms_scale(ss, DH, dm.eps);
#pragma unroll
        for (int j = 0; j < E; ++j) y[j] = rbf(__fmul_rn(bf2f(gn[lane + 32 * j]), rbf(__fmul_rn(y[j], rs))));
        if (pos >= rope_rows) {
            latch_error(status, DEV_BAD_POSITION);
            return;
        }
        // rotate-half RoPE: element e pairs with e + DH/2, both held by this lane
#pragma unroll
        for (int j = 0; j < E / 2; ++j) {
            const int e = lane + 32 * j;
            const float2 cs = rope_cs[(size_t)pos * (DH / 2) + e];
            const float a = y[j], c = y[j + E / 2];
            y[j] = rbf(__fsub_rn(__fmul_rn(a, cs.x), __fmul_rn(c, cs.y)));
            y[j + E / 2] = rbf(__fadd_rn(__fmul_rn(c, cs.x), __fmul_rn(a, cs.y)));
        }
    }
    if (kind == 0) {
        bf16 *dst = q_out + ((size_t)m * Hq + head) * DH;
#pragma unroll
        for (int j = 0; j < E; ++j) dst[lane + 32 * j] = f2bf(y[j]);
    } else {
        const int pg = pos / PAGE;
        if (pg >= kv.pages_per_seq) {
            latch_error(status, DEV_BAD_POSITION);
            return;
        }
        const int page = kv.page_table[b * kv.pages_per_seq + pg];
        const size_t off = ((((size_t)layer * kv.n_pages + page) * Hkv + head) * PAGE + (pos % PAGE)) * DH;
        bf16 *dst = static_cast<bf16 *>(kind == 1 ? kv.k : kv.v) + off;
#pragma unroll
        for (int j = 0; j < E; ++j) dst[lane + 32 * j] = f2bf(y[j]);
    }
}

cudaError_t launch_qkv_finalize(const Dims &dm, const PassDesc &pd, int layer, const Partials &part,
                                const void *lora_b_qkv, const void *q_norm, const void *k_norm,
                                const float2 *rope_cs, int rope_rows, const int *L, const KVCache &kv, void *q_out,
                                int *status, cudaStream_t st) {
    if (dm.r > MAX_R) return cudaErrorInvalidValue;
    dim3 grid(pd.M, (dm.Hq + 2 * dm.Hkv + 3) / 4);
    const bf16 *lb = static_cast<const bf16 *>(lora_b_qkv);
    if (dm.d == 128)
        k_qkv_finalize<128><<<grid, 128, 0, st>>>(dm, pd, layer, part, lb, static_cast<const bf16 *>(q_norm),
                                                 static_cast<const bf16 *>(k_norm), rope_cs, rope_rows, L, kv,
                                                 static_cast<bf16 *>(q_out), status);
    else if (dm.d == 64)
        k_qkv_finalize<64><<<grid, 128, 0, st>>>(dm, pd, layer, part, lb, static_cast<const bf16 *>(q_norm),
                                                static_cast<const bf16 *>(k_norm), rope_cs, rope_rows, L, kv,
                                                static_cast<bf16 *>(q_out), status);
    else
        return cudaErrorInvalidValue;
    return cudaGetLastError();
}

// One CTA per row: residual add of the linear's output (+ adapter), then RMSNorm for the next block.
__global__ void __launch_bounds__(ROW_THREADS)
    k_residual_norm(Dims dm, PassDesc pd, Partials P, int n_out, const bf16 *__restrict__ lora_b,
                    const bf16 *__restrict__ gain, bf16 *__restrict__ h, bf16 *__restrict__ x, bf16 *__restrict__ x_ro) {
    __shared__ float red[ROW_THREADS / 32];
    __shared__ float su[MAX_R];
    const int m = blockIdx.x;
    const int H = dm.H, r = dm.r;
    if (pd.adapter) {
        if ((int)threadIdx.x < r) su[threadIdx.x] = rbf(sum_splits(P, m, n_out + threadIdx.x));
        __syncthreads();
    }
    float hv[MAX_PER_THREAD];
    float ss = 0.f;
#pragma unroll
    for (int j = 0; j < MAX_PER_THREAD; ++j) {
        const int f = threadIdx.x + j * ROW_THREADS;
        if (f < H) {
            float acc = sum_splits(P, m, f);
            if (pd.adapter) acc = __fadd_rn(acc, __fmul_rn(dm.lora_scale, lora_dot(su, lora_b + (size_t)f * r, r)));
            const float y = rbf(acc);
            const float hn = rbf(__fadd_rn(bf2f(h[(size_t)m * H + f]), y));
            hv[j] = hn;
            h[(size_t)m * H + f] = f2bf(hn);
            ss = __fadd_rn(ss, __fmul_rn(hn, hn));
        }
    }
    ss = block_sum<ROW_THREADS>(ss, red);
    const float rs = rms_scale(ss, H, dm.eps);
    const int i = m % pd.R;
    const int ro = (x_ro != nullptr && i >= pd.ro_first && i < pd.ro_first + pd.ro_count)
                       ? (m / pd.R) * pd.ro_count + (i - pd.ro_first)
                       : -1;
#pragma unroll
    for (int j = 0; j < MAX_PER_THREAD; ++j) {
        const int f = threadIdx.x + j * ROW_THREADS;
        if (f < H) {
            const bf16 v = f2bf(__fmul_rn(bf2f(gain[f]), rbf(__fmul_rn(hv[j], rs))));
            x[(size_t)m * H + f] = v;
            if (ro >= 0) x_ro[(size_t)ro * H + f] = v;
        }
    }
}

cudaError_t launch_residual_norm(const Dims &dm, const PassDesc &pd, const Partials &part, int n_out,
                                 const void *lora_b, const void *gain, void *h, void *x, void *x_ro,
                                 cudaStream_t st) {
    if (dm.H > ROW_THREADS * MAX_PER_THREAD || dm.r > MAX_R) return cudaErrorInvalidValue;
    k_residual_norm<<<pd.M, ROW_THREADS, 0, st>>>(dm, pd, part, n_out, static_cast<const bf16 *>(lora_b),
                                                  static_cast<const bf16 *>(gain), static_cast<bf16 *>(h),
                                                  static_cast<bf16 *>(x), static_cast<bf16 *>(x_ro));
    return cudaGetLastError();
}

// SwiGLU on the fused gate|up partial sums: features [0, I) gate, [I, 2I) up; adapter rows
// [2I, 2I + r) belong to gate, [2I + r, 2I + 2r) to up.
__global__ void __launch_bounds__(ROW_THREADS)
    k_act(Dims dm, PassDesc pd, Partials P, const bf16 *__restrict__ lora_b, bf16 *__restrict__ act) {
    __shared__ float su[2 * MAX_R];
    const int m = blockIdx.x;
    const int I = dm.I, r = dm.r;
    if (pd.adapter) {
        if ((int)threadIdx.x < 2 * r) su[threadIdx.x] = rbf(sum_splits(P, m, 2 * I + threadIdx.x));
        __syncthreads();
    }
    const int f = blockIdx.y * ROW_THREADS + threadIdx.x;
    if (f >= I) return;
    float g = sum_splits(P, m, f);
    float u = sum_splits(P, m, I + f);
    if (pd.adapter) {
        g = __fadd_rn(g, __fmul_rn(dm.lora_scale, lora_dot(su, lora_b + (size_t)f * r, r)));
        u = __fadd_rn(u, __fmul_rn(dm.lora_scale, lora_dot(su + r, lora_b + (size_t)(I + f) * r, r)));
    }
    g = rbf(g);
    u = rbf(u);
    const float sg = __fdiv_rn(g, __fadd_rn(1.0f, expf(-g)));
    act[(size_t)m * I + f] = f2bf(__fmul_rn(sg, u));
}

cudaError_t launch_act(const Dims &dm, const PassDesc &pd, const Partials &part, const void *lora_b_gu, void *act,
                       cudaStream_t st) {
    if (dm.r > MAX_R) return cudaErrorInvalidValue;
    dim3 grid(pd.M, (dm.I + ROW_THREADS - 1) / ROW_THREADS);
    k_act<<<grid, ROW_THREADS, 0, st>>>(dm, pd, part, static_cast<const bf16 *>(lora_b_gu), static_cast<bf16 *>(act));
    return cudaGetLastError();
}

// Standalone linear epilogue: y = bf16(sum of splits + scale * u B^T), u = bf16(adapter rows).
__global__ void __launch_bounds__(ROW_THREADS)
    k_linear_finalize(Partials P, int N, int r, float scale, const bf16 *__restrict__ lora_b, bf16 *__restrict__ y) {
    __shared__ float su[MAX_R];
    const int m = blockIdx.x;
    if (r > 0) {
        if ((int)threadIdx.x < r) su[threadIdx.x] = rbf(sum_splits(P, m, N + threadIdx.x));
        __syncthreads();
    }
    const int f = blockIdx.y * ROW_THREADS + threadIdx.x;
    if (f >= N) return;
    float acc = sum_splits(P, m, f);
    if (r > 0) acc = __fadd_rn(acc, __fmul_rn(scale, lora_dot(su, lora_b + (size_t)f * r, r)));
    y[(size_t)m * N + f] = f2bf(acc);
}

cudaError_t launch_linear_finalize(const Partials &P, int M, int N, int r, float scale, const void *lora_b, void *y,
                                   cudaStream_t st) {
    if (r > MAX_R) return cudaErrorInvalidValue;
    dim3 grid(M, (N + ROW_THREADS - 1) / ROW_THREADS);
    k_linear_finalize<<<grid, ROW_THREADS, 0, st>>>(P, N, r, scale, static_cast<const bf16 *>(lora_b),
                                                    static_cast<bf16 *>(y));
    return cudaGetLastError();
}

// kind 0: draft rows [pending, -1 x D]; 1: verify rows [pending, d_1..d_D]; 2: decode [pending]
__global__ void k_build_ids(PassDesc pd, int kind, const int *__restrict__ pending, const int *__restrict__ drafts,
                            int D, int *__restrict__ ids) {
    const int m = blockIdx.x * blockDim.x + threadIdx.x;
    if (m >= pd.M) return;
    const int bl = m / pd.R, i = m % pd.R, b = pd.b0 + bl;
    int t;
    if (i == 0)
        t = pending[b];
    else if (kind == 0)
        t = -1;
    else
        t = drafts[bl * D + (i - 1)];
    ids[m] = t;
}

cudaError_t launch_build_ids(const PassDesc &pd, int kind, const int *pending, const int *drafts, int D, int *ids,
                             cudaStream_t st) {
    k_build_ids<<<(pd.M + 127) / 128, 128, 0, st>>>(pd, kind, pending, drafts, D, ids);
    return cudaGetLastError();
}

// Section 3, steps 4-5 on the device.  One thread per sequence.
__global__ void k_accept_commit(SeqState s, int nb, int D, const int *__restrict__ drafts,
                                const int *__restrict__ verify, const int *__restrict__ forced, int forced_stride,
                                int max_new, int out_cap, int *__restrict__ accepted_out) {
    const int b = threadIdx.x;
    const int round = *s.round;
    __syncthreads();
    if (b < nb) {
        if (s.done[b]) {
            if (accepted_out) accepted_out[b] = -1;
        } else {
            const int *d = drafts + (size_t)b * D;
            const int *v = verify + (size_t)b * (D + 1);
            int n = 0;
            while (n < D && d[n] == v[n]) ++n;
            if (forced != nullptr) n = min(max(forced[(size_t)round * forced_stride + b], 0), D);
            const int cnt = s.n_out[b];
            const int take = min(n + 1, max_new - cnt);
            for (int j = 0; j < take; ++j) s.out_tokens[(size_t)b * out_cap + cnt + j] = j < n ? d[j] : v[n];
            s.n_out[b] = cnt + take;
            s.L[b] += n + 1;
            s.pending[b] = v[n];
            if (cnt + take >= max_new) s.done[b] = 1;
            atomicAdd((unsigned long long *)&s.stats[0], 1ull);
            atomicAdd((unsigned long long *)&s.stats[1], (unsigned long long)n);
            atomicAdd((unsigned long long *)&s.stats[2], (unsigned long long)take);
            if (accepted_out) accepted_out[b] = n;
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int all = 1;
        for (int i = 0; i < nb; ++i) all &= s.done[i];
        *s.all_done = all;
        *s.round = round + 1;
    }
}

cudaError_t launch_accept_commit(const SeqState &s, int nb, int D, const int *drafts, const int *verify,
                                 const int *forced, int forced_stride, int max_new, int out_cap, int *accepted_out,
                                 cudaStream_t st) {
    const int threads = ((nb + 31) / 32) * 32;
    k_accept_commit<<<1, threads, 0, st>>>(s, nb, D, drafts, verify, forced, forced_stride, max_new, out_cap,
                                           accepted_out);
    return cudaGetLastError();
}

// Row-major [rows, K] bf16 -> 128 x 64 swizzled tiles; one 16-byte chunk per thread.
__global__ void k_repack_tiled(const uint4 *__restrict__ src, int rows, int K, bf16 *__restrict__ dst, int row0) {
    const size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int cpr = K / 8;
    if (idx >= (size_t)rows * cpr) return;
    const int i = (int)(idx / cpr), cg = (int)(idx % cpr);
    const int R = row0 + i;
    const int t = R >> 7, rr = R & 127, kt = cg >> 3, c = cg & 7;
    const size_t off = ((size_t)t * (K / KT) + kt) * (TILE_ROWS * KT) + rr * KT + ((c ^ (rr & 7)) << 3);
    *reinterpret_cast<uint4 *>(dst + off) = src[idx];
}

cudaError_t launch_repack_tiled(const void *src, int rows, int K, void *dst_tiles, int dst_row0, cudaStream_t st) {
    const size_t n = (size_t)rows * (K / 8);
    k_repack_tiled<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(static_cast<const uint4 *>(src), rows, K,
                                                                static_cast<bf16 *>(dst_tiles), dst_row0);
    return cudaGetLastError();
}

__global__ void k_read_kv(KVCache kv, int Hkv, int d, int layer, int seq, int n, bf16 *__restrict__ k_out,
                          bf16 *__restrict__ v_out) {
    const size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    const size_t per = (size_t)Hkv * d;
    if (idx >= (size_t)n * per) return;
    const int t = (int)(idx / per), rem = (int)(idx % per), g = rem / d, e = rem % d;
    const int page = kv.page_table[seq * kv.pages_per_seq + t / PAGE];
    const size_t off = ((((size_t)layer * kv.n_pages + page) * Hkv + g) * PAGE + (t % PAGE)) * d + e;
    k_out[idx] = static_cast<const bf16 *>(kv.k)[off];
    v_out[idx] = static_cast<const bf16 *>(kv.v)[off];
}

cudaError_t launch_read_kv(const Dims &dm, const KVCache &kv, int layer, int seq, int n, void *k_out, void *v_out,
                           cudaStream_t st) {
    const size_t total = (size_t)n * dm.Hkv * dm.d;
    if (total == 0) return cudaSuccess;
    k_read_kv<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(kv, dm.Hkv, dm.d, layer, seq, n,
                                                               static_cast<bf16 *>(k_out), static_cast<bf16 *>(v_out));
    return cudaGetLastError();
}

__global__ void k_set_len(int *L, int b, int value) { L[b] = value; }

__global__ void k_prefill_finish(SeqState s, int b, int P, const int *first_id, int max_new, int out_cap) {
    const int t = *first_id;
    s.L[b] = P;
    s.pending[b] = t;
    s.out_tokens[(size_t)b * out_cap] = t;
    s.n_out[b] = 1;
    s.done[b] = max_new <= 1 ? 1 : 0;
}

cudaError_t launch_prefill_finish(const SeqState &s, int b, int P, const int *first_id, int max_new, int out_cap,
                                  cudaStream_t st) {
    k_prefill_finish<<<1, 1, 0, st>>>(s, b, P, first_id, max_new, out_cap);
    return cudaGetLastError();
}

cudaError_t launch_set_len(int *L, int b, int value, cudaStream_t st) {
    k_set_len<<<1, 1, 0, st>>>(L, b, value);
    return cudaGetLastError();
}

}  // namespace pbd
