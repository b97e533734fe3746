// ops.cu -- small kernels around the persistent pass kernel:
//   k_build_ids       row token ids of a draft / verify / decode pass from the device state
//   k_accept_commit   longest accepted prefix, emission, KV commit (Section 3, steps 4-5)
//   k_prefill_finish  cached length and first token after a prompt
//   k_repack_tiled    row-major bf16 weights -> 128 x 64 tiles in the 128-byte swizzle layout
//   k_read_kv         paged cache -> contiguous rows (tests of the commit rule)
//   k_linear_finalize split-K sum + adapter delta of the standalone linear entry point
#include "common.cuh"
#include "pbd_internal.h"

namespace pbd {

constexpr int ROW_THREADS = 256;
constexpr int MAX_R = 64;

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

// Row-major [rows, K] bf16 -> 128 x 64 swizzled tiles; one 16-byte chunk per thread.  Source row
// i lands on tile row dst_row0 + (i / group) * stride + i % group (group == rows: contiguous).
__global__ void k_repack_tiled(const uint4 *__restrict__ src, int rows, int K, bf16 *__restrict__ dst, int row0,
                               int group, int stride) {
    const size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int cpr = K / 8;
    if (idx >= (size_t)rows * cpr) return;
    const int i = (int)(idx / cpr), cg = (int)(idx % cpr);
    const int R = row0 + (i / group) * stride + (i % group);
    const int t = R >> 7, rr = R & 127, kt = cg >> 3, c = cg & 7;
    const size_t off = ((size_t)t * (K / KT) + kt) * (TILE_ROWS * KT) + rr * KT + ((c ^ (rr & 7)) << 3);
    *reinterpret_cast<uint4 *>(dst + off) = src[idx];
}

cudaError_t launch_repack_tiled_map(const void *src, int rows, int K, void *dst_tiles, int dst_row0, int group,
                                    int stride, cudaStream_t st) {
    const size_t n = (size_t)rows * (K / 8);
    k_repack_tiled<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(static_cast<const uint4 *>(src), rows, K,
                                                                static_cast<bf16 *>(dst_tiles), dst_row0, group,
                                                                stride);
    return cudaGetLastError();
}

cudaError_t launch_repack_tiled(const void *src, int rows, int K, void *dst_tiles, int dst_row0, cudaStream_t st) {
    return launch_repack_tiled_map(src, rows, K, dst_tiles, dst_row0, rows, 0, st);
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

cudaError_t launch_set_len(int *L, int b, int value, cudaStream_t st) {
    k_set_len<<<1, 1, 0, st>>>(L, b, value);
    return cudaGetLastError();
}

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

}  // namespace pbd
