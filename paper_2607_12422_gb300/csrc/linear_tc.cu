// linear_tc.cu -- weight-streaming linear layers on the 5th-generation tensor core (sm_103a).
//
// Every projection of a decoder pass (q/k/v, o, gate/up, down, and the tied lm_head) is a
// skinny contraction: M = batch x (D+1) token rows (17 at batch 1, D = 16) against an
// [out, in] bf16 weight that is read exactly once per pass.  The kernel swaps the operands
// so the weight supplies the 128-row MMA dimension and the tokens the N dimension:
//     D[feature, token] += W[feature, k] * X[token, k]      (both K-major)
// Weights are pre-tiled in HBM as 128 x 64 tiles already in the 128-byte swizzle layout,
// so one 1-D bulk copy (TMA) per stage moves 16 KiB straight into the MMA's shared-memory
// operand.  Activations come through a 2-D TMA map (box 64 x BN, same swizzle).  One thread
// issues the copies, one thread issues tcgen05.mma into a TMEM accumulator, and all four
// warps read TMEM back for the epilogue.
//
// The split over K is fixed per linear and independent of M, and each output column of an
// MMA depends only on its own token row, so a row's result is bit-identical whatever the
// number of rows in the pass (batch invariance: verify row j == plain decode at that position).
//
// Epilogues:  EPI_PARTIAL writes fp32 split-K partial sums (the consumer kernel adds the
// splits in a fixed order, applies the adapter's B, rounds to bf16 and fuses the next step);
// EPI_ARGMAX is the lm_head: per 128-row vocabulary tile it writes the (max, argmax) of each
// token row, lowest index on ties, and optionally the fp32 logits.
#include "common.cuh"
#include "pbd_internal.h"

namespace pbd {

constexpr int LIN_THREADS = 128;
constexpr int NSTAGE = 4;
enum { EPI_PARTIAL = 0, EPI_ARGMAX = 1 };

template <int BN>
struct LinLayout {
    static constexpr int B_BYTES = BN * 128;
    static constexpr int A_OFF = 0;
    static constexpr int B_OFF = NSTAGE * TILE_BYTES;
    static constexpr int BAR_OFF = B_OFF + NSTAGE * B_BYTES;
    static constexpr int RED_OFF = BAR_OFF + 256;
    static constexpr int RED_BYTES = 4 * BN * 8;
    static constexpr int TOTAL = RED_OFF + RED_BYTES + 1024;  // + alignment slack
    static constexpr uint32_t TMEM_COLS = BN < 32 ? 32 : BN;
};

template <int BN, int EPI>
__global__ void __launch_bounds__(LIN_THREADS, 1)
    k_linear_tc(const __grid_constant__ CUtensorMap xmap, const uint8_t *__restrict__ wtiles, int k_tiles,
                int n_main_tiles, int lora_rows, int k_splits, int M, float *__restrict__ part, int rows_alloc,
                int n_total, float *__restrict__ tile_max, int *__restrict__ tile_arg, float *__restrict__ logits,
                int V, int *status) {
    using LY = LinLayout<BN>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sA = base + LY::A_OFF;
    uint8_t *sB = base + LY::B_OFF;
    uint64_t *full = reinterpret_cast<uint64_t *>(base + LY::BAR_OFF);
    uint64_t *empty = full + NSTAGE;
    uint64_t *done = empty + NSTAGE;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(done + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
    float *red_val = reinterpret_cast<float *>(base + LY::RED_OFF);
    int *red_idx = reinterpret_cast<int *>(red_val + 4 * BN);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tile = blockIdx.x, split = blockIdx.y, tok0 = blockIdx.z * BN;
    const bool lora_tile = tile >= n_main_tiles;
    const int rows_valid = lora_tile ? lora_rows : TILE_ROWS;
    const uint32_t a_bytes = (uint32_t)rows_valid * 128u;
    const int kt_per = k_tiles / k_splits;
    const int kt0 = split * kt_per;

    if (threadIdx.x == 0) {
        for (int s = 0; s < NSTAGE; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(done, 1);
        *abort_flag = 0;
        fence_mbarrier_init();
        prefetch_tensormap(&xmap);
    }
    if (warp == 0) tmem_alloc(tmem_slot, LY::TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // ---- producer: weight tile (bulk copy) + activation tile (tiled TMA) per stage
        const uint64_t pol = l2_policy_evict_first();
        const uint8_t *wsrc = wtiles + ((size_t)tile * k_tiles + kt0) * TILE_BYTES;
        int issued = 0;
        for (int s = 0; s < kt_per; ++s) {
            const int slot = s % NSTAGE;
            if (s >= NSTAGE &&
                !mbar_wait(&empty[slot], ((s / NSTAGE) - 1) & 1, status, DEV_TIMEOUT_SLOT, abort_flag))
                break;
            mbar_arrive_expect_tx(&full[slot], a_bytes + (uint32_t)LY::B_BYTES);
            bulk_g2s(sA + slot * TILE_BYTES, wsrc + (size_t)s * TILE_BYTES, a_bytes, &full[slot], pol);
            tma_load_2d(sB + slot * LY::B_BYTES, &xmap, (kt0 + s) * KT, tok0, &full[slot]);
            ++issued;
        }
        if (*abort_flag) {
            // error path: give the copies still in flight a bounded chance to land before exit
            for (int s = issued > NSTAGE ? issued - NSTAGE : 0; s < issued; ++s)
                mbar_wait(&full[s % NSTAGE], (s / NSTAGE) & 1, nullptr, 0, nullptr);
        }
    } else if (warp == 1 && lane == 0) {
        // ---- MMA issuer: 4 x (128 x BN x 16) per 64-wide stage into the TMEM accumulator
        const uint32_t idesc = idesc_bf16_f32(128, BN);
        bool ok = true;
        for (int s = 0; s < kt_per; ++s) {
            const int slot = s % NSTAGE;
            if (!mbar_wait(&full[slot], (s / NSTAGE) & 1, status, DEV_TIMEOUT_LOAD, abort_flag)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint64_t ad = sw128_kmajor_desc(sA + slot * TILE_BYTES);
            const uint64_t bd = sw128_kmajor_desc(sB + slot * LY::B_BYTES);
#pragma unroll
            for (int kk = 0; kk < KT / 16; ++kk)  // +32 bytes along K inside the swizzle atom
                mma_bf16_ss(tmem, ad + 2ull * kk, bd + 2ull * kk, idesc, (s | kk) != 0 ? 1u : 0u);
            mma_commit(&empty[slot]);
        }
        if (ok) mma_commit(done);
    }
    __syncwarp();

    // ---- epilogue: warp w owns TMEM lanes 32w..32w+31 = output features of the tile
    const bool have = mbar_wait(done, 0, status, DEV_TIMEOUT_MMA, abort_flag);
    tc_fence_after();
    const int row = warp * 32 + lane;
    const int feat = tile * TILE_ROWS + row;
    const uint32_t tbase = tmem + ((uint32_t)(warp * 32) << 16);
    if (have) {
        for (int c0 = 0; c0 < BN; c0 += 32) {
            if (tok0 + c0 >= M) break;  // uniform across the CTA
            uint32_t v[32];
            tmem_ld_32cols(tbase + (uint32_t)c0, v);
            tmem_ld_wait();
            if constexpr (EPI == EPI_PARTIAL) {
                if (row < rows_valid) {
                    float *dst = part + ((size_t)split * rows_alloc + tok0 + c0) * n_total + feat;
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (tok0 + c0 + j < M) dst[(size_t)j * n_total] = __uint_as_float(v[j]);
                }
            } else {
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    float bv = __uint_as_float(v[j]);
                    int bi = feat;
                    const int tok = tok0 + c0 + j;
                    if (logits != nullptr && tok < M) logits[(size_t)tok * V + feat] = bv;
#pragma unroll
                    for (int off = 16; off >= 1; off >>= 1) {
                        const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
                        const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
                        if (ov > bv || (ov == bv && oi < bi)) {
                            bv = ov;
                            bi = oi;
                        }
                    }
                    if (lane == 0) {
                        red_val[warp * BN + c0 + j] = bv;
                        red_idx[warp * BN + c0 + j] = bi;
                    }
                }
            }
        }
    }
    if constexpr (EPI == EPI_ARGMAX) {
        __syncthreads();
        for (int c = threadIdx.x; have && c < BN && tok0 + c < M; c += LIN_THREADS) {
            float bv = red_val[c];
            int bi = red_idx[c];
            for (int w = 1; w < 4; ++w) {
                const float ov = red_val[w * BN + c];
                const int oi = red_idx[w * BN + c];
                if (ov > bv || (ov == bv && oi < bi)) {
                    bv = ov;
                    bi = oi;
                }
            }
            tile_max[(size_t)tile * M + tok0 + c] = bv;
            tile_arg[(size_t)tile * M + tok0 + c] = bi;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, LY::TMEM_COLS);
}

// ------------------------------------------------------------------ persistent lm_head
//
// One CTA per SM walks vocabulary tiles t = blockIdx.x, + gridDim.x, ...: the token rows'
// activation operand (all K atoms) is loaded once and stays in shared memory, weight tiles
// stream through a ring across tile boundaries, and two TMEM accumulators let the argmax
// epilogue of one tile run under the MMAs of the next.  Warp 0 streams, warp 1 issues the
// MMAs, warps 2-5 (one per TMEM lane quarter) reduce each token row's (max, argmax) over the
// tile's 128 vocabulary rows, lowest index on ties, as k_linear_tc<BN, EPI_ARGMAX> does.
constexpr int LMH_THREADS = 192;
constexpr int LMH_STAGES = 4;

template <int BN>
struct LmhLayout {
    static constexpr int X_ATOM = BN * 128;  // one 64-wide K atom of the token rows
    static constexpr int RING_OFF = 0;
    static constexpr int X_OFF = LMH_STAGES * TILE_BYTES;
    static constexpr int MAX_ATOMS = 16;     // K <= 1024
    static constexpr int BAR_OFF = X_OFF + MAX_ATOMS * X_ATOM;
    static constexpr int RED_OFF = BAR_OFF + 256;
    static constexpr int RED_BYTES = 2 * 4 * BN * 8;  // [acc][quarter][token] (value, index)
    static constexpr int TOTAL = RED_OFF + RED_BYTES + 1024;
    static constexpr uint32_t TMEM_COLS = 2 * BN < 32 ? 32 : 2 * BN;
};

template <int BN>
__global__ void __launch_bounds__(LMH_THREADS, 1)
    k_lm_head(const __grid_constant__ CUtensorMap xmap, const uint8_t *__restrict__ wtiles, int k_tiles, int n_tiles,
              int M, float *__restrict__ tile_max, int *__restrict__ tile_arg, float *__restrict__ logits, int V,
              int *status) {
    using LY = LmhLayout<BN>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *ring = base + LY::RING_OFF;
    uint8_t *sx = base + LY::X_OFF;
    uint64_t *full = reinterpret_cast<uint64_t *>(base + LY::BAR_OFF);
    uint64_t *empty = full + LMH_STAGES;
    uint64_t *x_full = empty + LMH_STAGES;
    uint64_t *acc_full = x_full + 1;   // [2]
    uint64_t *acc_empty = acc_full + 2;  // [2]
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_empty + 2);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
    float *red_val = reinterpret_cast<float *>(base + LY::RED_OFF);
    int *red_idx = reinterpret_cast<int *>(red_val + 2 * 4 * BN);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_my = blockIdx.x < n_tiles ? (n_tiles - 1 - blockIdx.x) / gridDim.x + 1 : 0;

    if (threadIdx.x == 0) {
        for (int s = 0; s < LMH_STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(x_full, 1);
        mbar_init(&acc_full[0], 1);
        mbar_init(&acc_full[1], 1);
        mbar_init(&acc_empty[0], 1);
        mbar_init(&acc_empty[1], 1);
        *abort_flag = 0;
        fence_mbarrier_init();
        prefetch_tensormap(&xmap);
    }
    if (warp == 0) tmem_alloc(tmem_slot, LY::TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // ---- producer: the token rows once, then the CTA's weight tiles back to back
        mbar_arrive_expect_tx(x_full, (uint32_t)(k_tiles * LY::X_ATOM));
        for (int a = 0; a < k_tiles; ++a) tma_load_2d(sx + a * LY::X_ATOM, &xmap, a * KT, 0, x_full);
        const uint64_t pol = l2_policy_evict_first();
        int g = 0;
        for (int j = 0; j < n_my && !*abort_flag; ++j) {
            const uint8_t *wsrc = wtiles + (size_t)(blockIdx.x + j * gridDim.x) * k_tiles * TILE_BYTES;
            for (int s = 0; s < k_tiles; ++s, ++g) {
                const int slot = g % LMH_STAGES;
                if (g >= LMH_STAGES &&
                    !mbar_wait(&empty[slot], ((g / LMH_STAGES) - 1) & 1, status, DEV_TIMEOUT_SLOT, abort_flag))
                    break;
                mbar_arrive_expect_tx(&full[slot], (uint32_t)TILE_BYTES);
                bulk_g2s(ring + slot * TILE_BYTES, wsrc + (size_t)s * TILE_BYTES, TILE_BYTES, &full[slot], pol);
            }
        }
        if (*abort_flag) {
            // error path: give the copies still in flight a bounded chance to land before exit
            mbar_wait(x_full, 0, nullptr, 0, nullptr);
            for (int h = g > LMH_STAGES ? g - LMH_STAGES : 0; h < g; ++h)
                mbar_wait(&full[h % LMH_STAGES], (h / LMH_STAGES) & 1, nullptr, 0, nullptr);
        }
    } else if (warp == 1 && lane == 0) {
        // ---- MMA issuer: per tile 4 x (128 x BN x 16) per K atom into accumulator j & 1
        const uint32_t idesc = idesc_bf16_f32(128, BN);
        bool ok = mbar_wait(x_full, 0, status, DEV_TIMEOUT_LOAD, abort_flag);
        tc_fence_after();
        int g = 0;
        for (int j = 0; ok && j < n_my; ++j) {
            const int acc = j & 1;
            if (j >= 2 && !mbar_wait(&acc_empty[acc], ((j >> 1) - 1) & 1, status, DEV_TIMEOUT_MMA, abort_flag)) break;
            tc_fence_after();
            const uint32_t d = tmem + (uint32_t)(acc * BN);
            for (int s = 0; s < k_tiles; ++s, ++g) {
                const int slot = g % LMH_STAGES;
                if (!mbar_wait(&full[slot], (g / LMH_STAGES) & 1, status, DEV_TIMEOUT_LOAD, abort_flag)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint64_t ad = sw128_kmajor_desc(ring + slot * TILE_BYTES);
                const uint64_t bd = sw128_kmajor_desc(sx + s * LY::X_ATOM);
#pragma unroll
                for (int kk = 0; kk < KT / 16; ++kk)
                    mma_bf16_ss(d, ad + 2ull * kk, bd + 2ull * kk, idesc, (s | kk) != 0 ? 1u : 0u);
                mma_commit(&empty[slot]);
            }
            if (ok) mma_commit(&acc_full[acc]);
        }
    } else if (warp >= 2) {
        // ---- epilogue: warp w reads TMEM lane quarter w % 4 (32 vocabulary rows)
        const int q = warp & 3;
        const int row = q * 32 + lane;
        for (int j = 0; j < n_my; ++j) {
            const int acc = j & 1, tile = blockIdx.x + j * gridDim.x;
            if (!mbar_wait(&acc_full[acc], (j >> 1) & 1, status, DEV_TIMEOUT_MMA, abort_flag)) break;
            tc_fence_after();
            const int feat = tile * TILE_ROWS + row;
            float *rv = red_val + acc * 4 * BN;
            int *ri = red_idx + acc * 4 * BN;
            for (int c0 = 0; c0 < BN && c0 < M; c0 += 32) {
                uint32_t v[32];
                tmem_ld_32cols(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN + c0), v);
                tmem_ld_wait();
#pragma unroll
                for (int jj = 0; jj < 32; ++jj) {
                    const int tok = c0 + jj;
                    if (tok >= M) break;  // uniform across the warp
                    float bv = __uint_as_float(v[jj]);
                    int bi = feat;
                    if (logits != nullptr) logits[(size_t)tok * V + feat] = bv;
#pragma unroll
                    for (int off = 16; off >= 1; off >>= 1) {
                        const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
                        const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
                        if (ov > bv || (ov == bv && oi < bi)) {
                            bv = ov;
                            bi = oi;
                        }
                    }
                    if (lane == 0) {
                        rv[q * BN + tok] = bv;
                        ri[q * BN + tok] = bi;
                    }
                }
            }
            tc_fence_before();
            asm volatile("bar.sync 1, 128;" ::: "memory");  // the four epilogue warps
            if (warp == 2) {
                for (int c = lane; c < M; c += 32) {
                    float bv = rv[c];
                    int bi = ri[c];
#pragma unroll
                    for (int w = 1; w < 4; ++w) {
                        const float ov = rv[w * BN + c];
                        const int oi = ri[w * BN + c];
                        if (ov > bv || (ov == bv && oi < bi)) {
                            bv = ov;
                            bi = oi;
                        }
                    }
                    tile_max[(size_t)tile * M + c] = bv;
                    tile_arg[(size_t)tile * M + c] = bi;
                }
                __syncwarp();
                // the accumulator and this tile's reduction slots may be reused
                if (lane == 0) mbarrier_arrive_one(&acc_empty[acc]);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, LY::TMEM_COLS);
}

static int lm_head_grid() {
    static int sms = 0;
    if (sms == 0) {
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
            sms = 0;
    }
    return sms;
}

template <int BN, int EPI>
static cudaError_t configure_one() {
    return cudaFuncSetAttribute(k_linear_tc<BN, EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                LinLayout<BN>::TOTAL);
}

cudaError_t configure_linear_kernels() {
    cudaError_t e;
    if ((e = configure_one<32, EPI_PARTIAL>()) != cudaSuccess) return e;
    if ((e = configure_one<64, EPI_PARTIAL>()) != cudaSuccess) return e;
    if ((e = configure_one<128, EPI_PARTIAL>()) != cudaSuccess) return e;
    if ((e = configure_one<256, EPI_PARTIAL>()) != cudaSuccess) return e;
    if ((e = configure_one<32, EPI_ARGMAX>()) != cudaSuccess) return e;
    if ((e = configure_one<64, EPI_ARGMAX>()) != cudaSuccess) return e;
    if ((e = configure_one<128, EPI_ARGMAX>()) != cudaSuccess) return e;
    if ((e = configure_one<256, EPI_ARGMAX>()) != cudaSuccess) return e;
    if ((e = cudaFuncSetAttribute(k_lm_head<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, LmhLayout<32>::TOTAL)) !=
        cudaSuccess)
        return e;
    return cudaFuncSetAttribute(k_lm_head<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, LmhLayout<64>::TOTAL);
}

template <int BN, int EPI>
static cudaError_t launch_tc(const CUtensorMap *x_map, const TiledWeight &w, int n_tiles, int k_splits, int M,
                             float *part, int rows_alloc, int n_total, float *tmax, int *targ, float *logits,
                             int *status, cudaStream_t st) {
    constexpr int smem = LinLayout<BN>::TOTAL;
    dim3 grid(n_tiles, k_splits, (M + BN - 1) / BN);
    k_linear_tc<BN, EPI><<<grid, LIN_THREADS, smem, st>>>(*x_map, static_cast<const uint8_t *>(w.tiles), w.K / KT,
                                                          w.n_main / TILE_ROWS, w.lora_rows, k_splits, M, part,
                                                          rows_alloc, n_total, tmax, targ, logits, w.n_main, status);
    return cudaGetLastError();
}

cudaError_t launch_linear_partials(const CUtensorMap *x_map, int bn, const TiledWeight &w, int with_lora, int M,
                                   const Partials &out, int *status, cudaStream_t st) {
    const int n_tiles = w.n_main / TILE_ROWS + ((with_lora && w.lora_rows > 0) ? 1 : 0);
    switch (bn) {
        case 32: return launch_tc<32, EPI_PARTIAL>(x_map, w, n_tiles, out.k_splits, M, out.p, out.rows_alloc,
                                                   out.n_total, nullptr, nullptr, nullptr, status, st);
        case 64: return launch_tc<64, EPI_PARTIAL>(x_map, w, n_tiles, out.k_splits, M, out.p, out.rows_alloc,
                                                   out.n_total, nullptr, nullptr, nullptr, status, st);
        case 128: return launch_tc<128, EPI_PARTIAL>(x_map, w, n_tiles, out.k_splits, M, out.p, out.rows_alloc,
                                                     out.n_total, nullptr, nullptr, nullptr, status, st);
        case 256: return launch_tc<256, EPI_PARTIAL>(x_map, w, n_tiles, out.k_splits, M, out.p, out.rows_alloc,
                                                     out.n_total, nullptr, nullptr, nullptr, status, st);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_lm_head(const CUtensorMap *x_map, int bn, const TiledWeight &w, int M, float *tile_max,
                           int *tile_arg, float *logits, int *status, cudaStream_t st) {
    const int n_tiles = w.n_main / TILE_ROWS;
    const int k_tiles = w.K / KT;
    const int grid = std::min(lm_head_grid(), n_tiles);
    // a few token rows: the persistent kernel (operand resident, one CTA per SM)
    if ((bn == 32 || bn == 64) && k_tiles <= LmhLayout<32>::MAX_ATOMS && grid > 0) {
        if (bn == 32)
            k_lm_head<32><<<grid, LMH_THREADS, LmhLayout<32>::TOTAL, st>>>(
                *x_map, static_cast<const uint8_t *>(w.tiles), k_tiles, n_tiles, M, tile_max, tile_arg, logits, w.n_main,
                status);
        else
            k_lm_head<64><<<grid, LMH_THREADS, LmhLayout<64>::TOTAL, st>>>(
                *x_map, static_cast<const uint8_t *>(w.tiles), k_tiles, n_tiles, M, tile_max, tile_arg, logits, w.n_main,
                status);
        return cudaGetLastError();
    }
    switch (bn) {
        case 32: return launch_tc<32, EPI_ARGMAX>(x_map, w, n_tiles, 1, M, nullptr, 0, 0, tile_max, tile_arg, logits,
                                                  status, st);
        case 64: return launch_tc<64, EPI_ARGMAX>(x_map, w, n_tiles, 1, M, nullptr, 0, 0, tile_max, tile_arg, logits,
                                                  status, st);
        case 128: return launch_tc<128, EPI_ARGMAX>(x_map, w, n_tiles, 1, M, nullptr, 0, 0, tile_max, tile_arg,
                                                    logits, status, st);
        case 256: return launch_tc<256, EPI_ARGMAX>(x_map, w, n_tiles, 1, M, nullptr, 0, 0, tile_max, tile_arg,
                                                    logits, status, st);
        default: return cudaErrorInvalidValue;
    }
}

// Final argmax over the vocabulary tiles: lowest index among equal maxima.
__global__ void k_argmax_reduce(const float *__restrict__ tile_max, const int *__restrict__ tile_arg, int n_tiles,
                                int rows, int *__restrict__ ids_out) {
    const int r = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    __shared__ float sv[8];
    __shared__ int si[8];
    float bv = -INFINITY;
    int bi = 0x7fffffff;
    for (int t = threadIdx.x; t < n_tiles; t += blockDim.x) {
        const float v = tile_max[(size_t)t * rows + r];
        const int i = tile_arg[(size_t)t * rows + r];
        if (v > bv || (v == bv && i < bi)) {
            bv = v;
            bi = i;
        }
    }
    for (int off = 16; off >= 1; off >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
        if (ov > bv || (ov == bv && oi < bi)) {
            bv = ov;
            bi = oi;
        }
    }
    if (lane == 0) {
        sv[warp] = bv;
        si[warp] = bi;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        bv = sv[0];
        bi = si[0];
        for (int w = 1; w < (int)(blockDim.x >> 5); ++w)
            if (sv[w] > bv || (sv[w] == bv && si[w] < bi)) {
                bv = sv[w];
                bi = si[w];
            }
        ids_out[r] = bi;
    }
}

cudaError_t launch_argmax_reduce(const float *tile_max, const int *tile_arg, int n_tiles, int rows, int *ids_out,
                                 cudaStream_t st) {
    if (rows <= 0) return cudaSuccess;
    k_argmax_reduce<<<rows, 256, 0, st>>>(tile_max, tile_arg, n_tiles, rows, ids_out);
    return cudaGetLastError();
}

}  // namespace pbd
