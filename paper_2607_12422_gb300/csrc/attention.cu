// attention.cu -- block-diffusion / causal attention over the paged bf16 KV cache.
//
// Rows of a pass are the D+1 block positions of each sequence (or a prefill chunk).  The
// draft pass uses the block-diffusion mask of Section 3 (steps 1-2): the pending token's
// row sees the cache and itself, every masked row sees the cache, the pending row and the
// whole masked block.  The verify pass and plain decoding use the causal mask (Appendix A.4:
// verification runs "with a different attention mask").  GQA: query head h reads KV head
// h / (Hq / Hkv).
//
// Work split (flash-decoding): one CTA per (sequence, KV head, 128-key split).  Splits are
// aligned to absolute key positions, so a row's partial result never depends on how many
// rows share the pass.  Each CTA stages its K split (bf16) and V split (converted to fp16)
// in shared memory, then each warp takes 16 query vectors (row x head of the group) at a
// time: S = Q K^T with bf16 mma.sync, fp32 masked softmax statistics with quad shuffles in
// a fixed order, O = P V with fp16 mma.sync (P in fp16 keeps 11 significant bits).  The
// partial (m, l, O) per split goes to the workspace; k_attn_combine merges the splits in
// increasing order.
#include "common.cuh"
#include "pbd_internal.h"

namespace pbd {

constexpr int ATT_THREADS = 128;

template <int DH>
struct AttSmem {
    static constexpr int KSTR = DH + 8;  // bf16 elements per staged key row (bank-conflict padding)
    static constexpr int VSTR = DH + 8;  // fp16 elements per staged value row
    static constexpr int BYTES = ATT_SPLIT * KSTR * 2 + ATT_SPLIT * VSTR * 2;
};

__device__ __forceinline__ uint32_t ld_u32(const void *p) { return *reinterpret_cast<const uint32_t *>(p); }

template <int DH>
__global__ void __launch_bounds__(ATT_THREADS)
    k_attention(const bf16 *__restrict__ q, const bf16 *__restrict__ kc, const bf16 *__restrict__ vc, int layer,
                const int *__restrict__ page_table, int pages_per_seq, int n_pages, const int *__restrict__ Lbuf,
                PassDesc pd, int Hq, int Hkv, int n_splits, float scale, float *__restrict__ o_part,
                float2 *__restrict__ ml_part) {
    using SM = AttSmem<DH>;
    constexpr int NT = ATT_SPLIT / 8;  // key n-tiles of the score matrix
    constexpr int KS = DH / 16;        // k-steps of Q K^T
    constexpr int DT = DH / 8;         // dim n-tiles of the output

    const int s = blockIdx.x, g = blockIdx.y, bl = blockIdx.z;
    const int b = pd.b0 + bl;
    const int L = Lbuf[b];
    const int R = pd.R;
    const int T = L + R;  // keys [0, T) exist in this pass
    const int k0 = s * ATT_SPLIT;
    if (k0 >= T) return;
    const int grp = Hq / Hkv;
    const int QV = R * grp;
    const int n_mt = (QV + 15) / 16;

    extern __shared__ __align__(16) uint8_t smem[];
    bf16 *sK = reinterpret_cast<bf16 *>(smem);
    __half *sV = reinterpret_cast<__half *>(smem + ATT_SPLIT * SM::KSTR * 2);

    // ---- stage the split's keys and values through the page table; zero beyond T
    const size_t layer_off = (size_t)layer * n_pages * Hkv * PAGE * DH;
    for (int idx = threadIdx.x; idx < ATT_SPLIT * (DH / 8); idx += ATT_THREADS) {
        const int kk = idx / (DH / 8), c = idx % (DH / 8);
        const int kp = k0 + kk;
        uint4 k4 = make_uint4(0, 0, 0, 0), v4 = make_uint4(0, 0, 0, 0);
        if (kp < T && kp / PAGE < pages_per_seq) {
            const int page = page_table[b * pages_per_seq + kp / PAGE];
            const size_t off = layer_off + (((size_t)page * Hkv + g) * PAGE + (kp % PAGE)) * DH + (size_t)c * 8;
            k4 = *reinterpret_cast<const uint4 *>(kc + off);
            v4 = *reinterpret_cast<const uint4 *>(vc + off);
        }
        *reinterpret_cast<uint4 *>(sK + kk * SM::KSTR + c * 8) = k4;
        const bf16 *ve = reinterpret_cast<const bf16 *>(&v4);
        uint4 h4;
        uint32_t *hw = reinterpret_cast<uint32_t *>(&h4);
#pragma unroll
        for (int e = 0; e < 4; ++e) hw[e] = pack_half2(bf2f(ve[2 * e]), bf2f(ve[2 * e + 1]));
        *reinterpret_cast<uint4 *>(sV + kk * SM::VSTR + c * 8) = h4;
    }
    __syncthreads();

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int gq = lane >> 2, tq = lane & 3;

    for (int mt = warp; mt < n_mt; mt += ATT_THREADS / 32) {
        // query vectors of this m-tile: qv = mt*16 + gq (+8); qv -> (row i = qv / grp, head g*grp + qv % grp)
        const int qv0 = mt * 16 + gq, qv1 = qv0 + 8;
        const bool val0 = qv0 < QV, val1 = qv1 < QV;
        const int i0 = val0 ? qv0 / grp : 0, i1 = val1 ? qv1 / grp : 0;
        const int h0 = g * grp + (val0 ? qv0 % grp : 0), h1 = g * grp + (val1 ? qv1 % grp : 0);
        const bf16 *q0 = q + ((size_t)(bl * R + i0) * Hq + h0) * DH;
        const bf16 *q1 = q + ((size_t)(bl * R + i1) * Hq + h1) * DH;

        uint32_t qa[KS][4];
#pragma unroll
        for (int ks = 0; ks < KS; ++ks) {
            const int c = ks * 16 + 2 * tq;
            qa[ks][0] = val0 ? ld_u32(q0 + c) : 0u;
            qa[ks][1] = val1 ? ld_u32(q1 + c) : 0u;
            qa[ks][2] = val0 ? ld_u32(q0 + c + 8) : 0u;
            qa[ks][3] = val1 ? ld_u32(q1 + c + 8) : 0u;
        }

        float sc[NT][4];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
            sc[nt][0] = sc[nt][1] = sc[nt][2] = sc[nt][3] = 0.f;
            const bf16 *krow = sK + (nt * 8 + gq) * SM::KSTR + 2 * tq;
#pragma unroll
            for (int ks = 0; ks < KS; ++ks) mma_m16n8k16_bf16(sc[nt], qa[ks], ld_u32(krow + ks * 16), ld_u32(krow + ks * 16 + 8));
        }

        // ---- mask, scale, row max (rows r0 = qv0 and r1 = qv1; each thread holds 2 key columns per n-tile)
        const int qp0 = L + i0, qp1 = L + i1;
        const bool blk = pd.mask_mode == MASK_BLOCK_DRAFT;
        float m0 = -INFINITY, m1 = -INFINITY;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int kp = k0 + nt * 8 + 2 * tq + e;
                const bool vis0 = val0 && kp < T && (kp <= qp0 || (blk && i0 >= 1 && kp > L));
                const bool vis1 = val1 && kp < T && (kp <= qp1 || (blk && i1 >= 1 && kp > L));
                sc[nt][e] = vis0 ? __fmul_rn(sc[nt][e], scale) : -INFINITY;
                sc[nt][2 + e] = vis1 ? __fmul_rn(sc[nt][2 + e], scale) : -INFINITY;
                m0 = fmaxf(m0, sc[nt][e]);
                m1 = fmaxf(m1, sc[nt][2 + e]);
            }
        }
        m0 = fmaxf(m0, __shfl_xor_sync(0xffffffffu, m0, 1));
        m0 = fmaxf(m0, __shfl_xor_sync(0xffffffffu, m0, 2));
        m1 = fmaxf(m1, __shfl_xor_sync(0xffffffffu, m1, 1));
        m1 = fmaxf(m1, __shfl_xor_sync(0xffffffffu, m1, 2));
        const float mz0 = m0 == -INFINITY ? 0.f : m0, mz1 = m1 == -INFINITY ? 0.f : m1;

        float l0 = 0.f, l1 = 0.f;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const float p0 = sc[nt][e] == -INFINITY ? 0.f : __expf(sc[nt][e] - mz0);
                const float p1 = sc[nt][2 + e] == -INFINITY ? 0.f : __expf(sc[nt][2 + e] - mz1);
                sc[nt][e] = p0;
                sc[nt][2 + e] = p1;
                l0 += p0;
                l1 += p1;
            }
        }
        l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
        l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
        l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
        l1 += __shfl_xor_sync(0xffffffffu, l1, 2);

        // ---- O = P V  (P as fp16 A fragments straight from the score registers)
        float oc[DT][4];
#pragma unroll
        for (int dt = 0; dt < DT; ++dt) oc[dt][0] = oc[dt][1] = oc[dt][2] = oc[dt][3] = 0.f;
#pragma unroll
        for (int kstep = 0; kstep < ATT_SPLIT / 16; ++kstep) {
            uint32_t pa[4];
            pa[0] = pack_half2(sc[2 * kstep][0], sc[2 * kstep][1]);
            pa[1] = pack_half2(sc[2 * kstep][2], sc[2 * kstep][3]);
            pa[2] = pack_half2(sc[2 * kstep + 1][0], sc[2 * kstep + 1][1]);
            pa[3] = pack_half2(sc[2 * kstep + 1][2], sc[2 * kstep + 1][3]);
            // ldmatrix.trans of V[keys][dims]: matrices (keys 0-7 | 8-15) x (dims n0 | n0+8)
            const int vrow = kstep * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
            for (int dt = 0; dt < DT; dt += 2) {
                const int vcol = dt * 8 + (lane >> 4) * 8;
                const uint32_t addr = smem_u32(sV + vrow * SM::VSTR + vcol);
                uint32_t r0, r1, r2, r3;
                asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                             : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                             : "r"(addr));
                mma_m16n8k16_f16(oc[dt], pa, r0, r1);
                mma_m16n8k16_f16(oc[dt + 1], pa, r2, r3);
            }
        }

        // ---- write the split's partial result
        if (val0) {
            const int m = bl * R + i0;
            float *dst = o_part + (((size_t)m * Hq + h0) * n_splits + s) * DH;
#pragma unroll
            for (int dt = 0; dt < DT; ++dt)
                *reinterpret_cast<float2 *>(dst + dt * 8 + 2 * tq) = make_float2(oc[dt][0], oc[dt][1]);
            if (tq == 0) ml_part[((size_t)m * Hq + h0) * n_splits + s] = make_float2(m0, l0);
        }
        if (val1) {
            const int m = bl * R + i1;
            float *dst = o_part + (((size_t)m * Hq + h1) * n_splits + s) * DH;
#pragma unroll
            for (int dt = 0; dt < DT; ++dt)
                *reinterpret_cast<float2 *>(dst + dt * 8 + 2 * tq) = make_float2(oc[dt][2], oc[dt][3]);
            if (tq == 0) ml_part[((size_t)m * Hq + h1) * n_splits + s] = make_float2(m1, l1);
        }
    }
}

// Merge the splits of one (row, head) in increasing split order; splits where the row saw no
// key (l = 0) are skipped, so a row's result equals the one of a pass that never had them.
template <int DH>
__global__ void k_attn_combine(const int *__restrict__ Lbuf, PassDesc pd, int Hq, int n_splits,
                               const float *__restrict__ o_part, const float2 *__restrict__ ml_part,
                               bf16 *__restrict__ out) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int item = blockIdx.x * (blockDim.x >> 5) + warp;
    if (item >= pd.M * Hq) return;
    const int m = item / Hq, h = item % Hq;
    const int b = pd.b0 + m / pd.R;
    const int T = Lbuf[b] + pd.R;
    const int nv = min(n_splits, (T + ATT_SPLIT - 1) / ATT_SPLIT);
    const float2 *ml = ml_part + ((size_t)m * Hq + h) * n_splits;
    float mx = -INFINITY;
    for (int s = 0; s < nv; ++s) {
        const float2 v = ml[s];
        if (v.y > 0.f) mx = fmaxf(mx, v.x);
    }
    constexpr int E = DH / 32;
    float num[E];
#pragma unroll
    for (int e = 0; e < E; ++e) num[e] = 0.f;
    float den = 0.f;
    for (int s = 0; s < nv; ++s) {
        const float2 v = ml[s];
        if (!(v.y > 0.f)) continue;
        const float w = __expf(v.x - mx);
        den = __fadd_rn(den, __fmul_rn(w, v.y));
        const float *o = o_part + (((size_t)m * Hq + h) * n_splits + s) * DH;
#pragma unroll
        for (int e = 0; e < E; ++e) num[e] = __fadd_rn(num[e], __fmul_rn(w, o[lane + 32 * e]));
    }
    bf16 *dst = out + ((size_t)m * Hq + h) * DH;
#pragma unroll
    for (int e = 0; e < E; ++e) dst[lane + 32 * e] = f2bf(__fdiv_rn(num[e], den));
}

cudaError_t configure_attention_kernels() {
    cudaError_t e = cudaFuncSetAttribute(k_attention<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         AttSmem<128>::BYTES);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(k_attention<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, AttSmem<64>::BYTES);
}

cudaError_t launch_attention(const Dims &dm, const PassDesc &pd, int layer, const void *q, const KVCache &kv,
                             const int *L, int n_splits, float *o_part, float2 *ml_part, cudaStream_t st) {
    dim3 grid(n_splits, dm.Hkv, pd.nb);
    const float scale = (float)(1.0 / sqrt((double)dm.d));
    if (dm.d == 128) {
        k_attention<128><<<grid, ATT_THREADS, AttSmem<128>::BYTES, st>>>(
            static_cast<const bf16 *>(q), static_cast<const bf16 *>(kv.k), static_cast<const bf16 *>(kv.v), layer,
            kv.page_table, kv.pages_per_seq, kv.n_pages, L, pd, dm.Hq, dm.Hkv, n_splits, scale, o_part, ml_part);
    } else if (dm.d == 64) {
        k_attention<64><<<grid, ATT_THREADS, AttSmem<64>::BYTES, st>>>(
            static_cast<const bf16 *>(q), static_cast<const bf16 *>(kv.k), static_cast<const bf16 *>(kv.v), layer,
            kv.page_table, kv.pages_per_seq, kv.n_pages, L, pd, dm.Hq, dm.Hkv, n_splits, scale, o_part, ml_part);
    } else {
        return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

cudaError_t launch_attn_combine(const Dims &dm, const PassDesc &pd, const int *L, int n_splits, const float *o_part,
                                const float2 *ml_part, void *attn_out, cudaStream_t st) {
    const int items = pd.M * dm.Hq;
    const int grid = (items + 3) / 4;
    if (dm.d == 128)
        k_attn_combine<128><<<grid, 128, 0, st>>>(L, pd, dm.Hq, n_splits, o_part, ml_part,
                                                 static_cast<bf16 *>(attn_out));
    else if (dm.d == 64)
        k_attn_combine<64><<<grid, 128, 0, st>>>(L, pd, dm.Hq, n_splits, o_part, ml_part,
                                                static_cast<bf16 *>(attn_out));
    else
        return cudaErrorInvalidValue;
    return cudaGetLastError();
}

}  // namespace pbd
