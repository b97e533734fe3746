// ops_api.cu -- single-kernel C entry points (include/pbd_ops.h) and the TMA descriptor helper
// shared with the context code.  The linear entry point re-tiles W (and A) into the workspace,
// runs the same tensor-core kernel and split-K reduction as the decoder passes, and finishes
// with bf16(x W^T + s * bf16(x A^T) B^T).
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdio>
#include <string>

#include "../../include/pbd_ops.h"
#include "common.cuh"
#include "pbd_internal.h"

namespace pbd {

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// 2-D bf16 row-major [rows, cols] tensor map with box {64, box_rows}, 128-byte swizzle.
bool encode_bf16_map(CUtensorMap *map, const void *base, int rows, int cols, int box_rows) {
    static EncodeTiledFn enc = nullptr;
    if (!enc) {
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            fn == nullptr || q != cudaDriverEntryPointSuccess)
            return false;
        enc = reinterpret_cast<EncodeTiledFn>(fn);
    }
    if ((reinterpret_cast<uintptr_t>(base) & 15) || (cols * 2) % 16) return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    cuuint32_t box[2] = {(cuuint32_t)KT, (cuuint32_t)box_rows};
    cuuint32_t es[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int op_bn(int M) { return M <= 32 ? 32 : M <= 64 ? 64 : M <= 128 ? 128 : 256; }

}  // namespace pbd

using namespace pbd;

namespace {

thread_local std::string g_op_err;

pbd_status op_fail(pbd_status s, const char *msg, cudaError_t e = cudaSuccess) {
    char b[256];
    snprintf(b, sizeof b, "%s%s%s", msg, e != cudaSuccess ? ": " : "", e != cudaSuccess ? cudaGetErrorString(e) : "");
    g_op_err = b;
    return s;
}

struct LinearPlan {
    size_t tiles_off, part_off, status_off, total;
    int k_splits, row_tiles;
};

bool plan_linear(int M, int K, int N, int r, LinearPlan *p) {
    if (M < 1 || M > 4096 || K < 64 || K % 64 || N < 128 || N % 128 || r < 0 || r > 32) return false;
    const int kt = K / KT;
    p->k_splits = (kt % 4 == 0) ? kt / 4 : 1;
    p->row_tiles = N / TILE_ROWS + (r > 0 ? 1 : 0);
    size_t off = 0;
    auto take = [&](size_t bytes) {
        off = (off + 1023) / 1024 * 1024;
        const size_t o = off;
        off += bytes;
        return o;
    };
    p->status_off = take(256);
    p->tiles_off = take((size_t)p->row_tiles * kt * TILE_BYTES);
    p->part_off = take(sizeof(float) * (size_t)p->k_splits * M * (N + r));
    p->total = off;
    return true;
}

}  // namespace

namespace pbd {

// Waits for d_stream, then reads the status word a kernel may have latched (a DEV_* code).
pbd_status read_device_code(const int *d_status, cudaStream_t st, int *code, const char *who) {
    cudaError_t e = cudaStreamSynchronize(st);
    if (e == cudaSuccess) e = cudaMemcpy(code, d_status, sizeof(int), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) {
        char b[128];
        snprintf(b, sizeof b, "%s: reading the status word", who);
        return op_fail(PBD_ERR_CUDA, b, e);
    }
    return PBD_OK;
}

const char *device_code_name(int code) {
    switch (code) {
        case DEV_TIMEOUT_LOAD: return "a weight or operand copy never completed";
        case DEV_TIMEOUT_MMA: return "a tensor-core accumulation never completed";
        case DEV_TIMEOUT_SLOT: return "a shared-memory ring slot was never released";
        case DEV_BAD_TOKEN: return "token id outside the vocabulary";
        case DEV_BAD_POSITION: return "position beyond the reserved KV pages";
        case DEV_TIMEOUT_DEP: return "a work item's inputs never completed";
        default: return "unknown device code";
    }
}

pbd_status device_fail(int code, const char *who) {
    char b[256];
    snprintf(b, sizeof b, "%s: device status %d latched by a kernel (%s); the outputs of that call are invalid", who,
             code, device_code_name(code));
    g_op_err = b;
    return PBD_ERR_DEVICE;
}

}  // namespace pbd

extern "C" {

size_t pbd_op_linear_workspace_bytes(int32_t M, int32_t K, int32_t N, int32_t r) {
    LinearPlan p;
    return plan_linear(M, K, N, r, &p) ? p.total : 0;
}

pbd_status pbd_op_linear(int32_t M, int32_t K, int32_t N, int32_t r, float scale, const void *d_x, const void *d_w,
                         const void *d_a, const void *d_b, void *d_y, void *d_ws, size_t ws_bytes, void *d_stream) {
    const bool lora = r > 0 && d_a != nullptr && d_b != nullptr;
    const int rr = lora ? r : 0;
    LinearPlan p;
    if (!plan_linear(M, K, N, rr, &p)) return op_fail(PBD_ERR_INVALID_ARG, "pbd_op_linear: unsupported sizes");
    if (!d_x || !d_w || !d_y) return op_fail(PBD_ERR_INVALID_ARG, "pbd_op_linear: null pointer");
    if (!d_ws || (reinterpret_cast<uintptr_t>(d_ws) & 1023) || ws_bytes < p.total)
        return op_fail(PBD_ERR_WORKSPACE, "pbd_op_linear: workspace missing, misaligned or too small");
    cudaStream_t st = static_cast<cudaStream_t>(d_stream);
    uint8_t *ws = static_cast<uint8_t *>(d_ws);
    int *status = reinterpret_cast<int *>(ws + p.status_off);
    TiledWeight w;
    w.tiles = ws + p.tiles_off;
    w.n_main = N;
    w.lora_rows = rr;
    w.K = K;
    Partials P;
    P.p = reinterpret_cast<float *>(ws + p.part_off);
    P.k_splits = p.k_splits;
    P.rows_alloc = M;
    P.n_total = N + rr;
    const int bn = op_bn(M);
    CUtensorMap map;
    if (!encode_bf16_map(&map, d_x, M, K, bn)) return op_fail(PBD_ERR_INVALID_ARG, "pbd_op_linear: x not TMA-mappable");
    cudaError_t e;
    if ((e = configure_linear_kernels()) != cudaSuccess) return op_fail(PBD_ERR_CUDA, "configure", e);
    if ((e = cudaMemsetAsync(status, 0, 256, st)) != cudaSuccess) return op_fail(PBD_ERR_CUDA, "memset", e);
    if ((e = cudaMemsetAsync(const_cast<void *>(w.tiles), 0, (size_t)p.row_tiles * (K / KT) * TILE_BYTES, st)) !=
        cudaSuccess)
        return op_fail(PBD_ERR_CUDA, "memset", e);
    if ((e = launch_repack_tiled(d_w, N, K, const_cast<void *>(w.tiles), 0, st)) != cudaSuccess)
        return op_fail(PBD_ERR_CUDA, "repack W", e);
    if (lora && (e = launch_repack_tiled(d_a, rr, K, const_cast<void *>(w.tiles), N, st)) != cudaSuccess)
        return op_fail(PBD_ERR_CUDA, "repack A", e);
    if ((e = launch_linear_partials(&map, bn, w, lora ? 1 : 0, M, P, status, st)) != cudaSuccess)
        return op_fail(PBD_ERR_CUDA, "linear", e);
    if ((e = launch_linear_finalize(P, M, N, rr, scale, d_b, d_y, st)) != cudaSuccess)
        return op_fail(PBD_ERR_CUDA, "finalize", e);
    return PBD_OK;
}

size_t pbd_op_lm_head_workspace_bytes(int32_t M, int32_t H, int32_t V) {
    if (M < 1 || M > 256 || H < 64 || H % 64 || V < 128 || V % 128) return 0;
    size_t tiles = (size_t)(V / TILE_ROWS) * (H / KT) * TILE_BYTES;
    size_t red = (size_t)(V / TILE_ROWS) * M * 8;
    return 1024 + (tiles + 1023) / 1024 * 1024 + (red + 1023) / 1024 * 1024;
}

pbd_status pbd_op_lm_head_argmax(int32_t M, int32_t H, int32_t V, const void *d_x, const void *d_embed,
                                 int32_t *d_ids, float *d_logits_opt, void *d_ws, size_t ws_bytes, void *d_stream) {
    const size_t need = pbd_op_lm_head_workspace_bytes(M, H, V);
    if (need == 0) return op_fail(PBD_ERR_INVALID_ARG, "pbd_op_lm_head_argmax: unsupported sizes");
    if (!d_x || !d_embed || !d_ids) return op_fail(PBD_ERR_INVALID_ARG, "pbd_op_lm_head_argmax: null pointer");
    if (!d_ws || (reinterpret_cast<uintptr_t>(d_ws) & 1023) || ws_bytes < need)
        return op_fail(PBD_ERR_WORKSPACE, "pbd_op_lm_head_argmax: workspace missing, misaligned or too small");
    cudaStream_t st = static_cast<cudaStream_t>(d_stream);
    uint8_t *ws = static_cast<uint8_t *>(d_ws);
    int *status = reinterpret_cast<int *>(ws);
    const size_t tiles_bytes = (size_t)(V / TILE_ROWS) * (H / KT) * TILE_BYTES;
    TiledWeight w;
    w.tiles = ws + 1024;
    w.n_main = V;
    w.lora_rows = 0;
    w.K = H;
    float *tmax = reinterpret_cast<float *>(ws + 1024 + (tiles_bytes + 1023) / 1024 * 1024);
    int *targ = reinterpret_cast<int *>(tmax + (size_t)(V / TILE_ROWS) * M);
    const int bn = op_bn(M);
    CUtensorMap map;
    if (!encode_bf16_map(&map, d_x, M, H, bn))
        return op_fail(PBD_ERR_INVALID_ARG, "pbd_op_lm_head_argmax: x not TMA-mappable");
    cudaError_t e;
    if ((e = configure_linear_kernels()) != cudaSuccess) return op_fail(PBD_ERR_CUDA, "configure", e);
    if ((e = cudaMemsetAsync(status, 0, 256, st)) != cudaSuccess) return op_fail(PBD_ERR_CUDA, "memset", e);
    if ((e = launch_repack_tiled(d_embed, V, H, const_cast<void *>(w.tiles), 0, st)) != cudaSuccess)
        return op_fail(PBD_ERR_CUDA, "repack", e);
    if ((e = launch_lm_head(&map, bn, w, M, tmax, targ, d_logits_opt, status, st)) != cudaSuccess)
        return op_fail(PBD_ERR_CUDA, "lm_head", e);
    if ((e = launch_argmax_reduce(tmax, targ, V / TILE_ROWS, M, d_ids, st)) != cudaSuccess)
        return op_fail(PBD_ERR_CUDA, "argmax", e);
    return PBD_OK;
}

pbd_status pbd_op_status(const void *d_ws, void *d_stream, int32_t *h_device_code) {
    if (h_device_code) *h_device_code = 0;
    if (!d_ws || (reinterpret_cast<uintptr_t>(d_ws) & 1023))
        return op_fail(PBD_ERR_INVALID_ARG, "pbd_op_status: workspace missing or misaligned");
    int code = 0;
    pbd_status s = read_device_code(static_cast<const int *>(d_ws), static_cast<cudaStream_t>(d_stream), &code,
                                    "pbd_op_status");
    if (s != PBD_OK) return s;
    if (h_device_code) *h_device_code = code;
    return code == 0 ? PBD_OK : device_fail(code, "pbd_op_status");
}

const char *pbd_op_last_error(void) { return g_op_err.c_str(); }

}  // extern "C"

namespace pbd {
void op_record_error(const char *msg) { g_op_err = msg; }
}  // namespace pbd
