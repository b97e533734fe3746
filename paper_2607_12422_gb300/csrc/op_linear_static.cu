// op_linear_static.cu -- pbd_op_linear_static (include/pbd_ops.h): the block linear of
// pbd_op_linear, with its scratch taken from a fixed-size device array that belongs to this
// library instead of from a caller workspace.  A call therefore neither receives nor allocates
// device memory: it re-tiles the weight into the array, runs the same tensor-core kernel and
// split-K reduction, and writes y.
//
// The array exists once per device; it is created when the CUDA runtime loads this library's
// device code on that device, and its address is looked up once per device (first call with
// that device current).  Every call on a device uses the same bytes, so calls on one device
// must not overlap in time.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <cstdio>
#include <mutex>

#include "../../include/pbd_ops.h"
#include "pbd_internal.h"

// Layout inside the array (offsets from the first 1024-byte boundary in it):
//   [0, 256)         status word of the tensor-core kernel (cleared by every call)
//   [1024, ...)      the weight (and adapter A rows) re-tiled in 128 x 64 tiles of 16 KiB
//   [..., ...)       fp32 split-K partial sums [k_splits][M][N + r]
static __device__ __align__(256) unsigned char g_linear_scratch[PBD_OP_LINEAR_STATIC_SCRATCH_BYTES];

using namespace pbd;

namespace {

constexpr int MAX_DEVICES = 64;
constexpr size_t BASE_ALIGN = 1024;  // the array is 256-aligned; the tiles start on a 1 KiB boundary

std::mutex g_setup_mu;
uint8_t *g_scratch[MAX_DEVICES];  // aligned scratch base per device, nullptr until set up

struct StaticPlan {
    size_t tiles_off, part_off, total;  // total includes the alignment slack
    int k_splits, row_tiles;
};

size_t round_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

bool plan(int M, int K, int N, int r, StaticPlan *p) {
    if (M < 1 || M > 4096 || K < 64 || K % 64 || N < 128 || N % 128 || r < 0 || r > 32) return false;
    const int kt = K / KT;
    p->k_splits = (kt % 4 == 0) ? kt / 4 : 1;  // 256-wide K slices, as in pbd_op_linear
    p->row_tiles = N / TILE_ROWS + (r > 0 ? 1 : 0);
    p->tiles_off = BASE_ALIGN;
    p->part_off = round_up(p->tiles_off + (size_t)p->row_tiles * kt * TILE_BYTES, BASE_ALIGN);
    p->total = BASE_ALIGN + p->part_off + sizeof(float) * (size_t)p->k_splits * M * (N + r);
    return true;
}

pbd_status fail(pbd_status s, const char *fmt, size_t a = 0, size_t b = 0) {
    char msg[256];
    snprintf(msg, sizeof msg, fmt, a, b);
    op_record_error(msg);
    return s;
}

pbd_status fail_cuda(const char *what, cudaError_t e) {
    char msg[256];
    snprintf(msg, sizeof msg, "pbd_op_linear_static: %s: %s", what, cudaGetErrorString(e));
    op_record_error(msg);
    return PBD_ERR_CUDA;
}

// Address of this device's scratch; looked up (and the kernels configured) on the first call
// made with the device current.
pbd_status scratch_of_current_device(uint8_t **out) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail_cuda("cudaGetDevice", e);
    if (dev < 0 || dev >= MAX_DEVICES)
        return fail(PBD_ERR_INVALID_ARG, "pbd_op_linear_static: device ordinal %zu beyond %zu", (size_t)dev,
                    (size_t)MAX_DEVICES);
    std::lock_guard<std::mutex> lock(g_setup_mu);
    if (g_scratch[dev] == nullptr) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_linear_scratch);
        if (e != cudaSuccess) return fail_cuda("cudaGetSymbolAddress of the static scratch", e);
        if (p == nullptr) return fail(PBD_ERR_CUDA, "pbd_op_linear_static: static scratch has no address");
        if ((e = configure_linear_kernels()) != cudaSuccess) return fail_cuda("kernel attributes", e);
        const uintptr_t a = (reinterpret_cast<uintptr_t>(p) + BASE_ALIGN - 1) & ~(uintptr_t)(BASE_ALIGN - 1);
        g_scratch[dev] = reinterpret_cast<uint8_t *>(a);
    }
    *out = g_scratch[dev];
    return PBD_OK;
}

}  // namespace

extern "C" pbd_status pbd_op_linear_static(int32_t M, int32_t K, int32_t N, int32_t r, float scale, const void *d_x,
                                           const void *d_w, const void *d_a, const void *d_b, void *d_y,
                                           void *d_stream) {
    const bool lora = r > 0 && d_a != nullptr && d_b != nullptr;
    const int rr = lora ? r : 0;
    StaticPlan p;
    if (!plan(M, K, N, rr, &p)) return fail(PBD_ERR_INVALID_ARG, "pbd_op_linear_static: unsupported sizes");
    if (p.total > (size_t)PBD_OP_LINEAR_STATIC_SCRATCH_BYTES)
        return fail(PBD_ERR_CAPACITY, "pbd_op_linear_static: these sizes need %zu bytes of scratch; the static "
                    "scratch holds %zu (use pbd_op_linear with a workspace)", p.total,
                    (size_t)PBD_OP_LINEAR_STATIC_SCRATCH_BYTES);
    if (!d_x || !d_w || !d_y) return fail(PBD_ERR_INVALID_ARG, "pbd_op_linear_static: null pointer");

    uint8_t *ws = nullptr;
    const pbd_status s = scratch_of_current_device(&ws);
    if (s != PBD_OK) return s;

    const int bn = M <= 32 ? 32 : M <= 64 ? 64 : M <= 128 ? 128 : 256;
    CUtensorMap map;
    if (!encode_bf16_map(&map, d_x, M, K, bn))
        return fail(PBD_ERR_INVALID_ARG, "pbd_op_linear_static: x not TMA-mappable (16-byte alignment)");

    cudaStream_t st = static_cast<cudaStream_t>(d_stream);
    int *status = reinterpret_cast<int *>(ws);
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
    uint8_t *tiles = ws + p.tiles_off;

    cudaError_t e;
    // What must start at zero on every call: the status word, which the kernel only ever raises.
    // The weight tiles and the partial sums this call reads are written by this call first (the
    // kernel copies only the adapter tile's first r rows, and stores only rows it computed).
    if ((e = cudaMemsetAsync(status, 0, 256, st)) != cudaSuccess) return fail_cuda("clear status", e);
    if ((e = launch_repack_tiled(d_w, N, K, tiles, 0, st)) != cudaSuccess) return fail_cuda("repack W", e);
    if (lora && (e = launch_repack_tiled(d_a, rr, K, tiles, N, st)) != cudaSuccess) return fail_cuda("repack A", e);
    if ((e = launch_linear_partials(&map, bn, w, lora ? 1 : 0, M, P, status, st)) != cudaSuccess)
        return fail_cuda("linear", e);
    if ((e = launch_linear_finalize(P, M, N, rr, scale, d_b, d_y, st)) != cudaSuccess)
        return fail_cuda("finalize", e);
    return PBD_OK;
}

extern "C" pbd_status pbd_op_linear_static_status(void *d_stream, int32_t *h_device_code) {
    if (h_device_code) *h_device_code = 0;
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail_cuda("cudaGetDevice", e);
    uint8_t *ws = nullptr;
    {
        std::lock_guard<std::mutex> lock(g_setup_mu);
        if (dev >= 0 && dev < MAX_DEVICES) ws = g_scratch[dev];
    }
    if (ws == nullptr)
        return fail(PBD_ERR_STATE, "pbd_op_linear_static_status: no pbd_op_linear_static call on this device yet");
    int code = 0;
    const pbd_status s = read_device_code(reinterpret_cast<const int *>(ws), static_cast<cudaStream_t>(d_stream), &code,
                                          "pbd_op_linear_static_status");
    if (s != PBD_OK) return s;
    if (h_device_code) *h_device_code = code;
    return code == 0 ? PBD_OK : device_fail(code, "pbd_op_linear_static");
}
