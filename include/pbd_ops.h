/*
 * pbd_ops.h -- single-kernel entry points of libpbd, for per-kernel parity tests and for
 * callers that want one step of the pass on its own.  Same conventions as pbd.h: device
 * pointers (d_), asynchronous on the given stream, caller-provided workspace, pbd_status
 * return; the message of the last failure of these calls on this thread comes from
 * pbd_op_last_error().
 */
#ifndef PBD_OPS_H
#define PBD_OPS_H

#include "pbd.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Workspace bytes pbd_op_linear needs for these sizes (0 if unsupported). */
size_t pbd_op_linear_workspace_bytes(int32_t M, int32_t K, int32_t N, int32_t r);

/* One block linear with the switchable LoRA-like delta of the paper's adapter (Appendix A.2:
 * rank r, scale alpha/r, on every projection):
 *     u = bf16(x A^T)                    [M, r]
 *     y = bf16(x W^T + scale * u B^T)    [M, N]   (fp32 accumulation, one final rounding)
 * d_x [M, K], d_w [N, K], d_a [r, K], d_b [N, r], d_y [M, N]: bf16, row-major, 16-byte aligned.
 * d_a == NULL or d_b == NULL (or r == 0) switches the delta off.  Runs the same tensor-core
 * kernel as the decoder passes (K split in 256-wide slices, fp32 partial sums in the workspace,
 * fixed-order reduction).  Requirements: N % 128 == 0, K % 64 == 0, 1 <= M <= 4096, r <= 32.
 * The workspace (d_ws, >= pbd_op_linear_workspace_bytes, 1024-byte aligned) is scratch; its first
 * word is the kernel's status word, cleared by each call and read by pbd_op_status.
 * The return value covers argument checks and launches only: a bounded device wait that ran out
 * is reported by pbd_op_status(d_ws, ...) after the call (before the next call on d_ws). */
pbd_status pbd_op_linear(int32_t M, int32_t K, int32_t N, int32_t r, float scale, const void *d_x, const void *d_w,
                         const void *d_a, const void *d_b, void *d_y, void *d_ws, size_t ws_bytes, void *d_stream);

/* Bytes of the library's own device scratch behind pbd_op_linear_static, per device. */
#define PBD_OP_LINEAR_STATIC_SCRATCH_BYTES (16u << 20)

/* pbd_op_linear without a workspace.  This entry point has no counterpart in the paper: it is
 * an integration aid.  It computes exactly what pbd_op_linear computes, with the same kernels
 * and the same fixed-order sums, so for the same inputs the two give the same y.
 *
 * Who it is for: callers that cannot hand the library device memory.  For example a caller
 * that sits behind an interface which passes only its input and output tensors, a process whose
 * device memory is entirely owned by another allocator, or a loop that must not call cudaMalloc
 * or cudaFree because those calls can synchronise the device.  Such a caller gets a call that
 * never allocates or frees device memory (no cudaMalloc, cudaFree, stream-ordered or library
 * allocation of any kind).
 *
 * Where the scratch lives: a fixed array of PBD_OP_LINEAR_STATIC_SCRATCH_BYTES (16 MiB) in the
 * library's device code, one per device, created when the CUDA runtime loads that code on the
 * device.  Its address is looked up the first time this function is called with a device current
 * (also the time the kernels' attributes are set); make that first call on each device before
 * any stream capture begins.
 *
 * Size limit: the call needs 2048 + (N/128 + (r > 0)) * (K/64) * 16384 + 4 * s * M * (N + r)
 * bytes, s = K/256 when K is a multiple of 256 and 1 otherwise (the re-tiled weight, the
 * adapter rows and the fp32 split-K partial sums).  Larger problems return PBD_ERR_CAPACITY
 * before anything is launched, and the message gives both sizes; use pbd_op_linear for them.
 * Within 16 MiB fit, for instance, an N = 6144, K = 1024 weight with r = 16 up to M = 39, and
 * an N = 1024, K = 3072 weight with r = 16 up to M = 194.
 *
 * Zeroing: every call clears, on d_stream, the one part of the scratch that must start at zero,
 * the kernel's status word.  Every other byte a call reads (the re-tiled weight and adapter rows,
 * the partial sums) is written by that same call first, so a call never sees an earlier call's
 * data.
 *
 * Device errors: as for pbd_op_linear, the return value covers argument checks and launches;
 * pbd_op_linear_static_status reports a device wait that ran out.  Ask before the next call on
 * the device, which clears the status word.
 *
 * Concurrency: all calls on one device share the same scratch.  Two calls whose work can
 * overlap in time on the device (different streams without an ordering between them, or
 * several host threads with their own streams) race on it and can produce wrong results.
 * Issue them on one stream, or order the streams.
 *
 * Arguments as pbd_op_linear, without d_ws and ws_bytes; the work runs on the current device
 * and d_stream must belong to it.  Returns PBD_ERR_INVALID_ARG for unsupported sizes or null
 * pointers, PBD_ERR_CAPACITY when the scratch is too small, PBD_ERR_CUDA when a runtime call
 * fails (message from pbd_op_last_error()). */
pbd_status pbd_op_linear_static(int32_t M, int32_t K, int32_t N, int32_t r, float scale, const void *d_x,
                                const void *d_w, const void *d_a, const void *d_b, void *d_y, void *d_stream);

/* Device status of the last pbd_op_linear_static call on the current device: waits for d_stream,
 * then reads the status word in the library's static scratch.  PBD_OK (and *h_device_code = 0)
 * when no kernel latched an error; PBD_ERR_DEVICE with the latched code (the DEV_* values of the
 * pass kernel: 1 copy, 2 accumulation, 3 ring slot, 6 inputs) in *h_device_code otherwise, in
 * which case that call's y is invalid; PBD_ERR_STATE if no call was made on this device yet;
 * PBD_ERR_CUDA if the stream failed.  h_device_code may be NULL.  Allocates nothing. */
pbd_status pbd_op_linear_static_status(void *d_stream, int32_t *h_device_code);

/* Workspace bytes pbd_op_lm_head_argmax needs (0 if unsupported). */
size_t pbd_op_lm_head_workspace_bytes(int32_t M, int32_t H, int32_t V);

/* Tied lm_head with greedy readout (Section 3, step 4 uses the verifier's top-1 token):
 *     logits = x E^T (fp32, never rounded),  ids[m] = argmax_v logits[m, v], lowest v on ties.
 * d_x [M, H] and d_embed [V, H] bf16 row-major; d_ids [M] int32; d_logits_opt [M, V] fp32 or
 * NULL.  Requirements: V % 128 == 0, H % 64 == 0, 1 <= M <= 256.  The workspace's first word is
 * the kernel's status word: pbd_op_status(d_ws, ...) reports a device wait that ran out. */
pbd_status pbd_op_lm_head_argmax(int32_t M, int32_t H, int32_t V, const void *d_x, const void *d_embed,
                                 int32_t *d_ids, float *d_logits_opt, void *d_ws, size_t ws_bytes, void *d_stream);

/* Device status of the last pbd_op_linear or pbd_op_lm_head_argmax call that used the
 * workspace d_ws (the 1024-byte-aligned pointer that call was given): waits for d_stream, then
 * reads the status word at the start of d_ws.  PBD_OK when no kernel latched an error;
 * PBD_ERR_DEVICE with the latched code in *h_device_code (may be NULL) otherwise, and that call's
 * outputs are invalid; PBD_ERR_INVALID_ARG for a null or misaligned d_ws; PBD_ERR_CUDA if the
 * stream failed.  A device wait bounded at one second that runs out is the only way these kernels
 * latch an error (the kernels' bounds on their inputs are checked on the host). */
pbd_status pbd_op_status(const void *d_ws, void *d_stream, int32_t *h_device_code);

/* Message of the last failed pbd_op_* call on this thread ("" if none). */
const char *pbd_op_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* PBD_OPS_H */
