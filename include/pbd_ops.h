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
 * The workspace (d_ws, >= pbd_op_linear_workspace_bytes, 1024-byte aligned) is scratch. */
pbd_status pbd_op_linear(int32_t M, int32_t K, int32_t N, int32_t r, float scale, const void *d_x, const void *d_w,
                         const void *d_a, const void *d_b, void *d_y, void *d_ws, size_t ws_bytes, void *d_stream);

/* Workspace bytes pbd_op_lm_head_argmax needs (0 if unsupported). */
size_t pbd_op_lm_head_workspace_bytes(int32_t M, int32_t H, int32_t V);

/* Tied lm_head with greedy readout (Section 3, step 4 uses the verifier's top-1 token):
 *     logits = x E^T (fp32, never rounded),  ids[m] = argmax_v logits[m, v], lowest v on ties.
 * d_x [M, H] and d_embed [V, H] bf16 row-major; d_ids [M] int32; d_logits_opt [M, V] fp32 or
 * NULL.  Requirements: V % 128 == 0, H % 64 == 0, 1 <= M <= 256. */
pbd_status pbd_op_lm_head_argmax(int32_t M, int32_t H, int32_t V, const void *d_x, const void *d_embed,
                                 int32_t *d_ids, float *d_logits_opt, void *d_ws, size_t ws_bytes, void *d_stream);

/* Message of the last failed pbd_op_* call on this thread ("" if none). */
const char *pbd_op_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* PBD_OPS_H */
