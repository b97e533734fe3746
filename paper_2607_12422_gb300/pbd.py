"""Python binding of libpbd (include/pbd.h): argument marshalling only.

Every step of a pass runs in the library's CUDA kernels; PyTorch is used here only to
own device memory (weights, workspace, outputs) and the CUDA stream.  If the compiled
library is missing this module raises; there is no fallback path.
"""
from __future__ import annotations

import ctypes as C
import os
import re
from typing import Dict, List, Optional, Sequence

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "lib", "libpbd.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "pbd.h")

PBD_OK = 0
STATUS_NAMES = {0: "PBD_OK", 1: "PBD_ERR_INVALID_ARG", 2: "PBD_ERR_WORKSPACE", 3: "PBD_ERR_CAPACITY",
                4: "PBD_ERR_STATE", 5: "PBD_ERR_CUDA", 6: "PBD_ERR_DEVICE"}
LINEARS = ("q", "k", "v", "o", "gate", "up", "down")
TRACE_STAMPS = 16  # timestamps per work item of pbd_trace_pass


class PbdError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__("%s: %s" % (STATUS_NAMES.get(status, status), msg))
        self.status = status


class pbd_config(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("hidden", C.c_int32), ("n_q_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32), ("intermediate", C.c_int32),
                ("vocab", C.c_int32), ("rms_eps", C.c_float), ("rope_theta", C.c_float),
                ("lora_rank", C.c_int32), ("lora_scale", C.c_float), ("block_D", C.c_int32),
                ("max_batch", C.c_int32), ("max_seq_len", C.c_int32), ("page_size", C.c_int32),
                ("draft_layers", C.c_int32), ("denoise_steps", C.c_int32), ("draft_unanchored", C.c_int32),
                ("draft_skip_mask", C.c_uint64), ("max_ctas", C.c_int32)]


class pbd_base_weights(C.Structure):
    _fields_ = [("embed", C.c_void_p), ("final_norm", C.c_void_p), ("attn_norm", C.c_void_p),
                ("mlp_norm", C.c_void_p), ("q_norm", C.c_void_p), ("k_norm", C.c_void_p), ("w", C.c_void_p * 7)]


class pbd_adapter_weights(C.Structure):
    _fields_ = [("lora_a", C.c_void_p * 7), ("lora_b", C.c_void_p * 7), ("mask_embed", C.c_void_p)]


class pbd_stats(C.Structure):
    _fields_ = [("rounds", C.c_int64), ("accepted", C.c_int64), ("emitted", C.c_int64),
                ("draft_ms", C.c_double), ("verify_ms", C.c_double)]


_lib = None


def header_functions() -> List[str]:
    """Names of the functions include/pbd.h and include/pbd_ops.h declare."""
    names = set()
    for h in (HEADER, os.path.join(os.path.dirname(HEADER), "pbd_ops.h")):
        txt = re.sub(r"/\*.*?\*/", "", open(h).read(), flags=re.S)
        names.update(re.findall(r"\b(pbd_[a-z_]+)\s*\(", txt))
    return sorted(names)


def load(path: str = LIB_PATH) -> C.CDLL:
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError("libpbd.so is not built (%s); run __graft_entry__.build()" % path)
    L = C.CDLL(path)
    P = C.c_void_p
    I32 = C.c_int32
    L.pbd_workspace_bytes.restype = C.c_size_t
    L.pbd_workspace_bytes.argtypes = [C.POINTER(pbd_config)]
    L.pbd_create.argtypes = [C.POINTER(pbd_config), C.POINTER(pbd_base_weights), C.POINTER(pbd_adapter_weights),
                             P, C.c_size_t, P, C.POINTER(P)]
    L.pbd_destroy.argtypes = [P]
    L.pbd_prefill.argtypes = [P, I32, P, P, I32, P]
    L.pbd_draft_block.argtypes = [P, P, P]
    L.pbd_verify_block.argtypes = [P, P, P, P]
    L.pbd_accept_commit.argtypes = [P, P, P]
    L.pbd_decode_step.argtypes = [P, P, P]
    L.pbd_generate.argtypes = [P, I32, P, P, I32, I32, P, P, C.POINTER(pbd_stats)]
    L.pbd_get_state.argtypes = [P, P, P, P]
    L.pbd_get_tokens.argtypes = [P, P]
    L.pbd_read_kv.argtypes = [P, I32, I32, I32, P, P]
    L.pbd_sync.argtypes = [P]
    L.pbd_last_error.restype = C.c_char_p
    L.pbd_last_error.argtypes = [P]
    L.pbd_version.restype = C.c_char_p
    L.pbd_bench_rounds.argtypes = [P, I32, I32, I32, P, P, P]
    L.pbd_time_pass.argtypes = [P, I32, I32, P, P]
    L.pbd_trace_pass.argtypes = [P, I32, P, P, I32, P]
    L.pbd_trace_pass.restype = C.c_int
    L.pbd_bench_rounds.restype = C.c_int
    L.pbd_time_pass.restype = C.c_int
    L.pbd_check_stalled_pass.argtypes = [P, P]
    L.pbd_check_stalled_pass.restype = C.c_int
    L.pbd_plan_pass.argtypes = [C.POINTER(pbd_config), I32, I32, P, I32, I32, P, P, I32, P]
    L.pbd_plan_pass.restype = C.c_int
    L.pbd_op_linear_workspace_bytes.restype = C.c_size_t
    L.pbd_op_linear_workspace_bytes.argtypes = [I32, I32, I32, I32]
    L.pbd_op_linear.argtypes = [I32, I32, I32, I32, C.c_float, P, P, P, P, P, P, C.c_size_t, P]
    L.pbd_op_lm_head_workspace_bytes.restype = C.c_size_t
    L.pbd_op_lm_head_workspace_bytes.argtypes = [I32, I32, I32]
    L.pbd_op_lm_head_argmax.argtypes = [I32, I32, I32, P, P, P, P, P, C.c_size_t, P]
    L.pbd_op_last_error.restype = C.c_char_p
    L.pbd_op_linear_static.argtypes = [I32, I32, I32, I32, C.c_float, P, P, P, P, P, P]
    L.pbd_op_linear_static.restype = C.c_int
    L.pbd_op_status.argtypes = [P, P, P]
    L.pbd_op_status.restype = C.c_int
    L.pbd_op_linear_static_status.argtypes = [P, P]
    L.pbd_op_linear_static_status.restype = C.c_int
    for name in ("pbd_create", "pbd_destroy", "pbd_prefill", "pbd_draft_block", "pbd_verify_block",
                 "pbd_accept_commit", "pbd_decode_step", "pbd_generate", "pbd_get_state", "pbd_get_tokens",
                 "pbd_read_kv", "pbd_sync", "pbd_op_linear", "pbd_op_lm_head_argmax"):
        getattr(L, name).restype = C.c_int
    _lib = L
    return L


def _ws(torch, nbytes, device):
    """1024-byte-aligned view into a fresh uint8 device buffer."""
    buf = torch.empty(nbytes + 1024, dtype=torch.uint8, device=device)
    off = (-buf.data_ptr()) % 1024
    return buf, buf.data_ptr() + off


def _raise_if(L, s):
    if s != PBD_OK:
        raise PbdError(s, L.pbd_op_last_error().decode())


def pbd_op_linear(x, W, A=None, B=None, scale: float = 2.0):
    """y = bf16(x W^T + scale * bf16(x A^T) B^T) on the GPU (torch bf16 device tensors in, out).
    Waits for the result and raises PbdError(PBD_ERR_DEVICE) if a kernel latched an error."""
    import torch
    L = load()
    M, K = x.shape
    N = W.shape[0]
    r = A.shape[0] if (A is not None and B is not None) else 0
    need = L.pbd_op_linear_workspace_bytes(M, K, N, r)
    if need == 0:
        raise PbdError(1, "pbd_op_linear: unsupported sizes")
    with torch.cuda.device(x.device):  # the library runs on the current device
        buf, ws = _ws(torch, need, x.device)
        y = torch.empty(M, N, dtype=torch.bfloat16, device=x.device)
        st = torch.cuda.current_stream(x.device).cuda_stream
        _raise_if(L, L.pbd_op_linear(M, K, N, r, scale, x.data_ptr(), W.data_ptr(), _ptr(A) if r else None,
                                     _ptr(B) if r else None, y.data_ptr(), ws, need, st))
        _raise_if(L, L.pbd_op_status(ws, st, None))
    del buf
    return y


def pbd_op_linear_static(x, W, A=None, B=None, scale: float = 2.0, y=None, sync: bool = True):
    """pbd_op_linear through the entry point that takes no workspace (the library's own static
    scratch); y [M, N] bf16 is the caller's output tensor (allocated here when not given).
    With sync, waits and raises PbdError(PBD_ERR_DEVICE) if the kernel latched an error; without
    it the caller asks pbd_op_linear_static_status before the next call."""
    import torch
    L = load()
    M, K = x.shape
    N = W.shape[0]
    r = A.shape[0] if (A is not None and B is not None) else 0
    with torch.cuda.device(x.device):  # the library picks its scratch by the current device
        if y is None:
            y = torch.empty(M, N, dtype=torch.bfloat16, device=x.device)
        st = torch.cuda.current_stream(x.device).cuda_stream
        _raise_if(L, L.pbd_op_linear_static(M, K, N, r, scale, x.data_ptr(), W.data_ptr(), _ptr(A) if r else None,
                                            _ptr(B) if r else None, y.data_ptr(), st))
        if sync:
            _raise_if(L, L.pbd_op_linear_static_status(st, None))
    return y


def pbd_op_linear_static_status(device=None) -> int:
    """Device code of the last pbd_op_linear_static call on `device` (0 = none); raises PbdError
    on PBD_ERR_DEVICE, PBD_ERR_STATE (no call yet) or PBD_ERR_CUDA."""
    import torch
    L = load()
    dev = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
    code = C.c_int32(0)
    with torch.cuda.device(dev):
        s = L.pbd_op_linear_static_status(torch.cuda.current_stream(dev).cuda_stream, C.byref(code))
    if s != PBD_OK:
        raise PbdError(s, L.pbd_op_last_error().decode())
    return code.value


def pbd_op_lm_head_argmax(x, E, want_logits: bool = False):
    """(argmax ids [M] int32, logits [M, V] fp32 or None) of x E^T on the GPU.
    Waits for the result and raises PbdError(PBD_ERR_DEVICE) if a kernel latched an error."""
    import torch
    L = load()
    M, H = x.shape
    V = E.shape[0]
    need = L.pbd_op_lm_head_workspace_bytes(M, H, V)
    if need == 0:
        raise PbdError(1, "pbd_op_lm_head_argmax: unsupported sizes")
    with torch.cuda.device(x.device):
        buf, ws = _ws(torch, need, x.device)
        ids = torch.empty(M, dtype=torch.int32, device=x.device)
        lg = torch.empty(M, V, dtype=torch.float32, device=x.device) if want_logits else None
        st = torch.cuda.current_stream(x.device).cuda_stream
        _raise_if(L, L.pbd_op_lm_head_argmax(M, H, V, x.data_ptr(), E.data_ptr(), ids.data_ptr(), _ptr(lg), ws,
                                             need, st))
        _raise_if(L, L.pbd_op_status(ws, st, None))
    del buf
    return ids, lg


def make_config(shape, block_D: int, max_batch: int, max_seq_len: int, draft_layers: int = 0,
                denoise_steps: int = 1, anchored: bool = True, draft_skip: int = 0, max_ctas: int = 0) -> pbd_config:
    """pbd_config for a model shape; the draft variant defaults to the method of Section 3."""
    return pbd_config(shape.n_layers, shape.hidden, shape.n_q_heads, shape.n_kv_heads, shape.head_dim,
                      shape.intermediate, shape.vocab, shape.rms_eps, shape.rope_theta, shape.lora_rank,
                      shape.lora_alpha / shape.lora_rank, block_D, max_batch, max_seq_len, 16,
                      draft_layers, denoise_steps, 0 if anchored else 1, draft_skip, max_ctas)


def pbd_plan_pass(cfg: pbd_config, kind: int, prompt_lens: Sequence[int], max_new: int, grid: int,
                  cap: int = 1 << 20):
    """(items [n, 8] int32, cta_off [grid + 1] int32) of one pass's schedule, host only: per item
    {op | lin << 8 | layer << 16, a, b, c, wait counter, wait target, release counters 0, 1}."""
    L = load()
    lens = np.ascontiguousarray(np.asarray(prompt_lens, dtype=np.int32))
    items = np.zeros((cap, 8), np.int32)
    off = np.zeros(grid + 1, np.int32)
    n = np.zeros(1, np.int32)
    s = L.pbd_plan_pass(C.byref(cfg), kind, len(lens), lens.ctypes.data, max_new, grid, items.ctypes.data,
                        off.ctypes.data, cap, n.ctypes.data)
    if s != PBD_OK:
        raise PbdError(s, (L.pbd_last_error(None) or b"").decode())
    return items[: int(n[0])].copy(), off


def _ptr(t) -> int:
    return t.data_ptr() if t is not None else None


class Engine:
    """One pbd context on one GPU: owns the workspace and a private CUDA stream."""

    def __init__(self, shape, base: Dict[str, np.ndarray], adapter: Dict[str, np.ndarray], block_D: int,
                 max_batch: int, max_seq_len: int, device: str = "cuda:0", keep_host_weights: bool = False,
                 draft_layers: int = 0, denoise_steps: int = 1, anchored: bool = True, draft_skip: int = 0,
                 max_ctas: int = 0):
        import torch
        self.torch = torch
        self.lib = load()
        self.shape = shape
        self.D = block_D
        self.device = torch.device(device)
        self.cfg = make_config(shape, block_D, max_batch, max_seq_len, draft_layers, denoise_steps, anchored,
                               draft_skip, max_ctas)
        need = self.lib.pbd_workspace_bytes(C.byref(self.cfg))
        if need == 0:
            raise PbdError(1, "configuration rejected by pbd_workspace_bytes")
        self.workspace = torch.empty(need + 256, dtype=torch.uint8, device=self.device)
        self.stream = torch.cuda.Stream(device=self.device)

        def dev(a):
            return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(self.device).view(torch.bfloat16)

        bw = pbd_base_weights()
        tmp = {}
        for k in ("embed", "final_norm", "attn_norm", "mlp_norm", "q_norm", "k_norm"):
            tmp[k] = dev(base[k])
            setattr(bw, k, _ptr(tmp[k]))
        for i, n in enumerate(LINEARS):
            tmp["w" + n] = dev(base["w" + n])
            bw.w[i] = _ptr(tmp["w" + n])
        aw = pbd_adapter_weights()
        for i, n in enumerate(LINEARS):
            tmp["a_" + n] = dev(adapter["a_" + n])
            tmp["b_" + n] = dev(adapter["b_" + n])
            aw.lora_a[i] = _ptr(tmp["a_" + n])
            aw.lora_b[i] = _ptr(tmp["b_" + n])
        tmp["mask_embed"] = dev(adapter["mask_embed"])
        aw.mask_embed = _ptr(tmp["mask_embed"])
        torch.cuda.synchronize(self.device)
        base_addr = self.workspace.data_ptr()
        aligned = (base_addr + 255) // 256 * 256
        ctx = C.c_void_p()
        self._check(self.lib.pbd_create(C.byref(self.cfg), C.byref(bw), C.byref(aw), aligned,
                                        need + 256 - (aligned - base_addr), self.stream.cuda_stream, C.byref(ctx)),
                    None)
        self.ctx = ctx
        if keep_host_weights:
            self._weights = tmp
        del tmp
        self.batch = 0
        self.max_new = 0

    # -- helpers
    def _call(self, fn, *args):
        """Run one library call on the engine's stream, ordered after and before torch's current stream."""
        cur = self.torch.cuda.current_stream(self.device)
        self.stream.wait_stream(cur)
        status = fn(self.ctx, *args)
        cur.wait_stream(self.stream)
        self._check(status)

    def _check(self, status: int, ctx=None):
        if status != PBD_OK:
            msg = self.lib.pbd_last_error(ctx if ctx is not None else getattr(self, "ctx", None))
            raise PbdError(status, (msg or b"").decode())

    def close(self):
        if getattr(self, "ctx", None):
            self.lib.pbd_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _i32(self, n):
        return self.torch.empty(n, dtype=self.torch.int32, device=self.device)

    # -- C ABI calls, same names
    def pbd_prefill(self, prompts: Sequence[np.ndarray], max_new: int):
        torch = self.torch
        lens = np.array([len(p) for p in prompts], dtype=np.int32)
        packed = torch.from_numpy(np.concatenate([np.asarray(p, np.int32) for p in prompts])).to(self.device)
        first = self._i32(len(prompts))
        self._call(self.lib.pbd_prefill, len(prompts), packed.data_ptr(), lens.ctypes.data, max_new,
                   first.data_ptr())
        self.batch, self.max_new = len(prompts), max_new
        return first

    def pbd_draft_block(self, want_logits: bool = False):
        d = self._i32(self.batch * self.D)
        lg = (self.torch.empty(self.batch * self.D * self.shape.vocab, dtype=self.torch.float32, device=self.device)
              if want_logits else None)
        self._call(self.lib.pbd_draft_block, d.data_ptr(), _ptr(lg))
        return d.view(self.batch, self.D), (lg.view(self.batch, self.D, -1) if lg is not None else None)

    def pbd_verify_block(self, drafts=None, want_logits: bool = False):
        v = self._i32(self.batch * (self.D + 1))
        lg = (self.torch.empty(self.batch * (self.D + 1) * self.shape.vocab, dtype=self.torch.float32,
                               device=self.device) if want_logits else None)
        dp = None
        if drafts is not None:
            drafts = self.torch.as_tensor(drafts, dtype=self.torch.int32).to(self.device).contiguous()
            dp = drafts.data_ptr()
        self._call(self.lib.pbd_verify_block, dp, v.data_ptr(), _ptr(lg))
        return v.view(self.batch, self.D + 1), (lg.view(self.batch, self.D + 1, -1) if lg is not None else None)

    def pbd_accept_commit(self, forced_n=None):
        n = self._i32(self.batch)
        fp = None
        if forced_n is not None:
            forced_n = self.torch.as_tensor(forced_n, dtype=self.torch.int32).to(self.device).contiguous()
            fp = forced_n.data_ptr()
        self._call(self.lib.pbd_accept_commit, fp, n.data_ptr())
        return n

    def pbd_decode_step(self, want_logits: bool = False):
        t = self._i32(self.batch)
        lg = (self.torch.empty(self.batch * self.shape.vocab, dtype=self.torch.float32, device=self.device)
              if want_logits else None)
        self._call(self.lib.pbd_decode_step, t.data_ptr(), _ptr(lg))
        return t, (lg.view(self.batch, -1) if lg is not None else None)

    def pbd_generate(self, prompts: Sequence[np.ndarray], max_new: int, mode: int = 0, forced_n_seq=None):
        torch = self.torch
        lens = np.array([len(p) for p in prompts], dtype=np.int32)
        packed = torch.from_numpy(np.concatenate([np.asarray(p, np.int32) for p in prompts])).to(self.device)
        out = self._i32(len(prompts) * max_new)
        fp = None
        if forced_n_seq is not None:
            forced_n_seq = torch.as_tensor(forced_n_seq, dtype=torch.int32).to(self.device).contiguous()
            fp = forced_n_seq.data_ptr()
        st = pbd_stats()
        self._call(self.lib.pbd_generate, len(prompts), packed.data_ptr(), lens.ctypes.data, max_new,
                   mode, fp, out.data_ptr(), C.byref(st))
        self.batch, self.max_new = len(prompts), max_new
        return out.view(len(prompts), max_new), st

    def pbd_get_state(self):
        n = max(self.batch, 1)
        L = np.zeros(n, np.int32)
        p = np.zeros(n, np.int32)
        o = np.zeros(n, np.int32)
        self._call(self.lib.pbd_get_state, L.ctypes.data, p.ctypes.data, o.ctypes.data)
        return L, p, o

    def pbd_get_tokens(self):
        out = self._i32(self.batch * self.max_new)
        self._call(self.lib.pbd_get_tokens, out.data_ptr())
        self.pbd_sync()
        return out.view(self.batch, self.max_new)

    def pbd_read_kv(self, layer: int, seq: int, n: int):
        w = self.shape.n_kv_heads * self.shape.head_dim
        k = self.torch.empty(n * w, dtype=self.torch.bfloat16, device=self.device)
        v = self.torch.empty(n * w, dtype=self.torch.bfloat16, device=self.device)
        self._call(self.lib.pbd_read_kv, layer, seq, n, k.data_ptr(), v.data_ptr())
        self.pbd_sync()
        return k.view(n, w), v.view(n, w)

    def pbd_sync(self):
        self._call(self.lib.pbd_sync)

    def pbd_bench_rounds(self, mode: int, warmup: int, steps: int, forced_n_seq=None):
        """Returns (ms_draft, ms_verify_or_ar, ms_commit, ms_total, launches_per_round) summed over the steps."""
        ms = np.zeros(4, np.float64)
        launches = np.zeros(1, np.int32)
        fp = None
        if forced_n_seq is not None:
            forced_n_seq = self.torch.as_tensor(forced_n_seq, dtype=self.torch.int32).to(self.device).contiguous()
            fp = forced_n_seq.data_ptr()
        self._call(self.lib.pbd_bench_rounds, mode, warmup, steps, fp, ms.ctypes.data, launches.ctypes.data)
        return float(ms[0]), float(ms[1]), float(ms[2]), float(ms[3]), int(launches[0])

    def pbd_trace_pass(self, kind: int, cap: int = 400000):
        """(items [n, 4] int32 {op|lin<<8|layer<<16, a, b, c}, stamps [n, 16] uint64 ns) of one traced pass."""
        items = np.zeros(cap * 4, np.int32)
        tr = np.zeros(cap * TRACE_STAMPS, np.uint64)
        n = np.zeros(1, np.int32)
        self._call(self.lib.pbd_trace_pass, kind, items.ctypes.data, tr.ctypes.data, cap, n.ctypes.data)
        k = int(n[0])
        return items[: 4 * k].reshape(k, 4), tr[: TRACE_STAMPS * k].reshape(k, TRACE_STAMPS)

    def pbd_check_stalled_pass(self):
        """(status, device code) of a verify pass missing one item (see include/pbd.h)."""
        code = np.zeros(1, np.int32)
        status = self.lib.pbd_check_stalled_pass(self.ctx, code.ctypes.data)
        return int(status), int(code[0])

    def pbd_time_pass(self, kind: int, iters: int):
        """(ms per launch, algorithmic bytes per launch) of the persistent pass kernel timed alone
        (kind 0 draft, 1 verify, 2 plain decoding)."""
        ms = np.zeros(1, np.float64)
        nb = np.zeros(1, np.float64)
        self._call(self.lib.pbd_time_pass, kind, iters, ms.ctypes.data, nb.ctypes.data)
        return float(ms[0]), float(nb[0])
