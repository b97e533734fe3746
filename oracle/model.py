"""Python harness of the CPU oracle (test infrastructure; see the package docstring).

The C library (pbd_oracle.c) computes one forward pass.  This module owns the
speculative loop of the paper's Section 3:
  1. enable the adapter and append D masked positions after the pending token;
  2. denoise the block in one draft pass (row j proposes the token at position L+j+1);
  3. disable the adapter and run the causal verifier on [pending, d_1..d_D];
  4. accept the longest prefix d_1..d_n that matches the verifier's greedy tokens;
  5. append d_1..d_n and the verifier's token v_n, and repeat until the budget is met.
and plain greedy decoding by the verifier (the result that exact verification must
reproduce, Section 4.1 and Appendix A.1).
"""
from __future__ import annotations

import ctypes as C
from typing import Callable, Dict, List, Optional, Sequence

import numpy as np

from .build import build

MASK_CAUSAL = 0
MASK_BLOCK_DRAFT = 1

# The seven block linears carrying the adapter (Appendix A.2: "all linear projection
# modules in the transformer blocks"), in the C library's order.
LINEAR_NAMES = ("q", "k", "v", "o", "gate", "up", "down")


def _linear_dims(shape, name):
    H, q, kv, I = shape.hidden, shape.n_q_heads * shape.head_dim, shape.n_kv_heads * shape.head_dim, shape.intermediate
    return {"q": (H, q), "k": (H, kv), "v": (H, kv), "o": (q, H), "gate": (H, I), "up": (H, I), "down": (I, H)}[name]


def adapter_param_count(shape) -> int:
    """Trainable LoRA parameters the oracle's forward uses: per layer, r*(in+out) per adapted linear."""
    return shape.n_layers * sum(shape.lora_rank * sum(_linear_dims(shape, n)) for n in LINEAR_NAMES)


def base_param_count(shape) -> int:
    """Backbone parameters the oracle's forward reads: tied embedding, 7 linears and 4 norms per layer, final norm."""
    per_layer = sum(i * o for i, o in (_linear_dims(shape, n) for n in LINEAR_NAMES))
    per_layer += 2 * shape.hidden + 2 * shape.head_dim
    return shape.vocab * shape.hidden + shape.n_layers * per_layer + shape.hidden


class _Config(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("hidden", C.c_int32), ("n_q_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32), ("intermediate", C.c_int32),
                ("vocab", C.c_int32), ("rms_eps", C.c_float), ("rope_theta", C.c_float),
                ("lora_rank", C.c_int32), ("lora_scale", C.c_float)]


_U16P = C.POINTER(C.c_uint16)


class _Weights(C.Structure):
    _fields_ = [("embed", _U16P), ("final_norm", _U16P), ("attn_norm", _U16P), ("mlp_norm", _U16P),
                ("q_norm", _U16P), ("k_norm", _U16P), ("w", _U16P * 7), ("lora_a", _U16P * 7),
                ("lora_b", _U16P * 7), ("mask_embed", _U16P)]


_libs = {}


def lib(variant: str = "f32"):
    """The oracle library: 'f32' (reference) or 'f64acc' (fp64 accumulators, drift measurement only)."""
    if variant not in _libs:
        L = C.CDLL(build(variant=variant))
        F = C.POINTER(C.c_float)
        I32 = C.POINTER(C.c_int32)
        L.orc_cache_new.restype = C.c_void_p
        L.orc_cache_new.argtypes = [C.POINTER(_Config), C.c_int32]
        L.orc_cache_free.argtypes = [C.c_void_p]
        L.orc_cache_copy.argtypes = [C.POINTER(_Config), C.c_void_p, C.c_void_p, C.c_int32]
        L.orc_cache_read.argtypes = [C.POINTER(_Config), C.c_void_p, C.c_int32, C.c_int32, C.c_int32, F]
        L.orc_cache_write.argtypes = [C.POINTER(_Config), C.c_void_p, C.c_int32, C.c_int32, C.c_int32, F, F]
        L.orc_forward.argtypes = [C.POINTER(_Config), C.POINTER(_Weights), C.c_void_p, C.c_int32, C.c_int32, I32,
                                  C.c_int32, C.c_int32, C.c_int32, C.c_int32, F, I32, F, C.c_uint64]
        L.orc_forward.restype = C.c_int32
        L.orc_op_rmsnorm.argtypes = [C.c_int32, C.c_int32, F, _U16P, C.c_float, F]
        L.orc_op_linear.argtypes = [C.POINTER(_Config), C.c_int32, C.c_int32, C.c_int32, F, _U16P, _U16P, _U16P,
                                    C.c_int32, F]
        L.orc_op_rope.argtypes = [F, C.c_int32, C.c_int32, C.c_double]
        L.orc_op_swiglu.argtypes = [C.c_int32, F, F, F]
        L.orc_op_attention.argtypes = [C.POINTER(_Config), C.c_int32, C.c_void_p, C.c_int32, C.c_int32, C.c_int32,
                                       F, F]
        L.orc_round_bf16.argtypes = [C.c_float]
        L.orc_round_bf16.restype = C.c_float
        L.orc_num_threads.restype = C.c_int32
        _libs[variant] = L
    return _libs[variant]


def _fp(a: np.ndarray):
    return a.ctypes.data_as(C.POINTER(C.c_float))


def _u16(a: np.ndarray):
    return a.ctypes.data_as(_U16P)


def _i32(a: np.ndarray):
    return a.ctypes.data_as(C.POINTER(C.c_int32))


def make_config(shape) -> _Config:
    return _Config(shape.n_layers, shape.hidden, shape.n_q_heads, shape.n_kv_heads, shape.head_dim,
                   shape.intermediate, shape.vocab, shape.rms_eps, shape.rope_theta, shape.lora_rank,
                   shape.lora_alpha / shape.lora_rank)


class OracleCache:
    """Per-sequence KV cache: [layers][capacity][kv_heads*head_dim] fp32 holding bf16 values."""

    def __init__(self, model: "OracleModel", capacity: int):
        self.model = model
        self.capacity = capacity
        self.ptr = lib().orc_cache_new(C.byref(model.cfg), capacity)
        if not self.ptr:
            raise MemoryError("oracle cache allocation failed")

    def __del__(self):
        if getattr(self, "ptr", None):
            lib().orc_cache_free(self.ptr)
            self.ptr = None

    def read(self, layer: int, which: str, n: int) -> np.ndarray:
        s = self.model.shape
        out = np.empty((n, s.n_kv_heads * s.head_dim), dtype=np.float32)
        rc = lib().orc_cache_read(C.byref(self.model.cfg), self.ptr, layer, 0 if which == "k" else 1, n, _fp(out))
        assert rc == 0
        return out

    def write(self, layer: int, L: int, k: np.ndarray, v: np.ndarray):
        k = np.ascontiguousarray(k, dtype=np.float32)
        v = np.ascontiguousarray(v, dtype=np.float32)
        rc = lib().orc_cache_write(C.byref(self.model.cfg), self.ptr, layer, L, k.shape[0], _fp(k), _fp(v))
        assert rc == 0

    def copy_to(self, other: "OracleCache", n: int):
        assert lib().orc_cache_copy(C.byref(self.model.cfg), self.ptr, other.ptr, n) == 0


class OracleModel:
    """Holds the config and the bf16 weight arrays (uint16 bit patterns) for the C library."""

    def __init__(self, shape, base: Dict[str, np.ndarray], adapter: Dict[str, np.ndarray], acc: str = "f32"):
        self.shape = shape
        self.acc = acc
        self.cfg = make_config(shape)
        nl, r = shape.n_layers, shape.lora_rank
        keep = {}

        def arr(a, expect):
            a = np.ascontiguousarray(a, dtype=np.uint16)
            if tuple(a.shape) != tuple(expect):
                raise ValueError("shape %s != %s" % (a.shape, expect))
            keep[id(a)] = a
            return a

        H, d = shape.hidden, shape.head_dim
        W = _Weights()
        W.embed = _u16(arr(base["embed"], (shape.vocab, H)))
        W.final_norm = _u16(arr(base["final_norm"], (H,)))
        W.attn_norm = _u16(arr(base["attn_norm"], (nl, H)))
        W.mlp_norm = _u16(arr(base["mlp_norm"], (nl, H)))
        W.q_norm = _u16(arr(base["q_norm"], (nl, d)))
        W.k_norm = _u16(arr(base["k_norm"], (nl, d)))
        for t, name in enumerate(LINEAR_NAMES):
            fin, fout = _linear_dims(shape, name)
            W.w[t] = _u16(arr(base["w" + name], (nl, fout, fin)))
            W.lora_a[t] = _u16(arr(adapter["a_" + name], (nl, r, fin)))
            W.lora_b[t] = _u16(arr(adapter["b_" + name], (nl, fout, r)))
        W.mask_embed = _u16(arr(adapter["mask_embed"], (H,)))
        self.weights = W
        self._keep = keep

    def new_cache(self, capacity: int) -> OracleCache:
        return OracleCache(self, capacity)

    def forward(self, cache: OracleCache, L: int, tokens: Sequence[int], adapter_on: bool, mask_mode: int,
                read_first: int = 0, n_read: Optional[int] = None, want_logits: bool = False,
                want_hidden: bool = False, n_layers: Optional[int] = None, skip_layers: int = 0):
        """One pass over len(tokens) rows at positions L.. (token < 0 = mask row).

        n_layers: run only the first n_layers decoder layers, then the final norm and the tied
        head (the early exit of Section 6); the skipped layers' cache slots are left untouched.
        skip_layers: bit l set skips decoder layer l (layer skipping, Section 6); its cache slots
        are left untouched too.
        Returns (argmax[n_read], logits[n_read, V] or None, hidden[n_read, H] or None).
        """
        cfg = self.cfg
        if n_layers is not None:
            if not 1 <= n_layers <= self.shape.n_layers:
                raise ValueError("n_layers %d outside [1, %d]" % (n_layers, self.shape.n_layers))
            cfg = _Config.from_buffer_copy(self.cfg)
            cfg.n_layers = n_layers
        toks = np.ascontiguousarray(np.asarray(tokens, dtype=np.int32))
        n = toks.shape[0]
        if n_read is None:
            n_read = n - read_first
        am = np.empty(n_read, dtype=np.int32)
        logits = np.empty((n_read, self.shape.vocab), dtype=np.float32) if want_logits else None
        hidden = np.empty((n_read, self.shape.hidden), dtype=np.float32) if want_hidden else None
        rc = lib(self.acc).orc_forward(C.byref(cfg), C.byref(self.weights), cache.ptr, L, n, _i32(toks),
                               int(adapter_on), mask_mode, read_first, n_read,
                               _fp(logits) if logits is not None else None, _i32(am),
                               _fp(hidden) if hidden is not None else None, int(skip_layers))
        if rc != 0:
            raise ValueError("oracle forward rejected its arguments (cache capacity or token range)")
        return am, logits, hidden

    def prefill(self, prompt: Sequence[int], capacity: int, want_logits: bool = False):
        """Causal, adapter-off pass over the prompt; returns (cache, first token, logits of the last row)."""
        cache = self.new_cache(capacity)
        P = len(prompt)
        am, lg, _ = self.forward(cache, 0, prompt, False, MASK_CAUSAL, read_first=P - 1, n_read=1,
                                 want_logits=want_logits)
        return cache, int(am[0]), (lg[0] if lg is not None else None)


def accept_length(draft: Sequence[int], verify: Sequence[int]) -> int:
    """Longest accepted prefix (Section 3, step 4; exact greedy top-1 matching, Appendix A.1).

    draft = [d_1..d_D] and verify = [v_0..v_D], where v_j is the verifier's greedy token
    after the row holding d_j (d_0 = the pending token).  d_i is accepted while it
    equals v_{i-1}: n = max{k <= D : d_i == v_{i-1} for all i <= k}.
    """
    n = 0
    D = len(draft)
    while n < D and int(draft[n]) == int(verify[n]):
        n += 1
    return n


def draft_block(model: OracleModel, cache: OracleCache, L: int, p: int, D: int, draft_layers: Optional[int] = None,
                denoise_steps: int = 1, anchored: bool = True, want_logits: bool = False, draft_skip: int = 0):
    """The adapter-on draft of one round (Section 3, steps 1-2) and its variants.

    Step 1 runs rows [p, MASK x D] at positions L..L+D under the block mask.  The token it
    proposes for position L+j (j = 1..D) is d_j:
      anchored (the default): row j-1 proposes position L+j (rows 0..D-1 are read);
      unanchored (ablation of Sections 4.4 and 5.3): mask row j proposes its own position
        (rows 1..D are read; the pending token's row is context only).
    denoise_steps > 1 (the two-step ablation of Sections 4.4 and 5.3): each further step
    runs the same adapter-on block pass with the mask rows replaced by the previous step's
    proposals, rows [p, d_1..d_D], nothing remasked; its proposals replace the block.
    draft_layers: the draft exits after the first draft_layers decoder layers (the early exit
    Section 6 names as a cheaper draft path); None runs all of them.  draft_skip: a mask of
    decoder layers the draft skips (layer skipping, the other cheaper path Section 6 names).
    Returns (drafts of the last step, its logits or None, proposals of every step).
    """
    first = 0 if anchored else 1
    rows = [p] + [-1] * D
    steps = []
    lg = None
    for _ in range(max(1, denoise_steps)):
        am, lg, _ = model.forward(cache, L, rows, True, MASK_BLOCK_DRAFT, first, D, want_logits=want_logits,
                                  n_layers=draft_layers, skip_layers=draft_skip)
        drafts = [int(t) for t in am]
        steps.append(drafts)
        rows = [p] + drafts
    return steps[-1], lg, steps


def greedy_generate(model: OracleModel, prompt: Sequence[int], max_new: int):
    """Plain greedy decoding by the adapter-off verifier: the output exact verification must reproduce."""
    P = len(prompt)
    cache, tok, _ = model.prefill(prompt, P + max_new + 1)
    out = [tok]
    L = P
    while len(out) < max_new:
        am, _, _ = model.forward(cache, L, [out[-1]], False, MASK_CAUSAL, 0, 1)
        out.append(int(am[0]))
        L += 1
    return out


def spec_generate(model: OracleModel, prompt: Sequence[int], max_new: int, D: int,
                  forced_n: Optional[Sequence[int]] = None,
                  draft_override: Optional[Callable[[int, List[int]], List[int]]] = None,
                  want_logits: bool = False, max_rounds: Optional[int] = None, return_state: bool = False,
                  draft_layers: Optional[int] = None, denoise_steps: int = 1, anchored: bool = True,
                  draft_skip: int = 0):
    """PEFT-BD decoding (Section 3).  Returns (tokens, rounds[, (cache, L)]).

    rounds[i] = dict(L=cached length before the round, pending, draft, verify, n, emitted,
    draft_steps, [draft_logits, verify_logits]).  forced_n replaces the accepted length of
    round i by forced_n[i] (timing mode); draft_override(i, drafts) may replace the drafted
    block (adversarial drafters in the tests).  draft_layers, denoise_steps, anchored and
    draft_skip select the draft variant (draft_block).  The generation budget is the only stop rule:
    the last round is truncated to max_new tokens.
    """
    P = len(prompt)
    cache, p, _ = model.prefill(prompt, P + max_new + D + 1)
    out = [p]
    L = P
    rounds = []
    while len(out) < max_new and (max_rounds is None or len(rounds) < max_rounds):
        ri = len(rounds)
        drafts, d_lg, d_steps = draft_block(model, cache, L, p, D, draft_layers, denoise_steps, anchored,
                                            want_logits, draft_skip)
        if draft_override is not None:
            drafts = [int(t) for t in draft_override(ri, list(drafts))]
        v_am, v_lg, _ = model.forward(cache, L, [p] + drafts, False, MASK_CAUSAL, 0, D + 1,
                                      want_logits=want_logits)
        verify = [int(t) for t in v_am]
        n = accept_length(drafts, verify)
        if forced_n is not None:
            n = int(forced_n[ri])
        emitted = drafts[:n] + [verify[n]]
        take = min(len(emitted), max_new - len(out))
        rec = dict(L=L, pending=p, draft=drafts, verify=verify, n=n, emitted=emitted[:take], draft_steps=d_steps)
        if want_logits:
            rec["draft_logits"], rec["verify_logits"] = d_lg, v_lg
        rounds.append(rec)
        out.extend(emitted[:take])
        L += n + 1
        p = verify[n]
    if return_state:
        return out, rounds, (cache, L)
    return out, rounds
