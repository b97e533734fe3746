"""Seeded synthetic inputs: model shapes, random-init weights, adapters, prompts.

This module is data only.  It draws the numbers that both the GPU library and the
CPU oracle consume and holds none of the decoding arithmetic: no forward pass, no
acceptance rule, no attention.  Weights are drawn N(0, 0.02) in float32 from
numpy's PCG64 and stored as bfloat16 bit patterns (uint16) by round-to-nearest-even,
so every consumer sees identical bytes.

Shapes follow the paper's model (Qwen3-0.6B, Section 4.1) and its adapter
(rank 16, alpha 32, on all seven block linears, Appendix A.2).  The paper trains
the adapter; no trained weights exist here, so A, B and the mask embedding are
random too.  Norm gains are 1.0 (a random gain of scale 0.02 would shrink the
logits to a width where near-ties dominate the argmax).

Seeds are fixed per role: base weights 0, adapter 1, prompts 2, forced accepted
lengths 3.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional, Sequence

import numpy as np

# Order of the seven adapted linears, shared by the C ABI and the oracle.
LINEARS = ("q", "k", "v", "o", "gate", "up", "down")

SEED_WEIGHTS = 0
SEED_ADAPTER = 1
SEED_PROMPTS = 2
SEED_FORCED = 3
INIT_STD = 0.02


@dataclasses.dataclass(frozen=True)
class ModelShape:
    name: str
    n_layers: int
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    intermediate: int
    vocab: int
    rms_eps: float = 1e-6
    rope_theta: float = 1e6
    lora_rank: int = 16
    lora_alpha: float = 32.0

    @property
    def lora_scale(self) -> float:
        return self.lora_alpha / self.lora_rank

    def linear_dims(self, name: str):
        """(in_features, out_features) of one block linear."""
        H, q, kv, I = self.hidden, self.n_q_heads * self.head_dim, self.n_kv_heads * self.head_dim, self.intermediate
        return {"q": (H, q), "k": (H, kv), "v": (H, kv), "o": (q, H),
                "gate": (H, I), "up": (H, I), "down": (I, H)}[name]


TINY = ModelShape("tiny-qwen3", n_layers=2, hidden=256, n_q_heads=4, n_kv_heads=2, head_dim=64,
                  intermediate=768, vocab=4096, lora_rank=8, lora_alpha=16.0)
QWEN3_0_6B = ModelShape("qwen3-0.6b", n_layers=28, hidden=1024, n_q_heads=16, n_kv_heads=8, head_dim=128,
                        intermediate=3072, vocab=151936, lora_rank=16, lora_alpha=32.0)


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    shape: ModelShape
    batch: int
    block_D: int
    prompt_lens: tuple          # one entry per sequence
    max_new: int
    forced_means: tuple = ()    # forced-acceptance sweep (empty: natural acceptance)
    D_sweep: tuple = ()


def _cfg4_lens() -> tuple:
    rng = np.random.Generator(np.random.PCG64(SEED_PROMPTS))
    return tuple(int(x) for x in rng.integers(256, 2049, size=8))


WORKLOADS = {
    "tiny-b1-d16-p64-g64": Workload("tiny-b1-d16-p64-g64", TINY, 1, 16, (64,), 64),
    "qwen3-0.6b-b1-d16-p512-g256": Workload("qwen3-0.6b-b1-d16-p512-g256", QWEN3_0_6B, 1, 16, (512,), 256),
    "qwen3-0.6b-b1-d16-p4096-g512": Workload("qwen3-0.6b-b1-d16-p4096-g512", QWEN3_0_6B, 1, 16, (4096,), 512),
    "qwen3-0.6b-b8-d16-p256to2048-g256": Workload("qwen3-0.6b-b8-d16-p256to2048-g256", QWEN3_0_6B, 8, 16,
                                                  _cfg4_lens(), 256),
    "qwen3-0.6b-b1-p1024-dsweep-forced": Workload("qwen3-0.6b-b1-p1024-dsweep-forced", QWEN3_0_6B, 1, 16,
                                                  (1024,), 256, forced_means=(1.0, 3.0, 6.0),
                                                  D_sweep=(4, 8, 16, 32)),
}


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bfloat16 bit patterns by IEEE round-to-nearest-even (data encoding only)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    lsb = u >> 16
    lsb &= np.uint32(1)
    w = u + np.uint32(0x7FFF)
    w += lsb
    w >>= 16
    return w.astype(np.uint16)


def bf16_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _normal_bf16(rng: np.random.Generator, shape, std: float = INIT_STD) -> np.ndarray:
    out = np.empty(shape, dtype=np.uint16)
    flat = out.reshape(-1)
    n = flat.size
    chunk = 1 << 22
    buf = np.empty(min(n, chunk), dtype=np.float32)
    for s in range(0, n, chunk):
        e = min(n, s + chunk)
        v = buf[: e - s]
        rng.standard_normal(out=v, dtype=np.float32)
        v *= np.float32(std)
        flat[s:e] = bf16_bits(v)
    return out


def _ones_bf16(shape) -> np.ndarray:
    return np.full(shape, 0x3F80, dtype=np.uint16)


def gen_base_weights(shape: ModelShape, seed: int = SEED_WEIGHTS) -> Dict[str, np.ndarray]:
    """Base (verifier) weights, bf16 bit patterns, layer-stacked, [out, in] row-major.

    Draw order from one PCG64 stream: embed, then wq, wk, wv, wo, wgate, wup, wdown
    (each stacked over layers).  Norm gains are 1.0.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    nl, H, d = shape.n_layers, shape.hidden, shape.head_dim
    w = {"embed": _normal_bf16(rng, (shape.vocab, H))}
    for name in LINEARS:
        fin, fout = shape.linear_dims(name)
        w["w" + name] = _normal_bf16(rng, (nl, fout, fin))
    w["final_norm"] = _ones_bf16((H,))
    w["attn_norm"] = _ones_bf16((nl, H))
    w["mlp_norm"] = _ones_bf16((nl, H))
    w["q_norm"] = _ones_bf16((nl, d))
    w["k_norm"] = _ones_bf16((nl, d))
    return w


def with_random_norm_gains(w: Dict[str, np.ndarray], seed: int = SEED_WEIGHTS + 7) -> Dict[str, np.ndarray]:
    """A copy of base weights whose RMSNorm gains (final, attn, mlp, q, k) are drawn uniformly from
    [0.5, 1.5) and rounded to bf16, in that order from one PCG64 stream; the rest is shared."""
    rng = np.random.Generator(np.random.PCG64(seed))
    out = dict(w)
    for k in ("final_norm", "attn_norm", "mlp_norm", "q_norm", "k_norm"):
        out[k] = bf16_bits(rng.uniform(0.5, 1.5, size=w[k].shape).astype(np.float32))
    return out


def gen_adapter(shape: ModelShape, seed: int = SEED_ADAPTER, zero_B: bool = False) -> Dict[str, np.ndarray]:
    """Adapter weights: per linear A [nl, r, in] and B [nl, out, r], plus mask_embed [H].

    Draw order: A_q, B_q, A_k, B_k, ..., A_down, B_down, mask_embed.  With zero_B the
    B draws still happen (so A and mask_embed are unchanged) and B is then zeroed.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    nl, r = shape.n_layers, shape.lora_rank
    a = {}
    for name in LINEARS:
        fin, fout = shape.linear_dims(name)
        a["a_" + name] = _normal_bf16(rng, (nl, r, fin))
        b = _normal_bf16(rng, (nl, fout, r))
        a["b_" + name] = np.zeros_like(b) if zero_B else b
    a["mask_embed"] = _normal_bf16(rng, (shape.hidden,))
    return a


def gen_prompts(shape: ModelShape, lens: Sequence[int], seed: int = SEED_PROMPTS) -> List[np.ndarray]:
    """Uniform token ids in [0, V) per sequence (stand-in for the TULU-3 prompts)."""
    rng = np.random.Generator(np.random.PCG64(seed + 1000))
    return [rng.integers(0, shape.vocab, size=int(L), dtype=np.int64).astype(np.int32) for L in lens]


def forced_accept_lengths(mean: float, D: int, count: int, seed: int = SEED_FORCED) -> np.ndarray:
    """Seeded accepted-prefix lengths n (0..D) for the forced-acceptance timing mode.

    A = n + 1 follows a truncated geometric law P(A=k) ~ rho^(k-1) on k = 1..D+1, with
    rho found by bisection so that E[A] = mean.  mean <= 1 gives A = 1 always; a mean
    above D+1 gives A = D+1 always.  These are benchmark inputs, not model outputs.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    u = rng.random(count)
    K = D + 1
    if mean <= 1.0:
        return np.zeros(count, dtype=np.int32)
    if mean >= K:
        return np.full(count, D, dtype=np.int32)
    ks = np.arange(1, K + 1, dtype=np.float64)

    def probs(log_rho):
        lw = (ks - 1) * log_rho
        lw -= lw.max()
        p = np.exp(lw)
        return p / p.sum()

    lo, hi = -60.0, 60.0
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if float((probs(mid) * ks).sum()) < mean:
            lo = mid
        else:
            hi = mid
    cdf = np.cumsum(probs(0.5 * (lo + hi)))
    A = np.searchsorted(cdf, u, side="right") + 1
    A = np.minimum(A, K)
    return (A - 1).astype(np.int32)
