"""The benchmark's byte model and bookkeeping, pinned without a GPU.

- Algorithmic bytes of a pass (the roofline numerator): the closed form for the Qwen3-0.6B
  shape, 1,192,099,840 B of weights and norm gains per pass plus 114,688 B per token of KV
  (read for the cached tokens, written for the block's rows), and 20,185,088 B more for the
  adapter in the draft pass.  The closed form is re-derived here from the parameter counts the
  oracle pins against the paper (596,049,920 base and 10,092,544 adapter parameters).
- The traffic record keys on the kernel source without its comments.
"""
import importlib.util
import os

import numpy as np
import pytest

import oracle
from paper_2607_12422_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_module", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_pass_bytes_closed_form(bench):
    S = synth.QWEN3_0_6B
    # every base parameter once (bf16), the tied embedding once, the final norm gain once
    base = 2 * oracle.base_param_count(S)
    kv_tok = 2 * 2 * S.n_layers * S.n_kv_heads * S.head_dim
    assert base == 1_192_099_840 and kv_tok == 114_688
    for L in (0, 512, 613, 4096):
        assert bench.pass_bytes(S, L, 17, False) == base + kv_tok * (L + 17)
        assert bench.pass_bytes(S, L, 17, True) - bench.pass_bytes(S, L, 17, False) == 2 * oracle.adapter_param_count(S)
    assert 2 * oracle.adapter_param_count(S) == 20_185_088


def test_source_hash_ignores_comments(bench, tmp_path):
    a = tmp_path / "a.cu"
    b = tmp_path / "b.cu"
    c = tmp_path / "c.cu"
    a.write_text("int f(int x) {\n  return x + 1;  // one more\n}\n")
    b.write_text("/* header */\nint f(int x) {\n    return x + 1;\n}\n")
    c.write_text("int f(int x) {\n  return x + 2;\n}\n")
    assert bench.source_hash(str(a)) == bench.source_hash(str(b))
    assert bench.source_hash(str(a)) != bench.source_hash(str(c))


def test_verify_flops_closed_form(bench):
    """2 FLOPs per multiply-add over every linear and the tied head (the pinned base parameters
    less the 65,536 norm gains) for each of the 17 rows, plus causal attention: QK^T and PV of
    d = 128 per visible key, 16 query heads, 28 layers, row j seeing L + j + 1 keys."""
    S = synth.QWEN3_0_6B
    matmul_params = oracle.base_param_count(S) - (S.n_layers * (2 * S.hidden + 2 * S.head_dim) + S.hidden)
    assert matmul_params == 595_984_384
    for L in (0, 512, 4096):
        keys = sum(L + j + 1 for j in range(17))
        assert bench.verify_flops(S, L, 1, 16) == 2 * 17 * matmul_params + 4 * 128 * 16 * 28 * keys
    assert bench.verify_flops(S, 512, 1, 16) == 22_295_052_288
    # a batch: the linears scale with the rows, the attention with each sequence's own keys
    Ls = [420, 1757, 900]
    keys = sum(L + j + 1 for L in Ls for j in range(17))
    assert bench.verify_flops(S, sum(Ls), 3, 16) == 2 * 51 * matmul_params + 4 * 128 * 16 * 28 * keys


class _FakeEngine:
    """Stands in for the engine in the benchmark's bookkeeping: every speculative round emits the
    forced n + 1 tokens per sequence (2 without forcing) and reports 1, 2 and 0.01 ms for draft,
    verify and commit (3.01 ms in all); a plain-decoding step emits one token in 2.01 ms (no
    draft)."""

    def __init__(self, shape, base, adapter, block_D, max_batch, max_seq_len, device=None, **kw):
        self.D = block_D

    def pbd_prefill(self, prompts, max_new):
        self.G = max_new
        self.L = np.array([len(p) for p in prompts], np.int64)
        self.n = np.ones(len(prompts), np.int64)

    def pbd_get_state(self):
        return self.L.copy(), np.zeros_like(self.L), self.n.copy()

    def pbd_bench_rounds(self, mode, warmup, steps, forced=None):
        for i in range(steps):
            for b in range(len(self.n)):
                A = 1 if mode == 1 else (int(forced[i, b]) + 1 if forced is not None else 2)
                take = min(A, self.G - self.n[b])
                self.n[b] += take
                self.L[b] += take
        if mode == 1:
            return 0.0, 2.0 * steps, 0.01 * steps, 2.01 * steps, 5
        return 1.0 * steps, 2.0 * steps, 0.01 * steps, 3.01 * steps, 9

    def close(self):
        pass


class _FakePbd:
    Engine = _FakeEngine


def test_other_workloads_bookkeeping(bench):
    out = bench.measure_configs(_FakePbd, synth, None, None, "cpu", 6780.0, 3)
    tf, _ = bench.bf16_peak()
    S = synth.QWEN3_0_6B
    for name, B, P_sum in (("qwen3-0.6b-b1-d16-p4096-g512", 1, 4096),
                           ("qwen3-0.6b-b8-d16-p256to2048-g256", 8,
                            sum(synth.WORKLOADS["qwen3-0.6b-b8-d16-p256to2048-g256"].prompt_lens))):
        r = out[name]
        W = synth.WORKLOADS[name]
        assert r["batch"] == B and r["draft_us"] == pytest.approx(1000.0) and r["verify_us"] == pytest.approx(2000.0)
        assert r["mean_tokens_per_round_per_seq"] == pytest.approx(2.0)  # no timed round is cut by the budget
        assert r["tokens_per_s"] == pytest.approx(2.0 * B / 3.01e-3)
        assert P_sum < r["kv_tokens_mean"] < P_sum + B * W.max_new
        L = r["kv_tokens_mean"]
        assert r["verify_roofline_frac"] == pytest.approx(bench.pass_bytes(S, L, B * 17, False) / 6780e9 / 2e-3)
        assert r["verify_tensor_frac"] == pytest.approx(bench.verify_flops(S, L, B, 16) / 2e-3 / (tf * 1e12))
    sweep = out["qwen3-0.6b-b1-p1024-dsweep-forced"]
    for D in (4, 8, 16, 32):
        row = sweep["D=%d" % D]
        assert row["ar_us_per_token"] == pytest.approx(2010.0)
        assert row["break_even_accept"] == pytest.approx(3000.0 / 2010.0)  # draft + verify over one step
        assert row["mean_A_1"]["tokens_per_round"] == pytest.approx(1.0)
        for m in ("mean_A_1", "mean_A_3", "mean_A_6"):
            a = row[m]
            assert a["step_us"] == pytest.approx(3010.0)
            assert a["speedup_vs_ar"] == pytest.approx(a["tokens_per_round"] * 2010.0 / 3010.0)
            assert a["tokens_per_s"] == pytest.approx(a["tokens_per_round"] / 3.01e-3)
