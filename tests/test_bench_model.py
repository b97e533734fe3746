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
