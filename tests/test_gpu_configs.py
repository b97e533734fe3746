"""Full-size parity against the CPU oracle on the long-context, batched and block-size
workloads of the Qwen3-0.6B shape (28 layers, vocab 151936, rank 16), in lockstep over several
speculative rounds (see _parity.py for what is compared and recorded):

- 4096-token prompt, D = 16: three rounds;
- batch of 8 ragged prompts (420..1757 tokens), D = 16: three batched rounds, every sequence
  compared with its own oracle run (the longest ones exercise the deepest split-KV merges);
- 1024-token prompt, D in {4, 8, 16, 32} (the block-size sweep): three rounds each.
"""
import numpy as np
import pytest

import _parity
import oracle
from paper_2607_12422_gb300 import synth

pytestmark = pytest.mark.gpu
ROUNDS = 3


@pytest.fixture(scope="module")
def cenv():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_12422_gb300 import pbd
    S = synth.QWEN3_0_6B
    base, ad = synth.gen_base_weights(S), synth.gen_adapter(S)
    return dict(torch=torch, pbd=pbd, S=S, base=base, ad=ad, m=oracle.OracleModel(S, base, ad),
                m64=oracle.OracleModel(S, base, ad, acc="f64acc"))


def test_long_context_4096_rounds(cenv):
    W = synth.WORKLOADS["qwen3-0.6b-b1-d16-p4096-g512"]
    prompt = synth.gen_prompts(W.shape, list(W.prompt_lens))[0]
    eng = cenv["pbd"].Engine(cenv["S"], cenv["base"], cenv["ad"], block_D=W.block_D, max_batch=1,
                             max_seq_len=len(prompt) + 96)
    seqs = {0: _parity.Seq(cenv["m"], cenv["m64"], prompt, W.block_D, ROUNDS)}
    _parity.start(eng, [prompt], seqs, 64, W.name)
    _parity.rounds(eng, seqs, ROUNDS, W.name)
    eng.close()


def test_batch8_ragged_rounds(cenv):
    W = synth.WORKLOADS["qwen3-0.6b-b8-d16-p256to2048-g256"]
    prompts = synth.gen_prompts(W.shape, list(W.prompt_lens))
    eng = cenv["pbd"].Engine(cenv["S"], cenv["base"], cenv["ad"], block_D=W.block_D, max_batch=8,
                             max_seq_len=max(W.prompt_lens) + 96)
    seqs = {b: _parity.Seq(cenv["m"], cenv["m64"], prompts[b], W.block_D, ROUNDS) for b in range(len(prompts))}
    _parity.start(eng, prompts, seqs, 64, W.name)
    _parity.rounds(eng, seqs, ROUNDS, W.name)
    eng.close()


@pytest.fixture(scope="module")
def sweep(cenv):
    """The block-size sweep's 1024-token prompt, prefilled once on both oracles; each block size
    continues from a copy of that cache."""
    W = synth.WORKLOADS["qwen3-0.6b-b1-p1024-dsweep-forced"]
    prompt = synth.gen_prompts(W.shape, list(W.prompt_lens))[0]
    return W, prompt, _parity.Seq(cenv["m"], cenv["m64"], prompt, max(W.D_sweep), ROUNDS)


@pytest.mark.parametrize("D", [4, 8, 16, 32])
def test_block_size_sweep_rounds(cenv, sweep, D):
    W, prompt, base_sq = sweep
    assert D in W.D_sweep
    P = len(prompt)
    sq = _parity.Seq.__new__(_parity.Seq)
    sq.m, sq.m64, sq.D, sq.L, sq.p, sq.lg0 = base_sq.m, base_sq.m64, D, P, base_sq.p, base_sq.lg0
    cap = P + (ROUNDS + 1) * (max(W.D_sweep) + 1)
    sq.cache, sq.cache64 = sq.m.new_cache(cap), sq.m64.new_cache(cap)
    base_sq.cache.copy_to(sq.cache, P)
    base_sq.cache64.copy_to(sq.cache64, P)
    eng = cenv["pbd"].Engine(cenv["S"], cenv["base"], cenv["ad"], block_D=D, max_batch=1, max_seq_len=P + 160)
    seqs = {0: sq}
    _parity.start(eng, [prompt], seqs, 96, "%s-D%d" % (W.name, D))
    _parity.rounds(eng, seqs, ROUNDS, "%s-D%d" % (W.name, D))
    eng.close()
