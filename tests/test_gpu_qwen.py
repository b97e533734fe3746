"""Full-size parity on the Qwen3-0.6B shape (28 layers, vocab 151936, rank 16, D = 16).

The oracle runs the 512-token prefill and then six speculative rounds in lockstep with the GPU
(both sides on the GPU's tokens; what is compared and recorded is described in _parity.py), and
checks every token of the headline generation teacher-forced.  Properties that hold at any size
run on the GPU for the whole workloads: speculative output equals plain greedy decoding bit for
bit, verify rows equal decode rows bit for bit, and a sequence's tokens do not depend on the
batch it shares."""
import numpy as np
import pytest

import _parity
import oracle
from paper_2607_12422_gb300 import synth

pytestmark = pytest.mark.gpu
D = 16


@pytest.fixture(scope="module")
def big():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_12422_gb300 import pbd
    S = synth.QWEN3_0_6B
    base, ad = synth.gen_base_weights(S), synth.gen_adapter(S)
    eng = pbd.Engine(S, base, ad, block_D=D, max_batch=8, max_seq_len=4096 + 512 + 8)
    return dict(torch=torch, S=S, base=base, ad=ad, eng=eng, model=oracle.OracleModel(S, base, ad))


def test_lockstep_rounds_after_512_prefill(big):
    """Six speculative rounds after the 512-token prefill, in lockstep with the oracle (fp32 and
    fp64 accumulation; see _parity.py): logits within the bound, ids equal to the oracle's argmax
    up to counted near-ties, accepted and cached lengths exact."""
    eng, m = big["eng"], big["model"]
    m64 = oracle.OracleModel(big["S"], big["base"], big["ad"], acc="f64acc")
    W = synth.WORKLOADS["qwen3-0.6b-b1-d16-p512-g256"]
    prompt = synth.gen_prompts(W.shape, list(W.prompt_lens))[0]
    seqs = {0: _parity.Seq(m, m64, prompt, D, 6)}
    _parity.start(eng, [prompt], seqs, W.max_new, W.name)
    _parity.rounds(eng, seqs, 6, W.name)


def test_whole_generation_matches_oracle_greedy(big):
    """All 256 tokens of the headline generation (pbd_generate, speculative rounds on the GPU)
    against the oracle's greedy decoding, teacher-forced on the GPU's tokens: the oracle runs one
    causal pass over the prompt's continuation as generated, and every generated token must be
    that pass's argmax at its position, or a near-tie of the oracle's logits inside the bound
    measured there (twice the fp32-vs-fp64 oracle drift, at least 3e-2, at most 0.1), counted and
    reported."""
    eng, m = big["eng"], big["model"]
    m64 = oracle.OracleModel(big["S"], big["base"], big["ad"], acc="f64acc")
    W = synth.WORKLOADS["qwen3-0.6b-b1-d16-p512-g256"]
    prompt = synth.gen_prompts(W.shape, list(W.prompt_lens))[0]
    out, st = eng.pbd_generate([prompt], W.max_new, mode=0)
    gpu = [int(t) for t in out[0].cpu()]
    assert len(gpu) == W.max_new
    P = len(prompt)
    cap = P + W.max_new + 1
    cache, p0, lg0 = m.prefill(prompt, cap, want_logits=True)
    cache64, _, lg0_64 = m64.prefill(prompt, cap, want_logits=True)
    # logits after prompt + gpu[:i] for i = 1..255: rows gpu[0..254] at positions P..P+254
    _, lg, _ = m.forward(cache, P, gpu[:-1], False, oracle.MASK_CAUSAL, 0, W.max_new - 1, want_logits=True)
    _, lg64, _ = m64.forward(cache64, P, gpu[:-1], False, oracle.MASK_CAUSAL, 0, W.max_new - 1, want_logits=True)
    ref = np.concatenate([lg0[None], lg])
    ref64 = np.concatenate([lg0_64[None], lg64])
    ties = []
    for i, t in enumerate(gpu):
        best = int(np.argmax(ref[i]))
        if t != best:
            gap = float(ref[i][best] - ref[i][t])
            tol = _parity.bound(float(np.abs(ref[i] - ref64[i]).max()))
            assert gap <= tol, (i, t, best, gap, tol)
            ties.append((i, gap))
    _parity.record_tokens(W.name + ":generation", 0, len(gpu), ties)


def test_spec_equals_ar_bitwise_full_workload(big):
    eng = big["eng"]
    W = synth.WORKLOADS["qwen3-0.6b-b1-d16-p512-g256"]
    prompt = synth.gen_prompts(W.shape, list(W.prompt_lens))[0]
    spec, st = eng.pbd_generate([prompt], W.max_new, mode=0)
    ar, st_ar = eng.pbd_generate([prompt], W.max_new, mode=1)
    assert big["torch"].equal(spec, ar)
    assert st.emitted == W.max_new and st_ar.rounds == W.max_new - 1


def test_verify_rows_equal_decode_rows_long_context(big):
    """Batch invariance at a 4096-token context (several attention splits and pages)."""
    eng = big["eng"]
    W = synth.WORKLOADS["qwen3-0.6b-b1-d16-p4096-g512"]
    prompt = synth.gen_prompts(W.shape, list(W.prompt_lens))[0]
    ar, _ = eng.pbd_generate([prompt], 6, mode=1)
    cont = [int(t) for t in ar[0].cpu()]
    eng.pbd_prefill([prompt], max_new=40)
    drafts = cont[1:6] + [0] * (D - 5)
    _, v_lg = eng.pbd_verify_block(drafts=[drafts], want_logits=True)
    v_lg = v_lg[0].cpu().numpy()
    eng.pbd_accept_commit(forced_n=[0])
    eng.pbd_prefill([prompt], max_new=40)
    for j in range(5):
        _, lg = eng.pbd_decode_step(want_logits=True)
        assert np.array_equal(lg[0].cpu().numpy().view(np.uint32), v_lg[j].view(np.uint32)), j


def test_batch8_ragged_matches_solo_and_ar(big):
    """Batch of 8 ragged prompts (256..2048 tokens, paged KV): each sequence's speculative output
    equals its own plain greedy decoding and its solo run, bit for bit."""
    eng = big["eng"]
    W = synth.WORKLOADS["qwen3-0.6b-b8-d16-p256to2048-g256"]
    prompts = synth.gen_prompts(W.shape, list(W.prompt_lens))
    G = 64
    spec, st = eng.pbd_generate(prompts, G, mode=0)
    ar, _ = eng.pbd_generate(prompts, G, mode=1)
    assert big["torch"].equal(spec, ar)
    for b in (0, 7):
        solo, _ = eng.pbd_generate([prompts[b]], G, mode=0)
        assert big["torch"].equal(solo[0], spec[b]), b


def test_forced_acceptance_sweep_lengths(big):
    """Forced-acceptance timing mode (D sweep workload): committed lengths follow the seeded draws."""
    from paper_2607_12422_gb300 import pbd
    S = big["S"]
    W = synth.WORKLOADS["qwen3-0.6b-b1-p1024-dsweep-forced"]
    prompt = synth.gen_prompts(S, list(W.prompt_lens))[0]
    for Dk in (4, 32):
        e = pbd.Engine(S, big["base"], big["ad"], block_D=Dk, max_batch=1, max_seq_len=1024 + 64 + 8)
        forced = synth.forced_accept_lengths(3.0, Dk, 64)
        out, st = e.pbd_generate([prompt], 64, mode=0, forced_n_seq=forced.reshape(-1, 1))
        rounds = int(st.rounds)
        assert st.accepted == int(forced[:rounds].sum())
        # the rounds needed: the first whose cumulative emission (plus the prefill token) reaches 64
        cum = 1 + np.cumsum(forced + 1)
        assert rounds == int(np.argmax(cum >= 64)) + 1
        L, _, n_out = e.pbd_get_state()
        assert int(n_out[0]) == 64
        assert int(L[0]) == len(prompt) + int((forced[:rounds] + 1).sum())
        e.close()
