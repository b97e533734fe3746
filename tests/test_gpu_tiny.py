"""Pass-level parity of the GPU path against the CPU oracle on the tiny Qwen3-style model
(2 layers, hidden 256, vocab 4096, rank 8, D = 16): draft and verify logits within 3e-2,
token ids, accepted lengths and cached lengths exact, KV commit, batching, forced acceptance,
and the exactness properties on the GPU itself (speculative == greedy, verify rows == decode
rows bit for bit)."""
import numpy as np
import pytest

import _parity
import oracle
from paper_2607_12422_gb300 import synth

pytestmark = pytest.mark.gpu
TOL = 3e-2
D = 16


@pytest.fixture(scope="module")
def env():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_12422_gb300 import pbd
    S = synth.TINY
    base, ad = synth.gen_base_weights(S), synth.gen_adapter(S)
    prompts = synth.gen_prompts(S, [64, 40, 17, 100])
    eng = pbd.Engine(S, base, ad, block_D=D, max_batch=4, max_seq_len=256)
    return dict(torch=torch, pbd=pbd, S=S, base=base, ad=ad, prompts=prompts, eng=eng,
                model=oracle.OracleModel(S, base, ad))


def _check_ids(ids, ref_logits, tol=TOL):
    """GPU argmax equals the oracle's, except where the oracle's top two are within tol (reported)."""
    ids = np.asarray(ids).reshape(-1)
    ref_logits = ref_logits.reshape(len(ids), -1)
    for j, t in enumerate(ids):
        best = int(np.argmax(ref_logits[j]))
        if t != best:
            assert ref_logits[j][best] - ref_logits[j][t] <= tol, (j, t, best)


def test_lockstep_rounds_random_norm_gains(env):
    """Six lockstep rounds with every RMSNorm gain drawn from [0.5, 1.5) (the default synthetic
    gains are all 1, which would hide a gain applied to the wrong column or not at all): logits
    within 3e-2, every verify id equal to the oracle's argmax."""
    S, pbd = env["S"], env["pbd"]
    base = synth.with_random_norm_gains(env["base"])
    assert not np.all(base["attn_norm"] == env["base"]["attn_norm"])
    m = oracle.OracleModel(S, base, env["ad"])
    eng = pbd.Engine(S, base, env["ad"], block_D=D, max_batch=1, max_seq_len=256)
    prompt = env["prompts"][0]
    seqs = {0: _parity.Seq(m, None, prompt, D, 6)}
    _parity.start(eng, [prompt], seqs, 64, "tiny-b1-d16-p64-g64-random-gains")
    n0 = len(_parity.RECORDS)
    _parity.rounds(eng, seqs, 6, "tiny-b1-d16-p64-g64-random-gains")
    eng.close()
    new = _parity.RECORDS[n0:]
    assert all(r["bound"] == TOL for r in new)
    assert sum(r["id_mismatches"] for r in new if r["pass_kind"] == "verify") == 0


def test_few_ctas_last_item_merges_lockstep(env):
    """The pass kernel on 4 CTAs (many items per CTA) with a 1000-token prompt: each (sequence, KV
    head) then has more attention items than CTAs, so the last item to finish merges all of them
    (the path long batched contexts take on the full GPU).  Three lockstep rounds at 3e-2."""
    S, pbd = env["S"], env["pbd"]
    P, G = 1000, 48
    cfg = pbd.make_config(S, D, 1, P + G + 8, max_ctas=4)
    items, _ = pbd.pbd_plan_pass(cfg, 1, [P], G, 4)
    op, c, b = items[:, 0] & 0xFF, items[:, 3], items[:, 2]
    layer0 = (items[:, 0] >> 16) == 0
    assert min(int(c[(op == 2) & layer0 & (b == g)].max()) + 1 for g in range(S.n_kv_heads)) > 4
    prompt = synth.gen_prompts(S, [P], seed=11)[0]
    eng = pbd.Engine(S, env["base"], env["ad"], block_D=D, max_batch=1, max_seq_len=P + G + 8, max_ctas=4)
    seqs = {0: _parity.Seq(env["model"], None, prompt, D, 3)}
    _parity.start(eng, [prompt], seqs, G, "tiny-b1-d16-p1000-4ctas")
    n0 = len(_parity.RECORDS)
    _parity.rounds(eng, seqs, 3, "tiny-b1-d16-p1000-4ctas")
    eng.close()
    assert all(r["bound"] == TOL for r in _parity.RECORDS[n0:])


def test_round_matches_oracle(env):
    eng, m, prompt = env["eng"], env["model"], env["prompts"][0]
    P = len(prompt)
    first = eng.pbd_prefill([prompt], max_new=64)
    cache, p0, lg0 = m.prefill(prompt, P + 96, want_logits=True)
    assert int(first[0]) == p0
    d_ids, d_lg = eng.pbd_draft_block(want_logits=True)
    _, od, _ = m.forward(cache, P, [p0] + [-1] * D, True, oracle.MASK_BLOCK_DRAFT, 0, D, want_logits=True)
    d_lg = d_lg[0].cpu().numpy()
    assert np.abs(d_lg - od).max() <= TOL
    _check_ids(d_ids[0].cpu().numpy(), od)
    drafts = [int(t) for t in d_ids[0].cpu()]
    v_ids, v_lg = eng.pbd_verify_block(want_logits=True)
    _, ov, _ = m.forward(cache, P, [p0] + drafts, False, oracle.MASK_CAUSAL, 0, D + 1, want_logits=True)
    assert np.abs(v_lg[0].cpu().numpy() - ov).max() <= TOL
    _check_ids(v_ids[0].cpu().numpy(), ov)
    verify = [int(t) for t in v_ids[0].cpu()]
    n = eng.pbd_accept_commit()
    assert int(n[0]) == oracle.accept_length(drafts, verify)
    L, pend, n_out = eng.pbd_get_state()
    assert int(L[0]) == P + int(n[0]) + 1
    assert int(pend[0]) == verify[int(n[0])]
    assert int(n_out[0]) == 1 + int(n[0]) + 1


def test_lockstep_rounds_strict(env):
    """Eight rounds in lockstep at the stated tolerance of 3e-2 with no widening: every verify id
    and every generated token equals the oracle's argmax exactly (no near-tie allowed on the tiny
    model); draft ids may differ only inside 3e-2 (recorded)."""
    eng, m, prompt = env["eng"], env["model"], env["prompts"][0]
    seqs = {0: _parity.Seq(m, None, prompt, D, 8)}
    _parity.start(eng, [prompt], seqs, 64, "tiny-b1-d16-p64-g64")
    n0 = len(_parity.RECORDS)
    _parity.rounds(eng, seqs, 8, "tiny-b1-d16-p64-g64")
    new = _parity.RECORDS[n0:]
    assert all(r["bound"] == TOL for r in new)
    assert sum(r["id_mismatches"] for r in new if r["pass_kind"] == "verify") == 0


def test_generate_equals_oracle_greedy(env):
    eng, m, prompt = env["eng"], env["model"], env["prompts"][0]
    ref = oracle.greedy_generate(m, prompt, 64)
    out, st = eng.pbd_generate([prompt], 64, mode=0)
    assert [int(t) for t in out[0].cpu()] == ref
    assert st.emitted == 64
    ar, _ = eng.pbd_generate([prompt], 64, mode=1)
    assert [int(t) for t in ar[0].cpu()] == ref


def test_verify_rows_equal_decode_rows_bitwise(env):
    """Batch invariance: the verify pass's row j equals plain decoding at that position, bit for bit."""
    eng, prompt = env["eng"], env["prompts"][0]
    ar, _ = eng.pbd_generate([prompt], D + 2, mode=1)
    cont = [int(t) for t in ar[0].cpu()]
    eng.pbd_prefill([prompt], max_new=D + 2)
    v_ids, v_lg = eng.pbd_verify_block(drafts=[cont[1:D + 1]], want_logits=True)
    v_lg = v_lg[0].cpu().numpy()
    eng.pbd_accept_commit(forced_n=[0])  # leave the verify state
    eng.pbd_prefill([prompt], max_new=D + 2)
    for j in range(D + 1):
        t, lg = eng.pbd_decode_step(want_logits=True)
        assert np.array_equal(lg[0].cpu().numpy().view(np.uint32), v_lg[j].view(np.uint32)), j
        assert int(t[0]) == cont[j + 1]


def test_kv_commit_matches_fresh_prefill(env):
    """After rounds with forced acceptance, cached K/V [0, L) equal a fresh prefill of the same tokens."""
    eng, m, S, prompt = env["eng"], env["model"], env["S"], env["prompts"][1]
    P = len(prompt)
    forced = [3, 0, 16, 5, 1, 7]
    eng.pbd_prefill([prompt], max_new=120)
    for n in forced:
        eng.pbd_draft_block()
        eng.pbd_verify_block()
        eng.pbd_accept_commit(forced_n=[n])
    L, pend, n_out = eng.pbd_get_state()
    assert int(L[0]) == P + sum(n + 1 for n in forced)
    toks = eng.pbd_get_tokens()[0].cpu().numpy()[: int(n_out[0])]
    seq = np.concatenate([prompt, toks[:-1]]).astype(np.int32)
    assert len(seq) == int(L[0])
    kv_spec = [eng.pbd_read_kv(l, 0, int(L[0])) for l in range(S.n_layers)]
    eng.pbd_prefill([seq], max_new=2)
    for l in range(S.n_layers):
        k2, v2 = eng.pbd_read_kv(l, 0, int(L[0]))
        assert env["torch"].equal(kv_spec[l][0], k2) and env["torch"].equal(kv_spec[l][1], v2), l
    # and against the oracle's cache after the same forced rounds (bf16 values, small drift)
    out_o, rounds, (cache, Lo) = oracle.spec_generate(m, prompt, 120, D, forced_n=forced + [0] * 200,
                                                      max_rounds=len(forced), return_state=True)
    assert Lo == int(L[0])
    # committed slots agree with the oracle's cache (all of them when both committed the same tokens)
    n_cmp = Lo if list(out_o[: len(toks)]) == [int(t) for t in toks] else P
    for l in range(S.n_layers):
        for which, idx in (("k", 0), ("v", 1)):
            ko = cache.read(l, which, n_cmp)
            kg = kv_spec[l][idx][:n_cmp].float().cpu().numpy()
            assert np.abs(kg - ko).max() <= 0.05 * (1 + np.abs(ko).max()), (l, which)


def test_forced_acceptance_lockstep_with_oracle(env):
    """Forced lengths commit drafted tokens, and the masked rows' logits are nearly flat, so the
    GPU's own drafts may legitimately differ from the oracle's at near-ties.  The GPU therefore
    verifies the oracle's drafts; its own drafts are checked against the oracle's draft logits
    (argmax up to ties within the tolerance); verify tokens, lengths and outputs must be exact."""
    eng, m, prompt = env["eng"], env["model"], env["prompts"][2]
    forced = [int(x) for x in synth.forced_accept_lengths(3.0, D, 64)]
    ref, rounds = oracle.spec_generate(m, prompt, 48, D, forced_n=forced, want_logits=True)
    eng.pbd_prefill([prompt], max_new=48)
    for r in rounds:
        d_ids, d_lg = eng.pbd_draft_block(want_logits=True)
        assert np.abs(d_lg[0].cpu().numpy() - r["draft_logits"]).max() <= TOL
        _check_ids(d_ids[0].cpu().numpy(), r["draft_logits"])
        v_ids, v_lg = eng.pbd_verify_block(drafts=[r["draft"]], want_logits=True)
        assert np.abs(v_lg[0].cpu().numpy() - r["verify_logits"]).max() <= TOL
        assert [int(t) for t in v_ids[0].cpu()] == r["verify"]
        n = eng.pbd_accept_commit(forced_n=[r["n"]])
        assert int(n[0]) == r["n"]
        L, _, _ = eng.pbd_get_state()
        assert int(L[0]) == r["L"] + r["n"] + 1
    assert [int(t) for t in eng.pbd_get_tokens()[0].cpu()] == ref


def test_forced_generate_graph_equals_eager_rounds(env):
    """pbd_generate (one CUDA graph per round) reproduces the eager calls bit for bit."""
    eng, prompt = env["eng"], env["prompts"][2]
    forced = synth.forced_accept_lengths(3.0, D, 64)
    out, st = eng.pbd_generate([prompt], 48, mode=0, forced_n_seq=forced.reshape(-1, 1))
    eng.pbd_prefill([prompt], max_new=48)
    rounds = 0
    while True:
        _, _, n_out = eng.pbd_get_state()
        if int(n_out[0]) >= 48:
            break
        eng.pbd_draft_block()
        eng.pbd_verify_block()
        eng.pbd_accept_commit(forced_n=[int(forced[rounds])])
        rounds += 1
    assert env["torch"].equal(eng.pbd_get_tokens()[0], out[0])
    assert st.rounds == rounds and st.accepted == int(sum(forced[:rounds]))


def test_batch_of_ragged_prompts(env):
    eng, m, prompts = env["eng"], env["model"], env["prompts"][1:4]
    out, st = eng.pbd_generate(list(prompts), 32, mode=0)
    for b, p in enumerate(prompts):
        ref = oracle.greedy_generate(m, p, 32)
        assert [int(t) for t in out[b].cpu()] == ref, b
    # batch composition does not change a sequence's tokens
    solo, _ = eng.pbd_generate([prompts[1]], 32, mode=0)
    assert env["torch"].equal(solo[0], out[1])


def test_zero_B_block_of_one_is_greedy(env):
    from paper_2607_12422_gb300 import pbd
    S = env["S"]
    adz = synth.gen_adapter(S, zero_B=True)
    e1 = pbd.Engine(S, env["base"], adz, block_D=1, max_batch=1, max_seq_len=200)
    prompt = env["prompts"][0]
    out, st = e1.pbd_generate([prompt], 40, mode=0)
    assert [int(t) for t in out[0].cpu()] == oracle.greedy_generate(env["model"], prompt, 40)
    # one accepted draft in every full round
    assert st.accepted == st.rounds or st.accepted == st.rounds - 1
    e1.close()


def test_state_machine_errors(env):
    from paper_2607_12422_gb300 import pbd
    eng = env["eng"]
    eng.pbd_prefill([env["prompts"][0]], max_new=8)
    with pytest.raises(pbd.PbdError) as ei:
        eng.pbd_accept_commit()
    assert ei.value.status == 4
    with pytest.raises(pbd.PbdError) as ei:
        eng.pbd_prefill([np.zeros(300, np.int32)], max_new=8)
    assert ei.value.status == 3


def test_pass_timing_and_trace_entry_points(env):
    """pbd_time_pass and pbd_trace_pass run a pass on a prefilled context without advancing it:
    positive times and byte counts, every scheduled item traced once with ordered stamps, and
    the generation state unchanged afterwards."""
    eng, prompt, pbd = env["eng"], env["prompts"][1], env["pbd"]
    eng.pbd_prefill([prompt], max_new=32)
    before = [np.asarray(x).copy() for x in eng.pbd_get_state()]
    for kind in (0, 1, 2):
        ms, nbytes = eng.pbd_time_pass(kind, 2)
        assert ms > 0 and nbytes > 0
        items, st = eng.pbd_trace_pass(kind)
        assert len(items) == len(st) > 0
        assert st.shape[1] == pbd.TRACE_STAMPS == 16
        ops = items[:, 0] & 0xFF
        assert set(np.unique(ops)) <= {0, 1, 2, 3}
        # start <= inputs ready <= end for every item (all stamps from one global clock)
        assert (st[:, 0] > 0).all() and (st[:, 1] >= st[:, 0]).all() and (st[:, 3] >= st[:, 1]).all()
    after = [np.asarray(x) for x in eng.pbd_get_state()]
    for a, b in zip(before, after):
        assert np.array_equal(a, b)
    # the context is still in the state a round starts from
    d1, _ = eng.pbd_draft_block()
    assert d1.shape == (1, D)


def test_stalled_pass_is_reported_and_context_survives(env):
    """Failure detection without a GPU fault: a verify pass whose schedule lacks one q|k|v item
    never receives that item's partial sums; the bounded waits run out (about a second), the
    device code is latched and reported as PBD_ERR_DEVICE, the decoding state is untouched and
    the context keeps decoding exactly."""
    eng, m, prompt = env["eng"], env["model"], env["prompts"][0]
    P = len(prompt)
    eng.pbd_prefill([prompt], max_new=32)
    status, code = eng.pbd_check_stalled_pass()
    assert status == 6  # PBD_ERR_DEVICE
    assert code in (1, 2, 3, 6)  # a DEV_TIMEOUT_* code
    L, pend, n_out = eng.pbd_get_state()
    assert int(L[0]) == P and int(n_out[0]) == 1
    out, st = eng.pbd_generate([prompt], 32, mode=0)
    assert [int(t) for t in out[0].cpu()] == oracle.greedy_generate(m, prompt, 32)


def test_out_of_range_token_ids_are_latched_and_context_survives(env):
    """The device bounds latch on token ids (the one input the host cannot check: it is device
    memory): a prompt holding id V, or a negative id, is embedded from row 0 instead of read out
    of bounds, the prefill reports PBD_ERR_DEVICE with DEV_BAD_TOKEN (4), and so does a verify
    pass given a drafted id of V.  The same context then decodes a valid prompt exactly."""
    eng, m, prompt, pbd = env["eng"], env["model"], env["prompts"][0], env["pbd"]
    V = env["S"].vocab
    for bad in (V, -5, -1):  # -1 is a mask row, valid only in a draft pass
        p = np.array(prompt, np.int32).copy()
        p[3] = bad
        with pytest.raises(pbd.PbdError) as ei:
            eng.pbd_prefill([p], max_new=16)
        assert ei.value.status == 6 and "device status 4" in str(ei.value), bad
    eng.pbd_prefill([prompt], max_new=16)
    d_ids, _ = eng.pbd_draft_block()
    drafts = d_ids.clone()
    drafts[0, 2] = V
    eng.pbd_verify_block(drafts=drafts)
    with pytest.raises(pbd.PbdError) as ei:
        eng.pbd_sync()
    assert ei.value.status == 6 and "device status 4" in str(ei.value)
    out, st = eng.pbd_generate([prompt], 32, mode=0)
    assert [int(t) for t in out[0].cpu()] == oracle.greedy_generate(m, prompt, 32)


@pytest.mark.parametrize("P,G", [(1, 1), (1, 5), (1, 17), (1, 40), (64, 3), (236, 20)],
                         ids=["p1-g1", "p1-g5", "p1-g17", "p1-g40", "p64-g3", "p236-g20-full"])
def test_edge_lengths(env, P, G):
    """One-token prompts, budgets below one block (no full round), exactly one block, and a
    prompt plus budget that fills max_seq_len (256): the speculative output is the GPU's own
    greedy output bit for bit, and that is the oracle's greedy output up to reported near-ties."""
    eng, m, torch = env["eng"], env["model"], env["torch"]
    prompt = synth.gen_prompts(env["S"], [P], seed=11)[0]
    spec, st = eng.pbd_generate([prompt], G, mode=0)
    ar, _ = eng.pbd_generate([prompt], G, mode=1)
    assert spec.shape[1] >= G and torch.equal(spec[0, :G], ar[0, :G])
    assert st.emitted == G
    ref = oracle.greedy_generate(m, prompt, G)
    got = [int(t) for t in ar[0, :G].cpu()]
    if got != ref:  # the first disagreement must be a near-tie of the oracle's own logits
        j = next(i for i in range(G) if got[i] != ref[i])
        cache, _, lg0 = m.prefill(prompt, P + G + 1, want_logits=True)
        if j == 0:
            lg = lg0[None]
        else:  # the logits after ref[:j]: read-out row j - 1 of a pass over those tokens
            _, lg, _ = m.forward(cache, P, ref[:j], False, oracle.MASK_CAUSAL, j - 1, 1, want_logits=True)
        _check_ids([got[j]], lg, TOL)
