"""Pins of the oracle's draft variants (Sections 4.4, 5.3 and 6).

- Early exit after E decoder layers (a cheaper draft path, Section 6): the draft's logits
  equal those of a separately built model holding only the first E layers' weights, and
  E = n_layers is the default draft bit for bit.
- Layer skipping (the other cheaper draft path Section 6 names): the draft with a set of
  layers skipped equals a separately built model holding only the kept layers' weights, fed
  the kept layers' cache; an empty skip set is the default draft bit for bit.
- Unanchored readout (Sections 4.4 and 5.3): the same block pass read one row later, so
  the unanchored proposals d_1..d_{D-1} are the anchored proposals d_2..d_D.
- Two-step denoising (Sections 4.4 and 5.3): step 1 is the one-step draft; the pending
  row sees only the cache and itself, so its proposal cannot change in step 2, while the
  refilled mask rows do change.
- Any variant keeps exact verification: the output equals greedy decoding, and the
  committed KV equals a fresh prefill of the emitted tokens.
"""
import dataclasses

import numpy as np
import pytest

import oracle
from oracle import MASK_CAUSAL

VARIANTS = [
    dict(draft_layers=1),
    dict(draft_skip=1),
    dict(denoise_steps=2),
    dict(anchored=False),
    dict(draft_layers=1, denoise_steps=2, anchored=False),
]


@pytest.fixture(scope="module")
def greedy48(tiny):
    return oracle.greedy_generate(tiny["model"], tiny["prompt"], 48)


@pytest.mark.parametrize("D", [4, 16])
@pytest.mark.parametrize("var", VARIANTS, ids=lambda v: ",".join("%s=%s" % kv for kv in v.items()))
def test_variant_spec_equals_greedy(tiny, greedy48, D, var):
    out, rounds = oracle.spec_generate(tiny["model"], tiny["prompt"], 48, D, **var)
    assert out == greedy48
    steps = var.get("denoise_steps", 1)
    assert all(len(r["draft_steps"]) == steps and r["draft_steps"][-1] == r["draft"] for r in rounds)


def _sliced_model(tiny, E):
    """The same backbone and adapter cut to the first E decoder layers."""
    S = tiny["shape"]
    S2 = dataclasses.replace(S, n_layers=E)
    per_layer = ("attn_norm", "mlp_norm", "q_norm", "k_norm") + tuple("w" + n for n in oracle.LINEAR_NAMES)
    base = {k: (v[:E].copy() if k in per_layer else v) for k, v in tiny["base"].items()}
    ad = {k: (v[:E].copy() if k != "mask_embed" else v) for k, v in tiny["adapter"].items()}
    return oracle.OracleModel(S2, base, ad)


def test_early_exit_equals_truncated_model(tiny):
    m, prompt = tiny["model"], tiny["prompt"]
    P, D, E = len(prompt), 8, 1
    assert tiny["shape"].n_layers > E
    cache, p, _ = m.prefill(prompt, P + 32)
    d_ee, lg_ee, _ = oracle.draft_block(m, cache, P, p, D, draft_layers=E, want_logits=True)
    short = _sliced_model(tiny, E)
    cache2, p2, _ = short.prefill(prompt, P + 32)
    d_sh, lg_sh, _ = oracle.draft_block(short, cache2, P, p2, D, want_logits=True)
    assert np.array_equal(lg_ee.view(np.uint32), lg_sh.view(np.uint32))
    assert d_ee == d_sh
    # and the full model's own draft differs (the exit really skips layers)
    _, lg_full, _ = oracle.draft_block(m, cache, P, p, D, want_logits=True)
    assert not np.array_equal(lg_full, lg_ee)


def _kept_model(tiny, keep):
    """The same backbone and adapter holding only the decoder layers in `keep`, in order."""
    S = tiny["shape"]
    S2 = dataclasses.replace(S, n_layers=len(keep))
    per_layer = ("attn_norm", "mlp_norm", "q_norm", "k_norm") + tuple("w" + n for n in oracle.LINEAR_NAMES)
    base = {k: (np.ascontiguousarray(v[keep]) if k in per_layer else v) for k, v in tiny["base"].items()}
    ad = {k: (np.ascontiguousarray(v[keep]) if k != "mask_embed" else v) for k, v in tiny["adapter"].items()}
    return oracle.OracleModel(S2, base, ad)


def test_layer_skip_equals_model_of_kept_layers(tiny):
    """Skipping layer 0 of the two: the draft equals a one-layer model holding layer 1's weights,
    with layer 1's cache of the prefix; a wrong layer (the skipped one's weights) differs."""
    m, prompt, S = tiny["model"], tiny["prompt"], tiny["shape"]
    P, D = len(prompt), 8
    assert S.n_layers == 2
    cache, p, _ = m.prefill(prompt, P + 32)
    d_sk, lg_sk, _ = oracle.draft_block(m, cache, P, p, D, draft_skip=1, want_logits=True)
    for keep, same in (([1], True), ([0], False)):
        kept = _kept_model(tiny, keep)
        c2 = kept.new_cache(P + 32)
        c2.write(0, 0, cache.read(keep[0], "k", P), cache.read(keep[0], "v", P))
        d2, lg2, _ = oracle.draft_block(kept, c2, P, p, D, want_logits=True)
        assert np.array_equal(lg_sk.view(np.uint32), lg2.view(np.uint32)) == same, keep
        if same:
            assert d_sk == d2
    # an empty skip set is the default draft
    d0, l0, _ = oracle.draft_block(m, cache, P, p, D, want_logits=True)
    d1, l1, _ = oracle.draft_block(m, cache, P, p, D, draft_skip=0, want_logits=True)
    assert d0 == d1 and np.array_equal(l0.view(np.uint32), l1.view(np.uint32))
    # the skipped layer's cache slots are not written by the draft
    before = cache.read(0, "k", P + D + 1).copy()
    oracle.draft_block(m, cache, P, p, D, draft_skip=1)
    assert np.array_equal(cache.read(0, "k", P + D + 1)[P:], before[P:])


def test_early_exit_at_depth_is_default_draft(tiny):
    m, prompt = tiny["model"], tiny["prompt"]
    P, D = len(prompt), 8
    cache, p, _ = m.prefill(prompt, P + 32)
    d0, l0, _ = oracle.draft_block(m, cache, P, p, D, want_logits=True)
    d1, l1, _ = oracle.draft_block(m, cache, P, p, D, draft_layers=tiny["shape"].n_layers, want_logits=True)
    assert d0 == d1 and np.array_equal(l0.view(np.uint32), l1.view(np.uint32))
    with pytest.raises(ValueError):
        m.forward(cache, P, [p], False, MASK_CAUSAL, n_layers=0)


def test_unanchored_reads_one_row_later(tiny):
    m, prompt = tiny["model"], tiny["prompt"]
    P, D = len(prompt), 8
    cache, p, _ = m.prefill(prompt, P + 32)
    da, la, _ = oracle.draft_block(m, cache, P, p, D, want_logits=True)
    du, lu, _ = oracle.draft_block(m, cache, P, p, D, anchored=False, want_logits=True)
    assert du[:D - 1] == da[1:]
    assert np.array_equal(lu[:D - 1].view(np.uint32), la[1:].view(np.uint32))
    assert not np.array_equal(lu[D - 1], la[D - 1])


def test_two_step_keeps_step_one_and_the_anchor(tiny):
    m, prompt = tiny["model"], tiny["prompt"]
    P, D = len(prompt), 8
    cache, p, _ = m.prefill(prompt, P + 32)
    d1, l1, s1 = oracle.draft_block(m, cache, P, p, D, want_logits=True)
    d2, l2, s2 = oracle.draft_block(m, cache, P, p, D, denoise_steps=2, want_logits=True)
    assert s1 == [d1] and s2[0] == d1 and s2[1] == d2
    # the pending row proposes d_1 from the cache and itself only: unchanged by the refill
    assert d2[0] == d1[0]
    assert np.array_equal(l2[0].view(np.uint32), l1[0].view(np.uint32))
    # the mask rows now see proposals instead of the mask embedding
    assert all(not np.array_equal(l2[j], l1[j]) for j in range(1, D))


def test_variant_rounds_commit_prefill_kv(tiny):
    m, prompt, S = tiny["model"], tiny["prompt"], tiny["shape"]
    D = 4
    out, rounds, (cache, L) = oracle.spec_generate(m, prompt, 40, D, return_state=True, draft_layers=1,
                                                   denoise_steps=2, anchored=False, draft_skip=1)
    toks = list(prompt) + out[:-1]
    assert L == len(toks)
    fresh = m.new_cache(L + 8)
    m.forward(fresh, 0, toks, False, MASK_CAUSAL, L - 1, 1)
    for layer in range(S.n_layers):
        for which in ("k", "v"):
            assert np.array_equal(cache.read(layer, which, L), fresh.read(layer, which, L)), (layer, which)
