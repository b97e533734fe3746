"""The seeded input generator: determinism, bf16 encoding, forced-acceptance draws."""
import numpy as np
import torch

from paper_2607_12422_gb300 import synth


def test_bf16_bits_matches_torch_rne():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(100000).astype(np.float32) * 0.02,
                        np.array([0.0, -0.0, 1.0, 1.00390625, 1.01171875, 3.0e38, 1e-40], np.float32)])
    ours = synth.bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


def test_weights_deterministic_and_scaled():
    a = synth.gen_base_weights(synth.TINY)
    b = synth.gen_base_weights(synth.TINY)
    for k in a:
        assert np.array_equal(a[k], b[k])
    w = synth.bf16_to_f32(a["wq"])
    assert abs(w.std() - 0.02) < 1e-3 and abs(w.mean()) < 1e-3
    assert np.all(a["attn_norm"] == 0x3F80)


def test_zero_B_keeps_A_and_mask():
    a = synth.gen_adapter(synth.TINY)
    z = synth.gen_adapter(synth.TINY, zero_B=True)
    for n in synth.LINEARS:
        assert np.array_equal(a["a_" + n], z["a_" + n])
        assert not z["b_" + n].any()
    assert np.array_equal(a["mask_embed"], z["mask_embed"])


def test_forced_accept_lengths():
    for D in (4, 8, 16, 32):
        for mean in (1.0, 3.0, 6.0):
            n = synth.forced_accept_lengths(mean, D, 20000)
            assert n.min() >= 0 and n.max() <= D
            A = n + 1
            target = min(mean, D + 1)
            if mean > D + 1:
                assert np.all(A == D + 1)
            else:
                assert abs(A.mean() - target) < 0.05 * target
    assert np.all(synth.forced_accept_lengths(1.0, 16, 100) == 0)


def test_workloads_shapes():
    w = synth.WORKLOADS["qwen3-0.6b-b8-d16-p256to2048-g256"]
    assert len(w.prompt_lens) == 8 and all(256 <= L <= 2048 for L in w.prompt_lens)
    p = synth.gen_prompts(w.shape, w.prompt_lens)
    assert [len(x) for x in p] == list(w.prompt_lens)
    assert all(x.min() >= 0 and x.max() < w.shape.vocab for x in p)


def test_random_norm_gains():
    a = synth.gen_base_weights(synth.TINY)
    r = synth.with_random_norm_gains(a)
    r2 = synth.with_random_norm_gains(a)
    for k in ("final_norm", "attn_norm", "mlp_norm", "q_norm", "k_norm"):
        g = synth.bf16_to_f32(r[k])
        assert r[k].shape == a[k].shape and np.array_equal(r[k], r2[k])
        assert g.min() >= 0.5 and g.max() <= 1.5 and len(np.unique(g)) > 10
    for k in synth.LINEARS:
        assert r["w" + k] is a["w" + k]
    assert np.all(a["attn_norm"] == 0x3F80)  # the input dict is not modified
