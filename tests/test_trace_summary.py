"""The per-phase timeline summary of a traced pass, on the planner's real item list with
stamps laid out by hand (no GPU): every phase of layer l ends at 100 l + 20 (k + 1) us (k its
position in q|k|v, attention, o, gate|up, down), each item waits 1 us, works 2 us and spends
2 us after its work; the final-norm items end 10 us after the last layer."""
import numpy as np
import pytest

from paper_2607_12422_gb300 import pbd, synth, trace_pass

PHASES = ["qkv", "attn", "o", "gate_up", "down"]


def _timeline(items, n_layers):
    op = items[:, 0] & 0xFF
    lin = (items[:, 0] >> 8) & 0xFF
    layer = items[:, 0] >> 16
    end = np.zeros(len(items))
    for i in range(len(items)):
        if op[i] == 0:
            end[i] = 10.0
        elif op[i] == 3:
            end[i] = 100.0 * n_layers + 10.0
        else:
            k = 1 if op[i] == 2 else (0 if lin[i] == 0 else lin[i] + 1)
            end[i] = 100.0 * layer[i] + 20.0 * (k + 1) + 10.0
    tr = np.zeros((len(items), 8), np.uint64)
    base_ns = 5_000_000_000
    for col, back in ((0, 5.0), (1, 4.0), (2, 2.0), (3, 0.0)):
        tr[:, col] = (base_ns + 1e3 * (end - back)).astype(np.uint64)
    tr[:, 4] = tr[:, 1] + 500  # one sub-stamp: 0.5 us after the inputs were ready
    return tr


@pytest.mark.parametrize("kind", [0, 1])
def test_summary_of_a_known_timeline(kind):
    S = synth.TINY
    cfg = pbd.make_config(S, 16, 1, 160)
    items, _ = pbd.pbd_plan_pass(cfg, kind, [64], 32, 152)
    res = trace_pass.summarize(items, _timeline(items, S.n_layers))
    assert res["items"] == len(items)
    # from the embeddings' start (5 us) to the final-norm items' end
    assert res["pass_us"] == pytest.approx(100.0 * S.n_layers + 10.0 - 5.0)
    for name in PHASES:
        ph = res["phases"][name]
        assert ph["wait_us_med"] == pytest.approx(1.0)
        assert ph["work_us_med"] == pytest.approx(2.0)
        assert ph["post_us_med"] == pytest.approx(2.0)
        assert ph["item_us_max"] == pytest.approx(5.0)
        # each phase from the end of the one before it; q|k|v from the previous layer's down
        # (layer 0: the embedding, which ends at 10 us)
        assert ph["layer_span_us_mean"] == pytest.approx(20.0)
        key = "landed_us_med" if name == "attn" else "staged_us_med"
        assert ph["since_deps"][key] == pytest.approx(0.5)
    assert res["layer_us_mean"] == pytest.approx(100.0)
    assert res["phases"]["embed"]["items"] == 17
    assert res["phases"]["final"]["items"] == (16 if kind == 0 else 17)
