"""Timeline of one pass of the persistent kernel, summarized per phase.

    python -m paper_2607_12422_gb300.trace_pass --workload qwen3-0.6b-b1-d16-p512-g256 --kind verify

Prefills the workload's first prompt, traces one draft / verify / decode pass (pbd_trace_pass),
and prints, per phase kind: item count, median time waiting for inputs, median work time, median
time after the work (split reduction and signalling), and the mean per-layer span from the end
of the previous phase to the end of this one (the critical-path share of the phase).
"""
import argparse
import json

import numpy as np

OPS = {0: "embed", 1: "linear", 2: "attn", 3: "final"}
LINS = {0: "qkv", 1: "o", 2: "gate_up", 3: "down"}


def summarize(items, tr):
    op = items[:, 0] & 0xFF
    lin = (items[:, 0] >> 8) & 0xFF
    layer = items[:, 0] >> 16
    t = tr.astype(np.float64)
    t0 = t[:, 0].min()
    t = (t - t0) / 1e3  # us from the first item start
    names = np.array([OPS[o] if o != 1 else LINS[l] for o, l in zip(op, lin)])
    out = {"pass_us": float(t[:, 3].max()), "items": int(len(items)), "phases": {}}
    order = ["embed", "qkv", "attn", "o", "gate_up", "down", "final"]
    nl = int(layer.max()) + 1
    ends = {}
    for name in order:
        sel = names == name
        if not sel.any():
            continue
        wait = t[sel, 1] - t[sel, 0]
        work = t[sel, 2] - t[sel, 1]
        post = t[sel, 3] - t[sel, 2]
        out["phases"][name] = {"items": int(sel.sum()), "wait_us_med": float(np.median(wait)),
                               "work_us_med": float(np.median(work)), "post_us_med": float(np.median(post)),
                               "item_us_max": float((t[sel, 3] - t[sel, 0]).max())}
        # sub-stamps 4..7 (0 = not reached): linear = operand staged, accumulator ready, partials
        # stored, reduced; attention = K/V landed, pages ready for the compute (the same instant
        # now that V needs no conversion), all splits stored, merged
        sub = {}
        labels = (("staged", "acc_ready", "counted", "reduced") if name not in ("attn",)
                  else ("landed", "converted", "counted", "merged"))
        for j, lab in enumerate(labels):
            ok = sel & (tr[:, 4 + j] > 0)
            if ok.any():
                sub[lab + "_us_med"] = float(np.median(t[ok, 4 + j] - t[ok, 1]))
        # finer sub-steps 8..12 (present when the stamps are 16 wide), as means: the timer ticks
        # in steps of a few hundred ns, so means over many items resolve finer than medians
        labels2 = (("norm_or_act_ready", "first_row_summed", "first_row_computed", "reduce_stored")
                   if name not in ("attn",) else
                   ("block_requested", "scores_done", "softmax_done", "partials_stored", "merge_loaded"))
        if tr.shape[1] >= 16:
            for j, lab in enumerate(labels2):
                ok = sel & (tr[:, 8 + j] > 0)
                if ok.any():
                    sub[lab + "_us_mean"] = float(np.mean(t[ok, 8 + j] - t[ok, 1]))
        if sub:
            out["phases"][name]["since_deps"] = sub
        ends[name] = {int(l): float(t[sel & (layer == l), 3].max()) for l in np.unique(layer[sel])}
    # per-layer span of each phase: end of this phase minus end of the previous phase in the layer
    prev = {"qkv": None, "attn": "qkv", "o": "attn", "gate_up": "o", "down": "gate_up"}
    for name, p in prev.items():
        if name not in ends:
            continue
        spans = []
        for l in range(nl):
            if l not in ends[name]:
                continue
            if p is None:
                base = ends["down"].get(l - 1, ends.get("embed", {}).get(0, 0.0)) if "down" in ends else 0.0
            else:
                base = ends[p].get(l, 0.0)
            spans.append(ends[name][l] - base)
        out["phases"][name]["layer_span_us_mean"] = float(np.mean(spans))
    layer_end = [max(ends[n].get(l, 0.0) for n in ends if n not in ("embed", "final")) for l in range(nl)]
    out["layer_us_mean"] = float(np.mean(np.diff(layer_end))) if nl > 1 else layer_end[0]
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="qwen3-0.6b-b1-d16-p512-g256")
    ap.add_argument("--kind", default="verify", choices=["draft", "verify", "decode"])
    ap.add_argument("--repeat", type=int, default=3)
    ap.add_argument("--dump", default="", help="also save the raw items and stamps to this .npz file")
    a = ap.parse_args()
    from paper_2607_12422_gb300 import pbd, synth
    W = synth.WORKLOADS[a.workload]
    S = W.shape
    eng = pbd.Engine(S, synth.gen_base_weights(S), synth.gen_adapter(S), block_D=W.block_D, max_batch=W.batch,
                     max_seq_len=max(W.prompt_lens) + W.max_new + 8)
    prompts = synth.gen_prompts(S, list(W.prompt_lens))
    eng.pbd_prefill(prompts, max_new=W.max_new)
    kind = {"draft": 0, "verify": 1, "decode": 2}[a.kind]
    res = None
    for _ in range(a.repeat):  # the last (warm) trace is reported
        items, tr = eng.pbd_trace_pass(kind)
        res = summarize(items, tr)
    res["workload"], res["kind"] = a.workload, a.kind
    if a.dump:
        np.savez(a.dump, items=items, stamps=tr)
    print(json.dumps(res, indent=1))


if __name__ == "__main__":
    main()
