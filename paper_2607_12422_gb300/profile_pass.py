"""Small standalone driver of the persistent pass kernel, for profilers.

Builds a context for a workload (seeded weights), prefills its prompts, then launches
`--iters` draft / verify / decode passes through pbd_time_pass (one warm-up launch first) and
prints the mean device time per launch.  The prefill itself launches the pass kernel once per
64-token chunk of each prompt, so a profiler that wants the first timed pass skips the printed
prefill_launches + 1 launches.

    python -m paper_2607_12422_gb300.profile_pass --kind verify --iters 3
"""
import argparse
import json


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="qwen3-0.6b-b1-d16-p512-g256")
    ap.add_argument("--kind", default="verify", choices=["draft", "verify", "decode"])
    ap.add_argument("--iters", type=int, default=3)
    a = ap.parse_args()
    from paper_2607_12422_gb300 import pbd, synth
    W = synth.WORKLOADS[a.workload]
    S = W.shape
    lens = list(W.prompt_lens)
    eng = pbd.Engine(S, synth.gen_base_weights(S), synth.gen_adapter(S), block_D=W.block_D, max_batch=len(lens),
                     max_seq_len=max(lens) + W.max_new + 8)
    eng.pbd_prefill(synth.gen_prompts(S, lens), max_new=W.max_new)
    kind = {"draft": 0, "verify": 1, "decode": 2}[a.kind]
    ms, nbytes = eng.pbd_time_pass(kind, a.iters)
    print(json.dumps({"workload": a.workload, "kind": a.kind, "batch": len(lens),
                      "prefill_launches": sum(-(-P // 64) for P in lens), "ms_per_launch": ms,
                      "bytes_per_launch": nbytes}))


if __name__ == "__main__":
    main()
