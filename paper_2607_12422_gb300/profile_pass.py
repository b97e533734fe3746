"""Small standalone driver of the persistent pass kernel, for profilers.

Builds a context for a workload (seeded weights), prefills its first prompt, then launches
`--iters` draft / verify / decode passes through pbd_time_pass (one warm-up launch first) and
prints the mean device time per launch.  The prefill itself launches the pass kernel once per
64-token chunk, so a profiler that wants the first timed pass skips ceil(P / 64) + 1 launches.

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
    eng = pbd.Engine(S, synth.gen_base_weights(S), synth.gen_adapter(S), block_D=W.block_D, max_batch=1,
                     max_seq_len=W.prompt_lens[0] + W.max_new + 8)
    eng.pbd_prefill(synth.gen_prompts(S, [W.prompt_lens[0]]), max_new=W.max_new)
    kind = {"draft": 0, "verify": 1, "decode": 2}[a.kind]
    ms, nbytes = eng.pbd_time_pass(kind, a.iters)
    print(json.dumps({"workload": a.workload, "kind": a.kind, "prefill_launches": -(-W.prompt_lens[0] // 64),
                      "ms_per_launch": ms, "bytes_per_launch": nbytes}))


if __name__ == "__main__":
    main()
