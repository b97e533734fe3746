#!/usr/bin/env python3
"""Benchmark of the PEFT-BD hot path on one GB300 per rank.

Workload: Qwen3-0.6B shape (28 layers, hidden 1024, 16/8 heads, head 128, SwiGLU 3072,
vocab 151936, tied head), adapter rank 16 on all seven linears, batch 1, block D = 16,
a seeded uniform 512-token prompt and a 256-token generation budget.  Random-init bf16
weights and synthetic prompts stand in for the paper's trained adapter and TULU-3 prompts.

A step is one speculative round: adapter-on draft pass, adapter-off verify pass, device-side
accept/commit (Section 3 of the paper).  Rounds run as CUDA graphs; each step is bracketed by
CUDA events on the library's stream.  When a generation reaches its budget, the next prompt is
prefilled outside the timed region.  The weights streamed per pass (1.2 GB) exceed the 129 MB
L2, so no flush is needed between steps.

Prints one JSON line.  --impl reference times the CPU oracle on the same workload instead.
"""
import argparse
import hashlib
import json
import os
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

WORKLOAD = "qwen3-0.6b-b1-d16-p512-g256"
METRIC = "decoded tokens/s (PEFT-BD draft+verify rounds, Qwen3-0.6B shape, D=16)"
CHUNK = 32  # rounds per timed chunk
# draft variants measured beside the method of Section 3: early exit at half and quarter depth and
# layer skipping (the odd layers 5..23, 10 of 28; Section 6), two-step denoising and the
# unanchored readout (Sections 4.4 and 5.3)
VARIANTS = (("early_exit_14", dict(draft_layers=14)), ("early_exit_7", dict(draft_layers=7)),
            ("skip_odd_5_23", dict(draft_skip=sum(1 << l for l in range(5, 24, 2)))),
            ("denoise_2", dict(denoise_steps=2)), ("unanchored", dict(anchored=False)))


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def bf16_peak():
    """Sustained dense bf16 TFLOP/s (for steps timed inside a long loop) and where it came from."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops_sustained"]), "measured (sustained)"
    except Exception:
        return 1700.0, "fallback (sustained)"


def verify_flops(S, L_sum, B, D):
    """Algorithmic FLOPs of one verify step over B sequences of D + 1 rows: every linear and the
    tied lm_head on every row (2 per multiply-add), and causal attention (QK^T and PV, 4 d per
    visible key and query head), row j of sequence b seeing L_b + j + 1 keys; L_sum = sum of L_b."""
    M = B * (D + 1)
    lin = S.n_layers * sum(i * o for i, o in (S.linear_dims(n) for n in ("q", "k", "v", "o", "gate", "up", "down")))
    keys = (D + 1) * L_sum + B * (D + 1) * (D + 2) // 2
    return 2 * M * (lin + S.vocab * S.hidden) + 4 * S.head_dim * S.n_q_heads * S.n_layers * keys


def pass_bytes(S, L_mean, rows, adapter):
    """Algorithmic bytes of one pass: every weight once, the KV cache read once, the block's KV written."""
    lin = sum(S.linear_dims(n)[0] * S.linear_dims(n)[1] for n in ("q", "k", "v", "o", "gate", "up", "down"))
    w = 2 * (S.n_layers * lin + S.vocab * S.hidden)
    norms = 2 * (2 * S.n_layers * S.hidden + 2 * S.n_layers * S.head_dim + S.hidden)
    lora = 2 * S.n_layers * sum(S.lora_rank * sum(S.linear_dims(n))
                                for n in ("q", "k", "v", "o", "gate", "up", "down")) if adapter else 0
    kv_tok = 2 * 2 * S.n_layers * S.n_kv_heads * S.head_dim
    return w + norms + lora + kv_tok * (L_mean + rows)


class ClockSampler:
    """nvidia-smi clock/throttle samples while the timed region runs."""

    def __init__(self, index):
        self.index = index
        self.lines = []
        self.proc = None

    def __enter__(self):
        q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
             "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
             "clocks_event_reasons.sw_power_cap")
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), "--query-gpu=" + q,
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.t.join(timeout=2)

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx = float(parts[1])
            except ValueError:
                continue
            for n, v in zip(names, parts[3:7]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def source_hash(path):
    """Hash of a CUDA source with its comments and blank space removed: a comment edit leaves the
    compiled kernel, and therefore its measured traffic, unchanged."""
    import re
    txt = open(path).read()
    txt = re.sub(r"//[^\n]*", "", re.sub(r"/\*.*?\*/", "", txt, flags=re.S))
    txt = re.sub(r"\s+", " ", txt).strip()
    return hashlib.sha256(txt.encode()).hexdigest()[:16]


def traffic_for(kernel_src):
    """DRAM bytes per launch from the committed ncu summary, if the kernel source is unchanged since
    (comments aside)."""
    path = os.path.join(ROOT, "profiles", "k_pass_verify_qwen3_0.6b_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
        h = source_hash(kernel_src)
        if rec.get("source_sha256_16") == h:
            return float(rec["dram_bytes_per_launch"])
    except Exception:
        pass
    return None


def run_cpu_oracle(S, base, ad, prompt_len, D, rounds, max_seconds=None):
    """Times oracle speculative rounds after an untimed prefill; returns (tokens/s, sec, rounds, threads)."""
    import oracle
    from paper_2607_12422_gb300 import synth
    m = oracle.OracleModel(S, base, ad)
    prompt = synth.gen_prompts(S, [prompt_len])[0]
    cache, p, _ = m.prefill(prompt, prompt_len + (rounds + 2) * (D + 1))
    L = prompt_len
    toks = 0
    done = 0
    t0 = time.perf_counter()
    for _ in range(rounds):
        d_am, _, _ = m.forward(cache, L, [p] + [-1] * D, True, oracle.MASK_BLOCK_DRAFT, 0, D)
        v_am, _, _ = m.forward(cache, L, [p] + [int(t) for t in d_am], False, oracle.MASK_CAUSAL, 0, D + 1)
        n = oracle.accept_length([int(t) for t in d_am], [int(t) for t in v_am])
        toks += n + 1
        L += n + 1
        p = int(v_am[n])
        done += 1
        if max_seconds and time.perf_counter() - t0 > max_seconds:
            break
    dt = time.perf_counter() - t0
    return toks / dt, dt, done, int(oracle.model.lib().orc_num_threads())


def job_totals(dist, seconds, units, device):
    """(slowest rank's elapsed time, units summed over ranks) of one timed region.  The ranks run
    independent replicas, so the job's rate is the summed units over the slowest rank's time."""
    if dist is None:
        return float(seconds), float(units)
    import torch
    t = torch.tensor([float(seconds), float(units)], dtype=torch.float64, device=device)
    mx = t.clone()
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(mx[0]), float(t[1])


def dist_setup(args):
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def main_reference(args):
    ws, rank, local = dist_setup(args)
    if rank != 0:
        return 0
    from paper_2607_12422_gb300 import synth
    W = synth.WORKLOADS[WORKLOAD]
    S = W.shape
    base, ad = synth.gen_base_weights(S), synth.gen_adapter(S)
    import oracle
    m = oracle.OracleModel(S, base, ad)
    prompt = synth.gen_prompts(S, list(W.prompt_lens))[0]
    P, D = len(prompt), W.block_D
    total = args.warmup + args.steps
    cache, p, _ = m.prefill(prompt, P + (total + 2) * (D + 1))
    L = P
    toks = 0
    t_meas = 0.0
    timed = 0
    budget_s = 150.0  # keeps the reference arm within a few minutes on the host cores
    for i in range(total):
        if i >= args.warmup and t_meas > budget_s:
            break
        t0 = time.perf_counter()
        d_am, _, _ = m.forward(cache, L, [p] + [-1] * D, True, oracle.MASK_BLOCK_DRAFT, 0, D)
        drafts = [int(t) for t in d_am]
        v_am, _, _ = m.forward(cache, L, [p] + drafts, False, oracle.MASK_CAUSAL, 0, D + 1)
        n = oracle.accept_length(drafts, [int(t) for t in v_am])
        dt = time.perf_counter() - t0
        L += n + 1
        p = int(v_am[n])
        if i >= args.warmup:
            t_meas += dt
            toks += n + 1
            timed += 1
    value = toks / t_meas
    threads = int(oracle.model.lib().orc_num_threads())
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * t_meas / timed,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32 (bf16 storage)",
            "data": "synthetic",
            "config": {"workload": WORKLOAD, "batch": 1, "block_D": D, "prompt_len": P, "gen_len": W.max_new},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": threads, "kind": "oracle",
                             "sample": "%d timed speculative rounds (draft+verify+accept; at most %d requested, "
                                       "capped at %.0f s) after an untimed %d-token prefill and %d warm-up rounds"
                                       % (timed, args.steps, budget_s, P, args.warmup)},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def run_rounds(e, prompts, G, D, mode, steps, warmup, forced=None):
    """`warmup` then `steps` timed rounds over generations of `prompts` on engine e.  A chunk never
    holds more rounds than the budget left could absorb at full acceptance (for the sequence
    furthest along), so no timed round runs past a finished generation; the prompts are prefilled
    again (untimed) when the budget is spent.  Returns (per-phase ms sums, tokens emitted in timed
    rounds over all sequences, kernel launches, mean cached length summed over sequences).
    forced: [rounds, batch] accepted lengths, consumed in order across the calls."""
    acc = np.zeros(4)
    f_off = 0

    def chunk_forced(k):
        nonlocal f_off
        if forced is None:
            return None
        idx = (f_off + np.arange(k)) % len(forced)
        f_off += k
        return np.ascontiguousarray(forced[idx])
    tokens = 0
    launches = 0
    l_sum = 0.0
    per_round = (D + 1) if mode == 0 else 1
    e.pbd_prefill(prompts, max_new=G)
    done_w, left = 0, steps
    while done_w < warmup or left > 0:
        L0, _, n0 = e.pbd_get_state()
        room = (G - int(np.max(n0[:len(prompts)]))) // per_round
        if room < 1:
            e.pbd_prefill(prompts, max_new=G)
            continue
        if done_w < warmup:
            k = min(warmup - done_w, room, CHUNK)
            e.pbd_bench_rounds(mode, 0, k, chunk_forced(k))
            done_w += k
            continue
        k = min(left, room, CHUNK)
        r = e.pbd_bench_rounds(mode, 0, k, chunk_forced(k))
        L1, _, n1 = e.pbd_get_state()
        acc += np.array(r[:4])
        tokens += int(np.sum(n1[:len(prompts)])) - int(np.sum(n0[:len(prompts)]))
        launches += r[4] * k
        l_sum += 0.5 * (int(np.sum(L0[:len(prompts)])) + int(np.sum(L1[:len(prompts)]))) * k
        left -= k
    return acc, tokens, launches, l_sum / steps


def measure_configs(pbd, synth, base, ad, dev, hbm, warmup):
    """The other workloads of the 0.6B shape: a 4096-token prompt, a batch of 8 ragged prompts,
    and the block-size sweep with forced acceptance (means 1, 3, 6) beside plain decoding."""
    out = {}
    for name, steps in (("qwen3-0.6b-b1-d16-p4096-g512", 48), ("qwen3-0.6b-b8-d16-p256to2048-g256", 32)):
        W = synth.WORKLOADS[name]
        S, D = W.shape, W.block_D
        prompts = synth.gen_prompts(S, list(W.prompt_lens))
        e = pbd.Engine(S, base, ad, block_D=D, max_batch=len(prompts), max_seq_len=max(W.prompt_lens) + W.max_new + 8,
                       device=dev)
        acc, tok, _, L_sum = run_rounds(e, prompts, W.max_new, D, 0, steps, warmup)
        e.close()
        d_us, v_us = 1e3 * acc[0] / steps, 1e3 * acc[1] / steps
        B = len(prompts)
        # one verify pass of the batch: every weight once, each sequence's KV once, B (D+1) rows written
        fl_v = pass_bytes(S, L_sum, B * (D + 1), False) / (hbm * 1e9) * 1e6
        tf, _ = bf16_peak()
        out[name] = {"batch": B, "draft_us": d_us, "verify_us": v_us, "tokens_per_s": tok / (acc[3] / 1e3),
                     "mean_tokens_per_round_per_seq": tok / steps / B, "kv_tokens_mean": L_sum,
                     "verify_roofline_frac": fl_v / v_us,
                     "verify_tensor_frac": verify_flops(S, L_sum, B, D) / (v_us * 1e-6) / (tf * 1e12), "steps": steps}
    W = synth.WORKLOADS["qwen3-0.6b-b1-p1024-dsweep-forced"]
    S = W.shape
    prompt = synth.gen_prompts(S, list(W.prompt_lens))
    sweep = {}
    for D in W.D_sweep:
        e = pbd.Engine(S, base, ad, block_D=D, max_batch=1, max_seq_len=W.prompt_lens[0] + W.max_new + 2 * D + 8,
                       device=dev)
        acc_ar, tok_ar, _, _ = run_rounds(e, prompt, W.max_new, D, 1, 32, warmup)
        ar_us = 1e3 * acc_ar[3] / 32
        row = {"ar_us_per_token": ar_us}
        for mean in W.forced_means:
            steps = 48
            forced = synth.forced_accept_lengths(mean, D, steps + warmup).reshape(-1, 1)
            acc, tok, _, _ = run_rounds(e, prompt, W.max_new, D, 0, steps, warmup, forced)
            step_us = 1e3 * acc[3] / steps
            row["mean_A_%g" % mean] = {"step_us": step_us, "tokens_per_s": tok / (acc[3] / 1e3),
                                       "tokens_per_round": tok / steps, "speedup_vs_ar": (tok / steps) * ar_us / step_us}
        row["break_even_accept"] = (1e3 * acc[0] / steps + 1e3 * acc[1] / steps) / ar_us
        e.close()
        sweep["D=%d" % D] = row
    out[W.name] = sweep
    return out


def main(args):
    ws, rank, local = dist_setup(args)
    import torch
    dist = None
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = "cuda:%d" % local
    from paper_2607_12422_gb300 import pbd, synth
    Wl = synth.WORKLOADS[WORKLOAD]
    S, D = Wl.shape, Wl.block_D
    base, ad = synth.gen_base_weights(S), synth.gen_adapter(S)
    prompt = synth.gen_prompts(S, list(Wl.prompt_lens))[0]
    P, G = len(prompt), Wl.max_new
    eng = pbd.Engine(S, base, ad, block_D=D, max_batch=1, max_seq_len=P + G + 8, device=dev)

    def timed_rounds(mode, steps, warmup, forced=None, e=None):
        return run_rounds(e or eng, [prompt], G, D, mode, steps, warmup, forced)

    hbm, peak_kind = peaks()
    if args.profile_rounds:
        # profiler configuration: prefill, then warm-up and timed rounds only (no other legs)
        acc, tokens, launches, L_mean = timed_rounds(0, args.steps, args.warmup)
        print(json.dumps({"profile_rounds": args.steps, "ms_per_step": acc[3] / args.steps,
                          "launches_per_round": launches // args.steps}))
        eng.close()
        return 0
    # ---- main measurement: speculative rounds
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        acc, tokens, launches, L_mean = timed_rounds(0, args.steps, args.warmup)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    ms_total = acc[3]
    ms_job, tok_job = job_totals(dist, ms_total, tokens, dev)
    value = tok_job / (ms_job / 1e3)
    ms_per_step = ms_total / args.steps
    draft_us = 1e3 * acc[0] / args.steps
    verify_us = 1e3 * acc[1] / args.steps
    commit_us = 1e3 * acc[2] / args.steps
    mean_A = tokens / args.steps

    # ---- plain greedy decoding on the same kernels (the paper's AR baseline)
    ar_steps = max(64, args.steps // 2)
    acc_ar, tok_ar, _, L_ar = timed_rounds(1, ar_steps, args.warmup)
    ar_us = 1e3 * (acc_ar[1] + acc_ar[2]) / ar_steps
    ar_pass_us = 1e3 * acc_ar[1] / ar_steps

    # ---- pass-level roofline (weights + KV per pass over the measured copy bandwidth)
    b_verify = pass_bytes(S, L_mean, D + 1, False)
    b_draft = pass_bytes(S, L_mean, D + 1, True)
    floor_v = b_verify / (hbm * 1e9) * 1e6
    floor_d = b_draft / (hbm * 1e9) * 1e6

    # ---- dominant kernel: the persistent pass kernel (all 28 layers of a verify pass), timed alone
    eng.pbd_prefill([prompt], max_new=G)
    ms_k, k_bytes = eng.pbd_time_pass(1, 16)
    ms_kd, kd_bytes = eng.pbd_time_pass(0, 16)
    achieved = k_bytes / (ms_k * 1e-3) / 1e9
    traffic = traffic_for(os.path.join(ROOT, "paper_2607_12422_gb300", "csrc", "pass_kernel.cu"))

    # ---- end to end through the public call with host buffers
    # (host prompt ids in, host token ids out; the binding copies the prompt to the device),
    # whole-job over the replicas like the device-timed value
    e2e_vals = []
    for it in range(3):
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        out, st = eng.pbd_generate([prompt], G, mode=0)
        host_tokens = out.cpu().numpy()
        dt = time.perf_counter() - t0
        assert host_tokens.shape == (1, G)
        dt_job, tok_job_e2e = job_totals(dist, dt, G, dev)
        if it > 0:
            e2e_vals.append(tok_job_e2e / dt_job)
    e2e = float(np.median(e2e_vals))

    # ---- draft variants (Sections 4.4, 5.3 and 6): same workload, natural acceptance, one
    # engine each; the draft time covers every denoising pass and its lm_head
    variants = None
    if ws == 1 and not args.no_variants:
        variants = {}
        for name, kw in VARIANTS:
            ev = pbd.Engine(S, base, ad, block_D=D, max_batch=1, max_seq_len=P + G + 8, device=dev, **kw)
            v_steps = 64
            acc_v, tok_v, _, L_v = timed_rounds(0, v_steps, args.warmup, e=ev)
            ev.pbd_prefill([prompt], max_new=G)
            ms_vd, vd_bytes = ev.pbd_time_pass(0, 8)
            d_us, v_us = 1e3 * acc_v[0] / v_steps, 1e3 * acc_v[1] / v_steps
            variants[name] = {"config": kw, "draft_us": d_us, "verify_us": v_us,
                              "mean_tokens_per_round": tok_v / v_steps,
                              "tokens_per_s": tok_v / (acc_v[3] / 1e3), "draft_over_verify": d_us / v_us,
                              "draft_pass_kernel_us": ms_vd * 1e3,
                              "draft_pass_kernel_frac": vd_bytes / (ms_vd * 1e-3) / 1e9 / hbm,
                              "break_even_accept": (d_us + v_us) / ar_us, "steps": v_steps}
            ev.close()
            del ev

    configs = None
    if ws == 1 and not args.no_configs:
        configs = measure_configs(pbd, synth, base, ad, dev, hbm, args.warmup)

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        P0 = Wl.prompt_lens[0]
        tps, sec, done, threads = run_cpu_oracle(S, base, ad, P0, D, 96, max_seconds=15)
        cpu = {"value": tps, "unit": "tokens/s", "cores": threads, "kind": "oracle",
               "sample": "%d speculative rounds (draft+verify+accept) of the same model after an untimed prefill "
                         "of the workload's %d-token prompt, %.1f s (at most 96 rounds or 15 s)" % (done, P0, sec)}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": WORKLOAD, "batch": 1, "block_D": D, "prompt_len": P, "gen_len": G,
                       "acceptance": "natural (random-init adapter)",
                       "l2": "no flush: 1.19 GB of weights per pass exceeds the 129 MB L2",
                       "parallelism": "replicas" if ws > 1 else "single GPU"},
            "passes": {"draft_us": draft_us, "verify_us": verify_us, "commit_us": commit_us,
                       "draft_floor_us": floor_d, "verify_floor_us": floor_v,
                       "draft_roofline_frac": floor_d / draft_us, "verify_roofline_frac": floor_v / verify_us,
                       "draft_bytes": b_draft, "verify_bytes": b_verify, "L_mean": L_mean,
                       "verify_tensor_frac": verify_flops(S, L_mean, 1, D) / (verify_us * 1e-6) / (bf16_peak()[0] * 1e12),
                       "tensor_peak": "%.1f TFLOP/s bf16, %s" % bf16_peak(),
                       "mean_tokens_per_round": mean_A, "draft_over_verify": draft_us / verify_us},
            "ar": {"us_per_step": ar_us, "pass_us": ar_pass_us, "tokens_per_s": tok_ar / (acc_ar[3] / 1e3),
                   "break_even_accept": (draft_us + verify_us) / ar_us},
            "draft_variants": variants,
            "other_workloads": configs,
            "roofline": {"bound": "hbm", "kernel": "k_pass (persistent; 28 layers of one verify pass, 17 rows)",
                         "achieved": achieved, "peak": hbm, "peak_kind": peak_kind + " hbm_gbs (burst)",
                         "unit": "GB/s", "frac": achieved / hbm, "traffic": traffic,
                         "algorithmic_bytes": k_bytes, "us_per_launch": ms_k * 1e3,
                         "draft_kernel": {"us_per_launch": ms_kd * 1e3, "algorithmic_bytes": kd_bytes,
                                          "frac": kd_bytes / (ms_kd * 1e-3) / 1e9 / hbm}},
            "cpu_baseline": cpu,
            "e2e": {"value": e2e, "unit": "tokens/s", "h2d_bytes_per_step": 4 * P, "d2h_bytes_per_step": 4 * G,
                    "step": "one pbd_generate call (prefill + rounds) per generation"},
            "gpu_launches": int(launches),
            "clocks": clk.summary(),
            "paper_context": {"peft_bd_tok_s": 34.045, "greedy_ar_tok_s": 431.356, "hardware": "not stated"},
        }
        print(json.dumps(line))
    eng.close()
    if dist:
        dist.barrier()
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=256)
    ap.add_argument("--warmup", type=int, default=8)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-variants", action="store_true", help="skip the draft-variant measurements")
    ap.add_argument("--no-configs", action="store_true", help="skip the long-context, batch-8 and D-sweep workloads")
    ap.add_argument("--profile-rounds", action="store_true",
                    help="only prefill + warm-up + timed rounds (the configuration profiled under ncu)")
    a = ap.parse_args()
    if a.warmup < 3:
        a.warmup = 3
    sys.exit(main_reference(a) if a.impl == "reference" else main(a))
