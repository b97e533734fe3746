"""Small standalone driver of one tensor-core linear shape, for profilers.

Runs pbd_op_linear (the same kernel as the decoder passes) on seeded bf16 data:
  gate_up: 17 x 1024 -> 6144  (the fused gate|up projection of Qwen3-0.6B at D = 16)
  qkv:     17 x 1024 -> 4096,  o: 17 x 2048 -> 1024,  down: 17 x 3072 -> 1024
Device footprint is a few tens of MB, so a profiler can replay the kernel cheaply.

    python -m paper_2607_12422_gb300.profile_linear --which gate_up --rows 17 --iters 5
"""
import argparse

import numpy as np

SHAPES = {"gate_up": (1024, 6144), "qkv": (1024, 4096), "o": (2048, 1024), "down": (3072, 1024)}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--which", default="gate_up", choices=sorted(SHAPES))
    ap.add_argument("--rows", type=int, default=17)
    ap.add_argument("--iters", type=int, default=5)
    ap.add_argument("--lora", action="store_true")
    a = ap.parse_args()
    import torch

    from paper_2607_12422_gb300 import pbd, synth
    K, N = SHAPES[a.which]
    rng = np.random.default_rng(0)

    def dev(shape, std):
        bits = synth.bf16_bits((rng.standard_normal(shape) * std).astype(np.float32))
        return torch.from_numpy(bits.view(np.int16)).cuda().view(torch.bfloat16)

    x, W = dev((a.rows, K), 1.0), dev((N, K), 0.02)
    A, B = (dev((16, K), 0.02), dev((N, 16), 0.02)) if a.lora else (None, None)
    for _ in range(a.iters):
        y = pbd.pbd_op_linear(x, W, A, B, 2.0)
    torch.cuda.synchronize()
    print("ok", a.which, tuple(y.shape), float(y.float().abs().mean()))


if __name__ == "__main__":
    main()
