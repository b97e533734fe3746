"""The multi-GPU path is replicas only: every rank runs its own generation and the benchmark
combines the ranks' timed regions once, as the slowest rank's time and the summed tokens.
These run as two gloo ranks on the CPU."""
import importlib.util
import os
import socket

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_module", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    b = _bench()
    ws, r, local = b.dist_setup(None)
    seconds = [1.5, 2.25][rank]   # rank 1 is the slower replica
    units = [100, 37][rank]
    t, u = b.job_totals(dist, seconds, units, "cpu")
    with open(os.path.join(out_dir, "rank%d.txt" % rank), "w") as f:
        f.write("%d %d %d %r %r\n" % (ws, r, local, t, u))
    dist.barrier()
    dist.destroy_process_group()


def test_job_totals_two_gloo_ranks(tmp_path):
    mp = pytest.importorskip("torch.multiprocessing")
    port = _free_port()
    mp.spawn(_rank_main, args=(2, port, str(tmp_path)), nprocs=2, join=True)
    for rank in range(2):
        ws, r, local, t, u = open(tmp_path / ("rank%d.txt" % rank)).read().split()
        assert (int(ws), int(r), int(local)) == (2, rank, rank)
        assert float(t) == 2.25 and float(u) == 137.0  # every rank sees the job's totals


def test_job_totals_single_process():
    b = _bench()
    assert b.job_totals(None, 3.5, 12, "cpu") == (3.5, 12.0)


def test_reference_arm_other_ranks_do_no_work(monkeypatch):
    """Under torchrun only rank 0 times the oracle; the others exit 0 at once."""
    b = _bench()
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("LOCAL_RANK", "1")
    assert b.main_reference(None) == 0


def test_reference_arm_line(monkeypatch, capsys):
    """The reference arm (the CPU oracle on the same workload) prints one JSON line with the
    keys the driver reads; one timed round after the 512-token prefill keeps this short."""
    import json
    import types
    b = _bench()
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    args = types.SimpleNamespace(gpus=1, steps=1, warmup=0, impl="reference")
    assert b.main_reference(args) == 0
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["metric"] == b.METRIC and line["unit"] == "tokens/s"
    assert line["value"] > 0 and line["higher_is_better"] is True and line["steps"] == 1
    assert line["config"]["workload"] == b.WORKLOAD and line["config"]["prompt_len"] == 512
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["value"] == line["value"]
    assert line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"] == {"value": line["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
