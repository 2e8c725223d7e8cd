"""The benchmark's multi-replica path on CPU: two gloo ranks (no GPU).

Replicas share nothing on the data path; the job's step time is the slowest
replica's (a MAX all-reduce) and its throughput counts every replica's rows.
The reference arm runs on rank 0 only.
"""
import importlib.util
import io
import json
import os
import socket
import sys
from contextlib import redirect_stdout
from pathlib import Path

import torch.multiprocessing as mp

ROOT = Path(__file__).resolve().parents[1]


def _bench():
    spec = importlib.util.spec_from_file_location("bench", ROOT / "bench.py")
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out_dir):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    b = _bench()
    t = b.max_over_ranks(1.5 + rank)          # rank 1 is the slow replica
    v = b.whole_job_rate(1408, world, t)
    buf = io.StringIO()
    with redirect_stdout(buf):
        args = type("A", (), dict(workload="tiny", steps=1, warmup=0, cpu_seconds=0.5))()
        b.run_reference(args)
    dist.barrier()
    dist.destroy_process_group()
    (Path(out_dir) / f"r{rank}.json").write_text(json.dumps({"t": t, "v": v, "printed": buf.getvalue()}))


def test_two_replicas_on_gloo(tmp_path):
    sys.path.insert(0, str(ROOT))
    mp.spawn(_rank, args=(2, _free_port(), str(tmp_path)), nprocs=2, join=True)
    r0 = json.loads((tmp_path / "r0.json").read_text())
    r1 = json.loads((tmp_path / "r1.json").read_text())
    assert r0["t"] == r1["t"] == 2.5
    assert r0["v"] == r1["v"] == 2 * 1408 / 2.5e-3
    line = json.loads(r0["printed"].strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["value"] > 0
    assert r1["printed"] == ""


def test_single_process_needs_no_process_group():
    b = _bench()
    assert b.max_over_ranks(3.0) == 3.0
    assert b.whole_job_rate(10, 1, 2.0) == 5000.0
