"""The benchmark's multi-process path on CPU (gloo, world size 2): the job
time is the slowest rank's time on every rank, the whole-job value counts
every rank's tokens over that time, and the reference arm prints on rank 0
only. The decode path does not shard (each rank is an independent replica),
so this is all the data path needs across processes."""
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, ms, q):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from bench import job_value, max_over_ranks
    t = max_over_ranks(ms[rank], torch.device("cpu"))
    q.put((rank, t, job_value(world, 4, 65, 3, t)))
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_ranks_and_job_value_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ms = [10.0, 12.5]
    procs = [ctx.Process(target=_worker, args=(r, 2, port, ms, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = dict((r, (t, v)) for r, t, v in (q.get(timeout=120) for _ in procs))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in (0, 1):
        assert got[r][0] == 12.5                      # the slowest rank's time
        assert got[r][1] == pytest.approx(2 * 4 * 65 * 3 / 0.0125)


def test_single_process_is_identity():
    sys.path.insert(0, ROOT)
    from bench import job_value, max_over_ranks
    assert max_over_ranks(3.0, "cpu") == 3.0
    assert job_value(1, 2, 10, 5, 1000.0) == 100.0


def test_reference_arm_prints_on_rank_zero_only():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "0"], env=env, capture_output=True,
                       text=True, timeout=120)
    assert r.returncode == 0 and r.stdout.strip() == ""


def test_profiled_traffic_follows_the_committed_capture(monkeypatch, tmp_path):
    """The roofline's traffic comes from the committed ncu summary while the
    attention source still has the sha256 recorded there, scaled by the
    launch's algorithmic bytes; any other source or workload gives None."""
    import hashlib
    sys.path.insert(0, ROOT)
    import bench
    prof = os.path.join(ROOT, "profiles", "decode_step_lumina1024_rho4.md")
    src = os.path.join(ROOT, "paper_2605_20600_gb300", "csrc", "hkv_attention.cu")
    vals = dict(line.strip().partition(": ")[::2] for line in open(prof) if ": " in line)
    same = hashlib.sha256(open(src, "rb").read()).hexdigest() == vals.get("source_sha256")
    t = bench.profiled_traffic("lumina1024", 1e8)
    if same:
        exp = float(vals["attn_traffic_ratio"]) * 1e8 + float(vals["finish_traffic_bytes_per_launch"])
        assert t == pytest.approx(exp)
    else:
        assert t is None
    assert bench.profiled_traffic("llamagen_xl", 1e8) is None
    # a copy of the tree whose attention source differs: no traffic
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "decode_step_lumina1024_rho4.md").write_text(open(prof).read())
    d = tmp_path / "paper_2605_20600_gb300" / "csrc"
    d.mkdir(parents=True)
    (d / "hkv_attention.cu").write_text(open(src).read() + "\n// changed\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.profiled_traffic("lumina1024", 1e8) is None
