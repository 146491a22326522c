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
    """The roofline's traffic comes from a committed ncu summary of the same
    workload and decode-step design while the kernel sources still hash to
    the digest recorded there, scaled by the launch's algorithmic bytes; any
    other source, design or workload gives None."""
    import glob
    sys.path.insert(0, ROOT)
    import bench
    for launches in (1, 2):
        digest = bench.sources_digest(launches)
        caps = []
        for path in glob.glob(os.path.join(ROOT, "profiles", "*.md")):
            vals = dict(line.strip().partition(": ")[::2] for line in open(path) if ": " in line)
            if vals.get("capture_of") == "lumina1024" and vals.get("launches") == str(launches):
                caps.append(vals)
        t = bench.profiled_traffic("lumina1024", 1e8, launches)
        match = [v for v in caps if v.get("sources_sha256") == digest]
        if match:
            v = match[0]
            assert t == pytest.approx(float(v["traffic_ratio"]) * 1e8
                                      + float(v.get("extra_bytes_per_launch", "0")))
        else:
            assert t is None
        assert bench.profiled_traffic("no_such_workload", 1e8, launches) is None
    # a copy of the tree with a capture that matches, then a changed source
    (tmp_path / "profiles").mkdir()
    d = tmp_path / "paper_2605_20600_gb300" / "csrc"
    d.mkdir(parents=True)
    for f in bench.STEP_SOURCES[1]:
        (d / f).write_text(open(os.path.join(ROOT, "paper_2605_20600_gb300", "csrc", f)).read())
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    (tmp_path / "profiles" / "cap.md").write_text(
        f"capture_of: lumina1024\nlaunches: 1\nsources_sha256: {bench.sources_digest(1)}\n"
        "traffic_ratio: 1.01\nextra_bytes_per_launch: 5\n")
    assert bench.profiled_traffic("lumina1024", 1e8, 1) == pytest.approx(1.01e8 + 5)
    assert bench.profiled_traffic("lumina1024", 1e8, 2) is None
    (d / "hkv_step.cu").write_text(open(os.path.join(ROOT, "paper_2605_20600_gb300", "csrc",
                                                     "hkv_step.cu")).read() + "\n// changed\n")
    assert bench.profiled_traffic("lumina1024", 1e8, 1) is None
