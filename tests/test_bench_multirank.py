"""The benchmark's multi-rank host logic (replicas: each rank its own
sessions, max-over-ranks timing) run as two gloo ranks on the CPU."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), WORLD_SIZE=str(world),
                      RANK=str(rank), LOCAL_RANK=str(rank))
    import bench
    from paper_2607_13093_gb300 import workloads as wl
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w_, r_, l_ = bench.rank_env()
        assert (w_, r_, l_) == (world, rank, rank)
        # a timed region of a different length on every rank: all ranks
        # report the slowest
        ms = bench.max_over_ranks(10.0 + 5.0 * rank)
        # replicated head, own sessions
        w = wl.workload("tiny", device="cpu")
        g = torch.Generator().manual_seed(bench.rank_seed(rank))
        h = wl.make_hidden(w.rows, w.d, g, "cpu")
        W = w.W_h.float()
        hs = [torch.empty_like(h) for _ in range(world)]
        Ws = [torch.empty_like(W[:64]) for _ in range(world)]
        dist.all_gather(hs, h)
        dist.all_gather(Ws, W[:64].contiguous())
        out[rank] = (ms, bool(torch.equal(Ws[0], Ws[1])), bool(torch.equal(hs[0], hs[1])))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_replicas_and_max_timing():
    world, port = 2, _free_port()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_rank_main, args=(world, port, out), nprocs=world, join=True,
                       start_method="spawn")
    assert sorted(out.keys()) == [0, 1]
    for rank in range(world):
        ms, same_w, same_h = out[rank]
        assert ms == 15.0                  # the slower rank's time everywhere
        assert same_w                      # every rank holds the same head
        assert not same_h                  # but its own sessions


def test_job_throughput_counts_every_rank():
    import bench
    assert bench.job_rows_per_s(32, 4, 100, 1000.0) == 32 * 4 * 100 / 1.0
    assert bench.max_over_ranks(3.5) == 3.5          # no process group: identity


def test_reference_arm_under_torchrun_prints_once_from_rank_zero():
    # two ranks launched as the driver launches them; rank 0 alone times the
    # oracle and prints the one JSON line, rank 1 exits 0 without work
    import json
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
           "bench.py", "--impl", "reference", "--gpus", "2", "--steps", "2", "--warmup", "1",
           "--workload", "tiny", "--ref-seconds", "2"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    p = subprocess.run(cmd, cwd=root, env=env, capture_output=True, text=True, timeout=600)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [l for l in p.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    out = json.loads(lines[0])
    assert out["impl"] == "reference" and out["n_gpus"] == 2
    assert out["value"] > 0 and out["e2e"]["value"] == out["value"]
    assert out["cpu_baseline"]["kind"] == "oracle"
    for key in ("metric", "unit", "steps", "warmup", "ms_per_step", "higher_is_better",
                "config", "dtype"):
        assert key in out


def test_traffic_record_follows_its_own_sources(tmp_path, monkeypatch):
    # a committed DRAM-traffic record counts while the kernel sources it
    # lists hash as they did when it was taken, and is dropped once one of
    # them changes (a file the call does not launch does not matter)
    import json
    import bench
    src = tmp_path / "k.cu"
    other = tmp_path / "other.cu"
    src.write_text("kernel v1\n")
    other.write_text("unrelated v1\n")
    (tmp_path / "profiles").mkdir()
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    rec = {"call": {"bytes_per_launch": 1234, "source_files": ["k.cu"],
                    "source_hash": bench.source_hash(["k.cu"])}}
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(rec))
    assert bench.traffic_for("call", files=["k.cu", "other.cu"]) == 1234
    other.write_text("unrelated v2\n")
    assert bench.traffic_for("call", files=["k.cu", "other.cu"]) == 1234
    src.write_text("kernel v2\n")
    assert bench.traffic_for("call") is None
    assert bench.traffic_for("absent") is None


def test_every_traffic_record_is_one_the_bench_looks_up():
    # a record in profiles/traffic.json counts only under the key that the
    # default line (the sweep at 1024 rows over the full vocabulary) or a
    # two-call entry of its configuration block builds for its own call
    import json
    import os
    import bench
    from paper_2607_13093_gb300 import workloads as wl

    def key(name, rows, keep, act):
        cfg = wl.WORKLOADS[name]
        n = cfg["n_keep"] if keep is None else round(keep * cfg["V"])
        return bench.traffic_key(name, rows or cfg["rows"], n, act)

    built = {key("sweep", 1024, 1.0, "fp32")}
    built |= {key(name, rows, keep, act)
              for name, rows, keep, d_l, act, mode, chunk in bench.CONFIG_BLOCK
              if mode == "split" and d_l is None}
    with open(os.path.join(bench.ROOT, "profiles", "traffic.json")) as f:
        records = json.load(f)
    assert records and set(records) <= built, set(records) - built
    assert "cloud_decode_32_12000_fp32" in records
    assert "cloud_sweep_1024_256000_fp32" in records


def test_block_grids_extend_the_configuration_block():
    import bench
    assert len(bench.DEND_GRID) == 10 and len(bench.SWEEP_GRID) == 10
    assert {k for _, k in bench.SWEEP_GRID} == {0.1, 0.5}
    assert {r for r, _ in bench.SWEEP_GRID} == {1, 8, 64, 256, 1024}
