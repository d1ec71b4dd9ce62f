"""bench.py's multi-rank host logic on CPU: two gloo ranks (no GPU needed).

Under torchrun every rank times its own replica of the step; the job's time
is the slowest rank's and its throughput counts every rank's units.  The
reference arm runs on rank 0 only.
"""

import json
import os
import socket
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
torch = pytest.importorskip("torch")


def _bench():
    import importlib.util
    spec = importlib.util.spec_from_file_location("bench", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, ws, port, out_dir):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws))
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    b = _bench()
    local_ms = 100.0 + 50.0 * rank          # rank 1 is the slow one
    total = b.max_over_ranks(local_ms, ws)
    dist.barrier()
    value = b.job_throughput(1000.0, ws, 4, total)
    with open(os.path.join(out_dir, f"r{rank}.json"), "w") as f:
        json.dump({"total": total, "value": value}, f)
    dist.destroy_process_group()


def test_max_over_ranks_and_job_throughput_gloo(tmp_path):
    ws, port = 2, _free_port()
    torch.multiprocessing.spawn(_rank_main, args=(ws, port, str(tmp_path)), nprocs=ws, join=True)
    res = [json.load(open(tmp_path / f"r{r}.json")) for r in range(ws)]
    for r in res:
        assert r["total"] == 150.0                       # the slowest rank's time
        assert r["value"] == pytest.approx(1000.0 * 2 * 4 / 0.150)  # every rank's units


def test_single_rank_needs_no_process_group():
    b = _bench()
    assert b.max_over_ranks(12.5, 1) == 12.5
    assert b.job_throughput(10, 1, 3, 1000.0) == pytest.approx(30.0)


def _run_bench(rank, ws, extra):
    env = dict(os.environ, RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE=str(ws))
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py")] + extra, env=env, cwd=ROOT,
                          capture_output=True, text=True, timeout=600)


def test_reference_arm_runs_on_rank_zero_only():
    args = ["--impl", "reference", "--gpus", "2", "--config", "C1", "--steps", "1", "--warmup", "0"]
    r1 = _run_bench(1, 2, args)
    assert r1.returncode == 0 and r1.stdout.strip() == ""
    r0 = _run_bench(0, 2, args)
    assert r0.returncode == 0, r0.stderr[-2000:]
    line = json.loads(r0.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["n_gpus"] == 2
    assert line["value"] > 0 and line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0


def test_world_size_must_match_gpus():
    r = _run_bench(0, 2, ["--impl", "reference", "--gpus", "1", "--config", "C1", "--steps", "1"])
    assert r.returncode != 0 and "WORLD_SIZE" in (r.stderr + r.stdout)


def test_exact_topk_and_recall_at():
    """The recall diagnostic's exact top-k, streamed over row blocks, equals
    a full sort (score desc, row asc); Recall@x@y counts the exact top x
    among y results."""
    b = _bench()
    rng = np.random.default_rng(5)
    X = rng.standard_normal((1000, 16))
    X[500] = X[20]  # a tie: the lower row comes first
    Q = rng.standard_normal((4, 16))
    ex = b.ExactTopK(Q, 25)
    for lo in range(0, 1000, 300):
        ex.add(X[lo:lo + 300], lo)
    S = Q @ X.T
    for i in range(4):
        o = np.lexsort((np.arange(1000), -S[i]))[:25]
        assert np.array_equal(ex.ids[i], o)
    truth = ex.ids
    found = np.concatenate([truth[:, :15], np.full((4, 25), -1)], axis=1)  # 40 results
    assert ex.recall_at(found, 20) == 0.75
    assert ex.recall_at(found[:, :10], 20) == 0.5
    r = ex.recall(truth[:, :10], found)
    assert r["recall_k_at_k"] == 1.0 and r["recall_1_at_k"] == 1.0
    assert (r["recall_20_at_20"], r["recall_20_at_30"], r["recall_20_at_40"]) == (0.75, 0.75, 0.75)


def test_traffic_records_are_consistent():
    """Each ncu traffic record states its bytes per candidate as (read +
    write) / candidates, names the command that captured it, and is looked
    up only while its kernel's sources are unchanged (hash match)."""
    b = _bench()
    with open(os.path.join(ROOT, "profiles", "scan_kernel_traffic.json")) as f:
        recs = json.load(f)
    assert recs
    for key, r in recs.items():
        cfg, _, kernel = key.partition("/")
        assert kernel in b.SCAN_SOURCES, key
        assert r["command"].startswith("ncu ") and "--clock-control none" in r["command"], key
        per = (r["dram_bytes_read"] + r["dram_bytes_write"]) / r["candidates"]
        assert abs(per - r["dram_bytes_per_candidate"]) <= 1e-9 * per, key
        got = b.traffic_record(cfg, kernel)
        if r.get("kernel_hash") == b.scan_source_hash(kernel):
            assert got is not None and got["dram_bytes_per_candidate"] == r["dram_bytes_per_candidate"], key
        else:
            assert got is None, key


def test_launch_count_matches_the_profiled_lists():
    """gpu_launches per step for C4 and C5 equals the kernel launches of one
    search in the committed launch lists (23 and 38: probe, rotation, two
    list inversions, split, two passes, threshold, finalize, re-scan, and
    for C5 the GEMM probe chunks, the second rotation and the rescoring)."""
    b = _bench()
    import paper_2608_30384_gb300.workloads as W

    def desc(bits, D):
        g = {1: 4, 2: 2, 4: 1}[bits]
        Dp = (D + g - 1) // g * g
        return {"group": g, "score_bits": bits, "padded_dim": Dp, "code_bytes": (Dp // g + 1) // 2}

    for name, want in (("C4", 23), ("C5", 38)):
        w = W.WORKLOADS[name]
        assert b.launches_per_step(w, w.nq, True, b.finalize_launches(desc(w.bits, w.D), False)) == want, name
