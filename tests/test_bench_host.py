"""Host-side logic of bench.py's multi-rank path, on CPU with gloo (world size 2).

Ranks run independent trajectories (weak scaling); the only collectives are the
host-side timing reductions: iterations are summed and the slowest rank's time
is taken.
"""
import os
import socket

import pytest
import torch.multiprocessing as mp

import workload as W


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    import torch.distributed as dist
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    units, secs = bench.aggregate(10 * (rank + 1), 0.5 + rank)
    w = bench.rank_workload(W.BATCHED, rank)
    out[rank] = (units, secs, w.seed, bench.rank_info())
    dist.barrier()
    dist.destroy_process_group()


def test_aggregate_and_rank_seeds_gloo():
    world = 2
    port = _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    for r in range(world):
        units, secs, seed, info = out[r]
        assert units == 30.0 and secs == 1.5
        assert seed == W.BATCHED.seed + r * W.BATCHED.batch
        assert info == (r, world, r)


def test_single_process_aggregate_is_identity():
    import bench
    assert bench.aggregate(7, 0.25) == (7.0, 0.25)


def test_iteration_bytes_counts_rows():
    import numpy as np
    import bench
    w = W.TINY
    # iteration 0: t=0, p=8, 8 misses, stride 4, frontier 0 (all lazy), no hits;
    # iteration 1: t=4, p=8, 5 misses, stride 8, frontier 8, 3 hits at j >= 1
    log = np.zeros((2, 1, 8), dtype=np.int32)
    log[0, 0, :6] = (0, 8, 8, 4, 0, 0)
    log[1, 0, :6] = (4, 8, 5, 8, 8, 3)
    upd, gat, den = bench.iteration_bytes(log, w)
    row = w.D * 4
    assert upd[0] == (1 + 0 + 8 + 16 + 0 + 8) * row
    # iteration 1: lazy = 4 + 8 - 8 = 4; 3 ehat hits; 10 entry writes; 3 xhat reads
    assert upd[1] == (1 + 4 + 5 + 8) * row + (3 + 10 + 3) * row
    # the planning kernel gathers iteration 1's 5 rows after iteration 0 (read
    # and write), nothing after the last iteration; the fused step only writes
    assert gat[0] == 2 * 5 * row and gat[1] == 0
    _, gat_f, _ = bench.iteration_bytes(log, w, fused=True)
    assert gat_f[0] == 5 * row and gat_f[1] == 0
    assert den[0] == (2 * 8 + w.K) * row and den[1] == (2 * 5 + w.K) * row
    # bfloat16 entries: the 16 entry writes count half a row each
    upd16, _, _ = bench.iteration_bytes(log, w, entry_bytes=2)
    assert upd16[0] == (1 + 0 + 8 + 8) * row + 16 * (row // 2)


def test_cpu_baseline_legs(monkeypatch):
    """cpu_baseline reports the one-thread leg as its value, an all-cores leg
    beside it, the CPU model and the solver step with the denoiser excluded."""
    import bench
    calls = []

    def fake(name, budget, threads=1, cache_thresh=None):
        calls.append(threads)
        return {"iters": 8, "generations": 2, "seconds": 2.0, "denoiser_seconds": 1.5,
                "nfe_per_gen": 10, "iters_per_gen": 4}

    monkeypatch.setattr(bench, "time_oracle_subprocess", fake)
    cb = bench.cpu_baseline("tiny", budget_s=0.0)
    assert calls == [1, os.cpu_count() or 1]
    assert cb["cores"] == 1 and cb["value"] == 4.0 and cb["kind"] == "oracle"
    assert cb["host_cores"] == (os.cpu_count() or 1) and cb["cpu_model"]
    assert abs(cb["solver_step_us_per_iteration"] - 1e6 * 0.5 / 8) < 1e-6
    assert cb["all_cores"]["threads"] == (os.cpu_count() or 1)
    assert abs(cb["all_cores"]["solver_steps_per_s_denoiser_excluded"] - 16.0) < 1e-9


def test_reference_config_matches_ours():
    """Both arms carry the same workload-only config for the same workload."""
    import bench
    w = W.SD15
    c = bench.workload_config(w, 1, 4)
    assert c["workload"] == w.name and c["solver_steps_per_step"] == 4 and c["window"] == 100
    assert set(c) >= {"workload", "global_batch", "seq_len"}


@pytest.mark.parametrize("workload", ["tiny", "srds"])
def test_reference_arm_json_line(workload):
    """bench.py --impl reference times the fp64 oracle on the host and prints
    one JSON line with the contract's keys (CPU only, no GPU involved)."""
    import json
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference",
                        "--workload", workload, "--steps", "1", "--warmup", "0"],
                       capture_output=True, text=True, timeout=600, cwd=root)
    assert r.returncode == 0, r.stderr[-2000:]
    line = json.loads(r.stdout.strip().splitlines()[-1])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config", "e2e",
                "cpu_baseline"):
        assert key in line, key
    assert line["impl"] == "reference" and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] == 1
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["value"] == line["value"]
    assert line["config"]["workload"] == W.ALL[workload].name
    assert line["config"]["solver_steps_per_step"] >= 1
