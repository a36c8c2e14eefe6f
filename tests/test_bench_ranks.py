"""bench.py's multi-process bookkeeping on CPU, as two gloo ranks: the job's time is the
slowest rank's, the job's rate counts every replica's sequences, and the reference arm
runs on rank 0 only and prints one line of the benchmark's JSON contract. (The drafter runs as independent replicas, one per GPU, with no
exchange on the data path; these are the only cross-rank steps.)"""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, ws, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws))
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    try:
        times = [3.0, 5.0, 4.0, 1.0]
        slowest = bench.max_over_ranks(times[rank], ws, "cpu")
        q.put((rank, "max", slowest))
        q.put((rank, "dist_env", bench.dist_env()))
    finally:
        dist.destroy_process_group()


def test_slowest_rank_time_and_job_rate():
    import torch.multiprocessing as mp
    ws = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, ws, port, q)) for r in range(ws)]
    for p in procs:
        p.start()
    got = {}
    try:
        for _ in range(2 * ws):  # two results per rank
            r, what, v = q.get(timeout=120)
            got[(r, what)] = v
    finally:
        for p in procs:
            p.join(timeout=60)
            if p.exitcode is None:
                p.kill()
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    assert got[(0, "max")] == got[(1, "max")] == 5.0
    assert got[(0, "dist_env")] == (2, 0, 0) and got[(1, "dist_env")] == (2, 1, 0)


def test_single_process_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(2.5, 1, "cpu") == 2.5
    # two replicas of B = 32 sequences, 1.346 ms per step: 47548 drafts/s for the job
    assert bench.job_rate(2, 32, 1.346e-3) == pytest.approx(2 * 32 / 1.346e-3)
    assert bench.job_rate(1, 1, 1e-3) == pytest.approx(1000.0)


def test_reference_arm_runs_on_rank_zero_only(capsys):
    sys.path.insert(0, ROOT)
    import bench
    # a non-zero rank returns at once, before reading its arguments, building any input or
    # touching the oracle
    assert bench.run_reference(None, 2, 1) is None
    assert capsys.readouterr().out == ""


def test_reference_arm_prints_one_contract_line():
    """`bench.py --impl reference` (the oracle on the host cores) prints exactly one JSON
    line with the keys the benchmark contract names, on a workload small enough for CPU."""
    import json
    import subprocess
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny",
                        "--steps", "2", "--warmup", "1"], capture_output=True, text=True, timeout=300, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    line = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "impl", "cpu_baseline", "e2e"):
        assert key in line, key
    assert line["impl"] == "reference" and line["metric"] == line["unit"] == "drafts/s"
    assert line["value"] > 0 and line["higher_is_better"] is True and line["vs_baseline"] is None
    assert line["config"]["workload"] == "tiny"
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"] == {"value": line["value"], "unit": "drafts/s", "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}


def test_in_step_times_partition_the_stamped_span():
    """fe_profile_graph's stamps -> per-launch added time: with programmatic launches the
    spans overlap, and each launch is charged only the time its end lies past the previous
    end, so the charges sum to the run's span; bench.py folds operand preps into their
    phase's family."""
    sys.path.insert(0, ROOT)
    import importlib
    fe_binding = importlib.import_module("paper_2509_20416_gb300")
    import bench
    stamps = [("linear", 0.0, 10.0), ("attention", 8.0, 13.0), ("linear", 9.0, 20.0), ("lm_prep", 19.5, 21.0),
              ("lm_head", 20.0, 30.0), ("lm_head", 29.0, 31.0), ("copy", -1.0, -1.0), ("tree", 31.0, 31.5)]
    its = fe_binding.in_step_times(stamps)
    assert [k for k, _, _ in its] == ["linear", "attention", "linear", "lm_prep", "lm_head", "lm_head", "tree"]
    assert [a for _, _, a in its] == pytest.approx([10.0, 3.0, 7.0, 1.0, 9.0, 1.0, 0.5])
    assert sum(a for _, _, a in its) == pytest.approx(31.5)
    fam = bench.family_times(its + its, 2)
    assert fam["linear"]["launches_per_draft"] == 2 and fam["linear"]["us_per_draft"] == pytest.approx(17.0)
    assert fam["lm_head"]["launches_per_draft"] == 2 and fam["lm_head"]["us_per_draft"] == pytest.approx(11.0)
    assert sum(v["us_per_draft"] for v in fam.values()) == pytest.approx(31.5)
    assert fam["linear"]["span_us_per_draft"] == pytest.approx(21.0)
