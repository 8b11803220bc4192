"""The benchmark's multi-process path on the CPU: two gloo ranks, one
independent batch each (replicas, no data-path collective).  The job's time
is the slowest rank's and its work is the sum of every rank's."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, ms_of, units_of, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms, units = bench.reduce_over_ranks(ms_of[rank], units_of[rank], torch.device("cpu"))
        dist.barrier()
        q.put((rank, ms, units))
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time_and_the_total_work():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    ms_of, units_of = [12.5, 19.25], [6555 * 100, 6601 * 100]
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, ms_of, units_of, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, ms, units in got:
        assert ms == pytest.approx(19.25)
        assert units == pytest.approx(sum(units_of))


def test_one_process_is_the_identity():
    assert bench.reduce_over_ranks(3.5, 42, torch.device("cpu")) == (3.5, 42.0)


def test_ranks_get_independent_batches_of_the_same_shape():
    a = bench.make_structure(0x5EED0002)
    b = bench.make_structure(0x5EED0002 + 1000)
    assert a["token_ids"].shape == b["token_ids"].shape
    assert not np.array_equal(a["span_start"], b["span_start"])
    # weak scaling: about the same work per rank (30 % coverage of the same lengths)
    assert abs(len(a["span_start"]) - len(b["span_start"])) < 0.05 * len(a["span_start"])


def _run_bench(args, env_extra):
    import json
    import subprocess
    import sys
    env = dict(os.environ, **env_extra)
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, os.path.join(root, "bench.py")] + args, cwd=root, env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    return [json.loads(l) for l in lines]


def test_reference_arm_prints_one_line_with_the_contract_keys():
    """The oracle arm runs on the host cores only and prints one JSON line
    on the same metric, unit and workload as the GPU arm."""
    (line,) = _run_bench(["--impl", "reference", "--steps", "2", "--warmup", "3"], {})
    assert line["impl"] == "reference"
    # the steps it reports were timed, not extrapolated: they fit in the run's own wall time
    assert line["steps"] == 2 and line["ms_per_step"] * line["steps"] <= 1000.0 * line["wall_s"] + 1.0
    assert line["metric"] == bench.METRIC and line["unit"] == bench.UNIT
    assert line["higher_is_better"] is True and line["value"] > 0
    assert line["config"]["workload"].startswith("llama8b_layer")
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["value"] == line["value"]
    assert line["e2e"] == {"value": line["value"], "unit": bench.UNIT, "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}


def test_reference_arm_other_ranks_exit_without_work():
    assert _run_bench(["--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "3"],
                      {"RANK": "1", "WORLD_SIZE": "2", "LOCAL_RANK": "1"}) == []
