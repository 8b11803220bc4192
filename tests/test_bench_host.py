"""Host-side arithmetic of bench.py on the CPU: the algorithmic work that the
roofline fractions divide by, the per-kernel table, the traffic lookup keyed
to the profiled sources, and the serving loop's scheduler bookkeeping checked
against the oracle's append and rollback."""
import hashlib
import json
import os

import numpy as np
import pytest

import bench
import oracle
import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_algorithmic_work_of_the_bench_step():
    st = bench.make_structure(0x5EED0002)
    w = bench.WORKLOAD
    work = bench.algorithmic_work(st)
    B, L = w["B"], w["L"]
    entry = 2 * w["Hkv"] * w["D"] * 2
    offs, ss, ll = st["span_offsets"], st["span_start"], st["span_len"]
    # every entry after a sequence's first span that survives moves once: L - s_first - sum(k)
    moved = sum(L - int(ss[offs[b]]) - int(ll[offs[b]:offs[b + 1]].sum()) for b in range(B) if offs[b + 1] > offs[b])
    S = len(ss)
    assert work["S"] == S and work["T"] == int(ll.sum()) == len(st["span_tokens"])
    assert work["rollback_bytes"] == (moved + S) * entry * 2 + 4 * (3 * S + 3 * B)
    Lp = np.array([L - int((ll[offs[b]:offs[b + 1]] - 1).sum()) for b in range(B)])
    np.testing.assert_array_equal(work["Lp"], Lp)
    assert work["attention_bytes"] >= Lp.sum() * entry
    assert work["gemm1_flop"] == 2.0 * work["T"] * w["d_model"] ** 2
    assert work["gemm2_flop"] == 2.0 * S * w["d_model"] ** 2
    # the workload is the one the bench names: 30 % of positions in spans of 2..4
    assert abs(ll.sum() / (B * L) - 0.3) < 0.002 and ll.min() >= 2 and ll.max() <= 4


def test_kernel_table_shares_and_rates():
    recs = [("a", 2.0), ("b", 1.0), ("a", 2.0), ("b", 1.0), ("c", 0.5)]
    work = {"a": ("hbm", 4.0, "GB/s", 8000.0)}      # 4 GB per launch
    t = bench.kernel_table(recs, 2, work)
    assert abs(sum(v["share"] for v in t.values()) - 1.0) < 1e-3
    assert t["a"]["ms"] == 2.0 and t["a"]["launches_per_step"] == 1.0
    assert t["a"]["achieved"] == 2000.0 and t["a"]["frac"] == 0.25   # 4 GB in 2 ms
    assert "frac" not in t["c"]


def test_traffic_is_reported_only_for_unchanged_sources():
    prof = json.load(open(os.path.join(ROOT, "profiles", "ncu_traffic.json")))
    for label, e in prof.items():
        src = os.path.join(ROOT, "paper_2609_27233_gb300", "csrc", e["source"])
        same = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16] == e["source_sha"]
        got = bench.traffic_from_profile(label, e["workload"])
        assert (got == e["bytes_per_launch_full"]) if same else got is None, label
        # a capture is never reported for another workload's launch of the kernel
        assert bench.traffic_from_profile(label, "another_workload") is None, label
    assert bench.traffic_from_profile("no.such.kernel") is None


@pytest.mark.parametrize("seed", [1, 2])
def test_serving_plan_matches_the_oracle(seed):
    sl = W.serving_loop(seed, B=12, n_layers=1, n_q_heads=2, n_kv_heads=1, head_dim=8, steps=60, p=0.3,
                        lens=[1, 15, 16, 17, 31, 32, 33, 2, 100, 47, 48, 5])
    plan = bench.serving_plan(sl)
    pool = W.bits(sl.init_pool("cpu"))
    bt, lens = sl.block_table.copy(), sl.lens.copy()
    alloc = W.PageAllocator(sl.free_pages)
    for step, p in enumerate(plan):
        new_pages = alloc.take(lens)
        np.testing.assert_array_equal(new_pages, p["new_pages"])
        nk, nv = (W.bits(x) for x in sl.new_entries(step, "cpu"))
        pool, bt, lens, rej = oracle.kv_append(pool, bt, lens, nk, nv, new_pages)
        assert rej == []
        S = len(p["st"])
        sk = np.zeros((S, 1, 1, 8), np.uint16)
        pool, bt, lens, freed = oracle.kv_rollback(pool, bt, lens, p["offs"], p["st"], p["ln"], sk, sk)
        alloc.give_back(freed)
        np.testing.assert_array_equal(lens, p["lens_after"])
