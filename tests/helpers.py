"""Shared helpers of the GPU parity tests: run the CUDA path through the C ABI
and compare with the CPU oracle on the same seeded inputs."""
import json
import os

import numpy as np
import torch

import oracle
import workloads as W

# tolerances for floating-point outputs (bf16 in, fp32 accumulate)
MAX_ABS = 1e-2
REL_L2 = 2e-3


def float_close(got, want, what=""):
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    assert got.shape == want.shape, (what, got.shape, want.shape)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    err = np.abs(got - want)
    rel = np.linalg.norm(got - want) / max(np.linalg.norm(want), 1e-30)
    log = os.environ.get("UMIM_PARITY_LOG")
    if log:
        with open(log, "a") as f:
            f.write(json.dumps({"test": os.environ.get("PYTEST_CURRENT_TEST", "").split(" ")[0], "what": what,
                                "max_abs": float(err.max()), "rel_l2": float(rel)}) + "\n")
    assert err.max() <= MAX_ABS, f"{what}: max abs err {err.max():.3e}"
    assert rel <= REL_L2, f"{what}: rel L2 err {rel:.3e}"
    return float(err.max()), float(rel)


def umim():
    import paper_2609_27233_gb300 as m
    m.lib()
    return m


def dev():
    return torch.device("cuda:0")


def case_to_dev(c, d):
    return dict(pool=c.pool.to(d), bt=c.block_table.to(d), lens=c.seq_lens.to(d), offs=c.span_offsets.to(d),
                st=c.span_start.to(d), ln=c.span_len.to(d), sk=c.surrogate_k.to(d), sv=c.surrogate_v.to(d),
                q=c.q.to(d))


def oracle_rollback(c):
    return oracle.kv_rollback(W.bits(c.pool), c.block_table.cpu().numpy(), c.seq_lens.cpu().numpy(),
                              c.span_offsets.cpu().numpy(), c.span_start.cpu().numpy(),
                              c.span_len.cpu().numpy(), W.bits(c.surrogate_k), W.bits(c.surrogate_v))


def compare_rollback(g_pool, g_bt, g_lens, g_freed, ref):
    """Bit-exact: block table, lengths, freed pages, every valid KV byte."""
    rp, rbt, rl, rfreed = ref
    bt = g_bt.cpu().numpy()
    lens = g_lens.cpu().numpy()
    np.testing.assert_array_equal(bt, rbt)
    np.testing.assert_array_equal(lens, rl)
    f = g_freed.cpu().numpy()
    assert f[:len(rfreed)].tolist() == rfreed
    if len(rfreed) < len(f):
        assert f[len(rfreed)] == -1
    gp = W.bits(g_pool)
    for b in range(len(rl)):
        t = np.arange(int(rl[b]))
        pg, sl = rbt[b, t // 16], t % 16
        np.testing.assert_array_equal(gp[:, pg, :, :, sl, :], rp[:, pg, :, :, sl, :], err_msg=f"seq {b}")


def oracle_append_merge(pool, bt, lens, nk, nv, new_pages, merge_k, sk, sv):
    """kv_append, then kv_rollback of the suffix span (L + 1 - k, k) of every
    merging sequence (surrogate rows in sequence order); released pages per
    sequence from the rollback's freed list."""
    L0 = lens.copy()
    pool, bt, lens, rej = oracle.kv_append(pool, bt, lens, nk, nv, new_pages)
    assert rej == []
    B = len(L0)
    offs = np.zeros(B + 1, np.int32)
    st, ln = [], []
    for b in range(B):
        offs[b + 1] = offs[b]
        if merge_k[b] > 0:
            st.append(int(L0[b]) + 1 - int(merge_k[b]))
            ln.append(int(merge_k[b]))
            offs[b + 1] += 1
    pool, bt2, lens2, freed = oracle.kv_rollback(pool, bt, lens, offs, np.array(st, np.int32),
                                                 np.array(ln, np.int32), sk, sv)
    released = np.full(B, -1, np.int32)
    fi = iter(freed)
    for b in range(B):
        if (int(lens[b]) + 15) // 16 > (int(lens2[b]) + 15) // 16:
            released[b] = next(fi)
    return pool, bt2, lens2, released
