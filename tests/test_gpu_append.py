"""Decode-step KV append on the GPU against the oracle: bit-exact pool,
block tables and sequence lengths after every step, page boundaries and
rejected appends included."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from helpers import dev, oracle_append_merge, umim

pytestmark = pytest.mark.gpu


def _free_pages(bt, n_pages):
    used = set(int(x) for x in bt[bt >= 0].ravel())
    return [p for p in range(n_pages) if p not in used]


CASES = [
    # seed, lens, Hkv, D, layers, steps
    (21, [0, 1, 15, 16, 17, 31, 32, 100], 8, 128, 3, 20),
    (22, [5, 64, 2047], 2, 64, 2, 18),
    (23, list(range(0, 600, 3)), 4, 128, 1, 4),     # 200 sequences, every phase of a page
    # entries large enough that several CTAs share one sequence (2 and 8 of them)
    (25, [0, 15, 16, 33, 300], 8, 128, 5, 18),
    (26, [1, 16, 31, 64, 1000, 7], 8, 128, 32, 18),
]


@pytest.mark.parametrize("seed,lens,hkv,d,layers,steps", CASES)
def test_append_steps_match_oracle(seed, lens, hkv, d, layers, steps):
    m = umim()
    dv = dev()
    B = len(lens)
    extra = (steps + 15) // 16 + 1
    c = W.decode_case(seed, lens=lens, n_q_heads=hkv, n_kv_heads=hkv, head_dim=d, n_layers=layers,
                      coverage=0.0, spare_pages=B * extra, extra_max_pages=extra)
    pool = c.pool.to(dv)
    bt = c.block_table.to(dv)
    sl = c.seq_lens.to(dv)
    o_pool, o_bt, o_lens = W.bits(c.pool), c.block_table.numpy(), c.seq_lens.numpy()
    alloc = W.PageAllocator(_free_pages(o_bt, c.n_pages))
    status = m.new_status(dv)
    for step in range(steps):
        nk = W.bf16_normal((B, layers, hkv, d), 1.0, seed * 1000 + 2 * step, dv)
        nv = W.bf16_normal((B, layers, hkv, d), 1.0, seed * 1000 + 2 * step + 1, dv)
        new_pages = alloc.take(o_lens)
        m.umim_kv_append(pool, bt, sl, nk, nv, torch.from_numpy(new_pages).to(dv), dev_status=status)
        o_pool, o_bt, o_lens, rej = oracle.kv_append(o_pool, o_bt, o_lens, W.bits(nk), W.bits(nv), new_pages)
        assert rej == []
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        np.testing.assert_array_equal(bt.cpu().numpy(), o_bt)
        np.testing.assert_array_equal(sl.cpu().numpy(), o_lens)
    # every byte of the pool: appended slots and everything left alone
    np.testing.assert_array_equal(W.bits(pool), o_pool)


def test_impossible_appends_are_rejected_and_leave_the_sequence_unchanged():
    m = umim()
    dv = dev()
    lens = [32, 5, 16, 48, 16, 7]       # max_pages = 3: sequence 3 is full
    c = W.decode_case(24, lens=lens, n_q_heads=8, n_kv_heads=8, head_dim=128, n_layers=2, coverage=0.0,
                      spare_pages=4)
    assert c.max_pages == 3
    B = len(lens)
    pool, bt, sl = c.pool.to(dv), c.block_table.to(dv), c.seq_lens.to(dv)
    free = _free_pages(c.block_table.numpy(), c.n_pages)
    # 0: boundary, no page given; 2: page outside the pool; 4: a good new page
    new_pages = np.array([-1, -1, c.n_pages, 0, free[0], -1], np.int32)
    nk = W.bf16_normal((B, 2, 8, 128), 1.0, 901, dv)
    nv = W.bf16_normal((B, 2, 8, 128), 1.0, 902, dv)
    status = m.new_status(dv)
    m.umim_kv_append(pool, bt, sl, nk, nv, torch.from_numpy(new_pages).to(dv), dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 1   # UMIM_ERR_INVALID_ARG
    o_pool, o_bt, o_lens, rej = oracle.kv_append(W.bits(c.pool), c.block_table.numpy(), c.seq_lens.numpy(),
                                                 W.bits(nk), W.bits(nv), new_pages)
    assert rej == [0, 2, 3]
    np.testing.assert_array_equal(bt.cpu().numpy(), o_bt)
    np.testing.assert_array_equal(sl.cpu().numpy(), o_lens)
    np.testing.assert_array_equal(W.bits(pool), o_pool)


def test_no_page_list_needed_inside_pages():
    m = umim()
    dv = dev()
    c = W.decode_case(25, lens=[3, 17, 40], n_q_heads=4, n_kv_heads=4, head_dim=64, n_layers=1, coverage=0.0)
    pool, bt, sl = c.pool.to(dv), c.block_table.to(dv), c.seq_lens.to(dv)
    nk = W.bf16_normal((3, 1, 4, 64), 1.0, 903, dv)
    nv = W.bf16_normal((3, 1, 4, 64), 1.0, 904, dv)
    status = m.new_status(dv)
    m.umim_kv_append(pool, bt, sl, nk, nv, None, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    o_pool, o_bt, o_lens, rej = oracle.kv_append(W.bits(c.pool), c.block_table.numpy(), c.seq_lens.numpy(),
                                                 W.bits(nk), W.bits(nv), None)
    assert rej == []
    np.testing.assert_array_equal(sl.cpu().numpy(), o_lens)
    np.testing.assert_array_equal(W.bits(pool), o_pool)


# ---------------------------------------------------------------------------
# append or suffix merge in one call (the decode loop's cache update)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("seed,lens,hkv,d,layers,steps", [
    (41, [0, 1, 15, 16, 17, 31, 32, 100, 255, 256], 8, 128, 3, 30),
    (42, [3, 16, 47, 64, 2047], 2, 64, 2, 24),
    (44, [0, 14, 16, 17, 48, 500], 8, 128, 12, 20),   # 3 CTAs per sequence
    (45, [5, 15, 16, 31, 260], 8, 128, 32, 20),       # 8 CTAs per sequence
])
def test_append_merge_matches_append_then_suffix_rollback(seed, lens, hkv, d, layers, steps):
    m = umim()
    dv = dev()
    B = len(lens)
    extra = (steps + 15) // 16 + 1
    c = W.decode_case(seed, lens=lens, n_q_heads=hkv, n_kv_heads=hkv, head_dim=d, n_layers=layers,
                      coverage=0.0, spare_pages=B * extra, extra_max_pages=extra)
    pool, bt, sl = c.pool.to(dv), c.block_table.to(dv), c.seq_lens.to(dv)
    o_pool, o_bt, o_lens = W.bits(c.pool), c.block_table.numpy(), c.seq_lens.numpy()
    alloc = W.PageAllocator(_free_pages(o_bt, c.n_pages))
    r = W.rng(seed + 7)
    status = m.new_status(dv)
    n_merged = 0
    for step in range(steps):
        nk = W.bf16_normal((B, layers, hkv, d), 1.0, seed * 1000 + 2 * step, dv)
        nv = W.bf16_normal((B, layers, hkv, d), 1.0, seed * 1000 + 2 * step + 1, dv)
        new_pages = alloc.take(o_lens)
        # about a third of the sequences merge; k up to 16, never past the start
        merge_k = np.where(r.random(B) < 0.35, r.integers(1, 17, size=B), 0).astype(np.int32)
        merge_k = np.minimum(merge_k, o_lens + 1).astype(np.int32)
        rows = np.cumsum(merge_k > 0).astype(np.int32) - 1
        merge_row = np.where(merge_k > 0, rows, -1).astype(np.int32)
        S = int((merge_k > 0).sum())
        sk = W.bf16_normal((max(S, 1), layers, hkv, d), 1.0, seed * 1000 + 500 + 2 * step, dv)
        sv = W.bf16_normal((max(S, 1), layers, hkv, d), 1.0, seed * 1000 + 501 + 2 * step, dv)
        t = lambda x: torch.from_numpy(x).to(dv)
        rel = m.umim_decode_append_merge(pool, bt, sl, nk, nv, t(new_pages), t(merge_k), t(merge_row), sk, sv,
                                         dev_status=status)
        o_pool, o_bt, o_lens, o_rel = oracle_append_merge(o_pool, o_bt, o_lens, W.bits(nk), W.bits(nv), new_pages,
                                                           merge_k, W.bits(sk)[:S], W.bits(sv)[:S])
        alloc.give_back([p for p in o_rel if p >= 0])
        n_merged += S
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        np.testing.assert_array_equal(bt.cpu().numpy(), o_bt, err_msg=f"step {step}")
        np.testing.assert_array_equal(sl.cpu().numpy(), o_lens, err_msg=f"step {step}")
        np.testing.assert_array_equal(rel.cpu().numpy(), o_rel, err_msg=f"step {step}")
        gp = W.bits(pool)
        for b in range(B):
            tt = np.arange(int(o_lens[b]))
            pg, slot = o_bt[b, tt // 16], tt % 16
            np.testing.assert_array_equal(gp[:, pg, :, :, slot, :], o_pool[:, pg, :, :, slot, :],
                                          err_msg=f"step {step} seq {b}")
    assert n_merged > 0


@pytest.mark.parametrize("layers", [2, 32])   # one CTA, and 4 CTAs, per sequence
def test_impossible_merges_are_rejected_and_leave_the_sequence_unchanged(layers):
    m = umim()
    dv = dev()
    lens = [10, 20, 3, 40]
    c = W.decode_case(43, lens=lens, n_q_heads=4, n_kv_heads=4, head_dim=128, n_layers=layers, coverage=0.0,
                      spare_pages=4, extra_max_pages=1)
    pool, bt, sl = c.pool.to(dv), c.block_table.to(dv), c.seq_lens.to(dv)
    nk = W.bf16_normal((4, layers, 4, 128), 1.0, 905, dv)
    nv = W.bf16_normal((4, layers, 4, 128), 1.0, 906, dv)
    sk = W.bf16_normal((2, layers, 4, 128), 1.0, 907, dv)
    sv = W.bf16_normal((2, layers, 4, 128), 1.0, 908, dv)
    # 0: k = 17 (longer than supported); 1: row outside the surrogates; 2: k > L + 1; 3: a good merge
    merge_k = torch.tensor([17, 2, 5, 3], dtype=torch.int32, device=dv)
    merge_row = torch.tensor([0, 2, 0, 1], dtype=torch.int32, device=dv)
    status = m.new_status(dv)
    rel = m.umim_decode_append_merge(pool, bt, sl, nk, nv, None, merge_k, merge_row, sk, sv, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 1   # UMIM_ERR_INVALID_ARG
    got_lens = sl.cpu().numpy()
    assert list(got_lens) == [10, 20, 3, 40 + 1 - 3 + 1]
    np.testing.assert_array_equal(bt.cpu().numpy()[:3], c.block_table.numpy()[:3])
    gp, op = W.bits(pool), W.bits(c.pool)
    for b in range(3):
        tt = np.arange(lens[b])
        pg, slot = c.block_table.numpy()[b, tt // 16], tt % 16
        np.testing.assert_array_equal(gp[:, pg, :, :, slot, :], op[:, pg, :, :, slot, :])
    # the good merge: surrogate row 1 at slot 38
    p38 = c.block_table.numpy()[3, 38 // 16]
    np.testing.assert_array_equal(gp[:, p38, 0, :, 38 % 16, :], W.bits(sk)[1])
    np.testing.assert_array_equal(gp[:, p38, 1, :, 38 % 16, :], W.bits(sv)[1])
    assert rel.cpu().numpy()[3] == -1
