"""Decode-step KV append on the GPU against the oracle: bit-exact pool,
block tables and sequence lengths after every step, page boundaries and
rejected appends included."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from helpers import dev, umim

pytestmark = pytest.mark.gpu


def _free_pages(bt, n_pages):
    used = set(int(x) for x in bt[bt >= 0].ravel())
    return [p for p in range(n_pages) if p not in used]


CASES = [
    # seed, lens, Hkv, D, layers, steps
    (21, [0, 1, 15, 16, 17, 31, 32, 100], 8, 128, 3, 20),
    (22, [5, 64, 2047], 2, 64, 2, 18),
    (23, list(range(0, 600, 3)), 4, 128, 1, 4),     # 200 sequences, every phase of a page
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
