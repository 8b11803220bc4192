"""Failure detection on the GPU without faulting it: every bounded wait of
the library, given something that never happens, gives up after its limit
with UMIM_ERR_TIMEOUT and the context stays usable; memory outside the
pages a call may touch is left alone (canary pages around the pool)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from helpers import dev, umim

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("which", [0, 1])
def test_bounded_wait_gives_up_and_the_context_stays_usable(which):
    m, dv = umim(), dev()
    status, elapsed = m.umim_selftest_bounded_wait(which, 20000, dv)   # 20 ms
    torch.cuda.synchronize()
    assert int(status.item()) == 4   # UMIM_ERR_TIMEOUT
    assert 20e6 <= int(elapsed.item()) < 1e9
    # the context still runs ordinary work
    c = W.decode_case(5, lens=[40, 7], n_q_heads=4, n_kv_heads=2, head_dim=64, coverage=0.0)
    st = m.new_status(dv)
    out = m.umim_decode_attention(c.q.to(dv), c.pool.to(dv), 0, c.block_table.to(dv), c.seq_lens.to(dv),
                                  dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0 and torch.isfinite(out.float()).all()


def test_rollback_leaves_canary_pages_alone():
    """Pages no sequence owns (before, between and after the sequences' pages
    in the pool) keep their bytes through a rollback, and so do the slots of
    every sequence before its first span."""
    m, dv = umim(), dev()
    c = W.decode_case(6, lens=[300, 4096, 77, 1000], n_q_heads=8, n_kv_heads=8, head_dim=128, n_layers=2,
                      coverage=0.3, spare_pages=40)
    bt0 = c.block_table.numpy()
    owned = set(int(x) for x in bt0[bt0 >= 0].ravel())
    canary = np.array([p for p in range(c.n_pages) if p not in owned])
    assert len(canary) >= 40
    pool = c.pool.to(dv)
    m.umim_kv_rollback(pool, c.block_table.to(dv), c.seq_lens.to(dv), c.span_offsets.to(dv), c.span_start.to(dv),
                       c.span_len.to(dv), c.surrogate_k.to(dv), c.surrogate_v.to(dv))
    torch.cuda.synchronize()
    before, after = W.bits(c.pool), W.bits(pool)
    np.testing.assert_array_equal(after[:, canary], before[:, canary])
    offs, st = c.span_offsets.numpy(), c.span_start.numpy()
    for b in range(len(bt0)):
        first = int(st[offs[b]]) if offs[b + 1] > offs[b] else int(c.seq_lens[b])
        t = np.arange(first)
        pg, slot = bt0[b, t // 16], t % 16
        np.testing.assert_array_equal(after[:, pg, :, :, slot, :], before[:, pg, :, :, slot, :])
