"""KV rollback / compaction on the GPU against the oracle: bit-exact block
tables, sequence lengths, freed pages and every moved KV byte."""
import numpy as np
import pytest
import torch

import workloads as W
from helpers import case_to_dev, compare_rollback, dev, oracle_rollback, umim

pytestmark = pytest.mark.gpu


def _run(c, ws=None):
    m = umim()
    d = dev()
    g = case_to_dev(c, d)
    status = m.new_status(d)
    freed = m.umim_kv_rollback(g["pool"], g["bt"], g["lens"], g["offs"], g["st"], g["ln"], g["sk"], g["sv"],
                               workspace_buf=ws, dev_status=status)
    torch.cuda.synchronize()
    return g, freed, int(status.item())


CASES = [
    # seed, lens, Hq, Hkv, D, layers, coverage, kmin, kmax
    (1, [512], 8, 2, 64, 1, None, 2, 4),                                  # tiny: 40 spans below
    (2, [1, 15, 16, 17, 300, 1000, 0, 33], 32, 8, 128, 3, 0.3, 2, 4),     # ragged, 2 head groups
    (3, [2048, 777], 28, 4, 128, 2, 0.6, 2, 4),                           # dense coverage
    (4, [400, 129, 64], 16, 16, 64, 1, 0.5, 1, 4),                        # k = 1 spans, 2 head groups
    (5, [4096], 8, 1, 128, 1, 0.05, 2, 4),                                # sparse spans
    (6, [100, 50], 8, 8, 128, 2, 0.9, 3, 8),                              # long spans
]


@pytest.mark.parametrize("seed,lens,hq,hkv,d,layers,cov,kmin,kmax", CASES)
def test_rollback_matches_oracle(seed, lens, hq, hkv, d, layers, cov, kmin, kmax):
    n_spans = [40] if cov is None else None
    c = W.decode_case(seed, lens=lens, n_q_heads=hq, n_kv_heads=hkv, head_dim=d, n_layers=layers,
                      coverage=cov, n_spans=n_spans, kmin=kmin, kmax=kmax, spare_pages=5)
    g, freed, st = _run(c)
    assert st == 0
    compare_rollback(g["pool"], g["bt"], g["lens"], freed, oracle_rollback(c))


def test_spans_at_both_ends_and_page_aligned_lengths():
    c = W.decode_case(11, lens=[64, 48, 20, 16], n_q_heads=4, n_kv_heads=2, head_dim=128, n_spans=[0, 0, 0, 0])
    # seq 0: first and last entries; seq 1: start, middle, end; seq 2: none; seq 3: whole cache -> 1 entry
    c.span_offsets = torch.tensor([0, 2, 5, 5, 6], dtype=torch.int32)
    c.span_start = torch.tensor([0, 60, 0, 10, 44, 0], dtype=torch.int32)
    c.span_len = torch.tensor([3, 4, 5, 5, 4, 16], dtype=torch.int32)
    c.surrogate_k = W.bf16_normal((6, 1, 2, 128), 1.0, 5)
    c.surrogate_v = W.bf16_normal((6, 1, 2, 128), 1.0, 6)
    g, freed, st = _run(c)
    assert st == 0
    compare_rollback(g["pool"], g["bt"], g["lens"], freed, oracle_rollback(c))


def test_identity_when_k1_surrogate_is_stored_entry():
    c = W.decode_case(12, lens=[300, 31], n_q_heads=8, n_kv_heads=8, head_dim=64, n_layers=2, coverage=0.5,
                      kmin=1, kmax=1)
    pool = W.bits(c.pool)
    bt = c.block_table.numpy()
    sk, sv = W.bits(c.surrogate_k).copy(), W.bits(c.surrogate_v).copy()
    offs, st = c.span_offsets.numpy(), c.span_start.numpy()
    for b in range(2):
        for i in range(offs[b], offs[b + 1]):
            t = st[i]
            sk[i] = pool[:, bt[b, t // 16], 0, :, t % 16, :]
            sv[i] = pool[:, bt[b, t // 16], 1, :, t % 16, :]
    c.surrogate_k = torch.from_numpy(sk.view(np.int16)).view(torch.bfloat16)
    c.surrogate_v = torch.from_numpy(sv.view(np.int16)).view(torch.bfloat16)
    g, freed, s = _run(c)
    assert s == 0
    assert W.bits(g["pool"]).tobytes() == pool.tobytes()
    np.testing.assert_array_equal(g["bt"].cpu().numpy(), bt)
    np.testing.assert_array_equal(g["lens"].cpu().numpy(), c.seq_lens.numpy())
    assert int(freed[0].item()) == -1


def test_no_spans_changes_nothing():
    c = W.decode_case(13, lens=[100, 0, 37], n_q_heads=4, n_kv_heads=2, head_dim=128, n_spans=[0, 0, 0])
    pool = W.bits(c.pool).copy()
    g, freed, s = _run(c)
    assert s == 0
    assert W.bits(g["pool"]).tobytes() == pool.tobytes()
    np.testing.assert_array_equal(g["lens"].cpu().numpy(), c.seq_lens.numpy())
    assert int(freed[0].item()) == -1


@pytest.mark.parametrize("bad", ["overlap", "past_end", "zero_len", "bad_page", "len_too_big"])
def test_invalid_input_is_rejected_before_any_write(bad):
    c = W.decode_case(14, lens=[64, 64], n_q_heads=4, n_kv_heads=2, head_dim=128, n_spans=[3, 3])
    st, ln, bt, lens = c.span_start.clone(), c.span_len.clone(), c.block_table.clone(), c.seq_lens.clone()
    if bad == "overlap":
        st[1] = st[0]
    elif bad == "past_end":
        st[5] = 63
        ln[5] = 4
    elif bad == "zero_len":
        ln[4] = 0
    elif bad == "bad_page":
        bt[1, 2] = c.pool.shape[1] + 7
    elif bad == "len_too_big":
        lens[0] = bt.shape[1] * 16 + 1
    c.span_start, c.span_len, c.block_table, c.seq_lens = st, ln, bt, lens
    pool = W.bits(c.pool).copy()
    g, freed, s = _run(c)
    assert s == 1                                   # UMIM_ERR_INVALID_ARG
    assert W.bits(g["pool"]).tobytes() == pool.tobytes()
    np.testing.assert_array_equal(g["bt"].cpu().numpy(), bt.numpy())
    np.testing.assert_array_equal(g["lens"].cpu().numpy(), lens.numpy())


def test_workspace_reused_across_calls():
    """The call counter in the workspace keeps read-done flags of one call
    from satisfying the next call's waits."""
    m = umim()
    d = dev()
    c1 = W.decode_case(15, lens=[1500, 900], n_q_heads=8, n_kv_heads=2, head_dim=128, n_layers=2, coverage=0.4)
    c2 = W.decode_case(16, lens=[1500, 900], n_q_heads=8, n_kv_heads=2, head_dim=128, n_layers=2, coverage=0.4)
    S = max(c1.span_start.numel(), c2.span_start.numel())
    ws = m.workspace(m.umim_kv_rollback_workspace_size(2, S, c1.block_table.shape[1], 2, 2, 128), d)
    for c in (c1, c2, c1):
        g, freed, s = _run(c, ws)
        assert s == 0
        compare_rollback(g["pool"], g["bt"], g["lens"], freed, oracle_rollback(c))


@pytest.mark.parametrize("name", ["llama8b_layer", "long_context", "long_context_tr40"])
def test_full_size_configs(name):
    seed = W.SEEDS[name]
    if name == "llama8b_layer":
        c = W.decode_case(seed, lens=[4096] * 16, n_q_heads=32, n_kv_heads=8, head_dim=128, coverage=0.3)
    elif name == "long_context":
        c = W.decode_case(seed, lens=[32768] * 4, n_q_heads=28, n_kv_heads=4, head_dim=128, coverage=0.4)
    else:
        c = W.decode_case(seed, lens=[32768] * 4, n_q_heads=28, n_kv_heads=4, head_dim=128, coverage=0.6)
    g, freed, s = _run(c)
    assert s == 0
    compare_rollback(g["pool"], g["bt"], g["lens"], freed, oracle_rollback(c))
