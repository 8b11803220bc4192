"""Pins of the decode-attention oracle against things other than itself (CPU only).

  * torch's scaled_dot_product_attention (enable_gqa) on a contiguous cache
    rebuilt from the pages (library routine);
  * closed forms: one cached entry gives v_0, identical keys give the mean of
    the values, softmax weights sum to 1;
  * attention after a rollback equals attention over a cache rebuilt
    explicitly (Python lists) at the shorter length.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from oracle import bf16
import workloads as W

P = 16


def _contig(pool, bt_row, L, layer):
    t = np.arange(L)
    K = bf16.to_f64(pool[layer, bt_row[t // P], 0, :, t % P, :])
    V = bf16.to_f64(pool[layer, bt_row[t // P], 1, :, t % P, :])
    return K, V


@pytest.mark.parametrize("hq,hkv,d", [(8, 2, 64), (32, 8, 128), (28, 4, 128), (4, 4, 16)])
def test_matches_library_sdpa_gqa(hq, hkv, d):
    case = W.decode_case(10, lens=[1, 16, 17, 200], n_q_heads=hq, n_kv_heads=hkv, head_dim=d,
                         n_layers=2, n_spans=[0, 0, 0, 0])
    pool, bt, lens = W.bits(case.pool), case.block_table.numpy(), case.seq_lens.numpy()
    qb = W.bits(case.q)
    out = oracle.decode_attention(qb, pool, 1, bt, lens)
    q = bf16.to_f64(qb)
    for b in range(4):
        K, V = _contig(pool, bt[b], int(lens[b]), 1)
        qt = torch.from_numpy(q[b]).view(1, hq, 1, d)
        kt = torch.from_numpy(K).permute(1, 0, 2).unsqueeze(0)
        vt = torch.from_numpy(V).permute(1, 0, 2).unsqueeze(0)
        ref = F.scaled_dot_product_attention(qt, kt, vt, enable_gqa=True).view(hq, d).numpy()
        np.testing.assert_allclose(out[b], ref, rtol=0, atol=1e-12)


def test_closed_forms():
    case = W.decode_case(11, lens=[1, 40], n_q_heads=8, n_kv_heads=2, head_dim=32, n_spans=[0, 0])
    pool, bt = W.bits(case.pool), case.block_table.numpy()
    lens = case.seq_lens.numpy()
    qb = W.bits(case.q)
    out, wts = oracle.decode_attention(qb, pool, 0, bt, lens, return_weights=True)
    # one cached entry: the output is that entry's value
    K, V = _contig(pool, bt[0], 1, 0)
    for h in range(8):
        np.testing.assert_allclose(out[0, h], V[0, h // 4], atol=1e-15)
    for b in range(2):
        for h in range(8):
            assert abs(wts[b][h].sum() - 1.0) < 1e-12
    # identical keys: every weight is 1/L and the output is the mean value
    pool2 = pool.copy()
    page0, slot0 = bt[1, 0], 0
    for t in range(40):
        pool2[0, bt[1, t // P], 0, :, t % P, :] = pool[0, page0, 0, :, slot0, :]
    out2 = oracle.decode_attention(qb, pool2, 0, bt, lens)
    K, V = _contig(pool2, bt[1], 40, 0)
    for h in range(8):
        np.testing.assert_allclose(out2[1, h], V[:, h // 4].mean(axis=0), atol=1e-13)


def test_empty_cache_gives_zero():
    case = W.decode_case(12, lens=[0, 5], n_q_heads=2, n_kv_heads=1, head_dim=16, n_spans=[0, 0])
    out = oracle.decode_attention(W.bits(case.q), W.bits(case.pool), 0, case.block_table.numpy(),
                                  case.seq_lens.numpy())
    assert np.all(out[0] == 0)


def test_after_rollback_equals_rebuilt_cache():
    case = W.decode_case(13, lens=[300, 123], n_q_heads=8, n_kv_heads=2, head_dim=32, coverage=0.4)
    pool, bt, lens = W.bits(case.pool), case.block_table.numpy(), case.seq_lens.numpy()
    offs, st, ln = case.span_offsets.numpy(), case.span_start.numpy(), case.span_len.numpy()
    sk, sv = W.bits(case.surrogate_k), W.bits(case.surrogate_v)
    pool2, bt2, lens2, _ = oracle.kv_rollback(pool, bt, lens, offs, st, ln, sk, sv)
    out = oracle.decode_attention(W.bits(case.q), pool2, 0, bt2, lens2)
    q = bf16.to_f64(W.bits(case.q))
    for b in range(2):
        K, V = _contig(pool, bt[b], int(lens[b]), 0)
        Kl, Vl = list(K), list(V)
        for i in reversed(range(offs[b], offs[b + 1])):
            s, k = int(st[i]), int(ln[i])
            Kl[s:s + k] = [bf16.to_f64(sk[i, 0])]
            Vl[s:s + k] = [bf16.to_f64(sv[i, 0])]
        Kr, Vr = np.stack(Kl), np.stack(Vl)
        assert len(Kr) == lens2[b]
        for h in range(8):
            s_ = Kr[:, h // 4] @ q[b, h] / math.sqrt(32)
            e = np.exp(s_ - s_.max())
            np.testing.assert_allclose(out[b, h], (e / e.sum()) @ Vr[:, h // 4], atol=1e-12)


@pytest.mark.parametrize("pieces", [1, 2, 5, 40])
def test_split_keys_merged_by_log_sum_exp_equal_the_whole(pieces):
    """The split-K form: softmax statistics (max, sum, weighted values) of
    separate key ranges, merged with log-sum-exp weights, give the same
    output as attention over all keys at once (float64, any split)."""
    case = W.decode_case(15, lens=[333, 40], n_q_heads=8, n_kv_heads=2, head_dim=32, n_spans=[0, 0])
    pool, bt, lens = W.bits(case.pool), case.block_table.numpy(), case.seq_lens.numpy()
    qb = W.bits(case.q)
    out = oracle.decode_attention(qb, pool, 0, bt, lens)
    q = bf16.to_f64(qb)
    for b in range(2):
        K, V = _contig(pool, bt[b], int(lens[b]), 0)
        bounds = np.linspace(0, int(lens[b]), pieces + 1).astype(int)
        for h in range(8):
            parts = []
            for lo, hi in zip(bounds[:-1], bounds[1:]):
                if hi == lo:
                    continue
                s = K[lo:hi, h // 4] @ q[b, h] / math.sqrt(32)
                m = s.max()
                e = np.exp(s - m)
                parts.append((m, e.sum(), e @ V[lo:hi, h // 4]))
            M = max(p[0] for p in parts)
            l = sum(p[1] * math.exp(p[0] - M) for p in parts)
            acc = sum(p[2] * math.exp(p[0] - M) for p in parts)
            np.testing.assert_allclose(acc / l, out[b, h], rtol=0, atol=1e-12)
