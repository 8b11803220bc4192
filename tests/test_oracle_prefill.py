"""Pins of the oracle's prefill attention over packed compressed prompts.

  * torch's scaled_dot_product_attention (causal, grouped-query) on every
    sequence separately (a library routine);
  * closed forms: the first row of a sequence attends only to itself (out =
    v_0); with all keys of a sequence equal, row i is the mean of v_0..v_i;
  * packing: a batch gives each sequence what it gets alone;
  * the last row of a sequence equals decode attention (the separately pinned
    decode oracle) of that row's query over the sequence's keys and values.
"""
import numpy as np
import pytest
import torch

from oracle import bf16
from oracle.attention import attend
from oracle.prefill import prefill_attention


def _bits(x):
    return bf16.from_f64(np.asarray(x, dtype=np.float64))


def _case(seed, lens, hq, hkv, d):
    r = np.random.default_rng(seed)
    T = sum(lens)
    q = _bits(r.normal(0, 1, (T, hq, d)))
    k = _bits(r.normal(0, 1, (T, hkv, d)))
    v = _bits(r.normal(0, 1, (T, hkv, d)))
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    return q, k, v, cu


@pytest.mark.parametrize("hq,hkv,d", [(4, 4, 16), (8, 2, 32), (6, 3, 8)])
def test_matches_library_causal_sdpa(hq, hkv, d):
    lens = [1, 7, 13]
    q, k, v, cu = _case(hq * 10 + d, lens, hq, hkv, d)
    got = prefill_attention(q, k, v, cu)
    for b in range(len(lens)):
        lo, hi = cu[b], cu[b + 1]
        tq = torch.from_numpy(bf16.to_f64(q[lo:hi])).permute(1, 0, 2)[None]
        tk = torch.from_numpy(bf16.to_f64(k[lo:hi])).permute(1, 0, 2)[None]
        tv = torch.from_numpy(bf16.to_f64(v[lo:hi])).permute(1, 0, 2)[None]
        want = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, is_causal=True, enable_gqa=True)
        np.testing.assert_allclose(got[lo:hi], want[0].permute(1, 0, 2).numpy(), rtol=1e-12, atol=1e-12)


def test_closed_forms():
    q, k, v, cu = _case(1, [9, 5], 4, 2, 16)
    out = prefill_attention(q, k, v, cu)
    for b in range(2):
        lo = cu[b]
        np.testing.assert_allclose(out[lo], np.repeat(bf16.to_f64(v[lo]), 2, axis=0), rtol=1e-12)
    k_eq = k.copy()
    k_eq[:] = k[0]
    out = prefill_attention(q, k_eq, v, cu)
    vf = bf16.to_f64(v)
    for b in range(2):
        lo, hi = cu[b], cu[b + 1]
        for i in range(lo, hi):
            want = np.repeat(vf[lo:i + 1].mean(axis=0), 2, axis=0)
            np.testing.assert_allclose(out[i], want, rtol=1e-12, atol=1e-14)


def test_packing_is_per_sequence():
    lens = [5, 0, 11, 3]
    q, k, v, cu = _case(2, lens, 4, 4, 8)
    packed = prefill_attention(q, k, v, cu)
    for b in range(len(lens)):
        lo, hi = cu[b], cu[b + 1]
        alone = prefill_attention(q[lo:hi], k[lo:hi], v[lo:hi], np.array([0, hi - lo]))
        np.testing.assert_array_equal(packed[lo:hi], alone)


def test_last_row_is_decode_attention():
    lens = [6, 17]
    q, k, v, cu = _case(3, lens, 8, 2, 16)
    out = prefill_attention(q, k, v, cu)
    qf, kf, vf = bf16.to_f64(q), bf16.to_f64(k), bf16.to_f64(v)
    for b in range(2):
        lo, hi = cu[b], cu[b + 1]
        for h in range(8):
            want, _ = attend(qf[hi - 1, h], kf[lo:hi, h // 4], vf[lo:hi, h // 4], 1 / 4.0)
            np.testing.assert_allclose(out[hi - 1, h], want, rtol=1e-12, atol=1e-14)


def test_bad_offsets_are_refused():
    q, k, v, cu = _case(4, [3, 3], 2, 2, 8)
    for bad in ([1, 3, 6], [0, 4, 3], [0, 3, 7]):
        with pytest.raises(ValueError):
            prefill_attention(q, k, v, np.array(bad))
