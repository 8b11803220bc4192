"""Pins of the merge-module oracle against things other than itself (CPU only).

  * n = 1: the pooling is the identity, so z reduces to a chain of library
    routines (torch.nn.functional.linear / gelu / layer_norm in float64);
  * pooling alone equals torch's scaled_dot_product_attention with one query
    per head and keys = values = P_i (library routine);
  * invariants: sum(alpha) = 1, n copies of one token give the same z as the
    token alone, z does not depend on the order of the span's tokens,
    q = 0 gives mean pooling;
  * brute force with scalar Python loops at d = 8;
  * the parameter count printed in App. C.3.
"""
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from oracle import merge as M
from oracle import bf16
import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _weights(d, h, seed):
    w = W.merge_weights(d, h, seed)
    return {k: W.bits(v) for k, v in w.tensors().items()}


def _torch_chain(e, w, eps=1e-5):
    """z for a one-token span from library routines only."""
    t = {k: torch.from_numpy(v) for k, v in w.items()}
    x = torch.from_numpy(e)
    h1 = F.linear(x, t["w_kv"], t["b_kv"])
    p = F.layer_norm(F.gelu(h1), (x.shape[-1],), t["ln_kv_gamma"], t["ln_kv_beta"], eps)
    h2 = F.linear(p, t["w_o"], t["b_o"])
    return F.layer_norm(F.gelu(h2), (x.shape[-1],), t["ln_o_gamma"], t["ln_o_beta"], eps).numpy()


@pytest.mark.parametrize("d,h", [(64, 4), (512, 4), (256, 8)])
def test_single_token_span_is_library_chain(d, h):
    wb = _weights(d, h, 7)
    w = M.weights_f64(wb)
    case = W.merge_case(3, vocab=97, d=d, h=h, n_spans=6, kmin=1, kmax=1)
    tb = W.bits(case.table)
    z = oracle.merge_spans(tb, case.token_ids.numpy(), case.span_offsets.numpy(), w, h)
    e = bf16.to_f64(tb[case.token_ids.numpy()])
    ref = _torch_chain(e, w)
    np.testing.assert_allclose(z, ref, rtol=0, atol=1e-12)


def test_pooling_is_library_sdpa():
    r = np.random.default_rng(5)
    for n in (1, 2, 3, 4, 7):
        d, h = 64, 4
        dh = d // h
        P = r.standard_normal((n, d))
        q = r.standard_normal((h, dh))
        o, alphas = M.attention_pool(P, q, h)
        Pt = torch.from_numpy(P).view(1, n, h, dh).permute(0, 2, 1, 3)  # [1][h][n][dh]
        qt = torch.from_numpy(q).view(1, h, 1, dh)
        ref = F.scaled_dot_product_attention(qt, Pt, Pt).reshape(d).numpy()
        np.testing.assert_allclose(o, ref, rtol=0, atol=1e-12)
        np.testing.assert_allclose(alphas.sum(axis=1), np.ones(h), atol=1e-14)


def test_repeated_token_equals_single_token():
    d, h = 128, 4
    w = M.weights_f64(_weights(d, h, 11))
    table = W.bf16_normal((50, d), 0.02, 12)
    tb = W.bits(table)
    ids = np.array([17, 17, 17, 17, 17, 17, 17, 17, 17, 17], dtype=np.int32)
    offs = np.array([0, 1, 3, 6, 10], dtype=np.int32)   # n = 1, 2, 3, 4 of the same token
    z = oracle.merge_spans(tb, ids, offs, w, h)
    for i in range(1, 4):
        np.testing.assert_allclose(z[i], z[0], rtol=0, atol=1e-12)


def test_token_order_does_not_matter():
    d, h = 128, 4
    w = M.weights_f64(_weights(d, h, 21))
    tb = W.bits(W.bf16_normal((50, d), 0.02, 22))
    ids = np.array([3, 9, 41, 41, 3, 9, 9, 41, 3], dtype=np.int32)
    offs = np.array([0, 3, 6, 9], dtype=np.int32)
    z = oracle.merge_spans(tb, ids, offs, w, h)
    np.testing.assert_allclose(z[1], z[0], rtol=0, atol=1e-12)
    np.testing.assert_allclose(z[2], z[0], rtol=0, atol=1e-12)


def test_zero_query_is_mean_pooling():
    d, h = 64, 4
    w = M.weights_f64(_weights(d, h, 31))
    w["query"] = np.zeros_like(w["query"])
    tb = W.bits(W.bf16_normal((20, d), 0.02, 32))
    ids = np.array([1, 5, 7], dtype=np.int32)
    E = bf16.to_f64(tb[ids])
    P, alphas, o, z = M.merge_span_reference_steps(E, w, h)
    np.testing.assert_allclose(alphas, np.full((h, 3), 1 / 3), atol=1e-15)
    np.testing.assert_allclose(o, P.mean(axis=0), atol=1e-14)


def _brute(E, w, h, eps=1e-5):
    """Scalar loops, d tiny."""
    n, d = len(E), len(E[0])
    dh = d // h

    def lin(x, W_, b):
        return [sum(W_[o][i] * x[i] for i in range(d)) + b[o] for o in range(d)]

    def gel(v):
        return [0.5 * a * (1 + math.erf(a / math.sqrt(2))) for a in v]

    def ln(v, g, bb):
        mu = sum(v) / d
        var = sum((a - mu) ** 2 for a in v) / d
        return [(a - mu) / math.sqrt(var + eps) * g[i] + bb[i] for i, a in enumerate(v)]

    P = [ln(gel(lin(E[j], w["w_kv"], w["b_kv"])), w["ln_kv_gamma"], w["ln_kv_beta"]) for j in range(n)]
    o = [0.0] * d
    for i in range(h):
        sc = [sum(P[j][i * dh + c] * w["query"][i][c] for c in range(dh)) / math.sqrt(dh) for j in range(n)]
        m = max(sc)
        ex = [math.exp(s - m) for s in sc]
        tot = sum(ex)
        for c in range(dh):
            o[i * dh + c] = sum(ex[j] / tot * P[j][i * dh + c] for j in range(n))
    return ln(gel(lin(o, w["w_o"], w["b_o"])), w["ln_o_gamma"], w["ln_o_beta"])


def test_brute_force_tiny():
    d, h = 8, 4
    w = M.weights_f64(_weights(d, h, 41))
    wl = {k: v.tolist() for k, v in w.items()}
    tb = W.bits(W.bf16_normal((30, d), 0.5, 42))
    ids = np.array([2, 4, 6, 8, 10, 12, 1, 29, 0], dtype=np.int32)
    offs = np.array([0, 2, 5, 9], dtype=np.int32)
    z = oracle.merge_spans(tb, ids, offs, w, h)
    for s in range(3):
        E = bf16.to_f64(tb[ids[offs[s]:offs[s + 1]]]).tolist()
        np.testing.assert_allclose(z[s], _brute(E, wl, h), rtol=0, atol=1e-11)


def test_listing_semantics_batched():
    """The batched pooling of the App. C.6 listing (view into heads, einsum
    with the expanded query, softmax over the span, weighted sum), written
    with torch library ops on a batch of equal-length spans."""
    d, h, n, S = 256, 4, 3, 5
    dh = d // h
    w = M.weights_f64(_weights(d, h, 51))
    tb = W.bits(W.bf16_normal((40, d), 0.02, 52))
    ids = np.random.default_rng(0).integers(0, 40, size=S * n).astype(np.int32)
    offs = np.arange(0, S * n + 1, n).astype(np.int32)
    z = oracle.merge_spans(tb, ids, offs, w, h)
    t = {k: torch.from_numpy(v) for k, v in w.items()}
    tokens = torch.from_numpy(bf16.to_f64(tb[ids])).view(S, n, d)
    proc = F.layer_norm(F.gelu(F.linear(tokens, t["w_kv"], t["b_kv"])), (d,), t["ln_kv_gamma"], t["ln_kv_beta"], 1e-5)
    proc = proc.view(S, n, h, dh).permute(0, 2, 1, 3)
    query = t["query"].unsqueeze(0).unsqueeze(2).expand(S, h, 1, dh)
    scores = torch.einsum("bhqd,bhkd->bhk", query, proc) / math.sqrt(dh)
    weights = torch.softmax(scores, dim=2).unsqueeze(-1)
    pooled = (proc * weights).sum(dim=2).reshape(S, d)
    ref = F.layer_norm(F.gelu(F.linear(pooled, t["w_o"], t["b_o"])), (d,), t["ln_o_gamma"], t["ln_o_beta"], 1e-5)
    np.testing.assert_allclose(z, ref.numpy(), rtol=0, atol=1e-12)


def test_subset_selection_matches_full():
    d, h = 64, 4
    w = M.weights_f64(_weights(d, h, 61))
    case = W.merge_case(62, vocab=300, d=d, h=h, n_spans=20)
    tb = W.bits(case.table)
    ids, offs = case.token_ids.numpy(), case.span_offsets.numpy()
    z = oracle.merge_spans(tb, ids, offs, w, h)
    sub = [19, 0, 7]
    np.testing.assert_allclose(oracle.merge_spans(tb, ids, offs, w, h, which=sub), z[sub], rtol=0, atol=1e-12)


def test_parameter_count_matches_paper():
    g = json.load(open(os.path.join(GOLDEN, "parameter_count.json")))
    d = g["d"]
    n = M.parameter_count(d, 4)
    assert round(n / 1e6, 1) == g["approx_millions"]
    assert round(100 * n / 8e9, 2) == g["fraction_of_8B_percent"]
    # and the weight tensors the workloads hand to both sides have that many values
    w = W.merge_weights(64, 4, 1)
    assert sum(v.numel() for v in w.tensors().values()) == M.parameter_count(64, 4)


def test_gelu_is_erf_form():
    x = np.linspace(-6, 6, 1001)
    np.testing.assert_allclose(M.gelu(x), F.gelu(torch.from_numpy(x)).numpy(), atol=1e-15)
    # and differs from the tanh approximation, so a swap would be caught
    assert np.abs(M.gelu(x) - F.gelu(torch.from_numpy(x), approximate="tanh").numpy()).max() > 1e-5
