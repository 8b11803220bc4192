"""Pins of the compaction oracle and of the oracle's bf16 rounding (CPU only).

  * the worked example of App. C.5 / App. J.4 with positions [0, 1, 2];
  * the compressed-length formula of App. E;
  * bf16 round-to-nearest-even against torch's float32 -> bfloat16 cast
    (library routine), including ties, subnormals, infinities and NaN.
"""
import json
import os

import numpy as np
import torch

import oracle
from oracle import bf16
import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_worked_example():
    g = json.load(open(os.path.join(GOLDEN, "prompt_compaction_example.json")))
    d = 16
    tb = W.bits(W.bf16_normal((10, d), 0.02, 1))
    ids = np.array([[4, 7, 2, 9]], np.int32)    # x1..x4
    z = np.random.default_rng(0).standard_normal((1, d)).astype(np.float32)
    s, k = g["span"]["start"], g["span"]["length"]
    out, pos, cu = oracle.build_compressed(tb, ids, np.array([0, 1]), np.array([s]), np.array([k]), z)
    units = {"e(x1)": tb[4], "e(x4)": tb[9], "z23": bf16.from_f32(z[0])}
    np.testing.assert_array_equal(out, np.stack([units[u] for u in g["compressed_units"]]))
    assert pos.tolist() == g["compressed_positions"]
    assert cu.tolist() == [0, 3]


def test_compressed_length_formula():
    g = json.load(open(os.path.join(GOLDEN, "prompt_length.json")))
    for cs in g["cases"]:
        L = cs["L_p"]
        sp = cs["spans"]
        st = np.array([a for a, _ in sp], np.int32)
        ln = np.array([b - a for a, b in sp], np.int32)
        tb = W.bits(W.bf16_normal((L + 1, 8), 0.02, 2))
        ids = np.arange(L, dtype=np.int32)[None, :]
        z = np.zeros((len(sp), 8), np.float32)
        out, pos, cu = oracle.build_compressed(tb, ids, np.array([0, len(sp)]), st, ln, z)
        assert len(out) == cs["L_compressed"] == cu[-1]
        assert pos.tolist() == list(range(cs["L_compressed"]))


def test_no_spans_is_embedding_lookup():
    case = W.prompt_case(3, B=3, L=50, vocab=200, d=32, coverage=0.0)
    tb = W.bits(case.table)
    ids = case.token_ids.numpy()
    out, pos, cu = oracle.build_compressed(tb, ids, case.span_offsets.numpy(), case.span_start.numpy(),
                                           case.span_len.numpy(), np.zeros((0, 32), np.float32))
    np.testing.assert_array_equal(out, tb[ids.reshape(-1)])
    assert cu.tolist() == [0, 50, 100, 150]
    assert pos.tolist() == list(range(50)) * 3


def test_bf16_rounding_matches_torch():
    r = np.random.default_rng(1)
    x = np.concatenate([
        r.standard_normal(100000).astype(np.float32) * 10.0 ** r.integers(-40, 38, 100000),
        np.array([np.inf, -np.inf, 0.0, -0.0, 1e-45, -1e-40, 3.4e38], np.float32),
    ]).astype(np.float32)
    # exact ties: low 16 bits = 0x8000, both parities of the kept part
    u = r.integers(0, 2 ** 31, 1000, dtype=np.uint32)
    ties = ((u & np.uint32(0xFFFF0000)) | np.uint32(0x8000)).view(np.float32)
    ties = ties[np.isfinite(ties)]
    x = np.concatenate([x, ties])
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(bf16.from_f32(x), want)
    assert np.isnan(bf16.to_f64(bf16.from_f32(np.array([np.nan], np.float32))))[0]
    back = torch.from_numpy(want.view(np.int16)).view(torch.bfloat16).double().numpy()
    np.testing.assert_array_equal(bf16.to_f64(want), back)
