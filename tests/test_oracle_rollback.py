"""Pins of the rollback oracle against things other than itself (CPU only).

  * the worked example of App. C.5 ([x1,x2,x3,x4] -> [x1, z23, x4]);
  * the cache-length formula of App. E, L_C' = L_C - (n-1) + 1, and
    L' = L - sum(k - 1);
  * k = 1 with the stored entry as surrogate leaves everything byte-identical;
  * a brute force on Python lists (slice deletion and insertion, one span at
    a time from the right) equals the batched call;
  * pages before the first span are untouched; freed pages are exactly the
    emptied tail of each block table.
"""
import json
import os

import numpy as np
import pytest

import oracle
import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
P = 16


def _np(case):
    return dict(pool=W.bits(case.pool), bt=case.block_table.numpy(), lens=case.seq_lens.numpy(),
                offs=case.span_offsets.numpy(), st=case.span_start.numpy(), ln=case.span_len.numpy(),
                sk=W.bits(case.surrogate_k), sv=W.bits(case.surrogate_v))


def _run(c):
    return oracle.kv_rollback(c["pool"], c["bt"], c["lens"], c["offs"], c["st"], c["ln"], c["sk"], c["sv"])


def _logical(pool, bt_row, L, layer=0):
    """Logical entries of one sequence as a list of byte strings (K and V)."""
    out = []
    for t in range(L):
        page, slot = bt_row[t // P], t % P
        out.append(pool[layer, page, :, :, slot, :].tobytes())
    return out


def _sur(sk, sv, i, layer=0):
    return np.stack([sk[i, layer], sv[i, layer]]).tobytes()


def test_worked_example_app_c5():
    g = json.load(open(os.path.join(GOLDEN, "prompt_compaction_example.json")))
    case = W.decode_case(1, lens=[4], n_q_heads=2, n_kv_heads=1, head_dim=8, n_spans=[0])
    c = _np(case)
    s, k = g["span"]["start"], g["span"]["length"]
    c["offs"] = np.array([0, 1], np.int32)
    c["st"] = np.array([s], np.int32)
    c["ln"] = np.array([k], np.int32)
    c["sk"] = W.bits(W.bf16_normal((1, 1, 1, 8), 1.0, 5))
    c["sv"] = W.bits(W.bf16_normal((1, 1, 1, 8), 1.0, 6))
    before = _logical(c["pool"], c["bt"][0], 4)
    pool, bt, lens, freed = _run(c)
    assert lens[0] == len(g["compressed_units"])
    after = _logical(pool, bt[0], int(lens[0]))
    names = {"e(x1)": before[0], "e(x4)": before[3], "z23": _sur(c["sk"], c["sv"], 0)}
    assert after == [names[u] for u in g["compressed_units"]]
    assert freed == []


def test_decode_cache_length_formula():
    g = json.load(open(os.path.join(GOLDEN, "decode_cache_length.json")))
    for cs in g["cases"]:
        LC, n = cs["L_C"], cs["n"]
        # the n-1 cached entries of the suffix are replaced by the surrogate's one entry
        case = W.decode_case(2, lens=[LC], n_q_heads=1, n_kv_heads=1, head_dim=8, n_spans=[0])
        c = _np(case)
        c["offs"] = np.array([0, 1], np.int32)
        c["st"] = np.array([LC - (n - 1)], np.int32)
        c["ln"] = np.array([n - 1], np.int32)
        c["sk"] = W.bits(W.bf16_normal((1, 1, 1, 8), 1.0, 7))
        c["sv"] = W.bits(W.bf16_normal((1, 1, 1, 8), 1.0, 8))
        _, _, lens, _ = _run(c)
        assert lens[0] == cs["L_C_after"]


def test_length_formula_many_spans():
    case = W.decode_case(3, lens=[700, 33, 64, 0, 1], n_q_heads=4, n_kv_heads=2, head_dim=16,
                         coverage=0.4)
    c = _np(case)
    _, _, lens, _ = _run(c)
    for b in range(5):
        lo, hi = c["offs"][b], c["offs"][b + 1]
        assert lens[b] == c["lens"][b] - int((c["ln"][lo:hi] - 1).sum())


def test_k1_with_stored_entry_is_identity():
    case = W.decode_case(4, lens=[100, 37], n_q_heads=4, n_kv_heads=2, head_dim=16, n_layers=3,
                         coverage=0.5, kmin=1, kmax=1)
    c = _np(case)
    # surrogate = the entry already stored at the span's position
    for b in range(2):
        for i in range(c["offs"][b], c["offs"][b + 1]):
            t = c["st"][i]
            page, slot = c["bt"][b, t // P], t % P
            c["sk"][i] = c["pool"][:, page, 0, :, slot, :]
            c["sv"][i] = c["pool"][:, page, 1, :, slot, :]
    pool, bt, lens, freed = _run(c)
    assert pool.tobytes() == c["pool"].tobytes()
    np.testing.assert_array_equal(bt, c["bt"])
    np.testing.assert_array_equal(lens, c["lens"])
    assert freed == []


def _brute_lists(c, layer):
    """Python-list model: per sequence, delete each span's slice and insert its
    surrogate, handling spans from the rightmost to the leftmost."""
    res = []
    for b in range(len(c["lens"])):
        seq = _logical(c["pool"], c["bt"][b], int(c["lens"][b]), layer)
        for i in reversed(range(c["offs"][b], c["offs"][b + 1])):
            s, k = int(c["st"][i]), int(c["ln"][i])
            seq[s:s + k] = [_sur(c["sk"], c["sv"], i, layer)]
        res.append(seq)
    return res


@pytest.mark.parametrize("seed,lens,layers,cov", [
    (5, [512], 1, 0.4), (6, [100, 0, 17, 300, 16, 32], 2, 0.3), (7, [1000, 999], 3, 0.6)])
def test_against_list_brute_force(seed, lens, layers, cov):
    case = W.decode_case(seed, lens=lens, n_q_heads=4, n_kv_heads=2, head_dim=8, n_layers=layers,
                         coverage=cov)
    c = _np(case)
    pool, bt, nl, freed = _run(c)
    for layer in range(layers):
        want = _brute_lists(c, layer)
        for b in range(len(lens)):
            assert _logical(pool, bt[b], int(nl[b]), layer) == want[b]


def test_untouched_prefix_and_freed_pages():
    case = W.decode_case(8, lens=[400, 250, 77], n_q_heads=8, n_kv_heads=2, head_dim=16, n_layers=2,
                         coverage=0.35, spare_pages=3)
    c = _np(case)
    pool, bt, nl, freed = _run(c)
    exp_freed = []
    for b in range(3):
        L, Lp = int(c["lens"][b]), int(nl[b])
        first = int(c["st"][c["offs"][b]])
        for p in range(first // P):
            page = c["bt"][b, p]
            assert pool[:, page].tobytes() == c["pool"][:, page].tobytes()
        for p in range((Lp + P - 1) // P, (L + P - 1) // P):
            exp_freed.append(int(c["bt"][b, p]))
            assert bt[b, p] == -1
        np.testing.assert_array_equal(bt[b, :(Lp + P - 1) // P], c["bt"][b, :(Lp + P - 1) // P])
    assert freed == exp_freed
    assert len(set(freed)) == len(freed)


def test_invalid_spans_rejected_before_mutation():
    case = W.decode_case(9, lens=[64], n_q_heads=2, n_kv_heads=1, head_dim=8, n_spans=[0])
    c = _np(case)
    c["offs"] = np.array([0, 2], np.int32)
    c["sk"] = W.bits(W.bf16_normal((2, 1, 1, 8), 1.0, 5))
    c["sv"] = W.bits(W.bf16_normal((2, 1, 1, 8), 1.0, 6))
    for st, ln in [([4, 5], [2, 2]), ([10, 4], [2, 2]), ([60, 62], [2, 3]), ([3, 9], [0, 2])]:
        c["st"], c["ln"] = np.array(st, np.int32), np.array(ln, np.int32)
        with pytest.raises(ValueError):
            _run(c)


@pytest.mark.parametrize("L,spans,exp_len,exp_pages", [
    (20, [(0, 5)], 16, 1),        # L' lands exactly on a page boundary
    (32, [(3, 17)], 16, 1),       # L is a page multiple too
    (33, [(1, 2)], 32, 2),
    (16, [(0, 16)], 1, 1),        # the whole cache collapses into one entry
])
def test_page_aligned_lengths(L, spans, exp_len, exp_pages):
    case = W.decode_case(14, lens=[L], n_q_heads=2, n_kv_heads=1, head_dim=8, n_spans=[0])
    c = _np(case)
    c["offs"] = np.array([0, len(spans)], np.int32)
    c["st"] = np.array([s for s, _ in spans], np.int32)
    c["ln"] = np.array([k for _, k in spans], np.int32)
    c["sk"] = W.bits(W.bf16_normal((len(spans), 1, 1, 8), 1.0, 5))
    c["sv"] = W.bits(W.bf16_normal((len(spans), 1, 1, 8), 1.0, 6))
    pool, bt, lens, freed = _run(c)
    assert lens[0] == exp_len
    n_before = (L + P - 1) // P
    assert freed == [int(x) for x in c["bt"][0, exp_pages:n_before]]
    assert np.all(bt[0, exp_pages:] == -1)
    np.testing.assert_array_equal(bt[0, :exp_pages], c["bt"][0, :exp_pages])


@pytest.mark.parametrize("seed,lens,cov", [(21, [300, 64, 0, 17], 0.4), (22, [1000], 0.6)])
def test_one_span_at_a_time_right_to_left_equals_the_batched_call(seed, lens, cov):
    """Rolling back the spans one call at a time, rightmost first (so every
    start is still valid), ends in the state of the one batched call: same
    lengths, same block tables, same logical entries, same set of pages
    released."""
    case = W.decode_case(seed, lens=lens, n_q_heads=4, n_kv_heads=2, head_dim=8, n_layers=2, coverage=cov)
    c = _np(case)
    pool, bt, nl, freed = _run(c)
    B = len(lens)
    p1, b1, l1, f1 = c["pool"], c["bt"], c["lens"], []
    for b in range(B):
        for i in reversed(range(int(c["offs"][b]), int(c["offs"][b + 1]))):
            o = np.zeros(B + 1, np.int32)
            o[b + 1:] = 1
            p1, b1, l1, f = oracle.kv_rollback(p1, b1, l1, o, c["st"][i:i + 1], c["ln"][i:i + 1],
                                               c["sk"][i:i + 1], c["sv"][i:i + 1])
            f1 += f
    np.testing.assert_array_equal(l1, nl)
    np.testing.assert_array_equal(b1, bt)
    assert sorted(f1) == sorted(freed)
    for layer in range(2):
        for b in range(B):
            assert _logical(p1, b1[b], int(l1[b]), layer) == _logical(pool, bt[b], int(nl[b]), layer)
