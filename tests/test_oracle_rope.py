"""Pins of the oracle's position-aware rollback (App. J.4: compressed positions
pi(t) = t - r(t), and its RoPE discussion) and of its float64 -> bf16
rounding.

  * bf16.from_f64 against exact rational arithmetic (nearest, ties to even);
  * keys built as RoPE rotations of raw vectors at their original positions
    (numpy complex exponentials, the blockwise-rotation definition) become,
    after the rollback, the rotations at the compressed positions, within
    the two bf16 roundings involved;
  * the change of each moved key respects the paper's bound
    ||R_D - R_{D-d}||_2 = 2 max_m |sin(d w_m / 2)| (times the key norm);
  * inner products between keys moved by the same shift are unchanged
    (a common rotation);
  * everything that must not change is bit-exact: entries that do not move,
    V rows, surrogate entries, columns at or beyond rotary_dim.
"""
from fractions import Fraction

import numpy as np
import pytest

from oracle import bf16
from oracle.rollback import kv_rollback

P = 16


def _bf16_val(b):
    return Fraction(float(np.array([np.uint32(b) << 16], dtype=np.uint32).view(np.float32)[0]))


def test_from_f64_is_nearest_ties_to_even():
    r = np.random.default_rng(0)
    x = np.concatenate([r.normal(0, 1, 3000), r.normal(0, 1e-4, 300), r.normal(0, 1e5, 300), [0.0, -0.0]])
    got = bf16.from_f64(x)
    for xi, g in zip(x, got):
        g = int(g)
        d = abs(Fraction(float(xi)) - _bf16_val(g))
        for nb in (g - 1, g + 1):
            if 0 <= nb < 0x7F80 or 0x8000 <= nb < 0xFF80:
                assert d <= abs(Fraction(float(xi)) - _bf16_val(nb))
    # exact ties go to the even pattern
    base = r.integers(0x3F80, 0x4700, 500).astype(np.uint32)
    lo = (base << 16).view(np.float32).astype(np.float64)
    hi = ((base + 1) << 16).view(np.float32).astype(np.float64)
    got = bf16.from_f64((lo + hi) / 2)
    want = np.where(base % 2 == 0, base, base + 1).astype(np.uint16)
    np.testing.assert_array_equal(got, want)


def _inv_freq(D, base=500000.0, rotary_dim=None):
    rd = D if rotary_dim is None else rotary_dim
    return (base ** (-np.arange(0, rd, 2, dtype=np.float64) / rd)).astype(np.float32)


def _rope_case(seed, L, spans, D=64, hkv=2, layers=2, rotary_dim=None):
    """A one-sequence cache whose keys are raw vectors rotated at their
    positions: pair m of K_t is (x + i y) * exp(i t w_m)."""
    r = np.random.default_rng(seed)
    rd = D if rotary_dim is None else rotary_dim
    w = _inv_freq(D, rotary_dim=rd).astype(np.float64)
    raw = r.normal(0, 1, size=(L, layers, hkv, D))
    z = raw[..., :rd // 2] + 1j * raw[..., rd // 2:rd]
    zt = z * np.exp(1j * np.arange(L)[:, None, None, None] * w)
    keys = raw.copy()
    keys[..., :rd // 2], keys[..., rd // 2:rd] = zt.real, zt.imag
    pages = (L + P - 1) // P
    n_pages = pages + 2
    perm = r.permutation(n_pages).astype(np.int32)
    bt = perm[:pages][None, :].copy()
    pool = r.integers(0, 1 << 16, size=(layers, n_pages, 2, hkv, P, D), dtype=np.uint16) & 0x3FFF
    t = np.arange(L)
    kb = bf16.from_f64(keys)                                   # [L][layers][hkv][D]
    for layer in range(layers):
        pool[layer, bt[0, t // P], 0, :, t % P, :] = kb[:, layer]
    st = np.array([s for s, _ in spans], np.int32)
    ln = np.array([k for _, k in spans], np.int32)
    S = len(spans)
    sk = r.integers(0, 1 << 16, size=(S, layers, hkv, D), dtype=np.uint16) & 0x3FFF
    sv = r.integers(0, 1 << 16, size=(S, layers, hkv, D), dtype=np.uint16) & 0x3FFF
    return dict(pool=pool, bt=bt, lens=np.array([L], np.int32), offs=np.array([0, S], np.int32), st=st, ln=ln,
                sk=sk, sv=sv, raw=raw, z=z, w=w, rd=rd, D=D)


def _moves(L, spans):
    """(t, j, r) for every kept entry."""
    out, t, j, r = [], 0, 0, 0
    for s, k in list(spans) + [(L, 0)]:
        while t < s:
            out.append((t, j, r))
            t, j = t + 1, j + 1
        if k:
            t, j, r = s + k, j + 1, r + k - 1
    return out


def _run(c, rope=True):
    return kv_rollback(c["pool"], c["bt"], c["lens"], c["offs"], c["st"], c["ln"], c["sk"], c["sv"],
                       rope_inv_freq=c["w"].astype(np.float32) if rope else None, rotary_dim=c["rd"])


SPANS = [(5, 3), (20, 4), (21 + 10, 2), (60, 4), (100, 3)]


@pytest.mark.parametrize("rotary_dim", [None, 32])
def test_moved_keys_carry_their_compressed_positions(rotary_dim):
    L = 140
    c = _rope_case(1, L, SPANS, rotary_dim=rotary_dim)
    pool, bt, lens, _ = _run(c)
    rd, w, D = c["rd"], c["w"], c["D"]
    for (t, j, r) in _moves(L, SPANS):
        got = bf16.to_f64(pool[:, bt[0, j // P], 0, :, j % P, :])           # [layers][hkv][D]
        want = c["z"][t] * np.exp(1j * j * w)                                # rotation at pi(t) = j
        gz = got[..., :rd // 2] + 1j * got[..., rd // 2:rd]
        norm = np.abs(c["z"][t])
        # two roundings of a bf16 value (before and after the rotation), each <= 2^-9 of the pair norm per part
        assert np.all(np.abs(gz - want) <= 2 * 2.0 ** -8 * norm + 1e-30), (t, j, r)
        if rd < D:   # columns past rotary_dim are moved verbatim
            src = c["pool"][:, c["bt"][0, t // P], 0, :, t % P, rd:]
            np.testing.assert_array_equal(pool[:, bt[0, j // P], 0, :, j % P, rd:], src)


def test_a_sign_slip_in_the_rotation_fails_the_identity():
    """The identity above is strict enough to catch rotating the wrong way."""
    L = 140
    c = _rope_case(2, L, SPANS)
    wrong = dict(c)
    wrong["w"] = -c["w"]
    pool, bt, _, _ = _run(wrong)
    bad = 0
    for (t, j, r) in _moves(L, SPANS):
        if r == 0:
            continue
        got = bf16.to_f64(pool[:, bt[0, j // P], 0, :, j % P, :])
        gz = got[..., :32] + 1j * got[..., 32:64]
        want = c["z"][t] * np.exp(1j * j * c["w"])
        bad += int(np.any(np.abs(gz - want) > 2 * 2.0 ** -8 * np.abs(c["z"][t]) + 1e-30))
    assert bad > 0


def test_change_respects_the_rotation_bound_and_common_shifts_keep_inner_products():
    L = 140
    c = _rope_case(3, L, SPANS)
    pool, bt, _, _ = _run(c)
    w = c["w"]
    by_shift = {}
    for (t, j, r) in _moves(L, SPANS):
        old = bf16.to_f64(c["pool"][:, c["bt"][0, t // P], 0, :, t % P, :])
        new = bf16.to_f64(pool[:, bt[0, j // P], 0, :, j % P, :])
        bound = 2 * np.max(np.abs(np.sin(r * w / 2)))
        for layer in range(old.shape[0]):
            for h in range(old.shape[1]):
                n = np.linalg.norm(old[layer, h])
                assert np.linalg.norm(new[layer, h] - old[layer, h]) <= bound * n + 2 ** -7 * n
        by_shift.setdefault(r, []).append((old, new))
    for r, pairs in by_shift.items():
        for (a0, a1), (b0, b1) in zip(pairs, pairs[1:]):
            before = np.sum(a0 * b0, axis=-1)
            after = np.sum(a1 * b1, axis=-1)
            scale = np.linalg.norm(a0, axis=-1) * np.linalg.norm(b0, axis=-1)
            assert np.all(np.abs(after - before) <= 2 ** -6 * scale)


def test_what_does_not_move_or_is_not_a_key_is_unchanged():
    L = 140
    c = _rope_case(4, L, SPANS)
    pool, bt, lens, freed = _run(c)
    plain = _run(c, rope=False)
    np.testing.assert_array_equal(bt, plain[1])
    np.testing.assert_array_equal(lens, plain[2])
    assert freed == plain[3]
    Lp = int(lens[0])
    j = np.arange(Lp)
    pg, sl = bt[0, j // P], j % P
    # V rows and surrogate entries: the verbatim rollback's bytes
    np.testing.assert_array_equal(pool[:, pg, 1, :, sl, :], plain[0][:, pg, 1, :, sl, :])
    moved = {jj for (_, jj, r) in _moves(L, SPANS) if r > 0}
    same = np.array([x not in moved for x in j])
    np.testing.assert_array_equal(pool[:, pg[same], 0, :, sl[same], :], plain[0][:, pg[same], 0, :, sl[same], :])


def test_a_suffix_span_moves_and_rotates_nothing():
    """Decoding-time merges crop a suffix: no kept entry moves, no key rotates."""
    c = _rope_case(5, 64, [(61, 3)])
    pool, bt, lens, _ = _run(c)
    plain = _run(c, rope=False)
    np.testing.assert_array_equal(pool, plain[0])
