"""Pins of the oracle's aligned predictive distillation (App. F, Algorithm 1,
the masked distillation loss).

  * the paper's alignment example (tests/golden/distill_alignment_example.json);
  * the packed pairing equals the compressed-position map of App. J.4: a
    kept token t pairs with pi(t) = t - r(t) and a span's last position with
    its surrogate's index -- written here from the span list, not by masks;
  * with eps = 0 the loss is torch's soft-target cross-entropy (a library
    routine), and loss - H(P^T) is the mean KL divergence (>= 0, 0 when the
    student equals the teacher);
  * the closed-form gradient equals torch autograd of the loss with eps.
"""
import json
import os

import numpy as np
import pytest
import torch

from oracle.distill import align, soft_ce

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "distill_alignment_example.json")


def test_paper_alignment_example():
    with open(GOLDEN) as f:
        g = json.load(f)
    st = [s for s, _ in g["spans"]]
    ln = [n for _, n in g["spans"]]
    offs, tp, sp = align([g["L"]], [0, len(st)], st, ln)
    assert tp.tolist() == g["teacher_pos"] and sp.tolist() == g["student_pos"]
    tm = [int(j in set(tp.tolist())) for j in range(g["L"])]
    Lc = g["L"] - sum(n - 1 for n in ln)
    sm = [int(j in set(sp.tolist())) for j in range(Lc)]
    assert tm == g["teacher_mask"] and sm == g["student_mask"]


def _random_spans(r, L):
    st, ln, t = [], [], int(r.integers(0, 6))
    while t < L:
        n = int(r.integers(1, 5))
        if t + n > L:
            break
        if r.random() < 0.4:
            st.append(t)
            ln.append(n)
            t += n
        else:
            t += 1
    return st, ln


@pytest.mark.parametrize("seed", range(5))
def test_packed_pairs_follow_the_compressed_position_map(seed):
    r = np.random.default_rng(seed)
    lens, offs, st, ln = [], [0], [], []
    for b in range(6):
        L = int(r.integers(0, 90))
        s, n = _random_spans(r, L)
        lens.append(L)
        st += s
        ln += n
        offs.append(len(st))
    po, tp, sp = align(lens, offs, st, ln)
    for b in range(6):
        pairs = list(zip(tp[po[b]:po[b + 1]].tolist(), sp[po[b]:po[b + 1]].tolist()))
        spans = list(zip(st[offs[b]:offs[b + 1]], ln[offs[b]:offs[b + 1]]))
        if not spans:
            assert pairs == []
            continue
        want, removed, t = [], 0, 0
        for s, n in spans:
            want += [(u, u - removed) for u in range(t, s) if u >= spans[0][0]]
            want.append((s + n - 1, s - removed))          # the anchor pairs with the surrogate
            removed += n - 1
            t = s + n
        want += [(u, u - removed) for u in range(t, lens[b])]
        assert pairs == want


def _logits(seed, rows, V, scale=3.0):
    return np.random.default_rng(seed).normal(0, scale, size=(rows, V))


def test_loss_is_library_soft_cross_entropy_and_kl():
    T, S = _logits(1, 9, 50), _logits(2, 7, 50)
    tr, sr = np.array([0, 3, 4, 8]), np.array([1, 2, 5, 6])
    loss, _ = soft_ce(T, S, tr, sr, eps=0.0)
    pt = torch.softmax(torch.from_numpy(T[tr]), -1)
    want = torch.nn.functional.cross_entropy(torch.from_numpy(S[sr]), pt)
    assert abs(loss - float(want)) < 1e-12
    ent = float(-(pt * torch.log(pt)).sum(-1).mean())
    kl = float(torch.nn.functional.kl_div(torch.log_softmax(torch.from_numpy(S[sr]), -1), pt,
                                          reduction="batchmean"))
    assert abs((loss - ent) - kl) < 1e-12 and kl > 0
    same, _ = soft_ce(T, T, tr, tr, eps=0.0)
    assert abs(same - ent) < 1e-12


@pytest.mark.parametrize("eps", [0.0, 1e-8, 1e-3])
def test_gradient_matches_autograd(eps):
    T, S = _logits(3, 6, 40), _logits(4, 5, 40)
    tr, sr = np.array([0, 2, 5]), np.array([4, 1, 3])
    loss, grad = soft_ce(T, S, tr, sr, eps=eps)
    s = torch.from_numpy(S).requires_grad_(True)
    pt = torch.softmax(torch.from_numpy(T[tr]), -1)
    ls = -(pt * torch.log(torch.softmax(s[sr], -1) + eps)).sum(-1).mean()
    ls.backward()
    assert abs(ls.detach().item() - loss) < 1e-12
    np.testing.assert_allclose(grad, s.grad.numpy(), rtol=1e-9, atol=1e-14)
    assert np.all(grad[[0, 2]] == 0)   # rows in no pair


def test_no_spans_no_pairs_and_zero_loss():
    po, tp, sp = align([10, 0], [0, 0, 0], [], [])
    assert po.tolist() == [0, 0, 0] and len(tp) == 0 and len(sp) == 0
    loss, grad = soft_ce(np.zeros((2, 4)), np.zeros((2, 4)), tp, sp)
    assert loss == 0.0 and not grad.any()
