"""Aligned predictive distillation on the GPU against the oracle (App. F
"Predictive Distillation Loss and Alignment Metrics", Algorithm 1, the masked
distillation loss).

Alignment: pair offsets, teacher rows, student rows and the compressed-row
prefix sums bit-exact on ragged samples (empty ones, samples without spans,
spans at both ends, n = 1 spans) and on the Llama-3.1-8B training shape
(8 x 512 tokens); invalid spans and a too-small capacity are rejected with
nothing written.

Soft-target cross-entropy: loss, per-pair losses and the gradient with respect
to the student logits within max-abs 1e-2 and relative L2 2e-3 of the float64
oracle, on vocabularies that do and do not fill the last 16-byte vector and on
peaky distributions where eps matters; at the full Llama-3 vocabulary (128256)
sampled pairs are checked one by one, and properties that hold at any size
(zero gradient on unpaired rows, each gradient row summing to zero, the loss
being the mean of the per-pair losses) on all rows.  Invalid pairs are rejected
with nothing written; results are bit-identical from call to call.
"""
import numpy as np
import pytest
import torch

import oracle
from oracle import distill as OD
import workloads as W
from helpers import dev, float_close, umim

pytestmark = pytest.mark.gpu


def _np(t):
    return t.detach().cpu().numpy()


def _oracle_rows(c):
    """The oracle's pairs as rows of the packed teacher / student batches."""
    lens = _np(c.seq_lens)
    offs, tp, sp = OD.align(lens, _np(c.span_offsets), _np(c.span_start), _np(c.span_len))
    so = _np(c.span_offsets)
    sl = _np(c.span_len)
    Lc = np.array([int(lens[b]) - int(np.sum(sl[so[b]:so[b + 1]] - 1)) for b in range(len(lens))], np.int64)
    t_cu = np.concatenate([[0], np.cumsum(lens.astype(np.int64))])
    s_cu = np.concatenate([[0], np.cumsum(Lc)])
    b_of = np.repeat(np.arange(len(lens)), np.diff(offs))
    return offs, (t_cu[b_of] + tp).astype(np.int32), (s_cu[b_of] + sp).astype(np.int32), s_cu.astype(np.int32)


def _gpu_align(m, c, dv, capacity=None, status=None):
    status = m.new_status(dv) if status is None else status
    cap = int(c.seq_lens.sum()) if capacity is None else capacity
    out = m.umim_distill_align(c.seq_lens.to(dv), c.span_offsets.to(dv), c.span_start.to(dv), c.span_len.to(dv),
                               cap, dev_status=status)
    torch.cuda.synchronize()
    return out, status


def _check_align(out, ref):
    offs, tr, sr, s_cu = ref
    n = int(offs[-1])
    np.testing.assert_array_equal(_np(out["pair_offsets"]), offs)
    np.testing.assert_array_equal(_np(out["teacher_rows"])[:n], tr)
    np.testing.assert_array_equal(_np(out["student_rows"])[:n], sr)
    np.testing.assert_array_equal(_np(out["student_cu"]), s_cu)


def test_align_paper_example():
    m, dv = umim(), dev()
    c = W.DistillCase(seq_lens=torch.tensor([6], dtype=torch.int32),
                      span_offsets=torch.tensor([0, 2], dtype=torch.int32),
                      span_start=torch.tensor([1, 4], dtype=torch.int32),
                      span_len=torch.tensor([2, 2], dtype=torch.int32), teacher_logits=None)
    out, st = _gpu_align(m, c, dv)
    m.check_status(st)
    # App. F example: pairs (x3, z23), (x4, x4), (x6, z56) -> teacher 2, 3, 5; student 1, 2, 3
    assert _np(out["teacher_rows"])[:3].tolist() == [2, 3, 5]
    assert _np(out["student_rows"])[:3].tolist() == [1, 2, 3]
    assert _np(out["pair_offsets"]).tolist() == [0, 3]


@pytest.mark.parametrize("seed", range(4))
def test_align_ragged(seed):
    m, dv = umim(), dev()
    r = W.rng(100 + seed)
    lens = [int(x) for x in r.integers(0, 300, size=9)] + [0, 1, 2, 5000]
    c = W.distill_case(200 + seed, lens=lens, vocab=8, coverage=float(r.uniform(0.0, 0.9)), kmin=1, kmax=4)
    out, st = _gpu_align(m, c, dv)
    m.check_status(st)
    _check_align(out, _oracle_rows(c))


def test_align_edge_layouts():
    m, dv = umim(), dev()
    # sample 0: span at 0 covering the whole sample; 1: no spans; 2: n = 1 spans only;
    # 3: span at the end; 4: empty sample
    lens = torch.tensor([4, 7, 5, 9, 0], dtype=torch.int32)
    st = torch.tensor([0, 1, 3, 6], dtype=torch.int32)
    ln = torch.tensor([4, 1, 1, 3], dtype=torch.int32)
    offs = torch.tensor([0, 1, 1, 3, 4, 4], dtype=torch.int32)
    c = W.DistillCase(seq_lens=lens, span_offsets=offs, span_start=st, span_len=ln, teacher_logits=None)
    out, s = _gpu_align(m, c, dv)
    m.check_status(s)
    _check_align(out, _oracle_rows(c))


def test_align_llama_training_shape():
    m, dv = umim(), dev()
    c = W.distill_case(W.SEEDS["distillation"], lens=[512] * 8, vocab=8, coverage=0.4)
    out, st = _gpu_align(m, c, dv)
    m.check_status(st)
    _check_align(out, _oracle_rows(c))


@pytest.mark.parametrize("bad", ["overlap", "past_end", "empty_span", "negative_len", "capacity"])
def test_align_rejects_invalid_input(bad):
    m, dv = umim(), dev()
    lens = torch.tensor([10, 12], dtype=torch.int32)
    st = torch.tensor([1, 5, 2], dtype=torch.int32)
    ln = torch.tensor([2, 3, 2], dtype=torch.int32)
    offs = torch.tensor([0, 2, 3], dtype=torch.int32)
    cap = 100
    if bad == "overlap":
        st[1] = 2
    elif bad == "past_end":
        st[2] = 11
    elif bad == "empty_span":
        ln[0] = 0
    elif bad == "negative_len":
        lens[1] = -1
    elif bad == "capacity":
        cap = 5
    c = W.DistillCase(seq_lens=lens, span_offsets=offs, span_start=st, span_len=ln, teacher_logits=None)
    i32 = lambda n: torch.full((n,), -7, dtype=torch.int32, device=dv)
    out = dict(pair_offsets=i32(3), teacher_rows=i32(100), student_rows=i32(100), student_cu=i32(3))
    status = m.new_status(dv)
    m.umim_distill_align(c.seq_lens.to(dv), c.span_offsets.to(dv), c.span_start.to(dv), c.span_len.to(dv), cap,
                         out=out, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 1
    for k, v in out.items():
        assert bool((v == -7).all()), f"{k} written"


# ---------------------------------------------------------------------------
# soft-target cross-entropy
# ---------------------------------------------------------------------------
def _case_with_student(seed, lens, V, dv, std=2.0, noise=None, coverage=0.4):
    """Teacher logits and pairs; student logits an independent draw, or with
    `noise` the paired teacher row plus N(0, noise^2) (a nearly trained module)."""
    c = W.distill_case(seed, lens=lens, vocab=V, coverage=coverage, std=std, device=dv)
    offs, tr, sr, s_cu = _oracle_rows(c)
    ld = c.teacher_logits.shape[1]
    stu = W.distill_logits(seed + 7, int(s_cu[-1]), ld, std, dv)
    if noise is not None and len(sr):
        g = torch.Generator(device=dv).manual_seed(seed + 9)
        t_rows = torch.from_numpy(tr).long().to(dv)
        s_rows = torch.from_numpy(sr).long().to(dv)
        x = c.teacher_logits[t_rows].float() + noise * torch.randn((len(sr), ld), generator=g, device=dv)
        stu[s_rows] = x.to(torch.bfloat16)
    return c, stu, tr, sr


def _gpu_ce(m, c, stu, tr, sr, dv, V, eps=1e-8, n_pairs=None, status=None, **kw):
    status = m.new_status(dv) if status is None else status
    t_rows = torch.from_numpy(np.ascontiguousarray(tr)).to(dv)
    s_rows = torch.from_numpy(np.ascontiguousarray(sr)).to(dv)
    loss, pl, grad = m.umim_distill_soft_ce(c.teacher_logits, stu, t_rows, s_rows, n_pairs=n_pairs, vocab=V,
                                            eps=eps, dev_status=status, **kw)
    torch.cuda.synchronize()
    return loss, pl, grad, status


def _f64(t, V):
    return t[:, :V].double().cpu().numpy()


@pytest.mark.parametrize("V,std,noise", [(1000, 2.0, None), (1001, 2.0, 0.3), (4096, 1.0, None),
                                         (32000, 3.0, 0.2), (50257, 2.0, None)])
def test_soft_ce_matches_oracle(V, std, noise):
    m, dv = umim(), dev()
    c, stu, tr, sr = _case_with_student(31 + V, [40, 0, 75, 23, 9], V, dv, std=std, noise=noise)
    loss, pl, grad, st = _gpu_ce(m, c, stu, tr, sr, dv, V)
    m.check_status(st)
    rl, rg = OD.soft_ce(_f64(c.teacher_logits, V), _f64(stu, V), tr, sr)
    float_close([loss.item()], [rl], "loss")
    rpl = [OD.soft_ce(_f64(c.teacher_logits[[int(t)]], V), _f64(stu[[int(s)]], V), [0], [0])[0]
           for t, s in zip(tr, sr)]
    float_close(_np(pl)[:len(tr)], rpl, "pair losses")
    float_close(_f64(grad, V), rg, "gradient")


@pytest.mark.parametrize("eps,std", [(0.0, 2.0), (1e-3, 2.0), (1e-8, 8.0), (1e-4, 8.0)])
def test_soft_ce_eps_and_peaky_distributions(eps, std):
    m, dv = umim(), dev()
    V = 2048
    c, stu, tr, sr = _case_with_student(77, [64, 48], V, dv, std=std)
    loss, pl, grad, st = _gpu_ce(m, c, stu, tr, sr, dv, V, eps=eps)
    m.check_status(st)
    rl, rg = OD.soft_ce(_f64(c.teacher_logits, V), _f64(stu, V), tr, sr, eps=eps)
    float_close([loss.item()], [rl], "loss")
    float_close(_f64(grad, V), rg, "gradient")


def test_soft_ce_llama3_vocabulary_training_batch():
    """8 x 512 tokens at 40 % coverage over the 128256-entry Llama-3 vocabulary,
    pairs from the GPU alignment (its pair count read on the device)."""
    m, dv = umim(), dev()
    V = W.LLAMA3_VOCAB
    c = W.distill_case(W.SEEDS["distillation"], lens=[512] * 8, vocab=V, coverage=0.4, device=dv)
    al, st = _gpu_align(m, c, dv)
    m.check_status(st)
    ref = _oracle_rows(c)
    _check_align(al, ref)
    offs, tr, sr, s_cu = ref
    N, R_S = int(offs[-1]), int(s_cu[-1])
    stu = W.distill_logits(W.SEEDS["distillation"] + 7, R_S, V, 2.0, dv)
    status = m.new_status(dv)
    loss, pl, grad = m.umim_distill_soft_ce(c.teacher_logits, stu, al["teacher_rows"], al["student_rows"],
                                            n_pairs=al["pair_offsets"][-1:], dev_status=status)
    torch.cuda.synchronize()
    m.check_status(status)
    pln = _np(pl)[:N].astype(np.float64)
    assert abs(loss.item() - pln.mean()) <= 1e-6 * abs(pln.mean())
    # sampled pairs against the oracle, one by one
    pick = sorted(set([0, N - 1] + [int(x) for x in W.rng(5).choice(N, size=14, replace=False)]))
    got_pl, want_pl, got_g, want_g = [], [], [], []
    for k in pick:
        l1, g1 = OD.soft_ce(_f64(c.teacher_logits[[int(tr[k])]], V), _f64(stu[[int(sr[k])]], V), [0], [0])
        got_pl.append(pln[k])
        want_pl.append(l1)
        got_g.append(_f64(grad[[int(sr[k])]], V)[0])
        want_g.append(g1[0] / N)
    float_close(got_pl, want_pl, "sampled pair losses")
    float_close(np.stack(got_g), np.stack(want_g), "sampled gradient rows")
    # any size: unpaired rows zero, each gradient row sums to zero
    paired = np.zeros(R_S, bool)
    paired[sr] = True
    g = grad.float()
    unp = torch.from_numpy(np.nonzero(~paired)[0]).to(dv)
    assert bool((g[unp] == 0).all())
    rs = g.sum(dim=1).abs()
    assert bool((rs <= 4e-3 * g.abs().sum(dim=1) + 1e-30).all())


def test_soft_ce_rejects_invalid_pairs():
    m, dv = umim(), dev()
    V = 512
    c, stu, tr, sr = _case_with_student(5, [30, 30], V, dv)
    for bad in ("dup_student", "teacher_range", "student_range", "n_pairs"):
        t2, s2, n_pairs = tr.copy(), sr.copy(), None
        if bad == "dup_student":
            s2[1] = s2[0]
        elif bad == "teacher_range":
            t2[2] = c.teacher_logits.shape[0]
        elif bad == "student_range":
            s2[0] = -1
        else:
            n_pairs = torch.tensor([len(tr) + 1], dtype=torch.int32, device=dv)
        grad = torch.full_like(stu, 3.0)
        loss = torch.full((1,), 5.0, device=dv)
        _, _, g, st = _gpu_ce(m, c, stu, t2, s2, dv, V, n_pairs=n_pairs, grad=grad, loss=loss)
        assert int(st.item()) == 1, bad
        assert bool((g == 3.0).all()) and loss.item() == 5.0, bad


def test_soft_ce_repeatable_padding_loss_only_and_fewer_pairs():
    m, dv = umim(), dev()
    V = 1001   # ld 1008: elements 1001..1007 are padding
    c, stu, tr, sr = _case_with_student(8, [50, 31], V, dv)
    pad = torch.full_like(stu, -9.0)
    l1, p1, g1, st = _gpu_ce(m, c, stu, tr, sr, dv, V, grad=pad)
    m.check_status(st)
    assert bool((g1[:, V:] == -9.0).all())
    l2, p2, g2, st = _gpu_ce(m, c, stu, tr, sr, dv, V)
    assert torch.equal(l1, l2) and torch.equal(p1, p2) and torch.equal(g1[:, :V], g2[:, :V])
    l3, _, g3, st = _gpu_ce(m, c, stu, tr, sr, dv, V, with_grad=False)
    assert g3 is None and torch.equal(l1, l3)
    # only the first n pairs count when n_pairs is given
    n = len(tr) // 2
    l4, p4, g4, st = _gpu_ce(m, c, stu, tr, sr, dv, V, n_pairs=torch.tensor([n], dtype=torch.int32, device=dv))
    m.check_status(st)
    rl, rg = OD.soft_ce(_f64(c.teacher_logits, V), _f64(stu, V), tr[:n], sr[:n])
    float_close([l4.item()], [rl], "loss over the first pairs")
    float_close(_f64(g4, V), rg, "gradient over the first pairs")


def test_soft_ce_no_pairs():
    m, dv = umim(), dev()
    V = 256
    c, stu, tr, sr = _case_with_student(9, [12, 7], V, dv, coverage=0.0)
    assert len(tr) == 0
    loss, _, grad, st = _gpu_ce(m, c, stu, tr, sr, dv, V)
    m.check_status(st)
    assert loss.item() == 0.0 and bool((grad[:, :V] == 0).all())
