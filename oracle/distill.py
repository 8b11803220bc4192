"""Aligned predictive distillation of the oracle (test infrastructure only):
the training-side step of the method (App. F "Loss and Alignment Metric",
Algorithm 1 "Aligned Predictive Distillation", the masked distillation loss
equation).

Alignment.  For a sample with original length L and sorted, non-overlapping
merged spans (s_i, n_i):
  * the keep mask marks every retained token and, for each span, only its
    final position s_i + n_i - 1 (the surrogate is aligned with the span's
    last token); the span's other positions are inactive placeholders;
  * the teacher mask is the keep mask restricted to positions at or after
    the first span's start s_b (before it the two paths compute the same
    thing); N_b = its number of ones;
  * the compressed sequence has L~ = L - sum (n_i - 1) positions; the student
    mask drops its first L~ - N_b positions;
  * Pack keeps the marked positions in order, so the k-th teacher position
    pairs with the k-th student position.
A sample without spans contributes no pairs.

Loss.  With P^T = softmax(teacher logits), P^S = softmax(student logits) over
the whole vocabulary, over all N = sum_b N_b aligned pairs:
  L = -(1/N) sum_pairs sum_v P^T(v) log(P^S(v) + eps),
and its gradient with respect to the student logits s of a paired row
(differentiating log(P^S + eps) through the softmax):
  dL/ds_v = -(1/N) [ a_v - P^S(v) sum_u a_u ],  a_u = P^T(u) P^S(u) / (P^S(u) + eps).
Float64 throughout; the running maximum is subtracted before exp.
"""
import numpy as np


def align(lens, span_offsets, span_start, span_len):
    """Per sample b (original length lens[b], spans span_start/span_len over
    span_offsets[b] .. span_offsets[b+1]-1): the teacher positions (within
    the original sequence) and the student positions (within the compressed
    sequence) of its aligned pairs.  Returns (pair_offsets [B+1],
    teacher_pos [N], student_pos [N]) as int32 arrays."""
    offs, tpos, spos = [0], [], []
    for b in range(len(lens)):
        L = int(lens[b])
        lo, hi = int(span_offsets[b]), int(span_offsets[b + 1])
        if hi == lo:
            offs.append(len(tpos))
            continue
        keep = np.ones(L, bool)
        removed = 0
        for i in range(lo, hi):
            s, n = int(span_start[i]), int(span_len[i])
            keep[s:s + n - 1] = False          # placeholders; the last position stays as the anchor
            removed += n - 1
        first = int(span_start[lo])
        teacher = [j for j in range(L) if keep[j] and j >= first]
        N = len(teacher)
        Lc = L - removed
        student = list(range(Lc - N, Lc))
        tpos += teacher
        spos += student
        offs.append(len(tpos))
    i32 = lambda x: np.asarray(x, dtype=np.int32)
    return i32(offs), i32(tpos), i32(spos)


def _softmax(x):
    e = np.exp(x - x.max())
    return e / e.sum()


def soft_ce(teacher_logits, student_logits, teacher_rows, student_rows, eps=1e-8):
    """teacher_logits [R_T][V], student_logits [R_S][V] (float64 values);
    teacher_rows / student_rows [N]: the aligned pairs.  Returns (loss,
    grad [R_S][V]) with grad zero on rows that are not paired."""
    N = len(teacher_rows)
    grad = np.zeros(np.shape(student_logits))
    if N == 0:
        return 0.0, grad
    total = 0.0
    for t, s in zip(teacher_rows, student_rows):
        pt = _softmax(np.asarray(teacher_logits[t], dtype=np.float64))
        ps = _softmax(np.asarray(student_logits[s], dtype=np.float64))
        total += float(np.sum(pt * np.log(ps + eps)))
        a = pt * ps / (ps + eps)
        grad[s] += -(a - ps * a.sum()) / N
    return -total / N, grad
