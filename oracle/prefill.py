"""Prefill attention over packed compressed prompts, oracle (test
infrastructure only).

App. E ("Prompt Merging") and App. C.5: the compressed embeddings, with
contiguous positions, are passed to the frozen backbone for prefill, so the
backbone's causal self-attention runs over the shorter sequences.  The packed
form is the one umim_build_compressed produces: the sequences' rows
concatenated, sequence b owning rows cu_seqlens[b] .. cu_seqlens[b+1]-1.

Per sequence, with rows i, j counted inside it, this is the standard
grouped-query causal attention of a Llama-style decoder:

  out[i, h] = sum_{j <= i} softmax_j(scale * <q[i, h], k[j, g]>) v[j, g]
  g = floor(h / G),  G = Hq / Hkv,  scale = 1 / sqrt(D) unless given.

No sliding window, softcap or ALiBi; rotary embeddings are already applied to
q and k by the caller.  Float64 from the exact bf16 inputs, the running
maximum subtracted before exp.
"""
import math

import numpy as np

from . import bf16


def prefill_attention(q_bits, k_bits, v_bits, cu_seqlens, scale=None, rows=None):
    """q_bits [T][Hq][D], k_bits / v_bits [T][Hkv][D] uint16 (bf16 bits);
    cu_seqlens [B+1].  Returns out [T][Hq][D] float64 (rows outside every
    sequence stay 0).  rows: optional list of global row indices to compute
    (the others stay 0)."""
    q, k, v = bf16.to_f64(q_bits), bf16.to_f64(k_bits), bf16.to_f64(v_bits)
    T, Hq, D = q.shape
    Hkv = k.shape[1]
    if Hq % Hkv:
        raise ValueError("Hq must be a multiple of Hkv")
    G = Hq // Hkv
    if scale is None or scale == 0:
        scale = 1.0 / math.sqrt(D)
    cu = np.asarray(cu_seqlens)
    if cu[0] != 0 or np.any(np.diff(cu) < 0) or cu[-1] > T:
        raise ValueError("cu_seqlens")
    want = None if rows is None else set(int(r) for r in rows)
    out = np.zeros((T, Hq, D))
    for b in range(len(cu) - 1):
        lo, hi = int(cu[b]), int(cu[b + 1])
        for i in range(lo, hi):
            if want is not None and i not in want:
                continue
            for h in range(Hq):
                g = h // G
                s = (k[lo:i + 1, g, :] @ q[i, h]) * scale
                e = np.exp(s - s.max())
                out[i, h] = (e / e.sum()) @ v[lo:i + 1, g, :]
    return out
