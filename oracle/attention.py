"""Decode attention over the compacted paged cache, oracle (test infrastructure only).

After rollback the frozen backbone attends over the shorter cache in the usual
way (App. I.1: every decode step attends over whatever KV entries the cache
holds at that point; App. E: the surrogate's KV state is one ordinary cache
entry).  The paper gives no
formula of its own, so this is the standard grouped-query scaled dot-product
attention of a Llama-style decoder for one new query token:

  out[b, h] = sum_{j < L'_b} softmax_j(scale * <q[b, h], K[b, g, j]>) V[b, g, j]
  g = floor(h / G),  G = Hq / Hkv  (query heads h = gG .. gG+G-1 share KV head g)
  scale = 1 / sqrt(D) unless given.

Readings: no causal mask is needed (one query sees every cached entry), no
softcap, window or ALiBi.  An empty cache (L' = 0) gives a zero output.
Float64 throughout with the running maximum subtracted before exp.
"""
import math

import numpy as np

from . import bf16


def attend(q, K, V, scale):
    """Plain softmax attention of one query vector over K, V ([L][D])."""
    if K.shape[0] == 0:
        return np.zeros(V.shape[-1]), np.zeros(0)
    s = (K @ q) * scale
    e = np.exp(s - s.max())
    w = e / e.sum()
    return w @ V, w


def decode_attention(q_bits, pool_bits, layer, block_table, seq_lens, scale=None,
                     page_size=16, return_weights=False):
    """q_bits [B][Hq][D] uint16, pool_bits [layers][pages][2][Hkv][P][D] uint16.
    Returns out [B][Hq][D] float64 (and the softmax weights if asked)."""
    q = bf16.to_f64(q_bits)
    B, Hq, D = q.shape
    Hkv = pool_bits.shape[3]
    if Hq % Hkv:
        raise ValueError("Hq must be a multiple of Hkv")
    G = Hq // Hkv
    if scale is None or scale == 0:
        scale = 1.0 / math.sqrt(D)
    out = np.zeros((B, Hq, D))
    weights = []
    for b in range(B):
        L = int(seq_lens[b])
        t = np.arange(L)
        pages = np.asarray(block_table)[b, t // page_size]
        slots = t % page_size
        # only the pages this sequence uses are upcast
        K = bf16.to_f64(pool_bits[layer, pages, 0, :, slots, :])   # [L][Hkv][D]
        V = bf16.to_f64(pool_bits[layer, pages, 1, :, slots, :])
        wb = []
        for h in range(Hq):
            g = h // G
            out[b, h], w = attend(q[b, h], K[:, g, :], V[:, g, :], scale)
            wb.append(w)
        weights.append(wb)
    if return_weights:
        return out, weights
    return out
