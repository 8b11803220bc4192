"""Merge module M_phi of the oracle (test infrastructure only).

Follows App. C.1 ("Attention-based Pooling Architecture") step by step; the
main-text form is Sec. 3.2 Eq. 1, which App. C.1 extends with a GELU and a
LayerNorm on each side (App. C.3 counts both LayerNorms in |phi| = 2d^2 + 7d).

For one span s with n tokens and static embeddings E_s (n x d):
    P      = LN_kv(GELU(Linear_kv(E_s)))                  (n x d)
    P      = [P_1, ..., P_h],   P_i  (n x d_h),  d_h = d / h
    alpha_i = softmax(P_i q_i / sqrt(d_h))                (n)
    o_i    = alpha_i^T P_i                                 (d_h)
    z_s    = LN_o(GELU(Linear_o([o_1; ...; o_h])))         (d)

Readings where the paper is silent:
  * GELU is the exact erf form 0.5 x (1 + erf(x / sqrt(2))).
  * LayerNorm uses the biased variance, eps = 1e-5, elementwise affine
    (gamma, beta).
  * Linear(x) = W x + b with W stored [out][in].
  * Head i owns the contiguous columns [i d_h, (i+1) d_h) (the listing of
    App. C.6 views the last dimension as (heads, head_dim)).
Everything is float64; bf16 inputs are upcast exactly.
"""
import math

import numpy as np
from scipy.special import erf

from . import bf16

WEIGHT_NAMES = ("w_kv", "b_kv", "ln_kv_gamma", "ln_kv_beta", "query",
                "w_o", "b_o", "ln_o_gamma", "ln_o_beta")


def weights_f64(w_bits: dict) -> dict:
    """Upcast a dict of bf16 bit arrays (uint16) to float64 arrays."""
    return {k: bf16.to_f64(w_bits[k]) for k in WEIGHT_NAMES}


def gelu(x):
    return 0.5 * x * (1.0 + erf(x / math.sqrt(2.0)))


def layer_norm(x, gamma, beta, eps):
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * gamma + beta


def linear(x, w, b):
    return x @ w.T + b


def token_processor(E, w, eps):
    """P = LN_kv(GELU(Linear_kv(E)))  for a batch of token rows E (m x d)."""
    return layer_norm(gelu(linear(E, w["w_kv"], w["b_kv"])), w["ln_kv_gamma"], w["ln_kv_beta"], eps)


def attention_pool(P, q, n_heads):
    """alpha_i = softmax(P_i q_i / sqrt(d_h)),  o_i = alpha_i^T P_i,  o = [o_1;..;o_h]."""
    n, d = P.shape
    dh = d // n_heads
    o = np.empty(d)
    alphas = np.empty((n_heads, n))
    for i in range(n_heads):
        Pi = P[:, i * dh:(i + 1) * dh]
        s = Pi @ q[i] / math.sqrt(dh)
        e = np.exp(s - s.max())
        a = e / e.sum()
        alphas[i] = a
        o[i * dh:(i + 1) * dh] = a @ Pi
    return o, alphas


def output_processor(o, w, eps):
    """z = LN_o(GELU(Linear_o(o)))  for a batch of pooled rows o (m x d)."""
    return layer_norm(gelu(linear(o, w["w_o"], w["b_o"])), w["ln_o_gamma"], w["ln_o_beta"], eps)


def merge_span_reference_steps(E, w, n_heads, eps=1e-5):
    """One span, every intermediate returned: (P, alphas, o, z)."""
    P = token_processor(E, w, eps)
    o, alphas = attention_pool(P, w["query"], n_heads)
    z = output_processor(o[None, :], w, eps)[0]
    return P, alphas, o, z


def merge_spans(table_bits, token_ids, span_offsets, w, n_heads, eps=1e-5, which=None):
    """Surrogate embeddings z (float64, S x d) for the spans of a CSR list.

    table_bits   [V][d] uint16, bf16 embedding table e(.)
    token_ids    [T] span tokens, concatenated
    span_offsets [S+1] CSR offsets into token_ids
    w            dict of float64 weights (see ``weights_f64``)
    which        optional subset of span indices (returns rows in that order)
    """
    token_ids = np.asarray(token_ids)
    span_offsets = np.asarray(span_offsets)
    S = len(span_offsets) - 1
    idx = np.arange(S) if which is None else np.asarray(which)
    d = table_bits.shape[1]
    if len(idx) == 0:
        return np.zeros((0, d))
    # step 1: static embeddings of every token of the selected spans
    segs = [np.arange(span_offsets[i], span_offsets[i + 1]) for i in idx]
    tok_pos = np.concatenate(segs)
    if np.any(token_ids[tok_pos] < 0) or np.any(token_ids[tok_pos] >= table_bits.shape[0]):
        raise ValueError("token id out of range")
    E = bf16.to_f64(table_bits[token_ids[tok_pos]])
    # step 2: shared token projection (library matmul over all span tokens)
    P_all = token_processor(E, w, eps)
    # steps 3-4: per-span attention pooling with the learnable queries
    o = np.empty((len(idx), d))
    r = 0
    for j, seg in enumerate(segs):
        n = len(seg)
        o[j], _ = attention_pool(P_all[r:r + n], w["query"], n_heads)
        r += n
    # step 5: output processor
    return output_processor(o, w, eps)


def parameter_count(d: int, n_heads: int) -> int:
    """|phi| of App. C.3: Q (d) + two Linear (d^2 + d each) + two LayerNorm (2d each)."""
    q = n_heads * (d // n_heads)
    return q + 2 * (d * d + d) + 2 * (2 * d)
