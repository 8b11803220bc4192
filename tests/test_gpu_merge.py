"""Merge module on the GPU (tcgen05 GEMMs + pooling + LayerNorms) against the
float64 oracle, within max-abs 1e-2 and relative L2 2e-3."""
import numpy as np
import pytest
import torch

import oracle
from oracle import merge as M
import workloads as W
from helpers import dev, float_close, umim

pytestmark = pytest.mark.gpu


def _wf(w):
    return M.weights_f64({k: W.bits(v) for k, v in w.tensors().items()})


def _run(case):
    m = umim()
    d = dev()
    status = m.new_status(d)
    z = m.umim_merge_spans(case.table.to(d), case.token_ids.to(d), case.span_offsets.to(d),
                           case.weights.to(d), dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return z.cpu().double().numpy()


@pytest.mark.parametrize("seed,vocab,d,h,S,kmin,kmax", [
    (W.SEEDS["tiny"], 32000, 512, 4, 40, 2, 4),          # the tiny workload's merge module
    (21, 1000, 512, 4, 1, 1, 1),                         # one single-token span
    (22, 5000, 1024, 4, 129, 1, 4),                      # ragged M tiles in both GEMMs
    (23, 3000, 4096, 4, 97, 2, 4),                       # Llama-3-8B width, several M / all N tiles
    (24, 700, 2048, 8, 60, 1, 4),                        # 8 pooling heads
    (25, 700, 1536, 2, 33, 4, 4),                        # 2 heads, only 4-token spans
    (27, 700, 1536, 8, 21, 1, 4),                        # head width 192: 24 chunks, 3 column groups per head
    (28, 900, 4096, 2, 45, 1, 4),                        # head width 2048: the CTA-per-span pooling
    (29, 900, 2048, 1, 30, 2, 4),                        # one head over the whole width
    (30, 900, 512, 8, 50, 1, 4),                         # head width 64: 8 chunks per head
])
def test_merge_matches_oracle(seed, vocab, d, h, S, kmin, kmax):
    case = W.merge_case(seed, vocab=vocab, d=d, h=h, n_spans=S, kmin=kmin, kmax=kmax)
    z = _run(case)
    ref = oracle.merge_spans(W.bits(case.table), case.token_ids.numpy(), case.span_offsets.numpy(),
                             _wf(case.weights), h)
    float_close(z, ref)


def test_bad_token_id_is_flagged():
    m = umim()
    d = dev()
    case = W.merge_case(26, vocab=100, d=512, h=4, n_spans=5)
    ids = case.token_ids.clone()
    ids[3] = 100
    status = m.new_status(d)
    m.umim_merge_spans(case.table.to(d), ids.to(d), case.span_offsets.to(d), case.weights.to(d),
                       dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 1


def test_prompt_compression_sampled_spans():
    """Full prompt-compression workload: 64 prompts x 2048 tokens over a
    128256 x 4096 table, 40 % coverage; every span is merged on the GPU and a
    seeded sample of spans (plus all spans of prompts 0 and 63) is checked."""
    seed = W.SEEDS["prompt_compression"]
    d = dev()
    table = W.bf16_normal((128256, 4096), 0.02, seed + 101, d)
    pc = W.prompt_case(seed, B=64, L=2048, vocab=128256, d=4096, coverage=0.4, device=d, table=table)
    w = W.merge_weights(4096, 4, seed + 202, d)
    m = umim()
    status = m.new_status(d)
    z = m.umim_merge_spans(table, pc.span_token_ids, pc.span_token_offsets, w, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    S = pc.span_start.numel()
    offs = pc.span_offsets.cpu().numpy()
    r = W.rng(seed + 7)
    which = np.unique(np.concatenate([r.choice(S, 192, replace=False), np.arange(offs[0], offs[1]),
                                      np.arange(offs[63], offs[64])]))
    ids = pc.span_token_ids.cpu().numpy()
    toffs = pc.span_token_offsets.cpu().numpy()
    used = np.unique(ids[np.concatenate([np.arange(toffs[i], toffs[i + 1]) for i in which])])
    # only the rows the sample needs leave the GPU
    tb = np.zeros((128256, 4096), dtype=np.uint16)
    tb[used] = W.bits(table[torch.from_numpy(used).to(d)])
    wf = M.weights_f64({k: W.bits(v) for k, v in w.tensors().items()})
    ref = oracle.merge_spans(tb, ids, toffs, wf, 4, which=which)
    float_close(z[torch.from_numpy(which).to(d)].cpu().double().numpy(), ref)


# ---------------------------------------------------------------------------
# fp16 intermediates: values past fp16's range are refused, tiny W_o entries kept
# ---------------------------------------------------------------------------
def _weights_with(case, **over):
    w = case.weights
    kw = {k: v.clone() for k, v in w.tensors().items()}
    kw.update(over)
    return W.MergeWeights(w.d_model, w.n_heads, ln_eps=w.ln_eps, **kw)


def _refused_with_nothing_written(case, weights, table=None):
    m = umim()
    d = dev()
    S = case.span_offsets.numel() - 1
    status = m.new_status(d)
    sentinel = torch.full((S, case.weights.d_model), 12345.0, dtype=torch.float32, device=d)
    z = m.umim_merge_spans((case.table if table is None else table).to(d), case.token_ids.to(d),
                           case.span_offsets.to(d), weights.to(d), surrogates=sentinel.clone(), dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 2   # UMIM_ERR_UNSUPPORTED
    assert torch.equal(z, sentinel), "a refused call must leave the surrogates untouched"


def test_hidden_activation_past_fp16_range_is_refused():
    """A bias of 70000 on one column makes GELU(E W_kv^T + b_kv) exceed fp16's
    65504 in the first projection's output."""
    case = W.merge_case(61, vocab=300, d=512, h=4, n_spans=9)
    b = case.weights.b_kv.clone()
    b[7] = 70000.0
    _refused_with_nothing_written(case, _weights_with(case, b_kv=b))


def test_large_embeddings_past_fp16_range_are_refused():
    case = W.merge_case(62, vocab=300, d=1024, h=4, n_spans=9)
    table = case.table.clone()
    table[case.token_ids[0]] = 3.0e6   # one span token's row: |E W^T| far past fp16
    _refused_with_nothing_written(case, case.weights, table=table)


def test_output_projection_weight_past_the_scaled_range_is_refused():
    """W_o is staged in fp16 times 256: an entry of 300 does not fit."""
    case = W.merge_case(63, vocab=300, d=512, h=4, n_spans=9)
    wo = case.weights.w_o.clone()
    wo[3, 5] = 300.0
    _refused_with_nothing_written(case, _weights_with(case, w_o=wo))


@pytest.mark.parametrize("scale", [1e-3, 2e-5, 1e-6])
def test_tiny_output_projection_weights_keep_their_precision(scale):
    """W_o and b_o scaled down so far that every entry would be an fp16
    subnormal (below 6.1e-5) without the power-of-two staging: the surrogates
    still match the oracle."""
    case = W.merge_case(64, vocab=2000, d=1024, h=4, n_spans=70, kmin=1, kmax=4)
    wo = (case.weights.w_o.float() * scale).to(torch.bfloat16)
    bo = (case.weights.b_o.float() * scale).to(torch.bfloat16)
    wt = _weights_with(case, w_o=wo, b_o=bo)
    case2 = W.MergeCase(table=case.table, token_ids=case.token_ids, span_offsets=case.span_offsets, weights=wt)
    z = _run(case2)
    ref = oracle.merge_spans(W.bits(case.table), case.token_ids.numpy(), case.span_offsets.numpy(), _wf(wt), 4)
    float_close(z, ref, f"W_o scaled by {scale}")
