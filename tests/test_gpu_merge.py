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
