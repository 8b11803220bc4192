"""Prefill attention over packed compressed prompts on the GPU against the
oracle (App. E "Prompt Merging", App. C.5): causal grouped-query attention
within each sequence, within max-abs 1e-2 and relative L2 2e-3."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from helpers import dev, float_close, umim

pytestmark = pytest.mark.gpu


def _qkv(seed, T, hq, hkv, d, dv):
    return (W.bf16_normal((T, hq, d), 1.0, seed, dv), W.bf16_normal((T, hkv, d), 1.0, seed + 1, dv),
            W.bf16_normal((T, hkv, d), 1.0, seed + 2, dv))


@pytest.mark.parametrize("seed,lens,hq,hkv,d,pad", [
    (81, [1, 63, 64, 65, 200, 0, 130], 32, 8, 128, 0),   # tile edges, an empty sequence
    (82, [17, 129, 300], 8, 2, 64, 5),                  # head_dim 64, unused rows past the last sequence
    (83, [1000], 4, 4, 128, 0),                          # one long sequence, G = 1
    (84, [5, 77, 3, 250], 28, 4, 128, 0),                # G = 7 (the long-context model)
    # 32 query tiles x 32 heads = 1024 work units over 2 CTAs per SM: every CTA runs
    # several units, so barriers and rings count across units (checked on every row)
    (85, [1000, 1000, 700, 513, 300, 65, 1], 32, 8, 128, 0),
])
def test_prefill_matches_oracle(seed, lens, hq, hkv, d, pad):
    m, dv = umim(), dev()
    T = sum(lens) + pad
    q, k, v = _qkv(seed, T, hq, hkv, d, dv)
    cu = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int32, device=dv)
    out = torch.full_like(q, 7.0)
    status = m.new_status(dv)
    m.umim_prefill_attention(q, k, v, cu, out=out, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    want = oracle.prefill_attention(W.bits(q), W.bits(k), W.bits(v), cu.cpu().numpy())
    got = out.cpu().double().numpy()
    n = sum(lens)
    float_close(got[:n], want[:n], "prefill")
    assert np.all(got[n:] == 7.0)   # rows outside every sequence are left alone


def test_prefill_over_compressed_prompts_sampled():
    """64 prompts of 2048 tokens compressed at 40 % coverage (about 1500 rows
    each), Llama-3-8B attention (32/8 heads, head_dim 128); sampled rows,
    the first and last of every prompt among them."""
    m, dv = umim(), dev()
    pc = W.prompt_case(W.SEEDS["prompt_compression"], B=64, L=2048, vocab=128256, d=8, coverage=0.4)
    offs, ln = pc.span_offsets.numpy(), pc.span_len.numpy()
    lens = [2048 - int((ln[offs[b]:offs[b + 1]] - 1).sum()) for b in range(64)]
    T = sum(lens)
    q, k, v = _qkv(91, T, 32, 8, 128, dv)
    cu_np = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    cu = torch.from_numpy(cu_np).to(dv)
    status = m.new_status(dv)
    out = m.umim_prefill_attention(q, k, v, cu, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    r = W.rng(92)
    rows = sorted(set(cu_np[:-1].tolist()) | set((cu_np[1:] - 1).tolist()) |
                  set(r.integers(0, T, 64).tolist()))
    want = oracle.prefill_attention(W.bits(q), W.bits(k), W.bits(v), cu_np, rows=rows)
    got = out.cpu().double().numpy()
    float_close(got[rows], want[rows], "prefill sampled rows")


def test_bad_offsets_write_nothing():
    m, dv = umim(), dev()
    q, k, v = _qkv(93, 40, 4, 2, 64, dv)
    for bad in ([1, 20, 40], [0, 30, 20], [0, 20, 41]):
        out = torch.full_like(q, 3.0)
        status = m.new_status(dv)
        m.umim_prefill_attention(q, k, v, torch.tensor(bad, dtype=torch.int32, device=dv), out=out,
                                 dev_status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 1
        assert torch.all(out == 3.0)
