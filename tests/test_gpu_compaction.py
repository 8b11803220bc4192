"""Compressed prompt construction on the GPU against the oracle: bit-exact
embedding rows, position ids and cu_seqlens."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from helpers import dev, umim

pytestmark = pytest.mark.gpu


def _run(pc, z, capacity=None):
    m = umim()
    d = dev()
    B, L = pc.token_ids.shape
    status = m.new_status(d)
    out = None if capacity is None else torch.empty((capacity, pc.table.shape[1]), dtype=torch.bfloat16, device=d)
    emb, pos, cu = m.umim_build_compressed(pc.table.to(d), pc.token_ids.to(d), pc.span_offsets.to(d),
                                           pc.span_start.to(d), pc.span_len.to(d), z.to(d), out_embeds=out,
                                           dev_status=status)
    torch.cuda.synchronize()
    return emb, pos, cu, int(status.item())


@pytest.mark.parametrize("seed,B,L,d,cov", [(1, 1, 4, 512, 0.5), (2, 3, 100, 512, 0.4), (3, 5, 333, 1024, 0.7),
                                            (4, 2, 64, 512, 0.0), (5, 4, 17, 4096, 1.0)])
def test_compaction_matches_oracle(seed, B, L, d, cov):
    pc = W.prompt_case(seed, B=B, L=L, vocab=999, d=d, coverage=cov)
    z = torch.randn(pc.span_start.numel(), d, generator=torch.Generator().manual_seed(seed))
    emb, pos, cu, st = _run(pc, z)
    assert st == 0
    re, rpos, rcu = oracle.build_compressed(W.bits(pc.table), pc.token_ids.numpy(), pc.span_offsets.numpy(),
                                            pc.span_start.numpy(), pc.span_len.numpy(), z.numpy())
    n = int(rcu[-1])
    np.testing.assert_array_equal(cu.cpu().numpy(), rcu)
    np.testing.assert_array_equal(pos[:n].cpu().numpy(), rpos)
    np.testing.assert_array_equal(W.bits(emb[:n].cpu()), re)


def test_rounding_ties_of_surrogates():
    """Surrogate values exactly halfway between two bf16 numbers round to even."""
    pc = W.prompt_case(6, B=1, L=8, vocab=50, d=512, coverage=0.5)
    S = pc.span_start.numel()
    u = torch.randint(0, 2 ** 15, (S, 512), generator=torch.Generator().manual_seed(0), dtype=torch.int32)
    z = ((u << 16) | 0x8000).view(torch.float32)
    z = torch.where(torch.isfinite(z), z, torch.zeros_like(z))
    emb, pos, cu, st = _run(pc, z)
    assert st == 0
    re, rpos, rcu = oracle.build_compressed(W.bits(pc.table), pc.token_ids.numpy(), pc.span_offsets.numpy(),
                                            pc.span_start.numpy(), pc.span_len.numpy(), z.numpy())
    np.testing.assert_array_equal(W.bits(emb[:int(rcu[-1])].cpu()), re)


def test_capacity_too_small_writes_nothing():
    pc = W.prompt_case(7, B=2, L=50, vocab=100, d=512, coverage=0.2)
    z = torch.zeros(pc.span_start.numel(), 512)
    emb, pos, cu, st = _run(pc, z, capacity=10)
    assert st == 1


def test_prompt_compression_full_size():
    """64 x 2048 prompts, 128256 x 4096 table, 40 % coverage: position ids
    and cu_seqlens of all 64 prompts compared with the oracle, embedding rows
    of prompts 0, 31 and 63 compared."""
    seed = W.SEEDS["prompt_compression"]
    d = dev()
    table = W.bf16_normal((128256, 4096), 0.02, seed + 101, d)
    pc = W.prompt_case(seed, B=64, L=2048, vocab=128256, d=4096, coverage=0.4, device=d, table=table)
    z = torch.randn(pc.span_start.numel(), 4096, generator=torch.Generator(device=d).manual_seed(3), device=d)
    m = umim()
    status = m.new_status(d)
    emb, pos, cu = m.umim_build_compressed(table, pc.token_ids, pc.span_offsets, pc.span_start, pc.span_len, z,
                                           dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ids = pc.token_ids.cpu().numpy()
    offs = pc.span_offsets.cpu().numpy()
    st_, ln_ = pc.span_start.cpu().numpy(), pc.span_len.cpu().numpy()
    cu_h = cu.cpu().numpy()
    for b in (0, 31, 63):
        used = np.unique(ids[b])
        tb = np.zeros((128256, 4096), dtype=np.uint16)
        tb[used] = W.bits(table[torch.from_numpy(used).to(d)])
        lo, hi = offs[b], offs[b + 1]
        re, rpos, rcu = oracle.build_compressed(tb, ids[b:b + 1], np.array([0, hi - lo]), st_[lo:hi], ln_[lo:hi],
                                                z[lo:hi].cpu().numpy())
        assert cu_h[b + 1] - cu_h[b] == rcu[-1]
        np.testing.assert_array_equal(pos[cu_h[b]:cu_h[b + 1]].cpu().numpy(), rpos)
        np.testing.assert_array_equal(W.bits(emb[cu_h[b]:cu_h[b + 1]].cpu()), re)
    # position ids and cu_seqlens of every prompt: they do not depend on the
    # embedding width, so the oracle runs on a one-column table
    narrow = np.zeros((128256, 1), dtype=np.uint16)
    _, rpos_all, rcu_all = oracle.build_compressed(narrow, ids, offs, st_, ln_,
                                                   np.zeros((len(st_), 1), np.float32))
    np.testing.assert_array_equal(cu_h, rcu_all)
    np.testing.assert_array_equal(pos[:cu_h[-1]].cpu().numpy(), rpos_all)
    for b in range(64):
        lo, hi = offs[b], offs[b + 1]
        assert cu_h[b + 1] - cu_h[b] == 2048 - int((ln_[lo:hi] - 1).sum())
