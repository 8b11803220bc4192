"""Position-aware rollback on the GPU against the oracle (App. J.4 compressed
positions; moved keys re-rotated by -r(t) w_m on the half-split RoPE pairs).

Bit-exact: block tables, lengths, freed pages, V rows, surrogate entries,
entries that do not move and key columns past rotary_dim.  Re-rotated keys:
the GPU computes the rotation in fp32 (angle with its exact rounding error
folded in), the oracle in float64; both round to bf16, so a key element may
differ by one bf16 ulp where the exact value lies next to a rounding
boundary, which must be rare; where the rotated value nearly cancels, the
fp32 rounding of the two products (a few fp32 ulps of the pair's magnitude)
bounds the difference instead."""
import numpy as np
import pytest
import torch

import oracle
from oracle import bf16
import workloads as W
from helpers import dev, umim

pytestmark = pytest.mark.gpu


def _inv_freq(rd, base=500000.0):
    return (base ** (-np.arange(0, rd, 2, dtype=np.float64) / rd)).astype(np.float32)


@pytest.mark.parametrize("seed,lens,hkv,D,layers,rd,coverage", [
    (71, [512], 2, 64, 1, 64, 0.4),                       # the tiny workload's shape
    (72, [700, 33, 4096, 1], 8, 128, 1, 128, 0.3),        # Llama-8B-layer shape, ragged lengths
    (73, [300, 999, 17], 4, 128, 3, 64, 0.5),             # partial rotary dim, several layers
    (74, [2500, 2600], 4, 128, 2, 128, 0.6),              # long shifts (r in the hundreds)
])
def test_rope_rollback_matches_oracle(seed, lens, hkv, D, layers, rd, coverage):
    m, dv = umim(), dev()
    c = W.decode_case(seed, lens=lens, n_q_heads=hkv, n_kv_heads=hkv, head_dim=D, n_layers=layers,
                      coverage=coverage)
    w = _inv_freq(rd)
    pool, bt, sl = c.pool.to(dv), c.block_table.to(dv), c.seq_lens.to(dv)
    status = m.new_status(dv)
    freed = m.umim_kv_rollback(pool, bt, sl, c.span_offsets.to(dv), c.span_start.to(dv), c.span_len.to(dv),
                               c.surrogate_k.to(dv), c.surrogate_v.to(dv), dev_status=status,
                               rope_inv_freq=torch.from_numpy(w).to(dv), rotary_dim=rd)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    rp, rbt, rl, rfreed = oracle.kv_rollback(W.bits(c.pool), c.block_table.numpy(), c.seq_lens.numpy(),
                                              c.span_offsets.numpy(), c.span_start.numpy(), c.span_len.numpy(),
                                              W.bits(c.surrogate_k), W.bits(c.surrogate_v), rope_inv_freq=w,
                                              rotary_dim=rd)
    np.testing.assert_array_equal(bt.cpu().numpy(), rbt)
    np.testing.assert_array_equal(sl.cpu().numpy(), rl)
    f = freed.cpu().numpy()
    assert f[:len(rfreed)].tolist() == list(rfreed)
    gp = W.bits(pool)
    n_diff = n_rot = 0
    for b in range(len(lens)):
        t = np.arange(int(rl[b]))
        pg, slot = rbt[b, t // 16], t % 16
        g = gp[:, pg, :, :, slot, :]            # [layers][L'][2][Hkv][D] after fancy indexing: [L'][layers][2][Hkv][D]
        o = rp[:, pg, :, :, slot, :]
        np.testing.assert_array_equal(g[..., 1, :, :], o[..., 1, :, :], err_msg=f"V seq {b}")
        np.testing.assert_array_equal(g[..., 0, :, rd:], o[..., 0, :, rd:], err_msg=f"K past rotary_dim seq {b}")
        gk, ok = bf16.to_f64(g[..., 0, :, :rd]), bf16.to_f64(o[..., 0, :, :rd])
        # one bf16 ulp of the result, or the fp32 error of a rotation near cancellation (x c + y s
        # close to 0): a few fp32 ulps of the pair's magnitude
        pair = np.sqrt(ok[..., :rd // 2] ** 2 + ok[..., rd // 2:] ** 2)
        pair = np.concatenate([pair, pair], axis=-1)
        assert np.all(np.abs(gk - ok) <= np.maximum(2.0 ** -7 * np.abs(ok), 2.0 ** -20 * pair) + 1e-38), \
            f"K seq {b}: more than one bf16 ulp"
        same = g[..., 0, :, :rd] == o[..., 0, :, :rd]
        n_diff += int((~same).sum())
        n_rot += same.size
    assert n_diff <= max(8, 1e-3 * n_rot), (n_diff, n_rot)


def test_rope_rollback_rejects_a_bad_rotary_dim():
    m, dv = umim(), dev()
    c = W.decode_case(75, lens=[64], n_q_heads=2, n_kv_heads=2, head_dim=64, coverage=0.3)
    w = torch.from_numpy(_inv_freq(64)).to(dv)
    for rd in (0, 24, 80):
        with pytest.raises(m.UmimError):
            m.umim_kv_rollback(c.pool.to(dv), c.block_table.to(dv), c.seq_lens.to(dv), c.span_offsets.to(dv),
                               c.span_start.to(dv), c.span_len.to(dv), c.surrogate_k.to(dv), c.surrogate_v.to(dv),
                               rope_inv_freq=w, rotary_dim=rd)
