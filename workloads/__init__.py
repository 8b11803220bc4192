"""Seeded synthetic inputs for the UMIM decode step over a merged context.

This module only draws random numbers and does the bookkeeping a paged-cache
allocator would do (which physical page holds which logical page).  It holds
none of the method's arithmetic: no merge module, no rollback, no attention.
Both the CUDA path (through its binding) and the CPU oracle consume exactly
the tensors produced here, so a parity test compares like with like.

Shapes follow the workloads the paper evaluates (Llama-3-8B / 3.1-8B-shaped
layers, span lengths n in {2,3,4} from the merge rule of Sec. 3.1, 30-40 %
token coverage matching the reported token reduction, App. I.1 decode
setting).  The paper's corpora (WikiText-103 and others) are not available, so
uniform token ids and N(0, sigma^2) embeddings / KV entries stand in for them.

Randomness:
  * integer structure (token ids, span placement, page permutation, lengths)
    comes from numpy's PCG64 seeded per workload, so it is identical on any
    host;
  * bulk bf16 tensors (embedding tables, KV pools, q) come from a seeded
    ``torch.Generator`` on the device that will hold them (float32 normal,
    then rounded to bf16 by torch).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional, Sequence

import numpy as np
import torch

PAGE_SIZE = 16

# Seeds: one per named workload, 0x5EED000n.
SEEDS = {
    "tiny": 0x5EED0001,
    "llama8b_layer": 0x5EED0002,
    "prompt_compression": 0x5EED0003,
    "long_context": 0x5EED0004,
    "long_context_tr40": 0x5EED0014,
    "serving": 0x5EED0005,
    "rule_matching": 0x5EED0006,
    "distillation": 0x5EED0007,
}

# Retained merge rules per n-gram length for the Llama-3 tokenizer (the paper's
# table of rule counts, frequency threshold 5): 2-, 3- and 4-grams.
LLAMA3_RULE_COUNTS = (216_700, 684_793, 1_266_080)
LLAMA3_VOCAB = 128_256


def rng(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed))


def torch_gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


# ----------------------------------------------------------------------------
# span placement
# ----------------------------------------------------------------------------
def span_layout(r: np.random.Generator, L: int, *, n_spans: Optional[int] = None,
                coverage: Optional[float] = None, kmin: int = 2, kmax: int = 4):
    """Sorted, non-overlapping spans inside [0, L).

    Lengths are drawn uniformly from {kmin..kmax}, either exactly ``n_spans``
    of them or until they cover ``round(coverage * L)`` positions.  The L - sum(k)
    free positions are spread over the S+1 gaps by a uniform random
    composition (stars and bars).  Returns (start[S], length[S]) int32.
    """
    lens = []
    if n_spans is not None:
        lens = list(r.integers(kmin, kmax + 1, size=n_spans))
    else:
        target = int(round(coverage * L))
        tot = 0
        while tot < target:
            k = int(r.integers(kmin, kmax + 1))
            if tot + k > L:
                break
            lens.append(k)
            tot += k
    lens = np.asarray(lens, dtype=np.int64)
    S = len(lens)
    free = L - int(lens.sum())
    if free < 0:
        raise ValueError("spans do not fit")
    if S == 0:
        return np.zeros(0, np.int32), np.zeros(0, np.int32)
    # stars and bars: choose S bar positions among free + S slots
    bars = np.sort(r.choice(free + S, size=S, replace=False))
    gaps_before = bars - np.arange(S)          # free positions before span i (cumulative)
    starts = gaps_before + np.concatenate([[0], np.cumsum(lens)[:-1]])
    return starts.astype(np.int32), lens.astype(np.int32)


def suffix_span(r: np.random.Generator, L: int, kmin: int = 2, kmax: int = 4):
    k = int(r.integers(kmin, kmax + 1))
    k = min(k, L)
    return L - k, k


# ----------------------------------------------------------------------------
# bulk bf16 tensors
# ----------------------------------------------------------------------------
def bf16_normal(shape, std: float, seed: int, device="cpu") -> torch.Tensor:
    g = torch_gen(seed, device)
    # chunked so that very large tensors never need a full float32 copy
    out = torch.empty(shape, dtype=torch.bfloat16, device=device)
    of = out.view(-1)
    step = 1 << 26
    for i in range(0, of.numel(), step):
        j = min(of.numel(), i + step)
        of[i:j] = torch.randn(j - i, generator=g, device=device, dtype=torch.float32).mul_(std)
    return out


def bf16_uniform(shape, lo: float, hi: float, seed: int, device="cpu") -> torch.Tensor:
    g = torch_gen(seed, device)
    x = torch.rand(shape, generator=g, device=device, dtype=torch.float32)
    return (x * (hi - lo) + lo).to(torch.bfloat16)


def bits(t: torch.Tensor) -> np.ndarray:
    """Raw bf16 bit patterns of a bf16 tensor as a numpy uint16 array."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


# ----------------------------------------------------------------------------
# merge-module weights (random init; the trained checkpoints are not public)
# ----------------------------------------------------------------------------
@dataclasses.dataclass
class MergeWeights:
    d_model: int
    n_heads: int
    w_kv: torch.Tensor      # [d][d]  W[out][in]
    b_kv: torch.Tensor      # [d]
    ln_kv_gamma: torch.Tensor
    ln_kv_beta: torch.Tensor
    query: torch.Tensor     # [h][d/h]
    w_o: torch.Tensor       # [d][d]
    b_o: torch.Tensor
    ln_o_gamma: torch.Tensor
    ln_o_beta: torch.Tensor
    ln_eps: float = 1e-5

    def tensors(self):
        return dict(w_kv=self.w_kv, b_kv=self.b_kv, ln_kv_gamma=self.ln_kv_gamma,
                    ln_kv_beta=self.ln_kv_beta, query=self.query, w_o=self.w_o,
                    b_o=self.b_o, ln_o_gamma=self.ln_o_gamma, ln_o_beta=self.ln_o_beta)

    def to(self, device):
        kw = {k: v.to(device) for k, v in self.tensors().items()}
        return MergeWeights(self.d_model, self.n_heads, ln_eps=self.ln_eps, **kw)


def merge_weights(d: int, h: int, seed: int, device="cpu") -> MergeWeights:
    """Linear weights/biases ~ U(-1/sqrt(d), 1/sqrt(d)) (the usual Linear init),
    q ~ N(0,1), LayerNorm gamma = 1 + U(-0.1,0.1), beta ~ U(-0.1,0.1); all bf16."""
    a = 1.0 / math.sqrt(d)
    s = seed * 16
    return MergeWeights(
        d_model=d, n_heads=h,
        w_kv=bf16_uniform((d, d), -a, a, s + 1, device),
        b_kv=bf16_uniform((d,), -a, a, s + 2, device),
        ln_kv_gamma=bf16_uniform((d,), 0.9, 1.1, s + 3, device),
        ln_kv_beta=bf16_uniform((d,), -0.1, 0.1, s + 4, device),
        query=bf16_normal((h, d // h), 1.0, s + 5, device),
        w_o=bf16_uniform((d, d), -a, a, s + 6, device),
        b_o=bf16_uniform((d,), -a, a, s + 7, device),
        ln_o_gamma=bf16_uniform((d,), 0.9, 1.1, s + 8, device),
        ln_o_beta=bf16_uniform((d,), -0.1, 0.1, s + 9, device),
    )


# ----------------------------------------------------------------------------
# span tokens for the merge module
# ----------------------------------------------------------------------------
@dataclasses.dataclass
class MergeCase:
    table: torch.Tensor          # [V][d] bf16
    token_ids: torch.Tensor      # [T] int32, span tokens concatenated
    span_offsets: torch.Tensor   # [S+1] int32
    weights: MergeWeights


def merge_case(seed: int, *, vocab: int, d: int, h: int = 4, n_spans: int,
               kmin: int = 2, kmax: int = 4, device="cpu", table=None,
               weights=None) -> MergeCase:
    r = rng(seed)
    lens = r.integers(kmin, kmax + 1, size=n_spans)
    offs = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    ids = r.integers(0, vocab, size=int(offs[-1])).astype(np.int32)
    if table is None:
        table = bf16_normal((vocab, d), 0.02, seed + 101, device)
    if weights is None:
        weights = merge_weights(d, h, seed + 202, device)
    return MergeCase(table=table, token_ids=torch.from_numpy(ids).to(device),
                     span_offsets=torch.from_numpy(offs).to(device), weights=weights)


# ----------------------------------------------------------------------------
# paged KV cache with spans to roll back
# ----------------------------------------------------------------------------
@dataclasses.dataclass
class DecodeCase:
    pool: torch.Tensor           # [n_layers][n_pages][2][Hkv][P][D] bf16
    block_table: torch.Tensor    # [B][max_pages] int32 (-1 = no page)
    seq_lens: torch.Tensor       # [B] int32
    span_offsets: torch.Tensor   # [B+1] int32 (CSR over sequences)
    span_start: torch.Tensor     # [S] int32
    span_len: torch.Tensor       # [S] int32
    surrogate_k: torch.Tensor    # [S][n_layers][Hkv][D] bf16
    surrogate_v: torch.Tensor
    q: torch.Tensor              # [B][Hq][D] bf16
    n_q_heads: int
    page_size: int = PAGE_SIZE

    @property
    def n_layers(self):
        return self.pool.shape[0]

    @property
    def n_pages(self):
        return self.pool.shape[1]

    @property
    def n_kv_heads(self):
        return self.pool.shape[3]

    @property
    def head_dim(self):
        return self.pool.shape[5]

    @property
    def max_pages(self):
        return self.block_table.shape[1]


def decode_case(seed: int, *, lens: Sequence[int], n_q_heads: int, n_kv_heads: int,
                head_dim: int, n_layers: int = 1, coverage: Optional[float] = None,
                n_spans: Optional[Sequence[int]] = None, kmin: int = 2, kmax: int = 4,
                spare_pages: int = 0, extra_max_pages: int = 0, suffix_only: bool = False,
                device="cpu", pool_device=None, kv_std: float = 1.0) -> DecodeCase:
    """A paged bf16 KV cache holding ``lens[b]`` entries per sequence, spans to
    roll back in each sequence, surrogate K/V and one query token per sequence.

    Physical pages are a random permutation of the pool, so logical order and
    physical order differ.  Every slot of the pool (used or not) holds N(0,1)
    bf16 values."""
    r = rng(seed)
    B = len(lens)
    P = PAGE_SIZE
    lens = np.asarray(lens, dtype=np.int64)
    pages_per = (lens + P - 1) // P
    max_pages = int(max(1, pages_per.max() if B else 1)) + extra_max_pages
    n_pages = int(pages_per.sum()) + spare_pages
    n_pages = max(n_pages, 1)
    perm = r.permutation(n_pages).astype(np.int32)
    bt = np.full((B, max_pages), -1, dtype=np.int32)
    k = 0
    for b in range(B):
        for p in range(int(pages_per[b])):
            bt[b, p] = perm[k]
            k += 1
    starts, slens, offs = [], [], [0]
    for b in range(B):
        L = int(lens[b])
        if suffix_only:
            if L >= 1 and r.random() < (coverage if coverage is not None else 1.0):
                s, kk = suffix_span(r, L, kmin, kmax)
                st, ln = np.array([s], np.int32), np.array([kk], np.int32)
            else:
                st, ln = np.zeros(0, np.int32), np.zeros(0, np.int32)
        elif n_spans is not None:
            st, ln = span_layout(r, L, n_spans=int(n_spans[b]), kmin=kmin, kmax=kmax)
        else:
            st, ln = span_layout(r, L, coverage=coverage or 0.0, kmin=kmin, kmax=kmax)
        starts.append(st)
        slens.append(ln)
        offs.append(offs[-1] + len(st))
    S = offs[-1]
    span_start = np.concatenate(starts).astype(np.int32) if S else np.zeros(0, np.int32)
    span_len = np.concatenate(slens).astype(np.int32) if S else np.zeros(0, np.int32)
    pdev = pool_device or device
    pool = bf16_normal((n_layers, n_pages, 2, n_kv_heads, P, head_dim), kv_std, seed + 11, pdev)
    sk = bf16_normal((S, n_layers, n_kv_heads, head_dim), 1.0, seed + 12, device)
    sv = bf16_normal((S, n_layers, n_kv_heads, head_dim), 1.0, seed + 13, device)
    q = bf16_normal((B, n_q_heads, head_dim), 1.0, seed + 14, device)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(device)
    return DecodeCase(pool=pool, block_table=t(bt), seq_lens=t(lens.astype(np.int32)),
                      span_offsets=t(np.asarray(offs, np.int32)), span_start=t(span_start),
                      span_len=t(span_len), surrogate_k=sk, surrogate_v=sv, q=q,
                      n_q_heads=n_q_heads)


# ----------------------------------------------------------------------------
# prompts for compaction
# ----------------------------------------------------------------------------
@dataclasses.dataclass
class PromptCase:
    table: torch.Tensor          # [V][d] bf16
    token_ids: torch.Tensor      # [B][L] int32
    span_offsets: torch.Tensor   # [B+1]
    span_start: torch.Tensor     # [S] position within its prompt
    span_len: torch.Tensor       # [S]
    span_token_ids: torch.Tensor  # [T] span tokens concatenated (merge-module input)
    span_token_offsets: torch.Tensor  # [S+1]


def prompt_case(seed: int, *, B: int, L: int, vocab: int, d: int, coverage: float,
                kmin: int = 2, kmax: int = 4, device="cpu", table=None) -> PromptCase:
    r = rng(seed)
    ids = r.integers(0, vocab, size=(B, L)).astype(np.int32)
    starts, slens, offs = [], [], [0]
    for b in range(B):
        st, ln = span_layout(r, L, coverage=coverage, kmin=kmin, kmax=kmax)
        starts.append(st)
        slens.append(ln)
        offs.append(offs[-1] + len(st))
    span_start = np.concatenate(starts).astype(np.int32)
    span_len = np.concatenate(slens).astype(np.int32)
    toks, toffs = [], [0]
    i = 0
    for b in range(B):
        for j in range(offs[b], offs[b + 1]):
            s, k = int(span_start[j]), int(span_len[j])
            toks.append(ids[b, s:s + k])
            toffs.append(toffs[-1] + k)
    span_tokens = np.concatenate(toks).astype(np.int32) if toks else np.zeros(0, np.int32)
    if table is None:
        table = bf16_normal((vocab, d), 0.02, seed + 101, device)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(device)
    return PromptCase(table=table, token_ids=t(ids), span_offsets=t(np.asarray(offs, np.int32)),
                      span_start=t(span_start), span_len=t(span_len),
                      span_token_ids=t(span_tokens),
                      span_token_offsets=t(np.asarray(toffs, np.int32)))


# ----------------------------------------------------------------------------
# merge rules and prompts that use them
# ----------------------------------------------------------------------------
def _distinct_rows(a: np.ndarray) -> np.ndarray:
    """Rows of a with repeats removed (first occurrence kept), order kept."""
    if len(a) == 0:
        return a
    order = np.lexsort(a.T[::-1])
    srt = a[order]
    first = np.ones(len(a), bool)
    first[1:] = np.any(srt[1:] != srt[:-1], axis=1)
    keep = np.zeros(len(a), bool)
    keep[order[first]] = True
    return a[keep]


def random_rules(seed: int, counts, vocab: int) -> np.ndarray:
    """Distinct n-grams: counts[0] 2-grams, counts[1] 3-grams, counts[2]
    4-grams with uniform token ids in [0, vocab), in that order, each as a
    row [4] int32 padded with -1 (the rule id is the row), rows shuffled."""
    r = rng(seed)
    out = []
    for n, c in zip((2, 3, 4), counts):
        got = np.zeros((0, n), np.int32)
        while len(got) < c:
            more = r.integers(0, vocab, size=(c - len(got) + 16, n)).astype(np.int32)
            got = _distinct_rows(np.concatenate([got, more]))
        rows = np.full((c, 4), -1, np.int32)
        rows[:, :n] = got[:c]
        out.append(rows)
    rules = np.concatenate(out) if out else np.zeros((0, 4), np.int32)
    return rules[r.permutation(len(rules))]


def rule_prompts(seed: int, rules: np.ndarray, *, B: int, L: int, vocab: int, coverage: float,
                 lens=None) -> np.ndarray:
    """Prompts [B][L] int32 of uniform random tokens in which occurrences of
    rules are planted at non-overlapping places until they cover about
    ``coverage`` of each prompt: a length n uniform in {2, 3, 4} (among the
    lengths the rule set has), then a rule of that length uniformly, placed by
    stars and bars as in span_layout.  lens[b] < L leaves the tail of row b as
    padding (-1)."""
    r = rng(seed)
    ids = r.integers(0, vocab, size=(B, L)).astype(np.int32)
    n_of = (rules >= 0).sum(axis=1) if len(rules) else np.zeros(0, np.int64)
    by_n = [np.nonzero(n_of == n)[0] for n in (2, 3, 4)]
    by_n = [g for g in by_n if len(g)]
    for b in range(B):
        Lb = L if lens is None else int(lens[b])
        chosen, tot = [], 0
        target = int(round(coverage * Lb))
        while by_n and tot < target:
            g = by_n[int(r.integers(0, len(by_n)))]
            j = int(g[int(r.integers(0, len(g)))])
            if tot + n_of[j] > Lb:
                break
            chosen.append(j)
            tot += int(n_of[j])
        S = len(chosen)
        if S:
            ks = n_of[chosen]
            bars = np.sort(r.choice(Lb - tot + S, size=S, replace=False))
            starts = bars - np.arange(S) + np.concatenate([[0], np.cumsum(ks)[:-1]])
            for j, s0 in zip(chosen, starts):
                ids[b, s0:s0 + n_of[j]] = rules[j, :n_of[j]]
        ids[b, Lb:] = -1
    return ids


def rule_tuples(rules: np.ndarray):
    """Rule rows [R][4] (-1 padded) as a list of token tuples, rule id order."""
    n_of = (rules >= 0).sum(axis=1)
    out = [None] * len(rules)
    for n in (2, 3, 4):
        idx = np.nonzero(n_of == n)[0]
        for i, g in zip(idx.tolist(), rules[idx, :n].tolist()):
            out[i] = tuple(g)
    return out


# ----------------------------------------------------------------------------
# serving-loop lengths
# ----------------------------------------------------------------------------
def serving_lengths(r: np.random.Generator, B: int, median: int = 1024, sigma: float = 1.0,
                    lo: int = 256, hi: int = 8192) -> np.ndarray:
    x = np.exp(np.log(median) + sigma * r.standard_normal(B))
    return np.clip(np.round(x), lo, hi).astype(np.int32)


# ----------------------------------------------------------------------------
# the decode loop of a serving engine (append, sometimes merge, attend)
# ----------------------------------------------------------------------------
class PageAllocator:
    """First-in first-out free-page list of a paged cache: the bookkeeping a
    serving engine's block allocator does (which physical page a sequence
    gets when its length reaches a page boundary)."""

    def __init__(self, free_pages):
        import collections
        self.free = collections.deque(int(p) for p in free_pages)

    def take(self, lens) -> np.ndarray:
        """new_pages[b]: a page for every sequence whose length is a multiple
        of the page size (it opens a page with its next entry), else -1."""
        new_pages = np.full(len(lens), -1, np.int32)
        for b, L in enumerate(lens):
            if int(L) % PAGE_SIZE == 0:
                new_pages[b] = self.free.popleft()
        return new_pages

    def give_back(self, pages):
        self.free.extend(int(p) for p in pages)


@dataclasses.dataclass
class ServingLoop:
    """A decode loop over a paged cache: every step appends one entry per
    sequence and layer, then each sequence with probability p merges its last
    k ~ U{kmin..kmax} stored entries (the new one included) into one
    surrogate entry, then attention runs per layer.  Initial KV entries,
    appended entries, surrogates and queries are N(0,1) bf16 drawn from seeds
    derived from (seed, step, layer), so any of them can be drawn again
    without replaying the loop."""
    seed: int
    n_layers: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    steps: int
    p: float
    kmin: int
    kmax: int
    lens: np.ndarray          # [B] initial lengths
    block_table: np.ndarray   # [B][max_pages] initial layout (-1 = no page)
    n_pages: int
    free_pages: list          # pages not in the initial layout, allocator order

    @property
    def B(self):
        return len(self.lens)

    def _seed(self, kind, step=0, layer=0):
        return self.seed + 7919 * kind + 104729 * step + layer

    def init_layer(self, layer, device):
        """Initial contents of one layer of the pool, [n_pages][2][Hkv][P][D]."""
        return bf16_normal((self.n_pages, 2, self.n_kv_heads, PAGE_SIZE, self.head_dim), 1.0,
                           self._seed(1, 0, layer), device)

    def init_pool(self, device):
        pool = torch.empty((self.n_layers, self.n_pages, 2, self.n_kv_heads, PAGE_SIZE, self.head_dim),
                           dtype=torch.bfloat16, device=device)
        for layer in range(self.n_layers):
            pool[layer] = self.init_layer(layer, device)
        return pool

    def new_entries(self, step, device):
        shape = (self.B, self.n_layers, self.n_kv_heads, self.head_dim)
        return (bf16_normal(shape, 1.0, self._seed(2, step, 0), device),
                bf16_normal(shape, 1.0, self._seed(2, step, 1), device))

    def rollbacks(self, step):
        """[(b, k)]: the sequences that merge their last k stored entries after
        this step's append, in increasing b."""
        r = rng(self._seed(3, step))
        hit = r.random(self.B) < self.p
        ks = r.integers(self.kmin, self.kmax + 1, size=self.B)
        return [(b, int(ks[b])) for b in range(self.B) if hit[b]]

    def surrogates(self, step, n, device):
        shape = (n, self.n_layers, self.n_kv_heads, self.head_dim)
        return (bf16_normal(shape, 1.0, self._seed(4, step, 0), device),
                bf16_normal(shape, 1.0, self._seed(4, step, 1), device))

    def q(self, step, layer, device):
        return bf16_normal((self.B, self.n_q_heads, self.head_dim), 1.0, self._seed(5, step, layer), device)


def serving_loop(seed: int, *, B: int, n_layers: int, n_q_heads: int, n_kv_heads: int, head_dim: int,
                 steps: int, p: float = 0.1, kmin: int = 2, kmax: int = 4, lens=None, median: int = 1024,
                 sigma: float = 1.0, lo: int = 256, hi: int = 8192) -> ServingLoop:
    """Lengths lognormal(ln median, sigma) clipped to [lo, hi] unless given;
    every sequence has room for `steps` appends; physical pages are a random
    permutation, the pages not in the initial layout form the free list."""
    r = rng(seed)
    lens = serving_lengths(r, B, median, sigma, lo, hi) if lens is None else np.asarray(lens, np.int32)
    P = PAGE_SIZE
    pages_now = (lens.astype(np.int64) + P - 1) // P
    pages_max = (lens.astype(np.int64) + steps + P - 1) // P
    max_pages = int(max(1, pages_max.max()))
    n_pages = int(pages_max.sum()) + B
    perm = r.permutation(n_pages).astype(np.int32)
    bt = np.full((B, max_pages), -1, np.int32)
    k = 0
    for b in range(B):
        for pg in range(int(pages_now[b])):
            bt[b, pg] = perm[k]
            k += 1
    return ServingLoop(seed=seed, n_layers=n_layers, n_q_heads=n_q_heads, n_kv_heads=n_kv_heads,
                       head_dim=head_dim, steps=steps, p=p, kmin=kmin, kmax=kmax, lens=lens.astype(np.int32),
                       block_table=bt, n_pages=n_pages, free_pages=[int(x) for x in perm[k:]])


# ----------------------------------------------------------------------------
# aligned predictive distillation (training side)
# ----------------------------------------------------------------------------
@dataclasses.dataclass
class DistillCase:
    seq_lens: torch.Tensor        # [B] int32 original lengths
    span_offsets: torch.Tensor    # [B+1]
    span_start: torch.Tensor      # [S] position within its sample
    span_len: torch.Tensor        # [S]
    teacher_logits: torch.Tensor  # [sum L][ld] bf16: the backbone's logits on the original sequences


def distill_case(seed: int, *, lens: Sequence[int], vocab: int, coverage: float = 0.4, kmin: int = 2,
                 kmax: int = 4, ld: Optional[int] = None, std: float = 2.0, device="cpu") -> DistillCase:
    """Samples of the given lengths with seeded spans (as span_layout) and
    N(0, std^2) teacher logits over the vocabulary, rows of stride ld
    (default: vocab rounded up to a multiple of 8).  The student logits are a
    separate draw (distill_logits) once the caller knows how many compressed
    rows there are."""
    r = rng(seed)
    starts, slens, offs = [], [], [0]
    for L in lens:
        st, ln = span_layout(r, int(L), coverage=coverage, kmin=kmin, kmax=kmax)
        starts.append(st)
        slens.append(ln)
        offs.append(offs[-1] + len(st))
    ld = ((vocab + 7) // 8) * 8 if ld is None else ld
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(device)
    cat = lambda xs: np.concatenate(xs).astype(np.int32) if xs else np.zeros(0, np.int32)
    return DistillCase(seq_lens=t(np.asarray(lens, np.int32)), span_offsets=t(np.asarray(offs, np.int32)),
                       span_start=t(cat(starts)), span_len=t(cat(slens)),
                       teacher_logits=distill_logits(seed + 1, int(sum(lens)), ld, std, device))


def distill_logits(seed: int, rows: int, ld: int, std: float = 2.0, device="cpu") -> torch.Tensor:
    """[rows][ld] bf16 logits, N(0, std^2)."""
    return bf16_normal((rows, ld), std, seed, device)
