"""CPU oracle for the UMIM decode step over a merged context (arXiv 2609.27233).

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports, links or runs
this package: only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s
CPU-baseline / reference arm use it.  It shares no code with the CUDA library
(``paper_2609_27233_gb300``) and does not import it.

Every function is a plain, slow, obviously-correct restatement of what the
paper defines, in float64 for floating point and exact integer / byte logic
for indices and moved KV bytes:

  merge.merge_spans       App. C.1 (attention-based pooling), Sec. 3.2 Eq. 1
  rollback.kv_rollback    App. C.6 and App. E ("Decoding-Time Merging and
                          KV-Cache Update"), Fig. 2 caption
  append.kv_append        App. E and Fig. 2 step (2): one KV entry appended
                          per layer when no rule matches
  attention.decode_attention
                          the backbone's ordinary attention over the shorter
                          cache (App. I.1); grouped-query mapping of Llama
  compaction.build_compressed
                          App. C.5 and App. E ("Prompt Merging"), App. J.4
                          ("Compressed-position convention")
  spans.span_metadata     removed-position count r(t) and compressed index
                          pi(t) = t - r(t) of App. J.4
  rules.match_prompt / match_prompts
                          App. E ("Rule Matching", "Prompt Merging"):
                          left-to-right, longest-first n-gram matching
  rules.SuffixState / match_suffixes
                          App. E ("Decoding-Time Merging"): longest-first
                          test of the raw generated suffix after every token
  rules.lookup            App. E (potential engineering optimizations):
                          surrogates precomputed per rule, fetched by id
  prefill.prefill_attention
                          App. E ("Prompt Merging"), App. C.5: the backbone's
                          causal grouped-query attention over the packed
                          compressed prompts
  distill.align / soft_ce
                          App. F (Algorithm 1, the masked distillation
                          loss): teacher / student alignment masks packed
                          into pairs, the soft cross-entropy and its
                          gradient with respect to the student logits

bf16 values are represented by their raw bit patterns (numpy uint16) and
upcast exactly to float64.

Parity status per function (what pins it is in tests/test_oracle_*.py):
  merge_spans       pinned (library routines, invariants, brute force)
  kv_rollback       pinned (worked example, length formula, invariants); its
                    key re-rotation to compressed positions pinned by the
                    complex-exponential RoPE identity, the rotation bound and
                    inner-product invariance (tests/test_oracle_rope.py)
  kv_append         pinned (logical-list model, rollback identities)
  decode_attention  pinned (library SDPA, closed forms, invariants)
  build_compressed  pinned (worked example, length formula, library bf16)
  match_prompt(s)   pinned (worked example, independent greedy-condition
                    checker, closed forms)
  SuffixState       pinned (worked example, list model with markers,
                    equality with prompt matching for 2-gram rules)
  lookup            pinned (equals merging the matched spans)
  prefill_attention pinned (library causal SDPA, closed forms, packing,
                    last row = decode attention)
  align / soft_ce   pinned (the paper's alignment example, the compressed-
                    position map, library soft cross-entropy and KL,
                    autograd)
"""
from . import bf16, spans, merge, rollback, append, attention, compaction, rules, prefill, distill  # noqa: F401
from .merge import merge_spans, merge_span_reference_steps  # noqa: F401
from .rollback import kv_rollback  # noqa: F401
from .append import kv_append  # noqa: F401
from .attention import decode_attention  # noqa: F401
from .compaction import build_compressed  # noqa: F401
from .prefill import prefill_attention  # noqa: F401
