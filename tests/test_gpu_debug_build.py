"""The debug build, libumim_debug.so: the same calls compiled with UMIM_DEBUG,
whose kernels check at every access site that the indexes they computed from
device data (pages read from block tables, rows and offsets of their own
plans, partial-result slots) lie inside the buffers they address.  A failed
check records UMIM_ERR_BOUNDS | site << 8 and skips the access instead of
touching memory outside a buffer.

Here: the check itself (the store it guards is skipped and the site is
reported), then the small parity and rejection cases of every call re-run on
the debug build -- the same oracle comparisons as on libumim.so, byte for
byte where the outputs are bytes, and no access site may report, on valid
inputs or on the invalid inputs the calls must refuse.  The canary test checks
that a rollback leaves every page it may not touch unchanged."""
import os

import pytest
import torch

import paper_2609_27233_gb300 as umim_pkg
from helpers import dev, umim

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def debug_library():
    from paper_2609_27233_gb300 import _lib, build
    if not os.path.exists(_lib.DEBUG_LIB_PATH):
        build.build(variants=("debug",))
    umim_pkg.use_debug_library(True)
    try:
        assert umim_pkg.umim_debug_build() == 1
        yield
    finally:
        umim_pkg.use_debug_library(False)


def test_an_index_inside_the_buffer_is_stored():
    m, dv = umim(), dev()
    buf = torch.zeros(8, dtype=torch.int32, device=dv)
    st = m.umim_selftest_bounds_check(buf, 7)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert buf.tolist() == [0] * 7 + [1]


@pytest.mark.parametrize("index", [8, -1, 1 << 40])
def test_an_index_outside_the_buffer_is_reported_and_not_stored(index):
    """The check compares the index against the buffer's length and reports
    the site instead of storing, so no access outside the buffer is made."""
    m, dv = umim(), dev()
    guard = torch.zeros(64, dtype=torch.int32, device=dv)
    buf = guard[16:24]   # 8 words with 16 zero words on either side
    st = m.umim_selftest_bounds_check(buf, index)
    torch.cuda.synchronize()
    code = int(st.item())
    assert code & 0xff == m.UMIM_ERR_BOUNDS and code >> 8 == 1
    assert m.umim_debug_site_name(code) == "selftest"
    assert int(guard.abs().sum().item()) == 0
    with pytest.raises(m.UmimError, match="UMIM_ERR_BOUNDS at selftest"):
        m.check_status(st, "selftest")
    # the context still runs ordinary work afterwards
    st2 = m.umim_selftest_bounds_check(buf, 0)
    torch.cuda.synchronize()
    assert int(st2.item()) == 0 and int(buf[0].item()) == 1


# The small cases of each call, collected again here so that they run on the
# debug build (the autouse fixture above switches the library for every test
# of this module).  Each asserts the exact status it expects: 0 on valid
# inputs, UMIM_ERR_INVALID_ARG on the invalid ones.
from test_gpu_rollback import (  # noqa: E402,F401
    test_rollback_matches_oracle as test_debug_rollback_matches_oracle,
    test_spans_at_both_ends_and_page_aligned_lengths as test_debug_rollback_spans_at_both_ends,
    test_no_spans_changes_nothing as test_debug_rollback_no_spans,
    test_invalid_input_is_rejected_before_any_write as test_debug_rollback_rejects_invalid_input,
    test_workspace_reused_across_calls as test_debug_rollback_workspace_reused,
)
from test_gpu_rollback_rope import (  # noqa: E402,F401
    test_rope_rollback_matches_oracle as test_debug_rope_rollback_matches_oracle,
)
from test_gpu_failure import (  # noqa: E402,F401
    test_rollback_leaves_canary_pages_alone as test_debug_rollback_leaves_canary_pages_alone,
)
from test_gpu_append import (  # noqa: E402,F401
    test_append_steps_match_oracle as test_debug_append_steps_match_oracle,
    test_impossible_appends_are_rejected_and_leave_the_sequence_unchanged as test_debug_impossible_appends,
    test_append_merge_matches_append_then_suffix_rollback as test_debug_append_merge,
    test_impossible_merges_are_rejected_and_leave_the_sequence_unchanged as test_debug_impossible_merges,
)
from test_gpu_attention import (  # noqa: E402,F401
    test_attention_matches_oracle as test_debug_attention_matches_oracle,
    test_empty_sequences_give_zero as test_debug_attention_empty_sequences,
    test_garbage_past_the_end_is_ignored as test_debug_attention_garbage_past_the_end,
    test_after_gpu_rollback as test_debug_attention_after_gpu_rollback,
)
from test_gpu_layer_step import (  # noqa: E402,F401
    test_layer_steps_match_append_rollback_attention as test_debug_layer_steps,
    test_rejected_sequences_are_left_unchanged as test_debug_layer_step_rejected_sequences,
)
from test_gpu_merge import (  # noqa: E402,F401
    test_merge_matches_oracle as test_debug_merge_matches_oracle,
    test_bad_token_id_is_flagged as test_debug_merge_bad_token_id,
)
from test_gpu_compaction import (  # noqa: E402,F401
    test_compaction_matches_oracle as test_debug_compaction_matches_oracle,
    test_capacity_too_small_writes_nothing as test_debug_compaction_capacity_too_small,
)
from test_gpu_prefill import (  # noqa: E402,F401
    test_prefill_matches_oracle as test_debug_prefill_matches_oracle,
    test_bad_offsets_write_nothing as test_debug_prefill_bad_offsets,
)
from test_gpu_distill import (  # noqa: E402,F401
    test_align_ragged as test_debug_align_ragged,
    test_align_rejects_invalid_input as test_debug_align_rejects_invalid_input,
    test_soft_ce_matches_oracle as test_debug_soft_ce_matches_oracle,
    test_soft_ce_rejects_invalid_pairs as test_debug_soft_ce_rejects_invalid_pairs,
    test_soft_ce_repeatable_padding_loss_only_and_fewer_pairs as test_debug_soft_ce_padding_and_fewer_pairs,
)
from test_gpu_rules import (  # noqa: E402,F401
    test_prompt_matching_matches_oracle as test_debug_prompt_matching_matches_oracle,
    test_invalid_rules_and_tokens_are_reported as test_debug_invalid_rules_and_tokens,
    test_suffix_matching_every_step as test_debug_suffix_matching_every_step,
    test_lookup_matches_indexing as test_debug_lookup_matches_indexing,
)
from test_gpu_serving import (  # noqa: E402,F401
    test_small_serving_loop_matches_oracle_every_step as test_debug_small_serving_loop,
)
