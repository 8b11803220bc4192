"""The C ABI library builds, loads and exports every entry point its header
declares; host-side argument checks work without a GPU (no compute call)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", f) for f in os.listdir(os.path.join(ROOT, "include")) if f.endswith(".h")]


def declared_functions():
    names = set()
    for h in HEADERS:
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"^[A-Za-z_][\w \*]*?\b(umim_\w+)\s*\(", text, flags=re.M):
            names.add(m.group(1))
    return names


@pytest.fixture(scope="module", params=["release", "debug"])
def lib(request):
    """Each test below runs on libumim.so and on libumim_debug.so (UMIM_DEBUG)."""
    from paper_2609_27233_gb300 import build, _lib
    path = _lib.LIB_PATH if request.param == "release" else _lib.DEBUG_LIB_PATH
    if not os.path.exists(path):
        build.build(variants=(request.param,))
    return _lib.load(path)


def test_header_declares_the_four_calls():
    names = declared_functions()
    for n in ("umim_merge_spans", "umim_kv_rollback", "umim_decode_attention", "umim_build_compressed"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert names
    for n in names:
        assert hasattr(lib, n), n
    from paper_2609_27233_gb300 import _lib
    assert set(_lib.SIGNATURES) == names


def test_status_strings_and_version(lib):
    assert lib.umim_status_string(0) == b"UMIM_OK"
    assert lib.umim_status_string(4) == b"UMIM_ERR_TIMEOUT"
    assert lib.umim_version() >= 100


def test_debug_build_flag_and_status_words(lib, request):
    """The two builds say which they are; a debug build's UMIM_ERR_BOUNDS word
    carries the access site in bits 8 and up, and the release build refuses
    the bounds self-test without launching anything (no check would stop its
    store there)."""
    debug = request.node.callspec.params["lib"] == "debug"
    assert lib.umim_debug_build() == (1 if debug else 0)
    assert lib.umim_status_string(6) == b"UMIM_ERR_BOUNDS"
    assert lib.umim_status_string(6 | (3 << 8)) == b"UMIM_ERR_BOUNDS"
    assert lib.umim_debug_site_name(6 | (1 << 8)) == b"selftest"
    assert lib.umim_debug_site_name(6 | (3 << 8)) == b"rollback_move.dst_page"
    assert lib.umim_debug_site_name(6 | (23 << 8)) == b"rules.span_token"
    assert lib.umim_debug_site_name(6) == b""
    assert lib.umim_debug_site_name(6 | (999 << 8)) == b""
    null = ctypes.c_void_p(0)
    if debug:
        assert lib.umim_selftest_bounds_check(null, 4, 0, null, null) == 1        # no buffer
        assert lib.umim_selftest_bounds_check(ctypes.c_void_p(1 << 20), 0, 0, null, null) == 1   # empty
    else:
        assert lib.umim_selftest_bounds_check(ctypes.c_void_p(1 << 20), 4, 9, null, null) == 2


def test_every_site_of_the_kernels_has_a_name():
    """The site numbers the kernels record and the names the library gives
    them come from one enumeration, each name used once."""
    csrc = os.path.join(ROOT, "paper_2609_27233_gb300", "csrc")
    common = open(os.path.join(csrc, "common.cuh")).read()
    sites = dict((m.group(1), int(m.group(2))) for m in re.finditer(r"(kSite\w+) = (\d+)", common))
    count = sites.pop("kSiteCount")
    assert sorted(sites.values()) == list(range(1, count))
    used = set()
    for f in os.listdir(csrc):
        if f.endswith(".cu"):
            used |= set(re.findall(r"in_bounds\([^;]*?(kSite\w+)\)", open(os.path.join(csrc, f)).read(), flags=re.S))
    assert used == set(sites), set(sites) ^ used
    api = open(os.path.join(csrc, "api.cu")).read()
    names = re.search(r"names\[kSiteCount\] = \{(.*?)\};", api, flags=re.S).group(1)
    names = re.findall(r'"([^"]*)"', names)
    assert len(names) == count and names[0] == "" and len(set(names)) == count


def test_workspace_sizes_are_positive(lib):
    assert lib.umim_merge_spans_workspace_size(120, 40, 512) > 120 * 512 * 6
    assert lib.umim_kv_rollback_workspace_size(16, 6560, 256, 1, 8, 128) > 0
    assert lib.umim_kv_rollback_workspace_size(1, 1, 1, 1, 1, 96) == 0     # head_dim unsupported
    assert lib.umim_build_compressed_workspace_size(64, 17472) > 0
    assert lib.umim_decode_attention_workspace_size(16, 32, 8, 128) > 0


def test_host_checks_reject_bad_arguments_without_touching_the_gpu(lib):
    from paper_2609_27233_gb300._lib import PagedKVC, MergeWeightsC
    null = ctypes.c_void_p(0)
    kv = PagedKVC(0, 1, 1, 1, 16, 128)                                   # null base
    assert lib.umim_kv_rollback(ctypes.byref(kv), null, 1, null, 1, null, null, null, 0, null, null, null,
                                null, 0, null, null) == 1
    kv = PagedKVC(4096, 1, 1, 1, 8, 128)                                  # page size 8
    assert lib.umim_decode_attention(null, 1, ctypes.byref(kv), 0, null, 1, null, 1, 0.0, null, null, 0,
                                     null, null) == 2
    kv = PagedKVC(4096, 1, 1, 2, 16, 128)                                 # Hq not a multiple of Hkv
    assert lib.umim_decode_attention(null, 3, ctypes.byref(kv), 0, null, 1, null, 1, 0.0, null, null, 0,
                                     null, null) == 2
    w = MergeWeightsC(*([0] * 9), 500, 4, 1e-5)                           # d not a multiple of 512
    assert lib.umim_merge_spans(null, 10, null, 0, null, 1, ctypes.byref(w), null, null, 0, null, null) == 2
    w = MergeWeightsC(*([0] * 9), 512, 3, 1e-5)                           # 3 heads
    assert lib.umim_merge_spans(null, 10, null, 0, null, 1, ctypes.byref(w), null, null, 0, null, null) == 2
    # empty batches are a no-op that succeeds
    kv = PagedKVC(4096, 1, 1, 1, 16, 128)
    assert lib.umim_kv_rollback(ctypes.byref(kv), null, 1, null, 0, null, null, null, 0, null, null, null,
                                null, 0, null, null) == 0


def test_distillation_host_checks(lib):
    null = ctypes.c_void_p(0)
    fake = ctypes.c_void_p(1 << 20)      # never dereferenced: every call below fails its host checks
    loss = ctypes.c_void_p(1 << 21)
    assert lib.umim_distill_soft_ce_workspace_size(3000, 3000) > 3000 * 8
    assert lib.umim_distill_align_workspace_size(8, 1000) > 0
    ce = lambda V, ld, eps=1e-8, ws=null, grad=null, lo=loss: lib.umim_distill_soft_ce(
        fake, 4, fake, 4, V, ld, fake, fake, 4, null, eps, lo, null, grad, ws, 1 << 20, null, null)
    assert ce(163841, 163848) == 2               # vocabulary above the supported maximum
    assert ce(1000, 1001) == 1                   # row stride not a multiple of 8
    assert ce(1001, 1000) == 1                   # stride shorter than the vocabulary
    assert ce(1000, 1000, eps=-1.0) == 1         # negative eps
    assert ce(1000, 1000, eps=float("inf")) == 1
    assert ce(1000, 1000, lo=null) == 1          # no loss output
    assert ce(1000, 1000, grad=ctypes.c_void_p((1 << 20) + 2)) == 1   # misaligned gradient
    assert ce(1000, 1000) == 5                   # no workspace
    assert ce(1000, 1000, ws=ctypes.c_void_p((1 << 20) + 16)) == 5    # misaligned workspace
    assert lib.umim_distill_align(null, -1, null, null, null, 0, fake, null, null, 0, null, null, 0, null,
                                  null) == 1
    assert lib.umim_distill_align(fake, 2, fake, null, null, 3, fake, fake, fake, 10, null, fake, 1 << 20, null,
                                  null) == 1     # spans but no span arrays
    assert lib.umim_distill_align(fake, 2, fake, fake, fake, 3, fake, fake, fake, 10, null, null, 0, null,
                                  null) == 5     # no workspace


def test_product_path_and_oracle_share_nothing():
    """The library, its binding and its header never name the oracle, and the
    oracle never imports the library: the two sides meet only in the tests."""
    pkg = os.path.join(ROOT, "paper_2609_27233_gb300")
    product = [os.path.join(pkg, f) for f in os.listdir(pkg) if f.endswith(".py")]
    product += [os.path.join(pkg, "csrc", f) for f in os.listdir(os.path.join(pkg, "csrc"))]
    product += HEADERS
    for p in product:
        assert "oracle" not in open(p, errors="ignore").read(), p
    odir = os.path.join(ROOT, "oracle")
    for f in os.listdir(odir):
        if f.endswith(".py"):
            text = open(os.path.join(odir, f)).read()
            for bad in ("import paper_2609_27233_gb300", "from paper_2609_27233_gb300", "ctypes", "libumim"):
                assert bad not in text, (f, bad)


def test_allocation_free_attention_host_checks(lib):
    """Shapes and arguments are refused on the host, before the first CUDA call."""
    from paper_2609_27233_gb300._lib import PagedKVC
    null = ctypes.c_void_p(0)
    fake = ctypes.c_void_p(1 << 20)      # never dereferenced: every call below stops at a host check

    def call(kv, hq=8, layer=0, batch=2, q=fake, out=fake):
        return lib.umim_decode_attention_static(q, hq, ctypes.byref(kv), layer, fake, 4, fake, batch, 0.0, out,
                                                null, null)

    assert call(PagedKVC(0, 1, 4, 2, 16, 128)) == 1          # no pool
    assert call(PagedKVC(4096 + 8, 1, 4, 2, 16, 128)) == 1   # pool not 16-byte aligned
    assert call(PagedKVC(4096, 1, 4, 2, 8, 128)) == 2        # page size 8
    assert call(PagedKVC(4096, 1, 4, 2, 16, 96)) == 2        # head_dim 96
    assert call(PagedKVC(4096, 1, 4, 2, 16, 128), hq=34) == 2   # 17 query heads per KV head
    assert call(PagedKVC(4096, 1, 4, 2, 16, 128), hq=7) == 2    # not a multiple of the KV heads
    assert call(PagedKVC(4096, 2, 4, 2, 16, 128), layer=2) == 1
    assert call(PagedKVC(4096, 1, 4, 2, 16, 128), q=null) == 1
    assert call(PagedKVC(4096, 1, 4, 2, 16, 128), out=ctypes.c_void_p((1 << 20) + 1)) == 1
    assert call(PagedKVC(4096, 1, 4, 2, 16, 128), batch=0) == 0   # nothing to do


def test_other_entry_points_host_checks(lib):
    """Compressed prompts, append, surrogate lookup, prefill and the wait
    self-test refuse bad arguments on the host (no CUDA call is reached)."""
    from paper_2609_27233_gb300._lib import PagedKVC
    null = ctypes.c_void_p(0)
    fake = ctypes.c_void_p(1 << 20)
    odd = ctypes.c_void_p((1 << 20) + 4)

    def compressed(d=512, batch=2, emb=fake, ws=fake, wsb=1 << 24):
        return lib.umim_build_compressed(emb, 1000, d, fake, batch, 64, fake, fake, fake, 3, fake, fake, 1000,
                                         fake, fake, ws, wsb, null, null)
    assert compressed(d=500) == 2                # d_model not a multiple of 8
    assert compressed(batch=-1) == 1
    assert compressed(batch=0) == 0
    assert compressed(emb=null) == 1
    assert compressed(emb=odd) == 1              # table not 16-byte aligned
    assert compressed(ws=null) == 5
    assert compressed(wsb=16) == 5

    kv = PagedKVC(4096, 1, 4, 2, 16, 128)
    assert lib.umim_kv_append(ctypes.byref(kv), fake, 4, fake, 2, odd, fake, fake, null, null) == 1
    assert lib.umim_kv_append(ctypes.byref(kv), null, 4, fake, 2, fake, fake, fake, null, null) == 1
    assert lib.umim_kv_append(ctypes.byref(kv), fake, 4, fake, 0, fake, fake, fake, null, null) == 0
    kv64 = PagedKVC(4096, 1, 4, 2, 16, 96)
    assert lib.umim_kv_append(ctypes.byref(kv64), fake, 4, fake, 2, fake, fake, fake, null, null) == 2

    assert lib.umim_lookup_surrogates(fake, 10, 6, fake, 4, null, fake, null, null) == 1   # d % 4 != 0
    assert lib.umim_lookup_surrogates(odd, 10, 8, fake, 4, null, fake, null, null) == 1
    assert lib.umim_lookup_surrogates(fake, 10, 8, fake, 0, null, fake, null, null) == 0

    def prefill(hd=128, hq=32, hkv=8, q=fake, ws=fake, batch=2):
        return lib.umim_prefill_attention(q, fake, fake, 100, hq, hkv, hd, fake, batch, 0.0, fake, ws, 1 << 30,
                                          null, null)
    assert prefill(hd=96) == 2
    assert prefill(hq=30) == 2                   # not a multiple of the KV heads
    assert prefill(batch=0) == 0
    assert prefill(q=odd) == 1
    assert prefill(ws=null) == 5

    assert lib.umim_selftest_bounded_wait(2, 1000, null, null, null, null) == 1
    assert lib.umim_selftest_bounded_wait(0, 0, null, null, null, null) == 1
    assert lib.umim_selftest_bounded_wait(0, 2000000, null, null, null, null) == 1
    assert lib.umim_selftest_bounded_wait(1, 1000, null, null, null, null) == 1   # flags needed


def test_binding_scratch_size_matches_the_header():
    text = open(os.path.join(ROOT, "include", "umim.h")).read()
    m = re.search(r"#define UMIM_STATIC_SCRATCH_BYTES \((\d+)u << (\d+)\)", text)
    assert m
    import paper_2609_27233_gb300 as umim
    assert umim.STATIC_SCRATCH_BYTES == int(m.group(1)) << int(m.group(2))


def test_layer_step_host_checks(lib):
    """The per-layer decode step refuses bad shapes and arguments on the host,
    before the first CUDA call."""
    from paper_2609_27233_gb300._lib import PagedKVC
    null = ctypes.c_void_p(0)
    fake = ctypes.c_void_p(1 << 20)      # never dereferenced: every call below stops at a host check
    kv = PagedKVC(4096, 2, 4, 2, 16, 128)

    def call(kv=kv, hq=8, layer=0, batch=2, stride=0, q=fake, out=fake, nk=fake, rows=0, mk=null):
        return lib.umim_decode_layer_step(q, hq, ctypes.byref(kv), layer, fake, 4, fake, batch, nk, fake, stride,
                                          null, mk, null, rows, null, null, 0, null, 0.0, out, null, 0, null, null)

    assert lib.umim_decode_layer_step_workspace_size(128, 8, 128) > 0
    assert lib.umim_decode_layer_step_workspace_size(128, 8, 96) == 0
    assert call(kv=PagedKVC(0, 2, 4, 2, 16, 128)) == 1       # no pool
    assert call(kv=PagedKVC(4096, 2, 4, 2, 16, 96)) == 2     # head_dim 96
    assert call(hq=34) == 2                                  # 17 query heads per KV head
    assert call(batch=4097) == 2                             # above the largest batch
    assert call(layer=2) == 1                                # no such layer
    assert call(stride=100) == 1                             # row stride below n_kv_heads * head_dim
    assert call(stride=260) == 1                             # not a multiple of 8 elements
    assert call(nk=null) == 1                                # no new entries
    assert call(nk=ctypes.c_void_p((1 << 20) + 8)) == 1      # new entries not 16-byte aligned
    assert call(out=ctypes.c_void_p((1 << 20) + 2)) == 1     # output not 4-byte aligned
    assert call(rows=3, mk=fake) == 1                        # merges without surrogate arrays
    assert call(batch=0) == 0                                # an empty batch is a no-op


def test_merge_needs_a_token_per_span(lib):
    from paper_2609_27233_gb300._lib import MergeWeightsC
    null = ctypes.c_void_p(0)
    w = MergeWeightsC(*([1 << 20] * 9), 512, 4, 1e-5)
    assert lib.umim_merge_spans(null, 10, null, 3, null, 4, ctypes.byref(w), null, null, 0, null, null) == 1


def test_binding_switches_library_and_decodes_bounds_words():
    """use_debug_library routes the binding's calls to libumim_debug.so and back;
    a UMIM_ERR_BOUNDS word raises an error naming its access site."""
    import paper_2609_27233_gb300 as umim
    from paper_2609_27233_gb300 import build, _lib
    for path, v in ((_lib.LIB_PATH, "release"), (_lib.DEBUG_LIB_PATH, "debug")):
        if not os.path.exists(path):
            build.build(variants=(v,))
    try:
        umim.use_debug_library(True)
        assert umim.umim_debug_build() == 1
        err = umim.UmimError(umim.UMIM_ERR_BOUNDS | (12 << 8), "step")
        assert err.site == "decode_step.cache_write" and "UMIM_ERR_BOUNDS at decode_step.cache_write" in str(err)
    finally:
        umim.use_debug_library(False)
    assert umim.umim_debug_build() == 0
    assert "UMIM_ERR_TIMEOUT" in str(umim.UmimError(4, "x")) and umim.UmimError(4).site == ""
