"""The C ABI without a GPU: the library loads, exports every function that
include/spire.h declares, and rejects bad host arguments before launching."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "spire.h")


@pytest.fixture(scope="module")
def spire():
    import __graft_entry__
    __graft_entry__._load_build_module().build()
    import paper_2504_06419_gb300 as m
    return m


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"SPIRE_API\s+[\w\s\*]+?\b(spire_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    assert names == sorted([
        "spire_verify_workspace_bytes", "spire_verify_attention",
        "spire_verify_attention_noalloc", "spire_draft_workspace_bytes", "spire_draft_sparse_attention", "spire_draft_slot",
        "spire_feedback_append_workspace_bytes", "spire_feedback_append",
        "spire_verify_tokens_workspace_bytes", "spire_verify_tokens",
        "spire_magicdec_workspace_bytes", "spire_magicdec_attention",
        "spire_get_device_error", "spire_get_cta_times", "spire_stream_read",
        "spire_test_draft_slots", "spire_test_stall_next_call", "spire_status_string"]), names


def test_library_exports_every_declared_symbol(spire):
    lib = ctypes.CDLL(spire._lib.LIB_PATH)
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert set(spire._lib.EXPORTED) == set(declared_functions())


def test_status_strings(spire):
    assert spire.spire_status_string(0) == "SPIRE_OK"
    assert spire.spire_status_string(3) == "SPIRE_ERR_WORKSPACE"
    assert spire.spire_status_string(99) == "SPIRE_ERR_UNKNOWN"


def test_draft_slot_host(spire):
    assert spire.spire_draft_slot(3, 4, 64) == 3
    assert spire.spire_draft_slot(4, 4, 64) == 4
    assert spire.spire_draft_slot(68, 4, 64) == 4
    assert spire.spire_draft_slot(69, 4, 64) == 5
    assert spire.spire_draft_slot(-1, 4, 64) == -1
    assert spire.spire_draft_slot(5, 4, 0) == -1


def _desc(spire, **kw):
    d = dict(batch=2, num_q_heads=8, num_kv_heads=2, head_dim=128, page_size=64,
             max_pages_per_seq=4, num_pages=8, softmax_scale=1.0)
    d.update(kw)
    return spire.make_desc(**d)


FAKE = 1 << 20   # a 16-byte aligned non-null "device" address; never dereferenced here


def _verify(spire, desc, k=4, ws_bytes=None, **ptrs):
    p = dict(q=FAKE, kc=FAKE, vc=FAKE, bt=FAKE, cl=FAKE, out=FAKE, ws=FAKE)
    p.update(ptrs)
    if ws_bytes is None:
        ws_bytes = spire.spire_verify_workspace_bytes(desc, k)
    return spire.spire_verify_attention(p["q"], p["kc"], p["vc"], p["bt"], p["cl"], k, desc,
                                        p["out"], p["ws"], ws_bytes, 0)


@pytest.mark.parametrize("kw,code", [
    (dict(num_q_heads=7), 1),          # Hq % Hkv != 0
    (dict(num_kv_heads=0), 1),
    (dict(batch=-1), 1),
    (dict(head_dim=96), 2),            # unsupported head_dim
    (dict(page_size=32), 2),           # unsupported page size
    (dict(softmax_scale=0.0), 1),
    (dict(softmax_scale=float("nan")), 1),
    (dict(max_pages_per_seq=0), 1),
])
def test_verify_rejects_bad_desc(spire, kw, code):
    assert _verify(spire, _desc(spire, **kw), ws_bytes=1 << 30) == code


def test_verify_rejects_bad_args(spire):
    d = _desc(spire)
    assert _verify(spire, d, k=-1, ws_bytes=1 << 30) == 1
    assert _verify(spire, d, k=32, ws_bytes=1 << 30) == 2          # 4 * 33 > 128 rows
    assert _verify(spire, d, q=0) == 1
    assert _verify(spire, d, out=0) == 1
    assert _verify(spire, d, q=FAKE + 2) == 1                      # misaligned
    assert _verify(spire, d, ws=0) == 3
    assert _verify(spire, d, ws=FAKE + 16) == 3                    # workspace misaligned
    assert _verify(spire, d, ws_bytes=spire.spire_verify_workspace_bytes(d, 4) - 1) == 3
    assert _verify(spire, _desc(spire, batch=0), q=0, kc=0, ws=0, ws_bytes=0) == 0


def test_draft_rejects_bad_args(spire):
    d = _desc(spire)
    ws = spire.spire_draft_workspace_bytes(d, 4, 64)
    f = spire.spire_draft_sparse_attention
    assert f(FAKE, FAKE, FAKE, -1, 64, d, FAKE, FAKE, ws, 0) == 1
    assert f(FAKE, FAKE, FAKE, 4, 0, d, FAKE, FAKE, ws, 0) == 1
    assert f(0, FAKE, FAKE, 4, 64, d, FAKE, FAKE, ws, 0) == 1
    assert f(FAKE, FAKE, FAKE, 4, 64, d, FAKE, FAKE, ws - 1, 0) == 3
    assert f(FAKE, FAKE, FAKE, 4, 64, _desc(spire, head_dim=80), FAKE, FAKE, ws, 0) == 2
    assert spire.spire_draft_workspace_bytes(d, 4, 0) == 0


def test_workspace_sizes_depend_only_on_shapes(spire):
    d = _desc(spire, batch=64, num_q_heads=32, num_kv_heads=8)
    a = spire.spire_verify_workspace_bytes(d, 4)
    assert a > 0 and a % 256 == 0
    assert spire.spire_verify_workspace_bytes(d, 8) > a
    assert spire.spire_verify_workspace_bytes(_desc(spire, batch=64, num_q_heads=32,
                                                    num_kv_heads=8, num_pages=10 ** 6), 4) == a
    assert spire.spire_draft_workspace_bytes(d, 16, 512) == spire.spire_draft_workspace_bytes(d, 0, 9)
    assert spire.spire_verify_workspace_bytes(None, 4) == 0


def _adesc(spire, **kw):
    d = dict(batch=64, num_act=3, num_draft_layers=2, d_model=4096, num_kv_heads=8, head_dim=128,
             n_sink=16, window=512, rope_theta=10000.0)
    d.update(kw)
    return spire.make_append_desc(**d)


def test_append_workspace_depends_only_on_shapes(spire):
    # the header word and one device error word per CTA (at most 512): the
    # kernel keeps its split partials in shared memory, so no shape needs more
    d = _adesc(spire)
    n = 256 + 4 * 512
    assert spire.spire_feedback_append_workspace_bytes(d) == n
    assert spire.spire_feedback_append_workspace_bytes(_adesc(spire, batch=300)) == n
    assert spire.spire_feedback_append_workspace_bytes(_adesc(spire, num_act=16, d_model=64)) == n
    assert spire.spire_feedback_append_workspace_bytes(_adesc(spire, batch=0)) == n


def test_append_empty_batch_is_a_no_op(spire):
    # B = 0: the rest of the shape is still checked, nothing is read or launched
    assert spire.spire_feedback_append(0, 0, 0, 0, _adesc(spire, batch=0), 0, 0, 0, 0) == 0
    assert spire.spire_feedback_append(0, 0, 0, 0, _adesc(spire, batch=0, head_dim=96), 0, 0, 0,
                                       0) == spire._lib.SPIRE_ERR_UNSUPPORTED
    assert spire.spire_feedback_append(0, 0, 0, 0, _adesc(spire, batch=0, window=0), 0, 0, 0,
                                       0) == spire._lib.SPIRE_ERR_INVALID_ARG


@pytest.mark.parametrize("kw", [
    dict(batch=-1), dict(num_act=0), dict(num_act=17), dict(num_draft_layers=0),
    dict(d_model=100), dict(d_model=0), dict(num_kv_heads=0), dict(head_dim=96),
    dict(n_sink=-1), dict(window=0), dict(rope_theta=-1.0), dict(rope_theta=float("inf")),
])
def test_append_rejects_bad_desc(spire, kw):
    d = _adesc(spire, **kw)
    assert spire.spire_feedback_append_workspace_bytes(d) == 0
    good = 1 << 20
    st = spire.spire_feedback_append(good, good, good, good, d, good, good, 1 << 30, 0)
    want = spire._lib.SPIRE_ERR_UNSUPPORTED if "head_dim" in kw else spire._lib.SPIRE_ERR_INVALID_ARG
    assert st == want


def test_append_rejects_bad_args(spire):
    d = _adesc(spire)
    ws = spire.spire_feedback_append_workspace_bytes(d)
    good = 1 << 20
    E = spire._lib
    # null pointers, misalignment, small workspace: all refused before any launch
    for i in range(6):
        args = [good] * 6
        args[i] = 0
        x, mw, wkv, pos, kv, w = args
        assert spire.spire_feedback_append(x, mw, wkv, pos, d, kv, w, ws, 0) == E.SPIRE_ERR_INVALID_ARG
    assert spire.spire_feedback_append(good + 8, good, good, good, d, good, good, ws, 0) == \
        E.SPIRE_ERR_INVALID_ARG
    assert spire.spire_feedback_append(good, good, good, good, d, good, good + 16, ws, 0) == \
        E.SPIRE_ERR_INVALID_ARG
    assert spire.spire_feedback_append(good, good, good, good, d, good, good, ws - 1, 0) == \
        E.SPIRE_ERR_WORKSPACE
    assert spire.spire_feedback_append(good, good, good, good, None, good, good, ws, 0) == \
        E.SPIRE_ERR_INVALID_ARG


def test_tokens_workspace_and_host_checks(spire):
    E = spire._lib
    # header and error word, one 8-byte accept record per sequence (256-byte
    # aligned), one 24-byte partial per 4096-entry chunk
    assert spire.spire_verify_tokens_workspace_bytes(64, 4, 128256) == 512 + 512 + 64 * 32 * 24
    assert spire.spire_verify_tokens_workspace_bytes(1, 0, 1) == 512 + 256 + 24
    assert spire.spire_verify_tokens_workspace_bytes(0, 4, 100) == 512
    for bad in [(-1, 4, 100), (1, -1, 100), (1, 32, 100), (1, 4, 0), (70000, 1, 10)]:
        assert spire.spire_verify_tokens_workspace_bytes(*bad) == 0
    good = 1 << 20
    ws = spire.spire_verify_tokens_workspace_bytes(8, 4, 1000)
    call = lambda **kw: spire.spire_verify_tokens(**{**dict(
        p=good, q=good, draft_tokens=good, u=good, e=good, batch=8, k=4, vocab=1000,
        out_tokens=good, n_accepted=good, workspace=good, ws_bytes=ws, stream=0), **kw})
    for name in ("p", "q", "draft_tokens", "u", "e", "out_tokens", "n_accepted", "workspace"):
        assert call(**{name: 0}) == E.SPIRE_ERR_INVALID_ARG, name
    # with k = 0 the draft arguments may be NULL: refused only for the small workspace
    assert call(k=0, q=0, draft_tokens=0, u=0, ws_bytes=0) == E.SPIRE_ERR_WORKSPACE
    assert call(p=good + 4) == E.SPIRE_ERR_INVALID_ARG           # V % 4 == 0 needs 16 B
    assert call(p=good + 2, vocab=1001) == E.SPIRE_ERR_INVALID_ARG
    assert call(ws_bytes=ws - 1) == E.SPIRE_ERR_WORKSPACE
    assert call(k=40) == E.SPIRE_ERR_UNSUPPORTED
    # B = 0: nothing to do, any pointer may be NULL; k and V are still checked
    assert call(batch=0, p=0, q=0, draft_tokens=0, u=0, e=0, out_tokens=0, n_accepted=0,
                workspace=0, ws_bytes=0) == E.SPIRE_OK
    assert call(batch=0, k=40) == E.SPIRE_ERR_UNSUPPORTED
    assert call(batch=0, vocab=0) == E.SPIRE_ERR_INVALID_ARG
    assert call(batch=-1) == E.SPIRE_ERR_INVALID_ARG


def test_magicdec_host_checks(spire):
    E = spire._lib
    d = _desc(spire)
    ws = spire.spire_magicdec_workspace_bytes(d, 1, 64)
    assert ws > spire.spire_draft_workspace_bytes(d, 1, 64)
    assert spire.spire_magicdec_workspace_bytes(d, -1, 64) == 0
    assert spire.spire_magicdec_workspace_bytes(d, 1, 0) == 0
    good = 1 << 20
    call = lambda **kw: spire.spire_magicdec_attention(**{**dict(
        q=good, k_cache=good, v_cache=good, block_table=good, ctx_lens=good, n_sink=1,
        window=64, rope_theta=10000.0, desc=d, out=good, workspace=good, ws_bytes=ws,
        stream=0), **kw})
    for name in ("q", "k_cache", "v_cache", "block_table", "ctx_lens", "out"):
        assert call(**{name: 0}) == E.SPIRE_ERR_INVALID_ARG, name
    assert call(workspace=0) == E.SPIRE_ERR_WORKSPACE
    assert call(ws_bytes=ws - 1) == E.SPIRE_ERR_WORKSPACE
    assert call(rope_theta=-1.0) == E.SPIRE_ERR_INVALID_ARG
    assert call(rope_theta=float("nan")) == E.SPIRE_ERR_INVALID_ARG
    assert call(window=0) == E.SPIRE_ERR_INVALID_ARG
    assert call(q=good + 8) == E.SPIRE_ERR_INVALID_ARG
    assert call(desc=_desc(spire, page_size=32)) == E.SPIRE_ERR_UNSUPPORTED
    assert call(window=70000) == E.SPIRE_ERR_UNSUPPORTED


def test_cta_times_host_checks(spire):
    """Argument errors of spire_get_cta_times come back before any CUDA call."""
    lib = spire._lib.LIB
    n = ctypes.c_int32(-1)
    buf = (ctypes.c_uint64 * 4)()
    assert lib.spire_get_cta_times(None, 1 << 20, buf, 2, ctypes.byref(n), None) == 1
    assert lib.spire_get_cta_times(256, 1 << 20, buf, 2, None, None) == 1
    assert lib.spire_get_cta_times(256, 1 << 20, None, 2, ctypes.byref(n), None) == 1
    assert lib.spire_get_cta_times(256, 1 << 20, buf, -1, ctypes.byref(n), None) == 1
    assert lib.spire_get_cta_times(256, 255, buf, 2, ctypes.byref(n), None) == 3
    assert n.value == -1


def test_stream_read_host_checks(spire):
    # a zero-byte read is a no-op; null, misaligned or ragged sizes are refused
    # before anything is launched
    assert spire.spire_stream_read(None, 0, 0) == 0
    assert spire.spire_stream_read(None, 16, 0) == 1
    assert spire.spire_stream_read(1 << 20, 8, 0) == 1
    assert spire.spire_stream_read((1 << 20) + 8, 16, 0) == 1


def test_draft_slots_hook_host_checks(spire):
    # n = 0 is a no-op; a negative n, a null or a misaligned output is refused
    # before anything is launched
    assert spire.spire_test_draft_slots(None, 0, 4, 64, 0) == 0
    assert spire.spire_test_draft_slots(None, 10, 4, 64, 0) == 1
    assert spire.spire_test_draft_slots(1 << 20, -1, 4, 64, 0) == 1
    assert spire.spire_test_draft_slots((1 << 20) + 4, 10, 4, 64, 0) == 1


def test_stall_hook_host_checks(spire):
    # the hook arms nothing for an invalid pair
    assert spire.spire_test_stall_next_call(-1) == 1
