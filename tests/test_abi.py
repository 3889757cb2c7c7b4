"""The C-ABI library builds, loads without a GPU, and exports every entry point
include/wf.h declares; the binding's signature table covers the same set."""
import ctypes
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "wf.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(wf_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared()
    for must in ("wf_create", "wf_prefill_cross_kv", "wf_draft", "wf_verify_accept", "wf_step",
                 "wf_greedy_step", "wf_workspace_bytes", "wf_destroy", "wf_get_state"):
        assert must in names


def test_library_exports_every_declared_symbol():
    from paper_2609_32869_gb300 import build
    path = build.build()
    lib = ctypes.CDLL(path)
    missing = [n for n in _declared() if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_covers_the_header():
    from paper_2609_32869_gb300 import binding
    assert sorted(binding.EXPORTED) == _declared()


def test_host_validation_without_gpu():
    """Argument checks run on the host and need no device."""
    from paper_2609_32869_gb300 import binding as B
    from paper_2609_32869_gb300 import synthetic as syn
    cfg = B.make_config(syn.LARGE)
    n = B.wf_workspace_bytes(cfg, 1, 448)
    assert n > 2 * 32 * 448 * 1280 * 2          # at least the target's key/value cache
    bad = B.make_config(syn.LARGE)
    bad.n_heads = 7                              # head_dim would not be 64
    try:
        B.wf_workspace_bytes(bad, 1, 448)
        raise AssertionError("expected failure")
    except B.WfError as e:
        assert e.status == B.WF_ERR_UNSUPPORTED
    try:
        B.wf_workspace_bytes(cfg, 1, 449)           # beyond the learned positions
        raise AssertionError("expected failure")
    except B.WfError as e:
        assert e.status == B.WF_ERR_INVALID
    assert B.wf_gemm_scratch_bytes(9, 1280, 1000) == 0   # K not a multiple of 64


def test_null_handle_is_rejected_on_the_host():
    """Every call that takes a handle checks it before touching the device."""
    from paper_2609_32869_gb300 import binding as B
    lib = B.lib()
    sp = B.WfSampleParams()
    calls = {
        "wf_destroy": (None,),
        "wf_prefill_cross_kv": (None, 1, None, None, None, 4, None, None, None, None),
        "wf_draft": (None, None, None),
        "wf_verify_accept": (None, None, None, None, None, None, None),
        "wf_step": (None, None, None, None, None, None, None),
        "wf_greedy_step": (None, None, None, None, None),
        "wf_compact": (None, None, None),
        "wf_reset_slots": (None, 1, None, None),
        "wf_get_state": (None, None, None, None, None, None),
        "wf_get_error": (None, None, 0, None),
        "wf_set_option": (None, B.WF_OPT_PERSIST, 1),
        "wf_debug_view": (None, 1, None, None),
        "wf_profile_read": (None, None, None, None, None),
    }
    for name, args in calls.items():
        assert getattr(lib, name)(*args) == B.WF_ERR_INVALID, name
    # with a (non-null) sampling-parameter block the answer is the same
    assert lib.wf_draft(None, ctypes.byref(sp), None) == B.WF_ERR_INVALID


def test_status_strings_are_distinct():
    from paper_2609_32869_gb300 import binding as B
    lib = B.lib()
    codes = (B.WF_OK, B.WF_ERR_INVALID, B.WF_ERR_CAPACITY, B.WF_ERR_CUDA, B.WF_ERR_UNSUPPORTED,
             B.WF_ERR_DEVICE)
    texts = [lib.wf_status_str(c) for c in codes]
    assert all(t for t in texts) and len(set(texts)) == len(codes)


def test_workspace_grows_with_batch_and_context():
    """The caller-owned workspace holds per-slot caches: a second slot adds at
    least one slot's target key/value cache and acoustic keys/values."""
    from paper_2609_32869_gb300 import binding as B
    from paper_2609_32869_gb300 import synthetic as syn
    cfg = B.make_config(syn.LARGE)
    one, two = B.wf_workspace_bytes(cfg, 1, 448), B.wf_workspace_bytes(cfg, 2, 448)
    d, layers, frames = 1280, 32, 1500
    per_slot = 2 * layers * 448 * d * 2 + 2 * layers * frames * d * 2
    assert two - one >= per_slot
    assert B.wf_workspace_bytes(cfg, 1, 200) < one


def test_binding_constants_equal_the_header():
    """Every numeric #define and status code of include/wf.h that the binding
    names has the header's value (options, views, error bits, families)."""
    from paper_2609_32869_gb300 import binding as B
    src = open(os.path.join(ROOT, "include", "wf.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    values = {m.group(1): int(m.group(2), 0)
              for m in re.finditer(r"#define\s+(WF_[A-Z0-9_]+)\s+(0x[0-9a-fA-F]+|\d+)u?\b", src)}
    values.update({m.group(1): int(m.group(2)) for m in re.finditer(r"\b(WF_[A-Z_]+)\s*=\s*(\d+)", src)})
    assert len(values) >= 20
    named = {k: v for k, v in values.items() if hasattr(B, k)}
    assert {"WF_OPT_SKINNY", "WF_DEV_ERR_TIMEOUT", "WF_DEV_ERR_LAUNCH", "WF_ERR_CUDA"} <= set(named)
    for k, v in named.items():
        assert getattr(B, k) == v, k
