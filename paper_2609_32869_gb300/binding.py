"""ctypes binding of libwf.so (include/wf.h): argument marshalling only.

Every function below calls the C entry point of the same name; all compute
runs in the library's CUDA kernels.  PyTorch provides device memory and
streams.  Importing this module loads nothing; the first call loads
libwf.so and raises if it is missing (there is no CPU fallback).
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libwf.so")
_lib = None

WF_OK, WF_ERR_INVALID, WF_ERR_CAPACITY, WF_ERR_CUDA, WF_ERR_UNSUPPORTED, WF_ERR_DEVICE = range(6)
WF_DEV_ERR_TIMEOUT, WF_DEV_ERR_CAPACITY, WF_DEV_ERR_TOKEN, WF_DEV_ERR_LAUNCH = 1, 2, 4, 8
WF_MAX_TAPS = 8
WF_OPT_KEEP_LOGITS = 1
WF_OPT_PROFILE = 2
WF_OPT_GRAPHS = 3
WF_OPT_PDL = 4
WF_OPT_PERSIST = 5
WF_OPT_SPIN_LIMIT = 6
WF_OPT_SKINNY = 7
WF_FAMILIES = ("gemm", "head", "attn_self", "attn_cross", "layernorm", "other", "persist")
WF_VIEW_TARGET_LOGITS, WF_VIEW_DRAFT_LOGITS, WF_VIEW_TAPS, WF_VIEW_CANDIDATES = 1, 2, 3, 4


class WfError(RuntimeError):
    def __init__(self, fn, status):
        super().__init__(f"{fn} failed: {status_str(status)} ({status})")
        self.status = status


class WfConfig(C.Structure):
    _fields_ = [("d_model", C.c_int32), ("n_heads", C.c_int32), ("d_ff", C.c_int32),
                ("n_layers", C.c_int32), ("vocab", C.c_int32), ("max_pos", C.c_int32),
                ("enc_frames", C.c_int32), ("n_draft_layers", C.c_int32), ("block_k", C.c_int32),
                ("n_taps", C.c_int32), ("taps", C.c_int32 * WF_MAX_TAPS), ("eos_id", C.c_int32),
                ("rope_base", C.c_float), ("ln_eps", C.c_float)]


_LAYER_FIELDS = ("ln1_g", "ln1_b", "qkv_w", "qkv_b", "out_w", "out_b", "ln2_g", "ln2_b",
                 "xq_w", "xq_b", "xkv_w", "xkv_b", "xout_w", "xout_b", "ln3_g", "ln3_b",
                 "fc1_w", "fc1_b", "fc2_w", "fc2_b")


class WfLayerWeights(C.Structure):
    _fields_ = [(f, C.c_void_p) for f in _LAYER_FIELDS]


class WfTargetWeights(C.Structure):
    _fields_ = [("tok_emb", C.c_void_p), ("pos_emb", C.c_void_p), ("lnf_g", C.c_void_p),
                ("lnf_b", C.c_void_p), ("layers", C.POINTER(WfLayerWeights))]


class WfDrafterWeights(C.Structure):
    _fields_ = [("layers", C.POINTER(WfLayerWeights)), ("proj_w", C.c_void_p),
                ("proj_b", C.c_void_p), ("hln_g", C.c_void_p), ("hln_b", C.c_void_p),
                ("mask_emb", C.c_void_p)]


class WfSampleParams(C.Structure):
    _fields_ = [("temperature", C.c_float), ("_pad", C.c_uint32), ("seed", C.c_uint64),
                ("d_suppress", C.c_void_p)]


_P = C.c_void_p
_I = C.c_int32
_SZ = C.c_size_t
_SIGS = {
    "wf_workspace_bytes": (_I, [C.POINTER(WfConfig), _I, _I, C.POINTER(_SZ)]),
    "wf_create": (_I, [C.POINTER(WfConfig), C.POINTER(WfTargetWeights), C.POINTER(WfDrafterWeights),
                       _I, _I, _P, _SZ, _P, C.POINTER(_P)]),
    "wf_destroy": (_I, [_P]),
    "wf_prefill_cross_kv": (_I, [_P, _I, _P, _P, _P, _I, _P, _P, C.POINTER(WfSampleParams), _P]),
    "wf_draft": (_I, [_P, C.POINTER(WfSampleParams), _P]),
    "wf_verify_accept": (_I, [_P, C.POINTER(WfSampleParams), _P, _P, _P, _P, _P]),
    "wf_step": (_I, [_P, C.POINTER(WfSampleParams), _P, _P, _P, _P, _P]),
    "wf_greedy_step": (_I, [_P, C.POINTER(WfSampleParams), _P, _P, _P]),
    "wf_compact": (_I, [_P, _P, C.POINTER(_I)]),
    "wf_reset_slots": (_I, [_P, _I, _P, _P]),
    "wf_get_state": (_I, [_P, _P, _P, _P, _P, _P]),
    "wf_get_error": (_I, [_P, C.POINTER(C.c_uint32), _I, _P]),
    "wf_last_launch_count": (_I, [_P]),
    "wf_set_option": (_I, [_P, _I, _I]),
    "wf_debug_view": (_I, [_P, _I, C.POINTER(_P), C.POINTER(_SZ)]),
    "wf_profile_read": (_I, [_P, _P, _P, _P, _P]),
    "wf_status_str": (C.c_char_p, [_I]),
    "wf_gemm_bf16": (_I, [_P, _P, _P, _P, _I, _I, _I, _P, _SZ, _P]),
    "wf_gemm_scratch_bytes": (_SZ, [_I, _I, _I]),
    "wf_attention": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, C.c_float, _P, _P, _SZ, _P]),
    "wf_attention_scratch_bytes": (_SZ, [_I, _I, _I, _I]),
    "wf_attention_noalloc": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, C.c_float, _P, _P]),
}
EXPORTED = tuple(_SIGS)


def lib():
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"libwf.so not built ({_LIB_PATH}); run "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        handle = C.CDLL(_LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(handle, name)
            fn.restype = res
            fn.argtypes = args
        _lib = handle
    return _lib


def status_str(status: int) -> str:
    return lib().wf_status_str(int(status)).decode()


def _check(name, status):
    if status != WF_OK:
        raise WfError(name, status)


def _ptr(t):
    """Device pointer of a torch tensor (or an int / None)."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# ------------------------------------------------------------ structs ----
def make_config(cfg) -> WfConfig:
    c = WfConfig()
    c.d_model, c.n_heads, c.d_ff, c.n_layers = cfg.d_model, cfg.n_heads, cfg.d_ff, cfg.n_layers
    c.vocab, c.max_pos, c.enc_frames = cfg.vocab, cfg.max_pos, cfg.enc_frames
    c.n_draft_layers, c.block_k, c.n_taps = cfg.n_draft_layers, cfg.block_k, len(cfg.taps)
    for i, t in enumerate(cfg.taps):
        c.taps[i] = t
    c.eos_id, c.rope_base, c.ln_eps = cfg.eos_id, cfg.rope_base, cfg.ln_eps
    return c


def sample_params(temperature: float = 0.0, seed: int = 0, suppress=None) -> WfSampleParams:
    sp = WfSampleParams()
    sp.temperature = float(temperature)
    sp.seed = int(seed) & 0xFFFFFFFFFFFFFFFF
    sp.d_suppress = _ptr(suppress)
    return sp


def _layer_struct(tensors: dict) -> WfLayerWeights:
    lw = WfLayerWeights()
    for f in _LAYER_FIELDS:
        setattr(lw, f, tensors[f].data_ptr())
    return lw


def weight_structs(dev: dict, n_layers: int, n_draft: int):
    """ctypes structs over device tensors.  `dev` holds 'target', 'target_layers',
    'drafter', 'drafter_layers' (torch bf16 tensors).  The returned tuple keeps
    the layer arrays alive."""
    tl = (WfLayerWeights * n_layers)(*[_layer_struct(x) for x in dev["target_layers"]])
    dl = (WfLayerWeights * n_draft)(*[_layer_struct(x) for x in dev["drafter_layers"]])
    tw = WfTargetWeights()
    t = dev["target"]
    tw.tok_emb, tw.pos_emb = t["tok_emb"].data_ptr(), t["pos_emb"].data_ptr()
    tw.lnf_g, tw.lnf_b = t["lnf_g"].data_ptr(), t["lnf_b"].data_ptr()
    tw.layers = C.cast(tl, C.POINTER(WfLayerWeights))
    dw = WfDrafterWeights()
    dd = dev["drafter"]
    dw.layers = C.cast(dl, C.POINTER(WfLayerWeights))
    dw.proj_w, dw.proj_b = dd["proj_w"].data_ptr(), dd["proj_b"].data_ptr()
    dw.hln_g, dw.hln_b = dd["hln_g"].data_ptr(), dd["hln_b"].data_ptr()
    dw.mask_emb = dd["mask_emb"].data_ptr()
    return tw, dw, tl, dl


# --------------------------------------------------------- entry points --
def wf_workspace_bytes(cfg: WfConfig, max_batch: int, max_ctx: int) -> int:
    out = C.c_size_t(0)
    _check("wf_workspace_bytes", lib().wf_workspace_bytes(C.byref(cfg), max_batch, max_ctx,
                                                          C.byref(out)))
    return out.value


def wf_create(cfg: WfConfig, tw, dw, max_batch, max_ctx, workspace, workspace_bytes, stream=None):
    h = C.c_void_p()
    _check("wf_create", lib().wf_create(C.byref(cfg), C.byref(tw), C.byref(dw), max_batch, max_ctx,
                                        _ptr(workspace), workspace_bytes, _stream(stream),
                                        C.byref(h)))
    return h.value


def wf_destroy(h):
    _check("wf_destroy", lib().wf_destroy(h))


def wf_prefill_cross_kv(h, n, slots, enc, prompt, P, budget, first, sp=None, stream=None):
    _check("wf_prefill_cross_kv", lib().wf_prefill_cross_kv(
        h, n, _ptr(slots), _ptr(enc), _ptr(prompt), P, _ptr(budget), _ptr(first),
        C.byref(sp) if sp is not None else None, _stream(stream)))


def wf_draft(h, sp=None, stream=None):
    _check("wf_draft", lib().wf_draft(h, C.byref(sp) if sp is not None else None, _stream(stream)))


def wf_verify_accept(h, sp, forced, forced_q, out_tokens, out_count, stream=None):
    _check("wf_verify_accept", lib().wf_verify_accept(
        h, C.byref(sp) if sp is not None else None, _ptr(forced), _ptr(forced_q),
        _ptr(out_tokens), _ptr(out_count), _stream(stream)))


def wf_step(h, sp, forced, forced_q, out_tokens, out_count, stream=None):
    _check("wf_step", lib().wf_step(h, C.byref(sp) if sp is not None else None, _ptr(forced),
                                    _ptr(forced_q), _ptr(out_tokens), _ptr(out_count),
                                    _stream(stream)))


def wf_greedy_step(h, sp, out_tokens, out_count, stream=None):
    _check("wf_greedy_step", lib().wf_greedy_step(h, C.byref(sp) if sp is not None else None,
                                                  _ptr(out_tokens), _ptr(out_count),
                                                  _stream(stream)))


def wf_compact(h, stream=None) -> int:
    n = C.c_int32(0)
    _check("wf_compact", lib().wf_compact(h, _stream(stream), C.byref(n)))
    return n.value


def wf_reset_slots(h, n, slots, stream=None):
    _check("wf_reset_slots", lib().wf_reset_slots(h, n, _ptr(slots), _stream(stream)))


def wf_get_state(h, max_batch, stream=None):
    arrs = [np.zeros(max_batch, np.int32) for _ in range(4)]
    _check("wf_get_state", lib().wf_get_state(h, *[a.ctypes.data for a in arrs], _stream(stream)))
    return dict(zip(("len", "anchor", "remaining", "done"), arrs))


def wf_get_error(h, clear=False, stream=None) -> int:
    e = C.c_uint32(0)
    _check("wf_get_error", lib().wf_get_error(h, C.byref(e), int(clear), _stream(stream)))
    return e.value


def wf_last_launch_count(h) -> int:
    return lib().wf_last_launch_count(h)


def wf_set_option(h, option, value):
    _check("wf_set_option", lib().wf_set_option(h, option, value))


def wf_debug_view(h, which):
    p, n = C.c_void_p(), C.c_size_t()
    _check("wf_debug_view", lib().wf_debug_view(h, which, C.byref(p), C.byref(n)))
    return p.value, n.value


def wf_profile_read(h, stream=None) -> dict:
    n = len(WF_FAMILIES)
    ms, cnt, by = np.zeros(n), np.zeros(n, np.int32), np.zeros(n)
    _check("wf_profile_read", lib().wf_profile_read(h, _stream(stream), ms.ctypes.data,
                                                    cnt.ctypes.data, by.ctypes.data))
    return {f: {"ms": float(ms[i]), "launches": int(cnt[i]), "bytes": float(by[i])}
            for i, f in enumerate(WF_FAMILIES)}


def wf_gemm_scratch_bytes(M, N, K) -> int:
    return lib().wf_gemm_scratch_bytes(M, N, K)


def wf_gemm_bf16(x, w, b, y, M, N, K, scratch, scratch_bytes, stream=None):
    _check("wf_gemm_bf16", lib().wf_gemm_bf16(_ptr(x), _ptr(w), _ptr(b), _ptr(y), M, N, K,
                                              _ptr(scratch), scratch_bytes, _stream(stream)))


def wf_attention_scratch_bytes(n_seq, rps, n_heads, ctx) -> int:
    return lib().wf_attention_scratch_bytes(n_seq, rps, n_heads, ctx)


def wf_attention(q, kc, vc, slot, base, n_seq, rps, n_heads, ctx, mode, rope, rope_base, out,
                 scratch, scratch_bytes, stream=None):
    _check("wf_attention", lib().wf_attention(
        _ptr(q), _ptr(kc), _ptr(vc), _ptr(slot), _ptr(base), n_seq, rps, n_heads, ctx, mode,
        int(rope), float(rope_base), _ptr(out), _ptr(scratch), scratch_bytes, _stream(stream)))


def wf_attention_noalloc(q, kc, vc, slot, base, n_seq, rps, n_heads, ctx, mode, rope, rope_base,
                         out, stream=None):
    _check("wf_attention_noalloc", lib().wf_attention_noalloc(
        _ptr(q), _ptr(kc), _ptr(vc), _ptr(slot), _ptr(base), n_seq, rps, n_heads, ctx, mode,
        int(rope), float(rope_base), _ptr(out), _stream(stream)))
