"""Python binding of liblsp (include/lsp.h): argument marshalling only.

Every function here has the name of the C entry point it calls and does no
computation of its own: tensors are passed as raw device pointers, structs are
mirrored with ctypes, and a non-zero status raises LspError.  The library must
have been built (paper_2609_37029_gb300.build); importing this module without
it fails loudly -- there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import (POINTER, Structure, c_char_p, c_float, c_int, c_size_t, c_uint32, c_uint64,
                    c_void_p)

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "liblsp.so")

LSP_MAX_DRAFT_LAYERS = 16
LSP_OK, LSP_ERR_ARG, LSP_ERR_SHAPE, LSP_ERR_CUDA = 0, -1, -2, -3
LSP_ERR_TIMEOUT, LSP_ERR_STATE, LSP_ERR_NOMEM, LSP_ERR_UNSUPPORTED = -4, -5, -6, -7
LSP_DEV_TIMEOUT, LSP_DEV_BAD_TOKEN, LSP_DEV_BAD_DELTA = 1, 2, 4
LSP_NO_BOUNDARY = 1
LSP_DTYPE_BF16, LSP_DTYPE_F32 = 0, 1

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it with `python -m paper_2609_37029_gb300.build`"
                      " (the CUDA library is required; there is no CPU path)")
_lib = ctypes.CDLL(LIB_PATH)


class lsp_config(Structure):
    _fields_ = [(n, c_int) for n in "C B L D H nq nkv d F V W R rc dtype".split()] + [
        ("layer_map", c_int * LSP_MAX_DRAFT_LAYERS), ("rope_theta", c_float), ("rms_eps", c_float),
        ("flags", c_uint32)]


class lsp_target_feats(Structure):
    _fields_ = [("k", c_void_p), ("v", c_void_p), ("h", c_void_p), ("rows", c_int), ("h_rows", c_int)]


_LAYER_FIELDS = ["in_norm", "wq", "wk", "wv", "q_norm", "k_norm", "wo", "post_norm", "w_gate",
                 "w_up", "w_down"]
_TOP_FIELDS = ["embed", "final_norm", "lm_head", "fuse", "pos", "mask_emb", "Ec", "Wc"]


class lsp_layer_weights(Structure):
    _fields_ = [(n, c_void_p) for n in _LAYER_FIELDS]


class lsp_weights(Structure):
    _fields_ = [(n, c_void_p) for n in _TOP_FIELDS] + [
        ("layer", lsp_layer_weights * LSP_MAX_DRAFT_LAYERS)]


class lsp_sample_params(Structure):
    _fields_ = [("temperature", c_float), ("round", c_uint32), ("seed", c_uint64)]


class LspError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {lsp_status_string(status)} ({status})")


def _sig(name, res, *args):
    f = getattr(_lib, name)
    f.restype = res
    f.argtypes = list(args)
    return f


_f = {
    "lsp_status_string": _sig("lsp_status_string", c_char_p, c_int),
    "lsp_state_bytes": _sig("lsp_state_bytes", c_size_t, POINTER(lsp_config)),
    "lsp_config_check": _sig("lsp_config_check", c_int, POINTER(lsp_config)),
    "lsp_state_create": _sig("lsp_state_create", c_int, POINTER(lsp_config), POINTER(c_void_p)),
    "lsp_state_destroy": _sig("lsp_state_destroy", None, c_void_p),
    "lsp_state_init": _sig("lsp_state_init", c_int, c_void_p, c_void_p, c_void_p),
    "lsp_view_update": _sig("lsp_view_update", c_int, c_void_p, POINTER(lsp_target_feats), c_void_p,
                            c_void_p),
    "lsp_prefill": _sig("lsp_prefill", c_int, c_void_p, c_int, POINTER(lsp_target_feats), c_void_p),
    "lsp_verify": _sig("lsp_verify", c_int, c_void_p, c_void_p, c_void_p, c_void_p,
                       POINTER(lsp_sample_params), c_void_p, c_void_p, c_void_p),
    "lsp_draft": _sig("lsp_draft", c_int, c_void_p, c_void_p, POINTER(lsp_weights),
                      POINTER(lsp_sample_params), c_void_p, c_void_p, c_void_p),
    "lsp_sample": _sig("lsp_sample", c_int, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                       POINTER(lsp_sample_params), c_void_p, c_void_p, c_void_p),
    "lsp_sample_noalloc": _sig("lsp_sample_noalloc", c_int, c_void_p, c_void_p, c_void_p, c_void_p,
                               c_int, c_int, c_int, c_int, c_int, POINTER(lsp_sample_params),
                               c_void_p, c_void_p, c_void_p, c_void_p),
    "lsp_linear_workspace_bytes": _sig("lsp_linear_workspace_bytes", c_size_t, c_int, c_int, c_int),
    "lsp_gemm_plan_info": _sig("lsp_gemm_plan_info", c_int, c_int, c_int, c_int, c_int, c_int, c_int,
                               POINTER(c_int), POINTER(c_int), POINTER(c_int)),
    "lsp_linear": _sig("lsp_linear", c_int, c_void_p, c_void_p, c_void_p, c_int, c_int, c_int, c_int,
                       c_int, c_void_p, c_size_t, c_void_p),
    "lsp_philox_words": _sig("lsp_philox_words", c_int, c_uint64, c_uint32, c_uint32, c_uint32,
                             c_void_p, c_int, c_void_p),
    "lsp_get_error": _sig("lsp_get_error", c_int, c_void_p, POINTER(c_uint32), c_int, c_void_p),
    "lsp_stage_count": _sig("lsp_stage_count", c_int, c_void_p),
    "lsp_round_launches": _sig("lsp_round_launches", c_int, c_void_p),
    "lsp_stage_name": _sig("lsp_stage_name", c_char_p, c_void_p, c_int),
    "lsp_set_stage_events": _sig("lsp_set_stage_events", c_int, c_void_p, POINTER(c_void_p), c_int),
    "lsp_state_export": _sig("lsp_state_export", c_int, c_void_p, c_void_p, c_size_t, c_void_p),
    "lsp_state_import": _sig("lsp_state_import", c_int, c_void_p, c_void_p, c_size_t, c_void_p),
}


def _ptr(x):
    """Device/host address of a tensor (or an int address, or None)."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return stream if isinstance(stream, int) else stream.cuda_stream


def _check(rc, where):
    if rc != LSP_OK:
        raise LspError(rc, where)


# ------------------------------------------------------------------ struct builders
def make_config(shape) -> lsp_config:
    """lsp_config from any object with the shape fields (e.g. synth.LspShape)."""
    c = lsp_config()
    for n in "C B L D H nq nkv d F V W R rc".split():
        setattr(c, n, int(getattr(shape, n)))
    c.dtype = LSP_DTYPE_BF16 if shape.dtype == "bf16" else LSP_DTYPE_F32
    lm = list(getattr(shape, "layer_map", ()) or ())
    for j in range(LSP_MAX_DRAFT_LAYERS):
        c.layer_map[j] = int(lm[j]) if j < len(lm) else -1
    c.rope_theta = float(shape.rope_theta)
    c.rms_eps = float(shape.rms_eps)
    c.flags = LSP_NO_BOUNDARY if getattr(shape, "no_boundary", False) else 0
    return c


def make_weights(w: dict) -> lsp_weights:
    """lsp_weights of device pointers from a dict of tensors (synth.make_weights layout)."""
    s = lsp_weights()
    for n in _TOP_FIELDS:
        setattr(s, n, _ptr(w[n]))
    for j, lw in enumerate(w["layers"]):
        for n in _LAYER_FIELDS:
            setattr(s.layer[j], n, _ptr(lw[n]))
    return s


def make_sample_params(temperature=0.0, seed=0, rnd=0) -> lsp_sample_params:
    return lsp_sample_params(float(temperature), int(rnd) & 0xFFFFFFFF, int(seed) & (2 ** 64 - 1))


# ------------------------------------------------------------------ entry points
def lsp_status_string(status: int) -> str:
    return _f["lsp_status_string"](status).decode()


def lsp_config_check(cfg: lsp_config) -> int:
    return _f["lsp_config_check"](ctypes.byref(cfg))


def lsp_state_bytes(cfg: lsp_config) -> int:
    return _f["lsp_state_bytes"](ctypes.byref(cfg))


def lsp_state_create(cfg: lsp_config) -> int:
    h = c_void_p()
    _check(_f["lsp_state_create"](ctypes.byref(cfg), ctypes.byref(h)), "lsp_state_create")
    return h.value


def lsp_state_destroy(st) -> None:
    _f["lsp_state_destroy"](st)


def lsp_state_init(st, G, stream=None) -> None:
    _check(_f["lsp_state_init"](st, _ptr(G), _stream(stream)), "lsp_state_init")


def lsp_view_update(st, k, v, h, accepted_len, rows=None, stream=None, h_rows=0) -> None:
    """h_rows = 1: h is [C][L][1][H], the hidden state of each request's last new row only."""
    f = lsp_target_feats(_ptr(k), _ptr(v), _ptr(h), int(rows if rows is not None else k.shape[2]), int(h_rows))
    _check(_f["lsp_view_update"](st, ctypes.byref(f), _ptr(accepted_len), _stream(stream)),
           "lsp_view_update")


def lsp_prefill(st, b, k, v, h, rows=None, stream=None, h_rows=0) -> None:
    """k, v: [L][t][nkv][d], h: [L][t][H] of request b's whole prefix ([L][1][H], the last
    row only, with h_rows = 1)."""
    f = lsp_target_feats(_ptr(k), _ptr(v), _ptr(h), int(rows if rows is not None else k.shape[1]),
                         int(h_rows))
    _check(_f["lsp_prefill"](st, int(b), ctypes.byref(f), _stream(stream)), "lsp_prefill")


def lsp_verify(st, target_logits, draft_logits, draft_tokens, sp: lsp_sample_params, accepted_len,
               next_token, stream=None) -> None:
    _check(_f["lsp_verify"](st, _ptr(target_logits), _ptr(draft_logits), _ptr(draft_tokens),
                            ctypes.byref(sp), _ptr(accepted_len), _ptr(next_token), _stream(stream)),
           "lsp_verify")


def lsp_draft(st, block_tokens, weights: lsp_weights, sp: lsp_sample_params, out_tokens,
              out_logits=None, stream=None) -> None:
    _check(_f["lsp_draft"](st, _ptr(block_tokens), ctypes.byref(weights), ctypes.byref(sp),
                           _ptr(out_tokens), _ptr(out_logits), _stream(stream)), "lsp_draft")


def lsp_sample(st, base_logits, prev_token, Ec, Wc, sp: lsp_sample_params, out_tokens,
               out_logits=None, stream=None) -> None:
    _check(_f["lsp_sample"](st, _ptr(base_logits), _ptr(prev_token), _ptr(Ec), _ptr(Wc),
                            ctypes.byref(sp), _ptr(out_tokens), _ptr(out_logits), _stream(stream)),
           "lsp_sample")


def lsp_sample_noalloc(base_logits, prev_token, Ec, Wc, dtype, C, B, V, rc,
                       sp: lsp_sample_params, out_tokens, out_logits=None, dev_error=None,
                       stream=None) -> None:
    _check(_f["lsp_sample_noalloc"](_ptr(base_logits), _ptr(prev_token), _ptr(Ec), _ptr(Wc), dtype,
                                    C, B, V, rc, ctypes.byref(sp), _ptr(out_tokens),
                                    _ptr(out_logits), _ptr(dev_error), _stream(stream)),
           "lsp_sample_noalloc")


def lsp_linear_workspace_bytes(M: int, N: int, splits: int) -> int:
    return _f["lsp_linear_workspace_bytes"](M, N, splits)


def lsp_gemm_plan_info(dtype, M, N, K, swiglu, num_sms):
    """(splits, token groups, token rows per group) of the projection GEMM's plan (host only)."""
    s, g, r = c_int(0), c_int(0), c_int(0)
    _check(_f["lsp_gemm_plan_info"](dtype, M, N, K, int(bool(swiglu)), num_sms, ctypes.byref(s),
                                    ctypes.byref(g), ctypes.byref(r)), "lsp_gemm_plan_info")
    return s.value, g.value, r.value


def lsp_linear(X, W, Y, M, N, K, dtype, splits=1, workspace=None, workspace_bytes=0,
               stream=None) -> None:
    _check(_f["lsp_linear"](_ptr(X), _ptr(W), _ptr(Y), M, N, K, dtype, splits, _ptr(workspace),
                            workspace_bytes, _stream(stream)), "lsp_linear")


def lsp_philox_words(seed, rnd, b, i, out, count, stream=None) -> None:
    _check(_f["lsp_philox_words"](int(seed) & (2 ** 64 - 1), int(rnd), int(b), int(i), _ptr(out),
                                  int(count), _stream(stream)), "lsp_philox_words")


def lsp_get_error(st, clear=True, stream=None):
    """(status, LSP_DEV_* bits) of the state's device error word."""
    bits = c_uint32(0)
    rc = _f["lsp_get_error"](st, ctypes.byref(bits), 1 if clear else 0, _stream(stream))
    return rc, bits.value


def lsp_round_launches(st) -> int:
    return _f["lsp_round_launches"](st)


def lsp_stage_count(st) -> int:
    return _f["lsp_stage_count"](st)


def lsp_stage_name(st, k: int) -> str:
    r = _f["lsp_stage_name"](st, k)
    return r.decode() if r else ""


def lsp_set_stage_events(st, events) -> None:
    """events: a list of torch.cuda.Event(enable_timing=True) (or raw handles); [] turns it off."""
    handles = [e.cuda_event if hasattr(e, "cuda_event") else int(e) for e in events]
    for e in events:
        if hasattr(e, "cuda_event") and e.cuda_event == 0:
            raise ValueError("create each torch.cuda.Event before passing it (record it once)")
    arr = (c_void_p * max(1, len(handles)))(*handles)
    _check(_f["lsp_set_stage_events"](st, arr, len(handles)), "lsp_set_stage_events")


def lsp_state_export(st, host_buf, stream=None) -> None:
    _check(_f["lsp_state_export"](st, _ptr(host_buf), host_buf.numel() * host_buf.element_size(),
                                  _stream(stream)), "lsp_state_export")


def lsp_state_import(st, host_buf, stream=None) -> None:
    _check(_f["lsp_state_import"](st, _ptr(host_buf), host_buf.numel() * host_buf.element_size(),
                                  _stream(stream)), "lsp_state_import")


EXPORTED = sorted(_f)
