"""Thin ctypes binding of libalr (include/alr.h).

The ``alr_*`` functions here carry the C names and only marshal arguments: torch tensors
become device pointers, the current torch CUDA stream becomes the ``stream`` argument, and
a non-zero status becomes an :class:`AlrError`.  Every computation runs in the CUDA library;
if ``_lib/libalr.so`` is missing, loading raises instead of falling back to anything else.

``SlotLoss`` is a convenience owner of the output and workspace tensors for repeated calls.
"""

from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib", "libalr.so")

ALR_OK, ALR_ERR_INVALID_ARG, ALR_ERR_UNSUPPORTED, ALR_ERR_CUDA, ALR_ERR_TIMEOUT = range(5)
ALR_BF16, ALR_F32 = 0, 1
ALR_MODE_ALR, ALR_MODE_ERASE_SOFT, ALR_MODE_ERASE_HARD = 0, 1, 2

_c_int, _c_i32, _c_i64, _c_f, _c_p, _c_sz = (ctypes.c_int, ctypes.c_int32, ctypes.c_int64,
                                            ctypes.c_float, ctypes.c_void_p, ctypes.c_size_t)


class AlrParams(ctypes.Structure):
    _fields_ = [("N", _c_i64), ("d", _c_i32), ("V", _c_i32), ("B", _c_i32), ("dtype", _c_i32),
                ("mode", _c_i32), ("lam", _c_f), ("gamma", _c_f)]


_FWD_FIELDS = ("loss_row", "ent_row", "lse_d", "lse_t", "argmax_d", "argmax_t", "gap_d", "gap_t",
               "logp_x", "weight", "loss_total", "weight_sum", "wl_sum")


class AlrFwdOutputs(ctypes.Structure):
    _fields_ = [(f, _c_p) for f in _FWD_FIELDS]


_TOPK_FIELDS = ("loss_row", "lse_d", "tail_q", "argmax_d", "gap_d", "weight", "loss_total",
                "weight_sum", "wl_sum")
ALR_TOPK = 8


class AlrTopkFwdOutputs(ctypes.Structure):
    _fields_ = [(f, _c_p) for f in _TOPK_FIELDS]


# name -> (restype, argtypes); must match include/alr.h
SIGNATURES = {
    "alr_version": (ctypes.c_char_p, []),
    "alr_last_error": (ctypes.c_char_p, []),
    "alr_device_supported": (_c_int, []),
    "alr_device_status": (_c_int, [_c_p, _c_int]),
    "alr_kernel_forms": (_c_int, [_c_p, _c_p]),
    "alr_cluster_forms_error": (ctypes.c_char_p, []),
    "alr_debug_withhold_next_stage": (_c_int, [_c_int]),
    "alr_gather_ira_blocks": (_c_int, [_c_p, _c_i32, _c_i32, _c_i32, _c_i32, _c_p, _c_p, _c_p,
                                       _c_i32, _c_i32, _c_p, _c_p, _c_p]),
    "alr_fwd_workspace_size": (_c_sz, [ctypes.POINTER(AlrParams)]),
    "alr_slot_loss_fwd": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p, _c_p,
                                   ctypes.POINTER(AlrFwdOutputs), _c_p, _c_sz, _c_p]),
    "alr_slot_loss_fwd_noalloc": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p,
                                           _c_p, ctypes.POINTER(AlrFwdOutputs), _c_p]),
    "alr_bwd_workspace_size": (_c_sz, [ctypes.POINTER(AlrParams)]),
    "alr_slot_loss_bwd": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                                   _c_p, _c_p, _c_p, _c_p, _c_sz, _c_p]),
    "alr_logit_grad_workspace_size": (_c_sz, [ctypes.POINTER(AlrParams)]),
    "alr_logit_grad": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                                _c_p, _c_p, _c_p, _c_sz, _c_p]),
    "alr_kept_ref_groups": (_c_i32, [_c_i32]),
    "alr_slot_loss_fwd_keep_logits": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p,
                                               _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                                               ctypes.POINTER(AlrFwdOutputs), _c_p, _c_sz, _c_p]),
    "alr_logit_grad_from_logits": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p,
                                            _c_p, _c_p, _c_p, _c_p, _c_p, _c_p]),
    "alr_bwd_from_logits_workspace_size": (_c_sz, [ctypes.POINTER(AlrParams)]),
    "alr_slot_loss_bwd_from_logits": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p,
                                               _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                                               _c_p, _c_p, _c_sz, _c_p]),
    "alr_readout_workspace_size": (_c_sz, [ctypes.POINTER(AlrParams)]),
    "alr_label_readout": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                                   _c_p, _c_p, _c_p, _c_p, _c_p, _c_sz, _c_p]),
    "alr_topk_fwd_workspace_size": (_c_sz, [ctypes.POINTER(AlrParams)]),
    "alr_topk_loss_fwd": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                                   _c_p, ctypes.POINTER(AlrTopkFwdOutputs), _c_p, _c_sz, _c_p]),
    "alr_topk_logit_grad": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p, _c_p,
                                     _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_sz, _c_p]),
    "alr_topk_loss_bwd": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                                   _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_sz, _c_p]),
    "alr_topk_loss_fwd_keep_logits": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p,
                                               _c_p, _c_p, _c_p, _c_p, _c_p,
                                               ctypes.POINTER(AlrTopkFwdOutputs), _c_p, _c_sz,
                                               _c_p]),
    "alr_topk_logit_grad_from_logits": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p,
                                                 _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p]),
    "alr_topk_loss_bwd_from_logits": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p,
                                               _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                                               _c_p, _c_p, _c_p, _c_sz, _c_p]),
    "alr_ira_blocks": (_c_int, [_c_i32, _c_i32, _c_i32, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                                _c_p, _c_p, _c_p, _c_p]),
    "alr_loss_from_sums": (_c_int, [_c_p, _c_p, _c_f, _c_p, _c_p]),
    "alr_ira_draw": (_c_int, [_c_i32, _c_i32, _c_i32, _c_i32, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                              _c_p]),
    "alr_ira_context": (_c_int, [_c_p, _c_i32, _c_i32, _c_i32, _c_i32, _c_i32, _c_i32, _c_p, _c_p,
                                 _c_p, _c_p, _c_p, _c_p, _c_p, _c_p]),
    "alr_accept_len": (_c_int, [_c_p, _c_p, _c_p, _c_i32, _c_i32, _c_p, _c_p, _c_p]),
    "alr_erase_weights": (_c_int, [_c_p, _c_p, _c_p, _c_p, _c_i32, _c_i32, _c_f, _c_i32, _c_p,
                                   _c_p]),
    "alr_gemm": (_c_int, [_c_i32, _c_i32, _c_i32, _c_i32, _c_p, _c_p, _c_p, _c_i32, _c_i32,
                          _c_i32, _c_p]),
}


class AlrError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"libalr status {code}: {msg}")
        self.code = code


_lib = None


def lib():
    """Load libalr.so (built in-tree by ``build_lib.build()``); raise if it is absent."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -m paper_2609_38795_gb300.build_lib`")
        h = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(h, name)
            fn.restype, fn.argtypes = res, args
        _lib = h
    return _lib


def _check(rc):
    if rc != ALR_OK:
        raise AlrError(rc, lib().alr_last_error().decode())


_I32, _I64, _F32 = torch.int32, torch.int64, torch.float32


def _ptr(t, name="tensor", numel=None, dtype=None):
    """Device pointer of a tensor argument (None stays NULL), after the checks the C ABI cannot
    make on a bare pointer: a tensor on the current CUDA device, contiguous, of the expected
    element type, holding at least `numel` elements.  A wrong buffer is refused here rather
    than read or written out of bounds by a kernel."""
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name}: expected a torch.Tensor, got {type(t).__name__}")
    if not t.is_cuda or t.device.index != torch.cuda.current_device():
        raise ValueError(f"{name} must be on the current CUDA device (got {t.device})")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype} (got {t.dtype})")
    if numel is not None and t.numel() < numel:
        raise ValueError(f"{name} holds {t.numel()} elements, fewer than the {numel} needed")
    return t.data_ptr()


def _in_dtype(params):
    return torch.bfloat16 if params.dtype == ALR_BF16 else torch.float32


def _logit_dtype(params):
    return torch.float16 if params.dtype == ALR_BF16 else torch.float32


def _fwd_outputs(params, out):
    N = params.N
    spec = dict(loss_row=(N, _F32), ent_row=(N, _F32), lse_d=(N, _F32), lse_t=(N, _F32),
                argmax_d=(N, _I32), argmax_t=(N, _I32), gap_d=(N, _F32), gap_t=(N, _F32),
                logp_x=(N, _F32), weight=(N, _F32), loss_total=(1, _F32), weight_sum=(1, _F32),
                wl_sum=(1, _F32))
    return AlrFwdOutputs(**{f: _ptr(out.get(f), f, *spec[f]) for f in _FWD_FIELDS})


def _topk_outputs(params, out):
    N = params.N
    spec = dict(loss_row=(N, _F32), lse_d=(N, _F32), tail_q=(N, _F32), argmax_d=(N, _I32),
                gap_d=(N, _F32), weight=(N, _F32), loss_total=(1, _F32), weight_sum=(1, _F32),
                wl_sum=(1, _F32))
    return AlrTopkFwdOutputs(**{f: _ptr(out.get(f), f, *spec[f]) for f in _TOPK_FIELDS})


def _ws(ws):
    return _ptr(ws, "workspace")


def _stream(stream=None):
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


def dtype_code(t_dtype) -> int:
    if t_dtype == torch.bfloat16:
        return ALR_BF16
    if t_dtype == torch.float32:
        return ALR_F32
    raise ValueError(f"unsupported dtype {t_dtype}")


def make_params(N, d, V, B, dtype=torch.bfloat16, mode=ALR_MODE_ALR, lam=1.0, gamma=2.0):
    return AlrParams(N=N, d=d, V=V, B=B, dtype=dtype_code(dtype), mode=mode, lam=lam, gamma=gamma)


# ------------------------------------------------------------ C-named entry points ---
def alr_version() -> str:
    return lib().alr_version().decode()


def alr_last_error() -> str:
    return lib().alr_last_error().decode()


def alr_device_supported() -> int:
    return lib().alr_device_supported()


def alr_device_status(clear=True, stream=None) -> int:
    return lib().alr_device_status(_stream(stream), int(clear))


GEMM_FORMS = ("single", "mcast", "pair", "mcast4")
LOSS_FORMS = ("single", "mcast")


def alr_kernel_forms():
    """(GEMM form, loss-kernel form) names the next bf16 call will use in this process."""
    g, l = ctypes.c_int32(), ctypes.c_int32()
    _check(lib().alr_kernel_forms(ctypes.byref(g), ctypes.byref(l)))
    return GEMM_FORMS[g.value], LOSS_FORMS[l.value]


def alr_cluster_forms_error() -> str:
    """"" when libalr_cluster.so (the cluster kernel forms) is loaded in this process, else why
    it is not."""
    return lib().alr_cluster_forms_error().decode()


def alr_debug_withhold_next_stage(enable=True) -> int:
    return lib().alr_debug_withhold_next_stage(int(enable))


def alr_gather_ira_blocks(feat, seq, pos, B, out, row_valid=None, valid_len=None, stream=None):
    S, L, d = feat.shape
    A = seq.numel()
    dt = feat.dtype
    _check(lib().alr_gather_ira_blocks(_ptr(feat, "feat"), S, L, d, dtype_code(dt),
                                       _ptr(seq, "seq", A, _I32), _ptr(pos, "pos", A, _I32),
                                       _ptr(valid_len, "valid_len", A, _I32), A, B,
                                       _ptr(out, "out", A * B * d, dt),
                                       _ptr(row_valid, "row_valid", A * B, _F32),
                                       _stream(stream)))


def alr_fwd_workspace_size(params) -> int:
    return lib().alr_fwd_workspace_size(ctypes.byref(params))


def alr_bwd_workspace_size(params) -> int:
    return lib().alr_bwd_workspace_size(ctypes.byref(params))


def _heads(params, Hd=None, Ht=None, W=None):
    """Pointers of the hidden states [N, d] and the head [d, V] (input element type)."""
    N, d, V, dt = params.N, params.d, params.V, _in_dtype(params)
    return (_ptr(Hd, "Hd", N * d, dt), _ptr(Ht, "Ht", N * d, dt), _ptr(W, "W", d * V, dt))


def alr_slot_loss_fwd(params, Hd, Ht, W, out: dict, workspace, row_mask=None, corpus_tok=None,
                      stream=None):
    N = params.N
    hd, ht, w = _heads(params, Hd, Ht, W)
    o = _fwd_outputs(params, out)
    _check(lib().alr_slot_loss_fwd(ctypes.byref(params), hd, ht, w,
                                   _ptr(row_mask, "row_mask", N, _F32),
                                   _ptr(corpus_tok, "corpus_tok", N, _I32), ctypes.byref(o),
                                   _ws(workspace), _nbytes(workspace), _stream(stream)))


def alr_slot_loss_fwd_noalloc(params, Hd, Ht, W, out: dict, row_mask=None, corpus_tok=None,
                              stream=None):
    """alr_slot_loss_fwd without a workspace (scratch in the library's fixed device array)."""
    N = params.N
    hd, ht, w = _heads(params, Hd, Ht, W)
    o = _fwd_outputs(params, out)
    _check(lib().alr_slot_loss_fwd_noalloc(ctypes.byref(params), hd, ht, w,
                                           _ptr(row_mask, "row_mask", N, _F32),
                                           _ptr(corpus_tok, "corpus_tok", N, _I32),
                                           ctypes.byref(o), _stream(stream)))


def _row_stats(params, weight, weight_sum, lse_d, fourth=None, fourth_name="lse_t"):
    """Pointers of the per-row forward results the backward reads: weight [N], weight_sum [1],
    lse_d [N] and lse_t (full vocabulary) or tail_q (top-k) [N]."""
    N = params.N
    return (_ptr(weight, "weight", N, _F32), _ptr(weight_sum, "weight_sum", 1, _F32),
            _ptr(lse_d, "lse_d", N, _F32), _ptr(fourth, fourth_name, N, _F32))


def _head_grads(params, dHd, dW):
    N, d, V = params.N, params.d, params.V
    return _ptr(dHd, "dHd", N * d, _F32), _ptr(dW, "dW", d * V, _F32)


def alr_slot_loss_bwd(params, Hd, Ht, W, weight, weight_sum, lse_d, lse_t, dHd, dW, workspace,
                      stream=None):
    hd, ht, w = _heads(params, Hd, Ht, W)
    wt, ws_, ld, lt = _row_stats(params, weight, weight_sum, lse_d, lse_t)
    dh, dw = _head_grads(params, dHd, dW)
    _check(lib().alr_slot_loss_bwd(ctypes.byref(params), hd, ht, w, wt, ws_, ld, lt, dh, dw,
                                   _ws(workspace), _nbytes(workspace), _stream(stream)))


def alr_logit_grad_workspace_size(params) -> int:
    return lib().alr_logit_grad_workspace_size(ctypes.byref(params))


def _grad_matrix(params, G):
    return _ptr(G, "G", params.N * params.V, _in_dtype(params))


def alr_logit_grad(params, Hd, Ht, W, weight, weight_sum, lse_d, lse_t, G, workspace=None,
                   stream=None):
    hd, ht, w = _heads(params, Hd, Ht, W)
    wt, ws_, ld, lt = _row_stats(params, weight, weight_sum, lse_d, lse_t)
    _check(lib().alr_logit_grad(ctypes.byref(params), hd, ht, w, wt, ws_, ld, lt,
                                _grad_matrix(params, G), _ws(workspace), _nbytes(workspace),
                                _stream(stream)))


def _nbytes(ws):
    return 0 if ws is None else ws.numel() * ws.element_size()


def logits_dtype(t_dtype):
    """Element type of the kept logits for inputs of type t_dtype."""
    return torch.float16 if t_dtype == torch.bfloat16 else torch.float32


def _logits(params, Z, name):
    return _ptr(Z, name, params.N * params.V, _logit_dtype(params))


def alr_kept_ref_groups(V) -> int:
    """16-column groups of a row of V logits: the leading dimension of a kept-logit
    group-reference array [groups, N]."""
    return lib().alr_kept_ref_groups(int(V))


def _refs(params, R, name):
    """Group references of kept fp16 logits: [alr_kept_ref_groups(V), N] float16 (bf16 inputs);
    fp32 inputs keep plain logits and pass None."""
    if params.dtype != ALR_BF16:
        return _ptr(R, name)
    return _ptr(R, name, params.N * alr_kept_ref_groups(params.V), torch.float16)


def alr_slot_loss_fwd_keep_logits(params, Hd, Ht, W, Zd, Zt, Zd_ref, Zt_ref, out: dict,
                                  workspace, row_mask=None, corpus_tok=None, stream=None):
    N = params.N
    hd, ht, w = _heads(params, Hd, Ht, W)
    o = _fwd_outputs(params, out)
    _check(lib().alr_slot_loss_fwd_keep_logits(ctypes.byref(params), hd, ht, w,
                                               _ptr(row_mask, "row_mask", N, _F32),
                                               _ptr(corpus_tok, "corpus_tok", N, _I32),
                                               _logits(params, Zd, "Zd"), _logits(params, Zt, "Zt"),
                                               _refs(params, Zd_ref, "Zd_ref"),
                                               _refs(params, Zt_ref, "Zt_ref"),
                                               ctypes.byref(o), _ws(workspace),
                                               _nbytes(workspace), _stream(stream)))


def alr_logit_grad_from_logits(params, Zd, Zt, Zd_ref, Zt_ref, weight, weight_sum, lse_d, lse_t, G,
                               stream=None):
    wt, ws_, ld, lt = _row_stats(params, weight, weight_sum, lse_d, lse_t)
    _check(lib().alr_logit_grad_from_logits(ctypes.byref(params), _logits(params, Zd, "Zd"),
                                            _logits(params, Zt, "Zt"),
                                            _refs(params, Zd_ref, "Zd_ref"),
                                            _refs(params, Zt_ref, "Zt_ref"), wt, ws_, ld, lt,
                                            _grad_matrix(params, G), _stream(stream)))


def alr_bwd_from_logits_workspace_size(params) -> int:
    return lib().alr_bwd_from_logits_workspace_size(ctypes.byref(params))


def alr_slot_loss_bwd_from_logits(params, Hd, W, Zd, Zt, Zd_ref, Zt_ref, weight, weight_sum, lse_d,
                                  lse_t, G, dHd, dW, workspace=None, stream=None):
    hd, _, w = _heads(params, Hd, None, W)
    wt, ws_, ld, lt = _row_stats(params, weight, weight_sum, lse_d, lse_t)
    dh, dw = _head_grads(params, dHd, dW)
    _check(lib().alr_slot_loss_bwd_from_logits(ctypes.byref(params), hd, w,
                                               _logits(params, Zd, "Zd"),
                                               _logits(params, Zt, "Zt"),
                                               _refs(params, Zd_ref, "Zd_ref"),
                                               _refs(params, Zt_ref, "Zt_ref"), wt, ws_, ld, lt,
                                               _grad_matrix(params, G), dh, dw, _ws(workspace),
                                               _nbytes(workspace), _stream(stream)))


def alr_readout_workspace_size(params) -> int:
    return lib().alr_readout_workspace_size(ctypes.byref(params))


def alr_label_readout(params, Ht, W, out: dict, workspace, corpus_tok=None, stream=None):
    """out: top_idx [N, 8] int32, top_prob [N, 8], tail [N]; optional lse_t, argmax_t, gap_t,
    logp_x."""
    N, k = params.N, ALR_TOPK
    _, ht, w = _heads(params, None, Ht, W)
    _check(lib().alr_label_readout(ctypes.byref(params), ht, w,
                                   _ptr(corpus_tok, "corpus_tok", N, _I32),
                                   _ptr(out["top_idx"], "top_idx", N * k, _I32),
                                   _ptr(out["top_prob"], "top_prob", N * k, _F32),
                                   _ptr(out["tail"], "tail", N, _F32),
                                   _ptr(out.get("lse_t"), "lse_t", N, _F32),
                                   _ptr(out.get("argmax_t"), "argmax_t", N, _I32),
                                   _ptr(out.get("gap_t"), "gap_t", N, _F32),
                                   _ptr(out.get("logp_x"), "logp_x", N, _F32),
                                   _ws(workspace), _nbytes(workspace), _stream(stream)))


def alr_topk_fwd_workspace_size(params) -> int:
    return lib().alr_topk_fwd_workspace_size(ctypes.byref(params))


def _labels(params, top_idx, top_prob, tail):
    N, k = params.N, ALR_TOPK
    return (_ptr(top_idx, "top_idx", N * k, _I32), _ptr(top_prob, "top_prob", N * k, _F32),
            _ptr(tail, "tail", N, _F32))


def alr_topk_loss_fwd(params, Hd, W, top_idx, top_prob, tail, out: dict, workspace,
                      row_mask=None, weight_in=None, stream=None):
    N = params.N
    hd, _, w = _heads(params, Hd, None, W)
    o = _topk_outputs(params, out)
    _check(lib().alr_topk_loss_fwd(ctypes.byref(params), hd, w,
                                   *_labels(params, top_idx, top_prob, tail),
                                   _ptr(row_mask, "row_mask", N, _F32),
                                   _ptr(weight_in, "weight_in", N, _F32), ctypes.byref(o),
                                   _ws(workspace), _nbytes(workspace), _stream(stream)))


def alr_topk_logit_grad(params, Hd, W, top_idx, top_prob, tail, weight, weight_sum, lse_d,
                        tail_q, G, workspace=None, stream=None):
    hd, _, w = _heads(params, Hd, None, W)
    wt, ws_, ld, tq = _row_stats(params, weight, weight_sum, lse_d, tail_q, "tail_q")
    _check(lib().alr_topk_logit_grad(ctypes.byref(params), hd, w,
                                     *_labels(params, top_idx, top_prob, tail), wt, ws_, ld, tq,
                                     _grad_matrix(params, G), _ws(workspace), _nbytes(workspace),
                                     _stream(stream)))


def alr_topk_loss_bwd(params, Hd, W, top_idx, top_prob, tail, weight, weight_sum, lse_d, tail_q,
                      dHd, dW, workspace, stream=None):
    hd, _, w = _heads(params, Hd, None, W)
    wt, ws_, ld, tq = _row_stats(params, weight, weight_sum, lse_d, tail_q, "tail_q")
    dh, dw = _head_grads(params, dHd, dW)
    _check(lib().alr_topk_loss_bwd(ctypes.byref(params), hd, w,
                                   *_labels(params, top_idx, top_prob, tail), wt, ws_, ld, tq,
                                   dh, dw, _ws(workspace), _nbytes(workspace), _stream(stream)))


def alr_topk_loss_fwd_keep_logits(params, Hd, W, top_idx, top_prob, tail, Zd, Zd_ref, out: dict,
                                  workspace, row_mask=None, weight_in=None, stream=None):
    N = params.N
    hd, _, w = _heads(params, Hd, None, W)
    o = _topk_outputs(params, out)
    _check(lib().alr_topk_loss_fwd_keep_logits(ctypes.byref(params), hd, w,
                                               *_labels(params, top_idx, top_prob, tail),
                                               _ptr(row_mask, "row_mask", N, _F32),
                                               _ptr(weight_in, "weight_in", N, _F32),
                                               _logits(params, Zd, "Zd"),
                                               _refs(params, Zd_ref, "Zd_ref"), ctypes.byref(o),
                                               _ws(workspace), _nbytes(workspace),
                                               _stream(stream)))


def alr_topk_logit_grad_from_logits(params, Zd, Zd_ref, top_idx, top_prob, tail, weight,
                                    weight_sum, lse_d, tail_q, G, stream=None):
    wt, ws_, ld, tq = _row_stats(params, weight, weight_sum, lse_d, tail_q, "tail_q")
    _check(lib().alr_topk_logit_grad_from_logits(ctypes.byref(params), _logits(params, Zd, "Zd"),
                                                 _refs(params, Zd_ref, "Zd_ref"),
                                                 *_labels(params, top_idx, top_prob, tail),
                                                 wt, ws_, ld, tq, _grad_matrix(params, G),
                                                 _stream(stream)))


def alr_topk_loss_bwd_from_logits(params, Hd, W, Zd, Zd_ref, top_idx, top_prob, tail, weight,
                                  weight_sum, lse_d, tail_q, G, dHd, dW, workspace=None,
                                  stream=None):
    hd, _, w = _heads(params, Hd, None, W)
    wt, ws_, ld, tq = _row_stats(params, weight, weight_sum, lse_d, tail_q, "tail_q")
    dh, dw = _head_grads(params, dHd, dW)
    _check(lib().alr_topk_loss_bwd_from_logits(ctypes.byref(params), hd, w,
                                               _logits(params, Zd, "Zd"),
                                               _refs(params, Zd_ref, "Zd_ref"),
                                               *_labels(params, top_idx, top_prob, tail),
                                               wt, ws_, ld, tq, _grad_matrix(params, G), dh, dw,
                                               _ws(workspace), _nbytes(workspace),
                                               _stream(stream)))


def alr_ira_blocks(K, max_blocks, valid_anchors, rollout_len, offsets, out: dict,
                   rollout_tok=None, corpus_anchor_tok=None, stream=None):
    """out: seq, pos, valid_len (int32 [S*max_blocks]); optional ctx_len, anchor_tok."""
    S = valid_anchors.numel()
    half = max_blocks // 2
    P = max_blocks - half
    T = S * max_blocks
    _check(lib().alr_ira_blocks(S, K, max_blocks, _ptr(valid_anchors, "valid_anchors", S, _I32),
                                _ptr(rollout_len, "rollout_len", S * P, _I32),
                                _ptr(offsets, "offsets", S * half, _I32),
                                _ptr(rollout_tok, "rollout_tok", S * P * K, _I32),
                                _ptr(corpus_anchor_tok, "corpus_anchor_tok", T, _I32),
                                _ptr(out["seq"], "seq", T, _I32), _ptr(out["pos"], "pos", T, _I32),
                                _ptr(out["valid_len"], "valid_len", T, _I32),
                                _ptr(out.get("ctx_len"), "ctx_len", T, _I32),
                                _ptr(out.get("anchor_tok"), "anchor_tok", T, _I32),
                                _stream(stream)))


def alr_loss_from_sums(wl_sum, weight_sum, lam, loss_total, stream=None):
    """L = lambda * wl_sum / weight_sum (0 when weight_sum = 0) from reduced sums (one float
    each, on the device)."""
    _check(lib().alr_loss_from_sums(_ptr(wl_sum, "wl_sum", 1, _F32),
                                    _ptr(weight_sum, "weight_sum", 1, _F32), float(lam),
                                    _ptr(loss_total, "loss_total", 1, _F32), _stream(stream)))


def alr_ira_draw(K, max_blocks, anchor_ok, keys, offset_u, out: dict, stream=None):
    """anchor_ok [S, L] uint8, keys [S, L] and offset_u [S, max_blocks // 2] random integers
    (int32 tensors holding the uint32 bits); out: n_valid [S], anchor_pos [S, max_blocks],
    offsets [S, max_blocks // 2] (int32)."""
    S, L = anchor_ok.shape
    H = max_blocks // 2
    _check(lib().alr_ira_draw(S, L, K, max_blocks, _ptr(anchor_ok, "anchor_ok", S * L, torch.uint8),
                              _ptr(keys, "keys", S * L, _I32),
                              _ptr(offset_u, "offset_u", S * H, _I32),
                              _ptr(out["n_valid"], "n_valid", S, _I32),
                              _ptr(out["anchor_pos"], "anchor_pos", S * max_blocks, _I32),
                              _ptr(out["offsets"], "offsets", S * H, _I32), _stream(stream)))


def alr_ira_context(K, max_blocks, store, n_valid, rollout_len, offsets, anchor_pos, ctx,
                    ctx_len=None, prefix_end=None, stream=None):
    """store [S * P, C, F]; ctx [S, max_blocks // 2, C, F] (same dtype)."""
    SP, C, F = store.shape
    H, P = max_blocks // 2, max_blocks - max_blocks // 2
    S = SP // P
    dt = store.dtype
    _check(lib().alr_ira_context(_ptr(store, "store", SP * C * F, dt), C, F, dtype_code(dt), S, K,
                                 max_blocks, _ptr(n_valid, "n_valid", S, _I32),
                                 _ptr(rollout_len, "rollout_len", S * P, _I32),
                                 _ptr(offsets, "offsets", S * H, _I32),
                                 _ptr(anchor_pos, "anchor_pos", S * max_blocks, _I32),
                                 _ptr(ctx, "ctx", S * H * C * F, dt),
                                 _ptr(ctx_len, "ctx_len", S * H, _I32),
                                 _ptr(prefix_end, "prefix_end", S * H, _I32), _stream(stream)))


def _anchors(t, B, name):
    """Anchor count of a per-row tensor of A*B entries."""
    if B < 1 or t.numel() % B != 0:
        raise ValueError(f"{name} holds {t.numel()} rows, not a whole number of anchors of B = {B}")
    return t.numel() // B


def alr_accept_len(argmax_d, argmax_t, B, acc_len, hist=None, active=None, stream=None):
    A = _anchors(argmax_d, B, "argmax_d")
    N = A * B
    _check(lib().alr_accept_len(_ptr(argmax_d, "argmax_d", N, _I32),
                                _ptr(argmax_t, "argmax_t", N, _I32),
                                _ptr(active, "active", N, _F32), A, B,
                                _ptr(acc_len, "acc_len", A, _I32),
                                _ptr(hist, "hist", B + 1, _I64), _stream(stream)))


def alr_erase_weights(B, gamma, hard, weight, logp_x=None, corpus_tok=None, argmax_t=None,
                      row_mask=None, stream=None):
    A = _anchors(weight, B, "weight")
    N = A * B
    _check(lib().alr_erase_weights(_ptr(logp_x, "logp_x", N, _F32),
                                   _ptr(corpus_tok, "corpus_tok", N, _I32),
                                   _ptr(argmax_t, "argmax_t", N, _I32),
                                   _ptr(row_mask, "row_mask", N, _F32), A, B, float(gamma),
                                   int(hard), _ptr(weight, "weight", N, _F32), _stream(stream)))


def alr_gemm(A, B, C, M, Nc, K, a_mn=False, b_mn=False, accumulate=False, stream=None):
    dt = A.dtype
    _check(lib().alr_gemm(dtype_code(dt), int(a_mn), int(b_mn), int(accumulate),
                          _ptr(A, "A", M * K, dt), _ptr(B, "B", Nc * K, dt),
                          _ptr(C, "C", M * Nc, _F32), M, Nc, K, _stream(stream)))


# ------------------------------------------------------------------ convenience ---
@dataclass
class SlotLoss:
    """Owns the outputs and workspaces of the slot-loss calls for one problem size.

    keep_logits: the forward also writes z_d and z_t (``self.Zd``, ``self.Zt``, with their
    fp16 group references ``self.Zd_ref``, ``self.Zt_ref`` for bf16 inputs) and the backward
    computes G from them in place of z_d instead of recomputing the head products; each
    forward then allows one backward."""
    N: int
    d: int
    V: int
    B: int
    dtype: torch.dtype = torch.bfloat16
    mode: int = ALR_MODE_ALR
    lam: float = 1.0
    gamma: float = 2.0
    device: str = "cuda"
    keep_logits: bool = False

    def __post_init__(self):
        self.params = make_params(self.N, self.d, self.V, self.B, self.dtype, self.mode,
                                  self.lam, self.gamma)
        dev, N = self.device, self.N
        f = lambda: torch.empty(N, dtype=torch.float32, device=dev)  # noqa: E731
        i = lambda: torch.empty(N, dtype=torch.int32, device=dev)  # noqa: E731
        self.out = dict(loss_row=f(), ent_row=f(), lse_d=f(), lse_t=f(), argmax_d=i(),
                        argmax_t=i(), gap_d=f(), gap_t=f(), logp_x=f(), weight=f(),
                        loss_total=torch.zeros(1, dtype=torch.float32, device=dev),
                        weight_sum=torch.zeros(1, dtype=torch.float32, device=dev),
                        wl_sum=torch.zeros(1, dtype=torch.float32, device=dev))
        self.ws_fwd = torch.empty(max(alr_fwd_workspace_size(self.params), 16), dtype=torch.uint8,
                                  device=dev)
        self._ws_bwd = None
        self.Zd = self.Zt = self.Zd_ref = self.Zt_ref = None
        if self.keep_logits:
            lt = logits_dtype(self.dtype)
            self.Zd = torch.empty(N, self.V, dtype=lt, device=dev)
            self.Zt = torch.empty(N, self.V, dtype=lt, device=dev)
            if self.dtype == torch.bfloat16:
                ng = alr_kept_ref_groups(self.V)
                self.Zd_ref = torch.empty(ng, N, dtype=torch.float16, device=dev)
                self.Zt_ref = torch.empty(ng, N, dtype=torch.float16, device=dev)
        self.acc_len = torch.empty(N // self.B, dtype=torch.int32, device=dev)
        self.hist = torch.empty(self.B + 1, dtype=torch.int64, device=dev)

    @property
    def ws_bwd(self):
        if self._ws_bwd is None:
            self._ws_bwd = torch.empty(alr_bwd_workspace_size(self.params), dtype=torch.uint8,
                                       device=self.device)
        return self._ws_bwd

    def forward(self, Hd, Ht, W, row_mask=None, corpus_tok=None, stream=None):
        if self.keep_logits:
            alr_slot_loss_fwd_keep_logits(self.params, Hd, Ht, W, self.Zd, self.Zt, self.Zd_ref,
                                          self.Zt_ref, self.out, self.ws_fwd, row_mask=row_mask,
                                          corpus_tok=corpus_tok, stream=stream)
        else:
            alr_slot_loss_fwd(self.params, Hd, Ht, W, self.out, self.ws_fwd, row_mask=row_mask,
                              corpus_tok=corpus_tok, stream=stream)
        return self.out

    def accept(self, active=None, stream=None):
        alr_accept_len(self.out["argmax_d"], self.out["argmax_t"], self.B, self.acc_len,
                       self.hist, active=active, stream=stream)
        return self.acc_len, self.hist

    def backward(self, Hd, Ht, W, dHd, dW=None, weight_sum=None, stream=None):
        """weight_sum: the normaliser sum omega of Eq. 1 (default: this forward's own; a
        row-sharded batch passes the sum over all its shards)."""
        o = dict(self.out)
        if weight_sum is not None:
            o["weight_sum"] = weight_sum
        if self.keep_logits:
            if self._ws_bwd is None:
                n = alr_bwd_from_logits_workspace_size(self.params)
                self._ws_bwd = torch.empty(max(n, 16), dtype=torch.uint8, device=self.device)
            alr_slot_loss_bwd_from_logits(self.params, Hd, W, self.Zd, self.Zt, self.Zd_ref,
                                          self.Zt_ref, o["weight"], o["weight_sum"], o["lse_d"],
                                          o["lse_t"], self.G, dHd, dW, self._ws_bwd,
                                          stream=stream)
            return
        alr_slot_loss_bwd(self.params, Hd, Ht, W, o["weight"], o["weight_sum"], o["lse_d"],
                          o["lse_t"], dHd, dW, self.ws_bwd, stream=stream)

    @property
    def G(self):
        """With keep_logits, the logit gradient's storage: z_d's buffer, viewed as the input
        element type."""
        return None if self.Zd is None else self.Zd.view(self.dtype)
