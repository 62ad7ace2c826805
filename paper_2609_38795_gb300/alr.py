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
               "logp_x", "weight", "loss_total", "weight_sum")


class AlrFwdOutputs(ctypes.Structure):
    _fields_ = [(f, _c_p) for f in _FWD_FIELDS]


_TOPK_FIELDS = ("loss_row", "lse_d", "tail_q", "argmax_d", "gap_d", "weight", "loss_total",
                "weight_sum")
ALR_TOPK = 8


class AlrTopkFwdOutputs(ctypes.Structure):
    _fields_ = [(f, _c_p) for f in _TOPK_FIELDS]


# name -> (restype, argtypes); must match include/alr.h
SIGNATURES = {
    "alr_version": (ctypes.c_char_p, []),
    "alr_last_error": (ctypes.c_char_p, []),
    "alr_device_supported": (_c_int, []),
    "alr_device_status": (_c_int, [_c_p, _c_int]),
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
    "alr_slot_loss_fwd_keep_logits": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p,
                                               _c_p, _c_p, _c_p, _c_p,
                                               ctypes.POINTER(AlrFwdOutputs), _c_p, _c_sz, _c_p]),
    "alr_logit_grad_from_logits": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p,
                                            _c_p, _c_p, _c_p, _c_p]),
    "alr_bwd_from_logits_workspace_size": (_c_sz, [ctypes.POINTER(AlrParams)]),
    "alr_slot_loss_bwd_from_logits": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p,
                                               _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                                               _c_sz, _c_p]),
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
                                               _c_p, _c_p, _c_p, _c_p,
                                               ctypes.POINTER(AlrTopkFwdOutputs), _c_p, _c_sz,
                                               _c_p]),
    "alr_topk_logit_grad_from_logits": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p,
                                                 _c_p, _c_p, _c_p, _c_p, _c_p, _c_p]),
    "alr_topk_loss_bwd_from_logits": (_c_int, [ctypes.POINTER(AlrParams), _c_p, _c_p, _c_p, _c_p,
                                               _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                                               _c_p, _c_p, _c_sz, _c_p]),
    "alr_ira_blocks": (_c_int, [_c_i32, _c_i32, _c_i32, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                                _c_p, _c_p, _c_p, _c_p]),
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


def _ptr(t):
    return None if t is None else t.data_ptr()


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


def alr_debug_withhold_next_stage(enable=True) -> int:
    return lib().alr_debug_withhold_next_stage(int(enable))


def alr_gather_ira_blocks(feat, seq, pos, B, out, row_valid=None, valid_len=None, stream=None):
    S, L, d = feat.shape
    _check(lib().alr_gather_ira_blocks(_ptr(feat), S, L, d, dtype_code(feat.dtype), _ptr(seq),
                                       _ptr(pos), _ptr(valid_len), seq.numel(), B, _ptr(out),
                                       _ptr(row_valid), _stream(stream)))


def alr_fwd_workspace_size(params) -> int:
    return lib().alr_fwd_workspace_size(ctypes.byref(params))


def alr_bwd_workspace_size(params) -> int:
    return lib().alr_bwd_workspace_size(ctypes.byref(params))


def alr_slot_loss_fwd(params, Hd, Ht, W, out: dict, workspace, row_mask=None, corpus_tok=None,
                      stream=None):
    o = AlrFwdOutputs(**{f: _ptr(out.get(f)) for f in _FWD_FIELDS})
    _check(lib().alr_slot_loss_fwd(ctypes.byref(params), _ptr(Hd), _ptr(Ht), _ptr(W),
                                   _ptr(row_mask), _ptr(corpus_tok), ctypes.byref(o),
                                   _ptr(workspace), workspace.numel() * workspace.element_size(),
                                   _stream(stream)))


def alr_slot_loss_fwd_noalloc(params, Hd, Ht, W, out: dict, row_mask=None, corpus_tok=None,
                              stream=None):
    """alr_slot_loss_fwd without a workspace (scratch in the library's fixed device array)."""
    o = AlrFwdOutputs(**{f: _ptr(out.get(f)) for f in _FWD_FIELDS})
    _check(lib().alr_slot_loss_fwd_noalloc(ctypes.byref(params), _ptr(Hd), _ptr(Ht), _ptr(W),
                                           _ptr(row_mask), _ptr(corpus_tok), ctypes.byref(o),
                                           _stream(stream)))


def alr_slot_loss_bwd(params, Hd, Ht, W, weight, weight_sum, lse_d, lse_t, dHd, dW, workspace,
                      stream=None):
    _check(lib().alr_slot_loss_bwd(ctypes.byref(params), _ptr(Hd), _ptr(Ht), _ptr(W),
                                   _ptr(weight), _ptr(weight_sum), _ptr(lse_d), _ptr(lse_t),
                                   _ptr(dHd), _ptr(dW), _ptr(workspace),
                                   workspace.numel() * workspace.element_size(), _stream(stream)))


def alr_logit_grad_workspace_size(params) -> int:
    return lib().alr_logit_grad_workspace_size(ctypes.byref(params))


def alr_logit_grad(params, Hd, Ht, W, weight, weight_sum, lse_d, lse_t, G, workspace=None,
                   stream=None):
    nbytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(lib().alr_logit_grad(ctypes.byref(params), _ptr(Hd), _ptr(Ht), _ptr(W), _ptr(weight),
                                _ptr(weight_sum), _ptr(lse_d), _ptr(lse_t), _ptr(G),
                                _ptr(workspace), nbytes, _stream(stream)))


def _nbytes(ws):
    return 0 if ws is None else ws.numel() * ws.element_size()


def logits_dtype(t_dtype):
    """Element type of the kept logits for inputs of type t_dtype."""
    return torch.float16 if t_dtype == torch.bfloat16 else torch.float32


def alr_slot_loss_fwd_keep_logits(params, Hd, Ht, W, Zd, Zt, out: dict, workspace, row_mask=None,
                                  corpus_tok=None, stream=None):
    o = AlrFwdOutputs(**{f: _ptr(out.get(f)) for f in _FWD_FIELDS})
    _check(lib().alr_slot_loss_fwd_keep_logits(ctypes.byref(params), _ptr(Hd), _ptr(Ht), _ptr(W),
                                               _ptr(row_mask), _ptr(corpus_tok), _ptr(Zd),
                                               _ptr(Zt), ctypes.byref(o), _ptr(workspace),
                                               _nbytes(workspace), _stream(stream)))


def alr_logit_grad_from_logits(params, Zd, Zt, weight, weight_sum, lse_d, lse_t, G, stream=None):
    _check(lib().alr_logit_grad_from_logits(ctypes.byref(params), _ptr(Zd), _ptr(Zt), _ptr(weight),
                                            _ptr(weight_sum), _ptr(lse_d), _ptr(lse_t), _ptr(G),
                                            _stream(stream)))


def alr_bwd_from_logits_workspace_size(params) -> int:
    return lib().alr_bwd_from_logits_workspace_size(ctypes.byref(params))


def alr_slot_loss_bwd_from_logits(params, Hd, W, Zd, Zt, weight, weight_sum, lse_d, lse_t, G, dHd,
                                  dW, workspace=None, stream=None):
    _check(lib().alr_slot_loss_bwd_from_logits(ctypes.byref(params), _ptr(Hd), _ptr(W), _ptr(Zd),
                                               _ptr(Zt), _ptr(weight), _ptr(weight_sum),
                                               _ptr(lse_d), _ptr(lse_t), _ptr(G), _ptr(dHd),
                                               _ptr(dW), _ptr(workspace), _nbytes(workspace),
                                               _stream(stream)))


def alr_readout_workspace_size(params) -> int:
    return lib().alr_readout_workspace_size(ctypes.byref(params))


def alr_label_readout(params, Ht, W, out: dict, workspace, corpus_tok=None, stream=None):
    """out: top_idx [N, 8] int32, top_prob [N, 8], tail [N]; optional lse_t, argmax_t, gap_t,
    logp_x."""
    _check(lib().alr_label_readout(ctypes.byref(params), _ptr(Ht), _ptr(W), _ptr(corpus_tok),
                                   _ptr(out["top_idx"]), _ptr(out["top_prob"]), _ptr(out["tail"]),
                                   _ptr(out.get("lse_t")), _ptr(out.get("argmax_t")),
                                   _ptr(out.get("gap_t")), _ptr(out.get("logp_x")),
                                   _ptr(workspace), _nbytes(workspace), _stream(stream)))


def alr_topk_fwd_workspace_size(params) -> int:
    return lib().alr_topk_fwd_workspace_size(ctypes.byref(params))


def alr_topk_loss_fwd(params, Hd, W, top_idx, top_prob, tail, out: dict, workspace,
                      row_mask=None, weight_in=None, stream=None):
    o = AlrTopkFwdOutputs(**{f: _ptr(out.get(f)) for f in _TOPK_FIELDS})
    _check(lib().alr_topk_loss_fwd(ctypes.byref(params), _ptr(Hd), _ptr(W), _ptr(top_idx),
                                   _ptr(top_prob), _ptr(tail), _ptr(row_mask), _ptr(weight_in),
                                   ctypes.byref(o), _ptr(workspace), _nbytes(workspace),
                                   _stream(stream)))


def alr_topk_logit_grad(params, Hd, W, top_idx, top_prob, tail, weight, weight_sum, lse_d,
                        tail_q, G, workspace=None, stream=None):
    _check(lib().alr_topk_logit_grad(ctypes.byref(params), _ptr(Hd), _ptr(W), _ptr(top_idx),
                                     _ptr(top_prob), _ptr(tail), _ptr(weight), _ptr(weight_sum),
                                     _ptr(lse_d), _ptr(tail_q), _ptr(G), _ptr(workspace),
                                     _nbytes(workspace), _stream(stream)))


def alr_topk_loss_bwd(params, Hd, W, top_idx, top_prob, tail, weight, weight_sum, lse_d, tail_q,
                      dHd, dW, workspace, stream=None):
    _check(lib().alr_topk_loss_bwd(ctypes.byref(params), _ptr(Hd), _ptr(W), _ptr(top_idx),
                                   _ptr(top_prob), _ptr(tail), _ptr(weight), _ptr(weight_sum),
                                   _ptr(lse_d), _ptr(tail_q), _ptr(dHd), _ptr(dW),
                                   _ptr(workspace), _nbytes(workspace), _stream(stream)))


def alr_topk_loss_fwd_keep_logits(params, Hd, W, top_idx, top_prob, tail, Zd, out: dict,
                                  workspace, row_mask=None, weight_in=None, stream=None):
    o = AlrTopkFwdOutputs(**{f: _ptr(out.get(f)) for f in _TOPK_FIELDS})
    _check(lib().alr_topk_loss_fwd_keep_logits(ctypes.byref(params), _ptr(Hd), _ptr(W),
                                               _ptr(top_idx), _ptr(top_prob), _ptr(tail),
                                               _ptr(row_mask), _ptr(weight_in), _ptr(Zd),
                                               ctypes.byref(o), _ptr(workspace),
                                               _nbytes(workspace), _stream(stream)))


def alr_topk_logit_grad_from_logits(params, Zd, top_idx, top_prob, tail, weight, weight_sum,
                                    lse_d, tail_q, G, stream=None):
    _check(lib().alr_topk_logit_grad_from_logits(ctypes.byref(params), _ptr(Zd), _ptr(top_idx),
                                                 _ptr(top_prob), _ptr(tail), _ptr(weight),
                                                 _ptr(weight_sum), _ptr(lse_d), _ptr(tail_q),
                                                 _ptr(G), _stream(stream)))


def alr_topk_loss_bwd_from_logits(params, Hd, W, Zd, top_idx, top_prob, tail, weight, weight_sum,
                                  lse_d, tail_q, G, dHd, dW, workspace=None, stream=None):
    _check(lib().alr_topk_loss_bwd_from_logits(ctypes.byref(params), _ptr(Hd), _ptr(W), _ptr(Zd),
                                               _ptr(top_idx), _ptr(top_prob), _ptr(tail),
                                               _ptr(weight), _ptr(weight_sum), _ptr(lse_d),
                                               _ptr(tail_q), _ptr(G), _ptr(dHd), _ptr(dW),
                                               _ptr(workspace), _nbytes(workspace),
                                               _stream(stream)))


def alr_ira_blocks(K, max_blocks, valid_anchors, rollout_len, offsets, out: dict,
                   rollout_tok=None, corpus_anchor_tok=None, stream=None):
    """out: seq, pos, valid_len (int32 [S*max_blocks]); optional ctx_len, anchor_tok."""
    _check(lib().alr_ira_blocks(valid_anchors.numel(), K, max_blocks, _ptr(valid_anchors),
                                _ptr(rollout_len), _ptr(offsets), _ptr(rollout_tok),
                                _ptr(corpus_anchor_tok), _ptr(out["seq"]), _ptr(out["pos"]),
                                _ptr(out["valid_len"]), _ptr(out.get("ctx_len")),
                                _ptr(out.get("anchor_tok")), _stream(stream)))


def alr_accept_len(argmax_d, argmax_t, B, acc_len, hist=None, active=None, stream=None):
    A = argmax_d.numel() // B
    _check(lib().alr_accept_len(_ptr(argmax_d), _ptr(argmax_t), _ptr(active), A, B,
                                _ptr(acc_len), _ptr(hist), _stream(stream)))


def alr_erase_weights(B, gamma, hard, weight, logp_x=None, corpus_tok=None, argmax_t=None,
                      row_mask=None, stream=None):
    A = weight.numel() // B
    _check(lib().alr_erase_weights(_ptr(logp_x), _ptr(corpus_tok), _ptr(argmax_t), _ptr(row_mask),
                                   A, B, float(gamma), int(hard), _ptr(weight), _stream(stream)))


def alr_gemm(A, B, C, M, Nc, K, a_mn=False, b_mn=False, accumulate=False, stream=None):
    _check(lib().alr_gemm(dtype_code(A.dtype), int(a_mn), int(b_mn), int(accumulate), _ptr(A),
                          _ptr(B), _ptr(C), M, Nc, K, _stream(stream)))


# ------------------------------------------------------------------ convenience ---
@dataclass
class SlotLoss:
    """Owns the outputs and workspaces of the slot-loss calls for one problem size.

    keep_logits: the forward also writes z_d and z_t (``self.Zd``, ``self.Zt``) and the
    backward computes G from them in place of z_d instead of recomputing the head products;
    each forward then allows one backward."""
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
                        weight_sum=torch.zeros(1, dtype=torch.float32, device=dev))
        self.ws_fwd = torch.empty(max(alr_fwd_workspace_size(self.params), 16), dtype=torch.uint8,
                                  device=dev)
        self._ws_bwd = None
        self.Zd = self.Zt = None
        if self.keep_logits:
            lt = logits_dtype(self.dtype)
            self.Zd = torch.empty(N, self.V, dtype=lt, device=dev)
            self.Zt = torch.empty(N, self.V, dtype=lt, device=dev)
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
            alr_slot_loss_fwd_keep_logits(self.params, Hd, Ht, W, self.Zd, self.Zt, self.out,
                                          self.ws_fwd, row_mask=row_mask, corpus_tok=corpus_tok,
                                          stream=stream)
        else:
            alr_slot_loss_fwd(self.params, Hd, Ht, W, self.out, self.ws_fwd, row_mask=row_mask,
                              corpus_tok=corpus_tok, stream=stream)
        return self.out

    def accept(self, active=None, stream=None):
        alr_accept_len(self.out["argmax_d"], self.out["argmax_t"], self.B, self.acc_len,
                       self.hist, active=active, stream=stream)
        return self.acc_len, self.hist

    def backward(self, Hd, Ht, W, dHd, dW=None, stream=None):
        o = self.out
        if self.keep_logits:
            if self._ws_bwd is None:
                n = alr_bwd_from_logits_workspace_size(self.params)
                self._ws_bwd = torch.empty(max(n, 16), dtype=torch.uint8, device=self.device)
            alr_slot_loss_bwd_from_logits(self.params, Hd, W, self.Zd, self.Zt, o["weight"],
                                          o["weight_sum"], o["lse_d"], o["lse_t"], self.G, dHd,
                                          dW, self._ws_bwd, stream=stream)
            return
        alr_slot_loss_bwd(self.params, Hd, Ht, W, o["weight"], o["weight_sum"], o["lse_d"],
                          o["lse_t"], dHd, dW, self.ws_bwd, stream=stream)

    @property
    def G(self):
        """With keep_logits, the logit gradient's storage: z_d's buffer, viewed as the input
        element type."""
        return None if self.Zd is None else self.Zd.view(self.dtype)
