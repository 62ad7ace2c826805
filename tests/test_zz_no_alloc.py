"""alr_slot_loss_fwd_noalloc: the forward pass for callers that cannot allocate device memory
(their process pools all device memory up front, or a device allocation's synchronisation is
not acceptable on their path).  Its scratch is the library's fixed device array.

Checked through the C ABI on two calls in a row: bit for bit against alr_slot_loss_fwd with a
caller workspace (the same kernels over the same split plan), and against the CPU oracle at
the parity bars; plus the size limit and the absence of any device allocation by the call.
This file is collected last on purpose."""

import ctypes

import numpy as np
import pytest
import torch

from oracle import alr_oracle as orc
from paper_2609_38795_gb300 import alr, build_lib, synthetic
from tests import parity as P

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    build_lib.build()
    alr.lib()
    assert alr.alr_device_supported() == alr.ALR_OK, alr.alr_last_error()


def _outputs(N):
    f = lambda: torch.full((N,), float("nan"), device="cuda")  # noqa: E731
    i = lambda: torch.full((N,), -1, dtype=torch.int32, device="cuda")  # noqa: E731
    z = lambda: torch.zeros(1, device="cuda")  # noqa: E731
    return dict(loss_row=f(), ent_row=f(), lse_d=f(), lse_t=f(), argmax_d=i(), argmax_t=i(),
                gap_d=f(), gap_t=f(), logp_x=f(), weight=f(), loss_total=z(), weight_sum=z(),
                wl_sum=z())


def _bits(t):
    t = t.cpu()
    return t.view(torch.int32) if t.dtype == torch.float32 else t


def _oracle_view(o):
    out = {k: P.np64(o[k]) for k in ("loss_row", "ent_row", "lse_d", "lse_t", "gap_d", "gap_t",
                                     "weight", "logp_x")}
    out["argmax_d"], out["argmax_t"] = P.npi(o["argmax_d"]), P.npi(o["argmax_t"])
    out["loss_total"] = float(o["loss_total"].item())
    out["weight_sum"] = float(o["weight_sum"].item())
    return out


CASES = [
    # (dtype, A, B, d, V, mode): bf16 with 640 rows (5 row tiles) and a ragged V; fp32, whose
    # transposed head copy lives in the fixed array too
    (torch.bfloat16, 40, 16, 512, 3000, alr.ALR_MODE_ALR),
    (torch.bfloat16, 40, 16, 512, 3000, alr.ALR_MODE_ERASE_SOFT),
    (torch.float32, 8, 8, 256, 4096, alr.ALR_MODE_ALR),
]


@pytest.mark.parametrize("dtype,A,B,d,V,mode", CASES)
def test_noalloc_forward_matches_workspace_forward_twice(dtype, A, B, d, V, mode):
    b = synthetic.slot_batch(d, V, A, B, 0.5, dtype=dtype, device="cuda", seed=7 + mode)
    Hd, Ht, W = b["Hd"], b["Ht"], b["W"]
    N = A * B
    tok = None
    if mode:
        tok = torch.randint(0, V, (N,), dtype=torch.int32, device="cuda",
                            generator=torch.Generator(device="cuda").manual_seed(1))
    mask = torch.ones(N, device="cuda")
    mask[3::B] = 0.0
    params = alr.make_params(N, d, V, B, dtype, mode=mode, lam=1.013441)
    ref = _outputs(N)
    need = alr.alr_fwd_workspace_size(params)
    ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    alr.alr_slot_loss_fwd(params, Hd, Ht, W, ref, ws, row_mask=mask, corpus_tok=tok)
    torch.cuda.synchronize()
    r = orc.slot_loss_forward(P.np64(Hd), P.np64(Ht), P.np64(W), B, mode=mode, lam=1.013441,
                              row_mask=P.np64(mask), corpus_tok=None if tok is None else P.npi(tok))
    for call in range(2):                                 # the array keeps the last call's data
        out = _outputs(N)
        torch.cuda.synchronize()
        reserved, free = torch.cuda.memory_reserved(), torch.cuda.mem_get_info()[0]
        alr.alr_slot_loss_fwd_noalloc(params, Hd, Ht, W, out, row_mask=mask, corpus_tok=tok)
        torch.cuda.synchronize()
        # no device allocation: torch's pool is untouched, and on the second call the device's
        # free memory did not drop by a workspace (the driver may move a little memory of its
        # own between the two readings, hence the slack, which is below the workspace this
        # problem needs).  The first call's set-up may load the library's module on the
        # device, which places the fixed array itself (64 MiB) when modules load lazily.
        assert torch.cuda.memory_reserved() == reserved
        if call == 1:
            assert need > (1 << 20) and torch.cuda.mem_get_info()[0] >= free - (1 << 20)
        for k in ref:
            assert torch.equal(_bits(out[k]), _bits(ref[k])), (call, k)
        P.compare_forward(_oracle_view(out), r, mode=mode)
    assert alr.alr_device_status() == alr.ALR_OK


def test_noalloc_rejects_problems_beyond_the_fixed_scratch():
    lib = alr.lib()
    params = alr.make_params(1 << 20, 4096, 151936, 16, torch.bfloat16)
    need = alr.alr_fwd_workspace_size(params)
    assert need > (64 << 20)                              # ALR_NOALLOC_SCRATCH_BYTES
    out = alr.AlrFwdOutputs()
    rc = lib.alr_slot_loss_fwd_noalloc(ctypes.byref(params), None, None, None, None, None,
                                       ctypes.byref(out), None)
    assert rc == alr.ALR_ERR_INVALID_ARG
    msg = alr.alr_last_error()
    assert "scratch" in msg and str(64 << 20) in msg and str(need) in msg
