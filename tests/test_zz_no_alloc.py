"""alr_slot_loss_fwd_noalloc: the forward pass for callers that cannot allocate device memory
(their process pools all device memory up front, or a device allocation's synchronisation is
not acceptable on their path).  Its scratch is the library's fixed device array.

Checked through the C ABI against alr_slot_loss_fwd (caller workspace) on two calls in a
row, with the parity tolerances of the other GPU tests, plus the size limit and the absence
of any device allocation after the first call.  This file is collected last on purpose."""

import ctypes

import numpy as np
import pytest
import torch

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
    return dict(loss_row=f(), ent_row=f(), lse_d=f(), lse_t=f(), argmax_d=i(), argmax_t=i(),
                gap_d=f(), gap_t=f(), logp_x=f(), weight=f(),
                loss_total=torch.zeros(1, device="cuda"), weight_sum=torch.zeros(1, device="cuda"))


def _compare(g, r):
    """Same kernels, so the results should agree to rounding; checked with the parity bars."""
    assert P.rel_err(g["loss_row"], r["loss_row"]).max() <= P.LOSS_RTOL
    assert P.rel_err(g["ent_row"], r["ent_row"]).max() <= P.LOSS_RTOL
    np.testing.assert_allclose(g["lse_d"], r["lse_d"], rtol=2e-4)
    np.testing.assert_allclose(g["lse_t"], r["lse_t"], rtol=2e-4)
    clear = (r["gap_d"] >= P.NEAR_TIE) & (r["gap_t"] >= P.NEAR_TIE)
    assert np.array_equal(g["argmax_d"][clear], r["argmax_d"][clear])
    assert np.array_equal(g["argmax_t"][clear], r["argmax_t"][clear])
    np.testing.assert_allclose(g["weight"], r["weight"], rtol=1e-3, atol=1e-6)
    assert abs(g["loss_total"] - r["loss_total"]) <= P.LOSS_RTOL * abs(r["loss_total"])


def _np(o):
    out = {k: P.np64(v) for k, v in o.items() if v.dtype == torch.float32 and v.numel() > 1}
    out["argmax_d"], out["argmax_t"] = P.npi(o["argmax_d"]), P.npi(o["argmax_t"])
    out["loss_total"] = float(o["loss_total"].item())
    return out


@pytest.mark.parametrize("mode", [alr.ALR_MODE_ALR, alr.ALR_MODE_ERASE_SOFT])
def test_noalloc_forward_matches_workspace_forward_twice(mode):
    A, B, d, V = 40, 16, 512, 3000                        # 640 rows: 5 row tiles, ragged V
    b = synthetic.slot_batch(d, V, A, B, 0.5, dtype=torch.bfloat16, device="cuda", seed=7 + mode)
    Hd, Ht, W = b["Hd"], b["Ht"], b["W"]
    N = A * B
    tok = torch.randint(0, V, (N,), dtype=torch.int32, device="cuda") if mode else None
    mask = torch.ones(N, device="cuda")
    mask[3::B] = 0.0
    params = alr.make_params(N, d, V, B, torch.bfloat16, mode=mode, lam=1.013441)
    ref_out = _outputs(N)
    ws = torch.empty(alr.alr_fwd_workspace_size(params), dtype=torch.uint8, device="cuda")
    alr.alr_slot_loss_fwd(params, Hd, Ht, W, ref_out, ws, row_mask=mask, corpus_tok=tok)
    torch.cuda.synchronize()
    ref = _np(ref_out)
    for call in range(2):                                 # the array keeps the last call's data
        out = _outputs(N)
        if call == 1:
            torch.cuda.synchronize()
            free_before = torch.cuda.mem_get_info()[0]
        alr.alr_slot_loss_fwd_noalloc(params, Hd, Ht, W, out, row_mask=mask, corpus_tok=tok)
        torch.cuda.synchronize()
        if call == 1:
            assert torch.cuda.mem_get_info()[0] == free_before   # no device allocation
        _compare(_np(out), ref)
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
