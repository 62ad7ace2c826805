"""Failure detection without a GPU fault: a pipeline wait that nothing will satisfy runs out
after its bounded time, the kernel records ALR_ERR_TIMEOUT, the host reads it through
alr_device_status(), and the same context keeps computing correct results."""

import time

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


@pytest.mark.parametrize("form", ["single", "mcast"])
def test_withheld_stage_times_out_and_context_survives(form, monkeypatch):
    """Both forms of the fused kernel: single CTAs, and clusters of two CTAs that feed each
    other's stages by multicast (every CTA of the cluster then runs out on its own barriers
    and both meet at the closing cluster barrier)."""
    monkeypatch.setenv("ALR_LOSS_FORM", form)
    assert alr.alr_kernel_forms()[1] == form, alr.alr_cluster_forms_error()
    A, B, d, V = 16, 16, 256, 1024
    b = synthetic.slot_batch(d, V, A, B, 0.5, dtype=torch.bfloat16, device="cuda", seed=9)
    sl = alr.SlotLoss(A * B, d, V, B)
    assert alr.alr_device_status(clear=True) == alr.ALR_OK
    alr.alr_debug_withhold_next_stage(True)
    t0 = time.monotonic()
    sl.forward(b["Hd"], b["Ht"], b["W"])          # enqueues; the kernel gives up on its own
    rc = alr.alr_device_status(clear=True)
    waited = time.monotonic() - t0
    assert rc == alr.ALR_ERR_TIMEOUT, alr.alr_last_error()
    assert "timed out" in alr.alr_last_error()
    assert waited < 20.0
    # the hook disarmed itself; the next call is normal and correct
    sl.forward(b["Hd"], b["Ht"], b["W"])
    torch.cuda.synchronize()
    assert alr.alr_device_status() == alr.ALR_OK
    r = orc.slot_loss_forward(P.np64(b["Hd"]), P.np64(b["Ht"]), P.np64(b["W"]), B)
    P.compare_forward(P.fwd_to_numpy(sl), r)


@pytest.mark.parametrize("form", ["single", "mcast", "mcast4"])
def test_withheld_gemm_stage_times_out_and_context_survives(form, monkeypatch):
    """The tensor-core GEMM in its single-CTA and multicast-cluster forms: the withheld stage
    makes every CTA give up (one epilogue warp sees the abort and the others follow it out of
    their named barrier), the timeout is reported, and the next product is correct."""
    monkeypatch.setenv("ALR_GEMM_FORM", form)
    assert alr.alr_kernel_forms()[0] == form, alr.alr_cluster_forms_error()
    M, Nc, K = 1024, 768, 512
    g = torch.Generator(device="cuda").manual_seed(5)
    A = torch.randn(M, K, device="cuda", generator=g).to(torch.bfloat16)
    Bm = torch.randn(Nc, K, device="cuda", generator=g).to(torch.bfloat16)
    C = torch.zeros(M, Nc, device="cuda")
    assert alr.alr_device_status(clear=True) == alr.ALR_OK
    alr.alr_debug_withhold_next_stage(True)
    t0 = time.monotonic()
    alr.alr_gemm(A, Bm, C, M, Nc, K)
    rc = alr.alr_device_status(clear=True)
    waited = time.monotonic() - t0
    assert rc == alr.ALR_ERR_TIMEOUT, alr.alr_last_error()
    assert waited < 20.0
    alr.alr_gemm(A, Bm, C, M, Nc, K)
    torch.cuda.synchronize()
    assert alr.alr_device_status() == alr.ALR_OK
    ref = P.np64(A) @ P.np64(Bm).T
    assert P.max_norm_rel(P.np64(C), ref) <= 1e-3


def test_binding_refuses_wrong_device_buffers():
    """Buffers the kernels would read or write out of bounds, or misread, are refused by the
    binding with the argument's name, and nothing is launched (the status stays clean)."""
    N, d, V, B = 64, 64, 256, 16
    params = alr.make_params(N, d, V, B, torch.bfloat16)
    bf = lambda *s: torch.zeros(*s, dtype=torch.bfloat16, device="cuda")  # noqa: E731
    Hd, W = bf(N, d), bf(d, V)
    out = {f: torch.zeros(N, device="cuda") for f in alr._FWD_FIELDS}
    out["argmax_d"] = torch.zeros(N, dtype=torch.int32, device="cuda")
    out["argmax_t"] = torch.zeros(N, dtype=torch.int32, device="cuda")
    with pytest.raises(ValueError, match="Ht holds"):
        alr.alr_slot_loss_fwd_noalloc(params, Hd, bf(N - 1, d), W, out)
    with pytest.raises(ValueError, match="W must be contiguous"):
        alr.alr_slot_loss_fwd_noalloc(params, Hd, Hd, bf(V, d).t(), out)
    bad = dict(out, argmax_d=torch.zeros(N, dtype=torch.int64, device="cuda"))
    with pytest.raises(ValueError, match="argmax_d must be torch.int32"):
        alr.alr_slot_loss_fwd_noalloc(params, Hd, Hd, W, bad)
    with pytest.raises(ValueError, match="C holds"):
        alr.alr_gemm(Hd, Hd, torch.zeros(N, N - 1, device="cuda"), N, N, d)
    torch.cuda.synchronize()
    assert alr.alr_device_status() == alr.ALR_OK
