"""Run-to-run reproducibility of the whole step through the C ABI: the same inputs give
bit-identical outputs on every call.  No floating-point reduction of the path uses atomics:
the partial statistics of the vocabulary splits are merged in a fixed order and every GEMM
tile accumulates its K range in one fixed order; the only atomic adds are the integer counts
of the accepted-length histogram, which are exact in any order."""

import pytest
import torch

from paper_2609_38795_gb300 import alr, build_lib, synthetic

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    build_lib.build()
    alr.lib()
    assert alr.alr_device_supported() == alr.ALR_OK, alr.alr_last_error()


def _bits(t):
    t = t.detach()
    return t.view(torch.int16) if t.element_size() == 2 else (
        t.view(torch.int32) if t.element_size() == 4 else t.view(torch.int64))


def _step(sl, Hd, Ht, W):
    """forward -> accepted length -> backward; returns every output the step produces."""
    N, d, V = sl.N, sl.d, sl.V
    out = sl.forward(Hd, Ht, W)
    acc, hist = sl.accept()
    dH = torch.empty(N, d, device="cuda")
    dW = torch.zeros(d, V, device="cuda")
    sl.backward(Hd, Ht, W, dH, dW)
    torch.cuda.synchronize()
    res = {k: v.clone() for k, v in out.items()}
    res.update(acc=acc.clone(), hist=hist.clone(), dH=dH, dW=dW)
    if sl.keep_logits:
        res["G"] = sl.G.clone()
    return res


def _assert_identical(a, b):
    for k in a:
        if k == "logp_x":
            continue                              # written in the erase modes only
        assert torch.equal(_bits(a[k]), _bits(b[k])), k


@pytest.mark.parametrize("keep", [True, False])
def test_step_is_bit_reproducible(keep):
    """2560 rows (20 row blocks), a ragged vocabulary (5000 = 19.5 tiles of 256), d = 512."""
    A, B, d, V = 160, 16, 512, 5000
    b = synthetic.slot_batch(d, V, A, B, 0.5, dtype=torch.bfloat16, device="cuda", seed=21)
    sl = alr.SlotLoss(A * B, d, V, B, keep_logits=keep)
    first = _step(sl, b["Hd"], b["Ht"], b["W"])
    second = _step(sl, b["Hd"], b["Ht"], b["W"])
    _assert_identical(first, second)
    assert alr.alr_device_status() == alr.ALR_OK


def test_text8b_step_is_bit_reproducible():
    """The benchmarked step at full size (32768 rows, d = 4096, V = 151936), logits kept."""
    wl = synthetic.WORKLOADS["text8b"]
    b = synthetic.slot_batch(wl.d, wl.V, wl.A, wl.B, wl.sigma, dtype=torch.bfloat16,
                             device="cuda", seed=5)
    sl = alr.SlotLoss(wl.N, wl.d, wl.V, wl.B, keep_logits=True)
    first = _step(sl, b["Hd"], b["Ht"], b["W"])
    second = _step(sl, b["Hd"], b["Ht"], b["W"])
    _assert_identical(first, second)
    assert alr.alr_device_status() == alr.ALR_OK
