"""The kept-logits path through the C ABI against the CPU oracle: the forward that also writes
z_d and z_t, the logit gradient computed from those logits, and the backward built on it.

Bars: forward outputs bit-identical to the plain forward (same kernel arithmetic); kept
logits within their storage rounding of the oracle's fp64 logits (bf16 inputs: fp16 values
relative to 16-column group references, 2^-11 of the distance to the reference, plus the fp32
accumulation; fp32 inputs: the tf32 products' 2^-10 relative input rounding summed over d);
gradients 2e-2 relative in max-norm."""

import numpy as np
import pytest
import torch

from oracle import alr_oracle as orc
from paper_2609_38795_gb300 import alr, build_lib, synthetic
from tests import parity as P

pytestmark = pytest.mark.gpu

FWD_KEYS = ("loss_row", "ent_row", "lse_d", "lse_t", "argmax_d", "argmax_t", "gap_d", "gap_t",
            "weight", "logp_x", "loss_total", "weight_sum")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    build_lib.build()
    alr.lib()
    assert alr.alr_device_supported() == alr.ALR_OK, alr.alr_last_error()


def _inputs(d, V, A, B, sigma, dtype, seed):
    b = synthetic.slot_batch(d, V, A, B, sigma, dtype=dtype, device="cuda", seed=seed)
    return b["Hd"], b["Ht"], b["W"]


def _check_kept(sl, r):
    """Both kept logit matrices of a SlotLoss against the oracle's logits."""
    for Z, R, z_r in ((sl.Zd, sl.Zd_ref, r["z_d"]), (sl.Zt, sl.Zt_ref, r["z_t"])):
        if R is not None:
            P.check_kept(Z, R, z_r)
        else:
            # tf32 products: each operand keeps 10 mantissa bits (relative error below 2^-10),
            # so the error is at most about 2^-9 |z| plus a random part far below 4e-3 here
            err = np.abs(P.np64(Z) - z_r)
            assert np.all(err <= 2.0 ** -8 * np.abs(z_r) + 4e-3), err.max()


def _same(a, b):
    """Bit-identical tensors (NaN positions included)."""
    a, b = a.cpu(), b.cpu()
    if a.dtype.is_floating_point:
        return torch.equal(a.view(torch.int32), b.view(torch.int32))
    return torch.equal(a, b)


def _run_keep(Hd, Ht, W, B, mode=alr.ALR_MODE_ALR, lam=1.0, gamma=2.0, row_mask=None,
              corpus_tok=None):
    N, d = Hd.shape
    V = W.shape[1]
    plain = alr.SlotLoss(N, d, V, B, dtype=Hd.dtype, mode=mode, lam=lam, gamma=gamma)
    plain.forward(Hd, Ht, W, row_mask=row_mask, corpus_tok=corpus_tok)
    keep = alr.SlotLoss(N, d, V, B, dtype=Hd.dtype, mode=mode, lam=lam, gamma=gamma,
                        keep_logits=True)
    keep.forward(Hd, Ht, W, row_mask=row_mask, corpus_tok=corpus_tok)
    torch.cuda.synchronize()
    for k in FWD_KEYS:
        if k == "logp_x" and mode == alr.ALR_MODE_ALR:
            continue                                 # written in the erase modes only
        assert _same(plain.out[k], keep.out[k]), k
    return keep


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("mode", [alr.ALR_MODE_ALR, alr.ALR_MODE_ERASE_SOFT, alr.ALR_MODE_ERASE_HARD])
def test_keep_logits_forward_and_backward(dtype, mode):
    """Ragged sizes (N = 160: 1.25 row tiles; d = 200: a K tail; V = 1000: 3.9 vocabulary
    tiles, a 16-column chunk cut at 8), a masked row per anchor, lambda and gamma off their
    defaults: kept logits, forward outputs, and dH / dW from the kept logits with G written
    over z_d in place."""
    A, B, d, V, lam, gamma = 10, 16, 200, 1000, 1.013441, 0.5
    Hd, Ht, W = _inputs(d, V, A, B, 0.5, dtype, seed=61 + mode)
    mask = torch.ones(A * B, device="cuda")
    mask[5::B] = 0.0
    tok = None
    if mode != alr.ALR_MODE_ALR:
        greedy = np.argmax(P.np64(Ht) @ P.np64(W), axis=1)
        m, rnd = synthetic.corpus_replacement(A * B, V, 0.2, seed=9)
        tok = synthetic.corpus_tokens(torch.from_numpy(greedy), m, rnd).cuda()
    sl = _run_keep(Hd, Ht, W, B, mode=mode, lam=lam, gamma=gamma, row_mask=mask, corpus_tok=tok)
    r = orc.slot_loss_forward(P.np64(Hd), P.np64(Ht), P.np64(W), B, mode=mode, gamma=gamma,
                              lam=lam, row_mask=P.np64(mask),
                              corpus_tok=None if tok is None else P.npi(tok))
    P.compare_forward(P.fwd_to_numpy(sl), r, mode=mode)
    assert sl.Zd.dtype == alr.logits_dtype(dtype)
    _check_kept(sl, r)
    dH = torch.empty(A * B, d, device="cuda")
    dW0 = torch.randn(d, V, device="cuda") * 1e-3
    dW = dW0.clone()
    sl.backward(Hd, Ht, W, dH, dW)
    torch.cuda.synchronize()
    G = orc.logit_grad(r["z_d"], r["z_t"], r["weight"], lam)
    dH_r, dW_r = orc.slot_loss_backward(P.np64(Hd), P.np64(W), G)
    assert P.max_norm_rel(P.np64(dH), dH_r) <= P.GRAD_RTOL
    assert P.max_norm_rel(P.np64(dW - dW0), dW_r) <= P.GRAD_RTOL
    assert P.max_norm_rel(P.np64(sl.G), G) <= P.GRAD_RTOL      # G now occupies z_d's buffer
    assert np.all(P.np64(sl.G)[5::B] == 0)                     # masked rows
    assert np.all(P.np64(dH)[5::B] == 0)
    assert alr.alr_device_status() == alr.ALR_OK


@pytest.mark.parametrize("V,scale", [(8, 2.5), (1000, 2.5), (40000, 2.5), (40000, 12.0)])
@pytest.mark.parametrize("in_place", [False, True])
def test_logit_grad_from_logits_elementwise(V, scale, in_place):
    """G from given kept logits (oracle-made inputs: seeded logits in the kept storage, the
    exact logits that storage holds, their fp64 log-sum-exps) against the oracle's gradient
    element by element: bf16 output rounding, 2^-8 relative, plus the fp32 exponentials
    (exponent rounding a few 1e-6 relative on each of q and p, which q - p can cancel:
    1e-5 c (q + p)).  V = 8 (one vector, half a group), 1000 (one pass), 40000 (several unrolled
    passes per thread), and logits of magnitude up to ~60; one row masked, lambda off its
    default."""
    N, B, lam = 48, 16, 0.7
    g = torch.Generator().manual_seed(V)
    zd0 = (torch.randn(N, V, generator=g, dtype=torch.float64) * scale).numpy()
    zt0 = zd0 + torch.randn(N, V, generator=g, dtype=torch.float64).numpy()
    Zd, Rd = P.encode_kept(zd0)
    Zt, Rt = P.encode_kept(zt0)
    zd, zt = P.kept_logits(Zd, Rd), P.kept_logits(Zt, Rt)
    weight = orc.slot_weights(alr.ALR_MODE_ALR, B, 2.0, N)
    weight[7] = 0.0
    lse_d = orc.log_sum_exp(zd)
    lse_t = orc.log_sum_exp(zt)
    ref = orc.logit_grad(zd, zt, weight, lam)
    params = alr.make_params(N, 64, V, B, torch.bfloat16, lam=lam)
    f32 = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float32)).cuda()  # noqa: E731
    zd_dev, zt_dev = Zd.cuda(), Zt.cuda()
    G = zd_dev.view(torch.bfloat16) if in_place else torch.full((N, V), 3.0, dtype=torch.bfloat16,
                                                                 device="cuda")
    alr.alr_logit_grad_from_logits(params, zd_dev, zt_dev, Rd.cuda(), Rt.cuda(), f32(weight),
                                   f32([weight.sum()]), f32(lse_d), f32(lse_t), G)
    torch.cuda.synchronize()
    got = P.np64(G)
    c = lam * weight / weight.sum()
    # fp32 flushes results below its normal range (2^-126) to zero, and bf16 shares that range:
    # entries under ~1e-36 may come out as 0 (they do once logits span +-60)
    tol = (2.0 ** -8 * np.abs(ref) + 1e-5 * c[:, None] * (orc.softmax(zd) + orc.softmax(zt))
           + P.FLUSH_FLOOR)
    assert np.all(np.abs(got - ref) <= tol), np.abs(got - ref).max()
    assert np.all(got[7] == 0)


def test_logit_grad_from_logits_zero_total_weight():
    N, V = 16, 256
    Z = torch.randn(N, V).half().cuda()
    R = torch.zeros(alr.alr_kept_ref_groups(V), N, dtype=torch.float16, device="cuda")
    G = torch.full((N, V), 3.0, dtype=torch.bfloat16, device="cuda")
    params = alr.make_params(N, 64, V, 16, torch.bfloat16)
    w = torch.zeros(N, device="cuda")
    alr.alr_logit_grad_from_logits(params, Z, Z, R, R, w, torch.zeros(1, device="cuda"),
                                   torch.zeros(N, device="cuda"), torch.zeros(N, device="cuda"), G)
    torch.cuda.synchronize()
    assert G.abs().max().item() == 0.0


def test_keep_logits_small_workload():
    """The small workload (d=2048, V=32000, B=16, 4096 rows) through the kept-logits step:
    every kept logit and every dH row against the oracle, dW on a quarter of the columns."""
    wl = synthetic.WORKLOADS["small"]
    Hd, Ht, W = _inputs(wl.d, wl.V, wl.A, wl.B, wl.sigma, torch.bfloat16, seed=3)
    sl = _run_keep(Hd, Ht, W, wl.B)
    r = orc.slot_loss_forward(P.np64(Hd), P.np64(Ht), P.np64(W), wl.B)
    P.compare_forward(P.fwd_to_numpy(sl), r)
    _check_kept(sl, r)
    dH = torch.empty(wl.N, wl.d, device="cuda")
    dW = torch.zeros(wl.d, wl.V, device="cuda")
    sl.backward(Hd, Ht, W, dH, dW)
    torch.cuda.synchronize()
    G = orc.logit_grad(r["z_d"], r["z_t"], r["weight"], 1.0)
    Hd64, W64 = P.np64(Hd), P.np64(W)
    assert P.max_norm_rel(P.np64(dH), G @ W64.T) <= P.GRAD_RTOL
    cols = np.arange(0, wl.V, 4)
    assert P.max_norm_rel(P.np64(dW)[:, cols], Hd64.T @ G[:, cols]) <= P.GRAD_RTOL
