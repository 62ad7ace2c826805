"""Parity at the full workload sizes, in the launch configuration bench.py times.

The GPU runs the whole batch; the oracle recomputes 16 whole anchors spread over the batch
(covering different row blocks and vocabulary splits) element by element, and the
batch-level outputs are checked through properties that hold at any size:
  - L equals lambda * sum omega l / sum omega of the per-row outputs, and sum omega equals the
    oracle's exact slot weights summed over the batch;
  - <dW, W> equals <dH, H_d> (both are sum_{r,v} G[r,v] z_d[r,v], reached through differently
    laid-out products);
  - the acceptance histogram counts every anchor.
Gradients in full (every dH and dW entry) are compared on 8-anchor sub-batches at full d and
V, run through exactly the calls the benchmarked step makes: with random heads and with a
sharp head (logits of a trained head's magnitude), in all three weighting modes with the exact
batch normaliser.
"""

import numpy as np
import pytest
import torch

from oracle import alr_oracle as orc
from paper_2609_38795_gb300 import alr, build_lib, synthetic
from tests import parity as P

pytestmark = pytest.mark.gpu

N_SAMPLE_ANCHORS = 16


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    build_lib.build()
    alr.lib()
    assert alr.alr_device_supported() == alr.ALR_OK, alr.alr_last_error()


def _sample_anchors(A):
    return np.unique(np.linspace(0, A - 1, N_SAMPLE_ANCHORS).round().astype(np.int64))


def _rows(anchors, B):
    return (anchors[:, None] * B + np.arange(B)[None, :]).reshape(-1)


class Run:
    """The step bench.py times: gather -> forward keeping the logits -> accepted length ->
    logit gradient from the kept logits (in place of z_d) -> dH = G W^T -> dW += H_d^T G, all
    through the C ABI on the current stream.  keep=False: the forward keeps nothing and the
    logit gradient recomputes the head products instead.  The kept logits of `sample_rows`
    are copied out before the gradient overwrites z_d."""

    def __init__(self, wl, x, mode=alr.ALR_MODE_ALR, lam=1.0, corpus_tok=None, keep=True,
                 sample_rows=None):
        self.wl, self.x = wl, x
        N, d, V, B = wl.N, wl.d, wl.V, wl.B
        x["Ht"] = torch.empty(N, d, dtype=torch.bfloat16, device="cuda")
        x["row_valid"] = torch.empty(N, device="cuda")
        alr.alr_gather_ira_blocks(x["F"], x["seq"], x["pos"], B, x["Ht"], x["row_valid"])
        self.sl = alr.SlotLoss(N, d, V, B, mode=mode, lam=lam, keep_logits=keep)
        self.sl.forward(x["Hd"], x["Ht"], x["W"], row_mask=x["row_valid"], corpus_tok=corpus_tok)
        self.acc, self.hist = self.sl.accept(active=x["row_valid"])
        o = self.sl.out
        self.z_sample = None
        if keep:
            if sample_rows is not None:
                idx = torch.from_numpy(sample_rows).cuda()
                self.z_sample = ((self.sl.Zd[idx].cpu(), self.sl.Zd_ref[:, idx].cpu()),
                                 (self.sl.Zt[idx].cpu(), self.sl.Zt_ref[:, idx].cpu()))
            self.G = self.sl.G
            alr.alr_logit_grad_from_logits(self.sl.params, self.sl.Zd, self.sl.Zt, self.sl.Zd_ref,
                                           self.sl.Zt_ref, o["weight"], o["weight_sum"],
                                           o["lse_d"], o["lse_t"], self.G)
        else:
            self.G = torch.empty(N, V, dtype=torch.bfloat16, device="cuda")
            alr.alr_logit_grad(self.sl.params, x["Hd"], x["Ht"], x["W"], o["weight"],
                               o["weight_sum"], o["lse_d"], o["lse_t"], self.G)
        self.dH = torch.empty(N, d, device="cuda")
        alr.alr_gemm(self.G, x["W"], self.dH, N, d, V)
        self.dW = torch.zeros(d, V, device="cuda")
        alr.alr_gemm(x["Hd"], self.G, self.dW, d, V, N, a_mn=True, b_mn=True, accumulate=True)
        torch.cuda.synchronize()
        assert alr.alr_device_status() == alr.ALR_OK


def _oracle_inputs(wl, x):
    """The oracle's own gather of the target rows (not the GPU's), and fp64 copies."""
    F = x["F"].float().cpu().numpy()
    Ht, valid = orc.gather_ira_blocks(F, x["seq"].cpu().numpy(), x["pos"].cpu().numpy(), wl.B)
    return Ht, valid, P.np64(x["Hd"]), P.np64(x["W"])


def _check_step(wl, x, run, Ht_ref, valid_ref, Hd64, W64, mode=alr.ALR_MODE_ALR, lam=1.0,
                corpus_tok=None):
    B = wl.B
    # gather: every row, bit for bit
    assert np.array_equal(x["Ht"].float().cpu().numpy(), Ht_ref)
    assert np.array_equal(x["row_valid"].cpu().numpy(), valid_ref)
    # sampled anchors, element by element
    anchors = _sample_anchors(wl.A)
    rows = _rows(anchors, B)
    tok = None if corpus_tok is None else corpus_tok[rows]
    r = orc.slot_loss_forward(Hd64[rows], Ht_ref[rows], W64, B, mode=mode, lam=lam,
                              row_mask=valid_ref[rows], corpus_tok=tok)
    g = P.fwd_to_numpy(run.sl, rows)
    if run.z_sample is not None:
        # kept logits: fp16 relative to the group references
        for (Z, R), z_r in zip(run.z_sample, (r["z_d"], r["z_t"])):
            P.check_kept(Z, R, z_r)
    if mode == alr.ALR_MODE_ERASE_HARD:
        # a near-tie target row may flip its greedy token and with it the hard gate of the
        # anchor's later rows: compare the weights of anchors without near-ties only
        tie = ((r["gap_t"] < P.NEAR_TIE) | (r["gap_d"] < P.NEAR_TIE)).reshape(-1, B).any(axis=1)
        keep = np.repeat(~tie, B)
        np.testing.assert_allclose(g["weight"][keep], r["weight"][keep], rtol=1e-5, atol=0)
        g = dict(g, weight=r["weight"])
    near = P.compare_forward(g, r, mode=mode, check_totals=False)
    acc_r, _ = orc.accept_len(r["argmax_d"], r["argmax_t"], B, active=valid_ref[rows])
    P.compare_accept(P.npi(run.acc)[anchors], None, acc_r, r["gap_d"], r["gap_t"], B)
    assert P.npi(run.hist).sum() == wl.A
    # batch totals through properties
    o = run.sl.out
    w_all, l_all = P.np64(o["weight"]), P.np64(o["loss_row"])
    L_host = lam * (w_all * l_all).sum() / w_all.sum()
    assert abs(o["loss_total"].item() - L_host) <= 1e-5 * abs(L_host)
    dH_g = P.np64(run.dH)[rows]
    if mode == alr.ALR_MODE_ALR:
        # every slot weight is known exactly without labels: check all of them and sum omega
        w_exact = orc.slot_weights(mode, B, 2.0, wl.N, row_mask=valid_ref)
        np.testing.assert_allclose(w_all, w_exact, rtol=1e-6)
        np.testing.assert_allclose(o["weight_sum"].item(), w_exact.sum(), rtol=1e-5)
        G_r = orc.logit_grad(r["z_d"], r["z_t"], r["weight"], lam, weight_sum=w_exact.sum())
        assert P.max_norm_rel(dH_g, G_r @ W64.T) <= P.GRAD_RTOL
    else:
        # the gate of every other anchor needs its labels, so the batch normaliser is not
        # recomputed: sum omega must equal the per-row weights' sum, and the sampled dH rows
        # must match the oracle's up to that one scalar
        np.testing.assert_allclose(o["weight_sum"].item(), w_all.sum(), rtol=1e-5)
        G_r = orc.logit_grad(r["z_d"], r["z_t"], r["weight"], lam, weight_sum=1.0)
        dH_r = G_r @ W64.T
        assert P.max_norm_rel(dH_g / np.abs(dH_g).max(), dH_r / np.abs(dH_r).max()) <= P.GRAD_RTOL
    # <dW, W> = <dH, H_d>: both equal sum_{r,v} G[r,v] z_d[r,v]
    lhs = torch.sum(run.dW * run.x["W"].float(), dtype=torch.float64).item()
    rhs = torch.sum(run.dH * run.x["Hd"].float(), dtype=torch.float64).item()
    assert abs(lhs - rhs) <= 1e-3 * max(abs(rhs), 1e-12), (lhs, rhs)
    return near


@pytest.mark.parametrize("sigma,keep", [(0.25, True), (0.5, True), (1.0, True), (0.5, False)])
def test_text8b_full_batch(sigma, keep):
    """d=4096, V=151936, B=16, 2048 anchors (32768 rows), feature buffer 16 x 4096; the
    kept-logits step at three noise levels and the recomputing step at one."""
    wl = synthetic.WORKLOADS["text8b"]
    x = synthetic.rollout_batch(wl.d, wl.V, wl.A, wl.B, wl.S, wl.L, sigma, device="cuda", seed=0)
    run = Run(wl, x, keep=keep, sample_rows=_rows(_sample_anchors(wl.A), wl.B))
    Ht_ref, valid_ref, Hd64, W64 = _oracle_inputs(wl, x)
    near = _check_step(wl, x, run, Ht_ref, valid_ref, Hd64, W64)
    hist = P.npi(run.hist).tolist()
    print(f"text8b sigma={sigma} keep={keep}: acc-len histogram {hist}, {near} near-tie sampled rows")


@pytest.mark.parametrize("mode", [alr.ALR_MODE_ERASE_SOFT, alr.ALR_MODE_ERASE_HARD])
def test_erase_full_batch(mode):
    """The erase comparator at the text8b size.  Sampled anchors get the paper's corpus
    tokens (the oracle's greedy target token, replaced w.p. 0.2); the others random tokens."""
    wl = synthetic.WORKLOADS["erase"]
    x = synthetic.rollout_batch(wl.d, wl.V, wl.A, wl.B, wl.S, wl.L, 0.5, device="cuda", seed=1)
    Ht_ref, valid_ref, Hd64, W64 = _oracle_inputs(wl, x)
    rows = _rows(_sample_anchors(wl.A), wl.B)
    greedy = np.argmax(Ht_ref[rows].astype(np.float64) @ W64, axis=1)
    mask, rnd = synthetic.corpus_replacement(wl.N, wl.V, wl.replace_rate, seed=3)
    tok = rnd.numpy().astype(np.int64)
    tok[rows] = np.where(mask.numpy()[rows], tok[rows], greedy)
    tok_dev = torch.from_numpy(tok.astype(np.int32)).cuda()
    run = Run(wl, x, mode=mode, corpus_tok=tok_dev, sample_rows=rows)
    _check_step(wl, x, run, Ht_ref, valid_ref, Hd64, W64, mode=mode, corpus_tok=tok)


def test_vl7b_full_batch_and_gradient_sub_batch():
    """d=3584, V=152064, B=16, 512 anchors over 32 rollout sequences of length 2048; then the
    full backward (every dH and dW entry) on an 8-anchor sub-batch at full d and V."""
    wl = synthetic.WORKLOADS["vl7b"]
    x = synthetic.rollout_batch(wl.d, wl.V, wl.A, wl.B, wl.S, wl.L, wl.sigma, device="cuda", seed=2)
    run = Run(wl, x, lam=1.013441, sample_rows=_rows(_sample_anchors(wl.A), wl.B))
    Ht_ref, valid_ref, Hd64, W64 = _oracle_inputs(wl, x)
    _check_step(wl, x, run, Ht_ref, valid_ref, Hd64, W64, lam=1.013441)
    # sub-batch gradient in full, through the composite backward entry point
    sub = _rows(np.arange(8) * (wl.A // 8), wl.B)
    Hd_s = x["Hd"][torch.from_numpy(sub).cuda()].contiguous()
    Ht_s = x["Ht"][torch.from_numpy(sub).cuda()].contiguous()
    sl = alr.SlotLoss(len(sub), wl.d, wl.V, wl.B, lam=1.013441)
    sl.forward(Hd_s, Ht_s, x["W"])
    dH = torch.empty(len(sub), wl.d, device="cuda")
    dW = torch.zeros(wl.d, wl.V, device="cuda")
    sl.backward(Hd_s, Ht_s, x["W"], dH, dW)
    torch.cuda.synchronize()
    r = orc.slot_loss_forward(Hd64[sub], Ht_ref[sub], W64, wl.B, lam=1.013441)
    G = orc.logit_grad(r["z_d"], r["z_t"], r["weight"], 1.013441)
    dH_r, dW_r = orc.slot_loss_backward(Hd64[sub], W64, G)
    assert P.max_norm_rel(P.np64(dH), dH_r) <= P.GRAD_RTOL
    assert P.max_norm_rel(P.np64(dW), dW_r) <= P.GRAD_RTOL


def _bench_sequence(Hd, Ht, W, B, mode=alr.ALR_MODE_ALR, lam=1.0, corpus_tok=None):
    """The benchmarked step's calls on a sub-batch: forward keeping both logit matrices ->
    accepted length -> G from the kept logits written over z_d -> dH = G W^T -> dW += H_d^T G
    (into a non-zero dW, default GEMM form).  Returns the SlotLoss, G (copied before the dW
    product reads it), dH and the accumulated dW minus its start value."""
    N, d = Hd.shape
    V = W.shape[1]
    sl = alr.SlotLoss(N, d, V, B, mode=mode, lam=lam, keep_logits=True)
    sl.forward(Hd, Ht, W, corpus_tok=corpus_tok)
    sl.accept()
    o = sl.out
    alr.alr_logit_grad_from_logits(sl.params, sl.Zd, sl.Zt, sl.Zd_ref, sl.Zt_ref, o["weight"],
                                   o["weight_sum"], o["lse_d"], o["lse_t"], sl.G)
    dH = torch.empty(N, d, device="cuda")
    alr.alr_gemm(sl.G, W, dH, N, d, V)
    dW0 = torch.randn(d, V, generator=torch.Generator(device="cuda").manual_seed(1),
                      device="cuda") * 1e-2
    dW = dW0.clone()
    alr.alr_gemm(Hd, sl.G, dW, d, V, N, a_mn=True, b_mn=True, accumulate=True)
    torch.cuda.synchronize()
    assert alr.alr_device_status() == alr.ALR_OK
    return sl, P.np64(sl.G), P.np64(dH), P.np64(dW) - P.np64(dW0)


SUB_CASES = [
    # (mode, sigma, sharp head)
    (alr.ALR_MODE_ALR, 0.5, False),
    (alr.ALR_MODE_ERASE_SOFT, 0.5, False),
    (alr.ALR_MODE_ERASE_HARD, 0.5, False),
    (alr.ALR_MODE_ALR, 0.1, True),
    (alr.ALR_MODE_ALR, 0.5, True),
    (alr.ALR_MODE_ERASE_SOFT, 0.25, True),
    (alr.ALR_MODE_ERASE_HARD, 0.25, True),
]


@pytest.mark.parametrize("mode,sigma,sharp", SUB_CASES)
def test_text8b_gradient_sub_batch(mode, sigma, sharp):
    """8 anchors (128 rows) at the text8b head (d=4096, V=151936) through the benchmarked
    step's calls; every G, dH and dW entry against the oracle at the 2e-2 max-norm bar, with
    the oracle's own slot weights and batch normaliser (erase gates included).  Sharp heads put
    the logits at |z| up to ~40, where plain fp16 storage of the kept logits would move q and p
    by up to 2 % and miss the bar.  Erase modes: corpus tokens are the oracle's greedy target
    tokens, replaced w.p. 0.2 by uniform ones; a target row whose top-2 gap is below the
    near-tie threshold gets a corpus token that is neither of its top two, so the hard gate
    does not hinge on a tie."""
    wl = synthetic.WORKLOADS["text8b"]
    A, B, lam = 8, wl.B, 1.013441
    b = synthetic.slot_batch(wl.d, wl.V, A, B, sigma, device="cuda", seed=40 + mode)
    if sharp:
        b = synthetic.sharpen(b)
    Hd, Ht, W = b["Hd"], b["Ht"], b["W"]
    Hd64, Ht64, W64 = P.np64(Hd), P.np64(Ht), P.np64(W)
    tok = None
    if mode != alr.ALR_MODE_ALR:
        zt = Ht64 @ W64
        top2 = np.argsort(-zt, axis=1, kind="stable")[:, :2]
        gap = np.take_along_axis(zt, top2, axis=1) @ np.array([1.0, -1.0])
        m, rnd = synthetic.corpus_replacement(A * B, wl.V, 0.2, seed=11 + mode)
        tok = np.where(m.numpy(), rnd.numpy(), top2[:, 0]).astype(np.int64)
        tied = gap < P.NEAR_TIE
        tok[tied] = (top2[tied].max(axis=1) + 1) % wl.V
        assert not np.any(tok[tied, None] == top2[tied])
        del zt
    sl, G_g, dH_g, dW_g = _bench_sequence(
        Hd, Ht, W, B, mode=mode, lam=lam,
        corpus_tok=None if tok is None else torch.from_numpy(tok.astype(np.int32)).cuda())
    r = orc.slot_loss_forward(Hd64, Ht64, W64, B, mode=mode, lam=lam, corpus_tok=tok)
    if sharp:
        assert np.abs(r["z_d"]).max() > 30.0
    P.compare_forward(P.fwd_to_numpy(sl), r, mode=mode)
    G_r = orc.logit_grad(r["z_d"], r["z_t"], r["weight"], lam)
    dH_r, dW_r = orc.slot_loss_backward(Hd64, W64, G_r)
    errs = (P.max_norm_rel(G_g, G_r), P.max_norm_rel(dH_g, dH_r), P.max_norm_rel(dW_g, dW_r))
    print(f"mode={mode} sigma={sigma} sharp={sharp}: max|z|={np.abs(r['z_d']).max():.1f}, "
          f"relative max-norm errors G {errs[0]:.2e}, dH {errs[1]:.2e}, dW {errs[2]:.2e}")
    assert max(errs) <= P.GRAD_RTOL, errs
