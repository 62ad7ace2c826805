"""Shared helpers of the GPU parity tests: run the CUDA path, run the oracle on the same
(rounded) inputs, and compare with the tolerances the workload fixes:

  per-row loss          1e-3 relative
  gradients (dH, dW)    2e-2 relative in max-norm  (||gpu - ref||_inf / ||ref||_inf)
  argmax, acc-len       bit-exact, except rows whose oracle top-2 gap is below 1e-2
                        (counted and returned, never silently dropped)
"""

from __future__ import annotations

import numpy as np
import torch

from oracle import alr_oracle as orc
from paper_2609_38795_gb300 import alr

LOSS_RTOL = 1e-3
GRAD_RTOL = 2e-2
NEAR_TIE = 1e-2
# Elementwise gradient checks: values below fp32's normal range (2^-126 = 1.2e-38), which bf16
# shares, are flushed to zero by the fp32 exponentials; after the row factor c < 1 anything under
# about 1e-36 may read 0.
FLUSH_FLOOR = 1e-36


def np64(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def npi(t):
    return t.detach().cpu().numpy().astype(np.int64)


def gpu_forward(Hd, Ht, W, B, mode=alr.ALR_MODE_ALR, lam=1.0, gamma=2.0, row_mask=None,
                corpus_tok=None):
    N, d = Hd.shape
    V = W.shape[1]
    sl = alr.SlotLoss(N, d, V, B, dtype=Hd.dtype, mode=mode, lam=lam, gamma=gamma)
    sl.forward(Hd, Ht, W, row_mask=row_mask, corpus_tok=corpus_tok)
    torch.cuda.synchronize()
    return sl


def fwd_to_numpy(sl, rows=None):
    o = sl.out
    sel = (lambda x: x) if rows is None else (lambda x: x[rows])
    out = {k: sel(np64(o[k])) for k in ("loss_row", "ent_row", "lse_d", "lse_t", "gap_d",
                                         "gap_t", "weight", "logp_x")}
    out["argmax_d"] = sel(npi(o["argmax_d"]))
    out["argmax_t"] = sel(npi(o["argmax_t"]))
    out["loss_total"] = float(o["loss_total"].item())
    out["weight_sum"] = float(o["weight_sum"].item())
    return out


def rel_err(a, b):
    return np.abs(a - b) / np.maximum(np.abs(b), 1e-30)


def compare_forward(g, r, *, mode=alr.ALR_MODE_ALR, check_totals=True):
    """Compare GPU forward outputs `g` with oracle outputs `r` on the same rows.
    Returns the number of near-tie rows excluded from the argmax comparison."""
    assert np.all(np.isfinite(g["loss_row"]))
    assert rel_err(g["loss_row"], r["loss_row"]).max() <= LOSS_RTOL, rel_err(g["loss_row"], r["loss_row"]).max()
    assert rel_err(g["ent_row"], r["ent_row"]).max() <= LOSS_RTOL
    np.testing.assert_allclose(g["lse_d"], r["lse_d"], rtol=2e-4)
    np.testing.assert_allclose(g["lse_t"], r["lse_t"], rtol=2e-4)
    clear = (r["gap_d"] >= NEAR_TIE) & (r["gap_t"] >= NEAR_TIE)
    assert np.array_equal(g["argmax_d"][clear], r["argmax_d"][clear])
    assert np.array_equal(g["argmax_t"][clear], r["argmax_t"][clear])
    np.testing.assert_allclose(g["gap_d"][clear], r["gap_d"][clear], atol=2e-3)
    if mode == alr.ALR_MODE_ERASE_SOFT:
        # log-space gate; tiny gates underflow fp32, so abs 1e-6 + rel 1e-3
        np.testing.assert_allclose(g["weight"], r["weight"], rtol=1e-3, atol=1e-6)
        np.testing.assert_allclose(g["logp_x"], r["logp_x"], rtol=1e-3, atol=1e-3)
    else:
        np.testing.assert_allclose(g["weight"], r["weight"], rtol=1e-5, atol=0)
    if check_totals:
        np.testing.assert_allclose(g["weight_sum"], r["weight_sum"], rtol=1e-4)
        assert abs(g["loss_total"] - r["loss_total"]) <= LOSS_RTOL * abs(r["loss_total"]) + 1e-7
    return int((~clear).sum())


def max_norm_rel(g, r):
    den = np.abs(r).max()
    return np.abs(g - r).max() / (den if den > 0 else 1.0)


def compare_accept(acc_g, hist_g, acc_r, gaps_d, gaps_t, B):
    """acc-len bit-exact on anchors with no near-tie row among the slots the count scans.
    hist_g is the histogram of exactly these anchors, or None when they are a sample."""
    A = len(acc_r)
    near = ((gaps_d < NEAR_TIE) | (gaps_t < NEAR_TIE)).reshape(A, B)
    ok = np.ones(A, dtype=bool)
    for a in range(A):
        scan = min(acc_r[a] + 1, B)
        ok[a] = not near[a, :scan].any()
    assert np.array_equal(acc_g[ok], acc_r[ok])
    if hist_g is not None:
        if ok.all():
            assert np.array_equal(hist_g, np.bincount(acc_r, minlength=B + 1))
        assert hist_g.sum() == A
    return int((~ok).sum())


# ------------------------------------------------------------------ kept logits ---
KEEP_GROUP = 16


def _refs_per_column(R, V):
    """Group references [groups, rows] spread to one per logit: [rows, V] fp64."""
    return np.repeat(np64(R).T, KEEP_GROUP, axis=1)[:, :V]


def kept_logits(Z, R=None):
    """Logits a kept matrix holds, in fp64: fp32 values as they are, or fp16 values plus their
    16-column group references (bf16 inputs, group-major R[g, r]): z[r, v] = Z[r, v] +
    R[v // 16, r]."""
    z = np64(Z)
    return z if R is None else z + _refs_per_column(R, z.shape[1])


def fp16_round_up(x):
    """The smallest fp16 value >= x (elementwise, fp64 in, fp16 out)."""
    h = x.astype(np.float16)
    low = h.astype(np.float64) < x
    h[low] = np.nextafter(h[low], np.float16(np.inf))
    return h


def _group_max(z):
    rows, V = z.shape
    n_grp = (V + KEEP_GROUP - 1) // KEEP_GROUP
    pad = np.full((rows, n_grp * KEEP_GROUP), -np.inf)
    pad[:, :V] = z
    return pad.reshape(rows, n_grp, KEEP_GROUP).max(axis=2)


def encode_kept(z):
    """(Z, R) torch fp16 tensors holding fp64 logits z [rows, V] in the kept-logit storage of
    bf16 inputs: R [groups, rows] = each 16-column group's maximum rounded up to fp16,
    Z = fp16(z - R)."""
    R = np.ascontiguousarray(fp16_round_up(_group_max(z)).T)
    Z = (z - _refs_per_column(torch.from_numpy(R), z.shape[1])).astype(np.float16)
    return torch.from_numpy(Z), torch.from_numpy(R)


def check_kept(Z, R, z_ref):
    """Kept logits of bf16 inputs (Z [rows, V], R [groups, rows]) against the oracle's fp64
    logits z_ref:
      - every stored value is <= 0 (its group reference bounds the group from above);
      - each reference is the group maximum rounded up to fp16, up to the accumulation error;
      - |kept - z_ref| <= 2^-11 (R - z_ref) (the fp16 rounding of z - R) plus the fp32
        accumulation over d of exact bf16 products (1e-4 + 2^-16 |z|, far above its size)."""
    zs = np64(Z)
    assert np.all(zs <= 0.0)
    gmax, gref = _group_max(z_ref), np64(R).T
    ulp = np.abs(gmax) * 2.0 ** -10 + 2.0 ** -24
    tol_g = 1e-4 + 2.0 ** -16 * np.abs(gmax)
    assert np.all(gref >= gmax - tol_g) and np.all(gref <= gmax + ulp + tol_g)
    ref = _refs_per_column(R, z_ref.shape[1])
    acc = 1e-4 + 2.0 ** -16 * np.abs(z_ref)
    err = np.abs(zs + ref - z_ref)
    assert np.all(err <= 2.0 ** -11 * np.abs(ref - z_ref) + acc), err.max()
