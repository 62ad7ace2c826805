"""Compact-label path on the GPU against the oracle: the rollout label readout (top-8 target
probabilities, tail mass, greedy token) and the top-8 + tail-bin soft CE forward and
backward (Sec. 3.1 under Eq. 1; App. A).  Labels fed to the GPU loss come from the oracle's
readout (or are drawn at random), never from the GPU's."""

import numpy as np
import pytest
import torch

from oracle import alr_oracle as orc
from paper_2609_38795_gb300 import alr, build_lib, synthetic
from tests import parity as P

pytestmark = pytest.mark.gpu
K = alr.ALR_TOPK


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    build_lib.build()
    alr.lib()
    assert alr.alr_device_supported() == alr.ALR_OK, alr.alr_last_error()


def gpu_readout(Ht, W, B, corpus_tok=None):
    N, d = Ht.shape
    V = W.shape[1]
    params = alr.make_params(N, d, V, B, Ht.dtype)
    f = lambda *s: torch.full(s, float("nan"), device="cuda")  # noqa: E731
    out = dict(top_idx=torch.full((N, K), -7, dtype=torch.int32, device="cuda"), top_prob=f(N, K),
               tail=f(N), lse_t=f(N), argmax_t=torch.empty(N, dtype=torch.int32, device="cuda"),
               gap_t=f(N), logp_x=f(N))
    ws = torch.empty(alr.alr_readout_workspace_size(params), dtype=torch.uint8, device="cuda")
    alr.alr_label_readout(params, Ht, W, out, ws, corpus_tok=corpus_tok)
    torch.cuda.synchronize()
    return out


def separated_rows(z_t, k=K + 1, gap=P.NEAR_TIE):
    """Rows whose k largest target logits are pairwise at least `gap` apart (the top-8 set and
    its order are then unique beyond rounding)."""
    top = -np.sort(-z_t, axis=1)[:, :k]
    return (top[:, :-1] - top[:, 1:]).min(axis=1) >= gap


def compare_readout(g, r, prob_rtol=1e-3):
    """The GPU's label is a valid top-8 readout: every (token, probability) pair carries the
    oracle's probability of that token, the list is sorted and distinct, nothing outside it
    beats its last entry beyond the near-tie band, and rows whose top 9 logits are separated
    match the oracle's list exactly.  Returns the number of rows with near-ties."""
    idx_g, prob_g = P.npi(g["top_idx"]), P.np64(g["top_prob"])
    z = r["z_t"]
    N = len(z)
    rows = np.arange(N)[:, None]
    p = np.exp(z - r["lse_t"][:, None])
    np.testing.assert_allclose(prob_g, p[rows, idx_g], rtol=prob_rtol, atol=1e-7)
    zg = z[rows, idx_g]
    assert np.all(np.diff(zg, axis=1) <= P.NEAR_TIE)
    assert all(len(set(row)) == K for row in idx_g.tolist())
    rest = z.copy()
    rest[rows, idx_g] = -np.inf
    assert np.all(rest.max(axis=1) <= zg.min(axis=1) + P.NEAR_TIE)
    ok = separated_rows(z)
    assert np.array_equal(idx_g[ok], r["idx"][ok])
    np.testing.assert_allclose(P.np64(g["tail"]), 1.0 - p[rows, idx_g].sum(axis=1), rtol=1e-3,
                               atol=1e-5)
    np.testing.assert_allclose(P.np64(g["lse_t"]), r["lse_t"], rtol=2e-4)
    clear = r["gap_t"] >= P.NEAR_TIE
    assert np.array_equal(P.npi(g["argmax_t"])[clear], r["argmax_t"][clear])
    return int((~ok).sum())


@pytest.mark.parametrize("dtype,shape", [(torch.bfloat16, (10, 16, 200, 1000)),
                                         (torch.bfloat16, (17, 16, 200, 1000)),
                                         (torch.float32, (64, 8, 256, 4096)),
                                         (torch.bfloat16, (64, 16, 2048, 32000)),
                                         (torch.bfloat16, (125, 16, 1000, 60000))])
def test_readout_matches_oracle(dtype, shape):
    """Row counts of 1.25, 2.1, 4, 8 and 15.6 row blocks of 128: the readout's units take two
    row blocks each, so the last unit may hold a partial block or none; the last shape also
    has a K tail (d = 1000) and a partial vocabulary tile (V = 60000)."""
    A, B, d, V = shape
    b = synthetic.slot_batch(d, V, A, B, 0.5, dtype=dtype, device="cuda", seed=A + V)
    N = A * B
    tok = torch.randint(0, V, (N,), dtype=torch.int32, device="cuda")
    g = gpu_readout(b["Ht"], b["W"], B, corpus_tok=tok)
    r = orc.label_readout(P.np64(b["Ht"]), P.np64(b["W"]), k=K, corpus_tok=P.npi(tok))
    # fp32 inputs multiply as tf32 (10-bit mantissa): logits carry ~3e-4 absolute error at
    # d = 256, so a token's probability ~1e-3 relative; bf16 inputs multiply exactly
    near = compare_readout(g, r, prob_rtol=3e-3 if dtype == torch.float32 else 1e-3)
    np.testing.assert_allclose(P.np64(g["logp_x"]), r["logp_x"], rtol=1e-3, atol=1e-3)
    print(f"readout {shape}: {near} of {N} rows with near-ties among their top 9")


def test_readout_exact_ties_and_small_vocabulary():
    """Equal logits keep the lower id first; V = 8 tokens fills the list exactly (tail 0)."""
    A, B, d, V = 2, 4, 64, 8
    b = synthetic.slot_batch(d, V, A, B, 0.5, dtype=torch.bfloat16, device="cuda", seed=77)
    Ht = b["Ht"].abs().to(torch.bfloat16)
    W = b["W"].clone()
    W[:, 5] = 1.0
    W[:, 2] = 1.0
    g = gpu_readout(Ht, W, B)
    assert torch.all(g["top_idx"][:, 0] == 2) and torch.all(g["top_idx"][:, 1] == 5)
    assert torch.all(g["gap_t"] == 0)
    assert torch.all(g["tail"] == 0)
    r = orc.label_readout(P.np64(Ht), P.np64(W), k=K)
    assert np.array_equal(P.npi(g["top_idx"])[:, :2], r["idx"][:, :2])


def gpu_topk_forward(Hd, W, B, labels, row_mask=None, weight_in=None, lam=1.0, Zd=None,
                     Zd_ref=None):
    """The top-k forward; with Zd given, the variant that also keeps z_d there (and its group
    references in Zd_ref, bf16 inputs)."""
    N, d = Hd.shape
    V = W.shape[1]
    params = alr.make_params(N, d, V, B, Hd.dtype, lam=lam)
    f = lambda: torch.full((N,), float("nan"), device="cuda")  # noqa: E731
    out = dict(loss_row=f(), lse_d=f(), tail_q=f(), argmax_d=torch.empty(N, dtype=torch.int32, device="cuda"),
               gap_d=f(), weight=f(), loss_total=torch.zeros(1, device="cuda"),
               weight_sum=torch.zeros(1, device="cuda"))
    ws = torch.empty(alr.alr_topk_fwd_workspace_size(params), dtype=torch.uint8, device="cuda")
    if Zd is None:
        alr.alr_topk_loss_fwd(params, Hd, W, labels["idx"], labels["prob"], labels["tail"], out, ws,
                              row_mask=row_mask, weight_in=weight_in)
    else:
        alr.alr_topk_loss_fwd_keep_logits(params, Hd, W, labels["idx"], labels["prob"],
                                          labels["tail"], Zd, Zd_ref, out, ws, row_mask=row_mask,
                                          weight_in=weight_in)
    torch.cuda.synchronize()
    return params, out


def gpu_topk_backward(params, Hd, W, labels, out, dW=None):
    N, d = Hd.shape
    dH = torch.empty(N, d, device="cuda")
    ws = torch.empty(alr.alr_bwd_workspace_size(params), dtype=torch.uint8, device="cuda")
    alr.alr_topk_loss_bwd(params, Hd, W, labels["idx"], labels["prob"], labels["tail"],
                          out["weight"], out["weight_sum"], out["lse_d"], out["tail_q"], dH, dW, ws)
    torch.cuda.synchronize()
    return dH


def device_labels(r):
    return dict(idx=torch.from_numpy(r["idx"].astype(np.int32)).cuda(),
                prob=torch.from_numpy(r["prob"].astype(np.float32)).cuda(),
                tail=torch.from_numpy(r["tail"].astype(np.float32)).cuda())


def host_labels(lab):
    return P.npi(lab["idx"]), P.np64(lab["prob"]), P.np64(lab["tail"])


@pytest.mark.parametrize("dtype,shape,use_weight", [(torch.bfloat16, (10, 16, 200, 1000), False),
                                                    (torch.bfloat16, (10, 16, 200, 1000), True),
                                                    (torch.bfloat16, (17, 16, 200, 1000), False),
                                                    (torch.float32, (64, 8, 256, 4096), False)])
def test_topk_loss_forward_backward(dtype, shape, use_weight):
    A, B, d, V = shape
    lam = 1.013441
    b = synthetic.slot_batch(d, V, A, B, 0.5, dtype=dtype, device="cuda", seed=5 + V)
    N = A * B
    Hd, Ht, W = b["Hd"], b["Ht"], b["W"]
    lab_r = orc.label_readout(P.np64(Ht), P.np64(W), k=K)
    lab = device_labels(lab_r)
    mask = torch.ones(N, device="cuda")
    mask[3::B] = 0.0
    win = (torch.rand(N, generator=torch.Generator().manual_seed(3)) * mask.cpu()).cuda() if use_weight else None
    params, out = gpu_topk_forward(Hd, W, B, lab, row_mask=None if use_weight else mask,
                                   weight_in=win, lam=lam)
    idx, prob, tail = host_labels(lab)
    z_d = P.np64(Hd) @ P.np64(W)
    loss_r, tail_q_r = orc.top_k_soft_cross_entropy(z_d, idx, prob, tail)
    w_r = P.np64(win) if use_weight else orc.slot_weights(orc.MODE_ALR, B, 2.0, N, row_mask=P.np64(mask))
    assert P.rel_err(P.np64(out["loss_row"]), loss_r).max() <= P.LOSS_RTOL
    np.testing.assert_allclose(P.np64(out["tail_q"]), tail_q_r, rtol=1e-3, atol=1e-6)
    np.testing.assert_allclose(P.np64(out["lse_d"]), orc.log_sum_exp(z_d), rtol=2e-4)
    am_r, gap_r = orc.greedy(z_d)
    clear = gap_r >= P.NEAR_TIE
    assert np.array_equal(P.npi(out["argmax_d"])[clear], am_r[clear])
    np.testing.assert_allclose(P.np64(out["weight"]), w_r, rtol=1e-5, atol=0)
    L_r, ws_r = orc.weighted_loss(loss_r, w_r, lam)
    assert abs(out["loss_total"].item() - L_r) <= P.LOSS_RTOL * abs(L_r)
    np.testing.assert_allclose(out["weight_sum"].item(), ws_r, rtol=1e-5)
    dW = torch.zeros(d, V, device="cuda")
    dH = gpu_topk_backward(params, Hd, W, lab, out, dW)
    G = orc.top_k_logit_grad(z_d, idx, prob, tail, w_r, lam)
    dH_r, dW_r = orc.slot_loss_backward(P.np64(Hd), P.np64(W), G)
    assert P.max_norm_rel(P.np64(dH), dH_r) <= P.GRAD_RTOL
    assert P.max_norm_rel(P.np64(dW), dW_r) <= P.GRAD_RTOL


def random_labels(N, V, seed):
    """Valid compact labels drawn at random: 8 distinct tokens, probabilities with a tail."""
    rng = np.random.default_rng(seed)
    idx = np.stack([rng.choice(V, K, replace=False) for _ in range(N)])
    raw = rng.random((N, K + 1))
    raw /= raw.sum(axis=1, keepdims=True)
    return dict(idx=idx, prob=-np.sort(-raw[:, :K], axis=1), tail=raw[:, K])


@pytest.mark.parametrize("keep", [True, False])
def test_text8b_full_batch_compact_labels(keep):
    """The compact-label path at the text8b size (32768 rows, V = 151936): readout of every
    row on the GPU; sampled anchors against the oracle; the top-k loss with oracle labels on
    the sampled anchors and random labels elsewhere; totals through properties.  keep: the
    step bench.py times (forward keeping z_d, G from it in place, dH and dW as two GEMM calls);
    otherwise the recomputing backward."""
    wl = synthetic.WORKLOADS["text8b"]
    b = synthetic.slot_batch(wl.d, wl.V, wl.A, wl.B, 0.5, device="cuda", seed=4)
    Hd, Ht, W = b["Hd"], b["Ht"], b["W"]
    g = gpu_readout(Ht, W, wl.B)
    anchors = np.unique(np.linspace(0, wl.A - 1, 16).round().astype(np.int64))
    rows = (anchors[:, None] * wl.B + np.arange(wl.B)).reshape(-1)
    W64 = P.np64(W)
    r = orc.label_readout(P.np64(Ht)[rows], W64, k=K)
    compare_readout({k: v[rows] for k, v in g.items()}, r)
    lab_np = random_labels(wl.N, wl.V, seed=6)
    lab_np["idx"][rows], lab_np["prob"][rows], lab_np["tail"][rows] = r["idx"], r["prob"], r["tail"]
    lab = device_labels(lab_np)
    Zd = torch.empty(wl.N, wl.V, dtype=torch.float16, device="cuda") if keep else None
    Rd = (torch.empty(alr.alr_kept_ref_groups(wl.V), wl.N, dtype=torch.float16, device="cuda")
          if keep else None)
    params, out = gpu_topk_forward(Hd, W, wl.B, lab, Zd=Zd, Zd_ref=Rd)
    z_d = P.np64(Hd)[rows] @ W64
    if keep:
        sel = torch.from_numpy(rows).cuda()
        P.check_kept(Zd[sel], Rd[:, sel], z_d)
    loss_r, tq_r = orc.top_k_soft_cross_entropy(z_d, r["idx"], r["prob"], r["tail"])
    assert P.rel_err(P.np64(out["loss_row"])[rows], loss_r).max() <= P.LOSS_RTOL
    np.testing.assert_allclose(P.np64(out["tail_q"])[rows], tq_r, rtol=1e-3, atol=1e-6)
    w_all = orc.slot_weights(orc.MODE_ALR, wl.B, 2.0, wl.N)
    np.testing.assert_allclose(P.np64(out["weight"]), w_all, rtol=1e-6)
    l_all = P.np64(out["loss_row"])
    L_host = (w_all * l_all).sum() / w_all.sum()
    assert abs(out["loss_total"].item() - L_host) <= 1e-5 * abs(L_host)
    dW = torch.zeros(wl.d, wl.V, device="cuda")
    if keep:
        G_dev = Zd.view(torch.bfloat16)
        alr.alr_topk_logit_grad_from_logits(params, Zd, Rd, lab["idx"], lab["prob"], lab["tail"],
                                            out["weight"], out["weight_sum"], out["lse_d"],
                                            out["tail_q"], G_dev)
        dH = torch.empty(wl.N, wl.d, device="cuda")
        alr.alr_gemm(G_dev, W, dH, wl.N, wl.d, wl.V)
        alr.alr_gemm(Hd, G_dev, dW, wl.d, wl.V, wl.N, a_mn=True, b_mn=True, accumulate=True)
        torch.cuda.synchronize()
    else:
        dH = gpu_topk_backward(params, Hd, W, lab, out, dW)
    G = orc.top_k_logit_grad(z_d, r["idx"], r["prob"], r["tail"], w_all[rows], 1.0,
                             weight_sum=w_all.sum())
    assert P.max_norm_rel(P.np64(dH)[rows], G @ W64.T) <= P.GRAD_RTOL
    lhs = torch.sum(dW * W.float(), dtype=torch.float64).item()
    rhs = torch.sum(dH * Hd.float(), dtype=torch.float64).item()
    assert abs(lhs - rhs) <= 1e-3 * abs(rhs)
    assert alr.alr_device_status() == alr.ALR_OK


# ------------------------------------------------------------------ kept logits ---
@pytest.mark.parametrize("dtype,shape,use_weight", [(torch.bfloat16, (10, 16, 200, 1000), False),
                                                    (torch.bfloat16, (10, 16, 200, 1000), True),
                                                    (torch.float32, (64, 8, 256, 4096), False),
                                                    (torch.bfloat16, (16, 16, 1024, 40000), False),
                                                    (torch.bfloat16, (125, 16, 1000, 60000), False)])
def test_topk_keep_logits_forward_backward(dtype, shape, use_weight):
    """The kept-logits top-k path: forward outputs bit-identical to the plain forward, the kept
    z_d within its storage rounding of the oracle's, and G (written over z_d), dH and dW from
    the kept logits against the oracle; masked rows get G = 0."""
    A, B, d, V = shape
    lam = 1.013441
    b = synthetic.slot_batch(d, V, A, B, 0.5, dtype=dtype, device="cuda", seed=9 + V)
    N = A * B
    Hd, Ht, W = b["Hd"], b["Ht"], b["W"]
    lab_r = orc.label_readout(P.np64(Ht), P.np64(W), k=K)
    lab = device_labels(lab_r)
    mask = torch.ones(N, device="cuda")
    mask[3::B] = 0.0
    win = (torch.rand(N, generator=torch.Generator().manual_seed(3)) * mask.cpu()).cuda() if use_weight else None
    kw = dict(row_mask=None if use_weight else mask, weight_in=win, lam=lam)
    _, plain = gpu_topk_forward(Hd, W, B, lab, **kw)
    Zd = torch.empty(N, V, dtype=alr.logits_dtype(dtype), device="cuda")
    Rd = (torch.empty(alr.alr_kept_ref_groups(V), N, dtype=torch.float16, device="cuda")
          if dtype == torch.bfloat16 else None)
    params, out = gpu_topk_forward(Hd, W, B, lab, Zd=Zd, Zd_ref=Rd, **kw)
    for k in plain:
        a, c = plain[k].cpu(), out[k].cpu()
        assert torch.equal(a.view(torch.int32), c.view(torch.int32)), k
    idx, prob, tail = host_labels(lab)
    z_d = P.np64(Hd) @ P.np64(W)
    if dtype == torch.bfloat16:
        P.check_kept(Zd, Rd, z_d)
    else:
        assert np.all(np.abs(P.np64(Zd) - z_d) <= 2.0 ** -8 * np.abs(z_d) + 4e-3)
    w_r = P.np64(win) if use_weight else orc.slot_weights(orc.MODE_ALR, B, 2.0, N, row_mask=P.np64(mask))
    G = Zd.view(dtype)
    dH = torch.empty(N, d, device="cuda")
    dW = torch.zeros(d, V, device="cuda")
    ws = torch.empty(max(alr.alr_bwd_from_logits_workspace_size(params), 16), dtype=torch.uint8,
                     device="cuda")
    alr.alr_topk_loss_bwd_from_logits(params, Hd, W, Zd, Rd, lab["idx"], lab["prob"], lab["tail"],
                                      out["weight"], out["weight_sum"], out["lse_d"], out["tail_q"],
                                      G, dH, dW, ws)
    torch.cuda.synchronize()
    G_r = orc.top_k_logit_grad(z_d, idx, prob, tail, w_r, lam)
    assert P.max_norm_rel(P.np64(G), G_r) <= P.GRAD_RTOL
    dH_r, dW_r = orc.slot_loss_backward(P.np64(Hd), P.np64(W), G_r)
    assert P.max_norm_rel(P.np64(dH), dH_r) <= P.GRAD_RTOL
    assert P.max_norm_rel(P.np64(dW), dW_r) <= P.GRAD_RTOL
    if not use_weight:
        assert np.all(P.np64(G)[3::B] == 0)
    assert alr.alr_device_status() == alr.ALR_OK


@pytest.mark.parametrize("scale", [2.0, 12.0])
def test_topk_logit_grad_from_logits_elementwise(scale):
    """G from oracle-made kept logits (the kept storage of seeded logits, up to ~60 in
    magnitude at scale 12) and labels against the oracle element by element (bf16 output
    rounding 2^-8 relative, plus the fp32 exponentials), in place over z_d; the label tokens
    of each row, the tail factor and a masked row included."""
    N, B, V, lam = 32, 16, 5000, 0.9
    g = torch.Generator().manual_seed(21)
    Zd, Rd = P.encode_kept((torch.randn(N, V, generator=g, dtype=torch.float64) * scale).numpy())
    zd = P.kept_logits(Zd, Rd)
    lab = random_labels(N, V, seed=22)
    w = orc.slot_weights(orc.MODE_ALR, B, 2.0, N)
    w[5] = 0.0
    lse = orc.log_sum_exp(zd)
    q = orc.softmax(zd)
    tail_q = 1.0 - np.take_along_axis(q, lab["idx"], axis=1).sum(axis=1)
    ref = orc.top_k_logit_grad(zd, lab["idx"], lab["prob"], lab["tail"], w, lam)
    params = alr.make_params(N, 64, V, B, torch.bfloat16, lam=lam)
    f32 = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float32)).cuda()  # noqa: E731
    zd_dev = Zd.cuda()
    dl = device_labels(lab)
    G = zd_dev.view(torch.bfloat16)
    alr.alr_topk_logit_grad_from_logits(params, zd_dev, Rd.cuda(), dl["idx"], dl["prob"],
                                        dl["tail"], f32(w), f32([w.sum()]), f32(lse), f32(tail_q),
                                        G)
    torch.cuda.synchronize()
    got = P.np64(G)
    c = lam * w / w.sum()
    tol = 2.0 ** -8 * np.abs(ref) + 1e-5 * c[:, None] * (q + 1e-3) + P.FLUSH_FLOOR
    assert np.all(np.abs(got - ref) <= tol), np.abs(got - ref).max()
    assert np.all(got[5] == 0)


@pytest.mark.parametrize("sigma", [0.1, 0.5])
def test_text8b_sub_batch_sharp_head_compact_labels(sigma):
    """The compact-label step's calls on 8 anchors (128 rows) at the text8b head with a head
    scaled to trained-head logit sizes (|z| up to ~40): readout of H_t, top-8 forward keeping
    z_d, G from the kept z_d in place, dH and dW through alr_gemm.  Labels, per-row losses and
    every G, dH, dW entry against the oracle (1e-3 relative, 2e-2 max-norm)."""
    wl = synthetic.WORKLOADS["text8b"]
    A, B, lam = 8, wl.B, 1.013441
    b = synthetic.sharpen(synthetic.slot_batch(wl.d, wl.V, A, B, sigma, device="cuda", seed=81))
    Hd, Ht, W = b["Hd"], b["Ht"], b["W"]
    N = A * B
    Hd64, Ht64, W64 = P.np64(Hd), P.np64(Ht), P.np64(W)
    g = gpu_readout(Ht, W, B)
    r = orc.label_readout(Ht64, W64, k=K)
    assert np.abs(r["z_t"]).max() > 30.0
    compare_readout(g, r)
    lab = dict(idx=g["top_idx"], prob=g["top_prob"], tail=g["tail"])
    idx, prob, tail = host_labels(lab)
    Zd = torch.empty(N, wl.V, dtype=torch.float16, device="cuda")
    Rd = torch.empty(alr.alr_kept_ref_groups(wl.V), N, dtype=torch.float16, device="cuda")
    params, out = gpu_topk_forward(Hd, W, B, lab, lam=lam, Zd=Zd, Zd_ref=Rd)
    z_d = Hd64 @ W64
    P.check_kept(Zd, Rd, z_d)
    loss_r, tq_r = orc.top_k_soft_cross_entropy(z_d, idx, prob, tail)
    assert P.rel_err(P.np64(out["loss_row"]), loss_r).max() <= P.LOSS_RTOL
    w_r = orc.slot_weights(orc.MODE_ALR, B, 2.0, N)
    G = Zd.view(torch.bfloat16)
    alr.alr_topk_logit_grad_from_logits(params, Zd, Rd, lab["idx"], lab["prob"], lab["tail"],
                                        out["weight"], out["weight_sum"], out["lse_d"],
                                        out["tail_q"], G)
    dH = torch.empty(N, wl.d, device="cuda")
    dW = torch.zeros(wl.d, wl.V, device="cuda")
    alr.alr_gemm(G, W, dH, N, wl.d, wl.V)
    alr.alr_gemm(Hd, G, dW, wl.d, wl.V, N, a_mn=True, b_mn=True, accumulate=True)
    torch.cuda.synchronize()
    G_r = orc.top_k_logit_grad(z_d, idx, prob, tail, w_r, lam)
    dH_r, dW_r = orc.slot_loss_backward(Hd64, W64, G_r)
    errs = (P.max_norm_rel(P.np64(G), G_r), P.max_norm_rel(P.np64(dH), dH_r),
            P.max_norm_rel(P.np64(dW), dW_r))
    print(f"compact labels, sharp head, sigma={sigma}: loss rel err "
          f"{P.rel_err(P.np64(out['loss_row']), loss_r).max():.2e}, G/dH/dW {errs}")
    assert max(errs) <= P.GRAD_RTOL
    assert alr.alr_device_status() == alr.ALR_OK
