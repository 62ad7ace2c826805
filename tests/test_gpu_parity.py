"""GPU path (through the C ABI) against the CPU oracle, element by element, on seeded inputs
that span several tiles and ragged tails, plus the degenerate cases of the method."""

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


def _inputs(d, V, A, B, sigma, dtype, seed):
    b = synthetic.slot_batch(d, V, A, B, sigma, dtype=dtype, device="cuda", seed=seed)
    return b["Hd"], b["Ht"], b["W"]


def _oracle_fwd(Hd, Ht, W, B, **kw):
    return orc.slot_loss_forward(P.np64(Hd), P.np64(Ht), P.np64(W), B, **kw)


def _erase_tokens(Ht, W, rate, seed):
    """Corpus tokens: the oracle's greedy target token, replaced at `rate` by a random one."""
    greedy = np.argmax(P.np64(Ht) @ P.np64(W), axis=1)
    mask, tok = synthetic.corpus_replacement(len(greedy), W.shape[1], rate, seed=seed)
    return synthetic.corpus_tokens(torch.from_numpy(greedy), mask, tok).cuda()


# ------------------------------------------------------------------------- gather ---
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_gather_matches_oracle_bit_for_bit(dtype):
    g = torch.Generator().manual_seed(3)
    S, L, d, A, B = 5, 70, 264, 37, 16
    F = torch.randn(S, L, d, generator=g).to(dtype)
    seq = torch.randint(-1, S + 1, (A,), generator=g, dtype=torch.int32)      # some invalid
    pos = torch.randint(-2, L - 4, (A,), generator=g, dtype=torch.int32)      # some past L-B
    vlen = torch.randint(0, L + 3, (A,), generator=g, dtype=torch.int32)
    # extreme values: positions whose row index would overflow int32, the int32 ends as valid
    # lengths and sequence ids; all give zero rows, as in the oracle's unbounded integers
    i32 = torch.iinfo(torch.int32)
    pos[0], pos[1], pos[2] = i32.max - 5, i32.max, i32.min
    vlen[3], vlen[4] = i32.min, i32.max
    seq[5], seq[6] = i32.max, i32.min
    for use_vlen in (False, True):
        out = torch.full((A * B, d), 7.0, dtype=dtype, device="cuda")
        valid = torch.full((A * B,), -1.0, device="cuda")
        alr.alr_gather_ira_blocks(F.cuda(), seq.cuda(), pos.cuda(), B, out, valid,
                                  valid_len=vlen.cuda() if use_vlen else None)
        ref, rv = orc.gather_ira_blocks(F.float().numpy(), seq.numpy(), pos.numpy(), B,
                                        valid_len=vlen.numpy() if use_vlen else None)
        assert np.array_equal(out.float().cpu().numpy(), ref)
        assert np.array_equal(valid.cpu().numpy(), rv)


def test_chained_gathers_see_each_others_writes():
    """The gathers are launched with programmatic dependent launch: a gather may be scheduled
    while the one before it still runs, and must wait for it before any access.  Each gather
    here reads the previous one's output as its feature buffer (read after write), and the last
    one also overwrites the buffer its predecessor read (write after read); every buffer
    matches the oracle applied in the same order."""
    g = torch.Generator().manual_seed(8)
    S, L, d, A, B = 3, 256, 512, 48, 16                   # A * B = S * L: outputs are buffers
    draws = [(torch.randint(0, S, (A,), generator=g, dtype=torch.int32),
              torch.randint(0, L - B + 1, (A,), generator=g, dtype=torch.int32)) for _ in range(4)]
    F0 = torch.randn(S, L, d, generator=g).to(torch.bfloat16)
    bufs = [F0.cuda()] + [torch.empty(S, L, d, dtype=torch.bfloat16, device="cuda")
                          for _ in range(3)]
    for i in range(3):                                    # bufs[i + 1] = gather(bufs[i])
        seq, pos = draws[i]
        alr.alr_gather_ira_blocks(bufs[i], seq.cuda(), pos.cuda(), B, bufs[i + 1].view(A * B, d))
    seq, pos = draws[3]                                   # reads bufs[3], overwrites bufs[2]
    alr.alr_gather_ira_blocks(bufs[3], seq.cuda(), pos.cuda(), B, bufs[2].view(A * B, d))
    torch.cuda.synchronize()
    ref = [F0.float().numpy()]
    for i in range(3):
        r, v = orc.gather_ira_blocks(ref[i], draws[i][0].numpy(), draws[i][1].numpy(), B)
        assert v.all()
        ref.append(r.reshape(S, L, d))
    last, _ = orc.gather_ira_blocks(ref[3], draws[3][0].numpy(), draws[3][1].numpy(), B)
    assert np.array_equal(bufs[1].float().cpu().numpy(), ref[1])
    assert np.array_equal(bufs[3].float().cpu().numpy(), ref[3])
    assert np.array_equal(bufs[2].float().cpu().numpy(), last.reshape(S, L, d))
    assert not np.array_equal(ref[2], last.reshape(S, L, d))
    assert alr.alr_device_status() == alr.ALR_OK


def test_gather_ira_secondary_blocks_mask():
    """Secondary blocks at offsets j in 2..14 of 15 stored rows: valid rows are 1[j+k <= K]."""
    K, d, A = 15, 64, 13
    prim = torch.randn(A, K, d).to(torch.bfloat16).cuda()
    seq = torch.arange(A, dtype=torch.int32).cuda()
    j = torch.arange(2, K, dtype=torch.int32).cuda()
    out = torch.empty(A * K, d, dtype=torch.bfloat16, device="cuda")
    valid = torch.empty(A * K, device="cuda")
    alr.alr_gather_ira_blocks(prim, seq, j, K, out, valid,
                              valid_len=torch.full((A,), K, dtype=torch.int32, device="cuda"))
    v = valid.cpu().numpy().reshape(A, K)
    for a in range(A):
        jj = a + 2
        assert v[a].tolist() == [1.0 if jj + k <= K else 0.0 for k in range(1, K + 1)]
    assert v.sum(axis=1).mean() == 7.0


def test_gather_empty_batch():
    F = torch.zeros(1, 4, 8, dtype=torch.bfloat16, device="cuda")
    e = torch.empty(0, dtype=torch.int32, device="cuda")
    out = torch.empty(0, 8, dtype=torch.bfloat16, device="cuda")
    alr.alr_gather_ira_blocks(F, e, e, 4, out)


def test_empty_batches_elsewhere():
    """No anchors: the accepted-length call still writes an all-zero histogram, the erase
    weights and the IRA block plan are no-ops, and the loss refuses N = 0 (a loss over no rows
    has no normaliser) with an argument error; nothing faults and the status stays clean."""
    B = 16
    ei = torch.empty(0, dtype=torch.int32, device="cuda")
    ef = torch.empty(0, device="cuda")
    hist = torch.full((B + 1,), 7, dtype=torch.int64, device="cuda")
    alr.alr_accept_len(ei, ei, B, ei, hist)
    alr.alr_erase_weights(B, 2.0, False, ef, logp_x=ef)
    out = {k: torch.empty(0, dtype=torch.int32, device="cuda") for k in ("seq", "pos", "valid_len")}
    alr.alr_ira_blocks(15, 128, ei, ei, ei, out)
    torch.cuda.synchronize()
    assert hist.cpu().tolist() == [0] * (B + 1)
    with pytest.raises(alr.AlrError) as err:
        alr.alr_slot_loss_fwd_noalloc(alr.make_params(0, 64, 256, B), None, None, None, {})
    assert err.value.code == alr.ALR_ERR_INVALID_ARG
    assert alr.alr_device_status() == alr.ALR_OK


# ------------------------------------------------------------------------ forward ---
def test_tiny_fp32_forward_backward_full_parity():
    """The tiny fp32 workload (d=256, V=4096, B=8, 64 anchors), every row and gradient."""
    wl = synthetic.WORKLOADS["tiny"]
    Hd, Ht, W = _inputs(wl.d, wl.V, wl.A, wl.B, 0.5, torch.float32, seed=0)
    sl = P.gpu_forward(Hd, Ht, W, wl.B)
    g = P.fwd_to_numpy(sl)
    r = _oracle_fwd(Hd, Ht, W, wl.B)
    P.compare_forward(g, r)
    acc, hist = sl.accept()
    acc_r, _ = orc.accept_len(r["argmax_d"], r["argmax_t"], wl.B)
    P.compare_accept(P.npi(acc), P.npi(hist), acc_r, r["gap_d"], r["gap_t"], wl.B)
    dH = torch.empty(wl.N, wl.d, device="cuda")
    dW0 = torch.randn(wl.d, wl.V, device="cuda") * 1e-3
    dW = dW0.clone()
    sl.backward(Hd, Ht, W, dH, dW)
    torch.cuda.synchronize()
    G = orc.logit_grad(r["z_d"], r["z_t"], r["weight"], 1.0)
    dH_r, dW_r = orc.slot_loss_backward(P.np64(Hd), P.np64(W), G)
    assert P.max_norm_rel(P.np64(dH), dH_r) <= P.GRAD_RTOL
    assert P.max_norm_rel(P.np64(dW - dW0), dW_r) <= P.GRAD_RTOL
    assert alr.alr_device_status() == alr.ALR_OK


@pytest.mark.parametrize("mode", [alr.ALR_MODE_ALR, alr.ALR_MODE_ERASE_SOFT, alr.ALR_MODE_ERASE_HARD])
def test_ragged_bf16_forward_backward(mode):
    """Ragged everywhere: N = 160 rows (1.25 row tiles), d = 200 (K tail), V = 1000 (7.8
    vocabulary tiles), a masked row per anchor, lambda and gamma off their defaults."""
    A, B, d, V, lam, gamma = 10, 16, 200, 1000, 1.013441, 0.5
    Hd, Ht, W = _inputs(d, V, A, B, 0.5, torch.bfloat16, seed=11 + mode)
    mask = torch.ones(A * B, device="cuda")
    mask[5::B] = 0.0
    tok = _erase_tokens(Ht, W, 0.2, seed=5) if mode != alr.ALR_MODE_ALR else None
    sl = P.gpu_forward(Hd, Ht, W, B, mode=mode, lam=lam, gamma=gamma, row_mask=mask, corpus_tok=tok)
    g = P.fwd_to_numpy(sl)
    r = _oracle_fwd(Hd, Ht, W, B, mode=mode, gamma=gamma, lam=lam, row_mask=P.np64(mask),
                    corpus_tok=None if tok is None else P.npi(tok))
    P.compare_forward(g, r, mode=mode)
    dH = torch.empty(A * B, d, device="cuda")
    dW = torch.zeros(d, V, device="cuda")
    sl.backward(Hd, Ht, W, dH, dW)
    torch.cuda.synchronize()
    G = orc.logit_grad(r["z_d"], r["z_t"], r["weight"], lam)
    dH_r, dW_r = orc.slot_loss_backward(P.np64(Hd), P.np64(W), G)
    assert P.max_norm_rel(P.np64(dH), dH_r) <= P.GRAD_RTOL
    assert P.max_norm_rel(P.np64(dW), dW_r) <= P.GRAD_RTOL
    assert np.all(P.np64(dH)[5::B] == 0)                   # masked rows get no gradient


@pytest.mark.parametrize("keep", [True, False])
def test_large_ragged_step(keep):
    """Ragged at scale, through the whole step (forward, accepted length, backward), with the
    logits kept and recomputed: N = 2000 rows (15.6 row tiles, the last raster group partial),
    d = 1000 (a K tail of 40), V = 60000 (234.4 vocabulary tiles, split unevenly over the
    CTAs), one masked row per anchor, lambda off its default.  Every row of the forward and
    of dH against the oracle, dW on every 7th column."""
    A, B, d, V, lam = 125, 16, 1000, 60000, 1.013441
    Hd, Ht, W = _inputs(d, V, A, B, 0.5, torch.bfloat16, seed=31)
    mask = torch.ones(A * B, device="cuda")
    mask[7::B] = 0.0
    sl = alr.SlotLoss(A * B, d, V, B, lam=lam, keep_logits=keep)
    sl.forward(Hd, Ht, W, row_mask=mask)
    acc, hist = sl.accept(active=mask)
    dH = torch.empty(A * B, d, device="cuda")
    dW = torch.zeros(d, V, device="cuda")
    sl.backward(Hd, Ht, W, dH, dW)
    torch.cuda.synchronize()
    assert alr.alr_device_status() == alr.ALR_OK
    r = _oracle_fwd(Hd, Ht, W, B, lam=lam, row_mask=P.np64(mask))
    P.compare_forward(P.fwd_to_numpy(sl), r)
    acc_r, _ = orc.accept_len(r["argmax_d"], r["argmax_t"], B, active=P.np64(mask))
    P.compare_accept(P.npi(acc), P.npi(hist), acc_r, r["gap_d"], r["gap_t"], B)
    G = orc.logit_grad(r["z_d"], r["z_t"], r["weight"], lam)
    assert P.max_norm_rel(P.np64(dH), G @ P.np64(W).T) <= P.GRAD_RTOL
    cols = np.arange(0, V, 7)
    assert P.max_norm_rel(P.np64(dW)[:, cols], P.np64(Hd).T @ G[:, cols]) <= P.GRAD_RTOL
    assert np.all(P.np64(dH)[7::B] == 0)


@pytest.mark.parametrize("keep", [True, False])
def test_paper_block_of_fifteen_predicted_slots(keep):
    """The paper's own block (Sec. 3: K = 15 predicted slots after the anchor, App. A: blocks
    of 16 with slot 0 the anchor) as B = 15 rows per anchor, so anchors straddle the 128-row
    tiles (40 anchors, 600 rows, 4.7 row tiles), in the soft erase mode with gamma = 0.5 (the
    alternative erase schedule) and lambda = 1.013441, through the whole step, logits kept and
    recomputed: every row of the forward, the accepted lengths, dH and dW against the oracle."""
    A, B, d, V, lam, gamma = 40, 15, 256, 3000, 1.013441, 0.5
    mode = alr.ALR_MODE_ERASE_SOFT
    Hd, Ht, W = _inputs(d, V, A, B, 0.5, torch.bfloat16, seed=15)
    tok = _erase_tokens(Ht, W, 0.2, seed=15)
    sl = alr.SlotLoss(A * B, d, V, B, lam=lam, gamma=gamma, mode=mode, keep_logits=keep)
    sl.forward(Hd, Ht, W, corpus_tok=tok)
    acc, hist = sl.accept()
    dH = torch.empty(A * B, d, device="cuda")
    dW = torch.zeros(d, V, device="cuda")
    sl.backward(Hd, Ht, W, dH, dW)
    torch.cuda.synchronize()
    assert alr.alr_device_status() == alr.ALR_OK
    r = _oracle_fwd(Hd, Ht, W, B, mode=mode, gamma=gamma, lam=lam, corpus_tok=P.npi(tok))
    P.compare_forward(P.fwd_to_numpy(sl), r, mode=mode)
    acc_r, _ = orc.accept_len(r["argmax_d"], r["argmax_t"], B)
    P.compare_accept(P.npi(acc), P.npi(hist), acc_r, r["gap_d"], r["gap_t"], B)
    G = orc.logit_grad(r["z_d"], r["z_t"], r["weight"], lam)
    dH_r, dW_r = orc.slot_loss_backward(P.np64(Hd), P.np64(W), G)
    assert P.max_norm_rel(P.np64(dH), dH_r) <= P.GRAD_RTOL
    assert P.max_norm_rel(P.np64(dW), dW_r) <= P.GRAD_RTOL


def test_small_bf16_forward_full_parity():
    """The small workload (d=2048, V=32000, B=16, 256 anchors): every row, forward only."""
    wl = synthetic.WORKLOADS["small"]
    Hd, Ht, W = _inputs(wl.d, wl.V, wl.A, wl.B, wl.sigma, torch.bfloat16, seed=0)
    sl = P.gpu_forward(Hd, Ht, W, wl.B)
    g = P.fwd_to_numpy(sl)
    r = _oracle_fwd(Hd, Ht, W, wl.B)
    near = P.compare_forward(g, r)
    acc, hist = sl.accept()
    acc_r, _ = orc.accept_len(r["argmax_d"], r["argmax_t"], wl.B)
    excluded = P.compare_accept(P.npi(acc), P.npi(hist), acc_r, r["gap_d"], r["gap_t"], wl.B)
    # near-ties are a property of the data (top-2 gaps of 32000 logits of std ~0.9); the
    # count is reported, and every other row matched exactly
    print(f"small: {near} near-tie rows of {wl.N}, {excluded} anchors excluded from acc-len")
    assert near < wl.N // 4


@pytest.mark.parametrize("keep", [False, True])
@pytest.mark.parametrize("B", [1, 3, 32])
def test_degenerate_shapes(B, keep):
    """Vocabulary smaller than one tile, hidden size below one pipeline stage, B = 1 and 32,
    through the whole step; with the logits kept, the kept z_d / z_t (their 16-column store
    boxes cut at V = 24) are checked too."""
    A, d, V = 7, 8, 24
    Hd, Ht, W = _inputs(d, V, A, B, 1.0, torch.bfloat16, seed=B)
    W = (W.float() * 20).to(torch.bfloat16)                  # sharpen the tiny problem
    N = A * B
    sl = alr.SlotLoss(N, d, V, B, keep_logits=keep)
    sl.forward(Hd, Ht, W)
    torch.cuda.synchronize()
    r = _oracle_fwd(Hd, Ht, W, B)
    P.compare_forward(P.fwd_to_numpy(sl), r)
    if keep:
        P.check_kept(sl.Zd, sl.Zd_ref, r["z_d"])
        P.check_kept(sl.Zt, sl.Zt_ref, r["z_t"])
    dH = torch.empty(N, d, device="cuda")
    dW = torch.zeros(d, V, device="cuda")
    sl.backward(Hd, Ht, W, dH, dW)
    torch.cuda.synchronize()
    G = orc.logit_grad(r["z_d"], r["z_t"], r["weight"], 1.0)
    dH_r, dW_r = orc.slot_loss_backward(P.np64(Hd), P.np64(W), G)
    assert P.max_norm_rel(P.np64(dH), dH_r) <= P.GRAD_RTOL
    assert P.max_norm_rel(P.np64(dW), dW_r) <= P.GRAD_RTOL
    assert alr.alr_device_status() == alr.ALR_OK


def test_identical_hidden_states_give_entropy_and_full_acceptance():
    """H_d = H_t: the loss equals the label entropy (Gibbs equality) and every slot is
    accepted; the gradient vanishes up to rounding."""
    A, B, d, V = 8, 16, 128, 640
    Hd, _, W = _inputs(d, V, A, B, 0.5, torch.bfloat16, seed=21)
    sl = P.gpu_forward(Hd, Hd, W, B)
    g = P.fwd_to_numpy(sl)
    np.testing.assert_allclose(g["loss_row"], g["ent_row"], rtol=1e-5, atol=1e-5)
    acc, hist = sl.accept()
    assert P.npi(hist)[B] == A
    dH = torch.empty(A * B, d, device="cuda")
    sl.backward(Hd, Hd, W, dH)
    torch.cuda.synchronize()
    assert dH.abs().max().item() < 1e-4


def test_zero_total_weight():
    A, B, d, V = 4, 8, 64, 256
    Hd, Ht, W = _inputs(d, V, A, B, 0.5, torch.bfloat16, seed=31)
    sl = P.gpu_forward(Hd, Ht, W, B, row_mask=torch.zeros(A * B, device="cuda"))
    assert sl.out["loss_total"].item() == 0.0 and sl.out["weight_sum"].item() == 0.0
    dH = torch.full((A * B, d), 5.0, device="cuda")
    dW = torch.zeros(d, V, device="cuda")
    sl.backward(Hd, Ht, W, dH, dW)
    torch.cuda.synchronize()
    assert dH.abs().max().item() == 0.0 and dW.abs().max().item() == 0.0


def test_constructed_exact_ties_take_the_lower_id():
    """Head columns 3 and 9 identical (and dominant): both logits tie exactly, id 3 wins."""
    A, B, d, V = 2, 8, 64, 256
    Hd, Ht, W = _inputs(d, V, A, B, 0.5, torch.bfloat16, seed=41)
    Hd = Hd.abs().to(torch.bfloat16)
    Ht = Ht.abs().to(torch.bfloat16)
    W[:, 3] = 1.0
    W[:, 9] = 1.0
    W[:, 200] = 1.0
    sl = P.gpu_forward(Hd, Ht, W, B)
    assert torch.all(sl.out["argmax_d"] == 3) and torch.all(sl.out["argmax_t"] == 3)
    assert torch.all(sl.out["gap_d"] == 0)


# ------------------------------------------------------------- row-level kernels ---
@pytest.mark.parametrize("B", [1, 5, 16, 32])
def test_accept_len_bit_exact(B):
    g = torch.Generator().manual_seed(B)
    A = 301
    am_t = torch.randint(0, 3, (A * B,), generator=g, dtype=torch.int32)
    am_d = torch.where(torch.rand(A * B, generator=g) < 0.85, am_t,
                       torch.randint(0, 3, (A * B,), generator=g, dtype=torch.int32))
    active = (torch.rand(A * B, generator=g) < 0.95).float()
    acc = torch.empty(A, dtype=torch.int32, device="cuda")
    hist = torch.full((B + 1,), 99, dtype=torch.int64, device="cuda")
    alr.alr_accept_len(am_d.cuda(), am_t.cuda(), B, acc, hist, active=active.cuda())
    acc_r, hist_r = orc.accept_len(am_d.numpy(), am_t.numpy(), B, active=active.numpy())
    assert np.array_equal(P.npi(acc), acc_r)
    assert np.array_equal(P.npi(hist), hist_r)


@pytest.mark.parametrize("hard", [0, 1])
def test_erase_weights_kernel(hard):
    g = torch.Generator().manual_seed(7 + hard)
    A, B, gamma = 50, 16, 2.0
    logp = -torch.rand(A * B, generator=g) * 3
    am_t = torch.randint(0, 4, (A * B,), generator=g, dtype=torch.int32)
    tok = torch.where(torch.rand(A * B, generator=g) < 0.8, am_t,
                      torch.randint(0, 4, (A * B,), generator=g, dtype=torch.int32))
    mask = (torch.rand(A * B, generator=g) < 0.9).float()
    w = torch.empty(A * B, device="cuda")
    alr.alr_erase_weights(B, gamma, hard, w, logp_x=logp.cuda(), corpus_tok=tok.cuda(),
                          argmax_t=am_t.cuda(), row_mask=mask.cuda())
    gate = orc.erase_gate(B, logp_x=logp.double().numpy(), corpus_tok=tok.numpy(),
                          argmax_t=am_t.numpy(), hard=bool(hard))
    ref = np.tile(orc.slot_envelope(B, gamma), A) * mask.double().numpy() * gate
    np.testing.assert_allclose(P.np64(w), ref, rtol=1e-5, atol=1e-7)


# ------------------------------------------------------------- IRA block plan (f3) ---
def test_ira_block_plan_bit_exact_and_gather():
    """The device block plan equals the oracle's (integers, bit for bit), including m odd /
    even, v = 0, v > 128, an early-terminated rollout and out-of-range offsets; the plan then
    drives the gather of secondary-block label rows from the primary label buffer."""
    K, max_b, d = 15, 128, 64
    P_ = max_b - max_b // 2
    g = torch.Generator().manual_seed(12)
    valid = torch.tensor([0, 1, 2, 7, 128, 300, 65], dtype=torch.int32)
    S = len(valid)
    offsets = torch.randint(2, K, (S, max_b // 2), generator=g, dtype=torch.int32)
    offsets[6, 3] = 0                                     # outside the rollout: unused block
    offsets[6, 4] = K
    rlen = torch.full((S, P_), K, dtype=torch.int32)
    rlen[3, 1] = 9
    roll_tok = torch.randint(0, 1000, (S, P_, K), generator=g, dtype=torch.int32)
    corp_tok = torch.randint(0, 1000, (S, max_b), generator=g, dtype=torch.int32)
    out = {k: torch.full((S * max_b,), -9, dtype=torch.int32, device="cuda")
           for k in ("seq", "pos", "valid_len", "ctx_len", "anchor_tok")}
    alr.alr_ira_blocks(K, max_b, valid.cuda(), rlen.cuda(), offsets.cuda(), out,
                       rollout_tok=roll_tok.cuda(), corpus_anchor_tok=corp_tok.cuda())
    ref = orc.ira_blocks(valid.numpy(), rlen.numpy(), offsets.numpy(), K, max_b,
                         rollout_tok=roll_tok.numpy(), corpus_anchor_tok=corp_tok.numpy())
    for k in out:
        assert np.array_equal(P.npi(out[k]), ref[k].reshape(-1)), k
    # gather the K label rows of every block from a primary label buffer [S*P, K, d]
    lab = torch.randn(S * P_, K, d, generator=g).to(torch.bfloat16)
    rows = torch.empty(S * max_b * K, d, dtype=torch.bfloat16, device="cuda")
    valid_rows = torch.empty(S * max_b * K, device="cuda")
    alr.alr_gather_ira_blocks(lab.cuda(), out["seq"], out["pos"], K, rows, valid_rows,
                              valid_len=out["valid_len"])
    g_ref, v_ref = orc.gather_ira_blocks(lab.float().numpy(), ref["seq"].reshape(-1),
                                         ref["pos"].reshape(-1), K,
                                         valid_len=ref["valid_len"].reshape(-1))
    assert np.array_equal(rows.float().cpu().numpy(), g_ref)
    assert np.array_equal(valid_rows.cpu().numpy(), v_ref)


# ------------------------------------------------------ loss kernel forms (multicast) ---
def _all_outputs(Hd, Ht, W, B, mode, tok):
    """Every fused-kernel output of one problem: forward, kept logits, logit gradient
    (recomputed), label readout, top-8 forward and gradient."""
    N, d = Hd.shape
    V = W.shape[1]
    out = {}
    sl = P.gpu_forward(Hd, Ht, W, B, mode=mode, corpus_tok=tok)
    out.update({f"fwd.{k}": v.clone() for k, v in sl.out.items() if k != "logp_x" or tok is not None})
    keep = alr.SlotLoss(N, d, V, B, mode=mode, keep_logits=True)
    keep.forward(Hd, Ht, W, corpus_tok=tok)
    out["Zd"], out["Zt"] = keep.Zd.clone(), keep.Zt.clone()
    out["Zd_ref"], out["Zt_ref"] = keep.Zd_ref.clone(), keep.Zt_ref.clone()
    G = torch.empty(N, V, dtype=Hd.dtype, device="cuda")
    o = sl.out
    alr.alr_logit_grad(sl.params, Hd, Ht, W, o["weight"], o["weight_sum"], o["lse_d"], o["lse_t"], G)
    out["G"] = G
    f = lambda *sh: torch.empty(*sh, device="cuda")  # noqa: E731
    lab = dict(top_idx=torch.empty(N, 8, dtype=torch.int32, device="cuda"), top_prob=f(N, 8),
               tail=f(N), lse_t=f(N), argmax_t=torch.empty(N, dtype=torch.int32, device="cuda"),
               gap_t=f(N))
    ws = torch.empty(alr.alr_readout_workspace_size(sl.params), dtype=torch.uint8, device="cuda")
    alr.alr_label_readout(sl.params, Ht, W, lab, ws)
    out.update({f"readout.{k}": v for k, v in lab.items()})
    tk = dict(loss_row=f(N), lse_d=f(N), tail_q=f(N), argmax_d=torch.empty(N, dtype=torch.int32, device="cuda"),
              gap_d=f(N), weight=f(N), loss_total=f(1), weight_sum=f(1))
    ws = torch.empty(alr.alr_topk_fwd_workspace_size(sl.params), dtype=torch.uint8, device="cuda")
    alr.alr_topk_loss_fwd(sl.params, Hd, W, lab["top_idx"], lab["top_prob"], lab["tail"], tk, ws)
    out.update({f"topk.{k}": v for k, v in tk.items()})
    Gk = torch.empty(N, V, dtype=Hd.dtype, device="cuda")
    alr.alr_topk_logit_grad(sl.params, Hd, W, lab["top_idx"], lab["top_prob"], lab["tail"],
                            tk["weight"], tk["weight_sum"], tk["lse_d"], tk["tail_q"], Gk)
    out["topk.G"] = Gk
    torch.cuda.synchronize()
    assert alr.alr_device_status() == alr.ALR_OK
    return out


@pytest.mark.parametrize("N", [272, 2048])
def test_loss_kernel_forms_agree_bit_for_bit(N, monkeypatch):
    """The multicast form of the fused kernels (clusters of two row blocks sharing each head
    tile, ALR_LOSS_FORM=mcast) and the single-CTA default compute every unit identically, so all
    outputs agree bit for bit: N = 272 has an odd number of row blocks (the last cluster's
    second CTA has no rows), N = 2048 several raster groups of pairs."""
    B, d, V = 16, 520, 3000
    Hd, Ht, W = _inputs(d, V, N // B, B, 0.5, torch.bfloat16, seed=N)
    tok = torch.randint(0, V, (N,), dtype=torch.int32, device="cuda")
    monkeypatch.setenv("ALR_LOSS_FORM", "single")
    single = _all_outputs(Hd, Ht, W, B, alr.ALR_MODE_ERASE_SOFT, tok)
    monkeypatch.setenv("ALR_LOSS_FORM", "mcast")
    assert alr.alr_kernel_forms()[1] == "mcast", alr.alr_cluster_forms_error()
    mcast = _all_outputs(Hd, Ht, W, B, alr.ALR_MODE_ERASE_SOFT, tok)
    for k in single:
        a, b = single[k].cpu(), mcast[k].cpu()
        if a.dtype.is_floating_point:
            a, b = a.view(torch.int16 if a.element_size() == 2 else torch.int32), \
                b.view(torch.int16 if b.element_size() == 2 else torch.int32)
        assert torch.equal(a, b), k
