"""Pins of the CPU oracle against what the paper and the mathematics fix.

None of these checks re-types the oracle's formulas: each compares it with a textbook
routine, a closed form, an invariant, finite differences of its own forward pass, or a
brute-force enumeration, chosen so that a dropped term, a flipped sign, a wrong index or a
transposed operand in the oracle fails at least one of them.
"""

import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import alr_oracle as orc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_constants.json")


def _paper():
    with open(GOLDEN) as f:
        return {k: v["value"] for k, v in json.load(f).items() if not k.startswith("_")}


def _rand(shape, seed, scale=1.0):
    return np.random.default_rng(seed).standard_normal(shape) * scale


# ---------------------------------------------------------------- soft cross-entropy ---
def test_one_hot_label_is_textbook_cross_entropy():
    """With p = e_y the soft CE is the ordinary CE (torch's cross_entropy in fp64)."""
    z_d = _rand((9, 13), 1, 3.0)
    y = np.random.default_rng(2).integers(0, 13, 9)
    p = np.eye(13)[y]
    ref = torch.nn.functional.cross_entropy(torch.from_numpy(z_d), torch.from_numpy(y),
                                            reduction="none").numpy()
    np.testing.assert_allclose(orc.soft_cross_entropy(p, z_d), ref, rtol=1e-13, atol=1e-13)


def test_sharp_target_tends_to_cross_entropy_on_target_argmax():
    """Scaling h_t by 1e3 makes p one-hot at argmax z_t; the loss tends to CE at that id."""
    d, V, N, B = 6, 11, 8, 4
    W = _rand((d, V), 3, 0.5)
    Hd = _rand((N, d), 4)
    Ht = _rand((N, d), 5) * 1e3
    out = orc.slot_loss_forward(Hd, Ht, W, B)
    y = np.argmax(Ht @ W, axis=1)
    ref = torch.nn.functional.cross_entropy(torch.from_numpy(Hd @ W), torch.from_numpy(y),
                                            reduction="none").numpy()
    np.testing.assert_allclose(out["loss_row"], ref, rtol=1e-9, atol=1e-9)
    np.testing.assert_allclose(out["ent_row"], 0.0, atol=1e-9)


def test_gibbs_inequality_and_equality_case():
    """H(p, q) >= H(p), with equality exactly when the drafter and target logits coincide."""
    d, V, N, B = 8, 17, 12, 4
    W = _rand((d, V), 6, 0.7)
    Hd, Ht = _rand((N, d), 7), _rand((N, d), 8)
    out = orc.slot_loss_forward(Hd, Ht, W, B)
    assert np.all(out["loss_row"] >= out["ent_row"] - 1e-12)
    assert np.all(out["loss_row"] - out["ent_row"] > 1e-6)
    same = orc.slot_loss_forward(Ht, Ht, W, B)
    np.testing.assert_allclose(same["loss_row"], same["ent_row"], rtol=0, atol=1e-12)
    # entropy against scipy's definition
    from scipy.stats import entropy as sp_entropy
    p = orc.softmax(Ht @ W)
    np.testing.assert_allclose(out["ent_row"], [sp_entropy(r) for r in p], rtol=1e-12)


def test_zero_head_closed_form():
    """W = 0: every logit is 0, q = p = uniform, l = log V, G = 0, argmax 0 with gap 0."""
    d, V, N, B = 5, 19, 6, 3
    W = np.zeros((d, V))
    Hd, Ht = _rand((N, d), 9), _rand((N, d), 10)
    out = orc.slot_loss_forward(Hd, Ht, W, B)
    np.testing.assert_allclose(out["loss_row"], math.log(V), rtol=1e-14)
    np.testing.assert_allclose(out["lse_d"], math.log(V), rtol=1e-14)
    assert np.all(out["argmax_d"] == 0) and np.all(out["argmax_t"] == 0)
    assert np.all(out["gap_d"] == 0)
    G = orc.logit_grad(out["z_d"], out["z_t"], out["weight"], 1.0)
    np.testing.assert_allclose(G, 0.0, atol=1e-16)


def test_single_token_vocabulary():
    """V = 1: p = q = 1, so the loss and the gradient vanish."""
    Hd, Ht, W = _rand((4, 3), 11), _rand((4, 3), 12), _rand((3, 1), 13)
    out = orc.slot_loss_forward(Hd, Ht, W, 2)
    np.testing.assert_allclose(out["loss_row"], 0.0, atol=1e-15)
    G = orc.logit_grad(out["z_d"], out["z_t"], out["weight"], 1.0)
    np.testing.assert_allclose(G, 0.0, atol=1e-15)


def test_shift_invariance_of_logits():
    """Adding a per-row constant to all logits (a constant feature column) changes nothing."""
    d, V, N, B = 7, 23, 8, 4
    W = _rand((d, V), 14, 0.6)
    Hd, Ht = _rand((N, d), 15), _rand((N, d), 16)
    base = orc.slot_loss_forward(Hd, Ht, W, B)
    c = _rand((N, 1), 17, 5.0)
    W2 = np.vstack([W, np.ones((1, V))])
    sh = orc.slot_loss_forward(np.hstack([Hd, c]), np.hstack([Ht, -c]), W2, B)
    np.testing.assert_allclose(sh["loss_row"], base["loss_row"], rtol=1e-12)
    np.testing.assert_allclose(sh["lse_d"], base["lse_d"] + c[:, 0], rtol=1e-12)
    assert np.array_equal(sh["argmax_d"], base["argmax_d"])


# --------------------------------------------------------------------------- weights ---
def test_envelope_matches_paper_constants():
    P = _paper()
    w = orc.slot_envelope(P["K"], P["gamma_default"])
    assert w[0] == 1.0                                   # slot 1 carries weight 1
    np.testing.assert_allclose(w[1:] / w[:-1], math.exp(-1 / 2.0), rtol=1e-15)
    np.testing.assert_allclose(w[-1], math.exp(-(15 - 1) / 2.0), rtol=1e-15)
    w05 = orc.slot_envelope(4, P["gamma_erase_alt"])
    np.testing.assert_allclose(w05, [1, math.exp(-2), math.exp(-4), math.exp(-6)], rtol=1e-15)


def test_normalisation_is_scale_free_and_empty_batch_is_zero():
    """Eq. 1 divides by the total weight: rescaling all omega leaves L unchanged."""
    loss = _rand(24, 18) ** 2
    w = np.abs(_rand(24, 19))
    L1, _ = orc.weighted_loss(loss, w, 1.3)
    L2, _ = orc.weighted_loss(loss, 7.5 * w, 1.3)
    np.testing.assert_allclose(L1, L2, rtol=1e-14)
    np.testing.assert_allclose(L1, 1.3 * np.average(loss, weights=w), rtol=1e-14)
    assert orc.weighted_loss(loss, np.zeros(24), 1.0) == (0.0, 0.0)


def _erase_case(seed, N=4 * 6, B=6, d=5, V=7):
    W = _rand((d, V), seed, 0.8)
    Hd, Ht = _rand((N, d), seed + 1), _rand((N, d), seed + 2)
    x = np.random.default_rng(seed + 3).integers(0, V, N)
    return Hd, Ht, W, x, B


def test_erase_gate_properties():
    """Eq. 2: gate 1 at slot 1, never above 1, non-increasing, and equal to the product of
    the label probabilities of the preceding corpus tokens (computed entry by entry)."""
    Hd, Ht, W, x, B = _erase_case(20)
    out = orc.slot_loss_forward(Hd, Ht, W, B, mode=orc.MODE_ERASE_SOFT, corpus_tok=x)
    g = (out["weight"] / np.tile(orc.slot_envelope(B, 2.0), len(x) // B)).reshape(-1, B)
    assert np.all(g[:, 0] == 1.0)
    assert np.all(g <= 1.0 + 1e-15)
    assert np.all(np.diff(g, axis=1) <= 1e-15)
    p = orc.softmax(Ht @ W)
    for a in range(g.shape[0]):
        for s in range(B):
            prod = 1.0
            for sp in range(s):
                r = a * B + sp
                prod *= p[r, x[r]]
            np.testing.assert_allclose(g[a, s], prod, rtol=1e-12)


def test_hard_gate_is_one_on_greedy_rollout():
    """Sec. 3.2: on a greedy target rollout the hard gate equals 1 on every active slot."""
    Hd, Ht, W, _, B = _erase_case(30)
    greedy_x = np.argmax(Ht @ W, axis=1)
    out = orc.slot_loss_forward(Hd, Ht, W, B, mode=orc.MODE_ERASE_HARD, corpus_tok=greedy_x)
    np.testing.assert_array_equal(out["weight"], np.tile(orc.slot_envelope(B, 2.0), len(greedy_x) // B))


def test_hard_gate_drops_everything_after_first_mismatch():
    B = 5
    am_t = np.array([3, 1, 4, 1, 5])
    x = np.array([3, 1, 0, 1, 5])                       # mismatch at row 2
    g = orc.erase_gate(B, corpus_tok=x, argmax_t=am_t, hard=True)
    np.testing.assert_array_equal(g, [1, 1, 1, 0, 0])    # rows after the mismatched one


def test_slot_one_identical_across_modes():
    """Sec. 3.2: slot 1 gets the same label and weight under KD/erase and ALR."""
    Hd, Ht, W, x, B = _erase_case(40)
    alr = orc.slot_loss_forward(Hd, Ht, W, B, mode=orc.MODE_ALR)
    soft = orc.slot_loss_forward(Hd, Ht, W, B, mode=orc.MODE_ERASE_SOFT, corpus_tok=x)
    hard = orc.slot_loss_forward(Hd, Ht, W, B, mode=orc.MODE_ERASE_HARD, corpus_tok=x)
    for o in (soft, hard):
        np.testing.assert_array_equal(o["weight"][::B], alr["weight"][::B])
        np.testing.assert_array_equal(o["loss_row"][::B], alr["loss_row"][::B])


# ------------------------------------------------------------------------- gradients ---
def _loss_of(Hd, W, z_t, weight, lam):
    """Eq. 1 as a function of the drafter side only (labels and weights held fixed)."""
    p = orc.softmax(z_t)
    return orc.weighted_loss(orc.soft_cross_entropy(p, Hd @ W), weight, lam)[0]


@pytest.mark.parametrize("mode", [orc.MODE_ALR, orc.MODE_ERASE_SOFT, orc.MODE_ERASE_HARD])
def test_gradients_match_central_differences(mode):
    d, V, A, B, lam = 4, 7, 2, 3, 1.013441
    N = A * B
    W = _rand((d, V), 50 + mode, 0.9)
    Hd, Ht = _rand((N, d), 60 + mode), _rand((N, d), 70 + mode)
    x = np.random.default_rng(80 + mode).integers(0, V, N)
    mask = np.array([1, 1, 0, 1, 1, 1], dtype=np.float64)
    out = orc.slot_loss_forward(Hd, Ht, W, B, mode=mode, gamma=2.0, lam=lam,
                                row_mask=mask, corpus_tok=x)
    G = orc.logit_grad(out["z_d"], out["z_t"], out["weight"], lam)
    dW_in = _rand((d, V), 90)
    dHd, dW = orc.slot_loss_backward(Hd, W, G, dW_in=dW_in)
    z_t, wt = out["z_t"], out["weight"]
    np.testing.assert_allclose(_loss_of(Hd, W, z_t, wt, lam), out["loss_total"], rtol=1e-14)
    eps = 1e-6
    num_H = np.zeros_like(Hd)
    for i, j in itertools.product(range(N), range(d)):
        e = np.zeros_like(Hd); e[i, j] = eps
        num_H[i, j] = (_loss_of(Hd + e, W, z_t, wt, lam) - _loss_of(Hd - e, W, z_t, wt, lam)) / (2 * eps)
    num_W = np.zeros_like(W)
    for i, j in itertools.product(range(d), range(V)):
        e = np.zeros_like(W); e[i, j] = eps
        num_W[i, j] = (_loss_of(Hd, W + e, z_t, wt, lam) - _loss_of(Hd, W - e, z_t, wt, lam)) / (2 * eps)
    np.testing.assert_allclose(dHd, num_H, rtol=1e-6, atol=1e-9)
    np.testing.assert_allclose(dW - dW_in, num_W, rtol=1e-6, atol=1e-9)
    assert np.all(dHd[2] == 0)                           # a masked row gets no gradient


def test_logit_gradient_rows_sum_to_zero():
    d, V, N, B = 6, 29, 10, 5
    W = _rand((d, V), 91, 0.5)
    out = orc.slot_loss_forward(_rand((N, d), 92), _rand((N, d), 93), W, B)
    G = orc.logit_grad(out["z_d"], out["z_t"], out["weight"], 1.0)
    np.testing.assert_allclose(G.sum(axis=1), 0.0, atol=1e-16)


def test_zero_total_weight_gives_zero_loss_and_gradient():
    d, V, N, B = 3, 5, 4, 2
    out = orc.slot_loss_forward(_rand((N, d), 94), _rand((N, d), 95), _rand((d, V), 96), B,
                                row_mask=np.zeros(N))
    assert out["loss_total"] == 0.0 and out["weight_sum"] == 0.0
    G = orc.logit_grad(out["z_d"], out["z_t"], out["weight"], 1.0)
    assert np.all(G == 0)


# ------------------------------------------------------------------ greedy and acc-len ---
def test_exact_ties_go_to_the_lower_id():
    z = np.array([[0.5, 2.0, 2.0, -1.0],
                  [3.0, 3.0, 3.0, 3.0],
                  [-1.0, -2.0, -1.0, -3.0],
                  [1.0, 0.0, 0.0, 7.0]])
    idx, gap = orc.greedy(z)
    np.testing.assert_array_equal(idx, [1, 0, 0, 3])
    np.testing.assert_array_equal(gap, [0.0, 0.0, 0.0, 6.0])


def test_accept_len_brute_force():
    """Every pair of greedy sequences with B <= 4 over V <= 3 tokens, with and without
    masked rows: acc equals the largest n such that the first n slots all match."""
    for B in (1, 2, 3, 4):
        seqs = list(itertools.product(range(3), repeat=B))
        masks = list(itertools.product((0, 1), repeat=B))
        d_all, t_all, m_all, want = [], [], [], []
        for sd, st in itertools.product(seqs, seqs):
            for m in masks[:: max(1, len(masks) // 4)]:
                d_all += sd; t_all += st; m_all += m
                want.append(max(n for n in range(B + 1)
                                if all(sd[i] == st[i] and m[i] for i in range(n))))
        acc, hist = orc.accept_len(np.array(d_all), np.array(t_all), B, active=np.array(m_all))
        np.testing.assert_array_equal(acc, want)
        np.testing.assert_array_equal(hist, np.bincount(want, minlength=B + 1))
        assert hist.sum() == len(want)


# ---------------------------------------------------------------------- IRA (Eq. 4) ---
def test_ira_offsets_average_seven_supervised_slots():
    P = _paper()
    K = P["K"]
    js = range(P["ira_offset_min"], P["ira_offset_max"] + 1)
    assert list(js) == list(range(2, K))                 # j ~ U{2..K-1}
    counts = [orc.ira_supervised_slots(K, j) for j in js]
    assert counts == [K - j for j in js]
    assert sum(counts) / len(counts) == P["ira_mean_supervised_slots"]


def test_gather_index_by_index_and_secondary_block_mask():
    rng = np.random.default_rng(100)
    S, L, d, B, A = 3, 20, 4, 5, 7
    F = rng.standard_normal((S, L, d)).astype(np.float32)
    seq = np.array([0, 1, 2, 2, 5, 1, 0])                # seq 5 is out of range
    pos = np.array([0, 15, 3, 16, 2, -1, 10])            # rows past L, and pos < 0
    vlen = np.array([20, 20, 6, 20, 20, 20, 12])
    out, valid = orc.gather_ira_blocks(F, seq, pos, B, valid_len=vlen)
    for a in range(A):
        for s in range(B):
            r = a * B + s
            ok = 0 <= seq[a] < S and pos[a] >= 0 and pos[a] + s < min(vlen[a], L)
            assert valid[r] == float(ok)
            if ok:
                np.testing.assert_array_equal(out[r], F[seq[a], pos[a] + s])
            else:
                assert np.all(out[r] == 0)
    # secondary blocks: a primary buffer [A_prim, K, d] read at offset j with valid_len K
    K = 15
    prim = rng.standard_normal((2, K, d)).astype(np.float32)
    for j in range(2, K):
        o, v = orc.gather_ira_blocks(prim, np.array([1]), np.array([j]), K,
                                     valid_len=np.array([K]))
        assert v.tolist() == [1.0 if j + k <= K else 0.0 for k in range(1, K + 1)]
        np.testing.assert_array_equal(o[: K - j], prim[1, j:K])


# ------------------------------------------------------------- IRA block plan (Eq. 4) ---
def test_ira_block_split_and_inheritance():
    """ceil(m/2) primary and floor(m/2) secondary blocks with m = min(v, 128); a secondary at
    offset j supervises exactly the slots k with j + k <= K (Eq. 4), reading primary row
    j + k - 1; its anchor token is y*_j and its context holds j - 1 rollout features."""
    K, max_b = 15, 128
    P = max_b // 2
    rng = np.random.default_rng(5)
    valid = np.array([0, 1, 2, 7, 128, 300])
    offsets = rng.integers(2, K, size=(len(valid), P))
    rlen = np.full((len(valid), P), K)
    rlen[3, 1] = 9                                        # an early-terminated rollout
    offsets[3, 1] = 12                                    # ... whose secondary lies past it
    rlen[5, 2] = 11                                       # ... and one whose secondary fits
    offsets[5, 2] = 6
    roll_tok = rng.integers(0, 1000, size=(len(valid), P, K))
    corp_tok = rng.integers(0, 1000, size=(len(valid), max_b))
    out = orc.ira_blocks(valid, rlen, offsets, K, max_b, rollout_tok=roll_tok,
                         corpus_anchor_tok=corp_tok)
    for s, v in enumerate(valid):
        m = min(v, max_b)
        kinds = ["P" if b < (m + 1) // 2 else ("S" if b < m else "-") for b in range(max_b)]
        assert kinds.count("P") == -(-m // 2) and kinds.count("S") == m // 2
        for b, kind in enumerate(kinds):
            if kind == "-":
                assert out["seq"][s, b] == -1
                continue
            p = b if kind == "P" else b - (m + 1) // 2
            j = 0 if kind == "P" else offsets[s, p]
            if j > rlen[s, p]:                            # y*_j was never generated
                assert out["seq"][s, b] == -1 and out["anchor_tok"][s, b] == -1
                assert out["ctx_len"][s, b] == 0
                continue
            assert out["seq"][s, b] == s * P + p
            assert out["pos"][s, b] == j and out["valid_len"][s, b] == rlen[s, p]
            assert out["ctx_len"][s, b] == max(j - 1, 0)
            assert out["anchor_tok"][s, b] == (corp_tok[s, b] if kind == "P" else roll_tok[s, p, j - 1])
            # supervised slots through the gather's validity rule
            lab = np.arange(len(valid) * P * K, dtype=np.float32).reshape(len(valid) * P, K, 1)
            _, rv = orc.gather_ira_blocks(lab, out["seq"][s, b:b + 1],
                                          out["pos"][s, b:b + 1], K,
                                          valid_len=out["valid_len"][s, b:b + 1])
            assert rv.tolist() == [1.0 if j + k <= rlen[s, p] else 0.0 for k in range(1, K + 1)]
