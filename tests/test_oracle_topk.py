"""Pins of the oracle's compact-label path: the top-k label readout and the top-k + tail-bin
soft cross-entropy (Sec. 3.1 under Eq. 1; App. A)."""

import itertools

import numpy as np
import pytest
import torch
from scipy.stats import entropy as sp_entropy

from oracle import alr_oracle as orc


def _rand(shape, seed, scale=1.0):
    return np.random.default_rng(seed).standard_normal(shape) * scale


def test_readout_order_ties_and_mass():
    """Brute-force ordering (probability descending, equal values to the lower id), the
    probabilities with the tail summing to one, and the greedy token first."""
    W = np.zeros((3, 10))
    W[0, [2, 5, 7]] = 4.0          # three exact ties at the top
    W[1, [1, 5]] = 2.0
    H = np.array([[1.0, 0.0, 0.0], [1.0, 1.0, 0.0], [0.0, 1.0, 0.0], [0.0, 0.0, 0.0]])
    out = orc.label_readout(H, W, k=4)
    z = H @ W
    for r in range(len(H)):
        want = sorted(range(10), key=lambda v: (-z[r, v], v))[:4]
        assert out["idx"][r].tolist() == want
        assert out["argmax_t"][r] == want[0]
    np.testing.assert_allclose(out["prob"].sum(1) + out["tail"], 1.0, rtol=1e-14)
    assert out["idx"][0].tolist()[:3] == [2, 5, 7] and out["gap_t"][0] == 0.0


def test_full_vocabulary_label_reduces_to_full_soft_ce():
    """k = V: the tail is empty and the top-k loss is the full-vocabulary soft CE."""
    d, V, N = 6, 9, 8
    W = _rand((d, V), 1, 0.7)
    Hd, Ht = _rand((N, d), 2), _rand((N, d), 3)
    lab = orc.label_readout(Ht, W, k=V)
    assert np.all(lab["tail"] == 0)
    loss, _ = orc.top_k_soft_cross_entropy(Hd @ W, lab["idx"], lab["prob"], lab["tail"])
    full = orc.soft_cross_entropy(orc.softmax(Ht @ W), Hd @ W)
    np.testing.assert_allclose(loss, full, rtol=1e-12)


def test_one_hot_label_is_textbook_cross_entropy():
    N, V = 7, 11
    z = _rand((N, V), 4, 2.0)
    y = np.random.default_rng(5).integers(0, V, N)
    idx = np.stack([y] + [(y + j) % V for j in range(1, 8)], axis=1)
    prob = np.zeros((N, 8))
    prob[:, 0] = 1.0
    loss, _ = orc.top_k_soft_cross_entropy(z, idx, prob, np.zeros(N))
    ref = torch.nn.functional.cross_entropy(torch.from_numpy(z), torch.from_numpy(y),
                                            reduction="none").numpy()
    np.testing.assert_allclose(loss, ref, rtol=1e-13)


def test_gibbs_on_the_bins():
    """The loss is the CE of two (k+1)-bin distributions: at least the label's bin entropy,
    with equality when the drafter logits equal the target logits."""
    d, V, N = 8, 40, 10
    W = _rand((d, V), 6, 0.8)
    Ht, Hd = _rand((N, d), 7), _rand((N, d), 8)
    lab = orc.label_readout(Ht, W)
    bins = np.concatenate([lab["prob"], lab["tail"][:, None]], axis=1)
    h_bins = np.array([sp_entropy(b) for b in bins])
    same, _ = orc.top_k_soft_cross_entropy(Ht @ W, lab["idx"], lab["prob"], lab["tail"])
    np.testing.assert_allclose(same, h_bins, rtol=1e-12)
    other, tail_q = orc.top_k_soft_cross_entropy(Hd @ W, lab["idx"], lab["prob"], lab["tail"])
    assert np.all(other > h_bins)
    q = orc.softmax(Hd @ W)
    np.testing.assert_allclose(tail_q + q[np.arange(N)[:, None], lab["idx"]].sum(1), 1.0,
                               rtol=1e-13)


def _topk_loss_of(Hd, W, idx, prob, tail, weight, lam):
    loss, _ = orc.top_k_soft_cross_entropy(Hd @ W, idx, prob, tail)
    return orc.weighted_loss(loss, weight, lam)[0]


def test_top_k_gradient_matches_central_differences():
    d, V, A, B, lam = 4, 13, 2, 3, 1.013441
    N = A * B
    W = _rand((d, V), 9, 0.9)
    Hd, Ht = _rand((N, d), 10), _rand((N, d), 11)
    lab = orc.label_readout(Ht, W, k=4)
    weight = orc.slot_weights(orc.MODE_ALR, B, 2.0, N, row_mask=np.array([1, 1, 0, 1, 1, 1.0]))
    G = orc.top_k_logit_grad(Hd @ W, lab["idx"], lab["prob"], lab["tail"], weight, lam)
    dHd, dW = orc.slot_loss_backward(Hd, W, G)
    args = (lab["idx"], lab["prob"], lab["tail"], weight, lam)
    eps = 1e-6
    for i, j in itertools.product(range(N), range(d)):
        e = np.zeros_like(Hd); e[i, j] = eps
        num = (_topk_loss_of(Hd + e, W, *args) - _topk_loss_of(Hd - e, W, *args)) / (2 * eps)
        np.testing.assert_allclose(dHd[i, j], num, rtol=1e-6, atol=1e-9)
    for i, j in itertools.product(range(d), range(V)):
        e = np.zeros_like(W); e[i, j] = eps
        num = (_topk_loss_of(Hd, W + e, *args) - _topk_loss_of(Hd, W - e, *args)) / (2 * eps)
        np.testing.assert_allclose(dW[i, j], num, rtol=1e-6, atol=1e-9)
    np.testing.assert_allclose(G.sum(axis=1), 0.0, atol=1e-15)


def test_top_k_gradient_with_empty_tail_is_the_full_gradient():
    """k = V: the gradient is the full-vocabulary q - p form."""
    d, V, N = 5, 7, 4
    W = _rand((d, V), 12, 0.6)
    Hd, Ht = _rand((N, d), 13), _rand((N, d), 14)
    lab = orc.label_readout(Ht, W, k=V)
    w = np.ones(N)
    G8 = orc.top_k_logit_grad(Hd @ W, lab["idx"], lab["prob"], lab["tail"], w, 1.0)
    G = orc.logit_grad(Hd @ W, Ht @ W, w, 1.0)
    np.testing.assert_allclose(G8, G, rtol=1e-12, atol=1e-16)
