"""Pins of the oracle's IRA draws and context assembly (Sec. 3.2, In-rollout anchors;
App. A: 128 anchors per sample, j ~ U{2..14}, rollout features of five layers stored for
y*_1..y*_13), on CPU.

- The anchor draw is uniform without replacement: over many seeded draws, every valid
  position is drawn with frequency m/v and every ordered pair of first two draws is equally
  likely; invalid positions never are; v <= 128 draws every valid position.
- The offset rule maps uniform 32-bit integers onto {2, ..., K-1} with counts equal to within
  two on an even grid over the 2^32 values, and the drawn offsets supervise seven slots on
  average (the paper's statement).
- The context of a secondary block is its primary's stored rows y*_1..y*_{j-1}, checked index
  by index on a store whose entries encode their own coordinates, and the corpus prefix of
  its primary's anchor: context positions a + 1 + (j - 1).
"""

import json
import os
from collections import Counter

import numpy as np

from oracle import alr_oracle as orc

HERE = os.path.dirname(os.path.abspath(__file__))
P = {k: v["value"] for k, v in json.load(open(os.path.join(HERE, "golden", "paper_constants.json"))).items()
     if isinstance(v, dict)}


def test_anchor_draw_is_uniform_without_replacement():
    L, max_b, n_draws = 12, 3, 20000
    ok = np.zeros((1, L), dtype=np.uint8)
    valid = [1, 2, 4, 5, 8, 9, 11]
    ok[0, valid] = 1
    rng = np.random.default_rng(0)
    single, pairs = Counter(), Counter()
    for _ in range(n_draws):
        keys = rng.integers(0, 1 << 32, size=(1, L), dtype=np.int64)
        n_valid, pos, _ = orc.ira_draw(ok, keys, np.zeros((1, 1)), 15, max_b)
        drawn = pos[0].tolist()
        assert n_valid[0] == len(valid)
        assert len(set(drawn)) == max_b and set(drawn) <= set(valid)
        single.update(drawn)
        pairs[tuple(drawn[:2])] += 1
    v = len(valid)
    for a in valid:                                   # each position drawn w.p. m / v
        f = single[a] / n_draws
        assert abs(f - max_b / v) < 4 * np.sqrt(max_b / v * (1 - max_b / v) / n_draws)
    exp = n_draws / (v * (v - 1))                     # each ordered pair equally likely
    assert len(pairs) == v * (v - 1)
    assert all(abs(c - exp) < 5 * np.sqrt(exp) for c in pairs.values())


def test_anchor_draw_takes_every_valid_position_when_there_are_few():
    L = 300
    rng = np.random.default_rng(1)
    ok = (rng.random((3, L)) < np.array([[0.0], [0.3], [0.9]])).astype(np.uint8)
    keys = rng.integers(0, 1 << 32, size=(3, L), dtype=np.int64)
    n_valid, pos, _ = orc.ira_draw(ok, keys, np.zeros((3, 64)), 15, P["anchors_per_sample"])
    for s in range(3):
        v = int(ok[s].sum())
        assert n_valid[s] == v
        m = min(v, P["anchors_per_sample"])
        assert (pos[s] >= 0).sum() == m and np.all(pos[s, m:] == -1)
        if v <= P["anchors_per_sample"]:
            assert sorted(pos[s, :m].tolist()) == np.flatnonzero(ok[s]).tolist()
        else:                                         # the m smallest keys, in key order
            drawn_keys = keys[s, pos[s, :m]]
            assert np.all(np.diff(drawn_keys) >= 0)
            rest = np.setdiff1d(np.flatnonzero(ok[s]), pos[s, :m])
            assert keys[s, rest].min() >= drawn_keys.max()


def test_offsets_are_uniform_on_2_to_K_minus_1():
    K = P["K"]
    n = 13 * 7919                                     # grid of u evenly over [0, 2^32)
    u = (np.arange(n, dtype=np.int64) * (1 << 32)) // n
    _, _, j = orc.ira_draw(np.zeros((1, 1)), np.zeros((1, 1)), u.reshape(1, n), K, 2 * n)
    j = j.reshape(-1)
    assert j.min() == P["ira_offset_min"] and j.max() == P["ira_offset_max"] == K - 1
    counts = np.bincount(j, minlength=K)[2:K]
    assert counts.max() - counts.min() <= 2          # grid points and bin edges both rounded
    _, _, jj = orc.ira_draw(np.zeros((1, 1)), np.zeros((1, 1)),
                            np.array([[0, (1 << 32) - 1]]), K, 4)
    assert jj.tolist() == [[2, K - 1]]
    slots = np.mean([orc.ira_supervised_slots(K, x) for x in j])
    assert abs(slots - P["ira_mean_supervised_slots"]) < 1e-3


def test_secondary_context_is_the_primary_rollout_prefix():
    K, max_b = P["K"], 8
    C, layers, d = P["stored_rollout_rows"], P["feature_layers"], 3
    Pn, H = max_b - max_b // 2, max_b // 2
    S = 3
    n_valid = np.array([8, 5, 300])                   # m = 8, 5 (2 secondaries), 8
    rng = np.random.default_rng(2)
    offsets = rng.integers(2, K, size=(S, H))
    offsets[0, 0], offsets[0, 1] = 2, K - 1           # the shortest and the longest contexts
    rlen = np.full((S, Pn), K)
    rlen[2, 3] = 4
    offsets[2, 3] = 9                                 # past an early-terminated rollout
    anchor_pos = rng.integers(0, 4096, size=(S, max_b))
    F = layers * d
    # every store entry encodes (primary, row, feature)
    store = (np.arange(S * Pn)[:, None, None] * 10000 + np.arange(C)[None, :, None] * 100
             + np.arange(F)[None, None, :]).astype(np.float64)
    ctx, ctx_len, prefix_end = orc.ira_context(store, n_valid, rlen, offsets, anchor_pos, K, max_b)
    assert store.shape[1] == K - 2 == C               # y*_1..y*_13 for K = 15
    for s in range(S):
        m = min(int(n_valid[s]), max_b)
        for i in range(H):
            j = offsets[s, i]
            if i >= m // 2 or j > rlen[s, i]:
                assert ctx_len[s, i] == 0 and prefix_end[s, i] == -1
                assert not ctx[s, i].any()
                continue
            assert ctx_len[s, i] == j - 1 and 1 <= j - 1 <= C
            a = anchor_pos[s, i]
            assert prefix_end[s, i] == a
            # context positions: the corpus prefix x_0..x_a, then y*_1..y*_{j-1}
            assert (prefix_end[s, i] + 1) + ctx_len[s, i] == a + j
            for r in range(C):
                for f in range(F):
                    want = (s * Pn + i) * 10000 + r * 100 + f if r < j - 1 else 0
                    assert ctx[s, i, r, f] == want
