"""CPU oracle for the ALR slot-loss hot path.  TEST INFRASTRUCTURE ONLY.

This module is the plain, slow, fp64 statement of what the GPU path computes.  Only the
test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
or call it; the product path (the CUDA library and its Python binding) never does, and this
module imports nothing from the product package.

Every function takes the already-rounded inputs (bf16 or fp32 values) widened to float64 and
accumulates in float64.  Library primitives used as single steps: ``numpy.matmul`` (the
head projection and the gradient products), ``numpy.argmax`` (first index of the maximum).

Notation follows the paper ("Recovering Off-Policy Supervision for Speculative Decoding"):
an anchor block has slots k = 1..K predicted in parallel (Sec. 3).  A batch holds A anchors
with B rows each; buffer row r = a*B + s holds paper slot k = s + 1.  z_d = H_d W are the
drafter logits (q = softmax z_d), z_t = H_t W the target logits whose softmax p is the label
distribution pi_{a,k} (Eq. 3 for ALR rows, the corpus-prefix KD label of Sec. 3.1 otherwise).

Parity status: every function below is pinned by tests/test_oracle_pins.py against closed
forms, textbook special cases, finite differences or brute-force enumeration.
"""

from __future__ import annotations

import numpy as np

MODE_ALR = 0          # omega = w_k (Sec. 3.2: ALR keeps the envelope and omits the gate)
MODE_ERASE_SOFT = 1   # omega = w_k * g_{a,k}, soft survival gate (Eq. 2)
MODE_ERASE_HARD = 2   # omega = w_k * prod 1[x = greedy target]  (hard variant under Eq. 2)


def _f64(x):
    return np.asarray(x, dtype=np.float64)


# ----------------------------------------------------------------------------------------
# Eq. 1: slot envelope w_k = exp(-(k-1)/gamma)
# ----------------------------------------------------------------------------------------
def slot_envelope(B: int, gamma: float) -> np.ndarray:
    """Envelope of Eq. 1 for buffer slots s = 0..B-1 (paper slot k = s+1): exp(-s/gamma)."""
    k = np.arange(1, B + 1, dtype=np.float64)
    return np.exp(-(k - 1.0) / float(gamma))


# ----------------------------------------------------------------------------------------
# Head projection and the full-vocabulary normaliser
# ----------------------------------------------------------------------------------------
def head_logits(H, W) -> np.ndarray:
    """z = H W for H [N, d] and the vocabulary head W [d, V] (one matmul)."""
    return _f64(H) @ _f64(W)


def log_sum_exp(z) -> np.ndarray:
    """Row-wise log sum_v exp(z[r, v]), shifted by the row maximum for range safety."""
    z = _f64(z)
    m = z.max(axis=1, keepdims=True)
    return (m + np.log(np.exp(z - m).sum(axis=1, keepdims=True)))[:, 0]


def softmax(z) -> np.ndarray:
    z = _f64(z)
    return np.exp(z - log_sum_exp(z)[:, None])


# ----------------------------------------------------------------------------------------
# Soft cross-entropy l(pi, q) of Eq. 1, in its full-vocabulary form
# ----------------------------------------------------------------------------------------
def soft_cross_entropy(p, z_d) -> np.ndarray:
    """l_r = -sum_v p[r, v] log q[r, v] with log q = z_d - LSE(z_d)."""
    p = _f64(p)
    log_q = _f64(z_d) - log_sum_exp(z_d)[:, None]
    return -(p * log_q).sum(axis=1)


def entropy(p) -> np.ndarray:
    """H(p)_r = -sum_v p log p (terms with p = 0 contribute 0)."""
    p = _f64(p)
    safe = np.where(p > 0, p, 1.0)
    return -(p * np.log(safe)).sum(axis=1)


# ----------------------------------------------------------------------------------------
# Greedy choice with the paper's tie rule (App. A: greedy ties go to the lower token id)
# ----------------------------------------------------------------------------------------
def greedy(z):
    """Per row: the smallest index attaining the maximum, and the gap top1 - top2.

    top2 is the largest value at any other index, so an exact tie gives gap 0.  With V = 1
    there is no second value and the gap is +inf.
    """
    z = _f64(z)
    idx = np.argmax(z, axis=1)                  # numpy returns the first maximal index
    rows = np.arange(z.shape[0])
    top1 = z[rows, idx]
    if z.shape[1] == 1:
        return idx.astype(np.int64), np.full(z.shape[0], np.inf)
    rest = z.copy()
    rest[rows, idx] = -np.inf
    return idx.astype(np.int64), top1 - rest.max(axis=1)


# ----------------------------------------------------------------------------------------
# Eq. 2: survival gate of the erase comparator
# ----------------------------------------------------------------------------------------
def erase_gate(B, logp_x=None, corpus_tok=None, argmax_t=None, hard=False) -> np.ndarray:
    """g_{a,k} = prod_{1<=j<k} f_{a,j} per buffer row (Eq. 2).

    Buffer row s of anchor a carries the label of paper slot k = s+1, conditioned on the
    corpus prefix before position a+k, and corpus_tok[a*B+s] is the corpus token x_{a+k}
    that this label predicts.  So the factor for paper position a+j (j = s'+1) comes from
    row s' = j-1:
      soft: f = p_T(x_{a+j} | x_{<a+j}) = exp(logp_x[a*B+s'])
      hard: f = 1[x_{a+j} == greedy target after x_{<a+j}] = 1[corpus_tok == argmax_t] of row s'
    and row s multiplies the factors of rows s' < s; row 0 (slot 1) has the empty product 1.
    """
    if hard:
        f = (np.asarray(corpus_tok) == np.asarray(argmax_t)).astype(np.float64)
    else:
        f = np.exp(_f64(logp_x))
    f = f.reshape(-1, B)
    g = np.ones_like(f)
    for s in range(1, B):
        g[:, s] = g[:, s - 1] * f[:, s - 1]
    return g.reshape(-1)


def slot_weights(mode, B, gamma, N, row_mask=None, logp_x=None, corpus_tok=None,
                 argmax_t=None) -> np.ndarray:
    """omega_r of Eq. 1: envelope w_k, times the termination / IRA validity mask, times the
    erase gate of Eq. 2 in the erase modes (ALR omits the gate, Sec. 3.2)."""
    w = np.tile(slot_envelope(B, gamma), N // B)
    if row_mask is not None:
        w = w * _f64(row_mask)
    if mode == MODE_ERASE_SOFT:
        w = w * erase_gate(B, logp_x=logp_x)
    elif mode == MODE_ERASE_HARD:
        w = w * erase_gate(B, corpus_tok=corpus_tok, argmax_t=argmax_t, hard=True)
    return w


def weighted_loss(loss_row, weight, lam):
    """Eq. 1 scaled by the KD factor lambda: L = lam * sum omega l / sum omega (0 if sum omega = 0)."""
    weight = _f64(weight)
    wsum = weight.sum()
    if wsum == 0.0:
        return 0.0, 0.0
    return float(lam * (weight * _f64(loss_row)).sum() / wsum), float(wsum)


# ----------------------------------------------------------------------------------------
# Forward pass of the slot loss
# ----------------------------------------------------------------------------------------
def slot_loss_forward(Hd, Ht, W, B, mode=MODE_ALR, gamma=2.0, lam=1.0, row_mask=None,
                      corpus_tok=None):
    """All forward outputs of the slot loss for N = A*B rows.

    Returns a dict with z_d, z_t (kept for the backward), lse_d, lse_t, loss_row (l_r),
    ent_row (H(p_r)), argmax_d / argmax_t and gap_d / gap_t, logp_x (erase modes), weight
    (omega_r), loss_total (L) and weight_sum (sum omega).
    """
    Hd, Ht, W = _f64(Hd), _f64(Ht), _f64(W)
    N = Hd.shape[0]
    assert N % B == 0
    z_d = head_logits(Hd, W)
    z_t = head_logits(Ht, W)
    lse_d = log_sum_exp(z_d)
    lse_t = log_sum_exp(z_t)
    p = np.exp(z_t - lse_t[:, None])
    loss_row = soft_cross_entropy(p, z_d)
    ent_row = entropy(p)
    am_d, gap_d = greedy(z_d)
    am_t, gap_t = greedy(z_t)
    logp_x = None
    if mode in (MODE_ERASE_SOFT, MODE_ERASE_HARD):
        x = np.asarray(corpus_tok, dtype=np.int64)
        logp_x = z_t[np.arange(N), x] - lse_t
    weight = slot_weights(mode, B, gamma, N, row_mask=row_mask, logp_x=logp_x,
                          corpus_tok=corpus_tok, argmax_t=am_t)
    L, wsum = weighted_loss(loss_row, weight, lam)
    return dict(z_d=z_d, z_t=z_t, lse_d=lse_d, lse_t=lse_t, loss_row=loss_row,
                ent_row=ent_row, argmax_d=am_d, argmax_t=am_t, gap_d=gap_d, gap_t=gap_t,
                logp_x=logp_x, weight=weight, loss_total=L, weight_sum=wsum)


# ----------------------------------------------------------------------------------------
# Backward pass: gradient of L with respect to the drafter logits, H_d and W
# ----------------------------------------------------------------------------------------
def logit_grad(z_d, z_t, weight, lam, weight_sum=None) -> np.ndarray:
    """dL/dz_d[r, v] = lam * omega_r / sum omega * (q[r, v] - p[r, v]).

    From l_r = LSE(z_d) - sum_v p_v z_d,v: d l_r / d z_d,v = q_v - p_v.  The label p, the
    weights omega and the erase gate are target-side quantities and carry no gradient.
    weight_sum: the normaliser sum omega of Eq. 1 over the whole batch, when only some of its
    rows are passed (default: the sum of the given weights).
    """
    weight = _f64(weight)
    wsum = weight.sum() if weight_sum is None else float(weight_sum)
    if wsum == 0.0:
        return np.zeros_like(_f64(z_d))
    q = softmax(z_d)
    p = softmax(z_t)
    return (lam * weight / wsum)[:, None] * (q - p)


def slot_loss_backward(Hd, W, G, dW_in=None):
    """dH_d = G W^T and dW = dW_in + H_d^T G (the drafter path of z_d = H_d W)."""
    G, Hd, W = _f64(G), _f64(Hd), _f64(W)
    dHd = G @ W.T
    dW = Hd.T @ G
    if dW_in is not None:
        dW = dW + _f64(dW_in)
    return dHd, dW


# ----------------------------------------------------------------------------------------
# Accepted length (Sec. 3.2 and the MAT definition of Sec. 4)
# ----------------------------------------------------------------------------------------
def accept_len(argmax_d, argmax_t, B, active=None):
    """acc[a] = number of leading rows s with active[a*B+s] and argmax_d == argmax_t.

    A slot contributes only when every earlier slot matched, so the count stops at the first
    mismatch or inactive (masked) row.  hist[n] = #{a : acc[a] = n}, n = 0..B.
    """
    am_d = np.asarray(argmax_d).reshape(-1, B)
    am_t = np.asarray(argmax_t).reshape(-1, B)
    ok = am_d == am_t
    if active is not None:
        ok &= np.asarray(active).reshape(-1, B) > 0
    A = ok.shape[0]
    acc = np.zeros(A, dtype=np.int64)
    for a in range(A):
        n = 0
        while n < B and ok[a, n]:
            n += 1
        acc[a] = n
    hist = np.bincount(acc, minlength=B + 1).astype(np.int64)
    return acc, hist


# ----------------------------------------------------------------------------------------
# IRA placement (Eq. 4): gather slot features from a rollout feature buffer
# ----------------------------------------------------------------------------------------
def gather_ira_blocks(F, seq, pos, B, valid_len=None):
    """out[a*B+s] = F[seq_a, pos_a + s] and row_valid = 1 when that position exists.

    A row is invalid (zero features, row_valid 0) when seq_a is outside [0, S), pos_a < 0,
    or pos_a + s >= min(valid_len_a, L).  For an IRA secondary block at offset j inside a
    primary block's stored rows [K, d], pos = j and valid_len = K give exactly the indicator
    1[j + k <= K] of Eq. 4 (row s is paper slot k = s + 1 and reads primary row j + s).
    """
    F = np.asarray(F)
    S, L, d = F.shape
    A = len(seq)
    out = np.zeros((A * B, d), dtype=F.dtype)
    valid = np.zeros(A * B, dtype=np.float32)
    for a in range(A):
        sq, p0 = int(seq[a]), int(pos[a])
        lim = L if valid_len is None else min(int(valid_len[a]), L)
        if sq < 0 or sq >= S or p0 < 0:
            continue
        for s in range(B):
            if p0 + s < lim:
                out[a * B + s] = F[sq, p0 + s]
                valid[a * B + s] = 1.0
    return out, valid


def ira_supervised_slots(K: int, j: int) -> int:
    """Number of supervised slots of a secondary block at offset j (Eq. 4): #{k : j+k <= K}."""
    return sum(1 for k in range(1, K + 1) if j + k <= K)


# ----------------------------------------------------------------------------------------
# Compact labels: top-k target probabilities plus a tail bin (Sec. 3.1 under Eq. 1; App. A,
# KD loss and rollout label readout)
# ----------------------------------------------------------------------------------------
def label_readout(Ht, W, k=8, corpus_tok=None):
    """The label a rollout step keeps: the k most probable target tokens (probability
    descending, equal probabilities to the lower token id, App. A), their probabilities, the
    remaining mass (the tail bin) and the greedy token y* (the first of them).

    Returns idx [N, k] int64, prob [N, k], tail [N] (sum of p over the other tokens), lse_t,
    argmax_t, gap_t, and logp_x (log p of corpus_tok, for the erase gate) when given.
    """
    z_t = head_logits(Ht, W)
    N, V = z_t.shape
    lse_t = log_sum_exp(z_t)
    p = np.exp(z_t - lse_t[:, None])
    order = np.argsort(-z_t, axis=1, kind="stable")   # stable: equal logits keep id order
    idx = order[:, :k]
    rows = np.arange(N)[:, None]
    prob = p[rows, idx]
    outside = np.ones_like(p, dtype=bool)
    outside[rows, idx] = False
    tail = np.where(outside, p, 0.0).sum(axis=1)
    am_t, gap_t = greedy(z_t)
    logp_x = None
    if corpus_tok is not None:
        x = np.asarray(corpus_tok, dtype=np.int64)
        logp_x = z_t[np.arange(N), x] - lse_t
    return dict(z_t=z_t, idx=idx.astype(np.int64), prob=prob, tail=tail, lse_t=lse_t,
                argmax_t=am_t, gap_t=gap_t, logp_x=logp_x)


def top_k_soft_cross_entropy(z_d, idx, prob, tail):
    """l_r = -sum_i prob_i log q[idx_i] - tail * log(tail_q), the soft CE between the
    (k+1)-bin label (prob, tail) and the drafter's (q[idx], tail_q), with tail_q the drafter
    mass outside the label's k tokens.  A zero tail contributes nothing."""
    z_d = _f64(z_d)
    N, V = z_d.shape
    rows = np.arange(N)[:, None]
    log_q = z_d - log_sum_exp(z_d)[:, None]
    outside = np.ones((N, V), dtype=bool)
    outside[rows, idx] = False
    tail_q = np.where(outside, np.exp(log_q), 0.0).sum(axis=1)
    tail = _f64(tail)
    tail_term = np.where(tail > 0, tail * np.log(np.where(tail > 0, tail_q, 1.0)), 0.0)
    return -(_f64(prob) * log_q[rows, idx]).sum(axis=1) - tail_term, tail_q


def top_k_logit_grad(z_d, idx, prob, tail, weight, lam, weight_sum=None):
    """Gradient of Eq. 1 with the top-k + tail loss with respect to the drafter logits:
    c_r * (q_v - prob at v) for a label token v, c_r * q_v * (1 - tail / tail_q) otherwise,
    with c_r = lam * omega_r / sum omega (zero when sum omega = 0)."""
    z_d = _f64(z_d)
    N, V = z_d.shape
    weight = _f64(weight)
    wsum = weight.sum() if weight_sum is None else float(weight_sum)
    if wsum == 0.0:
        return np.zeros_like(z_d)
    rows = np.arange(N)[:, None]
    q = softmax(z_d)
    _, tail_q = top_k_soft_cross_entropy(z_d, idx, prob, tail)
    tail = _f64(tail)
    beta = 1.0 - np.where(tail > 0, tail / np.where(tail > 0, tail_q, 1.0), 0.0)
    G = q * beta[:, None]
    G[rows, idx] = q[rows, idx] - _f64(prob)
    return (lam * weight / wsum)[:, None] * G


# ----------------------------------------------------------------------------------------
# IRA block construction (Sec. 3.2, In-rollout anchors; Eq. 4; App. A)
# ----------------------------------------------------------------------------------------
def ira_blocks(valid_anchors, rollout_len, offsets, K, max_blocks=128, rollout_tok=None,
               corpus_anchor_tok=None):
    """Block plan of one batch of S samples.

    Sample s has v_s valid anchor positions and keeps m_s = min(v_s, max_blocks) blocks: the
    first ceil(m/2) are primary (they run the target rollout), the next floor(m/2) secondary;
    slots past m are unused.  Secondary block i sits in primary block i's rollout at offset
    j = offsets[s, i] in {2..K-1}.  Primary block p's stored rollout holds rollout_len[s, p]
    label rows (K, or fewer after early termination); a secondary whose offset lies past them
    (j > rollout_len) has no anchor token y*_j and stays unused.

    Per block (s, b), with P = max_blocks - max_blocks // 2 primary slots per sample, the
    gather of label rows from the primary label buffer viewed as [S * P, K, d]:
      primary p:      seq = s*P + p, pos = 0, valid_len = rollout_len[s, p]
      secondary i:    seq = s*P + i, pos = j, valid_len = rollout_len[s, i]
      unused:         seq = -1 (every row invalid)
    so row k of a secondary block reads primary row j + k - 1 and is supervised iff
    j + k <= rollout_len (Eq. 4's 1[j + k <= K] with early termination masked, Sec. 3.2).
    anchor_tok: the corpus token at the anchor (primary) or the rollout token y*_j (secondary);
    ctx_len: rollout features of y*_1..y*_{j-1} in the secondary context (0 for primaries).
    """
    S = len(valid_anchors)
    P = max_blocks - max_blocks // 2
    seq = np.full((S, max_blocks), -1, dtype=np.int64)
    pos = np.zeros((S, max_blocks), dtype=np.int64)
    vlen = np.zeros((S, max_blocks), dtype=np.int64)
    ctx = np.zeros((S, max_blocks), dtype=np.int64)
    tok = np.full((S, max_blocks), -1, dtype=np.int64)
    for s in range(S):
        m = min(int(valid_anchors[s]), max_blocks)
        n_prim = (m + 1) // 2
        for b in range(m):
            if b < n_prim:
                p, j = b, 0
            else:
                p, j = b - n_prim, int(offsets[s][b - n_prim])
                # an offset outside the rollout leaves the block unused: past K - 1, or past
                # the end of a primary rollout that terminated early, y*_j does not exist
                if j < 1 or j > K - 1 or j > int(rollout_len[s][p]):
                    continue
            seq[s, b] = s * P + p
            pos[s, b] = j
            vlen[s, b] = int(rollout_len[s][p])
            ctx[s, b] = max(j - 1, 0)
            if j == 0 and corpus_anchor_tok is not None:
                tok[s, b] = int(corpus_anchor_tok[s][b])
            if j > 0 and rollout_tok is not None:
                tok[s, b] = int(rollout_tok[s][p][j - 1])      # y*_j is rollout step j
    return dict(seq=seq, pos=pos, valid_len=vlen, ctx_len=ctx, anchor_tok=tok)


def ira_draw(anchor_ok, keys, offset_u, K, max_blocks=128):
    """The random draws of IRA (Sec. 3.2, In-rollout anchors; App. A: 128 anchors per sample,
    j ~ U{2, ..., K-1}), from uniform random numbers given as inputs.

    Anchors: sample s has v_s valid positions (anchor_ok[s, a] != 0); m_s = min(v_s,
    max_blocks) of them are drawn uniformly without replacement, as the valid positions in
    increasing order of their keys (uniform 32-bit integers; equal keys in position order),
    the first m_s taken, in that order.  Offsets: j = 2 + floor(u (K - 2) / 2^32) for a
    uniform 32-bit u, one per secondary slot.

    Returns n_valid [S], anchor_pos [S, max_blocks] (-1 past m_s), offsets [S, max_blocks // 2].
    """
    anchor_ok = np.asarray(anchor_ok)
    keys = np.asarray(keys, dtype=np.int64)
    S, L = anchor_ok.shape
    n_valid = np.zeros(S, dtype=np.int64)
    anchor_pos = np.full((S, max_blocks), -1, dtype=np.int64)
    for s in range(S):
        valid = [a for a in range(L) if anchor_ok[s, a]]
        n_valid[s] = len(valid)
        order = sorted(valid, key=lambda a: (int(keys[s, a]), a))
        for i, a in enumerate(order[:max_blocks]):
            anchor_pos[s, i] = a
    u = np.asarray(offset_u, dtype=np.int64).reshape(S, max_blocks // 2)
    offsets = 2 + (u * (K - 2)) // (1 << 32)
    return n_valid, anchor_pos, offsets


def ira_context(store, n_valid, rollout_len, offsets, anchor_pos, K, max_blocks=128):
    """Context of every secondary block (Sec. 3.2: the target representations of the corpus
    prefix up to the anchor a, then those stored for y*_1..y*_{j-1}; App. A: the rollout
    stores the outputs of the five target layers the drafter reads for y*_1..y*_13).

    store [S * P, C, F]: primary block p of sample s keeps C rows of F features (the five
    layers' outputs side by side), row r for rollout token y*_{r+1}.  Secondary i of sample s
    (i < floor(m_s / 2)) sits in primary i at offset j = offsets[s, i]; when 1 <= j <= K - 1
    and j <= rollout_len[s, i] it exists, its context takes the j - 1 rows of y*_1..y*_{j-1}
    and the corpus prefix ends at primary i's anchor anchor_pos[s, i].

    Returns ctx [S, H, C, F] (rows past the context zero), ctx_len [S, H], prefix_end [S, H]
    (-1 for a secondary slot without a block), with H = max_blocks // 2.
    """
    store = np.asarray(store)
    S = len(n_valid)
    P, H = max_blocks - max_blocks // 2, max_blocks // 2
    _, C, F = store.shape
    assert C >= K - 2, "the store must hold the rows of y*_1..y*_{K-2}"
    ctx = np.zeros((S, H, C, F), dtype=store.dtype)
    ctx_len = np.zeros((S, H), dtype=np.int64)
    prefix_end = np.full((S, H), -1, dtype=np.int64)
    for s in range(S):
        m = min(int(n_valid[s]), max_blocks)
        for i in range(m // 2):
            j = int(offsets[s][i])
            if j < 1 or j > K - 1 or j > int(rollout_len[s][i]):
                continue
            n = j - 1
            ctx[s, i, :n] = store[s * P + i, :n]
            ctx_len[s, i] = n
            prefix_end[s, i] = int(anchor_pos[s][i])
    return ctx, ctx_len, prefix_end
