"""Multi-rank host logic on CPU ranks (gloo, world size 2-4).

- Row sharding (data parallelism over anchors): with Eq. 1 normalised over the global batch,
  the product's collective steps (all-reduce of sum omega l and sum omega, backward with the
  batch's sum omega, all-reduce of the per-rank H_d^T G and of the histograms) reproduce the
  unsharded loss, dH, dW and accepted-length histogram.
- Vocabulary sharding: per-shard partial statistics (running max / sum-exp of both sides,
  label-weighted sums, greedy top-2) merged in rank order give the unsharded log-sum-exps,
  losses, entropies, argmaxes and gaps — the same merge the forward kernel applies across
  vocabulary splits.
- bench.py's max-over-ranks timing and whole-job throughput.
"""

import multiprocessing as mp
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist

from oracle import alr_oracle as orc


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(fn, rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        q.put((rank, fn(rank, world)))
    finally:
        dist.destroy_process_group()


def _run(fn, world):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(fn, r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    return [out[r] for r in range(world)]


def _problem(seed=0, d=12, V=37, A=6, B=4):
    rng = np.random.default_rng(seed)
    W = rng.standard_normal((d, V)) * 0.6
    Hd = rng.standard_normal((A * B, d))
    Ht = Hd + 0.5 * rng.standard_normal((A * B, d))
    mask = (rng.random(A * B) < 0.85).astype(np.float64)
    return Hd, Ht, W, mask, B


def _row_shard(rank, world):
    """One rank of a row-sharded batch: the product's sequence of collective steps
    (paper_2609_38795_gb300.sharded), with the oracle standing in for the library's compute on
    this CPU rank (the forward's partial sums, L from the reduced sums, the backward with the
    batch's sum omega, the accepted lengths)."""
    from paper_2609_38795_gb300 import sharded
    lam = 1.013441
    Hd, Ht, W, mask, B = _problem()
    A = Hd.shape[0] // B
    anchors = np.arange(rank, A, world)
    rows = (anchors[:, None] * B + np.arange(B)).reshape(-1)
    out = orc.slot_loss_forward(Hd[rows], Ht[rows], W, B, lam=lam, row_mask=mask[rows])   # 1
    sums = torch.tensor([(out["weight"] * out["loss_row"]).sum(), out["weight"].sum()],
                        dtype=torch.float64)
    sharded.reduce_sums(sums)                                                             # 2
    L = lam * float(sums[0]) / float(sums[1])                                             # 3
    G = orc.logit_grad(out["z_d"], out["z_t"], out["weight"], lam, weight_sum=float(sums[1]))
    dH, dW = orc.slot_loss_backward(Hd[rows], W, G)                                       # 4
    dW = torch.from_numpy(dW)
    sharded.reduce_weight_grad(dW)                                                        # 5
    _, hist = orc.accept_len(out["argmax_d"], out["argmax_t"], B, active=mask[rows])
    hist = torch.from_numpy(np.asarray(hist, dtype=np.int64))
    sharded.reduce_hist(hist)
    return L, dW.numpy(), rows, dH, hist.numpy()


@pytest.mark.parametrize("world", [2, 3, 4])
def test_row_sharded_loss_and_gradients_match_unsharded(world):
    """Every rank ends with the batch's L and dW; the ranks' dH rows together are the batch's
    dH; the reduced histogram counts every anchor of the batch."""
    res = _run(_row_shard, world)
    Hd, Ht, W, mask, B = _problem()
    lam = 1.013441
    full = orc.slot_loss_forward(Hd, Ht, W, B, lam=lam, row_mask=mask)
    G = orc.logit_grad(full["z_d"], full["z_t"], full["weight"], lam)
    dH, dW = orc.slot_loss_backward(Hd, W, G)
    _, hist = orc.accept_len(full["argmax_d"], full["argmax_t"], B, active=mask)
    dH_sharded = np.zeros_like(dH)
    for L, dW_r, rows, dH_r, hist_r in res:
        np.testing.assert_allclose(L, full["loss_total"], rtol=1e-13)
        np.testing.assert_allclose(dW_r, dW, rtol=1e-11, atol=1e-14)
        assert np.array_equal(hist_r, hist)
        dH_sharded[rows] = dH_r
    np.testing.assert_allclose(dH_sharded, dH, rtol=1e-12, atol=1e-15)


def _vocab_shard(rank, world):
    """Partial statistics of this rank's vocabulary shard, gathered to every rank."""
    Hd, Ht, W, _, _ = _problem(seed=1, V=53)
    V = W.shape[1]
    lo, hi = rank * V // world, (rank + 1) * V // world
    zd, zt = Hd @ W[:, lo:hi], Ht @ W[:, lo:hi]
    md, mt = zd.max(1), zt.max(1)
    et = np.exp(zt - mt[:, None])
    idx_d, idx_t = zd.argmax(1), zt.argmax(1)
    rows = np.arange(len(zd))

    def second(z, i):
        r = z.copy()
        r[rows, i] = -np.inf
        return r.max(1) if z.shape[1] > 1 else np.full(len(z), -np.inf)

    part = np.stack([md, np.exp(zd - md[:, None]).sum(1), mt, et.sum(1), (et * zd).sum(1),
                     (et * zt).sum(1), zd[rows, idx_d], idx_d + lo, second(zd, idx_d),
                     zt[rows, idx_t], idx_t + lo, second(zt, idx_t)], axis=1)
    t = torch.from_numpy(part)
    gathered = [torch.empty_like(t) for _ in range(world)]
    dist.all_gather(gathered, t)
    return np.stack([g.numpy() for g in gathered])          # [world, rows, 12]


def _merge(parts):
    """Merge per-shard statistics in rank order: rescale sums to the common maximum; the
    larger leader wins and equal leaders go to the lower token id."""
    Md = Mt = -np.inf
    Sd = St = U = Wt = 0.0
    bd = bt = sd_ = st_ = -np.inf
    id_ = it = None
    for p in parts:
        md, sd, mt, s_t, u, w, b2, i2, s2, b3, i3, s3 = p
        n = max(Md, md)
        Sd = Sd * np.exp(Md - n) + sd * np.exp(md - n)
        Md = n
        n = max(Mt, mt)
        f_old, f_new = np.exp(Mt - n), np.exp(mt - n)
        St, U, Wt = St * f_old + s_t * f_new, U * f_old + u * f_new, Wt * f_old + w * f_new
        Mt = n
        if b2 > bd or (b2 == bd and i2 < id_):
            sd_, bd, id_ = max(bd, s2), b2, i2
        else:
            sd_ = max(sd_, b2)
        if b3 > bt or (b3 == bt and i3 < it):
            st_, bt, it = max(bt, s3), b3, i3
        else:
            st_ = max(st_, b3)
    lse_d, lse_t = Md + np.log(Sd), Mt + np.log(St)
    return lse_d, lse_t, lse_d - U / St, lse_t - Wt / St, int(id_), int(it), bd - sd_, bt - st_


@pytest.mark.parametrize("world", [2, 4])
def test_vocab_sharded_statistics_merge_matches_unsharded(world):
    res = _run(_vocab_shard, world)
    Hd, Ht, W, _, B = _problem(seed=1, V=53)
    full = orc.slot_loss_forward(Hd, Ht, W, B)
    for gathered in res:
        for r in range(gathered.shape[1]):
            lse_d, lse_t, loss, ent, am_d, am_t, gap_d, gap_t = _merge(gathered[:, r, :])
            np.testing.assert_allclose([lse_d, lse_t, loss, ent],
                                       [full["lse_d"][r], full["lse_t"][r], full["loss_row"][r],
                                        full["ent_row"][r]], rtol=1e-12)
            assert (am_d, am_t) == (full["argmax_d"][r], full["argmax_t"][r])
            np.testing.assert_allclose([gap_d, gap_t], [full["gap_d"][r], full["gap_t"][r]],
                                       rtol=1e-12, atol=1e-12)


def _bench_reduce(rank, world):
    import bench
    ms = [10.0 + rank, 20.0 - rank]
    slowest = bench.max_over_ranks(ms, "cpu")
    return slowest, bench.job_rows_per_s(world, 32768, 10, slowest[0])


def test_bench_takes_the_slowest_rank():
    res = _run(_bench_reduce, 3)
    for slowest, rps in res:
        assert slowest == [12.0, 20.0]
        assert rps == pytest.approx(3 * 32768 * 10 / 0.012)
