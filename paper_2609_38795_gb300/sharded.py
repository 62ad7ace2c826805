"""Row-sharded (data-parallel) slot loss: the anchors of one batch spread over several ranks.

Eq. 1 normalises the weighted soft cross-entropy over the whole batch, L = lambda * sum omega l
/ sum omega, so the ranks that share a batch (App. A trains with FSDP data parallelism) need
one exchange between forward and backward and one after it:

  1. forward on the rank's own anchors -> its partial sums (sum omega l, sum omega);
  2. all-reduce (sum) of those two floats;
  3. L of the batch from the reduced sums (``alr_loss_from_sums``);
  4. backward with the reduced sum omega as the normaliser, so that the rank's
     G = lambda omega_r / sum omega (q - p) is its rows' share of the batch gradient; dH of
     its rows is final;
  5. all-reduce (sum) of dW = H_d^T G, a sum over rows (or a reduce-scatter when the head
     itself is sharded), and of the accepted-length histogram.

Every computation runs in libalr; the collectives are ``torch.distributed`` calls on the
tensors the library wrote (NCCL on GPUs).  ``RowShardedSlotLoss`` runs the sequence through a
process group; ``reduce_sums`` / ``reduce_weight_grad`` / ``reduce_hist`` are the collective
steps on their own.
"""

from __future__ import annotations

import torch
import torch.distributed as dist

from . import alr


def reduce_sums(sums, group=None):
    """Step 2: sum the per-rank [sum omega l, sum omega] (one float32 tensor of 2) in place."""
    dist.all_reduce(sums, op=dist.ReduceOp.SUM, group=group)
    return sums


def reduce_weight_grad(dW, group=None):
    """Step 5: sum the per-rank head gradients in place (every rank gets the batch's dW)."""
    dist.all_reduce(dW, op=dist.ReduceOp.SUM, group=group)
    return dW


def reduce_hist(hist, group=None):
    """Accepted-length histograms of the ranks' anchors, added up in place."""
    dist.all_reduce(hist, op=dist.ReduceOp.SUM, group=group)
    return hist


class RowShardedSlotLoss:
    """One rank's part of a row-sharded batch.

    ``forward`` runs the local forward, reduces the two sums over ``group`` and writes the
    batch's L to ``self.loss``; ``backward`` runs the local backward with the batch's sum omega
    and reduces dW.  The per-rank steps are also exposed (``forward_local``, ``finalize``,
    ``backward_local``) so that one process can stand in for several ranks by summing their
    ``sums`` itself."""

    def __init__(self, N, d, V, B, group=None, **slot_loss_kw):
        self.sl = alr.SlotLoss(N, d, V, B, **slot_loss_kw)
        self.group = group
        dev = self.sl.device
        self.sums = torch.zeros(2, dtype=torch.float32, device=dev)   # [sum omega l, sum omega]
        self.loss = torch.zeros(1, dtype=torch.float32, device=dev)

    def forward_local(self, Hd, Ht, W, row_mask=None, corpus_tok=None):
        """Step 1: this rank's forward; returns its sums [sum omega l, sum omega]."""
        out = self.sl.forward(Hd, Ht, W, row_mask=row_mask, corpus_tok=corpus_tok)
        self.sums[0:1].copy_(out["wl_sum"])
        self.sums[1:2].copy_(out["weight_sum"])
        return self.sums

    def finalize(self, sums):
        """Step 3: the batch's L from reduced sums."""
        alr.alr_loss_from_sums(sums[0:1], sums[1:2], self.sl.lam, self.loss)
        return self.loss

    def backward_local(self, sums, Hd, Ht, W, dHd, dW=None):
        """Step 4: this rank's backward with the batch's normaliser sums[1]; dHd of its rows,
        and H_d^T G of its rows added to dW."""
        self.sl.backward(Hd, Ht, W, dHd, dW, weight_sum=sums[1:2])

    def forward(self, Hd, Ht, W, row_mask=None, corpus_tok=None):
        self.forward_local(Hd, Ht, W, row_mask=row_mask, corpus_tok=corpus_tok)
        reduce_sums(self.sums, self.group)
        return self.finalize(self.sums)

    def backward(self, Hd, Ht, W, dHd, dW):
        """dW is reduced over the group after the local backward: pass this rank's
        accumulation buffer (zero, or its running sum of earlier steps' local terms)."""
        self.backward_local(self.sums, Hd, Ht, W, dHd, dW)
        reduce_weight_grad(dW, self.group)

    def accept(self, active=None):
        acc, hist = self.sl.accept(active=active)
        reduce_hist(hist, self.group)
        return acc, hist
