"""The row-sharded form of the slot loss through the C ABI (App. A: data-parallel training),
with one GPU standing in for P ranks: the batch's anchors are split into P uneven parts, each
part runs its own forward, the parts' (sum omega l, sum omega) are added up as an all-reduce
would, every part finalises L from the sums and runs its backward with the batch's sum omega,
and the parts' dW are added up.  The result must be the unsplit batch's: L, every dH row and
dW against the oracle (1e-3 relative, 2e-2 max-norm) and against the unsplit GPU run."""

import numpy as np
import pytest
import torch

from oracle import alr_oracle as orc
from paper_2609_38795_gb300 import alr, build_lib, sharded, synthetic
from tests import parity as P

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    build_lib.build()
    alr.lib()
    assert alr.alr_device_supported() == alr.ALR_OK, alr.alr_last_error()


def _split(A, parts):
    """Uneven contiguous anchor ranges: the first parts one anchor larger."""
    sizes = [A // parts + (1 if i < A % parts else 0) for i in range(parts)]
    edges = np.cumsum([0] + sizes)
    return [(edges[i], edges[i + 1]) for i in range(parts)]


@pytest.mark.parametrize("parts", [2, 3, 4])
@pytest.mark.parametrize("mode,keep", [(alr.ALR_MODE_ALR, True), (alr.ALR_MODE_ALR, False),
                                       (alr.ALR_MODE_ERASE_SOFT, True)])
def test_row_sharded_batch_matches_unsplit(parts, mode, keep):
    A, B, d, V, lam = 11, 16, 320, 5000, 1.013441
    b = synthetic.slot_batch(d, V, A, B, 0.5, device="cuda", seed=70 + parts)
    Hd, Ht, W = b["Hd"], b["Ht"], b["W"]
    N = A * B
    mask = torch.ones(N, device="cuda")
    mask[7::B] = 0.0
    tok = None
    if mode != alr.ALR_MODE_ALR:
        tok = torch.randint(0, V, (N,), dtype=torch.int32, device="cuda",
                            generator=torch.Generator(device="cuda").manual_seed(3))
    # every part's forward, then the sums an all-reduce would give every rank
    shards, total = [], torch.zeros(2, device="cuda")
    for a0, a1 in _split(A, parts):
        r0, r1 = a0 * B, a1 * B
        sh = sharded.RowShardedSlotLoss(r1 - r0, d, V, B, mode=mode, lam=lam, keep_logits=keep)
        total += sh.forward_local(Hd[r0:r1], Ht[r0:r1], W, row_mask=mask[r0:r1],
                                  corpus_tok=None if tok is None else tok[r0:r1]).clone()
        shards.append((sh, r0, r1))
    dH = torch.empty(N, d, device="cuda")
    dW = torch.zeros(d, V, device="cuda")
    losses = []
    for sh, r0, r1 in shards:
        losses.append(sh.finalize(total).clone())
        dW_part = torch.zeros(d, V, device="cuda")
        sh.backward_local(total, Hd[r0:r1], Ht[r0:r1], W, dH[r0:r1], dW_part)
        dW += dW_part                                   # the all-reduce of step 5
    torch.cuda.synchronize()
    assert alr.alr_device_status() == alr.ALR_OK

    r = orc.slot_loss_forward(P.np64(Hd), P.np64(Ht), P.np64(W), B, mode=mode, lam=lam,
                              row_mask=P.np64(mask), corpus_tok=None if tok is None else P.npi(tok))
    G = orc.logit_grad(r["z_d"], r["z_t"], r["weight"], lam)
    dH_r, dW_r = orc.slot_loss_backward(P.np64(Hd), P.np64(W), G)
    for L in losses:
        assert abs(L.item() - r["loss_total"]) <= P.LOSS_RTOL * abs(r["loss_total"])
    np.testing.assert_allclose(total[1].item(), r["weight_sum"], rtol=1e-5)
    assert P.max_norm_rel(P.np64(dH), dH_r) <= P.GRAD_RTOL
    assert P.max_norm_rel(P.np64(dW), dW_r) <= P.GRAD_RTOL

    # the unsplit batch on the GPU: the same L and the same gradients up to rounding order
    whole = alr.SlotLoss(N, d, V, B, mode=mode, lam=lam, keep_logits=keep)
    whole.forward(Hd, Ht, W, row_mask=mask, corpus_tok=tok)
    dH1 = torch.empty(N, d, device="cuda")
    dW1 = torch.zeros(d, V, device="cuda")
    whole.backward(Hd, Ht, W, dH1, dW1)
    torch.cuda.synchronize()
    for L in losses:
        assert abs(L.item() - whole.out["loss_total"].item()) <= 1e-5 * abs(r["loss_total"])
    assert P.max_norm_rel(P.np64(dH), P.np64(dH1)) <= 1e-3
    assert P.max_norm_rel(P.np64(dW), P.np64(dW1)) <= 1e-3


def test_loss_from_sums():
    """L = lambda * wl / ws, and 0 when no slot of the batch is supervised."""
    f = lambda v: torch.tensor([v], dtype=torch.float32, device="cuda")  # noqa: E731
    out = f(-1.0)
    alr.alr_loss_from_sums(f(3.0), f(4.0), 1.5, out)
    torch.cuda.synchronize()
    assert out.item() == pytest.approx(1.125, rel=1e-7)
    alr.alr_loss_from_sums(f(0.0), f(0.0), 1.5, out)
    torch.cuda.synchronize()
    assert out.item() == 0.0
