"""IRA block construction on the GPU against the oracle, bit for bit (Sec. 3.2, In-rollout
anchors; App. A): the anchor and offset draws from given random integers, the block plan they
drive, and the secondary blocks' context rows (the primaries' stored five-layer rollout
features of y*_1..y*_{j-1}) at the paper's sequence length and stored-row count."""

import numpy as np
import pytest
import torch

from oracle import alr_oracle as orc
from paper_2609_38795_gb300 import alr, build_lib
from tests import parity as P

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    build_lib.build()
    alr.lib()
    assert alr.alr_device_supported() == alr.ALR_OK, alr.alr_last_error()


def _u32(t):
    """The uint32 values an int32 tensor holds."""
    return t.cpu().numpy().view(np.uint32).astype(np.int64)


def _draws(S, L, K, max_b, density, seed):
    g = torch.Generator().manual_seed(seed)
    ok = (torch.rand(S, L, generator=g) < torch.tensor(density)[:, None]).to(torch.uint8)
    keys = torch.randint(-(1 << 31), 1 << 31, (S, L), generator=g, dtype=torch.int64).to(torch.int32)
    keys[0, :64] = 7                                      # equal keys: position order decides
    off_u = torch.randint(-(1 << 31), 1 << 31, (S, max_b // 2), generator=g,
                          dtype=torch.int64).to(torch.int32)
    out = dict(n_valid=torch.empty(S, dtype=torch.int32, device="cuda"),
               anchor_pos=torch.empty(S, max_b, dtype=torch.int32, device="cuda"),
               offsets=torch.empty(S, max_b // 2, dtype=torch.int32, device="cuda"))
    alr.alr_ira_draw(K, max_b, ok.cuda(), keys.cuda(), off_u.cuda(), out)
    torch.cuda.synchronize()
    ref = orc.ira_draw(ok.numpy(), _u32(keys), _u32(off_u), K, max_b)
    return out, ref, ok


@pytest.mark.parametrize("L", [1, 700, 4096])
def test_ira_draw_bit_exact(L):
    """Samples with no, few, exactly 128 and many valid positions; one with ties among keys."""
    K, max_b = 15, 128
    density = [0.0, 0.02, 128.5 / max(L, 1), 0.5, 1.0]
    out, (n_valid, anchor_pos, offsets), _ = _draws(5, L, K, max_b, density, seed=L)
    assert np.array_equal(P.npi(out["n_valid"]), n_valid)
    assert np.array_equal(P.npi(out["anchor_pos"]), anchor_pos)
    assert np.array_equal(P.npi(out["offsets"]), offsets)
    assert alr.alr_device_status() == alr.ALR_OK


def test_ira_plan_and_context_bit_exact():
    """Draws -> block plan -> context rows, at the paper's sequence length (4096), 128 anchors,
    K = 15 and 13 stored rows of five layers' features (d = 64 here), bf16; primary rollouts
    that end early, including one that ends before its secondary's offset."""
    S, L, K, max_b, C, layers, d = 6, 4096, 15, 128, 13, 5, 64
    Pn, H, F = max_b - max_b // 2, max_b // 2, layers * d
    out, (n_valid, anchor_pos, offsets), _ = _draws(S, L, K, max_b, [0.9, 0.01, 0.3, 0.05, 0.6, 0.02],
                                                   seed=9)
    g = torch.Generator().manual_seed(10)
    rlen = torch.full((S * Pn,), K, dtype=torch.int32)
    rlen[torch.randint(0, S * Pn, (40,), generator=g)] = torch.randint(1, K, (40,), generator=g,
                                                                        dtype=torch.int32)
    store = torch.randn(S * Pn, C, F, generator=g).to(torch.bfloat16)
    ctx = torch.full((S, H, C, F), 7.0, dtype=torch.bfloat16, device="cuda")
    ctx_len = torch.full((S, H), -5, dtype=torch.int32, device="cuda")
    prefix_end = torch.full((S, H), -5, dtype=torch.int32, device="cuda")
    alr.alr_ira_context(K, max_b, store.cuda(), out["n_valid"], rlen.cuda(), out["offsets"],
                        out["anchor_pos"], ctx, ctx_len, prefix_end)
    # the block plan from the same draws
    T = S * max_b
    plan = {k: torch.empty(T, dtype=torch.int32, device="cuda")
            for k in ("seq", "pos", "valid_len", "ctx_len")}
    alr.alr_ira_blocks(K, max_b, out["n_valid"], rlen.cuda(), out["offsets"], plan)
    torch.cuda.synchronize()
    c_ref, cl_ref, pe_ref = orc.ira_context(store.float().numpy(), n_valid, rlen.numpy().reshape(S, Pn),
                                            offsets, anchor_pos, K, max_b)
    assert torch.equal(ctx.float().cpu(), torch.from_numpy(c_ref).float())
    assert np.array_equal(P.npi(ctx_len), cl_ref)
    assert np.array_equal(P.npi(prefix_end), pe_ref)
    ref = orc.ira_blocks(n_valid, rlen.numpy().reshape(S, Pn), offsets, K, max_b)
    for k in ("seq", "pos", "valid_len", "ctx_len"):
        assert np.array_equal(P.npi(plan[k]).reshape(S, max_b), ref[k]), k
    # the plan's secondaries and the context agree on which blocks exist
    sec = (P.npi(plan["seq"]).reshape(S, max_b) >= 0) & (P.npi(plan["pos"]).reshape(S, max_b) > 0)
    assert sec.sum() == (pe_ref >= 0).sum()
    assert (cl_ref > 0).sum() > 100 and (rlen.numpy() < K).any()
    assert alr.alr_device_status() == alr.ALR_OK
