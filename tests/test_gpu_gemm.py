"""The tensor-core GEMM of the backward (alr_gemm) against an fp64 product, for every operand
layout, both element types, with ragged M, N and K tails and with accumulation.  The largest
shape has more 256 x 256 tiles (81) than a GB300 holds CTA pairs, so pairs run several tiles
and cycle through both accumulator buffers."""

import itertools

import pytest
import torch

from paper_2609_38795_gb300 import alr, build_lib

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    build_lib.build()
    alr.lib()
    assert alr.alr_device_supported() == alr.ALR_OK, alr.alr_last_error()


def _operands(M, Nc, K, dtype, a_mn, b_mn, seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    A = torch.randn(M, K, generator=g, device="cuda").to(dtype)
    Bm = torch.randn(K, Nc, generator=g, device="cuda").to(dtype)
    A_st = A.t().contiguous() if a_mn else A.contiguous()        # [K, M] or [M, K]
    B_st = Bm.contiguous() if b_mn else Bm.t().contiguous()      # [K, Nc] or [Nc, K]
    ref = A.double() @ Bm.double()
    return A_st, B_st, ref


@pytest.mark.parametrize("form", ["single", "mcast", "mcast4", "pair"])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("a_mn,b_mn", list(itertools.product([False, True], repeat=2)))
@pytest.mark.parametrize("shape", [(200, 264, 200), (256, 512, 1024), (8, 8, 8),
                                   (2200, 2056, 520)])
def test_gemm_layouts(form, dtype, a_mn, b_mn, shape, monkeypatch):
    """Every form of the bf16 product (ALR_GEMM_FORM): single CTAs, clusters sharing B by
    multicast, CTA pairs with M = 256 products; fp32 (tf32) runs on single CTAs whatever the
    setting, so its cases check that a cluster-form setting leaves the tf32 path intact."""
    monkeypatch.setenv("ALR_GEMM_FORM", form)
    assert alr.alr_kernel_forms()[0] == form, alr.alr_cluster_forms_error()
    M, Nc, K = shape
    if dtype == torch.float32 and (a_mn or b_mn):
        A_st, B_st, _ = _operands(M, Nc, K, dtype, a_mn, b_mn, seed=1)
        C = torch.empty(M, Nc, device="cuda")
        with pytest.raises(alr.AlrError) as ei:            # tf32 products are K-major only
            alr.alr_gemm(A_st, B_st, C, M, Nc, K, a_mn=a_mn, b_mn=b_mn)
        assert ei.value.code == alr.ALR_ERR_UNSUPPORTED
        return
    A_st, B_st, ref = _operands(M, Nc, K, dtype, a_mn, b_mn, seed=M + Nc + K)
    C = torch.full((M, Nc), float("nan"), device="cuda")
    alr.alr_gemm(A_st, B_st, C, M, Nc, K, a_mn=a_mn, b_mn=b_mn, accumulate=False)
    torch.cuda.synchronize()
    tol = 1e-4 if dtype == torch.bfloat16 else 5e-3      # tf32 products for fp32 inputs
    err = (C.double() - ref).abs().max().item() / ref.abs().max().item()
    assert err <= tol, err
    # accumulate into the result: C + A B
    alr.alr_gemm(A_st, B_st, C, M, Nc, K, a_mn=a_mn, b_mn=b_mn, accumulate=True)
    torch.cuda.synchronize()
    err2 = (C.double() - 2 * ref).abs().max().item() / (2 * ref.abs().max().item())
    assert err2 <= tol, err2
    assert alr.alr_device_status() == alr.ALR_OK
