"""The GEMM entry point that allocates nothing (for callers that cannot call cudaMalloc: all
device memory owned by another allocator, or a loop that must not pay its synchronisation).

Its split-K partials live in the library's fixed 8 MiB device array.  Checked through the C
ABI against vla_op_gemm_bf16 with a caller workspace, on two calls in a row (the second call
reuses the array the first one left behind, and a first call fills it with NaN partials): the
two entry points agree bit for bit, and both are within the GEMM tolerance of fp64.
This file is collected last so that a failure here leaves every other test already run."""
import math

import pytest
import torch

from paper_2505_18719_gb300 import inputs as I
from paper_2505_18719_gb300 import vla as V

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    from paper_2505_18719_gb300 import build
    build.build()
    return V.load()


def _operands(M, N, K, seed):
    A = I.normal_bf16((M, K), seed, 1, 1.0).cuda()
    A_lo = I.normal_bf16((M, K), seed, 2, 2.0 ** -9).cuda()
    W = I.normal_bf16((N, K), seed, 3, 1.0).cuda()
    return A, A_lo, W


def _poison_scratch():
    """A call whose partials are all NaN, with more splits and a larger M x N than the checked
    cases, so the scratch holds NaN wherever a later call could read a partial it did not write."""
    M, N, K, splits = 96, 512, 2048, 16
    A = torch.full((M, K), float("nan"), dtype=torch.bfloat16, device="cuda")   # NaN partials
    W = torch.ones(N, K, dtype=torch.bfloat16, device="cuda")
    C = torch.zeros(M, N, dtype=torch.float32, device="cuda")
    assert V.vla_op_gemm_bf16_noalloc(A.data_ptr(), 0, K, W.data_ptr(), K, C.data_ptr(), N, M, N, K, 128,
                                      splits, 0) == 0, V.vla_last_error()
    torch.cuda.synchronize()
    assert torch.isnan(C).all()


def test_noalloc_matches_workspace_entry_point_on_two_calls():
    # Both entry points run the same kernels and the same fixed-order split-K reduction, so the
    # results must agree bit for bit; a partial read but never rewritten would show as NaN.
    _poison_scratch()
    cases = [(64, 384, 4096, 128, 5, True), (130, 200, 688, 128, 2, False)]
    for i, (M, N, K, bn, splits, split_a) in enumerate(cases):
        A, A_lo, W = _operands(M, N, K, 500 + i)
        lo = A_lo.data_ptr() if split_a else 0
        ws = torch.empty(splits * M * N, dtype=torch.float32, device="cuda")
        C_ref = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
        C_na = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
        assert V.vla_op_gemm_bf16(A.data_ptr(), lo, K, W.data_ptr(), K, C_ref.data_ptr(), N, M, N, K, bn,
                                  splits, ws.data_ptr(), 0) == 0, V.vla_last_error()
        assert V.vla_op_gemm_bf16_noalloc(A.data_ptr(), lo, K, W.data_ptr(), K, C_na.data_ptr(), N, M, N,
                                          K, bn, splits, 0) == 0, V.vla_last_error()
        torch.cuda.synchronize()
        assert torch.isfinite(C_na).all()
        assert torch.equal(C_na, C_ref), (i, (C_na - C_ref).abs().max().item())
        # and both against fp64, with the GEMM tolerance of the other tests
        ref = ((A.double() + A_lo.double()) if split_a else A.double()) @ W.double().T
        err = (C_na.double() - ref).abs().max().item()
        assert err < 2e-5 * math.sqrt(K) * 8, (i, err)


def test_noalloc_rejects_sizes_beyond_the_scratch():
    M, N, K = 512, 4096, 512
    A, _, W = _operands(M, N, K, 900)
    C = torch.zeros(M, N, dtype=torch.float32, device="cuda")
    # 2 * 512 * 4096 * 4 bytes = 16 MiB > 8 MiB
    rc = V.vla_op_gemm_bf16_noalloc(A.data_ptr(), 0, K, W.data_ptr(), K, C.data_ptr(), N, M, N, K, 128, 2, 0)
    assert rc == V.VLA_ERR_CAPACITY
    assert "8 MiB" in V.vla_last_error()
    torch.cuda.synchronize()
    assert C.abs().max().item() == 0.0        # nothing ran
