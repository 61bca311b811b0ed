"""Failure detection without a GPU fault: the error paths are driven from the host.

* A kernel launch made to fail on the host (vla_test_inject_launch_error: the n-th launch
  returns a CUDA error without launching) surfaces as VLA_ERR_CUDA from vla_prefill /
  vla_decode_actions, leaves the handle's bookkeeping where it was, and the same calls then
  reproduce a clean run bit for bit.
* A bounded pipeline wait that nothing completes (vla_test_stall_next_gemm: CTA 0 of the next
  tile GEMM leaves one stage unfilled) runs out after a short limit: the status word gets
  VLA_STATUS_TIMEOUT, the other CTAs finish, and the context stays usable.
* An activation beyond the fp16 range is saturated with VLA_STATUS_SATURATED raised, in the
  RMSNorm op and end to end through a handle whose first norm gain is huge.
"""
import math

import numpy as np
import pytest
import torch

from paper_2505_18719_gb300 import inputs as I
from paper_2505_18719_gb300 import vla as V
from tests import parity as P

pytestmark = pytest.mark.gpu
WL = I.WORKLOADS["tiny_b4"]
CUDA_ERROR_LAUNCH_OUT_OF_RESOURCES = 701


@pytest.fixture(scope="module")
def wdev():
    from paper_2505_18719_gb300 import build
    build.build()
    V.load()
    return P.weights_to_device(I.make_weights(WL.shape, WL.weight_seed))


@pytest.fixture(autouse=True)
def disarm():
    yield
    V.vla_test_inject_launch_error(0, 0)
    V.vla_test_set_wait_limit_ns(0)


def _turn(pol, inp, forced=None):
    vis, ids = inp.visual.cuda(), inp.ids.cuda()
    pol.prefill(vis, ids, inp.lengths)
    out = pol.decode(inp.uniforms.cuda(), WL.temperature, forced=forced)
    pol.sync()
    return {k: v.cpu() for k, v in out.items() if v is not None}


def _same(a, b):
    for k in ("tokens", "logprobs", "actions", "logits"):
        assert torch.equal(a[k], b[k]), k


def test_injected_launch_error_leaves_handle_consistent(wdev):
    inp = I.make_turn_inputs(WL, 0)
    pol = V.Policy(WL.shape, wdev, WL.batch, 128, 512)
    ref = _turn(pol, inp)
    n_prefill = None
    # a prefill whose 5th kernel launch fails
    pol.reset()
    assert V.vla_test_inject_launch_error(5, CUDA_ERROR_LAUNCH_OUT_OF_RESOURCES) == 0
    with pytest.raises(V.VlaError) as ei:
        pol.prefill(inp.visual.cuda(), inp.ids.cuda(), inp.lengths)
    assert ei.value.code == V.VLA_ERR_CUDA and "701" in str(ei.value)
    assert all(V.vla_context_length(pol.h, b) == 0 for b in range(WL.batch))
    assert V.vla_sync(pol.h) == 0                    # nothing pending on the device side
    out = _turn(pol, inp)                            # the same turn again: identical results
    _same(out, ref)
    # a decode whose 20th kernel launch fails, after a good prefill
    pol.reset()
    pol.prefill(inp.visual.cuda(), inp.ids.cuda(), inp.lengths)
    lens = [V.vla_context_length(pol.h, b) for b in range(WL.batch)]
    assert V.vla_test_inject_launch_error(20, CUDA_ERROR_LAUNCH_OUT_OF_RESOURCES) == 0
    with pytest.raises(V.VlaError) as ei:
        pol.decode(inp.uniforms.cuda(), WL.temperature)
    assert ei.value.code == V.VLA_ERR_CUDA
    assert [V.vla_context_length(pol.h, b) for b in range(WL.batch)] == lens
    out = pol.decode(inp.uniforms.cuda(), WL.temperature)
    pol.sync()
    _same({k: v.cpu() for k, v in out.items() if v is not None}, ref)
    pol.close()


def test_gemm_wait_timeout_sets_status_and_recovers():
    M, N, K = 256, 512, 1024        # 2 x 2 output tiles of 128 x 256, one per CTA
    A = (I.normal_bf16((M, K), 71, 1, 1.0).float()).half().cuda()
    W = (I.normal_bf16((N, K), 71, 2, 1.0).float()).half().cuda()
    ref = A.double().cpu() @ W.double().cpu().T
    assert V.vla_op_read_status()[0] == 0                       # start from a clear word
    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    assert V.vla_test_set_wait_limit_ns(500_000) == 0          # 0.5 ms per wait
    assert V.vla_test_stall_next_gemm() == 0
    assert V.vla_op_gemm_f16(A.data_ptr(), 0, K, W.data_ptr(), K, C.data_ptr(), N, M, N, K, 256, 1, 0, 0) == 0
    rc, st = V.vla_op_read_status()
    assert rc == 0 and st & V.VLA_STATUS_TIMEOUT, st
    Cc = C.cpu()
    assert torch.isnan(Cc[:128, :256]).all()                   # CTA 0 wrote nothing
    tol = 2e-5 * math.sqrt(K) * 8
    for (r0, c0) in ((0, 256), (128, 0), (128, 256)):         # the other CTAs finished normally
        err = (Cc[r0:r0 + 128, c0:c0 + 256].double() - ref[r0:r0 + 128, c0:c0 + 256]).abs().max().item()
        assert err < tol, (r0, c0, err)
    # the context is usable: the same call, no stall, default limit
    assert V.vla_test_set_wait_limit_ns(0) == 0
    C.fill_(float("nan"))
    assert V.vla_op_gemm_f16(A.data_ptr(), 0, K, W.data_ptr(), K, C.data_ptr(), N, M, N, K, 256, 1, 0, 0) == 0
    rc, st = V.vla_op_read_status()
    assert rc == 0 and st == 0
    assert (C.cpu().double() - ref).abs().max().item() < tol


def test_engine_reports_gemm_timeout_then_runs_clean(wdev):
    inp = I.make_turn_inputs(WL, 0)
    pol = V.Policy(WL.shape, wdev, WL.batch, 128, 512)
    ref = _turn(pol, inp)
    pol.reset()
    assert V.vla_test_set_wait_limit_ns(500_000) == 0
    assert V.vla_test_stall_next_gemm() == 0
    pol.prefill(inp.visual.cuda(), inp.ids.cuda(), inp.lengths)
    rc = V.vla_sync(pol.h)
    assert rc == V.VLA_ERR_DEVICE_STATUS
    assert "timed out" in V.vla_last_error(pol.h)
    assert V.vla_test_set_wait_limit_ns(0) == 0
    assert V.vla_sync(pol.h) == 0                  # the word was cleared by the report
    pol.reset()
    _same(_turn(pol, inp), ref)
    pol.close()


def test_rmsnorm_saturation_sets_status():
    M, d = 3, 256
    h = torch.ones(M, d, dtype=torch.float32, device="cuda")
    h[1] *= -1.0
    h[2, :8] = float("nan")                                     # passes through, no saturation bit
    w = torch.full((d,), 1.0e5, dtype=torch.bfloat16, device="cuda")   # y = +-w: beyond fp16
    yh = torch.empty(M, d, dtype=torch.float16, device="cuda")
    yl = torch.empty_like(yh)
    assert V.vla_op_read_status()[0] == 0
    assert V.vla_op_rmsnorm(h.data_ptr(), d, 2, d, w.data_ptr(), 1e-6, yh.data_ptr(), yl.data_ptr(), True) == 0
    rc, st = V.vla_op_read_status()
    assert rc == 0 and st == V.VLA_STATUS_SATURATED, st
    assert (yh[0].float().cpu() == 65504.0).all() and (yh[1].float().cpu() == -65504.0).all()
    assert (yl[:2].float().cpu() == 0.0).all()
    # the bf16 form holds 1e5 (fp32 range): no saturation
    yb = torch.empty(M, d, dtype=torch.bfloat16, device="cuda")
    ybl = torch.empty_like(yb)
    assert V.vla_op_rmsnorm(h.data_ptr(), d, 2, d, w.data_ptr(), 1e-6, yb.data_ptr(), ybl.data_ptr(), False) == 0
    assert V.vla_op_read_status() == (0, 0)
    # ordinary gains: no bit; a NaN row stays NaN without the bit
    w1 = torch.ones(d, dtype=torch.bfloat16, device="cuda")
    assert V.vla_op_rmsnorm(h.data_ptr(), d, M, d, w1.data_ptr(), 1e-6, yh.data_ptr(), yl.data_ptr(), True) == 0
    assert V.vla_op_read_status() == (0, 0)
    assert torch.isnan(yh[2].float()).all()


def test_engine_reports_saturated_activation():
    # A handle whose first attention-norm gain is 1e5: every row's normalised input to the
    # first q|k|v projection is beyond the fp16 range.
    w = I.make_weights(WL.shape, WL.weight_seed)
    w["attn_norm"] = w["attn_norm"].clone()
    w["attn_norm"][0] = torch.full_like(w["attn_norm"][0], 1.0e5)
    wd = P.weights_to_device(w)
    pol = V.Policy(WL.shape, wd, WL.batch, 128, 512)
    inp = I.make_turn_inputs(WL, 0)
    pol.prefill(inp.visual.cuda(), inp.ids.cuda(), inp.lengths)
    assert V.vla_sync(pol.h) == V.VLA_ERR_DEVICE_STATUS
    assert "saturated" in V.vla_last_error(pol.h)
    pol.close()
