"""Boundary behaviour of the C ABI on the GPU: state and capacity errors, device status
word, context-length bookkeeping, batch invariance (paper §3.5: large-batch decoding must
not change an env's results)."""
import numpy as np
import pytest
import torch

import oracle.vla_oracle as O
from paper_2505_18719_gb300 import inputs as I
from paper_2505_18719_gb300 import vla as V
from tests import parity as P

pytestmark = pytest.mark.gpu
WL = I.WORKLOADS["tiny_b4"]


@pytest.fixture(scope="module")
def wdev():
    from paper_2505_18719_gb300 import build
    build.build()
    return P.weights_to_device(I.make_weights(WL.shape, WL.weight_seed))


def _policy(wdev, B=4, cap=128, max_tokens=512):
    return V.Policy(WL.shape, wdev, B, cap, max_tokens)


def test_state_capacity_and_args(wdev):
    pol = _policy(wdev)
    inp = I.make_turn_inputs(WL, 0)
    u = inp.uniforms.cuda()
    outs = [torch.empty(4, 7, dtype=t, device="cuda") for t in (torch.int32, torch.float32, torch.float32)]
    rc = V.vla_decode_actions(pol.h, u.data_ptr(), 1.0, 0, *[o.data_ptr() for o in outs])
    assert rc == V.VLA_ERR_STATE
    rc = V.vla_score_actions(pol.h, outs[0].data_ptr(), 1.0, outs[1].data_ptr())
    assert rc == V.VLA_ERR_STATE
    vis, ids = inp.visual.cuda(), inp.ids.cuda()
    # 64 visual + 16 text = 80 rows; capacity 128 leaves room for 80 + 6, not for a second turn
    assert V.vla_prefill(pol.h, 4, vis.data_ptr(), 64, ids.data_ptr(), [16] * 4, ids.shape[1]) == 0
    assert V.vla_context_length(pol.h, 0) == 80
    rc = V.vla_decode_actions(pol.h, u.data_ptr(), -1.0, 0, *[o.data_ptr() for o in outs])
    assert rc == V.VLA_ERR_ARG
    rc = V.vla_decode_actions(pol.h, u.data_ptr(), float("nan"), 0, *[o.data_ptr() for o in outs])
    assert rc == V.VLA_ERR_ARG
    assert V.vla_decode_actions(pol.h, u.data_ptr(), 1.0, 0, *[o.data_ptr() for o in outs]) == 0
    assert V.vla_sync(pol.h) == 0
    assert V.vla_context_length(pol.h, 3) == 86
    rc = V.vla_prefill(pol.h, 4, vis.data_ptr(), 64, ids.data_ptr(), [16] * 4, ids.shape[1])
    assert rc == V.VLA_ERR_CAPACITY
    assert V.vla_context_length(pol.h, 3) == 86        # rejected call changed nothing
    assert V.vla_reset(pol.h, [1, 0, 0, 0]) == 0
    assert V.vla_context_length(pol.h, 0) == 0 and V.vla_context_length(pol.h, 1) == 86
    rc = V.vla_decode_actions(pol.h, u.data_ptr(), 1.0, 0, *[o.data_ptr() for o in outs])
    assert rc == V.VLA_ERR_STATE                        # env 0 was reset since the prefill
    pol.close()


def test_device_status_bad_ids_and_tokens(wdev):
    pol = _policy(wdev)
    inp = I.make_turn_inputs(WL, 0)
    ids = inp.ids.clone()
    ids[2, 3] = 40000
    ids[1, 0] = -5
    vis = inp.visual.cuda()
    assert V.vla_prefill(pol.h, 4, vis.data_ptr(), 64, ids.cuda().data_ptr(), [16] * 4, ids.shape[1]) == 0
    rc = V.vla_sync(pol.h)
    assert rc == V.VLA_ERR_DEVICE_STATUS
    assert "token id out of range" in V.vla_last_error(pol.h)
    assert V.vla_sync(pol.h) == 0                      # cleared
    bad = torch.full((4, 7), 5, dtype=torch.int32, device="cuda")   # not action ids
    lp = torch.empty(4, 7, dtype=torch.float32, device="cuda")
    assert V.vla_score_actions(pol.h, bad.data_ptr(), 1.0, lp.data_ptr()) == 0
    assert V.vla_sync(pol.h) == V.VLA_ERR_DEVICE_STATUS
    assert "not an action-bin id" in V.vla_last_error(pol.h)
    pol.close()


def test_batch_invariance_env_alone_vs_in_batch(wdev):
    inp = I.make_turn_inputs(WL, 0)
    base = WL.shape.vocab - 256
    forced = (base + (torch.arange(7, dtype=torch.int32)[None, :] * 11 + torch.arange(4)[:, None] * 3) % 256)
    forced = forced.to(torch.int32).cuda()
    big = _policy(wdev)
    big.prefill(inp.visual.cuda(), inp.ids.cuda(), inp.lengths.tolist())
    ob = big.decode(inp.uniforms.cuda(), 1.0, forced=forced)
    big.sync()
    solo = _policy(wdev, B=1)
    b = 2
    solo.prefill(inp.visual[b:b + 1].cuda(), inp.ids[b:b + 1].cuda(), inp.lengths[b:b + 1].tolist())
    os_ = solo.decode(inp.uniforms[b:b + 1].cuda(), 1.0, forced=forced[b:b + 1])
    solo.sync()
    err = (ob["logits"][b] - os_["logits"][0]).abs().max().item()
    assert err < 1e-3, err
    assert (ob["logprobs"][b] - os_["logprobs"][0]).abs().max().item() < 1e-3
    big.close()
    solo.close()


def test_score_equals_decode_and_multiturn_lengths(wdev):
    pol = _policy(wdev, cap=256)
    inp = I.make_turn_inputs(WL, 0)
    pol.prefill(inp.visual.cuda(), inp.ids.cuda(), inp.lengths.tolist())
    d = pol.decode(inp.uniforms.cuda(), 1.0)
    s = pol.score(d["tokens"], 1.0)
    pol.sync()
    assert (s["logprobs"] - d["logprobs"]).abs().max().item() < 2e-2
    assert V.vla_context_length(pol.h, 0) == 80 + 6
    inp2 = I.make_turn_inputs(I.dataclasses.replace(WL, append_visual=32), 1)
    pol.prefill(inp2.visual.cuda(), None, [0] * 4)
    assert V.vla_context_length(pol.h, 0) == 86 + 1 + 32
    pol.decode(inp2.uniforms.cuda(), 1.0)
    pol.sync()
    pol.close()
