"""The handle's fp16 copy of the projection matrices, through the C ABI: vla_create fills it
from the caller's bf16 weights, an in-place change of those weights is seen only after
vla_sync_weights (the weight refresh between a learner update of θ and the next rollout,
Algorithm 1), and a weight outside the fp16 range is refused."""
import pytest
import torch

from paper_2505_18719_gb300 import inputs as I
from paper_2505_18719_gb300 import vla as V
from tests import parity as P

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    from paper_2505_18719_gb300 import build
    build.build()


WL = I.WORKLOADS["tiny_b4"]


def _policy(w):
    wl = WL
    max_tokens = wl.batch * (wl.n_visual + (wl.text_len or wl.text_len_range[1]) + 8)
    return V.Policy(wl.shape, w, wl.batch, wl.kv_capacity, max_tokens)


def _rollout(pol, inp, forced):
    pol.reset()
    pol.prefill(inp.visual.cuda(), inp.ids.cuda(), inp.lengths.tolist())
    out = pol.decode(inp.uniforms.cuda(), WL.temperature, forced=forced)
    pol.sync()
    return out["logits"].clone(), out["logprobs"].clone()


def test_sync_weights_reads_updated_projections():
    sh = WL.shape
    w = P.weights_to_device(I.make_weights(sh))
    inp = I.make_turn_inputs(WL, 0)
    base = sh.vocab - sh.n_bins
    forced = (base + (torch.arange(sh.action_dim)[None, :] * 37 + torch.arange(WL.batch)[:, None]) % 256)
    forced = forced.to(torch.int32).cuda()
    pol = _policy(w)
    z0, lp0 = _rollout(pol, inp, forced)
    for name in ("wqkv", "wo", "w_gate_up", "w_down"):
        w[name].mul_(0.75)
    torch.cuda.synchronize()
    z1, lp1 = _rollout(pol, inp, forced)          # the copy is unchanged: same results
    assert torch.equal(z0, z1) and torch.equal(lp0, lp1)
    pol.sync_weights()
    z2, lp2 = _rollout(pol, inp, forced)
    assert not torch.equal(z0, z2)
    fresh = _policy(w)
    z3, lp3 = _rollout(fresh, inp, forced)        # deterministic kernels: bit-equal
    assert torch.equal(z2, z3) and torch.equal(lp2, lp3)
    fresh.close()
    # a weight beyond the fp16 range: refused by the sync and by a new handle
    w["w_down"][0].view(-1)[5] = 70000.0
    torch.cuda.synchronize()
    with pytest.raises(V.VlaError) as e:
        pol.sync_weights()
    assert e.value.code == V.VLA_ERR_UNSUPPORTED
    with pytest.raises(V.VlaError) as e:
        _policy(w)
    assert e.value.code == V.VLA_ERR_UNSUPPORTED
    pol.close()
