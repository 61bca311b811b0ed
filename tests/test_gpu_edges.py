"""Edge cases of the rollout path through the C ABI, each against the fp64 oracle on the tiny
model (Algorithm 1's rollout: prefill of the state, then the 7 action tokens):
  * a prefill without visual rows and with ragged text down to a single row per env (a
    prefill this small, 31 rows, runs on the weight-streaming GEMMs);
  * a context that fills the KV cache exactly (chunk + 6 decoded positions == capacity), and
    the same chunk one position short refused;
  * forced tokens at the two edge bins (ids vocab-256 and vocab-1: the last embedding row)."""
import numpy as np
import pytest
import torch

import oracle.vla_oracle as O
from paper_2505_18719_gb300 import inputs as I
from paper_2505_18719_gb300 import vla as V
from tests import parity as P

pytestmark = pytest.mark.gpu
WL = I.WORKLOADS["tiny_b4"]
SH = WL.shape
BASE = SH.vocab - SH.n_bins


@pytest.fixture(scope="module")
def weights():
    from paper_2505_18719_gb300 import build
    build.build()
    w = I.make_weights(SH, WL.weight_seed)
    return w, P.weights_to_device(w)


def _rollout(weights, visual, ids, lengths, cap, forced=None, T=1.0):
    """Prefill + decode on the GPU and in the oracle; the GPU is teacher-forced on the oracle's
    tokens (or on `forced` for both)."""
    w, wd = weights
    B = len(lengths)
    nv = 0 if visual is None else visual.shape[1]
    envs = list(range(B))
    u = I.make_turn_inputs(WL, 0).uniforms[:B]
    orc = O.Oracle(O.shape_from(SH), w, B)
    empty = torch.zeros(0, SH.d_model, dtype=torch.bfloat16)
    orc.prefill(envs, [visual[b] if visual is not None else empty for b in envs],
                [ids[b, :lengths[b]].tolist() for b in envs])
    od = orc.decode(envs, u, T, forced=forced)
    feed = forced if forced is not None else torch.as_tensor(od["tokens"], dtype=torch.int32)
    pol = V.Policy(SH, wd, B, cap, B * (nv + max(lengths) + 8))
    try:
        pol.prefill(visual.cuda() if visual is not None else None, ids.cuda(), lengths)
        g = pol.decode(u.cuda(), T, forced=feed.cuda())
        pol.sync()
        g = {k: v.cpu().numpy() for k, v in g.items() if v is not None}
        lens = [V.vla_context_length(pol.h, b) for b in envs]
    finally:
        pol.close()
    rep = P.compare_decode(0, envs, od, g)
    print(rep)
    return rep, lens


def test_text_only_prefill_with_single_row_chunks(weights):
    inp = I.make_turn_inputs(WL, 0)
    lengths = [1, 5, 16, 9]
    rep, lens = _rollout(weights, None, inp.ids, lengths, cap=64)
    assert rep.ok(), rep
    assert lens == [n + 6 for n in lengths]


def test_context_fills_the_kv_cache_exactly(weights):
    inp = I.make_turn_inputs(WL, 0)
    lengths = [16] * 4                       # 64 visual + 16 text = 80 rows per env
    rep, lens = _rollout(weights, inp.visual, inp.ids, lengths, cap=86)
    assert rep.ok(), rep
    assert lens == [86] * 4
    w, wd = weights
    pol = V.Policy(SH, wd, 4, 85, 4 * 88)
    try:
        vis, ids = inp.visual.cuda(), inp.ids.cuda()
        rc = V.vla_prefill(pol.h, 4, vis.data_ptr(), 64, ids.data_ptr(), lengths, ids.shape[1])
        assert rc == V.VLA_ERR_CAPACITY
        assert V.vla_context_length(pol.h, 0) == 0
    finally:
        pol.close()


def test_forced_edge_bins(weights):
    inp = I.make_turn_inputs(WL, 0)
    edge = torch.tensor([0, 255, 0, 255, 255, 0, 255], dtype=torch.int32)
    forced = torch.stack([BASE + edge.roll(b) for b in range(4)]).to(torch.int32)
    rep, _ = _rollout(weights, inp.visual, inp.ids, inp.lengths.tolist(), cap=128, forced=forced)
    assert rep.ok(), rep
