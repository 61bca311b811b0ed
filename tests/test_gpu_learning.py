"""Learning-phase quantities on the GPU (C ABI) vs the fp64 oracle: GAE (Algorithm 1) and the
clipped PPO objective (Eq. 2).  Inputs are seeded; the value head and the rollout entropy are
checked on every workload inside the parity runs (tests/parity.py)."""
import numpy as np
import pytest
import torch

import oracle.vla_oracle as O
from paper_2505_18719_gb300 import inputs as I
from paper_2505_18719_gb300 import vla as V

pytestmark = pytest.mark.gpu


def _gae_inputs(M, B, seed):
    r = I.normal_bf16((M, B), seed, 1, 1.0).float()
    v = I.normal_bf16((M + 1, B), seed, 2, 2.0).float()
    dn = (I.uniform_f32((M, B), seed, 3) < 0.1).float()
    return r, v, dn


@pytest.mark.parametrize("M,B", [(1, 1), (5, 3), (37, 65), (128, 256)])
@pytest.mark.parametrize("gamma,lam", [(0.99, 0.95), (1.0, 1.0), (0.9, 0.0)])
def test_gae_matches_oracle(M, B, gamma, lam):
    r, v, dn = _gae_inputs(M, B, 100 + M + B)
    rd, vd, dd = r.cuda(), v.cuda(), dn.cuda()
    adv = torch.full((M, B), float("nan"), device="cuda")
    ret = torch.full((M, B), float("nan"), device="cuda")
    assert V.vla_gae(rd.data_ptr(), vd.data_ptr(), dd.data_ptr(), M, B, gamma, lam, adv.data_ptr(),
                     ret.data_ptr(), 0) == 0
    torch.cuda.synchronize()
    oa, orr = O.gae(r.double(), v.double(), dn.double(), gamma, lam)
    scale = 1.0 + float(oa.abs().max())
    assert float((adv.cpu().double() - oa).abs().max()) < 2e-6 * scale * M ** 0.5
    assert float((ret.cpu().double() - orr).abs().max()) < 2e-6 * scale * M ** 0.5


@pytest.mark.parametrize("N", [1, 7, 5000])
@pytest.mark.parametrize("eps", [0.2, 0.0])
def test_ppo_clip_matches_oracle_and_is_deterministic(N, eps):
    A = 7
    lp_old = -I.uniform_f32((N, A), 200 + N, 1) * 6.0
    lp_new = lp_old + (I.uniform_f32((N, A), 200 + N, 2) - 0.5) * 0.12
    adv = I.normal_bf16((N,), 200 + N, 3, 1.0).float()
    d = [t.cuda() for t in (lp_new, lp_old, adv)]
    outs = []
    for _ in range(2):
        obj = torch.full((1,), float("nan"), device="cuda")
        rho = torch.full((N,), float("nan"), device="cuda")
        cf = torch.full((1,), float("nan"), device="cuda")
        assert V.vla_ppo_clip(d[0].data_ptr(), d[1].data_ptr(), d[2].data_ptr(), N, A, eps, obj.data_ptr(),
                              rho.data_ptr(), cf.data_ptr(), 0) == 0
        torch.cuda.synchronize()
        outs.append((obj.item(), rho.cpu(), cf.item()))
    assert outs[0][0] == outs[1][0] and torch.equal(outs[0][1], outs[1][1])
    o_obj, o_rho, o_cf = O.ppo_clip_objective(lp_new.double(), lp_old.double(), adv.double(), eps)
    assert abs(outs[0][0] - o_obj) < 1e-5 * (1.0 + abs(o_obj))
    assert float((outs[0][1].double() - o_rho).abs().max()) < 1e-5
    # a sample within fp32 rounding of |rho - 1| = eps may be counted differently
    near = int(((o_rho - 1.0).abs() - eps).abs().lt(1e-5).sum())
    assert abs(outs[0][2] - o_cf) <= (near + 0.5) / N


def test_learning_entry_points_reject_bad_arguments():
    x = torch.zeros(4, device="cuda")
    p = x.data_ptr()
    assert V.vla_gae(p, p, p, 0, 1, 0.9, 0.9, p) == V.VLA_ERR_ARG
    assert V.vla_gae(p, p, p, 1, 1, 1.5, 0.9, p) == V.VLA_ERR_ARG
    assert V.vla_gae(0, p, p, 1, 1, 0.9, 0.9, p) == V.VLA_ERR_ARG
    assert V.vla_ppo_clip(p, p, p, 0, 7, 0.2, p) == V.VLA_ERR_ARG
    assert V.vla_ppo_clip(p, p, p, 1, 7, -0.1, p) == V.VLA_ERR_ARG
