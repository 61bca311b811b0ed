"""Pins of the rounding-attribution module (tests/attribution.py), CPU only.

The roundings are checked against hand-worked fp16 values (ties to even, the subnormal range,
the pair's residual, the 4-bit residual's encoding and clamp), and the restated layer with
every hook the identity is checked against the oracle's layer bit for bit, so the attribution
runs measure storage rounding and nothing else."""
import torch

import oracle.vla_oracle as O
from paper_2505_18719_gb300 import inputs as I
from tests import attribution as A
from tests.test_oracle_pins import MICRO, micro_rows, micro_weights

F64 = torch.float64


def t(*v):
    return torch.tensor(v, dtype=F64)


def test_round_f16_hand_values():
    # 1 + 2^-11 is halfway between 1 and 1 + 2^-10: ties go to the even mantissa (1)
    # 1 + 3*2^-11 is halfway between 1 + 2^-10 (odd) and 1 + 2^-9 (even)
    # 65519 is below the halfway point 65520 between 65504 and 2^16: rounds to the largest finite
    # 2^-25 is halfway between 0 and the smallest subnormal 2^-24: ties to 0; 3*2^-26 -> 2^-24
    x = t(1 + 2 ** -11, 1 + 3 * 2 ** -11, 65519.0, 2 ** -25, 3 * 2 ** -26, -2.5)
    want = t(1.0, 1 + 2 ** -9, 65504.0, 0.0, 2 ** -24, -2.5)
    assert torch.equal(A.round_f16(x), want)


def test_round_f16_pair_hand_values():
    # 1 + 2^-11: hi = 1, lo = 2^-11 exactly, so the pair is exact
    # pi: hi = 1608 * 2^-9 = 3.140625; pi - hi = 0.00096765... lies in [2^-11, 2^-10), where fp16
    # steps by 2^-21, and 0.00096765 / 2^-21 = 2029.33 -> lo = 2029 * 2^-21
    got = A.round_f16_pair(t(1 + 2 ** -11, 3.141592653589793))
    want = t(1 + 2 ** -11, 3.140625 + 2029 * 2 ** -21)
    assert torch.equal(got, want)


def test_f16_ulp_hand_values():
    x = t(1.0, 1.5, 2.0, 65504.0, 2 ** -14, 2 ** -20, 0.0, -3.0)
    want = t(2 ** -10, 2 ** -10, 2 ** -9, 32.0, 2 ** -24, 2 ** -24, 2 ** -24, 2 ** -9)
    assert torch.equal(A.f16_ulp(x), want)


def test_round_f16_r4_hand_values_and_bound():
    # x = 1 + 2^-11 + 2^-13 = 1 + 0.625 ulp (ulp 2^-10): hi = 1 + 2^-10, x - hi = -0.375 ulp lies
    # in the cell [-6/16, -5/16) -> j = -6, value hi - 11/32 ulp = 1 + 2^-10 - 11 * 2^-15.
    # x = 1 + 2^-11 (tie -> hi = 1): +0.5 ulp is the top edge -> j = 8 clamps to 7 -> 1 + 15 * 2^-15.
    # x = 3 (exact in fp16): j = 0 -> 3 + 2^-9 / 32.
    got = A.round_f16_r4(t(1 + 2 ** -11 + 2 ** -13, 1 + 2 ** -11, 3.0))
    want = t(1 + 2 ** -10 - 11 * 2 ** -15, 1 + 15 * 2 ** -15, 3.0 + 2 ** -14)
    assert torch.equal(got, want)
    x = I.normal_bf16((4096,), 5, 1, 1.0).double() * torch.exp(I.normal_bf16((4096,), 5, 2, 3.0).double())
    x = x.clamp(-6e4, 6e4)
    hi = A.round_f16(x)
    err = (A.round_f16_r4(x) - x).abs()
    assert (err <= A.f16_ulp(hi) / 32).all()          # 4 bits past fp16's 11
    assert (A.round_f16(A.round_f16_r4(x)) == hi).all()  # the hi part reads back unchanged


def test_rounded_layer_with_identity_hooks_is_the_oracle_layer():
    W = O.Weights(MICRO, micro_weights())
    lw = W.layer(0)
    H, hd = MICRO.n_heads, MICRO.head_dim
    past = O.f64(micro_rows(3, seed=12)).reshape(3, H, hd)
    for n, m in ((5, 0), (1, 3), (4, 3)):
        h = O.f64(micro_rows(n))
        pos = torch.arange(m, m + n)
        kc, vc = past[:m], (past[:m] * 0.5)
        ref = O.layer_forward(MICRO, lw, h, pos, kc, vc)
        got = A.layer_forward_rounded(MICRO, lw, h, pos, kc, vc, A.EXACT)
        for a, b in zip(ref, got):
            assert torch.equal(a, b)


def test_attribution_oracle_with_identity_is_the_oracle():
    w = micro_weights()
    orc = O.Oracle(MICRO, w, 1)
    att = A.AttributionOracle(MICRO, w, 1, rounding=A.EXACT)
    vis = I.normal_bf16((3, MICRO.d_model), 21, 100, 1.0)
    u = I.uniform_f32((1, MICRO.action_dim, MICRO.n_bins), 31, 5)
    outs = []
    for o in (orc, att):
        o.prefill([0], [vis], [[5, 6]])
        outs.append(o.decode([0], u, 1.0))
    for k in ("tokens", "logprobs", "logits"):
        assert (outs[0][k] == outs[1][k]).all(), k


def test_gpu_path_rounding_moves_the_result_a_little():
    # the GPU-path roundings change the micro model's logits, by far less than the gate
    w = micro_weights()
    vis = I.normal_bf16((3, MICRO.d_model), 21, 100, 1.0)
    u = I.uniform_f32((1, MICRO.action_dim, MICRO.n_bins), 31, 5)
    outs = []
    for o in (O.Oracle(MICRO, w, 1), A.AttributionOracle(MICRO, w, 1, rounding=A.GPU_PATH)):
        o.prefill([0], [vis], [[5, 6]])
        outs.append(o.decode([0], u, 1.0, forced=torch.full((1, 7), MICRO.vocab - 200))["logits"])
    d = abs(outs[0] - outs[1]).max()
    assert 0 < d < 1e-3
