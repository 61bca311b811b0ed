"""The number-format facts the fp16 operand form rests on, checked exhaustively or on a
dense sample on the CPU: every bf16 weight in [2^-14, 65504] is exact in fp16 and a smaller
one moves by at most 2^-25; the pair hi = fp16(x), lo = fp16(x - hi) holds an fp32 x to
2^-22 relative in the normal range, and hi alone to 2^-11 (bf16 hi alone: 2^-8)."""
import numpy as np
import torch


def all_bf16():
    bits = torch.arange(0, 1 << 16, dtype=torch.int32).to(torch.int16)
    v = bits.view(torch.bfloat16).float()
    return v[torch.isfinite(v)]


def test_bf16_weights_in_fp16_range_are_exact():
    v = all_bf16().double()
    a = v.abs()
    inr = (a >= 2.0 ** -14) & (a <= 65504.0)
    h = v.float().half().double()
    assert torch.equal(h[inr], v[inr])
    small = a < 2.0 ** -14
    assert (h[small] - v[small]).abs().max().item() <= 2.0 ** -25
    assert small.any() and inr.sum().item() == 30 * 128 * 2   # binades 2^-14 .. 2^15, both signs


def test_fp16_pair_and_single_relative_error():
    g = torch.Generator().manual_seed(7)
    x = (torch.randn(1 << 20, generator=g) * torch.exp2(torch.randint(-10, 12, (1 << 20,), generator=g).float()))
    x = x[(x.abs() > 2.0 ** -2) & (x.abs() < 30000.0)]
    xd = x.double()
    hi = x.half()
    lo = (x - hi.float()).half()
    rel_pair = ((hi.double() + lo.double() - xd).abs() / xd.abs()).max().item()
    rel_hi = ((hi.double() - xd).abs() / xd.abs()).max().item()
    rel_bf = ((x.bfloat16().double() - xd).abs() / xd.abs()).max().item()
    assert rel_pair <= 2.0 ** -22
    assert 2.0 ** -12 < rel_hi <= 2.0 ** -11
    assert 2.0 ** -9 < rel_bf <= 2.0 ** -8
    assert np.isclose(rel_bf / rel_hi, 8.0, rtol=0.01)


def test_residual_decode_half_arithmetic_is_the_definition():
    """The kernels decode a cached value's 4-bit residual code c with three fp16 operations and
    no conversion (kv_res_pair in csrc/common.cuh): k = half(0x6400 | 2c) - half(0x640F) = 2c - 15,
    s = half(bits(hi) & 0x7C00) * half(0x0200) = 2^(e-15) * 2^-15, lo = k * s.  Emulated here in
    IEEE fp16 (numpy rounds each operation to nearest) for every finite fp16 hi and every code:
    lo equals the residual's definition (2c - 15) ulp(hi) / 32, ulp(hi) = 2^(e-25), exactly for
    exponent fields e >= 6; below (|hi| < 2^-9) the term itself is under 2^-21 in magnitude and
    comes out as zero or a rounded subnormal, so the decoded value is off by less than 2^-21."""
    bits = np.arange(0, 1 << 16, dtype=np.uint32).astype(np.uint16)
    e = ((bits >> 10) & 31).astype(np.int64)
    finite = e < 31
    bits, e = bits[finite], e[finite]
    one_k = np.array([0x640F], dtype=np.uint16).view(np.float16)[0]
    unit = np.array([0x0200], dtype=np.uint16).view(np.float16)[0]
    assert float(one_k) == 1039.0 and float(unit) == 2.0 ** -15
    s = (bits & np.uint16(0x7C00)).view(np.float16) * unit
    for c in range(16):
        k = np.array([0x6400 | (2 * c)], dtype=np.uint16).view(np.float16)[0] - one_k
        assert float(k) == 2 * c - 15
        lo = (np.float16(k) * s).astype(np.float64)
        want = (2.0 * c - 15.0) * np.ldexp(1.0, np.maximum(e, 1) - 30)
        exact = e >= 6
        assert np.array_equal(lo[exact], want[exact]), c
        assert np.abs(want[~exact]).max() < 2.0 ** -21 and np.abs(lo[~exact] - want[~exact]).max() < 2.0 ** -21, c
