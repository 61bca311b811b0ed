"""Rounding attribution: the oracle's decoder layer restated with the GPU path's storage
precisions, to tell rounding error apart from bugs.  NOT the parity gate (the gate is the
plain fp64 oracle); used by tests/parity.py when asked for attribution and by the precision
studies that chose the operand forms.

Test infrastructure only.  It reuses the oracle's primitives (RMSNorm, RoPE, attention, SiLU)
and re-states one layer with hooks at each point where the GPU stores a value at reduced
precision: GEMM input activations, queries, cached keys / values, and the keys / values a
single-row (decode) attention reads.  With every hook the identity it equals the oracle's
layer bit for bit (pinned in tests/test_attribution_cpu.py).
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Optional

import torch

import oracle.vla_oracle as O

F64 = torch.float64


def round_f16(x: torch.Tensor) -> torch.Tensor:
    """Nearest fp16 value (round to nearest even), returned in fp64."""
    return x.to(torch.float32).to(torch.float16).to(F64)


def round_f16_pair(x: torch.Tensor) -> torch.Tensor:
    """x -> hi + lo with hi = fp16(x), lo = fp16(x - hi): the GPU's activation pair."""
    hi = round_f16(x)
    return hi + round_f16(x - hi)


def f16_ulp(hi: torch.Tensor) -> torch.Tensor:
    """Spacing of fp16 values at |hi| (2^-24 in the subnormal range, and for hi = 0)."""
    a = hi.abs()
    e = torch.floor(torch.log2(torch.where(a > 0, a, torch.ones_like(a))))
    ulp = torch.pow(2.0, e - 10.0)
    return torch.where(a >= 2.0 ** -14, ulp, torch.full_like(a, 2.0 ** -24))


def round_f16_r4(x: torch.Tensor) -> torch.Tensor:
    """fp16 hi plus a 4-bit residual code j in [-8, 7] naming the midpoint of one of the 16
    equal cells of [-ulp/2, ulp/2) around hi: hi + (2j + 1) * ulp(hi) / 32 with
    j = clamp(floor((x - hi) / ulp(hi) * 16), -8, 7), so |error| <= ulp(hi) / 32."""
    hi = round_f16(x)
    ulp = f16_ulp(hi)
    j = torch.clamp(torch.floor((x - hi) / ulp * 16.0), -8.0, 7.0)
    return hi + (2.0 * j + 1.0) * ulp / 32.0


def _same(x):
    return x


@dataclass(frozen=True)
class Rounding:
    """Where an implementation stores values at reduced precision (identity = exact)."""
    act: object = _same   # GEMM input activations (norm outputs, attention output, SwiGLU)
    q: object = _same     # queries after RoPE
    kv: object = _same    # keys (after RoPE) and values as cached
    # per-projection override of `act` for chunks of more than one row (prefill, score):
    # {"qkv" | "o" | "gate_up" | "down": rounding}; None = `act` everywhere
    act_chunk: Optional[dict] = None
    # what a single-row (decode) attention reads of the cached keys / values; None = as cached
    kv_read_decode: object = None


EXACT = Rounding()
# The GPU path: fp16 activation pairs (fp16 weights hold the bf16 ones exactly above 2^-14),
# fp32 queries, K/V cached as fp16 + 4-bit residual; the multi-row projections use the pair for
# q|k|v only (hi alone for o, gate|up and down); every attention reads the cache at its stored
# precision.  Approximate where the GPU's choice follows the whole call's rows rather than one
# env's chunk (the last prefill layer runs o, gate|up and down on each env's final row through
# the two-half weight-streaming GEMM; decode of more than 128 envs runs the tile GEMMs).
GPU_PATH = Rounding(act=round_f16_pair, q=lambda x: x.to(torch.float32).to(F64), kv=round_f16_r4,
                    act_chunk={"o": round_f16, "gate_up": round_f16, "down": round_f16})


def layer_forward_rounded(shape: O.Shape, lw: dict, h, pos, k_cache, v_cache, rnd: Rounding):
    """O.layer_forward with the storage roundings of `rnd` applied where the GPU stores."""
    n = h.shape[0]
    d, H, hd, F = shape.d_model, shape.n_heads, shape.head_dim, shape.d_ffn

    def act(site, x):
        f = rnd.act_chunk.get(site) if (rnd.act_chunk and n > 1) else None
        return (f or rnd.act)(x)

    y = act("qkv", O.rms_norm(h, lw["attn_norm"], shape.rms_eps))
    qkv = y @ lw["wqkv"].T
    q = qkv[:, 0:d].reshape(n, H, hd)
    k = qkv[:, d:2 * d].reshape(n, H, hd)
    v = rnd.kv(qkv[:, 2 * d:3 * d].reshape(n, H, hd))
    q = rnd.q(O.apply_rope(q, pos, shape.rope_theta))
    k = rnd.kv(O.apply_rope(k, pos, shape.rope_theta))
    k_all = torch.cat([k_cache, k], dim=0)
    v_all = torch.cat([v_cache, v], dim=0)
    k_pos = torch.arange(k_all.shape[0], dtype=torch.long)
    k_rd, v_rd = k_all, v_all
    if n == 1 and rnd.kv_read_decode is not None:
        k_rd, v_rd = rnd.kv_read_decode(k_all), rnd.kv_read_decode(v_all)
    o = act("o", O.causal_attention(q, k_rd, v_rd, pos, k_pos))
    h = h + o.reshape(n, d) @ lw["wo"].T
    y = act("gate_up", O.rms_norm(h, lw["ffn_norm"], shape.rms_eps))
    gu = y @ lw["w_gate_up"].T
    h = h + act("down", O.silu(gu[:, :F]) * gu[:, F:]) @ lw["w_down"].T
    return h, k_all, v_all


class AttributionOracle(O.Oracle):
    """The oracle's engine with every layer run by layer_forward_rounded(rnd)."""

    def __init__(self, shape: O.Shape, weights, n_envs: int, cache_f64: bool = True,
                 rounding: Rounding = GPU_PATH):
        super().__init__(shape, weights, n_envs, cache_f64=cache_f64)
        self.rnd = rounding

    def _layer(self, lw: dict, h, pos, k_cache, v_cache):
        return layer_forward_rounded(self.shape, lw, h, pos, k_cache, v_cache, self.rnd)
