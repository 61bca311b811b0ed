"""Seeded synthetic workloads for the VLA rollout hot path.

This module only produces inputs: model shapes, the five workload recipes, and the
bytes of weights / visual embeddings / token ids / noise, drawn from the counter-based
generator in ``vla_inputs.c``.  It contains none of the method's arithmetic, so the
oracle and the CUDA path may both consume what it writes.

Workloads stand in for OpenVLA-7B (a Llama-2-7B backbone, paper §3.1) rolling out on
LIBERO-like prefixes (§4): projected visual patch embeddings followed by instruction ids,
then 7 action tokens (Eq. 1, |A| = 7) drawn from the last 256 vocabulary ids.  No
dataset item, checkpoint or simulator state is reproduced; everything is seeded noise of
the stated shape and distribution.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
import threading
from typing import Dict, List, Optional

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "vla_inputs.c")
_LIB_PATH = os.path.join(_HERE, "libvla_inputs.so")
_lock = threading.Lock()
_lib = None

BASE_SEED = 20250524


def build_library(force: bool = False) -> str:
    """Compile ``vla_inputs.c`` into ``libvla_inputs.so`` next to it (plain gcc)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-pthread", _SRC,
                               "-o", tmp, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _library():
    global _lib
    with _lock:
        if _lib is None:
            build_library()
            lib = ctypes.CDLL(_LIB_PATH)
            i64, u64, vp = ctypes.c_int64, ctypes.c_uint64, ctypes.c_void_p
            lib.vla_gen_normal_bf16.argtypes = [vp, i64, u64, u64, ctypes.c_double, ctypes.c_double]
            lib.vla_gen_uniform_f32.argtypes = [vp, i64, u64, u64]
            lib.vla_gen_randint_i32.argtypes = [vp, i64, u64, u64, ctypes.c_int32, ctypes.c_int32]
            lib.vla_gen_raw_u64.argtypes = [vp, i64, u64, u64]
            lib.vla_gen_splitmix64.argtypes = [vp, i64, u64]
            for f in (lib.vla_gen_normal_bf16, lib.vla_gen_uniform_f32, lib.vla_gen_randint_i32,
                      lib.vla_gen_raw_u64, lib.vla_gen_splitmix64):
                f.restype = None
            _lib = lib
    return _lib


# --------------------------------------------------------------------------- primitives
def normal_bf16(shape, seed: int, stream: int, std: float = 1.0, mean: float = 0.0) -> torch.Tensor:
    t = torch.empty(shape, dtype=torch.bfloat16)
    _library().vla_gen_normal_bf16(t.data_ptr(), t.numel(), seed, stream, std, mean)
    return t


def uniform_f32(shape, seed: int, stream: int) -> torch.Tensor:
    t = torch.empty(shape, dtype=torch.float32)
    _library().vla_gen_uniform_f32(t.data_ptr(), t.numel(), seed, stream)
    return t


def randint_i32(shape, seed: int, stream: int, lo: int, hi: int) -> torch.Tensor:
    """Uniform integers in [lo, hi], both ends included."""
    t = torch.empty(shape, dtype=torch.int32)
    _library().vla_gen_randint_i32(t.data_ptr(), t.numel(), seed, stream, lo, hi)
    return t


def raw_u64(n: int, seed: int, stream: int) -> List[int]:
    buf = (ctypes.c_uint64 * n)()
    _library().vla_gen_raw_u64(ctypes.addressof(buf), n, seed, stream)
    return list(buf)


def splitmix64(n: int, state: int) -> List[int]:
    buf = (ctypes.c_uint64 * n)()
    _library().vla_gen_splitmix64(ctypes.addressof(buf), n, state)
    return list(buf)


# --------------------------------------------------------------------------- shapes
@dataclasses.dataclass(frozen=True)
class ModelShape:
    """Llama-style decoder shape (paper §3.1: OpenVLA-7B = Llama-2-7B backbone)."""
    name: str
    n_layers: int
    d_model: int
    n_heads: int
    head_dim: int
    d_ffn: int
    vocab: int = 32064
    n_bins: int = 256          # last 256 vocabulary ids are the action bins
    action_dim: int = 7        # |A| = 7 (Eq. 1)
    rms_eps: float = 1e-6
    rope_theta: float = 1e4
    weight_std: float = 0.02

    @property
    def params_per_layer(self) -> int:
        d, f = self.d_model, self.d_ffn
        return 3 * d * d + d * d + 2 * f * d + d * f


TINY = ModelShape("tiny", 2, 256, 4, 64, 688)
SMALL = ModelShape("small", 8, 1024, 16, 64, 2816)
LLAMA7B = ModelShape("llama2-7b-shape", 32, 4096, 32, 128, 11008)
SHAPES = {s.name: s for s in (TINY, SMALL, LLAMA7B)}
_SHAPE_SEED_OFFSET = {"tiny": 1, "small": 2, "llama2-7b-shape": 3}


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic rollout workload.

    turn 0 prefix = n_visual visual embeddings ~N(0,1) + text ids uniform in [0, vocab-256);
    turns >= 1 append (pending 7th action token) + `append_visual` fresh visual rows
    + `append_text` ids.
    """
    name: str
    shape: ModelShape
    batch: int
    n_visual: int
    text_len: Optional[int]           # fixed text length, or None for ragged
    text_len_range: Optional[tuple] = None   # (lo, hi) inclusive when ragged
    turns: int = 1
    append_visual: int = 256
    append_text: int = 0
    temperature: float = 1.0
    score: bool = False
    kv_capacity: int = 0
    index: int = 0
    # episode ends: (turn, env ids) = these envs are reset before that turn's prefill and
    # start a new episode whose first prefix is that turn's chunk (Algorithm 1 terminal flags)
    resets: tuple = ()

    @property
    def input_seed(self) -> int:
        return BASE_SEED + 100 + self.index

    @property
    def weight_seed(self) -> int:
        return BASE_SEED + _SHAPE_SEED_OFFSET[self.shape.name]


WORKLOADS: Dict[str, Workload] = {w.name: w for w in (
    Workload("tiny_b4", TINY, 4, 64, 16, kv_capacity=128, index=1),
    Workload("small_b16_score", SMALL, 16, 256, 24, score=True, kv_capacity=320, index=2),
    Workload("7b_b16", LLAMA7B, 16, 256, 32, kv_capacity=320, index=3),
    Workload("7b_b64_ragged_score", LLAMA7B, 64, 256, None, (16, 48), score=True,
             kv_capacity=320, index=4),
    Workload("7b_b256_multiturn", LLAMA7B, 256, 256, 64, turns=4, append_visual=256,
             append_text=0, kv_capacity=1152, index=5),
    # the same trajectory with the instruction's 64 ids re-sent every turn (up to 1307 positions),
    # the paper's sampling temperature 1.5, and three envs whose episode ends after turn 1
    Workload("7b_b256_multiturn_t15", LLAMA7B, 256, 256, 64, turns=4, append_visual=256,
             append_text=64, temperature=1.5, kv_capacity=1344, index=6, resets=((2, (0, 5, 131)),)),
)}


# --------------------------------------------------------------------------- weights
# stream ids: one per tensor (per layer for the stacked ones)
def _wstream(kind: int, layer: int = 0) -> int:
    return 16 + 8 * layer + kind


WEIGHT_NAMES = ("embed", "attn_norm", "wqkv", "wo", "ffn_norm", "w_gate_up", "w_down",
                "final_norm", "lm_head")


def make_weights(shape: ModelShape, seed: Optional[int] = None) -> Dict[str, torch.Tensor]:
    """bf16 CPU weights.  Matrices and embed/lm_head ~N(0, std); RMSNorm gains = 1.0.

    Layout (row-major, nn.Linear [out, in]):
      embed [V,d]; attn_norm [L,d]; wqkv [L,3d,d] rows q|k|v; wo [L,d,d]; ffn_norm [L,d];
      w_gate_up [L,2F,d] rows gate|up; w_down [L,d,F]; final_norm [d]; lm_head [V,d].
    """
    if seed is None:
        seed = BASE_SEED + _SHAPE_SEED_OFFSET[shape.name]
    L, d, f, V, s = shape.n_layers, shape.d_model, shape.d_ffn, shape.vocab, shape.weight_std
    w = {
        "embed": normal_bf16((V, d), seed, 1, s),
        "lm_head": normal_bf16((V, d), seed, 2, s),
        "final_norm": torch.ones(d, dtype=torch.bfloat16),
        "attn_norm": torch.ones(L, d, dtype=torch.bfloat16),
        "ffn_norm": torch.ones(L, d, dtype=torch.bfloat16),
        "wqkv": torch.empty(L, 3 * d, d, dtype=torch.bfloat16),
        "wo": torch.empty(L, d, d, dtype=torch.bfloat16),
        "w_gate_up": torch.empty(L, 2 * f, d, dtype=torch.bfloat16),
        "w_down": torch.empty(L, d, f, dtype=torch.bfloat16),
    }
    lib = _library()
    for l in range(L):
        for kind, name in enumerate(("wqkv", "wo", "w_gate_up", "w_down")):
            t = w[name][l]
            lib.vla_gen_normal_bf16(t.data_ptr(), t.numel(), seed, _wstream(kind, l), s, 0.0)
    return w


# --------------------------------------------------------------------------- per-turn inputs
@dataclasses.dataclass
class TurnInputs:
    visual: torch.Tensor      # bf16 [B, n_visual, d]
    ids: torch.Tensor         # int32 [B, max_len] (padded with 0 beyond each length)
    lengths: torch.Tensor     # int32 [B] (text lengths)
    uniforms: torch.Tensor    # f32 [B, 7, 256] in (0, 1)


def make_turn_inputs(wl: Workload, turn: int) -> TurnInputs:
    sh, B, seed = wl.shape, wl.batch, wl.input_seed
    n_vis = wl.n_visual if turn == 0 else wl.append_visual
    visual = normal_bf16((B, n_vis, sh.d_model), seed, 1_000_000 + turn, 1.0)
    if turn == 0:
        if wl.text_len is not None:
            lengths = torch.full((B,), wl.text_len, dtype=torch.int32)
        else:
            lo, hi = wl.text_len_range
            lengths = randint_i32((B,), seed, 3_000_000 + turn, lo, hi)
    else:
        lengths = torch.full((B,), wl.append_text, dtype=torch.int32)
    max_len = max(int(lengths.max()) if B else 0, 1)
    ids = randint_i32((B, max_len), seed, 2_000_000 + turn, 0, sh.vocab - sh.n_bins - 1)
    for b in range(B):
        ids[b, int(lengths[b]):] = 0
    uniforms = uniform_f32((B, sh.action_dim, sh.n_bins), seed, 4_000_000 + turn)
    return TurnInputs(visual, ids, lengths, uniforms)
