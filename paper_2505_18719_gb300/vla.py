"""ctypes binding of libvla.so (include/vla.h, include/vla_ops.h): argument marshalling only.

Every step of the hot path runs in the CUDA library.  There is no fallback: if the library
is missing or fails to load, importing this module's functions raises.

Functions keep the C names (``vla_create``, ``vla_prefill``, ``vla_decode_actions``,
``vla_score_actions``, ``vla_reset``, ``vla_sync``, ``vla_last_error``, ``vla_destroy``,
...).  ``Policy`` is a convenience wrapper that holds torch device tensors and a handle.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, Optional, Sequence

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libvla.so")

VLA_OK = 0
VLA_ERR_ARG = -1
VLA_ERR_CAPACITY = -2
VLA_ERR_STATE = -3
VLA_ERR_CUDA = -4
VLA_ERR_OOM = -5
VLA_ERR_DEVICE_STATUS = -6
VLA_ERR_UNSUPPORTED = -7

VLA_STATUS_BAD_TOKEN = 0x1
VLA_STATUS_NONFINITE = 0x2
VLA_STATUS_TIMEOUT = 0x4
VLA_STATUS_BAD_FORCED = 0x8
VLA_STATUS_SATURATED = 0x10

KCLASS = ("gemm_prefill", "gemm_decode", "attn_prefill", "attn_decode", "head", "other")


class VlaConfig(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in ("n_layers", "d_model", "n_heads", "head_dim", "d_ffn",
                                             "vocab", "n_action_bins", "action_dim", "max_batch",
                                             "kv_capacity", "max_tokens")] + \
               [("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float)]


class VlaWeights(ctypes.Structure):
    _fields_ = [("embed", ctypes.c_void_p),
                ("attn_norm", ctypes.POINTER(ctypes.c_void_p)),
                ("wqkv", ctypes.POINTER(ctypes.c_void_p)),
                ("wo", ctypes.POINTER(ctypes.c_void_p)),
                ("ffn_norm", ctypes.POINTER(ctypes.c_void_p)),
                ("w_gate_up", ctypes.POINTER(ctypes.c_void_p)),
                ("w_down", ctypes.POINTER(ctypes.c_void_p)),
                ("final_norm", ctypes.c_void_p),
                ("lm_head", ctypes.c_void_p)]


class VlaError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"vla error {code}: {msg}")
        self.code = code


_lib = None


def load(path: str = LIB_PATH):
    """Load libvla.so (raises if it is missing: build it with paper_2505_18719_gb300.build)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise FileNotFoundError(f"{path} is missing; run `python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(path)
    vp, i32, f32, u32, i64 = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_uint32, ctypes.c_int64
    sig = {
        "vla_create": (i32, [ctypes.POINTER(VlaConfig), ctypes.POINTER(VlaWeights), vp, ctypes.POINTER(vp)]),
        "vla_prefill": (i32, [vp, i32, vp, i32, vp, ctypes.POINTER(ctypes.c_int32), i32]),
        "vla_decode_actions": (i32, [vp, vp, f32, vp, vp, vp, vp, vp]),
        "vla_score_actions": (i32, [vp, vp, f32, vp, vp]),
        "vla_reset": (i32, [vp, vp]),
        "vla_sync": (i32, [vp]),
        "vla_sync_weights": (i32, [vp]),
        "vla_context_length": (i32, [vp, i32]),
        "vla_last_error": (ctypes.c_char_p, [vp]),
        "vla_destroy": (None, [vp]),
        "vla_profile": (i32, [vp, u32]),
        "vla_profile_read": (i32, [vp, vp, vp, vp, vp]),
        "vla_launch_count": (i64, [vp]),
        "vla_action_entropy": (i32, [vp, vp]),
        "vla_value": (i32, [vp, vp, f32, vp]),
        "vla_gae": (i32, [vp, vp, vp, i32, i32, f32, f32, vp, vp, vp]),
        "vla_ppo_clip": (i32, [vp, vp, vp, i32, i32, f32, vp, vp, vp, vp]),
        "vla_op_gemm_bf16": (i32, [vp, vp, i32, vp, i32, vp, i32, i32, i32, i32, i32, i32, vp, vp]),
        "vla_op_gemm_pair_bf16": (i32, [vp, vp, i32, vp, i32, vp, i32, i32, i32, i32, vp]),
        "vla_op_gemm_decode_bf16": (i32, [vp, vp, i32, vp, i32, vp, i32, i32, i32, i32, vp, ctypes.c_size_t, vp]),
        "vla_op_gemm_decode_workspace_bytes": (ctypes.c_size_t, [i32, i32, i32]),
        "vla_op_gemm_f16": (i32, [vp, vp, i32, vp, i32, vp, i32, i32, i32, i32, i32, i32, vp, vp]),
        "vla_op_gemm_pair_f16": (i32, [vp, vp, i32, vp, i32, vp, i32, i32, i32, i32, vp]),
        "vla_op_gemm_decode_f16": (i32, [vp, vp, i32, vp, i32, vp, i32, i32, i32, i32, vp, ctypes.c_size_t, vp]),
        "vla_op_gemm_bf16_noalloc": (i32, [vp, vp, i32, vp, i32, vp, i32, i32, i32, i32, i32, i32, vp]),
        "vla_op_action_head": (i32, [vp, i32, i32, i32, vp, vp, f32, vp, f32, vp, vp, vp, vp, vp, vp, vp]),
        "vla_op_num_sms": (i32, []),
        "vla_op_attn_decode": (i32, [vp, vp, i32, i32, i32, i32, vp, vp, i32, i32, i32, vp, vp, vp, ctypes.c_size_t, vp]),
        "vla_op_attn_decode_workspace_bytes": (ctypes.c_size_t, [i32, i32, i32, i32, i32]),
        "vla_op_attn_decode_res": (i32, [vp, vp, vp, i32, i32, i32, i32, vp, vp, i32, i32, i32, vp, vp, vp,
                                         ctypes.c_size_t, vp]),
        "vla_op_attn_chunk": (i32, [vp, vp, i32, i32, i32, i32, vp, i32, i32, vp, vp, vp, vp]),
        "vla_op_rmsnorm": (i32, [vp, i32, i32, i32, vp, f32, vp, vp, i32, vp]),
        "vla_op_attn_chunk_res": (i32, [vp, vp, vp, i32, i32, i32, i32, vp, i32, i32, vp, vp, vp, vp]),
        "vla_op_attn_rows_res": (i32, [vp, vp, vp, i32, i32, i32, i32, vp, i32, i32, vp, vp, vp, vp]),
        "vla_op_read_status": (i32, [vp, ctypes.POINTER(u32)]),
        "vla_test_inject_launch_error": (i32, [i64, i32]),
        "vla_test_set_wait_limit_ns": (i32, [ctypes.c_uint64]),
        "vla_test_stall_next_gemm": (i32, []),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


# ---------------------------------------------------------------------------- C-named wrappers
def vla_last_error(handle=None) -> str:
    s = load().vla_last_error(handle)
    return s.decode() if s else ""


def _check(rc: int, handle=None):
    if rc != VLA_OK:
        raise VlaError(rc, vla_last_error(handle))
    return rc


def vla_create(cfg: VlaConfig, weights: VlaWeights, stream: int = 0):
    h = ctypes.c_void_p()
    rc = load().vla_create(ctypes.byref(cfg), ctypes.byref(weights), ctypes.c_void_p(stream or None),
                           ctypes.byref(h))
    _check(rc)
    return h


def vla_prefill(h, batch: int, visual_ptr: int, n_visual: int, ids_ptr: int, lengths: Sequence[int],
                max_len: int) -> int:
    lens = (ctypes.c_int32 * len(lengths))(*[int(x) for x in lengths])
    return load().vla_prefill(h, batch, visual_ptr or None, n_visual, ids_ptr or None, lens, max_len)


def vla_decode_actions(h, uniforms_ptr: int, temperature: float, forced_ptr: int, tokens_ptr: int,
                       logprobs_ptr: int, actions_ptr: int, logits_ptr: int = 0) -> int:
    return load().vla_decode_actions(h, uniforms_ptr or None, float(temperature), forced_ptr or None,
                                     tokens_ptr or None, logprobs_ptr or None, actions_ptr or None,
                                     logits_ptr or None)


def vla_score_actions(h, tokens_ptr: int, temperature: float, logprobs_ptr: int, logits_ptr: int = 0) -> int:
    return load().vla_score_actions(h, tokens_ptr or None, float(temperature), logprobs_ptr or None,
                                    logits_ptr or None)


def vla_action_entropy(h, entropy_ptr: int) -> int:
    return load().vla_action_entropy(h, entropy_ptr or None)


def vla_value(h, w_value_ptr: int, bias: float, values_ptr: int) -> int:
    return load().vla_value(h, w_value_ptr or None, float(bias), values_ptr or None)


def vla_gae(rewards_ptr: int, values_ptr: int, dones_ptr: int, M: int, B: int, gamma: float, lam: float,
            adv_ptr: int, returns_ptr: int = 0, stream: int = 0) -> int:
    return load().vla_gae(rewards_ptr or None, values_ptr or None, dones_ptr or None, M, B, float(gamma),
                          float(lam), adv_ptr or None, returns_ptr or None, stream or None)


def vla_ppo_clip(lp_new_ptr: int, lp_old_ptr: int, adv_ptr: int, N: int, A: int, eps: float, objective_ptr: int,
                 ratio_ptr: int = 0, clip_frac_ptr: int = 0, stream: int = 0) -> int:
    return load().vla_ppo_clip(lp_new_ptr or None, lp_old_ptr or None, adv_ptr or None, N, A, float(eps),
                               objective_ptr or None, ratio_ptr or None, clip_frac_ptr or None, stream or None)


def vla_reset(h, env_mask: Optional[Sequence[int]] = None) -> int:
    if env_mask is None:
        return load().vla_reset(h, None)
    m = (ctypes.c_uint8 * len(env_mask))(*[1 if x else 0 for x in env_mask])
    return load().vla_reset(h, m)


def vla_sync(h) -> int:
    return load().vla_sync(h)


def vla_sync_weights(h) -> int:
    return load().vla_sync_weights(h)


def vla_context_length(h, env: int) -> int:
    return load().vla_context_length(h, env)


def vla_destroy(h) -> None:
    load().vla_destroy(h)


def vla_profile(h, class_mask: int) -> int:
    return load().vla_profile(h, class_mask)


def vla_profile_read(h) -> Dict[str, dict]:
    n = len(KCLASS)
    la = (ctypes.c_int64 * n)()
    ms = (ctypes.c_double * n)()
    fl = (ctypes.c_double * n)()
    by = (ctypes.c_double * n)()
    _check(load().vla_profile_read(h, la, ms, fl, by), h)
    return {KCLASS[i]: {"launches": la[i], "ms": ms[i], "flops": fl[i], "bytes": by[i]} for i in range(n)}


def vla_launch_count(h=None) -> int:
    return load().vla_launch_count(h)


def vla_op_gemm_bf16(A_ptr, A_lo_ptr, lda, W_ptr, ldw, C_ptr, ldc, M, N, K, block_n=256, splits=1,
                     ws_ptr=0, stream=0) -> int:
    return load().vla_op_gemm_bf16(A_ptr, A_lo_ptr or None, lda, W_ptr, ldw, C_ptr, ldc, M, N, K,
                                   block_n, splits, ws_ptr or None, stream or None)


def vla_op_gemm_pair_bf16(A_ptr, A_lo_ptr, lda, W_ptr, ldw, C_ptr, ldc, M, N, K, stream=0) -> int:
    return load().vla_op_gemm_pair_bf16(A_ptr, A_lo_ptr or None, lda, W_ptr, ldw, C_ptr, ldc, M, N, K,
                                        stream or None)


def vla_op_gemm_decode_bf16(A_ptr, A_lo_ptr, lda, W_ptr, ldw, C_ptr, ldc, M, N, K, ws_ptr, ws_bytes,
                            stream=0) -> int:
    return load().vla_op_gemm_decode_bf16(A_ptr, A_lo_ptr, lda, W_ptr, ldw, C_ptr, ldc, M, N, K, ws_ptr,
                                          ws_bytes, stream or None)


def vla_op_gemm_decode_workspace_bytes(M, N, K) -> int:
    return load().vla_op_gemm_decode_workspace_bytes(M, N, K)


def vla_op_gemm_f16(A_ptr, A_lo_ptr, lda, W_ptr, ldw, C_ptr, ldc, M, N, K, block_n=256, splits=1,
                    ws_ptr=0, stream=0) -> int:
    return load().vla_op_gemm_f16(A_ptr, A_lo_ptr or None, lda, W_ptr, ldw, C_ptr, ldc, M, N, K,
                                  block_n, splits, ws_ptr or None, stream or None)


def vla_op_gemm_pair_f16(A_ptr, A_lo_ptr, lda, W_ptr, ldw, C_ptr, ldc, M, N, K, stream=0) -> int:
    return load().vla_op_gemm_pair_f16(A_ptr, A_lo_ptr or None, lda, W_ptr, ldw, C_ptr, ldc, M, N, K,
                                       stream or None)


def vla_op_gemm_decode_f16(A_ptr, A_lo_ptr, lda, W_ptr, ldw, C_ptr, ldc, M, N, K, ws_ptr, ws_bytes,
                           stream=0) -> int:
    return load().vla_op_gemm_decode_f16(A_ptr, A_lo_ptr, lda, W_ptr, ldw, C_ptr, ldc, M, N, K, ws_ptr,
                                         ws_bytes, stream or None)


def vla_op_gemm_bf16_noalloc(A_ptr, A_lo_ptr, lda, W_ptr, ldw, C_ptr, ldc, M, N, K, block_n=256,
                             splits=1, stream=0) -> int:
    """vla_op_gemm_bf16 for callers that cannot allocate: split-K partials in the library's
    fixed 8 MiB device scratch (see include/vla_ops.h)."""
    return load().vla_op_gemm_bf16_noalloc(A_ptr, A_lo_ptr or None, lda, W_ptr, ldw, C_ptr, ldc, M, N,
                                           K, block_n, splits, stream or None)


def vla_op_action_head(h_ptr, ldh, B, d, final_norm_ptr, head_rows_ptr, eps, uniforms_ptr, temperature,
                       forced_ptr, bins_ptr, lp_ptr, act_ptr, logits_ptr, status_ptr, stream=0) -> int:
    return load().vla_op_action_head(h_ptr, ldh, B, d, final_norm_ptr, head_rows_ptr, float(eps),
                                     uniforms_ptr or None, float(temperature), forced_ptr or None,
                                     bins_ptr or None, lp_ptr, act_ptr or None, logits_ptr or None,
                                     status_ptr, stream or None)


def vla_op_attn_chunk(q_ptr, kv_ptr, max_env, H, hd, cap, tiles, rows, tiles_dev_ptr, out_hi_ptr, out_lo_ptr,
                      stream=0) -> int:
    """tiles: host sequence of (env, row0, nrows, pos0)."""
    flat = [int(x) for t in tiles for x in t]
    arr = (ctypes.c_int32 * len(flat))(*flat)
    return load().vla_op_attn_chunk(q_ptr or None, kv_ptr or None, max_env, H, hd, cap, arr, len(tiles), rows,
                                    tiles_dev_ptr or None, out_hi_ptr or None, out_lo_ptr or None, stream or None)


def vla_op_attn_chunk_res(q_ptr, kv_ptr, res_ptr, max_env, H, hd, cap, tiles, rows, tiles_dev_ptr, out_hi_ptr,
                          out_lo_ptr, stream=0) -> int:
    """tiles: host sequence of (env, row0, nrows <= 128, pos0); res: the cache's 4-bit codes."""
    flat = [int(x) for t in tiles for x in t]
    arr = (ctypes.c_int32 * len(flat))(*flat)
    return load().vla_op_attn_chunk_res(q_ptr or None, kv_ptr or None, res_ptr or None, max_env, H, hd, cap, arr,
                                        len(tiles), rows, tiles_dev_ptr or None, out_hi_ptr or None,
                                        out_lo_ptr or None, stream or None)


def vla_op_attn_rows_res(q_ptr, kv_ptr, res_ptr, max_env, H, hd, cap, tiles, rows, tiles_dev_ptr, out_hi_ptr,
                         out_lo_ptr, stream=0) -> int:
    """tiles: host sequence of (env, row0, nrows <= 16, pos0); res: the cache's 4-bit codes."""
    flat = [int(x) for t in tiles for x in t]
    arr = (ctypes.c_int32 * len(flat))(*flat)
    return load().vla_op_attn_rows_res(q_ptr or None, kv_ptr or None, res_ptr or None, max_env, H, hd, cap, arr,
                                       len(tiles), rows, tiles_dev_ptr or None, out_hi_ptr or None,
                                       out_lo_ptr or None, stream or None)


def vla_op_num_sms() -> int:
    return load().vla_op_num_sms()


def vla_op_attn_decode(q_ptr, kv_ptr, max_env, H, hd, cap, env_ptr, pos_ptr, B, max_ctx, out_hi_ptr, out_lo_ptr,
                       ws_ptr, ws_bytes, stream=0, max_keys_per_cta=0) -> int:
    return load().vla_op_attn_decode(q_ptr, kv_ptr, max_env, H, hd, cap, env_ptr, pos_ptr, B, max_ctx,
                                     max_keys_per_cta, out_hi_ptr, out_lo_ptr, ws_ptr, ws_bytes, stream or None)


def vla_op_attn_decode_res(q_ptr, kv_ptr, res_ptr, max_env, H, hd, cap, env_ptr, pos_ptr, B, max_ctx, out_hi_ptr,
                           out_lo_ptr, ws_ptr, ws_bytes, stream=0, max_keys_per_cta=0) -> int:
    """vla_op_attn_decode over the fp16 cache plus its 4-bit residual codes (res)."""
    return load().vla_op_attn_decode_res(q_ptr, kv_ptr, res_ptr, max_env, H, hd, cap, env_ptr, pos_ptr, B, max_ctx,
                                         max_keys_per_cta, out_hi_ptr, out_lo_ptr, ws_ptr, ws_bytes, stream or None)


def vla_op_attn_decode_workspace_bytes(B, H, hd, max_ctx, max_keys_per_cta=0) -> int:
    return load().vla_op_attn_decode_workspace_bytes(B, H, hd, max_ctx, max_keys_per_cta)


def vla_op_rmsnorm(h_ptr, ldh, M, d, w_ptr, eps, y_hi_ptr, y_lo_ptr, fp16=True, stream=0) -> int:
    return load().vla_op_rmsnorm(h_ptr or None, ldh, M, d, w_ptr or None, float(eps), y_hi_ptr or None,
                                 y_lo_ptr or None, 1 if fp16 else 0, stream or None)


def vla_op_read_status(stream=0):
    """(rc, status bits) of the op entry points on the current device; clears the word."""
    st = ctypes.c_uint32(0)
    rc = load().vla_op_read_status(stream or None, ctypes.byref(st))
    return rc, st.value


def vla_test_inject_launch_error(nth_launch: int, cuda_error: int) -> int:
    return load().vla_test_inject_launch_error(int(nth_launch), int(cuda_error))


def vla_test_set_wait_limit_ns(limit_ns: int) -> int:
    return load().vla_test_set_wait_limit_ns(int(limit_ns))


def vla_test_stall_next_gemm() -> int:
    return load().vla_test_stall_next_gemm()


# ---------------------------------------------------------------------------- convenience
class Policy:
    """A handle plus the torch device tensors it borrows (weights) or fills (outputs).

    The four projection matrices are read into the handle's fp16 copy when it is created;
    after changing them in place (a learner update), call ``sync_weights()``.  torch is used
    only to hold device memory and to name the stream; all compute is in libvla.so.
    """

    def __init__(self, shape, weights_dev: Dict, max_batch: int, kv_capacity: int, max_tokens: int,
                 stream=None):
        import torch
        self.torch = torch
        self.shape = shape
        self.w = weights_dev
        L = shape.n_layers
        cfg = VlaConfig(shape.n_layers, shape.d_model, shape.n_heads, shape.head_dim, shape.d_ffn,
                        shape.vocab, shape.n_bins, shape.action_dim, max_batch, kv_capacity, max_tokens,
                        shape.rms_eps, shape.rope_theta)
        arr = lambda name: (ctypes.c_void_p * L)(*[weights_dev[name][l].data_ptr() for l in range(L)])
        self._keep = {n: arr(n) for n in ("attn_norm", "wqkv", "wo", "ffn_norm", "w_gate_up", "w_down")}
        cast = lambda a: ctypes.cast(a, ctypes.POINTER(ctypes.c_void_p))
        wts = VlaWeights(weights_dev["embed"].data_ptr(), cast(self._keep["attn_norm"]),
                         cast(self._keep["wqkv"]), cast(self._keep["wo"]), cast(self._keep["ffn_norm"]),
                         cast(self._keep["w_gate_up"]), cast(self._keep["w_down"]),
                         weights_dev["final_norm"].data_ptr(), weights_dev["lm_head"].data_ptr())
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        self.h = vla_create(cfg, wts, self.stream.cuda_stream)
        self.max_batch = max_batch
        self.B = 0

    def close(self):
        if self.h:
            vla_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def check(self, rc):
        return _check(rc, self.h)

    def prefill(self, visual, ids, lengths):
        """visual bf16 [B, Nv, d] (device), ids int32 [B, L] (device), lengths host ints."""
        B = len(lengths)
        nv = visual.shape[1] if visual is not None else 0
        self.check(vla_prefill(self.h, B, visual.data_ptr() if visual is not None else 0, nv,
                               ids.data_ptr() if ids is not None else 0, list(lengths),
                               ids.shape[1] if ids is not None else 0))
        self.B = B

    def decode(self, uniforms, temperature: float, forced=None, want_logits: bool = True):
        t = self.torch
        B, A = self.B, self.shape.action_dim
        dev = uniforms.device if uniforms is not None else t.device("cuda")
        out = {"tokens": t.empty(B, A, dtype=t.int32, device=dev),
               "logprobs": t.empty(B, A, dtype=t.float32, device=dev),
               "actions": t.empty(B, A, dtype=t.float32, device=dev),
               "logits": t.empty(B, A, 256, dtype=t.float32, device=dev) if want_logits else None}
        self.check(vla_decode_actions(self.h, uniforms.data_ptr() if uniforms is not None else 0, temperature,
                                      forced.data_ptr() if forced is not None else 0, out["tokens"].data_ptr(),
                                      out["logprobs"].data_ptr(), out["actions"].data_ptr(),
                                      out["logits"].data_ptr() if want_logits else 0))
        out["entropy"] = self.entropy(dev)
        return out

    def entropy(self, device=None):
        """Entropies [B, action_dim] of the latest decode / score (vla_action_entropy)."""
        t = self.torch
        e = t.empty(self.B, self.shape.action_dim, dtype=t.float32, device=device or t.device("cuda"))
        self.check(vla_action_entropy(self.h, e.data_ptr()))
        return e

    def value(self, w_value, bias: float):
        """Value-model estimates [B] at the latest prefill (vla_value); w_value bf16 [d] on the GPU."""
        t = self.torch
        v = t.empty(self.B, dtype=t.float32, device=w_value.device)
        self.check(vla_value(self.h, w_value.data_ptr(), bias, v.data_ptr()))
        return v

    def score(self, tokens, temperature: float, want_logits: bool = True):
        t = self.torch
        B, A = self.B, self.shape.action_dim
        out = {"logprobs": t.empty(B, A, dtype=t.float32, device=tokens.device),
               "logits": t.empty(B, A, 256, dtype=t.float32, device=tokens.device) if want_logits else None}
        self.check(vla_score_actions(self.h, tokens.data_ptr(), temperature, out["logprobs"].data_ptr(),
                                     out["logits"].data_ptr() if want_logits else 0))
        out["entropy"] = self.entropy(tokens.device)
        return out

    def reset(self, mask=None):
        self.check(vla_reset(self.h, mask))

    def sync(self):
        self.check(vla_sync(self.h))

    def sync_weights(self):
        """Re-read the projection matrices into the handle's fp16 copy (after an in-place
        update of the bf16 weights this Policy was created with)."""
        self.check(vla_sync_weights(self.h))
