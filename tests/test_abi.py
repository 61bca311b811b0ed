"""The C-ABI library loads and exports every symbol its headers declare; host-side argument
checks return their documented codes without touching a GPU (CPU only)."""
import ctypes
import os
import re

import pytest

from paper_2505_18719_gb300 import build as B
from paper_2505_18719_gb300 import vla as V

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    B.build()
    return V.load()


def declared_functions():
    names = []
    for hdr in ("vla.h", "vla_ops.h"):
        src = open(os.path.join(ROOT, "include", hdr)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names += re.findall(r"\b(vla_[a-z0-9_]+)\s*\(", src)
    return sorted(set(names))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert "vla_create" in names and "vla_decode_actions" in names and "vla_op_gemm_bf16" in names
    for n in names:
        assert hasattr(lib, n), n


def test_host_argument_errors_without_gpu(lib):
    h = ctypes.c_void_p()
    assert lib.vla_create(None, None, None, ctypes.byref(h)) == V.VLA_ERR_ARG
    assert h.value is None
    assert "NULL" in V.vla_last_error(None)
    cfg = V.VlaConfig(2, 256, 4, 48, 688, 32064, 256, 7, 4, 128, 512, 1e-6, 1e4)  # head_dim 48
    w = V.VlaWeights()
    assert lib.vla_create(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(h)) == V.VLA_ERR_UNSUPPORTED
    cfg.head_dim = 64
    cfg.n_action_bins = 128
    assert lib.vla_create(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(h)) == V.VLA_ERR_UNSUPPORTED
    cfg.n_action_bins = 256
    assert lib.vla_create(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(h)) == V.VLA_ERR_ARG  # NULL weights
    assert lib.vla_prefill(None, 1, None, 0, None, None, 0) == V.VLA_ERR_ARG
    assert lib.vla_decode_actions(None, None, 1.0, None, None, None, None, None) == V.VLA_ERR_ARG
    assert lib.vla_score_actions(None, None, 1.0, None, None) == V.VLA_ERR_ARG
    assert lib.vla_reset(None, None) == V.VLA_ERR_ARG
    assert lib.vla_sync(None) == V.VLA_ERR_ARG
    assert lib.vla_context_length(None, 0) == -1
    lib.vla_destroy(None)  # no-op
    assert lib.vla_op_gemm_bf16(None, None, 0, None, 0, None, 0, 0, 0, 0, 256, 1, None, None) == V.VLA_ERR_ARG
    assert lib.vla_sync_weights(None) == V.VLA_ERR_ARG
    assert lib.vla_op_gemm_f16(None, None, 0, None, 0, None, 0, 0, 0, 0, 256, 1, None, None) == V.VLA_ERR_ARG
    assert "vla_op_gemm_f16" in V.vla_last_error(None)
    assert lib.vla_op_gemm_pair_f16(None, None, 0, None, 0, None, 0, 0, 0, 0, None) == V.VLA_ERR_ARG
    assert lib.vla_op_gemm_decode_f16(None, None, 0, None, 0, None, 0, 0, 0, 0, None, 0, None) == V.VLA_ERR_ARG
    assert "vla_op_gemm_decode_f16" in V.vla_last_error(None)
    assert lib.vla_op_action_head(None, 0, 0, 0, None, None, 1e-6, None, 1.0, None, None, None, None,
                                  None, None, None) == V.VLA_ERR_ARG
    assert lib.vla_op_rmsnorm(None, 0, 0, 0, None, 1e-6, None, None, 1, None) == V.VLA_ERR_ARG
    assert "vla_op_rmsnorm" in V.vla_last_error(None)
    assert lib.vla_op_read_status(None, None) == V.VLA_ERR_ARG
    # the chunk attentions check their tiles on the host before any copy or launch: a tile over
    # the kernel's row limit, outside the env range or past the cache capacity, and null buffers
    rows_res = lambda tiles, max_env=2, cap=64: V.vla_op_attn_rows_res(16, 16, 16, max_env, 2, 128, cap, tiles, 32,
                                                                        16, 16, 16)
    assert rows_res([(0, 0, 17, 0)]) == V.VLA_ERR_ARG                 # 17 rows > 16
    assert "16 rows" in V.vla_last_error(None)
    assert rows_res([(2, 0, 4, 0)]) == V.VLA_ERR_ARG                  # env >= max_env
    assert rows_res([(0, 0, 4, 62)]) == V.VLA_ERR_ARG                 # pos0 + nrows > cap
    assert rows_res([(0, 30, 4, 0)]) == V.VLA_ERR_ARG                 # row0 + nrows > rows
    assert V.vla_op_attn_rows_res(0, 16, 16, 2, 2, 128, 64, [(0, 0, 4, 0)], 32, 16, 16, 16) == V.VLA_ERR_ARG
    assert V.vla_op_attn_rows_res(16, 16, 16, 2, 2, 96, 64, [(0, 0, 4, 0)], 32, 16, 16, 16) == V.VLA_ERR_ARG
    assert V.vla_op_attn_chunk_res(16, 16, 16, 2, 2, 128, 64, [(0, 0, 129, 0)], 200, 16, 16, 16) == V.VLA_ERR_ARG
    # failure-injection hooks: argument checks, and arming / disarming touch no device
    assert lib.vla_test_inject_launch_error(-1, 701) == V.VLA_ERR_ARG
    assert lib.vla_test_inject_launch_error(3, 0) == V.VLA_ERR_ARG
    assert lib.vla_test_inject_launch_error(0, 0) == V.VLA_OK
    assert lib.vla_test_set_wait_limit_ns(0) == V.VLA_OK
