"""Single-kernel parity through the C ABI (vla_ops.h): the tcgen05 GEMM and the action head
against fp64 CPU references, on ragged shapes that span several tiles."""
import math
import types

import numpy as np
import pytest
import torch

import oracle.vla_oracle as O
from paper_2505_18719_gb300 import inputs as I
from paper_2505_18719_gb300 import vla as V

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    from paper_2505_18719_gb300 import build
    build.build()
    return V.load()


GEMM_CASES = [
    # M, N, K, block_n, splits, split A (hi/lo pair)
    (1, 128, 64, 128, 1, False),
    (4, 256, 256, 256, 1, True),
    (130, 384, 688, 128, 1, False),     # ragged M and K tails
    (130, 384, 688, 128, 1, True),
    (300, 512, 1024, 256, 1, True),
    (257, 200, 136, 128, 2, True),      # ragged N, split-K
    (64, 384, 4096, 128, 5, False),     # decode-like: few tiles, split-K
    (64, 384, 4096, 128, 5, True),
    (1000, 768, 256, 256, 1, False),    # many tiles (persistent loop, both accumulators)
    (2304, 1024, 512, 256, 1, True),    # > 16 m-tiles: grouped raster
]


@pytest.mark.parametrize("M,N,K,bn,splits,split_a", GEMM_CASES)
def test_gemm_matches_fp64(M, N, K, bn, splits, split_a):
    A = I.normal_bf16((M, K), 99, 1000 + M, 1.0)
    A_lo = I.normal_bf16((M, K), 99, 3000 + M, 2.0 ** -9)   # a realistic low half
    W = I.normal_bf16((N, K), 99, 2000 + N, 1.0)
    Ad, Ald, Wd = A.cuda(), A_lo.cuda(), W.cuda()
    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    ws = torch.empty(max(1, splits * M * N), dtype=torch.float32, device="cuda")
    rc = V.vla_op_gemm_bf16(Ad.data_ptr(), Ald.data_ptr() if split_a else 0, K, Wd.data_ptr(), K,
                            C.data_ptr(), N, M, N, K, bn, splits, ws.data_ptr(), 0)
    assert rc == 0, V.vla_last_error()
    torch.cuda.synchronize()
    Aref = A.double() + A_lo.double() if split_a else A.double()
    ref = Aref @ W.double().T
    err = (C.cpu().double() - ref).abs().max().item()
    # exact bf16 products, fp32 sums: error ~ sqrt(K) * |sum| * 2^-24
    assert err < 2e-5 * math.sqrt(K) * 8, err


PAIR_CASES = [
    # M, N, K, split A
    (1, 256, 64, False),
    (200, 512, 688, True),      # one pair tile in M, ragged K
    (300, 768, 1024, True),     # ragged M over two pair tiles
    (4608, 1024, 512, True),    # many tiles, persistent pairs
    (513, 300, 256, False),     # ragged N
]


@pytest.mark.parametrize("M,N,K,split_a", PAIR_CASES)
def test_pair_gemm_matches_fp64(M, N, K, split_a):
    A = I.normal_bf16((M, K), 97, 1000 + M, 1.0)
    A_lo = I.normal_bf16((M, K), 97, 3000 + M, 2.0 ** -9)
    W = I.normal_bf16((N, K), 97, 2000 + N, 1.0)
    Ad, Ald, Wd = A.cuda(), A_lo.cuda(), W.cuda()
    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    rc = V.vla_op_gemm_pair_bf16(Ad.data_ptr(), Ald.data_ptr() if split_a else 0, K, Wd.data_ptr(), K,
                                 C.data_ptr(), N, M, N, K, 0)
    assert rc == 0, V.vla_last_error()
    torch.cuda.synchronize()
    Aref = A.double() + A_lo.double() if split_a else A.double()
    err = (C.cpu().double() - Aref @ W.double().T).abs().max().item()
    assert err < 2e-5 * math.sqrt(K) * 8, err


DECODE_CASES = [
    # M (<= 128 rows), N, K
    (1, 128, 64),
    (4, 768, 256),
    (16, 3072, 1024),
    (24, 200, 688),        # ragged N and K, score-sized M
    (64, 512, 192),        # 1.5 k-steps of 128
    (64, 12288, 4096),     # 7B q|k|v decode step
    (64, 4096, 11008),     # 7B down-projection decode step
    (100, 1376, 256),
    (128, 4096, 4096),
]


@pytest.mark.parametrize("M,N,K", DECODE_CASES)
def test_decode_gemm_matches_fp64(M, N, K):
    A = I.normal_bf16((M, K), 98, 1000 + M, 1.0)
    A_lo = I.normal_bf16((M, K), 98, 3000 + M, 2.0 ** -9)
    W = I.normal_bf16((N, K), 98, 2000 + N, 1.0)
    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    nbytes = V.vla_op_gemm_decode_workspace_bytes(M, N, K)
    ws = torch.empty(max(1, nbytes // 4), dtype=torch.float32, device="cuda")
    Ad, Ald, Wd = A.cuda(), A_lo.cuda(), W.cuda()
    rc = V.vla_op_gemm_decode_bf16(Ad.data_ptr(), Ald.data_ptr(), K, Wd.data_ptr(), K, C.data_ptr(), N,
                                   M, N, K, ws.data_ptr(), nbytes, 0)
    assert rc == 0, V.vla_last_error()
    torch.cuda.synchronize()
    ref = (A.double() + A_lo.double()) @ W.double().T
    err = (C.cpu().double() - ref).abs().max().item()
    assert err < 2e-5 * math.sqrt(K) * 8, err


def test_gemm_rejects_bad_strides():
    A = torch.zeros(8, 12, dtype=torch.bfloat16, device="cuda")
    C = torch.zeros(8, 8, dtype=torch.float32, device="cuda")
    rc = V.vla_op_gemm_bf16(A.data_ptr(), 0, 12, A.data_ptr(), 12, C.data_ptr(), 8, 8, 8, 12, 128, 1, 0, 0)
    assert rc == V.VLA_ERR_ARG          # 12 * 2 bytes is not a multiple of 16


@pytest.mark.parametrize("T", [0.0, 1.0, 1.5])
@pytest.mark.parametrize("forced", [False, True])
def test_action_head_matches_fp64(T, forced):
    B, d = 16, 4096
    h = I.normal_bf16((B, d), 7, 1, 1.0).float() * 3.0
    fn = I.normal_bf16((d,), 7, 2, 0.1, 1.0)
    rows = I.normal_bf16((256, d), 7, 3, 0.02)
    u = I.uniform_f32((B, 256), 7, 4)
    fb = I.randint_i32((B,), 7, 5, 0, 255)
    dev = {k: v.cuda() for k, v in dict(h=h, fn=fn, rows=rows, u=u, fb=fb).items()}
    bins = torch.empty(B, dtype=torch.int32, device="cuda")
    lp = torch.empty(B, dtype=torch.float32, device="cuda")
    act = torch.empty(B, dtype=torch.float32, device="cuda")
    logits = torch.empty(B, 256, dtype=torch.float32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    rc = V.vla_op_action_head(dev["h"].data_ptr(), d, B, d, dev["fn"].data_ptr(), dev["rows"].data_ptr(),
                              1e-6, dev["u"].data_ptr(), T, dev["fb"].data_ptr() if forced else 0,
                              bins.data_ptr(), lp.data_ptr(), act.data_ptr(), logits.data_ptr(),
                              status.data_ptr(), 0)
    assert rc == 0
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    W = types.SimpleNamespace(final_norm=O.f64(fn), head_rows=O.f64(rows))
    sh = O.Shape(1, d, 32, 128, 8, 32064)
    checked = 0
    for b in range(B):
        z = O.head_logits(sh, W, O.f64(h[b]))
        k, lps, margin = O.sample_bins(z, T, u[b])
        assert np.max(np.abs(logits[b].cpu().numpy() - z.numpy())) < 1e-4
        want = int(fb[b]) if forced else k
        assert abs(lp[b].item() - float(lps[want])) < 1e-4
        if margin > 0.05:
            checked += 1
            assert int(bins[b].item()) == k
            assert act[b].item() == O.bin_centre(k)
    assert checked >= B // 2


@pytest.mark.parametrize("B,H,hd,cap,ctx", [(3, 2, 64, 64, [1, 7, 64]), (5, 4, 128, 1152, [1, 129, 300, 1116, 161]),
                                          (64, 32, 128, 320, None)])
def test_decode_attention_matches_fp64(B, H, hd, cap, ctx):
    """Flash-decoding over the fp16 cache vs brute-force softmax attention in fp64."""
    max_env = B + 1
    kv = I.normal_bf16((max_env, 2, H, cap, hd), 77, B, 1.0).float().half()   # fp16 cache values
    q = I.normal_bf16((B, H, hd), 77, 100 + B, 1.0).float()
    if ctx is None:
        ctx = I.randint_i32((B,), 77, 200, 272, 310).tolist()
    env = torch.tensor([(b * 7 + 1) % max_env for b in range(B)], dtype=torch.int32)
    pos = torch.tensor([c - 1 for c in ctx], dtype=torch.int32)
    max_ctx = max(ctx)
    nbytes = V.vla_op_attn_decode_workspace_bytes(B, H, hd, max_ctx, 0)
    ws = torch.empty(nbytes // 4 + 64, dtype=torch.float32, device="cuda")
    oh = torch.empty(B, H * hd, dtype=torch.bfloat16, device="cuda")
    ol = torch.empty(B, H * hd, dtype=torch.bfloat16, device="cuda")
    kvd, qd, envd, posd = kv.cuda(), q.cuda(), env.cuda(), pos.cuda()
    rc = V.vla_op_attn_decode(qd.data_ptr(), kvd.data_ptr(), max_env, H, hd, cap, envd.data_ptr(), posd.data_ptr(),
                              B, max_ctx, oh.data_ptr(), ol.data_ptr(), ws.data_ptr(), nbytes, 0)
    assert rc == 0, V.vla_last_error()
    torch.cuda.synchronize()
    got = (oh.double() + ol.double()).cpu().reshape(B, H, hd)
    kv64 = kv.double()
    for b in range(B):
        e, n = int(env[b]), ctx[b]
        k, v = kv64[e, 0, :, :n], kv64[e, 1, :, :n]                  # [H, n, hd]
        sc = torch.einsum("hd,hnd->hn", q[b].double(), k) / math.sqrt(hd)
        o = torch.einsum("hn,hnd->hd", torch.softmax(sc, -1), v)
        assert (got[b] - o).abs().max().item() < 1e-4, b


@pytest.mark.parametrize("B,H,hd,cap,ctx", [(3, 2, 64, 64, [1, 7, 64]), (5, 4, 128, 1152, [1, 129, 300, 1116, 161]),
                                          (64, 32, 128, 320, None)])
def test_decode_attention_res_matches_fp64(B, H, hd, cap, ctx):
    """The engine's decode attention, reading fp16 parts and 4-bit residual codes (random), vs
    brute-force softmax attention in fp64 over the values the cache stores (hi + residual);
    positions past each context hold NaN."""
    max_env = B + 1
    hi = I.normal_bf16((max_env, 2, H, cap, hd), 79, B, 1.0).float().half().numpy()
    packed = I.randint_i32((max_env, 2, H, cap, hd // 2), 79, 50 + B, 0, 256).to(torch.uint8).numpy()
    q = I.normal_bf16((B, H, hd), 79, 100 + B, 1.0).float()
    if ctx is None:
        ctx = I.randint_i32((B,), 79, 200, 272, 310).tolist()
    env = torch.tensor([(b * 7 + 1) % max_env for b in range(B)], dtype=torch.int32)
    pos = torch.tensor([c - 1 for c in ctx], dtype=torch.int32)
    value = _decode_res4(hi, packed)
    for b in range(B):
        hi[int(env[b]), :, :, ctx[b]:] = np.float16("nan")
    max_ctx = max(ctx)
    nbytes = V.vla_op_attn_decode_workspace_bytes(B, H, hd, max_ctx, 0)
    ws = torch.empty(nbytes // 4 + 64, dtype=torch.float32, device="cuda")
    oh = torch.empty(B, H * hd, dtype=torch.bfloat16, device="cuda")
    ol = torch.empty(B, H * hd, dtype=torch.bfloat16, device="cuda")
    kvd, rsd, qd = torch.from_numpy(hi).cuda(), torch.from_numpy(packed).cuda(), q.cuda()
    envd, posd = env.cuda(), pos.cuda()
    rc = V.vla_op_attn_decode_res(qd.data_ptr(), kvd.data_ptr(), rsd.data_ptr(), max_env, H, hd, cap, envd.data_ptr(),
                                  posd.data_ptr(), B, max_ctx, oh.data_ptr(), ol.data_ptr(), ws.data_ptr(), nbytes, 0)
    assert rc == 0, V.vla_last_error()
    torch.cuda.synchronize()
    got = (oh.double() + ol.double()).cpu().reshape(B, H, hd)
    kv64 = torch.from_numpy(value)
    err = err_hi = 0.0
    for b in range(B):
        e, n = int(env[b]), ctx[b]
        k, v = kv64[e, 0, :, :n], kv64[e, 1, :, :n]                  # [H, n, hd]
        sc = torch.einsum("hd,hnd->hn", q[b].double(), k) / math.sqrt(hd)
        o = torch.einsum("hn,hnd->hd", torch.softmax(sc, -1), v)
        err = max(err, (got[b] - o).abs().max().item())
        kh, vh = (torch.from_numpy(hi[e, i, :, :n].astype(np.float64)) for i in (0, 1))
        sh = torch.einsum("hd,hnd->hn", q[b].double(), kh) / math.sqrt(hd)
        err_hi = max(err_hi, (got[b] - torch.einsum("hn,hnd->hd", torch.softmax(sh, -1), vh)).abs().max().item())
    assert err < 1e-4, err
    assert err_hi > 4 * err, (err, err_hi)   # the residual is read, not just the fp16 part


@pytest.mark.parametrize("hd", [64, 128])
def test_chunk_attention_matches_fp64(hd):
    """Prefill / score chunk attention vs brute-force causal softmax attention in fp64: chunks of
    1..130 rows appended after 0..200 cached positions, split into tiles of <= 64 rows."""
    H, cap, max_env = 3, 384, 6
    chunks = [(0, 0, 1), (1, 0, 63), (2, 0, 64), (3, 7, 130), (4, 200, 17), (5, 100, 64)]  # (env, past, n)
    rows = sum(n for _, _, n in chunks)
    kv = I.normal_bf16((max_env, 2, H, cap, hd), 91, hd, 1.0).float().half()
    q = I.normal_bf16((rows, H * hd), 91, 1000 + hd, 1.0).float()
    tiles, qpos, qenv = [], [], []
    r = 0
    for env, past, n in chunks:
        for t0 in range(0, n, 64):
            tiles.append((env, r + t0, min(64, n - t0), past + t0))
        qpos += [past + i for i in range(n)]
        qenv += [env] * n
        r += n
    tiles_dev = torch.zeros(len(tiles) * 4, dtype=torch.int32, device="cuda")
    oh = torch.empty(rows, H * hd, dtype=torch.bfloat16, device="cuda")
    ol = torch.empty_like(oh)
    qd, kvd = q.cuda(), kv.cuda()
    rc = V.vla_op_attn_chunk(qd.data_ptr(), kvd.data_ptr(), max_env, H, hd, cap, tiles, rows,
                             tiles_dev.data_ptr(), oh.data_ptr(), ol.data_ptr())
    assert rc == 0, V.vla_last_error(None)
    torch.cuda.synchronize()
    out = oh.cpu().double() + ol.cpu().double()
    kv64 = kv.double()
    err = 0.0
    for i in range(rows):
        env, p = qenv[i], qpos[i]
        for hh in range(H):
            qi = q[i, hh * hd:(hh + 1) * hd].double()
            K = kv64[env, 0, hh, :p + 1]
            Vv = kv64[env, 1, hh, :p + 1]
            w = torch.softmax(K @ qi / math.sqrt(hd), dim=0)
            err = max(err, float((out[i, hh * hd:(hh + 1) * hd] - w @ Vv).abs().max()))
    assert err < 3e-3, err
    # a tile outside the buffers is refused on the host
    bad = [(0, 0, 65, 0)]
    assert V.vla_op_attn_chunk(qd.data_ptr(), kvd.data_ptr(), max_env, H, hd, cap, bad, rows,
                               tiles_dev.data_ptr(), oh.data_ptr(), ol.data_ptr()) == V.VLA_ERR_ARG



# ------------------------------------------------------------------ fp16 operands (engine form)
def _f16_operands(M, N, K, seed):
    """fp16 A (11 significant bits used), its low half, and fp16 W, built from the seeded bf16
    generators: bf16 values plus a finer bf16 term, rounded once to fp16."""
    A = (I.normal_bf16((M, K), seed, 1000 + M, 1.0).float()
         + I.normal_bf16((M, K), seed, 5000 + M, 2.0 ** -8).float()).half()
    A_lo = I.normal_bf16((M, K), seed, 3000 + M, 2.0 ** -12).half()
    W = (I.normal_bf16((N, K), seed, 2000 + N, 1.0).float()
         + I.normal_bf16((N, K), seed, 6000 + N, 2.0 ** -8).float()).half()
    return A, A_lo, W


@pytest.mark.parametrize("M,N,K,bn,splits,split_a", GEMM_CASES[1::2] + [GEMM_CASES[0]])
def test_gemm_f16_matches_fp64(M, N, K, bn, splits, split_a):
    A, A_lo, W = _f16_operands(M, N, K, 91)
    Ad, Ald, Wd = A.cuda(), A_lo.cuda(), W.cuda()
    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    ws = torch.empty(max(1, splits * M * N), dtype=torch.float32, device="cuda")
    rc = V.vla_op_gemm_f16(Ad.data_ptr(), Ald.data_ptr() if split_a else 0, K, Wd.data_ptr(), K,
                           C.data_ptr(), N, M, N, K, bn, splits, ws.data_ptr(), 0)
    assert rc == 0, V.vla_last_error()
    torch.cuda.synchronize()
    Aref = A.double() + A_lo.double() if split_a else A.double()
    err = (C.cpu().double() - Aref @ W.double().T).abs().max().item()
    # fp16 x fp16 products are exact in fp32; the error is the fp32 sums'
    assert err < 2e-5 * math.sqrt(K) * 8, err


@pytest.mark.parametrize("M,N,K,split_a", PAIR_CASES)
def test_pair_gemm_f16_matches_fp64(M, N, K, split_a):
    A, A_lo, W = _f16_operands(M, N, K, 92)
    Ad, Ald, Wd = A.cuda(), A_lo.cuda(), W.cuda()
    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    rc = V.vla_op_gemm_pair_f16(Ad.data_ptr(), Ald.data_ptr() if split_a else 0, K, Wd.data_ptr(), K,
                                C.data_ptr(), N, M, N, K, 0)
    assert rc == 0, V.vla_last_error()
    torch.cuda.synchronize()
    Aref = A.double() + A_lo.double() if split_a else A.double()
    err = (C.cpu().double() - Aref @ W.double().T).abs().max().item()
    assert err < 2e-5 * math.sqrt(K) * 8, err


@pytest.mark.parametrize("M,N,K", DECODE_CASES[::2])
def test_decode_gemm_f16_matches_fp64(M, N, K):
    A, A_lo, W = _f16_operands(M, N, K, 93)
    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    nbytes = V.vla_op_gemm_decode_workspace_bytes(M, N, K)
    ws = torch.empty(max(1, nbytes // 4), dtype=torch.float32, device="cuda")
    Ad, Ald, Wd = A.cuda(), A_lo.cuda(), W.cuda()
    rc = V.vla_op_gemm_decode_f16(Ad.data_ptr(), Ald.data_ptr(), K, Wd.data_ptr(), K, C.data_ptr(), N,
                                  M, N, K, ws.data_ptr(), nbytes, 0)
    assert rc == 0, V.vla_last_error()
    torch.cuda.synchronize()
    err = (C.cpu().double() - (A.double() + A_lo.double()) @ W.double().T).abs().max().item()
    assert err < 2e-5 * math.sqrt(K) * 8, err


# ------------------------------------------------------------------ RMSNorm (operand-pair output)
@pytest.mark.parametrize("fp16", [True, False])
def test_rmsnorm_matches_fp64(fp16):
    M, d, ldh = 37, 4096, 4100
    h = I.normal_bf16((M, ldh), 95, 1, 3.0).float()
    w = I.normal_bf16((d,), 95, 2, 1.0, mean=1.0)
    hd_, wd = h.cuda(), w.cuda()
    dt = torch.float16 if fp16 else torch.bfloat16
    yh = torch.empty(M, d, dtype=dt, device="cuda")
    yl = torch.empty_like(yh)
    assert V.vla_op_rmsnorm(hd_.data_ptr(), ldh, M, d, wd.data_ptr(), 1e-6, yh.data_ptr(), yl.data_ptr(),
                            fp16) == 0, V.vla_last_error()
    assert V.vla_op_read_status() == (0, 0)
    x = h[:, :d].double()
    ref = O.rms_norm(x, w.double(), 1e-6)
    got = yh.cpu().double() + yl.cpu().double()
    # the pair keeps ~21 (fp16) / ~16 (bf16) significant bits; fp32 math before the split
    rel = (got - ref).abs().max().item() / ref.abs().max().item()
    assert rel < (2e-6 if fp16 else 2e-5), rel
    # hi alone is the round-to-nearest of the value in that format
    assert (yh.cpu().double() - ref).abs().max().item() <= ref.abs().max().item() * (2.0 ** -11 if fp16 else 2.0 ** -8)


# ------------------------------------------------------------------ tcgen05 chunk attention (fp16 + 4-bit residual cache)
def _encode_res4(x32: np.ndarray):
    """Host encoding of the cache's 4-bit residual, written from its definition: hi = fp16(x),
    code c = 8 + clamp(floor((x - hi) / ulp(hi) * 16), -8, 7), value hi + (2c - 15) ulp(hi) / 32
    with ulp(hi) = 2^(e-25) (biased exponent e >= 1) or 2^-24.  Returns (hi, packed codes, value)."""
    hi = x32.astype(np.float16)
    e = ((hi.view(np.uint16) >> 10) & 31).astype(np.int64)
    ee = np.maximum(e, 1)
    j = np.floor((x32.astype(np.float64) - hi.astype(np.float64)) * np.ldexp(1.0, 29 - ee))
    c = (np.clip(j, -8, 7) + 8).astype(np.uint8)
    value = hi.astype(np.float64) + (2.0 * c - 15.0) * np.ldexp(1.0, ee - 30)
    packed = (c[..., 0::2] | (c[..., 1::2] << 4)).astype(np.uint8)
    return hi, packed, value


@pytest.mark.parametrize("hd", [128, 64])
def test_chunk_attention_tc_matches_fp64(hd):
    """The tcgen05 chunk attention vs brute-force causal softmax attention in fp64 over the values
    the cache stores (fp16 + residual): chunks of 1..200 rows after 0..300 cached positions, tiles
    of <= 128 rows, a context reaching the last cache position (cap not a multiple of 64).  Cache
    positions past each env's context hold NaN, as stale rows may: they must not reach the output."""
    H, cap, max_env = 3, 400, 6
    chunks = [(0, 0, 1), (1, 0, 127), (2, 0, 128), (3, 7, 200), (4, 300, 100), (5, 100, 64)]  # (env, past, n)
    rows = sum(n for _, _, n in chunks)
    x = (I.normal_bf16((max_env, 2, H, cap, hd), 93, hd, 1.0).float()
         + I.normal_bf16((max_env, 2, H, cap, hd), 93, 7 + hd, 2.0 ** -9).float()).numpy()
    hi, packed, value = _encode_res4(x)
    for env, past, n in chunks:
        hi[env, :, :, past + n:] = np.float16("nan")
    q = I.normal_bf16((rows, H * hd), 93, 1000 + hd, 1.0).float()
    tiles, qpos, qenv = [], [], []
    r = 0
    for env, past, n in chunks:
        for t0 in range(0, n, 128):
            tiles.append((env, r + t0, min(128, n - t0), past + t0))
        qpos += [past + i for i in range(n)]
        qenv += [env] * n
        r += n
    tiles_dev = torch.zeros(len(tiles) * 4, dtype=torch.int32, device="cuda")
    oh = torch.full((rows, H * hd), float("nan"), dtype=torch.bfloat16, device="cuda")
    ol = torch.full_like(oh, float("nan"))
    qd = q.cuda()
    kvd = torch.from_numpy(hi).cuda()
    rsd = torch.from_numpy(packed).cuda()
    assert V.vla_op_read_status()[0] == 0
    rc = V.vla_op_attn_chunk_res(qd.data_ptr(), kvd.data_ptr(), rsd.data_ptr(), max_env, H, hd, cap, tiles, rows,
                                 tiles_dev.data_ptr(), oh.data_ptr(), ol.data_ptr())
    assert rc == 0, V.vla_last_error(None)
    assert V.vla_op_read_status() == (0, 0)
    out = oh.cpu().double() + ol.cpu().double()
    kv64 = torch.from_numpy(value)
    kvhi = torch.from_numpy(hi.astype(np.float64))
    err = err_hi = 0.0
    for i in range(rows):
        env, p = qenv[i], qpos[i]
        for hh in range(H):
            qi = q[i, hh * hd:(hh + 1) * hd].double()
            o = out[i, hh * hd:(hh + 1) * hd]
            K, Vv = kv64[env, 0, hh, :p + 1], kv64[env, 1, hh, :p + 1]
            w = torch.softmax(K @ qi / math.sqrt(hd), dim=0)
            err = max(err, float((o - w @ Vv).abs().max()))
            Kh, Vh = kvhi[env, 0, hh, :p + 1], kvhi[env, 1, hh, :p + 1]
            wh = torch.softmax(Kh @ qi / math.sqrt(hd), dim=0)
            err_hi = max(err_hi, float((o - wh @ Vh).abs().max()))
    # hi / lo products in fp32, the bf16 output pair (~16 bits): far below the fp16 cache's own error
    assert err < 1e-4, err
    assert err_hi > 4 * err, (err, err_hi)   # the residual is read, not just the fp16 part
    bad = [(0, 0, 129, 0)]
    assert V.vla_op_attn_chunk_res(qd.data_ptr(), kvd.data_ptr(), rsd.data_ptr(), max_env, H, hd, cap, bad, rows,
                                   tiles_dev.data_ptr(), oh.data_ptr(), ol.data_ptr()) == V.VLA_ERR_ARG


@pytest.mark.parametrize("hd", [128, 64])
def test_attn_rows_res_matches_fp64(hd):
    """The few-row chunk attention (tiles of <= 16 rows) vs brute-force causal softmax attention in
    fp64 over the cached values (fp16 + residual): 1..16 rows after 0..300 cached positions, tiles
    crossing a 64-key block boundary, the context reaching the last cache position, NaN past each
    env's context; a 17-row tile is rejected on the host."""
    H, cap, max_env = 3, 316, 7
    chunks = [(0, 0, 1), (1, 0, 16), (2, 7, 5), (3, 300, 16), (4, 100, 6), (5, 60, 9), (6, 63, 1)]
    rows = sum(n for _, _, n in chunks)
    x = (I.normal_bf16((max_env, 2, H, cap, hd), 95, hd, 1.0).float()
         + I.normal_bf16((max_env, 2, H, cap, hd), 95, 7 + hd, 2.0 ** -9).float()).numpy()
    hi, packed, value = _encode_res4(x)
    for env, past, n in chunks:
        hi[env, :, :, past + n:] = np.float16("nan")
    q = I.normal_bf16((rows, H * hd), 95, 1000 + hd, 1.0).float()
    tiles, qpos, qenv = [], [], []
    r = 0
    for env, past, n in chunks:
        tiles.append((env, r, n, past))
        qpos += [past + i for i in range(n)]
        qenv += [env] * n
        r += n
    tiles_dev = torch.zeros(len(tiles) * 4, dtype=torch.int32, device="cuda")
    oh = torch.full((rows, H * hd), float("nan"), dtype=torch.bfloat16, device="cuda")
    ol = torch.full_like(oh, float("nan"))
    qd, kvd, rsd = q.cuda(), torch.from_numpy(hi).cuda(), torch.from_numpy(packed).cuda()
    rc = V.vla_op_attn_rows_res(qd.data_ptr(), kvd.data_ptr(), rsd.data_ptr(), max_env, H, hd, cap, tiles, rows,
                                tiles_dev.data_ptr(), oh.data_ptr(), ol.data_ptr())
    assert rc == 0, V.vla_last_error(None)
    out = oh.cpu().double() + ol.cpu().double()
    kv64 = torch.from_numpy(value)
    kvhi = torch.from_numpy(hi.astype(np.float64))
    err = err_hi = 0.0
    for i in range(rows):
        env, p = qenv[i], qpos[i]
        for hh in range(H):
            qi = q[i, hh * hd:(hh + 1) * hd].double()
            o = out[i, hh * hd:(hh + 1) * hd]
            K, Vv = kv64[env, 0, hh, :p + 1], kv64[env, 1, hh, :p + 1]
            w = torch.softmax(K @ qi / math.sqrt(hd), dim=0)
            err = max(err, float((o - w @ Vv).abs().max()))
            Kh, Vh = kvhi[env, 0, hh, :p + 1], kvhi[env, 1, hh, :p + 1]
            wh = torch.softmax(Kh @ qi / math.sqrt(hd), dim=0)
            err_hi = max(err_hi, float((o - wh @ Vh).abs().max()))
    assert err < 1e-4, err
    assert err_hi > 4 * err, (err, err_hi)   # the residual is read, not just the fp16 part
    bad = [(0, 0, 17, 0)]
    assert V.vla_op_attn_rows_res(qd.data_ptr(), kvd.data_ptr(), rsd.data_ptr(), max_env, H, hd, cap, bad, rows,
                                  tiles_dev.data_ptr(), oh.data_ptr(), ol.data_ptr()) == V.VLA_ERR_ARG


def _decode_res4(hi: np.ndarray, packed: np.ndarray) -> np.ndarray:
    """The cached values from the fp16 parts and their packed 4-bit codes, from the definition:
    hi + (2c - 15) ulp(hi) / 32 with ulp(hi) = 2^(e-25) (biased exponent e >= 1) or 2^-24."""
    c = np.empty(hi.shape, dtype=np.int64)
    c[..., 0::2] = packed & 15
    c[..., 1::2] = packed >> 4
    e = ((hi.view(np.uint16) >> 10) & 31).astype(np.int64)
    return hi.astype(np.float64) + (2.0 * c - 15.0) * np.ldexp(1.0, np.maximum(e, 1) - 30)


@pytest.mark.parametrize("score,growing", [(False, False), (True, False), (False, True), (True, True)])
def test_chunk_attention_tc_full_size_sampled(score, growing):
    """The engine's chunk attention at the bench step's size: 64 envs x 32 heads x 128, contexts
    of 256 + U{16..48} positions in a 320-position cache.  Prefill: each env's whole context as
    one chunk in tiles of <= 128 rows (192 tiles, 6144 (tile, head) items, ~41 per persistent
    CTA); score: 6 rows after the context (64 tiles, 2048 items).  Random fp16 parts and residual
    codes, NaN past each env's last position; sampled (row, head) outputs vs fp64 brute force.
    growing: logits rising by ~0.2 per key position (dimension 0 of every key grows along the
    sequence, every query has 8 there), so each 64-key block's maximum exceeds the running one
    by far more than the kernel's rescale threshold and O is rescaled at every block, while the
    S products of the following blocks are already in flight."""
    B, H, hd, cap = 64, 32, 128, 320
    ctx = (256 + I.randint_i32((B,), 97, 3, 16, 49)).tolist()
    lens = [6] * B if score else [c - 6 for c in ctx]
    past = [c - 6 for c in ctx] if score else [0] * B
    hi = I.normal_bf16((B, 2, H, cap, hd), 97, 1, 1.0).float().half().numpy()
    if growing:
        hi[:, 0, :, :, 0] = (0.21 * np.arange(cap)).astype(np.float16)
    packed = I.randint_i32((B, 2, H, cap, hd // 2), 97, 2, 0, 256).to(torch.uint8).numpy()
    for b in range(B):
        hi[b, :, :, past[b] + lens[b]:] = np.float16("nan")
    rows = sum(lens)
    q = I.normal_bf16((rows, H * hd), 97, 4, 1.0).float()
    if growing:
        q[:, ::hd] = 8.0
    tiles, row_env, row_pos, tile_of_row = [], [], [], []
    r = 0
    for b, n in enumerate(lens):
        for t0 in range(0, n, 128):
            tiles.append((b, r + t0, min(128, n - t0), past[b] + t0))
        row_env += [b] * n
        row_pos += [past[b] + i for i in range(n)]
        r += n
    tiles_dev = torch.zeros(len(tiles) * 4, dtype=torch.int32, device="cuda")
    oh = torch.full((rows, H * hd), float("nan"), dtype=torch.bfloat16, device="cuda")
    ol = torch.full_like(oh, float("nan"))
    qd, kvd, rsd = q.cuda(), torch.from_numpy(hi).cuda(), torch.from_numpy(packed).cuda()
    assert V.vla_op_read_status()[0] == 0
    assert V.vla_op_attn_chunk_res(qd.data_ptr(), kvd.data_ptr(), rsd.data_ptr(), B, H, hd, cap, tiles, rows,
                                   tiles_dev.data_ptr(), oh.data_ptr(), ol.data_ptr()) == 0
    assert V.vla_op_read_status() == (0, 0)
    outs = [oh.cpu().double() + ol.cpu().double()]
    if score:
        # the few-row kernel the engine runs on these tiles
        oh.fill_(float("nan"))
        ol.fill_(float("nan"))
        assert V.vla_op_attn_rows_res(qd.data_ptr(), kvd.data_ptr(), rsd.data_ptr(), B, H, hd, cap, tiles, rows,
                                      tiles_dev.data_ptr(), oh.data_ptr(), ol.data_ptr()) == 0
        outs.append(oh.cpu().double() + ol.cpu().double())
    for out in outs:
        assert torch.isfinite(out).all()
    rng = np.random.default_rng(11)
    picks = [(int(i), int(h)) for i, h in zip(rng.integers(0, rows, 48), rng.integers(0, H, 48))]
    picks += [(t[1] + t[2] - 1, (k * 7) % H) for k, t in enumerate(tiles[::9])]   # tiles' last rows
    err = 0.0
    for i, h in picks:
        b, p = row_env[i], row_pos[i]
        K = _decode_res4(hi[b, 0, h, :p + 1], packed[b, 0, h, :p + 1])
        Vv = _decode_res4(hi[b, 1, h, :p + 1], packed[b, 1, h, :p + 1])
        qi = q[i, h * hd:(h + 1) * hd].double().numpy()
        s = K @ qi / math.sqrt(hd)
        w = np.exp(s - s.max())
        ref = (w / w.sum()) @ Vv
        for out in outs:
            err = max(err, float(np.abs(out[i, h * hd:(h + 1) * hd].numpy() - ref).max()))
    assert err < 1e-4, err


def test_pair_gemm_f16_full_size_sampled():
    """The prefill q|k|v projection at the bench step's full size, M = 18385 rows (64 envs x
    (256 + U{16..48})), N = 12288, K = 4096, on CTA pairs with the fp16 activation pair: sampled
    outputs (random, every tile edge in m and n, the ragged last rows) vs fp64 sums over the same
    fp16 values, within fp32 accumulation error."""
    M, N, K = 18385, 12288, 4096
    A = I.normal_bf16((M, K), 31, 1, 1.0).float().half()
    A_lo = (I.normal_bf16((M, K), 31, 2, 1.0).float() * 2.0 ** -12).half()
    W = I.normal_bf16((N, K), 31, 3, 0.02).float().half()
    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    Ad, Ald, Wd = A.cuda(), A_lo.cuda(), W.cuda()
    assert V.vla_op_gemm_pair_f16(Ad.data_ptr(), Ald.data_ptr(), K, Wd.data_ptr(), K, C.data_ptr(), N, M, N, K, 0) == 0
    torch.cuda.synchronize()
    rng = np.random.default_rng(3)
    ms = list(rng.integers(0, M, 40)) + [0, 255, 256, 2047, 2048, M - 256, M - 2, M - 1]
    ns = list(rng.integers(0, N, 40)) + [0, 255, 256, 4095, 4096, 8191, 8192, N - 1]
    Cs = C[torch.tensor(ms)][:, torch.tensor(ns)].cpu().double()
    a = A[ms].double() + A_lo[ms].double()
    w = W[ns].double()
    ref = a @ w.T
    bound = (a.abs() @ w.abs().T) * 3e-5 + 1e-6
    assert torch.isfinite(Cs).all()
    assert ((Cs - ref).abs() <= bound).all(), float(((Cs - ref).abs() / bound).max())
