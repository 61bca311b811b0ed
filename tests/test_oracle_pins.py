"""Pins of the fp64 oracle against things other than itself (CPU only).

Each pin is a closed form, a hand-worked fixture under tests/golden/, an invariant the
method fixes, or a brute-force pure-Python restatement (tests/bruteforce.py) on tiny
inputs.  The mutation tests at the end plant plausible mistakes in the oracle and check
that a pin catches each of them.
"""
import math
import os
import types

import numpy as np
import pytest
import torch

import oracle.vla_oracle as O
from paper_2505_18719_gb300 import inputs as I
from tests import bruteforce as BF

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
MICRO = O.Shape(n_layers=2, d_model=8, n_heads=2, head_dim=4, d_ffn=12, vocab=300)


def read_fixture(name):
    vals = {}
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if not line:
                continue
            if "=" in line:
                k, v = line.split("=", 1)
                vals[k.strip()] = [float(t) for t in v.split()]
            else:
                rows.append([float(t) for t in line.split()])
    return vals, rows


def micro_weights(seed=7, std=0.3):
    sh = MICRO
    L, d, F, V = sh.n_layers, sh.d_model, sh.d_ffn, sh.vocab
    return {
        "embed": I.normal_bf16((V, d), seed, 1, 1.0),
        "lm_head": I.normal_bf16((V, d), seed, 2, std),
        "final_norm": I.normal_bf16((d,), seed, 3, 0.2, 1.0),
        "attn_norm": I.normal_bf16((L, d), seed, 4, 0.2, 1.0),
        "ffn_norm": I.normal_bf16((L, d), seed, 5, 0.2, 1.0),
        "wqkv": I.normal_bf16((L, 3 * d, d), seed, 6, std),
        "wo": I.normal_bf16((L, d, d), seed, 7, std),
        "w_gate_up": I.normal_bf16((L, 2 * F, d), seed, 8, std),
        "w_down": I.normal_bf16((L, d, F), seed, 9, std),
    }


def as_lists(w):
    out = {}
    for k, t in w.items():
        out[k] = t.double().tolist()
    return out


def micro_rows(n, seed=11):
    return I.normal_bf16((n, MICRO.d_model), seed, 1, 1.0)


# ============================================================================ layers
def test_rmsnorm_closed_form():
    d = 8
    w = torch.linspace(0.5, 2.0, d, dtype=torch.float64)
    c = -3.0
    x = torch.full((d,), c, dtype=torch.float64)
    y = O.rms_norm(x, w, 1e-6)
    expect = w * (c / math.sqrt(c * c + 1e-6))
    assert torch.allclose(y, expect, rtol=0, atol=1e-15)
    # [3, 4]: mean square 12.5
    y2 = O.rms_norm(torch.tensor([3.0, 4.0], dtype=torch.float64),
                    torch.ones(2, dtype=torch.float64), 0.0)
    assert abs(y2[0].item() - 3 / math.sqrt(12.5)) < 1e-15
    assert abs(y2[1].item() - 4 / math.sqrt(12.5)) < 1e-15


def test_rope_golden_fixture():
    v, _ = read_fixture("rope_hd4_pos1.txt")
    x = torch.tensor(v["x"], dtype=torch.float64).reshape(1, 1, 4)
    y = O.apply_rope(x, torch.tensor([int(v["pos"][0])]), v["theta"][0]).reshape(4)
    assert torch.allclose(y, torch.tensor(v["expected"], dtype=torch.float64), rtol=0, atol=1e-14)


def test_rope_invariants():
    g = torch.Generator().manual_seed(0)
    x = torch.randn(5, 3, 8, generator=g, dtype=torch.float64)
    # position 0 is the identity
    assert torch.equal(O.apply_rope(x[:1], torch.tensor([0]), 1e4), x[:1])
    # every (i, i + hd/2) pair keeps its norm
    pos = torch.tensor([0, 1, 7, 100, 1115])
    y = O.apply_rope(x, pos, 1e4)
    nx = x[..., :4] ** 2 + x[..., 4:] ** 2
    ny = y[..., :4] ** 2 + y[..., 4:] ** 2
    assert torch.allclose(nx, ny, rtol=0, atol=1e-12)
    # q(m) . k(n) depends only on m - n
    q, k = x[0:1], x[1:2]
    def dot(m, n):
        return (O.apply_rope(q, torch.tensor([m]), 1e4) * O.apply_rope(k, torch.tensor([n]), 1e4)).sum(-1)
    assert torch.allclose(dot(5, 2), dot(13, 10), rtol=0, atol=1e-12)
    assert torch.allclose(dot(300, 1), dot(1299, 1000), rtol=0, atol=1e-10)


def test_attention_golden_fixture():
    v, _ = read_fixture("attention_two_keys.txt")
    t = lambda a: torch.tensor(a, dtype=torch.float64).reshape(1, 1, 2)
    k = torch.cat([t(v["k0"]), t(v["k1"])], 0)
    val = torch.cat([t(v["v0"]), t(v["v1"])], 0)
    kpos = torch.tensor([0, 1])
    o1 = O.causal_attention(t(v["q"]), k, val, torch.tensor([1]), kpos).reshape(2)
    o0 = O.causal_attention(t(v["q"]), k, val, torch.tensor([0]), kpos).reshape(2)
    assert torch.allclose(o1, torch.tensor(v["expected_pos1"], dtype=torch.float64), atol=1e-14)
    assert torch.allclose(o0, torch.tensor(v["expected_pos0"], dtype=torch.float64), atol=1e-14)


def test_attention_causality_and_uniform():
    g = torch.Generator().manual_seed(1)
    q = torch.randn(4, 2, 8, generator=g, dtype=torch.float64)
    k = torch.randn(6, 2, 8, generator=g, dtype=torch.float64)
    v = torch.randn(6, 2, 8, generator=g, dtype=torch.float64)
    qpos, kpos = torch.tensor([2, 3, 4, 5]), torch.arange(6)
    o = O.causal_attention(q, k, v, qpos, kpos)
    k2, v2 = k.clone(), v.clone()
    k2[5] += 10.0
    v2[5] -= 3.0
    o2 = O.causal_attention(q, k2, v2, qpos, kpos)
    assert torch.equal(o[:3], o2[:3])        # future keys never leak backwards
    assert not torch.allclose(o[3], o2[3])
    # identical keys -> mean of the visible values
    ku = torch.ones(6, 2, 8, dtype=torch.float64)
    ou = O.causal_attention(q, ku, v, qpos, kpos)
    for i, p in enumerate(qpos.tolist()):
        assert torch.allclose(ou[i], v[:p + 1].mean(0), atol=1e-14)


def test_silu_closed_form():
    x = torch.tensor([0.0, 1.0, -2.0, 30.0], dtype=torch.float64)
    y = O.silu(x)
    assert y[0].item() == 0.0
    assert abs(y[1].item() - 1.0 / (1.0 + math.exp(-1.0))) < 1e-16
    assert abs(y[2].item() - (-2.0 / (1.0 + math.exp(2.0)))) < 1e-16
    assert abs(y[3].item() - 30.0) < 1e-9
    z = torch.linspace(-5, 5, 11, dtype=torch.float64)
    assert torch.allclose(O.silu(-z), O.silu(z) - z, atol=1e-14)


# ============================================================================ decoder
def test_decoder_matches_bruteforce():
    w = micro_weights()
    Wt = O.Weights(MICRO, w)
    x = micro_rows(6)
    ours = O.full_forward(MICRO, Wt, O.f64(x))
    wl = as_lists(w)
    ref = BF.decoder(x.double().tolist(), wl, MICRO.n_layers, MICRO.n_heads, MICRO.head_dim,
                     MICRO.d_ffn, MICRO.rms_eps, MICRO.rope_theta)
    assert np.max(np.abs(ours.numpy() - np.array(ref))) < 1e-12
    # head
    V, nb = MICRO.vocab, MICRO.n_bins
    for T in (1.0, 1.5):
        z_ref, lp_ref = BF.head(ref[-1], wl["final_norm"], wl["lm_head"][V - nb:], MICRO.rms_eps, T)
        z = O.head_logits(MICRO, Wt, ours[-1])
        _, lp, _ = O.sample_bins(z, T, None)
        assert np.max(np.abs(z.numpy() - np.array(z_ref))) < 1e-12
        assert np.max(np.abs(lp.numpy() - np.array(lp_ref))) < 1e-12


def _micro_oracle(n_envs):
    return O.Oracle(MICRO, micro_weights(), n_envs)


def _prefill(orc, envs, n_vis, lens, seed=21):
    vis = [I.normal_bf16((n_vis, MICRO.d_model), seed, 100 + b, 1.0) for b in envs]
    ids = [I.randint_i32((lens[j],), seed, 200 + b, 0, MICRO.vocab - MICRO.n_bins - 1).tolist()
           for j, b in enumerate(envs)]
    orc.prefill(envs, vis, ids)
    return vis, ids


def _uniforms(n, seed=31):
    return I.uniform_f32((n, MICRO.action_dim, MICRO.n_bins), seed, 5)


def test_kv_cached_decode_equals_full_recompute():
    orc = _micro_oracle(2)
    _prefill(orc, [0, 1], 3, [2, 4])
    out = orc.decode([0, 1], _uniforms(2), 1.0)
    V, nb = MICRO.vocab, MICRO.n_bins
    for j, b in enumerate([0, 1]):
        toks = out["tokens"][j].tolist()
        # state after decode: prefix + a1..a6 cached, a7 pending
        e = orc.envs[b]
        assert e.length == e.len_prefill + 6 and e.pending == toks[6]
        for i in range(MICRO.action_dim):
            # recompute from the prefix rows + a_1..a_{i-1} with no KV reuse
            rows = list(e.rows[:e.len_prefill]) + list(orc.W.embed_rows(toks[:i]))
            h = O.full_forward(MICRO, orc.W, torch.stack(rows))[-1]
            z = O.head_logits(MICRO, orc.W, h)
            _, lp, _ = O.sample_bins(z, 1.0, None)
            assert abs(float(lp[toks[i] - (V - nb)]) - out["logprobs"][j, i]) < 1e-12
            assert np.max(np.abs(z.numpy() - out["logits"][j, i])) < 1e-12
        # Eq. 1: the sequence log-prob is the sum of the token log-probs, i.e. the log of
        # the product of the seven conditional probabilities
        seq = float(np.sum(out["logprobs"][j]))
        prod = float(np.prod(np.exp(out["logprobs"][j])))
        assert abs(seq - math.log(prod)) < 1e-12


def test_multiturn_append_equals_full_recompute():
    orc = _micro_oracle(1)
    _prefill(orc, [0], 3, [2])
    out = orc.decode([0], _uniforms(1), 1.0)
    a7 = int(out["tokens"][0, 6])
    vis2 = [I.normal_bf16((2, MICRO.d_model), 9, 77, 1.0)]
    orc.prefill([0], vis2, [[5]])
    e = orc.envs[0]
    assert e.pending is None and e.length == 3 + 2 + 6 + 1 + 2 + 1
    # the next-turn chunk starts with the pending 7th token of the previous turn
    assert torch.equal(e.rows[11], orc.W.embed_rows([a7])[0])
    h = orc.recompute_last_hidden(0)
    assert torch.max(torch.abs(h - e.h_last_prefill)).item() < 1e-12


def test_batch_invariance_bit_identical():
    big = _micro_oracle(3)
    _prefill(big, [0, 1, 2], 3, [1, 4, 2])
    out_big = big.decode([0, 1, 2], _uniforms(3), 1.0)
    solo = _micro_oracle(3)
    vis = [I.normal_bf16((3, MICRO.d_model), 21, 101, 1.0)]
    ids = [I.randint_i32((4,), 21, 201, 0, MICRO.vocab - MICRO.n_bins - 1).tolist()]
    solo.prefill([1], vis, ids)
    out_solo = solo.decode([1], _uniforms(3)[1:2], 1.0)
    for k in ("tokens", "logprobs", "logits", "actions"):
        assert np.array_equal(out_big[k][1], out_solo[k][0]), k


def test_score_equals_decode_logprobs():
    orc = _micro_oracle(2)
    _prefill(orc, [0, 1], 3, [3, 1])
    out = orc.decode([0, 1], _uniforms(2), 1.5)
    sc = orc.score([0, 1], torch.as_tensor(out["tokens"]), 1.5)
    assert np.max(np.abs(sc["logprobs"] - out["logprobs"])) < 1e-12
    assert np.max(np.abs(sc["logits"] - out["logits"])) < 1e-12


def test_forced_decode_feeds_given_tokens():
    orc = _micro_oracle(1)
    _prefill(orc, [0], 3, [2])
    V, nb = MICRO.vocab, MICRO.n_bins
    forced = torch.tensor([[V - nb + k for k in (3, 250, 17, 0, 255, 128, 64)]])
    out = orc.decode([0], _uniforms(1), 1.0, forced=forced)
    sc = orc.score([0], forced, 1.0)
    assert np.max(np.abs(sc["logprobs"][0] - out["logprobs"][0])) < 1e-12
    assert orc.envs[0].pending == int(forced[0, 6])


# ============================================================================ head
def test_head_closed_form_logprobs():
    nb = 256
    z = torch.log(torch.arange(1, nb + 1, dtype=torch.float64))
    _, lp, _ = O.sample_bins(z, 1.0, None)
    total = nb * (nb + 1) // 2                       # sum of (k + 1) = 32896
    expect = torch.log(torch.arange(1, nb + 1, dtype=torch.float64) / total)
    assert torch.allclose(lp, expect, rtol=0, atol=1e-13)
    _, lp2, _ = O.sample_bins(z, 2.0, None)          # p_k proportional to sqrt(k + 1)
    s = math.fsum(math.sqrt(k + 1) for k in range(nb))
    expect2 = torch.tensor([0.5 * math.log(k + 1) - math.log(s) for k in range(nb)],
                           dtype=torch.float64)
    assert torch.allclose(lp2, expect2, rtol=0, atol=1e-13)


def test_softmax_sums_to_one_and_nonpositive():
    g = torch.Generator().manual_seed(3)
    for T in (0.0, 0.5, 1.0, 1.5):
        z = torch.randn(256, generator=g, dtype=torch.float64) * 3
        _, lp, _ = O.sample_bins(z, T, None)
        assert abs(float(torch.exp(lp).sum()) - 1.0) < 1e-12
        assert float(lp.max()) <= 0.0


def test_temperature_to_zero_is_argmax_and_ties_lowest():
    g = torch.Generator().manual_seed(4)
    z = torch.randn(256, generator=g, dtype=torch.float64)
    u = I.uniform_f32((256,), 3, 3)
    k_greedy, lp0, _ = O.sample_bins(z, 0.0, u)
    assert k_greedy == int(torch.argmax(z))
    k_cold, _, _ = O.sample_bins(z, 1e-6, u)
    assert k_cold == k_greedy
    # T = 0 log-probs are those of T = 1
    _, lp1, _ = O.sample_bins(z, 1.0, None)
    assert torch.equal(lp0, lp1)
    ztie = torch.zeros(256, dtype=torch.float64)
    ztie[[9, 40, 200]] = 1.0
    assert O.sample_bins(ztie, 0.0, None)[0] == 9
    # equal uniforms -> equal Gumbel noise -> the draw is argmax z
    assert O.sample_bins(z, 1.0, torch.full((256,), 0.3))[0] == k_greedy


def test_gumbel_max_matches_softmax_chi_square():
    scipy_stats = pytest.importorskip("scipy.stats")
    nb, n = 256, 100_000
    g = torch.Generator().manual_seed(5)
    z = torch.randn(nb, generator=g, dtype=torch.float64) * 1.2
    rng = np.random.default_rng(12345)
    for T in (1.0, 1.5):
        u = torch.from_numpy(rng.random((n, nb)))
        gz = O.gumbel(u)
        s = (z / T)[None, :] + gz
        ks = torch.argmax(s, dim=1).numpy()
        counts = np.bincount(ks, minlength=nb)
        p = torch.softmax(z / T, 0).numpy()
        # merge sparse bins so every expected count is >= 5
        order = np.argsort(p)
        exp_c, obs_c, acc_e, acc_o = [], [], 0.0, 0
        for i in order:
            acc_e += p[i] * n
            acc_o += counts[i]
            if acc_e >= 5:
                exp_c.append(acc_e)
                obs_c.append(acc_o)
                acc_e, acc_o = 0.0, 0
        if acc_e > 0:
            exp_c[-1] += acc_e
            obs_c[-1] += acc_o
        chi2 = float(np.sum((np.array(obs_c) - np.array(exp_c)) ** 2 / np.array(exp_c)))
        pval = scipy_stats.chi2.sf(chi2, len(exp_c) - 1)
        assert pval > 1e-3, (T, chi2, pval)
        # and the oracle's own per-draw sampler agrees with the vectorised argmax
        for r in range(50):
            assert O.sample_bins(z, T, u[r])[0] == int(ks[r])


def test_bin_centres_golden_and_exact_fp32():
    _, rows = read_fixture("action_bins.txt")
    for k, c in rows:
        assert O.bin_centre(int(k)) == c
    cs = [O.bin_centre(k) for k in range(256)]
    assert cs[0] == -1 + 1 / 256 and cs[255] == 1 - 1 / 256
    for k in range(256):
        assert float(np.float32(cs[k])) == cs[k]          # exactly representable
        assert cs[k] == -cs[255 - k]
        if k:
            assert cs[k] - cs[k - 1] == 2 / 256


def test_head_token_and_action_mapping():
    w = micro_weights()
    Wt = O.Weights(MICRO, w)
    h = O.f64(micro_rows(1)[0])
    ho = O.action_head(MICRO, Wt, h, 1.0, I.uniform_f32((256,), 1, 1))
    assert ho.token == MICRO.vocab - 256 + ho.k
    assert ho.action == -1 + (2 * ho.k + 1) / 256


def test_reset_env_restarts_like_a_fresh_env():
    """An env reset at an episode end (Algorithm 1 terminal flags) and prefilled again gives the
    same decode, bit for bit, as a never-used env given the same prefix."""
    orc = _micro_oracle(2)
    _prefill(orc, [0, 1], 3, [2, 4])
    orc.decode([0, 1], _uniforms(2), 1.0)
    orc.reset([0])
    fresh = _micro_oracle(1)
    _prefill(orc, [0], 5, [3])
    _prefill(fresh, [0], 5, [3])
    a = orc.decode([0], _uniforms(1), 1.5)
    b = fresh.decode([0], _uniforms(1), 1.5)
    assert np.array_equal(a["logits"], b["logits"]) and np.array_equal(a["tokens"], b["tokens"])


# ============================================================================ entropy, value, GAE, PPO
def test_entropy_closed_forms():
    """Rollout entropy (§4.2): uniform logits give log 256 at any T; a two-level z has the closed
    form -p1 log p1 - 255 p0 log p0; H(z, T) = H(z / T, 1); 0 <= H <= log 256."""
    z0 = torch.zeros(256, dtype=torch.float64)
    for T in (0.0, 0.5, 1.0, 1.5):
        assert abs(O.token_entropy(z0, T) - math.log(256.0)) < 1e-12
    a = 3.0
    z = torch.zeros(256, dtype=torch.float64)
    z[17] = a
    p1 = math.exp(a) / (math.exp(a) + 255.0)
    p0 = 1.0 / (math.exp(a) + 255.0)
    want = -p1 * math.log(p1) - 255.0 * p0 * math.log(p0)
    assert abs(O.token_entropy(z, 1.0) - want) < 1e-12
    g = torch.Generator().manual_seed(5)
    zr = torch.randn(256, generator=g, dtype=torch.float64) * 4.0
    for T in (0.5, 1.5):
        assert abs(O.token_entropy(zr, T) - O.token_entropy(zr / T, 1.0)) < 1e-12
        h = O.token_entropy(zr, T)
        assert 0.0 <= h <= math.log(256.0) + 1e-12
    z[17] = 1e4
    assert O.token_entropy(z, 1.0) < 1e-12


def test_value_head_closed_form():
    """V = RMSNorm(h_last) . w_value + b: a constant hidden row c normalises to sign(c) times
    the final-norm gains, so V = sign(c) * sum(g * w) + b; V is affine in (w, b)."""
    d = 8
    sh = O.Shape(1, d, 2, 4, 16, 300)
    g = torch.tensor([1.0, 0.5, 2.0, 1.0, 1.0, 0.25, 1.0, 1.0], dtype=torch.float64)
    W = types.SimpleNamespace(final_norm=g)
    w = torch.tensor([0.5, -1.0, 0.25, 2.0, 0.0, 4.0, -0.5, 1.0], dtype=torch.float64)
    for c in (3.0, -0.75):
        h = torch.full((d,), c, dtype=torch.float64)
        want = math.copysign(1.0, c) * float((g * w).sum()) / math.sqrt(1.0 + sh.rms_eps / c ** 2) + 0.125
        assert abs(O.value_head(sh, W, h, w, 0.125) - want) < 1e-12
    h = torch.randn(d, generator=torch.Generator().manual_seed(3), dtype=torch.float64)
    v1, v2 = O.value_head(sh, W, h, w, 0.0), O.value_head(sh, W, h, 2.0 * w, 0.0)
    assert abs(v2 - 2.0 * v1) < 1e-12
    assert abs(O.value_head(sh, W, h, w, 1.5) - v1 - 1.5) < 1e-12


def _golden_rows(name):
    rows = []
    for line in open(os.path.join(GOLDEN, name)):
        line = line.strip()
        if line and not line.startswith("#"):
            rows.append(line.split())
    return rows


def test_gae_golden_fixture():
    rows = _golden_rows("gae_m3.txt")
    r = [[float(x[1])] for x in rows[:3]]
    v = [[float(x[2])] for x in rows[:4]]
    dn = [[float(x[3])] for x in rows[:3]]
    adv, ret = O.gae(r, v, dn, 0.5, 0.5)
    for t in range(3):
        assert float(adv[t, 0]) == float(rows[t][4])
        assert float(ret[t, 0]) == float(rows[t][5])


def test_gae_special_cases():
    """lambda = 1, no terminal: A_t = sum_k gamma^k r_{t+k} + gamma^(M-t) V_M - V_t (discounted
    return minus value); lambda = 0: A_t is the one-step TD error; a terminal at t makes
    A_t = r_t - V_t; envs are independent columns."""
    g = torch.Generator().manual_seed(11)
    M, B, gam = 6, 3, 0.9
    r = torch.randn(M, B, generator=g, dtype=torch.float64)
    v = torch.randn(M + 1, B, generator=g, dtype=torch.float64)
    zero = torch.zeros(M, B, dtype=torch.float64)
    adv, _ = O.gae(r, v, zero, gam, 1.0)
    for t in range(M):
        ret = sum(gam ** k * r[t + k] for k in range(M - t)) + gam ** (M - t) * v[M]
        assert torch.allclose(adv[t], ret - v[t], atol=1e-12)
    adv0, _ = O.gae(r, v, zero, gam, 0.0)
    assert torch.allclose(adv0, r + gam * v[1:] - v[:M], atol=1e-12)
    dn = zero.clone()
    dn[2, 1] = 1.0
    adv2, _ = O.gae(r, v, dn, gam, 0.95)
    assert abs(float(adv2[2, 1]) - float(r[2, 1] - v[2, 1])) < 1e-12
    assert torch.allclose(adv2[:, 0], O.gae(r[:, :1], v[:, :1], zero[:, :1], gam, 0.95)[0][:, 0], atol=1e-12)


def test_ppo_clip_golden_fixture():
    rows = _golden_rows("ppo_clip_eps02.txt")
    rho = [float(x[0]) for x in rows]
    adv = [float(x[1]) for x in rows]
    lp_old = torch.full((4, 7), -1.25, dtype=torch.float64)
    lp_new = lp_old + torch.tensor([math.log(x) / 7.0 for x in rho], dtype=torch.float64)[:, None]
    obj, rr, frac = O.ppo_clip_objective(lp_new, lp_old, adv, 0.2)
    assert abs(obj - 0.725) < 1e-12
    assert abs(frac - 0.75) < 1e-12
    assert torch.allclose(rr, torch.tensor(rho, dtype=torch.float64), atol=1e-12)


def test_ppo_clip_unclipped_equals_ratio_times_advantage():
    """Inside the trust region the objective is the plain importance-weighted advantage, and at
    rho = 1 it is mean(A)."""
    g = torch.Generator().manual_seed(2)
    lp_old = -torch.rand(10, 7, generator=g, dtype=torch.float64) * 3.0
    adv = torch.randn(10, generator=g, dtype=torch.float64)
    obj, _, frac = O.ppo_clip_objective(lp_old, lp_old, adv, 0.2)
    assert abs(obj - float(adv.mean())) < 1e-12 and frac == 0.0
    lp_new = lp_old + 0.01 / 7.0
    obj2, rho, _ = O.ppo_clip_objective(lp_new, lp_old, adv, 0.2)
    assert abs(obj2 - float((rho * adv).mean())) < 1e-12


def test_decode_and_score_report_entropy_of_their_logits():
    orc = _micro_oracle(1)
    _prefill(orc, [0], 3, [2])
    out = orc.decode([0], _uniforms(1), 1.5)
    sc = orc.score([0], torch.tensor(out["tokens"]), 1.5)
    for i in range(MICRO.action_dim):
        z = torch.tensor(out["logits"][0, i], dtype=torch.float64)
        assert abs(out["entropy"][0, i] - O.token_entropy(z, 1.5)) < 1e-12
        assert abs(sc["entropy"][0, i] - out["entropy"][0, i]) < 1e-12


# ============================================================================ mutations
def _bruteforce_gap():
    w = micro_weights()
    Wt = O.Weights(MICRO, w)
    x = micro_rows(5)
    ours = O.full_forward(MICRO, Wt, O.f64(x))
    ref = BF.decoder(x.double().tolist(), as_lists(w), MICRO.n_layers, MICRO.n_heads,
                     MICRO.head_dim, MICRO.d_ffn, MICRO.rms_eps, MICRO.rope_theta)
    return float(np.max(np.abs(ours.numpy() - np.array(ref))))


def test_mutation_rope_sign_is_caught(monkeypatch):
    def bad_rope(x, pos, theta):
        half = x.shape[-1] // 2
        c, s = O.rope_cos_sin(pos, x.shape[-1], theta)
        c, s = c[:, None, :], s[:, None, :]
        x1, x2 = x[..., :half], x[..., half:]
        return torch.cat([x1 * c + x2 * s, x2 * c - x1 * s], dim=-1)
    monkeypatch.setattr(O, "apply_rope", bad_rope)
    assert _bruteforce_gap() > 1e-6


def test_mutation_attention_scale_is_caught(monkeypatch):
    orig = O.causal_attention
    monkeypatch.setattr(O, "causal_attention",
                        lambda q, k, v, qp, kp: orig(q * math.sqrt(q.shape[-1]), k, v, qp, kp))
    assert _bruteforce_gap() > 1e-6


def test_mutation_transposed_wo_is_caught(monkeypatch):
    orig = O.Weights.layer
    def layer(self, l):
        lw = dict(orig(self, l))
        lw["wo"] = lw["wo"].T.contiguous()
        return lw
    monkeypatch.setattr(O.Weights, "layer", layer)
    assert _bruteforce_gap() > 1e-6


def test_mutation_dropped_gate_activation_is_caught(monkeypatch):
    monkeypatch.setattr(O, "silu", lambda x: x)
    assert _bruteforce_gap() > 1e-6


def test_mutation_untempered_sampling_is_caught():
    # sampling from softmax(z) instead of softmax(z / T) must fail the frequency test
    scipy_stats = pytest.importorskip("scipy.stats")
    nb, n, T = 256, 50_000, 1.5
    g = torch.Generator().manual_seed(5)
    z = torch.randn(nb, generator=g, dtype=torch.float64) * 1.2
    u = torch.from_numpy(np.random.default_rng(7).random((n, nb)))
    ks = torch.argmax(z[None, :] + O.gumbel(u), dim=1).numpy()   # planted: T dropped
    counts = np.bincount(ks, minlength=nb)
    p = torch.softmax(z / T, 0).numpy()
    mask = p * n >= 5
    chi2 = float(np.sum((counts[mask] - p[mask] * n) ** 2 / (p[mask] * n)))
    assert scipy_stats.chi2.sf(chi2, int(mask.sum()) - 1) < 1e-6


def test_mutation_gae_without_terminal_mask_is_caught(monkeypatch):
    good = O.gae

    def bad_gae(rewards, values, dones, gamma, lam):
        return good(rewards, values, torch.zeros_like(torch.as_tensor(dones, dtype=torch.float64)), gamma, lam)
    monkeypatch.setattr(O, "gae", bad_gae)
    with pytest.raises(AssertionError):
        test_gae_golden_fixture()


def test_mutation_ppo_max_instead_of_min_is_caught(monkeypatch):
    def bad(lp_new, lp_old, adv, eps):
        ln = torch.as_tensor(lp_new, dtype=torch.float64).sum(-1)
        lo = torch.as_tensor(lp_old, dtype=torch.float64).sum(-1)
        a = torch.as_tensor(adv, dtype=torch.float64)
        rho = torch.exp(ln - lo)
        obj = torch.maximum(rho * a, torch.clamp(rho, 1 - eps, 1 + eps) * a)
        return float(obj.mean()), rho, float(((rho - 1).abs() > eps).to(torch.float64).mean())
    monkeypatch.setattr(O, "ppo_clip_objective", bad)
    with pytest.raises(AssertionError):
        test_ppo_clip_golden_fixture()
