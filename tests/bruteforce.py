"""Brute-force pure-Python restatement of the policy decoder, for tiny shapes only.

Written separately from the oracle (lists, loops and the `math` module, no torch, no
numpy) so that it can pin the oracle: the same Llama-2-style layer (paper §3.1) with
RMSNorm, rotate-half RoPE, causal softmax attention, SwiGLU FFN, then the 256-bin action
head.  Every row is recomputed from scratch for every position (no KV cache).
"""
import math


def rmsnorm(x, w, eps):
    ms = 0.0
    for v in x:
        ms += v * v
    ms /= len(x)
    r = 1.0 / math.sqrt(ms + eps)
    return [x[i] * r * w[i] for i in range(len(x))]


def matvec(W, x):
    """W as list of rows [out][in]."""
    out = []
    for row in W:
        acc = 0.0
        for i in range(len(x)):
            acc += row[i] * x[i]
        out.append(acc)
    return out


def rope(vec, pos, theta):
    hd = len(vec)
    half = hd // 2
    out = [0.0] * hd
    for i in range(half):
        ang = pos * theta ** (-2.0 * i / hd)
        c, s = math.cos(ang), math.sin(ang)
        a, b = vec[i], vec[i + half]
        out[i] = a * c - b * s
        out[i + half] = b * c + a * s
    return out


def decoder(rows, W, n_layers, n_heads, head_dim, d_ffn, eps, theta):
    """rows: list of input vectors at positions 0..n-1; W: dict of nested lists.

    Returns the final-layer hidden of every row.
    """
    n = len(rows)
    d = len(rows[0])
    h = [list(r) for r in rows]
    for l in range(n_layers):
        q_all, k_all, v_all = [], [], []
        for t in range(n):
            y = rmsnorm(h[t], W["attn_norm"][l], eps)
            qkv = matvec(W["wqkv"][l], y)
            q, k, v = qkv[0:d], qkv[d:2 * d], qkv[2 * d:3 * d]
            qh, kh, vh = [], [], []
            for hh in range(n_heads):
                sl = slice(hh * head_dim, (hh + 1) * head_dim)
                qh.append(rope(q[sl], t, theta))
                kh.append(rope(k[sl], t, theta))
                vh.append(v[sl])
            q_all.append(qh)
            k_all.append(kh)
            v_all.append(vh)
        new_h = []
        for t in range(n):
            o = []
            for hh in range(n_heads):
                scores = []
                for j in range(t + 1):
                    s = 0.0
                    for i in range(head_dim):
                        s += q_all[t][hh][i] * k_all[j][hh][i]
                    scores.append(s / math.sqrt(head_dim))
                m = max(scores)
                e = [math.exp(s - m) for s in scores]
                z = sum(e)
                for i in range(head_dim):
                    acc = 0.0
                    for j in range(t + 1):
                        acc += e[j] / z * v_all[j][hh][i]
                    o.append(acc)
            attn = matvec(W["wo"][l], o)
            x = [h[t][i] + attn[i] for i in range(d)]
            y = rmsnorm(x, W["ffn_norm"][l], eps)
            gu = matvec(W["w_gate_up"][l], y)
            act = []
            for i in range(d_ffn):
                g, u = gu[i], gu[d_ffn + i]
                act.append(g / (1.0 + math.exp(-g)) * u)
            down = matvec(W["w_down"][l], act)
            new_h.append([x[i] + down[i] for i in range(d)])
        h = new_h
    return h


def head(h_last, final_norm, lm_head_rows, eps, temperature):
    """Logits over the action bins and their log-softmax at temperature T."""
    y = rmsnorm(h_last, final_norm, eps)
    z = matvec(lm_head_rows, y)
    zt = [v / temperature for v in z]
    m = max(zt)
    lse = m + math.log(sum(math.exp(v - m) for v in zt))
    return z, [v - lse for v in zt]
