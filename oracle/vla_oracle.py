"""Plain fp64 CPU oracle of the VLA-RL rollout / re-scoring hot path.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import or call this module;
only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` do.
It shares no code with the CUDA library.

What it computes, in the order the paper gives it:

* The policy π_θ is an auto-regressive Llama-2-style decoder (paper §3.1: OpenVLA-7B,
  whose core is Llama-2-7B).  A rollout step feeds the state (image tokens from the
  vision-text processor h(o_t), then the instruction v_t^in) and the policy generates the
  action token sequence v_t^out, n = |A| = 7 tokens (Algorithm 1, rollout phase; §3.3).
* Each action token stands for one discretised bin of one action dimension (§3.1);
  a_t = f(v_t^out) maps the bins back to continuous values.
* log π(a_t | o_t, v_t^in) = Σ_i log π(v_out,i | ·) (Eq. 1), the quantity the PPO ratio
  of Eq. 2 re-computes in the learning phase.
* The trajectory is a multi-turn conversation (§3.3): every step appends to the same
  context.

Precision: everything in fp64, weights decoded exactly from their bf16 bits.  Each
environment is processed on its own (that is the definition of batch invariance the
paper's large-batch remark in §3.5 asks for).

Readings where the paper is silent (listed in the design notes with their reasons):
action ids are the last 256 vocabulary ids in ascending bin order; bin k maps to the
centre -1 + (2k+1)/256; sampling is restricted to the 256 bins; the log-prob is that of
the tempered 256-way softmax; T = 0 means greedy with T = 1 log-probs; ties go to the
lowest bin; Gumbel-max with caller-supplied uniforms u (clamped to [2^-24, 1-2^-24], the fp32-representable ends of (0,1));
RoPE is the rotate-half form with theta = 1e4; RMSNorm eps = 1e-6; the 7th action token's
KV is written as the first row of the next turn's chunk.

Pins (tests/test_oracle_pins.py): closed forms for RMSNorm, RoPE, SiLU and the head,
brute-force pure-Python decoder on tiny inputs, KV-cached decode == full recompute, the
softmax summing to 1, T -> 0 == argmax, a chi-square test of the sampler, bin centres.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Dict, List, Optional, Sequence

import numpy as np
import torch

F64 = torch.float64
U_MIN = 2.0 ** -24
U_MAX = 1.0 - 2.0 ** -24


@dataclass(frozen=True)
class Shape:
    n_layers: int
    d_model: int
    n_heads: int
    head_dim: int
    d_ffn: int
    vocab: int
    n_bins: int = 256
    action_dim: int = 7
    rms_eps: float = 1e-6
    rope_theta: float = 1e4


def shape_from(obj) -> Shape:
    return Shape(obj.n_layers, obj.d_model, obj.n_heads, obj.head_dim, obj.d_ffn, obj.vocab,
                 obj.n_bins, obj.action_dim, obj.rms_eps, obj.rope_theta)


def f64(t: torch.Tensor) -> torch.Tensor:
    """bf16 / fp32 -> fp64 (exact)."""
    return t.to(F64)


# =========================================================================== layers
def rms_norm(x: torch.Tensor, w: torch.Tensor, eps: float) -> torch.Tensor:
    """RMSNorm of the Llama-2 backbone (§3.1): x / sqrt(mean(x^2) + eps) * w."""
    return x / torch.sqrt((x * x).mean(dim=-1, keepdim=True) + eps) * w


def rope_cos_sin(pos: torch.Tensor, head_dim: int, theta: float):
    """Rotary angles pos * theta^(-2i/hd), i = 0 .. hd/2-1 (Llama-2 backbone, §3.1)."""
    i = torch.arange(head_dim // 2, dtype=F64)
    inv_freq = theta ** (-2.0 * i / head_dim)
    ang = pos.to(F64)[:, None] * inv_freq[None, :]
    return torch.cos(ang), torch.sin(ang)


def apply_rope(x: torch.Tensor, pos: torch.Tensor, theta: float) -> torch.Tensor:
    """Rotate-half RoPE on x [n, H, hd]: pair (i, i + hd/2) rotated by angle pos*w_i."""
    hd = x.shape[-1]
    half = hd // 2
    c, s = rope_cos_sin(pos, hd, theta)
    c, s = c[:, None, :], s[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return torch.cat([x1 * c - x2 * s, x2 * c + x1 * s], dim=-1)


def causal_attention(q, k, v, q_pos, k_pos):
    """softmax(q k^T / sqrt(hd) + causal mask) v, per head.

    q [n, H, hd] at absolute positions q_pos [n]; k, v [m, H, hd] at k_pos [m].
    Key j is visible to query i iff k_pos[j] <= q_pos[i].
    """
    hd = q.shape[-1]
    scores = torch.einsum("nhd,mhd->hnm", q, k) / math.sqrt(hd)
    hidden = k_pos[None, :] > q_pos[:, None]
    scores = scores.masked_fill(hidden[None, :, :], float("-inf"))
    p = torch.softmax(scores, dim=-1)
    return torch.einsum("hnm,mhd->nhd", p, v)


def silu(x: torch.Tensor) -> torch.Tensor:
    return x / (1.0 + torch.exp(-x))


# =========================================================================== weights
class Weights:
    """bf16 CPU weights with fp64 views per layer (cached when `cache_f64`)."""

    def __init__(self, shape: Shape, w: Dict[str, torch.Tensor], cache_f64: bool = True):
        self.shape = shape
        self.w = w
        self.cache_f64 = cache_f64
        self._cache: Dict[int, dict] = {}
        V, nb = shape.vocab, shape.n_bins
        self.final_norm = f64(w["final_norm"])
        self.head_rows = f64(w["lm_head"][V - nb:V])       # only the 256 action-bin rows

    def embed_rows(self, ids: Sequence[int]) -> torch.Tensor:
        return f64(self.w["embed"][torch.as_tensor(list(ids), dtype=torch.long)])

    def layer(self, l: int) -> dict:
        if l in self._cache:
            return self._cache[l]
        w = self.w
        lw = {
            "attn_norm": f64(w["attn_norm"][l]),
            "wqkv": f64(w["wqkv"][l]),
            "wo": f64(w["wo"][l]),
            "ffn_norm": f64(w["ffn_norm"][l]),
            "w_gate_up": f64(w["w_gate_up"][l]),
            "w_down": f64(w["w_down"][l]),
        }
        if self.cache_f64:
            self._cache[l] = lw
        return lw


def layer_forward(shape: Shape, lw: dict, h, pos, k_cache, v_cache):
    """One decoder layer over the chunk rows h [n, d] at positions pos [n].

    k_cache / v_cache: [m, H, hd] post-RoPE keys / values already in the context
    (positions 0 .. m-1); returns (h_out, k_all, v_all) with the chunk appended.
    """
    n = h.shape[0]
    d, H, hd, F = shape.d_model, shape.n_heads, shape.head_dim, shape.d_ffn
    y = rms_norm(h, lw["attn_norm"], shape.rms_eps)
    qkv = y @ lw["wqkv"].T
    q = qkv[:, 0:d].reshape(n, H, hd)
    k = qkv[:, d:2 * d].reshape(n, H, hd)
    v = qkv[:, 2 * d:3 * d].reshape(n, H, hd)
    q = apply_rope(q, pos, shape.rope_theta)
    k = apply_rope(k, pos, shape.rope_theta)
    k_all = torch.cat([k_cache, k], dim=0)
    v_all = torch.cat([v_cache, v], dim=0)
    k_pos = torch.arange(k_all.shape[0], dtype=torch.long)
    o = causal_attention(q, k_all, v_all, pos, k_pos)
    h = h + o.reshape(n, d) @ lw["wo"].T
    y = rms_norm(h, lw["ffn_norm"], shape.rms_eps)
    gu = y @ lw["w_gate_up"].T
    h = h + (silu(gu[:, :F]) * gu[:, F:]) @ lw["w_down"].T
    return h, k_all, v_all


# =========================================================================== action head
@dataclass
class HeadOut:
    logits: torch.Tensor      # fp64 [256]
    k: int                    # sampled bin
    token: int                # vocab id
    action: float             # bin centre
    logprobs: torch.Tensor    # fp64 [256] log softmax(z / T)   (T = 0: T = 1 values)
    margin: float             # top-1 minus top-2 of the perturbed score s
    entropy: float = 0.0      # -sum_k p_k log p_k of the same distribution


def bin_centre(k: int, n_bins: int = 256) -> float:
    """a = f(v_out): bin k -> centre of the k-th of n_bins equal cells of [-1, 1]."""
    return -1.0 + (2.0 * k + 1.0) / n_bins


def gumbel(u: torch.Tensor) -> torch.Tensor:
    u = u.to(F64).clamp(U_MIN, U_MAX)
    return -torch.log(-torch.log(u))


def head_logits(shape: Shape, W: Weights, h_last: torch.Tensor) -> torch.Tensor:
    """Final RMSNorm then the 256 action-bin logits z_k = y . lm_head[V-256+k] (§3.1)."""
    y = rms_norm(h_last, W.final_norm, shape.rms_eps)
    return W.head_rows @ y


def sample_bins(z: torch.Tensor, temperature: float, u: Optional[torch.Tensor]):
    """Temperature sampling over the bins and the per-token log-probs of Eq. 1.

    T > 0: Gumbel-max draw k = argmax_k (z_k / T + g_k), g_k = -log(-log u_k), which is an
    exact sample of softmax(z / T) (Gumbel 1954; the Gumbel-max trick).  T = 0: k = argmax z
    and the log-probs are those of T = 1.  Ties -> lowest k.  u = None: no draw, s = z/T.
    Returns (k, log softmax(z/T) [n_bins], margin of the top two of s).
    """
    if temperature > 0.0:
        zt = z / temperature
        s = zt + gumbel(u) if u is not None else zt
    else:
        zt = z
        s = z
    s_np = s.numpy()
    k = int(np.argmax(s_np))                     # first maximal index = lowest k on ties
    srt = np.sort(s_np)
    margin = float(srt[-1] - srt[-2])
    lp = zt - torch.logsumexp(zt, dim=0)
    return k, lp, margin


def token_entropy(z: torch.Tensor, temperature: float) -> float:
    """Entropy of one action token's distribution over the bins (the rollout entropy the
    paper tracks in its training dynamics, §4.2): H = -sum_k p_k log p_k with p = softmax(z/T),
    the distribution the sampler draws from; T = 0 uses T = 1, as the log-probs do."""
    zt = z / temperature if temperature > 0.0 else z
    lp = zt - torch.logsumexp(zt, dim=0)
    return float(-(torch.exp(lp) * lp).sum())


def action_head(shape: Shape, W: Weights, h_last: torch.Tensor, temperature: float,
                u: Optional[torch.Tensor]) -> HeadOut:
    """Logits, sample, log-probs and the de-tokenised action for one hidden state."""
    z = head_logits(shape, W, h_last)
    k, lp, margin = sample_bins(z, temperature, u)
    return HeadOut(z, k, shape.vocab - shape.n_bins + k, bin_centre(k, shape.n_bins), lp, margin,
                   token_entropy(z, temperature))


# =========================================================================== value head
def value_head(shape: Shape, W: Weights, h_last: torch.Tensor, w_value: torch.Tensor,
               bias: float) -> float:
    """V(o_t, v_t^in) of Algorithm 1 ("value model estimates") for a homogeneous value model
    (§3.2 / the pipeline figure: the same decoder as the policy): the final RMSNorm of the
    last prefix row, then one linear output, V = y . w_value + bias."""
    y = rms_norm(h_last, W.final_norm, shape.rms_eps)
    return float(y @ f64(w_value)) + float(bias)


# =========================================================================== learning phase
def gae(rewards, values, dones, gamma: float, lam: float):
    """Generalised advantage estimation (Algorithm 1, "compute advantages"; §3.3 cites
    Schulman et al. 2015) over M steps of B envs, walking t = M-1 .. 0:

      delta_t = r_t + gamma * (1 - done_t) * V_{t+1} - V_t
      A_t     = delta_t + gamma * lam * (1 - done_t) * A_{t+1},   A_M = 0
      R_t     = A_t + V_t                        (the value model's regression target)

    rewards [M, B]; values [M + 1, B] = V_0 .. V_M (V_M bootstraps the unfinished tail);
    dones [M, B]: 1 where the episode ended with step t (then nothing past t is used).
    Returns (A [M, B], R [M, B]) in fp64."""
    r = torch.as_tensor(rewards, dtype=F64)
    v = torch.as_tensor(values, dtype=F64)
    d = torch.as_tensor(dones, dtype=F64)
    M = r.shape[0]
    adv = torch.zeros_like(r)
    nxt = torch.zeros_like(r[0])
    for t in range(M - 1, -1, -1):
        live = 1.0 - d[t]
        delta = r[t] + gamma * live * v[t + 1] - v[t]
        nxt = delta + gamma * lam * live * nxt
        adv[t] = nxt
    return adv, adv + v[:M]


def ppo_clip_objective(lp_new, lp_old, adv, eps: float):
    """The clipped PPO objective of Eq. 2 over N samples (env-steps):

      log pi(a_t | .) = sum_i log pi(v_out,t,i | .)        (Eq. 1: the 7 token log-probs)
      rho_t = exp(log pi_theta(a_t | .) - log pi_theta_old(a_t | .))
      L     = mean_t min(rho_t A_t, clip(rho_t, 1 - eps, 1 + eps) A_t)

    lp_new, lp_old [N, A] token log-probs; adv [N].  Returns (L, rho [N], fraction of samples
    with |rho - 1| > eps) in fp64.  L is the objective to maximise; a loss is -L."""
    ln = torch.as_tensor(lp_new, dtype=F64).sum(dim=-1)
    lo = torch.as_tensor(lp_old, dtype=F64).sum(dim=-1)
    a = torch.as_tensor(adv, dtype=F64)
    rho = torch.exp(ln - lo)
    obj = torch.minimum(rho * a, torch.clamp(rho, 1.0 - eps, 1.0 + eps) * a)
    clipped = ((rho - 1.0).abs() > eps).to(F64)
    return float(obj.mean()), rho, float(clipped.mean())


# =========================================================================== engine
@dataclass
class EnvState:
    k: List[torch.Tensor] = field(default_factory=list)   # per layer [len, H, hd]
    v: List[torch.Tensor] = field(default_factory=list)
    rows: List[torch.Tensor] = field(default_factory=list)  # input rows (fp64 [d]) in order
    length: int = 0
    len_prefill: int = 0           # context length right after the latest prefill
    h_last_prefill: Optional[torch.Tensor] = None
    pending: Optional[int] = None  # 7th action token of the latest turn, KV not yet written


class Oracle:
    """Per-environment fp64 rollout engine with the C-ABI's call semantics.

    prefill  : chunk = [pending a7] + visual rows + text ids, appended to the context.
    decode   : 7 action tokens from the latest prefill; tokens 2..7 each need one
               KV-cached decoder forward of the previous token; a7 stays pending.
    score    : teacher-forced log-probs of given tokens for the latest turn (the PPO ratio
               pass of Eq. 2); the turn's actions become the given tokens.
    """

    def __init__(self, shape: Shape, weights: Dict[str, torch.Tensor], n_envs: int,
                 cache_f64: bool = True):
        self.shape = shape
        self.W = Weights(shape, weights, cache_f64)
        self.envs = [self._fresh() for _ in range(n_envs)]

    def _fresh(self) -> EnvState:
        sh = self.shape
        e = EnvState()
        e.k = [torch.zeros(0, sh.n_heads, sh.head_dim, dtype=F64) for _ in range(sh.n_layers)]
        e.v = [torch.zeros(0, sh.n_heads, sh.head_dim, dtype=F64) for _ in range(sh.n_layers)]
        return e

    def reset(self, envs: Optional[Sequence[int]] = None):
        for b in (range(len(self.envs)) if envs is None else envs):
            self.envs[b] = self._fresh()

    # ------------------------------------------------------------------ forward
    def _layer(self, lw: dict, h, pos, k_cache, v_cache):
        """One decoder layer (layer_forward); the single place the engine calls it."""
        return layer_forward(self.shape, lw, h, pos, k_cache, v_cache)

    def _forward(self, env_ids: Sequence[int], chunks: Sequence[torch.Tensor]):
        """Run chunk rows [n_b, d] of each env through all layers; append KV; return h."""
        sh = self.shape
        hs, poss = [], []
        for b, x in zip(env_ids, chunks):
            e = self.envs[b]
            hs.append(x.clone())
            poss.append(torch.arange(e.length, e.length + x.shape[0], dtype=torch.long))
        for l in range(sh.n_layers):
            lw = self.W.layer(l)
            for j, b in enumerate(env_ids):
                e = self.envs[b]
                hs[j], e.k[l], e.v[l] = self._layer(lw, hs[j], poss[j], e.k[l], e.v[l])
        for b, x in zip(env_ids, chunks):
            e = self.envs[b]
            e.rows.extend(list(x))
            e.length += x.shape[0]
        return hs

    def _truncate(self, b: int, length: int):
        e = self.envs[b]
        for l in range(self.shape.n_layers):
            e.k[l] = e.k[l][:length]
            e.v[l] = e.v[l][:length]
        e.rows = e.rows[:length]
        e.length = length

    # ------------------------------------------------------------------ API
    def prefill(self, env_ids: Sequence[int], visual: Sequence[torch.Tensor],
                ids: Sequence[Sequence[int]]):
        """visual[j] bf16 [Nv, d], ids[j] list of ints for env env_ids[j]."""
        chunks = []
        for b, vis, tid in zip(env_ids, visual, ids):
            e = self.envs[b]
            parts = []
            if e.pending is not None:
                parts.append(self.W.embed_rows([e.pending]))
            parts.append(f64(vis))
            if len(tid):
                parts.append(self.W.embed_rows(tid))
            chunks.append(torch.cat(parts, dim=0))
        hs = self._forward(env_ids, chunks)
        for b, h in zip(env_ids, hs):
            e = self.envs[b]
            e.pending = None
            e.len_prefill = e.length
            e.h_last_prefill = h[-1].clone()

    def decode(self, env_ids: Sequence[int], uniforms: torch.Tensor, temperature: float,
               forced: Optional[torch.Tensor] = None):
        """uniforms [len(env_ids), 7, 256]; forced [len(env_ids), 7] ints or None.

        Returns dict of tokens/ks/actions/logprob (of the token fed forward)/logits/margins,
        each indexed [j, i].
        """
        sh = self.shape
        A = sh.action_dim
        n = len(env_ids)
        out = {"tokens": np.zeros((n, A), np.int64), "bins": np.zeros((n, A), np.int64),
               "actions": np.zeros((n, A), np.float64), "logprobs": np.zeros((n, A)),
               "sampled_logprobs": np.zeros((n, A)), "logits": np.zeros((n, A, sh.n_bins)),
               "margins": np.zeros((n, A)), "entropy": np.zeros((n, A))}
        for b in env_ids:
            self._truncate(b, self.envs[b].len_prefill)
        h_cur = [self.envs[b].h_last_prefill for b in env_ids]
        fed = [0] * n
        for i in range(A):
            for j, b in enumerate(env_ids):
                ho = action_head(sh, self.W, h_cur[j], temperature, uniforms[j, i])
                tok = ho.token if forced is None else int(forced[j, i])
                kk = tok - (sh.vocab - sh.n_bins)
                out["tokens"][j, i] = ho.token
                out["bins"][j, i] = ho.k
                out["actions"][j, i] = ho.action
                out["sampled_logprobs"][j, i] = float(ho.logprobs[ho.k])
                out["logprobs"][j, i] = float(ho.logprobs[kk])
                out["logits"][j, i] = ho.logits.numpy()
                out["margins"][j, i] = ho.margin
                out["entropy"][j, i] = ho.entropy
                fed[j] = tok
            if i == A - 1:
                break
            chunks = [self.W.embed_rows([fed[j]]) for j in range(n)]
            hs = self._forward(env_ids, chunks)
            h_cur = [h[-1] for h in hs]
        for j, b in enumerate(env_ids):
            self.envs[b].pending = fed[j]
        return out

    def score(self, env_ids: Sequence[int], tokens: torch.Tensor, temperature: float):
        """Teacher-forced log-probs of tokens [len(env_ids), 7] for the latest turn."""
        sh = self.shape
        A = sh.action_dim
        n = len(env_ids)
        for b in env_ids:
            self._truncate(b, self.envs[b].len_prefill)
        chunks = [self.W.embed_rows([int(t) for t in tokens[j, :A - 1]]) for j in range(n)]
        hs = self._forward(env_ids, chunks)
        lp = np.zeros((n, A))
        ent = np.zeros((n, A))
        logits = np.zeros((n, A, sh.n_bins))
        base = sh.vocab - sh.n_bins
        for j, b in enumerate(env_ids):
            hrow = [self.envs[b].h_last_prefill] + [hs[j][i] for i in range(A - 1)]
            for i in range(A):
                ho = action_head(sh, self.W, hrow[i], temperature, None)
                lp[j, i] = float(ho.logprobs[int(tokens[j, i]) - base])
                ent[j, i] = ho.entropy
                logits[j, i] = ho.logits.numpy()
            self.envs[b].pending = int(tokens[j, A - 1])
        return {"logprobs": lp, "logits": logits, "entropy": ent}

    def value(self, env_ids: Sequence[int], w_value: torch.Tensor, bias: float) -> np.ndarray:
        """Value-model estimates at each env's latest prefill (the state of the step)."""
        return np.array([value_head(self.shape, self.W, self.envs[b].h_last_prefill, w_value, bias)
                         for b in env_ids])

    # ------------------------------------------------------------------ full recompute
    def recompute_last_hidden(self, b: int, extra_ids: Sequence[int] = ()) -> torch.Tensor:
        """Final-layer hidden of the last row, recomputing the whole context of env b from
        its input rows (plus `extra_ids` appended) with no KV reuse."""
        e = self.envs[b]
        rows = list(e.rows)
        if len(extra_ids):
            rows += list(self.W.embed_rows(extra_ids))
        x = torch.stack(rows, dim=0)
        return full_forward(self.shape, self.W, x)[-1]


def full_forward(shape: Shape, W: Weights, x: torch.Tensor) -> torch.Tensor:
    """All layers over rows x [n, d] at positions 0..n-1 from an empty context."""
    h = x.clone()
    pos = torch.arange(x.shape[0], dtype=torch.long)
    empty = torch.zeros(0, shape.n_heads, shape.head_dim, dtype=F64)
    for l in range(shape.n_layers):
        h, _, _ = layer_forward(shape, W.layer(l), h, pos, empty, empty)
    return h
