"""GPU-vs-oracle comparison of whole rollout workloads (used by the -m gpu tests and smoke()).

Tolerances (fixed by the method's bf16 weights / fp32 accumulation):
  * action tokens bit-exact in teacher-forced mode wherever the oracle's top-2 margin of the
    perturbed score exceeds 0.05;
  * actions bit-exact wherever the tokens match;
  * logits, log-probs and the rollout entropy within 2e-2 absolute.
The GPU decodes with forced_tokens = the oracle's tokens, so both sides condition on the
same trajectory.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Sequence

import numpy as np
import torch

import oracle.vla_oracle as O
from paper_2505_18719_gb300 import inputs as I
from tests import attribution as A
from paper_2505_18719_gb300 import vla as V

TOL = 2e-2
MARGIN = 0.05


@dataclasses.dataclass
class TurnReport:
    turn: int
    envs: List[int]
    max_lp_err: float
    max_logit_err: float
    token_checked: int
    token_mismatch: int
    action_mismatch: int
    score_lp_err: Optional[float] = None
    score_vs_decode_err: Optional[float] = None
    score_logit_err: Optional[float] = None
    logit_err_by_step: Optional[list] = None
    emul_logit_err: Optional[float] = None      # vs the GPU-rounding oracle (attribution)
    emul_lp_err: Optional[float] = None
    entropy_err: Optional[float] = None         # rollout entropy of decode (and score)
    value_err: Optional[float] = None           # value head at the turn's prefill

    def ok(self) -> bool:
        errs = [self.max_lp_err, self.max_logit_err]
        errs += [e for e in (self.score_lp_err, self.score_vs_decode_err, self.score_logit_err,
                             self.entropy_err, self.value_err) if e is not None]
        return self.token_mismatch == 0 and self.action_mismatch == 0 and max(errs) <= TOL


def weights_to_device(w: Dict[str, torch.Tensor], device="cuda") -> Dict[str, torch.Tensor]:
    return {k: v.to(device) for k, v in w.items()}


def check_envs(wl: I.Workload, lengths: torch.Tensor, n_check: Optional[int]) -> List[int]:
    if n_check is None or n_check >= wl.batch:
        return list(range(wl.batch))
    # the first env and the longest one (ragged workloads), else the last one
    longest = int(torch.argmax(lengths).item())
    other = longest if longest != 0 else wl.batch - 1
    return [0, other][:n_check]


def run_parity(wl: I.Workload, weights_cpu=None, weights_dev=None, n_check: Optional[int] = None,
               turns: Optional[int] = None, cache_f64: bool = True, temperature: Optional[float] = None,
               device="cuda", attribution: bool = False) -> List[TurnReport]:
    sh = wl.shape
    T = wl.temperature if temperature is None else temperature
    if weights_cpu is None:
        weights_cpu = I.make_weights(sh, wl.weight_seed)
    if weights_dev is None:
        weights_dev = weights_to_device(weights_cpu, device)
    n_turns = wl.turns if turns is None else turns
    max_tokens = wl.batch * (wl.n_visual + (wl.text_len or wl.text_len_range[1]) + 8)
    pol = V.Policy(sh, weights_dev, wl.batch, wl.kv_capacity, max_tokens)
    orc = O.Oracle(O.shape_from(sh), weights_cpu, wl.batch, cache_f64=cache_f64)
    emu = A.AttributionOracle(O.shape_from(sh), weights_cpu, wl.batch, cache_f64=cache_f64,
                              rounding=A.GPU_PATH) if attribution else None
    base = sh.vocab - sh.n_bins
    reports = []
    envs = None
    try:
        for t in range(n_turns):
            inp = I.make_turn_inputs(wl, t)
            if envs is None:
                envs = check_envs(wl, inp.lengths, n_check)
            for t_r, ended in wl.resets:
                if t_r == t:
                    pol.reset([1 if b in ended else 0 for b in range(wl.batch)])
                    for o_ in (orc, emu):
                        if o_ is not None and any(b in envs for b in ended):
                            o_.reset([b for b in ended if b in envs])
            pol.prefill(inp.visual.to(device), inp.ids.to(device), inp.lengths.tolist())
            for o_ in (orc, emu):
                if o_ is not None:
                    o_.prefill(envs, [inp.visual[b] for b in envs],
                               [inp.ids[b, :int(inp.lengths[b])].tolist() for b in envs])
            # value head (Algorithm 1: V_t) at the prefill, same decoder weights
            wv = I.normal_bf16((sh.d_model,), 2025, 77, 0.02)
            gv = pol.value(wv.to(device), 0.25).cpu().numpy()
            ov = orc.value(envs, wv, 0.25)
            value_err = float(np.max(np.abs(gv[envs] - ov)))
            u_cpu = inp.uniforms
            od = orc.decode(envs, u_cpu[envs], T)
            forced = torch.full((wl.batch, sh.action_dim), base, dtype=torch.int32)
            for j, b in enumerate(envs):
                forced[b] = torch.as_tensor(od["tokens"][j], dtype=torch.int32)
            # envs that are not compared follow a fixed valid action sequence
            for b in range(wl.batch):
                if b not in envs:
                    forced[b] = base + (torch.arange(sh.action_dim, dtype=torch.int32) * 37 + b) % 256
            gd = pol.decode(u_cpu.to(device), T, forced=forced.to(device))
            pol.sync()
            g = {k: v.cpu().numpy() for k, v in gd.items() if v is not None}
            rep = compare_decode(t, envs, od, g)
            rep.entropy_err = float(np.max(np.abs(g["entropy"][envs] - od["entropy"])))
            rep.value_err = value_err
            if emu is not None:
                ed = emu.decode(envs, u_cpu[envs], T, forced=forced[envs])
                rep.emul_logit_err = float(np.max(np.abs(g["logits"][envs] - ed["logits"])))
                rep.emul_lp_err = float(np.max(np.abs(g["logprobs"][envs] - ed["logprobs"])))
            if wl.score:
                sc = pol.score(forced.to(device), T)
                pol.sync()
                os_ = orc.score(envs, forced[envs], T)
                if emu is not None:
                    emu.score(envs, forced[envs], T)
                glp = sc["logprobs"].cpu().numpy()
                glg = sc["logits"].cpu().numpy()
                rep.score_lp_err = float(np.max(np.abs(glp[envs] - os_["logprobs"])))
                rep.score_logit_err = float(np.max(np.abs(glg[envs] - os_["logits"])))
                rep.score_vs_decode_err = float(np.max(np.abs(glp - g["logprobs"])))
                rep.entropy_err = max(rep.entropy_err,
                                      float(np.max(np.abs(sc["entropy"].cpu().numpy()[envs] - os_["entropy"]))))
            reports.append(rep)
    finally:
        pol.close()
    return reports


def compare_decode(turn: int, envs: Sequence[int], od: dict, g: dict) -> TurnReport:
    lp_err = float(np.max(np.abs(g["logprobs"][envs] - od["logprobs"])))
    lg_err = float(np.max(np.abs(g["logits"][envs] - od["logits"])))
    mask = od["margins"] > MARGIN
    tok_mis = int(np.sum((g["tokens"][envs] != od["tokens"]) & mask))
    same = g["tokens"][envs] == od["tokens"]
    act_mis = int(np.sum((g["actions"][envs] != od["actions"].astype(np.float32)) & same))
    by_step = np.max(np.abs(g["logits"][envs] - od["logits"]), axis=(0, 2)).round(5).tolist()
    return TurnReport(turn, list(envs), lp_err, lg_err, int(mask.sum()), tok_mis, act_mis,
                      logit_err_by_step=by_step)
