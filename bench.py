"""Benchmark of the rollout / re-scoring hot path on GB300 (one JSON line on stdout).

A step is one pass of the whole hot path over one batch: reset, prefill of every env's
prefix (visual embeddings + instruction ids), the 7-token decode (sampling, log-probs,
actions) and the teacher-forced re-scoring of those tokens (PPO ratio pass).  Workload:
the Llama-2-7B-shaped policy with 64 envs and ragged text lengths U{16..48} after 256
visual embeddings (synthetic, seeded, random-init weights).

value = action tokens per second over whole steps (64 envs x 7 tokens / step time), with
inputs resident in HBM.  e2e = the same through the C ABI with host buffers (pinned H2D of
the step's inputs, D2H of tokens / log-probs / actions / scores inside the timed region).

--impl reference times the fp64 CPU oracle (the deliberately slow reference of this
build) on a bounded sample of the same workload.

Multi-GPU: one process per GPU (torchrun); each rank runs an independent replica on its own
batch of 64 envs (envs are independent: weak scaling, no data-path collective); the step
time is the max over ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "7b_b64_ragged_score"


# DRAM bytes of one launch of the dominant kernel from an ncu capture (set to None whenever
# that kernel changes): gemm_tc2_kernel, the q|k|v projection of this step's prefill
# (18385 x 12288 x 4096, fp16 operand pair, case pair_prefill_qkv_18385_f16; fp32 output in
# the case).
PROFILED_TRAFFIC = {"bytes": 2.366113e9 + 0.880124e9,
                    "launch": "gemm_tc2_kernel q|k|v (fp16 operands), M=18385 N=12288 K=4096",
                    "algorithmic_bytes": 2.0 * 18385 * 4096 * 2 + 2.0 * 12288 * 4096 + 4.0 * 18385 * 12288,
                    "profile": "profiles/gemm_tc2_prefill_qkv_18385x12288x4096.md"}


def workload_config(wl, n_gpus):
    """The `config` object of the JSON line (both arms)."""
    text = f"U{{{wl.text_len_range[0]}..{wl.text_len_range[1]}}}" if wl.text_len is None else str(wl.text_len)
    step = ("reset + prefill + 7-token decode" if wl.turns == 1 else
            f"reset + {wl.turns} turns x (prefill/append + 7-token decode)") + (" + score" if wl.score else "")
    return {"workload": wl.name, "model": wl.shape.name, "batch_per_gpu": wl.batch, "n_visual": wl.n_visual,
            "text_len": text, "turns": wl.turns, "append_visual": wl.append_visual if wl.turns > 1 else 0,
            "append_text": wl.append_text if wl.turns > 1 else 0, "action_tokens": wl.shape.action_dim,
            "temperature": wl.temperature, "step": step,
            "l2": "no flush: 13 GB of weights streamed per forward (> 129 MB L2)",
            "parallelism": f"replicas x{n_gpus}"}


def phase_work(sh, past, chunk):
    """Algorithmic work of one turn's phases for envs whose chunk of chunk[b] rows lands after
    past[b] cached positions (7B: 6.476e9 matrix parameters; K+V per position and layer as
    cached: 16 KB of fp16 parts and 4 KB of 4-bit residual codes).  Prefill FLOPs count what the method needs: every row through every layer,
    except that the last layer only needs q|k|v for all rows (KV cache) and the rest for each
    env's final row; attention FLOPs are the causal ones.  Decode bytes are, per forward, all
    weights + the K/V each env reads (positions 0..pos) and writes + the 256 head rows.
    Score: one weight stream, K/V reads of the 6 teacher-forced rows, 2 P flops per row; its
    projections (384 rows) are tensor-bound, so the pass's floor is max(projection flops at the
    tensor peak, weights at HBM speed) + the K/V reads at HBM speed."""
    d, F, L = sh.d_model, sh.d_ffn, sh.n_layers
    per_layer = 4 * d * d + 3 * F * d
    qkv_params = 3 * d * d
    params = L * per_layer
    w_bytes = 2.0 * params
    kv_tok = 2.5 * 2 * d * L                    # K and V as cached (fp16 + 4-bit residual), all layers
    A = sh.action_dim
    B = len(chunk)
    T = sum(chunk)
    P = [p + n for p, n in zip(past, chunk)]    # context after the prefill
    attn = sum(2.0 * d * (2 * n * p + n * (n + 1)) for p, n in zip(past, chunk))  # per layer
    flops_pre = (L - 1) * (2.0 * T * per_layer + attn) \
        + 2.0 * T * qkv_params + 2.0 * B * (per_layer - qkv_params) + sum(4.0 * d * p for p in P)
    flops_pre_formula = 2.0 * params * T + L * attn
    dec_bytes = 0.0
    for i in range(1, A):
        dec_bytes += w_bytes + sum((p + i) * kv_tok for p in P) + B * kv_tok + 2.0 * 256 * d
    dec_bytes += 2.0 * 256 * d                  # head of the first action (prefill's last row)
    n = A - 1
    sc_bytes = w_bytes + sum((p + n) * kv_tok for p in P) + B * n * kv_tok + 2.0 * 256 * d
    sc_flops = 2.0 * params * B * n + L * sum(2.0 * d * (2 * n * p + n * (n + 1)) for p in P)
    return {"prefill_flops": flops_pre, "prefill_flops_all_rows": flops_pre_formula,
            "decode_bytes": dec_bytes, "score_bytes": sc_bytes, "score_flops": sc_flops,
            "score_gemm_flops": 2.0 * params * B * n, "score_weight_bytes": w_bytes + 2.0 * 256 * d, "rows": T}


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p["hbm_gbs"], p["bf16_tflops"], p["bf16_tflops_sustained"], "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while the timed region runs."""

    def __init__(self, index: int):
        self.index = index
        self.samples = []
        self.proc = None
        self.thread = None

    def __enter__(self):
        cmd = ["nvidia-smi", "-i", str(self.index),
               "--query-gpu=clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
               "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
               "clocks_event_reasons.sw_power_cap", "--format=csv,noheader,nounits", "-lms", "200"]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 7:
                self.samples.append(parts)

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm = [float(s[0]) for s in self.samples if s[0].replace(".", "").isdigit()]
        mx = [float(s[1]) for s in self.samples if s[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for s in self.samples for i in range(4) if s[3 + i].strip() == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(self.samples)}


def max_over_ranks(x: float, dist=None, device="cuda") -> float:
    """Largest value over all ranks (the job is as slow as its slowest replica)."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def oracle_sample(wl, weights_cpu, n_threads=None):
    """Time the fp64 oracle on one env of the workload: prefill + 7-token decode + score."""
    import torch
    import oracle.vla_oracle as O
    from paper_2505_18719_gb300 import inputs as I
    if n_threads:
        torch.set_num_threads(n_threads)
    inp = I.make_turn_inputs(wl, 0)
    orc = O.Oracle(O.shape_from(wl.shape), weights_cpu, wl.batch, cache_f64=False)
    t0 = time.perf_counter()
    orc.prefill([0], [inp.visual[0]], [inp.ids[0, :int(inp.lengths[0])].tolist()])
    d = orc.decode([0], inp.uniforms[:1], wl.temperature)
    if wl.score:
        orc.score([0], torch.as_tensor(d["tokens"]), wl.temperature)
    dt = time.perf_counter() - t0
    prefix = wl.n_visual + int(inp.lengths[0])
    return dt, prefix, torch.get_num_threads()


def run_reference(args):
    """--impl reference: the fp64 oracle on the host cores, bounded sample per step."""
    world, rank, _ = dist_setup()
    if rank != 0:
        return 0
    from paper_2505_18719_gb300 import inputs as I
    wl = I.WORKLOADS[args.workload]
    w = I.make_weights(wl.shape, wl.weight_seed)
    times = []
    threads = None
    for i in range(args.warmup + args.steps):
        dt, prefix, threads = oracle_sample(wl, w)
        if i >= args.warmup:
            times.append(dt)
    per_step = statistics.median(times)
    value = wl.shape.action_dim / per_step
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "action tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": per_step * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded; random-init weights)",
        "config": dict(workload_config(wl, world), sample="1 env per step (prefill + 7 tokens + score)"),
        "cpu_baseline": {"value": value, "unit": "action tokens/s", "cores": threads, "host_cpus": os.cpu_count(),
                         "kind": "oracle",
                         "sample": f"1 of {wl.batch} envs, prefix {prefix} tokens, prefill+decode+score, fp64"},
        "e2e": {"value": value, "unit": "action tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


METRIC = "action tokens/sec (batched decode, 7B shape) and prefill tok/s; % of HBM/TC roofline"

# Single-kernel cases (7B shapes) for profiling one kernel in isolation, e.g. under ncu.
CASES = {
    # name: (M, N, K, block_n, splits, split A)
    "gemm_prefill_qkv": (4608, 12288, 4096, 256, 1, True),     # 16 envs x 288-token prefixes
    "gemm_prefill_down": (4608, 4096, 11008, 256, 1, True),
    "gemm_decode_qkv": (64, 12288, 4096, 128, 2, True),        # one decode step, 64 envs
    "gemm_decode_o": (64, 4096, 4096, 128, 5, True),
    # weight-streaming decode GEMM (swap-AB, stream-K): block_n / splits unused
    "gemv_decode_qkv": (64, 12288, 4096, 0, 0, True),
    "gemv_decode_o": (64, 4096, 4096, 0, 0, True),
    "gemv_decode_gate_up": (64, 22016, 4096, 0, 0, True),
    "gemv_decode_down": (64, 4096, 11008, 0, 0, True),
    "attn_decode": None,                                       # see run_attn_case
    "attn_decode_res": None,
    "learning": None,                                          # see run_learning_case
    "attn_chunk": None,                                        # see run_attn_chunk_case
    "attn_score": None,                                        # 6 rows per env after the prefix
    "attn_chunk_res": None,                                    # the same over fp16 + 4-bit residual
    "attn_score_res": None,
    "attn_score_rows_res": None,                               # the few-row kernel (tiles <= 16 rows)
    # the same prefill shapes on CTA pairs (2-SM MMAs, 256 x 256 tiles)
    "pair_prefill_qkv": (4608, 12288, 4096, 256, 1, True),
    "pair_prefill_down": (4608, 4096, 11008, 256, 1, True),
    "pair_prefill_gate_up_18k": (18432, 22016, 4096, 256, 1, True),
    # the q|k|v launch of the bench step's prefill (64 envs, 18385 rows)
    "pair_prefill_qkv_18385": (18385, 12288, 4096, 256, 1, True),
    "gemm_prefill_gate_up_18k": (18432, 22016, 4096, 256, 1, True),
    # score-pass shapes (64 envs x 6 teacher-forced rows): tile / split choices
    "gemm_score_qkv_bn256": (384, 12288, 4096, 256, 1, True),
    "gemm_score_qkv_bn128": (384, 12288, 4096, 128, 1, True),
    "gemm_score_o_s1": (384, 4096, 4096, 128, 1, True),
    "gemm_score_o_s2": (384, 4096, 4096, 128, 2, True),
    "gemm_score_down_s1": (384, 4096, 11008, 128, 1, True),
    "gemm_score_down_s2": (384, 4096, 11008, 128, 2, True),
    "gemm_score_gate_up_bn256": (384, 22016, 4096, 256, 1, True),
    "gemm_score_gate_up_bn128": (384, 22016, 4096, 128, 1, True),
    "pair_score_gate_up": (384, 22016, 4096, 256, 1, True),
    "pair_score_qkv": (384, 12288, 4096, 256, 1, True),
    "pair_score_down": (384, 4096, 11008, 256, 1, True),
    "gemm_score_down_bn256": (384, 4096, 11008, 256, 1, True),
    # the same in the engine's form: fp16 operands, the activation's high half alone
    "gemm_score_o_s1_hi_f16": (384, 4096, 4096, 128, 1, False),
    "gemm_score_o_s2_hi_f16": (384, 4096, 4096, 128, 2, False),
    "gemm_score_o_bn256_s3_hi_f16": (384, 4096, 4096, 256, 3, False),
    "gemm_score_down_s1_hi_f16": (384, 4096, 11008, 128, 1, False),
    "gemm_score_down_s2_hi_f16": (384, 4096, 11008, 128, 2, False),
    "gemm_score_down_bn256_s3_hi_f16": (384, 4096, 11008, 256, 3, False),
    "gemm_score_gate_up_bn256_hi_f16": (384, 22016, 4096, 256, 1, False),
    "gemm_score_gate_up_bn128_hi_f16": (384, 22016, 4096, 128, 1, False),
    "gemm_score_qkv_bn128_f16": (384, 12288, 4096, 128, 1, True),
    "gemm_score_qkv_bn256_s2_f16": (384, 12288, 4096, 256, 2, True),
    "gemv_score_o_m128": (128, 4096, 4096, 0, 0, True),
    "gemv_score_down_m128": (128, 4096, 11008, 0, 0, True),
    # decode GEMM at 2x / 4x the weight bytes of the q|k|v step (fixed vs per-byte cost)
    "gemv_decode_k8192": (64, 12288, 8192, 0, 0, True),
    "gemv_decode_k16384": (64, 12288, 16384, 0, 0, True),
}

# every GEMM case also with fp16 operands (the engine's form): NAME_f16
CASES.update({k + "_f16": v for k, v in list(CASES.items()) if v is not None})


def run_attn_case(args):
    """Decode attention for 64 envs x 32 heads at ~290 cached positions (one layer); attn_decode_res
    reads the fp16 parts and their 4-bit residual codes (the engine's form)."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2505_18719_gb300 import inputs as I
    from paper_2505_18719_gb300 import vla as V
    B, H, hd = 64, 32, 128
    scale = max(1, args.attn_ctx_scale)
    cap = 320 * scale
    kv = I.normal_bf16((B, 2, H, cap, hd), 5, 1, 1.0).cuda().half()
    res = args.case.endswith("_res")
    codes = I.randint_i32((B * 2 * H * cap * hd // 2,), 5, 4, 0, 256).to(torch.uint8).cuda() if res else None
    q = I.normal_bf16((B, H, hd), 5, 2, 1.0).cuda().float()
    ctx = I.randint_i32((B,), 5, 3, 273, 311) * scale
    env = torch.arange(B, dtype=torch.int32, device="cuda")
    pos = (ctx - 1).cuda()
    max_ctx = int(ctx.max())
    keys = args.attn_keys
    nbytes = V.vla_op_attn_decode_workspace_bytes(B, H, hd, max_ctx, keys)
    ws = torch.empty(nbytes // 4 + 64, dtype=torch.float32, device="cuda")
    oh = torch.empty(B, H * hd, dtype=torch.bfloat16, device="cuda")
    ol = torch.empty_like(oh)
    stream = torch.cuda.current_stream()

    def launch():
        if res:
            rc = V.vla_op_attn_decode_res(q.data_ptr(), kv.data_ptr(), codes.data_ptr(), B, H, hd, cap, env.data_ptr(),
                                          pos.data_ptr(), B, max_ctx, oh.data_ptr(), ol.data_ptr(), ws.data_ptr(),
                                          nbytes, stream.cuda_stream, keys)
        else:
            rc = V.vla_op_attn_decode(q.data_ptr(), kv.data_ptr(), B, H, hd, cap, env.data_ptr(), pos.data_ptr(), B,
                                      max_ctx, oh.data_ptr(), ol.data_ptr(), ws.data_ptr(), nbytes,
                                      stream.cuda_stream, keys)
        assert rc == 0, V.vla_last_error()

    for _ in range(args.warmup):
        launch()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        launch()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    hbm, _, _, kind = peaks()
    bytes_ = float(ctx.sum()) * 2 * H * hd * (2.5 if res else 2) + B * H * hd * (4 + 4)
    print(json.dumps({"case": args.case, "B": B, "H": H, "hd": hd, "max_keys_per_cta": keys,
                      "kv_positions": int(ctx.sum()), "ms": ms,
                      "gbs": bytes_ / ms / 1e6, "hbm_frac": bytes_ / ms / 1e6 / hbm, "peaks": kind}))
    return 0


def run_attn_chunk_case(args):
    """Prefill chunk attention of one layer of the bench step: 64 envs, 256 visual + U{16..48}
    text rows each, 32 heads x 128.  attn_chunk / attn_score: the fp16-cache kernel, tiles of
    <= 64 query rows; attn_chunk_res / attn_score_res: the tcgen05 kernel over the fp16 +
    4-bit residual cache, tiles of <= 128 rows; attn_score_rows_res: the few-row kernel over the
    same cache (the engine's score-pass form)."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2505_18719_gb300 import inputs as I
    from paper_2505_18719_gb300 import vla as V
    B, H, hd, cap = 64, 32, 128, 320
    prefix = (256 + I.randint_i32((B,), 5, 7, 16, 48)).tolist()
    score = args.case.startswith("attn_score")   # the score pass: 6 rows per env after its prefix
    res = args.case.endswith("_res")
    few = args.case == "attn_score_rows_res"
    tile_rows = 128 if res else 64
    lens = [6] * B if score else prefix
    past = prefix if score else [0] * B
    rows = sum(lens)
    kv = I.normal_bf16((B, 2, H, cap, hd), 5, 1, 1.0).cuda().half()
    codes = I.randint_i32((B * 2 * H * cap * hd // 2,), 5, 3, 0, 256).to(torch.uint8).cuda() if res else None
    q = I.normal_bf16((rows, H * hd), 5, 2, 1.0).cuda().float()
    tiles, r = [], 0
    for b, n in enumerate(lens):
        for t0 in range(0, n, tile_rows):
            tiles.append((b, r + t0, min(tile_rows, n - t0), past[b] + t0))
        r += n
    tiles_dev = torch.zeros(len(tiles) * 4, dtype=torch.int32, device="cuda")
    oh = torch.empty(rows, H * hd, dtype=torch.bfloat16, device="cuda")
    ol = torch.empty_like(oh)

    def launch():
        if few:
            rc = V.vla_op_attn_rows_res(q.data_ptr(), kv.data_ptr(), codes.data_ptr(), B, H, hd, cap, tiles, rows,
                                        tiles_dev.data_ptr(), oh.data_ptr(), ol.data_ptr())
        elif res:
            rc = V.vla_op_attn_chunk_res(q.data_ptr(), kv.data_ptr(), codes.data_ptr(), B, H, hd, cap, tiles, rows,
                                         tiles_dev.data_ptr(), oh.data_ptr(), ol.data_ptr())
        else:
            rc = V.vla_op_attn_chunk(q.data_ptr(), kv.data_ptr(), B, H, hd, cap, tiles, rows, tiles_dev.data_ptr(),
                                     oh.data_ptr(), ol.data_ptr())
        assert rc == 0, V.vla_last_error(None)

    for _ in range(args.warmup):
        launch()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.steps):
        launch()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    flops = sum(2.0 * H * hd * n * (n + 1 + 2 * p) for n, p in zip(lens, past))   # causal QK^T + PV
    kv_bytes = sum((p + n) * 2.0 * H * hd * (2.5 if res else 2) for n, p in zip(lens, past))
    _, tf_burst, _, kind = peaks()
    print(json.dumps({"case": args.case, "B": B, "H": H, "hd": hd, "rows": rows, "tiles": len(tiles), "ms": ms,
                      "tflops": flops / ms / 1e9, "tc_frac_of_burst": flops / ms / 1e9 / tf_burst,
                      "issued_mma_tflops": (3 if res else 2) * flops / ms / 1e9, "kv_gbs": kv_bytes / ms / 1e6, "peaks": kind}))
    return 0


def run_learning_case(args):
    """GAE over 128 steps x 256 envs and the clipped PPO objective over those 32768 samples
    (7 token log-probs each): the learning-phase quantities of one rollout batch."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2505_18719_gb300 import inputs as I
    from paper_2505_18719_gb300 import vla as V
    M, B, A = 128, 256, 7
    r = I.normal_bf16((M, B), 9, 1, 1.0).float().cuda()
    v = I.normal_bf16((M + 1, B), 9, 2, 1.0).float().cuda()
    dn = (I.uniform_f32((M, B), 9, 3) < 0.05).float().cuda()
    adv = torch.empty(M, B, device="cuda")
    ret = torch.empty(M, B, device="cuda")
    lp_old = (-I.uniform_f32((M * B, A), 9, 4) * 6.0).cuda()
    lp_new = lp_old + 0.01
    obj = torch.empty(1, device="cuda")
    out = {"case": "learning", "M": M, "B": B, "A": A}
    for name, fn, nbytes in (
            ("gae", lambda: V.vla_gae(r.data_ptr(), v.data_ptr(), dn.data_ptr(), M, B, 0.99, 0.95, adv.data_ptr(),
                                      ret.data_ptr(), 0), 4.0 * (M * B * 5 + B)),
            ("ppo_clip", lambda: V.vla_ppo_clip(lp_new.data_ptr(), lp_old.data_ptr(), adv.data_ptr(), M * B, A, 0.2,
                                                obj.data_ptr(), 0, 0, 0), 4.0 * M * B * (2 * A + 1))):
        for _ in range(args.warmup):
            assert fn() == 0
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(args.steps):
            assert fn() == 0
        e1.record()
        torch.cuda.synchronize()
        us = e0.elapsed_time(e1) / args.steps * 1e3
        out[name] = {"us": round(us, 2), "bytes": nbytes, "gbs": round(nbytes / us / 1e3, 1)}
    print(json.dumps(out))
    return 0


def run_case(args):
    """Time one GEMM shape through the GEMM op entry points (CUDA events, device-resident
    operands); bf16 operands, or fp16 for the NAME_f16 cases."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2505_18719_gb300 import inputs as I
    from paper_2505_18719_gb300 import vla as V
    if args.case in ("attn_decode", "attn_decode_res"):
        return run_attn_case(args)
    if args.case == "learning":
        return run_learning_case(args)
    if args.case.startswith(("attn_chunk", "attn_score")):
        return run_attn_chunk_case(args)
    M, N, K, bn, splits, split_a = CASES[args.case]
    fp16 = args.case.endswith("_f16")
    A = I.normal_bf16((M, K), 1, 1, 1.0).cuda()
    A_lo = I.normal_bf16((M, K), 1, 2, 2.0 ** -9).cuda()
    W = I.normal_bf16((N, K), 1, 3, 0.02).cuda()
    if fp16:
        A, A_lo, W = A.half(), (A_lo * 2.0 ** -3).half(), W.half()
    op_gemm, op_pair, op_decode = ((V.vla_op_gemm_f16, V.vla_op_gemm_pair_f16, V.vla_op_gemm_decode_f16) if fp16
                                   else (V.vla_op_gemm_bf16, V.vla_op_gemm_pair_bf16, V.vla_op_gemm_decode_bf16))
    C = torch.empty(M, N, dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()
    if args.case.startswith("pair"):
        ws = None

        def launch():
            rc = op_pair(A.data_ptr(), A_lo.data_ptr() if split_a else 0, K, W.data_ptr(), K,
                         C.data_ptr(), N, M, N, K, stream.cuda_stream)
            assert rc == 0, V.vla_last_error()
    elif args.case.startswith("gemv"):
        nbytes = V.vla_op_gemm_decode_workspace_bytes(M, N, K)
        ws = torch.empty(max(1, nbytes // 4), dtype=torch.float32, device="cuda")

        def launch():
            rc = op_decode(A.data_ptr(), A_lo.data_ptr(), K, W.data_ptr(), K, C.data_ptr(), N,
                           M, N, K, ws.data_ptr(), nbytes, stream.cuda_stream)
            assert rc == 0, V.vla_last_error()
    else:
        ws = torch.empty(max(1, splits * M * N), dtype=torch.float32, device="cuda")

        def launch():
            rc = op_gemm(A.data_ptr(), A_lo.data_ptr() if split_a else 0, K, W.data_ptr(), K,
                         C.data_ptr(), N, M, N, K, bn, splits, ws.data_ptr(), stream.cuda_stream)
            assert rc == 0, V.vla_last_error()

    for _ in range(args.warmup):
        launch()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        launch()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    hbm, tf_burst, _, kind = peaks()
    flops = 2.0 * M * N * K
    bytes_ = 2.0 * (M * K * (2 if split_a else 1) + N * K) + 4.0 * M * N
    print(json.dumps({"case": args.case, "M": M, "N": N, "K": K, "block_n": bn, "splits": splits,
                      "split_a": split_a, "operands": "fp16" if fp16 else "bf16", "ms": ms, "tflops": flops / ms / 1e9,
                      "tc_frac_of_burst": flops / ms / 1e9 / tf_burst, "gbs": bytes_ / ms / 1e6,
                      "hbm_frac": bytes_ / ms / 1e6 / hbm, "peaks": kind}))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=WORKLOAD)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--case", choices=sorted(CASES), help="time one kernel shape instead of the hot path")
    ap.add_argument("--attn-keys", type=int, default=0, help="attn_decode case: max keys per CTA (0 = default)")
    ap.add_argument("--attn-ctx-scale", type=int, default=1, help="attn_decode case: context length multiplier")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)
    if args.case:
        return run_case(args)

    import torch
    world, rank, local = dist_setup()
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    import __graft_entry__
    __graft_entry__.build()
    from paper_2505_18719_gb300 import inputs as I
    from paper_2505_18719_gb300 import vla as V

    wl = I.WORKLOADS[args.workload]
    sh = wl.shape
    B, A = wl.batch, sh.action_dim
    w_cpu = I.make_weights(sh, wl.weight_seed)
    w_dev = {k: v.cuda() for k, v in w_cpu.items()}
    # each rank: its own batch of envs (weak scaling); rank 0 = the workload's own inputs
    wl_r = wl if rank == 0 else I.dataclasses.replace(wl, index=wl.index + 1000 * rank)
    turns = [I.make_turn_inputs(wl_r, t) for t in range(wl.turns)]
    lens = [tin.lengths.tolist() for tin in turns]
    max_tokens = B * max(tin.visual.shape[1] + max(l) + 8 for tin, l in zip(turns, lens))
    stream = torch.cuda.current_stream()
    pol = V.Policy(sh, w_dev, B, wl.kv_capacity, max_tokens, stream=stream)

    dev_in = [(tin.visual.cuda(), tin.ids.cuda(), tin.uniforms.cuda()) for tin in turns]
    tok = torch.empty(B, A, dtype=torch.int32, device="cuda")
    lp = torch.empty(B, A, dtype=torch.float32, device="cuda")
    act = torch.empty(B, A, dtype=torch.float32, device="cuda")
    slp = torch.empty(B, A, dtype=torch.float32, device="cuda")
    T = wl.temperature
    h = pol.h
    reset_masks = {t: [1 if b in ended else 0 for b in range(B)] for t, ended in wl.resets}

    def step(inputs, ev=None, before_turn=None, after_turn=None):
        """reset, then per turn: episode ends, prefill (append), 7-token decode; then the score
        pass of the last turn.  ev: events [turn][3] + [2] for the score, for phase times."""
        pol.check(V.vla_reset(h, None))
        for t, (vis, ids, u) in enumerate(inputs):
            if before_turn:
                before_turn(t)
            if t in reset_masks:
                pol.check(V.vla_reset(h, reset_masks[t]))
            if ev:
                ev[t][0].record(stream)
            pol.check(V.vla_prefill(h, B, vis.data_ptr(), vis.shape[1], ids.data_ptr(), lens[t], ids.shape[1]))
            if ev:
                ev[t][1].record(stream)
            pol.check(V.vla_decode_actions(h, u.data_ptr(), T, 0, tok.data_ptr(), lp.data_ptr(), act.data_ptr(), 0))
            if ev:
                ev[t][2].record(stream)
            if after_turn:
                after_turn(t)
        if wl.score:
            if ev:
                ev[-1][0].record(stream)
            pol.check(V.vla_score_actions(h, tok.data_ptr(), T, slp.data_ptr(), 0))
            if ev:
                ev[-1][1].record(stream)

    def barrier():
        if dist is not None:
            dist.barrier()

    # ---- warm-up
    for _ in range(args.warmup):
        step(dev_in)
    pol.sync()

    # ---- timed region (device-resident inputs)
    launches0 = V.vla_launch_count(h)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        ev0.record(stream)
        for _ in range(args.steps):
            step(dev_in)
        ev1.record(stream)
        torch.cuda.synchronize()
    barrier()
    ms_total = max_over_ranks(ev0.elapsed_time(ev1), dist)
    launches = V.vla_launch_count(h) - launches0
    pol.sync()
    ms_step = ms_total / args.steps
    # ---- the same steps again with the library's events around each GEMM (for the roofline);
    # the events keep consecutive kernels from overlapping, so they stay out of the region above
    V.vla_profile(h, (1 << 0) | (1 << 1))
    for _ in range(args.steps):
        step(dev_in)
    pol.sync()
    prof = V.vla_profile_read(h)
    V.vla_profile(h, 0)

    # ---- phase breakdown (separate, untimed for the headline)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(wl.turns)]
    evs.append([torch.cuda.Event(enable_timing=True) for _ in range(2)])
    step(dev_in, ev=evs)
    pol.sync()
    t_pre_t = [evs[t][0].elapsed_time(evs[t][1]) for t in range(wl.turns)]
    t_dec_t = [evs[t][1].elapsed_time(evs[t][2]) for t in range(wl.turns)]
    t_pre, t_dec = sum(t_pre_t), sum(t_dec_t)
    t_sc = evs[-1][0].elapsed_time(evs[-1][1]) if wl.score else 0.0
    # one more step with every kernel class bracketed by events (outside the timed region)
    V.vla_profile(h, (1 << len(V.KCLASS)) - 1)
    step(dev_in)
    per_class = V.vla_profile_read(h)
    V.vla_profile(h, 0)

    # algorithmic work per turn (context lengths tracked as the handle does)
    ctx, pending = [0] * B, [0] * B
    works = []
    for t in range(wl.turns):
        for b in (wl.resets and dict(wl.resets).get(t, ()) or ()):
            ctx[b], pending[b] = 0, 0
        chunk = [pending[b] + turns[t].visual.shape[1] + int(lens[t][b]) for b in range(B)]
        works.append(phase_work(sh, ctx, chunk))
        ctx = [ctx[b] + chunk[b] + A - 1 for b in range(B)]
        pending = [1] * B
    prefill_rows = sum(w_["rows"] for w_ in works)
    phase = {"prefill_ms": t_pre, "decode_ms": t_dec, "score_ms": t_sc,
             "prefill_tok_s": prefill_rows / (t_pre / 1e3), "decode_action_tok_s": wl.turns * B * A / (t_dec / 1e3),
             "kernel_classes_ms": {k: round(v["ms"], 3) for k, v in per_class.items()},
             "kernel_classes_launches": {k: v["launches"] for k, v in per_class.items()}}
    if wl.turns > 1:
        phase["prefill_ms_per_turn"] = [round(x, 3) for x in t_pre_t]
        phase["decode_ms_per_turn"] = [round(x, 3) for x in t_dec_t]
        phase["decode_action_tok_s_per_turn"] = [round(B * A / (x / 1e3), 1) for x in t_dec_t]

    # ---- e2e through the C ABI with host buffers: each turn's inputs are copied in before
    # its prefill and its tokens / log-probs / actions copied out after its decode
    host_in = [(tin.visual.pin_memory(), tin.ids.pin_memory(), tin.uniforms.pin_memory()) for tin in turns]
    e2e_in = [tuple(torch.empty_like(x) for x in di) for di in dev_in]
    out_h = [[torch.empty(B, A, dtype=t_).pin_memory() for t_ in (torch.int32, torch.float32, torch.float32)]
             for _ in range(wl.turns)]
    score_h = torch.empty(B, A, dtype=torch.float32).pin_memory()

    def copy_in(t):
        for dst, src in zip(e2e_in[t], host_in[t]):
            dst.copy_(src, non_blocking=True)

    def copy_out(t):
        for dst, src in zip(out_h[t], (tok, lp, act)):
            dst.copy_(src, non_blocking=True)

    def e2e_step():
        step(e2e_in, before_turn=copy_in, after_turn=copy_out)
        if wl.score:
            score_h.copy_(slp, non_blocking=True)

    e2e_step()
    pol.sync()
    barrier()
    torch.cuda.synchronize()
    ev0.record(stream)
    for _ in range(args.steps):
        e2e_step()
    ev1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(ev0.elapsed_time(ev1), dist) / args.steps
    h2d = sum(v_.numel() * 2 + i_.numel() * 4 + u_.numel() * 4 for v_, i_, u_ in host_in)
    d2h = sum(x.numel() * 4 for o in out_h for x in o) + (score_h.numel() * 4 if wl.score else 0)

    hbm, tf_burst, tf_sus, peak_kind = peaks()
    gp = prof["gemm_prefill"]
    gd = prof["gemm_decode"]
    roof = None
    if gp["ms"] > 0:
        achieved = gp["flops"] / (gp["ms"] / 1e3) / 1e12
        roof = {"bound": "tensor", "kernel": "gemm_tc (prefill/score projections)",
                "achieved": achieved, "peak": tf_sus, "unit": "TFLOP/s", "frac": achieved / tf_sus,
                "peak_kind": f"{peak_kind} bf16 sustained (fp16 operands: same nominal dense rate as bf16)",
                "traffic": PROFILED_TRAFFIC["bytes"] if PROFILED_TRAFFIC else None,
                "traffic_launch": PROFILED_TRAFFIC,
                "launches": gp["launches"], "avg_launch_ms": gp["ms"] / max(1, gp["launches"])}
        # the q|k|v tile GEMMs multiply both halves of the activation pair, o, gate|up and
        # down hi alone: the MMAs issued are (1 + the paired share of the projection work) x
        # the algorithmic product
        sh = wl.shape
        d_, f_ = float(sh.d_model), float(sh.d_ffn)
        paired_share = (3.0 * d_ * d_) / (4.0 * d_ * d_ + 3.0 * f_ * d_)
        roof["issued_mma_frac"] = (1.0 + paired_share) * achieved / tf_sus
    roof_dec = None
    if gd["ms"] > 0:
        gbs = gd["bytes"] / (gd["ms"] / 1e3) / 1e9
        roof_dec = {"bound": "hbm", "kernel": "gemv_tc + stream-K reduction (decode projections)",
                    "achieved": gbs, "peak": hbm, "unit": "GB/s", "frac": gbs / hbm,
                    "peak_kind": f"{peak_kind} HBM copy",
                    "note": "each launch bracketed by events, which also stops it overlapping its neighbours",
                    "launches": gd["launches"], "avg_launch_ms": gd["ms"] / max(1, gd["launches"])}
    pre_fl = sum(w_["prefill_flops"] for w_ in works)
    dec_by = sum(w_["decode_bytes"] for w_ in works)
    phase_roof = {
        # the prefill runs ~0.2 s of back-to-back GEMMs every step under the power cap: its peak
        # is the sustained one; the fraction of the burst peak is given beside it
        "prefill": {"bound": "tensor", "tflop": pre_fl / 1e12, "ms": t_pre,
                    "achieved": pre_fl / (t_pre / 1e3) / 1e12, "peak": tf_sus, "unit": "TFLOP/s",
                    "frac": pre_fl / (t_pre / 1e3) / 1e12 / tf_sus,
                    "frac_of_burst": pre_fl / (t_pre / 1e3) / 1e12 / tf_burst,
                    "peak_kind": f"{peak_kind} bf16 sustained (fp16 operands: same nominal dense rate)",
                    "tflop_if_every_row_ran_every_layer": sum(w_["prefill_flops_all_rows"] for w_ in works) / 1e12},
        "decode": {"bound": "hbm", "gb": dec_by / 1e9, "ms": t_dec,
                   "achieved": dec_by / (t_dec / 1e3) / 1e9, "peak": hbm, "unit": "GB/s",
                   "frac": dec_by / (t_dec / 1e3) / 1e9 / hbm, "peak_kind": f"{peak_kind} HBM copy"},
    }
    if wl.turns > 1:
        phase_roof["decode"]["frac_per_turn"] = [round(w_["decode_bytes"] / (x / 1e3) / 1e9 / hbm, 3)
                                                 for w_, x in zip(works, t_dec_t)]
    if wl.score:
        sw = works[-1]
        phase_roof["score"] = {"bound": "hbm", "gb": sw["score_bytes"] / 1e9, "tflop": sw["score_flops"] / 1e12,
                               "ms": t_sc, "achieved": sw["score_bytes"] / (t_sc / 1e3) / 1e9, "peak": hbm,
                               "unit": "GB/s", "frac": sw["score_bytes"] / (t_sc / 1e3) / 1e9 / hbm,
                               "tflops": sw["score_flops"] / (t_sc / 1e3) / 1e12,
                               "peak_kind": f"{peak_kind} HBM copy"}
        # projections tensor-bound at 384 rows: floor = max(their flops at the sustained tensor
        # peak, the weights at HBM speed) + the K/V reads at HBM speed
        floor_ms = 1e3 * (max(sw["score_gemm_flops"] / (tf_sus * 1e12), sw["score_weight_bytes"] / (hbm * 1e9))
                          + (sw["score_bytes"] - sw["score_weight_bytes"]) / (hbm * 1e9))
        phase_roof["score"]["floor_ms"] = floor_ms
        phase_roof["score"]["frac_of_floor"] = floor_ms / t_sc

    n_gpus = world
    acts = wl.turns * B * A                     # action tokens per step
    value = n_gpus * acts / (ms_step / 1e3)
    line = {
        "metric": METRIC, "value": value, "unit": "action tokens/s", "n_gpus": n_gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "fp16 operands (bf16 weights converted once), fp32 accumulate",
        "data": "synthetic (seeded; random-init weights)",
        "config": workload_config(wl, n_gpus),
        "phases": phase,
        "roofline": roof, "roofline_decode": roof_dec, "phase_roofline": phase_roof,
        "e2e": {"value": n_gpus * acts / (e2e_ms / 1e3), "unit": "action tokens/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms},
        "gpu_launches": launches,
        "clocks": clk.summary(),
    }
    pol.close()
    if rank == 0 and not args.no_cpu_baseline:
        dt, prefix, threads = oracle_sample(wl, w_cpu)
        line["cpu_baseline"] = {"value": A / dt, "unit": "action tokens/s", "cores": threads,
                                "host_cpus": os.cpu_count(), "kind": "oracle",
                                "sample": f"1 of {B} envs (prefix {prefix} tokens): prefill + 7-token decode + score, fp64, {dt:.1f} s"}
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    if rank == 0:
        print(json.dumps(line))
    return 0


if __name__ == "__main__":
    sys.exit(main())
