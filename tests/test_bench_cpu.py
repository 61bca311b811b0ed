"""bench.py's host-side pieces, on the CPU: the algorithmic work behind the phase rooflines
matches the arithmetic of the 7B configurations worked by hand (6.476e9 matrix parameters;
K+V per position and layer as cached: 16 KB of fp16 parts + 4 KB of 4-bit residual codes),
and both bench arms describe the same workload."""
import bench
from paper_2505_18719_gb300 import inputs as I

P7B = 32 * (4 * 4096 * 4096 + 3 * 11008 * 4096)   # 6.476e9 matrix parameters
KV_TOK = 2.5 * 2 * 4096 * 32                        # bytes of cached K and V per position, all layers


def _work(name, turn=0):
    wl = I.WORKLOADS[name]
    lens = I.make_turn_inputs(wl, turn).lengths.tolist()
    return wl, lens, bench.phase_work(wl.shape, [0] * wl.batch, [wl.n_visual + int(x) for x in lens])


def test_parameter_count():
    assert abs(P7B - 6.476e9) < 1e6


def test_prefill_flops_16_envs_288_rows():
    wl, lens, w = _work("7b_b16")
    T = 16 * 288
    dense = 2.0 * P7B * T
    attn = 32 * 16 * 2.0 * 4096 * 288 * 289              # causal QK^T + PV per layer
    assert abs(w["prefill_flops_all_rows"] - (dense + attn)) < 1e6
    assert abs(w["prefill_flops_all_rows"] / 1e12 - 60.0) < 0.1
    # the pruned last layer needs only q|k|v for every row
    assert w["prefill_flops"] < w["prefill_flops_all_rows"]


def test_decode_bytes_16_and_64_envs():
    wl, lens, w = _work("7b_b16")
    want = sum(2.0 * P7B + sum((288 + i) * KV_TOK for _ in range(16)) + 16 * KV_TOK + 2.0 * 256 * 4096
               for i in range(1, 7)) + 2.0 * 256 * 4096
    assert abs(w["decode_bytes"] - want) < 1.0
    assert abs(w["decode_bytes"] / 1e9 - 96.1) < 0.3
    wl, lens, w = _work("7b_b64_ragged_score")
    assert abs(w["decode_bytes"] / 1e9 - 151.2) < 0.5


def test_score_work_64_envs():
    wl, lens, w = _work("7b_b64_ragged_score")
    assert abs(w["score_flops"] / 1e12 - 4.97) < 0.1                 # 2 P x 384 rows + attention
    assert abs(w["score_bytes"] / 1e9 - (12.95 + 12.6)) < 0.5          # weights + cached K/V
    # the projections alone: 2 P x 64 envs x 6 rows; the weights (+ the 256 head rows)
    assert abs(w["score_gemm_flops"] - 2.0 * P7B * 64 * 6) < 1.0
    assert abs(w["score_weight_bytes"] - (2.0 * P7B + 2.0 * 256 * 4096)) < 1.0


def test_both_arms_share_the_config():
    wl = I.WORKLOADS["7b_b64_ragged_score"]
    c = bench.workload_config(wl, 1)
    assert c["workload"] == wl.name and c["batch_per_gpu"] == 64 and c["text_len"] == "U{16..48}"
    assert c["step"] == "reset + prefill + 7-token decode + score"
    c5 = bench.workload_config(I.WORKLOADS["7b_b256_multiturn"], 2)
    assert c5["turns"] == 4 and c5["append_visual"] == 256 and c5["parallelism"] == "replicas x2"
