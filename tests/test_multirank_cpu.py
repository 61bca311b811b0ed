"""Multi-rank path on the CPU (gloo, world size 2).

Environments are independent (paper §3.5: each worker owns its own set of environments), so
the rollout shards across ranks with no collective in the data path.  Two gloo ranks each run
the oracle on half of the envs of the tiny workload; the gathered tokens / log-probs / logits
must equal a single-process run over all envs, bit for bit.  The bench's max-over-ranks
timing reduction is exercised the same way."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rollout(envs, wl, w):
    import oracle.vla_oracle as O
    from paper_2505_18719_gb300 import inputs as I
    inp = I.make_turn_inputs(wl, 0)
    orc = O.Oracle(O.shape_from(wl.shape), w, wl.batch)
    orc.prefill(envs, [inp.visual[b] for b in envs], [inp.ids[b, :int(inp.lengths[b])].tolist() for b in envs])
    out = orc.decode(envs, inp.uniforms[envs], wl.temperature)
    return np.concatenate([out["tokens"].astype(np.float64).ravel(), out["logprobs"].ravel(),
                           out["logits"].ravel()])


def _worker(rank, world, port, q):
    import sys
    sys.path.insert(0, ROOT)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        from paper_2505_18719_gb300 import inputs as I
        import bench
        wl = I.WORKLOADS["tiny_b4"]
        w = I.make_weights(wl.shape, wl.weight_seed)
        per = wl.batch // world
        mine = list(range(rank * per, (rank + 1) * per))
        local = torch.from_numpy(_rollout(mine, wl, w))
        parts = [torch.empty_like(local) for _ in range(world)]
        dist.all_gather(parts, local)
        slowest = bench.max_over_ranks(float(rank + 1), dist, device="cpu")
        if rank == 0:
            q.put((torch.cat(parts).numpy(), slowest))
    finally:
        dist.destroy_process_group()


def test_env_sharding_over_two_gloo_ranks_matches_one_process():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    gathered, slowest = q.get(timeout=300)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    from paper_2505_18719_gb300 import inputs as I
    wl = I.WORKLOADS["tiny_b4"]
    w = I.make_weights(wl.shape, wl.weight_seed)
    # one process, all envs: the same numbers in the same (env-major) layout
    ref = [_rollout([b], wl, w) for b in range(wl.batch)]
    half = [_rollout([0, 1], wl, w), _rollout([2, 3], wl, w)]
    assert np.array_equal(gathered, np.concatenate(half))
    # and each env alone gives the same values as inside its shard (batch invariance)
    t0 = half[0]
    toks = t0[: 2 * 7]
    assert np.array_equal(toks[:7], ref[0][:7]) and np.array_equal(toks[7:], ref[1][:7])
    assert slowest == 2.0
