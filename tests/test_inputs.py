"""The seeded input generator: published SplitMix64 outputs, determinism, distributions."""
import numpy as np
import torch

from paper_2505_18719_gb300 import inputs as I


def test_splitmix64_published_outputs():
    # SplitMix64 from state 0: the reference outputs published with the generator
    assert I.splitmix64(3, 0) == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_counter_based_prefix_stable():
    a = I.normal_bf16((1000,), 5, 9, 1.0)
    b = I.normal_bf16((300_000,), 5, 9, 1.0)     # many threads, other chunking
    assert torch.equal(a, b[:1000])
    assert not torch.equal(I.normal_bf16((1000,), 5, 10, 1.0), a)
    assert not torch.equal(I.normal_bf16((1000,), 6, 9, 1.0), a)


def test_distributions():
    x = I.normal_bf16((1_000_000,), 1, 1, 0.02).float().numpy()
    assert abs(x.mean()) < 1e-4 and abs(x.std() - 0.02) < 2e-4
    u = I.uniform_f32((1_000_000,), 1, 2).numpy()
    assert u.min() > 0 and u.max() < 1 and abs(u.mean() - 0.5) < 2e-3
    m = u.astype(np.float64) * 2 ** 23 - 0.5
    assert np.array_equal(m, np.round(m))           # (m + 0.5) 2^-23, m integer, exact in fp32
    assert u.min() >= 2.0 ** -24 and u.max() <= 1 - 2.0 ** -24
    r = I.randint_i32((100_000,), 1, 3, 16, 48).numpy()
    assert r.min() == 16 and r.max() == 48
    assert np.all(np.bincount(r - 16, minlength=33) > 2500)


def test_workload_inputs_shapes():
    wl = I.WORKLOADS["7b_b64_ragged_score"]
    # per-turn inputs only (no 7B weights here)
    t = I.make_turn_inputs(wl, 0)
    assert t.visual.shape == (64, 256, 4096) and t.visual.dtype == torch.bfloat16
    assert t.uniforms.shape == (64, 7, 256)
    assert int(t.lengths.min()) >= 16 and int(t.lengths.max()) <= 48
    assert int(t.ids.max()) < 32064 - 256
    for b in range(64):
        assert int(t.ids[b, int(t.lengths[b]):].abs().sum()) == 0
