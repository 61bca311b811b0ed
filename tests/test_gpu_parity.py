"""End-to-end parity of the rollout workloads against the fp64 oracle, through the C ABI.

tiny and small: every env.  7B-shaped workloads: two envs (the first and the longest), the
GPU running the full batch."""
import pytest
import torch

from paper_2505_18719_gb300 import inputs as I
from tests import parity as P

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    from paper_2505_18719_gb300 import build
    build.build()


def _assert_ok(reports):
    for r in reports:
        print(r)
    assert reports and all(r.ok() for r in reports), reports


def test_tiny_b4_parity():
    _assert_ok(P.run_parity(I.WORKLOADS["tiny_b4"]))


def test_tiny_b4_parity_greedy_and_hot():
    for T in (0.0, 1.5):
        _assert_ok(P.run_parity(I.WORKLOADS["tiny_b4"], temperature=T))


def test_small_b16_parity_with_score():
    _assert_ok(P.run_parity(I.WORKLOADS["small_b16_score"]))


@pytest.fixture(scope="module")
def llama_weights():
    w = I.make_weights(I.LLAMA7B)
    return w, P.weights_to_device(w)


@pytest.mark.slow
def test_7b_b16_parity(llama_weights):
    w, wd = llama_weights
    _assert_ok(P.run_parity(I.WORKLOADS["7b_b16"], w, wd, n_check=2, cache_f64=False))


@pytest.mark.slow
def test_7b_b64_ragged_score_parity(llama_weights):
    w, wd = llama_weights
    _assert_ok(P.run_parity(I.WORKLOADS["7b_b64_ragged_score"], w, wd, n_check=2, cache_f64=False))


@pytest.mark.slow
def test_7b_b256_multiturn_parity(llama_weights):
    w, wd = llama_weights
    _assert_ok(P.run_parity(I.WORKLOADS["7b_b256_multiturn"], w, wd, n_check=2, cache_f64=False))


@pytest.mark.slow
def test_7b_b256_multiturn_t15_with_resets_parity(llama_weights):
    """Four turns with 64 text ids re-sent per turn (up to 1307 positions), T = 1.5, and three
    envs (one of them compared) whose episode ends after turn 1: their turn-2 prefill starts a
    fresh context in the same batch as the others' appends."""
    w, wd = llama_weights
    _assert_ok(P.run_parity(I.WORKLOADS["7b_b256_multiturn_t15"], w, wd, n_check=2, cache_f64=False))
