"""Failure detection on the GPU without a fault: a bounded device wait that runs
out (a counter that nothing raises) gives up after its time limit, reports
MOLT_DEV_TIMEOUT through the status word, and leaves the context usable: the
next calls run and match the oracle."""
import time

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2607_21653_gb300 as molt  # noqa: E402
from oracle import molt_oracle as O  # noqa: E402
from workloads import random_problem  # noqa: E402

from parity import LOGP_ATOL, bf, np_, t  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    molt.build()
    molt.load()


def test_a_wait_that_runs_out_reports_a_timeout_and_the_context_survives():
    assert molt.device_status() == 0
    n0 = molt.kernel_launches()
    t0 = time.monotonic()
    molt.selftest_wait_timeout()
    flags = molt.device_status()
    elapsed = time.monotonic() - t0
    assert molt.kernel_launches() == n0 + 1
    assert flags & molt.DEV_FLAGS["timeout"], flags
    assert 2.0 < elapsed < 60.0, elapsed          # the 4 s bound, not a hang
    assert molt.device_status() == 0             # reading the word cleared it
    rng = np.random.default_rng(5)
    T, H, V = 300, 256, 1000
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.2)
    lp, ent = molt.token_logprobs(bf(h), bf(W), t(x), t(m))
    assert molt.device_status() == 0
    lp_ref, ent_ref = O.token_logprobs(O.widen_bf16(h), O.widen_bf16(W), x, m)
    assert np.abs(np_(lp) - lp_ref).max() <= LOGP_ATOL
    assert np.abs(np_(ent) - ent_ref).max() <= LOGP_ATOL
