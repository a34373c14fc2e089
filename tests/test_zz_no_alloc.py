"""The allocation-free log-probability entry point against the allocating one.

molt_token_logprobs_fwd_noalloc is for callers that cannot let a library
allocate device memory (their runtime reserves the GPU's memory and hands it
out only through its own pool).  It keeps its scratch in a fixed device array
instead.  This test calls it through the C ABI twice in a row, on different
inputs, and checks each result against molt_token_logprobs_fwd within the
log-prob tolerance of the other parity tests.  It also checks that a batch above
the array's limit is refused before anything is launched.

The file name makes pytest collect it last; it also passes when run alone in
a fresh process (the first call then does the per-device set-up).
"""
import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2607_21653_gb300 as molt  # noqa: E402
from workloads import random_problem  # noqa: E402

from parity import LOGP_ATOL, bf, np_, t  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    molt.build()
    return molt.load()


def _noalloc(lib, h, W, x, m):
    T, H = h.shape
    V = W.shape[0]
    logp = torch.full((T,), float("nan"), dtype=torch.float32, device=h.device)
    ent = torch.full((T,), float("nan"), dtype=torch.float32, device=h.device)
    st = lib.molt_token_logprobs_fwd_noalloc(
        ctypes.c_void_p(h.data_ptr()), ctypes.c_void_p(W.data_ptr()), ctypes.c_void_p(x.data_ptr()),
        ctypes.c_void_p(m.data_ptr()) if m is not None else None, T, H, V, ctypes.c_void_p(logp.data_ptr()),
        ctypes.c_void_p(ent.data_ptr()), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 0, lib.molt_last_error().decode()
    return logp, ent


@pytest.mark.parametrize("first,second", [((1000, 192, 3000, 0.3), (257, 64, 777, 0.0))])
def test_noalloc_matches_allocating_call_twice(lib, first, second):
    for k, (T, H, V, mf) in enumerate((first, second)):
        rng = np.random.default_rng(100 + k)
        h, W, x, m = random_problem(rng, T, H, V, mask_frac=mf, w_std=0.05)
        hd, Wd, xd, md = bf(h), bf(W), t(x), t(m)
        lp_na, ent_na = _noalloc(lib, hd, Wd, xd, md)
        lp_ref, ent_ref = molt.token_logprobs(hd, Wd, xd, md)
        assert molt.device_status() == 0
        lp_na, ent_na, lp_ref, ent_ref = np_(lp_na), np_(ent_na), np_(lp_ref), np_(ent_ref)
        assert np.isfinite(lp_na).all() and np.isfinite(ent_na).all()
        assert np.abs(lp_na - lp_ref).max() <= LOGP_ATOL
        assert np.abs(ent_na - ent_ref).max() <= LOGP_ATOL
        assert (lp_na[m == 0] == 0).all() and (ent_na[m == 0] == 0).all()


def test_noalloc_rejects_batches_above_the_limit(lib):
    fake = ctypes.c_void_p(0x1000)   # never dereferenced: the size check comes first
    st = lib.molt_token_logprobs_fwd_noalloc(fake, fake, fake, None, molt.NOALLOC_MAX_TOKENS + 1, 64, 100, fake,
                                             None, None)
    assert molt.STATUS[st] == "MOLT_ERR_UNSUPPORTED_SHAPE"
    assert "at most" in lib.molt_last_error().decode()
