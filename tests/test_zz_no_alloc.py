"""The allocation-free log-probability entry point against the allocating one.

molt_token_logprobs_fwd_noalloc is for callers that cannot let a library
allocate device memory (their runtime reserves the GPU's memory and hands it
out only through its own pool).  It keeps its scratch in a fixed device array
instead.  This test calls it through the C ABI twice in a row, on different
inputs, and checks each result against molt_token_logprobs_fwd within the
log-prob tolerance of the other parity tests.  At the array's limit
(MOLT_NOALLOC_MAX_TOKENS rows, the most vocab splits) it also compares sampled
rows with the fp64 oracle, without a mask or an entropy output, and checks that
the calls allocate nothing: the device's memory pool (the one cudaMallocAsync
draws from) sees no use and the free device memory does not change.  A batch
above the limit is refused before anything is launched.

The file name makes pytest collect it last; it also passes when run alone in
a fresh process (the first call then does the per-device set-up).
"""
import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2607_21653_gb300 as molt  # noqa: E402
from oracle import molt_oracle as O  # noqa: E402
from workloads import random_problem  # noqa: E402

from parity import LOGP_ATOL, bf, np_, t  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    molt.build()
    return molt.load()


def _noalloc(lib, h, W, x, m, want_entropy=True, logp=None):
    T, H = h.shape
    V = W.shape[0]
    if logp is None:
        logp = torch.full((T,), float("nan"), dtype=torch.float32, device=h.device)
    ent = torch.full((T,), float("nan"), dtype=torch.float32, device=h.device) if want_entropy else None
    st = lib.molt_token_logprobs_fwd_noalloc(
        ctypes.c_void_p(h.data_ptr()), ctypes.c_void_p(W.data_ptr()), ctypes.c_void_p(x.data_ptr()),
        ctypes.c_void_p(m.data_ptr()) if m is not None else None, T, H, V, ctypes.c_void_p(logp.data_ptr()),
        ctypes.c_void_p(ent.data_ptr()) if ent is not None else None,
        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 0, lib.molt_last_error().decode()
    return logp, ent


class _Pool:
    """The current memory pool of the device (what cudaMallocAsync draws from),
    read through the CUDA runtime the library itself loaded."""
    USED_MEM_HIGH = 8       # cudaMemPoolAttrUsedMemHigh
    RESERVED_MEM_HIGH = 6   # cudaMemPoolAttrReservedMemHigh

    def __init__(self):
        self.rt = ctypes.CDLL("libcudart.so.13")
        self.pool = ctypes.c_void_p()
        assert self.rt.cudaDeviceGetMemPool(ctypes.byref(self.pool), torch.cuda.current_device()) == 0

    def reset_high_water(self):
        for attr in (self.USED_MEM_HIGH, self.RESERVED_MEM_HIGH):
            zero = ctypes.c_uint64(0)
            assert self.rt.cudaMemPoolSetAttribute(self.pool, attr, ctypes.byref(zero)) == 0

    def high_water(self):
        out = []
        for attr in (self.USED_MEM_HIGH, self.RESERVED_MEM_HIGH):
            v = ctypes.c_uint64(0)
            assert self.rt.cudaMemPoolGetAttribute(self.pool, attr, ctypes.byref(v)) == 0
            out.append(int(v.value))
        return out


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


def test_noalloc_at_its_limit_allocates_nothing(lib):
    """T = MOLT_NOALLOC_MAX_TOKENS at the mid workload's H and V: every vocab
    split the array holds is in use.  No mask and no entropy output.  Two calls
    in a row (the second on other hidden states) against the allocating call,
    sampled rows against the oracle, and no allocation by either call."""
    T, H, V = molt.NOALLOC_MAX_TOKENS, 2048, 32000
    rng = np.random.default_rng(2024)
    h, W, x, _ = random_problem(rng, T, H, V, mask_frac=0.0, w_std=0.02)
    Wd, xd = bf(W), t(x)
    hds = [bf(h), bf(h[::-1].copy())]
    outs = [torch.full((T,), float("nan"), dtype=torch.float32, device=Wd.device) for _ in hds]
    _noalloc(lib, hds[0][:128], Wd, xd[:128], None, want_entropy=False)     # per-device set-up done
    torch.cuda.synchronize()
    pool = _Pool()
    pool.reset_high_water()             # the high-water marks drop to the current use
    base = pool.high_water()
    free0 = torch.cuda.mem_get_info()[0]
    for hd, lp in zip(hds, outs):
        _noalloc(lib, hd, Wd, xd, None, want_entropy=False, logp=lp)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    assert pool.high_water() == base, "a call allocated from the device's memory pool"
    assert molt.device_status() == 0
    W64 = O.widen_bf16(W)
    for k, (hd, lp) in enumerate(zip(hds, outs)):
        lp_ref, _ = molt.token_logprobs(hd, Wd, xd, None, want_entropy=False)
        assert molt.device_status() == 0
        got, ref = np_(lp), np_(lp_ref)
        assert np.isfinite(got).all()
        assert np.abs(got - ref).max() <= LOGP_ATOL
        rows = np.unique(np.concatenate([rng.choice(T, 48, replace=False), [0, T - 1]]))
        h_src = h if k == 0 else h[::-1]
        lp_o, _ = O.token_logprobs(O.widen_bf16(h_src[rows]), W64, x[rows], None)
        assert np.abs(got[rows] - lp_o).max() <= LOGP_ATOL


def test_noalloc_python_wrapper(lib):
    """The binding's token_logprobs_noalloc reaches the same entry point and
    refuses a batch above the limit it reads from the header."""
    rng = np.random.default_rng(7)
    h, W, x, m = random_problem(rng, 640, 128, 1000, mask_frac=0.2, w_std=0.05)
    hd, Wd, xd, md = bf(h), bf(W), t(x), t(m)
    lp, ent = molt.token_logprobs_noalloc(hd, Wd, xd, md)
    lp_ref, ent_ref = molt.token_logprobs(hd, Wd, xd, md)
    assert molt.device_status() == 0
    assert np.abs(np_(lp) - np_(lp_ref)).max() <= LOGP_ATOL
    assert np.abs(np_(ent) - np_(ent_ref)).max() <= LOGP_ATOL
    with pytest.raises(molt.MoltError):
        big = molt.NOALLOC_MAX_TOKENS + 1
        molt.token_logprobs_noalloc(bf(np.zeros((big, 128), np.uint16)), Wd, t(np.zeros(big, np.int32)))
