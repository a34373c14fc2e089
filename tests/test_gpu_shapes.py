"""Seeded shape fuzzing of the policy-loss call against the fp64 oracle: token
counts that leave 1-3 tiles of the last quad empty, vocabularies with ragged
512-column blocks, H from 256 (two jobs per unit) upward, both the cluster
backward (H % 128 == 0, a last 128-column job when H % 256 == 128) and the
single-CTA one, the deterministic schedule, and caller-provided workspaces."""
import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2607_21653_gb300 as molt  # noqa: E402
from oracle import molt_oracle as O  # noqa: E402
from workloads import random_problem  # noqa: E402

from parity import LOGP_ATOL, assert_grad_close, assert_loss_close, behavior_from_oracle, bf, np_, t  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    molt.build()
    molt.load()


def _cases():
    rng = np.random.default_rng(2607)
    out = []
    for i in range(10):
        H = int(rng.choice([256, 384, 512, 640, 768, 896, 1024, 1280, 320]))
        T = int(rng.integers(1, 1800))
        V = int(rng.integers(1, 7000))
        out.append((i, T, H, V, bool(i % 3 == 0) and H % 128 == 0))
    return out


@pytest.mark.parametrize("i,T,H,V,det", _cases())
def test_random_shapes(i, T, H, V, det):
    rng = np.random.default_rng(100 + i)
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=float(rng.uniform(0.0, 0.6)), w_std=0.05)
    m[0] = 1
    adv = rng.standard_normal(T).astype(np.float32)
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    b = behavior_from_oracle(h64, W64, x, 0.3, 0.2, 0.28, 7 + i)
    if det:
        out = molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.28, deterministic=True)
    else:
        out = molt.policy_loss_fwd_bwd(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.28)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    ref = O.policy_loss(h64, W64, x, b.astype(np.float64), adv.astype(np.float64), m, 0.2, 0.28)
    ref["_adv"] = adv.astype(np.float64)
    assert_loss_close(float(out["loss"].item()), ref)
    assert np.abs(np_(out["logp"]) - ref["logp"]).max() <= LOGP_ATOL
    dh = np_(out["dhidden"])
    assert (dh[m == 0] == 0).all()
    assert_grad_close(dh, ref["dH"], f"dhidden case {i}")
    assert_grad_close(np_(out["dW"]), ref["dW"], f"dW case {i}")


@pytest.mark.parametrize("V", [18986, 19243])
def test_vocab_split_with_side_kernel(V):
    """The raster backward splits the vocabulary when that evens out the work:
    the cluster kernel takes the first whole 512-column blocks and the
    single-CTA kernel the rest, concurrently on a side stream over the SMs that
    no cluster of four can use.  With 700 tokens and these V (on a GB300: 36
    clusters, 8 spare SMs) the cluster kernel keeps 36 blocks and the side
    kernel takes the last 554 or 811 columns.  Targets are placed in both
    slices; the deterministic schedule does not split; with V = 18432 (whole
    blocks, nothing to even out) the call launches one kernel fewer."""
    T, H = 700, 256
    rng = np.random.default_rng(V)
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.2, w_std=0.05)
    m[:64] = 1
    x[:32] = rng.integers(V - 500, V, 32)     # in the side kernel's slice
    x[32:64] = rng.integers(0, 700, 32)       # in the cluster kernel's first block
    adv = rng.standard_normal(T).astype(np.float32)
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    b = behavior_from_oracle(h64, W64, x, 0.3, 0.2, 0.28, 11)
    args = (bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.28)
    n0 = molt.kernel_launches()
    out = molt.policy_loss_fwd_bwd_ex(*args, deterministic=False)
    n_split = molt.kernel_launches() - n0
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    ref = O.policy_loss(h64, W64, x, b.astype(np.float64), adv.astype(np.float64), m, 0.2, 0.28)
    ref["_adv"] = adv.astype(np.float64)
    assert_loss_close(float(out["loss"].item()), ref)
    assert np.abs(np_(out["logp"]) - ref["logp"]).max() <= LOGP_ATOL
    assert_grad_close(np_(out["dhidden"]), ref["dH"], f"dhidden V={V}")
    dW = np_(out["dW"])
    assert_grad_close(dW, ref["dW"], f"dW V={V}")
    assert_grad_close(dW[V - 1024:], ref["dW"][V - 1024:], f"dW last columns V={V}")
    # accumulating into a caller's dW: both kernels add onto it
    dW0 = torch.randn(V, H, device="cuda", generator=torch.Generator(device="cuda").manual_seed(V))
    acc = dW0.clone()
    molt.policy_loss_fwd_bwd_ex(*args, deterministic=False, dW=acc, accumulate_dW=True)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    assert_grad_close(np_(acc - dW0), ref["dW"], f"dW accumulated V={V}")
    det = molt.policy_loss_fwd_bwd_ex(*args, deterministic=True)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    assert_grad_close(np_(det["dW"]), ref["dW"], f"dW deterministic V={V}")
    # 36 whole blocks: the same kernels but the side one
    hs, Ws = h, W[:18432]
    xs = np.minimum(x, 18431).astype(x.dtype)
    n0 = molt.kernel_launches()
    molt.policy_loss_fwd_bwd_ex(bf(hs), bf(Ws), t(xs), t(b), t(adv), t(m), 0.2, 0.28, deterministic=False)
    n_plain = molt.kernel_launches() - n0
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    assert n_split in (n_plain, n_plain + 1)
    if torch.cuda.get_device_properties(0).multi_processor_count == 152:
        assert n_split == n_plain + 1


@pytest.mark.parametrize("H,V", [(384, 3000), (640, 4133), (896, 18986)])
def test_half_width_last_job(H, V):
    """H % 256 == 128: the cluster backward's last dH / dW job is 128 columns
    wide.  Parity with the oracle on the raster schedule (V = 18986 also splits
    the vocabulary with the side kernel) and on the deterministic one, which is
    bitwise reproducible."""
    T = 900
    rng = np.random.default_rng(H + V)
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.25, w_std=0.05)
    m[0] = 1
    adv = rng.standard_normal(T).astype(np.float32)
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    b = behavior_from_oracle(h64, W64, x, 0.3, 0.2, 0.28, H)
    ref = O.policy_loss(h64, W64, x, b.astype(np.float64), adv.astype(np.float64), m, 0.2, 0.28)
    ref["_adv"] = adv.astype(np.float64)
    args = (bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.28)
    runs = []
    for det in (False, True, True):
        out = molt.policy_loss_fwd_bwd_ex(*args, deterministic=det)
        torch.cuda.synchronize()
        assert molt.device_status() == 0
        assert_loss_close(float(out["loss"].item()), ref)
        assert_grad_close(np_(out["dhidden"]), ref["dH"], f"dhidden H={H} det={det}")
        assert_grad_close(np_(out["dW"]), ref["dW"], f"dW H={H} det={det}")
        runs.append(out)
    for k in ("dhidden", "dW"):
        np.testing.assert_array_equal(np_(runs[1][k]).view(np.uint8), np_(runs[2][k]).view(np.uint8), err_msg=k)


def test_caller_workspace_and_too_small_workspace():
    rng = np.random.default_rng(3)
    T, H, V = 700, 512, 3000
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.2, w_std=0.05)
    m[0] = 1
    adv = rng.standard_normal(T).astype(np.float32)
    b = behavior_from_oracle(O.widen_bf16(h), O.widen_bf16(W), x, 0.3, 0.2, 0.2, 5)
    opts = molt.LossOptions(0.0, 0.0, None, None, 0.0, 0.0, 1)
    need = molt.load().molt_policy_loss_workspace_bytes_ex(T, H, V, ctypes.byref(opts))
    assert need > molt.load().molt_policy_loss_workspace_bytes(T, H, V)
    ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    a = molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.2, deterministic=True,
                                    workspace=ws)
    c = molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.2, deterministic=True)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    assert torch.equal(a["dW"].view(torch.int32), c["dW"].view(torch.int32))
    small = torch.empty(need - 4096, dtype=torch.uint8, device="cuda")
    with pytest.raises(molt.MoltError):
        molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.2, deterministic=True,
                                    workspace=small)


def test_policy_loss_captured_in_a_cuda_graph():
    """The loss call captured into a CUDA graph and replayed gives the eager
    call's results.  The eager call runs first on the same stream, so the
    stream's workspace and side stream exist and the vocab split (chosen for
    700 tokens and V = 18986 on a GB300) forks onto the side stream and joins
    back inside the captured graph."""
    T, H, V = 700, 256, 18986
    rng = np.random.default_rng(77)
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.2, w_std=0.05)
    m[0] = 1
    adv = rng.standard_normal(T).astype(np.float32)
    b = behavior_from_oracle(O.widen_bf16(h), O.widen_bf16(W), x, 0.3, 0.2, 0.28, 78)
    args = (bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.28)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        eager = molt.policy_loss_fwd_bwd(*args, stream=s)
    s.synchronize()
    assert molt.device_status() == 0
    eager = {k: v.clone() for k, v in eager.items() if v is not None}
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        out = molt.policy_loss_fwd_bwd(*args, stream=s)
    for _ in range(2):
        g.replay()
        torch.cuda.synchronize()
        assert molt.device_status() == 0
        np.testing.assert_array_equal(np_(out["loss"]), np_(eager["loss"]))
        np.testing.assert_array_equal(np_(out["logp"]), np_(eager["logp"]))
        assert_grad_close(np_(out["dhidden"]), np_(eager["dhidden"]).astype(np.float64), "dhidden (graph replay)")
        assert_grad_close(np_(out["dW"]), np_(eager["dW"]).astype(np.float64), "dW (graph replay)")


def test_concurrent_calls_on_two_streams():
    """Two different problems issued on two streams at once: each result equals
    the same problem run alone (the binding gives each stream its workspace)."""
    probs = []
    for i in range(2):
        rng = np.random.default_rng(40 + i)
        T, H, V = 900, 512, 3000 + 500 * i
        h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.2, w_std=0.05)
        m[0] = 1
        adv = rng.standard_normal(T).astype(np.float32)
        b = behavior_from_oracle(O.widen_bf16(h), O.widen_bf16(W), x, 0.3, 0.2, 0.2, 50 + i)
        probs.append((bf(h), bf(W), t(x), t(b), t(adv), t(m)))
    alone = [molt.policy_loss_fwd_bwd(*p, 0.2, 0.2) for p in probs]
    torch.cuda.synchronize()
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    together = []
    for p, s in zip(probs, streams):
        with torch.cuda.stream(s):
            together.append(molt.policy_loss_fwd_bwd(*p, 0.2, 0.2, stream=s))
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    for a, c in zip(alone, together):
        np.testing.assert_array_equal(np_(a["loss"]), np_(c["loss"]))
        np.testing.assert_array_equal(np_(a["logp"]), np_(c["logp"]))
        assert_grad_close(np_(c["dhidden"]), np_(a["dhidden"]).astype(np.float64), "dhidden on a second stream")
        assert_grad_close(np_(c["dW"]), np_(a["dW"]).astype(np.float64), "dW on a second stream")


def test_deterministic_calls_on_two_streams():
    """Two deterministic calls issued on two streams at once.  Their clusters
    wait on one another's turns, so each launch needs all its clusters resident:
    the launch enqueued first takes the SMs, the other's clusters start as its
    clusters leave.  Each result equals the same problem run alone, bit for bit,
    and no wait times out."""
    probs = []
    for i in range(2):
        rng = np.random.default_rng(60 + i)
        T, H, V = 3000, 512, 9000 + 1000 * i
        h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.2, w_std=0.05)
        m[0] = 1
        adv = rng.standard_normal(T).astype(np.float32)
        b = behavior_from_oracle(O.widen_bf16(h), O.widen_bf16(W), x, 0.3, 0.2, 0.2, 70 + i)
        probs.append((bf(h), bf(W), t(x), t(b), t(adv), t(m)))
    alone = [molt.policy_loss_fwd_bwd_ex(*p, 0.2, 0.2, deterministic=True) for p in probs]
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    together = []
    for p, s in zip(probs, streams):
        with torch.cuda.stream(s):
            together.append(molt.policy_loss_fwd_bwd_ex(*p, 0.2, 0.2, deterministic=True, stream=s))
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    for a, c in zip(alone, together):
        np.testing.assert_array_equal(np_(c["dW"]).view(np.uint32), np_(a["dW"]).view(np.uint32))
        np.testing.assert_array_equal(np_(c["dhidden"]).view(np.uint16), np_(a["dhidden"]).view(np.uint16))
