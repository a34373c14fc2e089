"""GPU parity of the extended objective (KL to a reference policy, entropy
bonus, sequence-level importance gate; Sec. 4.5) against the fp64 oracle,
through molt_policy_loss_fwd_bwd_ex, on both backward kernels (H a multiple of
256 runs on CTA pairs, other H on single CTAs).

Gate cases are built so that no decision sits near a boundary: each sequence's
mean log-ratio is placed at least 0.3 (in log space) from the band edges, and
the per-token ratios of accepted sequences stay well inside the clip band, far
beyond the 2e-3 log-prob tolerance between the fp32 kernel and the oracle.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2607_21653_gb300 as molt  # noqa: E402
from oracle import molt_oracle as O  # noqa: E402
from workloads import random_problem  # noqa: E402

from parity import LOGP_ATOL, LOSS_RTOL, assert_grad_close, behavior_from_oracle, bf, np_, t  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    molt.build()
    molt.load()


def _run(h, W, x, m, b, adv, eps_lo, eps_hi, denom=0.0, **kw):
    out = molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(b), t(adv), t(m), eps_lo, eps_hi, denom=denom,
                                      **{k: (t(v) if isinstance(v, np.ndarray) else v) for k, v in kw.items()})
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    okw = {k: v for k, v in kw.items()}
    if "seq_of_token" in okw:
        okw["gate_lo"] = kw.get("gate_lo", 0.0)
        okw["gate_hi"] = kw.get("gate_hi", float("inf"))
    ref = O.policy_loss_ex(O.widen_bf16(h), O.widen_bf16(W), x, b.astype(np.float64), adv.astype(np.float64), m,
                           eps_lo, eps_hi, denom=denom if denom > 0 else None, **okw)
    return out, ref


def _check(out, ref, m, adv, kl_coef=0.0, entropy_coef=0.0):
    act = m != 0
    D = ref["denom"]
    scale = max(abs(ref["loss"]), float((np.abs(ref["ratio"] * adv) + kl_coef * ref["kl"]
                                         + abs(entropy_coef) * ref["entropy"])[act].sum() / D))
    L = float(out["loss"].item())
    assert abs(L - ref["loss"]) <= LOSS_RTOL * scale, (L, ref["loss"], scale)
    assert np.abs(np_(out["logp"]) - ref["logp"]).max() <= LOGP_ATOL
    assert np.abs(np_(out["entropy"]) - ref["entropy"]).max() <= LOGP_ATOL
    tl = np_(out["token_loss"])
    np.testing.assert_allclose(tl[act], ref["token_loss"][act], rtol=5e-3, atol=2e-5)
    assert (tl[~act] == 0).all()
    dh = np_(out["dhidden"])
    assert (dh[~act] == 0).all()
    assert_grad_close(dh, ref["dH"], "dhidden")
    assert_grad_close(np_(out["dW"]), ref["dW"], "dW")
    st = molt.stats_dict(out["stats"])
    assert st["n_active"] == int(act.sum()) and st["denom"] == D
    keep = ref["gate"] != 0
    assert st["n_tokens_rejected"] == int((act & ~keep).sum())
    assert st["n_clip_low"] == int((ref["clipped"] & (adv < 0) & act & keep).sum())
    assert st["n_clip_high"] == int((ref["clipped"] & (adv > 0) & act & keep).sum())
    kl_sum = float((ref["kl"] * keep)[act].sum())
    assert abs(st["sum_kl"] - kl_sum) <= 1e-2 * max(1e-6, kl_sum) + 1e-6 * act.sum()
    # the backward's rows: accepted active rows with a nonzero coefficient (an
    # entropy bonus gives every accepted row one)
    live = act & keep & ((ref["coef"] != 0) | (entropy_coef != 0.0))
    assert st["n_grad_rows"] == int(live.sum())
    assert (dh[act & ~live] == 0).all()
    return st


SHAPES = [(300, 128, 1000), (513, 192, 4133), (300, 256, 1000), (640, 512, 2304), (1, 256, 7)]


@pytest.mark.parametrize("T,H,V", SHAPES)
def test_options_disabled_match_plain_loss(T, H, V):
    rng = np.random.default_rng(T + H)
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.2, w_std=0.05)
    m[0] = 1
    adv = rng.standard_normal(T).astype(np.float32)
    b = behavior_from_oracle(O.widen_bf16(h), O.widen_bf16(W), x, 0.3, 0.2, 0.28, T)
    ex = molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.28)
    pl = molt.policy_loss_fwd_bwd(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.28)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    # the row quantities run the same fp32 arithmetic: identical bits
    for k in ("loss", "logp", "entropy", "token_loss"):
        np.testing.assert_array_equal(np_(ex[k]), np_(pl[k]), err_msg=k)
    assert_grad_close(np_(ex["dhidden"]), np_(pl["dhidden"]).astype(np.float64), "dhidden")
    assert_grad_close(np_(ex["dW"]), np_(pl["dW"]).astype(np.float64), "dW")


@pytest.mark.parametrize("T,H,V", SHAPES)
def test_kl_and_entropy_terms(T, H, V):
    rng = np.random.default_rng(3 * T + H)
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.25, w_std=0.05)
    m[0] = 1
    adv = rng.standard_normal(T).astype(np.float32)
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    b = behavior_from_oracle(h64, W64, x, 0.3, 0.2, 0.28, T + 1)
    lp, _ = O.token_logprobs(h64, W64, x, None)
    ref_logp = (lp + rng.normal(0, 0.4, T)).astype(np.float32)
    out, ref = _run(h, W, x, m, b, adv, 0.2, 0.28, kl_coef=0.2, ref_logp=ref_logp, entropy_coef=0.05)
    _check(out, ref, m, adv, 0.2, 0.05)


@pytest.mark.parametrize("T,H,V", [(400, 128, 3000), (400, 256, 3000)])
@pytest.mark.parametrize("term", ["entropy", "kl"])
def test_single_term_without_advantage(T, H, V, term):
    """With A = 0 the surrogate's coefficient is 0 on every row: the whole
    gradient comes from the extra term, and no tile may be skipped."""
    rng = np.random.default_rng(T + H + len(term))
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.1, w_std=0.2)
    m[0] = 1
    adv = np.zeros(T, np.float32)
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    lp, _ = O.token_logprobs(h64, W64, x, None)
    b = lp.astype(np.float32)
    if term == "entropy":
        kw = dict(entropy_coef=0.1)
    else:
        kw = dict(kl_coef=0.5, ref_logp=(lp + rng.normal(0, 0.5, T)).astype(np.float32))
    out, ref = _run(h, W, x, m, b, adv, 0.2, 0.2, **kw)
    assert np.abs(ref["dH"]).max() > 0
    _check(out, ref, m, adv, kw.get("kl_coef", 0.0), kw.get("entropy_coef", 0.0))


def _gated_problem(rng, H, V, lengths, mask_frac=0.2):
    T = int(sum(lengths))
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=mask_frac, w_std=0.05)
    seq = np.repeat(np.arange(len(lengths)), lengths).astype(np.int32) * 3 + 7   # sorted, not dense
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    lp, _ = O.token_logprobs(h64, W64, x, None)
    targets = rng.choice([-0.08, 0.0, 0.08, 0.75, -0.85], size=len(lengths))
    lr = np.zeros(T)
    start = 0
    for s, n in enumerate(lengths):
        sl = slice(start, start + n)
        noise = rng.uniform(-0.04, 0.04, n)
        a = m[sl] != 0
        if a.any():
            noise[a] -= noise[a].mean()
        lr[sl] = targets[s] + noise
        start += n
    b = (lp - lr).astype(np.float32)
    return h, W, x, m, seq, b, targets


@pytest.mark.parametrize("H", [128, 256])
def test_sequence_gate(H):
    rng = np.random.default_rng(H)
    lengths = [1, 3, 31, 32, 33, 64, 700, 5, 200, 2, 129, 90, 1, 17, 300, 64]
    h, W, x, m, seq, b, targets = _gated_problem(rng, H, 2500, lengths)
    T = seq.size
    m[:3] = 0            # a one-token sequence with no active token, and more
    adv = rng.standard_normal(T).astype(np.float32)
    out, ref = _run(h, W, x, m, b, adv, 0.3, 0.3, seq_of_token=seq, gate_lo=0.6, gate_hi=1.5)
    st = _check(out, ref, m, adv)
    # independent count: a sequence is rejected iff its target log-ratio lies
    # outside [log 0.6, log 1.5] and it has an active token
    start, n_rej = 0, 0
    for s, n in enumerate(lengths):
        if m[start:start + n].any() and not (np.log(0.6) <= targets[s] <= np.log(1.5)):
            n_rej += 1
        start += n
    assert n_rej > 0 and st["n_seq_rejected"] == n_rej
    tl = np_(out["token_loss"])
    assert (tl[ref["gate"] == 0] == 0).all()


@pytest.mark.parametrize("H", [128, 256])
def test_gate_kl_entropy_window_denominator(H):
    rng = np.random.default_rng(11 + H)
    lengths = list(rng.integers(1, 120, size=40))
    h, W, x, m, seq, b, _ = _gated_problem(rng, H, 3001, lengths, mask_frac=0.3)
    T = seq.size
    m[0] = 1
    adv = rng.standard_normal(T).astype(np.float32)
    lp, _ = O.token_logprobs(O.widen_bf16(h), O.widen_bf16(W), x, None)
    ref_logp = (lp + rng.normal(0, 0.3, T)).astype(np.float32)
    D = float(m.sum()) * 1.7
    out, ref = _run(h, W, x, m, b, adv, 0.3, 0.3, denom=D, kl_coef=0.1, ref_logp=ref_logp, entropy_coef=0.02,
                    seq_of_token=seq, gate_lo=0.6, gate_hi=1.5)
    _check(out, ref, m, adv, 0.1, 0.02)


def test_one_sequence_spanning_everything():
    rng = np.random.default_rng(5)
    h, W, x, m, seq, b, targets = _gated_problem(rng, 256, 1000, [3000])
    adv = rng.standard_normal(seq.size).astype(np.float32)
    out, ref = _run(h, W, x, m, b, adv, 0.3, 0.3, seq_of_token=seq, gate_lo=0.6, gate_hi=1.5)
    _check(out, ref, m, adv)
    rejected = not (np.log(0.6) <= targets[0] <= np.log(1.5))
    assert molt.stats_dict(out["stats"])["n_seq_rejected"] == int(rejected)


def test_unsorted_sequence_ids_flagged():
    rng = np.random.default_rng(9)
    h, W, x, m = random_problem(rng, 200, 128, 500)
    seq = np.repeat(np.arange(4), 50).astype(np.int32)
    seq[120] = 0          # ids decrease at token 120 (and rise again at 121)
    z = np.zeros(200, np.float32)
    molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(z), t(z), t(m), 0.2, 0.2, seq_of_token=t(seq),
                                gate_lo=0.5, gate_hi=2.0)
    assert molt.device_status() & molt.DEV_FLAGS["unsorted_groups"]


def test_bad_options_rejected():
    rng = np.random.default_rng(10)
    h, W, x, m = random_problem(rng, 64, 128, 300)
    z = np.zeros(64, np.float32)
    args = (bf(h), bf(W), t(x), t(z), t(z), t(m), 0.2, 0.2)
    with pytest.raises(molt.MoltError):
        molt.policy_loss_fwd_bwd_ex(*args, kl_coef=0.1)                       # no ref_logp
    with pytest.raises(molt.MoltError):
        molt.policy_loss_fwd_bwd_ex(*args, seq_of_token=t(np.zeros(64, np.int32)), gate_lo=2.0, gate_hi=1.0)
    with pytest.raises(molt.MoltError):
        molt.policy_loss_fwd_bwd_ex(*args, entropy_coef=float("nan"))


# ----------------------------------------------------------- deterministic mode
# (5000, 256, 9000): about 7 token quads (two groups of four) and 18 vocab
# blocks (two per residue class on a GB300), so both reduction orders of the
# schedule have more than one step
DET_SHAPES = [(1000, 256, 5000), (513, 512, 4133), (640, 768, 2304), (1, 256, 7), (5000, 256, 9000),
              (900, 384, 3000)]


@pytest.mark.parametrize("T,H,V", DET_SHAPES)
def test_deterministic_mode_is_bitwise_reproducible(T, H, V):
    rng = np.random.default_rng(T + 7 * H)
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.3, w_std=0.05)
    m[0] = 1
    adv = rng.standard_normal(T).astype(np.float32)
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    b = behavior_from_oracle(h64, W64, x, 0.3, 0.2, 0.28, T + 3)
    runs = []
    for _ in range(3):
        o = molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.28, deterministic=True)
        torch.cuda.synchronize()
        assert molt.device_status() == 0
        runs.append({k: np_(o[k]).copy() for k in ("loss", "dhidden", "dW", "logp", "token_loss")})
    for r in runs[1:]:
        for k in r:
            np.testing.assert_array_equal(r[k].view(np.uint8), runs[0][k].view(np.uint8), err_msg=k)
    ref = O.policy_loss_ex(h64, W64, x, b.astype(np.float64), adv.astype(np.float64), m, 0.2, 0.28)
    assert_grad_close(runs[0]["dhidden"], ref["dH"], "dhidden (deterministic)")
    assert_grad_close(runs[0]["dW"], ref["dW"], "dW (deterministic)")
    assert abs(float(runs[0]["loss"][0]) - ref["loss"]) <= LOSS_RTOL * max(
        abs(ref["loss"]), float(np.abs(ref["ratio"] * adv)[m != 0].sum() / ref["denom"]))


@pytest.mark.parametrize("T,H,V", [(5000, 256, 9000), (2100, 640, 20000)])
def test_deterministic_mode_does_not_depend_on_the_cluster_count(T, H, V):
    """The reduction order of the deterministic schedule is fixed by the turn
    counters (dW in token-quad order, dhidden in vocab-block order), not by which
    cluster runs which unit: 4, 8 and 16 clusters give the bits of the default
    count, although units, timing and the clusters' waits all change.  (2100,
    640, 20000) has a 128-column last job and 40 vocab blocks."""
    rng = np.random.default_rng(T + H)
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.25, w_std=0.05)
    m[0] = 1
    adv = rng.standard_normal(T).astype(np.float32)
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    b = behavior_from_oracle(h64, W64, x, 0.3, 0.2, 0.28, T + 5)
    runs = {}
    for n in (None, 16, 8, 4):
        o = molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.28, deterministic=True,
                                        det_clusters=n or 0)
        torch.cuda.synchronize()
        assert molt.device_status() == 0, n
        runs[n] = (np_(o["dW"]).copy(), np_(o["dhidden"]).copy())
    for n in (16, 8, 4):
        np.testing.assert_array_equal(runs[n][0].view(np.uint32), runs[None][0].view(np.uint32), err_msg=f"dW {n}")
        np.testing.assert_array_equal(runs[n][1].view(np.uint16), runs[None][1].view(np.uint16), err_msg=f"dh {n}")
    ref = O.policy_loss_ex(h64, W64, x, b.astype(np.float64), adv.astype(np.float64), m, 0.2, 0.28)
    assert_grad_close(runs[None][0], ref["dW"], "dW (deterministic)")
    assert_grad_close(runs[None][1], ref["dH"], "dhidden (deterministic)")


def test_deterministic_mode_accumulates_and_combines_with_extended_terms():
    rng = np.random.default_rng(21)
    lengths = [300, 1, 64, 400, 35]
    h, W, x, m, seq, b, _ = _gated_problem(rng, 512, 3000, lengths)
    T = seq.size
    m[0] = 1
    adv = rng.standard_normal(T).astype(np.float32)
    lp, _ = O.token_logprobs(O.widen_bf16(h), O.widen_bf16(W), x, None)
    ref_logp = (lp + rng.normal(0, 0.3, T)).astype(np.float32)
    kw = dict(kl_coef=0.1, ref_logp=ref_logp, entropy_coef=0.02, seq_of_token=seq, gate_lo=0.6, gate_hi=1.5)
    dW0 = (0.01 * rng.standard_normal((3000, 512))).astype(np.float32)
    outs = []
    for _ in range(2):
        dW = t(dW0.copy())
        o = molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.3, 0.3, dW=dW,
                                        accumulate_dW=True, deterministic=True,
                                        **{k: (t(v) if isinstance(v, np.ndarray) else v) for k, v in kw.items()})
        torch.cuda.synchronize()
        assert molt.device_status() == 0
        outs.append((np_(o["dW"]).copy(), np_(o["dhidden"]).copy()))
    np.testing.assert_array_equal(outs[0][0].view(np.uint32), outs[1][0].view(np.uint32))
    np.testing.assert_array_equal(outs[0][1].view(np.uint16), outs[1][1].view(np.uint16))
    ref = O.policy_loss_ex(O.widen_bf16(h), O.widen_bf16(W), x, b.astype(np.float64), adv.astype(np.float64), m,
                           0.3, 0.3, **kw)
    assert_grad_close(outs[0][0] - dW0, ref["dW"], "dW (accumulated, deterministic)")
    assert_grad_close(outs[0][1], ref["dH"], "dhidden (deterministic, extended terms)")


def test_deterministic_mode_needs_h_multiple_of_128():
    rng = np.random.default_rng(4)
    h, W, x, m = random_problem(rng, 64, 192, 300)
    z = np.zeros(64, np.float32)
    with pytest.raises(molt.MoltError):
        molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(z), t(z), t(m), 0.2, 0.2, deterministic=True)


def test_deterministic_cluster_count_is_validated():
    """det_clusters must be 0 or a multiple of 4 that fits on the device; other
    values are refused on the host and nothing is written."""
    rng = np.random.default_rng(5)
    h, W, x, m = random_problem(rng, 300, 256, 2000, mask_frac=0.1, w_std=0.05)
    adv = rng.standard_normal(300).astype(np.float32)
    b = np.full(300, -7.0, np.float32)
    for n in (2, 6, -4, 4000):
        with pytest.raises(molt.MoltError) as e:
            molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.2, deterministic=True,
                                        det_clusters=n)
        assert e.value.status == 1 and "det_clusters" in str(e.value)
