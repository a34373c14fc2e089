"""Pins for the fp64 oracle, against things other than the oracle itself:
hand-derived values, closed forms, library routines (scipy log_softmax /
entropy, torch autograd of cross-entropy), finite differences and the
invariances that Eq. 2 and the segment rule of Sec. 4.2 state."""
import math

import numpy as np
import pytest
import scipy.special
import scipy.stats

from oracle import molt_oracle as O
from workloads import bf16_bits_to_f32, f32_to_bf16_bits, make_workload

GOLDEN = __import__("os").path.join(__import__("os").path.dirname(__file__), "golden")


def _read_golden(name):
    rows = []
    with open(f"{GOLDEN}/{name}") as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                rows.append(line)
    return rows


# ----------------------------------------------------------------- advantages
def test_advantages_hand_values():
    """Hand-derived GRPO values (tests/golden/grpo_hand.txt)."""
    for row in _read_golden("grpo_hand.txt"):
        rs, want = row.split("|")
        r = np.array([float(v) for v in rs.split()], dtype=np.float32)
        want = np.array([float(v) for v in want.split()], dtype=np.float64)
        got = O.group_advantages(r, np.zeros(len(r), dtype=np.int32))
        np.testing.assert_array_equal(got, want.astype(np.float32), err_msg=row)


def test_advantages_degenerate_groups():
    r = np.array([0.3, 0.3, 0.3, 0.3, 7.0, 1.0, 1.0], dtype=np.float32)
    g = np.array([0, 0, 0, 0, 1, 2, 2], dtype=np.int32)
    a = O.group_advantages(r, g)
    assert (a == 0).all()          # zero-variance groups and a one-response group give exactly 0


def test_advantages_match_library_and_moments():
    rng = np.random.default_rng(11)
    for G in (2, 3, 4, 8, 16, 33, 64):
        r = rng.random(G).astype(np.float32)
        a = O.group_advantages(r, np.zeros(G, dtype=np.int32))
        r64 = r.astype(np.float64)
        ref = (r64 - r64.mean()) / (r64.std(ddof=1) + 1e-6)
        np.testing.assert_allclose(a, ref.astype(np.float32), rtol=2e-7, atol=1e-7)
        assert abs(float(a.astype(np.float64).sum())) < 1e-5 * G
        sd = r64.std(ddof=1)
        assert abs(a.astype(np.float64).std(ddof=1) - sd / (sd + 1e-6)) < 1e-5


def test_advantages_groups_are_independent_and_permute():
    rng = np.random.default_rng(3)
    r = rng.random(40).astype(np.float32)
    g = np.repeat(np.arange(5), 8).astype(np.int32)
    a = O.group_advantages(r, g)
    for k in range(5):
        np.testing.assert_array_equal(a[8 * k:8 * k + 8],
                                      O.group_advantages(r[8 * k:8 * k + 8], np.zeros(8, np.int32)))
    perm = np.array([3, 0, 4, 1, 2])
    rp = np.concatenate([r[8 * k:8 * k + 8] for k in perm])
    ap = O.group_advantages(rp, g)
    np.testing.assert_array_equal(ap, np.concatenate([a[8 * k:8 * k + 8] for k in perm]))


def test_segment_split_invariance():
    """Sec. 4.2: segments of one rollout share its reward, counted once."""
    w = make_workload("long_traj", with_tensors=False, T=8 * 512)
    a_resp = O.group_advantages(w.rewards, w.group_ids)
    a_tok = O.broadcast_advantages(a_resp, w.resp_of_token)
    seg = w.extra["segment_of_token"]
    for s in np.unique(seg):
        toks = np.nonzero(seg == s)[0]
        assert np.unique(a_tok[toks]).size == 1
        assert a_tok[toks[0]] == a_resp[w.resp_of_token[toks[0]]]
    # the same rewards without any split give the same advantages
    np.testing.assert_array_equal(a_resp, O.group_advantages(w.rewards, np.zeros(8, np.int32)))


# ----------------------------------------------------------- log-softmax etc.
def test_logprobs_sum_to_one_and_match_library():
    rng = np.random.default_rng(5)
    T, H, V = 6, 9, 13
    h = rng.standard_normal((T, H))
    W = rng.standard_normal((V, H)) * 0.7
    z = h @ W.T
    tot = np.zeros(T)
    for v in range(V):
        lp, ent = O.token_logprobs(h, W, np.full(T, v), None)
        tot += np.exp(lp)
        np.testing.assert_allclose(lp, scipy.special.log_softmax(z, axis=1)[:, v], rtol=0, atol=1e-12)
        p = scipy.special.softmax(z, axis=1)
        np.testing.assert_allclose(ent, scipy.stats.entropy(p, axis=1), rtol=0, atol=1e-12)
    np.testing.assert_allclose(tot, 1.0, rtol=0, atol=1e-12)


def test_uniform_logits_closed_form():
    T, H, V = 4, 8, 1000
    h = np.ones((T, H))
    W = np.zeros((V, H))
    lp, ent = O.token_logprobs(h, W, np.arange(T), None)
    np.testing.assert_allclose(lp, -math.log(V), atol=1e-13)
    np.testing.assert_allclose(ent, math.log(V), atol=1e-13)


def test_masked_rows_zero():
    rng = np.random.default_rng(2)
    h = rng.standard_normal((5, 4))
    W = rng.standard_normal((7, 4))
    mask = np.array([1, 0, 1, 0, 0], np.uint8)
    lp, ent = O.token_logprobs(h, W, np.arange(5) % 7, mask)
    assert (lp[mask == 0] == 0).all() and (ent[mask == 0] == 0).all()
    assert (lp[mask == 1] < 0).all()


def test_bf16_widening_exact():
    x = np.array([1.0, -2.5, 3.140625, 1e-3, 65504.0], dtype=np.float32)
    bits = f32_to_bf16_bits(x)
    np.testing.assert_array_equal(O.widen_bf16(bits), bf16_bits_to_f32(bits).astype(np.float64))
    assert O.widen_bf16(np.array([0x3F80], np.uint16))[0] == 1.0
    assert O.widen_bf16(np.array([0xC020], np.uint16))[0] == -2.5


# ---------------------------------------------------------- clipped surrogate
def _small_problem(seed, T=8, H=16, V=32, mask=None):
    rng = np.random.default_rng(seed)
    h = rng.standard_normal((T, H))
    W = rng.standard_normal((V, H)) * 0.3
    x = rng.integers(0, V, T)
    m = np.ones(T, np.uint8) if mask is None else np.asarray(mask, np.uint8)
    return h, W, x, m


def test_clip_special_values():
    """Hand values of l = -min(rho A, clip(rho) A) for chosen rho."""
    h, W, x, m = _small_problem(0, T=6)
    lp, _ = O.token_logprobs(h, W, x, None)
    rho = np.array([1.0, 1.5, 0.5, 0.5, 1.5, 1.1])
    adv = np.array([0.7, 2.0, -1.0, 3.0, -0.5, -2.0])
    b = lp - np.log(rho)
    r = O.policy_loss(h, W, x, b, adv, m, 0.2, 0.28)
    want_l = np.array([-0.7, -1.28 * 2.0, -0.8 * -1.0, -0.5 * 3.0, -1.5 * -0.5, -1.1 * -2.0])
    want_clip = np.array([False, True, True, False, False, False])
    np.testing.assert_allclose(r["token_loss"], want_l, rtol=1e-12)
    np.testing.assert_array_equal(r["clipped"], want_clip)
    assert (r["dH"][want_clip] == 0).all()
    assert np.abs(r["dH"][~want_clip]).max() > 0
    np.testing.assert_allclose(r["loss"], want_l.sum() / 6, rtol=1e-12)


def test_rho_one_equals_weighted_nll_gradient():
    """At rho = 1 the gradient is that of sum m A CE(z, x) / D (torch autograd)."""
    torch = pytest.importorskip("torch")
    h, W, x, m = _small_problem(1, T=10, H=12, V=20, mask=[1, 1, 0, 1, 1, 1, 0, 1, 1, 1])
    adv = np.random.default_rng(9).standard_normal(10)
    lp, _ = O.token_logprobs(h, W, x, None)
    r = O.policy_loss(h, W, x, lp, adv, m, 0.2, 0.2)
    th = torch.tensor(h, requires_grad=True)
    tW = torch.tensor(W, requires_grad=True)
    ce = torch.nn.functional.cross_entropy(th @ tW.T, torch.tensor(x), reduction="none")
    L = (torch.tensor(m, dtype=torch.float64) * torch.tensor(adv) * ce).sum() / float(m.sum())
    L.backward()
    np.testing.assert_allclose(r["dH"], th.grad.numpy(), rtol=1e-10, atol=1e-13)
    np.testing.assert_allclose(r["dW"], tW.grad.numpy(), rtol=1e-10, atol=1e-13)
    np.testing.assert_allclose(r["loss"], -(m * adv).sum() / m.sum(), rtol=1e-12)


def test_full_gradient_matches_autograd():
    """Independent derivation of the backward: torch autograd of the surrogate."""
    torch = pytest.importorskip("torch")
    h, W, x, m = _small_problem(4, T=12, H=10, V=24, mask=[1] * 9 + [0] * 3)
    rng = np.random.default_rng(8)
    adv = rng.standard_normal(12)
    lp, _ = O.token_logprobs(h, W, x, None)
    b = lp + rng.choice([-0.6, -0.1, 0.05, 0.4], size=12)
    D = 17.0
    r = O.policy_loss(h, W, x, b, adv, m, 0.2, 0.28, denom=D)
    th = torch.tensor(h, requires_grad=True)
    tW = torch.tensor(W, requires_grad=True)
    logp = torch.log_softmax(th @ tW.T, dim=1)[torch.arange(12), torch.tensor(x)]
    rho = torch.exp(logp - torch.tensor(b))
    A = torch.tensor(adv)
    l = -torch.minimum(rho * A, torch.clamp(rho, 0.8, 1.28) * A)
    L = (torch.tensor(m, dtype=torch.float64) * l).sum() / D
    L.backward()
    np.testing.assert_allclose(r["loss"], L.item(), rtol=1e-12)
    np.testing.assert_allclose(r["dH"], th.grad.numpy(), rtol=1e-9, atol=1e-13)
    np.testing.assert_allclose(r["dW"], tW.grad.numpy(), rtol=1e-9, atol=1e-13)


def test_finite_differences():
    h, W, x, m = _small_problem(7, T=8, H=16, V=32, mask=[1, 1, 1, 0, 1, 1, 1, 1])
    rng = np.random.default_rng(1)
    adv = rng.standard_normal(8)
    lp, _ = O.token_logprobs(h, W, x, None)
    b = lp - np.log(np.array([1.0, 1.5, 0.5, 1.0, 0.9, 1.1, 0.6, 1.4]))
    r = O.policy_loss(h, W, x, b, adv, m, 0.2, 0.2)
    step = 1e-6

    def f(hh, WW):
        return O.policy_loss(hh, WW, x, b, adv, m, 0.2, 0.2)["loss"]

    gh = np.zeros_like(h)
    for i in range(h.shape[0]):
        for j in range(h.shape[1]):
            hp, hm = h.copy(), h.copy()
            hp[i, j] += step
            hm[i, j] -= step
            gh[i, j] = (f(hp, W) - f(hm, W)) / (2 * step)
    gW = np.zeros_like(W)
    for i in range(W.shape[0]):
        for j in range(W.shape[1]):
            Wp, Wm = W.copy(), W.copy()
            Wp[i, j] += step
            Wm[i, j] -= step
            gW[i, j] = (f(h, Wp) - f(h, Wm)) / (2 * step)
    np.testing.assert_allclose(r["dH"], gh, rtol=1e-5, atol=1e-9)
    np.testing.assert_allclose(r["dW"], gW, rtol=1e-5, atol=1e-9)


def test_microbatch_split_invariance():
    """Eq. 2: with one window denominator, microbatch losses/gradients add up."""
    h, W, x, m = _small_problem(12, T=20, H=8, V=16, mask=[1, 0, 1, 1, 1] * 4)
    rng = np.random.default_rng(12)
    adv = rng.standard_normal(20)
    lp, _ = O.token_logprobs(h, W, x, None)
    b = lp + rng.normal(0, 0.2, 20)
    full = O.policy_loss(h, W, x, b, adv, m, 0.2, 0.2)
    D = full["denom"]
    parts = [slice(0, 7), slice(7, 8), slice(8, 20)]
    tot, dW = 0.0, np.zeros_like(W)
    for s in parts:
        p = O.policy_loss(h[s], W, x[s], b[s], adv[s], m[s], 0.2, 0.2, denom=D)
        tot += p["loss"]
        dW += p["dW"]
        np.testing.assert_allclose(p["dH"], full["dH"][s], rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(tot, full["loss"], rtol=1e-12)
    np.testing.assert_allclose(dW, full["dW"], rtol=1e-11, atol=1e-15)


def test_gradient_row_and_column_sums_vanish():
    """sum_v g_tv = 0 per token, hence sum_v dW[v,:] = 0 (closed form)."""
    h, W, x, m = _small_problem(13, T=16, H=8, V=40)
    rng = np.random.default_rng(13)
    adv = rng.standard_normal(16)
    lp, _ = O.token_logprobs(h, W, x, None)
    r = O.policy_loss(h, W, x, lp + rng.normal(0, .1, 16), adv, m, 0.2, 0.2)
    np.testing.assert_allclose(r["dW"].sum(axis=0), 0.0, atol=1e-13)
    # trace identity: sum_t <dH_t, h_t> = sum_v <dW_v, W_v>
    np.testing.assert_allclose((r["dH"] * h).sum(), (r["dW"] * W).sum(), rtol=1e-10)


def test_rows_subset_equals_full():
    h, W, x, m = _small_problem(14, T=30, H=8, V=12, mask=[1, 1, 0] * 10)
    rng = np.random.default_rng(14)
    adv = rng.standard_normal(30)
    b = rng.normal(-2.5, 0.5, 30)
    full = O.policy_loss(h, W, x, b, adv, m, 0.2, 0.2)
    rows = np.array([29, 3, 4, 17, 0])
    sub = O.policy_loss_rows(h, W, x, b, adv, m, 0.2, 0.2, full["denom"], rows)
    for k in ("logp", "entropy", "ratio", "token_loss", "coef"):
        np.testing.assert_array_equal(sub[k], full[k][rows])
    np.testing.assert_allclose(sub["dH"], full["dH"][rows], rtol=1e-13, atol=1e-16)


# ------------------------------------------------ other estimators (Sec. 4.5)
def test_estimators_hand_values():
    for row in _read_golden("estimators_hand.txt"):
        est, rs, gs, want = [x.strip() for x in row.split("|")]
        r = np.array([float(v) for v in rs.split()], dtype=np.float32)
        g = np.array([int(v) for v in gs.split()], dtype=np.int32)
        want = np.array([float(v) for v in want.split()], dtype=np.float64).astype(np.float32)
        np.testing.assert_array_equal(O.advantages(r, g, est), want, err_msg=row)


def test_estimators_match_numpy_and_relations():
    rng = np.random.default_rng(21)
    r = rng.random(48).astype(np.float32)
    g = np.repeat(np.arange(6), 8).astype(np.int32)
    r64 = r.astype(np.float64)
    gm = O.advantages(r, g, "group_mean")
    np.testing.assert_array_equal(gm, O.advantages(r, g, "dr_grpo"))
    rloo = O.advantages(r, g, "rloo")
    for k in range(6):
        s = slice(8 * k, 8 * k + 8)
        ref = r64[s] - r64[s].mean()
        np.testing.assert_allclose(gm[s], ref.astype(np.float32), rtol=1e-6, atol=1e-7)
        # leave-one-out = n/(n-1) times the group-mean baseline advantage
        np.testing.assert_allclose(rloo[s], (8 / 7 * ref).astype(np.float32), rtol=2e-6, atol=1e-7)
        # GRPO = group-mean advantage / (std + eps)
        np.testing.assert_allclose(O.advantages(r, g, "grpo")[s], (ref / (r64[s].std(ddof=1) + 1e-6)).astype(np.float32),
                                   rtol=2e-6, atol=1e-7)
    rpp = O.advantages(r, g, "reinforce_pp")
    np.testing.assert_allclose(rpp, ((r64 - r64.mean()) / (r64.std(ddof=1) + 1e-6)).astype(np.float32),
                               rtol=2e-6, atol=1e-7)
    assert abs(float(rpp.astype(np.float64).sum())) < 1e-4
    # singleton groups and a batch of one give 0
    assert (O.advantages(np.array([3.0], np.float32), np.array([0], np.int32), "rloo") == 0).all()
    assert (O.advantages(np.array([3.0], np.float32), np.array([0], np.int32), "reinforce_pp") == 0).all()


# ------------------------------------ extended objective (KL, entropy, gate)
def _ex_problem(seed, T=12, H=10, V=24):
    h, W, x, _ = _small_problem(seed, T=T, H=H, V=V)
    rng = np.random.default_rng(seed + 100)
    m = (rng.random(T) > 0.2).astype(np.uint8)
    m[0] = 1
    adv = rng.standard_normal(T)
    lp, _ = O.token_logprobs(h, W, x, None)
    b = lp + rng.choice([-0.6, -0.1, 0.05, 0.4], size=T)
    ref = lp + rng.normal(0, 0.3, T)
    return h, W, x, m, adv, b, ref


def test_ex_reduces_to_plain_loss():
    h, W, x, m, adv, b, ref = _ex_problem(1)
    plain = O.policy_loss(h, W, x, b, adv, m, 0.2, 0.28)
    ex = O.policy_loss_ex(h, W, x, b, adv, m, 0.2, 0.28)
    np.testing.assert_allclose(ex["loss"], plain["loss"], rtol=1e-13)
    np.testing.assert_allclose(ex["dH"], plain["dH"], rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(ex["dW"], plain["dW"], rtol=1e-12, atol=1e-15)
    # KL against the policy itself is zero and leaves the gradient unchanged
    lp, _ = O.token_logprobs(h, W, x, None)
    ex0 = O.policy_loss_ex(h, W, x, b, adv, m, 0.2, 0.28, kl_coef=0.7, ref_logp=lp)
    np.testing.assert_allclose(ex0["kl"], 0.0, atol=1e-12)
    np.testing.assert_allclose(ex0["dH"], plain["dH"], rtol=1e-9, atol=1e-14)


def test_ex_gradient_matches_autograd():
    """Independent derivation: torch autograd of PPO + k3 KL - entropy bonus."""
    torch = pytest.importorskip("torch")
    h, W, x, m, adv, b, ref = _ex_problem(2)
    kl_c, ent_c, D = 0.3, 0.05, 11.0
    r = O.policy_loss_ex(h, W, x, b, adv, m, 0.2, 0.28, denom=D, kl_coef=kl_c, ref_logp=ref, entropy_coef=ent_c)
    th = torch.tensor(h, requires_grad=True)
    tW = torch.tensor(W, requires_grad=True)
    logits = th @ tW.T
    logsm = torch.log_softmax(logits, dim=1)
    logp = logsm[torch.arange(len(x)), torch.tensor(x)]
    ent = -(logsm.exp() * logsm).sum(dim=1)
    rho = torch.exp(logp - torch.tensor(b))
    A = torch.tensor(adv)
    pg = -torch.minimum(rho * A, torch.clamp(rho, 0.8, 1.28) * A)
    rr = torch.tensor(ref) - logp
    kl = torch.exp(rr) - rr - 1
    L = (torch.tensor(m, dtype=torch.float64) * (pg + kl_c * kl - ent_c * ent)).sum() / D
    L.backward()
    np.testing.assert_allclose(r["loss"], L.item(), rtol=1e-12)
    np.testing.assert_allclose(r["dH"], th.grad.numpy(), rtol=1e-9, atol=1e-13)
    np.testing.assert_allclose(r["dW"], tW.grad.numpy(), rtol=1e-9, atol=1e-13)


def test_sequence_gate_rejects_without_renormalising():
    """Sec. 4.5: rejection weights live in l_i; Eq. 2 keeps its denominator."""
    h, W, x, _ = _small_problem(3, T=12, H=8, V=16)
    m = np.ones(12, np.uint8)
    adv = np.random.default_rng(3).standard_normal(12)
    lp, _ = O.token_logprobs(h, W, x, None)
    seq = np.repeat(np.arange(3), 4).astype(np.int32)
    # per-sequence log ratios: seq 0 all +0.1 (ratio 1.105, kept), seq 1 mean +0.6
    # (ratio 1.82, rejected above 1.5), seq 2 mean -1.0 (ratio 0.37, rejected below 0.5)
    lr = np.array([0.1] * 4 + [0.9, 0.3, 0.6, 0.6] + [-1.0, -1.2, -0.8, -1.0])
    b = lp - lr
    w = O.sequence_gate(lr, seq, m, 0.5, 1.5)
    np.testing.assert_array_equal(w, [1] * 4 + [0] * 8)
    ex = O.policy_loss_ex(h, W, x, b, adv, m, 0.2, 0.2, seq_of_token=seq, gate_lo=0.5, gate_hi=1.5)
    plain = O.policy_loss(h, W, x, b, adv, m, 0.2, 0.2)
    assert ex["denom"] == 12.0
    np.testing.assert_allclose(ex["token_loss"][:4], plain["token_loss"][:4], rtol=1e-13)
    assert (ex["token_loss"][4:] == 0).all() and (ex["dH"][4:] == 0).all()
    np.testing.assert_allclose(ex["loss"], plain["token_loss"][:4].sum() / 12.0, rtol=1e-13)
    # masked tokens do not enter the geometric mean
    m2 = m.copy()
    m2[4] = 0
    # with hi = 1.7: seq 1 with all four tokens has ratio e^0.6 = 1.82 (rejected);
    # without its masked 0.9 token the mean is 0.5, ratio 1.65 (kept)
    np.testing.assert_array_equal(O.sequence_gate(lr, seq, m, 0.5, 1.7)[4:8], 0.0)
    np.testing.assert_array_equal(O.sequence_gate(lr, seq, m2, 0.5, 1.7)[4:8], 1.0)
    # a sequence with no active token keeps weight 1 and contributes nothing
    m3 = m.copy()
    m3[8:] = 0
    np.testing.assert_array_equal(O.sequence_gate(lr, seq, m3, 0.5, 1.5)[8:], 1.0)


def test_ex_rows_is_a_slice_of_the_full_extended_loss():
    h, W, x, m, adv, b, ref = _ex_problem(4, T=20, H=12, V=30)
    seq = np.repeat(np.arange(4), 5).astype(np.int32)
    full = O.policy_loss_ex(h, W, x, b, adv, m, 0.2, 0.28, kl_coef=0.2, ref_logp=ref, entropy_coef=0.05,
                            seq_of_token=seq, gate_lo=0.8, gate_hi=1.25)
    rows = np.array([17, 3, 0, 11, 8])
    part = O.policy_loss_ex_rows(h, W, x, b, adv, m, 0.2, 0.28, full["denom"], rows, kl_coef=0.2, ref_logp=ref,
                                 entropy_coef=0.05, gate_w=full["gate"])
    for k in ("logp", "token_loss", "coef"):
        np.testing.assert_allclose(part[k], full[k][rows], rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(part["dH"], full["dH"][rows], rtol=1e-12, atol=1e-15)


# ------------------------------------- full-batch forward and sampled dW rows
def test_full_forward_rows_matches_library():
    """lse / logp / entropy of whole rows against scipy's logsumexp,
    log_softmax and entropy; thread splitting and row blocks change nothing;
    large logits do not overflow (the row max is shifted out)."""
    rng = np.random.default_rng(21)
    T, H, V = 37, 24, 3001
    h = rng.standard_normal((T, H))
    W = rng.standard_normal((V, H)) * 0.5
    x = rng.integers(0, V, T)
    rows = np.array([36, 0, 5, 5, 17, 2])
    z = h @ W.T
    lse, lp, ent = O.full_forward_rows(h, W, x, rows)
    np.testing.assert_allclose(lse, scipy.special.logsumexp(z[rows], axis=1), rtol=0, atol=1e-12)
    np.testing.assert_allclose(lp, scipy.special.log_softmax(z[rows], axis=1)[np.arange(6), x[rows]], atol=1e-12)
    np.testing.assert_allclose(ent, scipy.stats.entropy(scipy.special.softmax(z[rows], axis=1), axis=1),
                               atol=1e-12)
    a = O.full_forward_rows(h, W, x, np.arange(T), block=7, workers=3)
    b = O.full_forward_rows(h, W, x, np.arange(T), block=1024, workers=1)
    for u, v in zip(a, b):
        np.testing.assert_array_equal(u, v)
    # a constant shift of every logit of a row moves lse by it and leaves logp
    # and entropy alone (bias column through h)
    h2 = np.concatenate([h, np.full((T, 1), 40.0)], axis=1)
    W2 = np.concatenate([W, np.full((V, 1), 20.0)], axis=1)
    lse2, lp2, ent2 = O.full_forward_rows(h2, W2, x, rows)
    np.testing.assert_allclose(lse2, lse + 800.0, rtol=1e-14)
    np.testing.assert_allclose(lp2, lp, atol=1e-10)
    np.testing.assert_allclose(ent2, ent, atol=1e-9)


def test_full_forward_rows_uniform_closed_form():
    T, H, V = 3, 5, 777
    lse, lp, ent = O.full_forward_rows(np.ones((T, H)), np.zeros((V, H)), np.arange(T), np.arange(T))
    np.testing.assert_allclose(lse, math.log(V), atol=1e-13)
    np.testing.assert_allclose(lp, -math.log(V), atol=1e-13)
    np.testing.assert_allclose(ent, math.log(V), atol=1e-13)


def test_dW_rows_is_a_slice_of_the_full_backward():
    """dW_rows with the loss's own lse and m c / D reproduces rows of the full
    backward (itself pinned by autograd and finite differences), target rows
    (one-hot term) and non-target rows alike."""
    h, W, x, m = _small_problem(23, T=40, H=12, V=50, mask=[1, 1, 1, 0] * 10)
    rng = np.random.default_rng(23)
    adv = rng.standard_normal(40)
    lp, _ = O.token_logprobs(h, W, x, None)
    b = lp + rng.normal(0, 0.3, 40)
    full = O.policy_loss(h, W, x, b, adv, m, 0.2, 0.25)
    act = np.nonzero(m)[0]
    vr = np.unique(np.concatenate([x[act][:5], [0, 7, 49]]))
    got = O.dW_rows(h, W, x, full["lse"][act], full["coef"][act], act, vr, block=7)
    np.testing.assert_allclose(got, full["dW"][vr], rtol=1e-11, atol=1e-15)
    assert np.abs(full["dW"][vr]).max() > 0


def test_shard_merge_equals_whole_row():
    """Statistics of disjoint vocabulary shards merged in log space equal the
    whole row's lse, logp and entropy, for any split (uneven shards, shards
    without any target, one shard)."""
    rng = np.random.default_rng(29)
    T, H, V = 23, 16, 1000
    h = rng.standard_normal((T, H))
    W = rng.standard_normal((V, H)) * 0.8
    x = rng.integers(0, 300, T)                 # targets only in the first shards
    rows = np.arange(T)
    ref = O.full_forward_rows(h, W, x, rows)
    for bounds in ([0, V], [0, 500, V], [0, 1, 333, 334, V], [0, 123, 456, 789, 999, V]):
        parts = np.stack([O.shard_partials(h, W[a:b], x, a, rows) for a, b in zip(bounds[:-1], bounds[1:])])
        lse, lp, ent = O.merge_shard_partials(parts)
        np.testing.assert_allclose(lse, ref[0], rtol=0, atol=1e-12)
        np.testing.assert_allclose(lp, ref[1], rtol=0, atol=1e-12)
        np.testing.assert_allclose(ent, ref[2], rtol=0, atol=1e-11)
    # a shard's own statistics: lse of the shard alone = M + log S
    p = O.shard_partials(h, W[500:], x, 500, rows)
    np.testing.assert_allclose(p[:, 0] + np.log(p[:, 1]), scipy.special.logsumexp((h @ W[500:].T), axis=1),
                               atol=1e-12)
    assert np.isneginf(p[:, 3]).all()           # no target falls in [500, V)


def test_shard_dhidden_terms_sum_to_the_full_backward():
    """The shards' dhidden terms (each with the whole row's lse and m c / D)
    add up to dH of the full backward (pinned by autograd), for uneven
    shards and shards without targets."""
    h, W, x, m = _small_problem(31, T=30, H=10, V=60, mask=[1, 0, 1] * 10)
    rng = np.random.default_rng(31)
    adv = rng.standard_normal(30)
    lp, _ = O.token_logprobs(h, W, x, None)
    full = O.policy_loss(h, W, x, lp + rng.normal(0, 0.3, 30), adv, m, 0.2, 0.2)
    act = np.nonzero(m)[0]
    for bounds in ([0, 60], [0, 7, 60], [0, 1, 30, 31, 60]):
        tot = np.zeros((act.size, 10))
        for a, b in zip(bounds[:-1], bounds[1:]):
            tot += O.shard_dhidden(h, W[a:b], x, a, full["lse"][act], full["coef"][act], act)
        np.testing.assert_allclose(tot, full["dH"][act], rtol=1e-11, atol=1e-15)
