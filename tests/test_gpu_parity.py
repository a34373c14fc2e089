"""GPU parity of every step of the hot path against the fp64 oracle, through
the C ABI, on seeded inputs small enough for the full oracle: several tiles in
every dimension with ragged tails (T, V and H not multiples of the tiles)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2607_21653_gb300 as molt  # noqa: E402
from oracle import molt_oracle as O  # noqa: E402
from workloads import make_workload, random_problem  # noqa: E402

from parity import (LOGP_ATOL, assert_grad_close, assert_loss_close, behavior_from_oracle, bf, np_,  # noqa: E402
                    t)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    molt.build()
    molt.load()


# ------------------------------------------------------------------ advantages
@pytest.mark.parametrize("name", ["tiny", "mid", "large_vocab", "long_traj", "ragged"])
def test_group_advantages_bit_exact(name):
    w = make_workload(name, with_tensors=False)
    ref = O.group_advantages(w.rewards, w.group_ids)
    got = np_(molt.group_advantages(t(w.rewards), t(w.group_ids)))
    assert molt.device_status() == 0
    np.testing.assert_array_equal(got.view(np.uint32), ref.view(np.uint32))


def test_group_advantages_edge_cases():
    rng = np.random.default_rng(7)
    sizes = [1, 2, 3, 31, 32, 33, 64, 100, 1, 5]
    gids = np.concatenate([np.full(s, i, np.int32) for i, s in enumerate(sizes)])
    r = rng.random(gids.shape[0]).astype(np.float32)
    r[gids == 4] = 0.25                      # zero-variance group of 32
    r[gids == 6] = np.float32(1e30) * rng.standard_normal(64).astype(np.float32)  # huge magnitudes
    got = np_(molt.group_advantages(t(r), t(gids)))
    ref = O.group_advantages(r, gids)
    np.testing.assert_array_equal(got.view(np.uint32), ref.view(np.uint32))
    assert (got[gids == 4] == 0).all() and got[0] == 0 and got[gids == 8][0] == 0
    assert molt.device_status() == 0
    # a decreasing id is reported on the device
    bad = gids.copy()
    bad[-1] = 0
    molt.group_advantages(t(r), t(bad))
    assert molt.device_status() & molt.DEV_FLAGS["unsorted_groups"]


@pytest.mark.parametrize("estimator", ["grpo", "group_mean", "dr_grpo", "rloo", "reinforce_pp"])
@pytest.mark.parametrize("name", ["tiny", "mid", "large_vocab", "long_traj", "ragged"])
def test_estimators_bit_exact(name, estimator):
    w = make_workload(name, with_tensors=False)
    ref = O.advantages(w.rewards, w.group_ids, estimator)
    got = np_(molt.advantages(t(w.rewards), t(w.group_ids), estimator))
    assert molt.device_status() == 0
    np.testing.assert_array_equal(got.view(np.uint32), ref.view(np.uint32))


def test_estimators_edge_cases():
    r = np.array([1, 0, 0, 0, 5, 2, 2, 2, 7], np.float32)
    g = np.array([0, 0, 0, 0, 1, 2, 2, 2, 3], np.int32)
    for est in ("group_mean", "dr_grpo", "rloo", "reinforce_pp"):
        got = np_(molt.advantages(t(r), t(g), est))
        np.testing.assert_array_equal(got.view(np.uint32), O.advantages(r, g, est).view(np.uint32))
    one = np.array([3.5], np.float32)
    assert float(np_(molt.advantages(t(one), None, "reinforce_pp"))[0]) == 0.0
    assert molt.device_status() == 0


def test_broadcast_and_mask_count():
    w = make_workload("long_traj", with_tensors=False, T=8 * 1000)
    adv = O.group_advantages(w.rewards, w.group_ids)
    got = np_(molt.broadcast_advantages(t(adv), t(w.resp_of_token)))
    np.testing.assert_array_equal(got, O.broadcast_advantages(adv, w.resp_of_token))
    for T in (1, 15, 16, 17, 1000, 8000, 65537):
        m = (np.random.default_rng(T).random(T) < 0.37).astype(np.uint8)
        assert int(molt.mask_count(t(m)).item()) == int(m.sum())


# ------------------------------------------------------------ log-probs fwd
SHAPES = [
    # T, H, V, mask fraction
    (300, 128, 1000, 0.2),      # ragged T and V, 2 K-blocks
    (128, 64, 256, 0.0),        # exactly one tile, one K-block
    (513, 192, 4133, 0.5),      # ragged everything, H not a multiple of 128
    (1, 64, 7, 0.0),            # one row, vocab smaller than a tile
    (700, 320, 2304, 0.9),      # mostly masked
]


@pytest.mark.parametrize("T,H,V,mf", SHAPES)
def test_token_logprobs_small(T, H, V, mf):
    rng = np.random.default_rng(T * 7 + H)
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=mf, w_std=0.05)
    lp_ref, ent_ref = O.token_logprobs(O.widen_bf16(h), O.widen_bf16(W), x, m)
    lp, ent = molt.token_logprobs(bf(h), bf(W), t(x), t(m))
    lp, ent = np_(lp), np_(ent)
    assert molt.device_status() == 0
    assert np.abs(lp - lp_ref).max() <= LOGP_ATOL, np.abs(lp - lp_ref).max()
    assert np.abs(ent - ent_ref).max() <= LOGP_ATOL, np.abs(ent - ent_ref).max()
    assert (lp[m == 0] == 0).all() and (ent[m == 0] == 0).all()


def test_token_logprobs_tiny_config():
    w = make_workload("tiny")
    lp_ref, ent_ref = O.token_logprobs(O.widen_bf16(w.hidden), O.widen_bf16(w.weight), w.tokens, w.mask)
    lp, ent = molt.token_logprobs(bf(w.hidden), bf(w.weight), t(w.tokens), t(w.mask))
    assert np.abs(np_(lp) - lp_ref).max() <= LOGP_ATOL
    assert np.abs(np_(ent) - ent_ref).max() <= LOGP_ATOL


def test_token_range_flag():
    rng = np.random.default_rng(3)
    h, W, x, m = random_problem(rng, 64, 64, 300)
    x[5] = 300
    molt.token_logprobs(bf(h), bf(W), t(x), t(m))
    assert molt.device_status() & molt.DEV_FLAGS["token_range"]


# --------------------------------------------------------- policy loss fwd+bwd
def _loss_case(h, W, x, m, adv, sigma, eps_lo, eps_hi, seed, denom=0.0):
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    b = behavior_from_oracle(h64, W64, x, sigma, eps_lo, eps_hi, seed)
    ref = O.policy_loss(h64, W64, x, b.astype(np.float64), adv.astype(np.float64), m, eps_lo, eps_hi,
                        denom=denom if denom > 0 else None)
    ref["_adv"] = adv.astype(np.float64)
    out = molt.policy_loss_fwd_bwd(bf(h), bf(W), t(x), t(b), t(adv), t(m), eps_lo, eps_hi, denom=denom)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    return out, ref


def _check_loss(out, ref, m):
    assert_loss_close(float(out["loss"].item()), ref)
    act = m != 0
    lp = np_(out["logp"])
    assert np.abs(lp - ref["logp"]).max() <= LOGP_ATOL
    assert np.abs(np_(out["entropy"]) - ref["entropy"]).max() <= LOGP_ATOL
    tl = np_(out["token_loss"])
    np.testing.assert_allclose(tl[act], ref["token_loss"][act], rtol=5e-3, atol=1e-5)
    assert (tl[~act] == 0).all()
    dh = np_(out["dhidden"])
    assert (dh[~act] == 0).all(), "masked rows must have exactly zero dhidden"
    assert_grad_close(dh, ref["dH"], "dhidden")
    assert_grad_close(np_(out["dW"]), ref["dW"], "dW")
    st = molt.stats_dict(out["stats"])
    assert st["n_active"] == int(act.sum())
    assert st["n_clip_low"] == int(((ref["clipped"]) & (ref["_adv"] < 0) & act).sum())
    assert st["n_clip_high"] == int(((ref["clipped"]) & (ref["_adv"] > 0) & act).sum())
    # the backward processes exactly the rows with a gradient; the others have
    # exactly zero dhidden
    live = act & (ref["coef"] != 0)
    assert st["n_grad_rows"] == int(live.sum())
    assert (dh[act & ~live] == 0).all()


LOSS_SHAPES = [
    # single-CTA backward (H not a multiple of 256)
    (300, 128, 1000, 0.2),
    (513, 192, 4133, 0.3),
    (256, 320, 2304, 0.0),
    (1, 64, 7, 0.0),
    # CTA-pair backward (H a multiple of 256): odd and even tile counts, a pair
    # whose second CTA has no tile, several H chunks, ragged vocab tails
    (300, 256, 1000, 0.2),
    (513, 512, 4133, 0.3),
    (1, 256, 7, 0.0),
    (640, 768, 2304, 0.0),
    (1000, 256, 5000, 0.6),
]


@pytest.mark.parametrize("T,H,V,mf", LOSS_SHAPES)
def test_policy_loss_small(T, H, V, mf):
    rng = np.random.default_rng(T + 11 * H)
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=mf, w_std=0.05)
    m[0] = 1
    adv = rng.standard_normal(T).astype(np.float32)
    out, ref = _loss_case(h, W, x, m, adv, 0.3, 0.2, 0.28, seed=T)
    _check_loss(out, ref, m)


def test_policy_loss_tiny_config():
    w = make_workload("tiny")
    adv = O.broadcast_advantages(O.group_advantages(w.rewards, w.group_ids), w.resp_of_token)
    out, ref = _loss_case(w.hidden, w.weight, w.tokens, w.mask, adv, w.behavior_sigma, w.eps_lo, w.eps_hi, 0)
    _check_loss(out, ref, w.mask)


def test_policy_loss_window_denominator_and_accumulate():
    """Eq. 2: two microbatches with the window denominator add up to the whole."""
    rng = np.random.default_rng(21)
    T, H, V = 400, 128, 1500
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.25, w_std=0.05)
    adv = rng.standard_normal(T).astype(np.float32)
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    b = behavior_from_oracle(h64, W64, x, 0.2, 0.2, 0.2, 5)
    D = float(m.sum())
    whole = molt.policy_loss_fwd_bwd(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.2)
    dW = torch.zeros(V, H, dtype=torch.float32, device=whole["dW"].device)
    L = 0.0
    dh_parts = []
    for s in (slice(0, 170), slice(170, 400)):
        o = molt.policy_loss_fwd_bwd(bf(h[s]), bf(W), t(x[s]), t(b[s]), t(adv[s]), t(m[s]), 0.2, 0.2, denom=D,
                                     dW=dW, accumulate_dW=True)
        L += float(o["loss"].item())
        dh_parts.append(np_(o["dhidden"]))
    assert abs(L - float(whole["loss"].item())) <= 1e-5 * max(1.0, abs(L))
    np.testing.assert_allclose(np_(dW), np_(whole["dW"]), rtol=1e-4, atol=1e-6)
    assert_grad_close(np.concatenate(dh_parts), np_(whole["dhidden"]), "dhidden (microbatches)")


def test_policy_loss_all_masked():
    rng = np.random.default_rng(4)
    h, W, x, m = random_problem(rng, 200, 64, 500)
    m[:] = 0
    adv = rng.standard_normal(200).astype(np.float32)
    b = np.full(200, -6.0, np.float32)
    # with a window denominator: zero loss and zero gradients, no flag
    o = molt.policy_loss_fwd_bwd(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.2, denom=100.0)
    assert float(o["loss"].item()) == 0.0
    assert molt.device_status() == 0
    assert not np_(o["dhidden"]).any() and not np_(o["dW"]).any()
    # without one: the zero denominator is flagged, outputs still zero
    o = molt.policy_loss_fwd_bwd(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.2)
    assert float(o["loss"].item()) == 0.0
    assert molt.device_status() & molt.DEV_FLAGS["zero_denom"]
    assert not np_(o["dW"]).any()


def test_policy_loss_deterministic():
    rng = np.random.default_rng(8)
    h, W, x, m = random_problem(rng, 300, 128, 1000, mask_frac=0.1, w_std=0.05)
    adv = rng.standard_normal(300).astype(np.float32)
    b = rng.normal(-7.0, 0.5, 300).astype(np.float32)
    o1 = molt.policy_loss_fwd_bwd(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.2)
    o2 = molt.policy_loss_fwd_bwd(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.2)
    assert float(o1["loss"].item()) == float(o2["loss"].item())
    np.testing.assert_array_equal(np_(o1["logp"]), np_(o2["logp"]))


@pytest.mark.parametrize("H,det", [(64, False), (256, False), (256, True)])
def test_single_class_vocabulary(H, det):
    """V = 1, the degenerate softmax: p = 1, so logp = entropy = 0 and g = coef (p -
    1) = 0 (dW and dhidden vanish up to the rounding of p next to 1); the loss
    is the surrogate of rho = exp(-b) alone."""
    rng = np.random.default_rng(H + int(det))
    T = 300
    h, W, x, m = random_problem(rng, T, H, 1, mask_frac=0.2, w_std=0.05)
    m[0] = 1
    adv = rng.standard_normal(T).astype(np.float32)
    b = rng.normal(0.0, 0.3, T).astype(np.float32)
    out = molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.28, deterministic=det)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    assert np.abs(np_(out["logp"])).max() <= 1e-6 and np.abs(np_(out["entropy"])).max() <= 1e-6
    ref = O.policy_loss(O.widen_bf16(h), O.widen_bf16(W), x, b.astype(np.float64), adv.astype(np.float64), m,
                        0.2, 0.28)
    ref["_adv"] = adv.astype(np.float64)
    assert_loss_close(float(out["loss"].item()), ref)
    coef = np.abs(ref["coef"])
    h_max = float(np.abs(O.widen_bf16(h)).max())
    w_max = float(np.abs(O.widen_bf16(W)).max())
    assert np.abs(np_(out["dW"])).max() <= 1e-5 * coef.sum() * h_max
    assert np.abs(np_(out["dhidden"]).astype(np.float64)).max() <= 1e-5 * coef.max() * w_max


@pytest.mark.parametrize("H,det", [(192, False), (512, False), (512, True)])
def test_zero_advantages_skip_every_tile(H, det):
    """A = 0 on every token: every coefficient m c / D is 0, every backward tile
    is skipped, and the loss, dW and dhidden are exactly zero while logp and
    entropy still match the oracle."""
    rng = np.random.default_rng(7 * H + int(det))
    T, V = 900, 3000
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.2, w_std=0.05)
    m[0] = 1
    adv = np.zeros(T, np.float32)
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    b = behavior_from_oracle(h64, W64, x, 0.3, 0.2, 0.2, 9)
    dW = torch.full((V, H), 7.0, device="cuda")
    out = molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.2, deterministic=det, dW=dW)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    assert float(out["loss"].item()) == 0.0
    assert not np_(out["dW"]).any() and not np_(out["dhidden"]).any()
    lp_ref, ent_ref = O.token_logprobs(h64, W64, x, m)
    assert np.abs(np_(out["logp"]) - lp_ref).max() <= LOGP_ATOL
    assert np.abs(np_(out["entropy"]) - ent_ref).max() <= LOGP_ATOL


@pytest.mark.parametrize("det", [False, True])
def test_largest_hidden_size(det):
    """H = 65536, the largest supported: 1024 K-blocks per logit tile in the
    forward, 2048 logit stages per vocab half and 256 dH / dW jobs per unit in
    the backward."""
    rng = np.random.default_rng(65536 + int(det))
    T, H, V = 130, 65536, 300
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.1, w_std=0.01)
    m[0] = 1
    adv = rng.standard_normal(T).astype(np.float32)
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    b = behavior_from_oracle(h64, W64, x, 0.3, 0.2, 0.28, 3)
    ref = O.policy_loss(h64, W64, x, b.astype(np.float64), adv.astype(np.float64), m, 0.2, 0.28)
    ref["_adv"] = adv.astype(np.float64)
    out = molt.policy_loss_fwd_bwd_ex(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.28, deterministic=det)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    assert np.abs(np_(out["logp"]) - ref["logp"]).max() <= LOGP_ATOL
    assert_loss_close(float(out["loss"].item()), ref)
    assert_grad_close(np_(out["dhidden"]), ref["dH"], "dhidden (H = 65536)")
    assert_grad_close(np_(out["dW"]), ref["dW"], "dW (H = 65536)")


@pytest.mark.parametrize("T,H,V", [(700, 256, 3000), (700, 192, 3000), (2100, 512, 9000)])
def test_rows_without_gradient_are_left_out(T, H, V):
    """Clipped rows and rows with A = 0 carry no gradient: the backward runs on
    the other rows only (n_grad_rows), gives them the oracle's gradient, and
    leaves exactly zero dhidden on the rest.  About half the rows are on the
    clipped branch (behaviour log-probs 0.5 away from the current ones) and a
    fifth have A = 0."""
    rng = np.random.default_rng(T + H)
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=0.15, w_std=0.05)
    adv = rng.standard_normal(T).astype(np.float32)
    adv[rng.random(T) < 0.2] = 0.0
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    lp, _ = O.token_logprobs(h64, W64, x, None)
    off = np.where(rng.random(T) < 0.5, rng.choice([-0.5, 0.5], T), rng.uniform(-0.08, 0.08, T))
    b = (lp + off).astype(np.float32)
    ref = O.policy_loss(h64, W64, x, b.astype(np.float64), adv.astype(np.float64), m, 0.2, 0.2)
    ref["_adv"] = adv.astype(np.float64)
    act = m != 0
    live = act & (ref["coef"] != 0)
    assert 0.2 * act.sum() < live.sum() < 0.7 * act.sum()
    out = molt.policy_loss_fwd_bwd(bf(h), bf(W), t(x), t(b), t(adv), t(m), 0.2, 0.2)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    _check_loss(out, ref, m)
