"""The vocabulary-parallel LM head on one GPU.

The shards of W run one after another on the same device, and their outputs
are combined the way the ranks' exchange would combine them: the statistics
stacked in shard order, the dhidden terms summed, the dW shards side by side.
The results are compared with the unsharded call (molt_policy_loss_fwd_bwd)
and with the fp64 oracle: the shard statistics with the oracle's
shard_partials, the merged log-probs, entropies and loss with the whole-row
forward, dhidden and dW with the oracle's backward.
"""
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


def _sharded_step(hd, Wd, xd, md, bd, advd, n, eps_lo, eps_hi, denom=0.0):
    V, H = Wd.shape
    bounds = molt.vocab_shard_bounds(V, n)
    parts = torch.stack([molt.vp_partials(hd, Wd[a:e], xd, a, md) for a, e in bounds])
    out = molt.vp_loss(parts, bd, advd, md, eps_lo, eps_hi, denom)
    dh = torch.zeros(hd.shape[0], H, dtype=torch.float32, device=hd.device)
    dWs = []
    for a, e in bounds:
        dh_s, dW_s = molt.vp_backward(hd, Wd[a:e], xd, out["lse"], out["coef"], a)
        dh += dh_s
        dWs.append(dW_s)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    out.update(parts=parts, dhidden=dh, dW=torch.cat(dWs), bounds=bounds)
    return out


CASES = [
    # (T, H, V, shards, mask fraction): cluster backward (H % 128 == 0) and the
    # single-CTA one (H % 128 == 64), uneven shards, a shard narrower than one
    # vocab tile, ragged tails
    (700, 256, 3000, 2, 0.2),
    (700, 256, 3000, 4, 0.2),
    (1030, 192, 5001, 3, 0.1),
    (2100, 512, 9000, 4, 0.25),
    (300, 128, 1100, 4, 0.0),
]


@pytest.mark.parametrize("T,H,V,n,mf", CASES)
def test_vocab_parallel_matches_unsharded_and_oracle(T, H, V, n, mf):
    rng = np.random.default_rng(T + H + n)
    h, W, x, m = random_problem(rng, T, H, V, mask_frac=mf, w_std=0.05)
    m[0] = 1
    adv = rng.standard_normal(T).astype(np.float32)
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    b = behavior_from_oracle(h64, W64, x, 0.3, 0.2, 0.28, T + 1)
    hd, Wd, xd, md, bd, advd = bf(h), bf(W), t(x), t(m), t(b), t(adv)
    out = _sharded_step(hd, Wd, xd, md, bd, advd, n, 0.2, 0.28)
    act = m != 0
    # every shard's statistics against the oracle's
    parts = out["parts"].double().cpu().numpy()
    rows = np.nonzero(act)[0]
    for s, (a, e) in enumerate(out["bounds"]):
        ref = O.shard_partials(h64, W64[a:e], x, a, rows)
        got = parts[s][rows]
        assert np.abs(got[:, 0] + np.log(got[:, 1]) - (ref[:, 0] + np.log(ref[:, 1]))).max() <= LOGP_ATOL
        assert np.abs(got[:, 2] / got[:, 1] - ref[:, 2] / ref[:, 1]).max() <= LOGP_ATOL
        fin = np.isfinite(ref[:, 3])
        assert (np.isfinite(got[:, 3]) == fin).all()
        assert np.abs(got[fin, 3] - ref[fin, 3]).max(initial=0.0) <= LOGP_ATOL
        assert (parts[s][~act] == np.array([-np.inf, 0, 0, -np.inf])).all()
    # the merged step against the oracle
    ref = O.policy_loss(h64, W64, x, b.astype(np.float64), adv.astype(np.float64), m, 0.2, 0.28)
    ref["_adv"] = adv.astype(np.float64)
    assert_loss_close(float(out["loss"].item()), ref)
    assert np.abs(np_(out["logp"]) - ref["logp"]).max() <= LOGP_ATOL
    assert np.abs(np_(out["entropy"]) - ref["entropy"]).max() <= LOGP_ATOL
    np.testing.assert_allclose(np_(out["token_loss"])[act], ref["token_loss"][act], rtol=5e-3, atol=1e-5)
    dh = np_(out["dhidden"])
    live = act & (ref["coef"] != 0)
    assert (dh[~live] == 0).all()
    assert_grad_close(dh, ref["dH"], "dhidden (sum of the shards)")
    assert_grad_close(np_(out["dW"]), ref["dW"], "dW (shards side by side)")
    st = molt.stats_dict(out["stats"])
    assert st["n_active"] == int(act.sum()) and st["n_grad_rows"] == int(live.sum())
    assert st["n_clip_low"] == int((ref["clipped"] & (adv < 0) & act).sum())
    assert st["n_clip_high"] == int((ref["clipped"] & (adv > 0) & act).sum())
    # the same step unsharded
    un = molt.policy_loss_fwd_bwd(hd, Wd, xd, bd, advd, md, 0.2, 0.28)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    assert abs(float(un["loss"].item()) - float(out["loss"].item())) <= 1e-5 * max(1e-3, abs(ref["loss"]))
    assert np.abs(np_(un["logp"]) - np_(out["logp"])).max() <= 1e-4
    assert_grad_close(dh, np_(un["dhidden"]), "dhidden (sharded vs unsharded)")
    assert_grad_close(np_(out["dW"]), np_(un["dW"]), "dW (sharded vs unsharded)")


def test_vocab_parallel_mid_workload():
    """The mid workload (T=32768, H=2048, V=32000) split into 2 and 4 shards:
    each against the unsharded call, and the log-probs of every active row,
    the loss and 128 sampled dhidden rows against the oracle."""
    w = make_workload("mid")
    hd, Wd, xd, md = bf(w.hidden), bf(w.weight), t(w.tokens), t(w.mask)
    act = np.nonzero(w.mask)[0]
    W64 = O.widen_bf16(w.weight)
    h_act = O.widen_bf16(w.hidden[act])
    _, lp_all, ent_all = O.full_forward_rows(h_act, W64, w.tokens[act], np.arange(act.size), workers=8)
    rng = np.random.default_rng(8)
    from workloads import boundary_safe_noise
    from parity import BOUNDARY_DELTA
    b = np.zeros(w.T)
    b[act] = lp_all + boundary_safe_noise(rng, act.size, w.behavior_sigma, w.eps_lo, w.eps_hi, 2.5 * BOUNDARY_DELTA)
    b = b.astype(np.float32)
    adv = O.broadcast_advantages(O.group_advantages(w.rewards, w.group_ids), w.resp_of_token).astype(np.float32)
    un = molt.policy_loss_fwd_bwd(hd, Wd, xd, t(b), t(adv), md, w.eps_lo, w.eps_hi)
    torch.cuda.synchronize()
    rho = np.exp(lp_all - b[act].astype(np.float64))
    tl, c, _ = O.surrogate(rho, adv[act].astype(np.float64), w.eps_lo, w.eps_hi)
    L_ref = float(tl.sum() / act.size)
    scale = float(np.abs(rho * adv[act]).sum() / act.size)
    pos = np.sort(rng.choice(act.size, 128, replace=False))
    rows = act[pos]
    h_rows = np.zeros((w.T, w.H))
    h_rows[rows] = h_act[pos]
    r = O.policy_loss_rows(h_rows, W64, w.tokens, b.astype(np.float64), adv.astype(np.float64), w.mask, w.eps_lo,
                           w.eps_hi, float(act.size), rows)
    for n in (2, 4):
        out = _sharded_step(hd, Wd, xd, md, t(b), t(adv), n, w.eps_lo, w.eps_hi)
        assert abs(float(out["loss"].item()) - L_ref) <= 1e-3 * max(abs(L_ref), scale)
        assert np.abs(np_(out["logp"])[act] - lp_all).max() <= LOGP_ATOL
        assert np.abs(np_(out["entropy"])[act] - ent_all).max() <= LOGP_ATOL
        dh = out["dhidden"]
        assert_grad_close(np_(dh[torch.from_numpy(rows).to(dh.device)]), r["dH"], f"dhidden ({n} shards, sampled)")
        assert_grad_close(np_(dh), np_(un["dhidden"]), f"dhidden ({n} shards vs unsharded)")
        assert_grad_close(np_(out["dW"]), np_(un["dW"]), f"dW ({n} shards vs unsharded)")


def test_vocab_parallel_token_in_no_shard_is_flagged():
    """Statistics of shards that do not cover a row's token (here: only the
    first of two shards is merged) raise the token-range flag."""
    rng = np.random.default_rng(3)
    h, W, x, m = random_problem(rng, 256, 128, 1000)
    x[:] = 900                                   # every target in the second half
    hd, Wd, xd = bf(h), bf(W), t(x)
    p0 = molt.vp_partials(hd, Wd[:500], xd, 0)
    b = t(np.full(256, -7.0, np.float32))
    adv = t(np.ones(256, np.float32))
    molt.vp_loss(p0[None], b, adv, None, 0.2, 0.2)
    assert molt.device_status() & molt.DEV_FLAGS["token_range"]


def test_vocab_parallel_edge_cases():
    """A single token row; a one-column shard; every row masked (loss 0 and the
    zero-denominator flag, as the unsharded call); rows whose coefficient is 0
    (A = 0) leave the backward nothing to do; accumulation into a dW shard."""
    rng = np.random.default_rng(11)
    # one row, shards [0, 1), [1, 500), [500, 1000)
    h, W, x, m = random_problem(rng, 1, 128, 1000, w_std=0.05)
    x[0] = 0
    hd, Wd, xd = bf(h), bf(W), t(x)
    bounds = [(0, 1), (1, 500), (500, 1000)]
    parts = torch.stack([molt.vp_partials(hd, Wd[a:e], xd, a) for a, e in bounds])
    h64, W64 = O.widen_bf16(h), O.widen_bf16(W)
    b = behavior_from_oracle(h64, W64, x, 0.2, 0.2, 0.2, 3)
    adv = np.array([0.7], np.float32)
    out = molt.vp_loss(parts, t(b), t(adv), None, 0.2, 0.2)
    ref = O.policy_loss(h64, W64, x, b.astype(np.float64), adv.astype(np.float64), np.ones(1, np.uint8), 0.2, 0.2)
    assert molt.device_status() == 0
    assert abs(np_(out["logp"])[0] - ref["logp"][0]) <= LOGP_ATOL
    dh = torch.zeros(1, 128, dtype=torch.float32, device=hd.device)
    dWs = []
    for a, e in bounds:
        d, dw = molt.vp_backward(hd, Wd[a:e], xd, out["lse"], out["coef"], a)
        dh += d
        dWs.append(dw)
    torch.cuda.synchronize()
    assert_grad_close(np_(dh), ref["dH"], "dhidden (one row)")
    assert_grad_close(np_(torch.cat(dWs)), ref["dW"], "dW (one row, one-column shard)")
    # accumulate into an existing shard: dW += the same contribution
    d2, dw2 = molt.vp_backward(hd, Wd[1:500], xd, out["lse"], out["coef"], 1, dW=dWs[1].clone(), accumulate_dW=True)
    torch.cuda.synchronize()
    np.testing.assert_allclose(np_(dw2), 2 * np_(dWs[1]), rtol=1e-6, atol=1e-12)
    # every row masked
    h, W, x, _ = random_problem(rng, 300, 256, 2000, w_std=0.05)
    m = np.zeros(300, np.uint8)
    hd, Wd, xd, md = bf(h), bf(W), t(x), t(m)
    parts = torch.stack([molt.vp_partials(hd, Wd[a:e], xd, a, md) for a, e in molt.vocab_shard_bounds(2000, 2)])
    assert torch.isneginf(parts[..., 0]).all() and (parts[..., 1] == 0).all()
    out = molt.vp_loss(parts, t(np.zeros(300, np.float32)), t(np.ones(300, np.float32)), md, 0.2, 0.2)
    assert float(out["loss"].item()) == 0.0
    assert molt.device_status() & molt.DEV_FLAGS["zero_denom"]
    assert not np_(out["coef"]).any()
    # all advantages 0: nothing for the backward
    m = np.ones(300, np.uint8)
    md = t(m)
    parts = torch.stack([molt.vp_partials(hd, Wd[a:e], xd, a, md) for a, e in molt.vocab_shard_bounds(2000, 2)])
    out = molt.vp_loss(parts, t(np.full(300, -7.0, np.float32)), t(np.zeros(300, np.float32)), md, 0.2, 0.2)
    assert molt.stats_dict(out["stats"])["n_grad_rows"] == 0
    d, dw = molt.vp_backward(hd, Wd[:1000], xd, out["lse"], out["coef"], 0)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    assert not np_(d).any() and not np_(dw).any()
