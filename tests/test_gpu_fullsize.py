"""Parity at the full workload sizes, in the launch configuration the benchmark
times (same entry point, same shapes, same masks).

The fp64 oracle cannot afford the whole [T, V] computation at these sizes, so:
  * sampled rows (random active rows plus every row of one 128-row tile) are
    checked one by one against the oracle: logp, entropy, per-token loss and the
    dhidden row;
  * properties that hold at any size are checked on the full outputs: the loss
    equals the sum of the per-token losses over D, masked rows have exactly zero
    dhidden / logp / loss, sum_v dW[v, :] = 0 (each row of g sums to zero), and
    sum_t <dH_t, h_t> = sum_v <dW_v, W_v> (both equal sum g z);
  * a sparse-mask run at the full V and H (only a few hundred active rows) lets
    the oracle compute dW exactly, element by element.
Behaviour log-probs of the sampled rows are the oracle's current log-probs plus
offsets kept away from the clip boundaries; the other rows draw an independent
stale-policy value, which puts roughly half of them on the clipped branch.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2607_21653_gb300 as molt  # noqa: E402
from oracle import molt_oracle as O  # noqa: E402
from workloads import boundary_safe_noise, make_workload  # noqa: E402

from parity import (BOUNDARY_DELTA, LOGP_ATOL, assert_grad_close, bf, np_, t)  # noqa: E402

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

N_RANDOM_ROWS = 96


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    molt.build()
    molt.load()


_W64_CACHE = {}


def _w64(w):
    key = (w.name, w.V, w.H, w.seed)
    if key not in _W64_CACHE:
        _W64_CACHE.clear()
        _W64_CACHE[key] = O.widen_bf16(w.weight)
    return _W64_CACHE[key]


def _sample_rows(w, rng):
    act = np.nonzero(w.mask)[0]
    rand = rng.choice(act, size=min(N_RANDOM_ROWS, act.size), replace=False)
    tile = act[(act.size // 2) // 128 * 128:][:128]        # one packed tile, all rows
    return np.unique(np.concatenate([rand, tile]))


# the ragged window's first microbatch holds only the two constant-reward groups
# (every advantage 0, so every tile is skipped); microbatch 1 mixes them with
# live groups
_MICROBATCH = {"ragged": 1}


def _run_fullsize(name, denom_from_window=False):
    w = make_workload(name, microbatch=_MICROBATCH.get(name, 0))
    rng = np.random.default_rng(1234)
    W64 = _w64(w)
    rows = _sample_rows(w, rng)
    h_rows64 = np.zeros((w.T, w.H))
    h_rows64[rows] = O.widen_bf16(w.hidden[rows])
    # behaviour log-probs: exact oracle log-probs + safe offsets on the sampled
    # rows, an independent stale-policy draw elsewhere
    b = rng.normal(-np.log(w.V) - 1.0, 1.0, w.T)
    lp_rows, _ = O.token_logprobs(h_rows64, W64, w.tokens, None, rows=rows)
    b[rows] = lp_rows + boundary_safe_noise(rng, rows.size, w.behavior_sigma, w.eps_lo, w.eps_hi,
                                            2.5 * BOUNDARY_DELTA)
    b = b.astype(np.float32)
    adv_resp = O.group_advantages(w.rewards, w.group_ids)
    adv = O.broadcast_advantages(adv_resp, w.resp_of_token)
    D = float(w.extra["window_denominator"]) if denom_from_window else float(w.mask.sum())

    dev_adv = molt.broadcast_advantages(molt.group_advantages(t(w.rewards), t(w.group_ids)), t(w.resp_of_token))
    np.testing.assert_array_equal(np_(dev_adv), adv)
    hid = bf(w.hidden)
    Wd = bf(w.weight)
    out = molt.policy_loss_fwd_bwd(hid, Wd, t(w.tokens), t(b), dev_adv, t(w.mask), w.eps_lo, w.eps_hi,
                                   denom=D if denom_from_window else 0.0)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    ref = O.policy_loss_rows(h_rows64, W64, w.tokens, b.astype(np.float64), adv.astype(np.float64), w.mask,
                             w.eps_lo, w.eps_hi, D, rows)
    return w, rows, b, adv, D, out, ref, hid, Wd


@pytest.mark.parametrize("name,window", [("large_vocab", False), ("mid", False), ("long_traj", False),
                                         ("ragged", True)])
def test_fullsize_policy_loss(name, window):
    w, rows, b, adv, D, out, ref, hid, Wd = _run_fullsize(name, denom_from_window=window)
    act = w.mask != 0
    lp, ent, tl = np_(out["logp"]), np_(out["entropy"]), np_(out["token_loss"])
    # sampled rows against the oracle
    assert np.abs(lp[rows] - ref["logp"]).max() <= LOGP_ATOL
    assert np.abs(ent[rows] - ref["entropy"]).max() <= LOGP_ATOL
    np.testing.assert_allclose(tl[rows], ref["token_loss"], rtol=5e-3, atol=1e-6)
    dh = out["dhidden"]
    dh_rows = np_(dh[torch.from_numpy(rows).to(dh.device)])
    assert_grad_close(dh_rows, ref["dH"], "dhidden (sampled rows)")
    # properties of the whole call
    assert (lp[~act] == 0).all() and (tl[~act] == 0).all() and (ent[~act] == 0).all()
    masked = torch.from_numpy(np.nonzero(~act)[0]).to(dh.device)
    if masked.numel():
        assert int(torch.count_nonzero(dh[masked]).item()) == 0
    L = float(out["loss"].item())
    L_tok = float(tl.astype(np.float64).sum() / D)
    assert abs(L - L_tok) <= 1e-5 * max(1e-3, abs(L_tok)), (L, L_tok)
    st = molt.stats_dict(out["stats"])
    assert st["n_active"] == int(act.sum()) and st["denom"] == D
    assert np.abs(ref["dH"]).max() > 0, "the sampled rows must carry a gradient"
    dW = out["dW"]
    col = dW.double().sum(dim=0)
    col_abs = dW.double().abs().sum(dim=0)
    assert float((col.abs() / col_abs.clamp_min(1e-30)).max().item()) < 1e-3
    # sum_t <dH_t, h_t> = sum_v <dW_v, W_v>; the sum can cancel, so scale the
    # tolerance by the sum of absolute per-row contributions
    row_dots = (dh.double() * hid.double()).sum(dim=1)
    lhs, scale = float(row_dots.sum().item()), float(row_dots.abs().sum().item())
    rhs = float((dW.double() * Wd.double()).sum().item())
    assert abs(lhs - rhs) <= 1e-2 * scale, (lhs, rhs, scale)


def test_fullsize_sparse_mask_exact_dW():
    """Full V and H, a few hundred active rows: dW parity element by element."""
    w = make_workload("large_vocab")
    rng = np.random.default_rng(77)
    act = np.sort(rng.choice(w.T, size=300, replace=False))
    mask = np.zeros(w.T, np.uint8)
    mask[act] = 1
    W64 = _w64(w)
    h_rows64 = np.zeros((w.T, w.H))
    h_rows64[act] = O.widen_bf16(w.hidden[act])
    lp, _ = O.token_logprobs(h_rows64, W64, w.tokens, None, rows=act)
    b = np.full(w.T, -12.0)
    b[act] = lp + boundary_safe_noise(rng, act.size, 0.3, w.eps_lo, w.eps_hi, 2.5 * BOUNDARY_DELTA)
    b = b.astype(np.float32)
    adv = rng.standard_normal(w.T).astype(np.float32)
    out = molt.policy_loss_fwd_bwd(bf(w.hidden), bf(w.weight), t(w.tokens), t(b), t(adv), t(mask), w.eps_lo,
                                   w.eps_hi)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    ref = O.policy_loss_rows(h_rows64, W64, w.tokens, b.astype(np.float64), adv.astype(np.float64), mask,
                             w.eps_lo, w.eps_hi, float(act.size), act, want_dW=True)
    assert_grad_close(np_(out["dW"]), ref["dW"], "dW (sparse mask, full V x H)")
    dh = np_(out["dhidden"])
    assert_grad_close(dh[act], ref["dH"], "dhidden (sparse mask)")
    assert not dh[mask == 0].any()
    assert abs(float(out["loss"].item()) - ref["token_loss"].sum() / act.size) <= 1e-3 * max(
        1e-3, float(np.abs(ref["ratio"] * adv[act]).sum() / act.size))


def test_fullsize_token_logprobs():
    w = make_workload("large_vocab")
    rng = np.random.default_rng(5)
    rows = _sample_rows(w, rng)
    h_rows64 = np.zeros((w.T, w.H))
    h_rows64[rows] = O.widen_bf16(w.hidden[rows])
    lp_ref, ent_ref = O.token_logprobs(h_rows64, _w64(w), w.tokens, w.mask, rows=rows)
    lp, ent = molt.token_logprobs(bf(w.hidden), bf(w.weight), t(w.tokens), t(w.mask))
    assert molt.device_status() == 0
    lp, ent = np_(lp), np_(ent)
    assert np.abs(lp[rows] - lp_ref).max() <= LOGP_ATOL
    assert np.abs(ent[rows] - ent_ref).max() <= LOGP_ATOL
    assert (lp[w.mask == 0] == 0).all()


def test_fullsize_deterministic_mode():
    """Deterministic backward at the benchmark size: two calls agree bit for bit
    on dW and dhidden, and sampled rows match the oracle."""
    w, rows, b, adv, D, _, ref, hid, Wd = _run_fullsize("large_vocab")
    outs = []
    for _ in range(2):
        o = molt.policy_loss_fwd_bwd_ex(hid, Wd, t(w.tokens), t(b), t(adv.astype(np.float32)), t(w.mask),
                                        w.eps_lo, w.eps_hi, deterministic=True)
        torch.cuda.synchronize()
        assert molt.device_status() == 0
        outs.append(o)
    assert torch.equal(outs[0]["dW"].view(torch.int32), outs[1]["dW"].view(torch.int32))
    assert torch.equal(outs[0]["dhidden"].view(torch.int16), outs[1]["dhidden"].view(torch.int16))
    assert float(outs[0]["loss"].item()) == float(outs[1]["loss"].item())
    dh = outs[0]["dhidden"]
    assert_grad_close(np_(dh[torch.from_numpy(rows).to(dh.device)]), ref["dH"], "dhidden (deterministic, sampled)")


def test_fullsize_extended_objective():
    """KL, entropy bonus and sequence gate at the benchmark size.  One sequence
    per response; each sequence's mean log-ratio is placed (from the library's
    own log-probs) either inside the gate band or 0.3+ outside it, so every gate
    decision is fixed by construction; sampled rows are checked against the
    oracle with those gate weights, and the rejection counts exactly."""
    w = make_workload("large_vocab")
    rng = np.random.default_rng(99)
    W64 = _w64(w)
    rows = _sample_rows(w, rng)
    h_rows64 = np.zeros((w.T, w.H))
    h_rows64[rows] = O.widen_bf16(w.hidden[rows])
    hid, Wd = bf(w.hidden), bf(w.weight)
    lp_dev, _ = molt.token_logprobs(hid, Wd, t(w.tokens), None)
    lp = np_(lp_dev).astype(np.float64)
    seq = w.resp_of_token.astype(np.int32)
    assert (np.diff(seq) >= 0).all()
    n_seq = int(seq.max()) + 1
    act = w.mask != 0
    targets = rng.choice([-0.05, 0.0, 0.05, 0.8, -0.9], size=n_seq)
    noise = rng.uniform(-0.04, 0.04, w.T)
    cnt = np.bincount(seq, weights=act.astype(np.float64), minlength=n_seq)
    mean_noise = np.bincount(seq, weights=noise * act, minlength=n_seq) / np.maximum(cnt, 1)
    lr = targets[seq] + noise - mean_noise[seq]
    b = (lp - lr).astype(np.float32)
    ref_logp = (lp + rng.normal(0, 0.3, w.T)).astype(np.float32)
    adv = O.broadcast_advantages(O.group_advantages(w.rewards, w.group_ids), w.resp_of_token).astype(np.float32)
    lo, hi = 0.6, 1.5
    kept = (np.log(lo) <= targets) & (targets <= np.log(hi))
    gate_w = np.where(kept[seq], 1.0, 0.0)
    out = molt.policy_loss_fwd_bwd_ex(hid, Wd, t(w.tokens), t(b), t(adv), t(w.mask), w.eps_lo, w.eps_hi,
                                      kl_coef=0.05, ref_logp=t(ref_logp), entropy_coef=0.01,
                                      seq_of_token=t(seq), gate_lo=lo, gate_hi=hi)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    D = float(act.sum())
    ref = O.policy_loss_ex_rows(h_rows64, W64, w.tokens, b.astype(np.float64), adv.astype(np.float64), w.mask,
                                w.eps_lo, w.eps_hi, D, rows, kl_coef=0.05, ref_logp=ref_logp, entropy_coef=0.01,
                                gate_w=gate_w)
    assert np.abs(np_(out["logp"])[rows] - ref["logp"]).max() <= LOGP_ATOL
    np.testing.assert_allclose(np_(out["token_loss"])[rows], ref["token_loss"], rtol=5e-3, atol=2e-5)
    dh = out["dhidden"]
    assert_grad_close(np_(dh[torch.from_numpy(rows).to(dh.device)]), ref["dH"], "dhidden (extended, sampled)")
    st = molt.stats_dict(out["stats"])
    live_seq = cnt > 0
    assert st["n_seq_rejected"] == int((~kept & live_seq).sum())
    assert st["n_tokens_rejected"] == int((act & ~kept[seq]).sum())


def test_fullsize_whole_ragged_window_in_one_call():
    """The ragged configuration's first 16 microbatches (1,048,576 tokens, H =
    5120) in one call: T x H = 5.4e9 elements, past 2^32, so every row offset
    of the packing, the backward and the casts needs 64-bit arithmetic.
    Sampled rows (random active rows across the whole window plus one tile near
    its end) against the oracle, and the whole-call properties of the
    full-size tests, evaluated in row chunks."""
    w = make_workload("ragged", T=16 * 65536)
    assert w.T == 16 * 65536 and w.T * w.H > 2 ** 32
    rng = np.random.default_rng(4321)
    act_idx = np.nonzero(w.mask)[0]
    rows = np.unique(np.concatenate([rng.choice(act_idx, size=N_RANDOM_ROWS, replace=False),
                                     act_idx[-(act_idx.size % 128 + 128):][:128]]))
    assert rows.max() * w.H > 2 ** 32
    W64 = _w64(w)
    h_c = O.widen_bf16(w.hidden[rows])          # the sampled rows only (rows are independent)
    x_c = w.tokens[rows]
    lp_c, _ = O.token_logprobs(h_c, W64, x_c, None, rows=np.arange(rows.size))
    b = rng.normal(-np.log(w.V) - 1.0, 1.0, w.T)
    b[rows] = lp_c + boundary_safe_noise(rng, rows.size, w.behavior_sigma, w.eps_lo, w.eps_hi,
                                         2.5 * BOUNDARY_DELTA)
    b = b.astype(np.float32)
    adv = O.broadcast_advantages(O.group_advantages(w.rewards, w.group_ids), w.resp_of_token)
    D = float(w.extra["window_denominator"])
    hid = bf(w.hidden)
    Wd = bf(w.weight)
    out = molt.policy_loss_fwd_bwd(hid, Wd, t(w.tokens), t(b), t(adv.astype(np.float32)), t(w.mask), w.eps_lo,
                                   w.eps_hi, denom=D)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    ref = O.policy_loss_rows(h_c, W64, x_c, b[rows].astype(np.float64), adv[rows].astype(np.float64),
                             w.mask[rows], w.eps_lo, w.eps_hi, D, np.arange(rows.size))
    lp, ent, tl = np_(out["logp"]), np_(out["entropy"]), np_(out["token_loss"])
    assert np.abs(lp[rows] - ref["logp"]).max() <= LOGP_ATOL
    assert np.abs(ent[rows] - ref["entropy"]).max() <= LOGP_ATOL
    np.testing.assert_allclose(tl[rows], ref["token_loss"], rtol=5e-3, atol=1e-6)
    dh = out["dhidden"]
    assert_grad_close(np_(dh[torch.from_numpy(rows).to(dh.device)]), ref["dH"], "dhidden (sampled rows)")
    assert np.abs(ref["dH"]).max() > 0, "the sampled rows must carry a gradient"
    act = w.mask != 0
    assert (lp[~act] == 0).all() and (tl[~act] == 0).all()
    masked = torch.from_numpy(np.nonzero(~act)[0]).to(dh.device)
    assert masked.numel() > 0 and int(torch.count_nonzero(dh[masked]).item()) == 0
    L_tok = float(tl.astype(np.float64).sum() / D)
    assert abs(float(out["loss"].item()) - L_tok) <= 1e-5 * max(1e-3, abs(L_tok))
    dW = out["dW"]
    col = dW.double().sum(dim=0)
    col_abs = dW.double().abs().sum(dim=0)
    assert float((col.abs() / col_abs.clamp_min(1e-30)).max().item()) < 1e-3
    lhs = scale = 0.0
    for r0 in range(0, w.T, 65536):
        d = (dh[r0:r0 + 65536].double() * hid[r0:r0 + 65536].double()).sum(dim=1)
        lhs += float(d.sum().item())
        scale += float(d.abs().sum().item())
    rhs = float((dW.double() * Wd.double()).sum().item())
    assert abs(lhs - rhs) <= 1e-2 * scale, (lhs, rhs, scale)
