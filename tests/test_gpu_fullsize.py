"""Parity at the full workload sizes, in the launch configuration the benchmark
times (same entry point, same shapes, same masks).

Mid (T=32768, H=2048, V=32000) is checked whole: every active row's logp,
entropy, per-token loss and dhidden row and the whole 32000 x 2048 dW against
the fp64 oracle's full forward and backward.

For the three H x V = 4096 (or 5120) x 151936 workloads the oracle runs the
full forward once per workload (2 T H V fp64 flops on the host cores, every
active row against the whole vocabulary), which gives:
  * the loss L = sum m l / D of the whole call, compared with the library's;
  * logp, entropy and the per-token loss of EVERY active row;
  * behaviour log-probs b = oracle logp + N(0, sigma) with sigma the
    workload's, redrawn inside a band around the clip boundaries, so that every
    clip decision is unique at the log-prob tolerance and the clip counters
    are exact;
  * lse and m c / D of every row, from which dW rows follow at full density:
    dW is compared on 256 random vocab rows plus the target row of every
    sampled token row (the one-hot term).
dhidden is compared on 1024 random active rows plus every row of one packed
128-row tile.  Properties that hold at any size are checked on the whole
outputs as well (sum_v dW[v, :] = 0; sum_t <dH_t, h_t> = sum_v <dW_v, W_v>).
"""
import os
import time

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2607_21653_gb300 as molt  # noqa: E402
from oracle import molt_oracle as O  # noqa: E402
from workloads import boundary_safe_noise, make_workload  # noqa: E402

from parity import (BOUNDARY_DELTA, LOGP_ATOL, LOSS_RTOL, assert_grad_close, bf, np_, t)  # noqa: E402

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

N_RANDOM_ROWS = 1024        # sampled active rows for dhidden (plus one packed tile)
N_DW_RANDOM_ROWS = 256      # random vocab rows of dW (plus the sampled rows' targets)
WORKERS = max(1, os.cpu_count() or 1)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    molt.build()
    molt.load()


# the ragged window's first microbatch holds only the two constant-reward groups
# (every advantage 0, so every tile is skipped); microbatch 1 mixes them with
# live groups and uses the window's denominator
_MICROBATCH = {"ragged": 1}
_WINDOW_DENOM = {"ragged": True}

_CACHE = {}     # the latest workload's inputs and oracle full forward


def _setup(name):
    """Workload, fp64 operands, oracle full forward of the active rows, the
    behaviour log-probs built from it and the per-token advantages."""
    key = name
    if key in _CACHE:
        return _CACHE[key]
    _CACHE.clear()
    w = make_workload(name, microbatch=_MICROBATCH.get(name, 0))
    act = np.nonzero(w.mask)[0]
    W64 = O.widen_bf16(w.weight)
    h_act = O.widen_bf16(w.hidden[act])
    t0 = time.perf_counter()
    lse, logp, ent = O.full_forward_rows(h_act, W64, w.tokens[act], np.arange(act.size), workers=WORKERS)
    secs = time.perf_counter() - t0
    print(f"\n[oracle] full forward of {name}: {act.size} rows x H {w.H} x V {w.V} in {secs:.1f} s "
          f"({WORKERS} threads)")
    rng = np.random.default_rng(1234)
    b = rng.normal(-np.log(w.V) - 1.0, 1.0, w.T)          # masked rows: ignored by both sides
    b[act] = logp + boundary_safe_noise(rng, act.size, w.behavior_sigma, w.eps_lo, w.eps_hi,
                                        2.5 * BOUNDARY_DELTA)
    b = b.astype(np.float32)
    adv = O.broadcast_advantages(O.group_advantages(w.rewards, w.group_ids), w.resp_of_token)
    D = float(w.extra["window_denominator"]) if _WINDOW_DENOM.get(name) else float(act.size)
    # the oracle's loss terms for every active row (m = 1 there)
    rho = np.exp(logp - b[act].astype(np.float64))
    a_act = adv[act].astype(np.float64)
    tl, c, clipped = O.surrogate(rho, a_act, w.eps_lo, w.eps_hi)
    ref = {"lse": lse, "logp": logp, "entropy": ent, "ratio": rho, "token_loss": tl, "coef": c / D,
           "clipped": clipped, "loss": float(tl.sum() / D), "scale": float(np.abs(rho * a_act).sum() / D),
           "secs": secs}
    s = dict(w=w, act=act, W64=W64, h_act=h_act, b=b, adv=adv, D=D, ref=ref,
             window=_WINDOW_DENOM.get(name, False), rng=np.random.default_rng(99))
    _CACHE[key] = s
    return s


def _sample_rows(act, rng):
    """Positions (into the active rows) of N_RANDOM_ROWS random active rows
    plus one whole packed 128-row tile."""
    rand = rng.choice(act.size, size=min(N_RANDOM_ROWS, act.size), replace=False)
    k0 = (act.size // 2) // 128 * 128
    tile = np.arange(k0, min(act.size, k0 + 128))
    return np.unique(np.concatenate([rand, tile]))


def _check_call(s, out, check_dW=True, label=""):
    w, act, ref, D = s["w"], s["act"], s["ref"], s["D"]
    rng = np.random.default_rng(7)
    lp, ent, tl = np_(out["logp"]), np_(out["entropy"]), np_(out["token_loss"])
    # every active row
    assert np.abs(lp[act] - ref["logp"]).max() <= LOGP_ATOL, label
    assert np.abs(ent[act] - ref["entropy"]).max() <= LOGP_ATOL, label
    np.testing.assert_allclose(tl[act], ref["token_loss"], rtol=5e-3, atol=1e-6, err_msg=label)
    inact = np.ones(w.T, bool)
    inact[act] = False
    assert (lp[inact] == 0).all() and (tl[inact] == 0).all() and (ent[inact] == 0).all()
    # the loss of the whole call against the oracle's full forward
    L = float(out["loss"].item())
    assert abs(L - ref["loss"]) <= LOSS_RTOL * max(abs(ref["loss"]), ref["scale"]), (label, L, ref["loss"])
    st = molt.stats_dict(out["stats"])
    a_act = s["adv"][act]
    assert st["n_active"] == act.size and st["denom"] == D
    assert st["n_clip_low"] == int((ref["clipped"] & (a_act < 0)).sum())
    assert st["n_clip_high"] == int((ref["clipped"] & (a_act > 0)).sum())
    # dhidden: sampled rows against the oracle's rows
    pos = _sample_rows(act, rng)
    rows = act[pos]
    h_rows = np.zeros((w.T, w.H))
    h_rows[rows] = s["h_act"][pos]
    r = O.policy_loss_rows(h_rows, s["W64"], w.tokens, s["b"].astype(np.float64), s["adv"].astype(np.float64),
                           w.mask, w.eps_lo, w.eps_hi, D, rows)
    np.testing.assert_allclose(r["lse"], ref["lse"][pos], rtol=0, atol=1e-9)
    dh = out["dhidden"]
    dh_rows = np_(dh[torch.from_numpy(rows).to(dh.device)])
    assert_grad_close(dh_rows, r["dH"], f"dhidden ({label}, {rows.size} sampled rows)")
    masked = torch.from_numpy(np.nonzero(inact)[0]).to(dh.device)
    if masked.numel():
        assert int(torch.count_nonzero(dh[masked]).item()) == 0
    if not check_dW:
        return
    # dW: random vocab rows and the targets of the sampled rows, full density
    vr_rand = np.sort(rng.choice(w.V, size=N_DW_RANDOM_ROWS, replace=False))
    vr = np.unique(np.concatenate([vr_rand, w.tokens[rows]]))
    dW_ref = O.dW_rows(s["h_act"], s["W64"], w.tokens[act], ref["lse"], ref["coef"], np.arange(act.size), vr)
    dW = out["dW"]
    dW_got = dW[torch.from_numpy(vr).to(dW.device)].double().cpu().numpy()
    assert_grad_close(dW_got, dW_ref, f"dW ({label}, {vr.size} vocab rows)")
    # the random rows on their own (mostly no one-hot term: softmax terms only)
    k = np.searchsorted(vr, vr_rand)
    assert_grad_close(dW_got[k], dW_ref[k], f"dW ({label}, {vr_rand.size} random vocab rows)")
    # whole-call identities
    col = dW.double().sum(dim=0)
    col_abs = dW.double().abs().sum(dim=0)
    assert float((col.abs() / col_abs.clamp_min(1e-30)).max().item()) < 1e-3
    hid = s["hid"]
    lhs = scale = 0.0
    for r0 in range(0, w.T, 65536):
        d = (dh[r0:r0 + 65536].double() * hid[r0:r0 + 65536].double()).sum(dim=1)
        lhs += float(d.sum().item())
        scale += float(d.abs().sum().item())
    rhs = float((dW.double() * s["Wd"].double()).sum().item())
    assert abs(lhs - rhs) <= 1e-2 * scale, (lhs, rhs, scale)


def _device_inputs(s):
    w = s["w"]
    if "hid" not in s:
        s["hid"] = bf(w.hidden)
        s["Wd"] = bf(w.weight)
    return s["hid"], s["Wd"]


def _loss_call(s, **kw):
    w = s["w"]
    hid, Wd = _device_inputs(s)
    dev_adv = molt.broadcast_advantages(molt.group_advantages(t(w.rewards), t(w.group_ids)), t(w.resp_of_token))
    np.testing.assert_array_equal(np_(dev_adv), s["adv"])
    fn = molt.policy_loss_fwd_bwd_ex if kw else molt.policy_loss_fwd_bwd
    out = fn(hid, Wd, t(w.tokens), t(s["b"]), dev_adv, t(w.mask), w.eps_lo, w.eps_hi,
             denom=s["D"] if s["window"] else 0.0, **kw)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    return out


# ------------------------------------------------------------- large vocab
def test_large_vocab_policy_loss():
    s = _setup("large_vocab")
    _check_call(s, _loss_call(s), label="large_vocab")


def test_large_vocab_token_logprobs_every_row():
    s = _setup("large_vocab")
    w, act = s["w"], s["act"]
    hid, Wd = _device_inputs(s)
    lp, ent = molt.token_logprobs(hid, Wd, t(w.tokens), t(w.mask))
    assert molt.device_status() == 0
    lp, ent = np_(lp), np_(ent)
    assert np.abs(lp[act] - s["ref"]["logp"]).max() <= LOGP_ATOL
    assert np.abs(ent[act] - s["ref"]["entropy"]).max() <= LOGP_ATOL
    assert (lp[w.mask == 0] == 0).all()


def test_large_vocab_deterministic_mode():
    """Deterministic backward at the benchmark size: two calls agree bit for bit
    on dW and dhidden, and the outputs match the oracle like the raster's."""
    s = _setup("large_vocab")
    outs = [_loss_call(s, deterministic=True) for _ in range(2)]
    assert torch.equal(outs[0]["dW"].view(torch.int32), outs[1]["dW"].view(torch.int32))
    assert torch.equal(outs[0]["dhidden"].view(torch.int16), outs[1]["dhidden"].view(torch.int16))
    assert float(outs[0]["loss"].item()) == float(outs[1]["loss"].item())
    _check_call(s, outs[0], label="large_vocab deterministic")


def test_large_vocab_extended_objective():
    """KL, entropy bonus and sequence gate at the benchmark size.  One sequence
    per response; each sequence's mean log-ratio is placed (from the oracle's
    full-forward log-probs) either inside the gate band or 0.3+ outside it, so
    every gate decision is fixed by construction; sampled rows are checked
    against the oracle with those gate weights, and the rejection counts
    exactly."""
    s = _setup("large_vocab")
    w, act = s["w"], s["act"]
    rng = np.random.default_rng(99)
    lp = np.zeros(w.T)
    lp[act] = s["ref"]["logp"]
    seq = w.resp_of_token.astype(np.int32)
    assert (np.diff(seq) >= 0).all()
    n_seq = int(seq.max()) + 1
    am = w.mask != 0
    targets = rng.choice([-0.05, 0.0, 0.05, 0.8, -0.9], size=n_seq)
    noise = rng.uniform(-0.04, 0.04, w.T)
    cnt = np.bincount(seq, weights=am.astype(np.float64), minlength=n_seq)
    mean_noise = np.bincount(seq, weights=noise * am, minlength=n_seq) / np.maximum(cnt, 1)
    lr = targets[seq] + noise - mean_noise[seq]
    b = (lp - lr).astype(np.float32)
    ref_logp = (lp + rng.normal(0, 0.3, w.T)).astype(np.float32)
    adv = s["adv"].astype(np.float32)
    lo, hi = 0.6, 1.5
    kept = (np.log(lo) <= targets) & (targets <= np.log(hi))
    gate_w = np.where(kept[seq], 1.0, 0.0)
    hid, Wd = _device_inputs(s)
    out = molt.policy_loss_fwd_bwd_ex(hid, Wd, t(w.tokens), t(b), t(adv), t(w.mask), w.eps_lo, w.eps_hi,
                                      kl_coef=0.05, ref_logp=t(ref_logp), entropy_coef=0.01,
                                      seq_of_token=t(seq), gate_lo=lo, gate_hi=hi)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    D = float(act.size)
    pos = _sample_rows(act, rng)
    rows = act[pos]
    h_rows = np.zeros((w.T, w.H))
    h_rows[rows] = s["h_act"][pos]
    ref = O.policy_loss_ex_rows(h_rows, s["W64"], w.tokens, b.astype(np.float64), adv.astype(np.float64), w.mask,
                                w.eps_lo, w.eps_hi, D, rows, kl_coef=0.05, ref_logp=ref_logp, entropy_coef=0.01,
                                gate_w=gate_w)
    assert np.abs(np_(out["logp"])[rows] - ref["logp"]).max() <= LOGP_ATOL
    np.testing.assert_allclose(np_(out["token_loss"])[rows], ref["token_loss"], rtol=5e-3, atol=2e-5)
    dh = out["dhidden"]
    assert_grad_close(np_(dh[torch.from_numpy(rows).to(dh.device)]), ref["dH"], "dhidden (extended, sampled)")
    st = molt.stats_dict(out["stats"])
    live_seq = cnt > 0
    assert st["n_seq_rejected"] == int((~kept & live_seq).sum())
    assert st["n_tokens_rejected"] == int((am & ~kept[seq]).sum())


def test_large_vocab_sparse_mask_exact_dW():
    """Full V and H, a few hundred active rows: dW parity on every element."""
    s = _setup("large_vocab")
    w = s["w"]
    rng = np.random.default_rng(77)
    act = np.sort(rng.choice(w.T, size=300, replace=False))
    mask = np.zeros(w.T, np.uint8)
    mask[act] = 1
    h_rows64 = np.zeros((w.T, w.H))
    h_rows64[act] = O.widen_bf16(w.hidden[act])
    lp, _ = O.token_logprobs(h_rows64, s["W64"], w.tokens, None, rows=act)
    b = np.full(w.T, -12.0)
    b[act] = lp + boundary_safe_noise(rng, act.size, 0.3, w.eps_lo, w.eps_hi, 2.5 * BOUNDARY_DELTA)
    b = b.astype(np.float32)
    adv = rng.standard_normal(w.T).astype(np.float32)
    hid, Wd = _device_inputs(s)
    out = molt.policy_loss_fwd_bwd(hid, Wd, t(w.tokens), t(b), t(adv), t(mask), w.eps_lo, w.eps_hi)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    ref = O.policy_loss_rows(h_rows64, s["W64"], w.tokens, b.astype(np.float64), adv.astype(np.float64), mask,
                             w.eps_lo, w.eps_hi, float(act.size), act, want_dW=True)
    assert_grad_close(np_(out["dW"]), ref["dW"], "dW (sparse mask, full V x H)")
    dh = np_(out["dhidden"])
    assert_grad_close(dh[act], ref["dH"], "dhidden (sparse mask)")
    assert not dh[mask == 0].any()
    assert abs(float(out["loss"].item()) - ref["token_loss"].sum() / act.size) <= 1e-3 * max(
        1e-3, float(np.abs(ref["ratio"] * adv[act]).sum() / act.size))


# ------------------------------------------------- long trajectory, ragged
@pytest.mark.parametrize("name", ["long_traj", "ragged"])
def test_policy_loss_full_forward(name):
    s = _setup(name)
    _check_call(s, _loss_call(s), label=name)


# ---------------------------------------------------------------- mid, whole
def test_mid_whole():
    """Mid in one call against the oracle's full forward and backward: every
    active row's logp, entropy, per-token loss and dhidden row, and every
    element of the 32000 x 2048 dW."""
    _CACHE.clear()
    w = make_workload("mid")
    act = np.nonzero(w.mask)[0]
    W64 = O.widen_bf16(w.weight)
    h64 = O.widen_bf16(w.hidden)
    t0 = time.perf_counter()
    _, lp0, _ = O.full_forward_rows(h64, W64, w.tokens, act, workers=WORKERS)
    rng = np.random.default_rng(31)
    b = rng.normal(-np.log(w.V) - 1.0, 1.0, w.T)
    b[act] = lp0 + boundary_safe_noise(rng, act.size, w.behavior_sigma, w.eps_lo, w.eps_hi, 2.5 * BOUNDARY_DELTA)
    b = b.astype(np.float32)
    adv = O.broadcast_advantages(O.group_advantages(w.rewards, w.group_ids), w.resp_of_token)
    ref = O.policy_loss(h64, W64, w.tokens, b.astype(np.float64), adv.astype(np.float64), w.mask, w.eps_lo,
                        w.eps_hi, block=512)
    print(f"\n[oracle] mid forward + backward: {time.perf_counter() - t0:.1f} s")
    out = molt.policy_loss_fwd_bwd(bf(w.hidden), bf(w.weight), t(w.tokens), t(b), t(adv.astype(np.float32)),
                                   t(w.mask), w.eps_lo, w.eps_hi)
    torch.cuda.synchronize()
    assert molt.device_status() == 0
    lp, ent, tl = np_(out["logp"]), np_(out["entropy"]), np_(out["token_loss"])
    assert np.abs(lp - ref["logp"]).max() <= LOGP_ATOL
    assert np.abs(ent - ref["entropy"]).max() <= LOGP_ATOL
    np.testing.assert_allclose(tl, ref["token_loss"], rtol=5e-3, atol=1e-6)
    L = float(out["loss"].item())
    scale = max(abs(ref["loss"]), float(np.abs(ref["ratio"] * adv).sum() / ref["denom"]))
    assert abs(L - ref["loss"]) <= LOSS_RTOL * scale, (L, ref["loss"])
    dh = np_(out["dhidden"])
    assert_grad_close(dh[act], ref["dH"][act], "dhidden (mid, every active row)")
    assert not dh[w.mask == 0].any()
    assert_grad_close(np_(out["dW"]), ref["dW"], "dW (mid, every element)")
    st = molt.stats_dict(out["stats"])
    assert st["n_active"] == act.size
    clipped = ref["clipped"][act]
    assert st["n_clip_low"] == int((clipped & (adv[act] < 0)).sum())
    assert st["n_clip_high"] == int((clipped & (adv[act] > 0)).sum())


# ------------------------------------------------- the whole ragged window
def test_fullsize_whole_ragged_window_in_one_call():
    """The ragged configuration's first 16 microbatches (1,048,576 tokens, H =
    5120) in one call: T x H = 5.4e9 elements, past 2^32, so every row offset
    of the packing, the backward and the casts needs 64-bit arithmetic.
    Sampled rows (random active rows across the whole window plus one tile near
    its end) against the oracle, and the whole-call properties of the
    full-size tests, evaluated in row chunks."""
    _CACHE.clear()
    w = make_workload("ragged", T=16 * 65536)
    assert w.T == 16 * 65536 and w.T * w.H > 2 ** 32
    rng = np.random.default_rng(4321)
    act_idx = np.nonzero(w.mask)[0]
    rows = np.unique(np.concatenate([rng.choice(act_idx, size=96, replace=False),
                                     act_idx[-(act_idx.size % 128 + 128):][:128]]))
    assert rows.max() * w.H > 2 ** 32
    W64 = O.widen_bf16(w.weight)
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
