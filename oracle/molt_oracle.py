"""fp64 CPU oracle for the per-token policy-update path of MOLT (arxiv 2607.21653).

TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check of the package entry
file and the CPU-baseline leg of the benchmark may import this module.  It
shares no code with the CUDA library and imports nothing from it.

Every function is a plain restatement of a definition, in fp64, applied to the
exact bits the GPU reads (bf16 hidden states and weights widened exactly).
Library primitives used as steps: numpy matmul (the LM-head product), exp/log.
There is no blocking, fusion or reordering beyond splitting rows into blocks
to bound memory, which does not change any per-element result.

What the paper fixes and what is a stated reading (the paper describes the
method at framework level only):

* Group advantage (Sec. 4.5: GRPO among the estimators; Sec. 4.2: a rollout's
  reward is counted once and mapped back to its segments).  Reading: per
  contiguous prompt group, A_j = (r_j - mean) / (std + eps) with the unbiased
  (n-1) standard deviation, eps = 1e-6 added outside the square root, a group of
  one response gets A = 0, and a zero-variance group gets exactly 0.  The fp64
  sums run in index order; the result is rounded once to fp32.
* Recomputed log-probabilities (Sec. 4.5, "the actor's recomputed
  probabilities"): z = h W^T, lse = log sum exp z, logp = z[x] - lse.
* Entropy (not in the paper; part of the hot path's forward outputs): Shannon
  entropy of softmax(z) in nats, H = lse - sum_v p_v z_v.  No gradient.
* Importance ratio against recorded behaviour log-probs (Sec. 4.3, Sec. 4.5):
  rho = exp(logp - b).
* Clipped surrogate (Sec. 4.5 "masking and clipping"; PPO is the cited
  objective).  Reading: l = -min(rho*A, clip(rho, 1-eps_lo, 1+eps_hi)*A), with
  asymmetric clip bounds and no KL, entropy bonus or dual clip.  The clipped
  branch is selected when (A>0 and rho>1+eps_hi) or (A<0 and rho<1-eps_lo),
  which is the same minimum written as a rule; ties count as unclipped.
* Token-mean normalisation, Eq. 2: L = sum_i m_i l_i / D with one denominator D
  for the whole optimizer window; D defaults to sum_i m_i of the call.
* Backward: dL/dz_tv = (m_t / D) c_t (p_tv - [v == x_t]) with c_t = rho_t A_t on
  the unclipped branch and 0 on the clipped one; dH = G W, dW = G^T h.

* Extended objective (policy_loss_ex; Sec. 4.5 names KL control and
  rejection/weighting rules among the configurable pieces).  Readings: the KL
  penalty to a reference policy is the per-token non-negative estimator
  KL_t = e^r - r - 1 with r = ref_t - logp_t, weighted by kl_coef; the entropy
  bonus subtracts entropy_coef * H_t and, unlike the reported entropy, carries
  a gradient; the sequence gate rejects a whole sequence when the geometric
  mean of its active tokens' ratios lies outside [gate_lo, gate_hi], setting
  w_t = 0 for its tokens while D stays as given (Eq. 2 is not renormalised).
  Per-row gradient: (m w / D)[(c + kl_coef(e^r - 1))(p - onehot)
  + entropy_coef p (z - sum_v p_v z_v)].

Pins (tests/test_oracle.py): closed-form advantages, zero/one-response groups,
library log_softmax / entropy, sum exp(logp) = 1, the rho = 1 case against the
autograd gradient of advantage-weighted cross-entropy, clipped rows having zero
gradient, special clip values, finite differences of the loss, microbatch-split
invariance of Eq. 2 and segment-split invariance of the advantages; for the
extended objective, torch autograd of PPO + k3 KL - entropy bonus, the
reduction to the plain loss, hand-built gate cases, and policy_loss_ex_rows as
an exact slice of policy_loss_ex.
"""
from __future__ import annotations

import math
from concurrent.futures import ThreadPoolExecutor

import numpy as np

__all__ = [
    "widen_bf16", "group_advantages", "advantages", "ESTIMATORS", "broadcast_advantages", "logits_rows",
    "row_softmax_stats", "token_logprobs", "policy_loss", "policy_loss_rows",
    "clip_decision", "surrogate", "policy_loss_ex", "sequence_gate", "policy_loss_ex_rows",
    "full_forward_rows", "dW_rows", "shard_partials", "merge_shard_partials", "shard_dhidden",
]

DEFAULT_ADV_EPS = 1e-6


def widen_bf16(bits: np.ndarray) -> np.ndarray:
    """bf16 bit pattern -> fp64 value (exact)."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


# --------------------------------------------------------------------------- #
# Advantages (Sec. 4.5 GRPO; Sec. 4.2 segments share the rollout reward)
# --------------------------------------------------------------------------- #
def group_advantages(rewards: np.ndarray, group_ids: np.ndarray,
                     eps: float = DEFAULT_ADV_EPS) -> np.ndarray:
    """GRPO group-normalised advantage per response, groups = maximal runs of
    equal consecutive ids.  Plain fp64 loops in index order; each operation is
    one correctly rounded IEEE double operation, result rounded to fp32."""
    r = np.asarray(rewards, dtype=np.float32)
    g = np.asarray(group_ids)
    n = r.shape[0]
    out = np.zeros(n, dtype=np.float32)
    start = 0
    while start < n:
        end = start + 1
        while end < n and g[end] == g[start]:
            end += 1
        cnt = end - start
        if cnt > 1:
            s = 0.0
            for j in range(start, end):
                s = s + float(r[j])
            mean = s / float(cnt)
            ss = 0.0
            for j in range(start, end):
                d = float(r[j]) - mean
                ss = ss + d * d
            std = math.sqrt(ss / float(cnt - 1))
            den = std + eps
            for j in range(start, end):
                out[j] = np.float32((float(r[j]) - mean) / den)
        start = end
    return out


ESTIMATORS = ("grpo", "group_mean", "dr_grpo", "rloo", "reinforce_pp")


def _runs(group_ids):
    g = np.asarray(group_ids)
    n = g.shape[0]
    start = 0
    while start < n:
        end = start + 1
        while end < n and g[end] == g[start]:
            end += 1
        yield start, end
        start = end


def advantages(rewards: np.ndarray, group_ids: np.ndarray, estimator: str = "grpo",
               eps: float = DEFAULT_ADV_EPS) -> np.ndarray:
    """The advantage estimators Sec. 4.5 lists, one reward per rollout (Sec. 4.2):

    grpo          (r - mean_g) / (std_g + eps), unbiased std (see group_advantages)
    group_mean    r - mean_g                           (group-mean baseline)
    dr_grpo       r - mean_g  (Dr. GRPO drops the std division; its length
                  normalisation is already the token-mean of Eq. 2)
    rloo          r_j - (sum_g r - r_j) / (n_g - 1)    (leave-one-out baseline)
    reinforce_pp  (r - mean_B) / (std_B + eps) over the whole batch B

    Groups of one response (a batch of one for reinforce_pp) give 0.  fp64
    sums in index order, one correctly rounded IEEE op at a time, one final
    rounding to fp32."""
    if estimator == "grpo":
        return group_advantages(rewards, group_ids, eps)
    r = np.asarray(rewards, dtype=np.float32)
    n = r.shape[0]
    out = np.zeros(n, dtype=np.float32)
    if estimator == "reinforce_pp":
        runs = [(0, n)] if n > 0 else []
    elif estimator in ("group_mean", "dr_grpo", "rloo"):
        runs = list(_runs(group_ids))
    else:
        raise ValueError(f"unknown estimator {estimator!r}")
    for start, end in runs:
        cnt = end - start
        if cnt < 2:
            continue
        s = 0.0
        for j in range(start, end):
            s = s + float(r[j])
        if estimator == "rloo":
            for j in range(start, end):
                baseline = (s - float(r[j])) / float(cnt - 1)
                out[j] = np.float32(float(r[j]) - baseline)
            continue
        mean = s / float(cnt)
        if estimator in ("group_mean", "dr_grpo"):
            for j in range(start, end):
                out[j] = np.float32(float(r[j]) - mean)
            continue
        ss = 0.0
        for j in range(start, end):
            d = float(r[j]) - mean
            ss = ss + d * d
        den = math.sqrt(ss / float(cnt - 1)) + eps
        for j in range(start, end):
            out[j] = np.float32((float(r[j]) - mean) / den)
    return out


def broadcast_advantages(adv_resp: np.ndarray, resp_of_token: np.ndarray) -> np.ndarray:
    """Per-token advantage = advantage of the rollout the token belongs to."""
    return np.asarray(adv_resp, dtype=np.float32)[np.asarray(resp_of_token)]


# --------------------------------------------------------------------------- #
# Log-softmax, gather, entropy (Sec. 4.5 recomputed probabilities)
# --------------------------------------------------------------------------- #
def logits_rows(h_rows: np.ndarray, W: np.ndarray) -> np.ndarray:
    """z = h W^T for a block of rows (fp64)."""
    return h_rows @ W.T


def row_softmax_stats(z: np.ndarray, x: np.ndarray):
    """For each row of z: lse, logp of target x, entropy, probabilities p."""
    M = z.max(axis=1, keepdims=True)
    e = np.exp(z - M)
    ssum = e.sum(axis=1, keepdims=True)
    lse = (M + np.log(ssum))[:, 0]
    p = np.exp(z - lse[:, None])
    logp = z[np.arange(z.shape[0]), x] - lse
    ent = lse - (p * z).sum(axis=1)
    return lse, logp, ent, p


def token_logprobs(hidden: np.ndarray, W: np.ndarray, tokens: np.ndarray, mask: np.ndarray | None,
                   rows: np.ndarray | None = None, block: int = 64):
    """logp and entropy per token (fp64).  `hidden`/`W` are fp64 (use widen_bf16
    on bf16 bits).  Rows with mask 0 are not computed and return 0.  If `rows`
    is given, only those row indices are computed (returned in that order)."""
    T = hidden.shape[0]
    idx = np.arange(T) if rows is None else np.asarray(rows)
    logp = np.zeros(idx.shape[0])
    ent = np.zeros(idx.shape[0])
    act = np.ones(idx.shape[0], dtype=bool) if mask is None else (np.asarray(mask)[idx] != 0)
    sel = np.nonzero(act)[0]
    for b0 in range(0, sel.shape[0], block):
        k = sel[b0:b0 + block]
        t = idx[k]
        z = logits_rows(hidden[t], W)
        _, lp, en, _ = row_softmax_stats(z, np.asarray(tokens)[t])
        logp[k] = lp
        ent[k] = en
    return logp, ent


# --------------------------------------------------------------------------- #
# Ratio, clipped surrogate, Eq. 2 normalisation and the backward pass
# --------------------------------------------------------------------------- #
def clip_decision(rho: np.ndarray, adv: np.ndarray, eps_lo: float, eps_hi: float) -> np.ndarray:
    """True where the clipped term of min(rho*A, clip(rho)*A) is the smaller one."""
    lo = 1.0 - float(eps_lo)
    hi = 1.0 + float(eps_hi)
    return ((adv > 0) & (rho > hi)) | ((adv < 0) & (rho < lo))


def surrogate(rho: np.ndarray, adv: np.ndarray, eps_lo: float, eps_hi: float):
    """Per-token loss l = -min(rho A, clip(rho) A) and its derivative coefficient
    c = -dl/dlogp (rho A on the unclipped branch, 0 on the clipped one)."""
    lo = 1.0 - float(eps_lo)
    hi = 1.0 + float(eps_hi)
    clipped = clip_decision(rho, adv, eps_lo, eps_hi)
    rho_c = np.minimum(np.maximum(rho, lo), hi)
    loss = np.where(clipped, -rho_c * adv, -rho * adv)
    coef = np.where(clipped, 0.0, rho * adv)
    return loss, coef, clipped


def policy_loss_rows(hidden: np.ndarray, W: np.ndarray, tokens: np.ndarray,
                     behavior_logp: np.ndarray, adv: np.ndarray, mask: np.ndarray,
                     eps_lo: float, eps_hi: float, denom: float, rows: np.ndarray,
                     want_dW: bool = False, block: int = 64):
    """Per-row forward quantities and dH rows for the given row indices.

    Returns dict with logp, entropy, lse, ratio, token_loss (m*l), coef
    (m*c/D), clipped, dH (len(rows) x H) and, if want_dW, the contribution of
    these rows to dW (V x H).  Each row is independent of the others, so this
    is exactly the corresponding slice of the full computation."""
    rows = np.asarray(rows)
    n = rows.shape[0]
    H = hidden.shape[1]
    out = {k: np.zeros(n) for k in ("logp", "entropy", "lse", "ratio", "token_loss", "coef")}
    out["clipped"] = np.zeros(n, dtype=bool)
    out["dH"] = np.zeros((n, H))
    dW = np.zeros_like(W) if want_dW else None
    m_all = np.asarray(mask).astype(np.float64)
    for b0 in range(0, n, block):
        sl = slice(b0, min(n, b0 + block))
        t = rows[sl]
        m = m_all[t]
        act = m != 0
        if not act.any():
            continue
        t_a = t[act]
        pos = np.arange(sl.start, sl.stop)[act]
        h_a = hidden[t_a]
        x = np.asarray(tokens)[t_a]
        z = logits_rows(h_a, W)
        lse, logp, ent, p = row_softmax_stats(z, x)
        rho = np.exp(logp - np.asarray(behavior_logp, dtype=np.float64)[t_a])
        a = np.asarray(adv, dtype=np.float64)[t_a]
        loss, c, clipped = surrogate(rho, a, eps_lo, eps_hi)
        coef = c / denom                       # m = 1 on these rows
        g = coef[:, None] * p
        g[np.arange(g.shape[0]), x] -= coef
        out["logp"][pos] = logp
        out["entropy"][pos] = ent
        out["lse"][pos] = lse
        out["ratio"][pos] = rho
        out["token_loss"][pos] = loss
        out["coef"][pos] = coef
        out["clipped"][pos] = clipped
        out["dH"][pos] = g @ W
        if want_dW:
            dW += g.T @ h_a
    out["dW"] = dW
    return out


def policy_loss(hidden: np.ndarray, W: np.ndarray, tokens: np.ndarray, behavior_logp: np.ndarray,
                adv: np.ndarray, mask: np.ndarray, eps_lo: float, eps_hi: float,
                denom: float | None = None, block: int = 64):
    """Full fp64 forward + backward of the token-mean clipped surrogate (Eq. 2).

    hidden [T,H] and W [V,H] are fp64; adv is the per-token advantage.  Returns
    loss, per-token quantities (masked rows 0), dH [T,H], dW [V,H] and the
    window statistics."""
    T = hidden.shape[0]
    m = np.asarray(mask).astype(np.float64)
    D = float(m.sum()) if (denom is None or denom <= 0) else float(denom)
    if D == 0.0:
        raise ZeroDivisionError("Eq. 2 needs a nonzero denominator")
    r = policy_loss_rows(hidden, W, tokens, behavior_logp, adv, mask, eps_lo, eps_hi, D,
                         np.arange(T), want_dW=True, block=block)
    loss = float(r["token_loss"].sum() / D)
    act = m != 0
    a = np.asarray(adv, dtype=np.float64)
    n_act = int(act.sum())
    stats = {
        "n_active": n_act,
        "loss": loss,
        "clip_frac_low": float(((r["clipped"]) & (a < 0) & act).sum() / max(1, n_act)),
        "clip_frac_high": float(((r["clipped"]) & (a > 0) & act).sum() / max(1, n_act)),
        "mean_ratio": float(r["ratio"][act].mean()) if n_act else 0.0,
        "mean_entropy": float(r["entropy"][act].mean()) if n_act else 0.0,
        "max_abs_log_ratio": float(np.abs(np.log(r["ratio"][act])).max()) if n_act else 0.0,
    }
    r.update(loss=loss, denom=D, stats=stats)
    return r


# --------------------------------------------------------------------------- #
# Extended objective: KL to a reference policy, entropy bonus, sequence gate
# --------------------------------------------------------------------------- #
def sequence_gate(log_ratio: np.ndarray, seq: np.ndarray, mask: np.ndarray, lo: float, hi: float) -> np.ndarray:
    """Per-token weight w_t in {0, 1} of a sequence-level importance gate
    (Sec. 4.5: "a configurable rejection or weighting rule"; Sec. 4.3).
    Reading: a sequence (maximal run of equal consecutive ids) is rejected when
    the geometric mean of its active tokens' ratios, exp(mean_t (logp_t - b_t)),
    lies outside [lo, hi]; all its tokens get w = 0.  fp64 sums in index order.
    Tokens of sequences without active tokens keep w = 1 (they carry no loss)."""
    lr = np.asarray(log_ratio, dtype=np.float64)
    m = np.asarray(mask)
    w = np.ones(lr.shape[0])
    for start, end in _runs(seq):
        s, n = 0.0, 0
        for t in range(start, end):
            if m[t]:
                s = s + float(lr[t])
                n += 1
        if n == 0:
            continue
        g = math.exp(s / float(n))
        if g < lo or g > hi:
            w[start:end] = 0.0
    return w


def policy_loss_ex(hidden: np.ndarray, W: np.ndarray, tokens: np.ndarray, behavior_logp: np.ndarray,
                   adv: np.ndarray, mask: np.ndarray, eps_lo: float, eps_hi: float, denom: float | None = None,
                   kl_coef: float = 0.0, ref_logp: np.ndarray | None = None, entropy_coef: float = 0.0,
                   seq_of_token: np.ndarray | None = None, gate_lo: float = 0.0, gate_hi: float = float("inf"),
                   block: int = 64):
    """Full fp64 forward + backward of the extended per-token loss

        l_t = w_t (l_pg,t + kl_coef KL_t - entropy_coef H_t),   L = sum_t m_t l_t / D

    l_pg the clipped surrogate (see surrogate), KL_t = exp(r) - r - 1 with
    r = ref_t - logp_t (the non-negative "k3" estimator of KL(pi || ref)), H_t
    the token entropy, w_t the sequence-gate weight (1 without a gate).  D is
    the Eq. 2 denominator (sum of the mask by default); rejected sequences do
    not change it ("does not renormalize by the number of accepted sequences").
    Gradient per row: (m w / D) [ (c + kl_coef (e^r - 1)) (p - onehot)
                                  + entropy_coef p (z - sum_v p_v z_v) ]."""
    T = hidden.shape[0]
    m = np.asarray(mask).astype(np.float64)
    D = float(m.sum()) if (denom is None or denom <= 0) else float(denom)
    if D == 0.0:
        raise ZeroDivisionError("Eq. 2 needs a nonzero denominator")
    x_all = np.asarray(tokens)
    b_all = np.asarray(behavior_logp, dtype=np.float64)
    a_all = np.asarray(adv, dtype=np.float64)
    # pass 1: log-probs of every active row (needed by the gate)
    logp_all, ent_all = token_logprobs(hidden, W, x_all, mask, block=block)
    w = np.ones(T)
    if seq_of_token is not None:
        w = sequence_gate(logp_all - b_all, seq_of_token, mask, gate_lo, gate_hi)
    out = {k: np.zeros(T) for k in ("logp", "entropy", "ratio", "token_loss", "coef", "kl")}
    out["clipped"] = np.zeros(T, dtype=bool)
    out["gate"] = w
    dH = np.zeros_like(hidden)
    dW = np.zeros_like(W)
    act = np.nonzero(m != 0)[0]
    for b0 in range(0, act.shape[0], block):
        t = act[b0:b0 + block]
        z = logits_rows(hidden[t], W)
        lse, logp, ent, p = row_softmax_stats(z, x_all[t])
        rho = np.exp(logp - b_all[t])
        l_pg, c, clipped = surrogate(rho, a_all[t], eps_lo, eps_hi)
        if ref_logp is not None and kl_coef != 0.0:
            r = np.asarray(ref_logp, dtype=np.float64)[t] - logp
            kl = np.exp(r) - r - 1.0
            c_kl = kl_coef * (np.exp(r) - 1.0)
        else:
            kl = np.zeros_like(logp)
            c_kl = np.zeros_like(logp)
        wt = w[t]
        l_t = wt * (l_pg + kl_coef * kl - entropy_coef * ent)
        coef = wt * (c + c_kl) / D
        mu = (p * z).sum(axis=1)
        g = coef[:, None] * p
        g[np.arange(t.shape[0]), x_all[t]] -= coef
        if entropy_coef != 0.0:
            g += (wt * entropy_coef / D)[:, None] * p * (z - mu[:, None])
        dH[t] = g @ W
        dW += g.T @ hidden[t]
        out["logp"][t] = logp
        out["entropy"][t] = ent
        out["ratio"][t] = rho
        out["token_loss"][t] = l_t
        out["coef"][t] = coef
        out["kl"][t] = kl
        out["clipped"][t] = clipped
    out.update(loss=float(out["token_loss"].sum() / D), denom=D, dH=dH, dW=dW)
    return out


def policy_loss_ex_rows(hidden: np.ndarray, W: np.ndarray, tokens: np.ndarray, behavior_logp: np.ndarray,
                        adv: np.ndarray, mask: np.ndarray, eps_lo: float, eps_hi: float, denom: float,
                        rows: np.ndarray, kl_coef: float = 0.0, ref_logp: np.ndarray | None = None,
                        entropy_coef: float = 0.0, gate_w: np.ndarray | None = None, block: int = 64):
    """policy_loss_ex restricted to the given rows, with the sequence-gate
    weights w_t supplied (gate_w[t] for every token t; None = all 1): the gate
    needs every token of a sequence, the per-row terms only the row itself.
    Returns logp, entropy, ratio, kl, token_loss (m w l), coef and dH for the
    rows, in their order."""
    rows = np.asarray(rows)
    n = rows.shape[0]
    out = {k: np.zeros(n) for k in ("logp", "entropy", "ratio", "kl", "token_loss", "coef")}
    out["dH"] = np.zeros((n, hidden.shape[1]))
    m_all = np.asarray(mask).astype(np.float64)
    w_all = np.ones(len(m_all)) if gate_w is None else np.asarray(gate_w, dtype=np.float64)
    for b0 in range(0, n, block):
        pos = np.arange(b0, min(n, b0 + block))
        t = rows[pos]
        act = m_all[t] != 0
        if not act.any():
            continue
        pos, t = pos[act], t[act]
        x = np.asarray(tokens)[t]
        z = logits_rows(hidden[t], W)
        lse, logp, ent, p = row_softmax_stats(z, x)
        rho = np.exp(logp - np.asarray(behavior_logp, dtype=np.float64)[t])
        l_pg, c, _ = surrogate(rho, np.asarray(adv, dtype=np.float64)[t], eps_lo, eps_hi)
        if ref_logp is not None and kl_coef != 0.0:
            r = np.asarray(ref_logp, dtype=np.float64)[t] - logp
            kl, c_kl = np.exp(r) - r - 1.0, kl_coef * (np.exp(r) - 1.0)
        else:
            kl, c_kl = np.zeros_like(logp), np.zeros_like(logp)
        wt = w_all[t]
        coef = wt * (c + c_kl) / denom
        g = coef[:, None] * p
        g[np.arange(t.shape[0]), x] -= coef
        if entropy_coef != 0.0:
            mu = (p * z).sum(axis=1)
            g += (wt * entropy_coef / denom)[:, None] * p * (z - mu[:, None])
        out["logp"][pos] = logp
        out["entropy"][pos] = ent
        out["ratio"][pos] = rho
        out["kl"][pos] = kl
        out["token_loss"][pos] = wt * (l_pg + kl_coef * kl - entropy_coef * ent)
        out["coef"][pos] = coef
        out["dH"][pos] = g @ W
    return out


# --------------------------------------------------------------------------- #
# Whole-batch forward and sampled dW rows at the full vocabulary size
# --------------------------------------------------------------------------- #
def _row_stats_block(z: np.ndarray, x: np.ndarray):
    """lse, logp of target x and entropy for each row of z (the definitions of
    row_softmax_stats without returning the probabilities)."""
    M = z.max(axis=1)
    e = np.exp(z - M[:, None])
    s = e.sum(axis=1)
    lse = M + np.log(s)
    logp = z[np.arange(z.shape[0]), x] - lse
    # sum_v p_v z_v with p_v = e_v / s
    ent = lse - (e * z).sum(axis=1) / s
    return lse, logp, ent


def full_forward_rows(hidden: np.ndarray, W: np.ndarray, tokens: np.ndarray, rows: np.ndarray,
                      block: int = 1024, workers: int = 1):
    """lse, logp and entropy (fp64) of every given row against the whole
    vocabulary: z = h W^T, lse = max + log sum exp(z - max), logp = z[x] - lse,
    entropy = lse - sum_v p_v z_v (the definitions of Sec. 4.5's recomputed
    probabilities, as in row_softmax_stats).  One matmul per block of rows;
    the per-row reductions of a block may run on `workers` threads, each over
    its own rows, which changes no per-row result."""
    rows = np.asarray(rows)
    n = rows.shape[0]
    lse = np.zeros(n)
    logp = np.zeros(n)
    ent = np.zeros(n)
    x_all = np.asarray(tokens)
    pool = ThreadPoolExecutor(max_workers=workers) if workers > 1 else None
    try:
        for b0 in range(0, n, block):
            sl = np.arange(b0, min(n, b0 + block))
            t = rows[sl]
            z = logits_rows(hidden[t], W)
            x = x_all[t]
            if pool is None:
                lse[sl], logp[sl], ent[sl] = _row_stats_block(z, x)
                continue
            parts = np.array_split(np.arange(sl.shape[0]), workers)
            res = list(pool.map(lambda p: _row_stats_block(z[p], x[p]), [p for p in parts if p.size]))
            for p, (a, b, c) in zip([p for p in parts if p.size], res):
                lse[sl[p]], logp[sl[p]], ent[sl[p]] = a, b, c
    finally:
        if pool is not None:
            pool.shutdown()
    return lse, logp, ent


def dW_rows(hidden: np.ndarray, W: np.ndarray, tokens: np.ndarray, lse: np.ndarray, coef: np.ndarray,
            rows: np.ndarray, vocab_rows: np.ndarray, block: int = 8192) -> np.ndarray:
    """Rows `vocab_rows` of dW = G^T h, summed over the token rows `rows`:
    dW_v = sum_t g_tv h_t with g_tv = coef_t (exp(z_tv - lse_t) - [v == x_t])
    (the backward of Eq. 2; coef_t = m_t c_t / D and lse_t are per row, in the
    order of `rows`).  Returns len(vocab_rows) x H, fp64."""
    rows = np.asarray(rows)
    vr = np.asarray(vocab_rows)
    x_all = np.asarray(tokens)
    Wv = W[vr]
    out = np.zeros((vr.shape[0], hidden.shape[1]))
    for b0 in range(0, rows.shape[0], block):
        sl = slice(b0, min(rows.shape[0], b0 + block))
        t = rows[sl]
        h = hidden[t]
        z = h @ Wv.T
        g = np.asarray(coef)[sl][:, None] * np.exp(z - np.asarray(lse)[sl][:, None])
        g -= np.asarray(coef)[sl][:, None] * (x_all[t][:, None] == vr[None, :])
        out += g.T @ h
    return out


# --------------------------------------------------------------------------- #
# Vocabulary-parallel pieces (the LM head split by vocabulary ranges)
# --------------------------------------------------------------------------- #
def shard_partials(hidden: np.ndarray, W_shard: np.ndarray, tokens: np.ndarray, v_begin: int,
                   rows: np.ndarray):
    """Per-row statistics of one vocabulary shard (columns v_begin ..
    v_begin + V_shard - 1 of z = h W^T): the shard's max M_s, S_s = sum exp(z -
    M_s), Q_s = sum exp(z - M_s)(z - M_s) and the target logit z[x] when the
    target lies in the shard (-inf otherwise).  Returns an [n, 4] array."""
    rows = np.asarray(rows)
    out = np.zeros((rows.shape[0], 4))
    Vs = W_shard.shape[0]
    for b0 in range(0, rows.shape[0], 256):
        sl = slice(b0, min(rows.shape[0], b0 + 256))
        t = rows[sl]
        z = logits_rows(hidden[t], W_shard)
        M = z.max(axis=1)
        e = np.exp(z - M[:, None])
        out[sl, 0] = M
        out[sl, 1] = e.sum(axis=1)
        out[sl, 2] = (e * (z - M[:, None])).sum(axis=1)
        xl = np.asarray(tokens)[t] - int(v_begin)
        inside = (xl >= 0) & (xl < Vs)
        zx = np.full(t.shape[0], -np.inf)
        zx[inside] = z[np.nonzero(inside)[0], xl[inside]]
        out[sl, 3] = zx
    return out


def merge_shard_partials(parts: np.ndarray):
    """Combine the statistics of disjoint vocabulary shards ([n_shards, n, 4],
    see shard_partials) into lse, logp and entropy of the whole row: with M the
    largest shard max, S = sum_s S_s e^{M_s - M}, lse = M + log S, and
    sum_v p_v z_v = sum_s e^{M_s - M} (Q_s + (M_s - M) S_s) / S + M, so that
    entropy = lse - sum_v p_v z_v; logp = z[x] - lse from the one shard that
    holds the target."""
    parts = np.asarray(parts, dtype=np.float64)
    Ms, Ss, Qs, Zs = parts[..., 0], parts[..., 1], parts[..., 2], parts[..., 3]
    M = Ms.max(axis=0)
    f = np.exp(Ms - M[None, :])
    S = (Ss * f).sum(axis=0)
    lse = M + np.log(S)
    pz = (f * (Qs + (Ms - M[None, :]) * Ss)).sum(axis=0) / S + M
    zx = Zs.max(axis=0)
    return lse, zx - lse, lse - pz


def shard_dhidden(hidden: np.ndarray, W_shard: np.ndarray, tokens: np.ndarray, v_begin: int, lse: np.ndarray,
                  coef: np.ndarray, rows: np.ndarray) -> np.ndarray:
    """One vocabulary shard's term of dhidden for the given rows:
    sum over the shard's columns v of g_tv W_v, with g_tv = coef_t
    (exp(z_tv - lse_t) - [v == x_t]) and lse_t, coef_t of the whole row (in
    the order of `rows`).  The shards' terms sum to dH = G W."""
    rows = np.asarray(rows)
    Vs = W_shard.shape[0]
    out = np.zeros((rows.shape[0], hidden.shape[1]))
    for b0 in range(0, rows.shape[0], 256):
        sl = slice(b0, min(rows.shape[0], b0 + 256))
        t = rows[sl]
        z = logits_rows(hidden[t], W_shard)
        c = np.asarray(coef)[sl]
        g = c[:, None] * np.exp(z - np.asarray(lse)[sl][:, None])
        xl = np.asarray(tokens)[t] - int(v_begin)
        inside = np.nonzero((xl >= 0) & (xl < Vs))[0]
        g[inside, xl[inside]] -= c[inside]
        out[sl] = g @ W_shard
    return out
