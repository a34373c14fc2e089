"""Helpers shared by the GPU parity tests: device transfer of the seeded
inputs, oracle references and the tolerance checks.

Tolerances (fp32 results of bf16 tensor-core products with fp32 accumulation
against the fp64 oracle on the same bf16 bits):
  advantages          bit-exact
  logp, entropy       max abs error <= 2e-3
  loss                |dL| <= 1e-3 * max(|L|, sum m |rho A| / D)
  dhidden, dW         max|d| / max|ref| <= 2e-2 per tensor and cosine >= 0.9999
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import molt_oracle as O
from workloads import boundary_safe_noise

LOGP_ATOL = 2e-3
LOSS_RTOL = 1e-3
GRAD_NORMWISE = 2e-2
GRAD_COSINE = 0.9999
# clip decisions are compared only where the oracle's log-ratio is at least this
# far from a clip boundary (twice the log-prob tolerance)
BOUNDARY_DELTA = 2 * LOGP_ATOL


def dev():
    return torch.device("cuda", torch.cuda.current_device())


def t(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev())


def bf(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(dev()).view(torch.bfloat16)


def np_(x):
    return x.detach().float().cpu().numpy() if x.dtype == torch.bfloat16 else x.detach().cpu().numpy()


def behavior_from_oracle(h64, W64, tokens, sigma, eps_lo, eps_hi, seed, rows=None):
    """behaviour log-probs = oracle current log-probs + N(0, sigma) offsets kept
    BOUNDARY_DELTA away from the clip boundaries."""
    lp, _ = O.token_logprobs(h64, W64, tokens, None, rows=rows)
    rng = np.random.default_rng(seed)
    return (lp + boundary_safe_noise(rng, lp.shape[0], sigma, eps_lo, eps_hi, 2.5 * BOUNDARY_DELTA)).astype(np.float32)


def assert_grad_close(got, ref, name):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    scale = np.abs(ref).max()
    err = np.abs(got - ref).max()
    assert scale > 0 or err == 0, f"{name}: reference is zero but result is not"
    if scale == 0:
        return
    cos = float((got * ref).sum() / (np.linalg.norm(got) * np.linalg.norm(ref)))
    assert err <= GRAD_NORMWISE * scale, f"{name}: max err {err:.3e} vs max ref {scale:.3e} (ratio {err / scale:.3e})"
    assert cos >= GRAD_COSINE, f"{name}: cosine {cos:.6f}"


def assert_loss_close(L, ref):
    scale = max(abs(ref["loss"]), float(np.abs(ref["ratio"] * ref["_adv"]).sum() / ref["denom"]))
    assert abs(L - ref["loss"]) <= LOSS_RTOL * scale, f"loss {L} vs oracle {ref['loss']} (scale {scale})"
