"""Seeded synthetic workloads for the per-token policy-update path.

This module only draws inputs: hidden states, LM-head weights, sampled tokens,
loss masks, rollout rewards, prompt-group ids, the segment -> rollout map and
the behaviour-policy noise.  It holds none of the method's arithmetic (no
softmax, no ratio, no advantage); both the fp64 oracle side and the CUDA side
of the tests read the arrays it returns.

Shapes and distributions follow the five workloads of the fused policy-loss
benchmark (tiny, mid, large-vocab, long-trajectory, ragged).  The paper's own
datasets are not used; every array here is synthetic and seeded (numpy PCG64).

Hidden states and weights are returned as bf16 bit patterns (uint16), rounded
from fp32 to nearest-even, so every consumer sees identical bits.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

__all__ = [
    "f32_to_bf16_bits", "bf16_bits_to_f32", "Workload", "make_workload",
    "boundary_safe_noise", "CONFIG_NAMES", "draw_normal_bf16",
]

CONFIG_NAMES = ("tiny", "mid", "large_vocab", "long_traj", "ragged")


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit pattern, round to nearest even (inputs are finite)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def draw_normal_bf16(rng: np.random.Generator, shape, std: float, out: np.ndarray | None = None,
                     chunk_rows: int = 8192) -> np.ndarray:
    """N(0, std^2) fp32 draws rounded to bf16 bits, generated row-chunk by row-chunk
    so that a 151936 x 5120 matrix never needs a full fp32 temporary."""
    rows, cols = shape
    if out is None:
        out = np.empty((rows, cols), dtype=np.uint16)
    for r0 in range(0, rows, chunk_rows):
        r1 = min(rows, r0 + chunk_rows)
        x = rng.standard_normal((r1 - r0, cols), dtype=np.float32)
        if std != 1.0:
            x *= np.float32(std)
        out[r0:r1] = f32_to_bf16_bits(x)
    return out


def boundary_safe_noise(rng: np.random.Generator, n: int, sigma: float, eps_lo: float,
                        eps_hi: float, delta: float) -> np.ndarray:
    """N(0, sigma^2) offsets for behaviour log-probs, redrawn wherever -offset lies
    within `delta` of log(1-eps_lo) or log(1+eps_hi).

    With behaviour = current + offset the importance ratio is exp(-offset), so this
    keeps every token at least `delta` (in log-ratio) away from a clip boundary.
    Tests use it so that the clip decision is unique at the stated log-prob
    tolerance; the distribution differs from N(0, sigma^2) only on those bands."""
    lo, hi = math.log1p(-eps_lo), math.log1p(eps_hi)
    out = rng.normal(0.0, sigma, size=n)
    for _ in range(1000):
        bad = (np.abs(-out - lo) < delta) | (np.abs(-out - hi) < delta)
        k = int(bad.sum())
        if k == 0:
            break
        out[bad] = rng.normal(0.0, sigma, size=k)
    return out


@dataclass
class Workload:
    """One synthetic batch.  Token-level arrays have length T, response-level
    arrays length n_resp.  `hidden`/`weight` are bf16 bits ([T,H], [V,H])."""
    name: str
    T: int
    H: int
    V: int
    hidden: np.ndarray | None
    weight: np.ndarray | None
    tokens: np.ndarray            # int32 [T]
    mask: np.ndarray              # uint8 [T]
    rewards: np.ndarray           # fp32 [n_resp]
    group_ids: np.ndarray         # int32 [n_resp] (contiguous equal-id runs)
    resp_of_token: np.ndarray     # int32 [T]
    behavior_sigma: float
    eps_lo: float
    eps_hi: float
    seed: int
    extra: dict = field(default_factory=dict)


def _spans_mask(rng, T, frac, lmin, lmax, tol=0.01):
    """mask=1 everywhere except contiguous spans (uniform length in [lmin,lmax])
    placed at uniform positions until about `frac` of the tokens are covered."""
    mask = np.ones(T, dtype=np.uint8)
    target = frac * T
    covered = 0
    while covered < target - tol * T:
        L = int(rng.integers(lmin, lmax + 1))
        s = int(rng.integers(0, max(1, T - L)))
        seg = mask[s:s + L]
        covered += int(seg.sum())
        seg[:] = 0
    return mask


def _response_layout(n_groups, G, length):
    n_resp = n_groups * G
    group_ids = np.repeat(np.arange(n_groups, dtype=np.int32), G)
    resp_of_token = np.repeat(np.arange(n_resp, dtype=np.int32), length)
    return n_resp, group_ids, resp_of_token


def make_workload(name: str, *, with_tensors: bool = True, T: int | None = None,
                  H: int | None = None, V: int | None = None, seed: int | None = None,
                  microbatch: int = 0) -> Workload:
    """Build one of the five workloads.

    tiny        T=512 (8 groups x G=4 x 16 tok), H=256, V=4096, rewards Bernoulli(.5),
                mask all 1, behaviour offset N(0,.05), eps .2/.2, seed 0
    mid         T=32768 (64 x G=8 x 64), H=2048, V=32000, rewards uniform {0,1},
                offset N(0,.1), 20% masked in spans of 8-64 tokens, seed 1
    large_vocab T=65536 (128 x G=8 x 64), H=4096, V=151936, rewards U[0,1],
                30% masked in spans of 8-256, eps .2/.28, offset N(0,.05), seed 2
    long_traj   8 trajectories x 16384 (T=131072), one prompt group of G=8, each
                trajectory cut into 2-6 segments; H=4096, V=151936, rewards
                Bernoulli(.5), 50% masked in spans of 64-2048, offset N(0,.2), seed 3
    ragged      256 groups x G=16, lengths log-uniform in [32,8192] (~6M tokens),
                processed in 65536-token microbatches; H=5120, V=151936, rewards
                Bernoulli(.3) with group 0 all-0 and group 1 all-1, >=1% of
                responses fully masked, offset N(0,.1), seed 4.  `microbatch`
                selects which 65536-token slice the token arrays cover.

    T/H/V overrides shrink a workload (same structure recipe) for fast tests.
    """
    if name not in CONFIG_NAMES:
        raise ValueError(f"unknown workload {name!r}")
    idx = CONFIG_NAMES.index(name)
    seed = idx if seed is None else seed
    rng = np.random.Generator(np.random.PCG64(seed))
    extra: dict = {}

    if name == "tiny":
        Td, Hd, Vd = 512, 256, 4096
        n_groups, G, length = 8, 4, 16
        T_ = T or Td
        length = max(1, T_ // (n_groups * G)) if T else length
        n_resp, group_ids, rot = _response_layout(n_groups, G, length)
        rot = np.resize(rot, T_).astype(np.int32)
        rewards = (rng.random(n_resp) < 0.5).astype(np.float32)
        mask = np.ones(T_, dtype=np.uint8)
        sigma, eps_lo, eps_hi = 0.05, 0.2, 0.2
    elif name == "mid":
        Td, Hd, Vd = 32768, 2048, 32000
        n_groups, G, length = 64, 8, 64
        T_ = T or Td
        n_resp, group_ids, rot = _response_layout(n_groups, G, length)
        rot = np.resize(rot, T_).astype(np.int32)
        rewards = rng.integers(0, 2, size=n_resp).astype(np.float32)
        mask = _spans_mask(rng, T_, 0.20, 8, 64)
        sigma, eps_lo, eps_hi = 0.1, 0.2, 0.2
    elif name == "large_vocab":
        Td, Hd, Vd = 65536, 4096, 151936
        n_groups, G, length = 128, 8, 64
        T_ = T or Td
        n_resp, group_ids, rot = _response_layout(n_groups, G, length)
        rot = np.resize(rot, T_).astype(np.int32)
        rewards = rng.random(n_resp).astype(np.float32)
        mask = _spans_mask(rng, T_, 0.30, 8, min(256, max(8, T_ // 4)))
        sigma, eps_lo, eps_hi = 0.05, 0.2, 0.28
    elif name == "long_traj":
        Td, Hd, Vd = 131072, 4096, 151936
        n_traj, traj_len = 8, 16384
        T_ = T or Td
        traj_len = T_ // n_traj if T else traj_len
        n_resp = n_traj
        group_ids = np.zeros(n_traj, dtype=np.int32)          # one prompt group, G=8
        rot = np.repeat(np.arange(n_traj, dtype=np.int32), traj_len)
        rot = np.resize(rot, T_).astype(np.int32)
        # compaction points: each trajectory is cut into 2-6 segments; segments keep
        # their rollout id (resp_of_token) and so share the rollout's reward
        seg_id = np.zeros(T_, dtype=np.int32)
        sid = 0
        for r in range(n_traj):
            k = int(rng.integers(2, 7))
            cuts = np.sort(rng.choice(np.arange(1, traj_len), size=k - 1, replace=False))
            bounds = np.concatenate([[0], cuts, [traj_len]]) + r * traj_len
            for a, b in zip(bounds[:-1], bounds[1:]):
                seg_id[a:min(b, T_)] = sid
                sid += 1
        extra["segment_of_token"] = seg_id
        rewards = (rng.random(n_resp) < 0.5).astype(np.float32)
        mask = _spans_mask(rng, T_, 0.50, 64, min(2048, max(64, T_ // 4)))
        sigma, eps_lo, eps_hi = 0.2, 0.2, 0.2
    else:  # ragged
        Td, Hd, Vd = 65536, 5120, 151936
        n_groups, G = 256, 16
        n_resp = n_groups * G
        lengths = np.exp(rng.uniform(math.log(32), math.log(8192), size=n_resp)).astype(np.int64)
        group_ids = np.repeat(np.arange(n_groups, dtype=np.int32), G)
        rewards = (rng.random(n_resp) < 0.3).astype(np.float32)
        rewards[0:G] = 0.0
        rewards[G:2 * G] = 1.0
        fully_masked = rng.choice(n_resp, size=max(41, n_resp // 100), replace=False)
        starts = np.concatenate([[0], np.cumsum(lengths)[:-1]])
        total = int(lengths.sum())
        extra["window_tokens"] = total
        extra["lengths"] = lengths
        T_ = T or Td
        t0 = microbatch * T_
        if t0 >= total:
            raise ValueError("microbatch beyond the ragged window")
        t1 = min(total, t0 + T_)
        rot_full_slice = np.searchsorted(starts, np.arange(t0, t1), side="right") - 1
        rot = rot_full_slice.astype(np.int32)
        fm = np.zeros(n_resp, dtype=bool)
        fm[fully_masked] = True
        mask = (~fm[rot]).astype(np.uint8)
        # the window denominator spans every microbatch of the window (Eq. 2)
        all_rot_lengths = lengths.copy()
        all_rot_lengths[fm] = 0
        extra["window_denominator"] = float(all_rot_lengths.sum())
        extra["fully_masked_responses"] = np.sort(fully_masked)
        T_ = t1 - t0
        sigma, eps_lo, eps_hi = 0.1, 0.2, 0.2

    H_ = H or Hd
    V_ = V or Vd
    tokens = rng.integers(0, V_, size=T_, dtype=np.int64).astype(np.int32)
    hidden = weight = None
    if with_tensors:
        # separate streams so that shrinking T does not change W and vice versa
        rh = np.random.Generator(np.random.PCG64([seed, 1, microbatch]))
        rw = np.random.Generator(np.random.PCG64([seed, 2]))
        hidden = draw_normal_bf16(rh, (T_, H_), 1.0)
        weight = draw_normal_bf16(rw, (V_, H_), 0.02)
    return Workload(name=name, T=T_, H=H_, V=V_, hidden=hidden, weight=weight, tokens=tokens,
                    mask=mask, rewards=rewards, group_ids=group_ids, resp_of_token=rot,
                    behavior_sigma=sigma, eps_lo=eps_lo, eps_hi=eps_hi, seed=seed, extra=extra)


def random_problem(rng: np.random.Generator, T: int, H: int, V: int, mask_frac: float = 0.0,
                   w_std: float = 0.02):
    """Small free-form problem for ragged-shape tests: bf16 bits + tokens + mask."""
    hidden = draw_normal_bf16(rng, (T, H), 1.0)
    weight = draw_normal_bf16(rng, (V, H), w_std)
    tokens = rng.integers(0, V, size=T).astype(np.int32)
    mask = (rng.random(T) >= mask_frac).astype(np.uint8)
    return hidden, weight, tokens, mask
