"""Python binding of libmolt: the GB300 (sm_103a) policy-update hot path of
MOLT (arxiv 2607.21653).

Every function here only marshals arguments into the C ABI declared in
include/molt.h: torch CUDA tensors become raw device pointers, the current CUDA
stream is passed along, and every step runs in the library's CUDA kernels.
There is no CPU fallback: if the library is not built, or a tensor is not on a
CUDA device, the call raises.
"""
from __future__ import annotations

import ctypes
import os
import re
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

__all__ = [
    "build", "load", "lib_path", "MoltError", "STATUS", "DEV_FLAGS", "group_advantages",
    "broadcast_advantages", "mask_count", "token_logprobs", "policy_loss_fwd_bwd", "device_status",
    "token_logprobs_workspace_bytes", "policy_loss_workspace_bytes", "header_functions",
    "vp_partials", "vp_loss", "vp_backward", "vocab_shard_bounds", "gather_shard_partials", "sum_dhidden",
    "policy_loss_vocab_parallel",
]

_PKG = os.path.dirname(os.path.abspath(__file__))
_ROOT = os.path.dirname(_PKG)
_CSRC = os.path.join(_PKG, "csrc")
_INCLUDE = os.path.join(_ROOT, "include")
_BUILD = os.path.join(_ROOT, "_build")
_LIB = os.path.join(_PKG, "libmolt.so")
_SOURCES = ["rows.cu", "lmhead_fwd.cu", "lmhead_bwd.cu", "lmhead_bwd4.cu", "api.cu", "noalloc.cu"]
ARCH_FLAGS = ["-gencode", "arch=compute_103a,code=sm_103a"]

STATUS = {
    0: "MOLT_OK", 1: "MOLT_ERR_INVALID_ARG", 2: "MOLT_ERR_UNSUPPORTED_SHAPE", 3: "MOLT_ERR_UNSORTED_GROUPS",
    4: "MOLT_ERR_ZERO_DENOM", 5: "MOLT_ERR_CUDA", 6: "MOLT_ERR_DEVICE_TIMEOUT", 7: "MOLT_ERR_NO_MEMORY",
    8: "MOLT_ERR_TOKEN_RANGE", 9: "MOLT_ERR_WORKSPACE",
}
DEV_FLAGS = {"timeout": 1, "token_range": 2, "zero_denom": 4, "unsorted_groups": 8}


def lib_path() -> str:
    return _LIB


def _nvcc() -> str:
    for c in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", "nvcc"):
        if c and (os.path.sep not in c or os.path.exists(c)):
            return c
    return "nvcc"


def build(verbose: bool = False, force: bool = False) -> str:
    """Compile the CUDA sources for sm_103a (in parallel) and link libmolt.so
    into this package directory.  Returns the library path."""
    os.makedirs(_BUILD, exist_ok=True)
    srcs = [os.path.join(_CSRC, s) for s in _SOURCES]
    deps = srcs + [os.path.join(_CSRC, h) for h in os.listdir(_CSRC) if h.endswith(".cuh")] + [
        os.path.join(_INCLUDE, "molt.h")]
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= max(os.path.getmtime(d) for d in deps)):
        return _LIB
    nvcc = _nvcc()
    common = [nvcc, "-std=c++17", "-O3", "-lineinfo", *ARCH_FLAGS, "-Xcompiler", "-fPIC", "-I", _INCLUDE]

    def compile_one(src):
        obj = os.path.join(_BUILD, os.path.basename(src).replace(".cu", ".o"))
        cmd = common + ["-c", src, "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        if verbose:
            sys.stdout.write(r.stdout + r.stderr)
        return obj

    with ThreadPoolExecutor(max_workers=len(srcs)) as ex:
        objs = list(ex.map(compile_one, srcs))
    tmp = _LIB + ".tmp"
    cmd = [nvcc, "-shared", *ARCH_FLAGS, "-cudart", "shared", "-o", tmp, *objs,
           "-Xlinker", "-rpath,/usr/local/cuda/lib64"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, _LIB)
    return _LIB


class MoltError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


_lib = None


def load():
    """Load libmolt.so (build() must have run).  Raises if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB):
        raise RuntimeError(f"{_LIB} is not built; call paper_2607_21653_gb300.build() first")
    L = ctypes.CDLL(_LIB)
    P, I64, I32, F, D, SZ = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_float, ctypes.c_double,
                             ctypes.c_size_t)
    sig = {
        "molt_status_string": (ctypes.c_char_p, [I32]),
        "molt_last_error": (ctypes.c_char_p, []),
        "molt_version": (I32, []),
        "molt_kernel_launches": (ctypes.c_uint64, []),
        "molt_device_status": (I32, [P, ctypes.POINTER(ctypes.c_uint32)]),
        "molt_selftest_wait_timeout": (I32, [P]),
        "molt_group_advantages": (I32, [P, P, I64, D, P, P]),
        "molt_advantages": (I32, [P, P, I64, I32, D, P, P]),
        "molt_broadcast_advantages": (I32, [P, P, I64, I64, P, P]),
        "molt_mask_count": (I32, [P, I64, P, P]),
        "molt_token_logprobs_workspace_bytes": (SZ, [I64, I64, I64]),
        "molt_token_logprobs_fwd": (I32, [P, P, P, P, I64, I64, I64, P, P, P, SZ, P]),
        "molt_policy_loss_workspace_bytes": (SZ, [I64, I64, I64]),
        "molt_policy_loss_fwd_bwd": (I32, [P, P, P, P, P, P, I64, I64, I64, F, F, D, P, P, P, I32, P, P, P, P,
                                            P, SZ, P]),
        "molt_policy_loss_workspace_bytes_ex": (SZ, [I64, I64, I64, P]),
        "molt_policy_loss_fwd_bwd_ex": (I32, [P, P, P, P, P, P, I64, I64, I64, F, F, D, P, P, P, P, I32, P, P,
                                               P, P, P, SZ, P]),
        "molt_set_timing_events": (None, [P, P, I32]),
        "molt_token_logprobs_fwd_noalloc": (I32, [P, P, P, P, I64, I64, I64, P, P, P]),
        "molt_vp_partials_workspace_bytes": (SZ, [I64, I64, I64]),
        "molt_vp_partials": (I32, [P, P, P, P, I64, I64, I64, I64, P, P, SZ, P]),
        "molt_vp_loss_workspace_bytes": (SZ, [I64]),
        "molt_vp_loss": (I32, [P, I32, P, P, P, I64, F, F, D, P, P, P, P, P, P, P, P, SZ, P]),
        "molt_vp_backward_workspace_bytes": (SZ, [I64, I64, I64]),
        "molt_vp_backward": (I32, [P, P, P, P, P, I64, I64, I64, I64, P, P, I32, P, SZ, P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    _lib = L
    return L


TIMING_SLOTS = ("gather", "forward", "merge", "backward", "cast")


def _cudart():
    """The CUDA runtime already loaded in this process (libmolt links it)."""
    load()
    rt = ctypes.CDLL("libcudart.so.13")
    rt.cudaEventCreate.argtypes = [ctypes.POINTER(ctypes.c_void_p)]
    rt.cudaEventElapsedTime.argtypes = [ctypes.POINTER(ctypes.c_float), ctypes.c_void_p, ctypes.c_void_p]
    rt.cudaEventDestroy.argtypes = [ctypes.c_void_p]
    return rt


class KernelTimer:
    """Records CUDA events around the library's kernel groups (C-ABI timing hook)
    for a series of steps; `elapsed_ms()` sums each group's time over the steps.
    The events are raw cudaEvent_t handles created through the CUDA runtime."""

    def __init__(self, steps: int):
        self.rt = _cudart()
        n = len(TIMING_SLOTS)
        self.ev = []
        for _ in range(steps):
            row = []
            for _ in range(n):
                a, b = ctypes.c_void_p(), ctypes.c_void_p()
                if self.rt.cudaEventCreate(ctypes.byref(a)) or self.rt.cudaEventCreate(ctypes.byref(b)):
                    raise RuntimeError("cudaEventCreate failed")
                row.append((a, b))
            self.ev.append(row)
        self._arrays = []

    def arm(self, step: int):
        n = len(TIMING_SLOTS)
        starts = (ctypes.c_void_p * n)(*[e[0].value for e in self.ev[step]])
        stops = (ctypes.c_void_p * n)(*[e[1].value for e in self.ev[step]])
        self._arrays.append((starts, stops))
        load().molt_set_timing_events(starts, stops, n)

    @staticmethod
    def disarm():
        load().molt_set_timing_events(None, None, 0)

    def elapsed_ms(self) -> dict:
        """Call after the stream has been synchronised."""
        out = {k: 0.0 for k in TIMING_SLOTS}
        ms = ctypes.c_float()
        for row in self.ev:
            for k, (a, b) in zip(TIMING_SLOTS, row):
                if self.rt.cudaEventElapsedTime(ctypes.byref(ms), a, b) == 0:
                    out[k] += ms.value
        return out

    def close(self):
        for row in self.ev:
            for a, b in row:
                self.rt.cudaEventDestroy(a)
                self.rt.cudaEventDestroy(b)
        self.ev = []


def header_functions() -> list[str]:
    """Names of the functions declared in include/molt.h."""
    with open(os.path.join(_INCLUDE, "molt.h")) as f:
        txt = f.read()
    return sorted(set(re.findall(r"\b(molt_[a-z0-9_]+)\s*\(", txt)))


def _check(status: int):
    if status != 0:
        msg = load().molt_last_error().decode()
        raise MoltError(status, msg)


# ---------------------------------------------------------------- torch glue
def _torch():
    import torch
    return torch


def _ptr(t, dtype=None, name="tensor"):
    """Device pointer of a contiguous CUDA tensor (None -> NULL)."""
    if t is None:
        return None
    torch = _torch()
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t.data_ptr()


def _stream(stream=None):
    torch = _torch()
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


_ws_cache: dict = {}
_WS_CACHE_MAX = 16


def _workspace(nbytes: int, device, key: str, stream=None):
    """Workspace buffer from the torch caching allocator, reused per (device,
    call kind, stream): calls on one stream run in order and can share it, calls
    on different streams may overlap and get their own.  Each buffer is
    allocated on the stream that uses it, so that when it is replaced by a
    larger one or evicted (beyond 16 entries, oldest first) the allocator
    reuses its memory only after that stream's pending work."""
    torch = _torch()
    s = torch.cuda.current_stream(device) if stream is None else stream
    k = (str(device), key, s.cuda_stream)
    buf = _ws_cache.pop(k, None)
    if buf is None or buf.numel() < nbytes:
        buf = None
        with torch.cuda.stream(s):
            buf = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=device)
    _ws_cache[k] = buf                   # most recently used last
    while len(_ws_cache) > _WS_CACHE_MAX:
        _ws_cache.pop(next(iter(_ws_cache)))
    return buf


def device_status(stream=None) -> int:
    """Synchronise the stream and return (and clear) the device status bits."""
    flags = ctypes.c_uint32(0)
    st = load().molt_device_status(_stream(stream), ctypes.byref(flags))
    if st not in (0, 3, 4, 6, 8):
        _check(st)
    return int(flags.value)


def selftest_wait_timeout(stream=None) -> None:
    """Enqueue the wait self-test (molt_selftest_wait_timeout): a bounded device
    wait on a counter nothing raises, which gives up after about 4 s and sets
    the timeout bit; read it with device_status()."""
    _check(load().molt_selftest_wait_timeout(_stream(stream)))


def kernel_launches() -> int:
    """Process-wide number of kernels the library has enqueued so far."""
    return int(load().molt_kernel_launches())


def group_advantages(rewards, group_ids, eps: float = 1e-6, out=None, stream=None):
    torch = _torch()
    n = rewards.shape[0]
    out = torch.empty(n, dtype=torch.float32, device=rewards.device) if out is None else out
    _check(load().molt_group_advantages(_ptr(rewards, torch.float32, "rewards"), _ptr(group_ids, torch.int32, "group_ids"),
                                        n, float(eps), _ptr(out, torch.float32, "out"), _stream(stream)))
    return out


ESTIMATORS = {"grpo": 0, "group_mean": 1, "dr_grpo": 2, "rloo": 3, "reinforce_pp": 4}


def advantages(rewards, group_ids, estimator="grpo", eps: float = 1e-6, out=None, stream=None):
    """Per-rollout advantages with one of the estimators of Sec. 4.5."""
    torch = _torch()
    n = rewards.shape[0]
    out = torch.empty(n, dtype=torch.float32, device=rewards.device) if out is None else out
    gid = None if group_ids is None else _ptr(group_ids, torch.int32, "group_ids")
    _check(load().molt_advantages(_ptr(rewards, torch.float32, "rewards"), gid, n, ESTIMATORS[estimator], float(eps),
                                  _ptr(out, torch.float32, "out"), _stream(stream)))
    return out


def broadcast_advantages(adv_resp, resp_of_token, out=None, stream=None):
    torch = _torch()
    T = resp_of_token.shape[0]
    out = torch.empty(T, dtype=torch.float32, device=resp_of_token.device) if out is None else out
    _check(load().molt_broadcast_advantages(_ptr(adv_resp, torch.float32, "adv_resp"),
                                            _ptr(resp_of_token, torch.int32, "resp_of_token"), adv_resp.shape[0], T,
                                            _ptr(out, torch.float32, "out"), _stream(stream)))
    return out


def mask_count(mask, out=None, stream=None):
    torch = _torch()
    out = torch.empty(1, dtype=torch.int64, device=mask.device) if out is None else out
    _check(load().molt_mask_count(_ptr(mask, torch.uint8, "mask"), mask.shape[0], _ptr(out, torch.int64, "out"),
                                  _stream(stream)))
    return out


def token_logprobs_workspace_bytes(T, H, V) -> int:
    return int(load().molt_token_logprobs_workspace_bytes(T, H, V))


def policy_loss_workspace_bytes(T, H, V) -> int:
    return int(load().molt_policy_loss_workspace_bytes(T, H, V))


def _bf16_bits(t, name):
    torch = _torch()
    if t.dtype == torch.bfloat16:
        return _ptr(t, None, name)
    if t.dtype in (torch.uint16, torch.int16):
        return _ptr(t, None, name)
    raise TypeError(f"{name} must be bfloat16 (or its 16-bit pattern)")


def token_logprobs(hidden, weight, tokens, mask=None, want_entropy=True, stream=None, workspace=None):
    """logp[T] and entropy[T] (fp32) of the generated tokens; rows with mask 0 give 0."""
    torch = _torch()
    T, H = hidden.shape
    V = weight.shape[0]
    logp = torch.empty(T, dtype=torch.float32, device=hidden.device)
    ent = torch.empty(T, dtype=torch.float32, device=hidden.device) if want_entropy else None
    nbytes = token_logprobs_workspace_bytes(T, H, V)
    ws = workspace if workspace is not None else _workspace(nbytes, hidden.device, "logprobs", stream)
    _check(load().molt_token_logprobs_fwd(_bf16_bits(hidden, "hidden"), _bf16_bits(weight, "weight"),
                                          _ptr(tokens, torch.int32, "tokens"), _ptr(mask, torch.uint8, "mask"),
                                          T, H, V, _ptr(logp), _ptr(ent), ws.data_ptr(), ws.numel(),
                                          _stream(stream)))
    return logp, ent


def _header_define(name: str) -> int:
    with open(os.path.join(_INCLUDE, "molt.h")) as f:
        m = re.search(r"#define\s+" + name + r"\s+(\d+)", f.read())
    if m is None:
        raise RuntimeError(f"{name} is not defined in molt.h")
    return int(m.group(1))


# the largest T molt_token_logprobs_fwd_noalloc takes (MOLT_NOALLOC_MAX_TOKENS)
NOALLOC_MAX_TOKENS = _header_define("MOLT_NOALLOC_MAX_TOKENS")


def token_logprobs_noalloc(hidden, weight, tokens, mask=None, want_entropy=True, stream=None):
    """Like token_logprobs, through molt_token_logprobs_fwd_noalloc: the library
    allocates nothing (its scratch is a fixed device array); T is at most
    NOALLOC_MAX_TOKENS."""
    torch = _torch()
    T, H = hidden.shape
    V = weight.shape[0]
    logp = torch.empty(T, dtype=torch.float32, device=hidden.device)
    ent = torch.empty(T, dtype=torch.float32, device=hidden.device) if want_entropy else None
    _check(load().molt_token_logprobs_fwd_noalloc(_bf16_bits(hidden, "hidden"), _bf16_bits(weight, "weight"),
                                                  _ptr(tokens, torch.int32, "tokens"),
                                                  _ptr(mask, torch.uint8, "mask"), T, H, V, _ptr(logp), _ptr(ent),
                                                  _stream(stream)))
    return logp, ent


def policy_loss_fwd_bwd(hidden, weight, tokens, behavior_logp, adv, mask=None, clip_lo=0.2, clip_hi=0.2,
                        denom=0.0, dW=None, accumulate_dW=False, want_token_outputs=True, stream=None,
                        workspace=None):
    """Fused clipped-surrogate loss (Eq. 2 token-mean) forward + backward.

    Returns dict(loss [1] fp32, dhidden [T,H] bf16, dW [V,H] fp32, logp, entropy,
    token_loss [T] fp32 (None unless want_token_outputs), stats [9 x 8 bytes])."""
    torch = _torch()
    T, H = hidden.shape
    V = weight.shape[0]
    dev = hidden.device
    loss = torch.empty(1, dtype=torch.float32, device=dev)
    dh = torch.empty(T, H, dtype=torch.bfloat16, device=dev)
    if dW is None:
        dW = torch.empty(V, H, dtype=torch.float32, device=dev)
        accumulate_dW = False
    stats = torch.zeros(9, dtype=torch.float64, device=dev)
    logp = ent = tl = None
    if want_token_outputs:
        logp = torch.empty(T, dtype=torch.float32, device=dev)
        ent = torch.empty(T, dtype=torch.float32, device=dev)
        tl = torch.empty(T, dtype=torch.float32, device=dev)
    nbytes = policy_loss_workspace_bytes(T, H, V)
    ws = workspace if workspace is not None else _workspace(nbytes, dev, "policy_loss", stream)
    _check(load().molt_policy_loss_fwd_bwd(
        _bf16_bits(hidden, "hidden"), _bf16_bits(weight, "weight"), _ptr(tokens, torch.int32, "tokens"),
        _ptr(behavior_logp, torch.float32, "behavior_logp"), _ptr(adv, torch.float32, "adv"),
        _ptr(mask, torch.uint8, "mask"), T, H, V, float(clip_lo), float(clip_hi), float(denom), _ptr(loss),
        _ptr(dh), _ptr(dW, torch.float32, "dW"), 1 if accumulate_dW else 0, _ptr(logp), _ptr(ent), _ptr(tl),
        _ptr(stats), ws.data_ptr(), ws.numel(), _stream(stream)))
    return {"loss": loss, "dhidden": dh, "dW": dW, "logp": logp, "entropy": ent, "token_loss": tl,
            "stats": stats}


def stats_dict(stats_tensor) -> dict:
    """Decode molt_stats (5 doubles + 4 int64) or molt_stats_ex (those, then
    1 double + 2 int64) copied to the host."""
    import numpy as np
    raw = stats_tensor.detach().cpu().numpy().view(np.uint8).tobytes()
    d = np.frombuffer(raw[:40], dtype=np.float64)
    i = np.frombuffer(raw[40:72], dtype=np.int64)
    out = {"denom": float(d[0]), "loss": float(d[1]), "sum_ratio": float(d[2]), "sum_entropy": float(d[3]),
           "max_abs_log_ratio": float(d[4]), "n_active": int(i[0]), "n_clip_low": int(i[1]),
           "n_clip_high": int(i[2]), "n_grad_rows": int(i[3])}
    if len(raw) >= 96:
        out["sum_kl"] = float(np.frombuffer(raw[72:80], dtype=np.float64)[0])
        j = np.frombuffer(raw[80:96], dtype=np.int64)
        out["n_tokens_rejected"] = int(j[0])
        out["n_seq_rejected"] = int(j[1])
    return out


class LossOptions(ctypes.Structure):
    """molt_loss_options: KL-to-reference, entropy bonus, sequence gate."""
    _fields_ = [("kl_coef", ctypes.c_float), ("entropy_coef", ctypes.c_float), ("ref_logp", ctypes.c_void_p),
                ("seq_of_token", ctypes.c_void_p), ("gate_lo", ctypes.c_double), ("gate_hi", ctypes.c_double),
                ("deterministic", ctypes.c_int), ("det_clusters", ctypes.c_int)]


def policy_loss_fwd_bwd_ex(hidden, weight, tokens, behavior_logp, adv, mask=None, clip_lo=0.2, clip_hi=0.2,
                           denom=0.0, kl_coef=0.0, ref_logp=None, entropy_coef=0.0, seq_of_token=None,
                           gate_lo=0.0, gate_hi=float("inf"), deterministic=False, det_clusters=0, dW=None,
                           accumulate_dW=False, want_token_outputs=True, stream=None, workspace=None):
    """policy_loss_fwd_bwd with the extended objective
    l_t = w_t (l_pg,t + kl_coef KL_t - entropy_coef H_t) (molt_policy_loss_fwd_bwd_ex).
    det_clusters (deterministic mode): clusters of four CTAs to run, a multiple
    of 4, or 0 for all that fit; the results do not depend on it.
    Returns the same dict; stats is molt_stats_ex (12 x 8 bytes)."""
    torch = _torch()
    T, H = hidden.shape
    V = weight.shape[0]
    dev = hidden.device
    loss = torch.empty(1, dtype=torch.float32, device=dev)
    dh = torch.empty(T, H, dtype=torch.bfloat16, device=dev)
    if dW is None:
        dW = torch.empty(V, H, dtype=torch.float32, device=dev)
        accumulate_dW = False
    stats = torch.zeros(12, dtype=torch.float64, device=dev)
    logp = ent = tl = None
    if want_token_outputs:
        logp = torch.empty(T, dtype=torch.float32, device=dev)
        ent = torch.empty(T, dtype=torch.float32, device=dev)
        tl = torch.empty(T, dtype=torch.float32, device=dev)
    opts = LossOptions(float(kl_coef), float(entropy_coef), _ptr(ref_logp, torch.float32, "ref_logp"),
                       _ptr(seq_of_token, torch.int32, "seq_of_token"), float(gate_lo), float(gate_hi),
                       1 if deterministic else 0, int(det_clusters))
    nbytes = int(load().molt_policy_loss_workspace_bytes_ex(T, H, V, ctypes.byref(opts)))
    if nbytes == 0:
        raise MoltError(2, "unsupported shape for these options")
    ws = workspace if workspace is not None else _workspace(nbytes, dev, "policy_loss", stream)
    _check(load().molt_policy_loss_fwd_bwd_ex(
        _bf16_bits(hidden, "hidden"), _bf16_bits(weight, "weight"), _ptr(tokens, torch.int32, "tokens"),
        _ptr(behavior_logp, torch.float32, "behavior_logp"), _ptr(adv, torch.float32, "adv"),
        _ptr(mask, torch.uint8, "mask"), T, H, V, float(clip_lo), float(clip_hi), float(denom),
        ctypes.byref(opts), _ptr(loss), _ptr(dh), _ptr(dW, torch.float32, "dW"), 1 if accumulate_dW else 0,
        _ptr(logp), _ptr(ent), _ptr(tl), _ptr(stats), ws.data_ptr(), ws.numel(), _stream(stream)))
    return {"loss": loss, "dhidden": dh, "dW": dW, "logp": logp, "entropy": ent, "token_loss": tl,
            "stats": stats}


# ------------------------------------------------------- vocabulary parallel
def vocab_shard_bounds(V: int, n_shards: int) -> list:
    """[(v_begin, v_end)] of n_shards contiguous vocabulary ranges covering
    [0, V) in order (rank r holds the r-th)."""
    if n_shards < 1 or n_shards > V:
        raise ValueError("need 1 <= n_shards <= V")
    return [(r * V // n_shards, (r + 1) * V // n_shards) for r in range(n_shards)]


def vp_partials(hidden, weight_shard, tokens, v_begin, mask=None, stream=None, workspace=None):
    """Per-token statistics (M, S, Q, z_x) of one vocabulary shard
    (molt_vp_partials): fp32 [T, 4]."""
    torch = _torch()
    T, H = hidden.shape
    Vs = weight_shard.shape[0]
    out = torch.empty(T, 4, dtype=torch.float32, device=hidden.device)
    nbytes = int(load().molt_vp_partials_workspace_bytes(T, H, Vs))
    ws = workspace if workspace is not None else _workspace(nbytes, hidden.device, "logprobs", stream)
    _check(load().molt_vp_partials(_bf16_bits(hidden, "hidden"), _bf16_bits(weight_shard, "weight_shard"),
                                   _ptr(tokens, torch.int32, "tokens"), _ptr(mask, torch.uint8, "mask"), T, H, Vs,
                                   int(v_begin), _ptr(out), ws.data_ptr(), ws.numel(), _stream(stream)))
    return out


def vp_loss(partials, behavior_logp, adv, mask=None, clip_lo=0.2, clip_hi=0.2, denom=0.0, stream=None):
    """Merge of the shards' statistics ([n_shards, T, 4], shard order) with
    the clipped surrogate and Eq. 2 (molt_vp_loss).  Returns dict(loss, lse,
    coef, logp, entropy, token_loss, stats)."""
    torch = _torch()
    n, T, four = partials.shape
    if four != 4:
        raise ValueError("partials must be [n_shards, T, 4]")
    dev = partials.device
    out = {"loss": torch.empty(1, dtype=torch.float32, device=dev)}
    for k in ("lse", "coef", "logp", "entropy", "token_loss"):
        out[k] = torch.empty(T, dtype=torch.float32, device=dev)
    out["stats"] = torch.zeros(9, dtype=torch.float64, device=dev)
    nbytes = int(load().molt_vp_loss_workspace_bytes(T))
    ws = _workspace(nbytes, dev, "vp_loss", stream)
    _check(load().molt_vp_loss(
        _ptr(partials, torch.float32, "partials"), n, _ptr(behavior_logp, torch.float32, "behavior_logp"),
        _ptr(adv, torch.float32, "adv"), _ptr(mask, torch.uint8, "mask"), T, float(clip_lo), float(clip_hi),
        float(denom), _ptr(out["loss"]), _ptr(out["lse"]), _ptr(out["coef"]), _ptr(out["logp"]),
        _ptr(out["entropy"]), _ptr(out["token_loss"]), _ptr(out["stats"]), ws.data_ptr(), ws.numel(),
        _stream(stream)))
    return out


def vp_backward(hidden, weight_shard, tokens, lse, coef, v_begin, dW=None, accumulate_dW=False, stream=None):
    """One shard's backward (molt_vp_backward): returns (dhidden contribution
    fp32 [T, H], dW shard fp32 [V_shard, H])."""
    torch = _torch()
    T, H = hidden.shape
    Vs = weight_shard.shape[0]
    dev = hidden.device
    dh = torch.empty(T, H, dtype=torch.float32, device=dev)
    if dW is None:
        dW = torch.empty(Vs, H, dtype=torch.float32, device=dev)
        accumulate_dW = False
    nbytes = int(load().molt_vp_backward_workspace_bytes(T, H, Vs))
    ws = _workspace(nbytes, dev, "vp_backward", stream)
    _check(load().molt_vp_backward(
        _bf16_bits(hidden, "hidden"), _bf16_bits(weight_shard, "weight_shard"), _ptr(tokens, torch.int32, "tokens"),
        _ptr(lse, torch.float32, "lse"), _ptr(coef, torch.float32, "coef"), T, H, Vs, int(v_begin), _ptr(dh),
        _ptr(dW, torch.float32, "dW"), 1 if accumulate_dW else 0, ws.data_ptr(), ws.numel(), _stream(stream)))
    return dh, dW


def gather_shard_partials(local, group=None):
    """The exchange before the merge: every rank's [T, 4] statistics, stacked
    in rank order (rank r holds the r-th vocabulary range) -> [n_shards, T, 4].
    One all-gather of 16 bytes per token over torch.distributed."""
    torch = _torch()
    import torch.distributed as dist
    world = dist.get_world_size(group)
    bufs = [torch.empty_like(local) for _ in range(world)]
    dist.all_gather(bufs, local.contiguous(), group=group)
    return torch.stack(bufs)


def sum_dhidden(partial, group=None):
    """The exchange after the shards' backward: dhidden = the sum of every
    rank's contribution (all-reduce, in place)."""
    import torch.distributed as dist
    dist.all_reduce(partial, op=dist.ReduceOp.SUM, group=group)
    return partial


def policy_loss_vocab_parallel(hidden, weight_shard, v_begin, tokens, behavior_logp, adv, mask=None, clip_lo=0.2,
                               clip_hi=0.2, denom=0.0, group=None, stream=None):
    """One rank's policy-loss step with W split by vocabulary over the ranks
    of `group` (rank r holds W[v_begin_r : v_begin_r + V_r], in order):
    shard statistics -> all-gather -> merge and loss -> shard backward ->
    all-reduce of dhidden.  Returns the vp_loss dict plus dhidden (fp32, the
    sum over the ranks) and dW (this rank's shard)."""
    local = vp_partials(hidden, weight_shard, tokens, v_begin, mask, stream=stream)
    parts = gather_shard_partials(local, group)
    out = vp_loss(parts, behavior_logp, adv, mask, clip_lo, clip_hi, denom, stream=stream)
    dh, dW = vp_backward(hidden, weight_shard, tokens, out["lse"], out["coef"], v_begin, stream=stream)
    out["dhidden"] = sum_dhidden(dh, group)
    out["dW"] = dW
    return out
