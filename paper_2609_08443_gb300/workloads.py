"""Seeded synthetic inputs for the Sketch Attention sketching step.

This module only draws random numbers and lays them out; it holds none of the
method's arithmetic, so both the fp64 oracle (under ``oracle/``) and the CUDA
path consume the identical bytes it produces.

Layouts (all contiguous, row-major):
  K, V      [N, H, d]   packed history keys / values of all users (N = sum L_b)
  Q         [H, P, d]   prototypes, shared by every user (Sec. 3.1)
  cu_seqlens[B + 1]     int32 offsets of each user's rows in K and V
  dsketch   [B, H, P, d] float32 upstream gradient of the sketch

Shapes follow the paper's workloads: histories of up to 100K tokens per user
(Sec. 2.1), a few hundred to a few thousand prototypes (Sec. 3.1; Table of SA
ablations uses k in {512, 1K, 2K}) and width d in {64, 128} (App. G.3).

Two generators exist:
  * ``make_host``: numpy PCG64, one independent stream per (user, tensor), so a
    single user's rows can be regenerated on the CPU without the others;
  * ``make_device``: torch's CUDA generator, for workloads too large to draw on
    the host in seconds (the 100K-token batch is 2.6e10 values).  The oracle
    side of a comparison then copies the sampled users' rows back.
bf16 values are produced by rounding fp32 draws to nearest-even in both paths.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, Optional, Sequence

import numpy as np

F32 = "f32"
BF16 = "bf16"


@dataclasses.dataclass(frozen=True)
class Spec:
    """One synthetic workload: ragged lengths plus the tensor shapes."""

    name: str
    H: int
    P: int
    d: int
    dtype: str  # F32 or BF16
    seed: int
    bwd: bool
    q_std: float = 1.0
    # length recipe
    kind: str = "fixed"  # fixed | uniform | lognormal | extremes | explicit
    B: int = 1
    L: int = 0
    lo: int = 0
    hi: int = 0
    median: float = 0.0
    sigma: float = 1.0
    n_long: int = 0
    L_long: int = 0
    n_short: int = 0
    explicit: Optional[tuple] = None

    @property
    def scale(self) -> float:
        # 1/sqrt(d) applied inside the kernel (Sec. 3.1, affinity S)
        return 1.0 / math.sqrt(self.d)


def config(i: int) -> Spec:
    """The five evaluation workloads, numbered 1..5."""
    if i == 1:
        return Spec("single user L=4096 H=1 d=64 P=64 fp32 fwd", H=1, P=64, d=64,
                    dtype=F32, seed=0, bwd=False, kind="fixed", B=1, L=4096)
    if i == 2:
        return Spec("32 users U[1024,16384] H=4 d=64 P=256 bf16 fwd", H=4, P=256, d=64,
                    dtype=BF16, seed=2, bwd=False, kind="uniform", B=32, lo=1024, hi=16384)
    if i == 3:
        return Spec("64 users lognormal(median 20K) clip[512,100000] H=8 d=64 P=256 bf16 fwd+bwd",
                    H=8, P=256, d=64, dtype=BF16, seed=3, bwd=True, kind="lognormal", B=64,
                    median=20000.0, sigma=1.0, lo=512, hi=100000)
    if i == 4:
        return Spec("128 users x L=100000 H=8 d=128 P=512 bf16 fwd+bwd", H=8, P=512, d=128,
                    dtype=BF16, seed=4, bwd=True, q_std=0.02, kind="fixed", B=128, L=100000)
    if i == 5:
        return Spec("4 users L=1048576 + 4096 users U[1,512] H=8 d=64 P=256 bf16 fwd+bwd",
                    H=8, P=256, d=64, dtype=BF16, seed=5, bwd=True, kind="extremes",
                    n_long=4, L_long=1048576, n_short=4096, lo=1, hi=512)
    raise ValueError(f"no workload {i}")


def custom(lengths: Sequence[int], H: int, P: int, d: int, dtype: str = BF16, seed: int = 0,
           q_std: float = 1.0, bwd: bool = True, name: str = "custom") -> Spec:
    return Spec(name, H=H, P=P, d=d, dtype=dtype, seed=seed, bwd=bwd, q_std=q_std,
                kind="explicit", B=len(lengths), explicit=tuple(int(x) for x in lengths))


def lengths(spec: Spec) -> np.ndarray:
    """Per-user history lengths L_b (int64), drawn from the spec's seed."""
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([spec.seed, 7])))
    if spec.kind == "fixed":
        out = np.full(spec.B, spec.L, dtype=np.int64)
    elif spec.kind == "uniform":  # integers, both ends inclusive
        out = rng.integers(spec.lo, spec.hi + 1, size=spec.B, dtype=np.int64)
    elif spec.kind == "lognormal":
        x = rng.lognormal(mean=math.log(spec.median), sigma=spec.sigma, size=spec.B)
        out = np.clip(np.rint(x), spec.lo, spec.hi).astype(np.int64)
    elif spec.kind == "extremes":
        short = rng.integers(spec.lo, spec.hi + 1, size=spec.n_short, dtype=np.int64)
        allv = np.concatenate([np.full(spec.n_long, spec.L_long, dtype=np.int64), short])
        out = allv[rng.permutation(allv.size)]
    elif spec.kind == "explicit":
        out = np.asarray(spec.explicit, dtype=np.int64)
    else:
        raise ValueError(spec.kind)
    return out


def cu_seqlens(lens: np.ndarray) -> np.ndarray:
    cu = np.zeros(lens.size + 1, dtype=np.int64)
    np.cumsum(lens, out=cu[1:])
    if cu[-1] >= 2**31:
        raise ValueError("total tokens must stay below 2^31")
    return cu.astype(np.int32)


def sub_spec(spec: Spec, users: Sequence[int]) -> Spec:
    """A spec whose lengths are the given users' lengths (same shapes, same seed)."""
    lens = lengths(spec)
    return dataclasses.replace(spec, kind="explicit", B=len(users),
                               explicit=tuple(int(lens[u]) for u in users))


# ---------------------------------------------------------------- bf16 bits

def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (nearest, ties to even); returns the uint16 bit patterns."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounding = np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1))
    return ((b + rounding) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float64."""
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


# --------------------------------------------------------------- host path

def _stream(spec: Spec, *key: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([spec.seed, *key])))


def _user_rows(spec: Spec, user_id: int, L: int, which: int) -> np.ndarray:
    return _stream(spec, 11, which, user_id).standard_normal((L, spec.H, spec.d), dtype=np.float32)


def make_host(spec: Spec, users: Optional[Sequence[int]] = None,
              per_user_q: bool = False) -> Dict[str, np.ndarray]:
    """Draw the workload on the host.

    Returns fp32 arrays for F32 specs and uint16 bf16 bit patterns for BF16
    specs ("K", "V", "Q"), plus "cu_seqlens" (int32), "dsketch" (fp32),
    "lengths" and "users" (the original user indices kept).
    ``users`` restricts the batch to a subset of the spec's users; each user's
    rows are identical to the ones it has in the full batch.
    ``per_user_q`` replaces Q by per-user prototypes [B, H, P, d] (the queries of
    the stacked refinement steps), drawn from one stream per user with the same
    standard deviation.
    """
    lens_all = lengths(spec)
    users = list(range(spec.B)) if users is None else [int(u) for u in users]
    lens = lens_all[users]
    parts_k = [_user_rows(spec, u, int(lens_all[u]), 0) for u in users]
    parts_v = [_user_rows(spec, u, int(lens_all[u]), 1) for u in users]
    empty = np.zeros((0, spec.H, spec.d), dtype=np.float32)
    K = np.concatenate(parts_k) if parts_k else empty
    V = np.concatenate(parts_v) if parts_v else empty
    if per_user_q:
        Q = np.stack([_stream(spec, 19, u).standard_normal((spec.H, spec.P, spec.d), dtype=np.float32)
                      for u in users]) if users else np.zeros((0, spec.H, spec.P, spec.d), np.float32)
    else:
        Q = _stream(spec, 13).standard_normal((spec.H, spec.P, spec.d), dtype=np.float32)
    Q = np.ascontiguousarray((Q * np.float32(spec.q_std)).astype(np.float32))
    dS = np.stack([_stream(spec, 17, u).standard_normal((spec.H, spec.P, spec.d), dtype=np.float32)
                   for u in users]) if users else np.zeros((0, spec.H, spec.P, spec.d), np.float32)
    out = {"cu_seqlens": cu_seqlens(lens), "lengths": lens, "users": np.asarray(users),
           "dsketch": np.ascontiguousarray(dS)}
    if spec.dtype == BF16:
        out.update(K=f32_to_bf16_bits(K), V=f32_to_bf16_bits(V), Q=f32_to_bf16_bits(Q))
    else:
        out.update(K=np.ascontiguousarray(K), V=np.ascontiguousarray(V), Q=Q)
    return out


def host_as_f64(spec: Spec, arr: np.ndarray) -> np.ndarray:
    """The exact float64 values of a host-drawn K/V/Q array."""
    if spec.dtype == BF16:
        return bf16_bits_to_f64(arr)
    return np.asarray(arr, dtype=np.float64)


def host_to_torch(spec: Spec, host: Dict[str, np.ndarray], device="cuda"):
    """Move a host-drawn workload into torch tensors (bf16 bits reinterpreted)."""
    import torch

    def kv(a):
        if spec.dtype == BF16:
            return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).to(device)
        return torch.from_numpy(a).to(device)

    return {
        "K": kv(host["K"]), "V": kv(host["V"]), "Q": kv(host["Q"]),
        "cu_seqlens": torch.from_numpy(host["cu_seqlens"]).to(device),
        "dsketch": torch.from_numpy(host["dsketch"]).to(device),
    }


# ------------------------------------------------------------- device path

def make_device(spec: Spec, device="cuda"):
    """Draw the workload directly in device memory with torch's CUDA RNG.

    Used for the full-size workloads; values are N(0,1) fp32 draws rounded
    to bf16 (nearest-even) like the host path, but from a different stream.
    """
    import torch

    lens = lengths(spec)
    cu = cu_seqlens(lens)
    N = int(cu[-1])
    g = torch.Generator(device=device)
    g.manual_seed(1_000_003 * spec.seed + 17)
    tdt = torch.bfloat16 if spec.dtype == BF16 else torch.float32

    def normal(shape, std=1.0):
        out = torch.empty(shape, dtype=tdt, device=device)
        flat = out.view(-1)
        chunk = 1 << 28
        for s in range(0, flat.numel(), chunk):
            n = min(chunk, flat.numel() - s)
            x = torch.randn(n, generator=g, device=device, dtype=torch.float32)
            if std != 1.0:
                x.mul_(std)
            flat[s:s + n].copy_(x)
        return out

    K = normal((N, spec.H, spec.d))
    V = normal((N, spec.H, spec.d))
    Q = normal((spec.H, spec.P, spec.d), spec.q_std)
    dS = torch.randn((lens.size, spec.H, spec.P, spec.d), generator=g, device=device,
                     dtype=torch.float32)
    return {"K": K, "V": V, "Q": Q, "cu_seqlens": torch.from_numpy(cu).to(device),
            "dsketch": dS, "lengths": lens}


def torch_as_f64(t) -> np.ndarray:
    """Exact float64 copy of a (bf16 or fp32) torch tensor on any device."""
    import torch

    return t.detach().to("cpu", torch.float64).numpy()
