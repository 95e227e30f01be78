"""FLOP model of the paper (App. G) and the roofline of the sketching step.

The paper counts FLOPs of matrix products only (App. G.1: 2mrp for an m x r
by r x p product) and ignores softmax exponentials.  Its closed forms:

  SA layer   2 L d^2 + 14 L_s d^2 + 4 L_s L d      (Eq. sa_layer_total)
  SA total   N_sa * SA layer                         (Eq. sa_closed)
  STCA       N_stca (12 L D^2 + 4 L D h + 20 D^2)    (Eq. stca_closed)
  adapter    2 L_s d D                               (Eq. adapt_flops)
  hit        adapter + STCA(L_s)                     (Eq. hit_miss_closed)
  expected   hit + (1 - p_hit) SA(L)                 (Eq. expected_closed)
  MRLB       shared / R + per-target                 (Eqs. stca_mrlb_total, expected_mrlb)

The sketching step built here is the L-dependent part of one SA layer: the
affinity and aggregation products, 2 L_s L d each (App. G.3), per head.
Its backward is not in the paper; counting the same way it has four more
products of the same size (dV = A^T G, dA = G V^T, dK = dS^T Q, dQ = dS K),
8 L_s L d, plus the affinity recomputed (2 L_s L d) which is reported apart.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, Optional


# ------------------------------------------------------- paper App. G

def sa_layer_flops(L, Ls, d):
    return 2 * L * d * d + 14 * Ls * d * d + 4 * Ls * L * d


def sa_flops(L, n_sa, Ls, d):
    return n_sa * sa_layer_flops(L, Ls, d)


def stca_flops(L, n_stca, D, h):
    return n_stca * (12 * L * D * D + 4 * L * D * h + 20 * D * D)


def adapt_flops(Ls, d, D):
    return 2 * Ls * d * D


def seqo1_hit_flops(Ls, d, D, h, n_stca):
    return adapt_flops(Ls, d, D) + stca_flops(Ls, n_stca, D, h)


def seqo1_expected_flops(L, p_hit, Ls, d, D, h, n_sa, n_stca):
    return seqo1_hit_flops(Ls, d, D, h, n_stca) + (1 - p_hit) * sa_flops(L, n_sa, Ls, d)


def stca_mrlb_flops(L, R, n_stca, D, h):
    return 12 * n_stca * L * D * D / R + n_stca * (4 * L * D * h + 20 * D * D)


def seqo1_mrlb_expected_flops(L, R, p_hit, Ls, d, D, h, n_sa, n_stca):
    per_target = n_stca * (4 * Ls * D * h + 20 * D * D)
    shared = adapt_flops(Ls, d, D) + 12 * n_stca * Ls * D * D
    return per_target + (shared + (1 - p_hit) * sa_flops(L, n_sa, Ls, d)) / R


PAPER_HPARAMS = dict(Ls=1024, d=128, D=1024, h=16, n_sa=2, n_stca=4)  # App. G.4


# ----------------------------------------------- the sketching step

@dataclasses.dataclass
class Work:
    """Algorithmic work of one call over a batch (recompute excluded)."""

    tokens: int          # sum_b L_b (all heads share these tokens)
    flops: float         # tensor-core FLOPs counted as 2mrp
    bytes: float         # HBM bytes that must move at least once
    exps: float          # exponentials (one per token, head and prototype)
    recompute_flops: float = 0.0


def fwd_work(tokens, B, H, P, d, elem_bytes, lse=False) -> Work:
    th = tokens * H
    flops = 4.0 * P * d * th                       # affinity + aggregation
    byt = 2.0 * d * elem_bytes * th                # K and V read
    byt += B * H * P * d * 4.0                     # sketch written (fp32)
    byt += H * P * d * elem_bytes                  # prototypes read
    byt += (B + 1) * 4.0                           # offsets
    if lse:
        byt += th * 4.0
    return Work(tokens, flops, byt, float(P) * th)


def bwd_work(tokens, B, H, P, d, elem_bytes, lse_in=True) -> Work:
    th = tokens * H
    flops = 8.0 * P * d * th                       # dV, dA, dK, dQ products
    byt = 4.0 * d * elem_bytes * th                # K, V read; dK, dV written
    byt += B * H * P * d * 4.0                     # upstream dSketch read
    byt += H * P * d * (elem_bytes + 4.0)          # prototypes read, dQ written
    byt += (B + 1) * 4.0
    if lse_in:
        byt += th * 4.0
    return Work(tokens, flops, byt, float(P) * th, recompute_flops=2.0 * P * d * th)


def step_work(tokens, B, H, P, d, elem_bytes) -> Work:
    """Forward (saving lse) then backward reusing it: one training step."""
    f = fwd_work(tokens, B, H, P, d, elem_bytes, lse=True)
    b = bwd_work(tokens, B, H, P, d, elem_bytes, lse_in=True)
    return Work(tokens, f.flops + b.flops, f.bytes + b.bytes, f.exps,
                recompute_flops=b.recompute_flops)


# MUFU exp2 throughput of one GB300 SM, in ex2.approx results per SM clock.
# Measured on the GB300s: a grid of 8 blocks of 256 threads per SM,
# each thread running 8 independent chains x <- 2^-x, timed with CUDA events
# over 2000 back-to-back launches; rate / (SMs x maximum SM clock).
EX2_PER_SM_CLK = 31.8  # 1.002e13 ex2/s on 152 SMs at 2070 MHz (the clock sampled during the probe)


def exp_peak_per_s(num_sms: int, sm_mhz: float) -> float:
    """MUFU exp2 peak of the whole GPU at the given SM clock."""
    return EX2_PER_SM_CLK * num_sms * sm_mhz * 1e6


def roofline_time(work: Work, peak_tflops: float, peak_gbs: float,
                  exp_per_s: Optional[float] = None) -> Dict[str, float]:
    """Slowest of the tensor, HBM and exp bounds, in seconds."""
    t = {"tensor": work.flops / (peak_tflops * 1e12), "hbm": work.bytes / (peak_gbs * 1e9)}
    if exp_per_s:
        t["mufu"] = work.exps / exp_per_s
    bound = max(t, key=t.get)
    t["bound"] = bound
    t["time"] = t[bound]
    return t
