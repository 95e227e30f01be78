"""CUDA path vs the fp64 oracle, element by element, on seeded inputs.

Sizes span several 128-token tiles with ragged tails, empty users and users
long enough to be cut across workers.  Tolerance: max|gpu - oracle| <=
1e-4 max|oracle| for fp32 inputs, 2e-2 max|oracle| for bf16 inputs.
"""
import numpy as np
import pytest
import torch

import harness
from paper_2609_08443_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

RAGGED = [0, 1, 127, 128, 129, 300, 0, 1000, 17, 2049]

SHAPES = [
    # (P, d, dtype, H)
    (64, 64, wl.F32, 1),
    (256, 64, wl.BF16, 2),
    (512, 128, wl.BF16, 2),
    (256, 128, wl.BF16, 1),
    (512, 64, wl.BF16, 1),
    (128, 64, wl.BF16, 3),
    (128, 128, wl.BF16, 2),
    (96, 32, wl.BF16, 1),
    (200, 128, wl.F32, 1),
    (1024, 64, wl.BF16, 1),
    (1024, 128, wl.BF16, 1),
    (2048, 128, wl.BF16, 1),
    (2048, 64, wl.BF16, 1),
    (1, 8, wl.BF16, 1),
]


@pytest.mark.parametrize("P,d,dt,H", SHAPES, ids=lambda x: str(x))
def test_ragged_fwd_bwd(cuda_lib, P, d, dt, H):
    spec = wl.custom(RAGGED, H=H, P=P, d=d, dtype=dt, seed=P + d)
    harness.check_spec(spec, bwd=True)


# runs of empty users longer than the kernels' forward scan from one segment to
# the next (eight users), so the walk falls back to its binary search, between
# short and long users
EMPTY_RUNS = [300] + [0] * 20 + [129] + [0] * 9 + [1000, 1] + [0] * 12 + [2049, 0, 0, 5] + [0] * 30 + [128]


@pytest.mark.parametrize("P,d,dt,H", [(256, 64, wl.BF16, 2), (512, 128, wl.BF16, 2), (128, 128, wl.BF16, 1),
                                      (1024, 128, wl.BF16, 1), (64, 64, wl.F32, 1)], ids=lambda x: str(x))
def test_long_runs_of_empty_users(cuda_lib, P, d, dt, H):
    spec = wl.custom(EMPTY_RUNS, H=H, P=P, d=d, dtype=dt, seed=3 * P + d)
    harness.check_spec(spec, bwd=True)


@pytest.mark.parametrize("pass_lse", [True, False])
def test_bwd_with_and_without_saved_lse(cuda_lib, pass_lse):
    spec = wl.custom([513, 77, 0, 1300], H=2, P=256, d=64, dtype=wl.BF16, seed=5)
    harness.check_spec(spec, bwd=True, pass_lse=pass_lse)


def test_config1_full(cuda_lib):
    """Single user, L=4096, H=1, d=64, P=64, fp32, forward (full size)."""
    harness.check_spec(wl.config(1), bwd=False)


def test_config2_full(cuda_lib):
    """32 users U[1024,16384], H=4, d=64, P=256, bf16, forward (full size)."""
    harness.check_spec(wl.config(2), bwd=False)


def test_config3_subbatch(cuda_lib):
    """Training-step shape of config 3 on 6 of its users (full lengths)."""
    spec = wl.config(3)
    lens = wl.lengths(spec)
    users = [int(np.argmax(lens)), int(np.argmin(lens)), 0, 1, 2, 3]
    harness.check_spec(wl.sub_spec(spec, users), bwd=True)


def test_config4_subbatch(cuda_lib):
    """100K-token users, H=8, d=128, P=512, Q ~ N(0, 0.02): 2 users."""
    spec = wl.sub_spec(wl.config(4), [0, 1])
    harness.check_spec(spec, bwd=True)


def test_config5_subbatch(cuda_lib):
    """One 1M-token user mixed with 40 short users of config 5."""
    spec = wl.config(5)
    lens = wl.lengths(spec)
    long_u = int(np.nonzero(lens == 1048576)[0][0])
    short_u = [int(u) for u in np.nonzero(lens < 1048576)[0][:40]]
    harness.check_spec(wl.sub_spec(spec, [short_u[0], long_u] + short_u[1:]), bwd=True)


def test_large_p_100k_user(cuda_lib):
    """The paper's final sketch length k = 1K (ablation table: k in {512, 1K, 2K}):
    one 100K-token user, H=8, d=128, P=1024, Q ~ N(0, 0.02), bf16."""
    spec = wl.custom([100000], H=8, P=1024, d=128, dtype=wl.BF16, seed=41, q_std=0.02)
    harness.check_spec(spec, bwd=True)


@pytest.mark.parametrize("P,d", [(512, 128), (256, 64)])
def test_negative_scale(cuda_lib, P, d):
    """A negative scale (valid; the softmax then favours anti-aligned keys) runs on
    the tensor-core kernels, its sign folded into a negated copy of Q: same
    parity bar."""
    spec = wl.custom(RAGGED, H=2, P=P, d=d, dtype=wl.BF16, seed=P + d + 5)
    host = wl.make_host(spec)
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    from paper_2609_08443_gb300 import binding
    from oracle import sa_backward, sa_forward

    scale = -2.0 / np.sqrt(d)
    sk, lse = binding.sa_sketch_fwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], scale, want_lse=True)
    dK, dV, dQ = binding.sa_sketch_bwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], t["dsketch"], scale, lse=lse)
    dK2, dV2, dQ2 = binding.sa_sketch_bwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], t["dsketch"], scale)
    torch.cuda.synchronize()
    K, V, Q = (wl.host_as_f64(spec, host[k]) for k in ("K", "V", "Q"))
    O, l_ref = sa_forward(K, V, host["cu_seqlens"], Q, scale, with_lse=True)
    gK, gV, gQ = sa_backward(K, V, host["cu_seqlens"], Q, scale, host["dsketch"].astype(np.float64))
    tol = harness.TOL[wl.BF16]
    for name, got, ref in (("sketch", sk, O), ("dK", dK, gK), ("dV", dV, gV), ("dQ", dQ, gQ), ("dK (lse recomputed)", dK2, gK),
                           ("dQ (lse recomputed)", dQ2, gQ)):
        harness.assert_close(name, wl.torch_as_f64(got), ref, tol)
    assert np.max(np.abs(wl.torch_as_f64(lse) - l_ref)) <= 5e-3 * max(1.0, np.max(np.abs(l_ref)))


def test_max_heads(cuda_lib):
    """H = 64, the largest head count, on the tensor-core path."""
    spec = wl.custom([300, 0, 129, 17, 1000], H=64, P=128, d=64, dtype=wl.BF16, seed=64)
    harness.check_spec(spec, bwd=True)
