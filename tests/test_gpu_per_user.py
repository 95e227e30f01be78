"""Per-user queries (stacked refinement, Sec. 3.3) on the GPU: the C ABI
entry points sa_sketch_fwd_per_user / sa_sketch_bwd_per_user against the fp64
oracle's per-user functions, element by element on seeded inputs.

Q is [B, H, P, d]; dQ[b, h] holds only user b's tokens.  The lengths include
empty users, single-token users, ragged tails and users long enough to be cut
across workers (their dQ pieces are summed like the sketch's).  Tolerance:
1e-4 max|oracle| for fp32 inputs, 2e-2 for bf16.
"""
import numpy as np
import pytest
import torch

import harness
from paper_2609_08443_gb300 import binding, workloads as wl

pytestmark = pytest.mark.gpu

RAGGED = [0, 1, 127, 128, 129, 300, 0, 1000, 17, 2049]

SHAPES = [
    # (P, d, dtype, H): tensor-core forward and backward kernels, then CUDA-core shapes
    (512, 128, wl.BF16, 2),   # cluster-pair forward, token-side + sliced dQ backward
    (256, 128, wl.BF16, 1),
    (256, 64, wl.BF16, 2),    # fused forward, one-CTA backward
    (128, 128, wl.BF16, 2),
    (512, 64, wl.BF16, 1),    # pair forward, CUDA-core backward
    (1024, 128, wl.BF16, 1),  # sliced lse pass + 4 prototype slices; 8-chunk token side, 8 dQ slices
    (64, 64, wl.F32, 1),      # CUDA cores (fp32)
    (96, 32, wl.BF16, 1),
    (1024, 64, wl.BF16, 1),
]


@pytest.mark.parametrize("P,d,dt,H", SHAPES, ids=lambda x: str(x))
def test_per_user_fwd_bwd(cuda_lib, P, d, dt, H):
    spec = wl.custom(RAGGED, H=H, P=P, d=d, dtype=dt, seed=P + d + 7)
    harness.check_spec(spec, bwd=True, per_user_q=True)


def test_per_user_without_saved_lse(cuda_lib):
    spec = wl.custom([513, 77, 0, 1300], H=2, P=512, d=128, dtype=wl.BF16, seed=11)
    harness.check_spec(spec, bwd=True, pass_lse=False, per_user_q=True)


def test_per_user_100k_subbatch(cuda_lib):
    """Two 100K-token users of the 100K workload's shapes (H=8, d=128, P=512)."""
    spec = wl.sub_spec(wl.config(4), [0, 1])
    harness.check_spec(spec, bwd=True, per_user_q=True)


def test_broadcast_prototypes_match_shared(cuda_lib):
    """Every user given the shared prototypes: the same sketch bitwise (the
    same kernels read the same values), and per-user dQ summing to the shared dQ."""
    spec = wl.custom([700, 0, 128, 129, 3000, 1], H=2, P=512, d=128, dtype=wl.BF16, seed=5)
    host = wl.make_host(spec)
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    B = t["cu_seqlens"].numel() - 1
    Qu = t["Q"].unsqueeze(0).expand(B, -1, -1, -1).contiguous()
    s_sh, l_sh = binding.sa_sketch_fwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], spec.scale, want_lse=True)
    s_pu, l_pu = binding.sa_sketch_fwd_per_user(t["K"], t["V"], t["cu_seqlens"], Qu, spec.scale, want_lse=True)
    assert torch.equal(s_sh, s_pu) and torch.equal(l_sh, l_pu)
    _, _, dq_sh = binding.sa_sketch_bwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], t["dsketch"], spec.scale, lse=l_sh)
    dk, dv, dq_pu = binding.sa_sketch_bwd_per_user(t["K"], t["V"], t["cu_seqlens"], Qu, t["dsketch"], spec.scale,
                                                   lse=l_pu)
    torch.cuda.synchronize()
    assert dq_pu.shape == (B,) + tuple(t["Q"].shape)
    assert torch.all(dq_pu[1] == 0)  # the empty user
    ref = dq_sh.double().cpu().numpy()
    assert harness.rel_err(dq_pu.double().sum(0).cpu().numpy(), ref) <= 1e-5


def test_per_user_bitwise_deterministic(cuda_lib):
    spec = wl.custom([5000, 0, 3, 12000, 129], H=2, P=512, d=128, dtype=wl.BF16, seed=3)
    host = wl.make_host(spec, per_user_q=True)
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    runs = []
    for _ in range(3):
        s, lse = binding.sa_sketch_fwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], spec.scale, want_lse=True)
        dk, dv, dq = binding.sa_sketch_bwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], t["dsketch"], spec.scale,
                                           lse=lse)
        torch.cuda.synchronize()
        runs.append([x.clone() for x in (s, dk, dv, dq)])
    for r in runs[1:]:
        for a, b in zip(runs[0], r):
            assert torch.equal(a, b)
