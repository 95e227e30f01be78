"""Determinism, edge cases and device-detected errors of the CUDA path."""
import numpy as np
import pytest
import torch

import harness
from paper_2609_08443_gb300 import binding, workloads as wl

pytestmark = pytest.mark.gpu


def _inputs(spec):
    host = wl.make_host(spec)
    return host, wl.host_to_torch(spec, host, torch.device("cuda"))


@pytest.mark.parametrize("P,d", [(256, 64), (512, 128), (64, 64)])
def test_bitwise_deterministic(cuda_lib, P, d):
    spec = wl.custom([5000, 0, 3, 12000, 129], H=2, P=P, d=d, dtype=wl.BF16, seed=3)
    _, t = _inputs(spec)
    runs = []
    for _ in range(3):
        s, lse = binding.sa_sketch_fwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], spec.scale, want_lse=True)
        g = binding.sa_sketch_bwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], t["dsketch"], spec.scale, lse=lse)
        runs.append([s.clone(), lse.clone()] + [x.clone() for x in g])
    for r in runs[1:]:
        for a, b in zip(runs[0], r):
            assert torch.equal(a, b)


def test_all_users_empty(cuda_lib):
    spec = wl.custom([0, 0, 0], H=2, P=64, d=64, dtype=wl.BF16, seed=1)
    host, t = _inputs(spec)
    K = torch.empty((0, 2, 64), dtype=torch.bfloat16, device="cuda")
    s = binding.sa_sketch_fwd(K, K, t["cu_seqlens"], t["Q"], spec.scale)
    dK, dV, dQ = binding.sa_sketch_bwd(K, K, t["cu_seqlens"], t["Q"], t["dsketch"], spec.scale)
    torch.cuda.synchronize()
    assert torch.count_nonzero(s) == 0 and torch.count_nonzero(dQ) == 0


def test_outputs_overwrite_not_accumulate(cuda_lib):
    spec = wl.custom([300, 0, 50], H=1, P=64, d=64, dtype=wl.BF16, seed=2)
    host, t = _inputs(spec)
    out = torch.full((3, 1, 64, 64), 7.0, device="cuda")
    binding.sa_sketch_fwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], spec.scale, out=out)
    ref = harness.oracle_outputs(spec, host, bwd=False)["sketch"]
    harness.assert_close("sketch", wl.torch_as_f64(out), ref, 2e-2)


def test_large_scores_stay_finite(cuda_lib):
    spec = wl.custom([400, 31], H=1, P=128, d=64, dtype=wl.BF16, seed=4)
    host, t = _inputs(spec)
    s = binding.sa_sketch_fwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], 8.0)  # scores of O(60)
    torch.cuda.synchronize()
    assert torch.isfinite(s).all()
    K64, V64, Q64 = (wl.host_as_f64(spec, host[k]) for k in ("K", "V", "Q"))
    from oracle import sa_forward
    harness.assert_close("sketch", wl.torch_as_f64(s), sa_forward(K64, V64, host["cu_seqlens"], Q64, 8.0), 2e-2)


def test_conservation_on_gpu(cuda_lib):
    """V = 1: every sketch column sums to the user's length (Sec. 3.1)."""
    spec = wl.custom([1000, 1, 0, 4097], H=2, P=256, d=64, dtype=wl.BF16, seed=6)
    host, t = _inputs(spec)
    ones = torch.ones_like(t["V"])
    s = binding.sa_sketch_fwd(t["K"], ones, t["cu_seqlens"], t["Q"], spec.scale)
    col = s.sum(dim=2).double().cpu().numpy()  # [B, H, d]
    for b, L in enumerate([1000, 1, 0, 4097]):
        assert np.allclose(col[b], L, rtol=1e-2, atol=1e-3)


def test_bad_seqlens_reported_and_gpu_still_usable(cuda_lib):
    spec = wl.custom([100, 100], H=1, P=64, d=64, dtype=wl.BF16, seed=7)
    host, t = _inputs(spec)
    bad = torch.tensor([0, 150, 120], dtype=torch.int32, device="cuda")  # decreasing
    need = binding.sa_workspace_size(2, 200, 1, 64, 64, binding.SA_BF16, 0)
    ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    binding.sa_sketch_fwd(t["K"], t["V"], bad, t["Q"], spec.scale, ws=ws)
    assert binding.sa_get_device_error(ws) == 6
    wrong_total = torch.tensor([0, 100, 150], dtype=torch.int32, device="cuda")  # cu[B] != N
    binding.sa_sketch_fwd(t["K"], t["V"], wrong_total, t["Q"], spec.scale, ws=ws)
    assert binding.sa_get_device_error(ws) == 6
    s = binding.sa_sketch_fwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], spec.scale, ws=ws)
    assert binding.sa_get_device_error(ws) == 0
    ref = harness.oracle_outputs(spec, host, bwd=False)["sketch"]
    harness.assert_close("sketch", wl.torch_as_f64(s), ref, 2e-2)


def test_autograd_function(cuda_lib):
    spec = wl.custom([200, 0, 333], H=2, P=128, d=64, dtype=wl.BF16, seed=8)
    host, t = _inputs(spec)
    K = t["K"].clone().requires_grad_(True)
    V = t["V"].clone().requires_grad_(True)
    Q = t["Q"].clone().requires_grad_(True)
    s = binding.sa_sketch(K, V, t["cu_seqlens"], Q)
    s.backward(t["dsketch"])
    ref = harness.oracle_outputs(spec, host, bwd=True)
    harness.assert_close("sketch", wl.torch_as_f64(s), ref["sketch"], 2e-2)
    harness.assert_close("dK", wl.torch_as_f64(K.grad), ref["dK"], 2e-2)
    harness.assert_close("dV", wl.torch_as_f64(V.grad), ref["dV"], 2e-2)
    harness.assert_close("dQ", wl.torch_as_f64(Q.grad), ref["dQ"], 2e-2)


def test_launches_counted(cuda_lib):
    spec = wl.custom([300], H=1, P=64, d=64, dtype=wl.BF16, seed=9)
    _, t = _inputs(spec)
    n0 = binding.sa_launch_count()
    binding.sa_sketch_fwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], spec.scale)
    assert binding.sa_launch_count() > n0
