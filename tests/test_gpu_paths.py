"""The tensor-core kernels against the CUDA-core kernels on the same inputs
(two independent GPU implementations of Sec. 3.1), plus which kernel runs."""
import pytest
import torch

import harness
from paper_2609_08443_gb300 import binding, workloads as wl

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("P,d", [(128, 64), (256, 64), (128, 128), (256, 128), (512, 128), (512, 64),
                                 (1024, 128), (1024, 64), (2048, 128)])
def test_tensor_core_path_matches_cuda_core_path(cuda_lib, P, d):
    spec = wl.custom([700, 0, 128, 129, 3000, 1], H=2, P=P, d=d, dtype=wl.BF16, seed=P * 7 + d)
    host = wl.make_host(spec)
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    assert binding.sa_main_kernel_name(P, d, binding.SA_BF16, False).startswith("tc_")
    assert binding.sa_main_kernel_name(P, d, binding.SA_BF16, True).startswith("tc_")
    tc = harness.gpu_outputs(spec, t, bwd=True)
    binding.sa_select_path(1)
    try:
        assert binding.sa_main_kernel_name(P, d, binding.SA_BF16, False).startswith("simt")
        simt = harness.gpu_outputs(spec, t, bwd=True)
    finally:
        binding.sa_select_path(0)
    for k in ("sketch", "dK", "dV", "dQ"):
        assert harness.rel_err(tc[k], simt[k]) <= 2e-2, k
    assert abs(tc["lse"] - simt["lse"]).max() <= 5e-3 * max(1.0, abs(simt["lse"]).max())


def test_fp32_uses_cuda_cores(cuda_lib):
    assert binding.sa_main_kernel_name(64, 64, binding.SA_F32, False).startswith("simt")


@pytest.mark.parametrize("P,d", [(512, 128), (512, 64), (256, 128)])
def test_pair_forward_matches_lse_pass_and_slices(cuda_lib, P, d):
    """The cluster-pair forward (one kernel, per-token statistics exchanged
    between two CTAs) against the lse pass + prototype slices (two kernels)."""
    spec = wl.custom([700, 0, 128, 129, 3000, 1], H=2, P=P, d=d, dtype=wl.BF16, seed=P + 3 * d)
    host = wl.make_host(spec)
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    fused = harness.gpu_outputs(spec, t, bwd=False)
    binding.sa_select_path(2)
    try:
        assert "sliced" in binding.sa_main_kernel_name(P, d, binding.SA_BF16, False)
        sliced = harness.gpu_outputs(spec, t, bwd=False)
    finally:
        binding.sa_select_path(0)
    assert "sliced" not in binding.sa_main_kernel_name(P, d, binding.SA_BF16, False)
    assert harness.rel_err(fused["sketch"], sliced["sketch"]) <= 2e-2
    assert abs(fused["lse"] - sliced["lse"]).max() <= 5e-3 * max(1.0, abs(sliced["lse"]).max())


@pytest.mark.parametrize("P,d", [(512, 128), (512, 64)])
def test_wide_pair_forward_matches_narrow(cuda_lib, P, d):
    """The P = 512 cluster-pair forward with sixteen softmax warps per CTA
    (eight partial (max, sum) per token) against the pair kernel with eight
    softmax warps (four partials), on ragged users that end tiles, segments
    and worker ranges at every offset, with the backward that follows it, and
    against the oracle; the sixteen-warp kernel is also bitwise reproducible."""
    spec = wl.custom([700, 0, 128, 129, 3000, 1, 5000, 2, 255, 257], H=3, P=P, d=d, dtype=wl.BF16, seed=P + d + 1)
    host = wl.make_host(spec)
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    assert "wide" in binding.sa_main_kernel_name(P, d, binding.SA_BF16, False)
    wide = harness.gpu_outputs(spec, t, bwd=True)
    wide2 = harness.gpu_outputs(spec, t, bwd=True)
    binding.sa_select_path(3)
    try:
        assert "pair" in binding.sa_main_kernel_name(P, d, binding.SA_BF16, False)
        narrow = harness.gpu_outputs(spec, t, bwd=True)
    finally:
        binding.sa_select_path(0)
    for k in ("sketch", "lse", "dK", "dV", "dQ"):
        assert (wide[k] == wide2[k]).all(), k
    for k in ("sketch", "dK", "dV", "dQ"):
        assert harness.rel_err(wide[k], narrow[k]) <= 2e-2, k
    assert abs(wide["lse"] - narrow["lse"]).max() <= 5e-3 * max(1.0, abs(narrow["lse"]).max())
    ref = harness.oracle_outputs(spec, host, bwd=True)
    for k in ("sketch", "dK", "dV", "dQ"):
        harness.assert_close(k, wide[k], ref[k], harness.TOL[wl.BF16])
