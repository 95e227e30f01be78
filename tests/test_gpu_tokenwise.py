"""Token-wise ("vanilla") normalisation (Sec. 5.1, App. C) on the GPU:
sa_sketch_fwd_tokenwise / sa_sketch_bwd_tokenwise through the C ABI against the
fp64 oracle's sa_forward_tokenwise / sa_backward_tokenwise, element by element
on seeded inputs.

Tolerances.  The CUDA-core kernels compute in fp32 from inputs that both
sides read exactly, so their fp32 outputs (sketch, dQ) are held to 1e-4
max|oracle| (5e-4 for a 100K-token user, where the fp32 sums run over 1e5
terms); dK and dV are stored in the input dtype, so bf16 ones carry bf16
rounding and take the bf16 bound 2e-2.  The tensor-core forward (bf16 inputs,
d in {64, 128}, P a multiple of 128) rounds the weights to bf16 before the
aggregation, so its sketch -- and the backward, which reads that sketch through
D_j = G_j . O_j -- take the bf16 bound 2e-2 throughout.  lse_tok is compared
absolutely, like the per-token lse.
"""
import numpy as np
import pytest
import torch

import harness
from oracle import sa_backward_tokenwise, sa_forward_tokenwise
from paper_2609_08443_gb300 import binding, workloads as wl

pytestmark = pytest.mark.gpu

RAGGED = [0, 1, 31, 32, 33, 300, 0, 1000, 17, 2049]


def _run(spec, users=None, pass_fwd=True):
    host = wl.make_host(spec, users=users)
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    O, lse = binding.sa_sketch_fwd_tokenwise(t["K"], t["V"], t["cu_seqlens"], t["Q"], spec.scale, want_lse=True)
    dK, dV, dQ = binding.sa_sketch_bwd_tokenwise(t["K"], t["V"], t["cu_seqlens"], t["Q"], t["dsketch"], spec.scale,
                                                 sketch=O if pass_fwd else None, lse=lse if pass_fwd else None)
    torch.cuda.synchronize()
    got = {k: wl.torch_as_f64(v) for k, v in dict(sketch=O, lse=lse, dK=dK, dV=dV, dQ=dQ).items()}
    return host, got


def _oracle(spec, host):
    K = wl.host_as_f64(spec, host["K"])
    V = wl.host_as_f64(spec, host["V"])
    Q = wl.host_as_f64(spec, host["Q"])
    cu = host["cu_seqlens"]
    O, lse = sa_forward_tokenwise(K, V, cu, Q, spec.scale, with_lse=True)
    dK, dV, dQ = sa_backward_tokenwise(K, V, cu, Q, spec.scale, host["dsketch"].astype(np.float64))
    return dict(sketch=O, lse=lse, dK=dK, dV=dV, dQ=dQ)


def _tensor_core_fwd(spec):
    return (spec.dtype == wl.BF16 and spec.d in (64, 128) and spec.P % 128 == 0 and
            binding.sa_main_kernel_name(256, 128, binding.SA_BF16, False).startswith("tc_"))


def _compare(spec, got, ref, tol32=1e-4):
    tol_io = tol32 if spec.dtype == wl.F32 else harness.TOL[spec.dtype]
    if _tensor_core_fwd(spec):
        tol32 = tol_io
    harness.assert_close("sketch", got["sketch"], ref["sketch"], tol32)
    harness.assert_close("dQ", got["dQ"], ref["dQ"], tol32)
    harness.assert_close("dK", got["dK"], ref["dK"], tol_io)
    harness.assert_close("dV", got["dV"], ref["dV"], tol_io)
    fin = np.isfinite(ref["lse"])
    assert np.array_equal(fin, np.isfinite(got["lse"])), "lse_tok: -inf exactly for the empty users"
    if fin.any():
        assert np.max(np.abs(got["lse"][fin] - ref["lse"][fin])) <= 5e-5 * max(1.0, np.max(np.abs(ref["lse"][fin])))


@pytest.mark.parametrize("P,d,dt,H", [(64, 64, wl.F32, 2), (100, 64, wl.F32, 1), (512, 128, wl.BF16, 2),
                                      (256, 64, wl.BF16, 3), (1, 8, wl.BF16, 1), (2048, 128, wl.BF16, 1),
                                      (130, 128, wl.F32, 1)], ids=lambda x: str(x))
def test_tokenwise_matches_oracle(cuda_lib, P, d, dt, H):
    spec = wl.custom(RAGGED, H=H, P=P, d=d, dtype=dt, seed=3 * P + d)
    host, got = _run(spec)
    _compare(spec, got, _oracle(spec, host))


def test_tokenwise_backward_recomputes_forward(cuda_lib):
    """Passing no forward outputs recomputes them with the same kernels: equal bits."""
    spec = wl.custom(RAGGED, H=2, P=512, d=128, dtype=wl.BF16, seed=8)
    _, a = _run(spec, pass_fwd=True)
    _, b = _run(spec, pass_fwd=False)
    for k in ("dK", "dV", "dQ"):
        assert np.array_equal(a[k], b[k]), k


def test_tokenwise_deterministic(cuda_lib):
    spec = wl.custom(RAGGED * 3, H=2, P=256, d=128, dtype=wl.BF16, seed=9)
    _, a = _run(spec)
    _, b = _run(spec)
    for k in a:
        assert np.array_equal(a[k], b[k]), k


def test_tokenwise_single_empty_and_one_token_users(cuda_lib):
    spec = wl.custom([0, 0, 1, 0], H=2, P=64, d=64, dtype=wl.F32, seed=10)
    host, got = _run(spec)
    ref = _oracle(spec, host)
    _compare(spec, got, ref)
    # one token: every prototype's sketch row is that token's value row
    v = wl.host_as_f64(spec, host["V"])[0]
    assert np.allclose(got["sketch"][2], np.repeat(v[:, None, :], 64, axis=1), rtol=0, atol=1e-6)


def test_tokenwise_100k_user(cuda_lib):
    """One user at the paper's 100K-token history length (Sec. 3.1 workload),
    cut across many workers, next to two short users."""
    spec = wl.custom([3, 100_000, 129], H=1, P=512, d=128, dtype=wl.BF16, seed=11)
    host, got = _run(spec)
    _compare(spec, got, _oracle(spec, host), tol32=5e-4)


def test_tokenwise_no_tokens(cuda_lib):
    spec = wl.custom([0, 0], H=2, P=256, d=128, dtype=wl.BF16, seed=12)
    host, got = _run(spec)
    assert np.all(got["sketch"] == 0) and np.all(np.isneginf(got["lse"]))
    assert np.all(got["dQ"] == 0)


@pytest.mark.parametrize("P,d", [(512, 128), (256, 64), (128, 128), (384, 64), (1024, 128)])
def test_tokenwise_tensor_core_matches_cuda_core(cuda_lib, P, d):
    """The tcgen05 forward against the CUDA-core forward (two independent GPU
    implementations of the same normalisation) on the same inputs."""
    spec = wl.custom(RAGGED, H=2, P=P, d=d, dtype=wl.BF16, seed=P + d + 13)
    host = wl.make_host(spec)
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    tc = binding.sa_sketch_fwd_tokenwise(t["K"], t["V"], t["cu_seqlens"], t["Q"], spec.scale, want_lse=True)
    binding.sa_select_path(1)
    try:
        simt = binding.sa_sketch_fwd_tokenwise(t["K"], t["V"], t["cu_seqlens"], t["Q"], spec.scale, want_lse=True)
    finally:
        binding.sa_select_path(0)
    torch.cuda.synchronize()
    assert harness.rel_err(wl.torch_as_f64(tc[0]), wl.torch_as_f64(simt[0])) <= 2e-2
    a, b = wl.torch_as_f64(tc[1]), wl.torch_as_f64(simt[1])
    fin = np.isfinite(b)
    assert np.array_equal(np.isfinite(a), fin)
    assert np.max(np.abs(a[fin] - b[fin])) <= 5e-5 * max(1.0, np.max(np.abs(b[fin])))


@pytest.mark.parametrize("d", [128, 64])
def test_tokenwise_growing_scores_rescale(cuda_lib, d):
    """Keys whose norm grows along each history, so the running maximum of every
    prototype's scores keeps rising and the forward must re-shift its
    accumulator many times (on the tensor cores: the lazy rescale of O in TMEM)."""
    lens = [5000, 300, 0, 2500]
    spec = wl.custom(lens, H=1, P=256, d=d, dtype=wl.BF16, seed=14 + d, q_std=1.0)
    host = wl.make_host(spec)
    K = wl.host_as_f64(spec, host["K"])
    cu = host["cu_seqlens"]
    for b in range(len(lens)):
        n = cu[b + 1] - cu[b]
        K[cu[b]:cu[b + 1]] *= (1.0 + 24.0 * np.arange(n) / max(n, 1))[:, None, None]
    host["K"] = wl.f32_to_bf16_bits(K.astype(np.float32))
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    O, lse = binding.sa_sketch_fwd_tokenwise(t["K"], t["V"], t["cu_seqlens"], t["Q"], spec.scale, want_lse=True)
    torch.cuda.synchronize()
    ref_O, ref_lse = sa_forward_tokenwise(wl.host_as_f64(spec, host["K"]), wl.host_as_f64(spec, host["V"]), cu,
                                          wl.host_as_f64(spec, host["Q"]), spec.scale, with_lse=True)
    harness.assert_close("sketch", wl.torch_as_f64(O), ref_O, harness.TOL[wl.BF16])
    got_lse = wl.torch_as_f64(lse)
    fin = np.isfinite(ref_lse)
    assert np.max(np.abs(got_lse[fin] - ref_lse[fin])) <= 5e-5 * max(1.0, np.max(np.abs(ref_lse[fin])))


@pytest.mark.parametrize("P", [256, 512, 1024])
def test_tokenwise_backward_tensor_core_matches_cuda_core(cuda_lib, P):
    """The tcgen05 backward (token side + prototype slices) against the CUDA-core
    backward, both fed the same forward outputs."""
    spec = wl.custom(RAGGED, H=2, P=P, d=128, dtype=wl.BF16, seed=P + 15)
    host = wl.make_host(spec)
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    args = (t["K"], t["V"], t["cu_seqlens"], t["Q"])
    O, lse = binding.sa_sketch_fwd_tokenwise(*args, spec.scale, want_lse=True)
    tc = binding.sa_sketch_bwd_tokenwise(*args, t["dsketch"], spec.scale, sketch=O, lse=lse)
    binding.sa_select_path(1)
    try:
        simt = binding.sa_sketch_bwd_tokenwise(*args, t["dsketch"], spec.scale, sketch=O, lse=lse)
    finally:
        binding.sa_select_path(0)
    torch.cuda.synchronize()
    for name, x, y in zip(("dK", "dV", "dQ"), tc, simt):
        assert harness.rel_err(wl.torch_as_f64(x), wl.torch_as_f64(y)) <= 2e-2, name


def test_tokenwise_negative_scale(cuda_lib):
    """A negative scale runs the token-wise forward on the CUDA cores."""
    spec = wl.custom(RAGGED, H=2, P=256, d=128, dtype=wl.BF16, seed=17)
    host = wl.make_host(spec)
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    scale = -1.5 / np.sqrt(128)
    O, lse = binding.sa_sketch_fwd_tokenwise(t["K"], t["V"], t["cu_seqlens"], t["Q"], scale, want_lse=True)
    dK, dV, dQ = binding.sa_sketch_bwd_tokenwise(t["K"], t["V"], t["cu_seqlens"], t["Q"], t["dsketch"], scale,
                                                 sketch=O, lse=lse)
    torch.cuda.synchronize()
    K, V, Q = (wl.host_as_f64(spec, host[k]) for k in ("K", "V", "Q"))
    ref_O = sa_forward_tokenwise(K, V, host["cu_seqlens"], Q, scale)
    rK, rV, rQ = sa_backward_tokenwise(K, V, host["cu_seqlens"], Q, scale, host["dsketch"].astype(np.float64))
    tol = harness.TOL[wl.BF16]
    for name, got, ref in (("sketch", O, ref_O), ("dK", dK, rK), ("dV", dV, rV), ("dQ", dQ, rQ)):
        harness.assert_close(name, wl.torch_as_f64(got), ref, tol)
