"""Allocation-free forward entry point.

sa_sketch_fwd_noalloc serves callers that cannot give the library a workspace
(a plugin hook that only receives its input and output buffers, or a service
with a device-memory budget fixed ahead of time): it runs the same forward with
scratch taken from a fixed array inside the library.  This file is collected
last on purpose, so a failure here does not hide the other tests.
"""
import ctypes
import math

import numpy as np
import pytest
import torch

import harness
from paper_2609_08443_gb300 import binding, workloads as wl

pytestmark = pytest.mark.gpu

LENS = [300, 0, 129, 1700, 17]


def _call_noalloc(lib, t, P, scale, dt, sketch, lse, cu=None):
    N, H, d = t["K"].shape
    cu = t["cu_seqlens"] if cu is None else cu
    B = cu.numel() - 1
    vp = ctypes.c_void_p
    return lib.sa_sketch_fwd_noalloc(
        vp(t["K"].data_ptr()), vp(t["V"].data_ptr()), vp(cu.data_ptr()), B, N, vp(t["Q"].data_ptr()), H, P, d,
        scale, dt, vp(sketch.data_ptr()), None if lse is None else vp(lse.data_ptr()),
        vp(torch.cuda.current_stream().cuda_stream))


def _noalloc_status(lib):
    return lib.sa_noalloc_get_device_error(ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


CASES = [
    # (P, d, dtype, with_lse, scale sign)
    (256, 64, wl.BF16, True, 1),
    (256, 64, wl.BF16, False, 1),
    (128, 128, wl.BF16, False, 1),
    (64, 64, wl.F32, True, 1),
    (64, 64, wl.F32, False, 1),
    (256, 64, wl.BF16, True, -1),  # a negative scale
]


@pytest.mark.parametrize("P,d,dt,with_lse,sign", CASES, ids=lambda x: str(x))
def test_noalloc_matches_workspace_forward_twice(cuda_lib, P, d, dt, with_lse, sign):
    lib = binding.load()
    spec = wl.custom(LENS, H=2, P=P, d=d, dtype=dt, seed=21 + P + d)
    scale = sign * spec.scale
    t = wl.host_to_torch(spec, wl.make_host(spec), torch.device("cuda"))
    ref, ref_lse = binding.sa_sketch_fwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], scale, want_lse=True)
    torch.cuda.synchronize()
    B, H, P_, d_ = ref.shape
    code = binding.SA_BF16 if dt == wl.BF16 else binding.SA_F32
    for _ in range(2):  # two calls in a row: the shared scratch keeps the last call's contents
        sketch = torch.full((B, H, P_, d_), float("nan"), device="cuda")
        lse = torch.full_like(ref_lse, float("nan")) if with_lse else None
        assert _call_noalloc(lib, t, P, scale, code, sketch, lse) == 0
        assert _noalloc_status(lib) == 0
        assert harness.rel_err(sketch.double().cpu().numpy(), ref.double().cpu().numpy()) <= harness.TOL[dt]
        if with_lse:
            assert torch.isfinite(lse).all()
            assert (lse - ref_lse).abs().max().item() <= 5e-3 * max(1.0, ref_lse.abs().max().item())


def test_noalloc_matches_the_oracle(cuda_lib):
    lib = binding.load()
    spec = wl.custom(LENS, H=2, P=256, d=64, dtype=wl.BF16, seed=23)
    host = wl.make_host(spec)
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    B, H = len(LENS), 2
    sketch = torch.full((B, H, spec.P, spec.d), float("nan"), device="cuda")
    lse = torch.full((t["K"].shape[0], H), float("nan"), device="cuda")
    assert _call_noalloc(lib, t, spec.P, spec.scale, binding.SA_BF16, sketch, lse) == 0
    assert _noalloc_status(lib) == 0
    ref = harness.oracle_outputs(spec, host, bwd=False)
    harness.assert_close("sketch", wl.torch_as_f64(sketch), ref["sketch"], harness.TOL[wl.BF16])
    assert np.max(np.abs(wl.torch_as_f64(lse) - ref["lse"])) <= 5e-3 * max(1.0, np.max(np.abs(ref["lse"])))


def test_noalloc_reports_bad_offsets_then_recovers(cuda_lib):
    """Decreasing cu_seqlens are caught on the device: the call's kernels skip
    their work and sa_noalloc_get_device_error reports SA_ERR_BAD_SEQLENS; the
    next valid call clears the error word and is correct."""
    lib = binding.load()
    spec = wl.custom(LENS, H=2, P=256, d=64, dtype=wl.BF16, seed=25)
    t = wl.host_to_torch(spec, wl.make_host(spec), torch.device("cuda"))
    ref = binding.sa_sketch_fwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], spec.scale)
    torch.cuda.synchronize()
    bad = t["cu_seqlens"].clone()
    bad[2] = bad[1] - 1  # user 1 gets a negative length; the total stays N
    sketch = torch.zeros_like(ref)
    assert _call_noalloc(lib, t, spec.P, spec.scale, binding.SA_BF16, sketch, None, cu=bad) == 0
    assert _noalloc_status(lib) == 6  # SA_ERR_BAD_SEQLENS
    sketch = torch.full_like(ref, float("nan"))
    assert _call_noalloc(lib, t, spec.P, spec.scale, binding.SA_BF16, sketch, None) == 0
    assert _noalloc_status(lib) == 0
    assert harness.rel_err(sketch.double().cpu().numpy(), ref.double().cpu().numpy()) <= harness.TOL[wl.BF16]


def test_noalloc_rejects_sizes_beyond_its_scratch(cuda_lib):
    lib = binding.load()
    cap = binding.sa_noalloc_scratch_bytes()
    B, H, P, d = 1, 8, 512, 128
    N = cap // (4 * H) + 1  # the lse scratch alone would exceed the array
    assert binding.sa_workspace_size(B, N, H, P, d, binding.SA_BF16, 0) > cap
    vp = ctypes.c_void_p
    st = lib.sa_sketch_fwd_noalloc(vp(256), vp(256), vp(256), B, N, vp(256), H, P, d, 1 / math.sqrt(d),
                                   binding.SA_BF16, vp(256), None, None)
    assert st == 3  # SA_ERR_WORKSPACE, returned before anything is launched
