"""Allocation-free forward entry point.

sa_sketch_fwd_noalloc serves callers that cannot give the library a workspace
(a plugin hook that only receives its input and output buffers, or a service
with a device-memory budget fixed ahead of time): it runs the same forward with
scratch taken from a fixed array inside the library.  This file is collected
last on purpose, so a failure here does not hide the other tests.
"""
import ctypes
import math

import pytest
import torch

import harness
from paper_2609_08443_gb300 import binding, workloads as wl

pytestmark = pytest.mark.gpu


def _call_noalloc(lib, t, spec, sketch, lse):
    N, H, d = t["K"].shape
    B = t["cu_seqlens"].numel() - 1
    vp = ctypes.c_void_p
    return lib.sa_sketch_fwd_noalloc(
        vp(t["K"].data_ptr()), vp(t["V"].data_ptr()), vp(t["cu_seqlens"].data_ptr()), B, N,
        vp(t["Q"].data_ptr()), H, spec.P, d, spec.scale, binding.SA_BF16, vp(sketch.data_ptr()),
        vp(lse.data_ptr()), vp(torch.cuda.current_stream().cuda_stream))


def test_noalloc_matches_workspace_forward_twice(cuda_lib):
    lib = binding.load()
    spec = wl.custom([300, 0, 129, 1700, 17], H=2, P=256, d=64, dtype=wl.BF16, seed=21)
    host = wl.make_host(spec)
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    ref, ref_lse = binding.sa_sketch_fwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], spec.scale, want_lse=True)
    torch.cuda.synchronize()
    B, H, P, d = ref.shape
    for _ in range(2):  # two calls in a row: the shared scratch keeps the last call's contents
        sketch = torch.full((B, H, P, d), float("nan"), device="cuda")
        lse = torch.full_like(ref_lse, float("nan"))
        assert _call_noalloc(lib, t, spec, sketch, lse) == 0
        torch.cuda.synchronize()
        assert harness.rel_err(sketch.double().cpu().numpy(), ref.double().cpu().numpy()) <= 2e-2
        assert torch.isfinite(lse).all()
        assert (lse - ref_lse).abs().max().item() <= 5e-3 * max(1.0, ref_lse.abs().max().item())


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
