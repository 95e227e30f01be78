"""The step on a batch in host memory (sa_sketch_step_host): users in chunks,
copies overlapped with the step through three streams.  Checked against the
device-buffer calls on the whole batch and against the fp64 oracle.

dK and dV are per-token results, the same on every chunking: bitwise equal to
the whole-batch call.  A user's sketch and dQ are sums whose grouping depends on
the chunking (the workers of a chunk split the users differently; dQ is summed
chunk by chunk), so they agree with the whole-batch call to fp32 rounding:
1e-5 and 1e-4 of max|.|.
"""
import numpy as np
import pytest
import torch

import harness
from paper_2609_08443_gb300 import binding, workloads as wl

pytestmark = pytest.mark.gpu

RAGGED = [0, 1, 127, 128, 129, 300, 0, 1000, 17, 2049, 0, 0, 640]


def _host(spec, pinned):
    host = wl.make_host(spec)
    t = wl.host_to_torch(spec, host, torch.device("cpu"))
    if pinned:
        t = {k: v.pin_memory() if hasattr(v, "pin_memory") else v for k, v in t.items()}
    return host, t


@pytest.mark.parametrize("P,d,chunk,pinned", [(512, 128, 700, True), (256, 64, 2000, False), (128, 128, 0, True),
                                              (64, 64, 300, True)], ids=lambda x: str(x))
def test_host_step_matches_device_calls_and_oracle(cuda_lib, P, d, chunk, pinned):
    dt = wl.F32 if P == 64 else wl.BF16
    spec = wl.custom(RAGGED, H=2, P=P, d=d, dtype=dt, seed=P + d + chunk)
    host, t = _host(spec, pinned)
    sk, dK, dV, dQ = binding.sa_sketch_step_host(t["K"], t["V"], t["cu_seqlens"], t["Q"], t["dsketch"], spec.scale,
                                                 chunk_tokens=chunk)
    dev = torch.device("cuda")
    g = {k: v.to(dev) for k, v in t.items() if hasattr(v, "to")}
    s_ref, lse = binding.sa_sketch_fwd(g["K"], g["V"], g["cu_seqlens"], g["Q"], spec.scale, want_lse=True)
    dK_ref, dV_ref, dQ_ref = binding.sa_sketch_bwd(g["K"], g["V"], g["cu_seqlens"], g["Q"], g["dsketch"], spec.scale,
                                                   lse=lse)
    torch.cuda.synchronize()
    assert torch.equal(dK, dK_ref.cpu()) and torch.equal(dV, dV_ref.cpu())
    assert harness.rel_err(wl.torch_as_f64(sk), wl.torch_as_f64(s_ref)) <= 1e-5
    assert harness.rel_err(wl.torch_as_f64(dQ), wl.torch_as_f64(dQ_ref)) <= 1e-4
    ref = harness.oracle_outputs(spec, host, bwd=True)
    tol = harness.TOL[spec.dtype]
    for name, got in (("sketch", sk), ("dK", dK), ("dV", dV), ("dQ", dQ)):
        harness.assert_close(name, wl.torch_as_f64(got), ref[name], tol)


def test_host_step_deterministic_and_repeatable(cuda_lib):
    spec = wl.custom(RAGGED * 2, H=2, P=512, d=128, dtype=wl.BF16, seed=3)
    _, t = _host(spec, True)
    args = (t["K"], t["V"], t["cu_seqlens"], t["Q"], t["dsketch"], spec.scale)
    a = binding.sa_sketch_step_host(*args, chunk_tokens=1500)
    b = binding.sa_sketch_step_host(*args, chunk_tokens=1500)
    for x, y in zip(a, b):
        assert torch.equal(x, y)
