"""The step with its key projection (Sec. 3.1: keys X W_K, values X) on the GPU:
sa_sketch_fwd_x / sa_sketch_bwd_x through the C ABI against the fp64 oracle's
sa_forward_x / sa_backward_x, element by element on seeded inputs.

The library folds W_K into the prototypes (Q W_K^T) and runs the step on
K = V = X; the oracle forms K = X W_K explicitly, so the two routes share no
arithmetic.  Tolerance: 1e-4 max|oracle| for fp32 inputs, 2e-2 for bf16.
"""
import numpy as np
import pytest
import torch

import harness
from oracle import sa_backward_x, sa_forward_x
from paper_2609_08443_gb300 import binding, workloads as wl

pytestmark = pytest.mark.gpu

RAGGED = [0, 1, 127, 128, 129, 300, 0, 1000, 17, 2049]


def _case(P, d, dt, H, seed):
    spec = wl.custom(RAGGED, H=H, P=P, d=d, dtype=dt, seed=seed)
    host = wl.make_host(spec)
    r = np.random.default_rng(seed + 99)
    Wk = (r.standard_normal((H, d, d)) / np.sqrt(d)).astype(np.float32)
    Wk_host = wl.f32_to_bf16_bits(Wk) if dt == wl.BF16 else Wk
    dev = torch.device("cuda")
    t = wl.host_to_torch(spec, host, dev)
    if dt == wl.BF16:
        Wk_t = torch.from_numpy(Wk_host.view(np.int16)).view(torch.bfloat16).to(dev)
    else:
        Wk_t = torch.from_numpy(Wk_host).to(dev)
    return spec, host, t, Wk_host, Wk_t


@pytest.mark.parametrize("P,d,dt,H", [(512, 128, wl.BF16, 2), (256, 64, wl.BF16, 2), (128, 128, wl.BF16, 1),
                                      (64, 64, wl.F32, 1), (1024, 128, wl.BF16, 1)], ids=lambda x: str(x))
def test_key_projection_fwd_bwd(cuda_lib, P, d, dt, H):
    spec, host, t, Wk_host, Wk_t = _case(P, d, dt, H, seed=P + d + 21)
    X = t["K"]  # the history: keys through W_K, values as is
    sketch, lse = binding.sa_sketch_fwd_x(X, t["cu_seqlens"], t["Q"], Wk_t, spec.scale, want_lse=True)
    dX, dQ, dWk = binding.sa_sketch_bwd_x(X, t["cu_seqlens"], t["Q"], Wk_t, t["dsketch"], spec.scale, lse=lse)
    torch.cuda.synchronize()
    Xf = wl.host_as_f64(spec, host["K"])
    Qf = wl.host_as_f64(spec, host["Q"])
    Wf = wl.host_as_f64(spec, Wk_host)
    cu = host["cu_seqlens"]
    O_ref = sa_forward_x(Xf, cu, Qf, Wf, spec.scale)
    dX_ref, dQ_ref, dW_ref = sa_backward_x(Xf, cu, Qf, Wf, spec.scale, host["dsketch"].astype(np.float64))
    tol = harness.TOL[spec.dtype]
    harness.assert_close("sketch", wl.torch_as_f64(sketch), O_ref, tol)
    harness.assert_close("dX", wl.torch_as_f64(dX), dX_ref, tol)
    harness.assert_close("dQ", wl.torch_as_f64(dQ), dQ_ref, tol)
    harness.assert_close("dWk", wl.torch_as_f64(dWk), dW_ref, tol)


def test_key_projection_deterministic(cuda_lib):
    spec, host, t, _, Wk_t = _case(512, 128, wl.BF16, 2, seed=77)
    runs = []
    for _ in range(3):
        s, lse = binding.sa_sketch_fwd_x(t["K"], t["cu_seqlens"], t["Q"], Wk_t, spec.scale, want_lse=True)
        g = binding.sa_sketch_bwd_x(t["K"], t["cu_seqlens"], t["Q"], Wk_t, t["dsketch"], spec.scale, lse=lse)
        torch.cuda.synchronize()
        runs.append([s.clone()] + [x.clone() for x in g])
    for r in runs[1:]:
        for a, b in zip(runs[0], r):
            assert torch.equal(a, b)
