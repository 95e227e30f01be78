"""A negative scale on the tensor-core kernels.

Any finite scale is valid.  With shared prototypes the library folds a
negative one into a negated copy of Q (scale Q K^T = (-scale)(-Q) K^T exactly),
so the tensor-core kernels run unchanged.  Each case is compared with the fp64
oracle at the same negative scale, and bitwise with the positive-scale call on
-Q, which shows that the tensor-core kernels (not the CUDA-core fallback) ran.
"""
import numpy as np
import pytest
import torch

import harness
from oracle import sa_backward, sa_backward_tokenwise, sa_forward, sa_forward_tokenwise
from paper_2609_08443_gb300 import binding, workloads as wl

pytestmark = pytest.mark.gpu

RAGGED = [0, 1, 127, 128, 129, 300, 1000, 17, 2049]


def _problem(P, d, H, seed):
    spec = wl.custom(RAGGED, H=H, P=P, d=d, dtype=wl.BF16, seed=seed)
    host = wl.make_host(spec)
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    f64 = {k: wl.host_as_f64(spec, host[k]) for k in ("K", "V", "Q")}
    return spec, host, t, f64


@pytest.mark.parametrize("P,d,H", [(256, 64, 2), (128, 128, 2), (512, 128, 2), (512, 64, 1), (1024, 128, 1)],
                         ids=lambda x: str(x))
def test_negative_scale_prototype_wise(cuda_lib, P, d, H):
    spec, host, t, f = _problem(P, d, H, seed=400 + P + d)
    s = -spec.scale
    K, V, cu, Q, G = t["K"], t["V"], t["cu_seqlens"], t["Q"], t["dsketch"]
    sketch, lse = binding.sa_sketch_fwd(K, V, cu, Q, s, want_lse=True)
    dK, dV, dQ = binding.sa_sketch_bwd(K, V, cu, Q, G, s, lse=lse)
    dK_r, dV_r, dQ_r = binding.sa_sketch_bwd(K, V, cu, Q, G, s)  # lse recomputed
    torch.cuda.synchronize()
    O, L = sa_forward(f["K"], f["V"], host["cu_seqlens"], f["Q"], s, with_lse=True)
    rK, rV, rQ = sa_backward(f["K"], f["V"], host["cu_seqlens"], f["Q"], s, host["dsketch"].astype(np.float64))
    tol = harness.TOL[wl.BF16]
    harness.assert_close("sketch", wl.torch_as_f64(sketch), O, tol)
    assert np.max(np.abs(wl.torch_as_f64(lse) - L)) <= 5e-3 * max(1.0, np.max(np.abs(L)))
    for name, got, ref in (("dK", dK, rK), ("dV", dV, rV), ("dQ", dQ, rQ), ("dK (lse recomputed)", dK_r, rK),
                           ("dQ (lse recomputed)", dQ_r, rQ)):
        harness.assert_close(name, wl.torch_as_f64(got), ref, tol)
    # the same call at the positive scale on -Q: bitwise equal (dQ negated)
    Qn = (-Q).contiguous()
    sketch2, lse2 = binding.sa_sketch_fwd(K, V, cu, Qn, -s, want_lse=True)
    dK2, dV2, dQ2 = binding.sa_sketch_bwd(K, V, cu, Qn, G, -s, lse=lse2)
    torch.cuda.synchronize()
    assert torch.equal(sketch, sketch2) and torch.equal(lse, lse2)
    assert torch.equal(dK, dK2) and torch.equal(dV, dV2) and torch.equal(dQ, -dQ2)


@pytest.mark.parametrize("P,d", [(256, 64), (512, 128)], ids=lambda x: str(x))
def test_negative_scale_token_wise(cuda_lib, P, d):
    spec, host, t, f = _problem(P, d, 2, seed=500 + P + d)
    s = -spec.scale
    K, V, cu, Q, G = t["K"], t["V"], t["cu_seqlens"], t["Q"], t["dsketch"]
    O, lse = binding.sa_sketch_fwd_tokenwise(K, V, cu, Q, s, want_lse=True)
    dK, dV, dQ = binding.sa_sketch_bwd_tokenwise(K, V, cu, Q, G, s, sketch=O, lse=lse)
    torch.cuda.synchronize()
    rO, rL = sa_forward_tokenwise(f["K"], f["V"], host["cu_seqlens"], f["Q"], s, with_lse=True)
    rK, rV, rQ = sa_backward_tokenwise(f["K"], f["V"], host["cu_seqlens"], f["Q"], s,
                                       host["dsketch"].astype(np.float64))
    tol = harness.TOL[wl.BF16]
    harness.assert_close("sketch", wl.torch_as_f64(O), rO, tol)
    lt = wl.torch_as_f64(lse)
    fin = np.isfinite(rL)
    assert np.array_equal(np.isfinite(lt), fin)
    assert np.max(np.abs(lt[fin] - rL[fin])) <= 5e-3 * max(1.0, np.max(np.abs(rL[fin])))
    for name, got, ref in (("dK", dK, rK), ("dV", dV, rV), ("dQ", dQ, rQ)):
        harness.assert_close(name, wl.torch_as_f64(got), ref, tol)
    O2, lse2 = binding.sa_sketch_fwd_tokenwise(K, V, cu, (-Q).contiguous(), -s, want_lse=True)
    torch.cuda.synchronize()
    assert torch.equal(O, O2) and torch.equal(lse, lse2)
