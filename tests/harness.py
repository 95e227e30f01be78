"""Helpers shared by the GPU parity tests: run the C ABI and the fp64 oracle
on the same seeded inputs and compare element by element."""
from __future__ import annotations

import numpy as np

from oracle import sa_backward, sa_backward_per_user, sa_forward, sa_forward_per_user
from paper_2609_08443_gb300 import workloads as wl

TOL = {wl.F32: 1e-4, wl.BF16: 2e-2}  # max|gpu - oracle| <= TOL * max|oracle|


def rel_err(got, ref) -> float:
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    if ref.size == 0:
        return 0.0
    den = float(np.max(np.abs(ref)))
    num = float(np.max(np.abs(got - ref)))
    if den == 0.0:
        return num
    return num / den


def assert_close(name, got, ref, tol):
    assert np.all(np.isfinite(got)), f"{name}: non-finite values"
    e = rel_err(got, ref)
    assert e <= tol, f"{name}: max|gpu-oracle| / max|oracle| = {e:.3e} > {tol:.1e}"
    return e


def oracle_outputs(spec, host, bwd=True):
    K = wl.host_as_f64(spec, host["K"])
    V = wl.host_as_f64(spec, host["V"])
    Q = wl.host_as_f64(spec, host["Q"])
    cu = host["cu_seqlens"]
    per_user = Q.ndim == 4  # per-user queries of the stacked refinement (Sec. 3.3)
    fwd, bwd_fn = (sa_forward_per_user, sa_backward_per_user) if per_user else (sa_forward, sa_backward)
    O, lse = fwd(K, V, cu, Q, spec.scale, with_lse=True)
    out = {"sketch": O, "lse": lse}
    if bwd:
        dK, dV, dQ = bwd_fn(K, V, cu, Q, spec.scale, host["dsketch"].astype(np.float64))
        out.update(dK=dK, dV=dV, dQ=dQ)
    return out


def gpu_outputs(spec, t, bwd=True, pass_lse=True):
    import torch

    from paper_2609_08443_gb300 import binding

    sketch, lse = binding.sa_sketch_fwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], spec.scale, want_lse=True)
    out = {"sketch": sketch, "lse": lse}
    if bwd:
        dK, dV, dQ = binding.sa_sketch_bwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], t["dsketch"], spec.scale,
                                           lse=lse if pass_lse else None)
        out.update(dK=dK, dV=dV, dQ=dQ)
    torch.cuda.synchronize()
    return {k: wl.torch_as_f64(v) for k, v in out.items()}


def check_spec(spec, bwd=True, pass_lse=True, users=None, per_user_q=False):
    import torch

    host = wl.make_host(spec, users=users, per_user_q=per_user_q)
    t = wl.host_to_torch(spec, host, torch.device("cuda"))
    got = gpu_outputs(spec, t, bwd=bwd, pass_lse=pass_lse)
    ref = oracle_outputs(spec, host, bwd=bwd)
    tol = TOL[spec.dtype]
    errs = {}
    for k in ("sketch", "dK", "dV", "dQ") if bwd else ("sketch",):
        errs[k] = assert_close(k, got[k], ref[k], tol)
    # lse is an fp32 statistic: compare absolutely (it is O(log P) in size)
    if host["K"].shape[0]:
        assert np.max(np.abs(got["lse"] - ref["lse"])) <= 5e-3 * max(1.0, np.max(np.abs(ref["lse"])))
    return errs


def oracle_dq_chunk(job):
    """dQ [H, P, d] of one piece of one user's history (bf16 bit patterns of K
    and V, fp64 Q and that user's dsketch [H, P, d]).  The prototype-wise weights
    are per token, so a user's dQ is the sum of its pieces' dQ; worker function
    of the full-batch tests' process pool."""
    kbits, vbits, Q, G, scale = job
    K = wl.bf16_bits_to_f64(kbits)
    V = wl.bf16_bits_to_f64(vbits)
    _, _, dQ = sa_backward(K, V, np.array([0, K.shape[0]]), Q, scale, G[None])
    return dQ
