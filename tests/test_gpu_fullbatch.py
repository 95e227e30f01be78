"""Two more evaluation workloads at full batch, run as bench.py runs them (one
workspace, the library's own worker split), against the fp64 oracle:

  * training step: 64 users, log-normal lengths (median 20K) clipped to
    [512, 100000], H=8, d=64, P=256, bf16, fwd+bwd;
  * ragged extremes: 4 users of 1048576 tokens among 4096 users of 1..512
    tokens, H=8, d=64, P=256, bf16, fwd+bwd.

Sampled users' sketches and sampled tokens' lse, dK and dV are computed by the
oracle one by one (the prototype-wise weights are per token, so a token's lse,
dK and dV depend on that token and its user's dsketch only).  The full-batch
dQ is compared with the oracle's dQ of every user, summed; each user's dQ is
itself summed over pieces of at most 65536 tokens, computed in a pool of
worker processes (spawned, not forked, so no worker inherits the CUDA context).
Tolerance: max|gpu - oracle| <= 2e-2 max|oracle| per tensor.
"""
import multiprocessing as mp
import os

import numpy as np
import pytest
import torch

import harness
from oracle import sa_backward, sa_forward
from paper_2609_08443_gb300 import binding, workloads as wl

pytestmark = pytest.mark.gpu

PIECE = 65536


def _f64(t):
    return wl.torch_as_f64(t)


def _bits(t):
    return t.contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def _oracle_dq(spec, data, cu_h):
    """sum over users b and pieces of b of the oracle's dQ (fp64), in a pool."""
    Qf = _f64(data["Q"])
    G = data["dsketch"]
    B = cu_h.size - 1

    def jobs():
        for b in range(B):
            t0, t1 = int(cu_h[b]), int(cu_h[b + 1])
            Gb = _f64(G[b])
            for s in range(t0, t1, PIECE):
                e = min(t1, s + PIECE)
                yield _bits(data["K"][s:e]), _bits(data["V"][s:e]), Qf, Gb, spec.scale

    env = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")}
    for k in env:
        os.environ[k] = "1"  # one BLAS thread per worker process
    try:
        nproc = max(1, min(16, len(os.sched_getaffinity(0))))
        total = np.zeros(Qf.shape)
        with mp.get_context("spawn").Pool(nproc) as pool:
            for dq in pool.imap_unordered(harness.oracle_dq_chunk, jobs(), chunksize=1):
                total += dq
    finally:
        for k, v in env.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    return total


@pytest.mark.parametrize("cfg", [3, 5], ids=["training-64-users", "ragged-extremes"])
def test_full_batch_against_oracle(cuda_lib, cfg):
    spec = wl.config(cfg)
    dev = torch.device("cuda")
    data = wl.make_device(spec, dev)
    K, V, Q, cu, G = data["K"], data["V"], data["Q"], data["cu_seqlens"], data["dsketch"]
    B = cu.numel() - 1
    N, H, d = K.shape
    P = Q.shape[1]
    ws = torch.empty(binding.sa_workspace_size(B, N, H, P, d, binding.SA_BF16, 1), dtype=torch.uint8, device=dev)
    sketch, lse = binding.sa_sketch_fwd(K, V, cu, Q, spec.scale, want_lse=True, ws=ws)
    dK, dV, dQ = binding.sa_sketch_bwd(K, V, cu, Q, G, spec.scale, lse=lse, ws=ws)
    torch.cuda.synchronize()
    assert binding.sa_get_device_error(ws) == 0
    tol = harness.TOL[wl.BF16]
    cu_h = cu.cpu().numpy().astype(np.int64)
    lens = np.diff(cu_h)
    Qf = _f64(Q)
    rng = np.random.default_rng(100 + cfg)
    longest = np.argsort(lens)[::-1]
    users = sorted({int(longest[0]), int(longest[1]), int(np.argmin(lens)), 0, B - 1,
                    *rng.integers(0, B, 6).tolist()})
    for b in users:
        t0, t1 = int(cu_h[b]), int(cu_h[b + 1])
        ref = sa_forward(_f64(K[t0:t1]), _f64(V[t0:t1]), np.array([0, t1 - t0]), Qf, spec.scale)
        harness.assert_close(f"sketch[user {b}, L={t1 - t0}]", _f64(sketch[b:b + 1]), ref, tol)
        if t1 == t0:
            continue
        Gb = _f64(G[b:b + 1])
        one = np.array([0, 1])
        for t in sorted({t0, t1 - 1, *rng.integers(t0, t1, 8).tolist()}):
            k1, v1 = _f64(K[t:t + 1]), _f64(V[t:t + 1])
            _, l1 = sa_forward(k1, v1, one, Qf, spec.scale, with_lse=True)
            dk1, dv1, _ = sa_backward(k1, v1, one, Qf, spec.scale, Gb)
            assert np.max(np.abs(_f64(lse[t:t + 1]) - l1)) <= 5e-3 * max(1.0, np.max(np.abs(l1))), f"lse[{t}]"
            harness.assert_close(f"dK[token {t}]", _f64(dK[t:t + 1]), dk1, tol)
            harness.assert_close(f"dV[token {t}]", _f64(dV[t:t + 1]), dv1, tol)
    harness.assert_close("dQ (whole batch)", _f64(dQ), _oracle_dq(spec, data, cu_h), tol)
    del data, K, V, dK, dV, ws
    torch.cuda.empty_cache()
