"""The 100K-token training workload at full size (128 users x 100000 tokens,
H=8, d=128, P=512, bf16, Q ~ N(0, 0.02)), run exactly as bench.py runs it (one
workspace, the library's own worker split), checked on outputs the fp64 oracle
computes one by one and on properties that hold at any size.

Prototype-wise weights are per token, so lse_i, dK_i and dV_i of a sampled
token depend on that token alone (and on its user's dsketch): the oracle runs
on one-token "users".  A sampled user's sketch is the oracle's forward on that
user.  dQ sums over all 12.8M tokens; it is checked by (a) its additivity over
users (two calls on halves of the batch, each with its own worker split, must
sum to the full call's dQ) and (b) the shift invariance of the prototype-wise
softmax: adding one vector to every prototype changes no weight, so
sum_j dQ[h, j] = 0 (to bf16 rounding of dS: sqrt(P) 2^-9 ~ 0.044 of max|dQ|).
The token-wise variant is checked the same way on whole users (its weights
couple all of a user's tokens).  Tolerances as in the parity tests, except for
the additivity of dQ: per token the two runs compute the same dS, but each
worker accumulates its ~42K tokens per head in TMEM (fp32, about 2600 UMMA
steps) and the two splits group the tokens differently; the sums agree to a
few 1e-3 of max|dQ| (2.2e-3 measured), so the check uses 1e-2 -- a lost or
doubled worker piece would move dQ by about 1/sqrt(38 workers) ~ 16 %.

Device memory: K and V take 26 GB each and every backward allocates dK and dV of
the same size, so the tests hold up to ~140 GB (a GB300 has 288 GB).
"""
import numpy as np
import pytest
import torch

import harness
from oracle import sa_backward, sa_backward_tokenwise, sa_forward, sa_forward_tokenwise
from paper_2609_08443_gb300 import binding, workloads as wl

pytestmark = pytest.mark.gpu

SAMPLE_USERS = (0, 77, 127)


@pytest.fixture(scope="module")
def full():
    spec = wl.config(4)
    dev = torch.device("cuda")
    data = wl.make_device(spec, dev)
    yield spec, data
    del data
    torch.cuda.empty_cache()


def _f64(t):
    return wl.torch_as_f64(t)


def _user(data, b):
    cu = data["cu_seqlens"].cpu().numpy()
    t0, t1 = int(cu[b]), int(cu[b + 1])
    return t0, t1


def test_fullsize_prototype_wise(cuda_lib, full):
    spec, data = full
    K, V, Q, cu, G = data["K"], data["V"], data["Q"], data["cu_seqlens"], data["dsketch"]
    B = cu.numel() - 1
    N, H, d = K.shape
    P = Q.shape[1]
    ws = torch.empty(binding.sa_workspace_size(B, N, H, P, d, binding.SA_BF16, 1), dtype=torch.uint8,
                     device=K.device)
    sketch, lse = binding.sa_sketch_fwd(K, V, cu, Q, spec.scale, want_lse=True, ws=ws)
    dK, dV, dQ = binding.sa_sketch_bwd(K, V, cu, Q, G, spec.scale, lse=lse, ws=ws)
    torch.cuda.synchronize()
    assert binding.sa_get_device_error(ws) == 0
    Qf = _f64(Q)
    tol = harness.TOL[wl.BF16]
    rng = np.random.default_rng(2024)
    for b in SAMPLE_USERS:
        t0, t1 = _user(data, b)
        Kb, Vb = _f64(K[t0:t1]), _f64(V[t0:t1])
        ref = sa_forward(Kb, Vb, np.array([0, t1 - t0]), Qf, spec.scale)
        harness.assert_close(f"sketch[user {b}]", _f64(sketch[b:b + 1]), ref, tol)
        # tokens one by one: the first, the last and random ones in between
        toks = sorted({t0, t1 - 1, *rng.integers(t0, t1, 30).tolist()})
        Gb = _f64(G[b:b + 1])
        for t in toks:
            k1, v1 = _f64(K[t:t + 1]), _f64(V[t:t + 1])
            one = np.array([0, 1])
            _, l1 = sa_forward(k1, v1, one, Qf, spec.scale, with_lse=True)
            dk1, dv1, _ = sa_backward(k1, v1, one, Qf, spec.scale, Gb)
            assert np.max(np.abs(_f64(lse[t:t + 1]) - l1)) <= 5e-3 * max(1.0, np.max(np.abs(l1)))
            harness.assert_close(f"dK[token {t}]", _f64(dK[t:t + 1]), dk1, tol)
            harness.assert_close(f"dV[token {t}]", _f64(dV[t:t + 1]), dv1, tol)
    # dQ: shift invariance, and additivity over two halves of the batch
    dq = _f64(dQ)
    assert np.max(np.abs(dq.sum(axis=1))) <= 0.1 * np.max(np.abs(dq))
    half = B // 2
    n_half = int(cu[half].item())
    cu_a = cu[: half + 1].clone()
    cu_b = (cu[half:] - cu[half]).contiguous()
    _, lse_a = binding.sa_sketch_fwd(K[:n_half], V[:n_half], cu_a, Q, spec.scale, want_lse=True)
    dq_a = binding.sa_sketch_bwd(K[:n_half], V[:n_half], cu_a, Q, G[:half].contiguous(), spec.scale, lse=lse_a)[2]
    _, lse_b = binding.sa_sketch_fwd(K[n_half:], V[n_half:], cu_b, Q, spec.scale, want_lse=True)
    dq_b = binding.sa_sketch_bwd(K[n_half:], V[n_half:], cu_b, Q, G[half:].contiguous(), spec.scale, lse=lse_b)[2]
    torch.cuda.synchronize()
    harness.assert_close("dQ = dQ(first half) + dQ(second half)", _f64(dq_a) + _f64(dq_b), dq, 1e-2)


def test_fullsize_tokenwise(cuda_lib, full):
    spec, data = full
    K, V, Q, cu, G = data["K"], data["V"], data["Q"], data["cu_seqlens"], data["dsketch"]
    B = cu.numel() - 1
    N, H, d = K.shape
    P = Q.shape[1]
    lib = binding.load()
    ws = torch.empty(lib.sa_workspace_size_tokenwise(B, N, H, P, d, binding.SA_BF16, 1), dtype=torch.uint8,
                     device=K.device)
    O, lse = binding.sa_sketch_fwd_tokenwise(K, V, cu, Q, spec.scale, want_lse=True, ws=ws)
    dK, dV, dQ = binding.sa_sketch_bwd_tokenwise(K, V, cu, Q, G, spec.scale, sketch=O, lse=lse, ws=ws)
    torch.cuda.synchronize()
    assert binding.sa_get_device_error(ws) == 0
    Qf = _f64(Q)
    tol = harness.TOL[wl.BF16]
    for b in SAMPLE_USERS[:2]:
        t0, t1 = _user(data, b)
        Kb, Vb = _f64(K[t0:t1]), _f64(V[t0:t1])
        one = np.array([0, t1 - t0])
        ref_O, ref_l = sa_forward_tokenwise(Kb, Vb, one, Qf, spec.scale, with_lse=True)
        harness.assert_close(f"sketch[user {b}]", _f64(O[b:b + 1]), ref_O, tol)
        assert np.max(np.abs(_f64(lse[b:b + 1]) - ref_l)) <= 5e-5 * max(1.0, np.max(np.abs(ref_l)))
    # one user's dK, dV in one head (the token-wise weights couple the user's tokens)
    b, h = SAMPLE_USERS[2], 5
    t0, t1 = _user(data, b)
    one = np.array([0, t1 - t0])
    dk, dv, _ = sa_backward_tokenwise(_f64(K[t0:t1, h:h + 1]), _f64(V[t0:t1, h:h + 1]), one, Qf[h:h + 1],
                                      spec.scale, _f64(G[b:b + 1, h:h + 1]))
    harness.assert_close("dK[user, head]", _f64(dK[t0:t1, h:h + 1]), dk, tol)
    harness.assert_close("dV[user, head]", _f64(dV[t0:t1, h:h + 1]), dv, tol)
    # dQ additivity over two halves of the batch
    half = B // 2
    n_half = int(cu[half].item())
    parts = []
    for sl_t, sl_b, c in ((slice(0, n_half), slice(0, half), cu[: half + 1].clone()),
                          (slice(n_half, N), slice(half, B), (cu[half:] - cu[half]).contiguous())):
        o, l = binding.sa_sketch_fwd_tokenwise(K[sl_t], V[sl_t], c, Q, spec.scale, want_lse=True)
        parts.append(binding.sa_sketch_bwd_tokenwise(K[sl_t], V[sl_t], c, Q, G[sl_b].contiguous(), spec.scale,
                                                     sketch=o, lse=l)[2])
    torch.cuda.synchronize()
    harness.assert_close("dQ = dQ(first half) + dQ(second half)", _f64(parts[0]) + _f64(parts[1]), _f64(dQ), 1e-2)
