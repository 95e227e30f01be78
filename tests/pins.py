"""Pins of the SA oracle against facts the paper and mathematics fix.

Every ``pin_*`` takes the forward and backward functions under test (with the
signatures of ``oracle.sa_forward`` / ``oracle.sa_backward``) and raises
AssertionError when they disagree with:

  * a 50-digit brute-force evaluation of the paper's definition (Sec. 3.1:
    affinity S, prototype-wise softmax A, sketch A X), written as plain loops
    with no stabilising shift;
  * 50-digit central finite differences of that brute force (for the gradient,
    which the paper does not print);
  * the conservation law sum_j A[j, i] = 1 (Sec. 3.1, App. C): with V = 1 every
    sketch column sums to the user's history length;
  * closed forms: equal prototypes give uniform weights 1/P; P = 1 is sum
    pooling; L = 1 is one softmax (scipy.special.softmax); a huge scale gives
    a hard arg-max assignment;
  * invariances: token order within a user (SA has no positional term), ragged
    batch = users run alone, heads independent, linear in V, common shift of
    all prototypes; and the gradient facts those imply (sum_j dQ[h, j] = 0,
    dK = 0 for equal prototypes, dV_i = g when every row of G equals g).

``tests/test_oracle_mutants.py`` plants plausible mistakes in copies of the
oracle and checks that each is caught by at least one pin.
"""
from __future__ import annotations

import numpy as np


def _rng(seed):
    return np.random.default_rng(seed)


def _rand_problem(seed, lens, H, P, d, q_std=1.0):
    r = _rng(seed)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    N = int(cu[-1])
    K = r.standard_normal((N, H, d))
    V = r.standard_normal((N, H, d))
    Q = q_std * r.standard_normal((H, P, d))
    dO = r.standard_normal((len(lens), H, P, d))
    return K, V, cu, Q, dO


def _close(a, b, rtol, what):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    assert a.shape == b.shape, f"{what}: shape {a.shape} != {b.shape}"
    scale = max(1.0, float(np.max(np.abs(b)))) if b.size else 1.0
    err = float(np.max(np.abs(a - b))) if a.size else 0.0
    assert err <= rtol * scale, f"{what}: max err {err:.3e} > {rtol:.1e} * {scale:.3e}"


# ----------------------------------------------------------- brute force

def _mp_forward(K, V, cu, Q, scale, mp):
    """Plain-loop evaluation of O = softmax_proto(S) X in mpmath (no shift)."""
    H, P, d = len(Q), len(Q[0]), len(Q[0][0])
    B = len(cu) - 1
    O = [[[[mp.mpf(0)] * d for _ in range(P)] for _ in range(H)] for _ in range(B)]
    for b in range(B):
        for h in range(H):
            for i in range(int(cu[b]), int(cu[b + 1])):
                ex = []
                for j in range(P):
                    s = mp.mpf(0)
                    for c in range(d):
                        s += mp.mpf(Q[h][j][c]) * mp.mpf(K[i][h][c])
                    ex.append(mp.exp(mp.mpf(scale) * s))
                z = mp.fsum(ex)
                for j in range(P):
                    a = ex[j] / z
                    for c in range(d):
                        O[b][h][j][c] += a * mp.mpf(V[i][h][c])
    return O


def _mp_loss(K, V, cu, Q, scale, dO, mp):
    O = _mp_forward(K, V, cu, Q, scale, mp)
    tot = mp.mpf(0)
    B, H, P, d = dO.shape
    for b in range(B):
        for h in range(H):
            for j in range(P):
                for c in range(d):
                    tot += mp.mpf(dO[b, h, j, c]) * O[b][h][j][c]
    return tot


def pin_bruteforce_forward(fwd, bwd=None):
    import mpmath as mp
    mp.mp.dps = 50
    K, V, cu, Q, _ = _rand_problem(1, [3, 0, 2, 1], H=2, P=3, d=2)
    scale = 0.7
    ref = _mp_forward(K.tolist(), V.tolist(), cu, Q.tolist(), scale, mp)
    got = fwd(K, V, cu, Q, scale)
    refa = np.array([[[[float(x) for x in row] for row in hh] for hh in bb] for bb in ref])
    _close(got, refa, 1e-13, "brute-force sketch")


def pin_bruteforce_lse(fwd, bwd=None):
    import mpmath as mp
    mp.mp.dps = 50
    K, V, cu, Q, _ = _rand_problem(2, [2, 3], H=2, P=4, d=3)
    scale = 1.3
    _, lse = fwd(K, V, cu, Q, scale, with_lse=True)
    for i in range(K.shape[0]):
        for h in range(2):
            z = mp.fsum(mp.exp(mp.mpf(scale) * mp.fsum(mp.mpf(Q[h, j, c]) * mp.mpf(K[i, h, c])
                                                     for c in range(3))) for j in range(4))
            assert abs(float(mp.log(z)) - lse[i, h]) < 1e-12, "lse"


def pin_bruteforce_gradients(fwd, bwd):
    """50-digit central differences of sum(dO * O) against the backward."""
    import mpmath as mp
    mp.mp.dps = 50
    K, V, cu, Q, dO = _rand_problem(3, [2, 3], H=2, P=3, d=2)
    scale = 0.9
    dK, dV, dQ = bwd(K, V, cu, Q, scale, dO)
    eps = mp.mpf("1e-20")

    def fd(arr_name, idx):
        base = {"K": K.tolist(), "V": V.tolist(), "Q": Q.tolist()}

        def with_delta(delta):
            a = [list(map(list, x)) for x in base[arr_name]]
            i, j, k = idx
            a[i][j][k] = mp.mpf(a[i][j][k]) + delta
            args = dict(base)
            args[arr_name] = a
            return _mp_loss(args["K"], args["V"], cu, args["Q"], scale, dO, mp)

        return float((with_delta(eps) - with_delta(-eps)) / (2 * eps))

    for name, grad in (("K", dK), ("V", dV), ("Q", dQ)):
        for idx in np.ndindex(*grad.shape):
            ref = fd(name, idx)
            assert abs(grad[idx] - ref) <= 1e-11 * max(1.0, abs(ref)), \
                f"d{name}{idx}: {grad[idx]} vs finite difference {ref}"


# ------------------------------------------------------------ invariants

def pin_conservation(fwd, bwd=None):
    lens = [5, 1, 0, 17]
    K, V, cu, Q, _ = _rand_problem(4, lens, H=3, P=7, d=4)
    O = fwd(K, np.ones_like(V), cu, Q, 0.5)
    for b, L in enumerate(lens):
        _close(O[b].sum(axis=1), np.full((3, 4), float(L)), 1e-13, "column sums = L_b")


def pin_equal_prototypes(fwd, bwd):
    lens = [6, 3]
    K, V, cu, Q, dO = _rand_problem(5, lens, H=2, P=5, d=3)
    Q[:] = Q[:, :1, :]  # every prototype row identical
    O = fwd(K, V, cu, Q, 0.8)
    for b in range(2):
        t0, t1 = cu[b], cu[b + 1]
        mean = V[t0:t1].sum(axis=0) / 5.0  # (H, d)
        _close(O[b], np.repeat(mean[:, None, :], 5, axis=1), 1e-13, "uniform weights")
    dK, _, _ = bwd(K, V, cu, Q, 0.8, dO)
    _close(dK, np.zeros_like(dK), 1e-13, "dK = 0 for equal prototypes")


def pin_single_prototype(fwd, bwd=None):
    lens = [4, 9]
    K, V, cu, Q, _ = _rand_problem(6, lens, H=2, P=1, d=3)
    O = fwd(K, V, cu, Q, 1.1)
    for b in range(2):
        _close(O[b][:, 0, :], V[cu[b]:cu[b + 1]].sum(axis=0), 1e-13, "P=1 sum pooling")


def pin_single_token(fwd, bwd=None):
    from scipy.special import softmax
    K, V, cu, Q, _ = _rand_problem(7, [1], H=2, P=6, d=4)
    O = fwd(K, V, cu, Q, 0.3)
    for h in range(2):
        w = softmax(0.3 * (Q[h] @ K[0, h]))
        _close(O[0, h], np.outer(w, V[0, h]), 1e-13, "L=1 softmax")


def pin_hard_assignment(fwd, bwd=None):
    r = _rng(8)
    P, d, L = 4, 4, 12
    Q = np.eye(P, d)[None] * 1.0
    # each token points mostly at one prototype; the margin is large
    owner = r.integers(0, P, size=L)
    K = (np.eye(P, d)[owner] * 3.0 + 0.1 * r.standard_normal((L, d)))[:, None, :]
    V = r.standard_normal((L, 1, d))
    cu = np.array([0, L])
    O = fwd(K, V, cu, Q, 200.0)
    ref = np.zeros((P, d))
    for i in range(L):
        ref[owner[i]] += V[i, 0]
    _close(O[0, 0], ref, 1e-10, "hard assignment")


def pin_permutation(fwd, bwd):
    lens = [7, 5]
    K, V, cu, Q, dO = _rand_problem(9, lens, H=2, P=4, d=3)
    perm = np.concatenate([np.random.default_rng(1).permutation(7),
                           7 + np.random.default_rng(2).permutation(5)])
    O1 = fwd(K, V, cu, Q, 0.6)
    O2 = fwd(K[perm], V[perm], cu, Q, 0.6)
    _close(O2, O1, 1e-13, "token order")
    g1 = bwd(K, V, cu, Q, 0.6, dO)
    g2 = bwd(K[perm], V[perm], cu, Q, 0.6, dO)
    _close(g2[0], g1[0][perm], 1e-13, "dK permuted")
    _close(g2[1], g1[1][perm], 1e-13, "dV permuted")
    _close(g2[2], g1[2], 1e-12, "dQ order")


def pin_ragged_batch(fwd, bwd):
    lens = [3, 0, 8, 1]
    K, V, cu, Q, dO = _rand_problem(10, lens, H=2, P=5, d=3)
    O = fwd(K, V, cu, Q, 0.4)
    dK, dV, dQ = bwd(K, V, cu, Q, 0.4, dO)
    dQ_sum = np.zeros_like(dQ)
    for b in range(4):
        t0, t1 = cu[b], cu[b + 1]
        one = np.array([0, t1 - t0])
        _close(O[b:b + 1], fwd(K[t0:t1], V[t0:t1], one, Q, 0.4), 1e-13, "batch vs alone")
        gk, gv, gq = bwd(K[t0:t1], V[t0:t1], one, Q, 0.4, dO[b:b + 1])
        _close(dK[t0:t1], gk, 1e-13, "dK batch vs alone")
        _close(dV[t0:t1], gv, 1e-13, "dV batch vs alone")
        dQ_sum += gq
    _close(dQ, dQ_sum, 1e-12, "dQ is the sum over users")


def pin_heads_independent(fwd, bwd=None):
    lens = [6]
    K, V, cu, Q, _ = _rand_problem(11, lens, H=3, P=4, d=2)
    O = fwd(K, V, cu, Q, 0.7)
    K2, V2, Q2 = K.copy(), V.copy(), Q.copy()
    K2[:, 1] += 1.0
    V2[:, 1] *= -2.0
    Q2[1] = 0.0
    O2 = fwd(K2, V2, cu, Q2, 0.7)
    _close(O2[:, [0, 2]], O[:, [0, 2]], 1e-13, "other heads untouched")


def pin_linear_in_v(fwd, bwd=None):
    lens = [5, 4]
    K, V, cu, Q, _ = _rand_problem(12, lens, H=2, P=3, d=3)
    V2 = _rng(13).standard_normal(V.shape)
    lhs = fwd(K, 2.0 * V - 0.5 * V2, cu, Q, 0.5)
    rhs = 2.0 * fwd(K, V, cu, Q, 0.5) - 0.5 * fwd(K, V2, cu, Q, 0.5)
    _close(lhs, rhs, 1e-13, "linear in V")


def pin_prototype_shift(fwd, bwd):
    lens = [6, 2]
    K, V, cu, Q, dO = _rand_problem(14, lens, H=2, P=5, d=3)
    u = _rng(15).standard_normal((2, 1, 3))
    _close(fwd(K, V, cu, Q + u, 0.9), fwd(K, V, cu, Q, 0.9), 1e-12, "common shift")
    _, _, dQ = bwd(K, V, cu, Q, 0.9, dO)
    _close(dQ.sum(axis=1), np.zeros((2, 3)), 1e-12, "sum_j dQ = 0")


def pin_constant_upstream(fwd, bwd):
    lens = [4, 3]
    K, V, cu, Q, _ = _rand_problem(16, lens, H=2, P=6, d=3)
    g = _rng(17).standard_normal((2, 2, 1, 3))
    dO = np.repeat(g, 6, axis=2)
    _, dV, _ = bwd(K, V, cu, Q, 0.5, dO)
    for b in range(2):
        _close(dV[cu[b]:cu[b + 1]], np.repeat(g[b, :, 0][None], lens[b], axis=0), 1e-13,
               "dV = g")


def pin_fd_fp64(fwd, bwd):
    """fp64 central differences at a size brute force cannot reach."""
    lens = [9, 4]
    K, V, cu, Q, dO = _rand_problem(18, lens, H=2, P=8, d=5)
    scale = 1.0 / np.sqrt(5.0)
    dK, dV, dQ = bwd(K, V, cu, Q, scale, dO)
    r = _rng(19)

    def loss(K_, V_, Q_):
        return float(np.sum(dO * fwd(K_, V_, cu, Q_, scale)))

    for name, grad in (("K", dK), ("V", dV), ("Q", dQ)):
        for _ in range(12):
            idx = tuple(int(r.integers(0, s)) for s in grad.shape)
            args = {"K": K.copy(), "V": V.copy(), "Q": Q.copy()}
            h = 1e-6
            args[name][idx] += h
            lp = loss(args["K"], args["V"], args["Q"])
            args[name][idx] -= 2 * h
            lm = loss(args["K"], args["V"], args["Q"])
            ref = (lp - lm) / (2 * h)
            assert abs(grad[idx] - ref) <= 1e-6 * max(1.0, abs(ref)), f"d{name}{idx}"


ALL_PINS = [
    pin_bruteforce_forward, pin_bruteforce_lse, pin_bruteforce_gradients, pin_conservation,
    pin_equal_prototypes, pin_single_prototype, pin_single_token, pin_hard_assignment,
    pin_permutation, pin_ragged_batch, pin_heads_independent, pin_linear_in_v,
    pin_prototype_shift, pin_constant_upstream, pin_fd_fp64,
]


# ------------------------------------------- per-user queries (Sec. 3.3)
# Pins of (fwd_uq, bwd_uq) with the signatures of oracle.sa_forward_per_user /
# oracle.sa_backward_per_user: Q[b, h] per user, dQ[b, h] per user.  They are
# checked against the shared-query functions, which the pins above fix, and
# against their own central finite differences.

def _rand_problem_uq(seed, lens, H, P, d):
    K, V, cu, _, dO = _rand_problem(seed, lens, H, P, d)
    Qu = _rng(seed + 1000).standard_normal((len(lens), H, P, d))
    return K, V, cu, Qu, dO


def pin_uq_broadcast(fwd_uq, bwd_uq, fwd=None, bwd=None):
    """The same prototypes for every user: the shared-query results, and the
    per-user dQ summing to the shared dQ (Sec. 3.1: the prototypes are global)."""
    from oracle import sa_backward, sa_forward

    lens = [5, 0, 3, 7]
    K, V, cu, Q, dO = _rand_problem(31, lens, H=2, P=4, d=3)
    Qu = np.broadcast_to(Q, (len(lens),) + Q.shape).copy()
    scale = 0.7
    O_u, lse_u = fwd_uq(K, V, cu, Qu, scale, with_lse=True)
    O, lse = sa_forward(K, V, cu, Q, scale, with_lse=True)
    _close(O_u, O, 1e-12, "sketch, broadcast prototypes")
    _close(lse_u, lse, 1e-12, "lse, broadcast prototypes")
    dK_u, dV_u, dQ_u = bwd_uq(K, V, cu, Qu, scale, dO)
    dK, dV, dQ = sa_backward(K, V, cu, Q, scale, dO)
    _close(dK_u, dK, 1e-12, "dK, broadcast prototypes")
    _close(dV_u, dV, 1e-12, "dV, broadcast prototypes")
    _close(dQ_u.sum(axis=0), dQ, 1e-12, "sum over users of per-user dQ")
    assert np.all(dQ_u[1] == 0), "an empty user has no query gradient"


def pin_uq_users_alone(fwd_uq, bwd_uq, fwd=None, bwd=None):
    """Each user of a ragged batch equals that user alone with the shared-query
    functions and Q = that user's prototypes."""
    from oracle import sa_backward, sa_forward

    lens = [6, 2, 0, 9]
    K, V, cu, Qu, dO = _rand_problem_uq(32, lens, H=2, P=5, d=4)
    scale = 0.6
    O_u = fwd_uq(K, V, cu, Qu, scale)
    dK_u, dV_u, dQ_u = bwd_uq(K, V, cu, Qu, scale, dO)
    for b in range(len(lens)):
        t0, t1 = int(cu[b]), int(cu[b + 1])
        c1 = np.array([0, t1 - t0])
        O1 = sa_forward(K[t0:t1], V[t0:t1], c1, Qu[b], scale)
        _close(O_u[b:b + 1], O1, 1e-12, f"sketch of user {b}")
        dK1, dV1, dQ1 = sa_backward(K[t0:t1], V[t0:t1], c1, Qu[b], scale, dO[b:b + 1])
        _close(dK_u[t0:t1], dK1, 1e-12, f"dK of user {b}")
        _close(dV_u[t0:t1], dV1, 1e-12, f"dV of user {b}")
        _close(dQ_u[b], dQ1, 1e-12, f"dQ of user {b}")


def pin_uq_conservation(fwd_uq, bwd_uq=None, fwd=None, bwd=None):
    """V = 1: every sketch column sums to the user's length (sum_j A[j, i] = 1)."""
    lens = [4, 0, 11]
    K, _, cu, Qu, _ = _rand_problem_uq(33, lens, H=3, P=6, d=2)
    O = fwd_uq(K, np.ones_like(K), cu, Qu, 0.9)
    for b, L in enumerate(lens):
        _close(O[b].sum(axis=1), np.full((3, 2), float(L)), 1e-12, f"column sums of user {b}")


def pin_uq_fd_fp64(fwd_uq, bwd_uq, fwd=None, bwd=None):
    """fp64 central differences of the per-user forward, for dQ (per user) and dK."""
    lens = [7, 5]
    K, V, cu, Qu, dO = _rand_problem_uq(34, lens, H=2, P=6, d=4)
    scale = 0.5
    dK, _, dQ = bwd_uq(K, V, cu, Qu, scale, dO)
    r = _rng(35)

    def loss(K_, Q_):
        return float(np.sum(dO * fwd_uq(K_, V, cu, Q_, scale)))

    for name, grad in (("K", dK), ("Q", dQ)):
        for _ in range(12):
            idx = tuple(int(r.integers(0, s)) for s in grad.shape)
            args = {"K": K.copy(), "Q": Qu.copy()}
            h = 1e-6
            args[name][idx] += h
            lp = loss(args["K"], args["Q"])
            args[name][idx] -= 2 * h
            lm = loss(args["K"], args["Q"])
            ref = (lp - lm) / (2 * h)
            assert abs(grad[idx] - ref) <= 1e-6 * max(1.0, abs(ref)), f"d{name}{idx}"


UQ_PINS = [pin_uq_broadcast, pin_uq_users_alone, pin_uq_conservation, pin_uq_fd_fp64]


# --------------------------------- key projection in the step (Sec. 3.1)
# Pins of (fwd_x, bwd_x) with the signatures of oracle.sa_forward_x /
# oracle.sa_backward_x: X [N, H, d] serves as the values and, through
# W_K [H, d, d], as the keys.

def _rand_problem_x(seed, lens, H, P, d):
    X, _, cu, Q, dO = _rand_problem(seed, lens, H, P, d)
    Wk = _rng(seed + 2000).standard_normal((H, d, d)) / np.sqrt(d)
    return X, cu, Q, Wk, dO


def pin_x_identity_projection(fwd_x, bwd_x, fwd=None, bwd=None):
    """W_K = I: keys and values are the history itself; the gradient of X is
    then the sum of the plain oracle's dK and dV."""
    from oracle import sa_backward, sa_forward

    lens = [5, 0, 8]
    X, cu, Q, _, dO = _rand_problem_x(41, lens, H=2, P=4, d=3)
    eye = np.broadcast_to(np.eye(3), (2, 3, 3)).copy()
    _close(fwd_x(X, cu, Q, eye, 0.8), sa_forward(X, X, cu, Q, 0.8), 1e-12, "sketch, W_K = I")
    dX, dQ, _ = bwd_x(X, cu, Q, eye, 0.8, dO)
    dK, dV, dQ1 = sa_backward(X, X, cu, Q, 0.8, dO)
    _close(dX, dK + dV, 1e-12, "dX, W_K = I")
    _close(dQ, dQ1, 1e-12, "dQ, W_K = I")


def pin_x_folded_prototypes(fwd_x, bwd_x, fwd=None, bwd=None):
    """S = Q (X W_K)^T = (Q W_K^T) X^T: the sketch equals the plain oracle with
    prototypes Q W_K^T and K = V = X (associativity of the product)."""
    from oracle import sa_forward

    lens = [7, 3]
    X, cu, Q, Wk, _ = _rand_problem_x(42, lens, H=2, P=5, d=4)
    Qf = np.einsum("hjc,hec->hje", Q, Wk)
    _close(fwd_x(X, cu, Q, Wk, 0.6), sa_forward(X, X, cu, Qf, 0.6), 1e-12, "sketch with folded prototypes")


def pin_x_fd_fp64(fwd_x, bwd_x, fwd=None, bwd=None):
    """fp64 central differences of the forward for dX, dQ and dW_K."""
    lens = [6, 4]
    X, cu, Q, Wk, dO = _rand_problem_x(43, lens, H=2, P=5, d=4)
    scale = 0.5
    dX, dQ, dWk = bwd_x(X, cu, Q, Wk, scale, dO)
    r = _rng(44)

    def loss(X_, Q_, W_):
        return float(np.sum(dO * fwd_x(X_, cu, Q_, W_, scale)))

    for name, grad in (("X", dX), ("Q", dQ), ("W", dWk)):
        for _ in range(12):
            idx = tuple(int(r.integers(0, s)) for s in grad.shape)
            args = {"X": X.copy(), "Q": Q.copy(), "W": Wk.copy()}
            h = 1e-6
            args[name][idx] += h
            lp = loss(args["X"], args["Q"], args["W"])
            args[name][idx] -= 2 * h
            lm = loss(args["X"], args["Q"], args["W"])
            ref = (lp - lm) / (2 * h)
            assert abs(grad[idx] - ref) <= 1e-6 * max(1.0, abs(ref)), f"d{name}{idx}"


X_PINS = [pin_x_identity_projection, pin_x_folded_prototypes, pin_x_fd_fp64]


# ------------------------- token-wise ("vanilla") normalisation (Sec. 5.1)
# Pins of (fwd_tw, bwd_tw) with the signatures of oracle.sa_forward_tokenwise /
# oracle.sa_backward_tokenwise (weights normalised over each user's tokens).

def pin_tw_bruteforce(fwd_tw, bwd_tw=None, fwd=None, bwd=None):
    """50-digit plain loops of A[j, i] = exp(S[j, i]) / sum_i' exp(S[j, i']),
    O = A V, no stabilising shift."""
    import mpmath as mp

    mp.mp.dps = 50
    lens = [3, 0, 2]
    K, V, cu, Q, _ = _rand_problem(51, lens, H=2, P=3, d=2)
    scale = 0.9
    O = fwd_tw(K, V, cu, Q, scale)
    for b in range(len(lens)):
        t0, t1 = int(cu[b]), int(cu[b + 1])
        for h in range(2):
            for j in range(3):
                s = [mp.mpf(scale) * mp.fsum(mp.mpf(Q[h, j, c]) * mp.mpf(K[i, h, c]) for c in range(2))
                     for i in range(t0, t1)]
                z = mp.fsum(mp.exp(x) for x in s)
                for c in range(2):
                    ref = mp.fsum(mp.exp(s[i - t0]) / z * mp.mpf(V[i, h, c]) for i in range(t0, t1)) if s else 0
                    assert abs(O[b, h, j, c] - float(ref)) <= 1e-12 * max(1.0, abs(float(ref))), (b, h, j, c)


def pin_tw_bruteforce_lse(fwd_tw, bwd_tw=None, fwd=None, bwd=None):
    """50-digit plain loops of lse_tok[b, h, j] = log sum_i exp(S[j, i]) over
    user b's tokens (no stabilising shift), and -inf for a user with none."""
    import mpmath as mp

    mp.mp.dps = 50
    lens = [4, 0, 1, 3]
    K, V, cu, Q, _ = _rand_problem(58, lens, H=2, P=3, d=3, q_std=2.0)
    scale = 1.1
    _, lse = fwd_tw(K, V, cu, Q, scale, with_lse=True)
    assert lse.shape == (len(lens), 2, 3), f"lse_tok shape {lse.shape}"
    for b in range(len(lens)):
        t0, t1 = int(cu[b]), int(cu[b + 1])
        for h in range(2):
            for j in range(3):
                if t1 == t0:
                    assert lse[b, h, j] == -np.inf, (b, h, j)
                    continue
                z = mp.fsum(mp.exp(mp.mpf(scale) * mp.fsum(mp.mpf(Q[h, j, c]) * mp.mpf(K[i, h, c])
                                                         for c in range(3))) for i in range(t0, t1))
                ref = float(mp.log(z))
                assert abs(lse[b, h, j] - ref) <= 1e-12 * max(1.0, abs(ref)), (b, h, j, lse[b, h, j], ref)


def pin_tw_rows_sum_to_one(fwd_tw, bwd_tw=None, fwd=None, bwd=None):
    """V = 1: every sketch entry of a non-empty user is 1 (sum_i A[j, i] = 1)."""
    lens = [4, 0, 9]
    K, V, cu, Q, _ = _rand_problem(52, lens, H=2, P=5, d=3)
    O = fwd_tw(K, np.ones_like(V), cu, Q, 0.7)
    _close(O[0], np.ones((2, 5, 3)), 1e-12, "user 0")
    _close(O[2], np.ones((2, 5, 3)), 1e-12, "user 2")
    assert np.all(O[1] == 0), "an empty user has a zero sketch"


def pin_tw_closed_forms(fwd_tw, bwd_tw=None, fwd=None, bwd=None):
    """One token: O[j] = v_1 for every prototype.  Equal keys: O[j] is the mean
    of the user's values.  A huge scale: O[j] = v at arg max_i S[j, i]."""
    r = _rng(53)
    Q = r.standard_normal((1, 4, 3))
    K1, V1 = r.standard_normal((1, 1, 3)), r.standard_normal((1, 1, 3))
    _close(fwd_tw(K1, V1, np.array([0, 1]), Q, 0.5)[0, 0], np.repeat(V1[0], 4, axis=0), 1e-12, "one token")
    Ke = np.repeat(r.standard_normal((1, 1, 3)), 6, axis=0)
    Ve = r.standard_normal((6, 1, 3))
    _close(fwd_tw(Ke, Ve, np.array([0, 6]), Q, 0.5)[0, 0], np.repeat(Ve.mean(axis=0), 4, axis=0), 1e-12, "equal keys")
    Kh, Vh = r.standard_normal((7, 1, 3)), r.standard_normal((7, 1, 3))
    O = fwd_tw(Kh, Vh, np.array([0, 7]), Q, 1e4)[0, 0]
    arg = np.argmax(Q[0] @ Kh[:, 0, :].T, axis=1)
    _close(O, Vh[arg, 0, :], 1e-9, "hard selection")


def pin_tw_token_order(fwd_tw, bwd_tw, fwd=None, bwd=None):
    """Permuting a user's tokens permutes dK, dV and changes nothing else."""
    lens = [8]
    K, V, cu, Q, dO = _rand_problem(54, lens, H=2, P=4, d=3)
    perm = _rng(55).permutation(8)
    _close(fwd_tw(K[perm], V[perm], cu, Q, 0.6), fwd_tw(K, V, cu, Q, 0.6), 1e-12, "sketch under permutation")
    dK, dV, dQ = bwd_tw(K, V, cu, Q, 0.6, dO)
    dKp, dVp, dQp = bwd_tw(K[perm], V[perm], cu, Q, 0.6, dO)
    _close(dKp, dK[perm], 1e-12, "dK under permutation")
    _close(dVp, dV[perm], 1e-12, "dV under permutation")
    _close(dQp, dQ, 1e-12, "dQ under permutation")


def pin_tw_fd_fp64(fwd_tw, bwd_tw, fwd=None, bwd=None):
    """fp64 central differences for dK, dV, dQ."""
    lens = [7, 0, 5]
    K, V, cu, Q, dO = _rand_problem(56, lens, H=2, P=6, d=4)
    scale = 0.5
    dK, dV, dQ = bwd_tw(K, V, cu, Q, scale, dO)
    r = _rng(57)

    def loss(K_, V_, Q_):
        return float(np.sum(dO * fwd_tw(K_, V_, cu, Q_, scale)))

    for name, grad in (("K", dK), ("V", dV), ("Q", dQ)):
        for _ in range(12):
            idx = tuple(int(r.integers(0, s)) for s in grad.shape)
            args = {"K": K.copy(), "V": V.copy(), "Q": Q.copy()}
            h = 1e-6
            args[name][idx] += h
            lp = loss(args["K"], args["V"], args["Q"])
            args[name][idx] -= 2 * h
            lm = loss(args["K"], args["V"], args["Q"])
            ref = (lp - lm) / (2 * h)
            assert abs(grad[idx] - ref) <= 1e-6 * max(1.0, abs(ref)), f"d{name}{idx}"


TW_PINS = [pin_tw_bruteforce, pin_tw_bruteforce_lse, pin_tw_rows_sum_to_one, pin_tw_closed_forms, pin_tw_token_order, pin_tw_fd_fp64]
