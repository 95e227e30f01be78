"""fp64 CPU oracle of the Sketch Attention (SA) sketching step.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or
execute this module: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.  It shares
no code with the CUDA library; the two meet only in the seeded inputs drawn by
``paper_2609_08443_gb300.workloads`` (which holds none of the arithmetic).

What it computes (paper Sec. 3.1, equations for S, A and the sketch
``eq:sa-sketch``; the same three steps are listed in App. B):

  per user b (rows cu[b]..cu[b+1] of the packed K, V) and head h:
    S[j, i]  = scale * <Q[h, j, :], K_b[i, h, :]>          P x L_b   (affinity)
    A[:, i]  = softmax over the prototype axis j of S[:, i]          (prototype-wise
               normalisation: every token spreads unit mass over the P prototypes)
    O[b, h]  = A @ V_b[:, h, :]                             P x d     (sketch)

The paper normalises nothing further: the sketch is the plain weighted sum
over tokens (Sec. 3.1, "Sketch construction").  Heads are independent copies
of the single-head SA of the paper.  ``scale`` is passed in; the paper uses
1/sqrt(d) with d the SA width.

The paper prints no backward pass; it states only that the sketch is fully
differentiable and trained end to end (Sec. 3.1, App. F).  The gradient below
is the chain rule of the three forward steps with upstream G = dL/dO[b, h]:
    dV_b   = A^T G                                   (L_b x d)
    dA     = G V_b^T                                 (P x L_b)
    dS     = A * (dA - 1 colsum(A * dA))   (softmax Jacobian along the prototype axis)
    dK_b   = scale * dS^T Q[h]                       (L_b x d)
    dQ[h] += scale * dS K_b    summed over ALL users, because the prototypes are
                               shared globally (Sec. 3.1)

Stacked refinement (Sec. 3.3): from the second SA step on, the queries are the
user's own refined sketch times W_Q^(l), so every user b has its own
prototypes Q[b, h] ([B, H, P, d]); the three steps are otherwise unchanged and
dQ[b, h] = scale * dS K_b collects only user b's tokens
(``sa_forward_per_user`` / ``sa_backward_per_user``).

Key projection in the step (Sec. 3.1, S = (P W_Q)(X W_K)^T / sqrt(d), sketch
A X; App. G.3, K = X W_K): the history X serves as the values and, through
W_K, as the keys.  ``sa_forward_x`` / ``sa_backward_x`` take X [N, H, d] and
W_K [H, d, d] (per head, k_i = x_i W_K[h]) and return the gradients of X, Q and
W_K by the chain rule through K = X W_K.

Token-wise ("vanilla") normalisation, the comparison of Sec. 5.1 and App. C:
the same scores normalised over the user's tokens instead of the prototypes,
A[j, :] = softmax over i of S[j, i] (weights p(i | j), each prototype
selecting tokens), sketch = A V_b (``sa_forward_tokenwise`` /
``sa_backward_tokenwise``; the softmax Jacobian then runs along the token axis).

All arithmetic is float64; bf16 inputs arrive already widened exactly.
Parity pins for both functions live in ``tests/test_oracle.py`` (brute force
in 50-digit arithmetic, closed forms, invariants, finite differences).
"""
from __future__ import annotations

import numpy as np


def _user_slices(cu_seqlens):
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    return [(int(cu[b]), int(cu[b + 1])) for b in range(cu.size - 1)]


def affinity(Qh, Kbh, scale):
    """S = scale * Q K^T for one (user, head): P x L (Sec. 3.1, affinity S)."""
    return scale * (Qh @ Kbh.T)


def proto_softmax(S):
    """Softmax along axis 0 (the prototype axis) of a P x L score matrix.

    The per-column max is subtracted first; in exact arithmetic this shift
    cancels (Sec. 3.1, A = softmax_proto(S)).
    """
    m = S.max(axis=0, keepdims=True)
    e = np.exp(S - m)
    return e / e.sum(axis=0, keepdims=True)


def sa_forward(K, V, cu_seqlens, Q, scale, with_lse=False):
    """Sketch O[B, H, P, d] (and optionally per-token log-sum-exp lse[N, H]).

    K, V: [N, H, d] float64;  Q: [H, P, d] float64;  cu_seqlens: [B + 1].
    A user with no tokens gets an all-zero sketch (empty sum).
    """
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    Q = np.asarray(Q, dtype=np.float64)
    H, P, d = Q.shape
    sl = _user_slices(cu_seqlens)
    O = np.zeros((len(sl), H, P, d))
    lse = np.zeros((K.shape[0], H))
    for b, (t0, t1) in enumerate(sl):
        if t1 == t0:
            continue
        for h in range(H):
            S = affinity(Q[h], K[t0:t1, h, :], scale)
            A = proto_softmax(S)
            O[b, h] = A @ V[t0:t1, h, :]
            if with_lse:
                m = S.max(axis=0)
                lse[t0:t1, h] = m + np.log(np.exp(S - m).sum(axis=0))
    return (O, lse) if with_lse else O


def sa_backward(K, V, cu_seqlens, Q, scale, dO):
    """Gradients (dK [N,H,d], dV [N,H,d], dQ [H,P,d]) of L = sum(dO * O)."""
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    Q = np.asarray(Q, dtype=np.float64)
    dO = np.asarray(dO, dtype=np.float64)
    H, P, d = Q.shape
    dK = np.zeros_like(K)
    dV = np.zeros_like(V)
    dQ = np.zeros_like(Q)
    for b, (t0, t1) in enumerate(_user_slices(cu_seqlens)):
        if t1 == t0:
            continue
        for h in range(H):
            Kb, Vb, G = K[t0:t1, h, :], V[t0:t1, h, :], dO[b, h]
            A = proto_softmax(affinity(Q[h], Kb, scale))
            dV[t0:t1, h, :] = A.T @ G
            dA = G @ Vb.T
            dS = A * (dA - (A * dA).sum(axis=0, keepdims=True))
            dK[t0:t1, h, :] = scale * (dS.T @ Q[h])
            dQ[h] += scale * (dS @ Kb)
    return dK, dV, dQ


def sa_forward_per_user(K, V, cu_seqlens, Qu, scale, with_lse=False):
    """Sketch with per-user queries (Sec. 3.3, S^(l) = (X~^(l) W_Q^(l)) (X W_K^(l))^T / sqrt(d)):
    Qu[b, h] ([B, H, P, d]) replaces Q[h] for user b; everything else as ``sa_forward``."""
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    Qu = np.asarray(Qu, dtype=np.float64)
    B, H, P, d = Qu.shape
    sl = _user_slices(cu_seqlens)
    assert len(sl) == B
    O = np.zeros((B, H, P, d))
    lse = np.zeros((K.shape[0], H))
    for b, (t0, t1) in enumerate(sl):
        if t1 == t0:
            continue
        for h in range(H):
            S = affinity(Qu[b, h], K[t0:t1, h, :], scale)
            O[b, h] = proto_softmax(S) @ V[t0:t1, h, :]
            if with_lse:
                m = S.max(axis=0)
                lse[t0:t1, h] = m + np.log(np.exp(S - m).sum(axis=0))
    return (O, lse) if with_lse else O


def sa_backward_per_user(K, V, cu_seqlens, Qu, scale, dO):
    """Gradients (dK [N,H,d], dV [N,H,d], dQu [B,H,P,d]) of L = sum(dO * O) with
    per-user queries: dQu[b, h] = scale * dS K_b holds only user b's tokens."""
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    Qu = np.asarray(Qu, dtype=np.float64)
    dO = np.asarray(dO, dtype=np.float64)
    B, H, P, d = Qu.shape
    dK = np.zeros_like(K)
    dV = np.zeros_like(V)
    dQu = np.zeros_like(Qu)
    for b, (t0, t1) in enumerate(_user_slices(cu_seqlens)):
        if t1 == t0:
            continue
        for h in range(H):
            Kb, Vb, G = K[t0:t1, h, :], V[t0:t1, h, :], dO[b, h]
            A = proto_softmax(affinity(Qu[b, h], Kb, scale))
            dV[t0:t1, h, :] = A.T @ G
            dA = G @ Vb.T
            dS = A * (dA - (A * dA).sum(axis=0, keepdims=True))
            dK[t0:t1, h, :] = scale * (dS.T @ Qu[b, h])
            dQu[b, h] = scale * (dS @ Kb)
    return dK, dV, dQu


def _project_keys(X, Wk):
    """K[:, h, :] = X[:, h, :] @ Wk[h] (Sec. 3.1 / App. G.3, K = X W_K)."""
    return np.einsum("nhc,hce->nhe", X, Wk)


def sa_forward_x(X, cu_seqlens, Q, Wk, scale, with_lse=False):
    """Sketch with keys projected from the history and the history itself as
    values: ``sa_forward(X W_K, X, ...)`` (Sec. 3.1)."""
    X = np.asarray(X, dtype=np.float64)
    Wk = np.asarray(Wk, dtype=np.float64)
    return sa_forward(_project_keys(X, Wk), X, cu_seqlens, Q, scale, with_lse=with_lse)


def sa_backward_x(X, cu_seqlens, Q, Wk, scale, dO):
    """Gradients (dX [N,H,d], dQ [H,P,d], dWk [H,d,d]) of L = sum(dO * O) for
    ``sa_forward_x``: X reaches O twice, as the values and through K = X W_K, so
    dX = dV + dK W_K^T and dW_K[h] = X[:, h]^T dK[:, h]."""
    X = np.asarray(X, dtype=np.float64)
    Wk = np.asarray(Wk, dtype=np.float64)
    dK, dV, dQ = sa_backward(_project_keys(X, Wk), X, cu_seqlens, Q, scale, dO)
    dX = dV + np.einsum("nhe,hce->nhc", dK, Wk)
    dWk = np.einsum("nhc,nhe->hce", X, dK)
    return dX, dQ, dWk


def token_softmax(S):
    """Softmax along axis 1 (the token axis) of a P x L score matrix, max
    subtracted per row (Sec. 5.1 / App. C: weights p(i | j))."""
    m = S.max(axis=1, keepdims=True)
    e = np.exp(S - m)
    return e / e.sum(axis=1, keepdims=True)


def sa_forward_tokenwise(K, V, cu_seqlens, Q, scale, with_lse=False):
    """Sketch O[B, H, P, d] under token-wise normalisation (and, with
    ``with_lse``, the per-prototype log-sum-exp over the user's tokens,
    lse_tok[B, H, P]).  A user with no tokens gets O = 0 and lse_tok = -inf."""
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    Q = np.asarray(Q, dtype=np.float64)
    H, P, d = Q.shape
    sl = _user_slices(cu_seqlens)
    O = np.zeros((len(sl), H, P, d))
    lse = np.full((len(sl), H, P), -np.inf)
    for b, (t0, t1) in enumerate(sl):
        if t1 == t0:
            continue
        for h in range(H):
            S = affinity(Q[h], K[t0:t1, h, :], scale)
            O[b, h] = token_softmax(S) @ V[t0:t1, h, :]
            m = S.max(axis=1)
            lse[b, h] = m + np.log(np.exp(S - m[:, None]).sum(axis=1))
    return (O, lse) if with_lse else O


def sa_backward_tokenwise(K, V, cu_seqlens, Q, scale, dO):
    """Gradients (dK [N,H,d], dV [N,H,d], dQ [H,P,d]) of L = sum(dO * O) for
    ``sa_forward_tokenwise``: dS = A * (dA - rowsum(A * dA)) (softmax Jacobian
    along the token axis); dQ sums over all users (shared prototypes)."""
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    Q = np.asarray(Q, dtype=np.float64)
    dO = np.asarray(dO, dtype=np.float64)
    H, P, d = Q.shape
    dK = np.zeros_like(K)
    dV = np.zeros_like(V)
    dQ = np.zeros_like(Q)
    for b, (t0, t1) in enumerate(_user_slices(cu_seqlens)):
        if t1 == t0:
            continue
        for h in range(H):
            Kb, Vb, G = K[t0:t1, h, :], V[t0:t1, h, :], dO[b, h]
            A = token_softmax(affinity(Q[h], Kb, scale))
            dV[t0:t1, h, :] = A.T @ G
            dA = G @ Vb.T
            dS = A * (dA - (A * dA).sum(axis=1, keepdims=True))
            dK[t0:t1, h, :] = scale * (dS.T @ Q[h])
            dQ[h] += scale * (dS @ Kb)
    return dK, dV, dQ
