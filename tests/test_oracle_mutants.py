"""Plant plausible mistakes in copies of the oracle; each must fail a pin.

This shows that the pins in ``pins.py`` are strong enough to catch a dropped
term, a wrong sign, a wrong softmax axis, a missing scale or a transposed
operand anywhere in the oracle.
"""
import numpy as np
import pytest

import pins
from oracle import sa_oracle as so


def _fwd_variant(softmax=so.proto_softmax, use_scale=True, agg_from_k=False):
    def fwd(K, V, cu, Q, scale, with_lse=False):
        K = np.asarray(K, float); V = np.asarray(V, float); Q = np.asarray(Q, float)
        H, P, d = Q.shape
        sl = so._user_slices(cu)
        O = np.zeros((len(sl), H, P, d)); lse = np.zeros((K.shape[0], H))
        for b, (t0, t1) in enumerate(sl):
            if t1 == t0:
                continue
            for h in range(H):
                S = (scale if use_scale else 1.0) * (Q[h] @ K[t0:t1, h].T)
                A = softmax(S)
                O[b, h] = A @ (K if agg_from_k else V)[t0:t1, h]
                m = S.max(axis=0)
                lse[t0:t1, h] = m + np.log(np.exp(S - m).sum(axis=0))
        return (O, lse) if with_lse else O
    return fwd


def _bwd_variant(drop_d=False, flip=False, dk_scale=True, dq_overwrite=False, dv_transpose=False):
    def bwd(K, V, cu, Q, scale, dO):
        K = np.asarray(K, float); V = np.asarray(V, float); Q = np.asarray(Q, float)
        H, P, d = Q.shape
        dK = np.zeros_like(K); dV = np.zeros_like(V); dQ = np.zeros_like(Q)
        for b, (t0, t1) in enumerate(so._user_slices(cu)):
            if t1 == t0:
                continue
            for h in range(H):
                Kb, Vb, G = K[t0:t1, h], V[t0:t1, h], dO[b, h]
                A = so.proto_softmax(scale * (Q[h] @ Kb.T))
                dV[t0:t1, h] = (A.T @ G) if not dv_transpose else (A.T @ G[::-1])
                dA = G @ Vb.T
                Dv = 0.0 if drop_d else (A * dA).sum(axis=0, keepdims=True)
                dS = A * ((Dv - dA) if flip else (dA - Dv))
                dK[t0:t1, h] = (scale if dk_scale else 1.0) * (dS.T @ Q[h])
                if dq_overwrite:
                    dQ[h] = scale * (dS @ Kb)
                else:
                    dQ[h] += scale * (dS @ Kb)
        return dK, dV, dQ
    return bwd


def _token_softmax(S):
    e = np.exp(S - S.max(axis=1, keepdims=True))
    return e / e.sum(axis=1, keepdims=True)


def _no_shift_sum_softmax(S):  # forgets to normalise
    return np.exp(S - S.max(axis=0, keepdims=True))


MUTANTS = {
    "softmax over tokens": (_fwd_variant(softmax=_token_softmax), so.sa_backward),
    "unnormalised weights": (_fwd_variant(softmax=_no_shift_sum_softmax), so.sa_backward),
    "scale dropped in S": (_fwd_variant(use_scale=False), so.sa_backward),
    "aggregates K not V": (_fwd_variant(agg_from_k=True), so.sa_backward),
    "dS without the D term": (so.sa_forward, _bwd_variant(drop_d=True)),
    "dS sign flipped": (so.sa_forward, _bwd_variant(flip=True)),
    "dK without scale": (so.sa_forward, _bwd_variant(dk_scale=False)),
    "dQ not summed over users": (so.sa_forward, _bwd_variant(dq_overwrite=True)),
    "dV with prototypes reversed": (so.sa_forward, _bwd_variant(dv_transpose=True)),
}

CHEAP_PINS = [p for p in pins.ALL_PINS if p is not pins.pin_bruteforce_gradients]


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name):
    fwd, bwd = MUTANTS[name]
    caught = []
    for pin in CHEAP_PINS:
        if pin.__name__.startswith("pin_bruteforce"):
            pytest.importorskip("mpmath")
        try:
            pin(fwd, bwd)
        except AssertionError:
            caught.append(pin.__name__)
    assert caught, f"no pin catches the planted mistake '{name}'"


# ------------------------------------------- per-user queries (Sec. 3.3)
def _uq_variant(first_user_q=False, dq_summed=False, dq_scale=True):
    def fwd(K, V, cu, Qu, scale, with_lse=False):
        Qx = np.broadcast_to(Qu[:1], Qu.shape) if first_user_q else Qu
        return so.sa_forward_per_user(K, V, cu, np.array(Qx), scale, with_lse=with_lse)

    def bwd(K, V, cu, Qu, scale, dO):
        Qx = np.array(np.broadcast_to(Qu[:1], Qu.shape)) if first_user_q else Qu
        dK, dV, dQ = so.sa_backward_per_user(K, V, cu, Qx, scale, dO)
        if dq_summed:
            dQ = np.broadcast_to(dQ.sum(axis=0, keepdims=True), dQ.shape).copy()
        if not dq_scale:
            dQ = dQ / scale
        return dK, dV, dQ
    return fwd, bwd


UQ_MUTANTS = {
    "every user gets user 0's prototypes": _uq_variant(first_user_q=True),
    "dQ summed over users": _uq_variant(dq_summed=True),
    "dQ without scale": _uq_variant(dq_scale=False),
}


@pytest.mark.parametrize("name", sorted(UQ_MUTANTS))
def test_per_user_mutant_is_caught(name):
    fwd, bwd = UQ_MUTANTS[name]
    caught = []
    for pin in pins.UQ_PINS:
        try:
            pin(fwd, bwd)
        except AssertionError:
            caught.append(pin.__name__)
    assert caught, f"no pin catches the planted mistake '{name}'"


# --------------------------------- key projection in the step (Sec. 3.1)
def _x_variant(transpose_wk=False, drop_value_path=False, dwk_transposed=False):
    def fwd(X, cu, Q, Wk, scale, with_lse=False):
        W = np.swapaxes(Wk, 1, 2) if transpose_wk else Wk
        return so.sa_forward_x(X, cu, Q, W, scale, with_lse=with_lse)

    def bwd(X, cu, Q, Wk, scale, dO):
        W = np.swapaxes(Wk, 1, 2) if transpose_wk else Wk
        dX, dQ, dW = so.sa_backward_x(X, cu, Q, W, scale, dO)
        if drop_value_path:
            dK, dV, _ = so.sa_backward(so._project_keys(np.asarray(X, float), np.asarray(W, float)),
                                       np.asarray(X, float), cu, Q, scale, dO)
            dX = dX - dV
        if dwk_transposed:
            dW = np.swapaxes(dW, 1, 2)
        return dX, dQ, dW
    return fwd, bwd


X_MUTANTS = {
    "keys projected with W_K^T": _x_variant(transpose_wk=True),
    "dX without the value path": _x_variant(drop_value_path=True),
    "dW_K transposed": _x_variant(dwk_transposed=True),
}


@pytest.mark.parametrize("name", sorted(X_MUTANTS))
def test_key_projection_mutant_is_caught(name):
    fwd, bwd = X_MUTANTS[name]
    caught = []
    for pin in pins.X_PINS:
        try:
            pin(fwd, bwd)
        except AssertionError:
            caught.append(pin.__name__)
    assert caught, f"no pin catches the planted mistake '{name}'"


# ------------------------- token-wise ("vanilla") normalisation (Sec. 5.1)
def _tw_lse_variant(lse_axis=1, keep_max=True):
    """lse_tok computed with the reduction over the wrong axis (axis 0, the
    prototypes) or with the subtracted maximum not added back."""
    def lse_tok(S):
        m = S.max(axis=lse_axis, keepdims=True)
        r = np.log(np.exp(S - m).sum(axis=lse_axis, keepdims=True)) + (m if keep_max else 0.0)
        return np.broadcast_to(r, S.shape)[:, 0]
    return lse_tok


def _tw_variant(proto_axis=False, drop_d=False, dv_from_g_t=False, lse_fn=None):
    def fwd(K, V, cu, Q, scale, with_lse=False):
        if proto_axis:
            return so.sa_forward(K, V, cu, Q, scale, with_lse=with_lse)
        if lse_fn is None or not with_lse:
            return so.sa_forward_tokenwise(K, V, cu, Q, scale, with_lse=with_lse)
        O = so.sa_forward_tokenwise(K, V, cu, Q, scale)
        Qd = np.asarray(Q, float)
        lse = np.full(O.shape[:3], -np.inf)
        for b, (t0, t1) in enumerate(so._user_slices(cu)):
            if t1 == t0:
                continue
            for h in range(Qd.shape[0]):
                lse[b, h] = lse_fn(scale * (Qd[h] @ np.asarray(K, float)[t0:t1, h].T))
        return O, lse

    def bwd(K, V, cu, Q, scale, dO):
        K = np.asarray(K, float); V = np.asarray(V, float); Q = np.asarray(Q, float); dO = np.asarray(dO, float)
        H, P, d = Q.shape
        dK = np.zeros_like(K); dV = np.zeros_like(V); dQ = np.zeros_like(Q)
        for b, (t0, t1) in enumerate(so._user_slices(cu)):
            if t1 == t0:
                continue
            for h in range(H):
                Kb, Vb, G = K[t0:t1, h], V[t0:t1, h], dO[b, h]
                A = so.token_softmax(scale * (Q[h] @ Kb.T))
                dV[t0:t1, h] = (A.T @ G) if not dv_from_g_t else (A.T @ G[::-1])
                dA = G @ Vb.T
                Dv = 0.0 if drop_d else (A * dA).sum(axis=1, keepdims=True)
                dS = A * (dA - Dv)
                dK[t0:t1, h] = scale * (dS.T @ Q[h])
                dQ[h] += scale * (dS @ Kb)
        return dK, dV, dQ
    return fwd, bwd


TW_MUTANTS = {
    "normalised over prototypes": _tw_variant(proto_axis=True),
    "dS without the row term": _tw_variant(drop_d=True),
    "dV with prototypes reversed": _tw_variant(dv_from_g_t=True),
    "lse_tok reduced over the prototypes": _tw_variant(lse_fn=_tw_lse_variant(lse_axis=0)),
    "lse_tok without its maximum": _tw_variant(lse_fn=_tw_lse_variant(keep_max=False)),
}


@pytest.mark.parametrize("name", sorted(TW_MUTANTS))
def test_tokenwise_mutant_is_caught(name):
    fwd, bwd = TW_MUTANTS[name]
    caught = []
    for pin in pins.TW_PINS:
        if pin.__name__.endswith("bruteforce"):
            pytest.importorskip("mpmath")
        try:
            pin(fwd, bwd)
        except AssertionError:
            caught.append(pin.__name__)
    assert caught, f"no pin catches the planted mistake '{name}'"
