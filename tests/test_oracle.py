"""The fp64 oracle against its pins (no GPU needed)."""
import numpy as np
import pytest

import pins
from oracle import (sa_backward, sa_backward_per_user, sa_backward_tokenwise, sa_backward_x, sa_forward,
                    sa_forward_per_user, sa_forward_tokenwise, sa_forward_x)


@pytest.mark.parametrize("pin", pins.ALL_PINS, ids=lambda p: p.__name__)
def test_oracle_pin(pin):
    if pin.__name__.startswith("pin_bruteforce"):
        pytest.importorskip("mpmath")
    pin(sa_forward, sa_backward)


def test_empty_user_gives_zero_sketch_and_no_nan():
    K = np.random.default_rng(0).standard_normal((3, 1, 4))
    cu = np.array([0, 0, 3, 3])
    Q = np.random.default_rng(1).standard_normal((1, 5, 4))
    O = sa_forward(K, K, cu, Q, 0.5)
    assert np.all(O[0] == 0) and np.all(O[2] == 0) and np.all(np.isfinite(O))
    dK, dV, dQ = sa_backward(K, K, cu, Q, 0.5, np.ones((3, 1, 5, 4)))
    assert np.all(np.isfinite(dK)) and np.all(np.isfinite(dQ))


def test_large_scores_do_not_overflow():
    # scores far above exp's fp64 range still give a valid allocation
    K = np.full((2, 1, 2), 100.0)
    Q = np.array([[[100.0, 100.0], [99.0, 100.0]]])
    O, lse = sa_forward(K, np.ones_like(K), np.array([0, 2]), Q, 1.0, with_lse=True)
    assert np.all(np.isfinite(O)) and np.allclose(O[0, 0].sum() + O[0, 0].sum(), O[0, 0].sum() * 2)
    assert np.allclose(O[0, 0, :, 0].sum(), 2.0)
    assert np.all(np.isfinite(lse))


@pytest.mark.parametrize("pin", pins.UQ_PINS, ids=lambda p: p.__name__)
def test_oracle_per_user_pin(pin):
    pin(sa_forward_per_user, sa_backward_per_user)


@pytest.mark.parametrize("pin", pins.X_PINS, ids=lambda p: p.__name__)
def test_oracle_key_projection_pin(pin):
    pin(sa_forward_x, sa_backward_x)


@pytest.mark.parametrize("pin", pins.TW_PINS, ids=lambda p: p.__name__)
def test_oracle_tokenwise_pin(pin):
    if pin.__name__.endswith("bruteforce"):
        pytest.importorskip("mpmath")
    pin(sa_forward_tokenwise, sa_backward_tokenwise)


def test_dq_is_a_sum_over_pieces_of_a_history():
    """Prototype-wise weights are per token, so a user's dQ is the sum of the dQ
    of any split of its tokens into pieces (the full-batch GPU tests sum the
    oracle's dQ this way)."""
    import harness
    from paper_2609_08443_gb300 import workloads as wl

    spec = wl.custom([37], H=2, P=5, d=8, dtype=wl.BF16, seed=9)
    host = wl.make_host(spec)
    Q = wl.host_as_f64(spec, host["Q"])
    G = host["dsketch"].astype(np.float64)
    K, V = wl.host_as_f64(spec, host["K"]), wl.host_as_f64(spec, host["V"])
    _, _, dq_all = sa_backward(K, V, host["cu_seqlens"], Q, spec.scale, G)
    parts = sum(harness.oracle_dq_chunk((host["K"][s:e], host["V"][s:e], Q, G[0], spec.scale))
                for s, e in ((0, 10), (10, 11), (11, 37)))
    assert np.max(np.abs(parts - dq_all)) <= 1e-12 * np.max(np.abs(dq_all))
