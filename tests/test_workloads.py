"""Seeded input generator: determinism, shapes and the length recipes."""
import math

import numpy as np

from paper_2609_08443_gb300 import workloads as wl


def test_lengths_follow_the_recipes():
    assert list(wl.lengths(wl.config(1))) == [4096]
    l2 = wl.lengths(wl.config(2))
    assert l2.size == 32 and l2.min() >= 1024 and l2.max() <= 16384
    l3 = wl.lengths(wl.config(3))
    assert l3.size == 64 and l3.min() >= 512 and l3.max() <= 100000
    assert 5000 < np.median(l3) < 80000
    assert list(wl.lengths(wl.config(4))) == [100000] * 128
    l5 = wl.lengths(wl.config(5))
    assert l5.size == 4100 and (l5 == 1048576).sum() == 4
    assert l5[l5 < 1048576].max() <= 512 and l5.min() >= 1
    assert np.nonzero(l5 == 1048576)[0].tolist() != [0, 1, 2, 3]  # permuted


def test_host_draws_are_reproducible_and_per_user():
    spec = wl.custom([5, 0, 9], H=2, P=8, d=16, seed=3)
    a = wl.make_host(spec)
    b = wl.make_host(spec)
    for k in ("K", "V", "Q", "dsketch", "cu_seqlens"):
        assert np.array_equal(a[k], b[k])
    sub = wl.make_host(spec, users=[2])
    assert np.array_equal(sub["K"], a["K"][5:14])
    assert np.array_equal(sub["dsketch"][0], a["dsketch"][2])
    assert list(a["cu_seqlens"]) == [0, 5, 5, 14]


def test_bf16_rounding_is_nearest_even():
    x = np.array([1.0, 1.0 + 2**-8, 1.0 + 3 * 2**-8, -2.5, 3.0e-3], dtype=np.float32)
    bits = wl.f32_to_bf16_bits(x)
    back = wl.bf16_bits_to_f64(bits)
    assert back[0] == 1.0
    assert back[1] == 1.0                      # tie -> even
    assert back[2] == 1.0 + 4 * 2**-8          # tie -> even (up)
    assert back[3] == -2.5
    assert abs(back[4] - 3.0e-3) <= 3.0e-3 * 2**-8


def test_scale_is_inverse_sqrt_d():
    assert math.isclose(wl.config(4).scale, 1 / math.sqrt(128))
    assert wl.config(4).q_std == 0.02
