"""The seeded input generator: determinism, dtype exactness, recipe shape."""
import numpy as np

import grkv_inputs as gi


def test_units_are_reproducible_and_independent():
    wl = gi.workload(1).replace(n=512)
    a = gi.unit_arrays(wl, 3)
    b = gi.unit_arrays(wl, 3)
    c = gi.unit_arrays(wl, 4)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)
    assert not np.array_equal(a[1], c[1])


def test_bf16_values_are_exact_and_rounding_is_nearest_even():
    wl = gi.workload(1).replace(n=256)
    q, k, v = gi.unit_arrays(wl, 0)
    for x in (q, k, v):
        np.testing.assert_array_equal(gi.bf16_value(gi.bf16_bits(x)), x)
    x = np.array([1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5, 0.0], np.float32)
    np.testing.assert_array_equal(gi.bf16_value(gi.bf16_bits(x)), [1.0, 1.0 + 4 * 2 ** -8, -2.5, 0.0])


def test_shapes_and_fill():
    wl = gi.workload(1).replace(n=128, units=3)
    q = np.zeros((3, wl.group, wl.window, wl.d), np.uint16)
    k = np.zeros((3, wl.n, wl.d), np.uint16)
    v = np.zeros_like(k)
    gi.fill_units(wl, q, k, v, threads=2)
    q1, k1, v1 = gi.unit_arrays(wl, 1)
    np.testing.assert_array_equal(gi.bf16_value(k[1]), k1)
    np.testing.assert_array_equal(gi.bf16_value(q[1]), q1)


def test_outlier_recipe_has_four_scaled_channels():
    wl = gi.workload(2).replace(n=2048, units=1)
    _, k, _ = gi.unit_arrays(wl, 0)
    std = k.std(axis=0)
    assert np.sum(std > 5.0) == 4


def test_spans_recipe_aligns_with_the_queries():
    wl = gi.workload(3).replace(n=8192, units=1)
    q, k, _ = gi.unit_arrays(wl, 0)
    t = q.reshape(-1, wl.d).mean(axis=0)
    t /= np.linalg.norm(t)
    cos = (k @ t) / np.linalg.norm(k, axis=1)
    assert np.sum(np.abs(cos - 0.8) < 0.02) >= 16 * 256 * 0.95
