"""Pins of the sampling oracle against values fixed outside it: the published
SplitMix64 test vector, the uniform grid, the Gumbel CDF exp(-exp(-x)), and the
Gumbel-max theorem (argmax of z/tau + G is distributed as softmax(z/tau)),
checked statistically with bounds far outside sampling noise."""
import json
import math
import os

import numpy as np

import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def test_splitmix64_published_vector():
    g = json.load(open(os.path.join(GOLDEN, "splitmix64.json")))
    out = oracle.splitmix64_at(g["state"], np.arange(5))
    assert [int(x) for x in out] == g["outputs"]


def test_uniforms_on_the_24_bit_grid_inside_the_unit_interval():
    u = oracle.sample_uniforms(7, 3, 5, 1 << 16)
    assert np.all(u > 0.0) and np.all(u < 1.0)
    k = u * 2 ** 24 - 0.5
    assert np.array_equal(k, np.round(k))
    # rows, steps and tokens index disjoint counters: different (b, j) give different draws
    assert not np.array_equal(u, oracle.sample_uniforms(7, 3, 6, 1 << 16))
    assert not np.array_equal(u, oracle.sample_uniforms(7, 4, 5, 1 << 16))
    # mean and variance of U(0, 1): 1/2 and 1/12 within 6 standard errors
    n = u.size
    assert abs(u.mean() - 0.5) < 6 * math.sqrt(1 / 12 / n)
    assert abs(u.var() - 1 / 12) < 6 * math.sqrt(1 / 180 / n)


def test_gumbel_cdf():
    g = np.sort(oracle.gumbel(oracle.sample_uniforms(11, 0, 0, 200000)))
    emp = np.arange(1, g.size + 1) / g.size
    ks = np.max(np.abs(emp - np.exp(-np.exp(-g))))
    assert ks < 1.63 / math.sqrt(g.size) + 1e-4  # 1 % Kolmogorov-Smirnov critical value


def test_gumbel_max_draws_follow_softmax():
    z = np.array([0.0, 1.0, -1.0, 2.0, 0.5, -3.0, 1.5, 0.2])
    for tau in (1.0, 0.5, 2.0):
        p = np.exp(z / tau - np.max(z / tau))
        p /= p.sum()
        n = 20000
        counts = np.zeros(z.size)
        for i in range(n):
            c, lp, _ = oracle.sample_token(z, tau, 1234, i % 97, i // 97)
            counts[c] += 1
            assert abs(lp - math.log(p[c])) < 1e-12
        # chi-square with 7 degrees of freedom: 0.1 % critical value 24.3
        chi2 = float(np.sum((counts - n * p) ** 2 / (n * p)))
        assert chi2 < 24.3, (tau, chi2)


def test_same_counter_same_token():
    z = np.random.default_rng(0).normal(size=4096)
    a = oracle.sample_token(z, 1.0, 5, 2, 9)
    assert a == oracle.sample_token(z, 1.0, 5, 2, 9)
    # a one-hot logit far above the rest is always drawn
    z2 = np.zeros(100)
    z2[37] = 60.0
    assert all(oracle.sample_token(z2, 1.0, s, 0, 0)[0] == 37 for s in range(20))
