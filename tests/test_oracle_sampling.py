"""Pins of the oracle's counter-based generator and temperature sampling."""
import math

import numpy as np
import pytest

from oracle import cospec_oracle as O
from oracle import philox as P


@pytest.mark.parametrize("ctr,key,expect", [
    ((0, 0, 0, 0), (0, 0), (0x6627E8D5, 0xE169C58D, 0xBC57AC4C, 0x9B00DBD8)),
    ((0xFFFFFFFF,) * 4, (0xFFFFFFFF, 0xFFFFFFFF), (0x408F276D, 0x41C83B0E, 0xA20BC7C6, 0x6D5451FD)),
    ((0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344), (0xA4093822, 0x299F31D0),
     (0xD16CFE09, 0x94FDCCEB, 0x5001E420, 0x24126EA1)),
])
def test_philox_known_answers(ctr, key, expect):
    # known-answer vectors published with the generator (Random123 distribution)
    out = P.philox4x32_10(*[np.array([c]) for c in ctr], *key)
    assert tuple(int(o[0]) for o in out) == expect


def test_uniform23_is_open_interval_and_exact():
    u = P.uniform23(np.array([0, 511, 512, 0xFFFFFFFF], dtype=np.uint64))
    assert u[0] == 0.5 / 2 ** 23 and u[1] == u[0] and u[2] == 1.5 / 2 ** 23
    assert u[3] == (2 ** 23 - 0.5) / 2 ** 23 < 1.0
    assert np.all(np.float32(u).astype(np.float64) == u) and np.float32(u[3]) < 1.0


def test_gumbel_noise_statistics():
    g = P.gumbel_noise(1234, 8, 50000)
    # standard Gumbel: mean = Euler-Mascheroni constant, variance = pi^2 / 6
    assert abs(g.mean() - 0.5772156649) < 0.01
    assert abs(g.var() - math.pi ** 2 / 6) < 0.03


def test_gumbel_max_samples_the_softmax():
    # argmax(x + g) over many independent rows follows softmax(x)
    x = np.log(np.array([0.5, 0.3, 0.15, 0.05]))
    rows = 40000
    g = P.gumbel_noise(99, rows, 4)
    counts = np.bincount(np.argmax(x[None, :] + g, axis=1), minlength=4) / rows
    np.testing.assert_allclose(counts, [0.5, 0.3, 0.15, 0.05], atol=0.01)


def test_sampling_row_stats_match_argmax_at_zero_noise_scale():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((5, 300)) * 3
    s1, st1 = O.row_stats_sampled(x, np.full(5, -1), seed=7, temperature=1.0)
    am, st0 = O.row_stats(x, np.full(5, -1))
    # the statistics of the logits do not depend on the sampling
    np.testing.assert_array_equal(np.nan_to_num(st1), np.nan_to_num(st0))
    g = P.gumbel_noise(7, 5, 300)
    np.testing.assert_array_equal(s1, np.argmax(x + g, axis=1))
    # at a tiny temperature the sample is the argmax
    s2, _ = O.row_stats_sampled(x, np.full(5, -1), seed=7, temperature=1e-6)
    np.testing.assert_array_equal(s2, am)
