"""Pins of the oracle's primitives against values fixed outside the oracle.

- SplitMix64 finalizer: the published SplitMix64 generator seeded with 0
  returns 0xE220A8397B1DCDAF as its first output (state 0x9E3779B97F4A7C15).
- Philox4x32-10: the known-answer vectors distributed with Random123
  (Salmon et al., SC 2011), read from tests/golden/philox4x32_10_kat.txt.
- exp: accuracy against numpy's float64 exp (<= 1 ulp of float32).
- Worker selection, Eq. (2): argmin with lowest-index ties; the softmax draw
  against Eq. (2) probabilities computed here with numpy; tau limits (§4.3).
- Nearest-rank P99 against numpy's inverted-CDF percentile.
"""
import math
import os

import numpy as np
import pytest

import oracle as O


def test_splitmix64_published_first_output():
    assert O.mix64(0x9E3779B97F4A7C15) == 0xE220A8397B1DCDAF


def test_mix64_is_a_bijection_on_samples():
    rng = np.random.default_rng(1)
    xs = [int(v) for v in rng.integers(0, 2**63, size=20000, dtype=np.int64)]
    ys = {O.mix64(x) for x in xs}
    assert len(ys) == len(set(xs))


def _philox_kat():
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden",
                        "philox4x32_10_kat.txt")
    out = []
    with open(path) as fh:
        for ln in fh:
            if ln.strip() and not ln.startswith("#"):
                v = [int(x, 16) for x in ln.split()]
                out.append((tuple(v[0:4]), tuple(v[4:6]), tuple(v[6:10])))
    return out


@pytest.mark.parametrize("ctr,key,expect", _philox_kat())
def test_philox_known_answers(ctr, key, expect):
    assert O.philox4x32_10(ctr, key) == expect


def test_expf_accuracy_and_range():
    x = np.linspace(-87.0, 0.0, 400001, dtype=np.float32)
    y = O.expf(x).astype(np.float64)
    ref = np.exp(x.astype(np.float64))
    ulp = np.spacing(ref.astype(np.float32)).astype(np.float64)
    assert np.max(np.abs(y - ref) / ulp) <= 1.0
    assert O.expf(np.float32(0.0))[0] == 1.0
    assert O.expf(np.float32(-87.5))[0] == 0.0
    assert O.expf(np.float32(-np.inf))[0] == 0.0
    assert np.all(np.diff(y) >= 0.0)


def test_select_argmin_lowest_index():
    assert O.select([3.0, 1.0, 1.0, 2.0], 0.0) == 1
    assert O.select([5.0], 0.0) == 0
    assert O.select([2.0, 2.0, 2.0], 0.0) == 0
    assert O.select([np.inf, 7.0, np.inf], 0.0) == 1


def test_select_softmax_matches_eq2_probabilities():
    cost = np.array([3.0, 1.0, 2.5, 1.2, 8.0], np.float32)
    tau = 0.9
    # Eq. (2) probabilities, float64 numpy
    p = np.exp(-cost.astype(np.float64) / tau)
    p /= p.sum()
    N = 1 << 16
    u = (np.arange(N, dtype=np.int64) * ((1 << 24) // N)).astype(np.uint32)
    picks = np.array([O.select(cost, tau, int(v)) for v in u])
    freq = np.bincount(picks, minlength=5) / N
    # a regular grid of u reproduces the CDF to within the grid step
    assert np.max(np.abs(np.cumsum(freq) - np.cumsum(p))) < 2.0 / N + 1e-6


def test_select_softmax_philox_chi2():
    cost = np.array([0.0, 0.5, 1.0, 3.0], np.float32)
    tau = 1.0
    p = np.exp(-cost.astype(np.float64) / tau)
    p /= p.sum()
    N = 40000
    draws = [O.philox4x32_10((i, 0, 0, 0x53494D31), (7, 0))[0] >> 8 for i in range(N)]
    picks = np.array([O.select(cost, tau, d) for d in draws])
    obs = np.bincount(picks, minlength=4)
    chi2 = float(np.sum((obs - N * p) ** 2 / (N * p)))
    assert chi2 < 16.27   # chi-square, 3 dof, p = 0.001


def test_select_temperature_limits():
    cost = np.array([4.0, 1.0, 3.0], np.float32)
    # tau -> 0+: the draw concentrates on the argmin
    assert all(O.select(cost, 1e-4, u) == 1 for u in (0, 1 << 23, (1 << 24) - 1))
    # tau -> infinity: uniform
    N = 3000
    u = (np.arange(N) * ((1 << 24) // N)).astype(np.uint32)
    picks = np.array([O.select(cost, 1e9, int(v)) for v in u])
    assert np.allclose(np.bincount(picks, minlength=3) / N, 1 / 3, atol=2e-3)


@pytest.mark.parametrize("n", [1, 2, 50, 99, 100, 101, 200, 1234])
def test_p99_nearest_rank(n):
    v = np.random.default_rng(n).exponential(size=n)
    assert O.p99(v) == np.percentile(v, 99, method="inverted_cdf")
