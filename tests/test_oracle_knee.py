"""Pins of the saturation-knee detector in the oracle (§5.1, the PoA-growth
proposition, item 3; Experiment 2's difference quotients over a concurrency
sweep), each against something other than the oracle's own formula: numpy's
inverted-CDF percentile, exact divided differences of quadratics, the closed
second derivative of the Eq. (9) latency curve and its threshold crossing,
and the degenerate sweeps."""
import math

import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import workloads as wk

GRID = np.array([1, 4, 8, 16, 32, 64, 128, 256, 512], np.float64)   # Experiment 2's levels


def _one_row_per_replica(y):
    n = len(y)
    return (np.zeros(n, np.int32), np.asarray(y, np.float64), np.arange(n + 1, dtype=np.int64))


@pytest.mark.parametrize("pct", [1, 37, 50, 90, 99, 100])
def test_percentile_is_numpy_inverted_cdf(pct):
    rng = np.random.default_rng(pct)
    sizes = [1, 2, 7, 100, 101, 999, 2500]
    rows = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int64)
    n = int(rows[-1])
    ttft = np.round(rng.lognormal(-2.0, 0.8, n), 3)           # rounding makes ties
    worker = rng.integers(-1, 3, n).astype(np.int32)            # about a quarter unrouted
    worker[rows[:-1]] = 0                                       # every replica routes one
    out = O.sweep_knee(worker, ttft, rows, np.arange(len(sizes), dtype=np.float64),
                       [0, len(sizes)], pct=pct)
    for r in range(len(sizes)):
        v = ttft[rows[r]:rows[r + 1]][worker[rows[r]:rows[r + 1]] >= 0]
        assert out["stat"][r] == np.percentile(v, pct, method="inverted_cdf")


def test_empty_replica_and_rejected_percentiles():
    out = O.sweep_knee([-1, -1, 0], [0.1, 0.2, 0.3], [0, 0, 2, 3], [1.0, 2.0, 3.0], [0, 3])
    assert math.isnan(out["stat"][0]) and math.isnan(out["stat"][1])
    assert out["stat"][2] == 0.3
    for bad in (0, 101):
        with pytest.raises(ValueError):
            O.sweep_knee([0], [0.1], [0, 1], [1.0], [0, 1], pct=bad)


def test_quadratic_divided_differences_are_exact():
    # y = p x^2 + q x + r: d1 on [x_k, x_k+1] is p (x_k + x_k+1) + q and the
    # three-point second difference is 2p on any grid, here the paper's
    p, q, r = 0.5, 3.0, 1.0
    y = p * GRID ** 2 + q * GRID + r
    out = O.sweep_knee(*_one_row_per_replica(y), GRID, [0, GRID.size], theta=0.99)
    assert np.array_equal(out["d1"][:-1], p * (GRID[:-1] + GRID[1:]) + q)
    assert np.array_equal(out["d2"][1:-1], np.full(GRID.size - 2, 2 * p))
    assert math.isnan(out["d1"][-1]) and math.isnan(out["d2"][0]) and math.isnan(out["d2"][-1])
    assert out["knee_index"][0] == 1 and out["knee_load"][0] == GRID[1]
    flat = O.sweep_knee(*_one_row_per_replica(q * GRID + r), GRID, [0, GRID.size], theta=0.0)
    assert np.all(flat["d2"][1:-1] == 0.0) and flat["knee_index"][0] == -1


def test_eq9_curve_second_derivative_and_knee():
    # f(n) = a n + b + d / (n_sat - n)^beta has f'' = beta (beta + 1) d / (n_sat - n)^(beta + 2);
    # the central difference on a uniform grid is within O(h^2), and the first
    # grid point above theta lies within one step of the closed-form crossing
    a, b, d, beta, nsat = 0.005, 0.020, 0.010, 2.0, 64.0
    h = 0.05
    x = np.arange(1.0, 60.0, h)
    y = a * x + b + d / (nsat - x) ** beta
    theta = 1e-4                       # crossing near n = 59.05
    out = O.sweep_knee(*_one_row_per_replica(y), x, [0, x.size], theta=theta)
    exact = beta * (beta + 1) * d / (nsat - x[1:-1]) ** (beta + 2)
    rel = np.abs(out["d2"][1:-1] - exact) / exact
    assert rel.max() < 1e-3
    nstar = nsat - (beta * (beta + 1) * d / theta) ** (1.0 / (beta + 2))
    k = out["knee_index"][0]
    assert k > 0 and abs(x[k] - nstar) <= h


def test_degenerate_sweeps():
    y = [0.1, 0.2, 0.5, 0.9, 1.7, 3.0]
    worker, ttft, rows = _one_row_per_replica(y)
    load = np.array([1.0, 2.0, 4.0, 8.0, 8.0, 9.0])
    # sweeps: empty, one point, two points, a non-increasing pair, one replica outside
    out = O.sweep_knee(worker, ttft, rows, load, [0, 0, 1, 3, 5], theta=-1.0)
    assert list(out["knee_index"]) == [-1, -1, -1, -2]
    assert math.isnan(out["knee_load"][3])
    assert out["d1"][1] == (0.5 - 0.2) / 2.0 and math.isnan(out["d1"][2])
    assert np.all(np.isnan(out["d2"]))
    assert np.all(np.isnan(out["d1"][[0, 3, 4, 5]]))


def test_sweep_grouping_of_the_plans():
    p = wk.plan("sat")
    s = wk.sweeps(p.replicas)
    assert s == list(range(0, 55, 9))
    for a, b in zip(s[:-1], s[1:]):
        assert [r.C for r in p.replicas[a:b]] == list(GRID.astype(int))
    assert wk.sweeps(wk.plan("p2d").replicas)[-2:] == [60, 64]
    assert wk.sweeps([]) == [0]
