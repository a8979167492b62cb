"""Pins of the static counterfactual policies and the static PoA (the
routing-baselines discussion, §9) in the oracle, each against something other
than the oracle's own formula: closed forms, a special case that reduces to
the Eq. (1) argmin, distribution tests, and a feasibility bound."""
import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import workloads as wk


def _trace(n=1500, seed=3):
    spec = wk.TraceSpec(n_req=n, n_groups=12, prefix_min=64, prefix_max=320, len_median=384,
                        len_max=2048, out_median=64, out_max=512)
    return wk.make_trace(spec, seed)


def test_round_robin_is_i_mod_W():
    tr = _trace()
    for W in (2, 3, 5):
        r = O.simulate(O.OracleConfig(W=W, K=4096), tr, 24, policy=O.POLICY_ROUNDROBIN,
                       omega=1.0, seed=9)
        assert r["status"] == 0
        assert np.array_equal(r["worker"], np.arange(tr.n_req) % W)


def test_random_is_uniform_and_ignores_costs():
    tr = _trace(n=6000, seed=4)
    W = 4
    cfg = O.OracleConfig(W=W, K=4096)
    a = O.simulate(cfg, tr, 32, policy=O.POLICY_RANDOM, omega=1.0, seed=21)
    b = O.simulate(cfg, tr, 8, policy=O.POLICY_RANDOM, omega=0.0, seed=21)
    assert a["status"] == b["status"] == 0
    # the draw depends on the request and the seed only
    assert np.array_equal(a["worker"], b["worker"])
    obs = np.bincount(a["worker"], minlength=W)
    exp = tr.n_req / W
    chi2 = float(np.sum((obs - exp) ** 2 / exp))
    assert chi2 < 16.27   # chi-square, 3 dof, p = 0.001
    c = O.simulate(cfg, tr, 32, policy=O.POLICY_RANDOM, omega=1.0, seed=22)
    assert not np.array_equal(a["worker"], c["worker"])


def test_p2c_with_two_workers_is_the_argmin():
    # with W = 2 both workers are always sampled: the lower Eq. (1) cost wins,
    # ties to the lower index -- the tau = 0 choice of Eq. (2)
    tr = _trace(seed=5)
    cfg = O.OracleConfig(W=2, K=4096)
    for om in (0.0, 1.0):
        p = O.simulate(cfg, tr, 48, policy=O.POLICY_P2C, omega=om, seed=3)
        d = O.simulate(cfg, tr, 48, policy=O.POLICY_DYNAMO, omega=om, tau=0.0, seed=3)
        assert p["status"] == d["status"] == 0
        assert np.array_equal(p["worker"], d["worker"])


def test_p2c_takes_the_better_of_two():
    tr = _trace(n=4000, seed=6)
    W = 5
    r = O.simulate(O.OracleConfig(W=W, K=4096), tr, 64, policy=O.POLICY_P2C, omega=0.0,
                   seed=8)
    assert r["status"] == 0
    cost = r["cost"]
    ch = cost[np.arange(tr.n_req), r["worker"]]
    ranks = (cost < ch[:, None]).sum(axis=1)    # workers strictly cheaper than the choice
    # never the strictly most expensive worker, and the cheapest of two uniform
    # distinct samples: rank r (0-based, distinct costs) with probability
    # 2 (W - 1 - r) / (W (W - 1))
    distinct = np.array([len(set(row)) == W for row in cost])
    assert distinct.sum() > 1000
    rk = ranks[distinct]
    assert rk.max() <= W - 2
    obs = np.bincount(rk, minlength=W - 1)[:W - 1]
    p = np.array([2.0 * (W - 1 - q) / (W * (W - 1)) for q in range(W - 1)])
    exp = p * rk.size
    chi2 = float(np.sum((obs - exp) ** 2 / exp))
    assert chi2 < 16.27   # 3 dof, p = 0.001


def test_static_poa_equals_observed_without_queueing():
    # with no worker ever holding cap - 1 requests, TTFT_i is exactly the
    # frozen cost of its worker, so the two estimates coincide
    tr = _trace(seed=7)
    cfg = O.OracleConfig(W=3, K=4096)
    for pol in (O.POLICY_DYNAMO, O.POLICY_ROUNDROBIN, O.POLICY_RANDOM, O.POLICY_P2C):
        r = O.simulate(cfg, tr, 16, policy=pol, omega=1.0, seed=2)
        assert r["status"] == 0
        tot = O.poa(cfg, r)[3]
        st = O.poa_static(cfg, r)
        assert abs(st - tot) <= 1e-9 * tot


def test_static_poa_of_round_robin_is_at_least_one():
    # round robin puts at most ceil(m / W) requests of a window on a worker,
    # within the OPT capacity: the realized assignment is feasible for OPT
    tr = _trace(n=3000, seed=8)
    cfg = O.OracleConfig(W=3, K=4096)
    r = O.simulate(cfg, tr, 256, policy=O.POLICY_ROUNDROBIN, omega=1.0, seed=1)
    assert r["status"] == 0
    numer = O.static_numer(cfg, r)
    _, opt, cnt, _ = O.poa(cfg, r)
    assert np.all(numer >= opt - 1e-12 * np.maximum(opt, 1.0))
    assert O.poa_static(cfg, r) >= 1.0 - 1e-12


def test_static_numer_by_hand():
    # two requests in window 0 on workers 1 and 0, one in window 1 on worker 0
    cfg = O.OracleConfig(W=2, K=16)
    rec = {"worker": np.array([1, 0, 0], np.int32),
           "completion": np.array([1.0, 2.0, 6.0]),
           "ttft": np.array([0.1, 0.1, 0.1]),
           "nbt": np.array([4, 2, 8], np.int32),
           "n_frozen": np.array([[1, 2], [3, 1], [1, 1]], np.uint16),
           "prefix": np.array([[0, 4], [1, 0], [8, 0]], np.uint16)}

    def f(n, m, nbt):   # the §6.4 frozen cost, written out
        return 0.005 * n + 0.020 + 0.010 / ((64 - n) * (64 - n)) - 0.015 * (m / nbt)

    st = O.static_numer(cfg, rec)
    assert st.size == 2
    assert st[0] == pytest.approx(f(2, 4, 4) + f(3, 1, 2), rel=1e-14)
    assert st[1] == pytest.approx(f(1, 8, 8), rel=1e-14)
