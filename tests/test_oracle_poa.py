"""Pins of the PoA side of the oracle.

- OPT of Eq. (12): Hungarian on the replicated-column matrix (§6.4), min-cost
  flow and brute-force enumeration agree, and match scipy's independent
  linear_sum_assignment on the replicated matrix.
- Hand-computed windows: the frozen cost c_ij = a n + b + d/(C - n)^2 - w_c o
  at chosen points, with and without binding column capacity.
- A run without queueing has PoA-hat >= 1 in every window where the observed
  assignment fits the replicated columns (observed TTFT equals its frozen cost).
- The exhaustive one-shot game (Def. 3, 5, 7): PoA >= 1; omega = 0 with affine
  latency is a congestion game (Def. 6): pure equilibria exist, best-response
  dynamics converge, worst-NE PoA <= 5/2 (§4.3), equilibrium loads on identical
  workers differ by at most one (§5.1, proof of Prop. 4).
"""
import itertools

import numpy as np
import pytest
from scipy.optimize import linear_sum_assignment

import oracle as O
from paper_2606_17081_gb300 import workloads as Wk

F1 = 0.005 * 1 + 0.020 + 0.010 / 63 ** 2      # 0.02500251952632905
F2 = 0.005 * 2 + 0.020 + 0.010 / 62 ** 2      # 0.030002601456815817


@pytest.mark.parametrize("seed", range(12))
def test_assignment_methods_agree_small(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, 8))
    W = int(rng.integers(1, 4))
    capw = int(rng.integers(-(-n // W), n + 1))
    c = rng.uniform(0.01, 1.0, size=(n, W))
    vb, ab = O.assign(c, capw, 3)
    vh, ah = O.assign(c, capw, 1)
    vm, am = O.assign(c, capw, 2)
    assert abs(vb - vh) < 1e-12 and abs(vb - vm) < 1e-12
    for a in (ah, am):
        assert np.all(np.bincount(a, minlength=W) <= capw)
        assert abs(c[np.arange(n), a].sum() - vb) < 1e-12


@pytest.mark.parametrize("n,W,capw", [(40, 3, 14), (120, 6, 20), (200, 3, 70), (90, 2, 64)])
def test_assignment_matches_scipy_on_replicated_matrix(n, W, capw):
    rng = np.random.default_rng(n + W)
    c = rng.uniform(0.02, 0.4, size=(n, W))
    big = np.repeat(c, capw, axis=1)
    r, col = linear_sum_assignment(big)
    ref = big[r, col].sum()
    vh, _ = O.assign(c, capw, 1)
    vm, _ = O.assign(c, capw, 2)
    assert abs(vh - ref) <= 1e-10 * ref and abs(vm - ref) <= 1e-10 * ref


def _records(worker, completion, ttft, nbt, nfz, pre):
    return {"worker": np.asarray(worker, np.int32), "completion": np.asarray(completion, float),
            "ttft": np.asarray(ttft, float), "nbt": np.asarray(nbt, np.int32),
            "n_frozen": np.asarray(nfz, np.uint16), "prefix": np.asarray(pre, np.uint16)}


def test_poa_hand_window():
    # two requests in window 0; frozen loads (1, 63) on both rows, no overlap:
    # OPT sends both to worker 0 (capacity 64 >= 2): 2 f(1).
    rec = _records([1, 0], [1.0, 2.0], [1.0, 2.0], [4, 4], [[1, 63], [1, 63]], [[0, 0], [0, 0]])
    cfg = O.OracleConfig(W=2)
    num, opt, cnt, tot = O.poa(cfg, rec)
    assert cnt.tolist() == [2] and num.tolist() == [3.0]
    assert abs(opt[0] - 2 * F1) < 1e-15
    assert abs(tot - 3.0 / (2 * F1)) < 1e-10


def test_poa_hand_overlap_and_windows():
    # request 0 (window 0): overlap 3/4 on worker 1 -> cost f(1) - 0.015*0.75
    # request 1 (window 2, completion 10.5): only worker 0 at load 2
    rec = _records([0, 0], [4.9, 10.5], [0.5, 0.25], [4, 2], [[1, 1], [2, 63]],
                   [[0, 3], [1, 0]])
    num, opt, cnt, tot = O.poa(O.OracleConfig(W=2), rec)
    assert cnt.tolist() == [1, 0, 1]
    assert abs(opt[0] - (F1 - 0.015 * 0.75)) < 1e-15
    assert abs(opt[2] - (F2 - 0.015 * 0.5)) < 1e-15
    assert abs(tot - 0.75 / (opt[0] + opt[2])) < 1e-12


def test_poa_binding_capacity():
    # 130 requests in one window, every row prefers worker 0 (load 1) over
    # worker 1 (load 2); column capacity max(64, ceil(130/2)) = 65 binds.
    n = 130
    rec = _records(np.zeros(n), np.full(n, 0.5), np.full(n, 0.1), np.full(n, 3),
                   np.tile([1, 2], (n, 1)), np.zeros((n, 2)))
    for method in (1, 2):
        num, opt, cnt, tot = O.poa(O.OracleConfig(W=2), rec, method=method)
        assert abs(opt[0] - (65 * F1 + 65 * F2)) < 1e-12


def test_poa_at_least_one_without_queueing():
    spec = Wk.TraceSpec(n_req=1500, len_kind="uniform", len_min=16, len_max=600, n_groups=6,
                        prefix_min=64, prefix_max=256, zipf_s=1.1, rate=40.0,
                        out_kind="uniform", out_min=1, out_max=200)
    tr = Wk.make_trace(spec, 4)
    for policy, om in ((O.POLICY_DYNAMO, 1.0), (O.POLICY_LOADBAL, 0.0)):
        cfg = O.OracleConfig(W=3, K=1024)
        r = O.simulate(cfg, tr, 12, policy=policy, omega=om)
        assert np.all(r["start"] == r["arrival"])      # no queueing at C = 12
        num, opt, cnt, tot = O.poa(cfg, r)
        w = np.floor(r["completion"] / 5.0).astype(int)
        for k in np.nonzero(cnt)[0]:
            per = np.bincount(r["worker"][w == k], minlength=3)
            if per.max() <= max(64, -(-cnt[k] // 3)):
                assert num[k] / opt[k] >= 1 - 1e-12
            assert abs(num[k] - r["ttft"][w == k].sum()) <= 1e-12 * num[k]
        assert abs(tot - num.sum() / opt.sum()) < 1e-12


def _rand_game(rng, n, W):
    return rng.uniform(0.0, 1.0, size=(n, W))


@pytest.mark.parametrize("seed", range(40))
def test_game_affine_congestion_properties(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(2, 8))
    W = int(rng.integers(2, 4))
    a = float(rng.uniform(0.001, 0.02))
    b = float(rng.uniform(0.0, 0.05))
    g = O.game_exhaustive(_rand_game(rng, n, W), 0.0, lat_a=a, lat_b=b, lat_d=0.0)
    assert g["n_ne"] >= 1
    assert g["worst_ne"] >= g["opt"] - 1e-12
    assert g["worst_ne"] / g["opt"] <= 2.5 + 1e-12
    assert g["br_steps"] >= 0
    assert g["max_ne_spread"] <= 1
    # the sequential greedy pass is itself an equilibrium here
    assert g["greedy"] <= g["worst_ne"] + 1e-12 and g["greedy"] >= g["best_ne"] - 1e-12


@pytest.mark.parametrize("seed", range(20))
def test_game_with_overlap_and_pole(seed):
    rng = np.random.default_rng(100 + seed)
    n = int(rng.integers(2, 7))
    W = int(rng.integers(2, 4))
    g = O.game_exhaustive(_rand_game(rng, n, W), float(rng.uniform(0, 0.015)))
    assert g["opt"] > 0
    if g["n_ne"] > 0:
        assert g["worst_ne"] / g["opt"] >= 1 - 1e-12
    assert g["greedy"] >= g["opt"] - 1e-12


def test_game_brute_force_small_by_hand():
    # two requests, two workers, f(n) = n (a = 1, b = 0, d = 0), omega = 0:
    # profiles (0,0),(1,1) cost 4; split profiles cost 2 -> OPT = 2, both
    # split profiles are the only equilibria, PoA = 1.
    g = O.game_exhaustive(np.zeros((2, 2)), 0.0, lat_a=1.0, lat_b=0.0, lat_d=0.0)
    assert g["opt"] == 2.0 and g["worst_ne"] == 2.0 and g["n_ne"] == 2
    # Pigou-like instance with overlap: request 0 gains 1.5 on worker 0
    o = np.array([[1.0, 0.0], [1.0, 0.0]])
    g = O.game_exhaustive(o, 1.5, lat_a=1.0, lat_b=0.0, lat_d=0.0)
    # (0,0): 2*2 - 3 = 1 ; (0,1) and (1,0): 1 + 1 - 1.5 = 0.5 ; (1,1): 4
    assert g["opt"] == 0.5
    # (0,0): moving costs 1 vs staying 2 - 1.5 = 0.5 -> NE; split profiles: the
    # worker-1 player moving to 0 pays 2 - 1.5 = 0.5 < 1 -> not NE.
    assert g["n_ne"] == 1 and g["worst_ne"] == 1.0


@pytest.mark.parametrize("seed", range(6))
def test_assignment_with_heavy_ties(seed):
    # frozen-cost matrices repeat the same few rows many times (equal loads,
    # no overlap): every method must still return the same optimum
    rng = np.random.default_rng(seed)
    n, W = int(rng.integers(60, 140)), 3
    loads = rng.integers(1, 6, size=(n, W))
    c = 0.005 * loads + 0.020 + 0.010 / (64 - loads) ** 2
    capw = max(64, -(-n // W)) if seed % 2 else -(-n // W)
    vh, _ = O.assign(c, capw, 1)
    vm, am = O.assign(c, capw, 2)
    assert abs(vh - vm) <= 1e-12 * vh
    assert np.all(np.bincount(am, minlength=W) <= capw)
