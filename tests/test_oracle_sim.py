"""Pins of the oracle's simulation against rules checked independently.

- Block hash + first-miss probe + LRU (the readings fixed for §2.2's KV blocks):
  replayed with a cache keyed by the prompt prefix *content* (no hashing), on
  the oracle's own decisions; prefix lengths and final cache order must agree.
- LRU inclusion property (Mattson et al., 1970) with one worker.
- Event rules read back from the per-request records: the closed-loop
  semaphore of §7.4, b^active of Eq. (1), FIFO service, at most cap-1 requests
  in service, and the Eq. (9) latency decomposition of each TTFT.
- A hand-worked three-request timeline.
- The controller (Eq. (10), Eq. (11), hysteresis of §6.2) on a hand-computed
  sample sequence.
"""
from collections import OrderedDict

import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import workloads as Wk


def _small_trace(n=600, seed=3, rate=None, groups=8):
    spec = Wk.TraceSpec(n_req=n, len_kind="uniform", len_min=1, len_max=400, n_groups=groups,
                        prefix_min=32, prefix_max=200, zipf_s=1.1, out_kind="uniform",
                        out_min=1, out_max=300, rate=rate)
    return Wk.make_trace(spec, seed)


def _content_ids(trace, block=16):
    """Interned identity of every block prefix: (previous id, block bytes) -> id."""
    table = {}
    ids = []
    for i in range(trace.n_req):
        t = trace.tokens[trace.offsets[i]:trace.offsets[i + 1]]
        prev = -1
        row = []
        for k in range(len(t) // block):
            key = (prev, t[k * block:(k + 1) * block].tobytes())
            if key not in table:
                table[key] = len(table)
            prev = table[key]
            row.append(prev)
        ids.append(row)
    return ids


def test_hash_layout_and_prefix_property():
    tr = _small_trace(200)
    h = O.hash_blocks(tr.tokens, tr.offsets)
    ids = _content_ids(tr)
    seen = {}
    for i in range(tr.n_req):
        base = int(tr.offsets[i]) // 16
        for k, cid in enumerate(ids[i]):
            hv = int(h[base + k])
            assert hv >= 2
            # equal prefix content <-> equal chained hash (no collisions here)
            assert seen.setdefault(hv, cid) == cid
    assert len(set(seen.values())) == len(seen)


def test_hash_change_propagates_and_tail_ignored():
    rng = np.random.default_rng(5)
    t = rng.integers(0, 32000, size=16 * 12 + 7, dtype=np.int32)
    off = np.array([0, t.size], np.int64)
    h0 = O.hash_blocks(t, off)
    assert h0.size == 12
    for k in range(12):
        t2 = t.copy()
        t2[16 * k + int(rng.integers(0, 16))] ^= 1
        h1 = O.hash_blocks(t2, off)
        assert np.array_equal(h0[:k], h1[:k])
        assert np.all(h0[k:] != h1[k:])
    t3 = t.copy()
    t3[-3:] += 1      # partial tail block: not hashed
    assert np.array_equal(O.hash_blocks(t3, off), h0)
    assert not np.array_equal(O.hash_blocks(t, off, seed=1), h0)


@pytest.mark.parametrize("tau,K", [(0.0, 64), (0.7, 48), (0.0, 4096)])
def test_probe_and_lru_against_content_replay(tau, K):
    tr = _small_trace(500)
    cfg = O.OracleConfig(W=3, K=K)
    r = O.simulate(cfg, tr, 24, omega=1.0, tau=tau, seed=11, want_cache=True)
    assert r["status"] == 0
    ids = _content_ids(tr)
    h = O.hash_blocks(tr.tokens, tr.offsets)
    h2id = {}
    caches = [OrderedDict() for _ in range(3)]
    for i in range(tr.n_req):
        base = int(tr.offsets[i]) // 16
        for k, cid in enumerate(ids[i]):
            h2id[int(h[base + k])] = cid
        for j in range(3):
            m = 0
            while m < len(ids[i]) and ids[i][m] in caches[j]:
                m += 1
            assert r["prefix"][i, j] == m, (i, j)
        c = caches[int(r["worker"][i])]
        for cid in ids[i]:
            if cid in c:
                c.move_to_end(cid)
            else:
                if len(c) == K:
                    c.popitem(last=False)
                c[cid] = True
    for j in range(3):
        got = [h2id[int(x)] for x in r["cache"][j]]
        assert got == list(caches[j].keys())
    if K == 48:
        assert r["summary"]["evicted_blocks"] > 0


def test_lru_inclusion_single_worker():
    tr = _small_trace(400)
    sets, hits = [], []
    for K in (30, 31, 45, 90, 400):
        cfg = O.OracleConfig(W=1, K=K)
        r = O.simulate(cfg, tr, 8, want_cache=True)
        sets.append(set(int(x) for x in r["cache"][0]))
        hits.append(r["summary"]["hit_blocks"])
        assert len(r["cache"][0]) <= K
    for a, b in zip(sets, sets[1:]):
        assert a <= b
    assert all(x <= y for x, y in zip(hits, hits[1:]))


def _latency(n):
    return 0.005 * n + 0.020 + 0.010 / (64 - n) ** 2


@pytest.mark.parametrize("policy,C,rate", [(O.POLICY_DYNAMO, 256, None),
                                           (O.POLICY_LOADBAL, 300, None),
                                           (O.POLICY_DYNAMO, 40, 30.0)])
def test_event_rules_from_records(policy, C, rate):
    tr = _small_trace(1500, seed=9, rate=rate)
    cfg = O.OracleConfig(W=3, K=512)
    om = 1.0 if policy == O.POLICY_DYNAMO else 0.0
    r = O.simulate(cfg, tr, C, policy=policy, omega=om)
    assert r["status"] == 0
    n = tr.n_req
    a, s, ft, ct, tt = r["arrival"], r["start"], r["first_token"], r["completion"], r["ttft"]
    wk = r["worker"]
    L = np.diff(tr.offsets)
    blk = (L + tr.out_len + 15) // 16
    nbt = (L + 15) // 16
    assert np.array_equal(r["nbt"], nbt)
    assert np.all(np.diff(a) >= 0) and np.all(a >= tr.release)
    assert np.all(s >= a) and np.all(ft > s) and np.all(ct >= ft)
    assert np.allclose(tt, ft - a, rtol=0, atol=1e-12)
    queued = 0
    for i in range(n):
        prev = np.arange(i)
        live = ct[:i] > a[i]
        # closed-loop semaphore: at most C-1 others in flight at an arrival
        assert live.sum() <= C - 1
        if i > 0 and a[i] > max(tr.release[i], a[i - 1]):
            assert (ct[:i] >= a[i]).sum() >= C
        for j in range(3):
            on_j = wk[:i] == j
            # b^active of Eq. (1): unfinished requests routed to j
            A = int(blk[:i][on_j & live].sum())
            bp = int(nbt[i]) - int(r["prefix"][i, j])
            assert r["cost"][i, j] == np.float32(om) * np.float32(bp) + np.float32(A)
            inserv = int((on_j & live & (s[:i] <= a[i])).sum())
            assert r["n_frozen"][i, j] == min(inserv + 1, 63)
        if policy == O.POLICY_LOADBAL or True:
            assert wk[i] == int(np.argmin(r["cost"][i]))   # tau = 0: lowest-index argmin
        queued += s[i] > a[i]
    for j in range(3):
        idx = np.nonzero(wk == j)[0]
        assert np.all(np.diff(s[idx]) >= 0)                 # FIFO
        ev = sorted([(s[q], 1, q) for q in idx] + [(ct[q], 0, q) for q in idx])
        live = 0
        for _, kind, _ in ev:
            live += 1 if kind else -1
            assert live <= 63
    # TTFT = wait + f(n) - w_c * o with n the in-service count at start (incl. self)
    o = r["prefix"][np.arange(n), wk] / np.maximum(nbt, 1)
    f_obs = (ft - s) + 0.015 * o
    table = np.array([_latency(k) for k in range(1, 64)])
    for i in range(n):
        k = int(np.argmin(np.abs(table - f_obs[i])))
        assert abs(table[k] - f_obs[i]) < 1e-12
        same = (wk == wk[i]) & ((s < s[i]) | ((s == s[i]) & (np.arange(n) <= i))) & (ct > s[i])
        assert int(same.sum()) == k + 1
    summ = r["summary"]
    assert summ["n_routed"] == n
    assert np.isclose(summ["sum_ttft"], tt.sum(), rtol=1e-12)
    assert np.isclose(summ["makespan"], ct.max(), rtol=0)
    if C > 189:
        assert queued > 0


def test_hand_worked_timeline():
    """W=2, C=2, three identical 32-token prompts released at t=0, O=10 tokens.

    f(1) = 0.005 + 0.020 + 0.010/63^2 = 0.02500251952632905
    r0: both workers cost 2 (2 prefill blocks, no load) -> worker 0 (tie);
        TTFT = f(1); completes at f(1) + 10 * 0.012 = 0.14500251952632905.
    r1: worker 0 costs 0 + 3 (blocks cached, ceil(42/16) active) and worker 1
        costs 2 + 0 -> worker 1; TTFT = f(1); completes at the same instant.
    r2: the semaphore is full, so r2 arrives at the first completion (r0, the
        lower index of the tie); r1's completion at the same time is processed
        before routing.  Both workers cost 0 -> worker 0, overlap 1:
        TTFT = f(1) - 0.015 = 0.01000251952632905, completion at
        0.14500251952632905 + 0.01000251952632905 + 0.12 = 0.2750050390526581.
    """
    t = np.tile(np.arange(100, 132, dtype=np.int32), 3)
    tr = Wk.Trace(t, np.array([0, 32, 64, 96], np.int64), np.zeros(3), np.full(3, 10, np.int32),
                  np.zeros(3, np.int32))
    r = O.simulate(O.OracleConfig(W=2, K=16), tr, 2, omega=1.0, tau=0.0)
    assert list(r["worker"]) == [0, 1, 0]
    assert np.allclose(r["ttft"], [0.02500251952632905, 0.02500251952632905,
                                   0.01000251952632905], rtol=1e-13, atol=0)
    assert np.allclose(r["arrival"], [0.0, 0.0, 0.14500251952632905], rtol=1e-13, atol=0)
    assert np.allclose(r["completion"], [0.14500251952632905, 0.14500251952632905,
                                         0.2750050390526581], rtol=1e-13, atol=0)
    assert r["cost"].tolist() == [[2.0, 2.0], [3.0, 2.0], [0.0, 0.0]]
    assert r["prefix"].tolist() == [[0, 0], [2, 0], [2, 2]]


def test_controller_hand_trace():
    """theta1 = 0.3 s, theta2 = 2 s, alpha = 0.3, k = 3, epsilon = 0.1 theta."""
    nan = float("nan")
    L = [nan, 0.1, 0.5, 0.5, 0.5, 0.5, nan, 3.0, 3.0, 3.0, 3.0, 3.0,
         0.0, 0.0, 0.0, 0.0, 0.0, 0.0, 0.0, 0.0, 0.0]
    ewma, reg = O.controller_run(O.OracleConfig(), L)
    exp_ewma = [-1.0, 0.1, 0.22, 0.304, 0.3628, 0.40396, 0.432772, 1.2029404, 1.74205828,
                2.119440796, 2.3836085572, 2.56852599004, 1.797968193028, 1.2585777351196,
                0.88100441458372, 0.616703090208604, 0.4316921631460228,
                0.30218451420221596, 0.21152915994155117, 0.14807041195908582,
                0.10364928837136007]
    exp_reg = [0, 0, 0, 0, 0, 1, 1, 1, 1, 1, 1, 2, 2, 2, 1, 1, 1, 1, 1, 1, 0]
    assert np.allclose(ewma, exp_ewma, rtol=1e-12, atol=0)
    assert list(reg) == exp_reg


def test_controller_drives_regime_params_in_sim():
    """Saturated closed loop (C far above 6 x 63) pushes the EWMA past theta2."""
    spec = Wk.TraceSpec(n_req=6000, n_groups=16, prefix_min=64, prefix_max=256, len_median=256,
                        len_max=1024)
    tr = Wk.make_trace(spec, 2)
    cfg = O.OracleConfig(W=3, K=4096)
    r = O.simulate(cfg, tr, 600, controller=1, omega=1.0, tau=0.0, seed=1, max_ticks=4000)
    assert r["status"] == 0
    summ = r["summary"]
    assert summ["ticks"] > 3 and summ["max_regime"] == 2
    assert summ["sampled"] > 0        # tau switched to 0.7 / 0.8 after the first switch
    r0 = O.simulate(cfg, tr, 600, controller=0, omega=1.0, tau=0.0, seed=1)
    assert r0["summary"]["sampled"] == 0 and r0["summary"]["ticks"] == 0


def test_capacity_and_invalid_arguments():
    tr = _small_trace(50)
    r = O.simulate(O.OracleConfig(W=2, K=4), tr, 4)
    assert r["status"] == O.ERR_CAPACITY
    assert O.simulate(O.OracleConfig(W=2, K=64), tr, 0)["status"] == O.ERR_INVALID
    assert O.simulate(O.OracleConfig(W=2, K=64), tr, 4, tau=-1.0)["status"] == O.ERR_INVALID
    empty = O.simulate(O.OracleConfig(W=2, K=64), tr, 4, n_req=0)
    assert empty["status"] == 0 and empty["summary"]["n_routed"] == 0
