"""Pins of the oracle's live router (route_batch / route_release semantics)
against things other than its code: a batch routes exactly as the same
requests one call at a time; every Eq. (1) cost equals omega (nbt - m) + A
with A recounted from the routed requests' blocks less the released ones;
instances are independent; a release never drives a load below zero and
skips (and reports) a worker out of range."""
import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import workloads as Wk


def _trace(n, seed):
    spec = Wk.TraceSpec(n_req=n, len_kind="uniform", len_min=0, len_max=500, n_groups=6,
                        prefix_min=16, prefix_max=300, zipf_s=1.1, out_kind="uniform",
                        out_min=1, out_max=300)
    return Wk.make_trace(spec, seed)


def _sub(tr, lo, hi):
    return Wk.Trace(tr.tokens, tr.offsets[lo:hi + 1], tr.release[lo:hi], tr.out_len[lo:hi],
                    tr.group[lo:hi])


@pytest.mark.parametrize("W,K,omega,tau", [(3, 64, 1.0, 0.0), (4, 200, 0.5, 0.6)])
def test_batch_equals_single_calls(W, K, omega, tau):
    tr = _trace(300, W)
    cfg = O.OracleConfig(W=W, K=K)
    rb = O.Router(cfg, omega, tau, 17)
    rs_ = O.Router(cfg, omega, tau, 17)
    st, wb, cb, pb = rb.route(0, tr.tokens, tr.offsets, tr.out_len)
    assert st == 0
    ws, cs, ps = [], [], []
    for i in range(tr.n_req):
        one = _sub(tr, i, i + 1)
        st, w, c, p = rs_.route(0, one.tokens, one.offsets, one.out_len)
        assert st == 0
        ws.append(w[0]); cs.append(c[0]); ps.append(p[0])
    assert np.array_equal(wb, np.array(ws))
    assert np.array_equal(cb, np.array(cs))
    assert np.array_equal(pb, np.array(ps))
    for j in range(W):
        assert np.array_equal(rb.cache(0, j), rs_.cache(0, j))
    assert np.array_equal(rb.active(0), rs_.active(0))


def test_costs_from_recounted_loads_and_releases():
    W, K, om = 3, 80, 1.0
    tr = _trace(400, 7)
    r = O.Router(O.OracleConfig(W=W, K=K), om, 0.0, 0, n_instances=2)
    A = np.zeros(W, np.int64)
    L = np.diff(tr.offsets)
    blk = (L + tr.out_len + 15) // 16
    nbt = (L + 15) // 16
    rng = np.random.default_rng(1)
    routed = []
    for lo in range(0, 400, 50):
        sub = _sub(tr, lo, lo + 50)
        st, w, c, p = r.route(1, sub.tokens, sub.offsets, sub.out_len)
        assert st == 0
        for k in range(50):
            i = lo + k
            for j in range(W):
                want = np.float32(om) * np.float32(nbt[i] - p[k, j]) + np.float32(A[j])
                assert c[k, j] == want, (i, j)
            assert w[k] == int(np.argmin(c[k]))          # tau = 0: lowest-index argmin
            A[w[k]] += blk[i]
            routed.append((int(w[k]), int(blk[i])))
        # release a random subset of what is in flight
        take = rng.choice(len(routed), size=len(routed) // 3, replace=False)
        ww = np.array([routed[t][0] for t in take], np.int32)
        bb = np.array([routed[t][1] for t in take], np.int32)
        assert r.release(1, ww, bb) == 0
        for t in sorted(take, reverse=True):
            A[routed[t][0]] -= routed[t][1]
            routed.pop(t)
        assert np.array_equal(r.active(1), A)
    assert np.array_equal(r.active(0), np.zeros(W, np.int64))   # the other instance
    assert all(r.cache(0, j).size == 0 for j in range(W))


def test_release_floor_and_bad_worker():
    W = 2
    tr = _trace(10, 3)
    r = O.Router(O.OracleConfig(W=W, K=64), 1.0, 0.0, 0)
    assert r.route(0, tr.tokens, tr.offsets, tr.out_len)[0] == 0
    a0 = r.active(0).copy()
    st = r.release(0, np.array([0, 5, 1], np.int32), np.array([10 ** 6, 3, 1], np.int32))
    assert st == O.ERR_INVALID                                    # worker 5 skipped, reported
    assert r.active(0)[0] == 0                                    # floor at zero
    assert r.active(0)[1] == max(a0[1] - 1, 0)
