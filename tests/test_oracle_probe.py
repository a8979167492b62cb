"""Pins of the oracle's batch probe (orc_router_probe: S2, the b^prefill of
Eq. (1), for many requests against one cache snapshot) against things other
than its code: a replay of the routed requests through LRU caches keyed by
prompt content (no hashes, no hash map) gives the same m_ij; probing changes
nothing (the routing that follows is the one a router that never probed
makes); special cases by hand (empty caches, a request just routed, a tail
shorter than a block)."""
from collections import OrderedDict

import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import workloads as Wk


def _trace(n, seed, lo=0, hi=700, groups=6):
    spec = Wk.TraceSpec(n_req=n, len_kind="uniform", len_min=lo, len_max=hi, n_groups=groups,
                        prefix_min=16, prefix_max=300, zipf_s=1.1, out_kind="uniform",
                        out_min=1, out_max=300)
    return Wk.make_trace(spec, seed)


def _content_ids(trace, table, block=16):
    ids = []
    for i in range(trace.n_req):
        t = trace.tokens[trace.offsets[i]:trace.offsets[i + 1]]
        prev, row = -1, []
        for k in range(len(t) // block):
            key = (prev, t[k * block:(k + 1) * block].tobytes())
            if key not in table:
                table[key] = len(table)
            prev = table[key]
            row.append(prev)
        ids.append(row)
    return ids


def _sub(tr, lo, hi):
    return Wk.Trace(tr.tokens, tr.offsets[lo:hi + 1], tr.release[lo:hi], tr.out_len[lo:hi],
                    tr.group[lo:hi])


@pytest.mark.parametrize("W,K,tau,seed", [(3, 60, 0.0, 1), (4, 200, 0.5, 2), (2, 45, 0.0, 3)])
def test_probe_matches_content_replay(W, K, tau, seed):
    tr = _trace(600, seed)
    routed, probed = _sub(tr, 0, 400), _sub(tr, 400, 600)
    r = O.Router(O.OracleConfig(W=W, K=K), 1.0, tau, 9, n_instances=1)
    st, worker, _, _ = r.route(0, routed.tokens, routed.offsets, routed.out_len)
    assert st == 0
    table = {}
    ids_r = _content_ids(routed, table)
    ids_p = _content_ids(probed, table)
    caches = [OrderedDict() for _ in range(W)]
    for i, row in enumerate(ids_r):
        c = caches[int(worker[i])]
        for b in row:
            if b in c:
                c.move_to_end(b)
            else:
                if len(c) == K:
                    c.popitem(last=False)
                c[b] = True
    st, m = r.probe(0, probed.tokens, probed.offsets)
    assert st == 0
    for i, row in enumerate(ids_p):
        for j in range(W):
            want = 0
            while want < len(row) and row[want] in caches[j]:
                want += 1
            assert m[i, j] == want, (i, j)
    assert m.max() > 0 and (m == 0).any()


def test_probe_changes_nothing():
    tr = _trace(300, 4)
    a, b = _sub(tr, 0, 150), _sub(tr, 150, 300)
    cfg = O.OracleConfig(W=3, K=80)
    r1 = O.Router(cfg, 1.0, 0.3, 5)
    r2 = O.Router(cfg, 1.0, 0.3, 5)
    for r in (r1, r2):
        assert r.route(0, a.tokens, a.offsets, a.out_len)[0] == 0
    st, m1 = r1.probe(0, b.tokens, b.offsets)
    st2, m2 = r1.probe(0, b.tokens, b.offsets)
    assert st == st2 == 0 and np.array_equal(m1, m2)
    x1 = r1.route(0, b.tokens, b.offsets, b.out_len)
    x2 = r2.route(0, b.tokens, b.offsets, b.out_len)
    for u, v in zip(x1[1:], x2[1:]):
        assert np.array_equal(u, v)
    for j in range(3):
        assert np.array_equal(r1.cache(0, j), r2.cache(0, j))
    assert np.array_equal(r1.active(0), r2.active(0))


def test_probe_special_cases():
    # 3 requests: 40 tokens (2 blocks + 8), 16 tokens (1 block), 15 tokens (no block)
    rng = np.random.default_rng(0)
    toks = rng.integers(0, 32000, 80).astype(np.int32)
    offsets = np.array([0, 40, 56, 71], np.int64)
    tr = Wk.Trace(toks, offsets, np.zeros(3), np.ones(3, np.int32), np.zeros(3, np.int32))
    r = O.Router(O.OracleConfig(W=2, K=10), 1.0, 0.0, 0)
    st, m = r.probe(0, tr.tokens, tr.offsets)
    assert st == 0 and np.array_equal(m, np.zeros((3, 2), np.int32))      # empty caches
    one = _sub(tr, 0, 1)
    st, w, _, _ = r.route(0, one.tokens, one.offsets, one.out_len)
    assert st == 0 and w[0] == 0                                         # ties: lowest index
    st, m = r.probe(0, tr.tokens, tr.offsets)
    # request 0 on worker 0: both full blocks; its 8-token tail is no block.
    # request 1 starts with other tokens; request 2 has no full block
    assert np.array_equal(m, np.array([[2, 0], [0, 0], [0, 0]], np.int32))
    # a prompt that starts like request 0 but diverges inside block 1
    p2 = toks[0:40].copy()
    p2[20] += 1
    st, m = r.probe(0, np.concatenate([toks, p2]), np.array([80, 120], np.int64))
    assert st == 0 and np.array_equal(m, np.array([[1, 0]], np.int32))
    assert r.probe(5, tr.tokens, tr.offsets)[0] == O.ERR_INVALID
