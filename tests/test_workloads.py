"""The seeded input generator: determinism, shapes and layout rules."""
import numpy as np

from paper_2606_17081_gb300 import workloads as Wk


def test_trace_deterministic_and_padded():
    a = Wk.make_trace(Wk.TINY_SPEC, 0)
    b = Wk.make_trace(Wk.TINY_SPEC, 0)
    c = Wk.make_trace(Wk.TINY_SPEC, 1)
    assert np.array_equal(a.tokens, b.tokens) and np.array_equal(a.offsets, b.offsets)
    assert not np.array_equal(a.tokens[:1000], c.tokens[:1000])
    assert a.tokens.size % 4 == 0 and a.tokens.size >= a.n_tokens
    L = np.diff(a.offsets)
    assert L.min() >= 64 and L.max() <= 512 and a.n_req == 512
    assert np.all(np.diff(a.release) >= 0) and a.release[0] > 0
    assert a.tokens.min() >= 0 and a.tokens.max() < 32000


def test_prefix_groups_share_leading_tokens():
    t = Wk.make_trace(Wk.TraceSpec(n_req=300, n_groups=4, prefix_min=64, prefix_max=64,
                                   len_kind="uniform", len_min=80, len_max=200), 3)
    for g in range(4):
        idx = np.nonzero(t.group == g)[0]
        heads = {t.tokens[t.offsets[i]:t.offsets[i] + 64].tobytes() for i in idx}
        assert len(heads) == 1


def test_plans_shapes():
    p = Wk.plan("p2d")
    assert p.W == 3 and len(p.replicas) == 64 and len(p.trace_seeds) == 7
    assert sorted({r.C for r in p.replicas}) == [16, 32, 64, 128, 256]
    g = Wk.plan("grid")
    assert len(g.replicas) == 8192 and g.K == 32768
    q = Wk.plan("p5d", n_req=1000, replicas=[0, 17, 255])
    assert [r.trace for r in q.replicas] == [0, 1, 2] and q.trace_seeds == [0, 1, 17]
    assert all(r.n_req == 1000 for r in q.replicas)
    h = Wk.make_trace(Wk.TINY_SPEC, 0).head(10)
    assert h.n_req == 10 and h.tokens.size % 4 == 0
