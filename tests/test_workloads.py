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


def test_splitmix64_published_outputs():
    # SplitMix64 (Steele, Lea & Flood 2014) from seed 0: its first outputs are
    # the published e220a8397b1dcdaf, 6e789e6aa1b965f4, 06c45d188009454f
    z = Wk.sm_output_np(np.array([0, 1, 2], np.int64), 0)
    assert [int(v) for v in z] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_counter_trace_random_access_and_prefixes():
    spec = Wk.TraceSpec(n_req=400, n_groups=8, prefix_min=40, prefix_max=90, len_kind="uniform",
                        len_min=16, len_max=300, tokens="counter", n_meta=1000)
    m = Wk.trace_meta(spec, 5)
    t = Wk.make_trace(spec, 5)
    assert t.n_req == 400 and t.tokens.size % 4 == 0
    # tokens of any range on their own equal the same range of the whole trace
    for x0, x1 in ((0, 1), (17, 933), (t.n_tokens - 50, t.n_tokens)):
        assert np.array_equal(m.tokens(x0, x1), t.tokens[x0:x1])
    # a shorter n_req keeps the same first requests (lengths, times, tokens)
    u = Wk.make_trace(Wk.TraceSpec(**{**spec.__dict__, "n_req": 100}), 5)
    assert np.array_equal(u.offsets, t.offsets[:101])
    assert np.array_equal(u.tokens[:u.n_tokens], t.tokens[:u.n_tokens])
    # every request starts with min(prefix length, L) tokens of its group's prefix
    for i in range(t.n_req):
        g, a = int(t.group[i]), int(t.offsets[i])
        k = int(m.kpref[i])
        plen = int(m.pool_off[g + 1] - m.pool_off[g])
        assert k == min(plen, int(t.offsets[i + 1] - a))
        assert np.array_equal(t.tokens[a:a + k], m.pool[m.pool_off[g]:m.pool_off[g] + k])
    assert t.tokens.min() >= 0 and t.tokens.max() < spec.vocab


def test_counter_tokens_torch_equal_numpy():
    torch = __import__("pytest").importorskip("torch")
    spec = Wk.TraceSpec(n_req=3000, tokens="counter", n_meta=3000, len_max=4000)
    m = Wk.trace_meta(spec, 11)
    d = m.device("cpu")
    end = int(m.offsets[-1])
    for x0, n in ((0, 5000), (int(m.offsets[1234]) + 3, 70001), (end - 777, 900)):
        out = torch.full((n,), -1, dtype=torch.int32)
        m.fill_device(d, x0, x0 + n, out, step=4096)
        assert np.array_equal(out.numpy(), m.tokens(x0, x0 + n))


def test_large_plan_uses_counter_tokens():
    p = Wk.plan("large", n_req=50, replicas=[0, 8])
    assert p.spec.tokens == "counter" and p.spec.n_meta == 1_000_000 and p.K == 1 << 20
    m = p.metas()[0]
    assert m.n_req == 50 and m.offsets[-1] == p.traces()[0].offsets[-1]
