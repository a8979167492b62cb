"""Parity of the Game 2 tiers (§4.2, Eq. kv-cost) through the C ABI with the
oracle: decisions, G1 prefixes, the per-request charge and its categories,
rho, and every worker's whole recency stack (G3, G2, G1) bit-exact."""
import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import routesim as rs
from paper_2606_17081_gb300 import workloads as wk

from gpu_helpers import assert_replica_equal, gpu_run, oracle_cfg, oracle_run

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA device", allow_module_level=True)


def _rand_trace(n, seed, len_hi=640, rate=None, groups=6):
    spec = wk.TraceSpec(n_req=n, len_kind="uniform", len_min=0, len_max=len_hi,
                        n_groups=groups, prefix_min=16, prefix_max=300, zipf_s=1.1,
                        out_kind="uniform", out_min=0, out_max=300, rate=rate)
    return wk.make_trace(spec, seed)


def _ctx(W, K, k2, k3, node=1, **kw):
    return rs.Context(W=W, K=K, tiered=1, tier_k2=k2, tier_k3=k3, tier_node=node, **kw)


def _check(ctx, trs, reps, W, stack):
    st, g = gpu_run(ctx, trs, reps)
    assert st == 0
    cfg = oracle_cfg(ctx)
    for k, r in enumerate(reps):
        o = oracle_run(cfg, trs[r.trace], r, want_cache=True)
        assert_replica_equal(g[k], o, W)
        for j in range(W):
            assert np.array_equal(rs.route_cache_dump(ctx.h, 1, k, j, stack), o["cache"][j]), (k, j)
    return g


@pytest.mark.parametrize("W,K,k2,k3,node,C,tau", [
    (3, 48, 64, 200, 1, 24, 0.0),
    (4, 40, 40, 80, 2, 40, 0.6),
    (4, 60, 0, 120, 2, 16, 0.0),     # no G2
    (3, 80, 50, 0, 3, 30, 0.3),      # no G3, one node
    (3, 64, 0, 0, 1, 24, 0.0),       # G1 only: remote copies and recomputation
])
def test_tier_parity(W, K, k2, k3, node, C, tau):
    tr = _rand_trace(800, 3 + K, rate=40.0)
    reps = [wk.Replica(0, C, wk.POLICY_DYNAMO, 0, 1.0, tau, 9, tr.n_req),
            wk.Replica(0, C, wk.POLICY_LOADBAL, 0, 0.0, 0.0, 9, tr.n_req)]
    ctx = _ctx(W, K, k2, k3, node)
    g = _check(ctx, [tr], reps, W, K + k2 + k3)
    r = g[0]["result"]
    assert r["kv_remote"] > 0 and r["kv_recompute"] > 0 and r["evicted_blocks"] > 0
    if k2 + k3:
        assert r["kv_g2"] + r["kv_g3"] > 0


def test_tier_g1_routing_equals_lru_of_g1():
    tr = _rand_trace(700, 8)
    reps = [wk.Replica(0, 20, wk.POLICY_DYNAMO, 0, 1.0, 0.5, 4, tr.n_req)]
    _, plain = gpu_run(rs.Context(W=3, K=50), [tr], reps)
    _, tier = gpu_run(_ctx(3, 50, 70, 90), [tr], reps)
    for f in ("worker", "prefix", "ttft", "completion"):
        assert np.array_equal(plain[0][f], tier[0][f]), f
    assert plain[0]["result"]["hit_blocks"] == tier[0]["result"]["hit_blocks"]


def test_tier_rebuilds_and_slow_path():
    # long shared prefixes against small stacks: compactions and the exact
    # sequential update, with the band boundaries carried through both
    spec = wk.TraceSpec(n_req=3000, len_kind="uniform", len_min=100, len_max=900, n_groups=40,
                        prefix_min=200, prefix_max=800, zipf_s=0.6, out_kind="uniform",
                        out_min=1, out_max=64)
    tr = wk.make_trace(spec, 5)
    ctx = _ctx(2, 60, 30, 30, 1)
    reps = [wk.Replica(0, 16, wk.POLICY_DYNAMO, 0, 2.0, 0.0, 0, tr.n_req)]
    g = _check(ctx, [tr], reps, 2, 120)
    r = g[0]["result"]
    assert r["slow_path"] > 0 and r["rebuilds"] > 0


def test_tier_hand_worked_round_robin():
    # the two-worker sequence worked by hand in the oracle pins
    names = "ABBACAADEB"
    n = len(names)
    tokens = np.zeros(16 * n, np.int32)
    for i, nm in enumerate(names):
        tokens[16 * i:16 * (i + 1)] = 500 + 41 * (ord(nm) - ord("A")) + np.arange(16)
    tr = wk.Trace(tokens, np.arange(0, 16 * (n + 1), 16, dtype=np.int64),
                  np.array([0.1 * i for i in range(n)]), np.ones(n, np.int32),
                  np.zeros(n, np.int32))
    ctx = _ctx(2, 1, 1, 1, 1)
    reps = [wk.Replica(0, 100, wk.POLICY_ROUNDROBIN, 0, 1.0, 0.0, 0, n)]
    st, g = gpu_run(ctx, [tr], reps)
    assert st == 0
    assert list(g[0]["kv_cost"]) == [100, 100, 11, 14, 100, 1, 20, 100, 100, 20]
    r = g[0]["result"]
    assert (r["kv_g1"], r["kv_g2"], r["kv_g3"], r["kv_remote"], r["kv_recompute"]) == (1, 0, 2, 2, 5)
    assert r["kv_cost"] == 566.0 and r["first_evict_t"] == 0.2
    assert r["rho_first_evict"] == 1.5 and r["rho_end"] == 3.0
    h = O.hash_blocks(tr.tokens, tr.offsets)
    nm = {int(h[i]): names[i] for i in range(n)}
    assert [nm[int(x)] for x in rs.route_cache_dump(ctx.h, 1, 0, 0, 3)] == list("CAE")
    assert [nm[int(x)] for x in rs.route_cache_dump(ctx.h, 1, 0, 1, 3)] == list("ADB")


def test_tier_limits_and_rejections():
    spec = wk.TraceSpec(n_req=40, len_kind="uniform", len_min=16 * 690, len_max=16 * 700,
                        n_groups=4, prefix_min=16, prefix_max=300, zipf_s=1.1,
                        out_kind="uniform", out_min=1, out_max=30)
    tr = wk.make_trace(spec, 2)                      # 690 .. 700 blocks
    ctx = _ctx(3, 800, 10, 10)
    st, _ = gpu_run(ctx, [tr], [wk.Replica(0, 4, wk.POLICY_DYNAMO, 0, 1.0, 0.0, 0, 40)])
    assert st == rs.RS_ERR_CAPACITY                  # 3 * 700 pairs > 2048
    small = _rand_trace(20, 1)
    r = wk.Replica(0, 4, wk.POLICY_DYNAMO, 0, 1.0, 0.0, 0, 20)
    r.eviction = rs.RS_EVICT_FREQ
    st, _ = gpu_run(_ctx(2, 64, 8, 8), [small], [r])
    assert st == rs.RS_ERR_INVALID                   # no frequency rule with tiers
    for kw in ({"tier_alpha": (1.0, 1.0, 20.0)}, {"tier_gamma": 10.0}, {"tier_node": 0},
               {"tier_d_far": -1.0}):
        base = {"tiered": 1, "tier_k2": 8, "tier_k3": 8, "tier_node": 1}
        base.update(kw)
        with pytest.raises(rs.RoutesimError):
            rs.Context(W=2, K=64, **base)
