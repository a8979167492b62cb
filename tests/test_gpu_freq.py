"""Parity of the frequency eviction (the KV Block Manager rule of §2.2) and of
the cache-pressure outputs (§5.3) through the C ABI with the oracle:
decisions, cached prefixes, counters, rho and the final caches in recency
order bit-exact, per-request times within 1e-12."""
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


def _rand_trace(n, seed, len_lo=0, len_hi=700, groups=6, rate=None, out_hi=300, pmax=300):
    spec = wk.TraceSpec(n_req=n, len_kind="uniform", len_min=len_lo, len_max=len_hi,
                        n_groups=groups, prefix_min=16, prefix_max=pmax, zipf_s=1.1,
                        out_kind="uniform", out_min=0, out_max=out_hi, rate=rate)
    return wk.make_trace(spec, seed)


def _freq(r, fmax, decay):
    r.eviction, r.freq_max, r.decay_s = rs.RS_EVICT_FREQ, fmax, decay
    return r


def _check_caches(ctx, g, o, W, K, index=0):
    for j in range(W):
        assert np.array_equal(rs.route_cache_dump(ctx.h, 1, index, j, K), o["cache"][j]), j


@pytest.mark.parametrize("K,C,tau,fmax,decay,rate", [
    (64, 24, 0.0, 8, 0.5, 40.0),        # decays often
    (200, 40, 0.7, 64, 5.0, 40.0),      # sampling, long protection
    (48, 16, 0.0, 4, 1e9, None),        # never decays: hot blocks pile up
    (120, 24, 0.0, 1 << 20, 0.05, 60.0),
    (600, 8, 0.3, 16, 2.0, None),       # few evictions
])
def test_frequency_eviction_parity(K, C, tau, fmax, decay, rate):
    tr = _rand_trace(900, 11 + K, len_hi=640, rate=rate)
    W = 3
    reps = [_freq(wk.Replica(0, C, wk.POLICY_DYNAMO, 0, 1.0, tau, 7, tr.n_req), fmax, decay)]
    ctx = rs.Context(W=W, K=K)
    st, g = gpu_run(ctx, [tr], reps)
    assert st == 0
    o = oracle_run(oracle_cfg(ctx), tr, reps[0], want_cache=True)
    assert_replica_equal(g[0], o, W)
    _check_caches(ctx, g, o, W, K)
    if K < 300:
        assert g[0]["result"]["evicted_blocks"] > 0


def test_frequency_eviction_under_pressure():
    # prompts of up to 23 blocks against 24-block caches, long shared
    # prefixes and no decay: hits make most of a cache hot, so requests evict
    # hot blocks and their own blocks (the exact sequential path)
    spec = wk.TraceSpec(n_req=1500, len_kind="uniform", len_min=16, len_max=380, n_groups=5,
                        prefix_min=100, prefix_max=300, zipf_s=0.8, out_kind="uniform",
                        out_min=1, out_max=32)
    tr = wk.make_trace(spec, 9)
    W, K = 2, 24
    reps = [_freq(wk.Replica(0, 12, wk.POLICY_DYNAMO, 0, 2.0, 0.0, 3, tr.n_req), 8, 1e9),
            _freq(wk.Replica(0, 12, wk.POLICY_DYNAMO, 0, 2.0, 0.0, 3, tr.n_req), 2, 0.2),
            _freq(wk.Replica(0, 12, wk.POLICY_LOADBAL, 0, 0.0, 0.0, 3, tr.n_req), 1 << 20, 50.0)]
    ctx = rs.Context(W=W, K=K)
    st, g = gpu_run(ctx, [tr], reps)
    assert st == 0
    cfg = oracle_cfg(ctx)
    for k, r in enumerate(reps):
        o = oracle_run(cfg, tr, r, want_cache=True)
        assert_replica_equal(g[k], o, W)
        _check_caches(ctx, g[k], o, W, K, index=k)
    assert sum(x["result"]["slow_path"] for x in g) > 0


def test_frequency_cap_one_equals_lru_on_gpu():
    tr = _rand_trace(800, 5, len_hi=700)
    W, K = 3, 60
    base = wk.Replica(0, 30, wk.POLICY_DYNAMO, 0, 1.0, 0.5, 4, tr.n_req)
    reps = [base, _freq(wk.Replica(**vars(base)), 1, 0.3)]
    ctx = rs.Context(W=W, K=K)
    st, g = gpu_run(ctx, [tr], reps)
    assert st == 0
    for f in ("worker", "prefix", "ttft", "completion"):
        assert np.array_equal(g[0][f], g[1][f]), f
    for j in range(W):
        assert np.array_equal(rs.route_cache_dump(ctx.h, 1, 0, j, K),
                              rs.route_cache_dump(ctx.h, 1, 1, j, K))
    o = oracle_run(oracle_cfg(ctx), tr, reps[1], want_cache=True)
    assert_replica_equal(g[1], o, W)


def test_hand_worked_sequence_on_gpu():
    # the single-worker sequence worked by hand in the oracle pins: K = 3, one
    # decay step per second, cap 4; the cache ends with I, J, K
    names = "ABCADEFGEEHIJK"
    times = [0.0, 0.1, 0.2, 0.3, 0.4, 0.5, 0.6, 1.2, 1.3, 1.35, 1.4, 2.5, 2.6, 4.5]
    n = len(names)
    tokens = np.zeros(16 * n, np.int32)
    for i, nm in enumerate(names):
        tokens[16 * i:16 * (i + 1)] = 1000 + 37 * (ord(nm) - ord("A")) + np.arange(16)
    tr = wk.Trace(tokens, np.arange(0, 16 * (n + 1), 16, dtype=np.int64),
                  np.array(times), np.ones(n, np.int32), np.zeros(n, np.int32))
    ctx = rs.Context(W=1, K=3)
    reps = [_freq(wk.Replica(0, 100, wk.POLICY_DYNAMO, 0, 1.0, 0.0, 0, n), 4, 1.0)]
    st, g = gpu_run(ctx, [tr], reps)
    assert st == 0
    h = O.hash_blocks(tr.tokens, tr.offsets)
    name_of = {int(h[i]): names[i] for i in range(n)}
    got = [name_of[int(x)] for x in rs.route_cache_dump(ctx.h, 1, 0, 0, 3)]
    assert got == list("IJK")
    r = g[0]["result"]
    assert (r["inserted_blocks"], r["evicted_blocks"], r["hit_blocks"]) == (11, 8, 3)
    assert r["first_evict_t"] == 0.4 and r["rho_first_evict"] == 1.0 and r["rho_end"] == 1.0


def test_lru_and_frequency_replicas_in_one_launch():
    trs = [_rand_trace(700, s, len_hi=800, rate=(30.0 if s else None)) for s in range(2)]
    reps = []
    for k in range(12):
        r = wk.Replica(k % 2, [8, 40, 120][k % 3], wk.POLICY_DYNAMO, k % 2, 1.0,
                       [0.0, 0.6][k % 2], 20 + k, 700 - 31 * (k % 4))
        if k % 3:
            _freq(r, [4, 64][k % 2], [0.5, 3.0][(k // 2) % 2])
        reps.append(r)
    ctx = rs.Context(W=4, K=150)
    st, g = gpu_run(ctx, trs, reps)
    assert st == 0
    cfg = oracle_cfg(ctx)
    for k, r in enumerate(reps):
        o = oracle_run(cfg, trs[r.trace], r, want_cache=True)
        assert_replica_equal(g[k], o, 4)
        _check_caches(ctx, g[k], o, 4, 150, index=k)


def test_frequency_arguments_rejected():
    tr = _rand_trace(20, 1)
    ctx = rs.Context(W=2, K=64)
    for fmax, decay in ((0, 1.0), ((1 << 20) + 1, 1.0), (4, 0.0), (4, float("inf"))):
        r = _freq(wk.Replica(0, 4, wk.POLICY_DYNAMO, 0, 1.0, 0.0, 0, 20), fmax, decay)
        st, _ = gpu_run(ctx, [tr], [r])
        assert st == rs.RS_ERR_INVALID
