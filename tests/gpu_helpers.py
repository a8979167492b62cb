"""Shared helpers of the GPU parity tests: run a replica grid through the C ABI
and the same replicas through the oracle, on identical seeded inputs."""
import numpy as np

import oracle as O
from paper_2606_17081_gb300 import routesim as rs
from paper_2606_17081_gb300 import workloads as wk

REC_FIELDS = ("worker", "arrival", "start", "first_token", "completion", "ttft", "nbt")


def gpu_run(ctx, traces, replicas, trace_mem=rs.RS_MEM_DEVICE, with_cost=True, flags=0):
    """Returns (results list of dict, records dict of numpy arrays per replica)."""
    import torch
    W = ctx.W
    bufs = [rs.device_trace(t) if trace_mem == rs.RS_MEM_DEVICE else rs.host_trace(t)
            for t in traces]
    rows = sum(r.n_req for r in replicas)
    with_kv = bool(ctx.cfg.tiered)
    rec, t = rs.device_records(max(rows, 1), W, with_cost=with_cost, with_kv=with_kv)
    try:
        res = rs.simulate_replicas(ctx.h, [b.desc() for b in bufs], trace_mem,
                                   [rs.replica_params(r) for r in replicas], rec, flags)
        status = rs.RS_OK
    except rs.RoutesimError as e:
        res = e.results
        status = e.status
    torch.cuda.synchronize()
    host = {k: v.cpu().numpy() for k, v in t.items()}
    out = []
    base = 0
    for k, r in enumerate(replicas):
        n = r.n_req
        d = {f: host[f][base:base + n] for f in REC_FIELDS + (("kv_cost",) if with_kv else ())}
        for f in ("n_frozen", "prefix") + (("cost",) if with_cost else ()):
            a = host[f][base * W:(base + n) * W].reshape(n, W)
            d[f] = a.view(np.uint16) if a.dtype == np.int16 else a
        d["result"] = res[k].as_dict()
        out.append(d)
        base += n
    return status, out


def oracle_cfg(ctx_or_W, K=None, **kw):
    if K is None:
        c = ctx_or_W.cfg
        if c.tiered:   # the context's Game 2 tiers
            kw.update(tiered=1, tier_node=c.tier_node, tier_k2=c.tier_k2, tier_k3=c.tier_k3,
                      tier_alpha=tuple(c.tier_alpha), tier_gamma=c.tier_gamma,
                      tier_d_near=c.tier_d_near, tier_d_far=c.tier_d_far)
        return O.OracleConfig(W=ctx_or_W.W, K=ctx_or_W.K, **kw)
    return O.OracleConfig(W=ctx_or_W, K=K, **kw)


def oracle_run(cfg, trace, r, want_cache=False, max_ticks=0):
    sched = (r.c_t1, r.c_t2, r.c_mid, r.c_end) if getattr(r, "c_mid", 0) > 0 else None
    return O.simulate(cfg, trace, r.C, policy=r.policy, controller=r.controller, omega=r.omega,
                      tau=r.tau, seed=r.seed, n_req=r.n_req, want_cache=want_cache,
                      max_ticks=max_ticks, schedule=sched, eviction=getattr(r, "eviction", 0),
                      freq_max=getattr(r, "freq_max", 64), decay_s=getattr(r, "decay_s", 1.0))


def assert_replica_equal(g, o, W, times_rtol=1e-12, check_cost=True):
    n = o["worker"].size
    assert g["result"]["status"] == o["status"] == 0, (g["result"]["status"], o["status"])
    assert np.array_equal(g["worker"], o["worker"]), _first_diff(g["worker"], o["worker"])
    assert np.array_equal(g["prefix"], o["prefix"]), "m_ij differ"
    assert np.array_equal(g["n_frozen"], o["n_frozen"]), "frozen loads differ"
    assert np.array_equal(g["nbt"], o["nbt"])
    if check_cost:
        assert np.array_equal(g["cost"], o["cost"]), "Eq. (1) costs differ"
    for f in ("arrival", "start", "first_token", "completion", "ttft"):
        assert np.allclose(g[f], o[f], rtol=times_rtol, atol=0), f
    gr, orr = g["result"], o["summary"]
    assert gr["first_switch_t"] == orr["first_switch_t"], (gr["first_switch_t"], orr["first_switch_t"])
    for f in ("first_evict_t", "rho_first_evict", "rho_end", "kv_g1", "kv_g2", "kv_g3",
              "kv_remote", "kv_recompute", "kv_cost"):
        assert gr[f] == orr[f], (f, gr[f], orr[f])
    if "kv_cost" in g:
        assert np.array_equal(g["kv_cost"], o["kv_cost"]), "Eq. kv-cost per request differs"
    for f in ("n_routed", "near_ties", "exact_ties", "sampled", "near_boundary", "hit_blocks",
              "inserted_blocks", "evicted_blocks", "ticks", "regime_switches", "final_regime",
              "max_regime"):
        assert gr[f] == orr[f], (f, gr[f], orr[f])
    assert list(gr["ticks_in_regime"]) == list(orr["ticks_in_regime"])
    for f in ("sum_ttft", "sum_e2e", "makespan"):
        assert abs(gr[f] - orr[f]) <= 1e-9 * max(1.0, abs(orr[f])), (f, gr[f], orr[f])
    if orr["final_ewma"] < 0:
        assert gr["final_ewma"] < 0
    else:
        assert abs(gr["final_ewma"] - orr["final_ewma"]) <= 1e-12 * orr["final_ewma"]
    assert n == gr["n_routed"]


def _first_diff(a, b):
    idx = np.nonzero(a != b)[0]
    return f"first decision difference at request {idx[0] if idx.size else None}"
