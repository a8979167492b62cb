"""Parity at the workloads' own sizes, in the launch configuration the
benchmark times: every replica of a grid runs in one simulate_replicas call;
the oracle recomputes sampled replicas one by one."""
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


def _check(p, sample, poa=True):
    traces = p.traces()
    ctx = rs.Context(W=p.W, K=p.K, theta1=p.theta1, theta2=p.theta2)
    st, g = gpu_run(ctx, traces, p.replicas, with_cost=False,
                    flags=0 if poa else rs.RS_SIM_NO_POA)
    assert st == 0
    cfg = oracle_cfg(ctx, theta1=p.theta1, theta2=p.theta2)
    for k in sample:
        r = p.replicas[k]
        o = oracle_run(cfg, traces[r.trace], r)
        assert_replica_equal(g[k], o, p.W, check_cost=False)
        if poa:
            _, opt, _, tot = O.poa(cfg, o)
            assert abs(g[k]["result"]["poa_total"] - tot) <= 1e-4 * tot
            st = float(np.sum(O.static_numer(cfg, o))) / float(np.sum(opt))
            assert abs(g[k]["result"]["poa_static"] - st) <= 1e-4 * st
    return g


def test_p2d_full_size_sampled_replicas():
    p = wk.plan("p2d")
    g = _check(p, [0, 5, 37, 63])
    assert all(x["result"]["status"] == 0 for x in g)
    assert sum(x["result"]["evicted_blocks"] for x in g) > 0


def test_p5d_grid_reduced():
    p = wk.plan("p5d", n_req=3000, replicas=list(range(0, 256, 17)) + [255])
    _check(p, range(len(p.replicas)))


def test_grid_reduced():
    p = wk.plan("grid", n_req=1500, replicas=list(range(0, 8192, 173)))
    _check(p, range(len(p.replicas)))


def test_large_shape_w64_reduced():
    # the W = 64 workload's prompt shape (median 2048 tokens, up to 32768, i.e.
    # 2048 blocks; 1024 prefix groups) and its concurrency C = 4096: the
    # chunked probe, 64 lanes of costs, the per-request slots and event heap in
    # global memory (4096 in flight do not fit beside 2048-block prompts in
    # shared memory) and the wide PoA solver (64 workers, one warp per window,
    # windows over the per-worker capacity).  Smaller caches and fewer
    # requests so that the oracle finishes in seconds.
    p = wk.plan("large", n_req=6000, replicas=[0, 8])
    p.K = 1 << 14
    assert all(r.C == 4096 for r in p.replicas)
    g = _check(p, range(len(p.replicas)))
    assert all(x["result"]["status"] == 0 for x in g)
    assert max(x["result"]["hashed_blocks"] for x in g) > 0


def test_load_spike_static_and_adaptive():
    # Experiment 3's load spike (C = 32 -> 128 -> 32 for 120 / 180 / 120 s, two
    # decode workers), static and adaptive replicas over three seeds, all in
    # one launch; the first regime switch times must agree too
    p = wk.plan("spike")
    g = _check(p, range(len(p.replicas)))
    for k, r in enumerate(p.replicas):
        fs = g[k]["result"]["first_switch_t"]
        if r.controller:
            assert fs > r.c_t1          # the adaptive replicas switch during the spike
        else:
            assert fs == -1.0


def _full_launch(p, flags=0, **ctx_fields):
    """One simulate_replicas call over the whole plan (the benchmark's launch
    configuration); records stay on the device."""
    traces = p.traces()
    ctx = rs.Context(W=p.W, K=p.K, theta1=p.theta1, theta2=p.theta2, **ctx_fields)
    bufs = [rs.device_trace(t) for t in traces]
    rows = sum(r.n_req for r in p.replicas)
    rec, t = rs.device_records(rows, p.W, with_kv=bool(ctx.cfg.tiered))
    res = rs.simulate_replicas(ctx.h, [b.desc() for b in bufs], rs.RS_MEM_DEVICE,
                               [rs.replica_params(r) for r in p.replicas], rec, flags)
    torch.cuda.synchronize()
    base = np.concatenate([[0], np.cumsum([r.n_req for r in p.replicas])]).astype(np.int64)
    return ctx, traces, res, t, base


def _rows(t, b0, n, W):
    d = {f: t[f][b0:b0 + n].cpu().numpy() for f in ("worker", "arrival", "start", "first_token",
                                                     "completion", "ttft", "nbt")}
    for f in ("n_frozen", "prefix"):
        d[f] = t[f][b0 * W:(b0 + n) * W].cpu().numpy().view(np.uint16).reshape(n, W)
    return d


def _prefix_equal(g, o, W):
    # a replica's first N requests do not depend on later ones: the full-size
    # run's first N records equal those of the oracle's N-request run
    assert np.array_equal(g["worker"], o["worker"])
    assert np.array_equal(g["prefix"], o["prefix"])
    assert np.array_equal(g["n_frozen"], o["n_frozen"])
    assert np.array_equal(g["nbt"], o["nbt"])
    for f in ("arrival", "start", "first_token", "completion", "ttft"):
        assert np.allclose(g[f], o[f], rtol=1e-12, atol=0), f


def test_p5d_full_size_prefix_of_sampled_replicas():
    # 256 replicas x 50 000 requests (two replicas per SM): every replica's
    # first 4000 requests checked on a sample
    p = wk.plan("p5d")
    ctx, traces, res, t, base = _full_launch(p)
    assert all(r.status == 0 for r in res)
    cfg = oracle_cfg(ctx, theta1=p.theta1, theta2=p.theta2)
    N = 4000
    for k in (0, 101, 255):
        r = p.replicas[k]
        rr = wk.Replica(**{**vars(r), "n_req": N})
        o = oracle_run(cfg, traces[r.trace], rr)
        _prefix_equal(_rows(t, int(base[k]), N, p.W), o, p.W)
    assert sum(x.regime_switches for x in res) > 0
    # one replica whole (C = 64, tau = 1: sampled decisions, controller on),
    # its PoA included
    k = 101
    r = p.replicas[k]
    assert r.tau == 1.0 and r.controller == 1
    g, o = _whole_equal(p, ctx, traces, res, t, base, k,
                        extra=("sampled", "near_ties", "exact_ties", "near_boundary", "ticks",
                               "regime_switches", "final_regime", "max_regime"))
    res_k = res[k].as_dict()
    assert res_k["sampled"] > 0 and res_k["ticks"] > 0
    assert list(res_k["ticks_in_regime"]) == list(o["summary"]["ticks_in_regime"])
    cfg = oracle_cfg(ctx, theta1=p.theta1, theta2=p.theta2)
    num, opt, cnt, tot = O.poa(cfg, o)
    assert res_k["n_windows"] == num.size
    assert abs(res_k["poa_total"] - tot) <= 1e-4 * tot
    ctx.close()


def test_grid_full_size_sampled_replicas():
    # 8192 replicas x 10 000 requests in one launch; sampled replicas whole,
    # PoA included
    p = wk.plan("grid")
    ctx, traces, res, t, base = _full_launch(p)
    assert all(r.status == 0 for r in res)
    cfg = oracle_cfg(ctx, theta1=p.theta1, theta2=p.theta2)
    for k in (0, 1, 4321, 8191):
        r = p.replicas[k]
        o = oracle_run(cfg, traces[r.trace], r)
        g = _rows(t, int(base[k]), r.n_req, p.W)
        _prefix_equal(g, o, p.W)
        res_k = res[k].as_dict()
        for f in ("n_routed", "hit_blocks", "inserted_blocks", "evicted_blocks", "exact_ties",
                  "near_ties"):
            assert res_k[f] == o["summary"][f], f
        _, _, _, tot = O.poa(cfg, o)
        assert abs(res_k["poa_total"] - tot) <= 1e-4 * tot
    ctx.close()


def _whole_equal(p, ctx, traces, res, t, base, k, extra=()):
    cfg = oracle_cfg(ctx, theta1=p.theta1, theta2=p.theta2)
    r = p.replicas[k]
    o = oracle_run(cfg, traces[r.trace], r)
    g = _rows(t, int(base[k]), r.n_req, p.W)
    _prefix_equal(g, o, p.W)
    res_k = res[k].as_dict()
    for f in ("n_routed", "hit_blocks", "inserted_blocks", "evicted_blocks", "first_evict_t",
              "rho_first_evict", "rho_end") + tuple(extra):
        assert res_k[f] == o["summary"][f], (f, res_k[f], o["summary"][f])
    return g, o


def test_frequency_eviction_p2d_full_size():
    # the p2d launch with every replica evicting by the frequency rule
    p = wk.plan("p2d")
    for r in p.replicas:
        r.eviction, r.freq_max, r.decay_s = rs.RS_EVICT_FREQ, 64, 1.0
    ctx, traces, res, t, base = _full_launch(p, flags=rs.RS_SIM_NO_POA)
    assert all(r.status == 0 for r in res)
    for k in (0, 37):
        _whole_equal(p, ctx, traces, res, t, base, k)
    assert sum(x.evicted_blocks for x in res) > 0
    ctx.close()


def test_game2_tiers_p2d_full_size():
    # the p2d launch with G2 = 64K and G3 = 128K blocks per worker beside the
    # 64K-block G1; the charge of every request compared
    p = wk.plan("p2d")
    ctx, traces, res, t, base = _full_launch(p, flags=rs.RS_SIM_NO_POA, tiered=1,
                                             tier_k2=p.K, tier_k3=2 * p.K, tier_node=1)
    assert all(r.status == 0 for r in res)
    for k in (5, 63):
        r = p.replicas[k]
        g, o = _whole_equal(p, ctx, traces, res, t, base, k,
                            extra=("kv_g1", "kv_g2", "kv_g3", "kv_remote", "kv_recompute",
                                   "kv_cost"))
        b0 = int(base[k])
        assert np.array_equal(t["kv_cost"][b0:b0 + r.n_req].cpu().numpy(), o["kv_cost"])
    assert sum(x.kv_g2 + x.kv_g3 for x in res) > 0
    ctx.close()


def test_probe_batch_in_the_bench_configuration():
    # the batch probe as aux.probe_batch runs it: a 64-worker router instance
    # of 65 536-block caches, the first 2 000 requests of p2d trace 0 routed,
    # the other 18 000 probed; every (request, worker) prefix bit-exact
    p = wk.plan("p2d")
    tr = p.traces()[0]
    W, K, nr = 64, 65536, 2000
    ctx = rs.Context(W=W, K=K, n_instances=1)
    ref = O.Router(O.OracleConfig(W=W, K=K), 1.0, 0.0, 0)
    d = rs.device_trace(tr)
    wo = torch.zeros(nr, dtype=torch.int32, device="cuda")
    rs.route_batch(ctx.h, 0, d.tokens, d.offsets, nr, d.out_len, wo)
    head = wk.Trace(tr.tokens, tr.offsets[:nr + 1], tr.release[:nr], tr.out_len[:nr],
                    tr.group[:nr])
    st, rw, _, _ = ref.route(0, head.tokens, head.offsets, head.out_len)
    assert st == 0 and np.array_equal(wo.cpu().numpy(), rw)
    m = tr.n_req - nr
    po = torch.full((m * W,), -1, dtype=torch.int32, device="cuda")
    rs.route_probe(ctx.h, 0, d.tokens, d.offsets[nr:], m, po)
    torch.cuda.synchronize()
    got = po.cpu().numpy().reshape(m, W)
    st, want = ref.probe(0, tr.tokens, tr.offsets[nr:])
    assert st == 0 and np.array_equal(got, want)
    assert got.mean() > 1.0
