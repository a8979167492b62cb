"""Parity of the saturation-knee detector (§5.1 PoA-growth proposition, item 3;
Experiment 2) through the C ABI with the oracle: percentiles, divided
differences and knees bit-exact on the same records; on a simulated sweep,
the GPU simulation's records against the oracle simulation's."""
import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import routesim as rs
from paper_2606_17081_gb300 import workloads as wk

from gpu_helpers import oracle_cfg, oracle_run

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA device", allow_module_level=True)


def _same(a, b):
    a, b = np.asarray(a), np.asarray(b)
    return a.shape == b.shape and np.array_equal(np.isnan(a), np.isnan(b)) and \
        np.array_equal(a[~np.isnan(a)], b[~np.isnan(b)])


def _device_records(worker, ttft):
    n = max(worker.size, 1)
    rec, t = rs.device_records(n, 1)
    if worker.size:
        t["worker"].copy_(torch.from_numpy(worker))
        t["ttft"].copy_(torch.from_numpy(ttft))
    return rec, t


@pytest.mark.parametrize("pct", [1, 50, 99, 100])
def test_knee_bit_exact_on_ragged_records(pct):
    rng = np.random.default_rng(40 + pct)
    # replicas: empty, one row, all unrouted, heavy ties, large, ...
    sizes = [0, 1, 5, 300, 4096, 33333, 2, 17, 900, 64, 64, 1000, 7]
    rows = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int64)
    n = int(rows[-1])
    ttft = rng.lognormal(-2.0, 1.0, n)
    ttft[rows[3]:rows[4]] = np.round(ttft[rows[3]:rows[4]], 2)     # ties
    worker = rng.integers(-1, 3, n).astype(np.int32)
    worker[rows[2]:rows[3]] = -1                                     # routes nothing
    load = np.array([1, 2, 4, 8, 16, 32, 64, 3, 5, 9, 9, 1, 2], np.float64)
    # sweeps: 0..6 increasing, 7..8, 9..10 (equal loads: rejected), 11..12,
    # plus an empty one; replica 12 ends the last
    sweep_start = [0, 7, 9, 11, 11, 13]
    theta = 0.0
    ctx = rs.Context(W=1, K=16)
    rec, _ = _device_records(worker, ttft)
    g = rs.sweep_knee(ctx.h, rec, rows, load, sweep_start, pct=pct, theta=theta)
    o = O.sweep_knee(worker, ttft, rows, load, sweep_start, pct=pct, theta=theta)
    for k in ("stat", "d1", "d2", "knee_load"):
        assert _same(g[k], o[k]), k
    assert np.array_equal(g["knee_index"], o["knee_index"])
    assert o["knee_index"][2] == -2 and np.isnan(o["stat"][0]) and np.isnan(o["stat"][2])


def test_knee_rejects_bad_arguments():
    ctx = rs.Context(W=1, K=16)
    rec, _ = _device_records(np.zeros(4, np.int32), np.ones(4))
    rows = np.array([0, 2, 4], np.int64)
    for kw in ({"pct": 0}, {"pct": 101}, {"theta": float("nan")}):
        with pytest.raises(rs.RoutesimError):
            rs.sweep_knee(ctx.h, rec, rows, [1.0, 2.0], [0, 2], **kw)
    with pytest.raises(rs.RoutesimError):          # sweeps past the replicas
        rs.sweep_knee(ctx.h, rec, rows, [1.0, 2.0], [0, 3])
    with pytest.raises(rs.RoutesimError):          # rows decrease
        rs.sweep_knee(ctx.h, rec, np.array([0, 3, 2], np.int64), [1.0, 2.0], [0, 2])


def test_knee_of_a_simulated_concurrency_sweep():
    # Experiment 2's nine levels, static and adaptive, one seed, prefix of the trace
    p = wk.plan("sat", n_req=1500, replicas=list(range(18)))
    traces = p.traces()
    ctx = rs.Context(W=p.W, K=p.K, theta1=p.theta1, theta2=p.theta2)
    bufs = [rs.device_trace(t) for t in traces]
    n = sum(r.n_req for r in p.replicas)
    rec, _ = rs.device_records(n, p.W)
    rs.simulate_replicas(ctx.h, [b.desc() for b in bufs], rs.RS_MEM_DEVICE,
                         [rs.replica_params(r) for r in p.replicas], rec)
    rows = np.concatenate([[0], np.cumsum([r.n_req for r in p.replicas])]).astype(np.int64)
    load = np.array([r.C for r in p.replicas], np.float64)
    sw = wk.sweeps(p.replicas)
    assert sw == [0, 9, 18]
    cfg = oracle_cfg(ctx, theta1=p.theta1, theta2=p.theta2)
    os_ = [oracle_run(cfg, traces[r.trace], r) for r in p.replicas]
    ow = np.concatenate([o["worker"] for o in os_])
    ot = np.concatenate([o["ttft"] for o in os_])
    o = O.sweep_knee(ow, ot, rows, load, sw, pct=99, theta=0.0)
    # a threshold between two well-separated second differences
    d2 = np.sort(o["d2"][~np.isnan(o["d2"])])
    gaps = np.diff(d2)
    k = int(np.argmax(gaps))
    theta = 0.5 * (d2[k] + d2[k + 1])
    o = O.sweep_knee(ow, ot, rows, load, sw, pct=99, theta=theta)
    g = rs.sweep_knee(ctx.h, rec, rows, load, sw, pct=99, theta=theta)
    assert np.allclose(g["stat"], o["stat"], rtol=1e-12, atol=0)
    scale = np.nanmax(np.abs(o["stat"]))
    for f in ("d1", "d2"):
        assert np.array_equal(np.isnan(g[f]), np.isnan(o[f]))
        m = ~np.isnan(o[f])
        assert np.allclose(g[f][m], o[f][m], rtol=0, atol=1e-9 * scale)
    assert np.array_equal(g["knee_index"], o["knee_index"])
    # the P99 grows with the concurrency level on the static sweep
    assert o["stat"][8] > o["stat"][0]
