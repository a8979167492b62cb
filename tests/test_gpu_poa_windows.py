"""PoA of Eq. (12) on sparse records: the records span far more 5-s windows
than they have rows (a slow Poisson client, long outputs), so every window the
records reach must get a slot.  The estimate of simulate_replicas, of
poa_estimate and of poa_estimate_noalloc must all equal the oracle's per
window (numerator, count, OPT) and in total."""
import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import routesim as rs
from paper_2606_17081_gb300 import workloads as wk

from gpu_helpers import gpu_run, oracle_cfg, oracle_run

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA device", allow_module_level=True)


def _sparse_trace(n, seed):
    spec = wk.TraceSpec(n_req=n, len_kind="uniform", len_min=16, len_max=600, n_groups=4,
                        prefix_min=32, prefix_max=200, zipf_s=None, out_kind="uniform",
                        out_min=1000, out_max=4000, rate=0.05)
    return wk.make_trace(spec, seed)


def _to_device(o, n, W):
    rec, t = rs.device_records(n, W)
    for f in ("worker", "completion", "ttft", "nbt"):
        t[f].copy_(torch.from_numpy(np.ascontiguousarray(o[f])))
    for f in ("n_frozen", "prefix"):
        t[f].copy_(torch.from_numpy(np.ascontiguousarray(o[f]).reshape(-1).view(np.int16)))
    return rec, t


@pytest.mark.parametrize("W,C", [(3, 4), (5, 64)])
def test_sparse_windows_match_oracle(W, C):
    tr = _sparse_trace(400, 60 + W)
    ctx = rs.Context(W=W, K=300)
    reps = [wk.Replica(0, C, wk.POLICY_DYNAMO, 0, 1.0, 0.0, 0, tr.n_req)]
    st, g = gpu_run(ctx, [tr], reps)
    assert st == 0
    cfg = oracle_cfg(ctx)
    o = oracle_run(cfg, tr, reps[0])
    num, opt, cnt, tot = O.poa(cfg, o)
    assert num.size > 3 * (tr.n_req + 2)         # far more windows than rows
    res = g[0]["result"]
    assert res["n_windows"] == num.size
    assert abs(res["poa_total"] - tot) <= 1e-9 * tot
    rec, keep = _to_device(o, tr.n_req, W)
    gn, go, gc, gt, nw = rs.poa_estimate(ctx.h, rec, tr.n_req, num.size)
    assert nw == num.size and np.array_equal(gc, cnt)
    assert np.allclose(gn, num, rtol=1e-12, atol=0)
    assert np.allclose(go, opt, rtol=1e-12, atol=0)
    assert abs(gt - tot) <= 1e-12 * tot
    # the allocation-free entry point: the windows take what the rows leave
    cap = num.size
    dn = torch.full((cap,), -1.0, dtype=torch.float64, device="cuda")
    do = torch.full((cap,), -1.0, dtype=torch.float64, device="cuda")
    dc = torch.full((cap,), -1, dtype=torch.int64, device="cuda")
    dt = torch.zeros(1, dtype=torch.float64, device="cuda")
    dw = torch.zeros(1, dtype=torch.int64, device="cuda")
    rs.poa_estimate_noalloc(ctx.cfg, rec, tr.n_req, dn, do, dc, cap, dt, dw)
    torch.cuda.synchronize()
    assert int(dw.item()) == num.size
    assert np.array_equal(dc.cpu().numpy(), cnt)
    assert np.allclose(dn.cpu().numpy(), num, rtol=1e-12, atol=0)
    assert np.allclose(do.cpu().numpy(), opt, rtol=1e-12, atol=0)
    assert abs(dt.item() - tot) <= 1e-12 * tot


def test_windows_far_apart_and_empty_records():
    # three routed rows thousands of windows apart; and no routed row at all
    W = 2
    ctx = rs.Context(W=W, K=16)
    cfg = oracle_cfg(ctx)
    o = {"worker": np.array([0, -1, 1, 0], np.int32),
         "completion": np.array([1.0, 7.0, 52_345.5, 9_999_999.0]),
         "ttft": np.array([0.1, 0.2, 0.3, 0.4]),
         "nbt": np.array([4, 1, 8, 2], np.int32),
         "n_frozen": np.array([[1, 2], [3, 4], [5, 6], [7, 8]], np.uint16),
         "prefix": np.array([[0, 1], [0, 0], [8, 2], [1, 1]], np.uint16)}
    num, opt, cnt, tot = O.poa(cfg, o)
    assert num.size == 2_000_000
    rec, keep = _to_device(o, 4, W)
    gn, go, gc, gt, nw = rs.poa_estimate(ctx.h, rec, 4, num.size)
    assert nw == num.size and np.array_equal(gc, cnt)
    assert np.allclose(gn, num, rtol=1e-12, atol=0) and np.allclose(go, opt, rtol=1e-12, atol=0)
    assert abs(gt - tot) <= 1e-12 * tot
    o["worker"][:] = -1
    rec, keep = _to_device(o, 4, W)
    gn, go, gc, gt, nw = rs.poa_estimate(ctx.h, rec, 4, 4)
    assert nw == 0 and gt == 0.0
