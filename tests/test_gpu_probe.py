"""Parity of the batch probe (route_probe) through the C ABI with the oracle
router: after routed batches, every (request, worker) prefix of a probed batch
bit-exact; the probe changes no state (routing afterwards matches the oracle
and the caches dump equal); prompts longer than the cache, empty prompts,
several instances, and a batch larger than one wave of the grid."""
import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import routesim as rs
from paper_2606_17081_gb300 import workloads as wk

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA device", allow_module_level=True)


def _trace(n, seed, lo=0, hi=700, groups=6):
    spec = wk.TraceSpec(n_req=n, len_kind="uniform", len_min=lo, len_max=hi, n_groups=groups,
                        prefix_min=16, prefix_max=300, zipf_s=1.1, out_kind="uniform",
                        out_min=1, out_max=300)
    return wk.make_trace(spec, seed)


def _sub(tr, lo, hi):
    return wk.Trace(tr.tokens, tr.offsets[lo:hi + 1], tr.release[lo:hi], tr.out_len[lo:hi],
                    tr.group[lo:hi])


def _route(ctx, ref, inst, sub, W):
    d = rs.device_trace(sub)
    n = sub.n_req
    wo = torch.zeros(n, dtype=torch.int32, device="cuda")
    rs.route_batch(ctx.h, inst, d.tokens, d.offsets, n, d.out_len, wo)
    st, rw, _, _ = ref.route(inst, sub.tokens, sub.offsets, sub.out_len)
    assert st == 0
    assert np.array_equal(wo.cpu().numpy(), rw)


def _probe(ctx, inst, sub, W):
    d = rs.device_trace(sub)
    n = sub.n_req
    po = torch.full((max(n, 1) * W,), -7, dtype=torch.int32, device="cuda")
    rs.route_probe(ctx.h, inst, d.tokens, d.offsets, n, po)
    torch.cuda.synchronize()
    return po.cpu().numpy()[: n * W].reshape(n, W)


@pytest.mark.parametrize("W,K,tau", [(3, 64, 0.0), (5, 300, 0.6), (2, 45, 0.0)])
def test_probe_matches_oracle(W, K, tau):
    tr = _trace(700, 21 + W)
    ctx = rs.Context(W=W, K=K, n_instances=2, tau=tau, omega=1.0, seed=13)
    ref = O.Router(O.OracleConfig(W=W, K=K), 1.0, tau, 13, n_instances=2)
    _route(ctx, ref, 0, _sub(tr, 0, 300), W)
    _route(ctx, ref, 1, _sub(tr, 300, 420), W)
    for inst in (0, 1):
        probed = _sub(tr, 420, 700)
        got = _probe(ctx, inst, probed, W)
        st, want = ref.probe(inst, probed.tokens, probed.offsets)
        assert st == 0
        assert np.array_equal(got, want), inst
        assert got.max() > 0
    # nothing changed: the next routed batch and the caches agree with the oracle
    _route(ctx, ref, 0, _sub(tr, 420, 560), W)
    for j in range(W):
        assert np.array_equal(rs.route_cache_dump(ctx.h, 0, 0, j, K), ref.cache(0, j))
    assert np.array_equal(rs.route_active(ctx.h, 0, W), ref.active(0))


def test_probe_long_and_empty_prompts():
    W, K = 3, 40
    tr = _trace(400, 5, lo=0, hi=600)                       # up to 37 blocks: routable
    ctx = rs.Context(W=W, K=K, n_instances=1)
    ref = O.Router(O.OracleConfig(W=W, K=K), 1.0, 0.0, 0)
    _route(ctx, ref, 0, _sub(tr, 0, 250), W)
    # probe-only batch: prompts up to 3000 tokens (longer than the cache) and
    # empty or sub-block prompts
    lng = _trace(300, 6, lo=0, hi=3000)
    got = _probe(ctx, 0, lng, W)
    st, want = ref.probe(0, lng.tokens, lng.offsets)
    assert st == 0 and np.array_equal(got, want)
    nb = np.diff(lng.offsets) // 16
    assert (got <= np.minimum(nb, K)[:, None]).all()
    assert (nb > K).any() and (nb == 0).any()


def test_probe_large_batch_grid_stride():
    # 20 000 requests x 16 workers = 320 000 pairs: more than 152 x 8 x 256
    # threads, so the grid-stride loop runs twice on a GB300
    W, K = 16, 2048
    tr = _trace(21000, 8, lo=0, hi=1200, groups=32)
    ctx = rs.Context(W=W, K=K, n_instances=1)
    ref = O.Router(O.OracleConfig(W=W, K=K), 1.0, 0.0, 0)
    _route(ctx, ref, 0, _sub(tr, 0, 1000), W)
    probed = _sub(tr, 1000, 21000)
    got = _probe(ctx, 0, probed, W)
    st, want = ref.probe(0, probed.tokens, probed.offsets)
    assert st == 0 and np.array_equal(got, want)


def test_probe_arguments():
    ctx = rs.Context(W=2, K=16, n_instances=1)
    tr = _trace(4, 1)
    d = rs.device_trace(tr)
    po = torch.zeros(8, dtype=torch.int32, device="cuda")
    rs.route_probe(ctx.h, 0, d.tokens, d.offsets, 0, po)             # nothing to do
    for inst, n, out in ((1, 4, po), (-1, 4, po), (0, -1, po), (0, 4, None)):
        with pytest.raises(rs.RoutesimError) as e:
            rs.route_probe(ctx.h, inst, d.tokens, d.offsets, n, out)
        assert e.value.status == rs.RS_ERR_INVALID
