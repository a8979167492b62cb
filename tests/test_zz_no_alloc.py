"""poa_estimate_noalloc: the PoA estimate for callers that cannot allocate
device memory (their GPU memory is owned by another allocator, or
cudaMalloc's device synchronisation is not acceptable on their path).

It must give the result of poa_estimate, the entry point that uses
library-allocated scratch, on consecutive calls that share its one static
scratch array; and refuse, before doing any work, a size beyond that array.
This file is collected last on purpose."""
import numpy as np
import pytest

from paper_2606_17081_gb300 import routesim as rs
from paper_2606_17081_gb300 import workloads as wk

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA device", allow_module_level=True)


def _simulated_records(ctx, seed, C, policy):
    spec = wk.TraceSpec(n_req=2500, len_kind="uniform", len_min=16, len_max=900, n_groups=8,
                        prefix_min=64, prefix_max=400, zipf_s=1.1, out_kind="uniform",
                        out_min=1, out_max=300)
    tr = wk.make_trace(spec, seed)
    rep = wk.Replica(0, C, policy, 0, 1.0 if policy == wk.POLICY_DYNAMO else 0.0, 0.0, seed,
                     tr.n_req)
    rec, t = rs.device_records(tr.n_req, ctx.W)
    d = rs.device_trace(tr)
    rs.simulate_replicas(ctx.h, [d.desc()], rs.RS_MEM_DEVICE, [rs.replica_params(rep)], rec,
                         rs.RS_SIM_NO_POA)
    return rec, t, tr.n_req


def test_noalloc_matches_poa_estimate_on_consecutive_calls():
    ctx = rs.Context(W=3, K=400)
    cases = [_simulated_records(ctx, 3, 256, wk.POLICY_DYNAMO),
             _simulated_records(ctx, 4, 24, wk.POLICY_LOADBAL)]
    for rec, keep, n in cases:        # two calls in a row on the shared static scratch
        maxw = n + 2
        ref_num, ref_opt, ref_cnt, ref_tot, ref_nw = rs.poa_estimate(ctx.h, rec, n, maxw)
        num = torch.full((maxw,), -1.0, dtype=torch.float64, device="cuda")
        opt = torch.full((maxw,), -1.0, dtype=torch.float64, device="cuda")
        cnt = torch.full((maxw,), -1, dtype=torch.int64, device="cuda")
        tot = torch.zeros(1, dtype=torch.float64, device="cuda")
        nw = torch.zeros(1, dtype=torch.int64, device="cuda")
        rs.poa_estimate_noalloc(ctx.cfg, rec, n, num, opt, cnt, maxw, tot, nw)
        torch.cuda.synchronize()
        assert int(nw.item()) == ref_nw > 0
        k = ref_nw
        assert np.array_equal(cnt.cpu().numpy()[:k], ref_cnt)
        assert np.allclose(num.cpu().numpy()[:k], ref_num, rtol=1e-12, atol=0)
        assert np.allclose(opt.cpu().numpy()[:k], ref_opt, rtol=1e-12, atol=0)
        assert abs(tot.item() - ref_tot) <= 1e-12 * ref_tot


def test_noalloc_rejects_sizes_beyond_its_array():
    ctx = rs.Context(W=3, K=16)
    rec, keep = rs.device_records(4, 3)
    tot = torch.zeros(1, dtype=torch.float64, device="cuda")
    nw = torch.zeros(1, dtype=torch.int64, device="cuda")
    with pytest.raises(rs.RoutesimError) as e:
        rs.poa_estimate_noalloc(ctx.cfg, rec, 5_000_000, None, None, None, 0, tot, nw)
    assert e.value.status == rs.RS_ERR_CAPACITY
