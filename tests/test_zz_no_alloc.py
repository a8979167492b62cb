"""poa_estimate_noalloc: the PoA estimate for callers that cannot allocate
device memory (their GPU memory is owned by another allocator, or
cudaMalloc's device synchronisation is not acceptable on their path).

It must give the result of poa_estimate, the entry point that uses
library-allocated scratch, on consecutive calls that share its one static
scratch array, on the narrow and the wide (W > 16) solver; honour the
caller's window capacity and NULL outputs; report records that span more
windows than the array holds with -1; and refuse, before doing any work, a
size beyond that array.  This file is collected last on purpose."""
import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import routesim as rs
from paper_2606_17081_gb300 import workloads as wk

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA device", allow_module_level=True)

BYTES = 32 * 1024 * 1024      # RS_NOALLOC_POA_BYTES


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


def _outputs(maxw):
    return (torch.full((max(maxw, 1),), -1.0, dtype=torch.float64, device="cuda"),
            torch.full((max(maxw, 1),), -1.0, dtype=torch.float64, device="cuda"),
            torch.full((max(maxw, 1),), -1, dtype=torch.int64, device="cuda"),
            torch.zeros(1, dtype=torch.float64, device="cuda"),
            torch.zeros(1, dtype=torch.int64, device="cuda"))


def _oracle_poa(ctx, t, n):
    rec = {f: t[f].cpu().numpy() for f in ("worker", "completion", "ttft", "nbt")}
    for f in ("n_frozen", "prefix"):
        rec[f] = t[f].cpu().numpy().view(np.uint16).reshape(n, ctx.W)
    return O.poa(O.OracleConfig(W=ctx.W, K=ctx.K), rec)


@pytest.mark.parametrize("W", [3, 17])
def test_noalloc_matches_poa_estimate_on_consecutive_calls(W):
    ctx = rs.Context(W=W, K=400)
    cases = [_simulated_records(ctx, 3, 256, wk.POLICY_DYNAMO),
             _simulated_records(ctx, 4, 24, wk.POLICY_LOADBAL)]
    for rec, keep, n in cases:        # two calls in a row on the shared static scratch
        maxw = n + 2
        ref_num, ref_opt, ref_cnt, ref_tot, ref_nw = rs.poa_estimate(ctx.h, rec, n, maxw)
        num, opt, cnt, tot, nw = _outputs(maxw)
        rs.poa_estimate_noalloc(ctx.cfg, rec, n, num, opt, cnt, maxw, tot, nw)
        torch.cuda.synchronize()
        assert int(nw.item()) == ref_nw > 0
        k = ref_nw
        assert np.array_equal(cnt.cpu().numpy()[:k], ref_cnt)
        assert np.allclose(num.cpu().numpy()[:k], ref_num, rtol=1e-12, atol=0)
        assert np.allclose(opt.cpu().numpy()[:k], ref_opt, rtol=1e-12, atol=0)
        assert abs(tot.item() - ref_tot) <= 1e-12 * ref_tot
        # and the oracle's Eq. (12) on the same records, directly
        o_num, o_opt, o_cnt, o_tot = _oracle_poa(ctx, keep, n)
        assert o_num.size == k and np.array_equal(cnt.cpu().numpy()[:k], o_cnt)
        assert np.allclose(opt.cpu().numpy()[:k], o_opt, rtol=1e-9, atol=0)
        assert abs(tot.item() - o_tot) <= 1e-4 * o_tot


def test_noalloc_window_capacity_and_null_outputs():
    ctx = rs.Context(W=3, K=400)
    rec, keep, n = _simulated_records(ctx, 5, 64, wk.POLICY_DYNAMO)
    ref_num, _, ref_cnt, ref_tot, ref_nw = rs.poa_estimate(ctx.h, rec, n, n + 2)
    assert ref_nw > 3
    num, opt, cnt, tot, nw = _outputs(ref_nw)
    rs.poa_estimate_noalloc(ctx.cfg, rec, n, num, opt, cnt, 3, tot, nw)
    torch.cuda.synchronize()
    assert int(nw.item()) == ref_nw                 # windows spanned, not written
    c = cnt.cpu().numpy()
    assert np.array_equal(c[:3], ref_cnt[:3]) and np.all(c[3:] == -1)
    assert np.all(num.cpu().numpy()[3:] == -1.0)
    _, _, _, tot2, nw2 = _outputs(1)
    rs.poa_estimate_noalloc(ctx.cfg, rec, n, None, None, None, 0, tot2, nw2)
    torch.cuda.synchronize()
    assert int(nw2.item()) == ref_nw and abs(tot2.item() - ref_tot) <= 1e-12 * ref_tot


def test_noalloc_reports_more_windows_than_its_array():
    # two rows whose completions are 2 * 10^8 windows apart: more windows than
    # the array holds beside the rows, so no estimate (-1)
    ctx = rs.Context(W=3, K=16)
    rec, t = rs.device_records(2, 3)
    t["worker"].copy_(torch.tensor([0, 1], dtype=torch.int32))
    t["completion"].copy_(torch.tensor([1.0, 1.0e9], dtype=torch.float64))
    t["ttft"].fill_(0.1)
    t["nbt"].fill_(1)
    num, opt, cnt, tot, nw = _outputs(4)
    rs.poa_estimate_noalloc(ctx.cfg, rec, 2, num, opt, cnt, 4, tot, nw)
    torch.cuda.synchronize()
    assert int(nw.item()) == -1


def test_noalloc_rejects_sizes_beyond_its_array():
    # accepted exactly while n (8 W + 60) + 4096 <= RS_NOALLOC_POA_BYTES
    W = 3
    nmax = (BYTES - 4096) // (8 * W + 60)
    ctx = rs.Context(W=W, K=16)
    rec, keep = rs.device_records(nmax + 1, W)      # no routed row: nothing to estimate
    num, opt, cnt, tot, nw = _outputs(1)
    rs.poa_estimate_noalloc(ctx.cfg, rec, nmax, None, None, None, 0, tot, nw)
    torch.cuda.synchronize()
    assert int(nw.item()) == 0
    for n in (nmax + 1, 5_000_000):
        with pytest.raises(rs.RoutesimError) as e:
            rs.poa_estimate_noalloc(ctx.cfg, rec, n, None, None, None, 0, tot, nw)
        assert e.value.status == rs.RS_ERR_CAPACITY
