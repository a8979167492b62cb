"""The W = 64 workload at its own shape: 16 replicas x 10^6 requests, 2^20-block
LRU caches per worker, prompts up to 32 768 tokens from 1024 Zipf(1.0) prefix
groups, C = 4096.  Its 8 traces hold about 2.7 G tokens each, so the tokens
are produced on the device chunk by chunk by the seeded generator and hashed
there (S1, route_hash_blocks); simulate_replicas takes the traces by their
block hashes.  Checked here: the device generator equals the host one, the
streamed hashes equal the oracle's, a trace given by its hashes simulates
exactly as the same trace given by its tokens, and the whole launch returns
status 0 with sampled replicas equal to the oracle on their first 20 000
requests (a replica's first N requests do not depend on later ones)."""
import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import routesim as rs
from paper_2606_17081_gb300 import streaming as stm
from paper_2606_17081_gb300 import workloads as wk

from gpu_helpers import assert_replica_equal, gpu_run, oracle_cfg, oracle_run

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA device", allow_module_level=True)


def test_counter_tokens_device_equal_host():
    m = wk.plan("large").metas()[3]
    d = m.device("cuda")
    end = int(m.offsets[-1])
    for x0, n in ((0, 1 << 20), (int(m.offsets[654_321]) + 7, 3_000_001), (end - 1000, 1000)):
        out = torch.full((n,), -1, dtype=torch.int32, device="cuda")
        m.fill_device(d, x0, x0 + n, out)
        assert np.array_equal(out.cpu().numpy(), m.tokens(x0, x0 + n))


def test_streamed_hashes_equal_oracle():
    # small chunks: many rebased launches, chunk starts at every alignment
    p = wk.plan("large", n_req=3000)
    m = p.metas()[0]
    tr = p.traces()[0]
    ctx = rs.Context(W=p.W, K=64)
    b = stm.hash_streamed(ctx, m, chunk_tokens=50_000)
    torch.cuda.synchronize()
    got = b.hashes.cpu().numpy().view(np.uint64)
    ref = O.hash_blocks(tr.tokens, tr.offsets)
    starts = tr.offsets[:-1] // 16
    lens = np.diff(tr.offsets) // 16
    idx = np.concatenate([np.arange(s, s + l) for s, l in zip(starts, lens)])
    assert np.array_equal(got[idx], ref[idx])
    # and the same as hashing the whole batch of tokens at once
    d = rs.device_trace(tr)
    out = torch.zeros(int(tr.offsets[-1]) // 16 + 1, dtype=torch.int64, device="cuda")
    rs.route_hash_blocks(ctx.h, d.tokens, d.offsets, tr.n_req, out)
    torch.cuda.synchronize()
    assert np.array_equal(out.cpu().numpy().view(np.uint64)[idx], got[idx])


@pytest.mark.parametrize("mem", [rs.RS_MEM_DEVICE, rs.RS_MEM_HOST])
def test_prehashed_traces_equal_token_traces(mem):
    p = wk.plan("p2d", n_req=1500, replicas=[0, 5, 17, 63])
    traces = p.traces()
    ctx = rs.Context(W=p.W, K=600)
    st, g_tok = gpu_run(ctx, traces, p.replicas, trace_mem=mem, with_cost=True)
    assert st == 0
    descs, keep = [], []
    for tr in traces:
        h = torch.zeros(int(tr.offsets[-1]) // 16 + 1, dtype=torch.int64, device="cuda")
        d = rs.device_trace(tr)
        rs.route_hash_blocks(ctx.h, d.tokens, d.offsets, tr.n_req, h)
        torch.cuda.synchronize()
        if mem == rs.RS_MEM_HOST:
            hb = rs.host_trace(tr)
            b = rs.TraceBuffers(None, hb.offsets, hb.release, hb.out_len, tr.n_req,
                                h.cpu().pin_memory())
        else:
            b = rs.TraceBuffers(None, d.offsets, d.release, d.out_len, tr.n_req, h)
        keep.append((b, d))
        descs.append(b.desc())
    rows = sum(r.n_req for r in p.replicas)
    rec, t = rs.device_records(rows, p.W, with_cost=True)
    res = rs.simulate_replicas(ctx.h, descs, mem, [rs.replica_params(r) for r in p.replicas], rec)
    torch.cuda.synchronize()
    base = 0
    for k, r in enumerate(p.replicas):
        n = r.n_req
        for f in ("worker", "arrival", "completion", "ttft", "nbt"):
            assert np.array_equal(t[f][base:base + n].cpu().numpy(), g_tok[k][f]), f
        for f in ("prefix", "n_frozen", "cost"):
            a = t[f][base * p.W:(base + n) * p.W].cpu().numpy().reshape(n, p.W)
            assert np.array_equal(a.view(g_tok[k][f].dtype), g_tok[k][f]), f
        assert res[k].poa_total == g_tok[k]["result"]["poa_total"]
        base += n
    assert rs.route_last_timing(ctx.h).hashed_tokens == 0


def test_large_full_launch_sampled_prefixes():
    p = wk.plan("large")
    assert p.W == 64 and p.K == 1 << 20 and len(p.replicas) == 16
    assert all(r.n_req == 1_000_000 and r.C == 4096 for r in p.replicas)
    metas = p.metas()
    ctx = rs.Context(W=p.W, K=p.K, theta1=p.theta1, theta2=p.theta2)
    bufs = [stm.hash_streamed(ctx, m) for m in metas]
    assert max(int(np.diff(m.offsets).max()) for m in metas) == 32768
    rows = sum(r.n_req for r in p.replicas)
    rec, t = rs.device_records(rows, p.W)
    res = rs.simulate_replicas(ctx.h, [b.desc() for b in bufs], rs.RS_MEM_DEVICE,
                               [rs.replica_params(r) for r in p.replicas], rec)
    torch.cuda.synchronize()
    assert all(r.status == 0 and r.n_routed == 1_000_000 for r in res)
    assert sum(r.evicted_blocks for r in res) > 0          # the 2^20-block caches fill
    assert all(r.n_windows > 0 and np.isfinite(r.poa_total) and r.poa_total > 0 for r in res)
    cfg = oracle_cfg(ctx, theta1=p.theta1, theta2=p.theta2)
    N = 20000
    head = metas[0].trace(N)
    for k in (0, 8):               # trace 0 under the selfish and the coordinated policy
        r = p.replicas[k]
        assert r.trace == 0
        o = oracle_run(cfg, head, wk.Replica(**{**vars(r), "n_req": N}))
        b0 = k * r.n_req
        assert np.array_equal(t["worker"][b0:b0 + N].cpu().numpy(), o["worker"])
        for f in ("prefix", "n_frozen"):
            a = t[f][b0 * p.W:(b0 + N) * p.W].cpu().numpy().view(np.uint16).reshape(N, p.W)
            assert np.array_equal(a, o[f]), f
        assert np.array_equal(t["nbt"][b0:b0 + N].cpu().numpy(), o["nbt"])
        for f in ("arrival", "start", "first_token", "completion", "ttft"):
            assert np.allclose(t[f][b0:b0 + N].cpu().numpy(), o[f], rtol=1e-12, atol=0), f
    ctx.close()
