"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Bar: block hashes, decisions, cached-prefix lengths, frozen loads, Eq. (1)
costs and final cache contents (LRU order) bit-exact; per-request times
within 1e-12 relative (both sides round every fp64 operation in the same
order, so they agree exactly in practice); accumulated latencies within 1e-9
and PoA values within 1e-4 relative.
"""
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


def _rand_trace(n, seed, len_lo=0, len_hi=700, groups=6, rate=None, out_hi=300):
    spec = wk.TraceSpec(n_req=n, len_kind="uniform", len_min=len_lo, len_max=len_hi,
                        n_groups=groups, prefix_min=16, prefix_max=300, zipf_s=1.1,
                        out_kind="uniform", out_min=0, out_max=out_hi, rate=rate)
    return wk.make_trace(spec, seed)


# ------------------------------------------------------------------ block hash (K1)

@pytest.mark.parametrize("seed,n,lo,hi", [(0, 1, 0, 15), (1, 333, 0, 700), (2, 2000, 16, 5000),
                                          (3, 64, 511, 513)])
def test_block_hash_bit_exact(seed, n, lo, hi):
    tr = _rand_trace(n, seed, len_lo=lo, len_hi=hi)
    ctx = rs.Context(W=2, K=64)
    d = rs.device_trace(tr)
    nh = int(tr.offsets[-1]) // 16
    out = torch.zeros(max(nh, 1), dtype=torch.int64, device="cuda")
    rs.route_hash_blocks(ctx.h, d.tokens, d.offsets, tr.n_req, out)
    torch.cuda.synchronize()
    got = out.cpu().numpy().view(np.uint64)[:nh]
    ref = O.hash_blocks(tr.tokens, tr.offsets)
    mask = np.zeros(nh, bool)
    for i in range(tr.n_req):
        b = int(tr.offsets[i]) // 16
        mask[b:b + (int(tr.offsets[i + 1] - tr.offsets[i]) // 16)] = True
    assert np.array_equal(got[mask], ref[mask])


def test_block_hash_large_ragged():
    # several tiles of warps, every start alignment, long prompts
    tr = wk.make_trace(wk.TraceSpec(n_req=5000, len_max=8192), 11)
    ctx = rs.Context(W=2, K=64)
    d = rs.device_trace(tr)
    nh = int(tr.offsets[-1]) // 16
    out = torch.zeros(nh, dtype=torch.int64, device="cuda")
    rs.route_hash_blocks(ctx.h, d.tokens, d.offsets, tr.n_req, out)
    torch.cuda.synchronize()
    got = out.cpu().numpy().view(np.uint64)
    ref = O.hash_blocks(tr.tokens, tr.offsets)
    starts = tr.offsets[:-1] // 16
    lens = np.diff(tr.offsets) // 16
    idx = np.concatenate([np.arange(s, s + l) for s, l in zip(starts, lens)])
    assert np.array_equal(got[idx], ref[idx])
    assert set(int(o) % 4 for o in tr.offsets[:-1]) == {0, 1, 2, 3}


# ------------------------------------------------------------------ simulation (K3)

def test_tiny_config_full():
    p = wk.plan("tiny")
    tr = p.traces()[0]
    ctx = rs.Context(W=p.W, K=p.K)
    st, g = gpu_run(ctx, [tr], p.replicas)
    assert st == 0
    cfg = oracle_cfg(ctx)
    o = oracle_run(cfg, tr, p.replicas[0], want_cache=True)
    assert_replica_equal(g[0], o, p.W)
    for j in range(p.W):
        assert np.array_equal(rs.route_cache_dump(ctx.h, 1, 0, j, p.K), o["cache"][j])
    _, _, _, tot = O.poa(cfg, o)
    assert abs(g[0]["result"]["poa_total"] - tot) <= 1e-4 * tot


@pytest.mark.parametrize("K,C,tau,policy,W", [
    (48, 24, 0.0, wk.POLICY_DYNAMO, 3),      # eviction-heavy, exact ties
    (40, 60, 0.7, wk.POLICY_DYNAMO, 3),      # sampling + slow-path evictions
    (200, 300, 0.0, wk.POLICY_LOADBAL, 3),   # queueing (C > W * 63)
    (64, 8, 1.0, wk.POLICY_DYNAMO, 6),
    (45, 5, 0.0, wk.POLICY_DYNAMO, 1),       # single FIFO server
    (1000, 1, 0.3, wk.POLICY_DYNAMO, 5),     # C = 1
])
def test_sim_parity_small(K, C, tau, policy, W):
    tr = _rand_trace(700, 7 + K, len_hi=640)
    om = 1.0 if policy == wk.POLICY_DYNAMO else 0.0
    reps = [wk.Replica(0, C, policy, 0, om, tau, 99, tr.n_req)]
    ctx = rs.Context(W=W, K=K)
    st, g = gpu_run(ctx, [tr], reps)
    assert st == 0
    cfg = oracle_cfg(ctx)
    o = oracle_run(cfg, tr, reps[0], want_cache=True)
    assert_replica_equal(g[0], o, W)
    for j in range(W):
        assert np.array_equal(rs.route_cache_dump(ctx.h, 1, 0, j, K), o["cache"][j])
    if K < 100:
        assert g[0]["result"]["evicted_blocks"] > 0


def test_sim_slow_path_and_rebuilds_exercised():
    # small caches with long shared prefixes put present blocks at the LRU end
    spec = wk.TraceSpec(n_req=3000, len_kind="uniform", len_min=100, len_max=900, n_groups=40,
                        prefix_min=200, prefix_max=800, zipf_s=0.6, out_kind="uniform",
                        out_min=1, out_max=64)
    tr = wk.make_trace(spec, 5)
    ctx = rs.Context(W=2, K=120)
    reps = [wk.Replica(0, 16, wk.POLICY_DYNAMO, 0, 2.0, 0.0, 0, tr.n_req)]
    st, g = gpu_run(ctx, [tr], reps)
    assert st == 0
    o = oracle_run(oracle_cfg(ctx), tr, reps[0], want_cache=True)
    assert_replica_equal(g[0], o, 2)
    r = g[0]["result"]
    assert r["slow_path"] > 0 and r["rebuilds"] > 0
    for j in range(2):
        assert np.array_equal(rs.route_cache_dump(ctx.h, 1, 0, j, 120), o["cache"][j])


def test_sim_controller_parity():
    spec = wk.TraceSpec(n_req=6000, n_groups=16, prefix_min=64, prefix_max=256,
                        len_median=256, len_max=1024)
    tr = wk.make_trace(spec, 2)
    reps = [wk.Replica(0, 600, wk.POLICY_DYNAMO, 1, 1.0, 0.0, 1, tr.n_req),
            wk.Replica(0, 150, wk.POLICY_DYNAMO, 1, 1.0, 0.5, 2, tr.n_req),
            wk.Replica(0, 600, wk.POLICY_LOADBAL, 1, 0.0, 0.0, 3, tr.n_req)]
    ctx = rs.Context(W=3, K=4096)
    st, g = gpu_run(ctx, [tr], reps)
    assert st == 0
    cfg = oracle_cfg(ctx)
    for k, r in enumerate(reps):
        o = oracle_run(cfg, tr, r)
        assert_replica_equal(g[k], o, 3)
    assert g[0]["result"]["max_regime"] == 2 and g[0]["result"]["regime_switches"] >= 2


def test_sim_many_replicas_one_launch():
    trs = [_rand_trace(900, s, len_hi=900, rate=(None if s % 2 else 30.0)) for s in range(3)]
    reps = []
    for k in range(24):
        pol = wk.POLICY_DYNAMO if k % 3 else wk.POLICY_LOADBAL
        reps.append(wk.Replica(k % 3, [4, 32, 200][k % 3], pol, k % 2, 1.0 if pol == 0 else 0.0,
                               [0.0, 0.5][k % 2], k, 900 - 37 * (k % 5)))
    ctx = rs.Context(W=4, K=300)
    st, g = gpu_run(ctx, trs, reps)
    assert st == 0
    cfg = oracle_cfg(ctx)
    for k, r in enumerate(reps):
        assert_replica_equal(g[k], oracle_run(cfg, trs[r.trace], r), 4)


def test_host_traces_equal_device_traces():
    tr = _rand_trace(500, 21)
    reps = [wk.Replica(0, 20, wk.POLICY_DYNAMO, 0, 1.0, 0.4, 5, tr.n_req)]
    ctx = rs.Context(W=3, K=90)
    _, gd = gpu_run(ctx, [tr], reps, rs.RS_MEM_DEVICE)
    _, gh = gpu_run(ctx, [tr], reps, rs.RS_MEM_HOST)
    for f in ("worker", "prefix", "ttft", "completion"):
        assert np.array_equal(gd[0][f], gh[0][f])


def test_edge_cases():
    tr = _rand_trace(50, 31, len_lo=0, len_hi=40)      # empty and sub-block prompts
    ctx = rs.Context(W=2, K=8)
    reps = [wk.Replica(0, 3, wk.POLICY_DYNAMO, 0, 1.0, 0.0, 0, 50),
            wk.Replica(0, 3, wk.POLICY_DYNAMO, 0, 1.0, 0.0, 0, 0)]
    st, g = gpu_run(ctx, [tr], reps)
    assert st == 0
    assert_replica_equal(g[0], oracle_run(oracle_cfg(ctx), tr, reps[0]), 2)
    assert g[1]["result"]["n_routed"] == 0 and g[1]["result"]["status"] == 0
    # a prompt longer than a cache: capacity error on both sides
    tr2 = _rand_trace(20, 32, len_lo=200, len_hi=300)
    rep = [wk.Replica(0, 3, wk.POLICY_DYNAMO, 0, 1.0, 0.0, 0, 20)]
    st, g = gpu_run(ctx, [tr2], rep)
    assert st == rs.RS_ERR_CAPACITY == g[0]["result"]["status"]
    assert oracle_run(oracle_cfg(ctx), tr2, rep[0])["status"] == O.ERR_CAPACITY
    # invalid arguments are rejected before any launch
    for bad in (wk.Replica(0, 0, 0, 0, 1.0, 0.0, 0, 5), wk.Replica(3, 2, 0, 0, 1.0, 0.0, 0, 5),
                wk.Replica(0, 2, 0, 0, -1.0, 0.0, 0, 5), wk.Replica(0, 2, 7, 0, 1.0, 0.0, 0, 5),
                wk.Replica(0, 2, 0, 0, 1.0, 0.0, 0, 51)):
        st, _ = gpu_run(ctx, [tr], [bad])
        assert st == rs.RS_ERR_INVALID


# ------------------------------------------------------------------ PoA (K4)

# W = 3 and W = 6 run the solver compiled for exactly that many workers, the
# others the one compiled for up to 16; the selfish replicas' windows bind
# their capacity (thousands of augmentations)
@pytest.mark.parametrize("W,C", [(3, 256), (6, 512), (5, 320), (12, 768)])
def test_poa_matches_oracle_per_window(W, C):
    tr = _rand_trace(3000, 41, len_hi=900)
    reps = [wk.Replica(0, C, wk.POLICY_DYNAMO, 0, 1.0, 0.0, 0, tr.n_req),
            wk.Replica(0, 8 * W, wk.POLICY_LOADBAL, 0, 0.0, 0.0, 0, tr.n_req)]
    ctx = rs.Context(W=W, K=500)
    st, g = gpu_run(ctx, [tr], reps)
    assert st == 0
    cfg = oracle_cfg(ctx)
    for k, r in enumerate(reps):
        o = oracle_run(cfg, tr, r)
        num, opt, cnt, tot = O.poa(cfg, o)
        assert abs(g[k]["result"]["poa_total"] - tot) <= 1e-4 * tot
        assert g[k]["result"]["n_windows"] == num.size
        # per-window values through poa_estimate on the same records
        rec, t = rs.device_records(tr.n_req, W)
        for f in ("worker", "completion", "ttft", "nbt"):
            t[f].copy_(torch.from_numpy(np.ascontiguousarray(o[f])))
        for f in ("n_frozen", "prefix"):
            t[f].copy_(torch.from_numpy(o[f].reshape(-1).view(np.int16)))
        gn, go, gc, gt, nw = rs.poa_estimate(ctx.h, rec, tr.n_req, num.size + 5)
        assert nw == num.size and np.array_equal(gc, cnt)
        assert np.allclose(gn, num, rtol=1e-12, atol=0)
        nz = cnt > 0
        assert np.allclose(go[nz], opt[nz], rtol=1e-9, atol=0)
        assert abs(gt - tot) <= 1e-9 * tot


@pytest.mark.parametrize("W", [17, 40, 64])
def test_poa_wide_solver_per_window(W):
    # more workers than the per-warp solver holds: four cheap workers take
    # most requests of every window far over the capacity, so that most
    # requests are put back along augmenting paths through the other workers
    rng = np.random.default_rng(300 + W)
    n = 3000
    ctx = rs.Context(W=W, K=16)
    cfg = oracle_cfg(ctx)
    nbt = rng.integers(1, 200, n).astype(np.int32)
    nf = rng.integers(24, 63, (n, W))
    nf[:, :4] = rng.integers(0, 6, (n, 4))
    pf = np.minimum(rng.integers(0, 200, (n, W)), nbt[:, None])
    o = {"worker": rng.integers(0, W, n).astype(np.int32),
         "completion": rng.uniform(0.0, 3.5 * cfg.poa_window, n),
         "ttft": rng.uniform(0.01, 0.5, n),
         "nbt": nbt,
         "n_frozen": nf.astype(np.uint16),
         "prefix": pf.astype(np.uint16)}
    o["worker"][::97] = -1          # a few unrouted rows
    num, opt, cnt, tot = O.poa(cfg, o)
    assert num.size == 4 and cnt.min() > 4 * 64
    rec, t = rs.device_records(n, W)
    for f in ("worker", "completion", "ttft", "nbt"):
        t[f].copy_(torch.from_numpy(np.ascontiguousarray(o[f])))
    for f in ("n_frozen", "prefix"):
        t[f].copy_(torch.from_numpy(o[f].reshape(-1).view(np.int16)))
    gn, go, gc, gt, nw = rs.poa_estimate(ctx.h, rec, n, num.size + 2)
    assert nw == num.size and np.array_equal(gc, cnt)
    assert np.allclose(gn, num, rtol=1e-12, atol=0)
    assert np.allclose(go, opt, rtol=1e-9, atol=0)
    assert abs(gt - tot) <= 1e-9 * tot


def test_poa_binding_capacity_on_gpu():
    F1 = 0.005 + 0.020 + 0.010 / 63 ** 2
    F2 = 0.010 + 0.020 + 0.010 / 62 ** 2
    n = 130
    ctx = rs.Context(W=2, K=16)
    rec, t = rs.device_records(n, 2)
    t["worker"].zero_()
    t["completion"].fill_(0.5)
    t["ttft"].fill_(0.1)
    t["nbt"].fill_(3)
    t["n_frozen"].copy_(torch.tensor([1, 2] * n, dtype=torch.int16))
    t["prefix"].zero_()
    gn, go, gc, gt, nw = rs.poa_estimate(ctx.h, rec, n, 4)
    assert nw == 1 and gc[0] == n
    assert abs(go[0] - (65 * F1 + 65 * F2)) < 1e-12


# ------------------------------------------------------------------ live router

@pytest.mark.parametrize("tau,K", [(0.0, 64), (0.6, 40)])
def test_route_batch_parity(tau, K):
    tr = _rand_trace(400, 51, len_hi=500)
    W = 3
    ctx = rs.Context(W=W, K=K, n_instances=2, tau=tau, omega=1.0, seed=77)
    ref = O.Router(O.OracleConfig(W=W, K=K), 1.0, tau, 77, n_instances=2)
    rng = np.random.default_rng(0)
    for inst in (1, 0):
        for lo, hi in ((0, 150), (150, 151), (151, 400)):
            sub = wk.Trace(tr.tokens, tr.offsets[lo:hi + 1], tr.release[lo:hi], tr.out_len[lo:hi],
                           tr.group[lo:hi])
            d = rs.device_trace(sub)
            n = hi - lo
            wo = torch.zeros(n, dtype=torch.int32, device="cuda")
            co = torch.zeros(n * W, dtype=torch.float32, device="cuda")
            po = torch.zeros(n * W, dtype=torch.int32, device="cuda")
            rs.route_batch(ctx.h, inst, d.tokens, d.offsets, n, d.out_len, wo, co, po)
            st, rw, rc, rp = ref.route(inst, sub.tokens, sub.offsets, sub.out_len)
            assert st == 0
            assert np.array_equal(wo.cpu().numpy(), rw)
            assert np.array_equal(co.cpu().numpy().reshape(n, W), rc)
            assert np.array_equal(po.cpu().numpy().reshape(n, W), rp)
            # release a random subset of what was routed
            k = int(rng.integers(0, n + 1))
            blocks = ((np.diff(sub.offsets) + sub.out_len + 15) // 16).astype(np.int32)[:k]
            wd = torch.from_numpy(rw[:k].copy()).cuda()
            bd = torch.from_numpy(blocks).cuda()
            rs.route_release(ctx.h, inst, wd, bd, k)
            ref.release(inst, rw[:k], blocks)
            assert np.array_equal(rs.route_active(ctx.h, inst, W), ref.active(inst))
        for j in range(W):
            assert np.array_equal(rs.route_cache_dump(ctx.h, 0, inst, j, K), ref.cache(inst, j))


def test_route_release_rejects_bad_worker():
    ctx = rs.Context(W=2, K=16, n_instances=1)
    wd = torch.tensor([0, 5, 1], dtype=torch.int32, device="cuda")
    bd = torch.tensor([1, 1, 1], dtype=torch.int32, device="cuda")
    with pytest.raises(rs.RoutesimError) as e:
        rs.route_release(ctx.h, 0, wd, bd, 3)
    assert e.value.status == rs.RS_ERR_INVALID
    assert np.array_equal(rs.route_active(ctx.h, 0, 2), [0, 0])


@pytest.mark.gpu
@pytest.mark.parametrize("W", [3, 5])
def test_static_policies_and_static_poa(W):
    # round robin, uniform random and power of two choices (the routing
    # baselines of §9), below and above saturation (C = 256 > 63 W for W = 3)
    spec = wk.TraceSpec(n_req=2500, n_groups=16, prefix_min=64, prefix_max=512,
                        len_median=512, len_max=4096, out_median=128, out_max=1024)
    tr = wk.make_trace(spec, 11)
    reps = []
    for k, (pol, om) in enumerate([(wk.POLICY_ROUNDROBIN, 1.0), (wk.POLICY_RANDOM, 1.0),
                                   (wk.POLICY_P2C, 0.0), (wk.POLICY_P2C, 1.0)]):
        for C in (8, 64, 256):
            reps.append(wk.Replica(0, C, pol, 0, om, 0.0, 100 + k, tr.n_req))
    ctx = rs.Context(W=W, K=8192)
    st, g = gpu_run(ctx, [tr], reps)
    assert st == 0
    cfg = oracle_cfg(ctx)
    for k, r in enumerate(reps):
        o = oracle_run(cfg, tr, r)
        assert_replica_equal(g[k], o, W)
        tot = O.poa(cfg, o)[3]
        sp = O.poa_static(cfg, o)
        res = g[k]["result"]
        assert abs(res["poa_total"] - tot) <= 1e-9 * tot
        assert abs(res["poa_static"] - sp) <= 1e-9 * sp
    if W == 3:   # queueing at C = 256: the observed estimate exceeds the static one
        sat = [g[k]["result"] for k, r in enumerate(reps) if r.C == 256]
        assert all(x["poa_total"] > x["poa_static"] for x in sat)


# W nb above the 2048 pairs the full probe captures: the prompts' cached
# prefixes come from the rounds of first-miss walks (four lookups in flight
# per thread with one replica per SM under LRU, one with two per SM or under
# frequency eviction), checked in both launch modes against the oracle
@pytest.mark.parametrize("nrep,freq", [(8, False), (160, False), (8, True)])
def test_long_prompts_first_miss_rounds(nrep, freq):
    spec = wk.TraceSpec(n_req=120, len_kind="uniform", len_min=4200, len_max=8000, n_groups=5,
                        prefix_min=1000, prefix_max=4000, zipf_s=0.8, out_kind="uniform",
                        out_min=1, out_max=200)
    tr = wk.make_trace(spec, 13)
    W = 8
    assert int((np.diff(tr.offsets) // 16).min()) * W > 2048
    ctx = rs.Context(W=W, K=1024)
    reps = [wk.Replica(0, 4 + (k % 5) * 8, wk.POLICY_DYNAMO if k % 2 == 0 else wk.POLICY_LOADBAL,
                       0, 1.0 if k % 2 == 0 else 0.0, 0.5 if k % 4 == 0 else 0.0, k, tr.n_req)
            for k in range(nrep)]
    if freq:
        for r in reps:
            r.eviction, r.freq_max, r.decay_s = rs.RS_EVICT_FREQ, 6, 2.0
    st, g = gpu_run(ctx, [tr], reps)
    assert st == 0
    cfg = oracle_cfg(ctx)
    for k in sorted({0, 1, nrep // 2 + 1, nrep - 1}):
        o = oracle_run(cfg, tr, reps[k])
        assert_replica_equal(g[k], o, W)
    assert max(x["result"]["evicted_blocks"] for x in g) > 0
