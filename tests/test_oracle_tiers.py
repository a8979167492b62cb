"""Pins of the Game 2 tiers (§4.2, Eq. kv-cost) in the oracle, against things
other than its code: routing sees G1, whose contents are those of an LRU
cache of K blocks (the LRU inclusion property); a replay keyed by prompt
content that keeps three separate tiers with demotion and promotion, and a
second replay with one recency stack cut into tier bands, both give the
oracle's per-request categories, costs and final caches; a hand-worked
two-worker sequence; rejected arguments."""
from collections import OrderedDict

import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import workloads as Wk


def _trace(n=500, seed=3, rate=40.0, groups=8):
    spec = Wk.TraceSpec(n_req=n, len_kind="uniform", len_min=1, len_max=400, n_groups=groups,
                        prefix_min=32, prefix_max=200, zipf_s=1.1, out_kind="uniform",
                        out_min=1, out_max=300, rate=rate)
    return Wk.make_trace(spec, seed)


def _content_ids(trace, block=16):
    table, ids = {}, []
    for i in range(trace.n_req):
        t = trace.tokens[trace.offsets[i]:trace.offsets[i + 1]]
        prev, row = -1, []
        for k in range(len(t) // block):
            key = (prev, t[k * block:(k + 1) * block].tobytes())
            if key not in table:
                table[key] = len(table)
            prev = table[key]
            row.append(prev)
        ids.append(row)
    return ids


def _tiered(W, K, k2, k3, node=1, **kw):
    return O.OracleConfig(W=W, K=K, tiered=1, tier_k2=k2, tier_k3=k3, tier_node=node, **kw)


@pytest.mark.parametrize("K,k2,k3,tau", [(48, 64, 200, 0.0), (90, 30, 0, 0.7), (40, 0, 60, 0.0)])
def test_g1_is_the_lru_cache_of_K_blocks(K, k2, k3, tau):
    tr = _trace()
    plain = O.simulate(O.OracleConfig(W=3, K=K), tr, 24, tau=tau, seed=5, want_cache=True)
    tier = O.simulate(_tiered(3, K, k2, k3), tr, 24, tau=tau, seed=5, want_cache=True)
    assert plain["status"] == tier["status"] == 0
    for f in ("worker", "prefix", "ttft", "completion"):
        assert np.array_equal(plain[f], tier[f]), f
    assert plain["summary"]["hit_blocks"] == tier["summary"]["hit_blocks"]
    for j in range(3):
        g1 = plain["cache"][j]
        assert np.array_equal(tier["cache"][j][-len(g1):], g1)   # the stack's top K
    assert tier["summary"]["first_evict_t"] == plain["summary"]["first_evict_t"]


def _replays(tr, r, cfg):
    """Categories per request from (a) three tiers with demotion and
    promotion and (b) one recency stack cut into bands; final stacks."""
    W, K, k2, k3 = cfg.W, cfg.K, cfg.tier_k2, cfg.tier_k3
    caps = [K, k2, k3]
    ids = _content_ids(tr)
    tiers = [[OrderedDict() for _ in range(3)] for _ in range(W)]     # least recent first
    stacks = [OrderedDict() for _ in range(W)]
    al, dn, df, gam = cfg.tier_alpha, cfg.tier_d_near, cfg.tier_d_far, cfg.tier_gamma

    def tier_a(j, b):
        for t in range(3):
            if b in tiers[j][t]:
                return t + 1
        return 0

    def tier_b(j, b):
        if b not in stacks[j]:
            return 0
        rank = list(reversed(stacks[j])).index(b)          # 0 = most recent
        return 1 if rank < K else (2 if rank < K + k2 else 3)

    out = []
    dropped = 0
    for i in range(tr.n_req):
        s = int(r["worker"][i])
        cnt = [0] * 10
        for b in ids[i]:
            ta, tb = tier_a(s, b), tier_b(s, b)
            assert ta == tb
            if ta:
                cnt[ta - 1] += 1
                continue
            best, cat = np.inf, 9
            for rr in (0, 1):
                for q in (1, 2, 3):
                    has = any(tier_a(j, b) == q for j in range(W)
                              if j != s and ((j // cfg.tier_node == s // cfg.tier_node) == (rr == 0)))
                    if has and (dn if rr == 0 else df) + al[q - 1] < best:
                        best, cat = (dn if rr == 0 else df) + al[q - 1], 3 + 3 * rr + (q - 1)
            cnt[cat] += 1
        c = al[0] * cnt[0]
        c = c + al[1] * cnt[1]
        c = c + al[2] * cnt[2]
        for q in range(3):
            c = c + (dn + al[q]) * cnt[3 + q]
        for q in range(3):
            c = c + (df + al[q]) * cnt[6 + q]
        c = c + gam * cnt[9]
        out.append((cnt, c))
        # the update: (a) tiers
        T = tiers[s]
        for b in ids[i]:
            if b in T[0]:
                T[0].move_to_end(b)
                continue
            for t in (1, 2):
                T[t].pop(b, None)
            key = b
            for t in range(3):
                if caps[t] == 0:
                    continue
                T[t][key] = True
                if len(T[t]) <= caps[t]:
                    key = None
                    break
                key, _ = T[t].popitem(last=False)
            if key is not None:
                dropped += 1
        # (b) one stack of K + k2 + k3
        S = stacks[s]
        for b in ids[i]:
            if b in S:
                S.move_to_end(b)
            else:
                S[b] = True
                if len(S) > K + k2 + k3:
                    S.popitem(last=False)
    return out, tiers, stacks, dropped


@pytest.mark.parametrize("K,k2,k3,node", [(30, 40, 80, 1), (50, 0, 100, 2), (40, 60, 0, 3),
                                          (25, 25, 25, 2)])
def test_tier_replay(K, k2, k3, node):
    tr = _trace(400)
    W = 4
    cfg = _tiered(W, K, k2, k3, node)
    r = O.simulate(cfg, tr, 24, omega=1.0, seed=11, want_cache=True)
    assert r["status"] == 0
    out, tiers, stacks, dropped = _replays(tr, r, cfg)
    cats = np.array([c for c, _ in out])
    s = r["summary"]
    assert s["kv_g1"] == cats[:, 0].sum() and s["kv_g2"] == cats[:, 1].sum()
    assert s["kv_g3"] == cats[:, 2].sum() and s["kv_recompute"] == cats[:, 9].sum()
    assert s["kv_remote"] == cats[:, 3:9].sum()
    assert np.array_equal(r["kv_cost"], np.array([c for _, c in out]))
    total = 0.0
    for _, c in out:
        total = total + c
    assert s["kv_cost"] == total
    assert s["evicted_blocks"] == dropped
    ids = _content_ids(tr)
    h = O.hash_blocks(tr.tokens, tr.offsets)
    h2id = {}
    for i in range(tr.n_req):
        base = int(tr.offsets[i]) // 16
        for k, cid in enumerate(ids[i]):
            h2id[int(h[base + k])] = cid
    for j in range(W):
        got = [h2id[int(x)] for x in r["cache"][j]]
        assert got == list(stacks[j].keys())
        assert got == list(tiers[j][2]) + list(tiers[j][1]) + list(tiers[j][0])
    assert cats[:, 1].sum() + cats[:, 2].sum() > 0 or k2 + k3 == 0
    assert cats[:, 3:9].sum() > 0
    # rho counts every tier against the G1 capacity
    assert s["rho_end"] == sum(len(x) for x in stacks) / (W * K)


def _one_block_trace(names, times):
    n = len(names)
    tokens = np.zeros(16 * n, np.int32)
    for i, nm in enumerate(names):
        tokens[16 * i:16 * (i + 1)] = 500 + 41 * (ord(nm) - ord("A")) + np.arange(16)
    return Wk.Trace(tokens, np.arange(0, 16 * (n + 1), 16, dtype=np.int64),
                    np.array(times, np.float64), np.ones(n, np.int32), np.zeros(n, np.int32))


def test_hand_worked_round_robin_two_workers():
    # two workers on different nodes (tier_node 1), G1 = 1 block, G2 = 1,
    # G3 = 1; round robin sends request i to worker i mod 2.  alpha = 1, 4, 20,
    # gamma = 100, d_far = 10.  By hand (worker: G1 / G2 / G3 after the request):
    #  A -> w0: nowhere, 100            w0: A / - / -
    #  B -> w1: nowhere, 100            w1: B / - / -
    #  B -> w0: w1 G1, 10 + 1 = 11      w0: B / A / -
    #  A -> w1: w0 G2, 10 + 4 = 14      w1: A / B / -
    #  C -> w0: nowhere, 100            w0: C / B / A
    #  A -> w1: own G1, 1               w1: A / B / -
    #  A -> w0: own G3, 20              w0: A / C / B
    #  D -> w1: nowhere, 100            w1: D / A / B
    #  E -> w0: nowhere, 100            w0: E / A / C   (B dropped)
    #  B -> w1: own G3, 20              w1: B / D / A
    names = "ABBACAADEB"
    tr = _one_block_trace(names, [0.1 * i for i in range(len(names))])
    cfg = _tiered(2, 1, 1, 1, node=1, tier_d_near=2.0, tier_d_far=10.0)
    r = O.simulate(cfg, tr, 100, policy=O.POLICY_ROUNDROBIN, want_cache=True)
    assert r["status"] == 0
    assert list(r["kv_cost"]) == [100, 100, 11, 14, 100, 1, 20, 100, 100, 20]
    s = r["summary"]
    assert (s["kv_g1"], s["kv_g2"], s["kv_g3"], s["kv_remote"], s["kv_recompute"]) == \
        (1, 0, 2, 2, 5)
    assert s["kv_cost"] == 566.0
    assert (s["inserted_blocks"], s["evicted_blocks"]) == (7, 1)
    h = O.hash_blocks(tr.tokens, tr.offsets)
    nm = {int(h[i]): names[i] for i in range(len(names))}
    assert [nm[int(x)] for x in r["cache"][0]] == list("CAE")
    assert [nm[int(x)] for x in r["cache"][1]] == list("ADB")
    # first block to leave a G1: request 2 (B onto w0 pushes A down), at t = 0.2
    assert s["first_evict_t"] == 0.2 and s["rho_first_evict"] == 3 / 2
    assert s["rho_end"] == 6 / 2


@pytest.mark.parametrize("kw", [{"tier_alpha": (1.0, 1.0, 20.0)}, {"tier_alpha": (1.0, 4.0, 3.0)},
                                {"tier_gamma": 20.0}, {"tier_node": 0}, {"tier_k2": -1},
                                {"tier_d_far": -1.0}, {"tier_d_near": float("inf")}])
def test_tier_arguments_rejected(kw):
    tr = _trace(20)
    base = {"W": 2, "K": 32, "tiered": 1, "tier_k2": 8, "tier_k3": 8, "tier_node": 1}
    base.update(kw)
    cfg = O.OracleConfig(**base)
    assert O.simulate(cfg, tr, 4)["status"] == O.ERR_INVALID


def test_tiers_with_frequency_eviction_rejected():
    tr = _trace(20)
    r = O.simulate(_tiered(2, 32, 8, 8), tr, 4, eviction=O.EVICT_FREQ)
    assert r["status"] == O.ERR_INVALID
