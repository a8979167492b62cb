"""Pins of the frequency eviction (the KV Block Manager of §2.2: frequency 1 on
insertion, doubled on a hit, lowered by 1 per decay step; frequency 1 cold,
2 and more hot) and of the cache-pressure outputs (the regime-transition
proposition of §5.3, rho = resident blocks over W K) in the oracle, against
things other than the oracle's code: the frequency cap 1 reduces to exact LRU;
a hand-worked single-worker sequence; a replay keyed by prompt content with
an eagerly decayed frequency table; conservation of blocks."""
from collections import OrderedDict

import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import workloads as Wk


def _small_trace(n=600, seed=3, rate=None, groups=8):
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


@pytest.mark.parametrize("K,tau,policy", [(48, 0.0, O.POLICY_DYNAMO), (90, 0.7, O.POLICY_DYNAMO),
                                          (64, 0.0, O.POLICY_LOADBAL)])
def test_frequency_cap_one_is_lru(K, tau, policy):
    # with freq_max = 1 a hit cannot raise a block above 1: every block stays
    # cold and the victim is always the least recently used block
    tr = _small_trace(500)
    cfg = O.OracleConfig(W=3, K=K)
    a = O.simulate(cfg, tr, 24, policy=policy, omega=1.0, tau=tau, seed=5, want_cache=True)
    b = O.simulate(cfg, tr, 24, policy=policy, omega=1.0, tau=tau, seed=5, want_cache=True,
                   eviction=O.EVICT_FREQ, freq_max=1, decay_s=0.25)
    assert a["status"] == b["status"] == 0
    for k in ("worker", "prefix", "ttft", "completion"):
        assert np.array_equal(a[k], b[k]), k
    for j in range(3):
        assert np.array_equal(a["cache"][j], b["cache"][j])
    assert a["summary"] == b["summary"]
    assert a["summary"]["evicted_blocks"] > 0


def _one_block_trace(names, times):
    # one 16-token block per request, the same tokens for the same name
    n = len(names)
    tokens = np.zeros(16 * n, np.int32)
    for i, nm in enumerate(names):
        tokens[16 * i:16 * (i + 1)] = 1000 + 37 * (ord(nm) - ord("A")) + np.arange(16)
    offsets = np.arange(0, 16 * (n + 1), 16, dtype=np.int64)
    return Wk.Trace(tokens, offsets, np.array(times, np.float64), np.ones(n, np.int32),
                    np.zeros(n, np.int32))


def test_hand_worked_single_worker():
    # K = 3, one decay step per second, frequency cap 4.  By hand (cache listed
    # least to most recent, frequencies in brackets):
    #  0.0 A, 0.1 B, 0.2 C          A1 B1 C1
    #  0.3 A hit                    B1 C1 A2
    #  0.4 D: cold LRU B out        C1 A2 D1
    #  0.5 E: C out                 A2 D1 E1
    #  0.6 F: A is hot, D out       A2 E1 F1
    #  1.2 G (step 1: A1): A out    E1 F1 G1
    #  1.3 E hit, 1.35 E hit        F1 G1 E4 (2, then 4 = the cap)
    #  1.4 H: F out                 G1 E4 H1
    #  2.5 I (step 2: E3): G out    E3 H1 I1
    #  2.6 J: E hot, H out          E3 I1 J1
    #  4.5 K (step 4: E1): E out    I1 J1 K1
    names = "ABCADEFGEEHIJK"
    times = [0.0, 0.1, 0.2, 0.3, 0.4, 0.5, 0.6, 1.2, 1.3, 1.35, 1.4, 2.5, 2.6, 4.5]
    tr = _one_block_trace(names, times)
    cfg = O.OracleConfig(W=1, K=3)
    r = O.simulate(cfg, tr, 100, want_cache=True, eviction=O.EVICT_FREQ, freq_max=4,
                   decay_s=1.0)
    assert r["status"] == 0
    assert np.array_equal(r["arrival"], tr.release)       # nothing waits for a slot
    h = O.hash_blocks(tr.tokens, tr.offsets)
    name_of = {int(h[i]): names[i] for i in range(len(names))}
    assert [name_of[int(x)] for x in r["cache"][0]] == list("IJK")
    s = r["summary"]
    assert (s["inserted_blocks"], s["evicted_blocks"], s["hit_blocks"]) == (11, 8, 3)
    assert s["first_evict_t"] == 0.4 and s["rho_first_evict"] == 1.0 and s["rho_end"] == 1.0
    # exact LRU on the same sequence ends with the three most recent
    lru = O.simulate(cfg, tr, 100, want_cache=True)
    assert [name_of[int(x)] for x in lru["cache"][0]] == list("IJK")
    assert lru["summary"]["evicted_blocks"] == 8


@pytest.mark.parametrize("K,decay,fmax,tau", [(64, 0.5, 8, 0.0), (200, 5.0, 64, 0.7),
                                              (48, 1e9, 4, 0.0), (120, 0.05, 1 << 20, 0.0)])
def test_frequency_rules_against_content_replay(K, decay, fmax, tau):
    tr = _small_trace(500, rate=40.0)
    W = 3
    cfg = O.OracleConfig(W=W, K=K)
    r = O.simulate(cfg, tr, 24, omega=1.0, tau=tau, seed=11, want_cache=True,
                   eviction=O.EVICT_FREQ, freq_max=fmax, decay_s=decay)
    assert r["status"] == 0
    ids = _content_ids(tr)
    h = O.hash_blocks(tr.tokens, tr.offsets)
    h2id = {}
    caches = [OrderedDict() for _ in range(W)]     # id -> frequency, least recent first
    step = 0
    first_ev, rho_first, evicted, inserted = -1.0, -1.0, 0, 0
    for i in range(tr.n_req):
        base = int(tr.offsets[i]) // 16
        for k, cid in enumerate(ids[i]):
            h2id[int(h[base + k])] = cid
        for j in range(W):
            m = 0
            while m < len(ids[i]) and ids[i][m] in caches[j]:
                m += 1
            assert r["prefix"][i, j] == m, (i, j)
        a = float(r["arrival"][i])
        d = int(np.floor(a / decay))
        while step < d:                      # one decay step at a time, every block
            step += 1
            for c in caches:
                for key in c:
                    c[key] = max(1, c[key] - 1)
        c = caches[int(r["worker"][i])]
        ev0 = evicted
        for cid in ids[i]:
            if cid in c:
                c[cid] = min(2 * c[cid], fmax)
                c.move_to_end(cid)
            else:
                if len(c) == K:
                    cold = [key for key, f in c.items() if f == 1]
                    victim = cold[0] if cold else next(iter(c))
                    del c[victim]
                    evicted += 1
                c[cid] = 1
                inserted += 1
        if ev0 == 0 and evicted > 0:
            first_ev = a
            rho_first = sum(len(x) for x in caches) / (W * K)
    for j in range(W):
        assert [h2id[int(x)] for x in r["cache"][j]] == list(caches[j].keys())
    s = r["summary"]
    assert (s["inserted_blocks"], s["evicted_blocks"]) == (inserted, evicted)
    assert s["first_evict_t"] == first_ev and s["rho_first_evict"] == rho_first
    assert s["rho_end"] == sum(len(x) for x in caches) / (W * K)
    assert evicted > 0


def test_rho_conservation_and_no_eviction():
    tr = _small_trace(300)
    for K in (40, 100000):
        cfg = O.OracleConfig(W=3, K=K)
        r = O.simulate(cfg, tr, 16, eviction=O.EVICT_FREQ, freq_max=16, decay_s=2.0)
        s = r["summary"]
        assert s["rho_end"] == (s["inserted_blocks"] - s["evicted_blocks"]) / (3 * K)
        if s["evicted_blocks"] == 0:
            assert s["first_evict_t"] == -1.0 and s["rho_first_evict"] == -1.0
        else:
            assert 0 < s["rho_first_evict"] <= 1.0 and s["first_evict_t"] >= 0.0
    assert O.simulate(O.OracleConfig(W=3, K=100000), tr, 16)["summary"]["evicted_blocks"] == 0


@pytest.mark.parametrize("fmax,decay", [(0, 1.0), (1 << 21, 1.0), (4, 0.0), (4, float("inf")),
                                        (4, float("nan"))])
def test_frequency_arguments_rejected(fmax, decay):
    tr = _small_trace(20)
    r = O.simulate(O.OracleConfig(W=2, K=64), tr, 4, eviction=O.EVICT_FREQ, freq_max=fmax,
                   decay_s=decay)
    assert r["status"] == O.ERR_INVALID
    r = O.simulate(O.OracleConfig(W=2, K=64), tr, 4, eviction=2)
    assert r["status"] == O.ERR_INVALID
