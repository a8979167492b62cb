"""Pin of the oracle's event and latency rules by an independent
discrete-event replay written from the rules themselves: the closed-loop
client of §7.4 (at most C requests in flight; a request waits for a
completion, taken in (time, request) order), the per-worker service limit
(C_j - 1 = 63 concurrent, FIFO beyond it) and the Eq. (9) latency with n the
in-service count at service start, including the request.  Given the oracle's
decisions and cached prefixes, the replay recomputes every arrival, service
start, first token and completion."""
import heapq

import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import workloads as Wk

LAT_A, LAT_B, LAT_D, W_C, ITL, CAP = 0.005, 0.020, 0.010, 0.015, 0.012, 64


def _f(n):
    return LAT_A * n + LAT_B + LAT_D / ((CAP - n) * (CAP - n))


def _replay(tr, worker, prefix_chosen, C, W):
    n = tr.n_req
    L = np.diff(tr.offsets)
    nbt = (L + 15) // 16
    arrival, start, first, done = (np.zeros(n) for _ in range(4))
    heap = []                       # (completion time, request)
    serving = [0] * W
    waiting = [[] for _ in range(W)]
    in_flight = 0

    def begin(r, t):
        j = worker[r]
        serving[j] += 1
        o = prefix_chosen[r] / nbt[r] if nbt[r] > 0 else 0.0
        start[r] = t
        first[r] = t + (_f(serving[j]) - W_C * o)
        done[r] = first[r] + tr.out_len[r] * ITL
        heapq.heappush(heap, (done[r], r))

    def complete():
        nonlocal in_flight
        t, q = heapq.heappop(heap)
        in_flight -= 1
        j = worker[q]
        serving[j] -= 1
        if waiting[j]:
            begin(waiting[j].pop(0), t)
        return t

    t_prev = 0.0
    for i in range(n):
        tw = t_prev
        while in_flight >= C:                       # wait for a free client slot
            tw = max(tw, complete())
        a = max(float(tr.release[i]), tw)
        while heap and heap[0][0] <= a:              # every completion up to the arrival
            complete()
        arrival[i] = a
        j = worker[i]
        if serving[j] < CAP - 1:
            begin(i, a)
        else:
            waiting[j].append(i)
        in_flight += 1
        t_prev = a
    while heap:
        complete()
    return arrival, start, first, done


@pytest.mark.parametrize("policy,C,rate,W,seed", [(O.POLICY_DYNAMO, 256, None, 3, 9),
                                                  (O.POLICY_LOADBAL, 300, None, 3, 4),
                                                  (O.POLICY_DYNAMO, 40, 30.0, 3, 5),
                                                  (O.POLICY_DYNAMO, 3, None, 2, 6),
                                                  (O.POLICY_DYNAMO, 150, None, 1, 7)])
def test_events_match_independent_replay(policy, C, rate, W, seed):
    spec = Wk.TraceSpec(n_req=1200, len_kind="uniform", len_min=1, len_max=400, n_groups=8,
                        prefix_min=32, prefix_max=200, zipf_s=1.1, out_kind="uniform",
                        out_min=1, out_max=300, rate=rate)
    tr = Wk.make_trace(spec, seed)
    om = 1.0 if policy == O.POLICY_DYNAMO else 0.0
    r = O.simulate(O.OracleConfig(W=W, K=512), tr, C, policy=policy, omega=om)
    assert r["status"] == 0
    wk = r["worker"].astype(int)
    m = r["prefix"][np.arange(tr.n_req), wk]
    a, s, ft, ct = _replay(tr, wk, m, C, W)
    for name, mine in (("arrival", a), ("start", s), ("first_token", ft), ("completion", ct)):
        assert np.allclose(r[name], mine, rtol=1e-12, atol=0), name
    assert np.allclose(r["ttft"], ft - a, rtol=1e-12, atol=1e-15)
    # the cases exercise the rules: waiting for a slot, and (one worker, many
    # in flight) queueing behind the service limit
    if C <= 40:
        assert (a > tr.release).any()
    if W == 1:
        assert (s > a).any()


def _controller_replay(first, ttft, n_ticks, dt=5.0, alpha=0.3, th=(0.3, 2.0), eps=0.1, k=3):
    """The controller of §6.2 from the records: at t_k = k dt the window is
    every request whose first token came in [t_{k-1}, t_k); its nearest-rank
    P99 (an empty window repeats the last value) feeds the EWMA of Eq. (10),
    which starts at the first sample; Eq. (11)'s regime moves one step up
    after k samples at or above the next threshold, one step down after k
    samples below the current threshold less eps of it."""
    ewmas, regs = [], []
    ewma, last, regime, up, down = None, None, 0, 0, 0
    for kk in range(1, n_ticks + 1):
        lo, hi = (kk - 1) * dt, kk * dt
        w = np.sort(ttft[(first >= lo) & (first < hi)])
        if w.size:
            last = float(w[int(np.ceil(0.99 * w.size)) - 1])
        if last is not None:
            ewma = last if ewma is None else alpha * last + (1.0 - alpha) * ewma
            go_up = regime < 2 and ewma >= th[regime]
            go_down = regime > 0 and ewma < th[regime - 1] * (1.0 - eps)
            up = up + 1 if go_up else 0
            down = down + 1 if go_down else 0
            if up >= k:
                regime, up, down = regime + 1, 0, 0
            elif down >= k:
                regime, up, down = regime - 1, 0, 0
        ewmas.append(-1.0 if ewma is None else ewma)
        regs.append(regime)
    return np.array(ewmas), np.array(regs)


@pytest.mark.parametrize("C,seed", [(600, 2), (250, 3)])
def test_controller_matches_replay_from_records(C, seed):
    # a closed loop that saturates, so that the regime moves
    spec = Wk.TraceSpec(n_req=6000, n_groups=16, prefix_min=64, prefix_max=256, len_median=256,
                        len_max=1024)
    tr = Wk.make_trace(spec, seed)
    r = O.simulate(O.OracleConfig(W=3, K=4096), tr, C, controller=1, omega=1.0, tau=0.0,
                   seed=1, max_ticks=4000)
    assert r["status"] == 0
    # ticks taken while requests were still arriving: all their windows' first
    # tokens are known from the records
    n_ticks = int(np.floor(r["arrival"][-1] / 5.0))
    assert n_ticks > 5
    ewma, reg = _controller_replay(r["first_token"], r["ttft"], n_ticks)
    assert np.allclose(r["tick_ewma"][:n_ticks], ewma, rtol=1e-12, atol=0)
    assert np.array_equal(r["tick_regime"][:n_ticks], reg)
    assert reg.max() >= 1
