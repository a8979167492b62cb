"""Pins of the load-spike schedule (Experiment 3) in the oracle: the client's
semaphore against C(t), admission as soon as a slot frees, the step-up, and
the first regime switch as a controller sample time."""
import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import workloads as wk

T1, T2 = 60.0, 150.0


def _conc(t, C=32, mid=128, end=32):
    return np.where(t < T1, C, np.where(t < T2, mid, end))


@pytest.fixture(scope="module")
def runs():
    tr = wk.make_trace(wk.TraceSpec(n_req=8000), 3)
    cfg = O.OracleConfig(W=2, K=65536)
    out = {}
    for ctl in (0, 1):
        out[ctl] = O.simulate(cfg, tr, 32, omega=1.0, tau=0.0, seed=1, controller=ctl,
                              schedule=(T1, T2, 128, 32), max_ticks=400)
    return tr, out


def _in_flight_before(a, c, i):
    # requests admitted earlier and not completed by a_i (completions at a_i
    # come first, so they no longer count)
    return int(np.sum((a[:i] <= a[i]) & (c[:i] > a[i])))


def test_semaphore_holds_C_of_t(runs):
    tr, out = runs
    for r in out.values():
        assert r["status"] == 0
        a, c = r["arrival"], r["completion"]
        lim = _conc(a)
        for i in range(0, tr.n_req, 7):
            assert _in_flight_before(a, c, i) < lim[i]


def test_admission_as_soon_as_a_slot_frees(runs):
    # closed loop (all releases at 0): request i arrives either with the
    # previous one or exactly when a completion frees a slot or the schedule
    # steps up
    tr, out = runs
    r = out[0]
    a, c = r["arrival"], r["completion"]
    cs = set(np.round(c, 12))
    for i in range(1, tr.n_req, 5):
        if a[i] > a[i - 1]:
            assert round(a[i], 12) in cs or a[i] in (T1,)
            # just before a_i the client was full
            t = np.nextafter(a[i], -np.inf)
            busy = int(np.sum((a[:i] <= t) & (c[:i] > t)))
            assert busy >= _conc(np.array([t]))[0]


def test_step_up_admits_at_T1(runs):
    _, out = runs
    a = out[0]["arrival"]
    k = int(np.sum(a == T1))
    assert k == 128 - 32   # the 96 new slots fill at the step


def test_step_down_drains_before_admitting(runs):
    _, out = runs
    a, c = out[0]["arrival"], out[0]["completion"]
    after = np.nonzero(a >= T2)[0]
    first = after[0]
    assert _in_flight_before(a, c, first) < 32


def test_first_switch_is_a_controller_sample(runs):
    _, out = runs
    s0, s1 = out[0]["summary"], out[1]["summary"]
    assert s0["first_switch_t"] == -1.0   # no controller: no switch
    fs = s1["first_switch_t"]
    assert fs > T1                          # the spike starts the switch
    cfg = O.OracleConfig(W=2, K=65536)
    k = int(round(fs / cfg.dt))
    assert fs == k * cfg.dt
    reg = out[1]["tick_regime"]
    assert reg[k - 1] != 0 and np.all(reg[:k - 1] == 0)
