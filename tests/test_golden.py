"""Values printed outside the code, kept as text fixtures under tests/golden/
(each file cites its source), against the oracle's and the library's
constants: the controller's Eq. (10)-(11) constants (§6.2), Table 2's regime
parameters (§6.3), the cost-matrix constants of the PoA estimate (§6.4), and
the Philox4x32-10 known-answer vectors of Random123.  The library is only
loaded and asked for its default configuration (host code; no GPU call)."""
import inspect
import os

import pytest

import oracle as O
from paper_2606_17081_gb300 import build as B
from paper_2606_17081_gb300 import routesim as rs
from paper_2606_17081_gb300 import workloads as wk

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _rows(name):
    with open(os.path.join(GOLDEN, name)) as fh:
        return [ln.split() for ln in fh if ln.strip() and not ln.lstrip().startswith("#")]


def _pairs(name):
    return {k: float(v) for k, v in _rows(name)}


@pytest.fixture(scope="module")
def lib_config():
    B.build()
    return rs.rs_config_default()


def test_controller_constants(lib_config):
    g = _pairs("controller_constants.txt")
    o = O.OracleConfig()
    for src in (o, lib_config):
        assert src.alpha == g["alpha"]
        assert src.dt == g["dt"]
        # the defaults are the 70B thresholds
        assert (src.theta1, src.theta2) == (g["theta1_70b"], g["theta2_70b"])
    p = wk.Plan.__dataclass_fields__   # the workloads' thresholds
    assert (p["theta1"].default, p["theta2"].default) == (g["theta1_70b"], g["theta2_70b"])
    # 340B thresholds: larger than the 70B ones by the paper's own figures
    assert g["theta1_340b"] > g["theta1_70b"] and g["theta2_340b"] > g["theta2_70b"]


def test_regime_parameters_table2(lib_config):
    rows = {r[0]: (float(r[1]), float(r[2])) for r in _rows("regime_params_table2.txt")}
    assert set(rows) == {"below", "transition", "saturated"}
    o = O.OracleConfig()
    for name, k in (("transition", 1), ("saturated", 2)):
        tau, om = rows[name]
        assert (o.regime_tau[k], o.regime_omega[k]) == (tau, om)
        # the library keeps them as float32
        assert lib_config.regime_tau[k] == pytest.approx(tau, rel=1e-7)
        assert lib_config.regime_omega[k] == pytest.approx(om, rel=1e-7)
    # Below: the replica's own tau and omega (the plan's cells start at the
    # paper's Below row: argmin with full cache weight)
    assert rows["below"] == (0.0, 1.0)


def test_cost_matrix_constants(lib_config):
    g = _pairs("cost_matrix_constants.txt")
    o = O.OracleConfig()
    for src in (o, lib_config):
        assert (src.lat_a, src.lat_b, src.lat_d) == (g["a"], g["b"], g["d"])
        assert src.cap == int(g["C_j"])
        assert src.w_c == g["w_c"]
    # beta = 2 is fixed in Eq. (9) on both sides (d / (C_j - n)^2)
    assert g["beta"] == 2.0
    # the exhaustive Game 1 solver's defaults are the same constants
    sig = inspect.signature(O.game_exhaustive).parameters
    assert (sig["lat_a"].default, sig["lat_b"].default, sig["lat_d"].default) == (g["a"], g["b"], g["d"])
    assert sig["cap"].default == int(g["C_j"])


def test_philox_known_answer_vectors():
    rows = _rows("philox4x32_10_kat.txt")
    assert len(rows) == 3
    for r in rows:
        v = [int(x, 16) for x in r]
        assert O.philox4x32_10(tuple(v[0:4]), tuple(v[4:6])) == tuple(v[6:10])
