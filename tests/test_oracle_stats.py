"""Pin of the oracle's decision statistics (the near-tie count of the
acceptance criteria: decisions whose two lowest Eq. (1) costs lie within
1e-6 relative, and exact ties) by a recount from the per-request cost
records."""
import numpy as np
import pytest

import oracle as O
from paper_2606_17081_gb300 import workloads as Wk


@pytest.mark.parametrize("W,omega,tau,seed", [(3, 1.0, 0.0, 1), (5, 0.0, 0.0, 2), (2, 0.5, 0.7, 3),
                                              (4, 1.0, 0.3, 4)])
def test_tie_counts_match_recount(W, omega, tau, seed):
    spec = Wk.TraceSpec(n_req=2000, len_kind="uniform", len_min=1, len_max=400, n_groups=8,
                        prefix_min=32, prefix_max=200, zipf_s=1.1, out_kind="uniform",
                        out_min=1, out_max=300)
    tr = Wk.make_trace(spec, seed)
    r = O.simulate(O.OracleConfig(W=W, K=512), tr, 64, omega=omega, tau=tau, seed=seed)
    assert r["status"] == 0
    c = np.sort(r["cost"].astype(np.float64), axis=1)
    c1, c2 = c[:, 0], c[:, 1]
    near = int(np.sum(c2 - c1 <= 1e-6 * np.abs(c2)))
    exact = int(np.sum(c2 == c1))
    s = r["summary"]
    assert (s["near_ties"], s["exact_ties"]) == (near, exact)
    assert exact > 0                      # integer-valued costs tie often
    assert s["sampled"] == (tr.n_req if tau > 0 else 0)
