"""CPU oracle of the routing simulation -- test infrastructure.

Only `tests/`, `__graft_entry__.smoke()` and the CPU-baseline leg of `bench.py`
import this package.  The product path (the CUDA library and its binding)
never does, and this package never imports the product.
"""
from .routesim_oracle import *  # noqa: F401,F403
from .routesim_oracle import build_oracle, OracleConfig  # noqa: F401
