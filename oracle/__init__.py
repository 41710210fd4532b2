"""CPU oracle (fp64 numpy) for the Flash-BoN draft path.

Test infrastructure: only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline /
reference leg may import it. It shares no code with the CUDA path.
"""
from .flashbon_oracle import *  # noqa: F401,F403
from .flashbon_oracle import OracleModel, plan_from_phi, resolve_plan, taylor_forecast  # noqa: F401
