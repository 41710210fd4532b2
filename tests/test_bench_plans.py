"""The bench's workload variants on the host: the plans, candidate counts and config keys
the JSON line reports (no GPU; the phi* plan comes from the library's host code)."""
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402
from _plans import knob_plan  # noqa: E402
from oracle import flashbon_oracle as O  # noqa: E402


def test_base_plan_is_the_draft_pool():
    cfg, sched, skip, proxy, s_draft = bench.plan_for("base")
    assert s_draft == bench.S_DRAFT == 10 and skip.shape == proxy.shape == (10, cfg.depth)
    assert len(sched) == bench.S_TOTAL + 1
    assert bench.n_candidates("base") == 32
    assert bench.N_CAND * bench.computed_blocks(skip, proxy) == 4800


def test_phi_star_plan_counts():
    """The paper's phi* (S = 50, S' = 49, blocks 22-23 skipped from step 3, a full step
    every 5, order 2) on 30 layers: 10 full steps; on the others every block outside
    22-23 proxied."""
    pytest.importorskip("ctypes")
    try:
        cfg, sched, skip, proxy, s_draft = bench.plan_for("phi_star")
    except (FileNotFoundError, OSError):
        pytest.skip("library not built")
    assert s_draft == 49 and skip.shape == (49, 30)
    assert int(skip.sum()) == (49 - 3) * 2           # blocks 22, 23 from step 3 on
    full_steps = [k for k in range(49) if (proxy[k] == -1).all() or
                  ((proxy[k] == -1) | (skip[k] == 1)).all()]
    assert full_steps == list(range(0, 49, 5))
    assert bench.computed_blocks(skip, proxy) == 282
    assert bench.n_candidates("phi_star") == 8
    assert bench.config_dict(cfg, "phi_star")["draft_steps"] == 49


def test_full50_computes_every_block():
    cfg, sched, skip, proxy, s_draft = bench.plan_for("full50")
    assert s_draft == 50 and not skip.any() and (proxy == -1).all()
    assert bench.computed_blocks(skip, proxy) == 50 * cfg.depth
    assert bench.config_dict(cfg, "full50")["refine_steps"] == 0


def test_split_schedule_variants():
    assert set(bench.SPLIT_VARIANTS) == {"base", "sde"}
    assert bench.REFINE_SMS % 8 == 0


def test_knob_plans_use_every_proxy_order():
    """The plans above really forecast at the orders named (anchor counts per proxy)."""
    an = O.resolve_plan(*knob_plan("1k"))
    assert an[(3, 0)] == [2, 1, 0] and an[(3, 1)] == [2, 1] and an[(4, 2)] == [3, 1]
    an = O.resolve_plan(*knob_plan("14b"))
    assert an[(1, 0)] == [0] and an[(3, 1)] == [2, 1, 0] and an[(3, 2)] == [2]
