"""Hand-written (skip_mask, proxy_plan) tables shared by the parity tests."""
from paper_2607_04461_gb300 import synth


def knob_plan(kind):
    """Hand-written plans (0-indexed steps and blocks; codes as synth.proxy_code).
    '1k': five steps; block 0 forecasts at order 2 from three anchors (steps 2, 1, 0),
    block 1 at order 1, block 2 at order 1 from anchors (3, 1) after a skip at step 2.
    '14b': four steps; order-0 proxies and an order-2 forecast of block 1 at step 3."""
    if kind == "1k":
        skip, proxy = synth.empty_plan(5, 3)
        skip[2, 2] = 1
        proxy[3, 0] = synth.proxy_code(2, 2)
        proxy[3, 1] = synth.proxy_code(2, 1)
        skip[4, 1] = 1
        proxy[4, 2] = synth.proxy_code(3, 1)
    else:
        skip, proxy = synth.empty_plan(4, 3)
        proxy[1, 0] = synth.proxy_code(0, 0)
        skip[1, 2] = 1
        skip[3, 0] = 1
        proxy[3, 1] = synth.proxy_code(2, 2)
        proxy[3, 2] = synth.proxy_code(2, 0)
    return skip, proxy
