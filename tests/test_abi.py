"""Host-side checks of the C-ABI library (no GPU needed): it loads, exports every
entry point include/flashbon.h declares, its weight layout matches the generator's, and
its host-only logic (phi expansion, argument validation) behaves as documented."""
import ctypes
import json
import os
import re

import numpy as np
import pytest

from oracle import flashbon_oracle as O
from paper_2607_04461_gb300 import flashbon as fb
from paper_2607_04461_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(fb.LIB_PATH):
        from paper_2607_04461_gb300 import build
        build.build()
    return fb.load_library()


def declared_functions():
    names = []
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            src = open(os.path.join(ROOT, "include", f)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names += re.findall(r"\b(fb_\w+)\s*\(", src)
    return sorted(set(names))


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert len(names) >= 15
    for n in names:
        assert hasattr(lib, n), f"{n} declared but not exported"
    assert set(names) == set(fb.EXPORTS)


@pytest.mark.parametrize("cfg", [synth.TINY, synth.SMALL, synth.WAN13], ids=["tiny", "small", "wan13"])
def test_weight_layout_matches_generator(lib, cfg):
    c = fb.make_cfg(cfg)
    count, total = ctypes.c_int(), ctypes.c_size_t()
    assert lib.fb_weights_count(ctypes.byref(c), ctypes.byref(count), ctypes.byref(total)) == 0
    specs = synth.weight_specs(cfg)
    assert count.value == len(specs)
    name, off, numel = ctypes.c_char_p(), ctypes.c_size_t(), ctypes.c_size_t()
    pos = 0
    for i, (n, shape, _) in enumerate(specs):
        assert lib.fb_weights_entry(ctypes.byref(c), i, ctypes.byref(name), ctypes.byref(off),
                                    ctypes.byref(numel)) == 0
        assert name.value.decode() == n
        assert off.value == pos and numel.value == int(np.prod(shape))
        pos += numel.value
    assert pos == total.value
    assert lib.fb_weights_entry(ctypes.byref(c), count.value, None, None, None) == fb.FB_EINVAL


def test_wan13_parameter_count(lib):
    c = fb.make_cfg(synth.WAN13)
    count, total = ctypes.c_int(), ctypes.c_size_t()
    lib.fb_weights_count(ctypes.byref(c), ctypes.byref(count), ctypes.byref(total))
    # a Wan2.1-1.3B-shaped DiT: about 1.3e9 parameters
    assert 1.2e9 < total.value < 1.5e9


def test_pack_weights_roundtrip(lib):
    cfg = synth.TINY
    w = synth.make_weights(cfg, bf16=False)
    buf = fb.pack_weights(cfg, w)
    c = fb.make_cfg(cfg)
    name, off, numel = ctypes.c_char_p(), ctypes.c_size_t(), ctypes.c_size_t()
    for i, (n, shape, _) in enumerate(synth.weight_specs(cfg)):
        lib.fb_weights_entry(ctypes.byref(c), i, ctypes.byref(name), ctypes.byref(off),
                             ctypes.byref(numel))
        np.testing.assert_array_equal(buf[off.value: off.value + numel.value], w[n].ravel())


def _phi_cases():
    with open(os.path.join(ROOT, "tests", "golden", "phi_star.json")) as fh:
        return json.load(fh)["cases"]


@pytest.mark.parametrize("case", _phi_cases(), ids=lambda c: c["name"])
@pytest.mark.parametrize("order", [0, 2])
def test_plan_from_phi_matches_oracle_and_golden(lib, case, order):
    args = (case["S"], case["S_prime"], case["n_skip"], case["l_start"], case["l_end"],
            case["f_full"], order, case["depth"])
    skip, proxy = fb.fb_plan_from_phi(*args)
    rs, rp = O.plan_from_phi(*args)
    np.testing.assert_array_equal(skip, rs)
    np.testing.assert_array_equal(proxy, rp)
    assert int(skip.sum()) == case["n_skip_entries"]
    assert int((proxy != -1).sum()) == case["n_proxy_entries"]


@pytest.mark.parametrize("bad", [
    (50, 0, 3, 22, 23, 5, 0, 30),     # S' < 1
    (50, 51, 3, 22, 23, 5, 0, 30),    # S' > S
    (50, 49, 3, 24, 23, 5, 0, 30),    # l_start > l_end
    (50, 49, 3, 22, 31, 5, 0, 30),    # l_end > depth
    (50, 49, 3, 22, 23, 0, 0, 30),    # f_full < 1
    (50, 49, -1, 22, 23, 5, 0, 30),   # n_skip < 0
    (50, 49, 3, 22, 23, 5, 3, 30),    # order 3
])
def test_plan_from_phi_rejects(lib, bad):
    with pytest.raises(fb.FlashBonError) as e:
        fb.fb_plan_from_phi(*bad)
    assert e.value.status == fb.FB_EINVAL
    with pytest.raises(ValueError):
        O.plan_from_phi(*bad)


@pytest.mark.parametrize("field,value", [("head_dim", 96), ("dim", 130), ("latent_h", 7),
                                         ("latent_c", 3), ("max_n", 0), ("eps_ln", 0.0)])
def test_init_rejects_bad_cfg_before_touching_the_device(lib, field, value):
    cfg = synth.TINY.with_(**{field: value})
    if field == "dim":
        cfg = cfg.with_(heads=1, head_dim=130)
    c = fb.make_cfg(cfg)
    h = ctypes.c_void_p()
    assert lib.fb_init_model(ctypes.byref(c), None, ctypes.byref(h)) == fb.FB_EINVAL
    assert h.value is None
    assert lib.fb_last_error()


def test_null_model_is_rejected(lib):
    assert lib.fb_draft(None, None, 1, None, None, 1, None, None) == fb.FB_EINVAL
    assert lib.fb_refine(None, None, None, None, 1) == fb.FB_EINVAL
    assert lib.fb_block_forward(None, 0, None, 1, 0.5) == fb.FB_EINVAL
    lib.fb_free(None)


@pytest.mark.parametrize("call", [
    lambda lib, out: lib.fb_probe_mma_gap(-1, out),
    lambda lib, out: lib.fb_probe_mma_gap(100001, out),
    lambda lib, out: lib.fb_probe_mufu(4, out),
    lambda lib, out: lib.fb_probe_mma_rate(3, 256, 16, out),   # 3 x 256 > 512 TMEM columns
    lambda lib, out: lib.fb_probe_mma_rate(1, 96, 16, out),
    lambda lib, out: lib.fb_probe_mma_mix(14, 0, 0, out),
    lambda lib, out: lib.fb_probe_mma_mix(0, 8, 0, out),
    lambda lib, out: lib.fb_probe_mma_mix(0, 7, 100001, out),
    lambda lib, out: lib.fb_probe_tmem_load(0, None),
])
def test_probes_reject_bad_arguments_before_touching_the_device(lib, call):
    out = ctypes.c_double()
    assert call(lib, ctypes.byref(out)) == fb.FB_EINVAL
    assert lib.fb_last_error()


# ---- Stage 2 selection (host logic) ---------------------------------------------------

@pytest.mark.parametrize("seed", range(12))
def test_select_elo_matches_oracle(lib, seed):
    g = np.random.default_rng(seed)
    M = int(g.integers(1, 40))
    quality = g.standard_normal(M)
    scores = np.clip(np.round(5 + 2 * quality + g.standard_normal(M)), 1, 10).astype(np.int32)
    noise = g.standard_normal((M, M))

    def cmp(a, b):   # noisy, confidence from the margin
        d = quality[a] - quality[b] + 0.3 * noise[a, b]
        return d > 0, 0 if abs(d) > 1 else (1 if abs(d) > 0.3 else 2)
    rho1, rho2, kappa = [(0.5, 0.5, 1.5), (1.0, 0.25, 3.0), (0.3, 1.0, 0.0)][seed % 3]
    if seed == 5:
        M, rho1 = 20, 0.3     # ceil(0.3 * 20) = 6 on both sides
        scores, quality = scores[:M] if len(scores) >= M else np.resize(scores, M), \
            np.resize(quality, M)
        noise = np.resize(noise, (M, M))
    w, r, calls = fb.fb_select_elo(scores, cmp, rho1, rho2, kappa)
    w0, r0, calls0 = O.elo_select(scores, cmp, rho1, rho2, kappa)
    assert (w, calls) == (w0, calls0)
    np.testing.assert_allclose(r, r0, rtol=0, atol=1e-9)


def test_select_elo_rejects_bad_confidence(lib):
    with pytest.raises(fb.FlashBonError) as e:
        fb.fb_select_elo([5, 6, 7], lambda a, b: (True, 5), 1.0, 1.0, 1.0)
    assert e.value.status == fb.FB_EINVAL
    with pytest.raises(fb.FlashBonError):
        fb.fb_select_elo([5, 6], lambda a, b: (True, 0), 0.0, 1.0, 1.0)
