"""Failure detection without a GPU fault.

* A device-side wait that runs out: with the stream-K tile counters poisoned (as a
  crashed launch could leave them) a finisher waits for a count no launch reaches; with a
  short wait limit the wait gives up, the call must return FB_ECUDA with "device wait
  timed out", and the model must work again at once.
* Host-injected allocation failures: every device allocation of fb_init_model is made to
  fail in turn; each attempt must return FB_ENOMEM, leave *out NULL and leak no device
  memory. A failure inside a sampling call leaves the model usable.
* fb_pipeline_step's worker thread makes the refiner's device current (two devices)."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2607_04461_gb300 import flashbon as fb
from paper_2607_04461_gb300 import synth

pytestmark = pytest.mark.gpu

SHORT_WAIT_NS = 20_000_000  # 20 ms: far beyond any wait of a correct launch of these shapes


def randn(shape, seed, scale=1.0, dtype=torch.bfloat16):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(shape, generator=g) * scale).to(dtype).cuda()


@pytest.fixture(scope="module")
def model():
    fb.load_library()
    m = fb.Model(synth.TINY, synth.make_weights(synth.TINY))
    yield m
    m.close()


def _ffn_down_operands():
    M, N, K = 1560, 1536, 8960          # the refine's FFN down-projection shape
    A, W = randn((M, K), 1), randn((N, K), 2, scale=K ** -0.5)
    bias, gate = randn((N,), 3, dtype=torch.float32), randn((N,), 4, dtype=torch.float32)
    resid = randn((M, N), 5, dtype=torch.float32)
    return M, N, K, A, W, bias, gate, resid


def test_stream_k_wait_times_out_then_recovers(model):
    M, N, K, A, W, bias, gate, resid = _ffn_down_operands()
    ref = torch.empty((M, N), dtype=torch.float32, device="cuda")
    fb.fb_op_gemm(model.handle, M, N, K, A, W, bias, 2, ref, resid, gate, None, None, 4)
    out = torch.zeros((M, N), dtype=torch.float32, device="cuda")
    fb.fb_test_poison_counters(model.handle)   # a count no launch will reach
    fb.fb_set_device_wait_limit(SHORT_WAIT_NS)
    try:
        with pytest.raises(fb.FlashBonError) as e:
            fb.fb_op_gemm(model.handle, M, N, K, A, W, bias, 2, out, resid, gate, None, None, 4)
    finally:
        fb.fb_set_device_wait_limit(0)
    assert e.value.status == fb.FB_ECUDA
    assert "device wait timed out" in str(e.value)
    # the call cleared the counters: the same call now matches bit for bit, twice
    for _ in range(2):
        again = torch.empty_like(ref)
        fb.fb_op_gemm(model.handle, M, N, K, A, W, bias, 2, again, resid, gate, None, None, 4)
        torch.cuda.synchronize()
        assert torch.equal(again, ref)


def _raw_init(cfg, weights):
    """fb_init_model through ctypes: (status, handle value)."""
    L = fb.load_library()
    packed = fb.pack_weights(cfg, weights)
    c = fb.make_cfg(cfg)
    h = ctypes.c_void_p(12345)           # must come back NULL on failure
    st = L.fb_init_model(ctypes.byref(c), packed.ctypes.data_as(ctypes.c_void_p),
                         ctypes.byref(h))
    return st, h.value


def test_init_model_allocation_failures_leak_nothing():
    cfg = synth.SMALL
    w = synth.make_weights(cfg, seed=4)
    fb.fb_test_fail_alloc(-1)
    with fb.Model(cfg, w):               # warm-up: loads the library's device code
        pass
    torch.cuda.synchronize()
    fb.fb_test_fail_alloc(-1)
    with fb.Model(cfg, w):
        n_alloc = fb.fb_test_alloc_calls()
    assert n_alloc >= 20
    free0, _ = torch.cuda.mem_get_info()
    try:
        for k in range(n_alloc):
            fb.fb_test_fail_alloc(k)
            st, h = _raw_init(cfg, w)
            assert st == fb.FB_ENOMEM, f"allocation {k}: status {st}"
            assert h is None, f"allocation {k}: *out not NULL"
            assert "injected" in fb.load_library().fb_last_error().decode()
            free1, _ = torch.cuda.mem_get_info()
            assert free1 == free0, f"allocation {k}: {free0 - free1} bytes leaked"
    finally:
        fb.fb_test_fail_alloc(-1)
    with fb.Model(cfg, w):               # disarmed: creation works again
        pass


def test_allocation_failure_inside_a_call_leaves_the_model_usable():
    """The first guided draft allocates the unconditional context's K/V; make that fail."""
    cfg = synth.SMALL.with_(max_n=4)
    w = synth.make_weights(cfg, bf16=True, norm_std=0.2)
    z = synth.make_latents(cfg, 2)
    ctx, ctx_u = synth.make_text(cfg), synth.make_text(cfg, seed=8)
    sched = synth.make_schedule(3)
    skip, proxy = synth.empty_plan(3, cfg.depth)
    opts = fb.make_opts(guidance=4.0, text_uncond=ctx_u)
    with fb.Model(cfg, w) as m:
        zd = torch.from_numpy(z).cuda()
        fb.fb_test_fail_alloc(0)
        try:
            with pytest.raises(fb.FlashBonError) as e:
                m.draft(zd, ctx, sched, skip, proxy, opts=opts)
        finally:
            fb.fb_test_fail_alloc(-1)
        assert e.value.status == fb.FB_ENOMEM
        assert torch.equal(zd, torch.from_numpy(z).cuda())   # nothing was written
        m.draft(zd, ctx, sched, skip, proxy, opts=opts)
        got = zd.cpu().numpy()
    with fb.Model(cfg, w) as m2:
        ze = torch.from_numpy(z).cuda()
        m2.draft(ze, ctx, sched, skip, proxy, opts=opts)
        assert np.array_equal(got, ze.cpu().numpy())


@pytest.mark.skipif(torch.cuda.device_count() < 2, reason="needs two CUDA devices")
def test_pipeline_step_refines_on_the_refiners_device():
    cfg = synth.SMALL
    w = synth.make_weights(cfg, bf16=True, norm_std=0.2)
    z = synth.make_latents(cfg, 2)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(4)
    skip, proxy = synth.empty_plan(2, cfg.depth)
    prev = torch.cuda.current_device()
    try:
        torch.cuda.set_device(1)
        with fb.Model(cfg, w) as d, fb.Model(cfg, w) as r:
            zd = torch.from_numpy(z).cuda(1)
            zr = torch.from_numpy(z[0]).cuda(1)
            fb.fb_pipeline_step(d.handle, zd, 2, ctx, sched[:3], skip, proxy,
                                refiner=r.handle, refine_latent=zr, refine_schedule=sched[2:])
            want = torch.from_numpy(z[0]).cuda(1)
            r.refine(want, ctx, sched[2:])
            assert torch.equal(zr, want)
    finally:
        torch.cuda.set_device(prev)
