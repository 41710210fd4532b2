"""Parity of the CUDA draft path (through the C-ABI) with the fp64 oracle.

Small shapes are compared in full; the Wan2.1-1.3B-shaped workloads are run at full
size in the configuration the benchmark uses and checked on sampled candidates the
oracle computes one by one, plus properties that hold at any size."""
import os

import numpy as np
import pytest
import torch

from oracle import flashbon_oracle as O
from paper_2607_04461_gb300 import flashbon as fb
from paper_2607_04461_gb300 import synth
from _metrics import BLOCK_TOL, COS_MIN, check_latents, cosine, rel_max
from _plans import knob_plan

pytestmark = pytest.mark.gpu


def cuda(x):
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


@pytest.fixture(scope="module")
def tiny():
    cfg = synth.TINY
    w = synth.make_weights(cfg, bf16=False, norm_std=0.2)
    m = fb.Model(cfg, w)
    yield cfg, w, m, O.OracleModel(cfg, w)
    m.close()


@pytest.fixture(scope="module")
def small():
    cfg = synth.SMALL
    w = synth.make_weights(cfg, bf16=True, norm_std=0.2)
    m = fb.Model(cfg, w)
    yield cfg, w, m, O.OracleModel(cfg, w)
    m.close()


# ---- tiny DiT (2 blocks, hidden 128, 16 tokens, N=4, 4 steps, skip + proxy) ----------

def test_tiny_draft_matches_oracle(tiny):
    cfg, w, m, ref = tiny
    z = synth.make_latents(cfg, 4)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(4)
    skip, proxy = synth.tiny_plan()
    zd = cuda(z)
    m.draft(zd, ctx, sched, skip, proxy)
    got = zd.cpu().numpy()
    want = ref.draft(z, ctx, sched, skip, proxy)
    for j in range(4):
        check_latents(got[j], want[j], z[j], label=f"tiny cand {j}")


def test_tiny_host_and_device_latents_agree(tiny):
    cfg, w, m, _ = tiny
    z = synth.make_latents(cfg, 3)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(4)
    skip, proxy = synth.tiny_plan()
    zh = z.copy()
    m.draft(zh, ctx, sched, skip, proxy)
    zd = cuda(z)
    m.draft(zd, cuda(ctx), sched, skip, proxy)
    np.testing.assert_array_equal(zh, zd.cpu().numpy())


# ---- small shape: several tiles with ragged tails -------------------------------------

def test_small_block_forward_each_layer(small):
    cfg, w, m, ref = small
    ctx = synth.make_text(cfg)
    m.encode_text(ctx)
    kv = ref.encode_text(ctx)
    rng = np.random.default_rng(5)
    n = cfg.max_n
    h = rng.standard_normal((n * cfg.tokens, cfg.dim)).astype(np.float32)
    t = 0.63
    _, mod = ref.time_embed(np.float32(t))
    for l in range(cfg.depth):
        hd = cuda(h)
        m.block_forward(l, hd, n, t)
        got = hd.cpu().numpy().astype(np.float64) - h
        for j in range(n):
            hj = h[j * cfg.tokens:(j + 1) * cfg.tokens].astype(np.float64)
            want = ref.block(l, hj, mod, kv[l]) - hj
            e = rel_max(got[j * cfg.tokens:(j + 1) * cfg.tokens], want)
            assert e <= BLOCK_TOL, f"layer {l} cand {j}: {e:.3e}"


PLANS = {
    "empty": lambda S, L: synth.empty_plan(S, L),
    "skip_third_proxy_half": lambda S, L: synth.random_plan(S, L, 1 / 3, 0.5, seed=3),
    "order1": lambda S, L: synth.random_plan(S, L, 0.0, 1.0, seed=4, order=1),
    "phi_order2": lambda S, L: O.plan_from_phi(S + 2, S, 2, 2, 2, 2, 2, L),
}


@pytest.mark.parametrize("plan", list(PLANS))
def test_small_draft_matches_oracle(small, plan):
    cfg, w, m, ref = small
    S = 5
    z = synth.make_latents(cfg, cfg.max_n)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(S)
    skip, proxy = PLANS[plan](S, cfg.depth)
    zd = cuda(z)
    m.draft(zd, ctx, sched, skip, proxy)
    got = zd.cpu().numpy()
    want = ref.draft(z, ctx, sched, skip, proxy)
    for j in range(cfg.max_n):
        check_latents(got[j], want[j], z[j], label=f"{plan} cand {j}")


def test_small_order2_taylor_with_three_anchors(small):
    """Steps 0, 1, 2 computed; step 3 forecasts from three anchors (Eqs. 3-5)."""
    cfg, w, m, ref = small
    skip, proxy = synth.empty_plan(4, cfg.depth)
    proxy[3, :] = synth.proxy_code(2, 2)
    z = synth.make_latents(cfg, 2)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(8)[:5]
    zd = cuda(z)
    m.draft(zd, ctx, sched, skip, proxy, n=2)
    want = ref.draft(z, ctx, sched, skip, proxy)
    for j in range(2):
        check_latents(zd.cpu().numpy()[j], want[j], z[j], label=f"order2 cand {j}")


def test_small_refine_and_markov(small):
    """Refine matches the oracle; draft to step k then refine equals one full run
    (bit-exact: same kernels on the same rows in the same order)."""
    cfg, w, m, ref = small
    S, k = 6, 2
    z = synth.make_latents(cfg, 1)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(S)
    full = cuda(z)
    m.draft(full, ctx, sched, *synth.empty_plan(S, cfg.depth))
    part = cuda(z)
    m.draft(part, ctx, sched[:k + 1], *synth.empty_plan(k, cfg.depth))
    r = part[0].clone()
    m.refine(r, ctx, sched[k:])
    assert torch.equal(r, full[0])
    want = ref.refine(part[0].cpu().numpy(), ctx, sched[k:])
    check_latents(r.cpu().numpy(), want, part[0].cpu().numpy(), label="refine")


def test_small_all_skipped_and_all_proxied(small):
    cfg, w, m, ref = small
    S = 3
    z = synth.make_latents(cfg, 2)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(S)
    skip, proxy = synth.empty_plan(S, cfg.depth)
    skip[0, :] = 1                      # step 0: every block skipped
    proxy[2, :] = synth.proxy_code(1, 0)  # step 2: every block proxied from step 1
    zd = cuda(z)
    m.draft(zd, ctx, sched, skip, proxy, n=2)
    want = ref.draft(z, ctx, sched, skip, proxy)
    for j in range(2):
        check_latents(zd.cpu().numpy()[j], want[j], z[j], label=f"skip/proxy-all cand {j}")


def test_small_candidate_permutation_is_exact(small):
    """Rows of different candidates never mix: permuting candidates permutes results."""
    cfg, w, m, _ = small
    z = synth.make_latents(cfg, 3)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(3)
    skip, proxy = synth.random_plan(3, cfg.depth, 1 / 3, 0.5, seed=9)
    a, b = cuda(z), cuda(z[::-1])
    m.draft(a, ctx, sched, skip, proxy)
    m.draft(b, ctx, sched, skip, proxy)
    assert torch.equal(a, b.flip(0))


def test_edge_cases_and_errors(small):
    cfg, w, m, _ = small
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(3)
    z = cuda(synth.make_latents(cfg, 1))
    z0 = z.clone()
    m.draft(z, ctx, sched, n=0)                       # n == 0: no-op
    assert torch.equal(z, z0)
    fb.fb_draft(m.handle, z, 1, ctx, sched[:1])        # zero steps: no-op
    assert torch.equal(z, z0)

    def status(fn):
        with pytest.raises(fb.FlashBonError) as e:
            fn()
        return e.value.status

    big = cuda(synth.make_latents(cfg, cfg.max_n + 1))
    assert status(lambda: m.draft(big, ctx, sched)) == fb.FB_EINVAL
    assert status(lambda: m.draft(z, ctx, sched[::-1].copy())) == fb.FB_EINVAL
    bad = sched.copy()
    bad[1] = bad[0]
    assert status(lambda: m.draft(z, ctx, bad)) == fb.FB_EINVAL
    skip, proxy = synth.empty_plan(3, cfg.depth)
    proxy[1, 0] = synth.proxy_code(1, 0)
    assert status(lambda: m.draft(z, ctx, sched, skip, proxy)) == fb.FB_EPLAN
    skip, proxy = synth.empty_plan(3, cfg.depth)
    skip[0, 1] = 1
    proxy[2, 1] = synth.proxy_code(0, 0)
    assert status(lambda: m.draft(z, ctx, sched, skip, proxy)) == fb.FB_EPLAN
    skip, proxy = synth.empty_plan(3, cfg.depth)
    skip[2, 0] = 1
    proxy[2, 0] = synth.proxy_code(0, 0)
    assert status(lambda: m.draft(z, ctx, sched, skip, proxy)) == fb.FB_EPLAN
    assert torch.equal(z, z0)                          # rejected calls changed nothing
    assert status(lambda: m.block_forward(cfg.depth, z, 1, 0.5)) == fb.FB_EINVAL


def test_block_forward_requires_text(small):
    cfg, w, _, _ = small
    with fb.Model(cfg.with_(depth=1, max_n=1), {k: v for k, v in w.items()
                                                if not k.startswith("blocks.") or
                                                k.startswith("blocks.0.")}) as m1:
        h = torch.zeros((cfg.tokens, cfg.dim), device="cuda")
        with pytest.raises(fb.FlashBonError) as e:
            m1.block_forward(0, h, 1, 0.5)
        assert e.value.status == fb.FB_ESTATE


# ---- Wan2.1-1.3B shape at full size --------------------------------------------------

def test_wan13_single_block_n16_sampled():
    """One Wan2.1-1.3B-shaped block, N=16 (1560 tokens each), candidates 0 and 15."""
    cfg = synth.WAN13.with_(depth=1, max_n=16)
    w = synth.make_weights(cfg)
    ctx = synth.make_text(cfg)
    rng = np.random.default_rng(11)
    n = 16
    h = rng.standard_normal((n * cfg.tokens, cfg.dim)).astype(np.float32)
    t = 0.5
    with fb.Model(cfg, w) as m:
        m.encode_text(ctx)
        hd = cuda(h)
        m.block_forward(0, hd, n, t)
        got = hd.cpu().numpy().astype(np.float64) - h
    ref = O.OracleModel(cfg, w)
    kv = ref.encode_text(ctx)
    _, mod = ref.time_embed(np.float32(t))
    for j in (0, n - 1):
        sl = slice(j * cfg.tokens, (j + 1) * cfg.tokens)
        want = ref.block(0, h[sl].astype(np.float64), mod, kv[0]) - h[sl]
        e = rel_max(got[sl], want)
        assert e <= BLOCK_TOL, f"cand {j}: {e:.3e}"


@pytest.fixture(scope="module")
def wan13_pool():
    cfg = synth.WAN13
    w = synth.make_weights(cfg)
    m = fb.Model(cfg, w)
    yield cfg, w, m
    m.close()


def test_wan13_draft_pool_full_size(wan13_pool):
    """The benchmark's draft pool: 30 blocks, N=32, 10 of 50 steps, 1/3 skipped per
    step, half of the rest proxied on odd steps. Checked: candidate permutation is exact
    at full size; the first two steps of candidate 0 match the oracle."""
    cfg, w, m = wan13_pool
    n, S = 32, 10
    sched = synth.make_schedule(50)[:S + 1]
    skip, proxy = synth.random_plan(S, cfg.depth, 1 / 3, 0.5, seed=7)
    z = synth.make_latents(cfg, n)
    ctx = synth.make_text(cfg)
    a = cuda(z)
    m.draft(a, ctx, sched, skip, proxy)
    assert torch.isfinite(a).all()
    perm = np.roll(np.arange(n), 5)
    b = cuda(z[perm])
    m.draft(b, ctx, sched, skip, proxy)
    assert torch.equal(b, a[torch.from_numpy(perm).cuda()])
    # oracle on candidate 0, first two steps of the same plan
    two = cuda(z[:1])
    m.draft(two, ctx, sched[:3], skip[:2], proxy[:2])
    ref = O.OracleModel(cfg, w)
    want = ref.draft(z[:1], ctx, sched[:3], skip[:2], proxy[:2])
    check_latents(two.cpu().numpy()[0], want[0], z[0], label="wan13 cand 0, 2 steps")


GOLD13 = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "wan13_pool_cand0.npz")


def test_wan13_pool_whole_trajectory_matches_oracle(wan13_pool):
    """The benchmark's whole path at full size against the oracle's trajectory of
    candidate 0 (stored by tests/golden/make_wan13_trajectory.py, which calls only the
    oracle): the 32-candidate draft over 10 of 50 steps with a third of the blocks
    skipped per step and half of the rest proxied on odd steps (§4.1, Eqs. 3-7), then
    candidate 0's draft latent refined over the remaining 40 steps with phi_full (§4.2
    Stage 3) on the 40-SM partition the benchmark refines on. Checked after the draft,
    after 20 refine steps and at the end."""
    g = np.load(GOLD13)
    cfg, w, m = wan13_pool
    n, S = 32, 10
    sched = synth.make_schedule(50)
    skip, proxy = synth.random_plan(S, cfg.depth, 1 / 3, 0.5, seed=7)
    assert np.array_equal(skip, g["skip"]) and np.array_equal(proxy, g["proxy"])
    assert np.array_equal(sched, g["schedule"])
    mid = int(g["refine_mid_step"])
    z = synth.make_latents(cfg, n)
    ctx = synth.make_text(cfg)
    a = cuda(z)
    m.draft(a, ctx, sched[:S + 1], skip, proxy)
    zd = a[0].clone()
    zd_h = zd.cpu().numpy()
    check_latents(zd_h, g["z_draft"], z[0], label="draft, 10 steps")
    try:
        sp = fb.SmSplit(40)
    except fb.FlashBonError:
        sp = None                        # no SM partitions from the driver: whole GPU
    try:
        if sp is not None:
            m.set_stream(sp.streams[0])
            m.set_sm_budget(sp.sms[0])
        m.refine(zd, ctx, sched[S:mid + 1])
        zm_h = zd.cpu().numpy()
        m.refine(zd, ctx, sched[mid:])
        zr_h = zd.cpu().numpy()
    finally:
        m.set_stream(None)
        m.set_sm_budget(0)
        if sp is not None:
            sp.close()
    check_latents(zm_h, g["z_refine_mid"], z[0], label=f"refine to step {mid}")
    check_latents(zr_h, g["z_refine"], z[0], label="refine, 40 steps")
    # the refine's own displacement, each side from its own draft latent
    assert cosine(zr_h - zd_h, g["z_refine"] - g["z_draft"]) >= COS_MIN


# ---- the other shapes of the scope table: Wan2.1-14B width, 4096 tokens ---------------
# One-block models: every kernel shape of the full models (D = 5120 with 40 heads and
# FFN 13824; 4096 tokens per candidate, 32 key tiles), at an oracle cost of seconds.

@pytest.fixture(scope="module", params=["wan14", "wan13_1k"])
def wide(request):
    cfg = {"wan14": synth.WAN14, "wan13_1k": synth.WAN13_1K}[request.param].with_(depth=1,
                                                                                 max_n=2)
    w = synth.make_weights(cfg)
    m = fb.Model(cfg, w)
    yield request.param, cfg, w, m
    m.close()


def test_wide_single_block_n2(wide):
    """One block at N=2: both candidates against the oracle."""
    name, cfg, w, m = wide
    ctx = synth.make_text(cfg)
    rng = np.random.default_rng(12)
    n, t = 2, 0.7
    h = rng.standard_normal((n * cfg.tokens, cfg.dim)).astype(np.float32)
    m.encode_text(ctx)
    hd = cuda(h)
    m.block_forward(0, hd, n, t)
    got = hd.cpu().numpy().astype(np.float64) - h
    ref = O.OracleModel(cfg, w)
    kv = ref.encode_text(ctx)
    _, mod = ref.time_embed(np.float32(t))
    for j in range(n):
        sl = slice(j * cfg.tokens, (j + 1) * cfg.tokens)
        want = ref.block(0, h[sl].astype(np.float64), mod, kv[0]) - h[sl]
        e = rel_max(got[sl], want)
        assert e <= BLOCK_TOL, f"{name} cand {j}: {e:.3e}"


def test_wide_two_step_draft(wide):
    """Two full steps of one candidate: patch embedding, time embedding, block and head
    at these widths against the oracle."""
    name, cfg, w, m = wide
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(50)[:3]
    skip, proxy = synth.empty_plan(2, cfg.depth)
    z = synth.make_latents(cfg, 1)
    a = cuda(z)
    m.draft(a, ctx, sched, skip, proxy)
    want = O.OracleModel(cfg, w).draft(z, ctx, sched, skip, proxy)
    check_latents(a.cpu().numpy()[0], want[0], z[0], label=f"{name} 2 steps")


def test_wan13_refine_on_a_partition_matches_the_whole_gpu(wan13_pool):
    """The refine as the bench runs it: one candidate on a 40-SM partition, where the FFN
    down-projection takes the stream-K split and attention three 256-query items per
    persistent CTA. Against the same refine on the whole GPU (whose draft path the oracle
    checks above) only fp32 summation orders differ."""
    cfg, w, m = wan13_pool
    z = synth.make_latents(cfg, 1)[0]
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(50)[10:13]          # two steps from t_10
    whole = cuda(z)
    m.refine(whole, ctx, sched)
    with fb.SmSplit(40) as sp:
        m.set_stream(sp.streams[0])
        m.set_sm_budget(sp.sms[0])
        part = cuda(z)
        m.refine(part, ctx, sched)
        m.set_stream(None)
        m.set_sm_budget(0)
    assert torch.isfinite(part).all()
    e = rel_max(part.cpu().double().numpy() - z, whole.cpu().double().numpy() - z)
    assert e <= 1e-2, f"displacement {e:.3e}"


def test_model_from_device_weights_equals_host_weights():
    """fb_init_model reads device-resident weights as it reads host ones."""
    cfg = synth.SMALL
    wd = synth.make_weights_device(cfg, seed=3)
    wh = {k: v.cpu().numpy() for k, v in wd.items()}
    z = synth.make_latents(cfg, 2)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(3)
    skip, proxy = synth.empty_plan(3, cfg.depth)
    outs = []
    for w in (wd, wh):
        with fb.Model(cfg, w) as m:
            a = cuda(z)
            m.draft(a, ctx, sched, skip, proxy)
            outs.append(a)
    assert torch.equal(outs[0], outs[1])


# ---- classifier-free guidance and SDE steps (App. A.1) -------------------------------

@pytest.fixture(scope="module")
def small4():
    cfg = synth.SMALL.with_(max_n=4)
    w = synth.make_weights(cfg, bf16=True, norm_std=0.2)
    m = fb.Model(cfg, w)
    yield cfg, w, m, O.OracleModel(cfg, w)
    m.close()


@pytest.mark.parametrize("mode", ["cfg", "sde", "cfg_sde"])
def test_small_guidance_and_sde_match_oracle(small4, mode):
    cfg, w, m, ref = small4
    S, n = 4, 2
    z = synth.make_latents(cfg, n)
    ctx, ctx_u = synth.make_text(cfg), synth.make_text(cfg, seed=8)
    sched = synth.make_schedule(S)
    skip, proxy = synth.random_plan(S, cfg.depth, 1 / 3, 0.5, seed=5, order=1)
    guided, sde = "cfg" in mode, "sde" in mode
    noise = synth.make_noise(cfg, S, n) if sde else None
    opts = fb.make_opts(guidance=4.5 if guided else 1.0, text_uncond=ctx_u if guided else None,
                        sde_a=0.7 if sde else 0.0, noise=noise)
    zd = cuda(z)
    m.draft(zd, ctx, sched, skip, proxy, opts=opts)
    want = ref.draft(z, ctx, sched, skip, proxy, ctx_uncond=ctx_u if guided else None,
                     guidance=4.5, sde_a=0.7 if sde else 0.0, noise=noise)
    for j in range(n):
        check_latents(zd.cpu().numpy()[j], want[j], z[j], label=f"{mode} cand {j}")


def test_guided_refine_with_sde_matches_oracle(small4):
    cfg, w, m, ref = small4
    S = 3
    z = synth.make_latents(cfg, 1)[0]
    ctx, ctx_u = synth.make_text(cfg), synth.make_text(cfg, seed=8)
    sched = synth.make_schedule(6)[3:]
    noise = synth.make_noise(cfg, S, 1, seed=77)
    zd = cuda(z)
    m.refine(zd, ctx, sched, opts=fb.make_opts(5.0, ctx_u, 0.3, cuda(noise)))
    want = ref.refine(z, ctx, sched, ctx_uncond=ctx_u, guidance=5.0, sde_a=0.3, noise=noise[:, 0])
    check_latents(zd.cpu().numpy(), want, z, label="guided SDE refine")


def test_guidance_weight_one_is_the_conditional_draft(small4):
    cfg, w, m, _ = small4
    z = synth.make_latents(cfg, 2)
    ctx, ctx_u = synth.make_text(cfg), synth.make_text(cfg, seed=8)
    sched = synth.make_schedule(3)
    a, b = cuda(z), cuda(z)
    m.draft(a, ctx, sched)
    m.draft(b, ctx, sched, opts=fb.make_opts(1.0, ctx_u))
    d = (a - b).abs().max().item()
    assert d <= 1e-5 * max(1.0, a.abs().max().item()), d


def test_guidance_and_sde_argument_errors(small4):
    cfg, w, m, _ = small4
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(2)
    z = cuda(synth.make_latents(cfg, 3))
    with pytest.raises(fb.FlashBonError) as e:      # 2n > max_n
        m.draft(z, ctx, sched, opts=fb.make_opts(3.0, ctx))
    assert e.value.status == fb.FB_EINVAL
    with pytest.raises(fb.FlashBonError) as e:      # SDE without draws
        m.draft(z, ctx, sched, opts=fb.make_opts(sde_a=0.5))
    assert e.value.status == fb.FB_EINVAL


def test_pipeline_draft_select_refine(small4):
    """Stage 1 -> Stage 2 -> Stage 3 (§4.2): drafts on the GPU, a synthetic verifier (the
    drafts' cosine to a hidden target; pairwise confidence from the margin) through the
    library's Elo selection, and a full refine of the selected draft."""
    cfg, w, m, ref = small4
    n, S, Sp = 4, 6, 3
    z = synth.make_latents(cfg, n)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(S)
    skip, proxy = synth.random_plan(Sp, cfg.depth, 1 / 3, 0.5, seed=11)
    zd = cuda(z)
    m.draft(zd, ctx, sched[:Sp + 1], skip, proxy)
    drafts = zd.cpu().numpy().astype(np.float64)
    target = synth.make_latents(cfg, 1, seed_base=99)[0].astype(np.float64).ravel()
    q = np.array([d.ravel() @ target / np.linalg.norm(d) / np.linalg.norm(target)
                  for d in drafts])
    scores = np.clip(np.round(5 + 50 * q), 1, 10).astype(np.int32)

    def cmp(a, b):
        d = q[a] - q[b]
        return d > 0, 0 if abs(d) > 0.02 else (1 if abs(d) > 0.005 else 2)
    win, ratings, calls = fb.fb_select_elo(scores, cmp, 0.5, 0.5, 1.5)
    assert win == O.elo_select(scores, cmp, 0.5, 0.5, 1.5)[0]
    assert win == int(np.argmax(q))
    r = zd[win].clone()
    m.refine(r, ctx, sched[Sp:])
    want = ref.refine(drafts[win], ctx, sched[Sp:])
    check_latents(r.cpu().numpy(), want, drafts[win], label="refine of the selected draft")


# ---- cached-state offload and a warm-started refine (§4.2 Stage 3) --------------------

def _parse_state(cfg, buf):
    """(t per layer, Delta per layer as fp32 [tokens][dim]) from a state buffer."""
    raw = (buf.cpu() if torch.is_tensor(buf) else torch.from_numpy(buf)).numpy().view(np.uint8)
    L, pd = cfg.depth, cfg.tokens * cfg.dim
    hb = (4 * L + 255) // 256 * 256
    assert raw.size == hb + L * pd * 2
    tau = raw[:4 * L].view(np.float32).copy()
    u16 = raw[hb:].view(np.uint16).astype(np.uint32) << 16
    return tau, u16.view(np.float32).reshape(L, cfg.tokens, cfg.dim)


def _state_dict(tau, delta):
    return {l: (float(tau[l]), delta[l].astype(np.float64))
            for l in range(len(tau)) if not np.isnan(tau[l])}


def _check_state(cfg, buf, want, label):
    tau, delta = _parse_state(cfg, buf)
    for l in range(cfg.depth):
        if l in want:
            assert tau[l] == np.float32(want[l][0]), (label, l)
            err = rel_max(delta[l], want[l][1])
            assert err <= 5e-2, f"{label} layer {l}: {err:.3e}"
        else:
            assert np.isnan(tau[l]) and not delta[l].any(), (label, l)


def test_state_offload_matches_oracle(small4):
    cfg, w, m, ref = small4
    S, n = 4, 3
    z = synth.make_latents(cfg, n)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(S)
    skip, proxy = synth.random_plan(S, cfg.depth, 1 / 3, 0.5, seed=5, order=1)
    zd = cuda(z)
    m.draft(zd, ctx, sched, skip, proxy, opts=fb.make_opts(keep_state=True))
    bufs = [torch.empty(m.state_bytes(), dtype=torch.uint8).pin_memory() for _ in range(n)]
    m.state_offload(0, bufs[:1])
    m.state_offload(1, bufs[1:])
    m.state_wait()
    want_z, states = ref.draft(z, ctx, sched, skip, proxy, keep_state=True)
    for j in range(n):
        check_latents(zd.cpu().numpy()[j], want_z[j], z[j], label=f"keep_state cand {j}")
        _check_state(cfg, bufs[j], states[j], f"state cand {j}")


def test_state_offload_overlapped_with_the_next_draft(small4):
    """The copies of draft A's state run while draft B rewrites the cache; B waits for
    them per slot, so A's offloaded state and B's latents are both intact."""
    cfg, w, m, ref = small4
    S = 4
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(S)
    skip, proxy = synth.random_plan(S, cfg.depth, 1 / 3, 0.5, seed=9, order=0)
    za = synth.make_latents(cfg, 2)
    zb = synth.make_latents(cfg, 2, seed_base=555)
    da, db = cuda(za), cuda(zb)
    m.draft(da, ctx, sched, skip, proxy, opts=fb.make_opts(keep_state=True))
    bufs = [torch.empty(m.state_bytes(), dtype=torch.uint8).pin_memory() for _ in range(2)]
    m.state_offload(0, bufs)
    m.draft(db, ctx, sched, skip, proxy, opts=fb.make_opts(keep_state=True))
    m.state_wait()
    _, states_a = ref.draft(za, ctx, sched, skip, proxy, keep_state=True)
    want_b = ref.draft(zb, ctx, sched, skip, proxy)
    for j in range(2):
        _check_state(cfg, bufs[j], states_a[j], f"draft A state cand {j}")
        check_latents(db.cpu().numpy()[j], want_b[j], zb[j], label=f"draft B cand {j}")


def test_warm_started_refine_matches_oracle(small4):
    cfg, w, m, ref = small4
    z = synth.make_latents(cfg, 2)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(5)
    zd = cuda(z)
    m.draft(zd, ctx, sched[:3], *synth.empty_plan(2, cfg.depth),
            opts=fb.make_opts(keep_state=True))
    buf = torch.empty(m.state_bytes(), dtype=torch.uint8).pin_memory()
    m.state_offload(1, [buf])
    m.state_wait()
    start = zd[1].cpu().numpy()
    state = _state_dict(*_parse_state(cfg, buf))
    assert sorted(state) == list(range(cfg.depth))
    for warm in (1, 2):
        r = zd[1].clone()
        m.refine(r, ctx, sched[2:], opts=fb.make_opts(state=buf, warm_steps=warm))
        want = ref.refine(start, ctx, sched[2:], state=state, warm_steps=warm)
        check_latents(r.cpu().numpy(), want, start, label=f"warm refine, {warm} warm steps")
        rd = zd[1].clone()                                   # the state from device memory
        m.refine(rd, ctx, sched[2:], opts=fb.make_opts(state=buf.cuda(), warm_steps=warm))
        assert torch.equal(r, rd)
    r0, r1 = zd[1].clone(), zd[1].clone()
    m.refine(r0, ctx, sched[2:])
    m.refine(r1, ctx, sched[2:], opts=fb.make_opts(state=buf, warm_steps=0))
    assert torch.equal(r0, r1)


def test_state_errors(small4):
    cfg, w, m, _ = small4
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(2)
    z = cuda(synth.make_latents(cfg, 2))
    buf = torch.empty(m.state_bytes(), dtype=torch.uint8)
    m.draft(z, ctx, sched)                                   # no keep_state
    with pytest.raises(fb.FlashBonError) as e:
        m.state_offload(0, [buf])
    assert e.value.status == fb.FB_ESTATE
    m.draft(z, ctx, sched, opts=fb.make_opts(keep_state=True))
    with pytest.raises(fb.FlashBonError) as e:
        m.state_offload(1, [buf, buf])                      # candidates 1..2 of 2
    assert e.value.status == fb.FB_EINVAL
    m.state_offload(1, [buf])
    m.state_wait()
    with pytest.raises(fb.FlashBonError) as e:               # no warm start under guidance
        m.refine(z[0].clone(), ctx, sched,
                 opts=fb.make_opts(2.0, ctx, state=buf, warm_steps=1))
    assert e.value.status == fb.FB_EINVAL


# ---- SM partitions: a model confined to part of the GPU ----------------------------

def test_sm_split_and_budget_reproduce_the_whole_gpu_run():
    """A draft on a 40-SM partition (green context) with the matching SM budget gives the
    same latents, bit for bit, as on the whole GPU: the kernels' choices are the same at
    this size and each output element's arithmetic does not depend on the grid."""
    cfg = synth.SMALL
    w = synth.make_weights(cfg, bf16=True, norm_std=0.2)
    z = synth.make_latents(cfg, cfg.max_n)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(4)
    skip, proxy = synth.random_plan(4, cfg.depth, 1 / 3, 0.5, seed=3)
    with fb.Model(cfg, w) as m:
        whole = cuda(z)
        m.draft(whole, ctx, sched, skip, proxy)
        with fb.SmSplit(40) as sp:
            assert sp.sms[0] >= 2 and sp.sms[1] >= 2
            assert sp.sms[0] + sp.sms[1] == torch.cuda.get_device_properties(0).multi_processor_count
            m.set_stream(sp.streams[0])
            m.set_sm_budget(sp.sms[0])
            part = cuda(z)
            m.draft(part, ctx, sched, skip, proxy)
            m.set_stream(None)
            m.set_sm_budget(0)
        assert torch.equal(part, whole)


def test_stream_k_on_a_partition():
    """On 20 SM pairs the 1560 x 1536 x 8960 GEMM's 42 tiles take 3 rounds, so the
    automatic choice is the stream-K split; every contributor must be resident inside the
    partition. Bit-identical to the forced split, within fp32 summation order of whole
    tiles, and right against the oracle."""
    M, N, K = 1560, 1536, 8960
    g = torch.Generator().manual_seed(91)
    A = (torch.randn(M, K, generator=g)).to(torch.bfloat16).cuda()
    W = (torch.randn(N, K, generator=g) * K ** -0.5).to(torch.bfloat16).cuda()
    resid = torch.randn(M, N, generator=g).cuda()
    with fb.Model(synth.TINY, synth.make_weights(synth.TINY)) as m, fb.SmSplit(40) as sp:
        m.set_stream(sp.streams[0])
        m.set_sm_budget(sp.sms[0])
        outs = []
        for impl in (0, 4, 3):
            out = torch.empty(M, N, device="cuda")
            fb.fb_op_gemm(m.handle, M, N, K, A, W, None, 2, out, resid, None, None, None, impl)
            outs.append(out)
        torch.cuda.synchronize()
        m.set_stream(None)
    assert torch.equal(outs[0], outs[1])
    assert rel_max(outs[0].cpu().double().numpy(), outs[2].cpu().double().numpy()) <= 1e-5
    want = resid.cpu().double().numpy() + O.linear(A.float().cpu().double().numpy(),
                                                   W.float().cpu().double().numpy())
    assert rel_max(outs[0].cpu().double().numpy(), want) <= 1e-4


def test_pipeline_step_equals_the_calls_one_after_the_other():
    """fb_pipeline_step (draft of a new pool on one partition while the previous pool's
    candidate 0 is refined on the other, a library worker thread) gives what the same
    two calls give one after the other, bit for bit."""
    cfg = synth.SMALL
    w = synth.make_weights(cfg, bf16=True, norm_std=0.2)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(8)
    dsched, rsched = sched[:4], sched[3:]
    skip, proxy = synth.random_plan(3, cfg.depth, 1 / 3, 0.5, seed=5)
    z_a, z_b = synth.make_latents(cfg, 3), synth.make_latents(cfg, 3, first=3)
    with fb.Model(cfg, w) as md, fb.Model(cfg.with_(max_n=2), w) as mr, \
            fb.SmSplit(40) as sp:
        mr.set_stream(sp.streams[0]); mr.set_sm_budget(sp.sms[0])
        md.set_stream(sp.streams[1]); md.set_sm_budget(sp.sms[1])
        # pipelined: pool a alone, then pool b beside the refine of a's candidate 0
        pa, pb = cuda(z_a), cuda(z_b)
        fb.fb_pipeline_step(md.handle, pa, 3, ctx, dsched, skip, proxy)
        torch.cuda.synchronize()
        ra = pa[0].clone()
        fb.fb_pipeline_step(md.handle, pb, 3, ctx, dsched, skip, proxy, mr.handle, ra, rsched)
        torch.cuda.synchronize()
        # the same calls one after the other
        qa, qb = cuda(z_a), cuda(z_b)
        md.draft(qa, ctx, dsched, skip, proxy)
        torch.cuda.synchronize()
        ra2 = qa[0].clone()
        md.draft(qb, ctx, dsched, skip, proxy)
        mr.refine(ra2, ctx, rsched)
        torch.cuda.synchronize()
        with pytest.raises(fb.FlashBonError) as e:   # the refine needs a model of its own
            fb.fb_pipeline_step(md.handle, cuda(z_b), 3, ctx, dsched, skip, proxy, md.handle,
                                ra.clone(), rsched)
        assert e.value.status == fb.FB_EINVAL
        pc = cuda(z_b)                                # (this call still drafts pc)
        with pytest.raises(fb.FlashBonError) as e:   # a refine error comes back, prefixed
            fb.fb_pipeline_step(md.handle, pc, 3, ctx, dsched, skip, proxy, mr.handle,
                                ra.clone(), np.array([0.5, 0.7], np.float32))  # increasing
        assert "refine:" in str(e.value)
        md.set_stream(None); mr.set_stream(None)
    assert torch.equal(pa, qa) and torch.equal(pb, qb) and torch.equal(ra, ra2)


def test_sm_budget_and_split_reject_bad_sizes():
    with fb.Model(synth.TINY, synth.make_weights(synth.TINY)) as m:
        for n in (1, 100000):
            with pytest.raises(fb.FlashBonError) as e:
                m.set_sm_budget(n)
            assert e.value.status == fb.FB_EINVAL
    for n in (1, 100000):
        with pytest.raises(fb.FlashBonError) as e:
            fb.SmSplit(n)
        assert e.value.status == fb.FB_EINVAL


# ---- multi-step plans with the method's knobs at the larger shapes (§4.1, Eqs. 3-7) ----
# Three-block models keep the oracle's cost to a minute while every step mixes computed,
# skipped and proxied blocks.

def test_wan13_4096_tokens_knob_plan_matches_oracle():
    """Wan2.1-1.3B dims at 1024x1024 (4096 tokens per candidate, 32 key tiles), three
    blocks, N=2, five steps of a plan with skips and order-1/2 proxies: both candidates."""
    cfg = synth.WAN13_1K.with_(depth=3, max_n=2)
    w = synth.make_weights(cfg)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(50)[:6]
    skip, proxy = knob_plan("1k")
    z = synth.make_latents(cfg, 2)
    with fb.Model(cfg, w) as m:
        a = cuda(z)
        m.draft(a, ctx, sched, skip, proxy)
        got = a.cpu().numpy()
    want = O.OracleModel(cfg, w).draft(z, ctx, sched, skip, proxy)
    for j in range(2):
        check_latents(got[j], want[j], z[j], label=f"4096 tokens cand {j}")


def test_wan14_width_knob_plan_matches_oracle():
    """Wan2.1-14B dims (hidden 5120, 40 heads, FFN 13824), three blocks, four steps with
    skips, order-0 proxies and an order-2 forecast; candidate 0 of N=2."""
    cfg = synth.WAN14.with_(depth=3, max_n=2)
    w = synth.make_weights(cfg)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(50)[:5]
    skip, proxy = knob_plan("14b")
    z = synth.make_latents(cfg, 2)
    with fb.Model(cfg, w) as m:
        a = cuda(z)
        m.draft(a, ctx, sched, skip, proxy)
        got = a.cpu().numpy()
    want = O.OracleModel(cfg, w).draft(z[:1], ctx, sched, skip, proxy)
    check_latents(got[0], want[0], z[0], label="14B width cand 0")
