"""Pins for the CPU oracle: each check compares it with something other than itself
(a library routine, brute force, a closed form, an invariant, or values derived by hand
from the paper's printed configurations)."""
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as Fn

from oracle import flashbon_oracle as O
from paper_2607_04461_gb300 import synth

GOLD = os.path.join(os.path.dirname(__file__), "golden")
rng = np.random.default_rng(123)


def t64(x):
    return torch.from_numpy(np.asarray(x, np.float64))


# -- primitives against library routines ----------------------------------------------

def test_layer_norm_matches_torch():
    x = rng.standard_normal((7, 48)) * 3 + 1
    w, b = rng.standard_normal(48), rng.standard_normal(48)
    ref = Fn.layer_norm(t64(x), (48,), t64(w), t64(b), eps=1e-6).numpy()
    np.testing.assert_allclose(O.layer_norm(x, 1e-6, w, b), ref, rtol=1e-12, atol=1e-12)
    ref0 = Fn.layer_norm(t64(x), (48,), eps=1e-6).numpy()
    np.testing.assert_allclose(O.layer_norm(x, 1e-6), ref0, rtol=1e-12, atol=1e-12)


def test_rms_norm_matches_torch():
    x = rng.standard_normal((5, 64)) * 2
    w = rng.standard_normal(64)
    ref = Fn.rms_norm(t64(x), (64,), t64(w), eps=1e-6).numpy()
    np.testing.assert_allclose(O.rms_norm(x, w, 1e-6), ref, rtol=1e-12, atol=1e-12)


def test_activations_match_torch():
    x = np.linspace(-8, 8, 1001)
    np.testing.assert_allclose(O.gelu_tanh(x), Fn.gelu(t64(x), approximate="tanh").numpy(),
                               rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(O.silu(x), Fn.silu(t64(x)).numpy(), rtol=1e-12, atol=1e-14)


def test_linear_matches_torch():
    x, w, b = rng.standard_normal((6, 10)), rng.standard_normal((4, 10)), rng.standard_normal(4)
    np.testing.assert_allclose(O.linear(x, w, b), Fn.linear(t64(x), t64(w), t64(b)).numpy(),
                               rtol=1e-12, atol=1e-12)


def test_timestep_embedding_hand_values():
    e = O.timestep_embedding(0.37, dim=256)
    assert e.shape == (256,)
    # frequency 0 is 1: the first cos/sin entries see 1000 t directly
    assert e[0] == pytest.approx(math.cos(370.0), abs=1e-12)
    assert e[128] == pytest.approx(math.sin(370.0), abs=1e-12)
    # last frequency 10000^(-127/128)
    f = 10000.0 ** (-127 / 128)
    assert e[127] == pytest.approx(math.cos(370.0 * f), abs=1e-12)
    assert e[255] == pytest.approx(math.sin(370.0 * f), abs=1e-12)
    z = O.timestep_embedding(0.0)
    assert np.all(z[:128] == 1.0) and np.all(z[128:] == 0.0)


# -- attention against brute force and the library --------------------------------------

def test_attention_brute_force():
    Lq, Lk, H, dh = 3, 4, 2, 5
    q, k, v = (rng.standard_normal((L, H, dh)) for L in (Lq, Lk, Lk))
    out = O.attention(q, k, v)
    for h in range(H):
        for i in range(Lq):
            s = [sum(q[i, h, d] * k[j, h, d] for d in range(dh)) / math.sqrt(dh)
                 for j in range(Lk)]
            m = max(s)
            e = [math.exp(x - m) for x in s]
            z = sum(e)
            for d in range(dh):
                ref = sum(e[j] / z * v[j, h, d] for j in range(Lk))
                assert out[i, h, d] == pytest.approx(ref, rel=1e-12, abs=1e-12)


def test_attention_matches_sdpa():
    q, k, v = rng.standard_normal((17, 3, 8)), rng.standard_normal((11, 3, 8)), \
        rng.standard_normal((11, 3, 8))
    ref = Fn.scaled_dot_product_attention(t64(q).transpose(0, 1), t64(k).transpose(0, 1),
                                          t64(v).transpose(0, 1)).transpose(0, 1).numpy()
    np.testing.assert_allclose(O.attention(q, k, v), ref, rtol=1e-10, atol=1e-12)


# -- RoPE --------------------------------------------------------------------------------

def test_rope_is_complex_rotation():
    gh, gw, dh, theta = 3, 5, 16, 10000.0
    cos, sin = O.rope_tables(gh, gw, dh, theta)
    x = rng.standard_normal((gh * gw, 2, dh))
    y = O.apply_rope(x, cos, sin)
    # independent statement: pair j of a token at grid (r, c) is multiplied by e^{i pos w_j}
    half = dh // 2
    for tok in range(gh * gw):
        r, c = divmod(tok, gw)
        for j in range(dh // 2):
            pos = r if j < half // 2 else c
            w = theta ** (-2.0 * (j % (half // 2)) / half)
            zc = complex(x[tok, 1, 2 * j], x[tok, 1, 2 * j + 1]) * complex(
                math.cos(pos * w), math.sin(pos * w))
            assert y[tok, 1, 2 * j] == pytest.approx(zc.real, abs=1e-12)
            assert y[tok, 1, 2 * j + 1] == pytest.approx(zc.imag, abs=1e-12)


def test_rope_invariants():
    gh, gw, dh = 4, 6, 32
    cos, sin = O.rope_tables(gh, gw, dh, 10000.0)
    x = rng.standard_normal((gh * gw, 3, dh))
    y = O.apply_rope(x, cos, sin)
    np.testing.assert_allclose(y[0], x[0], atol=0)            # grid (0, 0): identity
    np.testing.assert_allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1),
                               rtol=1e-12)
    # relative positions: <R(m)q, R(n)k> depends on m - n only
    q, k = rng.standard_normal(dh), rng.standard_normal(dh)
    X = np.tile(q, (gh * gw, 1, 1)).astype(np.float64)
    K = np.tile(k, (gh * gw, 1, 1)).astype(np.float64)
    Rq, Rk = O.apply_rope(X, cos, sin)[:, 0], O.apply_rope(K, cos, sin)[:, 0]
    tok = lambda r, c: r * gw + c  # noqa: E731
    assert Rq[tok(2, 3)] @ Rk[tok(1, 1)] == pytest.approx(Rq[tok(3, 5)] @ Rk[tok(2, 3)], rel=1e-10)


# -- patchify / embedding -------------------------------------------------------------

def test_patch_embed_is_strided_conv():
    cfg = synth.SMALL
    w = {"patch.w": rng.standard_normal((cfg.dim, cfg.patch_dim)),
         "patch.b": rng.standard_normal(cfg.dim)}
    m = O.OracleModel(cfg.with_(depth=0), w)
    z = rng.standard_normal((cfg.latent_c, cfg.latent_h, cfg.latent_w))
    h = m.patch_embed(z)
    conv = Fn.conv2d(t64(z)[None], t64(w["patch.w"]).reshape(cfg.dim, cfg.latent_c, 2, 2),
                     t64(w["patch.b"]), stride=2)[0]          # [D, gh, gw]
    np.testing.assert_allclose(h, conv.reshape(cfg.dim, -1).T.numpy(), rtol=1e-12, atol=1e-12)
    np.testing.assert_array_equal(O.unpatchify(O.patchify(z, 2), cfg.latent_c, cfg.latent_h,
                                               cfg.latent_w, 2), z)


# -- Taylor proxy (Eqs. 3-5) closed forms --------------------------------------------------

@pytest.mark.parametrize("coef", [(0.7, 0.0, 0.0), (0.7, -1.3, 0.0), (0.7, -1.3, 2.1)])
def test_taylor_forecast_closed_forms(coef):
    a, b, c = coef
    f = lambda tau: a + b * tau + c * tau * tau  # noqa: E731
    s = 0.1
    taus = [0.6, 0.6 + s, 0.6 + 2 * s]            # most recent (smallest t) first
    t = 0.6 - 0.05
    an = [(tau, np.array([f(tau)])) for tau in taus]
    dt = t - taus[0]
    # order 0: the cached value, exactly
    assert O.taylor_forecast(an[:1], t)[0] == f(taus[0])
    # order 1: exact for a linear history
    if c == 0.0:
        assert O.taylor_forecast(an[:2], t)[0] == pytest.approx(f(t), abs=1e-13)
    # order 2 with uniform spacing: error c * dt * (tau2 - tau1) (derived from Eqs. 3-5)
    err = O.taylor_forecast(an, t)[0] - f(t)
    assert err == pytest.approx(c * dt * (taus[1] - taus[0]), abs=1e-13)


# -- plan expansion against the paper's phi* (golden) --------------------------------------

def _phi_cases():
    with open(os.path.join(GOLD, "phi_star.json")) as fh:
        return json.load(fh)["cases"]


@pytest.mark.parametrize("case", _phi_cases(), ids=lambda c: c["name"])
def test_plan_from_phi_golden(case):
    skip, proxy = O.plan_from_phi(case["S"], case["S_prime"], case["n_skip"], case["l_start"],
                                  case["l_end"], case["f_full"], 0, case["depth"])
    assert skip.shape == (case["S_prime"], case["depth"])
    assert int(skip.sum()) == case["n_skip_entries"]
    assert int((proxy != -1).sum()) == case["n_proxy_entries"]
    assert int(((proxy == -1) & (skip == 0)).sum()) == case["n_compute_entries"]
    full = [k for k in range(case["S_prime"]) if np.all(proxy[k] == -1)]
    assert full == case["full_steps"]
    # skipped layers are exactly L_skip (1-indexed) from step n_skip on
    for k in range(case["S_prime"]):
        on = set(np.flatnonzero(skip[k]) + 1)
        want = set(range(case["l_start"], case["l_end"] + 1)) if k >= case["n_skip"] else set()
        assert on == want
    O.resolve_plan(skip, proxy)  # valid


def test_resolve_plan_rejects_bad_plans():
    skip, proxy = synth.empty_plan(3, 2)
    proxy[1, 0] = synth.proxy_code(1, 0)      # source not earlier
    with pytest.raises(ValueError):
        O.resolve_plan(skip, proxy)
    skip, proxy = synth.empty_plan(3, 2)
    skip[0, 1] = 1
    proxy[1, 1] = synth.proxy_code(0, 0)      # layer skipped at the source step
    with pytest.raises(ValueError):
        O.resolve_plan(skip, proxy)
    skip, proxy = synth.empty_plan(3, 2)
    skip[1, 0] = 1
    proxy[1, 0] = synth.proxy_code(0, 0)      # skip and proxy both set
    with pytest.raises(ValueError):
        O.resolve_plan(skip, proxy)
    skip, proxy = synth.empty_plan(3, 2)
    proxy[2, 0] = synth.proxy_code(1, 3)      # order 3
    with pytest.raises(ValueError):
        O.resolve_plan(skip, proxy)


def test_resolve_plan_anchor_ramp():
    skip, proxy = synth.empty_plan(6, 1)
    for k in (1, 3, 5):
        proxy[k, 0] = synth.proxy_code(k - 1, 2)
    an = O.resolve_plan(skip, proxy)
    assert an[(1, 0)] == [0] and an[(3, 0)] == [2, 0] and an[(5, 0)] == [4, 2, 0]


# -- model-level invariants --------------------------------------------------------------

def _tiny(norm_std=0.2):
    cfg = synth.TINY
    w = synth.make_weights(cfg, bf16=False, norm_std=norm_std)
    return cfg, w


def test_block_matches_library_composition():
    """The block restated with torch library routines (layer_norm, linear, rms_norm,
    scaled_dot_product_attention, gelu) on the same weights."""
    cfg, w = _tiny()
    m = O.OracleModel(cfg, w)
    h = rng.standard_normal((cfg.tokens, cfg.dim))
    temb, mod = m.time_embed(0.7)
    kv = m.encode_text(synth.make_text(cfg))
    out = m.block(1, h, mod, kv[1])

    T = {k: t64(v) for k, v in w.items()}
    p = "blocks.1."
    D, H, dh = cfg.dim, cfg.heads, cfg.head_dim
    md = t64(mod) + T[p + "table"]
    x = t64(h)
    a = Fn.layer_norm(x, (D,), eps=1e-6) * (1 + md[1]) + md[0]
    qkv = Fn.linear(a, T[p + "attn.wqkv"], T[p + "attn.bqkv"])
    q = Fn.rms_norm(qkv[:, :D], (D,), T[p + "attn.norm_q"], eps=1e-6)
    k = Fn.rms_norm(qkv[:, D:2 * D], (D,), T[p + "attn.norm_k"], eps=1e-6)
    v = qkv[:, 2 * D:]
    cos, sin = O.rope_tables(cfg.grid_h, cfg.grid_w, dh, cfg.rope_theta)

    def rope(u):  # complex-multiplication form
        uc = torch.view_as_complex(u.reshape(-1, H, dh // 2, 2).contiguous())
        rot = torch.polar(torch.ones_like(t64(cos)), torch.atan2(t64(sin), t64(cos)))
        return torch.view_as_real(uc * rot[:, None, :]).reshape(-1, H, dh)

    q, k = rope(q), rope(k)
    o = Fn.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1),
                                        v.reshape(-1, H, dh).transpose(0, 1)).transpose(0, 1)
    x = x + md[2] * Fn.linear(o.reshape(-1, D), T[p + "attn.wo"], T[p + "attn.bo"])
    a = Fn.layer_norm(x, (D,), T[p + "norm3.w"], T[p + "norm3.b"], eps=1e-6)
    qc = Fn.rms_norm(Fn.linear(a, T[p + "cross.wq"], T[p + "cross.bq"]), (D,),
                     T[p + "cross.norm_q"], eps=1e-6)
    ctx = t64(synth.make_text(cfg))
    ctx = Fn.linear(Fn.gelu(Fn.linear(ctx, T["text.w1"], T["text.b1"]), approximate="tanh"),
                    T["text.w2"], T["text.b2"])
    kvc = Fn.linear(ctx, T[p + "cross.wkv"], T[p + "cross.bkv"])
    kc = Fn.rms_norm(kvc[:, :D], (D,), T[p + "cross.norm_k"], eps=1e-6)
    vc = kvc[:, D:]
    oc = Fn.scaled_dot_product_attention(qc.reshape(-1, H, dh).transpose(0, 1),
                                         kc.reshape(-1, H, dh).transpose(0, 1),
                                         vc.reshape(-1, H, dh).transpose(0, 1)).transpose(0, 1)
    x = x + Fn.linear(oc.reshape(-1, D), T[p + "cross.wo"], T[p + "cross.bo"])
    a = Fn.layer_norm(x, (D,), eps=1e-6) * (1 + md[4]) + md[3]
    f = Fn.gelu(Fn.linear(a, T[p + "ffn.w1"], T[p + "ffn.b1"]), approximate="tanh")
    x = x + md[5] * Fn.linear(f, T[p + "ffn.w2"], T[p + "ffn.b2"])
    np.testing.assert_allclose(out, x.numpy(), rtol=1e-9, atol=1e-11)


def test_time_embed_matches_library_composition():
    """temb = Linear(SiLU(Linear(emb(1000 t)))) and mod = Linear(SiLU(temb)) as [6, D],
    restated with torch library routines at several t."""
    cfg, w = _tiny()
    m = O.OracleModel(cfg, w)
    T = {k: t64(v) for k, v in w.items()}
    for t in (1.0, 0.7, 0.13):
        temb, mod = m.time_embed(t)
        e = t64(O.timestep_embedding(t, cfg.freq_dim))
        want_t = Fn.linear(Fn.silu(Fn.linear(e, T["time.w1"], T["time.b1"])),
                           T["time.w2"], T["time.b2"])
        want_m = Fn.linear(Fn.silu(want_t), T["mod.w"], T["mod.b"]).reshape(6, cfg.dim)
        np.testing.assert_allclose(temb, want_t.numpy(), rtol=1e-12, atol=1e-13)
        np.testing.assert_allclose(mod, want_m.numpy(), rtol=1e-12, atol=1e-13)


def test_head_matches_library_composition():
    """Head: LayerNorm (no affine) * (1 + table_1 + temb) + table_0 + temb, then
    Linear(D -> C p p), restated with torch library routines; head.w is non-zero."""
    cfg, w = _tiny()
    w = dict(w)
    w["head.table"] = (rng.standard_normal((2, cfg.dim)) * 0.3).astype(np.float32)
    m = O.OracleModel(cfg, w)
    h = rng.standard_normal((cfg.tokens, cfg.dim)) * 2 + 0.5
    temb, _ = m.time_embed(0.45)
    got = m.head(h, temb)
    T = {k: t64(v) for k, v in w.items()}
    tb = T["head.table"]
    a = Fn.layer_norm(t64(h), (cfg.dim,), eps=cfg.eps_ln) * (1 + tb[1] + t64(temb)) \
        + tb[0] + t64(temb)
    want = Fn.linear(a, T["head.w"], T["head.b"]).numpy()
    assert np.abs(w["head.w"]).max() > 0 and np.abs(want).max() > 0.1
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)


def _hand_cfg(dim, heads=1, head_dim=None):
    """One token (a 2x2 latent with one channel, patch 2), so RoPE is the identity and
    attention returns its single value row; LayerNorm eps 0 keeps hand values exact."""
    return synth.Cfg(depth=1, dim=dim, heads=heads, head_dim=head_dim or dim, ffn=dim,
                     text_len=1, text_dim=dim, latent_c=1, latent_h=2, latent_w=2,
                     freq_dim=4, eps_ln=0.0)


def _zero_weights(cfg):
    return {n: np.zeros(s, np.float64) for n, s, _ in synth.weight_specs(cfg)}


# logistic sigmoid at the points used below: 1/(1+e^-x)
SIG2, SIGM1 = 0.8807970779778823, 0.2689414213699951


def test_time_embed_hand_values_fix_silu_and_chunk_order():
    """D = 2, t = 0: the sinusoid is [cos 0, cos 0, sin 0, sin 0] = [1, 1, 0, 0].
    Case 1 pins the first SiLU and the cos-first order: pre-activation [2, -1] gives
    temb = [2 sig(2), -sig(-1)]. Case 2 pins the SiLU before the modulation and the
    row order of the [6, D] split: row k of mod is output features 2k, 2k+1."""
    cfg = _hand_cfg(2, head_dim=4)
    w = _zero_weights(cfg)
    w["time.w1"][0, 0], w["time.w1"][1, 1] = 2.0, -1.0
    w["time.w2"][:] = np.eye(2)
    w["mod.b"][:] = np.arange(12)
    temb, mod = O.OracleModel(cfg, w).time_embed(0.0)
    np.testing.assert_allclose(temb, [2 * SIG2, -SIGM1], rtol=1e-14)
    np.testing.assert_allclose(mod, np.arange(12).reshape(6, 2), atol=0)
    # case 2: temb = b2 = [2, -1] exactly; mod row 2 (the first gate) reads SiLU(temb)
    w["time.w1"][:] = 0
    w["time.w2"][:] = 0
    w["time.b2"][:] = [2.0, -1.0]
    w["mod.b"][:] = 0
    w["mod.w"][4] = [1.0, 0.0]          # row 2, feature 0 <- SiLU(temb)_0
    w["mod.w"][11] = [0.0, 3.0]         # row 5, feature 1 <- 3 SiLU(temb)_1
    temb, mod = O.OracleModel(cfg, w).time_embed(0.0)
    np.testing.assert_allclose(temb, [2.0, -1.0], atol=0)
    want = np.zeros((6, 2))
    want[2, 0], want[5, 1] = 2 * SIG2, -3 * SIGM1
    np.testing.assert_allclose(mod, want, rtol=1e-14, atol=1e-300)


def test_head_hand_values_fix_shift_and_scale():
    """D = 2, h = [1, -1] (LayerNorm with eps 0 is the identity on it), table rows
    [0.5, 0.25] and [1, 2], temb [0.125, 0.5]: scale 1 + [1.125, 2.5], shift
    [0.625, 0.75], a = [2.75, -2.75]; head rows [1,0], [0,1], [1,1], [1,-1] with bias
    [0, 0, 0, 1] give v = [2.75, -2.75, 0, 6.5]. Swapping the rows, or dropping temb
    from either, changes v."""
    cfg = _hand_cfg(2, head_dim=4)
    w = _zero_weights(cfg)
    w["head.table"][:] = [[0.5, 0.25], [1.0, 2.0]]
    w["head.w"][:] = [[1, 0], [0, 1], [1, 1], [1, -1]]
    w["head.b"][:] = [0, 0, 0, 1]
    v = O.OracleModel(cfg, w).head(np.array([[1.0, -1.0]]), np.array([0.125, 0.5]))
    np.testing.assert_allclose(v, [[2.75, -2.75, 0.0, 6.5]], atol=1e-15)


def test_block_hand_values_fix_the_modulation_chunks():
    """D = 4, one head, one token, h = [1, -1, 1, -1] (its own LayerNorm with eps 0).
    All matrices are zero except the value part of W_qkv, W_o, W_1 and W_2 (identity),
    so attention returns v = a and the cross branch adds nothing. Given
    mod rows s1 = 0.5, c1 = 1, g1 = [1, 2, 3, 4], s2 = 0, c2 = -1, g2 = [10, 20, 30, 40]
    and b_2 = 1:
      a1 = LN(h)(1 + c1) + s1 = [2.5, -1.5, 2.5, -1.5];  h1 = h + g1 a1 = [3.5, -4, 8.5, -7]
      a2 = LN(h1)(1 + c2) + s2 = 0;  FFN = W_2 GELU(0) + b_2 = 1;  h2 = h1 + g2.
    A swapped shift/scale or a wrong gate row changes the result."""
    cfg = _hand_cfg(4)
    w = _zero_weights(cfg)
    p = "blocks.0."
    w[p + "attn.wqkv"][8:12] = np.eye(4)
    w[p + "attn.wo"][:] = np.eye(4)
    w[p + "ffn.w1"][:] = np.eye(4)
    w[p + "ffn.w2"][:] = np.eye(4)
    w[p + "ffn.b2"][:] = 1.0
    for n in ("attn.norm_q", "attn.norm_k", "cross.norm_q", "cross.norm_k", "norm3.w"):
        w[p + n][:] = 1.0
    m = O.OracleModel(cfg, w)
    mod = np.array([[0.5] * 4, [1.0] * 4, [1, 2, 3, 4], [0.0] * 4, [-1.0] * 4,
                    [10, 20, 30, 40]], np.float64)
    kv = (np.zeros((1, 4)), np.zeros((1, 4)))
    out = m.block(0, np.array([[1.0, -1.0, 1.0, -1.0]]), mod, kv)
    np.testing.assert_allclose(out, [[13.5, 16.0, 38.5, 33.0]], atol=1e-13)


def test_skip_equals_zero_contribution_block():
    """Eq. 6: skipping block l equals running a model whose block l adds nothing."""
    cfg, w = _tiny()
    z = synth.make_latents(cfg, 1)[0]
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(3)
    skip, proxy = synth.empty_plan(3, cfg.depth)
    skip[:, 1] = 1
    a = O.OracleModel(cfg, w).sample_one(z, O.OracleModel(cfg, w).encode_text(ctx), sched,
                                         skip, proxy)
    w0 = dict(w)
    for n in ("attn.wo", "attn.bo", "cross.wo", "cross.bo", "ffn.w2", "ffn.b2"):
        w0["blocks.1." + n] = np.zeros_like(w["blocks.1." + n])
    m0 = O.OracleModel(cfg, w0)
    b = m0.sample_one(z, m0.encode_text(ctx), sched, *synth.empty_plan(3, cfg.depth))
    np.testing.assert_allclose(a, b, rtol=1e-13, atol=1e-13)


def test_order0_proxy_step_adds_cached_contributions():
    """An all-proxy order-0 step: h_L = h_0 + sum_l Delta_l^(src)."""
    cfg, w = _tiny()
    m = O.OracleModel(cfg, w)
    z = synth.make_latents(cfg, 1)[0]
    kv = m.encode_text(synth.make_text(cfg))
    sched = synth.make_schedule(4)[:3]
    skip, proxy = synth.empty_plan(2, cfg.depth)
    proxy[1, :] = synth.proxy_code(0, 0)
    trace = []
    m.sample_one(z, kv, sched, skip, proxy, trace=trace)
    # step 0 by hand from the components
    temb0, mod0 = m.time_embed(sched[0])
    h = m.patch_embed(z)
    deltas = []
    for l in range(cfg.depth):
        hn = m.block(l, h, mod0, kv[l])
        deltas.append(hn - h)
        h = hn
    v = m.head(h, temb0)
    z1 = z + (sched[1] - sched[0]) * O.unpatchify(v, cfg.latent_c, cfg.latent_h, cfg.latent_w, 2)
    h1 = m.patch_embed(z1) + sum(deltas)
    last = [x for x in trace if x[0] == 1][-1][2]
    np.testing.assert_allclose(last, h1, rtol=1e-12, atol=1e-12)


def test_constant_velocity_integrates_exactly():
    """dx = v dt with a constant field: z(t_end) = z(t_0) + (t_end - t_0) v."""
    cfg, w = _tiny()
    w = dict(w)
    w["head.w"] = np.zeros_like(w["head.w"])
    w["head.b"] = np.linspace(-1, 1, cfg.patch_dim).astype(np.float32)
    m = O.OracleModel(cfg, w)
    z = synth.make_latents(cfg, 1)[0]
    sched = synth.make_schedule(5)
    out = m.sample_one(z, m.encode_text(synth.make_text(cfg)), sched, *synth.empty_plan(5, 2))
    v = O.unpatchify(np.tile(w["head.b"], (cfg.tokens, 1)), cfg.latent_c, cfg.latent_h,
                     cfg.latent_w, 2)
    want = z.astype(np.float64) + (float(sched[-1]) - float(sched[0])) * v
    np.testing.assert_allclose(out, want, rtol=1e-12, atol=1e-12)


def test_markov_draft_then_refine_equals_full_run():
    """Stage 3: resuming from the step-k latent with phi_full equals one full run."""
    cfg, w = _tiny()
    m = O.OracleModel(cfg, w)
    z = synth.make_latents(cfg, 1)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(6)
    full = m.draft(z, ctx, sched, *synth.empty_plan(6, 2))[0]
    part = m.draft(z, ctx, sched[:3], *synth.empty_plan(2, 2))[0]
    np.testing.assert_array_equal(m.refine(part, ctx, sched[2:]), full)


def test_candidates_are_independent():
    cfg, w = _tiny()
    m = O.OracleModel(cfg, w)
    z = synth.make_latents(cfg, 3)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(4)
    sk, px = synth.tiny_plan()
    all3 = m.draft(z, ctx, sched, sk, px)
    np.testing.assert_array_equal(m.draft(z, ctx, sched, sk, px, candidates=[2])[0], all3[2])


# -- the cached state and a warm-started refine (§4.2 Stage 3, reading R12) ------------------

def test_state_holds_each_layers_last_computed_contribution():
    """keep_state returns, per layer, Delta_l = h_after - h_before at the layer's last
    computed step and that step's t; checked against the trace of h after each layer."""
    cfg, w = _tiny()
    m = O.OracleModel(cfg, w)
    z = synth.make_latents(cfg, 1)[0]
    ctx = synth.make_text(cfg)
    kv = m.encode_text(ctx)
    sched = synth.make_schedule(4)
    skip, proxy = synth.tiny_plan()          # layer 1 skipped at step 2, layer 0 proxied at 3
    trace = []
    zo, state = m.sample_one(z, kv, sched, skip, proxy, trace=trace, keep_state=True)
    np.testing.assert_array_equal(zo, m.sample_one(z, kv, sched, skip, proxy))
    h = {(i, l): x for i, l, x in trace}
    z2 = m.sample_one(z, kv, sched[:3], skip[:2], proxy[:2])
    assert sorted(state) == [0, 1]
    assert state[0][0] == sched[2] and state[1][0] == sched[3]
    np.testing.assert_allclose(state[0][1], h[(2, 0)] - m.patch_embed(z2), rtol=0, atol=1e-12)
    np.testing.assert_allclose(state[1][1], h[(3, 1)] - h[(3, 0)], rtol=0, atol=1e-12)


def test_refine_without_warm_steps_is_phi_full():
    cfg, w = _tiny()
    m = O.OracleModel(cfg, w)
    z = synth.make_latents(cfg, 1)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(5)
    zd, states = m.draft(z, ctx, sched[:3], *synth.empty_plan(2, 2), keep_state=True)
    np.testing.assert_array_equal(m.refine(zd[0], ctx, sched[2:], state=states[0], warm_steps=0),
                                  m.refine(zd[0], ctx, sched[2:]))


def test_warm_step_adds_the_cached_state():
    """A warm step proxies every layer from the state: h_L = PatchEmbed(z) + sum_l Delta_l,
    then the Euler step; the steps after it are phi_full."""
    cfg, w = _tiny()
    m = O.OracleModel(cfg, w)
    z = synth.make_latents(cfg, 1)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(6)
    zd, states = m.draft(z, ctx, sched[:3], *synth.empty_plan(2, 2), keep_state=True)
    st = states[0]
    t0, t1 = sched[2], sched[3]
    temb, _ = m.time_embed(t0)
    hL = m.patch_embed(zd[0]) + st[0][1] + st[1][1]
    v = O.unpatchify(m.head(hL, temb), cfg.latent_c, cfg.latent_h, cfg.latent_w, cfg.patch)
    z1 = zd[0].astype(np.float64) + (float(t1) - float(t0)) * v
    np.testing.assert_allclose(m.refine(zd[0], ctx, sched[2:], state=st, warm_steps=1),
                               m.refine(z1, ctx, sched[3:]), rtol=0, atol=1e-12)


def test_state_proxy_rules():
    skip = np.zeros((2, 2), np.uint8)
    proxy = np.full((2, 2), O.COMPUTE, np.int32)
    proxy[0, 1] = O.STATE_SRC
    assert O.resolve_plan(skip, proxy, state_layers=(0, 1))[(0, 1)] == ["state"]
    with pytest.raises(ValueError):
        O.resolve_plan(skip, proxy, state_layers=(0,))         # layer 1 not in the state
    proxy[0, 1] = O.STATE_SRC | (1 << 16)
    with pytest.raises(ValueError):
        O.resolve_plan(skip, proxy, state_layers=(0, 1))       # order 1 from a single anchor


# -- classifier-free guidance and the SDE step (App. A.1) -----------------------------------

def test_sde_step_hand_value():
    # t = 0.5, t' = 0.4, a = 0.3: sigma = 0.3; drift 2 + 0.09/1.0 * (1 + 0.5*2) = 2.18
    z = O.euler_maruyama_step(np.array([1.0]), np.array([2.0]), 0.5, 0.4, 0.3, np.array([0.5]))
    assert z[0] == pytest.approx(1.0 - 0.218 + 0.3 * math.sqrt(0.1) * 0.5, abs=1e-14)


def test_sde_step_with_a0_is_the_ode_step():
    z, v, eps = rng.standard_normal(50), rng.standard_normal(50), rng.standard_normal(50)
    np.testing.assert_array_equal(O.euler_maruyama_step(z, v, 0.7, 0.6, 0.0, eps), z + (0.6 - 0.7) * v)


def test_sde_sigma_at_t1_uses_next_timestep():
    assert O.sde_sigma(1.0, 0.98, 0.7) == pytest.approx(0.7 * math.sqrt(0.98 / 0.02))
    assert O.sde_sigma(0.5, 0.48, 0.7) == pytest.approx(0.7)


def test_sde_preserves_rectified_flow_marginals():
    """App. A.1: the SDE keeps the ODE's marginals. Toy problem with a known velocity:
    x_0 ~ N(0, s^2), x_1 ~ N(0, 1), x_t = (1-t) x_0 + t x_1 has variance
    (1-t)^2 s^2 + t^2 and marginal velocity v(x, t) = x (t - (1-t) s^2) / var_t. Start
    from N(0, 1) at t = 1 and integrate to t = 0.25 with many particles."""
    s2 = 0.25
    var = lambda t: (1 - t) ** 2 * s2 + t * t  # noqa: E731
    vel = lambda x, t: x * (t - (1 - t) * s2) / var(t)  # noqa: E731
    g = np.random.default_rng(3)
    x = g.standard_normal(200_000)
    ts = np.linspace(1.0, 0.25, 301)
    for t, tn in zip(ts[:-1], ts[1:]):
        x = O.euler_maruyama_step(x, vel(x, t), t, tn, 0.7, g.standard_normal(x.size))
    assert x.var() == pytest.approx(var(0.25), rel=0.03)
    # a drift correction with the wrong sign does not preserve the marginals
    y = g.standard_normal(200_000)
    for t, tn in zip(ts[:-1], ts[1:]):
        sig = O.sde_sigma(t, tn, 0.7)
        v = vel(y, t)
        y = y + (v - sig * sig / (2 * t) * (y + (1 - t) * v)) * (tn - t) + \
            sig * math.sqrt(t - tn) * g.standard_normal(y.size)
    assert abs(y.var() / var(0.25) - 1) > 0.1


def test_guided_velocity_endpoints():
    vc, vu = rng.standard_normal(9), rng.standard_normal(9)
    np.testing.assert_array_equal(O.guided_velocity(vc, vu, 1.0), vu + (vc - vu))
    np.testing.assert_allclose(O.guided_velocity(vc, vu, 1.0), vc, rtol=0, atol=1e-15)
    np.testing.assert_array_equal(O.guided_velocity(vc, vu, 0.0), vu)


def test_cfg_with_identical_contexts_is_unguided():
    cfg, w = _tiny()
    m = O.OracleModel(cfg, w)
    z = synth.make_latents(cfg, 1)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(3)
    sk, px = synth.empty_plan(3, 2)
    px[2, 0] = synth.proxy_code(1, 1)
    a = m.draft(z, ctx, sched, sk, px)
    b = m.draft(z, ctx, sched, sk, px, ctx_uncond=ctx, guidance=4.0)
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-12)


# -- multi-stage Elo selection (§4.2 Stage 2) ------------------------------------------------

def test_elo_seed_values_from_the_paper():
    assert O.elo_seed(5) == 1500.0 and O.elo_seed(10) == 2000.0 and O.elo_seed(1) == 1100.0


def test_elo_update_hand_values():
    # equal ratings: E = 1/2; high confidence K = 32 * 1.2 = 38.4 -> +/- 19.2
    ra, rb = O.elo_update(1500.0, 1500.0, True, 32.0 * O.CONF_MULT[0])
    assert (ra, rb) == (pytest.approx(1519.2), pytest.approx(1480.8))
    # 400 points apart: E_a = 1/11; an upset with K = 32 moves a by 32 * 10/11
    ra, rb = O.elo_update(1500.0, 1900.0, True, 32.0)
    assert ra == pytest.approx(1500.0 + 32.0 * 10.0 / 11.0)
    assert ra + rb == pytest.approx(3400.0)  # zero-sum


def test_elo_select_call_counts_and_survivors():
    """Defaults at M = 32: M1 = 16, C2 = 24 adjacent comparisons, M2 = 8, 28 tournament
    games: 52 pairwise calls, the paper's 'roughly 3/2 M'."""
    g = np.random.default_rng(0)
    quality = g.standard_normal(32)
    scores = np.clip(np.round(5 + 2 * quality), 1, 10).astype(int)
    seen = []

    def cmp(a, b):
        seen.append((a, b))
        return quality[a] > quality[b], 0
    w, r, calls = O.elo_select(scores, cmp)
    assert calls == 52 == len(seen)
    assert len({x for p in seen for x in p}) <= 16          # only survivors of stage 1 play
    assert w in {x for p in seen[24:] for x in p}           # the winner played the tournament


def test_elo_select_finds_the_best_with_a_consistent_verifier():
    g = np.random.default_rng(1)
    for trial in range(20):
        quality = g.standard_normal(24)
        scores = np.clip(np.round(5 + 2 * quality), 1, 10).astype(int)
        w, _, _ = O.elo_select(scores, lambda a, b: (quality[a] > quality[b], 1))
        assert w == int(np.argmax(quality))


def test_elo_select_ties_go_to_lower_index():
    w, r, calls = O.elo_select([7, 7, 7, 7], lambda a, b: (a < b, 2), rho1=1.0, rho2=1.0,
                               kappa=0.0)
    assert w == 0 and calls == 6
