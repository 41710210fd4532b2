"""CPU oracle for the Flash-BoN draft-generation path (fp64, plain numpy).

TEST INFRASTRUCTURE ONLY. Only tests/, __graft_entry__.smoke() and bench.py's
cpu_baseline / reference leg may import or run this module. The product path (the
C-ABI library and its Python binding) never calls it, and this module imports nothing
from the product package: weights and inputs are passed in as arrays.

What it computes (paper: "Flash-BoN", §3-§4 and App. A.1):
  * the sampler of §3: S steps z_{t_{i-1}} = f_theta(z_{t_i}, x, t_i) (Eq. 2), each a
    pass through L sequential blocks B_1..B_L, truncated to the first S' steps
    (§4.1 knob 1, early timestep stopping);
  * the flow-matching ODE dx = v dt (App. A.1) integrated with the Euler step
    z <- z + (t' - t) v, time running from noise t=1 to data t=0;
  * layer skipping (§4.1 knob 3, Eq. 6): a skipped block passes h^(l-1) through;
  * activation proxies (§4.1 knob 2, Eqs. 3-5): the second-order Taylor forecast
    from cached features at earlier (larger-t) steps, used in place of the block;
  * Stage 1 draft generation over M seeds (§4.2, Eq. 8) and Stage 3 selective
    refinement with phi_full (§4.2): the Markov property lets refinement resume from
    the cached latent;
  * the configuration phi = (S', n_skip, l_start, l_end, f_full) (§4.1,
    "Configuration Space") expanded into per-(step, layer) decisions.

The denoiser f_theta is a black box in the paper (§3 names a DiT). The block below is a
Wan2.1-style DiT block: adaLN with 6-way modulation from the time embedding, q/k
RMSNorm, 2-D axial RoPE, self-attention, affine LayerNorm + cross-attention to the
projected text, and a GELU(tanh) FFN; gated residuals.

Readings where the paper is silent or ambiguous (all arithmetic in fp64):
  R1 the cache holds a block's contribution Delta_l = B_l(h) - h; a proxied block
     adds its forecast Delta (the Taylor forecast is linear in the anchors, so this
     equals forecasting per sub-branch and summing);
  R2 Taylor anchors are the most recent computed steps of that layer at or before the
     proxy's source step, most recent first (tau1 < tau2 < tau3 in t); Eqs. 3-5 are
     applied literally with tau in place of t_{i+1}, t_{i+2}, t_{i+3}; with fewer anchors
     than order+1 the order drops (0 -> 1 -> 2 as anchors accumulate);
  R3 f_full: draft step k (0-based) is full iff k mod f_full == 0; other steps proxy
     every non-skipped layer from the last full step;
  R4 n_skip: layers in L_skip (1-indexed in the paper) are skipped at steps k >= n_skip;
  R5 schedule t_i = 1 - i/S; the embedding sees 1000 t.
  R6 classifier-free guidance (used by the paper only for its GRPO experiments): the
     conditional and unconditional passes run through the same plan, each with its own
     proxy cache, and the step uses v = v_u + w (v_c - v_u);
  R7 SDE sampling (App. A.1, Euler-Maruyama form of the reverse SDE): with dt = t' - t < 0
     the noise term is sigma_t sqrt(|dt|) eps; sigma_t = a sqrt(t / (1 - t)) is undefined
     at t = 1, where it is evaluated at the next timestep t' instead.
  R8 Elo selection (§4.2 Stage 2): base K and the expected-score formula are not given;
     K = 32 and the logistic 400-point expected score are used; the adjacent comparisons
     are passes over the rating-sorted survivors; ties go to the lower index.
  R12 cached state (§4.2 Stage 3): the optional layer activations kept for warm-starting
     activation proxies are, under R1, each layer's contribution Delta_l from its last
     computed draft step, with that step's t. A refine step may proxy layer l from it
     (order 0: h <- h + Delta_l); with no such steps the refine is phi_full exactly.
"""
from __future__ import annotations

import numpy as np

F64 = np.float64
COMPUTE = -1
STATE_SRC = 0xFFFF  # proxy source: the cached state of an earlier call (R12), order 0


# ----------------------------------------------------------------------------------
# primitives
# ----------------------------------------------------------------------------------

def linear(x, w, b=None):
    """y = x W^T + b with W stored [out, in]."""
    y = x @ w.T
    return y if b is None else y + b


def layer_norm(x, eps, weight=None, bias=None):
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    y = (x - mu) / np.sqrt(var + eps)
    if weight is not None:
        y = y * weight
    if bias is not None:
        y = y + bias
    return y


def rms_norm(x, weight, eps):
    return x / np.sqrt((x * x).mean(axis=-1, keepdims=True) + eps) * weight


def silu(x):
    return x / (1.0 + np.exp(-x))


def gelu_tanh(x):
    return 0.5 * x * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (x + 0.044715 * x ** 3)))


def timestep_embedding(t, dim=256, max_period=10000.0, scale=1000.0):
    """Sinusoidal embedding of scale*t: [cos(scale t f_k), sin(scale t f_k)],
    f_k = max_period^(-k/half), k = 0..half-1."""
    half = dim // 2
    freqs = np.exp(-np.log(max_period) * np.arange(half, dtype=F64) / half)
    args = scale * F64(t) * freqs
    return np.concatenate([np.cos(args), np.sin(args)])


def rope_tables(grid_h, grid_w, head_dim, theta):
    """cos/sin [P, head_dim/2] for 2-D axial RoPE: the first head_dim/2 dims rotate by
    the token's row, the last head_dim/2 by its column; in each half pair j uses
    frequency theta^(-2j/half)."""
    half = head_dim // 2
    freqs = theta ** (-np.arange(0, half, 2, dtype=F64) / half)         # [half/2]
    rows = np.repeat(np.arange(grid_h, dtype=F64), grid_w)             # token -> row
    cols = np.tile(np.arange(grid_w, dtype=F64), grid_h)               # token -> col
    ang = np.concatenate([rows[:, None] * freqs, cols[:, None] * freqs], axis=1)
    return np.cos(ang), np.sin(ang)


def apply_rope(x, cos, sin):
    """x [P, H, dh]; rotates adjacent pairs (x[2j], x[2j+1]) by the angle of pair j:
    (a, b) -> (a cos - b sin, a sin + b cos)."""
    a, b = x[..., 0::2], x[..., 1::2]
    c, s = cos[:, None, :], sin[:, None, :]
    out = np.empty_like(x)
    out[..., 0::2] = a * c - b * s
    out[..., 1::2] = a * s + b * c
    return out


def attention(q, k, v):
    """softmax(q k^T / sqrt(dh)) v per head; q [Lq, H, dh], k/v [Lk, H, dh]."""
    dh = q.shape[-1]
    out = np.empty_like(q)
    for h in range(q.shape[1]):
        s = q[:, h, :] @ k[:, h, :].T / np.sqrt(dh)
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p = p / p.sum(axis=1, keepdims=True)
        out[:, h, :] = p @ v[:, h, :]
    return out


def patchify(z, p):
    """[C, H, W] -> [P, C p p]; token (r, c) is row r*(W/p) + c, its vector element
    ch*p*p + dy*p + dx is z[ch, r p + dy, c p + dx]."""
    C, H, W = z.shape
    return z.reshape(C, H // p, p, W // p, p).transpose(1, 3, 0, 2, 4).reshape(
        (H // p) * (W // p), C * p * p)


def unpatchify(x, C, H, W, p):
    return x.reshape(H // p, W // p, C, p, p).transpose(2, 0, 3, 1, 4).reshape(C, H, W)


def taylor_forecast(anchors, t):
    """Eqs. 3-5 with cached anchors [(tau1, h1), (tau2, h2), (tau3, h3)], most recent
    (smallest tau) first, forecasting the value at t (< tau1):
        dh  = (h1 - h2) / (tau1 - tau2)
        ddh = (h1 - 2 h2 + h3) / (tau1 - tau2)^2
        h~  = h1 + dt dh + dt^2 ddh / 2,   dt = t - tau1.
    One anchor: h1 (order 0). Two anchors: the first-order truncation."""
    tau1, h1 = anchors[0]
    if len(anchors) == 1:
        return h1
    tau2, h2 = anchors[1]
    dt = F64(t) - F64(tau1)
    hdot = (h1 - h2) / (F64(tau1) - F64(tau2))
    if len(anchors) == 2:
        return h1 + dt * hdot
    _, h3 = anchors[2]
    hddot = (h1 - 2.0 * h2 + h3) / (F64(tau1) - F64(tau2)) ** 2
    return h1 + dt * hdot + 0.5 * dt * dt * hddot


def sde_sigma(t, t_next, a):
    """sigma_t = a sqrt(t / (1 - t)) (App. A.1); at t = 1 evaluated at t_next (R7)."""
    te = F64(t_next) if F64(t) >= 1.0 else F64(t)
    return F64(a) * np.sqrt(te / (1.0 - te))


def euler_maruyama_step(z, v, t, t_next, a, eps):
    """One step of App. A.1's update, with dt = t_next - t:
        z + [v + sigma^2 / (2 t) (z + (1 - t) v)] dt + sigma sqrt(|dt|) eps."""
    t, t_next = F64(t), F64(t_next)
    dt = t_next - t
    sig = sde_sigma(t, t_next, a)
    return z + (v + sig * sig / (2.0 * t) * (z + (1.0 - t) * v)) * dt + sig * np.sqrt(abs(dt)) * eps


def guided_velocity(v_cond, v_uncond, w):
    """Classifier-free guidance: v = v_u + w (v_c - v_u)."""
    return v_uncond + F64(w) * (v_cond - v_uncond)


# ----------------------------------------------------------------------------------
# plan: phi expansion and validation
# ----------------------------------------------------------------------------------

def plan_from_phi(S, S_prime, n_skip, l_start, l_end, f_full, order, depth):
    """Expand phi = (S', n_skip, l_start, l_end, f_full) (§4.1) into
    skip_mask [S'][L] (uint8) and proxy_plan [S'][L] (int32: -1 compute, else
    src_step | order << 16). Readings R3, R4; layers are 1-indexed in phi."""
    if not (1 <= S_prime <= S) or f_full < 1 or not (1 <= l_start <= l_end <= depth) \
            or n_skip < 0 or not (0 <= order <= 2):
        raise ValueError("invalid phi")
    skip = np.zeros((S_prime, depth), np.uint8)
    proxy = np.full((S_prime, depth), COMPUTE, np.int32)
    for k in range(S_prime):
        full = (k % f_full) == 0
        last_full = k - (k % f_full)
        for l in range(depth):
            if k >= n_skip and (l_start - 1) <= l <= (l_end - 1):
                skip[k, l] = 1
            elif not full:
                proxy[k, l] = last_full | (order << 16)
    return skip, proxy


def resolve_plan(skip, proxy, state_layers=()):
    """Validate a plan and list, per proxied (step, layer), its anchor steps (most recent
    first); a proxy from the cached state (source STATE_SRC, R12) has the anchor "state".
    Raises ValueError on: skip and proxy both set; source step not earlier than the step;
    layer not computed at the source step; order outside 0..2; a state proxy of order > 0
    or of a layer the state does not hold."""
    skip = np.asarray(skip)
    proxy = np.asarray(proxy)
    S, L = skip.shape
    computed = {l: [] for l in range(L)}
    anchors = {}
    for k in range(S):
        for l in range(L):
            code = int(proxy[k, l])
            if code == COMPUTE:
                if not skip[k, l]:
                    computed[l].append(k)
                continue
            if skip[k, l]:
                raise ValueError(f"step {k} layer {l}: skipped and proxied")
            if code < 0:
                raise ValueError(f"step {k} layer {l}: bad proxy code {code}")
            src, order = code & 0xFFFF, code >> 16
            if src == STATE_SRC:
                if order != 0 or l not in state_layers:
                    raise ValueError(f"step {k} layer {l}: bad proxy from the cached state")
                anchors[(k, l)] = ["state"]
                continue
            if order > 2:
                raise ValueError(f"step {k} layer {l}: order {order} > 2")
            if src >= k:
                raise ValueError(f"step {k} layer {l}: source step {src} not earlier")
            if src not in computed[l]:
                raise ValueError(f"step {k} layer {l}: not computed at source step {src}")
            past = [s for s in computed[l] if s <= src][::-1]
            anchors[(k, l)] = past[: order + 1]
    return anchors


# ----------------------------------------------------------------------------------
# model
# ----------------------------------------------------------------------------------

class OracleModel:
    """fp64 DiT denoiser f_theta plus the Flash-BoN sampler around it."""

    def __init__(self, cfg, weights):
        self.cfg = cfg
        self.w = {k: np.asarray(v, dtype=F64) for k, v in weights.items()}
        self.cos, self.sin = rope_tables(cfg.grid_h, cfg.grid_w, cfg.head_dim,
                                         cfg.rope_theta)

    # -- conditioning ---------------------------------------------------------------
    def time_embed(self, t):
        """temb = W2 SiLU(W1 emb(1000 t) + b1) + b2; mod = W_mod SiLU(temb) + b_mod,
        as [6, D] rows (shift1, scale1, gate1, shift2, scale2, gate2)."""
        w = self.w
        e = timestep_embedding(t, self.cfg.freq_dim)
        temb = linear(silu(linear(e, w["time.w1"], w["time.b1"])), w["time.w2"], w["time.b2"])
        mod = linear(silu(temb), w["mod.w"], w["mod.b"]).reshape(6, self.cfg.dim)
        return temb, mod

    def encode_text(self, ctx):
        """Text projection Linear-GELU(tanh)-Linear, then per block the cross-attention
        keys (RMSNorm) and values. Invariant across steps and candidates."""
        w, cfg = self.w, self.cfg
        x = linear(gelu_tanh(linear(np.asarray(ctx, F64), w["text.w1"], w["text.b1"])),
                   w["text.w2"], w["text.b2"])
        kv = []
        for l in range(cfg.depth):
            p = f"blocks.{l}."
            if p + "cross.wkv" not in w:
                kv.append(None)
                continue
            y = linear(x, w[p + "cross.wkv"], w[p + "cross.bkv"])
            k = rms_norm(y[:, : cfg.dim], w[p + "cross.norm_k"], cfg.eps_rms)
            v = y[:, cfg.dim:]
            kv.append((k, v))
        return kv

    def patch_embed(self, z):
        return linear(patchify(np.asarray(z, F64), self.cfg.patch), self.w["patch.w"],
                      self.w["patch.b"])

    # -- one block B_l (Eq. 7) ------------------------------------------------------
    def block(self, l, h, mod, ctx_kv):
        cfg, w = self.cfg, self.w
        p = f"blocks.{l}."
        D, H, dh = cfg.dim, cfg.heads, cfg.head_dim
        P = h.shape[0]
        s1, c1, g1, s2, c2, g2 = mod + w[p + "table"]
        # self-attention branch
        a = layer_norm(h, cfg.eps_ln) * (1.0 + c1) + s1
        qkv = linear(a, w[p + "attn.wqkv"], w[p + "attn.bqkv"])
        q = rms_norm(qkv[:, :D], w[p + "attn.norm_q"], cfg.eps_rms)
        k = rms_norm(qkv[:, D:2 * D], w[p + "attn.norm_k"], cfg.eps_rms)
        v = qkv[:, 2 * D:]
        q = apply_rope(q.reshape(P, H, dh), self.cos, self.sin)
        k = apply_rope(k.reshape(P, H, dh), self.cos, self.sin)
        o = attention(q, k, v.reshape(P, H, dh)).reshape(P, D)
        h = h + g1 * linear(o, w[p + "attn.wo"], w[p + "attn.bo"])
        # cross-attention branch (affine LayerNorm, no modulation, no gate)
        a = layer_norm(h, cfg.eps_ln, w[p + "norm3.w"], w[p + "norm3.b"])
        q = rms_norm(linear(a, w[p + "cross.wq"], w[p + "cross.bq"]),
                     w[p + "cross.norm_q"], cfg.eps_rms)
        kc, vc = ctx_kv
        T = kc.shape[0]
        o = attention(q.reshape(P, H, dh), kc.reshape(T, H, dh), vc.reshape(T, H, dh))
        h = h + linear(o.reshape(P, D), w[p + "cross.wo"], w[p + "cross.bo"])
        # feed-forward branch
        a = layer_norm(h, cfg.eps_ln) * (1.0 + c2) + s2
        f = gelu_tanh(linear(a, w[p + "ffn.w1"], w[p + "ffn.b1"]))
        return h + g2 * linear(f, w[p + "ffn.w2"], w[p + "ffn.b2"])

    def head(self, h, temb):
        """Output head: LayerNorm with 2-way modulation (table + temb), then
        Linear(D -> C p p); returns the velocity patches [P, C p p]."""
        w, cfg = self.w, self.cfg
        shift = w["head.table"][0] + temb
        scale = w["head.table"][1] + temb
        a = layer_norm(h, cfg.eps_ln) * (1.0 + scale) + shift
        return linear(a, w["head.w"], w["head.b"])

    # -- sampler ----------------------------------------------------------------------
    def _blocks(self, i, h, t, mod, ctx_kv, skip, proxy, anchors, needed, cache, trace,
                last=None):
        """Blocks of step i on h: skip (Eq. 6), compute (Eq. 7, caching Delta_l when a
        later proxy needs it; with `last`, also recording each layer's latest (t, Delta_l),
        R12) or proxy (Eqs. 3-5)."""
        for l in range(self.cfg.depth):
            if skip[i][l]:
                continue
            if int(proxy[i][l]) == COMPUTE:
                h_new = self.block(l, h, mod, ctx_kv[l])
                if (i, l) in needed:
                    cache[(i, l)] = (t, h_new - h)
                if last is not None:
                    last[l] = (t, h_new - h)
                h = h_new
            else:
                h = h + taylor_forecast([cache[(s, l)] if s != "state" else cache[("state", l)]
                                         for s in anchors[(i, l)]], t)
            if trace is not None:
                trace.append((i, l, h.copy()))
        return h

    def sample_one(self, z, ctx_kv, schedule, skip, proxy, trace=None, ctx_kv_uncond=None,
                   guidance=1.0, sde_a=0.0, noise=None, keep_state=False, state=None):
        """One candidate through len(schedule)-1 steps under (skip, proxy).

        Step i goes from t = schedule[i] to t' = schedule[i+1]: h_0 = PatchEmbed(z);
        the blocks; v = Head(h); z <- z + (t' - t) v (the Euler step of dx = v dt).
        With ctx_kv_uncond the step runs a second, unconditional pass with its own proxy
        cache and uses the guided velocity (R6). With sde_a > 0 the step is App. A.1's
        Euler-Maruyama update with the standard normal draws noise[i] (R7).

        keep_state: also return the cached state, {layer: (t, Delta_l)} of each layer's
        last computed step (R12; the conditional pass). state: such a dict, the source of
        proxies coded STATE_SRC (single pass only)."""
        cfg = self.cfg
        sched = np.asarray(schedule, F64)
        n_steps = len(sched) - 1
        if state is not None and ctx_kv_uncond is not None:
            raise ValueError("a cached state warm-starts a single (unguided) pass")
        anchors = resolve_plan(skip, proxy, () if state is None else tuple(state))
        needed = {(s, l) for (k, l), steps in anchors.items() for s in steps if s != "state"}
        passes = [ctx_kv] if ctx_kv_uncond is None else [ctx_kv, ctx_kv_uncond]
        caches = [{} for _ in passes]
        if state is not None:
            for l, tl_d in state.items():
                caches[0][("state", l)] = tl_d
        last = {} if keep_state else None
        z = np.asarray(z, F64).copy()
        for i in range(n_steps):
            t, t_next = sched[i], sched[i + 1]
            temb, mod = self.time_embed(t)
            vs = []
            for kv, cache in zip(passes, caches):
                cond = kv is ctx_kv
                h = self._blocks(i, self.patch_embed(z), t, mod, kv, skip, proxy, anchors,
                                 needed, cache, trace if cond else None,
                                 last if cond else None)
                vs.append(unpatchify(self.head(h, temb), cfg.latent_c, cfg.latent_h,
                                     cfg.latent_w, cfg.patch))
            v = vs[0] if len(vs) == 1 else guided_velocity(vs[0], vs[1], guidance)
            if sde_a > 0:
                z = euler_maruyama_step(z, v, t, t_next, sde_a, np.asarray(noise[i], F64))
            else:
                z = z + (t_next - t) * v
        return (z, last) if keep_state else z

    def draft(self, z_T, ctx, schedule, skip, proxy, candidates=None, ctx_uncond=None,
              guidance=1.0, sde_a=0.0, noise=None, keep_state=False):
        """Stage 1 (Eq. 8): each candidate's z_T through the truncated, accelerated
        schedule. Candidates are independent; `candidates` picks a subset. noise, when
        sde_a > 0, is [n_steps][N][C][H][W] (indexed by the candidate's position in z_T).
        keep_state: also return each candidate's cached state (R12), a list of dicts."""
        z_T = np.asarray(z_T)
        idx = range(z_T.shape[0]) if candidates is None else candidates
        kv = self.encode_text(ctx)
        kvu = None if ctx_uncond is None else self.encode_text(ctx_uncond)
        out, states = [], []
        for j in idx:
            nz = None if noise is None else np.asarray(noise)[:, j]
            r = self.sample_one(z_T[j], kv, schedule, skip, proxy, ctx_kv_uncond=kvu,
                                guidance=guidance, sde_a=sde_a, noise=nz, keep_state=keep_state)
            if keep_state:
                out.append(r[0])
                states.append(r[1])
            else:
                out.append(r)
        return (np.stack(out), states) if keep_state else np.stack(out)

    def refine(self, z, ctx, schedule, ctx_uncond=None, guidance=1.0, sde_a=0.0, noise=None,
               state=None, warm_steps=0):
        """Stage 3: resume from a cached latent with phi_full (no skip, no proxy).
        noise, when sde_a > 0, is [n_steps][C][H][W]. With a cached state (R12) the first
        warm_steps steps proxy every layer the state holds from it (order 0)."""
        n = len(schedule) - 1
        skip = np.zeros((n, self.cfg.depth), np.uint8)
        proxy = np.full((n, self.cfg.depth), COMPUTE, np.int32)
        if state is not None:
            for i in range(min(warm_steps, n)):
                for l in state:
                    proxy[i, l] = STATE_SRC
        kvu = None if ctx_uncond is None else self.encode_text(ctx_uncond)
        return self.sample_one(z, self.encode_text(ctx), schedule, skip, proxy,
                               ctx_kv_uncond=kvu, guidance=guidance, sde_a=sde_a, noise=noise,
                               state=state)


# ----------------------------------------------------------------------------------
# Stage 2: multi-stage selection with Elo ratings (§4.2)
# ----------------------------------------------------------------------------------

CONF_MULT = (1.2, 1.0, 0.7)  # confidence high / medium / low scales K (§4.2 footnote)


def elo_seed(score):
    """r^(0) = 1500 + (s - 5) * 100."""
    return 1500.0 + (float(score) - 5.0) * 100.0


def elo_update(ra, rb, a_wins, k):
    """Standard Elo: expected score E_a = 1 / (1 + 10^((r_b - r_a) / 400)) (R8: the
    paper does not print it)."""
    ea = 1.0 / (1.0 + 10.0 ** ((rb - ra) / 400.0))
    sa = 1.0 if a_wins else 0.0
    return ra + k * (sa - ea), rb + k * ((1.0 - sa) - (1.0 - ea))


def _top(ids, r, count):
    """The `count` best by rating; ties go to the lower index."""
    return sorted(ids, key=lambda j: (-r[j], j))[:count]


def elo_select(scores, compare, rho1=0.5, rho2=0.5, kappa=1.5, k_base=32.0):
    """Pointwise pruning + Elo seeding, sparse adjacent comparisons, dense tournament.

    compare(a, b) -> (a_preferred: bool, confidence in {0, 1, 2}). Readings (R8): base K
    = k_base; the ceil(kappa M1) adjacent comparisons are passes over the list sorted by
    rating (from the top), the list re-sorted before each pass; the tournament plays the
    pairs (i, j), i < j, of the survivors in rating order. Returns (winner, ratings,
    pairwise calls)."""
    import math
    M = len(scores)
    r = {j: elo_seed(scores[j]) for j in range(M)}
    calls = 0

    def play(a, b):
        nonlocal calls
        a_wins, conf = compare(a, b)
        calls += 1
        r[a], r[b] = elo_update(r[a], r[b], a_wins, k_base * CONF_MULT[conf])

    ceil = lambda x: math.ceil(x - 1e-9)  # noqa: E731  (0.3 * 20 is 6, not 7)
    s1 = _top(range(M), r, ceil(rho1 * M))
    c2 = ceil(kappa * len(s1))
    done = 0
    while done < c2 and len(s1) > 1:
        order = _top(s1, r, len(s1))
        for i in range(len(order) - 1):
            if done == c2:
                break
            play(order[i], order[i + 1])
            done += 1
    s2 = _top(s1, r, ceil(rho2 * len(s1)))
    order = _top(s2, r, len(s2))
    for i in range(len(order)):
        for j in range(i + 1, len(order)):
            play(order[i], order[j])
    winner = _top(s2, r, 1)[0]
    return winner, [r[j] for j in range(M)], calls
