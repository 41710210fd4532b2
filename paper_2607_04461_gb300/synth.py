"""Seeded synthetic inputs for the Flash-BoN draft path.

This module produces DATA only: model configurations, random-init weights, initial
latents z_T, text contexts, timestep schedules and (skip_mask, proxy_plan) tables. It
holds none of the method's arithmetic. Both the CUDA path (through the C-ABI binding)
and the CPU oracle consume what it returns; neither imports the other.

Recipe (the paper's benchmarks and trained weights are not available, so seeded
synthetic stand-ins with the workloads' shapes are used):
  * weights: N(0, 0.02) per tensor, each tensor drawn from its own PCG64 stream seeded
    by (seed, tensor ordinal); norm scales are 1 + N(0, norm_std). For bf16 configs
    the values are rounded to bf16 (round to nearest even) here, so both sides see the
    identical numbers.
  * initial latents z_T^(j) ~ N(0, I), candidate j from seed 1000 + j (Stage 1, Eq. 8:
    one Gaussian draw per seed).
  * text context ~ N(0, 1) of shape [text_len, text_dim] (a padded prompt embedding).
  * schedule t_i = 1 - i/S, i = 0..S (flow-matching time runs from noise t=1 to data t=0).
"""
from __future__ import annotations

import dataclasses
import numpy as np

FREQ_DIM = 256  # sinusoidal timestep-embedding width


@dataclasses.dataclass(frozen=True)
class Cfg:
    depth: int
    dim: int
    heads: int
    head_dim: int
    ffn: int
    text_len: int
    text_dim: int
    latent_c: int
    latent_h: int
    latent_w: int
    patch: int = 2
    max_n: int = 1
    eps_ln: float = 1e-6
    eps_rms: float = 1e-6
    rope_theta: float = 10000.0
    freq_dim: int = FREQ_DIM

    @property
    def grid_h(self) -> int:
        return self.latent_h // self.patch

    @property
    def grid_w(self) -> int:
        return self.latent_w // self.patch

    @property
    def tokens(self) -> int:
        return self.grid_h * self.grid_w

    @property
    def patch_dim(self) -> int:
        return self.latent_c * self.patch * self.patch

    def with_(self, **kw) -> "Cfg":
        return dataclasses.replace(self, **kw)


# Tiny DiT: 2 blocks, hidden 128, 2 heads of 64, FFN 512; 8x8x4 latent -> 16 tokens;
# text 8 x 128; fp32 weights.
TINY = Cfg(depth=2, dim=128, heads=2, head_dim=64, ffn=512, text_len=8, text_dim=128,
           latent_c=4, latent_h=8, latent_w=8, max_n=4)
# Wan2.1-1.3B shape: 30 blocks, hidden 1536, 12 x 128 heads, FFN 8960, text 512 x 4096,
# 480x832 image -> 16 x 60 x 104 latent -> 1560 tokens.
WAN13 = Cfg(depth=30, dim=1536, heads=12, head_dim=128, ffn=8960, text_len=512,
            text_dim=4096, latent_c=16, latent_h=60, latent_w=104, max_n=32)
# Wan2.1-14B shape: 40 blocks, hidden 5120, 40 x 128 heads, FFN 13824.
WAN14 = WAN13.with_(depth=40, dim=5120, heads=40, ffn=13824, max_n=8)
# 1024x1024 image -> 16 x 128 x 128 latent -> 4096 tokens, Wan2.1-1.3B dims.
WAN13_1K = WAN13.with_(latent_h=128, latent_w=128, max_n=64)
# Small test shape: spans several GEMM / attention tiles with ragged tails
# (150 tokens per candidate, 40 text tokens).
SMALL = Cfg(depth=3, dim=256, heads=2, head_dim=128, ffn=1024, text_len=40, text_dim=256,
            latent_c=16, latent_h=20, latent_w=30, max_n=3)


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bf16 (ties to even); returns float32."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


def weight_specs(cfg: Cfg):
    """Ordered (name, shape, kind) of every model tensor; kind in {w, b, norm, table}.

    Linear weights are [out, in]. The order and names match the packed weight layout
    of the C-ABI (fb_weights_entry)."""
    D, F, C = cfg.dim, cfg.ffn, cfg.patch_dim
    specs = [
        ("patch.w", (D, C), "w"), ("patch.b", (D,), "b"),
        ("time.w1", (D, cfg.freq_dim), "w"), ("time.b1", (D,), "b"),
        ("time.w2", (D, D), "w"), ("time.b2", (D,), "b"),
        ("mod.w", (6 * D, D), "w"), ("mod.b", (6 * D,), "b"),
        ("text.w1", (D, cfg.text_dim), "w"), ("text.b1", (D,), "b"),
        ("text.w2", (D, D), "w"), ("text.b2", (D,), "b"),
        ("head.table", (2, D), "table"), ("head.w", (C, D), "w"), ("head.b", (C,), "b"),
    ]
    for l in range(cfg.depth):
        p = f"blocks.{l}."
        specs += [
            (p + "table", (6, D), "table"),
            (p + "attn.wqkv", (3 * D, D), "w"), (p + "attn.bqkv", (3 * D,), "b"),
            (p + "attn.norm_q", (D,), "norm"), (p + "attn.norm_k", (D,), "norm"),
            (p + "attn.wo", (D, D), "w"), (p + "attn.bo", (D,), "b"),
            (p + "norm3.w", (D,), "norm"), (p + "norm3.b", (D,), "b"),
            (p + "cross.wq", (D, D), "w"), (p + "cross.bq", (D,), "b"),
            (p + "cross.wkv", (2 * D, D), "w"), (p + "cross.bkv", (2 * D,), "b"),
            (p + "cross.norm_q", (D,), "norm"), (p + "cross.norm_k", (D,), "norm"),
            (p + "cross.wo", (D, D), "w"), (p + "cross.bo", (D,), "b"),
            (p + "ffn.w1", (F, D), "w"), (p + "ffn.b1", (F,), "b"),
            (p + "ffn.w2", (D, F), "w"), (p + "ffn.b2", (D,), "b"),
        ]
    return specs


def make_weights(cfg: Cfg, seed: int = 0, std: float = 0.02, norm_std: float = 0.02,
                 bf16: bool = True, layers=None) -> dict:
    """Random-init weights, one PCG64 stream per tensor (seeded by (seed, ordinal)).

    layers: optional iterable of block indices to generate (others are omitted), used
    when only some blocks are needed."""
    keep = None if layers is None else {f"blocks.{l}." for l in layers}
    out = {}
    for idx, (name, shape, kind) in enumerate(weight_specs(cfg)):
        if keep is not None and name.startswith("blocks.") and \
                name[: name.index(".", 7) + 1] not in keep:
            continue
        rng = np.random.default_rng([seed, idx])
        x = rng.standard_normal(shape, dtype=np.float32)
        if kind == "norm":
            x = 1.0 + np.float32(norm_std) * x
        else:
            x = np.float32(std) * x
        out[name] = bf16_round(x) if bf16 else x.astype(np.float32)
    return out


def make_weights_device(cfg: Cfg, seed: int = 0, std: float = 0.02,
                        norm_std: float = 0.02) -> dict:
    """make_weights' distributions drawn on the current CUDA device (torch, one seeded
    stream per tensor, values rounded to bf16): random-init weights for shapes whose
    host generation takes minutes (the 14B model). Not the host generator's numbers."""
    import torch
    out = {}
    for idx, (name, shape, kind) in enumerate(weight_specs(cfg)):
        g = torch.Generator(device="cuda").manual_seed(seed * 1_000_003 + idx)
        x = torch.randn(shape, generator=g, device="cuda", dtype=torch.float32)
        x = 1.0 + norm_std * x if kind == "norm" else std * x
        out[name] = x.to(torch.bfloat16).to(torch.float32)
    return out


def make_latents(cfg: Cfg, n: int, seed_base: int = 1000, first: int = 0) -> np.ndarray:
    """z_T for candidates first..first+n-1; candidate j is N(0, I) from seed seed_base + j."""
    z = np.empty((n, cfg.latent_c, cfg.latent_h, cfg.latent_w), dtype=np.float32)
    for i in range(n):
        rng = np.random.default_rng(seed_base + first + i)
        z[i] = rng.standard_normal(z.shape[1:], dtype=np.float32)
    return z


def make_text(cfg: Cfg, seed: int = 7) -> np.ndarray:
    rng = np.random.default_rng(seed)
    return rng.standard_normal((cfg.text_len, cfg.text_dim), dtype=np.float32)


def make_noise(cfg: Cfg, n_steps: int, n: int, seed: int = 2000) -> np.ndarray:
    """Standard normal draws for SDE steps: [n_steps][n][C][H][W] float32."""
    rng = np.random.default_rng(seed)
    return rng.standard_normal((n_steps, n, cfg.latent_c, cfg.latent_h, cfg.latent_w),
                               dtype=np.float32)


def make_schedule(S: int) -> np.ndarray:
    """t_i = 1 - i/S for i = 0..S (float32)."""
    return (1.0 - np.arange(S + 1, dtype=np.float64) / S).astype(np.float32)


COMPUTE = -1


def proxy_code(src_step: int, order: int) -> int:
    """proxy_plan entry: reuse/forecast from anchors at or before src_step."""
    return int(src_step) | (int(order) << 16)


def empty_plan(n_steps: int, depth: int):
    return (np.zeros((n_steps, depth), np.uint8),
            np.full((n_steps, depth), COMPUTE, np.int32))


def tiny_plan():
    """Tiny config plan: 4 steps, block 1 skipped at step 2, block 0 at step 3 reuses
    the step-1 contribution (0-indexed steps and blocks)."""
    skip, proxy = empty_plan(4, 2)
    skip[2, 1] = 1
    proxy[3, 0] = proxy_code(1, 0)
    return skip, proxy


def random_plan(n_steps: int, depth: int, skip_frac: float, proxy_frac: float,
                seed: int = 7, order: int = 0):
    """Seeded plan: at every step a uniform-random subset of round(skip_frac*depth)
    blocks is skipped; on odd steps round(proxy_frac * remaining) of the non-skipped
    blocks that were computed at the previous step reuse that step's contribution
    (proxy_code(k-1, order)); everything else is computed."""
    rng = np.random.default_rng(seed)
    skip, proxy = empty_plan(n_steps, depth)
    n_skip = int(round(skip_frac * depth))
    for k in range(n_steps):
        s = rng.choice(depth, size=n_skip, replace=False) if n_skip else []
        skip[k, s] = 1
        if k % 2 == 1 and proxy_frac > 0:
            live = np.flatnonzero(skip[k] == 0)
            eligible = [l for l in live if skip[k - 1, l] == 0 and proxy[k - 1, l] == COMPUTE]
            want = int(round(proxy_frac * len(live)))
            pick = rng.permutation(eligible)[:want]
            for l in pick:
                proxy[k, l] = proxy_code(k - 1, order)
    return skip, proxy
