"""Benchmark of the Flash-BoN draft path on GB300: draft candidates/s at the
Wan2.1-1.3B shape.

Workload (one "step" = one pass of the whole hot path over one batch):
  Wan2.1-1.3B-shaped DiT (30 blocks, hidden 1536, 12 x 128 heads, FFN 8960, text
  512 x 4096 projected to 1536), 480x832 image -> 16 x 60 x 104 latent -> 1560 tokens;
  N = 32 candidates drafted over the first 10 steps of a 50-step flow-matching schedule
  (t_i = 1 - i/50) with 1/3 of the blocks skipped per step (seeded) and, on odd steps,
  half of the remaining blocks proxied from the previous step's cached contribution;
  then candidate 0 is refined with full computation over the remaining 40 steps.
  Synthetic bf16 random-init weights N(0, 0.02), latents and text context N(0, 1).

value = candidates per second (N / step time) with inputs resident in HBM; e2e = the
same through the C-ABI with host (pinned) latents and text, copies inside the timed
region. The working set (2.6 GB of weights, 0.5-1 GB activations per kernel) is far
larger than L2, so no L2 flush is done between steps.

--impl reference times the CPU oracle (fp64 numpy) on a bounded sample of the same
workload and extrapolates the same metric.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2607_04461_gb300 import synth  # noqa: E402

METRIC = "draft candidates/sec at Wan2.1-1.3B shape (1 GB300); tensor-pipe % of bf16 peak"
N_CAND, S_TOTAL, S_DRAFT = 32, 50, 10
SKIP_FRAC, PROXY_FRAC, PLAN_SEED = 1 / 3, 0.5, 7


def workload():
    cfg = synth.WAN13.with_(max_n=N_CAND)
    sched = synth.make_schedule(S_TOTAL)
    skip, proxy = synth.random_plan(S_DRAFT, cfg.depth, SKIP_FRAC, PROXY_FRAC, seed=PLAN_SEED)
    return cfg, sched, skip, proxy


# The paper's searched configuration phi* on the Wan2.1-1.3B shape (Sec. 4.1): S = 50,
# S' = 49 draft steps, blocks 22-23 skipped from step 3 on, a full step every 5 steps, the
# others forecast with second-order proxies; N = 8 candidates; the remaining step refines
# candidate 0.
PHI_STAR = dict(S=50, S_prime=49, n_skip=3, l_start=22, l_end=23, f_full=5, order=2)
PHI_N = 8
# The 14B draft pool: N = 8, the first 10 of 50 steps, a seeded quarter of the blocks
# skipped per step, every remaining block proxied on odd steps; the drafts only.
W14_N = 8


def plan_for(variant):
    """(cfg, schedule, skip, proxy, draft steps) of a bench variant."""
    if variant == "wan14":  # the 14B draft pool; the schedule ends with the draft
        cfg = synth.WAN14.with_(max_n=W14_N)
        skip, proxy = synth.random_plan(S_DRAFT, cfg.depth, 0.25, 1.0, seed=PLAN_SEED)
        return cfg, synth.make_schedule(S_TOTAL)[: S_DRAFT + 1], skip, proxy, S_DRAFT
    if variant == "full50":  # the same N and schedule sampled without any acceleration
        cfg = synth.WAN13.with_(max_n=PHI_N)
        skip, proxy = synth.empty_plan(PHI_STAR["S"], cfg.depth)
        return cfg, synth.make_schedule(PHI_STAR["S"]), skip, proxy, PHI_STAR["S"]
    if variant != "phi_star":
        cfg, sched, skip, proxy = workload()
        return cfg, sched, skip, proxy, S_DRAFT
    from paper_2607_04461_gb300 import flashbon as fb
    cfg = synth.WAN13.with_(max_n=PHI_N)
    ph = PHI_STAR
    skip, proxy = fb.fb_plan_from_phi(ph["S"], ph["S_prime"], ph["n_skip"], ph["l_start"],
                                      ph["l_end"], ph["f_full"], ph["order"], cfg.depth)
    return cfg, synth.make_schedule(ph["S"]), skip, proxy, ph["S_prime"]


VARIANTS = {
    "base": "",
    "cfg": "; classifier-free guidance w=5 (16 candidates, 32 rows with the unconditional pass)",
    "sde": "; Euler-Maruyama SDE steps, a=0.7, caller-supplied N(0,1) draws",
    "offload": "; every candidate's cached state (each layer's last contribution, bf16, "
               "144 MB per candidate) copied to pinned host memory behind the refine and "
               "the next draft",
    "phi_star": "",
    "full50": "",
    "wan14": "",
    "sweep": "",
}


# variants whose value pass may run with the split schedule (see run_gb300). Not the
# guided one: its refine runs two rows and two cross-attention passes per block and on
# 40 SMs outlasts the draft (13.71 against 15.86 cand/s sequential).
SPLIT_VARIANTS = ("base", "sde")
REFINE_SMS = 40


def n_candidates(variant):
    return {"cfg": N_CAND // 2, "phi_star": PHI_N, "full50": PHI_N,
            "wan14": W14_N}.get(variant, N_CAND)


def config_dict(cfg, variant="base"):
    n = n_candidates(variant)
    if variant == "phi_star":
        ph = PHI_STAR
        return {"workload": f"wan2.1-1.3B, the paper's phi*: N={n}, 480x832 (1560 tokens), "
                            f"{ph['S_prime']} of {ph['S']} steps, blocks {ph['l_start']}-"
                            f"{ph['l_end']} skipped from step {ph['n_skip']}, a full step "
                            f"every {ph['f_full']}, order-{ph['order']} proxies between, "
                            "then the remaining step of candidate 0",
                "n_candidates": n, "tokens": cfg.tokens, "dim": cfg.dim, "depth": cfg.depth,
                "draft_steps": ph["S_prime"], "refine_steps": ph["S"] - ph["S_prime"],
                "l2": "inputs larger than L2 (2.6 GB weights), no flush"}
    if variant == "wan14":
        return {"workload": f"wan2.1-14B draft pool: N={n}, 480x832 (1560 tokens), 10 of 50 "
                            "steps, 1/4 of the blocks skipped per step, on odd steps every "
                            "remaining block the previous step computed proxied; the drafts "
                            "only (no refine); random-init weights drawn on the GPU",
                "n_candidates": n, "tokens": cfg.tokens, "dim": cfg.dim, "depth": cfg.depth,
                "draft_steps": S_DRAFT, "refine_steps": 0,
                "l2": "inputs larger than L2 (28 GB weights), no flush"}
    if variant == "full50":
        return {"workload": f"wan2.1-1.3B: N={n}, 480x832 (1560 tokens), all 50 steps, every "
                            "block computed (sampling without the paper's acceleration)",
                "n_candidates": n, "tokens": cfg.tokens, "dim": cfg.dim, "depth": cfg.depth,
                "draft_steps": PHI_STAR["S"], "refine_steps": 0,
                "l2": "inputs larger than L2 (2.6 GB weights), no flush"}
    return {"workload": f"wan2.1-1.3B draft pool: N={n}, 480x832 (1560 tokens), 10 of 50 "
                        "steps, 1/3 blocks skipped, half of the rest proxied on odd steps, "
                        "then a 40-step full refine of candidate 0" + VARIANTS[variant],
            "n_candidates": n, "tokens": cfg.tokens, "dim": cfg.dim, "depth": cfg.depth,
            "draft_steps": S_DRAFT, "refine_steps": S_TOTAL - S_DRAFT,
            "l2": "inputs larger than L2 (2.6 GB weights), no flush"}


def block_flops(cfg):
    """Algorithmic FLOPs of one block for one candidate (cross K/V hoisted)."""
    P, D, F, T = cfg.tokens, cfg.dim, cfg.ffn, cfg.text_len
    lin = 2 * P * D * (3 * D + D + D + D) + 4 * P * D * F
    attn = 4 * P * P * D + 4 * P * T * D
    return lin + attn


def computed_blocks(skip, proxy):
    return int(((skip == 0) & (proxy == -1)).sum())


# ---------------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------------
class ClockSampler:
    Q = ("clocks.sm,clocks.max.sm,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index, self.proc = index, None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        self.lines = []
        if self.proc:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()
                out = ""
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for l in getattr(self, "lines", []):
            f = [x.strip() for x in l.split(",")]
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except (ValueError, IndexError):
                continue
            for n, v in zip(names, f[2:]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------------
# oracle (CPU) timing: bounded sample, extrapolated
# ---------------------------------------------------------------------------------
def oracle_sample(cfg, sched, skip, proxy, budget_s):
    """Times the oracle's block on candidate 0 at step 0 (blocks in order) until the
    budget is spent; returns (seconds per computed block, blocks timed)."""
    from oracle import OracleModel
    n_blocks = max(1, min(cfg.depth, int(budget_s // 2) or 1))
    w = synth.make_weights(cfg, layers=range(n_blocks))
    sub = cfg.with_(depth=n_blocks)
    ref = OracleModel(sub, {k: v for k, v in w.items()})
    ctx = synth.make_text(cfg)
    kv = ref.encode_text(ctx)
    z = synth.make_latents(cfg, 1)[0]
    temb, mod = ref.time_embed(sched[0])
    h = ref.patch_embed(z)
    t0 = time.perf_counter()
    done = 0
    for l in range(n_blocks):
        h = ref.block(l, h, mod, kv[l])
        done += 1
        if time.perf_counter() - t0 > budget_s:
            break
    return (time.perf_counter() - t0) / done, done


def oracle_cands_per_s(per_block_s, cfg, skip, proxy):
    blocks = N_CAND * computed_blocks(skip, proxy) + (S_TOTAL - S_DRAFT) * cfg.depth
    return N_CAND / (blocks * per_block_s)


# ---------------------------------------------------------------------------------
def read_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as fh:
            d = json.load(fh)
        return d, "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


def gemm_traffic():
    """DRAM traffic of the tcgen05 GEMM per algorithmic byte, from the committed ncu
    captures (profiles/gemm_tc_traffic.json), if they were taken on the current kernel
    source; else None. Returns (combined ratio, {probe: ratio})."""
    src = os.path.join(ROOT, "paper_2607_04461_gb300", "csrc", "gemm_tc.cu")
    summ = os.path.join(ROOT, "profiles", "gemm_tc_traffic.json")
    if not os.path.exists(summ):
        return None
    sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    with open(summ) as fh:
        d = json.load(fh)
    if d.get("kernel_sha") != sha:
        return None
    probes = d["probes"]
    tot_t = sum(v["dram_read_bytes"] + v["dram_write_bytes"] for v in probes.values())
    tot_a = sum(v["algorithmic_bytes"] for v in probes.values())
    return tot_t / tot_a, {k: (v["dram_read_bytes"] + v["dram_write_bytes"]) /
                           v["algorithmic_bytes"] for k, v in probes.items()}


def aggregate(ms_local, n_local, world, reduce_max=None):
    """Whole-job throughput: every rank drafts n_local candidates; the job's time is the
    slowest rank's (max over ranks). reduce_max(x) returns the max of x over ranks."""
    ms = reduce_max(ms_local) if reduce_max else ms_local
    return ms, world * n_local / (ms / 1e3)


def rank_candidates(rank, n_local):
    """Candidate indices (latent seeds 1000 + index) drafted by `rank`."""
    return list(range(rank * n_local, (rank + 1) * n_local))


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def run_reference(args):
    ws, rank, _ = dist_env()
    if rank != 0:
        return 0
    cfg, sched, skip, proxy = workload()
    per_step = max(2.0, min(20.0, 120.0 / max(1, args.steps + args.warmup)))
    times = []
    for i in range(args.warmup + args.steps):
        pb, nb = oracle_sample(cfg, sched, skip, proxy, per_step)
        if i >= args.warmup:
            times.append(pb)
    pb = float(np.median(times))
    v = oracle_cands_per_s(pb, cfg, skip, proxy)
    cores = os.cpu_count()
    sample = (f"fp64 numpy oracle: Wan2.1-1.3B block forward of candidate 0 at step 0, "
              f"{nb} block(s) per step ({pb:.2f} s per block), extrapolated to the "
              f"workload's {N_CAND * computed_blocks(skip, proxy)} draft + "
              f"{(S_TOTAL - S_DRAFT) * cfg.depth} refine block evaluations")
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "candidates/s",
            "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * N_CAND / v, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_dict(cfg),
            "cpu_baseline": {"value": v, "unit": "candidates/s", "cores": cores,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": v, "unit": "candidates/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def run_gb300(args):
    import torch
    from paper_2607_04461_gb300 import flashbon as fb

    ws, rank, local = dist_env()
    torch.cuda.set_device(local)
    pg = None
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        pg = dist
    cfg, sched, skip, proxy, s_draft = plan_for(args.variant)
    NC = n_candidates(args.variant)
    t_setup = time.time()
    w = synth.make_weights_device(cfg) if args.variant == "wan14" else synth.make_weights(cfg)
    model = fb.Model(cfg, w)
    # the split schedule: step k's refine on a small SM partition beside step k + 1's
    # draft on the rest (green contexts); a second model instance serves the refine
    split, split_note, model_r = None, None, None
    if args.schedule != "seq" and args.variant in SPLIT_VARIANTS:
        try:
            split = fb.SmSplit(args.refine_sms)
        except fb.FlashBonError as e:
            if args.schedule == "split":
                raise
            split_note = f"sequential: no SM partition ({e})"
    if split:
        model_r = fb.Model(cfg.with_(max_n=2), w)
    del w
    torch.cuda.empty_cache()  # the generator's buffers (56 GB for the 14B weights)
    stream = torch.cuda.Stream()
    model.set_stream(stream)
    # each rank drafts its own candidates (weak scaling, no collective on the path)
    z0 = torch.from_numpy(synth.make_latents(cfg, NC, first=rank_candidates(rank, NC)[0])).cuda()
    ctx_h = synth.make_text(cfg)
    ctx = torch.from_numpy(ctx_h).cuda()
    z = torch.empty_like(z0)
    zr = torch.empty_like(z0[0])
    draft_sched, tail = sched[: s_draft + 1], sched[s_draft:]
    opts_d = opts_r = None
    if args.variant == "cfg":
        ctx_u = torch.from_numpy(synth.make_text(cfg, seed=8)).cuda()
        opts_d = opts_r = fb.make_opts(5.0, ctx_u)
    elif args.variant == "sde":
        nd = torch.from_numpy(synth.make_noise(cfg, S_DRAFT, NC, seed=2000 + rank)).cuda()
        nr = torch.from_numpy(synth.make_noise(cfg, S_TOTAL - S_DRAFT, 1, seed=3000 + rank)).cuda()
        opts_d, opts_r = fb.make_opts(sde_a=0.7, noise=nd), fb.make_opts(sde_a=0.7, noise=nr)
    states = []
    if args.variant == "offload":
        states = [torch.empty(model.state_bytes(), dtype=torch.uint8).pin_memory()
                  for _ in range(NC)]
        opts_d = fb.make_opts(keep_state=True)
    setup_s = time.time() - t_setup
    if split:
        s_ref, s_dr = split.streams
        t_dr = torch.cuda.ExternalStream(s_dr)
        zr2 = [torch.empty_like(z0[0]) for _ in range(2)]
        pipe = {"k": 0}

        def use_split():
            model.set_stream(s_dr)
            model.set_sm_budget(split.sms[1])
            model_r.set_stream(s_ref)
            model_r.set_sm_budget(split.sms[0])

        def pipe_step(z_in, z_buf, zr_bufs, ctx_in, to_dev):
            """Draft of a new pool (large part) while candidate 0 of the previous pool is
            refined (small part) on a worker thread of the library
            (fb_pipeline_step); both finished on return."""
            k = pipe["k"]
            if to_dev:  # on the drafter's stream, ahead of its draft
                with torch.cuda.stream(t_dr):
                    z_buf.copy_(z_in)
            else:
                z_buf.copy_(z_in)
            fb.fb_pipeline_step(model.handle, z_buf, z_buf.shape[0], ctx_in, draft_sched, skip,
                                proxy, model_r.handle if k > 0 else None,
                                zr_bufs[(k - 1) % 2] if k > 0 else None, tail, opts_d, opts_r)
            if to_dev:
                with torch.cuda.stream(t_dr):
                    zr_bufs[k % 2].copy_(z_buf[0])
                t_dr.synchronize()
            else:
                zr_bufs[k % 2].copy_(z_buf[0])
            pipe["k"] = k + 1
        use_split()

    def dev_step(after=None):
        with torch.cuda.stream(stream):
            z.copy_(z0)
        model.draft(z, ctx, draft_sched, skip, proxy, opts=opts_d)
        if after:
            after("draft")
        if states:   # every candidate's state to pinned host memory, behind the refine
            model.state_offload(0, states)
        with torch.cuda.stream(stream):
            zr.copy_(z[0])
        model.refine(zr, ctx, tail, opts=opts_r)
        if after:
            after("refine")

    def finish():  # the last step's offload copies belong to the timed region
        if states:
            model.state_wait()

    def value_step():
        if split:
            pipe_step(z0, z, zr2, ctx, True)
        else:
            dev_step()
    tstream = t_dr if split else stream
    # at least one untimed step with the split schedule: it fills the pipeline, so that
    # every timed step holds a draft and a refine
    for _ in range(max(args.warmup, 1 if split else 0)):
        value_step()
    finish()
    torch.cuda.synchronize()
    model.reset_stats()
    if model_r:
        model_r.reset_stats()
    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    # timed pass 1 (the reported value): no per-kernel instrumentation. With the split
    # schedule each timed step drafts a new pool and refines candidate 0 of the previous
    # one (the pipeline was filled in the warm-up); every call has returned, so all of
    # that work lies between the two events.
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        ev0.record(tstream)
        for _ in range(args.steps):
            value_step()
        finish()
        ev1.record(tstream)
        torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1)
    launch_stats = model.stats()
    if model_r:
        for k, v in model_r.stats().items():
            for f in ("launches", "flops", "bytes", "ms"):
                launch_stats[k][f] += v[f]
        # the roofline pass runs the steps one after the other on the whole GPU
        model.set_stream(stream)
        model.set_sm_budget(0)
    # timed pass 2 (roofline of the dominant kernel): the same K steps with CUDA events
    # around every tcgen05 GEMM launch on the library's stream. The events themselves
    # cost a few per cent of the step, which is why pass 1 runs without them.
    model.reset_stats()
    model.set_timing(1 << fb.K["gemm_tc"])
    e2, e3 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    finish()
    # the GEMM statistics of the draft and of the refine separately (each call collects
    # its launches' event times before it returns)
    by_phase = {ph: {"launches": 0, "ms": 0.0, "flops": 0.0} for ph in ("draft", "refine")}
    last = [model.stats()["gemm_tc"]]

    def after(ph):
        cur = model.stats()["gemm_tc"]
        for k in by_phase[ph]:
            by_phase[ph][k] += cur[k] - last[0][k]
        last[0] = cur
    with ClockSampler(local) as clk2s:
        e2.record(stream)
        for _ in range(args.steps):
            dev_step(after)
        finish()
        e3.record(stream)
        torch.cuda.synchronize()
    stats = model.stats()
    model.set_timing(0)
    ms_instrumented = e2.elapsed_time(e3)
    def reduce_max(x):
        t = torch.tensor([x], device="cuda")
        pg.all_reduce(t, op=pg.ReduceOp.MAX)
        return float(t.item())
    ms_step, value = aggregate(ms / args.steps, NC, ws, reduce_max if pg else None)
    if pg:
        pg.barrier()

    # end to end through the C-ABI with host buffers (pinned), copies inside the region
    zh = torch.empty(z0.shape, dtype=torch.float32, pin_memory=True)
    zrh = torch.empty(z0.shape[1:], dtype=torch.float32, pin_memory=True)
    zrh2 = [torch.empty(z0.shape[1:], dtype=torch.float32, pin_memory=True) for _ in range(2)]
    ctxh = torch.from_numpy(ctx_h).pin_memory()
    z0h = z0.cpu()
    if split:
        use_split()
        pipe["k"] = 0
    else:
        model.set_stream(None)

    def host_step():
        if split:
            pipe_step(z0h, zh, zrh2, ctxh, False)
            return
        zh.copy_(z0h)
        model.draft(zh, ctxh, draft_sched, skip, proxy, opts=opts_d)
        if states:
            model.state_offload(0, states)
        zrh.copy_(zh[0])
        model.refine(zrh, ctxh, tail, opts=opts_r)

    host_step()
    finish()
    torch.cuda.synchronize()
    if pg:
        pg.barrier()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        host_step()
    finish()
    e2e_s = (time.perf_counter() - t0) / args.steps
    if pg:
        t = torch.tensor([e2e_s], device="cuda")
        pg.all_reduce(t, op=pg.ReduceOp.MAX)
        e2e_s = float(t.item())
    zbytes = z0.numel() * 4
    h2d = zbytes + 2 * ctx_h.nbytes + zbytes // NC
    d2h = zbytes + zbytes // NC + sum(b.numel() for b in states)

    peaks, peak_kind = read_peaks()
    g = stats["gemm_tc"]
    achieved = g["flops"] / (g["ms"] / 1e3) / 1e12 if g["ms"] > 0 else None
    peak = peaks["bf16_tflops_sustained"]
    tr = gemm_traffic()
    ratio, per_probe = tr if tr else (None, None)
    traffic = ratio * g["bytes"] / g["launches"] if (ratio and g["launches"]) else None
    n_sm = torch.cuda.get_device_properties(local).multi_processor_count
    clk2 = clk2s.summary()

    def per_clock(tflops, mhz):
        """MACs per SM clock per SM: independent of the clock the work ran at."""
        return tflops * 1e12 / 2 / (mhz * 1e6 * n_sm) if (tflops and mhz) else None
    # the measured peak's own rate per clock: the sustained cuBLAS loop at its median clock
    peak_mhz = (peaks.get("clocks_under_load") or {}).get("sm_mhz_median")
    peak_pc = per_clock(peak, peak_mhz)
    launches = sum(s["launches"] for s in launch_stats.values())
    passes = 2 if args.variant == "cfg" else 1
    algo_flops = passes * (NC * computed_blocks(skip, proxy) * block_flops(cfg) +
                           (len(tail) - 1) * cfg.depth * block_flops(cfg))
    out = {"metric": METRIC, "value": value, "unit": "candidates/s", "n_gpus": ws,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
           "data": "synthetic",
           "config": {**config_dict(cfg, args.variant),
                      "schedule": (f"split: step k's refine of candidate 0 on {split.sms[0]} "
                                   f"SMs beside step k+1's draft on {split.sms[1]} (SM "
                                   "partitions); each timed step drafts a pool and refines "
                                   "the previous pool's candidate 0"
                                   if split else split_note or "sequential")},
           "roofline": {"bound": "tensor", "kernel": "gemm_tc (tcgen05/TMEM GEMM, all "
                        "projections)", "achieved": achieved, "peak": peak,
                        "unit": "TFLOP/s", "frac": (achieved / peak) if achieved else None,
                        "peak_kind": f"bf16 sustained, {peak_kind}",
                        "frac_burst": (achieved / peaks["bf16_tflops"]) if achieved else None,
                        "per_clock": {
                            "sm_mhz": clk2.get("sm_mhz"),
                            "mac_per_clk_per_sm": per_clock(achieved, clk2.get("sm_mhz")),
                            "peak_mac_per_clk_per_sm": peak_pc, "peak_sm_mhz": peak_mhz,
                            "frac": (per_clock(achieved, clk2.get("sm_mhz")) / peak_pc
                                     if (achieved and peak_pc and clk2.get("sm_mhz"))
                                     else None),
                            "note": "the GEMM launches' MACs per SM clock (median SM clock "
                                    "sampled during this pass) against the sustained cuBLAS "
                                    "loop's at its own median clock"},
                        "traffic": traffic,
                        "traffic_kind": "estimated" if traffic else None,
                        "traffic_note": "DRAM bytes per launch estimated as the ncu "
                                        "traffic/algorithmic ratio of three 8192-row probes "
                                        "(profiles/gemm_tc_traffic.json) x this run's "
                                        "algorithmic bytes per GEMM launch; null when the "
                                        "kernel source differs from the captured one",
                        "traffic_ratio_by_probe": per_probe,
                        "launches": g["launches"], "ms": g["ms"] / args.steps,
                        "measured_in": "timed pass 2 (same steps, one after the other on "
                                       "the whole GPU, per-launch CUDA events on the "
                                       "library stream)",
                        "pass2_ms_per_step": ms_instrumented / args.steps,
                        "by_phase": {ph: {"launches": v["launches"],
                                          "achieved": (v["flops"] / (v["ms"] / 1e3) / 1e12
                                                       if v["ms"] > 0 else None),
                                          "frac": (v["flops"] / (v["ms"] / 1e3) / 1e12 / peak
                                                   if v["ms"] > 0 else None),
                                          "frac_burst": (v["flops"] / (v["ms"] / 1e3) / 1e12
                                                         / peaks["bf16_tflops"]
                                                         if v["ms"] > 0 else None)}
                                     for ph, v in by_phase.items()}},
           "step_tflops": algo_flops / (ms_step / 1e3) / 1e12,
           "step_frac_of_peak": algo_flops / (ms_step / 1e3) / 1e12 / peak,
           "e2e": {"value": ws * NC / e2e_s, "unit": "candidates/s",
                   "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h)},
           "gpu_launches": int(launches),
           "clocks": clk.summary(),
           "kernels": {k: {"launches": v["launches"] // args.steps,
                           "gflop": v["flops"] / args.steps / 1e9}
                       for k, v in launch_stats.items() if v["launches"]},
           "setup_s": setup_s}
    if rank == 0 and ws == 1 and not args.no_cpu_baseline and args.variant == "base":
        pb, nb = oracle_sample(cfg, sched, skip, proxy, args.cpu_budget)
        v = oracle_cands_per_s(pb, cfg, skip, proxy)
        out["cpu_baseline"] = {
            "value": v, "unit": "candidates/s", "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"fp64 numpy oracle, {nb} Wan2.1-1.3B block forward(s) of one candidate "
                      f"({pb:.2f} s each), extrapolated to the step's "
                      f"{N_CAND * computed_blocks(skip, proxy)} draft + "
                      f"{(S_TOTAL - S_DRAFT) * cfg.depth} refine block evaluations"}
    if rank == 0:
        print(json.dumps(out))
    model.set_stream(None)
    model.close()
    if model_r:
        model_r.close()
    if split:
        split.close()
    if pg:
        pg.destroy_process_group()
    return 0


def run_probe(args):
    """A few launches of one kernel on a case sized for an ncu capture (inputs larger
    than L2, a few hundred MB on the device): gemm = the FFN up-projection shape
    (8192 x 1536 -> 8960, GELU epilogue); gemm_resid = FFN down (8192 x 8960 -> 1536,
    gated residual + contribution write); gemm_out = attention output projection
    (8192 x 1536 -> 1536, gated fp32 residual); attn = self-attention over 1560 tokens,
    4 candidates x 12 heads x 128; attn_pool = the same for the draft pool's 32
    candidates."""
    import torch
    from paper_2607_04461_gb300 import flashbon as fb
    torch.cuda.set_device(0)
    cfg = synth.TINY
    m = fb.Model(cfg, synth.make_weights(cfg))
    g = torch.Generator().manual_seed(0)
    rnd = lambda *s, dt=torch.bfloat16: (torch.randn(*s, generator=g) * 0.5).to(dt).cuda()  # noqa
    if args.probe == "pointwise":
        m.close()
        return probe_pointwise(args)
    if args.probe == "mma_rate":
        res = {f"N{n}/issuers{k}": round(fb.fb_probe_mma_rate(k, n), 1)
               for n in (64, 128, 256) for k in (1, 2, 4) if k * n <= 512}
        print(json.dumps({"probe": "mma_rate", "unit": "MAC per SM clock",
                          "nominal": 4096, "res": res}))
        m.close()
        return 0
    if args.probe == "pipes":
        MIX_FORMS = ("ss", "ss_mn", "ts_mn", "attn_step", "attn_step_commits",
                     "attn_step_hoisted", "attn_step_hoisted_commits")
        res = {"mma_gap_mac_per_clk": {str(g): round(fb.fb_probe_mma_gap(g), 1)
                                       for g in (0, 64, 128, 256, 512)},
               "mufu_per_clk": {name: round(fb.fb_probe_mufu(op), 2)
                                for op, name in enumerate(("ex2", "tanh", "rcp", "ex2_f16x2"))},
               "tmem_load_128_columns_clocks": {"tensor_idle": round(fb.fb_probe_tmem_load(False), 1),
                                                "tensor_busy": round(fb.fb_probe_tmem_load(True), 1)},
               "mma_mix_mac_per_clk": {f"{fname}/loaders{ld}/gap{gp}": round(fb.fb_probe_mma_mix(f, ld, gp), 1)
                                       for f, fname in enumerate(MIX_FORMS)
                                       for ld, gp in ((0, 0), (7, 800), (7, 0))},
               "mma_mix_softmax_loaders_mac_per_clk": {
                   f"{fname}/loaders{ld}/gap{gp}": round(fb.fb_probe_mma_mix(7 + f, ld, gp), 1)
                   for f, fname in enumerate(MIX_FORMS)
                   for ld, gp in ((3, 0), (7, 0), (7, 400))}}
        print(json.dumps({"probe": "pipes", "res": res}))
        m.close()
        return 0
    if args.probe in ("gemm_shapes", "gemm_shapes_part", "attn_shapes", "breakdown"):
        call = None
    elif args.probe in ("gemm_refine_out", "gemm_refine_down"):
        # the refine pass's attention output projection / FFN down-projection (one
        # candidate, 1560 rows), once over whole tiles (impl 3) and once with the
        # stream-K split (impl 4) per step
        M, D = 1560, 1536
        K = D if args.probe == "gemm_refine_out" else 8960
        A, W, b = rnd(M, K), rnd(D, K), rnd(D, dt=torch.float32)
        h, gt = rnd(M, D, dt=torch.float32), rnd(D, dt=torch.float32)
        out = torch.empty(M, D, dtype=torch.float32, device="cuda")

        def call():
            for impl in (3, 4):
                fb.fb_op_gemm(m.handle, M, D, K, A, W, b, 2, out, h, gt, None, None, impl)
    elif args.probe == "gemm_out":
        M, D = 8192, 1536
        A, W, b = rnd(M, D), rnd(D, D), rnd(D, dt=torch.float32)
        h, gt = rnd(M, D, dt=torch.float32), rnd(D, dt=torch.float32)
        out = torch.empty(M, D, dtype=torch.float32, device="cuda")
        call = lambda: fb.fb_op_gemm(m.handle, M, D, D, A, W, b, 2, out, h, gt)  # noqa
    elif args.probe in ("gemm", "gemm_resid"):
        M, D, F = 8192, 1536, 8960
        if args.probe == "gemm":
            A, W, out = rnd(M, D), rnd(F, D), torch.empty(M, F, dtype=torch.bfloat16, device="cuda")
            b = rnd(F, dt=torch.float32)
            call = lambda: fb.fb_op_gemm(m.handle, M, F, D, A, W, b, 1, out)  # noqa
        else:
            A, W, b = rnd(M, F), rnd(D, F), rnd(D, dt=torch.float32)
            h, hb, gt = rnd(M, D, dt=torch.float32), rnd(M, D, dt=torch.float32), rnd(D, dt=torch.float32)
            dl = torch.empty(M, D, dtype=torch.bfloat16, device="cuda")
            call = lambda: fb.fb_op_gemm(m.handle, M, D, F, A, W, b, 3, h, hb, gt, h, dl)  # noqa
    elif args.probe == "attn_pool_cross":
        # the draft pool's cross-attention: 32 candidates x 1560 queries, 512 text keys
        n, P, H, dh, T = 32, 1560, 12, 128, 512
        q, kv = rnd(n * P, H * dh), rnd(T, 2 * H * dh)
        o = torch.empty(n * P, H * dh, dtype=torch.bfloat16, device="cuda")
        D = H * dh
        call = lambda: fb.fb_op_attention(m.handle, q, D, kv.data_ptr(), 2 * D,  # noqa
                                          kv.data_ptr() + 2 * D, 2 * D, o, D, n, P, T, 0, H, dh, 0)
    else:
        n, P, H, dh = (32 if args.probe == "attn_pool" else 4), 1560, 12, 128
        qkv, o = rnd(n * P, 3 * H * dh), torch.empty(n * P, H * dh, dtype=torch.bfloat16, device="cuda")
        base, D = qkv.data_ptr(), H * dh
        call = lambda: fb.fb_op_attention(m.handle, base, 3 * D, base + 2 * D, 3 * D,  # noqa
                                          base + 4 * D, 3 * D, o, D, n, P, P, P, H, dh,
                                          1 if args.probe == "attn_mma" else
                                          (0 if args.probe == "attn_pool" else 3))
    if args.probe in ("gemm_shapes", "gemm_shapes_part"):
        return probe_gemm_shapes(m, rnd, args, part=args.probe == "gemm_shapes_part")
    if args.probe == "attn_shapes":
        return probe_attn_shapes(m, rnd, args)
    if args.probe == "breakdown":
        m.close()
        return probe_breakdown(args)
    m.reset_stats()
    for _ in range(args.steps):
        call()
    torch.cuda.synchronize()
    st = {k: v for k, v in m.stats().items() if v["launches"]}
    print(json.dumps({"probe": args.probe, "launches": args.steps, "stats": st}))
    m.close()
    return 0


def probe_gemm_shapes(m, rnd, args, part=False):
    """Per-launch time of each block GEMM shape at the draft (N=32) and refine (N=1) row
    counts: `reps` back-to-back launches inside one call, timed with CUDA events on the
    library's stream (fb_get_stats), for the automatic choice and each forced variant.
    part: the refine's row count only, on an SM partition of --refine-sms SMs (the split
    schedule's refine side)."""
    import torch
    from paper_2607_04461_gb300 import flashbon as fb
    D, F = 1536, 8960
    shapes = {"qkv": (3 * D, D, 0), "out": (D, D, 2), "cross_q": (D, D, 0),
              "cross_out": (D, D, 2), "ffn_up": (F, D, 1), "ffn_down": (D, F, 3)}
    res = {}
    reps = max(5, args.steps)
    split = None
    if part:
        split = fb.SmSplit(args.refine_sms)
        m.set_stream(split.streams[0])
        m.set_sm_budget(split.sms[0])
        res["partition_sms"] = split.sms[0]
    for M in ((1560,) if part else (49920, 1560)):
        for name, (N, K, epi) in shapes.items():
            A, W, b = rnd(M, K), rnd(N, K), rnd(N, dt=torch.float32)
            out = torch.empty(M, N, dtype=torch.bfloat16 if epi < 2 else torch.float32, device="cuda")
            r = rnd(M, N, dt=torch.float32) if epi >= 2 else None
            dl = torch.empty(M, N, dtype=torch.bfloat16, device="cuda") if epi == 3 else None
            for impl, tag in ((0, "auto"), (2, "1sm"), (3, "2sm_tiles"), (4, "2sm_streamk")):
                f = lambda: fb.fb_op_gemm(m.handle, M, N, K, A, W, b, epi, out, r, b if epi >= 2 else None,  # noqa
                                          r if epi == 3 else None, dl, impl)
                try:
                    f()
                except fb.FlashBonError:
                    continue   # stream-K needs enough K blocks per SM pair
                fb.fb_set_op_repeat(m.handle, reps)
                m.reset_stats()
                m.set_timing(1 << fb.K["gemm_tc"])
                f()
                m.set_timing(0)
                st = m.stats()["gemm_tc"]
                us = st["ms"] * 1e3 / st["launches"]
                # back to back without per-launch events (chained as in the model)
                fb.fb_set_op_repeat(m.handle, 10 * reps)
                t0 = time.perf_counter()
                f()
                chain_us = (time.perf_counter() - t0) * 1e6 / (10 * reps)
                fb.fb_set_op_repeat(m.handle, 1)
                res[f"M{M}/{name}/{tag}"] = {
                    "us": round(us, 2), "tflops": round(2 * M * N * K / us / 1e6, 1),
                    "chained_us": round(chain_us, 2)}
            del A, W, out, r, dl
    if split:
        torch.cuda.synchronize()
        m.set_sm_budget(0)
        m.set_stream(None)
        split.close()
    print(json.dumps({"probe": "gemm_shapes", "res": res}))
    return 0


def probe_attn_shapes(m, rnd, args):
    """Per-launch and back-to-back time of the block's attention shapes at the draft
    (N=32) and refine (N=1) batch sizes for the tcgen05 kernel with 128- and 256-query
    CTAs."""
    import torch
    from paper_2607_04461_gb300 import flashbon as fb
    H, dh, P, T = 12, 128, 1560, 512
    D = H * dh
    res = {}
    reps = max(5, args.steps)
    for n in (32, 1):
        qkv = rnd(n * P, 3 * D)
        kv = rnd(T, 2 * D)
        o = torch.empty(n * P, D, dtype=torch.bfloat16, device="cuda")
        base = qkv.data_ptr()
        cases = {
            "self": lambda impl: fb.fb_op_attention(m.handle, base, 3 * D, base + 2 * D, 3 * D,
                                                    base + 4 * D, 3 * D, o, D, n, P, P, P, H,
                                                    dh, impl),
            "cross": lambda impl: fb.fb_op_attention(m.handle, base, 3 * D, kv.data_ptr(),
                                                     2 * D, kv.data_ptr() + 2 * D, 2 * D, o, D,
                                                     n, P, T, 0, H, dh, impl)}
        for name, f in cases.items():
            flops = 4.0 * n * H * P * (P if name == "self" else T) * dh
            for impl, tag in ((0, "auto"), (2, "q128"), (3, "q256")):
                f(impl)
                fb.fb_set_op_repeat(m.handle, reps)
                m.reset_stats()
                m.set_timing(1 << fb.K["attn_self"])
                f(impl)
                m.set_timing(0)
                st = m.stats()["attn_self"]
                us = st["ms"] * 1e3 / st["launches"]
                fb.fb_set_op_repeat(m.handle, 10 * reps)
                t0 = time.perf_counter()
                f(impl)
                chain_us = (time.perf_counter() - t0) * 1e6 / (10 * reps)
                fb.fb_set_op_repeat(m.handle, 1)
                res[f"N{n}/{name}/{tag}"] = {"us": round(us, 2), "chained_us": round(chain_us, 2),
                                             "tflops": round(flops / chain_us / 1e6, 1)}
        del qkv, kv, o
    print(json.dumps({"probe": "attn_shapes", "res": res}))
    return 0


def probe_breakdown(args):
    """One bench step (draft + refine) with CUDA-event timing of every kernel class."""
    import torch
    from paper_2607_04461_gb300 import flashbon as fb
    cfg, sched, skip, proxy = workload()
    model = fb.Model(cfg, synth.make_weights(cfg))
    z0 = torch.from_numpy(synth.make_latents(cfg, N_CAND)).cuda()
    ctx = torch.from_numpy(synth.make_text(cfg)).cuda()
    out = {}
    for phase in ("draft", "refine"):
        z = z0.clone()
        for it in range(2):
            model.reset_stats()
            model.set_timing((1 << len(fb.KERNEL_KINDS)) - 1 if it else 0)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            e0.record()
            if phase == "draft":
                z.copy_(z0)
                model.draft(z, ctx, sched[: S_DRAFT + 1], skip, proxy)
            else:
                zr = z0[0].clone()
                model.refine(zr, ctx, sched[S_DRAFT:])
            e1.record()
            torch.cuda.synchronize()
            if it:
                st = model.stats()
                out[phase] = {"wall_ms": e0.elapsed_time(e1),
                              "kernels": {k: {"ms": round(v["ms"], 2), "launches": v["launches"],
                                              "tflops": round(v["flops"] / v["ms"] / 1e9, 1) if v["ms"] else None,
                                              "gbs": round(v["bytes"] / v["ms"] / 1e6, 1) if v["ms"] else None}
                                          for k, v in st.items() if v["launches"]}}
            else:
                out[phase + "_untimed_ms"] = e0.elapsed_time(e1)
    print(json.dumps({"probe": "breakdown", **out}))
    model.close()
    return 0


def probe_pointwise(args):
    """The HBM-bound kernels on a case sized for an ncu capture: a 16-candidate
    Wan2.1-1.3B draft (24960 rows, the fp32 residual stream 153 MB, above L2) over the
    first two steps of the bench plan (step 1 proxies), `steps` times."""
    import torch
    from paper_2607_04461_gb300 import flashbon as fb
    torch.cuda.set_device(0)
    n = 16
    cfg, sched, skip, proxy = workload()
    cfg = cfg.with_(max_n=n)
    model = fb.Model(cfg, synth.make_weights(cfg))
    z0 = torch.from_numpy(synth.make_latents(cfg, n)).cuda()
    ctx = torch.from_numpy(synth.make_text(cfg)).cuda()
    z = torch.empty_like(z0)
    model.reset_stats()
    model.set_timing((1 << len(fb.KERNEL_KINDS)) - 1)
    for _ in range(args.steps):
        z.copy_(z0)
        model.draft(z, ctx, sched[:3], skip[:2], proxy[:2])
    torch.cuda.synchronize()
    st = {k: {"launches": v["launches"], "ms": round(v["ms"], 3),
              "gbs": round(v["bytes"] / v["ms"] / 1e6, 1) if v["ms"] else None,
              "bytes_per_launch": v["bytes"] / v["launches"]}
          for k, v in model.stats().items() if v["launches"]}
    print(json.dumps({"probe": "pointwise", "candidates": n, "stats": st}))
    model.close()
    return 0


SWEEP_N = (1, 4, 16, 64)
SWEEP_SKIP = (0.0, 0.25, 0.5)
SWEEP_PROXY = (0.0, 0.5)


def run_sweep(args):
    """The 4096-token throughput sweep: Wan2.1-1.3B dims at 1024x1024 (16 x 128 x 128 latent,
    4096 tokens), 10 draft steps of the 50-step schedule, N in SWEEP_N, a seeded fraction
    of the blocks skipped per step (SWEEP_SKIP) and, on odd steps, a fraction of the
    remaining blocks proxied from the previous step (SWEEP_PROXY). One JSON line per point:
    candidates/s from `steps` timed drafts (CUDA events, inputs resident), then one draft
    with per-launch events for the GEMM and attention rates."""
    import torch
    from paper_2607_04461_gb300 import flashbon as fb
    torch.cuda.set_device(0)
    peaks, peak_kind = read_peaks()
    cfg = synth.WAN13_1K.with_(max_n=max(SWEEP_N))
    model = fb.Model(cfg, synth.make_weights(cfg))
    ctx = torch.from_numpy(synth.make_text(cfg)).cuda()
    sched = synth.make_schedule(S_TOTAL)[: S_DRAFT + 1]
    stream = torch.cuda.Stream()
    model.set_stream(stream)
    kinds = (1 << fb.K["gemm_tc"]) | (1 << fb.K["attn_self"]) | (1 << fb.K["attn_cross"])
    for n in SWEEP_N:
        z0 = torch.from_numpy(synth.make_latents(cfg, n)).cuda()
        z = torch.empty_like(z0)
        for sf in SWEEP_SKIP:
            for pf in SWEEP_PROXY:
                skip, proxy = synth.random_plan(S_DRAFT, cfg.depth, sf, pf, seed=PLAN_SEED)

                def draft():
                    with torch.cuda.stream(stream):
                        z.copy_(z0)
                    model.draft(z, ctx, sched, skip, proxy)
                for _ in range(args.warmup):
                    draft()
                torch.cuda.synchronize()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                with ClockSampler(0) as clk:
                    e0.record(stream)
                    for _ in range(args.steps):
                        draft()
                    e1.record(stream)
                    torch.cuda.synchronize()
                ms = e0.elapsed_time(e1) / args.steps
                model.reset_stats()
                model.set_timing(kinds)
                draft()
                model.set_timing(0)
                st = model.stats()
                flops = n * computed_blocks(skip, proxy) * block_flops(cfg)

                def rate(*ks):
                    f = sum(st[k]["flops"] for k in ks)
                    t = sum(st[k]["ms"] for k in ks)
                    return (f / (t / 1e3) / 1e12, t) if t else (None, 0.0)
                g, g_ms = rate("gemm_tc")
                a, a_ms = rate("attn_self", "attn_cross")
                print(json.dumps({
                    "variant": "sweep", "metric": "draft candidates/sec", "unit": "candidates/s",
                    "value": n / (ms / 1e3), "ms_per_draft": ms, "n_candidates": n,
                    "skip_frac": sf, "proxy_frac": pf, "tokens": cfg.tokens,
                    "draft_steps": S_DRAFT, "computed_blocks": computed_blocks(skip, proxy),
                    "algorithmic_tflop": flops / 1e12,
                    "step_tflops": flops / (ms / 1e3) / 1e12,
                    "gemm": {"tflops": g, "ms": g_ms,
                             "frac_burst": g / peaks["bf16_tflops"] if g else None},
                    "attention": {"tflops": a, "ms": a_ms,
                                  "frac_burst": a / peaks["bf16_tflops"] if a else None},
                    "peak_kind": f"bf16 burst, {peak_kind}", "clocks": clk.summary()}),
                    flush=True)
        del z0, z
    model.set_stream(None)
    model.close()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--cpu-budget", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--schedule", choices=["auto", "seq", "split"], default="auto",
                    help="auto: the split schedule (refine on a small SM partition beside "
                         "the next draft) where the variant allows it and the driver offers "
                         "SM partitions, else sequential")
    ap.add_argument("--refine-sms", type=int, default=REFINE_SMS)
    ap.add_argument("--variant", choices=list(VARIANTS), default="base",
                    help="base: the draft-pool workload; cfg / sde: the same with guidance "
                         "or SDE steps")
    ap.add_argument("--probe", choices=["gemm", "gemm_resid", "gemm_out", "gemm_refine_out",
                                        "gemm_refine_down", "attn", "attn_mma", "gemm_shapes", "gemm_shapes_part", "pipes",
                                        "attn_shapes", "breakdown", "pointwise",
                                        "attn_pool", "attn_pool_cross", "mma_rate"],
                    default=None)
    args = ap.parse_args()
    if args.probe:
        return run_probe(args)
    if args.impl == "reference":
        return run_reference(args)
    if args.variant == "sweep":
        return run_sweep(args)
    return run_gb300(args)


if __name__ == "__main__":
    sys.exit(main())
