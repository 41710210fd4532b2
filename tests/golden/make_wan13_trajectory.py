"""Writes wan13_pool_cand0.npz: the fp64 oracle's trajectory of candidate 0 of the
Wan2.1-1.3B draft pool, the stored expected values of the full-trajectory parity test.

Only the oracle (oracle/) and the seeded input generators (synth) are called; nothing
here touches the CUDA path. Workload (the draft pool the benchmark times):
  * Wan2.1-1.3B shape, 30 blocks, 1560 tokens, synth.make_weights(seed 0, bf16);
  * z_T of candidate 0 (seed 1000), text context seed 7;
  * schedule t_i = 1 - i/50; the draft runs steps 0..9 under
    synth.random_plan(10, 30, 1/3, 0.5, seed=7) (a third of the blocks skipped per
    step, half of the remaining ones proxied at order 0 on odd steps; §4.1, Eqs. 3-7);
  * the refine (§4.2 Stage 3, phi_full) resumes from the oracle's draft latent over
    steps 10..49.
Stored (float32): z_draft (after the 10 draft steps), z_refine_mid (after 20 of the 40
refine steps) and z_refine (after all 40). Candidates are independent (Eq. 8), so
candidate 0 alone is exact for the pool.

Run from the repository root:  python tests/golden/make_wan13_trajectory.py
(about an hour of fp64 CPU time on 8 cores)."""
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

from oracle import flashbon_oracle as O  # noqa: E402
from paper_2607_04461_gb300 import synth  # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "wan13_pool_cand0.npz")
S_TOTAL, S_DRAFT, PLAN_SEED = 50, 10, 7


def main():
    cfg = synth.WAN13
    t0 = time.time()
    w = synth.make_weights(cfg)
    ref = O.OracleModel(cfg, w)
    del w
    z = synth.make_latents(cfg, 1)
    ctx = synth.make_text(cfg)
    sched = synth.make_schedule(S_TOTAL)
    skip, proxy = synth.random_plan(S_DRAFT, cfg.depth, 1 / 3, 0.5, seed=PLAN_SEED)
    print(f"weights {time.time() - t0:.0f} s", flush=True)
    zd = ref.draft(z, ctx, sched[: S_DRAFT + 1], skip, proxy)[0]
    print(f"draft {time.time() - t0:.0f} s", flush=True)
    mid = S_DRAFT + (S_TOTAL - S_DRAFT) // 2
    zm = ref.refine(zd, ctx, sched[S_DRAFT: mid + 1])
    print(f"refine half {time.time() - t0:.0f} s", flush=True)
    zr = ref.refine(zm, ctx, sched[mid:])          # Markov: resuming equals one run
    print(f"refine {time.time() - t0:.0f} s", flush=True)
    np.savez(OUT, z_draft=zd.astype(np.float32), z_refine_mid=zm.astype(np.float32),
             z_refine=zr.astype(np.float32), skip=skip, proxy=proxy,
             schedule=sched, refine_mid_step=np.int32(mid))
    print("wrote", OUT)


if __name__ == "__main__":
    main()
