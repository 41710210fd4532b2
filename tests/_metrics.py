"""Error metrics shared by the GPU parity tests.

Tolerances (all compare the CUDA path, bf16 storage / fp32 accumulation, with the fp64
oracle on identical bf16-representable weights and inputs):
  * per-block contribution: max|D_gpu - D_ref| / max|D_ref| <= 2e-2, where
    D = B_l(h) - h (relative error of what the block adds; the block output itself
    would be dominated by the exact input h);
  * final latent: cosine(z_gpu, z_ref) >= 0.999 and the same cosine on the displacement
    z - z_T (the part the model computed), plus a max-error bound on the displacement.
"""
import numpy as np

BLOCK_TOL = 2e-2
COS_MIN = 0.999


def rel_max(got, want):
    got, want = np.asarray(got, np.float64), np.asarray(want, np.float64)
    return float(np.abs(got - want).max() / max(np.abs(want).max(), 1e-30))


def cosine(a, b):
    a, b = np.asarray(a, np.float64).ravel(), np.asarray(b, np.float64).ravel()
    return float(a @ b / (np.linalg.norm(a) * np.linalg.norm(b)))


def check_latents(got, want, z0, disp_tol=5e-2, label=""):
    """Final latents of the CUDA path vs the oracle."""
    got, want, z0 = (np.asarray(x, np.float64) for x in (got, want, z0))
    assert np.isfinite(got).all(), f"{label}: non-finite output"
    c_full = cosine(got, want)
    c_disp = cosine(got - z0, want - z0)
    e_disp = rel_max(got - z0, want - z0)
    msg = f"{label}: cos={c_full:.6f} cos_disp={c_disp:.6f} disp_err={e_disp:.3e}"
    assert c_full >= COS_MIN and c_disp >= COS_MIN and e_disp <= disp_tol, msg
    return c_full, c_disp, e_disp
