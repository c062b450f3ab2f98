"""Shared helpers of the parity tests: tolerances and comparisons.

Tolerances (floating point, bf16 storage with fp32 accumulation): a GPU tensor
passes if max|gpu - oracle| <= 2e-2 * RMS(oracle), per tensor.  Where the
quantity is a small update on top of a bf16-rounded output (X_out - X), the
bound adds half a bf16 ulp of |X_out| for the output rounding itself.
"""
import numpy as np

BF16_TOL = 2e-2
F32_TOL = 1e-4


def rms(a):
    a = np.asarray(a, np.float64)
    return float(np.sqrt(np.mean(a * a))) if a.size else 0.0


def max_rel_err(gpu, ref):
    """max |gpu - ref| / RMS(ref)."""
    g = np.asarray(gpu, np.float64)
    r = np.asarray(ref, np.float64)
    den = rms(r)
    return float(np.abs(g - r).max() / den) if den > 0 else float(np.abs(g - r).max())


def assert_close(name, gpu, ref, tol=BF16_TOL):
    e = max_rel_err(gpu, ref)
    assert e <= tol, f"{name}: max|gpu-ref|/rms(ref) = {e:.3e} > {tol:.1e}"
    return e


def bf16_half_ulp(x):
    """Half a unit in the last place of bf16 at |x| (8 significant bits)."""
    ax = np.maximum(np.abs(np.asarray(x, np.float64)), 1e-30)
    return 2.0 ** (np.floor(np.log2(ax)) - 8)


def assert_update_close(name, X, gpu_out, ref_out, tol=BF16_TOL):
    """Compare the injected update X_out - X with allowance for rounding X_out."""
    X = np.asarray(X, np.float64)
    du_g = np.asarray(gpu_out, np.float64) - X
    du_r = np.asarray(ref_out, np.float64) - X
    bound = tol * rms(du_r) + bf16_half_ulp(ref_out)
    bad = np.abs(du_g - du_r) > bound
    assert not bad.any(), (f"{name}: {int(bad.sum())} elements outside tol*rms(update) + "
                           f"half-ulp; worst excess {float((np.abs(du_g - du_r) - bound).max()):.3e}")
