"""Comparison helpers shared by the parity tests.

Every floating-point comparison applies two bounds with the same rtol (the stated
tolerance of the storage dtype):
  norm-wise:    max|gpu - ref| / max|ref| <= rtol
  elementwise:  |gpu - ref| <= atol + rtol |ref| for every element, atol = rtol RMS(ref)
The norm-wise bound reads "max relative error" per tensor; the elementwise one also
catches an error confined to the small-magnitude rows or columns of a tensor, which
the norm-wise bound would let through. A stack of independent tensors (one weight
gradient per expert, one router gradient per party) is compared slice by slice
(assert_close_slices): each slice's own scale sets its bounds, so neither a small
expert's error hides under a large expert's max nor a large expert's rounding is
held to a small expert's RMS.
"""
import numpy as np

# max relative error bound per storage dtype
TOL = {"f32": 1e-4, "bf16": 2e-2}


def np64(t):
    if hasattr(t, "detach"):
        t = t.detach()
        if t.dtype.is_floating_point:
            t = t.float()
        t = t.cpu().numpy()
    return np.asarray(t, dtype=np.float64)


def rel_err(gpu, ref) -> float:
    g, r = np64(gpu), np.asarray(ref, np.float64)
    assert g.shape == r.shape, (g.shape, r.shape)
    den = np.abs(r).max() if r.size else 0.0
    if den == 0.0:
        return float(np.abs(g).max()) if g.size else 0.0
    return float(np.abs(g - r).max() / den)


def elem_ratio(gpu, ref, rtol) -> float:
    """max over elements of |g - r| / (atol + rtol |r|) with atol = rtol RMS(r); the
    elementwise bound holds when this is <= 1 (0 for identical tensors)."""
    g, r = np64(gpu), np.asarray(ref, np.float64)
    assert g.shape == r.shape, (g.shape, r.shape)
    if not r.size:
        return 0.0
    diff = np.abs(g - r)
    bound = rtol * np.sqrt(np.mean(r * r)) + rtol * np.abs(r)
    with np.errstate(divide="ignore", invalid="ignore"):
        q = np.where(diff == 0.0, 0.0, diff / bound)
    return float(np.max(q))


class Err(float):
    """The norm-wise relative error, carrying the elementwise ratio as ``.elem``."""

    def __new__(cls, norm, elem):
        obj = super().__new__(cls, norm)
        obj.elem = elem
        return obj

    def __format__(self, spec):
        return f"{float(self):{spec}}/{self.elem:.2f}" if spec else f"{float(self)}/{self.elem:.2f}"


def assert_close(name, gpu, ref, tol):
    e = rel_err(gpu, ref)
    assert e <= tol, f"{name}: max rel err {e:.3e} > {tol:.1e}"
    q = elem_ratio(gpu, ref, tol)
    assert q <= 1.0, (f"{name}: elementwise |gpu-ref| exceeds {tol:.1e} (RMS(ref) + |ref|) "
                      f"by a factor {q:.2f}")
    return Err(e, q)


def assert_close_slices(name, gpu, ref, tol):
    """assert_close on every slice along the first axis; returns the worst slice's Err.
    A slice whose reference is all zero (an expert no token picked) must be exactly
    zero."""
    ref = np.asarray(ref, np.float64)
    worst = Err(0.0, 0.0)
    for i in range(ref.shape[0]):
        e = assert_close(f"{name}[{i}]", gpu[i], ref[i], tol)
        worst = Err(max(float(e), float(worst)), max(e.elem, worst.elem))
    return worst


def ints(t):
    return t.detach().cpu().numpy().astype(np.int64)
