"""Comparison helpers shared by the parity tests."""
import numpy as np

# max relative error bound per storage dtype (norm-wise: max|gpu-ref| / max|ref|)
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


def assert_close(name, gpu, ref, tol):
    e = rel_err(gpu, ref)
    assert e <= tol, f"{name}: max rel err {e:.3e} > {tol:.1e}"
    return e


def ints(t):
    return t.detach().cpu().numpy().astype(np.int64)
