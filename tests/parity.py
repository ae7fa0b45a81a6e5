"""Comparison helpers for the GPU parity tests (test infrastructure).

Errors are normwise per tensor, max|x - y| / max|y|, and taken per layer and
separately for the weights W_l and the bias weights b_l of each layer, so that
a small layer's error is not hidden behind a larger layer's entries.

Cancellation factor.  A pooled change G_l = D_l^T A_{l-1} is a sum of
products; the error of any floating-point evaluation of such a sum is bounded
by a multiple of the unit roundoff times the sum of the products' magnitudes,
|D_l|^T |A_{l-1}|, not times |G_l| (the standard forward error bound of a dot
product).  The hidden deltas are themselves such sums, so the magnitudes
propagate through the backward pass:

    |D|_L = |D_L|,   |D|_l = (|D|_{l+1} |W_{l+1}|) * |A_l (1 - A_l)|.

kappa_l = max(|D|_l^T |A_{l-1}|) / max|G_l| is 1 when nothing cancels and
grows when the terms of the sums cancel (deep nets whose first-layer changes
are much smaller than their terms).  The float32 bar of 1e-5 is applied to the
sum's magnitude: the allowed normwise error of layer l is 1e-5 * max(1, kappa_l).
kappa uses the same floor for max|G_l| as normwise() does for the reference's
size, so that for a change that is exactly zero the bar is the absolute bound
1e-5 * max(|D|_l^T |A_{l-1}|).
"""
import numpy as np

from oracle import bp_oracle as O
from paper_1801_01554_gb300 import synth


def normwise(x, y):
    x = np.asarray(x, dtype=np.float64)
    y = np.asarray(y, dtype=np.float64)
    return float(np.max(np.abs(x - y)) / max(np.max(np.abs(y)), 1e-30))


def layer_parts(sizes):
    """[(label, slice)] of the packed parameter vector: W_l and b_l of each layer."""
    offs, _ = synth.param_layout(sizes)
    out = []
    for l, (wo, bo) in enumerate(offs, start=1):
        out.append((f"W{l}", slice(wo, wo + sizes[l] * sizes[l - 1])))
        out.append((f"b{l}", slice(bo, bo + sizes[l])))
    return out


def kappa(sizes, theta, X, T, squash="logistic"):
    """Cancellation factor of each part (W_l, b_l) of the pooled change of one
    group, as a packed-layout-ordered list matching layer_parts()."""
    Ws, bs = O.unpack(sizes, theta)
    As = O.forward(Ws, bs, X, squash)
    Ds = O.deltas(Ws, As, T)
    L = len(Ws)
    mag = [None] * L
    mag[L - 1] = np.abs(Ds[L - 1])
    for l in range(L - 1, 0, -1):
        mag[l - 1] = (mag[l] @ np.abs(Ws[l])) * np.abs(As[l] * (1.0 - As[l]))
    out = []
    for l in range(L):
        G = Ds[l].T @ As[l]
        Gm = mag[l].T @ np.abs(As[l])
        g = Ds[l].sum(axis=0)
        gm = mag[l].sum(axis=0)
        out.append(max(1.0, float(Gm.max() / max(np.abs(G).max(), 1e-30))))
        out.append(max(1.0, float(gm.max() / max(np.abs(g).max(), 1e-30))))
    return out


def layer_errors(sizes, got, ref):
    """{label: normwise error} per part."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    return {lab: normwise(got[sl], ref[sl]) for lab, sl in layer_parts(sizes)}


def assert_layers(sizes, got, ref, tol, scale=None, what=""):
    """Every part within tol (times its scale factor, if given)."""
    errs = layer_errors(sizes, got, ref)
    scale = scale or [1.0] * len(errs)
    bad = {lab: (e, tol * s) for (lab, e), s in zip(errs.items(), scale) if not e <= tol * s}
    assert not bad, f"{what}: parts over the bar (error, bar): {bad}"
    return errs
