"""Helpers shared by the GPU parity tests: oracle evaluation of one layer over its
whole output (epilogue included, through the oracle's own add / ReLU / pool) and
the error-bound check.

Bound: |gpu - oracle| <= 1e-5 * S for every output, S = |bias| + sum |w * x|
(+ |skip| when a residual is added; the largest S of the window for a pooled
output; ReLU leaves S unchanged).  An output with S = 0 must be exact.
"""
import numpy as np

from paper_2004_11250_gb300 import synth

REL_TOL = 1e-5


def oracle_layer_full(orc, layer, x, skip=None, relu=False, pool=False):
    """Oracle output and budget S of one layer on input x (original channel order)."""
    if isinstance(layer, synth.DenseLayer):
        y, s = orc.conv_dense(x, layer.w, layer.bias)
    else:
        pat = orc.pattern_ids(layer.w, layer.mask, layer.taps)
        y, s = orc.conv_pruned(x, layer.w, pat, layer.taps, layer.bias)
    return orc.epilogue(y, s, relu_on=relu, skip=skip, pool=pool)


def to_original(a, layout):
    """An activation [N][C][H][W] stored in channel order `layout` (position c holds original channel
    layout[c]) rearranged into the original channel order."""
    if layout is None:
        return a
    out = np.empty_like(a)
    out[:, np.asarray(layout)] = a
    return out


def check_within(gpu, y, s, what=""):
    """Assert the bound element by element; returns the worst |err| / S."""
    gpu = np.asarray(gpu, np.float64)
    err = np.abs(gpu - y)
    assert np.isfinite(gpu).all(), f"{what}: non-finite GPU output"
    zero = s == 0
    assert (err[zero] == 0).all(), f"{what}: outputs with zero budget must be exact"
    bad = err > REL_TOL * s
    if bad.any():
        k = int(np.argmax(bad.ravel()))
        raise AssertionError(f"{what}: {int(bad.sum())} outputs out of bound; e.g. flat index {k}: gpu "
                             f"{gpu.ravel()[k]!r} oracle {y.ravel()[k]!r} budget {s.ravel()[k]!r}")
    nz = ~zero
    return float((err[nz] / s[nz]).max()) if nz.any() else 0.0
