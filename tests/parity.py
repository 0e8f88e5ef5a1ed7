"""Helpers shared by the GPU parity tests: oracle evaluation of one layer (whole
output or sampled points, epilogue included) and the error-bound check.

Bound: |gpu - oracle| <= 1e-5 * S for every output, S = |bias| + sum |w * x|
(+ |skip| when a residual is added; the largest S of the window for a pooled
output; ReLU leaves S unchanged).  An output with S = 0 must be exact.
"""
import numpy as np

from paper_2004_11250_gb300 import synth

REL_TOL = 1e-5


def oracle_layer_full(orc, layer, x, skip=None, relu=False, pool=False):
    if isinstance(layer, synth.DenseLayer):
        y, s = orc.conv_dense(x, layer.w, layer.bias)
    else:
        pat = orc.pattern_ids(layer.w, layer.mask, layer.taps)
        y, s = orc.conv_pruned(x, layer.w, pat, layer.taps, layer.bias)
    return orc.epilogue(y, s, relu_on=relu, skip=skip, pool=pool)


def sample_points(rng, N, Co, Ho, Wo, count):
    """Random output points plus every corner and the first/last row and column of a few channels."""
    pts = [np.stack([rng.integers(0, N, count), rng.integers(0, Co, count), rng.integers(0, Ho, count),
                     rng.integers(0, Wo, count)], axis=1)]
    edge = []
    for o in sorted({0, Co - 1, int(rng.integers(0, Co))}):
        n = int(rng.integers(0, N))
        for r in sorted({0, Ho - 1, min(Ho - 1, 15), min(Ho - 1, 16)}):
            for c in sorted({0, Wo - 1, min(Wo - 1, 7), min(Wo - 1, 8), min(Wo - 1, 16)}):
                edge.append((n, o, r, c))
    pts.append(np.array(edge, np.int64))
    return np.concatenate(pts).astype(np.int64)


def oracle_layer_points(orc, layer, x, pts, skip=None, relu=False, pool=False, pat=None):
    """Oracle output (and budget) of one layer at output points pts [k][4] = (n, o, r, c)."""
    pts = np.asarray(pts, np.int64)
    if pool:
        sub = []
        for dy in (0, 1):
            for dx in (0, 1):
                q = pts.copy()
                q[:, 2] = 2 * q[:, 2] + dy
                q[:, 3] = 2 * q[:, 3] + dx
                sub.append(q)
        conv_pts = np.concatenate(sub)
    else:
        conv_pts = pts
    if isinstance(layer, synth.DenseLayer):
        y, s = orc.conv_dense_points(x, layer.w, layer.bias, conv_pts)
    else:
        if pat is None:
            pat = orc.pattern_ids(layer.w, layer.mask, layer.taps)
        y, s = orc.conv_pruned_points(x, layer.w, pat, layer.taps, layer.bias, conv_pts)
    if skip is not None:
        sv = skip[tuple(conv_pts.T)].astype(np.float64)
        y = y + sv
        s = s + np.abs(sv)
    if relu:
        y = np.maximum(y, 0.0)
    if pool:
        k = len(pts)
        y = y.reshape(4, k).max(axis=0)
        s = s.reshape(4, k).max(axis=0)
    return y, s


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
