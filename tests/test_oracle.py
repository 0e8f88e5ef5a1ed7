"""Pins of the fp64 oracle against things other than itself (CPU only).

Each test fixes the oracle to an independent fact: a value worked by hand from
the definition (tests/golden), a library routine the method reduces to
(torch conv2d in float64 for the dense-with-mask special case, numpy lexsort
and bincount for the reorder keys), a closed form (shifts, constants,
all-pruned layers), or an invariant of the paper's definitions (Section 2:
4 taps per kept kernel from the pattern set, pruned kernels all zero; Section
3: compact storage is lossless).
"""
import json
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from paper_2004_11250_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def torch_conv(x, w, bias):
    """Library convolution in float64 (a dense 3x3 conv with zeros = the pruned layer)."""
    Co, Ci = w.shape[:2]
    xt = torch.from_numpy(np.asarray(x, np.float64))
    wt = torch.from_numpy(np.asarray(w, np.float64).reshape(Co, Ci, 3, 3))
    bt = None if bias is None else torch.from_numpy(np.asarray(bias, np.float64))
    return F.conv2d(xt, wt, bt, padding=1).numpy()


def torch_bound(x, w, bias):
    """|bias| + sum |w * x| computed by the library as conv(|x|, |w|) + |bias|."""
    return torch_conv(np.abs(np.asarray(x, np.float64)), np.abs(np.asarray(w, np.float64)),
                      None if bias is None else np.abs(np.asarray(bias, np.float64)))


# --------------------------------------------------------------------------- pattern sets / invariants


def test_pattern_sets_shape():
    r8 = synth.ring8_patterns()
    assert r8.shape == (8, 4)
    assert all(4 in p for p in r8)
    assert len({tuple(p) for p in r8}) == 8
    allp = synth.all_centre_patterns()
    assert allp.shape == (56, 4) and len({tuple(p) for p in allp}) == 56
    assert all((np.diff(p) > 0).all() and 4 in p for p in allp)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_generated_layer_invariants(oracle_mod, seed):
    rng = np.random.default_rng(seed)
    L = synth.small_random_layer(rng, 12, 10, P=8, keep=0.35)
    assert L.nk == int(np.floor(0.35 * 120 + 0.5))
    nz = (L.w != 0).sum(axis=2)
    assert (nz[L.mask == 1] == 4).all()  # exactly 4 taps kept per kept kernel
    assert (nz[L.mask == 0] == 0).all()  # connectivity-pruned kernels are all zero
    pat = oracle_mod.pattern_ids(L.w, L.mask, L.taps)
    # with 4 nonzero taps the pattern is unique, so inference recovers the drawn id
    assert (pat[L.mask == 1] == L.pattern_ids[L.mask == 1]).all()
    assert (pat[L.mask == 0] == -1).all()
    pat2 = oracle_mod.pattern_ids(L.w, L.mask, L.taps, given=L.pattern_ids)
    assert (pat2 == pat).all()


def test_validation_errors(oracle_mod):
    rng = np.random.default_rng(3)
    L = synth.small_random_layer(rng, 4, 4, P=8, keep=0.5)
    o, i = np.argwhere(L.mask == 0)[0]
    w = L.w.copy()
    w[o, i, 4] = 1.0
    with pytest.raises(oracle_mod.OracleError) as e:
        oracle_mod.pattern_ids(w, L.mask, L.taps)
    assert e.value.code == oracle_mod.OR_PRUNED_NONZERO
    o, i = np.argwhere(L.mask == 1)[0]
    w = L.w.copy()
    w[o, i, :] = 1.0  # 9 nonzero taps fit no pattern
    with pytest.raises(oracle_mod.OracleError) as e:
        oracle_mod.pattern_ids(w, L.mask, L.taps)
    assert e.value.code == oracle_mod.OR_TAP_NOT_IN_PATTERN
    given = L.pattern_ids.copy()
    given[o, i] = (given[o, i] + 1) % 8
    with pytest.raises(oracle_mod.OracleError) as e:
        oracle_mod.pattern_ids(L.w, L.mask, L.taps, given=given)
    assert e.value.code == oracle_mod.OR_PATTERN_ID_MISMATCH
    for bad in ([[0, 1, 2, 9]], [[1, 0, 2, 4]], [[0, 1, 2, 4], [0, 1, 2, 4]], [[0, 0, 1, 4]]):
        with pytest.raises(oracle_mod.OracleError) as e:
            oracle_mod.pattern_ids(np.zeros((1, 1, 9), np.float32), np.zeros((1, 1), np.uint8),
                                   np.array(bad, np.uint8))
        assert e.value.code == oracle_mod.OR_BAD_PATTERN_SET


def test_lowest_pattern_rule(oracle_mod):
    """A kept kernel whose support fits several patterns takes the lowest one."""
    taps = synth.ring8_patterns()
    w = np.zeros((1, 1, 9), np.float32)
    w[0, 0, 4] = 2.0  # centre only: inside every pattern
    assert oracle_mod.pattern_ids(w, np.ones((1, 1), np.uint8), taps)[0, 0] == 0
    w[0, 0, 5] = 1.0  # centre + right: patterns 1, 2, 3 contain {4, 5}
    assert oracle_mod.pattern_ids(w, np.ones((1, 1), np.uint8), taps)[0, 0] == 1


# --------------------------------------------------------------------------- convolution


def test_hand_worked_fixture(oracle_mod):
    g = json.load(open(os.path.join(GOLDEN, "hand_worked_3x3.json")))
    taps = np.array(g["taps"], np.uint8)
    w = np.zeros((1, 1, 9), np.float32)
    w[0, 0, taps[0]] = g["w_on_taps"]
    x = np.array(g["x"], np.float32)[None, None]
    pat = oracle_mod.pattern_ids(w, np.ones((1, 1), np.uint8), taps)
    y, s = oracle_mod.conv_pruned(x, w, pat, taps, np.array([g["bias"]], np.float32))
    assert (y[0, 0] == np.array(g["y"], np.float64)).all()
    assert (s[0, 0] == np.array(g["y"], np.float64)).all()  # all terms positive: budget = value


@pytest.mark.parametrize("N,Ci,Co,H,W", [(1, 1, 1, 1, 1), (2, 3, 4, 5, 7), (1, 4, 2, 2, 3), (2, 8, 6, 7, 5),
                                         (1, 5, 3, 3, 1)])
def test_conv_vs_torch_small(oracle_mod, N, Ci, Co, H, W):
    rng = np.random.default_rng(N * 1000 + Ci * 100 + Co * 10 + H + W)
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.6)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    pat = oracle_mod.pattern_ids(L.w, L.mask, L.taps)
    y, s = oracle_mod.conv_pruned(x, L.w, pat, L.taps, L.bias)
    ref = torch_conv(x, L.w, L.bias)
    np.testing.assert_allclose(y, ref, rtol=0, atol=1e-12)
    np.testing.assert_allclose(s, torch_bound(x, L.w, L.bias), rtol=1e-13, atol=1e-13)


@pytest.mark.parametrize("seed,P,ring", [(0, 8, True), (1, 4, False), (2, 12, False)])
def test_conv_vs_torch_medium(oracle_mod, seed, P, ring):
    rng = np.random.default_rng(seed)
    L = synth.small_random_layer(rng, 24, 20, P=P, keep=0.3, ring=ring)
    x = rng.uniform(-1, 1, (2, 20, 19, 23)).astype(np.float32)
    pat = oracle_mod.pattern_ids(L.w, L.mask, L.taps)
    y, s = oracle_mod.conv_pruned(x, L.w, pat, L.taps, L.bias)
    np.testing.assert_allclose(y, torch_conv(x, L.w, L.bias), rtol=0, atol=1e-11)
    yd, sd = oracle_mod.conv_dense(x, L.w, L.bias)
    np.testing.assert_allclose(yd, y, rtol=0, atol=1e-12)
    np.testing.assert_allclose(sd, s, rtol=1e-13)


def test_dense_vs_torch(oracle_mod):
    rng = np.random.default_rng(7)
    D = synth.make_dense_layer(rng, 5, 3, 0.3, 0.01)
    x = rng.uniform(0, 1, (1, 3, 9, 11)).astype(np.float32)
    y, s = oracle_mod.conv_dense(x, D.w, D.bias)
    np.testing.assert_allclose(y, torch_conv(x, D.w, D.bias), rtol=0, atol=1e-12)
    np.testing.assert_allclose(s, torch_bound(x, D.w, D.bias), rtol=1e-13)


@pytest.mark.parametrize("t", range(9))
def test_single_tap_is_a_shift(oracle_mod, t):
    """Closed form: one kept kernel with weight 1 on tap t and 0 on its other taps shifts the input by
    (t//3 - 1, t%3 - 1) with zero fill, exactly."""
    taps = synth.all_centre_patterns()
    p = next(k for k, pp in enumerate(taps) if t in pp)
    w = np.zeros((1, 1, 9), np.float32)
    w[0, 0, t] = 1.0
    rng = np.random.default_rng(t)
    x = rng.uniform(-1, 1, (1, 1, 6, 7)).astype(np.float32)
    pat = oracle_mod.pattern_ids(w, np.ones((1, 1), np.uint8), taps, given=np.array([[p]], np.uint8))
    y, _ = oracle_mod.conv_pruned(x, w, pat, taps, None)
    dy, dx = t // 3 - 1, t % 3 - 1
    ref = np.zeros((6, 7))
    for r in range(6):
        for c in range(7):
            if 0 <= r + dy < 6 and 0 <= c + dx < 7:
                ref[r, c] = x[0, 0, r + dy, c + dx]
    assert (y[0, 0] == ref).all()


def test_all_pruned_gives_bias(oracle_mod):
    rng = np.random.default_rng(11)
    taps = synth.ring8_patterns()
    w = np.zeros((3, 4, 9), np.float32)
    bias = rng.standard_normal(3).astype(np.float32)
    x = rng.uniform(-1, 1, (2, 4, 5, 5)).astype(np.float32)
    pat = oracle_mod.pattern_ids(w, np.zeros((3, 4), np.uint8), taps)
    y, s = oracle_mod.conv_pruned(x, w, pat, taps, bias)
    assert (y == bias[None, :, None, None].astype(np.float64)).all()
    assert (s == np.abs(bias)[None, :, None, None].astype(np.float64)).all()


def test_constant_input_closed_form(oracle_mod):
    """x = 1 everywhere: an interior output is bias + sum of the filter's kept weights; a corner output
    keeps only the taps that stay inside the map."""
    rng = np.random.default_rng(5)
    L = synth.small_random_layer(rng, 3, 4, P=8, keep=0.5)
    x = np.ones((1, 4, 6, 6), np.float32)
    pat = oracle_mod.pattern_ids(L.w, L.mask, L.taps)
    y, _ = oracle_mod.conv_pruned(x, L.w, pat, L.taps, L.bias)
    wd = L.w.astype(np.float64)
    for o in range(3):
        assert abs(y[0, o, 3, 3] - (L.bias[o] + wd[o].sum())) < 1e-12
        inside = [4, 5, 7, 8]  # top-left corner: taps with ky >= 1 and kx >= 1
        assert abs(y[0, o, 0, 0] - (L.bias[o] + wd[o][:, inside].sum())) < 1e-12


def test_points_match_full(oracle_mod):
    rng = np.random.default_rng(9)
    L = synth.small_random_layer(rng, 6, 5, P=8, keep=0.4)
    x = rng.uniform(-1, 1, (2, 5, 8, 9)).astype(np.float32)
    pat = oracle_mod.pattern_ids(L.w, L.mask, L.taps)
    y, s = oracle_mod.conv_pruned(x, L.w, pat, L.taps, L.bias)
    pts = np.stack([rng.integers(0, d, 50) for d in (2, 6, 8, 9)], axis=1)
    yp, sp = oracle_mod.conv_pruned_points(x, L.w, pat, L.taps, L.bias, pts)
    assert (yp == y[tuple(pts.T)]).all() and (sp == s[tuple(pts.T)]).all()
    yd, sd = oracle_mod.conv_dense_points(x, L.w, L.bias, pts)
    np.testing.assert_allclose(yd, yp, rtol=0, atol=1e-12)


def test_epilogue_ops(oracle_mod):
    rng = np.random.default_rng(4)
    y = rng.standard_normal((2, 3, 6, 8))
    s = np.abs(rng.standard_normal((2, 3, 6, 8)))
    assert (oracle_mod.relu(y) == np.maximum(y, 0)).all()
    skip = rng.standard_normal(y.shape).astype(np.float32)
    ya, sa = oracle_mod.add(y, s, skip)
    assert (ya == y + skip.astype(np.float64)).all() and (sa == s + np.abs(skip.astype(np.float64))).all()
    yp, sp = oracle_mod.pool2(y, s)
    ref = y.reshape(2, 3, 3, 2, 4, 2).max(axis=(3, 5))
    assert (yp == ref).all() and (sp == s.reshape(2, 3, 3, 2, 4, 2).max(axis=(3, 5))).all()
    t = torch.from_numpy(y)
    assert (yp == F.max_pool2d(t, 2).numpy()).all()
    # odd sizes floor
    yo, _ = oracle_mod.pool2(y[:, :, :5, :7], s[:, :, :5, :7])
    assert yo.shape == (2, 3, 2, 3)
    assert (yo == F.max_pool2d(torch.from_numpy(np.ascontiguousarray(y[:, :, :5, :7])), 2).numpy()).all()


def test_flipped_taps_would_be_caught(oracle_mod):
    """Sensitivity of the library pin: an oracle that read the kernel mirrored (a plausible index slip)
    would disagree with torch; emulate the slip by mirroring the weights fed to the same oracle."""
    rng = np.random.default_rng(21)
    L = synth.small_random_layer(rng, 4, 3, P=8, keep=1.0)
    x = rng.uniform(-1, 1, (1, 3, 6, 6)).astype(np.float32)
    wm = np.ascontiguousarray(L.w[:, :, ::-1])
    y, _ = oracle_mod.conv_dense(x, wm, L.bias)
    assert np.abs(y - torch_conv(x, L.w, L.bias)).max() > 1e-3


# --------------------------------------------------------------------------- storage / reorder


def test_hand_packed_fixture(oracle_mod):
    g = json.load(open(os.path.join(GOLDEN, "hand_packed_layer.json")))
    taps = np.array(g["taps"], np.uint8)
    w = np.zeros((g["Co"], g["Ci"], 9), np.float32)
    mask = np.zeros((g["Co"], g["Ci"]), np.uint8)
    for o, i, p in g["kept"]:
        mask[o, i] = 1
        for t in taps[p]:
            w[o, i, t] = 100 * o + 10 * i + t + 1
    pk = oracle_mod.pack(w, mask, taps)
    assert pk.perm.tolist() == g["perm"]
    assert pk.kptr.tolist() == g["kptr"]
    assert pk.kidx.tolist() == g["kidx"]
    assert pk.kpat.tolist() == g["kpat"]
    assert pk.kw.tolist() == g["kw"]


def check_packed_properties(L, pat, pk):
    """Invariants of the reading of Section 3's storage + reorder, checked with numpy."""
    Co, Ci = L.mask.shape
    P = L.taps.shape[0]
    cnt = L.mask.sum(axis=1).astype(np.int64)
    dom = np.array([np.bincount(pat[o][pat[o] >= 0], minlength=P).argmax() if cnt[o] else 0 for o in range(Co)])
    expect_perm = np.lexsort((np.arange(Co), dom, -cnt))  # last key is primary; lexsort is stable
    assert (pk.perm == expect_perm).all()
    assert pk.kptr[0] == 0 and (np.diff(pk.kptr) == cnt[pk.perm]).all()
    assert len(pk.kidx) == L.nk
    w_rec = np.zeros_like(L.w)
    for j in range(Co):
        o = pk.perm[j]
        seg = slice(pk.kptr[j], pk.kptr[j + 1])
        keys = list(zip(pk.kpat[seg].tolist(), pk.kidx[seg].tolist()))
        assert keys == sorted(keys) and len(set(keys)) == len(keys)
        for e in range(pk.kptr[j], pk.kptr[j + 1]):
            i, p = pk.kidx[e], pk.kpat[e]
            assert pat[o, i] == p
            w_rec[o, i, L.taps[p]] = pk.kw[e]
    # lossless: unpacking the compact form gives back W * M bit for bit
    assert (w_rec.view(np.uint32) == (L.w * L.mask[:, :, None]).view(np.uint32)).all()


@pytest.mark.parametrize("seed,Co,Ci,P,keep", [(0, 16, 16, 8, 0.5), (1, 64, 48, 4, 0.2), (2, 33, 7, 12, 0.9),
                                               (3, 5, 1, 8, 1.0), (4, 40, 40, 8, 0.02)])
def test_pack_properties(oracle_mod, seed, Co, Ci, P, keep):
    rng = np.random.default_rng(seed)
    L = synth.small_random_layer(rng, Co, Ci, P=P, keep=keep, ring=(P == 8))
    pat = oracle_mod.pattern_ids(L.w, L.mask, L.taps)
    pk = oracle_mod.pack(L.w, L.mask, L.taps)
    check_packed_properties(L, pat, pk)


def test_pack_empty_layer(oracle_mod):
    taps = synth.ring8_patterns()
    pk = oracle_mod.pack(np.zeros((3, 2, 9), np.float32), np.zeros((3, 2), np.uint8), taps)
    assert pk.perm.tolist() == [0, 1, 2] and pk.kptr.tolist() == [0, 0, 0, 0] and len(pk.kidx) == 0
