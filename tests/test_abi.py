"""The C-ABI library on the host (CPU only): it loads, exports every declared
symbol, and its host packer matches the oracle bit for bit (Section 3 storage
and reorder), including the validation errors of Section 2's invariants."""
import os
import re

import numpy as np
import pytest

from paper_2004_11250_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def pp():
    from paper_2004_11250_gb300 import build
    build.build()
    from paper_2004_11250_gb300 import ppconv
    return ppconv


def declared_symbols():
    src = open(os.path.join(ROOT, "include", "ppconv.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(pp_[a-z0-9_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(pp):
    names = declared_symbols()
    assert len(names) >= 20
    for name in names:
        assert hasattr(pp.lib, name), name


def test_status_strings(pp):
    assert pp.pp_status_string(0) == "PP_OK"
    assert pp.pp_status_string(6) == "PP_ERR_UNSUPPORTED"
    assert pp.pp_status_string(999) == "PP_ERR_UNKNOWN"
    assert pp.pp_version() >= 100


def layers_for_pack():
    rng = np.random.default_rng(0)
    out = [synth.small_random_layer(rng, 16, 16, P=8, keep=0.5),
           synth.small_random_layer(rng, 64, 48, P=4, keep=0.2, ring=False),
           synth.small_random_layer(rng, 33, 7, P=12, keep=0.9, ring=False),
           synth.small_random_layer(rng, 5, 1, P=8, keep=1.0),
           synth.small_random_layer(rng, 40, 40, P=8, keep=0.02),
           synth.cfg0_single().ops[0].layer,
           synth.cfg1_vgg16().ops[3].layer]
    return out


@pytest.mark.parametrize("idx", range(7))
def test_pack_matches_oracle_bit_exact(pp, oracle_mod, idx):
    L = layers_for_pack()[idx]
    ref = oracle_mod.pack(L.w, L.mask, L.taps)
    for ids in (None, L.pattern_ids):
        pk = pp.pp_pack_layer(L.w, L.mask, L.taps, ids)
        try:
            a = pp.pp_packed_arrays(pk)
            assert pp.pp_packed_info(pk) == (L.nk, L.Co, L.Ci, L.taps.shape[0])
            assert (a["perm"] == ref.perm).all()
            assert (a["kptr"] == ref.kptr).all()
            assert (a["kidx"] == ref.kidx).all()
            assert (a["kpat"] == ref.kpat).all()
            assert (a["kw"].view(np.uint32) == ref.kw.view(np.uint32)).all()
            assert (a["taps"] == L.taps).all()
            w, m = pp.pp_unpack_layer(pk)
            assert (m == L.mask).all()
            assert (w.view(np.uint32) == L.w.view(np.uint32)).all()
        finally:
            pp.pp_packed_destroy(pk)


def test_pack_hand_fixture(pp):
    import json
    g = json.load(open(os.path.join(ROOT, "tests", "golden", "hand_packed_layer.json")))
    taps = np.array(g["taps"], np.uint8)
    w = np.zeros((g["Co"], g["Ci"], 9), np.float32)
    mask = np.zeros((g["Co"], g["Ci"]), np.uint8)
    for o, i, p in g["kept"]:
        mask[o, i] = 1
        for t in taps[p]:
            w[o, i, t] = 100 * o + 10 * i + t + 1
    pk = pp.pp_pack_layer(w, mask, taps)
    a = pp.pp_packed_arrays(pk)
    pp.pp_packed_destroy(pk)
    for k in ("perm", "kptr", "kidx", "kpat", "kw"):
        assert a[k].tolist() == g[k], k


def test_validation_errors_match_oracle(pp, oracle_mod):
    rng = np.random.default_rng(3)
    L = synth.small_random_layer(rng, 6, 5, P=8, keep=0.5)
    cases = []
    o, i = np.argwhere(L.mask == 0)[0]
    w = L.w.copy()
    w[o, i, 0] = 0.5
    cases.append((w, L.mask, L.taps, None, pp.PP_ERR_PRUNED_NONZERO))
    o, i = np.argwhere(L.mask == 1)[0]
    w = L.w.copy()
    w[o, i, :] = 1.0
    cases.append((w, L.mask, L.taps, None, pp.PP_ERR_TAP_NOT_IN_PATTERN))
    ids = L.pattern_ids.copy()
    ids[o, i] = (ids[o, i] + 1) % 8
    cases.append((L.w, L.mask, L.taps, ids, pp.PP_ERR_PATTERN_ID_MISMATCH))
    for bad in ([[0, 1, 2, 9]], [[1, 0, 2, 4]], [[0, 1, 2, 4], [0, 1, 2, 4]]):
        cases.append((np.zeros((1, 1, 9), np.float32), np.zeros((1, 1), np.uint8), np.array(bad, np.uint8), None,
                      pp.PP_ERR_BAD_PATTERN_SET))
    for w, m, t, ids, code in cases:
        with pytest.raises(pp.PPError) as e:
            pp.pp_pack_layer(w, m, t, ids)
        assert e.value.code == code
        with pytest.raises(oracle_mod.OracleError) as e2:
            oracle_mod.pack(w, m, t, ids)
        assert e2.value.code == code  # the oracle uses the same numbering


def test_pack_empty_and_invalid(pp):
    taps = synth.ring8_patterns()
    pk = pp.pp_pack_layer(np.zeros((3, 2, 9), np.float32), np.zeros((3, 2), np.uint8), taps)
    a = pp.pp_packed_arrays(pk)
    pp.pp_packed_destroy(pk)
    assert a["perm"].tolist() == [0, 1, 2] and a["kptr"].tolist() == [0, 0, 0, 0] and a["kidx"].size == 0
    with pytest.raises(pp.PPError) as e:
        pp.pp_pack_layer(np.zeros((0, 2, 9), np.float32), np.zeros((0, 2), np.uint8), taps)
    assert e.value.code == pp.PP_ERR_INVALID_ARG
    # null handle arguments are rejected, not dereferenced
    assert pp.lib.pp_packed_info(None, None, None, None, None) == pp.PP_ERR_INVALID_ARG
    assert pp.lib.pp_conv_forward(None, None, None, None, 1, 1, 1, 0, None) == pp.PP_ERR_INVALID_ARG
    assert pp.lib.pp_net_run(None, None, None, None) == pp.PP_ERR_INVALID_ARG
    pp.pp_packed_destroy(None)
    pp.pp_layer_destroy(None)
    pp.pp_net_destroy(None)


def test_net_shape_validation_host_only(pp):
    """Network construction checks that need no device: bad shapes and flags."""
    with pytest.raises(pp.PPError):
        pp.pp_net_create(0, 1, 1, 1)
    net = pp.pp_net_create(1, 3, 8, 8)
    assert pp.pp_net_output_shape(net) == (1, 3, 8, 8)
    with pytest.raises(pp.PPError):
        pp.pp_net_finalize(net)  # no ops
    pp.pp_net_destroy(net)


def test_fold_batchnorm_against_definition(pp, oracle_mod):
    """pp_fold_batchnorm: conv with the folded weights and bias equals, in fp64, batch normalisation
    (gamma (z - mean) / sqrt(var + eps) + beta per output channel) applied to the original conv z,
    within the fp32 rounding of the folded values; zeros stay zero so the pruned layer packs the same."""
    rng = np.random.default_rng(23)
    Co, Ci = 12, 7
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.6, ring=False)
    gamma = rng.uniform(-2, 2, Co).astype(np.float32)
    beta = rng.standard_normal(Co).astype(np.float32)
    mean = rng.standard_normal(Co).astype(np.float32)
    var = rng.uniform(0.05, 3, Co).astype(np.float32)
    eps = 1e-3
    w2, b2 = pp.pp_fold_batchnorm(L.w, L.bias, gamma, beta, mean, var, eps)
    assert ((w2.reshape(Co, Ci, 9) != 0) == (L.w.reshape(Co, Ci, 9) != 0)).all()
    pat = oracle_mod.pattern_ids(L.w, L.mask, L.taps)
    assert (oracle_mod.pattern_ids(w2, L.mask, L.taps) == pat).all()
    x = rng.uniform(-1, 1, (2, Ci, 9, 11)).astype(np.float32)
    z, _ = oracle_mod.conv_pruned(x, L.w, pat, L.taps, L.bias)
    g = gamma.astype(np.float64) / np.sqrt(var.astype(np.float64) + eps)
    want = (z - mean[None, :, None, None]) * g[None, :, None, None] + beta[None, :, None, None]
    got, s2 = oracle_mod.conv_pruned(x, w2, pat, L.taps, b2)
    # each folded weight and the bias carry one fp32 rounding (2^-24 relative)
    assert (np.abs(got - want) <= 2.0 ** -23 * s2 + 1e-12).all()
    # a wrong per-filter index or sign would be far outside that
    assert np.abs(got - want).max() < 1e-5
    with pytest.raises(pp.PPError):
        pp.pp_fold_batchnorm(L.w, L.bias, gamma, beta, mean, -np.ones(Co, np.float32), 0.0)


def test_wait_probe_rejects_bad_arguments(pp):
    """Argument checks come before any device work (this runs without a GPU)."""
    for polls in (0, -1, (1 << 20) + 1):
        with pytest.raises(pp.PPError) as e:
            pp.pp_wait_probe(polls)
        assert e.value.code == pp.PP_ERR_INVALID_ARG


def test_peak_probe_rejects_bad_arguments(pp):
    """Argument checks come before any device work (this runs without a GPU)."""
    for kind, iters in ((pp.PP_PROBE_FFMA, 0), (pp.PP_PROBE_MMA_TF32, (1 << 24) + 1), (7, 100), (-1, 100)):
        with pytest.raises(pp.PPError) as e:
            pp.pp_peak_probe(kind, iters)
        assert e.value.code == pp.PP_ERR_INVALID_ARG


@pytest.mark.parametrize("idx", [0, 1, 2, 6])
def test_permuted_input_channels_pack_matches_oracle(pp, oracle_mod, idx):
    """Folding the filter reorder of one layer into the next (Section 3 "Matrix reorder"): the next
    layer's input channels are permuted on the host before packing.  pp_permute_input_channels equals
    numpy fancy indexing bit for bit, and the packed metadata of the permuted layer equals the oracle's
    packing of the numpy-permuted layer bit for bit."""
    L = layers_for_pack()[idx]
    rng = np.random.default_rng(100 + idx)
    layout = rng.permutation(L.Ci).astype(np.int32)
    w2, m2, i2 = pp.pp_permute_input_channels(L.w, L.mask, layout, L.pattern_ids)
    wn = L.w.reshape(L.Co, L.Ci, 9)[:, layout]
    assert (w2.view(np.uint32) == wn.view(np.uint32)).all()
    assert (m2 == L.mask[:, layout]).all() and (i2 == L.pattern_ids[:, layout]).all()
    ref = oracle_mod.pack(wn, L.mask[:, layout], L.taps)
    pk = pp.pp_pack_layer(w2, m2, L.taps)
    try:
        a = pp.pp_packed_arrays(pk)
        for k in ("perm", "kptr", "kidx", "kpat"):
            assert (a[k] == getattr(ref, k)).all(), k
        assert (a["kw"].view(np.uint32) == ref.kw.view(np.uint32)).all()
    finally:
        pp.pp_packed_destroy(pk)
    # the identity layout is a no-op; a repeated channel is not a permutation
    w3, _, _ = pp.pp_permute_input_channels(L.w, L.mask, np.arange(L.Ci, dtype=np.int32))
    assert (w3.view(np.uint32) == L.w.reshape(L.Co, L.Ci, 9).view(np.uint32)).all()
    if L.Ci > 1:
        bad = layout.copy()
        bad[0] = bad[1]
        with pytest.raises(pp.PPError) as e:
            pp.pp_permute_input_channels(L.w, L.mask, bad)
        assert e.value.code == pp.PP_ERR_INVALID_ARG


def test_fold_groups_of_the_workloads():
    """Host logic of the permutation folding: which activations keep the original channel order."""
    from paper_2004_11250_gb300 import runner
    g = runner.fold_groups(synth.cfg1_vgg16())
    assert g[0] and g[-1] and not any(g[1:-1])
    net = synth.cfg2_style()
    g = runner.fold_groups(net)
    # block inputs and outputs are tied to the network input through the skips; conv1 outputs are free
    assert g == [True] + [op.skip_from >= 0 for op in net.ops]
    net = synth.cfg3_vdsr(H=8, W=8)
    g = runner.fold_groups(net)
    # dense end layers and the global skip keep the original order, the 18 pruned layers' outputs are free
    assert g[0] and g[1] and g[-1] and g[-2] is False and not any(g[2:-2])
