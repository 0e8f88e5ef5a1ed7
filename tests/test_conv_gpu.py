"""GPU parity: the CUDA path, called through the C-ABI, against the fp64 oracle.

Every output is compared: small layers, and the five workloads at full size
layer by layer (each layer's oracle runs on the GPU's own input to that layer),
including all 48 sweep points and the multi-tile repeatability shapes.  Bound:
|gpu - oracle| <= 1e-5 * S per output (see tests/parity.py); integer-valued
cases must be bit-exact.
"""
import numpy as np
import pytest
import torch

from paper_2004_11250_gb300 import synth
from parity import check_within, oracle_layer_full, to_original

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pp():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2004_11250_gb300 import build
    build.build()
    from paper_2004_11250_gb300 import ppconv
    return ppconv


@pytest.fixture(scope="module")
def runner(pp):
    from paper_2004_11250_gb300 import runner
    return runner


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def run_layer(pp, runner, layer, x, skip=None, relu=False, pool=False, kernel=None, precision=0):
    L = runner.DeviceLayer(layer, precision=precision)
    try:
        if kernel is not None:
            pp.pp_layer_set_kernel(L.handle, kernel)
        N, _, H, W = x.shape
        Ho, Wo = (H // 2, W // 2) if pool else (H, W)
        y = torch.full((N, layer.Co, Ho, Wo), float("nan"), device="cuda")
        flags = (pp.PP_ADD_SKIP if skip is not None else 0) | (pp.PP_RELU if relu else 0) | (pp.PP_POOL2 if pool else 0)
        L.forward(dev(x), y, None if skip is None else dev(skip), N, H, W, flags, torch.cuda.current_stream())
        torch.cuda.synchronize()
        if not L.dense:
            assert pp.pp_layer_device_status(L.handle) == 0
        return y.cpu().numpy()
    finally:
        L.close()


SMALL = [
    # N, Ci, Co, H, W, P, ring, keep
    (1, 1, 1, 1, 1, 8, True, 1.0),
    (1, 3, 5, 7, 9, 8, True, 0.6),
    (2, 16, 16, 32, 32, 8, True, 0.5),
    (1, 17, 33, 17, 33, 8, True, 0.3),
    (2, 40, 20, 19, 40, 4, False, 0.35),
    (1, 20, 40, 16, 16, 12, False, 0.5),
    (1, 35, 18, 33, 18, 8, True, 1.0),
    (3, 5, 7, 2, 3, 8, False, 0.9),
    (1, 64, 64, 12, 44, 8, True, 0.2),
    (1, 40, 24, 14, 14, 8, True, 0.3),   # maps <= 16 wide: warps split each stage's channels
    (2, 64, 64, 10, 16, 8, True, 0.5),
    (1, 24, 20, 9, 17, 8, True, 0.6),    # 17 wide: the second tile half holds one column
    (1, 3, 70, 6, 4, 8, True, 1.0),
]


@pytest.mark.parametrize("case", SMALL)
@pytest.mark.parametrize("flags", ["none", "relu", "skip_relu", "pool_relu"])
def test_layer_parity_small(pp, runner, oracle_mod, case, flags):
    N, Ci, Co, H, W, P, ring, keep = case
    if flags == "pool_relu" and (H % 2 or W % 2):
        pytest.skip("pool needs even sizes")
    rng = np.random.default_rng(hash((case, flags)) % (2 ** 32))
    L = synth.small_random_layer(rng, Co, Ci, P=P, keep=keep, ring=ring)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32) if flags == "skip_relu" else None
    relu = flags != "none"
    pool = flags == "pool_relu"
    g = run_layer(pp, runner, L, x, skip, relu, pool)
    y, s = oracle_layer_full(oracle_mod, L, x, skip, relu, pool)
    check_within(g, y, s, f"{case} {flags}")


@pytest.mark.parametrize("case", [c for c in SMALL if c[6]])
@pytest.mark.parametrize("flags", ["none", "skip_relu", "pool_relu"])
def test_register_kernel_on_ring_layers(pp, runner, oracle_mod, case, flags):
    """Ring-set layers run the tensor-memory kernel by default; the register kernel must agree too."""
    N, Ci, Co, H, W, P, ring, keep = case
    if flags == "pool_relu" and (H % 2 or W % 2):
        pytest.skip("pool needs even sizes")
    rng = np.random.default_rng(sum(case[:5]) + len(flags))
    L = synth.small_random_layer(rng, Co, Ci, P=P, keep=keep, ring=ring)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32) if flags == "skip_relu" else None
    g = run_layer(pp, runner, L, x, skip, flags != "none", flags == "pool_relu", kernel=pp.PP_KERNEL_REGISTER)
    y, s = oracle_layer_full(oracle_mod, L, x, skip, flags != "none", flags == "pool_relu")
    check_within(g, y, s, f"register kernel {case} {flags}")


@pytest.mark.parametrize("case", SMALL)
@pytest.mark.parametrize("flags", ["none", "skip_relu", "pool_relu"])
def test_tensor_core_kernel(pp, runner, oracle_mod, case, flags):
    """The 3xTF32 implicit-GEMM kernel on every small case (fewer than 8 input channels: one ragged chunk)."""
    N, Ci, Co, H, W, P, ring, keep = case
    if flags == "pool_relu" and (H % 2 or W % 2):
        pytest.skip("pool needs even sizes")
    rng = np.random.default_rng(7 * sum(case[:5]) + len(flags))
    L = synth.small_random_layer(rng, Co, Ci, P=P, keep=keep, ring=ring)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32) if flags == "skip_relu" else None
    g = run_layer(pp, runner, L, x, skip, flags != "none", flags == "pool_relu", kernel=pp.PP_KERNEL_TC)
    y, s = oracle_layer_full(oracle_mod, L, x, skip, flags != "none", flags == "pool_relu")
    check_within(g, y, s, f"tensor-core kernel {case} {flags}")


@pytest.mark.parametrize("shape,flags,kernel", [
    ((1, 3, 64, 224, 224), "relu", "TC"),          # a network's first layer (RGB input), 224 wide
    ((1, 1, 64, 72, 128), "relu", "TC"),           # one input channel
    ((2, 5, 130, 20, 24), "skip_pool_relu", "TC_FLAT"),
    ((1, 7, 200, 14, 14), "relu", "TC_FLAT"),
])
@pytest.mark.parametrize("precision", [0, 1])
def test_tensor_core_few_input_channels(pp, runner, oracle_mod, shape, flags, kernel, precision):
    """Layers with fewer input channels than one chunk (8, or 16 in fp16): the channels past Ci come
    from the input box's zero fill and meet zero weights."""
    N, Ci, Co, H, W = shape
    rng = np.random.default_rng(Ci * 1000 + Co + precision)
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=1.0 if Ci <= 3 else 0.6)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32) if "skip" in flags else None
    pool = "pool" in flags
    g = run_layer(pp, runner, L, x, skip, True, pool, kernel=getattr(pp, "PP_KERNEL_" + kernel),
                  precision=precision)
    y, s = oracle_layer_full(oracle_mod, L, x, skip, True, pool)
    check_within(g, y, s, f"{kernel} precision {precision} {shape} {flags}")


def test_tensor_core_split_and_tiles(pp, runner, oracle_mod):
    """Shapes that exercise every tile width (16/32/64/128 pixels), ragged blocks and persistent CTAs with several tiles."""
    rng = np.random.default_rng(31)
    for (N, Ci, Co, H, W) in ((1, 72, 130, 12, 14), (1, 40, 64, 20, 30), (1, 24, 128, 9, 60), (1, 16, 33, 5, 140),
                              (2, 136, 200, 7, 9)):
        L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.4)
        x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
        g = run_layer(pp, runner, L, x, None, True, False, kernel=pp.PP_KERNEL_TC)
        y, s = oracle_layer_full(oracle_mod, L, x, None, True, False)
        check_within(g, y, s, f"tensor-core kernel {(N, Ci, Co, H, W)}")


@pytest.mark.parametrize("shape", [(1, 40, 130, 7, 100), (2, 16, 200, 4, 144), (1, 24, 64, 6, 160)])
@pytest.mark.parametrize("flags", ["none", "skip_relu", "pool_relu"])
def test_tensor_core_pixel_major(pp, runner, oracle_mod, shape, flags):
    """Maps at least 96 wide: the row-tiled kernel's pixel-major tiles (merged hi/lo weight operand), 64- and
    128-filter blocks, ragged filter blocks and row ends; pooled 128-filter layers take filter-major tiles."""
    N, Ci, Co, H, W = shape
    if flags == "pool_relu" and (H % 2 or W % 2):
        pytest.skip("pool needs even sizes")
    rng = np.random.default_rng(13 * sum(shape) + len(flags))
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.45)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32) if flags == "skip_relu" else None
    g = run_layer(pp, runner, L, x, skip, flags != "none", flags == "pool_relu", kernel=pp.PP_KERNEL_TC)
    y, s = oracle_layer_full(oracle_mod, L, x, skip, flags != "none", flags == "pool_relu")
    check_within(g, y, s, f"pixel-major tensor-core kernel {shape} {flags}")


FLAT_CASES = [
    # N, Ci, Co, H, W: every map width class, ragged filter blocks and channel
    # chunks, tiles that overhang the map, split and persistent launches
    (1, 72, 130, 14, 14),
    (1, 136, 256, 28, 28),
    (2, 20, 200, 18, 30),
    (1, 64, 129, 56, 56),
    (3, 24, 160, 12, 8),
    (1, 16, 130, 22, 112),
    (1, 40, 192, 10, 126),
    (1, 48, 136, 6, 128),
    (4, 32, 256, 20, 20),
    (1, 8, 136, 3, 2),
    (1, 64, 130, 13, 15),
]


PFR_CASES = [
    # N, Ci, Co, H, W: 64-filter layers on maps at most 62 wide run the row-tiled
    # kernel with whole rows flattened into the 128-pixel M side (16/32/64-pixel pitch)
    (1, 64, 64, 56, 56),
    (2, 24, 40, 20, 14),
    (1, 16, 64, 33, 30),
    (3, 40, 33, 9, 5),
    (1, 72, 64, 23, 62),
]


@pytest.mark.parametrize("case", PFR_CASES)
@pytest.mark.parametrize("flags", ["none", "skip_relu"])
def test_tensor_core_flattened_rows(pp, runner, oracle_mod, case, flags):
    """Row-tiled tensor-core kernel, pixel-major with flattened rows, against the oracle."""
    N, Ci, Co, H, W = case
    rng = np.random.default_rng(13 * sum(case) + len(flags))
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.4)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32) if flags == "skip_relu" else None
    g = run_layer(pp, runner, L, x, skip, flags != "none", False, kernel=pp.PP_KERNEL_TC)
    y, s = oracle_layer_full(oracle_mod, L, x, skip, flags != "none", False)
    check_within(g, y, s, f"flattened-row tensor-core kernel {case} {flags}")


@pytest.mark.parametrize("case", FLAT_CASES)
@pytest.mark.parametrize("flags", ["none", "skip_relu", "pool_relu", "skip_pool_relu"])
def test_tensor_core_flat_kernel(pp, runner, oracle_mod, case, flags):
    """The flat tensor-core kernel (whole rows per MMA, cluster split for few tiles) against the oracle."""
    N, Ci, Co, H, W = case
    pool = "pool" in flags
    if pool and (H % 2 or W % 2):
        pytest.skip("pool needs even sizes")
    rng = np.random.default_rng(11 * sum(case) + len(flags))
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.45, ring=sum(case) % 2 == 0)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32) if "skip" in flags else None
    g = run_layer(pp, runner, L, x, skip, flags != "none", pool, kernel=pp.PP_KERNEL_TC_FLAT)
    y, s = oracle_layer_full(oracle_mod, L, x, skip, flags != "none", pool)
    check_within(g, y, s, f"flat tensor-core kernel {case} {flags}")


def test_flat_geometry_pin(pp, runner, oracle_mod):
    """Every flat-kernel geometry the planner accepts for a shape gives results
    within the bound; pins are reported back, rejected pairs raise, R = 0 unpins."""
    N, Ci, Co, H, W = 1, 72, 130, 14, 14
    rng = np.random.default_rng(5)
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.45)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    y, s = oracle_layer_full(oracle_mod, L, x, None, True, True)
    dl = runner.DeviceLayer(L)
    flags = pp.PP_RELU | pp.PP_POOL2
    try:
        pp.pp_layer_set_kernel(dl.handle, pp.PP_KERNEL_TC_FLAT)
        assert pp.pp_layer_flat_geometry(dl.handle, N, H, W, flags) == (0, 0)
        accepted = []
        for R in range(1, 17):
            for S in (1, 2, 4, 8, 16) + tuple(pp.PP_FLAT_PAIRED | s for s in (1, 2, 4, 8)):
                try:
                    pp.pp_layer_pin_flat_geometry(dl.handle, N, H, W, flags, R, S)
                except pp.PPError as e:
                    assert e.code == pp.PP_ERR_UNSUPPORTED
                    continue
                assert pp.pp_layer_flat_geometry(dl.handle, N, H, W, flags) == (R, S)
                out = torch.full((N, Co, H // 2, W // 2), float("nan"), device="cuda")
                dl.forward(dev(x), out, None, N, H, W, flags, torch.cuda.current_stream())
                torch.cuda.synchronize()
                check_within(out.cpu().numpy(), y, s, f"flat geometry R={R} S={S}")
                accepted.append((R, S))
        assert len(accepted) >= 3 and any(S > 1 for _, S in accepted), accepted
        assert any(S & pp.PP_FLAT_PAIRED for _, S in accepted), accepted  # 130 filters: two blocks, a pair
        assert all(R % 2 == 0 for R, _ in accepted)  # pooling needs row pairs
        # another shape's pin is not reported for this one; R = 0 unpins
        assert pp.pp_layer_flat_geometry(dl.handle, N, H + 2, W, flags) == (0, 0)
        pp.pp_layer_pin_flat_geometry(dl.handle, N, H, W, flags, 0, 0)
        assert pp.pp_layer_flat_geometry(dl.handle, N, H, W, flags) == (0, 0)
    finally:
        dl.close()


PAIR_CASES = [
    # N, Ci, Co, H, W, flags: filter blocks in pairs (cta_group::2), every accepted paired geometry
    (1, 136, 256, 28, 28, "relu"),
    (1, 72, 512, 14, 14, "pool_relu"),
    (2, 40, 250, 20, 30, "skip_relu"),   # the second block ragged (122 filters)
    (1, 24, 384, 8, 126, "none"),        # three filter blocks: no pairs
    (1, 64, 256, 56, 56, "skip_pool_relu"),
]


@pytest.mark.parametrize("case", PAIR_CASES)
@pytest.mark.parametrize("precision", [0, 1])
def test_flat_kernel_cta_pairs(pp, runner, oracle_mod, case, precision):
    """The flat kernel with two filter blocks per MMA over a CTA pair (M = 256, each SM staging half of the
    tile's columns), at every paired geometry the planner accepts, against the oracle (every output)."""
    N, Ci, Co, H, W, flags = case
    rng = np.random.default_rng(Co + W + precision)
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.35)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32) if "skip" in flags else None
    relu, pool = "relu" in flags, "pool" in flags
    y, s = oracle_layer_full(oracle_mod, L, x, skip, relu, pool)
    f = (pp.PP_RELU if relu else 0) | (pp.PP_POOL2 if pool else 0) | (pp.PP_ADD_SKIP if skip is not None else 0)
    Ho, Wo = (H // 2, W // 2) if pool else (H, W)
    dl = runner.DeviceLayer(L, precision=precision)
    try:
        pp.pp_layer_set_kernel(dl.handle, pp.PP_KERNEL_TC_FLAT)
        accepted = []
        for R in range(1, 17):
            for S in (1, 2, 4, 8):
                try:
                    pp.pp_layer_pin_flat_geometry(dl.handle, N, H, W, f, R, pp.PP_FLAT_PAIRED | S)
                except pp.PPError as e:
                    assert e.code == pp.PP_ERR_UNSUPPORTED
                    continue
                for rep in range(2):  # twice: the pair's barriers and TMEM are set up afresh each launch
                    out = torch.full((N, Co, Ho, Wo), float("nan"), device="cuda")
                    dl.forward(dev(x), out, None if skip is None else dev(skip), N, H, W, f,
                               torch.cuda.current_stream())
                    torch.cuda.synchronize()
                    assert pp.pp_layer_device_status(dl.handle) == 0
                    check_within(out.cpu().numpy(), y, s, f"{case} precision {precision} pair R={R} S={S} #{rep}")
                accepted.append((R, S))
        if Co == 384:
            assert accepted == []
        else:
            assert accepted, "no paired geometry accepted"
    finally:
        dl.close()


@pytest.mark.parametrize("shape", [(1, 40, 130, 18, 30), (2, 24, 136, 14, 14), (1, 16, 132, 9, 50)])
@pytest.mark.parametrize("precision", [0, 1])
def test_flat_geometry_sweep_unaligned_rows(pp, runner, oracle_mod, shape, precision):
    """Maps whose rows are not 16-byte aligned (W % 4 != 0): the flat kernel stages the tile's rows packed
    through a tensor map over [N][Ci][H * W] when the planes are aligned and the box fits (at most 256
    elements), else with per-thread loads; every geometry the planner accepts, both arithmetics."""
    N, Ci, Co, H, W = shape
    rng = np.random.default_rng(W * 100 + precision)
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.5)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32)
    y, s = oracle_layer_full(oracle_mod, L, x, skip, True, False)
    dl = runner.DeviceLayer(L, precision=precision)
    flags = pp.PP_RELU | pp.PP_ADD_SKIP
    try:
        pp.pp_layer_set_kernel(dl.handle, pp.PP_KERNEL_TC_FLAT)
        accepted = []
        for R in range(1, 17):
            for S in (1, 2, 4, 8) + tuple(pp.PP_FLAT_PAIRED | s for s in (1, 2, 4, 8)):
                try:
                    pp.pp_layer_pin_flat_geometry(dl.handle, N, H, W, flags, R, S)
                except pp.PPError as e:
                    assert e.code == pp.PP_ERR_UNSUPPORTED
                    continue
                out = torch.full((N, Co, H, W), float("nan"), device="cuda")
                dl.forward(dev(x), out, dev(skip), N, H, W, flags, torch.cuda.current_stream())
                torch.cuda.synchronize()
                assert pp.pp_layer_device_status(dl.handle) == 0
                check_within(out.cpu().numpy(), y, s, f"{shape} precision {precision} R={R} S={S}")
                accepted.append((R, S))
        assert len(accepted) >= 2, accepted
    finally:
        dl.close()


@pytest.mark.parametrize("shape", [(1, 136, 130, 28, 28), (6, 40, 200, 14, 14)])
def test_tensor_core_flat_integer_bit_exact(pp, runner, oracle_mod, shape):
    """Integer weights and inputs: tf32 holds them exactly (lo parts are zero) and
    every partial sum, including the split's partial tiles, is an exact fp32
    integer, so the flat kernel equals the oracle bit for bit."""
    N, Ci, Co, H, W = shape
    rng = np.random.default_rng(Co + W)
    L = synth.integer_layer(rng, Co, Ci, synth.ring8_patterns(), 0.5)
    x = rng.integers(-8, 9, (N, Ci, H, W)).astype(np.float32)
    g = run_layer(pp, runner, L, x, None, True, False, kernel=pp.PP_KERNEL_TC_FLAT)
    y, _ = oracle_layer_full(oracle_mod, L, x, None, True, False)
    assert (g.astype(np.float64) == y).all()


@pytest.mark.parametrize("shape,kernel", [((12, 256, 256, 56, 56), "TC"), ((8, 64, 64, 128, 128), "TC"),
                                          ((12, 256, 256, 56, 56), "TC_FLAT"), ((1, 512, 512, 28, 28), "TC_FLAT"),
                                          ((1, 512, 512, 14, 14), "TC_FLAT"), ((2, 128, 128, 112, 112), "TC_FLAT")])
def test_tensor_core_repeatable_multi_tile(pp, runner, oracle_mod, shape, kernel):
    """Several tiles per persistent CTA, so every operand ring and both accumulator
    buffers wrap many times, or (flat kernel, few tiles) channel chunks split over
    clusters.  The kernels' summation order is fixed, so repeated
    runs must agree bit for bit (a pipeline race shows up as a run-to-run
    difference); one run is also checked against the oracle on every output."""
    N, Ci, Co, H, W = shape
    rng = np.random.default_rng(Ci + W)
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=1.0)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    dl = runner.DeviceLayer(L)
    try:
        pp.pp_layer_set_kernel(dl.handle, getattr(pp, "PP_KERNEL_" + kernel))
        xd = dev(x)
        outs = []
        for _ in range(5):
            y = torch.full((N, Co, H, W), float("nan"), device="cuda")
            dl.forward(xd, y, None, N, H, W, 0, torch.cuda.current_stream())
            outs.append(y)
        torch.cuda.synchronize()
        for k in range(1, 5):
            assert torch.equal(outs[0], outs[k]), f"run {k} differs from run 0"
        assert pp.pp_layer_device_status(dl.handle) == 0
        yr, s = oracle_layer_full(oracle_mod, L, x)
        check_within(outs[0].cpu().numpy(), yr, s, f"multi-tile {shape}")
    finally:
        dl.close()


def test_autotune_keeps_parity(pp, runner, oracle_mod):
    rng = np.random.default_rng(44)
    L = synth.small_random_layer(rng, 96, 64, P=8, keep=0.4)
    x = rng.uniform(-1, 1, (1, 64, 24, 40)).astype(np.float32)
    dl = runner.DeviceLayer(L)
    try:
        pp.pp_layer_autotune(dl.handle, 1, 24, 40, pp.PP_RELU, None)
        assert pp.pp_layer_kernel(dl.handle) in (pp.PP_KERNEL_TC, pp.PP_KERNEL_TC_FLAT, pp.PP_KERNEL_TMEM)
        y = torch.empty((1, 96, 24, 40), device="cuda")
        dl.forward(dev(x), y, None, 1, 24, 40, pp.PP_RELU, torch.cuda.current_stream())
        torch.cuda.synchronize()
        yr, s = oracle_layer_full(oracle_mod, L, x, None, True, False)
        check_within(y.cpu().numpy(), yr, s, "autotuned layer")
        assert pp.pp_layer_device_status(dl.handle) == 0
    finally:
        dl.close()


def test_kernel_selection(pp, runner):
    rng = np.random.default_rng(2)
    ring = runner.DeviceLayer(synth.small_random_layer(rng, 8, 8, ring=True))
    other = runner.DeviceLayer(synth.small_random_layer(rng, 8, 8, P=8, ring=False))
    try:
        assert pp.pp_layer_kernel(ring.handle) == pp.PP_KERNEL_TMEM
        assert pp.pp_layer_kernel(other.handle) == pp.PP_KERNEL_REGISTER
        with pytest.raises(pp.PPError) as e:
            pp.pp_layer_set_kernel(other.handle, pp.PP_KERNEL_TMEM)
        assert e.value.code == pp.PP_ERR_UNSUPPORTED
        pp.pp_layer_set_kernel(ring.handle, pp.PP_KERNEL_REGISTER)
        assert pp.pp_layer_kernel(ring.handle) == pp.PP_KERNEL_REGISTER
        pp.pp_layer_set_kernel(ring.handle, pp.PP_KERNEL_AUTO)
        assert pp.pp_layer_kernel(ring.handle) == pp.PP_KERNEL_TMEM
        pp.pp_layer_set_kernel(ring.handle, pp.PP_KERNEL_TC)
        assert pp.pp_layer_kernel(ring.handle) == pp.PP_KERNEL_TC
        assert pp.pp_layer_device_status(ring.handle) == 0
    finally:
        ring.close()
        other.close()


@pytest.mark.parametrize("ring", [True, False])
def test_integer_layer_bit_exact(pp, runner, oracle_mod, ring):
    """Small-integer weights and inputs: every partial sum is exact in fp32, so GPU == oracle bit for bit."""
    rng = np.random.default_rng(5 if ring else 6)
    taps = synth.ring8_patterns() if ring else synth.seeded_patterns(rng, 8)
    L = synth.integer_layer(rng, 37, 29, taps, 0.5)
    x = rng.integers(-8, 9, (2, 29, 21, 35)).astype(np.float32)
    g = run_layer(pp, runner, L, x)
    y, _ = oracle_layer_full(oracle_mod, L, x)
    assert (g.astype(np.float64) == y).all()
    if ring:
        g2 = run_layer(pp, runner, L, x, kernel=pp.PP_KERNEL_REGISTER)
        assert (g2.astype(np.float64) == y).all()
    # integers below 2^11 are exact in tf32, so the 3xTF32 kernel is exact too
    g3 = run_layer(pp, runner, L, x, kernel=pp.PP_KERNEL_TC)
    assert (g3.astype(np.float64) == y).all()


DIRECT_CASES = [
    # N, Ci, Co, H, W: first-layer and last-layer shapes, ragged tiles and filter blocks
    (1, 3, 64, 37, 46),
    (2, 1, 64, 33, 64),
    (1, 16, 16, 32, 32),
    (1, 64, 1, 40, 72),
    (3, 2, 5, 17, 23),
    (1, 5, 17, 64, 30),
    (2, 16, 3, 8, 8),
    (1, 4, 20, 1, 1),
]


@pytest.mark.parametrize("case", DIRECT_CASES)
@pytest.mark.parametrize("flags", ["none", "skip_relu", "pool_relu", "skip_pool_relu"])
def test_direct_kernel(pp, runner, oracle_mod, case, flags):
    """The direct FMA kernel (dense 9-tap weights, few input or output channels) against the oracle."""
    N, Ci, Co, H, W = case
    pool = "pool" in flags
    if pool and (H % 2 or W % 2):
        pytest.skip("pool needs even sizes")
    rng = np.random.default_rng(7 * sum(case) + len(flags))
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.6, ring=sum(case) % 2 == 1)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32) if "skip" in flags else None
    g = run_layer(pp, runner, L, x, skip, flags != "none", pool, kernel=pp.PP_KERNEL_DIRECT)
    y, s = oracle_layer_full(oracle_mod, L, x, skip, flags != "none", pool)
    check_within(g, y, s, f"direct kernel {case} {flags}")


def test_direct_kernel_input_only_4_byte_aligned(pp, runner, oracle_mod):
    """An input that starts 4 bytes past a 16-byte boundary takes the 4-byte copy path (same results)."""
    N, Ci, Co, H, W = 1, 3, 24, 20, 36
    rng = np.random.default_rng(41)
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.8)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    dl = runner.DeviceLayer(L)
    try:
        pp.pp_layer_set_kernel(dl.handle, pp.PP_KERNEL_DIRECT)
        buf = torch.zeros(x.size + 1, device="cuda")
        xs = buf[1:].view(N, Ci, H, W)
        xs.copy_(torch.from_numpy(x))
        assert xs.data_ptr() % 16 == 4
        out = torch.full((N, Co, H, W), float("nan"), device="cuda")
        dl.forward(xs, out, None, N, H, W, pp.PP_RELU, torch.cuda.current_stream())
        torch.cuda.synchronize()
        y, s = oracle_layer_full(oracle_mod, L, x, None, True, False)
        check_within(out.cpu().numpy(), y, s, "direct kernel, 4-byte aligned input")
    finally:
        dl.close()


def test_direct_kernel_integer_bit_exact_and_selection(pp, runner, oracle_mod):
    """Integer weights and inputs are summed exactly; a 3-channel first layer picks the direct
    kernel by default, a wide layer cannot set it."""
    rng = np.random.default_rng(31)
    L = synth.integer_layer(rng, 16, 12, synth.seeded_patterns(rng, 8), 0.5)
    x = rng.integers(-8, 9, (2, 12, 19, 27)).astype(np.float32)
    g = run_layer(pp, runner, L, x, kernel=pp.PP_KERNEL_DIRECT)
    y, _ = oracle_layer_full(oracle_mod, L, x)
    assert (g.astype(np.float64) == y).all()
    first = runner.DeviceLayer(synth.small_random_layer(rng, 64, 3, P=8, keep=1.0))
    wide = runner.DeviceLayer(synth.small_random_layer(rng, 32, 32, P=8, keep=0.5))
    try:
        assert pp.pp_layer_kernel(first.handle) == pp.PP_KERNEL_DIRECT
        with pytest.raises(pp.PPError) as e:
            pp.pp_layer_set_kernel(wide.handle, pp.PP_KERNEL_DIRECT)
        assert e.value.code == pp.PP_ERR_UNSUPPORTED
    finally:
        first.close()
        wide.close()


@pytest.mark.parametrize("kernel", ["AUTO", "REGISTER", "TMEM", "TC", "TC_FLAT", "DIRECT"])
def test_single_pattern_layer(pp, runner, oracle_mod, kernel):
    """Column pruning (one pattern for every kept kernel of the layer, Section 2's demo variant) is the
    one-pattern case of the same format: every kernel that can run it matches the oracle."""
    rng = np.random.default_rng(17)
    taps = synth.ring8_patterns()[3:4]  # a single ring pattern, so the TMEM kernel applies too
    Co, Ci = (130, 16) if kernel != "DIRECT" else (16, 12)
    L = synth.make_pruned_layer(rng, Co, Ci, taps, 0.6, 0.1, 0.01)
    assert L.taps.shape[0] == 1
    x = rng.uniform(-1, 1, (1, Ci, 18, 22)).astype(np.float32)
    g = run_layer(pp, runner, L, x, None, True, True, kernel=getattr(pp, "PP_KERNEL_" + kernel))
    y, s = oracle_layer_full(oracle_mod, L, x, None, True, True)
    check_within(g, y, s, f"single-pattern layer, {kernel}")


@pytest.mark.parametrize("kernel", ["AUTO", "TC", "TC_FLAT", "TMEM", "DIRECT"])
def test_batchnorm_folded_layer(pp, runner, oracle_mod, kernel):
    """Section 3's conv + BN fusion: an inference batch normalisation folded into a pruned layer's
    weights and bias on the host (pp_fold_batchnorm), then packed and run through pp_conv_forward,
    equals BN applied to the oracle's fp64 conv of the unfolded layer within 1e-5 * S, S the budget of
    the folded layer (the one-rounding-per-weight fold error is far below it)."""
    rng = np.random.default_rng(77)
    Co, Ci, N, H, W = (130, 24, 2, 18, 20) if kernel != "DIRECT" else (12, 3, 2, 18, 20)
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.5)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    gamma = rng.uniform(0.5, 2.0, Co).astype(np.float32)
    beta = rng.normal(0, 0.3, Co).astype(np.float32)
    mean = rng.normal(0, 0.2, Co).astype(np.float32)
    var = rng.uniform(0.2, 3.0, Co).astype(np.float32)
    eps = 1e-5
    wf, bf = pp.pp_fold_batchnorm(L.w, L.bias, gamma, beta, mean, var, eps)
    folded = synth.PrunedLayer(w=wf, mask=L.mask, taps=L.taps, bias=bf, pattern_ids=L.pattern_ids)
    g = run_layer(pp, runner, folded, x, None, True, False,
                  kernel=None if kernel == "AUTO" else getattr(pp, "PP_KERNEL_" + kernel))
    # BN(conv(x) + b) in fp64 from the unfolded layer, then ReLU
    pat = oracle_mod.pattern_ids(L.w, L.mask, L.taps)
    z, _ = oracle_mod.conv_pruned(x, L.w, pat, L.taps, L.bias)
    scale = gamma.astype(np.float64) / np.sqrt(var.astype(np.float64) + eps)
    ybn = (z - mean.astype(np.float64)[None, :, None, None]) * scale[None, :, None, None] + beta.astype(np.float64)[None, :, None, None]
    ybn = oracle_mod.relu(ybn)
    # budget of the layer as run: |b'| + sum |w' x|
    pat_f = oracle_mod.pattern_ids(wf, L.mask, L.taps)
    _, s = oracle_mod.conv_pruned(x, wf, pat_f, L.taps, bf)
    check_within(g, ybn, s, f"BN-folded layer, kernel {kernel}")


def test_all_pruned_layer_gives_bias(pp, runner, oracle_mod):
    rng = np.random.default_rng(8)
    L = synth.small_random_layer(rng, 20, 10, P=8, keep=0.0)
    assert L.nk == 0
    x = rng.uniform(-1, 1, (1, 10, 9, 9)).astype(np.float32)
    g = run_layer(pp, runner, L, x)
    assert (g == L.bias[None, :, None, None]).all()


def test_dense_layers(pp, runner, oracle_mod):
    rng = np.random.default_rng(12)
    for Co, Ci, H, W, relu, skip in ((64, 1, 37, 50, True, False), (1, 64, 40, 33, False, True),
                                     (7, 5, 16, 16, True, False)):
        D = synth.make_dense_layer(rng, Co, Ci, synth.he_std(Ci), 0.01)
        x = rng.uniform(0, 1, (1, Ci, H, W)).astype(np.float32)
        sk = rng.uniform(0, 1, (1, Co, H, W)).astype(np.float32) if skip else None
        g = run_layer(pp, runner, D, x, sk, relu)
        y, s = oracle_layer_full(oracle_mod, D, x, sk, relu)
        check_within(g, y, s, f"dense {Co}x{Ci}")


def test_cfg0_full(pp, runner, oracle_mod):
    net = synth.cfg0_single()
    L = net.ops[0].layer
    g = run_layer(pp, runner, L, net.x)
    y, s = oracle_layer_full(oracle_mod, L, net.x)
    check_within(g, y, s, "cfg0")


def layerwise_check(pp, runner, oracle_mod, net, check_net=True, fold_perm=False, precision=0):
    """Run a network op by op on the GPU and check every output of every op against the oracle
    evaluated on the GPU's own input to that op (rearranged into the original channel order when the
    filter reorder is folded into the next layer); then check the executor reproduces the op-by-op
    result bit for bit (direct launches and CUDA-graph replay) and the host-buffer path too."""
    dn = runner.DeviceNet(net, use_graph=True, fold_perm=fold_perm, precision=precision)
    try:
        x = dev(net.x)
        acts = dn.run_layerwise(x)
        torch.cuda.synchronize()
        worst = 0.0
        for k, op in enumerate(net.ops):
            xin = to_original(acts[k].cpu().numpy(), dn.layouts[k])
            out = to_original(acts[k + 1].cpu().numpy(), dn.layouts[k + 1])
            skip = to_original(acts[op.skip_from].cpu().numpy(), dn.layouts[op.skip_from]) if op.skip_from >= 0 else None
            y, s = oracle_layer_full(oracle_mod, op.layer, xin, skip, op.relu, op.pool)
            worst = max(worst, check_within(out, y, s, f"{net.name} op {k}"))
            del y, s, xin, out, skip
        if check_net:
            final = acts[-1]
            y1 = torch.empty_like(final)
            dn.run(x, y1)
            dn.run(x, y1)  # second call replays the captured graph
            torch.cuda.synchronize()
            assert torch.equal(y1, final)
            xh = torch.from_numpy(net.x).pin_memory()
            yh = torch.empty(final.shape, dtype=torch.float32).pin_memory()
            dn.run_host(xh, yh)
            assert torch.equal(yh, final.cpu())
        for L in dn.layers:
            if not L.dense:
                assert pp.pp_layer_device_status(L.handle) == 0
        return worst
    finally:
        dn.close()


def test_cfg1_vgg16(pp, runner, oracle_mod):
    assert layerwise_check(pp, runner, oracle_mod, synth.cfg1_vgg16()) < 1e-5


def test_cfg2_style(pp, runner, oracle_mod):
    assert layerwise_check(pp, runner, oracle_mod, synth.cfg2_style()) < 1e-5


def test_cfg3_vdsr(pp, runner, oracle_mod):
    assert layerwise_check(pp, runner, oracle_mod, synth.cfg3_vdsr()) < 1e-5


@pytest.mark.parametrize("name", ["vgg16", "style"])
def test_permutation_folded_networks(pp, runner, oracle_mod, name):
    """Section 3's filter reorder folded into the next layer (activations kept in reordered channel
    order between layers, the next layer's input channels permuted at pack time): every op still
    matches the oracle on every output, the network output is in the original order, and the folded
    executor reproduces its own op-by-op result bit for bit."""
    net = synth.cfg1_vgg16() if name == "vgg16" else synth.cfg2_style()
    assert layerwise_check(pp, runner, oracle_mod, net, fold_perm=True) < 1e-5


def test_permutation_folded_layouts(pp, runner):
    """Which activations the folding keeps in the original order: the network input and output, the
    skip chain of the style trunk; every other VGG activation is in its producer's reordered order."""
    dn = runner.DeviceNet(synth.cfg1_vgg16(), use_graph=False, fold_perm=True)
    try:
        ident = [bool((l == np.arange(len(l))).all()) for l in dn.layouts]
        assert ident[0] and ident[-1] and not any(ident[1:-1])
        for k, L in enumerate(dn.layers[:-1]):
            assert (dn.layouts[k + 1] == L.perm()).all()
    finally:
        dn.close()
    net = synth.cfg2_style()
    dn = runner.DeviceNet(net, use_graph=False, fold_perm=True)
    try:
        for k, op in enumerate(net.ops):
            l = dn.layouts[k + 1]
            assert bool((l == np.arange(len(l))).all()) == (op.skip_from >= 0)
    finally:
        dn.close()


def test_cfg3_small_full(pp, runner, oracle_mod):
    """The VDSR-shaped stack on a small ragged image, every output of every op checked."""
    net = synth.cfg3_vdsr(H=37, W=45)
    dn = runner.DeviceNet(net, use_graph=False)
    try:
        acts = dn.run_layerwise(dev(net.x))
        torch.cuda.synchronize()
        for k, op in enumerate(net.ops):
            skip = acts[op.skip_from].cpu().numpy() if op.skip_from >= 0 else None
            y, s = oracle_layer_full(oracle_mod, op.layer, acts[k].cpu().numpy(), skip, op.relu, op.pool)
            check_within(acts[k + 1].cpu().numpy(), y, s, f"vdsr small op {k}")
    finally:
        dn.close()


@pytest.mark.parametrize("point", synth.cfg4_points())
def test_cfg4_sweep_point(pp, runner, oracle_mod, point):
    """Every output of every sweep point, at the kernel autotuning picks for its shape (as the bench runs it)."""
    C, P, keep = point
    net = synth.cfg4_point(C, P, keep)
    L = net.ops[0].layer
    N, _, H, W = net.x.shape
    dl = runner.DeviceLayer(L)
    try:
        pp.pp_layer_autotune(dl.handle, N, H, W, 0, torch.cuda.current_stream())
        y = torch.full((N, C, H, W), float("nan"), device="cuda")
        dl.forward(dev(net.x), y, None, N, H, W, 0, torch.cuda.current_stream())
        torch.cuda.synchronize()
        assert pp.pp_layer_device_status(dl.handle) == 0
        g = y.cpu().numpy()
    finally:
        dl.close()
    yr, s = oracle_layer_full(oracle_mod, L, net.x)
    check_within(g, yr, s, f"sweep {point}")


def test_bad_arguments_rejected(pp, runner):
    rng = np.random.default_rng(1)
    L = runner.DeviceLayer(synth.small_random_layer(rng, 4, 4))
    x = torch.zeros((1, 4, 5, 5), device="cuda")
    y = torch.zeros((1, 4, 5, 5), device="cuda")
    try:
        with pytest.raises(pp.PPError) as e:
            L.forward(x, y, None, 1, 5, 5, pp.PP_POOL2, None)
        assert e.value.code == pp.PP_ERR_UNSUPPORTED
        with pytest.raises(pp.PPError) as e:
            L.forward(x, y, None, 1, 5, 5, pp.PP_ADD_SKIP, None)
        assert e.value.code == pp.PP_ERR_INVALID_ARG
        with pytest.raises(pp.PPError) as e:
            L.forward(x, y, None, 1, 5, 5, 64, None)
        assert e.value.code == pp.PP_ERR_INVALID_ARG
        with pytest.raises(pp.PPError) as e:
            L.forward(x, y, None, 0, 5, 5, 0, None)
        assert e.value.code == pp.PP_ERR_INVALID_ARG
    finally:
        L.close()


def test_bounded_wait_gives_up_and_device_stays_usable(pp, runner, oracle_mod):
    """A wait that nothing completes (the poll of the tensor-core kernels' waits, on an mbarrier nobody
    arrives on) gives up and says so; a full wait of PP_WAIT_POLLS polls is bounded in time; the context
    stays usable (a tensor-core conv right after is within the bound)."""
    best = None
    for _ in range(3):  # the fastest of three probes: a stall during one probe does not count
        gave_up, ns = pp.pp_wait_probe(1024)
        assert gave_up == 1 and ns > 0
        best = ns if best is None else min(best, ns)
    full_wait_s = best / 1024 * pp.PP_WAIT_POLLS / 1e9
    print(f"one poll {best / 1024:.1f} ns; a full wait gives up after ~{full_wait_s:.2f} s")
    assert full_wait_s < 5.0
    rng = np.random.default_rng(404)
    L = synth.small_random_layer(rng, 40, 24, P=8, keep=0.4)
    x = rng.uniform(-1, 1, (1, 24, 12, 20)).astype(np.float32)
    g = run_layer(pp, runner, L, x, None, True, False, kernel=pp.PP_KERNEL_TC)
    y, s = oracle_layer_full(oracle_mod, L, x, None, True, False)
    check_within(g, y, s, "tensor-core conv after a given-up wait")


def test_run_host_graph_and_plain_paths(pp, runner):
    """pp_net_run_host on a non-default stream: page-locked buffers take the captured graph (copies and ops
    in one graph, replayed on the second call and re-captured for other buffers), pageable buffers the
    op-by-op path, and graphs off the plain path; all give the device run's output bit for bit."""
    for spec in (synth.cfg0_single(), synth.cfg2_style()):
        run_host_paths(pp, runner, spec)


def run_host_paths(pp, runner, spec):
    dn = runner.DeviceNet(spec, use_graph=True)
    try:
        s = torch.cuda.Stream()
        x = torch.from_numpy(spec.x).cuda()
        ref = torch.empty(dn.out_shape, device="cuda")
        dn.run(x, ref, s)
        s.synchronize()
        ref = ref.cpu()
        outs = []
        xh = torch.from_numpy(spec.x).pin_memory()
        for _ in range(2):
            yh = torch.full(dn.out_shape, float("nan")).pin_memory()
            dn.run_host(xh, yh, s)
            outs.append(yh)
        yh2 = torch.full(dn.out_shape, float("nan")).pin_memory()  # other buffers: captured again
        dn.run_host(xh, yh2, s)
        outs.append(yh2)
        yp = torch.full(dn.out_shape, float("nan"))  # pageable: copies issued one by one
        dn.run_host(torch.from_numpy(spec.x.copy()), yp, s)
        outs.append(yp)
        pp.pp_net_use_graph(dn.net, False)
        yo = torch.full(dn.out_shape, float("nan")).pin_memory()
        dn.run_host(xh, yo, s)
        outs.append(yo)
        for o in outs:
            assert torch.equal(o, ref)
    finally:
        dn.close()


@pytest.mark.parametrize("kernel", ["TC", "TC_FLAT", "TMEM", "REGISTER", "DIRECT"])
def test_output_order_every_kernel(pp, runner, oracle_mod, kernel):
    """pp_layer_set_output_order: original filter o lands in channel order[o] on every kernel (skip read at
    the same channel, pooling included), NULL restores the original order."""
    rng = np.random.default_rng(91)
    Co, Ci = (12, 3) if kernel == "DIRECT" else (136, 24)
    N, H, W = 2, 14, 18
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.5)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32)
    order = rng.permutation(Co).astype(np.int32)
    flags = pp.PP_ADD_SKIP | pp.PP_RELU | pp.PP_POOL2
    y, s = oracle_layer_full(oracle_mod, L, x, skip, True, True)
    dl = runner.DeviceLayer(L)
    try:
        pp.pp_layer_set_kernel(dl.handle, getattr(pp, "PP_KERNEL_" + kernel))
        for ordv in (order, None):
            pp.pp_layer_set_output_order(dl.handle, ordv, torch.cuda.current_stream())
            sk = skip.copy()
            if ordv is not None:
                sk[:, ordv] = skip  # the skip tensor in the output's channel order
            out = torch.full((N, Co, H // 2, W // 2), float("nan"), device="cuda")
            dl.forward(dev(x), out, dev(sk), N, H, W, flags, torch.cuda.current_stream())
            torch.cuda.synchronize()
            g = out.cpu().numpy()
            g = g[:, ordv] if ordv is not None else g  # back to the original order
            check_within(g, y, s, f"output order {kernel} {'set' if ordv is not None else 'reset'}")
        bad = order.copy()
        bad[0] = bad[1]
        with pytest.raises(pp.PPError) as e:
            pp.pp_layer_set_output_order(dl.handle, bad, torch.cuda.current_stream())
        assert e.value.code == pp.PP_ERR_INVALID_ARG
    finally:
        dl.close()


def test_peak_probes(pp):
    """pp_peak_probe: the FFMA probe runs near the FP32 lanes' rate at the SM clock it reports, and the
    tensor-core probes well above it (f16 above tf32)."""
    props = torch.cuda.get_device_properties(0)
    tf, mhz, ms = pp.pp_peak_probe(pp.PP_PROBE_FFMA, 1 << 14)
    assert 300 < mhz < 2500 and ms > 0
    lanes_rate = props.multi_processor_count * 128 * 2 * mhz * 1e6 / 1e12
    assert 0.5 * lanes_rate < tf < 1.05 * lanes_rate, (tf, lanes_rate)
    t32, m32, _ = pp.pp_peak_probe(pp.PP_PROBE_MMA_TF32, 1 << 12)
    t16, m16, _ = pp.pp_peak_probe(pp.PP_PROBE_MMA_F16, 1 << 12)
    assert t32 > 5 * tf and t16 > 1.3 * t32, (tf, t32, t16)
    assert 300 < m32 < 2500 and 300 < m16 < 2500


# ----------------------------------------------------------------------------- fp16 split (PP_PRECISION_F16X3)

F16 = 1  # PP_PRECISION_F16X3


@pytest.mark.parametrize("case", SMALL)
@pytest.mark.parametrize("flags", ["none", "skip_relu", "pool_relu"])
@pytest.mark.parametrize("kernel", ["TC", "TC_FLAT"])
def test_f16_small(pp, runner, oracle_mod, case, flags, kernel):
    """The fp16-split arithmetic on every small case, both tensor-core kernels (layers with at most 64
    filters run the row-tiled kernel for TC_FLAT), every output."""
    N, Ci, Co, H, W, P, ring, keep = case
    if flags == "pool_relu" and (H % 2 or W % 2):
        pytest.skip("pool needs even sizes")
    rng = np.random.default_rng(13 * sum(case[:5]) + len(flags))
    L = synth.small_random_layer(rng, Co, Ci, P=P, keep=keep, ring=ring)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32) if flags == "skip_relu" else None
    k = getattr(pp, "PP_KERNEL_" + kernel) if (kernel == "TC" or Co > 64) else pp.PP_KERNEL_TC
    g = run_layer(pp, runner, L, x, skip, flags != "none", flags == "pool_relu", kernel=k, precision=F16)
    y, s = oracle_layer_full(oracle_mod, L, x, skip, flags != "none", flags == "pool_relu")
    check_within(g, y, s, f"f16 {kernel} {case} {flags}")


@pytest.mark.parametrize("case", FLAT_CASES)
@pytest.mark.parametrize("flags", ["none", "skip_pool_relu"])
def test_f16_flat_kernel(pp, runner, oracle_mod, case, flags):
    N, Ci, Co, H, W = case
    pool = "pool" in flags and H % 2 == 0 and W % 2 == 0
    rng = np.random.default_rng(17 * sum(case) + len(flags))
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.45, ring=sum(case) % 2 == 0)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32) if "skip" in flags else None
    g = run_layer(pp, runner, L, x, skip, flags != "none", pool, kernel=pp.PP_KERNEL_TC_FLAT, precision=F16)
    y, s = oracle_layer_full(oracle_mod, L, x, skip, flags != "none", pool)
    check_within(g, y, s, f"f16 flat {case} {flags}")


WIDE_F16_CASES = [
    # N, Ci, Co, H, W, flags, whether split geometries exist; flat-kernel f16 tiles of more than 128 columns
    # (the second accumulator in the other TMEM buffer, single-buffered)
    (8, 64, 100, 56, 56, "relu", False),           # unsplit: 152 or 112 tiles of 3 or 4 rows; ragged filter block
    (8, 48, 256, 56, 56, "skip_relu", False),      # unsplit, 304 or 224 tiles: several per CTA, one buffer
    (1, 96, 200, 28, 28, "skip_pool_relu", True),  # 8 or 10 tiles of 8 or 6 rows, unsplit and split 2 / 4
    (2, 40, 130, 20, 30, "skip_relu", True),       # ragged channel chunk and filter block, unsplit and split 2
]


@pytest.mark.parametrize("case", WIDE_F16_CASES)
def test_f16_flat_wide_tiles(pp, runner, oracle_mod, case):
    """Every f16 flat-kernel geometry wider than 128 columns the planner accepts, two launches each, against
    the oracle on every output (single-buffered: with several tiles per CTA each tile's MMAs wait for the
    previous tile's epilogue)."""
    N, Ci, Co, H, W, flags, split = case
    rng = np.random.default_rng(N * 1000 + Ci + W)
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.4)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32) if "skip" in flags else None
    relu, pool = "relu" in flags, "pool" in flags
    y, s = oracle_layer_full(oracle_mod, L, x, skip, relu, pool)
    f = (pp.PP_RELU if relu else 0) | (pp.PP_POOL2 if pool else 0) | (pp.PP_ADD_SKIP if skip is not None else 0)
    Ho, Wo = (H // 2, W // 2) if pool else (H, W)
    bcols = (W + 2 + 7) // 8 * 8
    dl = runner.DeviceLayer(L, precision=F16)
    try:
        pp.pp_layer_set_kernel(dl.handle, pp.PP_KERNEL_TC_FLAT)
        wide = []
        for R in range(1, 17):
            if (R * bcols + 15) // 16 * 16 <= 128:
                continue
            for S in (1, 2, 4, 8, 16):
                try:
                    pp.pp_layer_pin_flat_geometry(dl.handle, N, H, W, f, R, S)
                except pp.PPError as e:
                    assert e.code == pp.PP_ERR_UNSUPPORTED
                    continue
                for rep in range(2):
                    out = torch.full((N, Co, Ho, Wo), float("nan"), device="cuda")
                    dl.forward(dev(x), out, None if skip is None else dev(skip), N, H, W, f,
                               torch.cuda.current_stream())
                    torch.cuda.synchronize()
                    assert pp.pp_layer_device_status(dl.handle) == 0
                    check_within(out.cpu().numpy(), y, s, f"{case} wide f16 R={R} S={S} #{rep}")
                wide.append((R, S))
        assert any(S == 1 for _, S in wide), wide
        assert any(S > 1 for _, S in wide) == split, wide
        # CTA pairs keep f16 tiles within 128 columns
        for R in range(1, 17):
            if (R * bcols + 15) // 16 * 16 > 128:
                for S in (2, 4, 8):
                    with pytest.raises(pp.PPError):
                        pp.pp_layer_pin_flat_geometry(dl.handle, N, H, W, f, R, pp.PP_FLAT_PAIRED | S)
    finally:
        dl.close()


@pytest.mark.parametrize("shape", [(1, 40, 130, 7, 100), (2, 16, 200, 4, 144), (1, 24, 64, 6, 160)] + PFR_CASES)
@pytest.mark.parametrize("flags", ["none", "skip_relu", "pool_relu"])
def test_f16_row_tiled(pp, runner, oracle_mod, shape, flags):
    """Row-tiled kernel under f16: pixel-major (128- and 64-filter blocks), flattened rows, filter-major."""
    N, Ci, Co, H, W = shape
    pool = flags == "pool_relu"
    if pool and (H % 2 or W % 2):
        pytest.skip("pool needs even sizes")
    rng = np.random.default_rng(19 * sum(shape) + len(flags))
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.4)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32) if flags == "skip_relu" else None
    g = run_layer(pp, runner, L, x, skip, flags != "none", pool, kernel=pp.PP_KERNEL_TC, precision=F16)
    y, s = oracle_layer_full(oracle_mod, L, x, skip, flags != "none", pool)
    check_within(g, y, s, f"f16 row-tiled {shape} {flags}")


@pytest.mark.parametrize("shape,kernel", [((1, 136, 130, 28, 28), "TC_FLAT"), ((6, 40, 200, 14, 14), "TC_FLAT"),
                                          ((1, 40, 64, 20, 150), "TC"), ((2, 24, 130, 9, 40), "TC")])
def test_f16_integer_bit_exact(pp, runner, oracle_mod, shape, kernel):
    """Integer weights in [-4, 4] and inputs in [-8, 8]: f16 holds them exactly (lo parts zero), the
    power-of-two scales are exact and every partial sum is an exact fp32 value, so the result equals
    the oracle bit for bit."""
    N, Ci, Co, H, W = shape
    rng = np.random.default_rng(Co + W + 1)
    L = synth.integer_layer(rng, Co, Ci, synth.ring8_patterns(), 0.5)
    x = rng.integers(-8, 9, (N, Ci, H, W)).astype(np.float32)
    g = run_layer(pp, runner, L, x, None, True, False, kernel=getattr(pp, "PP_KERNEL_" + kernel), precision=F16)
    y, _ = oracle_layer_full(oracle_mod, L, x, None, True, False)
    assert (g.astype(np.float64) == y).all()


@pytest.mark.parametrize("shape,kernel", [((12, 256, 256, 56, 56), "TC"), ((8, 64, 64, 128, 128), "TC"),
                                          ((12, 256, 256, 56, 56), "TC_FLAT"), ((1, 512, 512, 28, 28), "TC_FLAT"),
                                          ((1, 512, 512, 14, 14), "TC_FLAT"), ((2, 128, 128, 112, 112), "TC_FLAT")])
def test_f16_repeatable_multi_tile(pp, runner, oracle_mod, shape, kernel):
    """As test_tensor_core_repeatable_multi_tile, under f16: five runs bit for bit equal, every output
    within the bound, device status clear."""
    N, Ci, Co, H, W = shape
    rng = np.random.default_rng(Ci + W + 2)
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=1.0)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    dl = runner.DeviceLayer(L, precision=F16)
    try:
        pp.pp_layer_set_kernel(dl.handle, getattr(pp, "PP_KERNEL_" + kernel))
        xd = dev(x)
        outs = []
        for _ in range(5):
            y = torch.full((N, Co, H, W), float("nan"), device="cuda")
            dl.forward(xd, y, None, N, H, W, 0, torch.cuda.current_stream())
            outs.append(y)
        torch.cuda.synchronize()
        for k in range(1, 5):
            assert torch.equal(outs[0], outs[k]), f"run {k} differs from run 0"
        assert pp.pp_layer_device_status(dl.handle) == 0
        yr, s = oracle_layer_full(oracle_mod, L, x)
        check_within(outs[0].cpu().numpy(), yr, s, f"f16 multi-tile {shape}")
    finally:
        dl.close()


@pytest.mark.parametrize("name", ["vgg16", "style", "vdsr"])
def test_f16_workloads(pp, runner, oracle_mod, name):
    """The three networks under f16 (every pruned layer with a tensor-core layout), every output of
    every op against the oracle on the GPU's own input, executor replays bit for bit."""
    net = {"vgg16": synth.cfg1_vgg16, "style": synth.cfg2_style, "vdsr": synth.cfg3_vdsr}[name]()
    assert layerwise_check(pp, runner, oracle_mod, net, precision=F16) < 1e-5


@pytest.mark.parametrize("point", synth.cfg4_points())
def test_f16_sweep_point(pp, runner, oracle_mod, point):
    """Every output of every sweep point under f16, at the kernel autotuning picks for its shape."""
    C, P, keep = point
    net = synth.cfg4_point(C, P, keep)
    L = net.ops[0].layer
    N, _, H, W = net.x.shape
    dl = runner.DeviceLayer(L, precision=F16)
    try:
        pp.pp_layer_autotune(dl.handle, N, H, W, 0, torch.cuda.current_stream())
        y = torch.full((N, C, H, W), float("nan"), device="cuda")
        dl.forward(dev(net.x), y, None, N, H, W, 0, torch.cuda.current_stream())
        torch.cuda.synchronize()
        assert pp.pp_layer_device_status(dl.handle) == 0
        g = y.cpu().numpy()
    finally:
        dl.close()
    yr, s = oracle_layer_full(oracle_mod, L, net.x)
    check_within(g, yr, s, f"f16 sweep {point}")


@pytest.mark.parametrize("kernel", ["TC", "TC_FLAT"])
def test_f16_input_range(pp, runner, oracle_mod, kernel):
    """An input that overflows fp16 after the layer's input scale (70000 at scale 1) is flagged in the
    device status word (bit 1), not silently wrong; with a bound that covers it (input scale 2^-3 for a
    bound of 1e5) the same input is within the error bound; the precision and scale read back."""
    rng = np.random.default_rng(5)
    Co, Ci, N, H, W = 136, 16, 1, 12, 20
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.5)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    x[0, 3, 5, 7] = 70000.0
    dl = runner.DeviceLayer(L, precision=F16)
    try:
        pp.pp_layer_set_kernel(dl.handle, getattr(pp, "PP_KERNEL_" + kernel))
        assert pp.pp_layer_precision(dl.handle) == (F16, 1.0)
        y = torch.empty((N, Co, H, W), device="cuda")
        dl.forward(dev(x), y, None, N, H, W, 0, torch.cuda.current_stream())
        torch.cuda.synchronize()
        assert pp.pp_layer_device_status(dl.handle) == pp.PP_STATUS_F16_RANGE
        assert pp.pp_layer_device_status(dl.handle) == 0  # cleared by the read
        pp.pp_layer_set_precision(dl.handle, F16, 1e5)
        assert pp.pp_layer_precision(dl.handle) == (F16, 2.0 ** -3)
        dl.forward(dev(x), y, None, N, H, W, 0, torch.cuda.current_stream())
        torch.cuda.synchronize()
        assert pp.pp_layer_device_status(dl.handle) == 0
        yr, s = oracle_layer_full(oracle_mod, L, x)
        check_within(y.cpu().numpy(), yr, s, f"f16 {kernel} with a bound of 1e5")
        pp.pp_layer_set_precision(dl.handle, 0)
        assert pp.pp_layer_precision(dl.handle) == (0, 1.0)
    finally:
        dl.close()
