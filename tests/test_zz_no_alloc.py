"""pp_conv_forward_noalloc: the flat tensor-core kernel run without any device
allocation by the call, for callers that cannot allocate while they run layers
(their device memory is reserved up front by another allocator, or their loop
cannot take the device-wide synchronisation of cudaMalloc / cudaFree).  Its
cluster-split partial tiles are reduced through distributed shared memory, so
the call needs no workspace.  Checked against pp_conv_forward and the oracle on
two calls in a row, with an unsplit (persistent) and a split geometry pinned,
on a layer whose selected kernel is another one, and against the device's free
memory.  Kept in its own file, named to be collected last, so it runs both
alone in a fresh process and after every other GPU test."""
import numpy as np
import pytest
import torch

from paper_2004_11250_gb300 import synth
from parity import check_within, oracle_layer_full

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pp():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2004_11250_gb300 import build
    build.build()
    from paper_2004_11250_gb300 import ppconv
    return ppconv


# (N, Ci, Co, H, W), flags, pinned (R, S) or None, kernel the layer keeps selected
CASES = [
    ((1, 512, 512, 14, 14), "relu", (14, 4), "TC_FLAT"),      # cluster split, read back through the pin
    ((4, 128, 256, 28, 28), "pool_relu", (8, 1), "TC_FLAT"),  # unsplit, persistent over tiles
    ((2, 64, 200, 20, 30), "skip_relu", None, "TC"),          # the layer runs the row-tiled kernel otherwise
    ((1, 96, 144, 16, 24), "relu", None, "REGISTER"),         # ... or an FMA kernel
]


@pytest.mark.parametrize("shape,flags,geo,kernel", CASES)
def test_noalloc_matches_forward(pp, oracle_mod, shape, flags, geo, kernel):
    from paper_2004_11250_gb300 import runner
    N, Ci, Co, H, W = shape
    rng = np.random.default_rng(Ci + Co + W)
    L = synth.small_random_layer(rng, Co, Ci, P=8, keep=0.3)
    x = rng.uniform(-1, 1, (N, Ci, H, W)).astype(np.float32)
    skip = rng.uniform(-1, 1, (N, Co, H, W)).astype(np.float32) if flags == "skip_relu" else None
    pool = flags == "pool_relu"
    f = pp.PP_RELU | (pp.PP_POOL2 if pool else 0) | (pp.PP_ADD_SKIP if skip is not None else 0)
    Ho, Wo = (H // 2, W // 2) if pool else (H, W)
    dl = runner.DeviceLayer(L)
    try:
        pp.pp_layer_set_kernel(dl.handle, getattr(pp, "PP_KERNEL_" + kernel))
        if geo is not None:
            pp.pp_layer_pin_flat_geometry(dl.handle, N, H, W, f, *geo)
            assert pp.pp_layer_flat_geometry(dl.handle, N, H, W, f) == geo
        xd = torch.from_numpy(x).cuda()
        sd = None if skip is None else torch.from_numpy(skip).cuda()
        ref = torch.full((N, Co, Ho, Wo), float("nan"), device="cuda")
        dl.forward(xd, ref, sd, N, H, W, f, torch.cuda.current_stream())
        outs = [torch.full((N, Co, Ho, Wo), float("nan"), device="cuda") for _ in range(3)]
        # a first call loads the kernel's code (lazy module loading) and sets its attributes
        pp.pp_conv_forward_noalloc(dl.handle, xd, outs.pop(), sd, N, H, W, f, torch.cuda.current_stream())
        torch.cuda.synchronize()
        free0, _ = torch.cuda.mem_get_info()
        for y in outs:  # two calls in a row on the same layer
            pp.pp_conv_forward_noalloc(dl.handle, xd, y, sd, N, H, W, f, torch.cuda.current_stream())
        torch.cuda.synchronize()
        free1, _ = torch.cuda.mem_get_info()
        assert free1 == free0, "the call changed the device's free memory"
        assert pp.pp_layer_device_status(dl.handle) == 0
        assert pp.pp_layer_kernel(dl.handle) == getattr(pp, "PP_KERNEL_" + kernel)  # selection untouched
        yr, s = oracle_layer_full(oracle_mod, L, x, skip, True, pool)
        r = ref.cpu().numpy()
        for k, y in enumerate(outs):
            g = y.cpu().numpy()
            assert np.isfinite(g).all(), f"call {k}: outputs left unwritten"
            # the two entry points agree within the tests' bound of each other ...
            check_within(g, r.astype(np.float64), s, f"noalloc call {k} vs pp_conv_forward")
            # ... and with the oracle
            check_within(g, yr, s, f"noalloc call {k} vs oracle")
        assert torch.equal(outs[0], outs[1])
    finally:
        dl.close()


def test_noalloc_rejects(pp):
    from paper_2004_11250_gb300 import runner
    rng = np.random.default_rng(3)
    small = runner.DeviceLayer(synth.small_random_layer(rng, 32, 16, P=8, keep=0.5))  # 32 filters: no flat kernel
    try:
        x = torch.zeros((1, 16, 8, 8), device="cuda")
        y = torch.zeros((1, 32, 8, 8), device="cuda")
        with pytest.raises(pp.PPError) as e:
            pp.pp_conv_forward_noalloc(small.handle, x, y, None, 1, 8, 8, 0, torch.cuda.current_stream())
        assert e.value.code == pp.PP_ERR_UNSUPPORTED
        with pytest.raises(pp.PPError) as e:
            pp.pp_conv_forward_noalloc(small.handle, x, y, None, 1, 8, 8, 64, torch.cuda.current_stream())
        assert e.value.code == pp.PP_ERR_INVALID_ARG
    finally:
        small.close()
