"""pp_conv_forward_noalloc: the flat tensor-core kernel with its split partials in
a static device array, against pp_conv_forward on the same layer.  Kept in its
own file, named to be collected last, so it runs both alone in a fresh process
and after every other GPU test."""
import numpy as np
import pytest
import torch

from paper_2004_11250_gb300 import synth
from parity import check_within, oracle_layer_points, sample_points

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pp():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2004_11250_gb300 import build
    build.build()
    from paper_2004_11250_gb300 import ppconv
    return ppconv


@pytest.mark.parametrize("shape,flags", [((1, 512, 512, 14, 14), "relu"), ((1, 256, 512, 28, 28), "pool_relu"),
                                         ((2, 64, 200, 20, 30), "skip_relu")])
def test_noalloc_matches_forward(pp, oracle_mod, shape, flags):
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
        pp.pp_layer_set_kernel(dl.handle, pp.PP_KERNEL_TC_FLAT)
        xd = torch.from_numpy(x).cuda()
        sd = None if skip is None else torch.from_numpy(skip).cuda()
        ref = torch.full((N, Co, Ho, Wo), float("nan"), device="cuda")
        dl.forward(xd, ref, sd, N, H, W, f, torch.cuda.current_stream())
        outs = []
        for _ in range(2):  # two calls in a row reuse the static workspace
            y = torch.full((N, Co, Ho, Wo), float("nan"), device="cuda")
            pp.pp_conv_forward_noalloc(dl.handle, xd, y, sd, N, H, W, f, torch.cuda.current_stream())
            outs.append(y)
        torch.cuda.synchronize()
        assert pp.pp_layer_device_status(dl.handle) == 0
        pts = sample_points(rng, N, Co, Ho, Wo, 1500)
        yr, s = oracle_layer_points(oracle_mod, L, x, pts, skip, True, pool)
        idx = tuple(pts.T)
        r = ref.cpu().numpy()
        for k, y in enumerate(outs):
            g = y.cpu().numpy()
            assert np.isfinite(g).all(), f"call {k}: outputs left unwritten"
            # the two entry points agree within the tests' bound of each other ...
            check_within(g[idx], r[idx].astype(np.float64), s, f"noalloc call {k} vs pp_conv_forward")
            # ... and with the oracle
            check_within(g[idx], yr, s, f"noalloc call {k} vs oracle")
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
