"""Python binding of the C-ABI library (``include/ppconv.h``), by ctypes.

Same names as the C entry points; each wrapper only marshals arguments
(numpy arrays for host data, integers or torch tensors for device pointers,
``torch.cuda.Stream``/int/None for streams) and raises ``PPError`` on a
non-zero status.  Every step of the computation runs in the compiled library.
Importing this module loads ``_build/libppconv.so`` and fails loudly if it has
not been built (``paper_2004_11250_gb300.build.build()``).
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import numpy as np

from .build import LIB as _LIB_PATH

if not os.path.exists(_LIB_PATH):
    raise ImportError(f"{_LIB_PATH} is missing: build it with paper_2004_11250_gb300.build.build() "
                      "(or __graft_entry__.build()); there is no fallback path")

lib = ctypes.CDLL(_LIB_PATH)

PP_OK = 0
PP_ERR_INVALID_ARG = 1
PP_ERR_BAD_PATTERN_SET = 2
PP_ERR_TAP_NOT_IN_PATTERN = 3
PP_ERR_PRUNED_NONZERO = 4
PP_ERR_PATTERN_ID_MISMATCH = 5
PP_ERR_UNSUPPORTED = 6
PP_ERR_CUDA = 7
PP_ERR_OOM = 8

PP_KERNEL_AUTO = 0
PP_KERNEL_TMEM = 1
PP_KERNEL_REGISTER = 2
PP_KERNEL_TC = 3
PP_KERNEL_TC_FLAT = 4
PP_KERNEL_DIRECT = 5

PP_WAIT_POLLS = 1 << 18

PP_PROBE_FFMA = 0
PP_PROBE_MMA_TF32 = 1
PP_PROBE_MMA_F16 = 2

PP_PRECISION_TF32X3 = 0
PP_PRECISION_F16X3 = 1
PP_FLAT_PAIRED = 256  # or-ed into a flat-kernel split: CTA pairs over two filter blocks

PP_STATUS_TIMEOUT = 1
PP_STATUS_F16_RANGE = 2

PP_ADD_SKIP = 1
PP_RELU = 2
PP_POOL2 = 4

_P = ctypes.c_void_p
_I = ctypes.c_int
_I64 = ctypes.c_int64
_PP = ctypes.POINTER(ctypes.c_void_p)

_SIGS = {
    "pp_status_string": ([_I], ctypes.c_char_p),
    "pp_version": ([], _I),
    "pp_pack_layer": ([_P, _P, _P, _I, _I, _I, _P, _PP], _I),
    "pp_packed_info": ([_P, _P, _P, _P, _P], _I),
    "pp_packed_arrays": ([_P, _PP, _PP, _PP, _PP, _PP, _PP], _I),
    "pp_unpack_layer": ([_P, _P, _P], _I),
    "pp_fold_batchnorm": ([_P, _P, _P, _P, _P, _P, ctypes.c_float, _I, _I], _I),
    "pp_packed_destroy": ([_P], None),
    "pp_layer_create": ([_P, _P, _P, _PP], _I),
    "pp_layer_info": ([_P, _P, _P, _P], _I),
    "pp_conv_forward": ([_P, _P, _P, _P, _I, _I, _I, _I, _P], _I),
    "pp_conv_forward_noalloc": ([_P, _P, _P, _P, _I, _I, _I, _I, _P], _I),
    "pp_layer_set_kernel": ([_P, _I], _I),
    "pp_layer_set_output_order": ([_P, _P, _P], _I),
    "pp_layer_set_precision": ([_P, _I, ctypes.c_float, _P], _I),
    "pp_layer_precision": ([_P, _P, _P], _I),
    "pp_permute_input_channels": ([_P, _P, _P, _I, _I, _P, _P, _P, _P], _I),
    "pp_layer_kernel": ([_P, _P], _I),
    "pp_layer_device_status": ([_P, _P], _I),
    "pp_wait_probe": ([ctypes.c_longlong, _P, _P], _I),
    "pp_peak_probe": ([_I, ctypes.c_longlong, _P, _P, _P], _I),
    "pp_layer_autotune": ([_P, _I, _I, _I, _I, _P], _I),
    "pp_layer_flat_geometry": ([_P, _I, _I, _I, _I, _P, _P], _I),
    "pp_layer_pin_flat_geometry": ([_P, _I, _I, _I, _I, _I, _I], _I),
    "pp_layer_destroy": ([_P], None),
    "pp_dense_create": ([_P, _P, _I, _I, _P, _PP], _I),
    "pp_dense_forward": ([_P, _P, _P, _P, _I, _I, _I, _I, _P], _I),
    "pp_dense_info": ([_P, _P, _P], _I),
    "pp_dense_destroy": ([_P], None),
    "pp_net_create": ([_I, _I, _I, _I, _PP], _I),
    "pp_net_add_conv": ([_P, _P, _I, _I], _I),
    "pp_net_add_dense": ([_P, _P, _I, _I], _I),
    "pp_net_finalize": ([_P], _I),
    "pp_net_output_shape": ([_P, _P, _P, _P, _P], _I),
    "pp_net_use_graph": ([_P, _I], _I),
    "pp_net_run": ([_P, _P, _P, _P], _I),
    "pp_net_run_host": ([_P, _P, _P, _P], _I),
    "pp_net_destroy": ([_P], None),
}
for _name, (_args, _res) in _SIGS.items():
    _fn = getattr(lib, _name)
    _fn.argtypes = _args
    _fn.restype = _res


class PPError(RuntimeError):
    def __init__(self, code: int, where: str = ""):
        super().__init__(f"{where}: {pp_status_string(code)} ({code})")
        self.code = code


def pp_fold_batchnorm(w, bias, gamma, beta, mean, var, eps=1e-5):
    """Batch normalisation after the conv folded into (w [Co][Ci][3][3] or [Co][Ci][9], bias [Co] or None):
    returns new fp32 arrays (w in the shape given, bias [Co])."""
    import numpy as np
    w2 = np.array(w, dtype=np.float32, order="C", copy=True)
    Co, Ci = w2.shape[0], w2.shape[1]
    b2 = np.zeros(Co, np.float32) if bias is None else np.array(bias, dtype=np.float32, copy=True)
    arrs = [np.ascontiguousarray(a, dtype=np.float32) for a in (gamma, beta, mean, var)]
    for a in arrs:
        if a.shape != (Co,):
            raise ValueError("batch-norm parameters must have shape [Co]")
    _check(lib.pp_fold_batchnorm(w2.ctypes.data, b2.ctypes.data, *[a.ctypes.data for a in arrs], float(eps), Co, Ci),
           "pp_fold_batchnorm")
    return w2, b2


def pp_permute_input_channels(w, mask, layout, pattern_ids=None):
    """(w, mask, ids) with input channel c of the result = original channel layout[c]; ids None if not given."""
    w = _host(w, np.float32)
    Co, Ci = w.shape[0], w.shape[1]
    w = w.reshape(Co, Ci, 9)
    mask = _host(mask, np.uint8)
    ids = _host(pattern_ids, np.uint8)
    lay = _host(layout, np.int32)
    if mask.shape != (Co, Ci) or lay.shape != (Ci,) or (ids is not None and ids.shape != (Co, Ci)):
        raise PPError(PP_ERR_INVALID_ARG, "pp_permute_input_channels shapes")
    w2 = np.empty_like(w)
    m2 = np.empty_like(mask)
    i2 = None if ids is None else np.empty_like(ids)
    _check(lib.pp_permute_input_channels(_hp(w), _hp(mask), _hp(ids), Co, Ci, _hp(lay), _hp(w2), _hp(m2), _hp(i2)),
           "pp_permute_input_channels")
    return w2, m2, i2


def pp_status_string(code: int) -> str:
    return lib.pp_status_string(code).decode()


def pp_version() -> int:
    return lib.pp_version()


def _check(st: int, where: str):
    if st != PP_OK:
        raise PPError(st, where)


def _host(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


def _hp(a):
    return None if a is None else a.ctypes.data


def _dp(t) -> Optional[int]:
    """Device pointer of a torch tensor or an int; None stays NULL."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(s) -> Optional[int]:
    if s is None:
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


# ------------------------------------------------------------------ packer


def pp_pack_layer(w, mask, pattern_taps, pattern_ids=None) -> int:
    """Pack a pruned layer; returns an opaque handle (free with pp_packed_destroy)."""
    w = _host(w, np.float32)
    Co, Ci = w.shape[0], w.shape[1]
    w = w.reshape(Co, Ci, 9)
    mask = _host(mask, np.uint8)
    taps = _host(pattern_taps, np.uint8)
    ids = _host(pattern_ids, np.uint8)
    if mask.shape != (Co, Ci) or taps.ndim != 2 or taps.shape[1] != 4 or (ids is not None and ids.shape != (Co, Ci)):
        raise PPError(PP_ERR_INVALID_ARG, "pp_pack_layer shapes")
    out = ctypes.c_void_p()
    _check(lib.pp_pack_layer(_hp(w), _hp(mask), _hp(taps), taps.shape[0], Co, Ci, _hp(ids), ctypes.byref(out)),
           "pp_pack_layer")
    return out.value


def pp_packed_info(pk):
    nk, co, ci, p = _I64(), _I(), _I(), _I()
    _check(lib.pp_packed_info(pk, ctypes.byref(nk), ctypes.byref(co), ctypes.byref(ci), ctypes.byref(p)),
           "pp_packed_info")
    return nk.value, co.value, ci.value, p.value


def pp_packed_arrays(pk) -> dict:
    """Copies of the stored arrays: perm, kptr, kidx, kpat, kw [nk][4], taps [P][4]."""
    nk, Co, Ci, P = pp_packed_info(pk)
    ptrs = [ctypes.c_void_p() for _ in range(6)]
    _check(lib.pp_packed_arrays(pk, *[ctypes.byref(p) for p in ptrs]), "pp_packed_arrays")

    def view(ptr, ctype, n, dtype):
        if n == 0:
            return np.zeros(0, dtype)
        buf = (ctype * n).from_address(ptr.value)
        return np.frombuffer(buf, dtype=dtype, count=n).copy()

    return {
        "perm": view(ptrs[0], ctypes.c_int32, Co, np.int32),
        "kptr": view(ptrs[1], ctypes.c_int32, Co + 1, np.int32),
        "kidx": view(ptrs[2], ctypes.c_int32, nk, np.int32),
        "kpat": view(ptrs[3], ctypes.c_uint8, nk, np.uint8),
        "kw": view(ptrs[4], ctypes.c_float, 4 * nk, np.float32).reshape(nk, 4),
        "taps": view(ptrs[5], ctypes.c_uint8, 4 * P, np.uint8).reshape(P, 4),
    }


def pp_unpack_layer(pk):
    nk, Co, Ci, P = pp_packed_info(pk)
    w = np.empty((Co, Ci, 9), np.float32)
    mask = np.empty((Co, Ci), np.uint8)
    _check(lib.pp_unpack_layer(pk, _hp(w), _hp(mask)), "pp_unpack_layer")
    return w, mask


def pp_packed_destroy(pk):
    lib.pp_packed_destroy(pk)


# ------------------------------------------------------------------ device layers


def pp_layer_create(pk, bias=None, stream=None) -> int:
    b = _host(bias, np.float32)
    out = ctypes.c_void_p()
    _check(lib.pp_layer_create(pk, _hp(b), _stream(stream), ctypes.byref(out)), "pp_layer_create")
    return out.value


def pp_layer_info(layer):
    co, ci, nb = _I(), _I(), _I64()
    _check(lib.pp_layer_info(layer, ctypes.byref(co), ctypes.byref(ci), ctypes.byref(nb)), "pp_layer_info")
    return co.value, ci.value, nb.value


def pp_conv_forward(layer, x, y, skip, N, H, W, flags, stream=None):
    _check(lib.pp_conv_forward(layer, _dp(x), _dp(y), _dp(skip), N, H, W, flags, _stream(stream)),
           "pp_conv_forward")


def pp_conv_forward_noalloc(layer, x, y, skip, N, H, W, flags, stream=None):
    """pp_conv_forward through the flat tensor-core kernel, whose split reduction needs no workspace (no device allocation)."""
    _check(lib.pp_conv_forward_noalloc(layer, _dp(x), _dp(y), _dp(skip), N, H, W, flags, _stream(stream)),
           "pp_conv_forward_noalloc")


def pp_layer_set_kernel(layer, kernel: int):
    _check(lib.pp_layer_set_kernel(layer, kernel), "pp_layer_set_kernel")


def pp_layer_set_output_order(layer, order=None, stream=None):
    """order[o] = output channel of original filter o (None: original order); see the header."""
    o = _host(order, np.int32)
    _check(lib.pp_layer_set_output_order(layer, _hp(o), _stream(stream)), "pp_layer_set_output_order")


def pp_layer_set_precision(layer, precision: int, input_bound: float = 0.0, stream=None):
    """PP_PRECISION_TF32X3 or PP_PRECISION_F16X3 for the tensor-core kernels (see the header)."""
    _check(lib.pp_layer_set_precision(layer, precision, float(input_bound), _stream(stream)), "pp_layer_set_precision")


def pp_layer_precision(layer):
    """(precision, input scale)."""
    p, sc = _I(), ctypes.c_float()
    _check(lib.pp_layer_precision(layer, ctypes.byref(p), ctypes.byref(sc)), "pp_layer_precision")
    return p.value, sc.value


def pp_layer_kernel(layer) -> int:
    k = _I()
    _check(lib.pp_layer_kernel(layer, ctypes.byref(k)), "pp_layer_kernel")
    return k.value


def pp_layer_autotune(layer, N, H, W, flags, stream=None):
    _check(lib.pp_layer_autotune(layer, N, H, W, flags, _stream(stream)), "pp_layer_autotune")


def pp_layer_flat_geometry(layer, N, H, W, flags):
    """(R, S) pinned for the flat tensor-core kernel at this shape, (0, 0) if none."""
    R, S = _I(), _I()
    _check(lib.pp_layer_flat_geometry(layer, N, H, W, flags, ctypes.byref(R), ctypes.byref(S)), "pp_layer_flat_geometry")
    return R.value, S.value


def pp_layer_pin_flat_geometry(layer, N, H, W, flags, R, S):
    _check(lib.pp_layer_pin_flat_geometry(layer, N, H, W, flags, R, S), "pp_layer_pin_flat_geometry")


def pp_layer_device_status(layer) -> int:
    v = _I()
    _check(lib.pp_layer_device_status(layer, ctypes.byref(v)), "pp_layer_device_status")
    return v.value


def pp_wait_probe(polls: int):
    """(gave_up, elapsed_ns) of `polls` polls of an mbarrier that nothing completes (see the header)."""
    g, ns = _I(), ctypes.c_longlong()
    _check(lib.pp_wait_probe(polls, ctypes.byref(g), ctypes.byref(ns)), "pp_wait_probe")
    return g.value, ns.value


def pp_peak_probe(kind: int, iters: int):
    """(TFLOP/s, SM MHz, ms) of one launch of a peak-rate probe (PP_PROBE_*; see the header)."""
    tf, mhz, ms = ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
    _check(lib.pp_peak_probe(kind, iters, ctypes.byref(tf), ctypes.byref(mhz), ctypes.byref(ms)), "pp_peak_probe")
    return tf.value, mhz.value, ms.value


def pp_layer_destroy(layer):
    lib.pp_layer_destroy(layer)


def pp_dense_create(w, bias=None, stream=None) -> int:
    w = _host(w, np.float32)
    Co, Ci = w.shape[0], w.shape[1]
    b = _host(bias, np.float32)
    out = ctypes.c_void_p()
    _check(lib.pp_dense_create(_hp(w.reshape(Co, Ci, 9)), _hp(b), Co, Ci, _stream(stream), ctypes.byref(out)),
           "pp_dense_create")
    return out.value


def pp_dense_forward(layer, x, y, skip, N, H, W, flags, stream=None):
    _check(lib.pp_dense_forward(layer, _dp(x), _dp(y), _dp(skip), N, H, W, flags, _stream(stream)),
           "pp_dense_forward")


def pp_dense_info(layer):
    co, ci = _I(), _I()
    _check(lib.pp_dense_info(layer, ctypes.byref(co), ctypes.byref(ci)), "pp_dense_info")
    return co.value, ci.value


def pp_dense_destroy(layer):
    lib.pp_dense_destroy(layer)


# ------------------------------------------------------------------ network


def pp_net_create(N, C, H, W) -> int:
    out = ctypes.c_void_p()
    _check(lib.pp_net_create(N, C, H, W, ctypes.byref(out)), "pp_net_create")
    return out.value


def pp_net_add_conv(net, layer, flags, skip_from=-1):
    _check(lib.pp_net_add_conv(net, layer, flags, skip_from), "pp_net_add_conv")


def pp_net_add_dense(net, layer, flags, skip_from=-1):
    _check(lib.pp_net_add_dense(net, layer, flags, skip_from), "pp_net_add_dense")


def pp_net_finalize(net):
    _check(lib.pp_net_finalize(net), "pp_net_finalize")


def pp_net_output_shape(net):
    v = [_I() for _ in range(4)]
    _check(lib.pp_net_output_shape(net, *[ctypes.byref(a) for a in v]), "pp_net_output_shape")
    return tuple(a.value for a in v)


def pp_net_use_graph(net, enable: bool):
    _check(lib.pp_net_use_graph(net, 1 if enable else 0), "pp_net_use_graph")


def pp_net_run(net, x, y, stream=None):
    _check(lib.pp_net_run(net, _dp(x), _dp(y), _stream(stream)), "pp_net_run")


def pp_net_run_host(net, x_host, y_host, stream=None):
    """x_host / y_host: host buffers (numpy arrays or pinned CPU torch tensors)."""
    xp = x_host.data_ptr() if hasattr(x_host, "data_ptr") else x_host.ctypes.data
    yp = y_host.data_ptr() if hasattr(y_host, "data_ptr") else y_host.ctypes.data
    _check(lib.pp_net_run_host(net, xp, yp, _stream(stream)), "pp_net_run_host")


def pp_net_destroy(net):
    lib.pp_net_destroy(net)
