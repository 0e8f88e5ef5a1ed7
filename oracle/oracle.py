"""Python side of the fp64 CPU oracle for pattern- and connectivity-pruned 3x3 conv.

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` use it.  The product library never imports,
links or runs anything under ``oracle/``, and this module imports nothing from
the product package.

The arithmetic lives in ``ppconv_oracle.c`` (plain loops, fp64); this module
only builds it with gcc and marshals numpy arrays.  Section references are to
Niu et al., IJCAI-20 demo paper (Section 2: structured pruning; Section 3:
sparse storage and matrix reorder).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ppconv_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")

OR_OK = 0
OR_INVALID_ARG = 1
OR_BAD_PATTERN_SET = 2
OR_TAP_NOT_IN_PATTERN = 3
OR_PRUNED_NONZERO = 4
OR_PATTERN_ID_MISMATCH = 5

_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP when available).  Returns the .so path."""
    os.makedirs(_BUILD, exist_ok=True)
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    base = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    lib = ctypes.CDLL(build())
    P = ctypes.c_void_p
    i32 = ctypes.c_int
    i64 = ctypes.c_int64
    lib.oracle_num_threads.restype = i32
    lib.oracle_pattern_ids.argtypes = [P, P, P, i32, i32, i32, P, P]
    lib.oracle_pattern_ids.restype = i32
    lib.oracle_pack.argtypes = [P, P, P, i32, i32, i32, P, P, P, P, P, P, P]
    lib.oracle_pack.restype = i32
    lib.oracle_conv_pruned.argtypes = [P, i32, i32, i32, i32, P, P, P, P, i32, P, P]
    lib.oracle_conv_pruned_points.argtypes = [P, i32, i32, i32, i32, P, P, P, P, i32, i64, P, P, P]
    lib.oracle_conv_dense.argtypes = [P, i32, i32, i32, i32, P, P, i32, P, P]
    lib.oracle_conv_dense_points.argtypes = [P, i32, i32, i32, i32, P, P, i32, i64, P, P, P]
    lib.oracle_relu.argtypes = [P, i64]
    lib.oracle_add.argtypes = [P, P, P, i64]
    lib.oracle_pool2.argtypes = [P, P, i64, i32, i32, P, P]
    _lib = lib
    return lib


def _p(a):
    return None if a is None else a.ctypes.data


def _c(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


class OracleError(ValueError):
    def __init__(self, code: int):
        super().__init__(f"oracle validation failed with code {code}")
        self.code = code


def num_threads() -> int:
    return int(_load().oracle_num_threads())


def pattern_ids(w, mask, taps, given=None) -> np.ndarray:
    """Pattern id of every kept kernel, -1 for pruned ones (Section 2).

    w [Co][Ci][9] (or [Co][Ci][3][3]) fp32, mask [Co][Ci] uint8, taps [P][4] uint8.
    Raises OracleError on a violated invariant.
    """
    w = _c(w, np.float32).reshape(w.shape[0], w.shape[1], 9)
    Co, Ci = w.shape[:2]
    mask = _c(mask, np.uint8)
    taps = _c(taps, np.uint8)
    given = _c(given, np.uint8)
    pat = np.empty((Co, Ci), np.int32)
    rc = _load().oracle_pattern_ids(_p(w), _p(mask), _p(taps), taps.shape[0], Co, Ci, _p(given), _p(pat))
    if rc != OR_OK:
        raise OracleError(rc)
    return pat


@dataclass
class Packed:
    perm: np.ndarray  # [Co] int32
    kptr: np.ndarray  # [Co+1] int32
    kidx: np.ndarray  # [nk] int32
    kpat: np.ndarray  # [nk] uint8
    kw: np.ndarray  # [nk][4] float32


def pack(w, mask, taps, given=None) -> Packed:
    """Compact storage + matrix reorder of Section 3, in the oracle's reading."""
    w = _c(w, np.float32).reshape(w.shape[0], w.shape[1], 9)
    Co, Ci = w.shape[:2]
    mask = _c(mask, np.uint8)
    taps = _c(taps, np.uint8)
    given = _c(given, np.uint8)
    cap = max(1, Co * Ci)
    perm = np.empty(Co, np.int32)
    kptr = np.empty(Co + 1, np.int32)
    kidx = np.empty(cap, np.int32)
    kpat = np.empty(cap, np.uint8)
    kw = np.empty((cap, 4), np.float32)
    nk = ctypes.c_int64(0)
    rc = _load().oracle_pack(_p(w), _p(mask), _p(taps), taps.shape[0], Co, Ci, _p(given), _p(perm), _p(kptr),
                             _p(kidx), _p(kpat), _p(kw), ctypes.addressof(nk))
    if rc != OR_OK:
        raise OracleError(rc)
    n = nk.value
    return Packed(perm, kptr, kidx[:n].copy(), kpat[:n].copy(), kw[:n].copy())


def conv_pruned(x, w, pat, taps, bias=None):
    """fp64 pruned conv (definition).  Returns (y, s), both [N][Co][H][W] float64."""
    x = _c(x, np.float32)
    N, Ci, H, W = x.shape
    w = _c(w, np.float32).reshape(-1, Ci, 9)
    Co = w.shape[0]
    pat = _c(pat, np.int32)
    taps = _c(taps, np.uint8)
    bias = _c(bias, np.float32)
    y = np.empty((N, Co, H, W), np.float64)
    s = np.empty_like(y)
    _load().oracle_conv_pruned(_p(x), N, Ci, H, W, _p(w), _p(pat), _p(taps), _p(bias), Co, _p(y), _p(s))
    return y, s


def conv_pruned_points(x, w, pat, taps, bias, pts):
    """The pruned conv at output points pts[k] = (n, o, r, c).  Returns (y, s) [npts]."""
    x = _c(x, np.float32)
    N, Ci, H, W = x.shape
    w = _c(w, np.float32).reshape(-1, Ci, 9)
    Co = w.shape[0]
    pts = _c(pts, np.int64).reshape(-1, 4)
    y = np.empty(pts.shape[0], np.float64)
    s = np.empty_like(y)
    _load().oracle_conv_pruned_points(_p(x), N, Ci, H, W, _p(w), _p(_c(pat, np.int32)), _p(_c(taps, np.uint8)),
                                      _p(_c(bias, np.float32)), Co, pts.shape[0], _p(pts), _p(y), _p(s))
    return y, s


def conv_dense(x, w, bias=None):
    """fp64 dense 3x3 conv over all 9 taps.  Returns (y, s)."""
    x = _c(x, np.float32)
    N, Ci, H, W = x.shape
    w = _c(w, np.float32).reshape(-1, Ci, 9)
    Co = w.shape[0]
    bias = _c(bias, np.float32)
    y = np.empty((N, Co, H, W), np.float64)
    s = np.empty_like(y)
    _load().oracle_conv_dense(_p(x), N, Ci, H, W, _p(w), _p(bias), Co, _p(y), _p(s))
    return y, s


def conv_dense_points(x, w, bias, pts):
    x = _c(x, np.float32)
    N, Ci, H, W = x.shape
    w = _c(w, np.float32).reshape(-1, Ci, 9)
    Co = w.shape[0]
    pts = _c(pts, np.int64).reshape(-1, 4)
    y = np.empty(pts.shape[0], np.float64)
    s = np.empty_like(y)
    _load().oracle_conv_dense_points(_p(x), N, Ci, H, W, _p(w), _p(_c(bias, np.float32)), Co, pts.shape[0],
                                     _p(pts), _p(y), _p(s))
    return y, s


def relu(y):
    y = np.ascontiguousarray(y, dtype=np.float64).copy()
    _load().oracle_relu(_p(y), y.size)
    return y


def add(y, s, skip):
    y = np.ascontiguousarray(y, dtype=np.float64).copy()
    s = np.ascontiguousarray(s, dtype=np.float64).copy()
    skip = _c(skip, np.float32)
    assert skip.shape == y.shape
    _load().oracle_add(_p(y), _p(s), _p(skip), y.size)
    return y, s


def pool2(y, s):
    y = np.ascontiguousarray(y, dtype=np.float64)
    s = np.ascontiguousarray(s, dtype=np.float64)
    N, C, H, W = y.shape
    y2 = np.empty((N, C, H // 2, W // 2), np.float64)
    s2 = np.empty_like(y2)
    _load().oracle_pool2(_p(y), _p(s), N * C, H, W, _p(y2), _p(s2))
    return y2, s2


def epilogue(y, s, relu_on=False, skip=None, pool=False):
    """Apply the layer epilogue in the library's order: +skip, then ReLU, then 2x2 max pool."""
    if skip is not None:
        y, s = add(y, s, skip)
    if relu_on:
        y = relu(y)
    if pool:
        y, s = pool2(y, s)
    return y, s
