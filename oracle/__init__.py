"""CPU oracle for the Codec-Gauge encode/decode path (arxiv 2607.20538).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py``. The product package never
imports it. The arithmetic lives in ``cg_oracle.c`` (plain C, compiled with
``-ffp-contract=off`` and no fast-math); this module only marshals numpy arrays.

Pins: ``tests/test_oracle_pins.py``, ``tests/test_oracle_tile_pins.py`` and
``tests/test_oracle_stream_pins.py``, ``tests/test_oracle_attention_pins.py`` (closed forms,
brute force, worked examples, library routines). No function here is "parity unpinned".
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libcgoracle.so")
SRC_PATH = os.path.join(_HERE, "cg_oracle.c")

BU, KIVI, NONE, TILE = 0, 1, 2, 3
TILE_TOKENS = 16  # T_b: tokens per block-uniform tile (Sec. 4.2, Sec. 4.3)


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no fast-math, no FMA contraction)."""
    if force or not os.path.exists(LIB_PATH) or os.path.getmtime(LIB_PATH) < os.path.getmtime(SRC_PATH):
        tmp = LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call([
            "gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math",
            "-pthread", SRC_PATH, "-o", tmp, "-lm"])
        os.replace(tmp, LIB_PATH)
    return LIB_PATH


class _Shape(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("L", "B", "H", "T", "d", "t0", "T_cap")]


class _Params(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("backend", "group", "bits", "block", "residual")]


_lib = None


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(LIB_PATH)
        P = ctypes.POINTER
        L.cgo_f32_to_f16.restype = ctypes.c_uint16
        L.cgo_f32_to_f16.argtypes = [ctypes.c_float]
        L.cgo_f16_to_f32.restype = ctypes.c_float
        L.cgo_f16_to_f32.argtypes = [ctypes.c_uint16]
        L.cgo_kivi_nq.restype = ctypes.c_int64
        L.cgo_kivi_nq.argtypes = [ctypes.c_int64] * 3
        L.cgo_packed_bytes.restype = ctypes.c_int
        L.cgo_packed_bytes.argtypes = [P(_Shape), P(_Params), P(ctypes.c_int64), P(ctypes.c_int64), P(ctypes.c_int64)]
        vp = ctypes.c_void_p
        L.cgo_encode.restype = ctypes.c_int
        L.cgo_encode.argtypes = [P(_Shape), P(_Params), vp, vp, vp, vp, vp, vp, vp, ctypes.c_int, P(ctypes.c_int32)]
        L.cgo_decode.restype = ctypes.c_int
        L.cgo_decode.argtypes = [P(_Shape), P(_Params), vp, vp, vp, vp, vp, ctypes.c_int]
        L.cgo_pack.restype = None
        L.cgo_pack.argtypes = [vp, ctypes.c_int, ctypes.c_int, vp]
        L.cgo_unpack.restype = None
        L.cgo_unpack.argtypes = [vp, ctypes.c_int, ctypes.c_int, vp]
        L.cgo_kivi_stream_bytes.restype = ctypes.c_int
        L.cgo_kivi_stream_bytes.argtypes = [P(_Shape), P(_Params), P(ctypes.c_int64), P(ctypes.c_int64),
                                            P(ctypes.c_int64)]
        L.cgo_kivi_append.restype = ctypes.c_int
        L.cgo_kivi_append.argtypes = [P(_Shape), P(_Params), vp, vp, vp, vp, vp, ctypes.c_int, P(ctypes.c_int32)]
        L.cgo_kivi_stream_decode.restype = ctypes.c_int
        L.cgo_kivi_stream_decode.argtypes = [P(_Shape), P(_Params), vp, vp, vp, vp, vp, ctypes.c_int]
        L.cgo_attention.restype = ctypes.c_int
        L.cgo_attention.argtypes = [ctypes.c_int] * 6 + [vp, vp, ctypes.c_double, vp]
        L.cgo_gauge_coord.restype = ctypes.c_float
        L.cgo_gauge_coord.argtypes = [vp, vp, ctypes.c_int]
        _lib = L
    return _lib


def _ptr(a):
    return None if a is None else ctypes.c_void_p(a.ctypes.data)


def _shape(L, B, H, T, d, t0=0, T_cap=0):
    return _Shape(L, B, H, T, d, t0, T_cap)


def f32_to_f16_bits(x: float) -> int:
    return int(lib().cgo_f32_to_f16(ctypes.c_float(x)))


def f16_bits_to_f32(h: int) -> float:
    return float(lib().cgo_f16_to_f32(ctypes.c_uint16(h)))


def kivi_nq(T: int, R: int, Gt: int) -> int:
    return int(lib().cgo_kivi_nq(T, R, Gt))


def packed_bytes(shape: dict, params: dict):
    c, s, r = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
    rc = lib().cgo_packed_bytes(ctypes.byref(_shape(**shape)), ctypes.byref(_Params(**params)),
                                ctypes.byref(c), ctypes.byref(s), ctypes.byref(r))
    if rc:
        raise ValueError(f"oracle packed_bytes rc={rc}")
    return c.value, s.value, r.value


def pack(q: np.ndarray, bits: int) -> np.ndarray:
    q = np.ascontiguousarray(q, dtype=np.uint8)
    out = np.zeros(q.size * bits // 8, np.uint8)
    lib().cgo_pack(_ptr(q), q.size, bits, _ptr(out))
    return out


def unpack(b: np.ndarray, n: int, bits: int) -> np.ndarray:
    b = np.ascontiguousarray(b, dtype=np.uint8)
    out = np.zeros(n, np.uint8)
    lib().cgo_unpack(_ptr(b), n, bits, _ptr(out))
    return out


def gauge_coord(Grow: np.ndarray, x: np.ndarray) -> np.float32:
    Grow = np.ascontiguousarray(Grow, np.float32)
    x = np.ascontiguousarray(x, np.float32)
    return np.float32(lib().cgo_gauge_coord(_ptr(Grow), _ptr(x), Grow.size))


def encode(shape: dict, params: dict, x_bf16: np.ndarray, gauges: np.ndarray, *, want_z=False,
           want_flags=False, nthreads: int = 0):
    """Returns dict(codes, scales (uint16 pairs), residual, z, flags, status)."""
    sh = dict(t0=0, T_cap=0)
    sh.update(shape)
    nc, ns, nr = packed_bytes(sh, params)
    x = np.ascontiguousarray(x_bf16).view(np.uint16)
    G = np.ascontiguousarray(gauges, np.float32)
    codes = np.zeros(nc, np.uint8)
    scales = np.zeros(ns // 2, np.uint16)
    resid = np.zeros(nr // 2, np.uint16)
    n = sh["L"] * 2 * sh["B"] * sh["H"] * sh["T"] * sh["d"]
    assert x.size == n, (x.size, n)
    z = np.zeros(n, np.float32) if want_z else None
    fl = np.zeros(n, np.uint8) if want_flags else None
    st = ctypes.c_int32(0)
    rc = lib().cgo_encode(ctypes.byref(_shape(**sh)), ctypes.byref(_Params(**params)), _ptr(x), _ptr(G),
                          _ptr(codes), _ptr(scales), _ptr(resid), _ptr(z), _ptr(fl),
                          nthreads or (os.cpu_count() or 1), ctypes.byref(st))
    if rc:
        raise ValueError(f"oracle encode rc={rc}")
    return dict(codes=codes, scales=scales, residual=resid, z=z, flags=fl, status=st.value)


def decode(shape: dict, params: dict, codes, scales, residual, gauges, *, nthreads: int = 0) -> np.ndarray:
    """Returns the recovered cache as float64 [L][2][B][H][T][d] (flattened)."""
    sh = dict(t0=0, T_cap=0)
    sh.update(shape)
    n = sh["L"] * 2 * sh["B"] * sh["H"] * sh["T"] * sh["d"]
    out = np.zeros(n, np.float64)
    codes = np.ascontiguousarray(codes, np.uint8)
    scales = None if scales is None else np.ascontiguousarray(scales).view(np.uint16)
    residual = None if residual is None else np.ascontiguousarray(residual).view(np.uint16)
    G = np.ascontiguousarray(gauges, np.float32)
    rc = lib().cgo_decode(ctypes.byref(_shape(**sh)), ctypes.byref(_Params(**params)), _ptr(codes),
                          _ptr(scales), _ptr(residual), _ptr(G), _ptr(out), nthreads or (os.cpu_count() or 1))
    if rc:
        raise ValueError(f"oracle decode rc={rc}")
    return out


# ---------------------------------------------------------------- KIVI streaming
def kivi_stream_bytes(shape: dict, params: dict):
    """(codes, scales, ring) bytes of a KIVI stream of capacity shape["T_cap"]."""
    c, s, r = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
    sh = dict(t0=0, T_cap=0)
    sh.update(shape)
    rc = lib().cgo_kivi_stream_bytes(ctypes.byref(_shape(**sh)), ctypes.byref(_Params(**params)),
                                     ctypes.byref(c), ctypes.byref(s), ctypes.byref(r))
    if rc:
        raise ValueError(f"oracle kivi_stream_bytes rc={rc}")
    return c.value, s.value, r.value


def kivi_stream_alloc(shape: dict, params: dict):
    """Zeroed stream buffers (codes u8, scales u16 pairs, ring u16) for capacity shape["T_cap"]."""
    nc, ns, nr = kivi_stream_bytes(shape, params)
    return np.zeros(nc, np.uint8), np.zeros(ns // 2, np.uint16), np.zeros(nr // 2, np.uint16)


def kivi_append(shape: dict, params: dict, x_new: np.ndarray, gauges: np.ndarray, codes, scales, ring,
                *, nthreads: int = 0) -> int:
    """Append tokens [t0, t0 + T) to the stream buffers in place; returns the status bits."""
    sh = dict(t0=0, T_cap=0)
    sh.update(shape)
    x = np.ascontiguousarray(x_new).view(np.uint16)
    assert x.size == sh["L"] * 2 * sh["B"] * sh["H"] * sh["T"] * sh["d"]
    G = np.ascontiguousarray(gauges, np.float32)
    st = ctypes.c_int32(0)
    rc = lib().cgo_kivi_append(ctypes.byref(_shape(**sh)), ctypes.byref(_Params(**params)), _ptr(x), _ptr(G),
                               _ptr(codes), _ptr(scales), _ptr(ring), nthreads or (os.cpu_count() or 1),
                               ctypes.byref(st))
    if rc:
        raise ValueError(f"oracle kivi_append rc={rc}")
    return st.value


def kivi_stream_decode(shape: dict, params: dict, codes, scales, ring, gauges, *, nthreads: int = 0) -> np.ndarray:
    """fp64 [L][2][B][H][T][d] of the first T tokens of the stream (t0 = 0)."""
    sh = dict(t0=0, T_cap=0)
    sh.update(shape)
    out = np.zeros(sh["L"] * 2 * sh["B"] * sh["H"] * sh["T"] * sh["d"], np.float64)
    G = np.ascontiguousarray(gauges, np.float32)
    rc = lib().cgo_kivi_stream_decode(ctypes.byref(_shape(**sh)), ctypes.byref(_Params(**params)),
                                      _ptr(np.ascontiguousarray(codes, np.uint8)),
                                      _ptr(np.ascontiguousarray(scales).view(np.uint16)),
                                      _ptr(np.ascontiguousarray(ring).view(np.uint16)), _ptr(G), _ptr(out),
                                      nthreads or (os.cpu_count() or 1))
    if rc:
        raise ValueError(f"oracle kivi_stream_decode rc={rc}")
    return out


# ---------------------------------------------------------------- attention
def attention(shape: dict, n_rep: int, q_bf16: np.ndarray, xhat: np.ndarray, scale: float) -> np.ndarray:
    """fp64 softmax attention of one query per sequence (n_rep query heads per KV head) over the
    decoded cache xhat [L][2][B][H][T][d]; q bf16 [L][B][H][n_rep][d]. Returns [L][B][H][n_rep][d]."""
    L, B, H, T, d = (shape[k] for k in ("L", "B", "H", "T", "d"))
    q = np.ascontiguousarray(q_bf16).view(np.uint16)
    assert q.size == L * B * H * n_rep * d
    xh = np.ascontiguousarray(xhat, np.float64)
    assert xh.size == L * 2 * B * H * T * d
    out = np.zeros(L * B * H * n_rep * d, np.float64)
    rc = lib().cgo_attention(L, B, H, T, d, n_rep, _ptr(q), _ptr(xh), float(scale), _ptr(out))
    if rc:
        raise ValueError(f"oracle attention rc={rc}")
    return out.reshape(L, B, H, n_rep, d)
