"""codecgauge: GB300-native encode/decode path of Codec-Gauge's cache-coordinate layer.

Thin Python binding over the C ABI of ``libcodecgauge.so`` (declared in
``include/codecgauge.h``): the functions below only marshal torch device tensors into
pointers and the current CUDA stream. Every step of encode (gauge rotation, block ranges,
scales, codes, packing) and decode (unpacking, dequantization, inverse rotation) runs in
the library's CUDA kernels. There is no CPU fallback: if the shared library is missing
or fails to load, every call raises.

Names follow the paper's notation (Sec. 3): X the cache tensor [L][2][B][H][T][d], G the
gauges [L][2][H][d/g][g][g], g the group size, B_c the compressed buffers.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

__all__ = ["CG_BLOCK_UNIFORM", "CG_KIVI", "CG_NONE", "CG_BLOCK_TILE", "CG_TILE_TOKENS", "Shape", "Params",
           "packed_bytes", "encode", "decode", "get_status", "lib_path", "load", "CodecGaugeError",
           "kivi_stream_bytes", "kivi_stream_alloc", "kivi_append", "kivi_stream_decode",
           "attention_workspace_bytes", "attention", "encode_hadamard", "decode_hadamard"]

CG_BLOCK_UNIFORM, CG_KIVI, CG_NONE, CG_BLOCK_TILE = 0, 1, 2, 3
CG_TILE_TOKENS = 16
CG_FLAG_NONFINITE_INPUT, CG_FLAG_FP16_OVERFLOW, CG_FLAG_PIPE_TIMEOUT = 1, 2, 4
_STATUS = {0: "CG_OK", -1: "CG_EINVAL", -2: "CG_EUNSUPPORTED", -3: "CG_ECUDA", -4: "CG_ERANGE"}

_HERE = os.path.dirname(os.path.abspath(__file__))


def lib_path() -> str:
    return os.path.join(_HERE, "libcodecgauge.so")


class CodecGaugeError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{_STATUS.get(code, code)}: {msg}")
        self.code = code


class _CShape(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("L", "B", "H", "T", "d", "t0", "T_cap")]


class _CParams(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("backend", "group", "bits", "block", "residual")]


@dataclass(frozen=True)
class Shape:
    L: int
    B: int
    H: int
    T: int
    d: int
    t0: int = 0
    T_cap: int = 0

    def c(self) -> _CShape:
        return _CShape(self.L, self.B, self.H, self.T, self.d, self.t0, self.T_cap)


@dataclass(frozen=True)
class Params:
    backend: int
    group: int
    bits: int = 4
    block: int = 64
    residual: int = 0

    def c(self) -> _CParams:
        return _CParams(self.backend, self.group, self.bits, self.block, self.residual)


_lib = None


def load():
    """Load libcodecgauge.so (raises if it is missing: build it with ``__graft_entry__.build()``)."""
    global _lib
    if _lib is None:
        p = lib_path()
        if not os.path.exists(p):
            raise CodecGaugeError(-3, f"CUDA extension not built: {p} is missing")
        L = ctypes.CDLL(p)
        P, vp = ctypes.POINTER, ctypes.c_void_p
        L.cg_packed_bytes.restype = ctypes.c_int
        L.cg_packed_bytes.argtypes = [P(_CShape), P(_CParams), P(ctypes.c_size_t), P(ctypes.c_size_t),
                                      P(ctypes.c_size_t)]
        L.cg_encode.restype = ctypes.c_int
        L.cg_encode.argtypes = [P(_CShape), P(_CParams), vp, vp, vp, vp, vp, vp]
        L.cg_decode.restype = ctypes.c_int
        L.cg_decode.argtypes = [P(_CShape), P(_CParams), vp, vp, vp, vp, vp, vp]
        L.cg_kivi_stream_bytes.restype = ctypes.c_int
        L.cg_kivi_stream_bytes.argtypes = [P(_CShape), P(_CParams)] + [P(ctypes.c_size_t)] * 4
        L.cg_kivi_append.restype = ctypes.c_int
        L.cg_kivi_append.argtypes = [P(_CShape), P(_CParams), vp, vp, vp, vp, vp, vp, ctypes.c_size_t, vp]
        L.cg_kivi_stream_decode.restype = ctypes.c_int
        L.cg_kivi_stream_decode.argtypes = [P(_CShape), P(_CParams), vp, vp, vp, vp, vp, vp]
        L.cg_attention_workspace_bytes.restype = ctypes.c_int
        L.cg_attention_workspace_bytes.argtypes = [P(_CShape), P(_CParams), ctypes.c_int, P(ctypes.c_size_t)]
        L.cg_attention.restype = ctypes.c_int
        L.cg_attention.argtypes = [P(_CShape), P(_CParams), ctypes.c_int, ctypes.c_float, vp, vp, vp, vp, vp, vp,
                                   ctypes.c_size_t, vp]
        L.cg_encode_hadamard.restype = ctypes.c_int
        L.cg_encode_hadamard.argtypes = [P(_CShape), P(_CParams), vp, vp, vp, vp]
        L.cg_decode_hadamard.restype = ctypes.c_int
        L.cg_decode_hadamard.argtypes = [P(_CShape), P(_CParams), vp, vp, vp, vp]
        L.cg_get_status.restype = ctypes.c_int
        L.cg_get_status.argtypes = [vp, P(ctypes.c_int32)]
        L.cg_last_error.restype = ctypes.c_char_p
        L.cg_last_error.argtypes = []
        _lib = L
    return _lib


def _check(rc: int):
    if rc != 0:
        raise CodecGaugeError(rc, load().cg_last_error().decode())


def packed_bytes(shape: Shape, params: Params) -> tuple[int, int, int]:
    """(codes, scales, residual) byte counts of the packed buffers (closed form)."""
    c, s, r = ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_size_t()
    _check(load().cg_packed_bytes(ctypes.byref(shape.c()), ctypes.byref(params.c()), ctypes.byref(c),
                                  ctypes.byref(s), ctypes.byref(r)))
    return c.value, s.value, r.value


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def encode(shape: Shape, params: Params, kv, gauges, codes, scales=None, residual=None, stream=None) -> None:
    """Encode (Z = G X, B_c = C(Z)) into caller-allocated device buffers (torch tensors)."""
    _check(load().cg_encode(ctypes.byref(shape.c()), ctypes.byref(params.c()), _ptr(kv), _ptr(gauges),
                            _ptr(codes), _ptr(scales), _ptr(residual), _stream(stream)))


def decode(shape: Shape, params: Params, codes, scales, residual, gauges, out, stream=None) -> None:
    """Decode (Zhat = D(B_c), Xhat = G^T Zhat) into the caller's bf16 output tensor."""
    _check(load().cg_decode(ctypes.byref(shape.c()), ctypes.byref(params.c()), _ptr(codes), _ptr(scales),
                            _ptr(residual), _ptr(gauges), _ptr(out), _stream(stream)))


def kivi_stream_bytes(shape: Shape, params: Params) -> tuple[int, int, int, int]:
    """(codes, scales, ring, workspace) byte counts of a KIVI stream of capacity shape.T_cap."""
    v = [ctypes.c_size_t() for _ in range(4)]
    _check(load().cg_kivi_stream_bytes(ctypes.byref(shape.c()), ctypes.byref(params.c()),
                                       *[ctypes.byref(x) for x in v]))
    return tuple(x.value for x in v)


def kivi_stream_alloc(shape: Shape, params: Params, device="cuda"):
    """Zero-filled device buffers (codes, scales, ring, workspace) of a KIVI stream."""
    import torch
    nc, ns, nr, nw = kivi_stream_bytes(shape, params)
    return (torch.zeros(max(nc, 16), dtype=torch.uint8, device=device),
            torch.zeros(max(ns // 4, 4), dtype=torch.int32, device=device),
            torch.zeros(max(nr // 2, 8), dtype=torch.int16, device=device),
            torch.zeros(max(nw // 2, 8), dtype=torch.int16, device=device))


def kivi_append(shape: Shape, params: Params, kv_new, gauges, codes, scales, ring, workspace=None,
                stream=None) -> None:
    """Append tokens [t0, t0 + T) (kv_new holds only them) to a KIVI stream holding t0 tokens."""
    nbytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(load().cg_kivi_append(ctypes.byref(shape.c()), ctypes.byref(params.c()), _ptr(kv_new), _ptr(gauges),
                                 _ptr(codes), _ptr(scales), _ptr(ring), _ptr(workspace), nbytes,
                                 _stream(stream)))


def kivi_stream_decode(shape: Shape, params: Params, codes, scales, ring, gauges, out, stream=None) -> None:
    """Decode the T tokens a KIVI stream holds (shape.t0 = 0) into the caller's bf16 output."""
    _check(load().cg_kivi_stream_decode(ctypes.byref(shape.c()), ctypes.byref(params.c()), _ptr(codes),
                                        _ptr(scales), _ptr(ring), _ptr(gauges), _ptr(out), _stream(stream)))


def attention_workspace_bytes(shape: Shape, params: Params, n_rep: int) -> int:
    """Workspace bytes of cg_attention for this cache shape and query heads per KV head."""
    v = ctypes.c_size_t()
    _check(load().cg_attention_workspace_bytes(ctypes.byref(shape.c()), ctypes.byref(params.c()), n_rep,
                                               ctypes.byref(v)))
    return v.value


def attention(shape: Shape, params: Params, n_rep: int, scale: float, q, codes, scales, gauges, out, workspace,
              stream=None) -> None:
    """Softmax attention of one query per sequence (q bf16 [L][B][H][n_rep][d]) over tokens
    [t0, t0 + T) of a block-uniform cache, straight from its codes; out fp32 [L][B][H][n_rep][d]."""
    nbytes = workspace.numel() * workspace.element_size()
    _check(load().cg_attention(ctypes.byref(shape.c()), ctypes.byref(params.c()), n_rep, scale, _ptr(q), _ptr(codes),
                               _ptr(scales), _ptr(gauges), _ptr(out), _ptr(workspace), nbytes, _stream(stream)))


def encode_hadamard(shape: Shape, params: Params, kv, codes, scales, stream=None) -> None:
    """cg_encode with the Hadamard gauge H_g / sqrt(g), by fast Walsh-Hadamard transform."""
    _check(load().cg_encode_hadamard(ctypes.byref(shape.c()), ctypes.byref(params.c()), _ptr(kv), _ptr(codes),
                                     _ptr(scales), _stream(stream)))


def decode_hadamard(shape: Shape, params: Params, codes, scales, out, stream=None) -> None:
    """cg_decode with the Hadamard gauge H_g / sqrt(g), by fast Walsh-Hadamard transform."""
    _check(load().cg_decode_hadamard(ctypes.byref(shape.c()), ctypes.byref(params.c()), _ptr(codes), _ptr(scales),
                                     _ptr(out), _stream(stream)))


def get_status(stream=None) -> int:
    """Synchronize the stream, return and clear the device's CG_FLAG_* bits."""
    v = ctypes.c_int32()
    _check(load().cg_get_status(_stream(stream), ctypes.byref(v)))
    return v.value


def alloc_outputs(shape: Shape, params: Params, device="cuda"):
    """Zero-filled device buffers (codes, scales, residual) sized by packed_bytes."""
    import torch
    nc, ns, nr = packed_bytes(shape, params)
    codes = torch.zeros(max(nc, 16), dtype=torch.uint8, device=device)
    scales = torch.zeros(max(ns // 4, 4), dtype=torch.int32, device=device)
    resid = torch.zeros(max(nr // 2, 8), dtype=torch.int16, device=device)
    return codes, scales, resid
