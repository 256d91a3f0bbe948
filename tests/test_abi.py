"""C-ABI checks that need no GPU: the library loads, exports every symbol the header
declares, computes byte counts equal to the oracle's closed form, and rejects invalid
arguments with the documented status before touching the device."""
import ctypes
import os
import re

import pytest

import oracle
from paper_2607_20538_gb300 import synth

cg = pytest.importorskip("paper_2607_20538_gb300")
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(cg.lib_path()):
        from paper_2607_20538_gb300 import build
        build.build()
    return cg.load()


def _declared_symbols():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            src = open(os.path.join(ROOT, "include", f)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"^\s*(?:const\s+)?\w+[\s\*]+(cg_\w+)\s*\(", src, flags=re.M))
    return names


def test_exports_every_declared_symbol(lib):
    names = _declared_symbols()
    assert {"cg_packed_bytes", "cg_encode", "cg_decode", "cg_get_status", "cg_last_error"} <= names
    for n in names:
        assert hasattr(lib, n), n


@pytest.mark.parametrize("name", list(synth.WORKLOADS))
def test_packed_bytes_match_oracle(lib, name):
    w = synth.WORKLOADS[name]
    assert cg.packed_bytes(cg.Shape(**w.shape), cg.Params(**w.params)) == oracle.packed_bytes(w.shape, w.params)
    for backend in (0, 1, 2, 3):
        for T in (0, 1, 15, 16, 17, 127, 128, 129, 300):
            ww = w.replace(backend=backend, T=T, T_cap=0, L=2, B=2, H=3)
            assert cg.packed_bytes(cg.Shape(**ww.shape), cg.Params(**ww.params)) == \
                oracle.packed_bytes(ww.shape, ww.params)


@pytest.mark.parametrize("bad", [
    dict(group=12), dict(group=256), dict(bits=5), dict(bits=1), dict(block=24), dict(block=4),
    dict(block=256), dict(backend=7), dict(d=48), dict(d=512), dict(T=-1), dict(L=0),
    dict(block=8, bits=3, d=64, group=8, _ok=True),
])
def test_validation(lib, bad):
    kw = dict(L=1, B=1, H=1, T=16, d=128, group=64, backend=0, bits=4, block=64, residual=0)
    ok = bad.pop("_ok", False)
    kw.update(bad)
    shape = cg.Shape(L=kw["L"], B=kw["B"], H=kw["H"], T=kw["T"], d=kw["d"])
    params = cg.Params(kw["backend"], kw["group"], kw["bits"], kw["block"], kw["residual"])
    if ok:
        cg.packed_bytes(shape, params)
        return
    with pytest.raises(cg.CodecGaugeError) as e:
        cg.packed_bytes(shape, params)
    assert e.value.code in (-1, -2)
    assert lib.cg_last_error().decode()


def test_tile_history_offsets(lib):
    """Block-uniform tiles: a call starts at a tile boundary (t0 % 16 == 0); the scales of a
    T_cap history are one pair per tile block, as the oracle counts them."""
    params = cg.Params(cg.CG_BLOCK_TILE, 32, 4, 64)
    for t0, T, T_cap, ok in ((0, 5, 40, True), (16, 9, 40, True), (32, 8, 40, True), (8, 4, 40, False),
                             (17, 1, 40, False), (16, 30, 40, False)):
        sh = dict(L=1, B=2, H=3, T=T, d=128, t0=t0, T_cap=T_cap)
        if ok:
            assert cg.packed_bytes(cg.Shape(**sh), params) == oracle.packed_bytes(sh, params.__dict__)
        else:
            with pytest.raises(cg.CodecGaugeError) as e:
                cg.packed_bytes(cg.Shape(**sh), params)
            assert e.value.code == (-1 if t0 + T > T_cap else -2)


def test_kivi_stream_bytes_and_validation(lib):
    """Stream byte counts as the oracle counts them; argument errors before any device work."""
    params = cg.Params(cg.CG_KIVI, 16, 3, 16, 20)
    for T_cap in (1, 20, 36, 37, 300):
        sh = dict(L=2, B=2, H=3, T=0, d=64, t0=0, T_cap=T_cap)
        nc, ns, nr, nw = cg.kivi_stream_bytes(cg.Shape(**sh), params)
        assert (nc, ns, nr) == oracle.kivi_stream_bytes(sh, params.__dict__)
        assert nw == 2 * 2 * 2 * 3 * 16 * 64 * 2
    S = lambda **k: ctypes.byref(cg.Shape(**{**dict(L=1, B=1, H=1, T=1, d=64, t0=0, T_cap=64), **k}).c())
    P = ctypes.byref(params.c())
    fake = ctypes.c_void_p(0x10000)
    assert lib.cg_kivi_stream_bytes(S(T_cap=0), P, None, None, None, None) == -1
    assert lib.cg_kivi_stream_bytes(S(t0=60, T=5), P, None, None, None, None) == -1
    assert lib.cg_kivi_stream_bytes(S(), ctypes.byref(cg.Params(0, 16, 3, 16).c()), None, None, None, None) == -1
    # appends after the first call carry at most `block` tokens
    assert lib.cg_kivi_append(S(t0=4, T=17), P, fake, fake, fake, fake, fake, fake, 1 << 20, None) == -2
    # an append that completes a key group (t0 = 35 -> 36 tokens: n_q 0 -> 16) needs the workspace
    assert lib.cg_kivi_append(S(t0=35, T=1), P, fake, fake, fake, fake, fake, fake, 16, None) == -1
    assert "workspace" in lib.cg_last_error().decode()
    assert lib.cg_kivi_stream_decode(S(t0=1, T=2), P, fake, fake, fake, fake, fake, None) == -2


def test_attention_validation(lib):
    """cg_attention: supported caches and query-head counts are checked on the host."""
    sh = cg.Shape(L=2, B=3, H=2, T=1100, d=128)
    nb = cg.attention_workspace_bytes(sh, cg.Params(0, 128, 4, 64), 4)
    assert nb == -(-2 * 3 * 2 * 4 * 128 * 4 // 256) * 256 + 2 * 3 * 2 * 9 * 4 * 130 * 4   # queries, 9 chunks
    for params, n_rep in ((cg.Params(cg.CG_KIVI, 64, 3, 128, 128), 4), (cg.Params(0, 16, 4, 16), 4),
                          (cg.Params(0, 16, 4, 64), 3)):
        with pytest.raises(cg.CodecGaugeError):
            cg.attention_workspace_bytes(sh, params, n_rep)
    with pytest.raises(cg.CodecGaugeError):
        cg.attention_workspace_bytes(cg.Shape(L=1, B=1, H=1, T=64, d=64), cg.Params(0, 16, 4, 32), 1)
    fake = ctypes.c_void_p(0x10000)
    S, P = ctypes.byref(sh.c()), ctypes.byref(cg.Params(0, 128, 4, 64).c())
    assert lib.cg_attention(S, P, 4, ctypes.c_float(float("nan")), fake, fake, fake, fake, fake, fake, 1 << 30,
                            None) == -1
    assert lib.cg_attention(S, P, 4, ctypes.c_float(0.1), fake, fake, fake, fake, fake, fake, 16, None) == -1
    assert "workspace" in lib.cg_last_error().decode()


def test_hadamard_validation(lib):
    fake = ctypes.c_void_p(0x10000)
    S = ctypes.byref(cg.Shape(L=1, B=1, H=1, T=4, d=128).c())
    for bad in (cg.Params(cg.CG_KIVI, 64, 3, 128, 0), cg.Params(cg.CG_BLOCK_TILE, 64, 4, 64)):
        assert lib.cg_encode_hadamard(S, ctypes.byref(bad.c()), fake, fake, fake, None) == -2
        assert lib.cg_decode_hadamard(S, ctypes.byref(bad.c()), fake, fake, fake, None) == -2
    P = ctypes.byref(cg.Params(0, 64, 4, 64).c())
    assert lib.cg_encode_hadamard(S, P, None, fake, fake, None) == -1
    assert lib.cg_encode_hadamard(S, P, ctypes.c_void_p(0x10008), fake, fake, None) == -1


def test_pointer_checks_fail_before_device(lib):
    shape = cg.Shape(L=1, B=1, H=1, T=4, d=64)
    params = cg.Params(0, 16, 4, 32)
    S, P = ctypes.byref(shape.c()), ctypes.byref(params.c())
    assert lib.cg_encode(S, P, None, None, None, None, None, None) == -1
    assert lib.cg_decode(S, P, None, None, None, None, None, None) == -1
    assert lib.cg_encode(S, P, ctypes.c_void_p(0x1001), ctypes.c_void_p(0x2000), ctypes.c_void_p(0x3000),
                         ctypes.c_void_p(0x4000), None, None) == -1
    assert "aligned" in lib.cg_last_error().decode()
    kp = cg.Params(1, 16, 4, 32, 8)
    assert lib.cg_encode(ctypes.byref(cg.Shape(L=1, B=1, H=1, T=4, d=64, t0=2, T_cap=8).c()),
                         ctypes.byref(kp.c()), None, None, None, None, None, None) == -2
    assert lib.cg_get_status(None, None) == -1
    # history overflow: t0 + T > T_cap
    assert lib.cg_packed_bytes(ctypes.byref(cg.Shape(L=1, B=1, H=1, T=4, d=64, t0=6, T_cap=8).c()), P,
                               None, None, None) == -1
