"""cg_kivi_append_static through the C ABI: the KIVI stream append whose staging workspace is
the library's own fixed device array, for callers that cannot allocate device memory.

Two streams receive the same appends: one through cg_kivi_append with a caller-allocated
workspace, one through cg_kivi_append_static. Each of two appends in a row completes a key
group (so both stage through the workspace); after each, codes, scales and ring must be
identical to the bytes (the same kernels run on the same inputs, so bit equality is within
the parity tolerance of the other tests), and the stream decode must agree. A shape whose
workspace exceeds the array is rejected before any launch.
"""
import ctypes

import numpy as np
import pytest

from paper_2607_20538_gb300 import synth

torch = pytest.importorskip("torch")
cg = pytest.importorskip("paper_2607_20538_gb300")

pytestmark = pytest.mark.gpu


def _p(t):
    return ctypes.c_void_p(t.data_ptr())


def _stream():
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def test_static_append_matches_workspace_append():
    lib = cg.load()
    lib.cg_kivi_append_static.restype = ctypes.c_int
    lib.cg_kivi_append_static.argtypes = [ctypes.c_void_p] * 8
    w = synth.Workload(name="noalloc", L=2, B=2, H=2, T=0, d=128, group=64, backend=1, bits=3, block=128,
                       residual=128)
    T_cap = 600
    params = cg.Params(**w.params)
    cap = cg.Shape(L=w.L, B=w.B, H=w.H, T=0, d=w.d, t0=0, T_cap=T_cap)
    x = synth.kv_cache(w.replace(T=512), threads=4)
    dG = torch.from_numpy(synth.gauges(w).reshape(-1)).cuda()
    ref = cg.kivi_stream_alloc(cap, params)      # codes, scales, ring, workspace
    got = cg.kivi_stream_alloc(cap, params)[:3]  # no workspace
    # a prefill of 255 tokens (all still raw: n_q(255) = 0), identical for both streams
    pre = cg.Shape(L=w.L, B=w.B, H=w.H, T=255, d=w.d, t0=0, T_cap=T_cap)
    dx = torch.from_numpy(np.ascontiguousarray(x[..., :255, :]).reshape(-1).view(np.int16)).cuda()
    for bufs in (ref, got):
        cg.kivi_append(pre, params, dx, dG, *bufs[:3])
    # two appends in a row, each completing a key group: 255 -> 256 and 256 -> 384
    for t0, n in ((255, 1), (256, 128)):
        sh = cg.Shape(L=w.L, B=w.B, H=w.H, T=n, d=w.d, t0=t0, T_cap=T_cap)
        dn = torch.from_numpy(np.ascontiguousarray(x[..., t0:t0 + n, :]).reshape(-1).view(np.int16)).cuda()
        cg.kivi_append(sh, params, dn, dG, *ref)
        rc = lib.cg_kivi_append_static(ctypes.byref(sh.c()), ctypes.byref(params.c()), _p(dn), _p(dG),
                                       _p(got[0]), _p(got[1]), _p(got[2]), _stream())
        assert rc == 0, lib.cg_last_error().decode()
        assert cg.get_status() == 0
        for a, b in zip(ref[:3], got):
            assert torch.equal(a, b)
        T = t0 + n
        full = cg.Shape(L=w.L, B=w.B, H=w.H, T=T, d=w.d, t0=0, T_cap=T_cap)
        oa = torch.empty(w.L * 2 * w.B * w.H * T * w.d, dtype=torch.int16, device="cuda")
        ob = torch.empty_like(oa)
        cg.kivi_stream_decode(full, params, *ref[:3], dG, oa)
        cg.kivi_stream_decode(full, params, *got, dG, ob)
        assert cg.get_status() == 0
        assert torch.equal(oa, ob)


def test_static_append_rejects_shapes_beyond_the_array():
    lib = cg.load()
    lib.cg_kivi_append_static.restype = ctypes.c_int
    lib.cg_kivi_append_static.argtypes = [ctypes.c_void_p] * 8
    params = cg.Params(cg.CG_KIVI, 64, 3, 128, 128)
    # 600 units x 128 tokens x 128 channels x 2 bytes = 19.7 MB fits; 2048 units = 67 MB does not
    ok = cg.Shape(L=75, B=2, H=2, T=1, d=128, t0=4, T_cap=4096)
    big = cg.Shape(L=64, B=4, H=4, T=1, d=128, t0=4, T_cap=4096)
    assert cg.kivi_stream_bytes(ok, params)[3] <= 32 << 20 < cg.kivi_stream_bytes(big, params)[3]
    fake = ctypes.c_void_p(0x10000)
    rc = lib.cg_kivi_append_static(ctypes.byref(big.c()), ctypes.byref(params.c()), fake, fake, fake, fake, fake,
                                   None)
    assert rc == -4
    assert "static workspace" in lib.cg_last_error().decode()
