"""The bounded pipeline waits of the tensor-core kernels give up cleanly.

Every mbarrier wait in the tensor-core encode and decode kernels is bounded. When one runs
out, the kernel raises CG_FLAG_PIPE_TIMEOUT, drains the bulk copies and MMAs it has in
flight (those drains keep the normal 4 s limit), frees its tensor memory and returns.
CODECGAUGE_PIPE_WAIT_NS lowers the limit of the pipeline waits only; below 1 ms the waits
poll without suspending. A limit of 100 ns cannot be met (no stage of the pipeline completes
that fast: the first bulk copy alone waits on HBM), so the calls below must come back with
the flag and without any fault, and the next calls on the same stream, with the normal
limit, must match the oracle again.
"""
import os

import numpy as np
import pytest

import oracle
from paper_2607_20538_gb300 import synth

from cgcheck import compare_codes, compare_decode, compare_scales, scales_as_elements

torch = pytest.importorskip("torch")
cg = pytest.importorskip("paper_2607_20538_gb300")

pytestmark = pytest.mark.gpu

ENV = "CODECGAUGE_PIPE_WAIT_NS"


def _wl(**kw):
    base = dict(name="case", L=2, B=1, H=2, T=1024, d=128, group=128, backend=0, bits=4, block=64, residual=0)
    base.update(kw)
    return synth.Workload(**base)


# each case runs only tensor-core kernels (d = 128, at least 64 tokens per unit)
CASES = {
    "bu4_g128_blk64": _wl(),
    "bu6_g32_blk32": _wl(group=32, bits=6, block=32, B=2),
    "kivi3_g64": _wl(backend=1, group=64, bits=3, block=128, residual=128, T=1152),
}


@pytest.mark.parametrize("name", list(CASES))
def test_pipe_wait_limit(name, monkeypatch):
    w = CASES[name]
    x = synth.kv_cache(w, threads=4)
    G = synth.gauges(w)
    dx = torch.from_numpy(np.ascontiguousarray(x).reshape(-1).view(np.int16)).cuda()
    dG = torch.from_numpy(np.ascontiguousarray(G).reshape(-1)).cuda()
    shape, params = cg.Shape(**w.shape), cg.Params(**w.params)
    nc, ns, nr = cg.packed_bytes(shape, params)
    codes, scales, resid = cg.alloc_outputs(shape, params)
    out = torch.empty_like(dx)
    assert cg.get_status() == 0

    monkeypatch.setenv(ENV, "100")
    cg.encode(shape, params, dx, dG, codes, scales, resid)
    assert cg.get_status() & cg.CG_FLAG_PIPE_TIMEOUT
    cg.decode(shape, params, codes, scales, resid, dG, out)
    assert cg.get_status() & cg.CG_FLAG_PIPE_TIMEOUT

    monkeypatch.delenv(ENV)
    codes.zero_()
    scales.zero_()
    cg.encode(shape, params, dx, dG, codes, scales, resid)
    cg.decode(shape, params, codes, scales, resid, dG, out)
    assert cg.get_status() == 0
    ref = oracle.encode(w.shape, w.params, x, G, want_flags=True)
    mism = compare_codes(w, codes.cpu().numpy().view(np.uint8)[:nc], ref["codes"], ref["flags"])
    compare_scales(scales.cpu().numpy().view(np.uint16)[: ns // 2], ref["scales"])
    if nr:
        np.testing.assert_array_equal(resid.cpu().numpy().view(np.uint16)[: nr // 2], ref["residual"])
    xr = oracle.decode(w.shape, w.params, ref["codes"], ref["scales"], ref["residual"], G)
    got = out.cpu().numpy().view(np.uint16)[: xr.size]
    step = scales_as_elements(w, ref["scales"]) * mism if mism.any() else None
    compare_decode(w, got, xr, G, step, codes=ref["codes"], scales_u16=ref["scales"])


def test_pipe_wait_env_is_bounded(monkeypatch):
    """A limit above the default or a malformed value falls back to the 4 s default."""
    w = CASES["bu4_g128_blk64"]
    x = synth.kv_cache(w, threads=4)
    G = synth.gauges(w)
    dx = torch.from_numpy(np.ascontiguousarray(x).reshape(-1).view(np.int16)).cuda()
    dG = torch.from_numpy(np.ascontiguousarray(G).reshape(-1)).cuda()
    shape, params = cg.Shape(**w.shape), cg.Params(**w.params)
    codes, scales, resid = cg.alloc_outputs(shape, params)
    for v in ("junk", "99999999999999999999", "12x"):
        monkeypatch.setenv(ENV, v)
        cg.encode(shape, params, dx, dG, codes, scales, resid)
        assert cg.get_status() == 0
    monkeypatch.delenv(ENV)
    os.environ.pop(ENV, None)
