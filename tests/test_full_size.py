"""Full-size parity: the large cache workloads, encoded and decoded by whole-workload
calls (the launch configuration the benchmark times), checked against the oracle on sampled
(layer, batch, head) units, keys and values.

The oracle runs on one unit pair at a time: the unit's K and V tokens with the gauges of
its (layer, head), as a 1-layer, 1-sequence, 1-head cache.
"""
import numpy as np
import pytest

import oracle
from paper_2607_20538_gb300 import synth

from cgcheck import compare_codes, compare_decode, compare_scales, scales_as_elements

torch = pytest.importorskip("torch")
cg = pytest.importorskip("paper_2607_20538_gb300")

pytestmark = pytest.mark.gpu


def _units(w, n_random=4, seed=7):
    rng = np.random.default_rng(seed)
    u = {(0, 0, 0), (w.L - 1, w.B - 1, w.H - 1)}
    while len(u) < 2 + n_random:
        u.add((int(rng.integers(w.L)), int(rng.integers(w.B)), int(rng.integers(w.H))))
    return sorted(u)


def _sub_bu(t, w, T_cap, l, b, h, per_row):
    """Rows [0, w.T) of both s of unit (l, b, h) from a block-uniform buffer [L][2][B][H][T_cap][per_row]."""
    v = t.view(w.L, 2, w.B, w.H, T_cap, per_row)[l, :, b, h, : w.T]
    return v.contiguous().cpu().numpy().ravel()


def _sub_kivi(t, w, l, b, h, k_per, v_per):
    """Unit (l, b, h) of a KIVI buffer laid out per layer as keys [B][H][k_per], values [B][H][v_per]."""
    per_layer = w.B * w.H * (k_per + v_per)
    lay = t[l * per_layer:(l + 1) * per_layer]
    kk = lay[: w.B * w.H * k_per].view(w.B, w.H, k_per)[b, h]
    vv = lay[w.B * w.H * k_per:].view(w.B, w.H, v_per)[b, h]
    return torch.cat([kk, vv]).cpu().numpy()


def _check_unit(w, G, x_unit, l, h, codes_u8, scales_u16, resid_u16, out_u16):
    """Oracle on one unit pair [1][2][1][1][T][d] (gauges of layer l, head h) vs the GPU's bytes."""
    w1 = w.replace(L=1, B=1, H=1, T_cap=0)
    G1 = np.ascontiguousarray(G[l:l + 1, :, h:h + 1])
    ref = oracle.encode(w1.shape, w1.params, x_unit, G1, want_flags=True)
    mism = compare_codes(w1, codes_u8, ref["codes"], ref["flags"])
    compare_scales(scales_u16, ref["scales"])
    if ref["residual"].size:
        np.testing.assert_array_equal(resid_u16, ref["residual"])
    xr = oracle.decode(w1.shape, w1.params, ref["codes"], ref["scales"], ref["residual"], G1)
    step = scales_as_elements(w1, ref["scales"]) * mism if mism.any() else None
    st = compare_decode(w1, out_u16, xr, G1, step, codes=ref["codes"], scales_u16=ref["scales"])
    print(f"unit (l={l}, h={h}): {int(mism.sum())} flagged code mismatches of {mism.size}; decode checked "
          f"tightly on {st['tight']} values ({st['tight_not_rne']} not bf16(ref)); "
          f"{st['rms_floor_only']} pass only through the rms floor")


@pytest.fixture(autouse=True)
def _release_device_memory():
    """Each test holds up to ~180 GB; hand the cached blocks back around every test."""
    torch.cuda.empty_cache()
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


@pytest.mark.parametrize("name", ["llama3_8b", "gemma27b", "kivi3_qwen", "llama3_8b_tile"])
def test_full_size_sampled(name):
    w = synth.WORKLOADS[name]
    x = synth.kv_cache(w, threads=16)
    G = synth.gauges(w)
    shape, params = cg.Shape(**w.shape), cg.Params(**w.params)
    dx = torch.from_numpy(x.reshape(-1).view(np.int16)).cuda()
    dG = torch.from_numpy(G.reshape(-1)).cuda()
    codes, scales, resid = cg.alloc_outputs(shape, params)
    out = torch.empty_like(dx)
    cg.encode(shape, params, dx, dG, codes, scales, resid)
    cg.decode(shape, params, codes, scales, resid, dG, out)
    assert cg.get_status() == 0
    del dx
    c8 = codes.view(torch.uint8)
    s32 = scales.view(torch.int32)
    o16 = out.view(torch.int16)
    for (l, b, h) in _units(w):
        xu = np.ascontiguousarray(x[l:l + 1, :, b:b + 1, h:h + 1])
        ou = o16.view(w.L, 2, w.B, w.H, w.T, w.d)[l, :, b, h].contiguous().cpu().numpy().view(np.uint16).ravel()
        if w.backend in (0, 3):
            cu = _sub_bu(c8, w, w.T, l, b, h, w.d * w.bits // 8)
            if w.backend == 0:
                su = _sub_bu(s32, w, w.T, l, b, h, w.d // w.block).view(np.uint16)
            else:  # one pair per 16-token tile block
                nt = -(-w.T // oracle.TILE_TOKENS)
                su = s32.view(w.L, 2, w.B, w.H, nt, w.d // w.block)[l, :, b, h].contiguous().cpu().numpy()
                su = su.ravel().view(np.uint16)
            ru = np.zeros(0, np.uint16)
        else:
            nq = oracle.kivi_nq(w.T, w.residual, w.block)
            pay = w.block * w.bits // 8
            cu = _sub_kivi(c8, w, l, b, h, (nq // w.block) * w.d * pay, nq * (w.d // w.block) * pay)
            su = _sub_kivi(s32, w, l, b, h, (nq // w.block) * w.d, nq * (w.d // w.block)).view(np.uint16)
            ru = resid.view(torch.int16).view(w.L, 2, w.B, w.H, w.T - nq, w.d)[l, :, b, h]
            ru = ru.contiguous().cpu().numpy().view(np.uint16).ravel()
        _check_unit(w, G, xu, l, h, cu, su, ru, ou)


def test_rolling_full_size_step():
    """Rolling decode step at full size: a 16k-token history per sequence (batch 64, 32 layers),
    one appended token per sequence, then the whole history decoded in one call."""
    w = synth.WORKLOADS["rolling"]
    Tc = w.T_cap
    free, _ = torch.cuda.mem_get_info()
    need = w.L * 2 * w.B * w.H * Tc * w.d * (2 + 0.5 + 4 / w.block) + 8e9
    if free < need:
        pytest.skip(f"needs {need / 1e9:.0f} GB of device memory, {free / 1e9:.0f} GB free")
    G = synth.gauges(w)
    dG = torch.from_numpy(G.reshape(-1)).cuda()
    params = cg.Params(**w.params)
    hist1 = synth.rolling_history_layer(w, threads=16)          # [1][2][B][H][Tc-1][d]
    xnew = synth.rolling_new_token(w, threads=16)               # [L][2][B][H][1][d]
    full = cg.Shape(L=w.L, B=w.B, H=w.H, T=Tc, d=w.d, t0=0, T_cap=Tc)
    codes, scales, _ = cg.alloc_outputs(full, params)
    # history: layer by layer (L = 1 calls), tokens [0, Tc - 1)
    lay = cg.Shape(L=1, B=w.B, H=w.H, T=Tc - 1, d=w.d, t0=0, T_cap=Tc)
    nc1, ns1, _ = cg.packed_bytes(lay, params)
    dh = torch.from_numpy(hist1.reshape(-1).view(np.int16)).cuda()
    per_g = dG.numel() // w.L
    for l in range(w.L):
        cg.encode(lay, params, dh, dG[l * per_g:(l + 1) * per_g], codes[l * nc1:(l + 1) * nc1],
                  scales[l * ns1 // 4:(l + 1) * ns1 // 4], None)
    del dh
    # the step: append one token per sequence, decode the whole history
    app = cg.Shape(L=w.L, B=w.B, H=w.H, T=1, d=w.d, t0=Tc - 1, T_cap=Tc)
    cg.encode(app, params, torch.from_numpy(xnew.reshape(-1).view(np.int16)).cuda(), dG, codes, scales, None)
    out = torch.empty(w.L * 2 * w.B * w.H * Tc * w.d, dtype=torch.int16, device="cuda")
    cg.decode(full, params, codes, scales, None, dG, out)
    assert cg.get_status() == 0
    wu = w.replace(T=Tc)
    for (l, b, h) in _units(w):
        xu = np.concatenate([hist1[0:1, :, b:b + 1, h:h + 1], xnew[l:l + 1, :, b:b + 1, h:h + 1]], axis=4)
        cu = _sub_bu(codes.view(torch.uint8), wu, Tc, l, b, h, w.d * w.bits // 8)
        su = _sub_bu(scales.view(torch.int32), wu, Tc, l, b, h, w.d // w.block).view(np.uint16)
        ou = out.view(w.L, 2, w.B, w.H, Tc, w.d)[l, :, b, h].contiguous().cpu().numpy().view(np.uint16).ravel()
        _check_unit(wu, G, np.ascontiguousarray(xu), l, h, cu, su, np.zeros(0, np.uint16), ou)


def test_kivi_stream_full_size_step():
    """KIVI decode-loop step at full size (the benchmark's kivi3_stream): a 32k-token stream per
    sequence (28 layers, batch 4, 4 heads), one appended token that completes a key group, then
    the whole history decoded; sampled units against the batch oracle of all 32768 tokens."""
    from cgcheck import stream_to_batch
    w = synth.WORKLOADS["kivi3_stream"]
    Tc = w.T_cap
    G = synth.gauges(w)
    dG = torch.from_numpy(G.reshape(-1)).cuda()
    params = cg.Params(**w.params)
    hist1 = synth.rolling_history_layer(w, threads=16)          # [1][2][B][H][Tc-1][d]
    xnew = synth.rolling_new_token(w, threads=16)               # [L][2][B][H][1][d]
    full = cg.Shape(L=w.L, B=w.B, H=w.H, T=Tc, d=w.d, t0=0, T_cap=Tc)
    codes, scales, ring, work = cg.kivi_stream_alloc(full, params)
    lay = cg.Shape(L=1, B=w.B, H=w.H, T=Tc - 1, d=w.d, t0=0, T_cap=Tc)
    nc1, ns1, nr1, _ = cg.kivi_stream_bytes(lay, params)
    dh = torch.from_numpy(hist1.reshape(-1).view(np.int16)).cuda()
    per_g = dG.numel() // w.L
    for l in range(w.L):
        cg.kivi_append(lay, params, dh, dG[l * per_g:(l + 1) * per_g], codes[l * nc1:(l + 1) * nc1],
                       scales[l * ns1 // 4:(l + 1) * ns1 // 4], ring[l * nr1 // 2:(l + 1) * nr1 // 2])
    del dh
    app = cg.Shape(L=w.L, B=w.B, H=w.H, T=1, d=w.d, t0=Tc - 1, T_cap=Tc)
    cg.kivi_append(app, params, torch.from_numpy(xnew.reshape(-1).view(np.int16)).cuda(), dG, codes, scales, ring,
                   work)
    out = torch.empty(w.L * 2 * w.B * w.H * Tc * w.d, dtype=torch.int16, device="cuda")
    cg.kivi_stream_decode(full, params, codes, scales, ring, dG, out)
    assert cg.get_status() == 0
    # one unit's slices of the stream buffers, as a 1-layer, 1-sequence, 1-head stream
    w1 = w.replace(L=1, B=1, H=1, T=Tc, T_cap=Tc)
    Gt, pay = w.block, w.block * w.bits // 8
    ncap = oracle.kivi_nq(Tc, w.residual, Gt)
    kc, vc = (ncap // Gt) * w.d * pay, ncap * (w.d // Gt) * pay     # code bytes per (b, h)
    ks, vs = (ncap // Gt) * w.d, ncap * (w.d // Gt)                 # scale pairs (u32) per (b, h)
    c8, s32 = codes.view(torch.uint8), scales.view(torch.int32)
    BH = w.B * w.H
    W = w.residual + w.block
    for (l, b, h) in _units(w):
        bh = b * w.H + h
        lc, ls = c8[l * nc1:(l + 1) * nc1], s32[l * ns1 // 4:(l + 1) * ns1 // 4]
        cu = torch.cat([lc[bh * kc:(bh + 1) * kc], lc[BH * kc + bh * vc:BH * kc + (bh + 1) * vc]]).cpu().numpy()
        su = torch.cat([ls[bh * ks:(bh + 1) * ks], ls[BH * ks + bh * vs:BH * ks + (bh + 1) * vs]]).cpu().numpy()
        ru = ring.view(w.L, 2, w.B, w.H, W, w.d)[l, :, b, h].contiguous().cpu().numpy()
        c1, s1, r1 = stream_to_batch(w1, Tc, Tc, cu, su.view(np.uint16), ru.view(np.uint16))
        xu = np.concatenate([hist1[0:1, :, b:b + 1, h:h + 1], xnew[l:l + 1, :, b:b + 1, h:h + 1]], axis=4)
        ou = out.view(w.L, 2, w.B, w.H, Tc, w.d)[l, :, b, h].contiguous().cpu().numpy().view(np.uint16).ravel()
        _check_unit(w1.replace(T_cap=0), G, np.ascontiguousarray(xu), l, h, c1, s1, r1, ou)
