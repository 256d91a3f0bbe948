"""Benchmark: encode + decode of a KV cache through libcodecgauge on GB300.

One step = one pass of the hot path over the workload: cg_encode (gauge rotation, block
ranges, scales, codes, packing) then cg_decode (unpacking, dequantization, inverse gauge)
of the whole cache, with inputs resident in HBM (1 GiB of bf16 for the Llama-3-8B-shaped
cache, larger than the 129 MB L2, so no flush is needed between steps).

value  = (bf16 bytes encoded + bf16 bytes decoded) / (encode + decode time), GB/s
e2e    = the same through the C ABI with host buffers: pinned host -> device copy of the
         cache, encode, decode, device -> pinned host copy of the recovered cache.
roofline: the slower of the two kernels; algorithmic bytes per launch / its average
         CUDA-event duration, against the measured copy bandwidth.

workloads: with the default 8B-shaped workload the same process then times the other target
         workloads (27B-shaped 6-bit, KIVI-3, the rolling decode step) with fewer steps:
         device-timed encode/decode ms, GB/s and HBM fractions per kernel.
cpu_baseline: the oracle on the host cores (all of them, and one thread).

Multi-GPU (torchrun): every rank encodes/decodes its own cache of the same shape (the
units (l, s, b, h) are independent; no collective on the data path), weak scaling.
--impl reference times the CPU oracle on the host cores on a bounded sample.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "encode/decode KV GB/s (bf16 bytes) and % of HBM roofline at 1 GB300"
FALLBACK_HBM_GBS = 6800.0


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def rank_reduce(v: float, op: str, device=None) -> float:
    """Max or min of a per-rank scalar over the job (identity without a process group)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return v
    t = torch.tensor([v], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX if op == "max" else dist.ReduceOp.MIN)
    return float(t.item())


def job_throughput(bytes_per_rank_step: int, world: int, ms_per_step: float) -> float:
    """Whole-job GB/s: every rank processes its own shard of the same size (weak scaling)."""
    return world * bytes_per_rank_step / (ms_per_step * 1e-3) / 1e9


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, dev_index: int):
        self.dev = dev_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(prefix="cg_clocks_", suffix=".csv")
            os.close(fd)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.dev}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "20"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None

    def stop(self):
        if not self.proc:
            return None
        time.sleep(0.05)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            f = [v.strip() for v in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        try:
            os.remove(self.path)
        except OSError:
            pass
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def _kernel_traffic(kind: str, workload: str):
    """ncu DRAM bytes (read + write) per launch of the kernel on this workload, recorded in
    profiles/dram_traffic_<workload>.json, or None when there is no record or any source file
    of the kernel changed since the counters were taken."""
    p = os.path.join(ROOT, "profiles", f"dram_traffic_{workload}.json")
    try:
        rec = json.load(open(p))[kind]
        h = hashlib.sha256()
        for name in rec["sources"]:
            h.update(open(os.path.join(ROOT, "paper_2607_20538_gb300", "csrc", name), "rb").read())
    except Exception:
        return None
    return rec["bytes_per_launch"] if h.hexdigest()[:16] == rec["sources_sha"] else None


def cpu_sample(w, G, seconds=12.0, nthreads=None, start=0):
    """Time the oracle (as it stands) on whole (layer, sequence) slices of the workload: the K and
    V units of every head of one (l, b), one slice after the other from slice `start`, until
    `seconds` of oracle time have accumulated (at least one slice)."""
    import numpy as np

    import oracle
    from paper_2607_20538_gb300 import synth
    nthreads = nthreads or os.cpu_count() or 1
    sub = w.replace(L=1, B=1, T_cap=0)
    done_bytes, t_total, n = 0, 0.0, 0
    n_slices = w.L * w.B
    while n < n_slices:
        l, b = divmod((start + n) % n_slices, w.B)
        x = np.stack([np.stack([np.stack([synth.kv_unit(w, l, s, b, h) for h in range(w.H)])
                                for s in range(2)])])[:, :, None]
        Gl = np.ascontiguousarray(G[l:l + 1])
        t0 = time.perf_counter()
        r = oracle.encode(sub.shape, sub.params, x, Gl, nthreads=nthreads)
        oracle.decode(sub.shape, sub.params, r["codes"], r["scales"], r["residual"], Gl, nthreads=nthreads)
        t_total += time.perf_counter() - t0
        done_bytes += 2 * x.nbytes
        n += 1
        if t_total >= seconds:
            break
    return {"value": done_bytes / t_total / 1e9, "unit": "GB/s", "cores": nthreads, "kind": "oracle",
            "sample": f"encode+decode of {n} of {n_slices} (layer, sequence) slices of the {w.name} cache "
                      f"({n * 2 * w.H} (l,s,b,h) units, {done_bytes // 2} bf16 bytes), "
                      f"{t_total:.2f} s on {nthreads} threads"}


def workload_config(w, ws):
    """The `config` of a bench line for workload `w` on `ws` ranks (both arms print the same)."""
    config = {"workload": w.name, "L": w.L, "B": w.B, "H": w.H, "T": w.T, "d": w.d,
              "group": w.group, "backend": ["block-uniform", "kivi", "none", "block-uniform-tile"][w.backend],
              "bits": w.bits, "block": w.block, "residual": w.residual, "kv_dtype": "bf16",
              "parallelism": f"replicas{ws}", "l2": "inputs larger than L2 (no flush)",
              "value_def": "(bf16 bytes encoded + bf16 bytes decoded) / (encode+decode time)"}
    if w.T_cap:
        config.update({"T_cap": w.T_cap,
                       "step": "append 1 token per sequence at T_cap - 1, decode all T_cap tokens"})
    return config


def _workload(args):
    """The workload of --workload, cut to --layers and with the --shape overrides."""
    from paper_2607_20538_gb300 import synth
    w = synth.WORKLOADS[args.workload]
    if args.layers:
        w = w.replace(L=min(args.layers, w.L))
    if args.shape:
        w = w.replace(**{k: int(v) for k, v in (kv.split("=") for kv in args.shape.split(","))})
    return w


def run_reference(args):
    ws, rank, _ = _dist()
    if rank != 0:
        return
    from paper_2607_20538_gb300 import synth
    w = _workload(args)
    G = synth.gauges(w)
    cores = os.cpu_count() or 1
    for i in range(args.warmup):
        cpu_sample(w, G, seconds=0.0, nthreads=cores, start=i)
    vals = []
    t0 = time.perf_counter()
    for i in range(args.steps):
        # one step: a bounded sample (one or more (layer, sequence) slices, ~0.25 s)
        vals.append(cpu_sample(w, G, seconds=0.25, nthreads=cores, start=args.warmup + i))
    el = time.perf_counter() - t0
    v = statistics.median(x["value"] for x in vals)
    line = {"impl": "reference", "metric": METRIC, "value": round(v, 4), "unit": "GB/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(el / args.steps * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic", "config": workload_config(w, args.gpus),
            "cpu_baseline": {"value": round(v, 4), "unit": "GB/s", "cores": cores, "kind": "oracle",
                             "sample": vals[-1]["sample"]},
            "e2e": {"value": round(v, 4), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


class _Problem:
    """What one step runs and how its bytes count (set up by _setup_cache / _setup_rolling)."""


def _setup_cache(w, dev, ws, stream):
    """Whole-cache step: encode the workload's cache, then decode it."""
    import numpy as np
    import torch

    import paper_2607_20538_gb300 as cg
    from paper_2607_20538_gb300 import synth
    P = _Problem()
    shape, params = cg.Shape(**w.shape), cg.Params(**w.params)
    nc, ns, nr = cg.packed_bytes(shape, params)
    x = synth.kv_cache(w, threads=max(4, (os.cpu_count() or 8) // max(ws, 1)))
    hadamard = w.extra.get("gauge") == "hadamard"
    P.G = synth.gauges(w, "hadamard" if hadamard else "random")
    dx = torch.from_numpy(x.reshape(-1).view(np.int16)).to(dev)
    dG = torch.from_numpy(P.G.reshape(-1)).to(dev)
    codes, scales, resid = cg.alloc_outputs(shape, params, device=dev)
    out = torch.empty_like(dx)
    n = x.nbytes
    P.enc_bytes = P.dec_bytes = n
    P.enc_alg = P.dec_alg = n + nc + ns + nr + (0 if hadamard else P.G.nbytes)
    P.launches = 2 if w.backend != 1 else 2 * 3
    P.config = {"gauge": "hadamard by fast Walsh-Hadamard transform (no gauge tensor)"} if hadamard else {}

    if hadamard:
        def encode():
            cg.encode_hadamard(shape, params, dx, codes, scales, stream=stream)

        def decode():
            cg.decode_hadamard(shape, params, codes, scales, out, stream=stream)
    else:
        def encode():
            cg.encode(shape, params, dx, dG, codes, scales, resid, stream=stream)

        def decode():
            cg.decode(shape, params, codes, scales, resid, dG, out, stream=stream)

    P.encode, P.decode = encode, decode
    hx = torch.from_numpy(x.reshape(-1).view(np.int16)).pin_memory()
    hout = torch.empty_like(hx).pin_memory()

    # End to end, layers streamed through per-layer calls (the layout is layer-major, so a
    # layer's input, codes, scales, residual and gauges are contiguous): the host->device copy
    # of layer l+1 and the device->host copy of layer l-1 overlap the coding of layer l. Each
    # step starts after the previous one has finished.
    shape1 = cg.Shape(**{**w.shape, "L": 1})
    nc1, ns1, nr1 = cg.packed_bytes(shape1, params)
    px, pg = dx.numel() // w.L, dG.numel() // w.L
    aligned = all(v % 16 == 0 for v in (nc1, ns1, nr1, 2 * px, 4 * pg))
    s_in, s_out = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    ev_in = [torch.cuda.Event() for _ in range(w.L)]
    ev_done = [torch.cuda.Event() for _ in range(w.L)]

    def e2e_layers():
        s_in.wait_stream(stream)
        for l in range(w.L):
            xs, gs = slice(l * px, (l + 1) * px), slice(l * pg, (l + 1) * pg)
            with torch.cuda.stream(s_in):
                dx[xs].copy_(hx[xs], non_blocking=True)
                ev_in[l].record(s_in)
            stream.wait_event(ev_in[l])
            c1 = codes[l * nc1:(l + 1) * nc1]
            sc1 = scales[l * (ns1 // 4):(l + 1) * (ns1 // 4)]
            r1 = resid[l * (nr1 // 2):(l + 1) * (nr1 // 2)] if nr1 else None
            if hadamard:
                cg.encode_hadamard(shape1, params, dx[xs], c1, sc1, stream=stream)
                cg.decode_hadamard(shape1, params, c1, sc1, out[xs], stream=stream)
            else:
                cg.encode(shape1, params, dx[xs], dG[gs], c1, sc1, r1, stream=stream)
                cg.decode(shape1, params, c1, sc1, r1, dG[gs], out[xs], stream=stream)
            ev_done[l].record(stream)
            s_out.wait_event(ev_done[l])
            with torch.cuda.stream(s_out):
                hout[xs].copy_(out[xs], non_blocking=True)
        stream.wait_stream(s_out)

    def e2e_whole():
        dx.copy_(hx, non_blocking=True)
        encode()
        decode()
        hout.copy_(out, non_blocking=True)

    e2e_step = e2e_layers if (aligned and w.L > 1) else e2e_whole
    P.e2e_step, P.h2d, P.d2h = e2e_step, n, n
    P.e2e_bytes = 2 * n
    return P


def _setup_rolling(w, dev, ws, stream):
    """Rolling decode step over a history of T_cap tokens per sequence: encode one new token per
    sequence into position T_cap - 1, then decode the whole history. The history is encoded once
    before timing (layer by layer; every layer holds one draw of layer 0's tokens, see synth)."""
    import numpy as np
    import torch

    import paper_2607_20538_gb300 as cg
    from paper_2607_20538_gb300 import synth
    P = _Problem()
    Tc = w.T_cap
    params = cg.Params(**w.params)
    full = cg.Shape(L=w.L, B=w.B, H=w.H, T=Tc, d=w.d, t0=0, T_cap=Tc)
    app = cg.Shape(L=w.L, B=w.B, H=w.H, T=1, d=w.d, t0=Tc - 1, T_cap=Tc)
    lay = cg.Shape(L=1, B=w.B, H=w.H, T=Tc - 1, d=w.d, t0=0, T_cap=Tc)
    nc, ns, _ = cg.packed_bytes(full, params)
    nc1, ns1, _ = cg.packed_bytes(lay, params)
    P.G = synth.gauges(w)
    dG = torch.from_numpy(P.G.reshape(-1)).to(dev)
    codes, scales, _ = cg.alloc_outputs(full, params, device=dev)
    threads = max(4, (os.cpu_count() or 8) // max(ws, 1))
    dh = torch.from_numpy(synth.rolling_history_layer(w, threads=threads).reshape(-1).view(np.int16)).to(dev)
    per_g = dG.numel() // w.L
    for l in range(w.L):
        cg.encode(lay, params, dh, dG[l * per_g:(l + 1) * per_g], codes[l * nc1:(l + 1) * nc1],
                  scales[l * ns1 // 4:(l + 1) * ns1 // 4], None, stream=stream)
    del dh
    xnew = synth.rolling_new_token(w, threads=threads)
    dnew = torch.from_numpy(xnew.reshape(-1).view(np.int16)).to(dev)
    n_out = w.L * 2 * w.B * w.H * Tc * w.d
    out = torch.empty(n_out, dtype=torch.int16, device=dev)
    P.enc_bytes, P.dec_bytes = xnew.nbytes, 2 * n_out
    tok_codes = w.L * 2 * w.B * w.H * (w.d * w.bits // 8)
    tok_scales = w.L * 2 * w.B * w.H * (w.d // w.block) * 4
    P.enc_alg = xnew.nbytes + tok_codes + tok_scales + P.G.nbytes
    P.dec_alg = nc + ns + P.G.nbytes + 2 * n_out
    P.launches = 2
    P.config = {"T_cap": Tc, "step": "append 1 token per sequence at T_cap - 1, decode all T_cap tokens"}
    n_rep = w.extra.get("n_rep", 0)
    if n_rep:
        # the step's second half is attention of one query per sequence over the whole history,
        # read straight from the codes (no bf16 cache written)
        del out
        nq = w.L * w.B * w.H * n_rep * w.d
        dq = torch.from_numpy(synth.f32_to_bf16_bits(
            np.random.default_rng(w.kv_seed + 900).normal(0.0, 1.0, nq).astype(np.float32)).view(np.int16)).to(dev)
        out = torch.empty(nq, dtype=torch.float32, device=dev)
        work = torch.empty(cg.attention_workspace_bytes(full, params, n_rep), dtype=torch.uint8, device=dev)
        P.dec_bytes = 2 * n_out  # bf16 bytes of the cache the attention reads through its codes
        P.dec_alg = nc + ns + P.G.nbytes + dq.numel() * 2 + nq * 4
        P.launches = 1 + 3
        P.config = {"T_cap": Tc, "n_rep": n_rep,
                    "step": "append 1 token per sequence at T_cap - 1, then attention of 1 query per sequence "
                            f"({n_rep} query heads per KV head) over all T_cap tokens, from the codes"}
        scale = 1.0 / float(np.sqrt(w.d))

        def decode():
            cg.attention(full, params, n_rep, scale, dq, codes, scales, dG, out, work, stream=stream)

        last = out
    else:
        def decode():
            cg.decode(full, params, codes, scales, None, dG, out, stream=stream)

        last = out.view(w.L * 2 * w.B * w.H, Tc, w.d)[:, Tc - 1, :]

    def encode():
        cg.encode(app, params, dnew, dG, codes, scales, None, stream=stream)

    P.encode, P.decode = encode, decode
    hnew = torch.from_numpy(xnew.reshape(-1).view(np.int16)).pin_memory()
    hlast = torch.empty(last.shape, dtype=last.dtype).pin_memory()

    def e2e_step():
        # the new tokens in, the step, and the decoded newest token (or the attention output) out
        dnew.copy_(hnew, non_blocking=True)
        encode()
        decode()
        hlast.copy_(last, non_blocking=True)

    P.e2e_step, P.h2d, P.d2h = e2e_step, hnew.numel() * 2, hlast.numel() * hlast.element_size()
    P.e2e_bytes = P.enc_bytes + P.dec_bytes
    return P


def _setup_kivi_stream(w, dev, ws, stream):
    """KIVI decode-loop step over a stream of capacity T_cap holding T_cap - 1 tokens: append one
    token per sequence at T_cap - 1 (it completes a key group, so the step also stages and
    quantizes that group's 128 keys and values), then decode all T_cap tokens. The history is
    prefilled once before timing, layer by layer (every layer holds one draw of layer 0's tokens).
    Re-running the step rewrites the same bytes: the staged tokens come from ring slots that the
    step does not write."""
    import numpy as np
    import torch

    import paper_2607_20538_gb300 as cg
    from paper_2607_20538_gb300 import synth
    P = _Problem()
    Tc = w.T_cap
    params = cg.Params(**w.params)
    full = cg.Shape(L=w.L, B=w.B, H=w.H, T=Tc, d=w.d, t0=0, T_cap=Tc)
    app = cg.Shape(L=w.L, B=w.B, H=w.H, T=1, d=w.d, t0=Tc - 1, T_cap=Tc)
    lay = cg.Shape(L=1, B=w.B, H=w.H, T=Tc - 1, d=w.d, t0=0, T_cap=Tc)
    nc, ns, nr, nw = cg.kivi_stream_bytes(full, params)
    nc1, ns1, nr1, _ = cg.kivi_stream_bytes(lay, params)
    P.G = synth.gauges(w)
    dG = torch.from_numpy(P.G.reshape(-1)).to(dev)
    codes, scales, ring, work = cg.kivi_stream_alloc(full, params, device=dev)
    threads = max(4, (os.cpu_count() or 8) // max(ws, 1))
    dh = torch.from_numpy(synth.rolling_history_layer(w, threads=threads).reshape(-1).view(np.int16)).to(dev)
    per_g = dG.numel() // w.L
    for l in range(w.L):
        cg.kivi_append(lay, params, dh, dG[l * per_g:(l + 1) * per_g], codes[l * nc1:(l + 1) * nc1],
                       scales[l * ns1 // 4:(l + 1) * ns1 // 4], ring[l * nr1 // 2:(l + 1) * nr1 // 2], None,
                       stream=stream)
    del dh
    xnew = synth.rolling_new_token(w, threads=threads)
    dnew = torch.from_numpy(xnew.reshape(-1).view(np.int16)).to(dev)
    n_out = w.L * 2 * w.B * w.H * Tc * w.d
    out = torch.empty(n_out, dtype=torch.int16, device=dev)
    Gt, units = w.block, w.L * 2 * w.B * w.H
    P.enc_bytes, P.dec_bytes = xnew.nbytes, 2 * n_out
    grp_codes = units * Gt * w.d * w.bits // 8
    grp_scales = w.L * w.B * w.H * (w.d + Gt * (w.d // Gt)) * 4
    # staging: the group's tokens read from the ring and written to the workspace, read again
    # by the quantizers; the new token in and into the ring
    P.enc_alg = 2 * xnew.nbytes + 3 * units * Gt * w.d * 2 + grp_codes + grp_scales + P.G.nbytes
    nq = (Tc - w.residual) // Gt * Gt
    P.dec_alg = nc + ns + units * (Tc - nq) * w.d * 2 + P.G.nbytes + 2 * n_out
    P.launches = 4 + 3
    P.config = {"T_cap": Tc, "step": "KIVI stream: append 1 token per sequence at T_cap - 1 (completes a key "
                                     "group), decode all T_cap tokens"}

    def encode():
        cg.kivi_append(app, params, dnew, dG, codes, scales, ring, work, stream=stream)

    def decode():
        cg.kivi_stream_decode(full, params, codes, scales, ring, dG, out, stream=stream)

    P.encode, P.decode = encode, decode
    hnew = torch.from_numpy(xnew.reshape(-1).view(np.int16)).pin_memory()
    last = out.view(units, Tc, w.d)[:, Tc - 1, :]
    hlast = torch.empty(last.shape, dtype=torch.int16).pin_memory()

    def e2e_step():
        dnew.copy_(hnew, non_blocking=True)
        encode()
        decode()
        hlast.copy_(last, non_blocking=True)

    P.e2e_step, P.h2d, P.d2h = e2e_step, hnew.numel() * 2, hlast.numel() * 2
    P.e2e_bytes = P.enc_bytes + P.dec_bytes
    return P


def _setup(w, dev, ws, stream):
    if w.T_cap:
        return (_setup_kivi_stream if w.backend == 1 else _setup_rolling)(w, dev, ws, stream)
    return _setup_cache(w, dev, ws, stream)


def _time_problem(P, stream, steps: int, warmup: int, dev, ws: int, clock_dev: int):
    """Warm-up, then `steps` timed steps of problem P on `stream` (CUDA events per kernel and
    around the whole region, nvidia-smi clocks sampled during it)."""
    import torch

    import paper_2607_20538_gb300 as cg

    def step(ev=None):
        if ev is not None:
            ev[0].record(stream)
        P.encode()
        if ev is not None:
            ev[1].record(stream)
        P.decode()
        if ev is not None:
            ev[2].record(stream)

    for _ in range(warmup):
        step()
    torch.cuda.synchronize()
    flags = cg.get_status()
    if flags:
        raise RuntimeError(f"device status flags {flags} after warm-up")
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    clocks = Clocks(clock_dev)
    clocks.start()
    if ws > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for i in range(steps):
        step(evs[i])
    t_end.record(stream)
    torch.cuda.synchronize()
    if ws > 1:
        torch.distributed.barrier()
    clk = clocks.stop()
    flags = cg.get_status()
    if flags:
        raise RuntimeError(f"device status flags {flags} after the timed region")
    total_ms = rank_reduce(t_start.elapsed_time(t_end), "max", dev)
    return {"ms_step": total_ms / steps,
            "enc_ms": statistics.mean(e[0].elapsed_time(e[1]) for e in evs),
            "dec_ms": statistics.mean(e[1].elapsed_time(e[2]) for e in evs),
            "clocks": clk}


def _kernel_figures(P, t, peak):
    return {"encode_ms": round(t["enc_ms"], 5), "decode_ms": round(t["dec_ms"], 5),
            "encode_gbs": round(P.enc_bytes / (t["enc_ms"] * 1e-3) / 1e9, 2),
            "decode_gbs": round(P.dec_bytes / (t["dec_ms"] * 1e-3) / 1e9, 2),
            "enc_frac": round(P.enc_alg / (t["enc_ms"] * 1e-3) / 1e9 / peak, 4),
            "dec_frac": round(P.dec_alg / (t["dec_ms"] * 1e-3) / 1e9 / peak, 4),
            "enc_alg_bytes": P.enc_alg, "dec_alg_bytes": P.dec_alg}


# Context only: the paper prints no encode/decode throughput; these are its own figures for
# the storage/timing side of the method and the hardware it states.
PAPER_CONTEXT = {
    "hardware": "NVIDIA RTX PRO 6000 Blackwell (CC 12.0, 97,887 MiB), AMD Ryzen 9 9950X, CUDA 13.2, PyTorch 2.12.1",
    "throughput": "not reported (the serial storage/timing run is shown as a normalized figure only)",
    "zfp4_actual_bits_per_value": 4.0,
    "zfp_rate_accuracy_bits_per_value": 6e-5,
    "inverse_gauge_round_trip_nrmse": "< 5.1e-8 (identity clone: 0)",
    "kl_reduction_learned_gauge": {"block_uniform": "44.2% (18/18 pairs)", "kivi": "27.2% (18/18 pairs)"},
}

# The other target workloads, timed in the same process after the headline one.
EXTRA_WORKLOADS = ("gemma27b", "kivi3_qwen", "rolling", "rolling_attn", "kivi3_stream", "llama3_8b_tile",
                   "llama3_8b_hadamard")


def run_cuda(args):
    import gc

    import torch

    from paper_2607_20538_gb300 import synth

    ws, rank, local = _dist()
    if ws > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    dev = torch.cuda.current_device()
    clock_dev = dev if ws == 1 else local
    w = _workload(args)
    stream = torch.cuda.current_stream()
    P = _setup(w, dev, ws, stream)
    t = _time_problem(P, stream, args.steps, args.warmup, dev, ws, clock_dev)
    ms_step = t["ms_step"]
    value = job_throughput(P.enc_bytes + P.dec_bytes, ws, ms_step)
    enc_avg, dec_avg = t["enc_ms"], t["dec_ms"]
    peak, peak_kind = _peaks()
    if dec_avg >= enc_avg:
        dom, dom_ms, dom_alg = "decode", dec_avg, P.dec_alg
    else:
        dom, dom_ms, dom_alg = "encode", enc_avg, P.enc_alg
    achieved = dom_alg / (dom_ms * 1e-3) / 1e9

    # end to end through the C ABI with host buffers
    e2e_steps = max(3, min(args.steps, 20))
    for _ in range(2):
        P.e2e_step()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(e2e_steps):
        P.e2e_step()
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = rank_reduce(e0.elapsed_time(e1) / e2e_steps, "max", dev)
    e2e_val = job_throughput(P.e2e_bytes, ws, e2e_ms)
    import paper_2607_20538_gb300 as cg
    flags = cg.get_status()
    if flags:
        raise RuntimeError(f"device status flags {flags} after the end-to-end steps")

    line = None
    if rank == 0:
        config = workload_config(w, ws)
        config.update(P.config)
        line = {
            "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(ms_step, 5), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic", "config": config,
            "encode_gbs": round(P.enc_bytes / (enc_avg * 1e-3) / 1e9, 2),
            "decode_gbs": round(P.dec_bytes / (dec_avg * 1e-3) / 1e9, 2),
            "encode_ms": round(enc_avg, 5), "decode_ms": round(dec_avg, 5),
            "steps_per_s": round(1e3 / ms_step, 3),
            "roofline": {"bound": "hbm", "kernel": dom, "achieved": round(achieved, 2), "peak": peak,
                         "peak_kind": peak_kind, "unit": "GB/s", "frac": round(achieved / peak, 4),
                         "traffic": None if (args.layers or args.shape) else _kernel_traffic(dom, w.name),
                         "alg_bytes_per_launch": dom_alg,
                         "enc_frac": round(P.enc_alg / (enc_avg * 1e-3) / 1e9 / peak, 4),
                         "dec_frac": round(P.dec_alg / (dec_avg * 1e-3) / 1e9 / peak, 4)},
            "e2e": {"value": round(e2e_val, 2), "unit": "GB/s", "h2d_bytes_per_step": P.h2d,
                    "d2h_bytes_per_step": P.d2h},
            "gpu_launches": P.launches * args.steps,
            "clocks": t["clocks"],
            "paper_context": PAPER_CONTEXT,
        }
    G_main = P.G
    del P
    gc.collect()
    torch.cuda.empty_cache()

    # the other target workloads, device-timed in the same process (fewer steps)
    extra = {}
    if not args.layers and not args.shape and not args.no_extra and args.workload == "llama3_8b":
        for name in EXTRA_WORKLOADS:
            we = synth.WORKLOADS[name]
            Pe = _setup(we, dev, ws, stream)
            te = _time_problem(Pe, stream, args.extra_steps, 3, dev, ws, clock_dev)
            fig = _kernel_figures(Pe, te, peak)
            fig["steps"] = args.extra_steps
            fig["ms_per_step"] = round(te["ms_step"], 5)
            fig["value_gbs"] = round(job_throughput(Pe.enc_bytes + Pe.dec_bytes, ws, te["ms_step"]), 2)
            if we.T_cap:
                fig["steps_per_s"] = round(1e3 / te["ms_step"], 3)
            fig["config"] = {**workload_config(we, ws), **Pe.config}
            fig["gpu_launches_per_step"] = Pe.launches
            fig["clocks"] = te["clocks"]
            extra[name] = fig
            del Pe
            gc.collect()
            torch.cuda.empty_cache()

    if rank == 0:
        if extra:
            line["workloads"] = extra
        if not args.no_cpu_baseline:
            line["cpu_baseline"] = cpu_sample(w, G_main, seconds=args.cpu_seconds)
            one = cpu_sample(w, G_main, seconds=args.cpu_seconds_1t, nthreads=1)
            line["cpu_baseline"]["one_thread"] = {"value": one["value"], "unit": one["unit"], "cores": 1,
                                                  "sample": one["sample"]}
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="cuda", choices=["cuda", "reference"])
    ap.add_argument("--workload", default="llama3_8b")
    ap.add_argument("--layers", type=int, default=0,
                    help="keep only the first N layers of the workload (small cases for profiling)")
    ap.add_argument("--shape", default="",
                    help="profiling slices: comma-separated workload overrides, e.g. L=1,d=256,T=32768")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--cpu-seconds-1t", type=float, default=4.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extra", action="store_true",
                    help="time only --workload (by default the 8B-shaped headline run also times the other targets)")
    ap.add_argument("--extra-steps", type=int, default=10)
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_cuda(args)


if __name__ == "__main__":
    main()
