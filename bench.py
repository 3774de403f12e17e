#!/usr/bin/env python
"""Throughput of the AWSRC hot path on GB300.

One step = one pass of the whole path over one synthetic Qwen2.5-3B-shaped
layer (7 modules, 77,070,336 BF16 weights, 1,204,224 tiles of C = 64):
seed search over S = 4096 seeds (P = 4 atoms, INT4 codes, power-of-two scale),
AWSRC-U selection at 0.162 bits/weight with the stream written, and a dense
decode-apply of every module. Inputs are resident in HBM (308 MB of W and W0,
larger than the 129 MB L2) when the timed region starts.

Reported: (tile, seed) candidates/s for the whole step (`value`), layers/s,
decode-apply GB/s, the search kernel against the pipe its contraction runs on
(`roofline`: the method's 2*C*P flop of correlation per candidate against the
measured dense bf16 tensor peak, fp16 having the same rate; the FP32 epilogue,
the executed tensor work and the DRAM traffic beside it), the end-to-end
figure through the public API with host buffers (`e2e`), the whole
Qwen2.5-3B, Qwen2.5-7B (AWSRC-P_F) and Qwen2.5-32B (AWSRC-U and AWSRC-P_F)
synthetic models (`model_stack`, `full_models`), and the CPU oracle on a
bounded sample (`cpu_baseline`). `--impl reference` times the oracle alone
(the baseline arm). Under torchrun each rank encodes its own layer (weak
scaling, no collective on the data path).
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

WORKLOAD = "qwen2.5-3b_layer"
RATE = 0.162
METRIC = "AWSRC encode (tile,seed) candidates/s + layers/s; decode-apply HBM GB/s"
UNIT = "candidates/s"
# The method's own work per (tile, seed) candidate of the C = 64, P = 4 search:
# the correlation b = B_s^T (D r) of Eq. 3, C*P multiply-adds = 2*C*P flop. It
# is a dense contraction (128 tiles x 64 inputs by 64 inputs x 4 atoms per
# seed) and runs on the tensor cores, so it is the roofline's work, against
# the dense fp16/bf16 tensor peak.
METHOD_FLOP_PER_CANDIDATE = 2 * 64 * 4
# What the kernel executes on the tensor cores: the exact fixed-point
# correlation takes two fp16 halves of Y, so twice the method's flop.
TENSOR_FLOP_PER_CANDIDATE = 2 * METHOD_FLOP_PER_CANDIDATE
# FP32-pipe operations every candidate needs before it can be pruned: forming
# the rounded correlation from its two halves (1 per atom), the forward
# substitution (6), z * (D^-1 m) (4) and the bound z^T (z D^-1 m) (4). The ~0.5%
# of candidates that survive the bound add about 50 more each, not counted.
OPS_PER_CANDIDATE = 4 + 6 + 4 + 4
# Bytes the search must move per launch at the least: W and W0 of the layer
# (BF16, read once) and the 16-byte candidates written.
def search_algorithmic_bytes(weights: int, tiles: int) -> int:
    return 4 * weights + 16 * tiles
# DRAM traffic (read + write) of one full-layer search launch, from an ncu launch
# list of this workload; valid only for the kernel source it was measured on.
SEARCH_TRAFFIC = {"source_sha256": "1ec4496c84e47a59c8b2fdba2e99964251f41e20adbb67b77e1e7ad911cb1316",
                  "bytes_per_launch": 443022848 + 16460032,
                  # the same kernel's pipe utilisation in an ncu --set full capture (gate + up)
                  "ncu_fma_pipe_pct": 40.23, "ncu_issue_active_pct": 48.50,
                  "ncu_tensor_pipe_pct": 24.69}


def search_source_sha() -> str:
    """SHA-256 of the search kernel's source and the headers it includes, with
    comments and blank lines removed: the committed DRAM traffic and ncu
    figures hold only for that exact code."""
    import re
    h = hashlib.sha256()
    for f in ("search_c64p4.cu", "tc05.cuh", "common.cuh", "internal.h"):
        src = open(os.path.join(ROOT, "paper_2608_23144_gb300", "csrc", f)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        src = "\n".join(l.split("//")[0].rstrip() for l in src.splitlines())
        h.update("\n".join(l for l in src.splitlines() if l.strip()).encode())
    return h.hexdigest()


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--cpu-seconds", type=float, default=15.0,
                    help="target CPU time of the oracle baseline sample")
    ap.add_argument("--ref-step-seconds", type=float, default=4.0,
                    help="target CPU time of one step of the reference (oracle) arm")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-pf", action="store_true", help="skip the P_F encode measurement")
    ap.add_argument("--no-full-models", action="store_true",
                    help="skip the whole 28-layer Qwen2.5-7B (P_F) and 64-layer Qwen2.5-32B (U and P_F) "
                         "synthetic models (encode, select, decode; about a minute of GPU time)")
    ap.add_argument("--no-model", action="store_true",
                    help="skip the whole 36-layer Qwen2.5-3B stack (encode, select, decode)")
    ap.add_argument("--modules", default="",
                    help="comma-separated subset of the layer's modules (profiling runs only)")
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(x: float, device=None) -> float:
    """Largest value of x over all ranks (the job's time is its slowest rank's)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device if device is not None else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(units_per_rank_step: int, world: int, steps: int, seconds_max: float) -> float:
    """Whole-job throughput: units every rank processed / the slowest rank's time."""
    return world * units_per_rank_step * steps / seconds_max


def rank_layer(rank: int) -> int:
    """Weak scaling: rank r encodes layer r of the stack (its own synthetic draw)."""
    return rank


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            return json.load(f), "measured"
    return {"hbm_gbs": 6800.0, "sm_max_mhz": 2070.0}, "fallback"


# ------------------------------------------------------------------ clocks --
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200"]
        if self.gpu_id:
            cmd += ["-i", self.gpu_id]
        try:
            self.proc = subprocess.Popen(cmd, stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        rows = []
        if self.path and os.path.exists(self.path):
            for line in open(self.path):
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
            os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
        pw = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows), "power_w_max": max(pw) if pw else None}


def gpu_id_for(dev) -> str:
    import torch
    try:
        p = torch.cuda.get_device_properties(dev)
        return "%08X:%02X:%02X.0" % (p.pci_domain_id, p.pci_bus_id, p.pci_device_id)
    except Exception:
        vis = os.environ.get("CUDA_VISIBLE_DEVICES", "")
        return vis.split(",")[dev.index or 0] if vis else str(dev.index or 0)


# ----------------------------------------------------------- cpu baseline --
def oracle_sample(wl, mods_host, target_s: float, seed: int = 0):
    """Time the oracle (as it stands, all host cores) on whole rows sampled from
    every module of the layer; returns (candidates/s, cores, description)."""
    import numpy as np
    from oracle import oracle as orc
    oprm = orc.params(C=wl.C, P=wl.P, b=wl.b, S=wl.S)
    masks = orc.basis_masks(oprm)
    rng = np.random.default_rng(seed)

    def run(rows_per_module):
        n = 0
        t0 = time.perf_counter()
        for m in mods_host:
            rows = rng.choice(m["W"].shape[0], rows_per_module, replace=False)
            orc.encode_tiles(oprm, m["W"][rows], m["W0"][rows], m["act"], masks=masks)
            n += rows_per_module * m["W"].shape[1] // wl.C
        return n, time.perf_counter() - t0

    n1, t1 = run(1)                       # calibration: one row of every module
    per_tile = t1 / n1
    rows = max(1, int(target_s / (per_tile * sum(m["W"].shape[1] // wl.C for m in mods_host))))
    n, t = run(rows)
    cands = n * wl.S
    desc = (f"{rows} random whole rows of each of the {len(mods_host)} modules ({n} tiles x {wl.S} seeds = "
            f"{cands:,} candidates) in {t:.1f} s")
    return cands / t, orc.num_threads(), desc


def host_modules(mods):
    return [{"W": m["W"].float().cpu().numpy(), "W0": m["W0"].float().cpu().numpy(),
             "act": m["act"].cpu().numpy()} for m in mods]


# ------------------------------------------------------------- reference --
def paper_points(dev, hbm_gbs):
    """The paper's own operating points (Sec. 4) on the three MLP projections of
    one Qwen2.5-3B-shaped layer (gate/up 11008x2048, down 2048x11008, BF16):
    AWSRC-U at (C, P, b, S) = (128, 2, 4, 2) and AWSRC-P_F at (16, 4, 4, 16) with
    the 0.25/0.75 activation/Fisher blend. Encode, select (0.162 bpw) and dense
    decode, each timed on the device (mean of 3 runs after one warm-up)."""
    import torch
    import paper_2608_23144_gb300 as aw
    from synth.workloads import make_module, module_seed
    shapes = [(11008, 2048), (11008, 2048), (2048, 11008)]
    out = {}
    for name, kw, fisher, blend in [
            ("U_c128_p2_s2", dict(C=128, P=2, b=4, S=2), False, (1.0, 0.0)),
            ("PF_c16_p4_s16", dict(C=16, P=4, b=4, S=16, variant=1), True, (0.25, 0.75))]:
        mods = [make_module(r, c, seed=module_seed(0, 0, 4 + i), device=dev, fisher=fisher, blend=blend)
                for i, (r, c) in enumerate(shapes)]
        prm = aw.params(**kw)
        N = sum(r * c for r, c in shapes)
        T = N // kw["C"]
        cands = aw.awsrc_encode_tiles(prm, mods)
        ws = cands._awsrc_workspace
        stream, counts, nbytes = aw.awsrc_select_records(prm, mods, cands, [0.162])
        outs = aw.awsrc_decode_apply(prm, mods, stream, -1)
        torch.cuda.synchronize()
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        reps = 3
        ev[0].record()
        for _ in range(reps):
            aw.awsrc_encode_tiles(prm, mods, out=cands, workspace=ws)
        ev[1].record()
        for _ in range(reps):
            aw.awsrc_select_records(prm, mods, cands, [0.162])
        ev[2].record()
        for _ in range(reps):
            aw.awsrc_decode_apply(prm, mods, stream, -1, outs=outs)
        ev[3].record()
        torch.cuda.synchronize()
        assert aw.awsrc_workspace_status(ws) == 0, "encoder self-check fault"
        enc, sel, dec = (ev[i].elapsed_time(ev[i + 1]) / reps for i in range(3))
        read = N * (2 + 2 + (4 if fisher else 0))  # W, W0 (BF16) and the Fisher diagonal
        out[name] = {"params": kw, "blend": list(blend), "tiles": T, "records": int(counts.sum().item()),
                     "encode_ms": enc, "candidates_per_s": T * kw["S"] / (enc * 1e-3),
                     "encode_read_gbs": read / (enc * 1e-3) / 1e9,
                     "encode_frac_of_hbm": read / (enc * 1e-3) / 1e9 / hbm_gbs,
                     "select_ms": sel, "decode_ms": dec,
                     "decode_gbs": N * 4 / (dec * 1e-3) / 1e9}
        del mods, cands, ws, stream, outs
    out["workload"] = ("gate/up/down projections of one Qwen2.5-3B-shaped layer (67,633,152 BF16 weights); "
                       "the paper's (C,P,b,S) points, 0.162 bpw")
    return out


def backbone_and_serving(dev, prm, mods, outs, stream, records, hbm_gbs):
    """The RTN-INT4 backbone with scale double quantisation (Sec. 3.3) and the
    sidecar applied inside an INT4 GEMV (the packed inference of Sec. 5) on the
    benchmark layer, against the HBM copy ceiling. The seven calls of each (or
    the one batched call) are captured in a CUDA graph and the graph replayed
    (mean of 10 replays after one warm-up), so the device time is measured,
    not the Python marshalling of each call. Algorithmic bytes: the backbone reads W (2 B/weight) and
    writes the 4-bit codes, the SDQ scale codes and constants and W0 (BF16);
    the GEMV (one vector) reads the codes, the SDQ scale codes and constants,
    the prepared sidecar's tile map (8 B per tile), record slots (16 B per
    record) and nibble tables, x and writes y; it is timed as seven calls and
    as one batched call. cuBLAS's BF16 GEMV of the decoded weights (2 B/weight)
    is timed the same way for context."""
    import torch
    import paper_2608_23144_gb300 as aw
    reps = 10
    N = sum(m["rows"] * m["cols"] for m in mods)
    G = N // 128
    T = N // prm.C
    shapes = [(m["rows"], m["cols"]) for m in mods]
    bb = [aw.awsrc_rtn_quantize(m["W"], sdq=True) for m in mods]
    side = aw.awsrc_sidecar_prepare(prm, shapes, stream)
    xs = [torch.randn(1, m["cols"], device=dev, dtype=torch.float32) for m in mods]
    ys = [torch.empty(1, m["rows"], device=dev, dtype=torch.float32) for m in mods]
    xb = [x.to(torch.bfloat16) for x in xs]
    yb = [torch.empty(1, m["rows"], device=dev, dtype=torch.bfloat16) for m in mods]

    def quantise():
        for m, b in zip(mods, bb):
            aw.awsrc_rtn_quantize(m["W"], sdq=True, out=b)

    Wl = [m["W"] for m in mods]

    def quantise_batch():
        aw.awsrc_rtn_quantize_batch(Wl, sdq=True, outs=bb)

    def gemv():
        for i in range(len(mods)):
            aw.awsrc_packed_gemv(prm, shapes, i, bb[i], xs[i], sidecar=side, y=ys[i])

    batch = [(i, bb[i], xs[i], ys[i]) for i in range(len(mods))]

    def gemv_batch():
        aw.awsrc_packed_gemv_batch(prm, shapes, batch, sidecar=side)

    def dense():
        for o, x, y in zip(outs, xb, yb):
            torch.matmul(x, o.t(), out=y)

    def graph_ms(fn):
        side_stream = torch.cuda.Stream(device=dev)
        side_stream.wait_stream(torch.cuda.current_stream(dev))
        with torch.cuda.stream(side_stream):
            fn()                                 # warm-up outside the capture
        torch.cuda.current_stream(dev).wait_stream(side_stream)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            fn()
        g.replay()
        torch.cuda.synchronize()
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
        ev[0].record()
        for _ in range(reps):
            g.replay()
        ev[1].record()
        torch.cuda.synchronize()
        return ev[0].elapsed_time(ev[1]) / reps

    q_ms = graph_ms(quantise)
    qb_ms = graph_ms(quantise_batch)
    g_ms = graph_ms(gemv)
    b_ms = graph_ms(gemv_batch)
    d_ms = graph_ms(dense)
    q_bytes = N * 2 + N // 2 + G + 8 * ((G + 255) // 256) + N * 2
    # codes, SDQ codes and constants, tile map (8 B per tile), record slots
    # (16 B per record), the seeds' nibble tables (16 B per 8 elements), x, y
    g_bytes = (N // 2 + G + 8 * ((G + 255) // 256) + 8 * T + 16 * records + 16 * prm.S * (prm.C // 8)
               + 4 * sum(m["cols"] + m["rows"] for m in mods))
    return {"workload": "the 7 modules of the benchmark layer (77,070,336 weights), 0.162-bpw stream; "
                        "7 calls per figure (or one batched call), captured in a CUDA graph",
            "rtn_sdq": {"ms": qb_ms, "gbs": q_bytes / (qb_ms * 1e-3) / 1e9,
                        "frac_of_hbm": q_bytes / (qb_ms * 1e-3) / 1e9 / hbm_gbs, "bytes": q_bytes,
                        "call": "awsrc_rtn_quantize_batch, the 7 modules in one launch"},
            "rtn_sdq_per_module_calls": {"ms": q_ms, "gbs": q_bytes / (q_ms * 1e-3) / 1e9,
                                         "frac_of_hbm": q_bytes / (q_ms * 1e-3) / 1e9 / hbm_gbs},
            "packed_gemv_m1": {"ms": b_ms, "gbs": g_bytes / (b_ms * 1e-3) / 1e9,
                               "frac_of_hbm": g_bytes / (b_ms * 1e-3) / 1e9 / hbm_gbs, "bytes": g_bytes,
                               "call": "awsrc_packed_gemv_batch, the 7 modules in one launch"},
            "packed_gemv_m1_per_module_calls": {"ms": g_ms, "gbs": g_bytes / (g_ms * 1e-3) / 1e9,
                                                "frac_of_hbm": g_bytes / (g_ms * 1e-3) / 1e9 / hbm_gbs},
            "cublas_bf16_gemv_of_decoded_m1_ms": d_ms}


def model_stack(dev, hbm_gbs):
    """The full Qwen2.5-3B-shaped stack (36 layers x 7 modules, 2,774,532,096
    BF16 weights): every layer encoded (S = 4096) into one candidate array,
    one AWSRC-U selection over all 252 modules at 0.162 bits/weight, then one
    dense decode-apply call over every module. Timed on the device with CUDA
    events, each phase once after a warm-up pass over the whole model. The
    decode's algorithmic bytes are W0 read + W_hat written (4 B/weight) +
    the stream."""
    import torch
    import paper_2608_23144_gb300 as aw
    from synth import WORKLOADS, make_layer
    wl = WORKLOADS["qwen2.5-3b_stack"]
    mods = []
    for layer in range(wl.layers):
        for m in make_layer(wl, layer=layer, device=dev):
            del m["W"]  # the encoder reads W; it is regenerated per layer below
            mods.append(m)
    prm = aw.params(C=wl.C, P=wl.P, b=wl.b, S=wl.S)
    per_layer = len(wl.shapes)
    T_layer = wl.tiles_per_layer
    cands = torch.empty((T_layer * wl.layers, 16), dtype=torch.uint8, device=dev)
    ws = None
    outs = [torch.empty_like(m["W0"]) for m in mods]

    def encode_all():
        nonlocal ws
        ms = 0.0
        e = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
        for layer in range(wl.layers):
            lm = make_layer(wl, layer=layer, device=dev)  # W and W0 of this layer, regenerated
            sl = cands[layer * T_layer:(layer + 1) * T_layer]
            torch.cuda.synchronize()
            e[0].record()
            out = aw.awsrc_encode_tiles(prm, lm, out=sl, workspace=ws)
            e[1].record()
            torch.cuda.synchronize()
            ws = out._awsrc_workspace
            ms += e[0].elapsed_time(e[1])
            del lm
        return ms

    encode_all()                       # warm-up
    enc_ms = encode_all()
    assert aw.awsrc_workspace_status(ws) == 0, "encoder self-check fault"
    stream, counts, nbytes = aw.awsrc_select_records(prm, mods, cands, [RATE])
    sel_ws = stream._awsrc_workspace
    aw.awsrc_decode_apply(prm, mods, stream, -1, outs=outs)
    dec_ws = outs[0]._awsrc_workspace
    torch.cuda.synchronize()
    e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    e[0].record()
    aw.awsrc_select_records(prm, mods, cands, [RATE], workspace=sel_ws, out=stream, counts=counts, nbytes=nbytes)
    e[1].record()
    aw.awsrc_decode_apply(prm, mods, stream, -1, outs=outs, workspace=dec_ws)
    e[2].record()
    torch.cuda.synchronize()
    assert aw.awsrc_workspace_status(dec_ws) == 0, "decoder fault"
    sel_ms, dec_ms = e[0].elapsed_time(e[1]), e[1].elapsed_time(e[2])
    N = sum(m["rows"] * m["cols"] for m in mods)
    sb = int(nbytes[0].item())
    dec_bytes = 4 * N + sb
    out = {"workload": wl.description, "layers": wl.layers, "modules": len(mods), "weights": N,
           "encode_ms": enc_ms, "layers_per_s": wl.layers / (enc_ms * 1e-3),
           "encode_candidates_per_s": T_layer * wl.layers * wl.S / (enc_ms * 1e-3),
           "select_ms": sel_ms, "records": int(counts.sum().item()), "stream_bytes": sb,
           "decode_ms": dec_ms, "decode_gbs": dec_bytes / (dec_ms * 1e-3) / 1e9,
           "decode_frac_of_hbm": dec_bytes / (dec_ms * 1e-3) / 1e9 / hbm_gbs,
           "timing": "encode: 36 calls (one per layer, W regenerated between calls, outside the timed "
                     "events); select and decode: one call over all 252 modules"}
    del mods, outs, cands, stream
    torch.cuda.empty_cache()
    return out


def full_model(dev, hbm_gbs, name):
    """A whole synthetic model of the Qwen2.5-7B (28 layers, AWSRC-P_F) or
    Qwen2.5-32B (64 layers, AWSRC-U plus AWSRC-P_F) shape, streamed one layer
    at a time: each layer's W, W0, activation moments and Fisher diagonal are
    generated on the device, encoded for every variant into model-wide
    candidate arrays, then W and F are dropped (W0 stays for the decoder).
    After the last layer: one selection per variant over all modules (U at
    0.162 bits/weight; P_F prefixes at 0.05/0.10/0.162/0.25 with the 0.5/0.5
    activation/Fisher blend) and one dense decode-apply call over every
    module (the U stream, else each P_F prefix). Encode time is the sum of the
    per-layer CUDA-event times (generation outside them); select and decode
    are single calls, timed likewise."""
    import torch
    import paper_2608_23144_gb300 as aw
    from synth import WORKLOADS
    from synth.workloads import make_module, module_seed
    wl = WORKLOADS[name]
    PF_RATES = [0.05, 0.10, 0.162, 0.25]
    variants = [1] if wl.variant == 1 else [0, 1]
    prm = {v: aw.params(C=wl.C, P=wl.P, b=wl.b, S=wl.S, variant=v) for v in variants}
    T_layer = wl.tiles_per_layer
    cands = {v: torch.empty((T_layer * wl.layers, 16), dtype=torch.uint8, device=dev) for v in variants}
    ws = {v: None for v in variants}
    enc_ms = {v: 0.0 for v in variants}
    keep = []  # W0 and shapes of every module, for selection and decode
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    for layer in range(wl.layers):
        lm = []
        for mi, (_, rows, cols) in enumerate(wl.shapes):
            m = make_module(rows, cols, seed=module_seed(wl.seed, layer, mi), device=dev, w_dtype=wl.w_dtype,
                            outlier=wl.outlier, fisher=True, blend=(0.5, 0.5))
            lm.append(m)
        for v in variants:
            mv = lm if v == 1 else [{**m, "fisher": None, "w_act": 1.0, "w_fisher": 0.0} for m in lm]
            torch.cuda.synchronize()
            ev[0].record()
            out = aw.awsrc_encode_tiles(prm[v], mv, out=cands[v][layer * T_layer:(layer + 1) * T_layer],
                                        workspace=ws[v])
            ev[1].record()
            torch.cuda.synchronize()
            ws[v] = out._awsrc_workspace
            enc_ms[v] += ev[0].elapsed_time(ev[1])
        for m in lm:
            keep.append({"W0": m["W0"], "rows": m["rows"], "cols": m["cols"], "act": m["act"], "fisher": None,
                         "w_act": 1.0, "w_fisher": 0.0})
        del lm
    for v in variants:
        assert aw.awsrc_workspace_status(ws[v]) == 0, "encoder self-check fault"
    N = sum(m["rows"] * m["cols"] for m in keep)
    outs = [torch.empty_like(m["W0"]) for m in keep]
    res = {"workload": wl.description, "layers": wl.layers, "modules": len(keep), "weights": N}
    e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    for v in variants:
        rates = PF_RATES if v == 1 else [RATE]
        stream, counts, nbytes = aw.awsrc_select_records(prm[v], keep, cands[v], rates)   # warm-up
        torch.cuda.synchronize()
        e[0].record()
        aw.awsrc_select_records(prm[v], keep, cands[v], rates, workspace=stream._awsrc_workspace, out=stream,
                                counts=counts, nbytes=nbytes)
        e[1].record()
        torch.cuda.synchronize()
        key = "U" if v == 0 else "P_F"
        r = {"encode_ms": enc_ms[v], "layers_per_s": wl.layers / (enc_ms[v] * 1e-3),
             "encode_candidates_per_s": T_layer * wl.layers * wl.S / (enc_ms[v] * 1e-3),
             "select_ms": e[0].elapsed_time(e[1]), "rates_bpw": rates,
             "records": [int(x) for x in counts.tolist()] if v == 1 else int(counts.sum().item()),
             "stream_bytes": [int(x) for x in nbytes.tolist()]}
        Ks = [int(x) for x in counts.tolist()] if v == 1 else [-1]
        dec = []
        dws = None
        for ki, K in enumerate(Ks):
            aw.awsrc_decode_apply(prm[v], keep, stream, K, outs=outs, workspace=dws)
            dws = outs[0]._awsrc_workspace
            torch.cuda.synchronize()
            e[1].record()
            aw.awsrc_decode_apply(prm[v], keep, stream, K, outs=outs, workspace=dws)
            e[2].record()
            torch.cuda.synchronize()
            assert aw.awsrc_workspace_status(dws) == 0, "decoder fault"
            ms = e[1].elapsed_time(e[2])
            sb = int(nbytes[ki].item())  # the bytes of this prefix of the stream
            gbs = (4 * N + sb) / (ms * 1e-3) / 1e9
            dec.append({"K": K, "ms": ms, "gbs": gbs, "frac_of_hbm": gbs / hbm_gbs})
        r["decode"] = dec
        res[key] = r
        del stream
    del keep, outs, cands
    torch.cuda.empty_cache()
    return res


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    import numpy as np
    import torch
    from oracle import oracle as orc
    from synth import WORKLOADS, make_layer
    wl = WORKLOADS[WORKLOAD]
    orc.build()
    mods = host_modules(make_layer(wl, layer=0, device="cpu"))
    oprm = orc.params(C=wl.C, P=wl.P, b=wl.b, S=wl.S)
    masks = orc.basis_masks(oprm)
    rng = np.random.default_rng(1)
    tiles_per_row = sum(m["W"].shape[1] // wl.C for m in mods)

    # one step = `rows` random whole rows of every module, enough tiles per
    # oracle call to keep every host core busy
    def step(rows):
        n = 0
        for m in mods:
            r = rng.choice(m["W"].shape[0], rows, replace=False)
            orc.encode_tiles(oprm, m["W"][r], m["W0"][r], m["act"], masks=masks)
            n += rows * m["W"].shape[1] // wl.C
        return n * wl.S
    t0 = time.perf_counter()
    step(4)                                          # calibration (and warm-up)
    per_row = (time.perf_counter() - t0) / 4
    rows = max(1, min(min(m["W"].shape[0] for m in mods), int(args.ref_step_seconds / per_row)))
    for _ in range(args.warmup):
        step(rows)
    t0 = time.perf_counter()
    cands = sum(step(rows) for _ in range(args.steps))
    dt = time.perf_counter() - t0
    v = cands / dt
    sample = (f"per step {rows} random whole rows of each of the 7 modules "
              f"({rows * tiles_per_row:,} tiles x {wl.S} seeds = {cands // args.steps:,} candidates)")
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic", "config": {"workload": wl.description},
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": orc.num_threads(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ ours --
def run_ours(args):
    import torch
    import torch.distributed as dist

    import paper_2608_23144_gb300 as aw
    from synth import WORKLOADS, make_layer

    rank, world, local = dist_env()
    if world > 1:
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    wl = WORKLOADS[WORKLOAD]
    if args.modules:
        keep = args.modules.split(",")
        idx = [i for i, (name, _, _) in enumerate(wl.shapes) if name in keep]
        assert idx, f"no module of {wl.name} in {keep}"
        mods = make_layer(wl, layer=rank_layer(rank), device=dev, modules=idx)
    else:
        mods = make_layer(wl, layer=rank_layer(rank), device=dev)
    prm = aw.params(C=wl.C, P=wl.P, b=wl.b, S=wl.S)
    T = sum(m["rows"] * m["cols"] // wl.C for m in mods)
    cands_per_step = T * wl.S
    enc_ws = torch.empty(aw.awsrc_encode_workspace_bytes(prm, mods), dtype=torch.uint8, device=dev)
    cands = torch.empty((T, 16), dtype=torch.uint8, device=dev)
    outs = [torch.empty_like(m["W0"]) for m in mods]
    cap = aw.awsrc_stream_capacity(prm, mods, [RATE])
    sel_out = torch.zeros(cap, dtype=torch.uint8, device=dev)
    sel_counts = torch.empty(len(mods), dtype=torch.int64, device=dev)
    sel_bytes = torch.empty(1, dtype=torch.int64, device=dev)
    stream_dev = [None]
    sel_ws = [None]
    dec_ws = [None]

    def step(ev_dec=None, layer_mods=None):
        lm = mods if layer_mods is None else layer_mods
        aw.awsrc_encode_tiles(prm, lm, out=cands, workspace=enc_ws)
        s, counts, nbytes = aw.awsrc_select_records(prm, lm, cands, [RATE], workspace=sel_ws[0],
                                                    out=sel_out, counts=sel_counts, nbytes=sel_bytes)
        sel_ws[0] = s._awsrc_workspace
        stream_dev[0] = (s, counts, nbytes)
        if ev_dec is not None:
            ev_dec[0].record()
        aw.awsrc_decode_apply(prm, lm, s, -1, outs=outs, workspace=dec_ws[0])
        dec_ws[0] = outs[0]._awsrc_workspace
        if ev_dec is not None:
            ev_dec[1].record()

    def barrier():
        if world > 1:
            dist.barrier()

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    assert aw.awsrc_workspace_status(enc_ws) == 0, "encoder self-check fault"

    # timed region: K steps, events on the launching stream
    ev_s = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ev_e = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ev_d = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            for _ in range(args.steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    for ev in ev_s + ev_e:   # torch creates the CUDA event on first record
        ev.record()
    torch.cuda.synchronize()
    l0 = aw.awsrc_kernel_launches()
    barrier()
    torch.cuda.synchronize()
    with ClockSampler(gpu_id_for(dev)) as clk:
        start.record()
        for k in range(args.steps):
            aw.awsrc_set_timing_events(ev_s[k], ev_e[k])
            step(ev_d[k])
        end.record()
        torch.cuda.synchronize()
    barrier()
    aw.awsrc_set_timing_events(None, None)
    launches = aw.awsrc_kernel_launches() - l0
    ms = max_over_ranks(start.elapsed_time(end), dev)
    search_ms = statistics.mean(a.elapsed_time(b) for a, b in zip(ev_s, ev_e))
    dec_ms = statistics.mean(a.elapsed_time(b) for a, b in ev_d)
    s, counts, nbytes = stream_dev[0]
    stream_bytes = int(nbytes[0].item())
    w0_bytes = sum(m["W0"].numel() * m["W0"].element_size() for m in mods)
    out_bytes = sum(o.numel() * o.element_size() for o in outs)
    dec_gbs = (w0_bytes + out_bytes + stream_bytes) / (dec_ms * 1e-3) / 1e9

    peaks, peak_kind = measured_peaks()
    nsm = torch.cuda.get_device_properties(dev).multi_processor_count
    fp32_peak = nsm * 128 * float(peaks.get("sm_max_mhz", 2070.0)) * 1e6
    tensor_peak = float(peaks.get("bf16_tflops", 1900.0)) * 1e12
    method_flops = cands_per_step * METHOD_FLOP_PER_CANDIDATE / (search_ms * 1e-3)
    executed_flops = cands_per_step * TENSOR_FLOP_PER_CANDIDATE / (search_ms * 1e-3)
    fp32_ops = cands_per_step * OPS_PER_CANDIDATE / (search_ms * 1e-3)
    counters_valid = SEARCH_TRAFFIC["source_sha256"] == search_source_sha()
    traffic = SEARCH_TRAFFIC["bytes_per_launch"] if counters_valid else None
    weights = sum(m["rows"] * m["cols"] for m in mods)
    alg_bytes = search_algorithmic_bytes(weights, T)
    roofline = {"bound": "tensor", "kernel": "search_c64p4", "achieved": method_flops / 1e12,
                "peak": tensor_peak / 1e12, "unit": "TFLOP/s", "frac": method_flops / tensor_peak,
                "traffic": traffic,
                "peak_kind": f"{peak_kind} dense bf16 burst (fp16, the operands' type, has the same rate)",
                "work": f"{METHOD_FLOP_PER_CANDIDATE} flop per (tile, seed) candidate (2*C*P, the Eq. 3 "
                        f"correlation) x {cands_per_step:,} candidates per launch",
                "search_ms": search_ms,
                "executed_tensor": {"flop_per_candidate": TENSOR_FLOP_PER_CANDIDATE,
                                    "tflops": executed_flops / 1e12, "frac": executed_flops / tensor_peak},
                "fp32_epilogue": {"ops_per_candidate_before_pruning": OPS_PER_CANDIDATE,
                                  "gops": fp32_ops / 1e9, "peak_gops": fp32_peak / 1e9,
                                  "frac": fp32_ops / fp32_peak,
                                  "peak_kind": f"{nsm} SMs x 128 FP32 lanes x "
                                               f"{peaks.get('sm_max_mhz', 2070.0):.0f} MHz"},
                "dram": {"algorithmic_bytes": alg_bytes, "traffic_bytes": traffic,
                         "traffic_over_algorithmic": traffic / alg_bytes if traffic else None},
                "ncu": ({k: SEARCH_TRAFFIC[k] for k in ("ncu_fma_pipe_pct", "ncu_issue_active_pct",
                                                         "ncu_tensor_pipe_pct")} if counters_valid else None)}
    decode = {"gbs": dec_gbs, "ms": dec_ms, "frac_of_hbm": dec_gbs / float(peaks.get("hbm_gbs", 6800.0)),
              "hbm_peak_gbs": float(peaks.get("hbm_gbs", 6800.0))}

    # End to end through the public API with host buffers: every step uploads
    # its layer's W, W0 and activation moments from pinned host memory and reads
    # the stream and counts back. Uploads run on a copy stream into two device
    # buffer sets, so step i+1's upload overlaps step i's compute, as when the
    # layers of a model are streamed through the GPU; the compute stream waits
    # for its buffer's upload, the upload for the compute that last used it.
    e2e = None
    if not args.no_e2e:
        host = [{k: (v.cpu().pin_memory() if torch.is_tensor(v) else v) for k, v in m.items()} for m in mods]
        h2d = sum(v.numel() * v.element_size() for m in host for k, v in m.items()
                  if k in ("W", "W0", "act") and torch.is_tensor(v))
        # two pinned result buffers: step i's read-back lands in one while step
        # i + 1 is queued behind it
        host_stream = [torch.empty(s.numel(), dtype=torch.uint8).pin_memory() for _ in range(2)]
        host_counts = [torch.empty(counts.numel() + nbytes.numel(), dtype=torch.int64).pin_memory()
                       for _ in range(2)]
        d2h = host_stream[0].numel() + host_counts[0].numel() * 8
        bufs = [mods, [{**m, **{k: torch.empty_like(m[k]) for k in ("W", "W0", "act")}} for m in mods]]
        comp = torch.cuda.current_stream(dev)
        copy_stream = torch.cuda.Stream(device=dev)
        ev_copied = [torch.cuda.Event(), torch.cuda.Event()]
        ev_used = [torch.cuda.Event(), torch.cuda.Event()]
        ev_read = [torch.cuda.Event(), torch.cuda.Event()]
        records_read = []

        def upload(i):
            b = i % 2
            copy_stream.wait_event(ev_used[b])
            with torch.cuda.stream(copy_stream):
                for m, hm in zip(bufs[b], host):
                    for k in ("W", "W0", "act"):
                        m[k].copy_(hm[k], non_blocking=True)
            ev_copied[b].record(copy_stream)

        def e2e_step(i):
            b = i % 2
            comp.wait_event(ev_copied[b])
            step(layer_mods=bufs[b])
            ev_used[b].record(comp)
            s2, c2, n2 = stream_dev[0]
            host_stream[b].copy_(s2, non_blocking=True)
            host_counts[b][: c2.numel()].copy_(c2, non_blocking=True)
            host_counts[b][c2.numel():].copy_(n2, non_blocking=True)
            ev_read[b].record(comp)

        def read_back(i):
            # the result of step i on the host (its record count), every step
            ev_read[i % 2].synchronize()
            records_read.append(int(host_counts[i % 2][: counts.numel()].sum()))

        def run(n):
            # step i + 1 is queued before the host waits for step i's result,
            # so the host's launch work overlaps the GPU's
            upload(0)
            for i in range(n):
                if i + 1 < n:
                    upload(i + 1)
                e2e_step(i)
                if i >= 1:
                    read_back(i - 1)
            read_back(n - 1)

        for ev in ev_used:
            ev.record(comp)
        run(2)
        torch.cuda.synchronize()
        barrier()
        t0 = time.perf_counter()
        run(args.steps)
        dt = time.perf_counter() - t0
        torch.cuda.synchronize()
        barrier()
        dt = max_over_ranks(dt, dev)
        assert all(r == int(counts.sum()) for r in records_read), "read-back record counts differ"
        e2e = {"value": job_value(cands_per_step, world, args.steps, dt), "unit": UNIT,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "ms_per_step": 1e3 * dt / args.steps,
               "uploads": "copy stream, double-buffered; each step's result read on the host "
                          "while the next step runs"}
        del bufs[1]

    # the P_F variant of the search on one Qwen2.5-7B-shaped layer (blended
    # activation/Fisher weights), timed on the device outside the step
    pf = None
    if rank == 0 and not args.no_pf and not args.modules:
        wl7 = WORKLOADS["qwen2.5-7b_stack_pf"]
        m7 = make_layer(wl7, layer=0, device=dev)
        p7 = aw.params(C=wl7.C, P=wl7.P, b=wl7.b, S=wl7.S, variant=1)
        c7 = aw.awsrc_encode_tiles(p7, m7)
        ws7 = c7._awsrc_workspace
        torch.cuda.synchronize()
        e7 = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
        reps = 3
        e7[0].record()
        for _ in range(reps):
            aw.awsrc_encode_tiles(p7, m7, out=c7, workspace=ws7)
        e7[1].record()
        torch.cuda.synchronize()
        assert aw.awsrc_workspace_status(ws7) == 0, "P_F encoder self-check fault"
        ms7 = e7[0].elapsed_time(e7[1]) / reps
        T7 = wl7.tiles_per_layer
        pf = {"workload": "one Qwen2.5-7B-shaped layer (7 modules, 233,046,016 weights) BF16, "
                          "AWSRC-P_F 0.5/0.5 activation/Fisher blend, C=64 P=4 b=4 S=4096",
              "encode_ms": ms7, "candidates_per_s": T7 * wl7.S / (ms7 * 1e-3)}
        del m7, c7, ws7

    paper = serving = None
    if rank == 0 and not args.no_pf and not args.modules:
        paper = paper_points(dev, float(peaks.get("hbm_gbs", 6800.0)))
        serving = backbone_and_serving(dev, prm, mods, outs, s, int(counts.sum().item()),
                                       float(peaks.get("hbm_gbs", 6800.0)))
    model = None
    if rank == 0 and world == 1 and not args.no_model and not args.modules:
        model = model_stack(dev, float(peaks.get("hbm_gbs", 6800.0)))
    models = None
    if rank == 0 and world == 1 and not args.no_full_models and not args.modules:
        models = {n: full_model(dev, float(peaks.get("hbm_gbs", 6800.0)), n)
                  for n in ("qwen2.5-7b_stack_pf", "qwen2.5-32b_stack")}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, cores, desc = oracle_sample(wl, host_modules(mods), args.cpu_seconds)
        cpu = {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": desc}

    if rank == 0:
        value = job_value(cands_per_step, world, args.steps, ms * 1e-3)
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": max(3, args.warmup), "ms_per_step": ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": wl.description if not args.modules else
                       f"{wl.name} modules {args.modules} (profiling subset)", "tiles_per_gpu": T, "seeds": wl.S, "C": wl.C,
                       "P": wl.P, "b": wl.b, "rate_bpw": RATE, "variant": "U",
                       "parallelism": f"{world} independent layers" if world > 1 else "single GPU",
                       "l2": "inputs larger than L2 (W and W0 of the layer: 308 MB per step)"},
            "layers_per_s": world * args.steps / (ms * 1e-3) if not args.modules else None,
            "encode_candidates_per_s_kernel": cands_per_step / (search_ms * 1e-3),
            "decode_apply": decode,
            "records_per_step": int(counts.sum().item()), "stream_bytes": stream_bytes,
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "pf": pf, "paper_points": paper, "backbone_and_serving": serving, "model_stack": model,
            "full_models": models,
            "gpu_launches": launches, "clocks": clk.summary(),
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
