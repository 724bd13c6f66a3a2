#!/usr/bin/env python3
"""Benchmark of the frame-quantized linear layer forward (libframequant) on GB300.

One step = the forward pass of every linear layer of a Llama-2-7B decoder block (q, k, v, o
4096x4096; gate, up 11008x4096; down 4096x11008) on one batch of tokens: analysis z = T_in x,
2-bit frame-coefficient product with per-row dequantization, synthesis y = T_out^T u, at
redundancy r = 1.1 with rho = 16.  The headline is decode (M = 16 tokens, HBM-bound); the
prefill regime (M = 2048, tensor-core-bound) is measured in the same run.

Inputs are seeded and synthetic (workloads/): W ~ N(0, 0.02^2), tokens ~ N(0, 1) in bf16 with
1% of channels x30.  The frames, frame coefficients and 2-bit codes are produced on the GPU by
the library's own offline entry points (fq_frame_build, fq_coefficients, fq_quantize_rtn,
fq_pack) before timing starts.

Usage:  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
Under torchrun each rank runs its own batch (no collective on the data path); the timing is
the maximum over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = ("frame-quant linear µs/layer; HBM GB/s (M≤16) & TFLOP/s (M=2048) vs "
          "GB300 peak")
UNIT = "us/layer"
RHO = 16
# the launches of one decoder block: independent layers share a launch
GROUPS = (("q", "k", "v"), ("o",), ("gate", "up"), ("down",))
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
SMI_FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


# --------------------------------------------------------------------------- accounting
def layer_bytes(d_in, d_out, n_in, n_out, M):
    """Algorithmic bytes of one layer forward: 2-bit codes, fp16 scale and zero, bf16 T_in and
    T_out, bf16 tokens in and out (z and u are intermediates and not counted)."""
    return (n_out * n_in // 4 + 4 * n_out + 2 * n_in * d_in + 2 * n_out * d_out
            + 2 * M * (d_in + d_out))


def layer_flops(d_in, d_out, n_in, n_out, M):
    return 2 * M * (n_in * d_in + n_out * n_in + d_out * n_out)


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {k: float(p[k]) for k in FALLBACK_PEAKS}, "measured"
    except (OSError, KeyError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def source_hash():
    """Hash of the sources that define the decode kernel: its code, the device helpers and the
    workspace constants it is built with (its traffic record is only valid for these exact
    sources)."""
    h = hashlib.sha256()
    pkg = os.path.join(ROOT, "paper_2403_06082_gb300", "csrc")
    for path in (os.path.join(pkg, "fq_decode.cu"), os.path.join(pkg, "fq_device.cuh"),
                 os.path.join(pkg, "fq_internal.h")):
        with open(path, "rb") as f:
            h.update(os.path.basename(path).encode())
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(key):
    """DRAM bytes per call from the committed ncu summary, if taken on the current kernels."""
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            rec = json.load(f)
    except (OSError, ValueError):
        return None
    if rec.get("source_hash") != source_hash():
        return None
    ent = rec.get(key)
    return None if ent is None else ent.get("dram_bytes_per_call")


# --------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 100 ms while running."""

    def __init__(self, uuid=None):
        self.uuid = uuid
        self.proc = None

    def __enter__(self):
        cmd = ["nvidia-smi", f"--query-gpu={SMI_FIELDS}", "--format=csv,noheader,nounits",
               "-lms", "100"]
        if self.uuid:
            cmd += ["-i", self.uuid]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                         text=True)
        except OSError:
            self.proc = None
        time.sleep(0.25)
        return self

    def __exit__(self, *exc):
        self.out = ""
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self):
        rows = []
        for line in (self.out or "").strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[4:9]))
            except ValueError:
                continue
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for _, _, r in rows for n, v in zip(names, r[1:])
                          if v.lower().startswith("active")})
        loaded = [s for s, _, _ in rows if s > 0] or [rows[0][0]]
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(m for _, m, _ in rows),
                "reasons": reasons, "samples": len(rows)}


# --------------------------------------------------------------------------- device layers
def prepare_layer(fq, wl, torch, wk, layer, r, dev):
    """Frames, coefficients, codes and packed words of one layer, made on the GPU by the
    library's offline entry points; returns the inference-time operands."""
    k_in, k_out = wl.k_for(r, layer.d_in), wl.k_for(r, layer.d_out)
    n_in, n_out = k_in * RHO, k_out * RHO

    def frame(k, d, side):
        dr = wl.rotation_draws(wk.seed, wk.key, layer.name, side, d=d)
        nb = fq.fq_frame_workspace_bytes(k, RHO, d, dr.a, dr.b)
        ws = torch.empty(nb, dtype=torch.uint8, device=dev)
        T = torch.empty(k * RHO, d, dtype=torch.float32, device=dev)
        fq.fq_frame_build(k, RHO, d, (dr.a, dr.b, dr.ga, dr.gb, dr.perm, dr.signs), T, ws, nb)
        return T

    T_in = frame(k_in, layer.d_in, "in")
    T_out = frame(k_out, layer.d_out, "out")
    W = torch.from_numpy(wl.weight(wk, layer)).to(dev, torch.float32)
    C = torch.empty(n_out, n_in, dtype=torch.float32, device=dev)
    nb = fq.fq_coefficients_workspace_bytes(layer.d_out, n_in)
    ws = torch.empty(nb, dtype=torch.uint8, device=dev)
    fq.fq_coefficients(W, layer.d_out, layer.d_in, T_in, n_in, T_out, n_out, C, ws, nb)
    del W, ws
    codes = torch.empty(n_out, n_in, dtype=torch.uint8, device=dev)
    scale = torch.empty(n_out, dtype=torch.int16, device=dev)
    zero = torch.empty(n_out, dtype=torch.int16, device=dev)
    gamma = torch.empty(n_out, dtype=torch.float32, device=dev)
    fq.fq_quantize_rtn(C, n_out, n_in, codes, scale, zero, gamma)
    del C
    words = torch.empty(fq.fq_packed_words(n_out, n_in), dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    C_packed = fq.fq_pack(codes, scale, zero, n_out, n_in, words, status)
    if fq.fq_check(status) != 0:
        raise RuntimeError("fq_pack reported out-of-range codes or a non-finite scale or zero")
    del codes
    return {
        "name": layer.name, "d_in": layer.d_in, "d_out": layer.d_out, "n_in": n_in,
        "n_out": n_out, "k_in": k_in, "k_out": k_out,
        "T_in": T_in.to(torch.bfloat16), "T_out_t": T_out.t().contiguous().to(torch.bfloat16),
        "C": C_packed, "gamma": gamma,
    }


class Regime:
    """All layers of one workload at one token count, with inputs, outputs and workspaces."""

    def __init__(self, fq, wl, torch, wl_key, M, dev, rank, use_gamma=False):
        self.fq, self.torch, self.dev, self.M = fq, torch, dev, M
        self.wk = wl.WORKLOADS[wl_key]
        self.r = self.wk.redundancy[0]
        self.layers = [prepare_layer(fq, wl, torch, self.wk, l, self.r, dev)
                       for l in self.wk.layers]
        self.use_gamma = use_gamma
        # independent layers of the block, one fq_linear_forward_group launch each (a
        # transformer's q, k and v read the same input, and so do gate and up)
        by = {L["name"]: L for L in self.layers}
        self.groups = [[by[n] for n in names] for names in GROUPS if all(n in by for n in names)]
        ws_bytes = max(fq.fq_workspace_bytes(M, L["d_in"], L["n_in"], L["n_out"], L["d_out"], 0)
                       for L in self.layers)
        # The step's activations and outputs live in one device buffer each (every layer a
        # 256-byte aligned slice), mirrored by one pinned host buffer each, so a step moves its
        # inputs in one host-to-device copy and its results in one device-to-host copy.
        def offsets(sizes):
            offs, tot = [], 0
            for n in sizes:
                offs.append(tot)
                tot += -(-n // 128) * 128
            return offs, tot
        xo, xt = offsets([M * L["d_in"] for L in self.layers])
        yo, yt = offsets([M * L["d_out"] for L in self.layers])
        self.x_all = torch.zeros(xt, dtype=torch.bfloat16, device=dev)
        self.y_all = torch.zeros(yt, dtype=torch.bfloat16, device=dev)
        self.x_host_all = torch.zeros(xt, dtype=torch.bfloat16).pin_memory()
        self.y_host_all = torch.zeros(yt, dtype=torch.bfloat16).pin_memory()
        for L, layer, x0, y0 in zip(self.layers, self.wk.layers, xo, yo):
            X = wl.activations(self.wk, layer, M)
            if rank:
                X = wl.round_bf16(wl.rng(rank, wl_key, layer.name, "X-rank").standard_normal(X.shape))
            L["x_host"] = self.x_host_all[x0:x0 + M * L["d_in"]].view(M, L["d_in"])
            L["x_host"].copy_(torch.from_numpy(X).to(torch.bfloat16))
            L["x"] = self.x_all[x0:x0 + M * L["d_in"]].view(M, L["d_in"])
            L["x"].copy_(L["x_host"])
            L["y"] = self.y_all[y0:y0 + M * L["d_out"]].view(M, L["d_out"])
            L["y_host"] = self.y_host_all[y0:y0 + M * L["d_out"]].view(M, L["d_out"])
        # the decode launches read the frames as pre-swizzled tiles (fq_frame_tile): the same
        # values, one contiguous 16 KiB copy per 128 x 64 block
        self.use_tiles = M <= 64
        if self.use_tiles:
            for L in self.layers:
                for src, rows, cols, key in ((L["T_in"], L["n_in"], L["d_in"], "T_in_tiles"),
                                             (L["T_out_t"], L["d_out"], L["n_out"],
                                              "T_out_tiles")):
                    nb = fq.fq_frame_tiles_bytes(rows, cols)
                    L[key] = torch.empty(nb, dtype=torch.uint8, device=dev)
                    fq.fq_frame_tile(src, rows, cols, L[key], nb)
        for grp in self.groups:
            ws_bytes = max(ws_bytes, fq.fq_group_workspace_bytes(M, self.group_layers(grp)))
        self.ws_bytes = ws_bytes
        self.ws = torch.zeros(ws_bytes, dtype=torch.uint8, device=dev)
        # one eager call per layer before any capture (sets kernel attributes, checks status)
        for L in self.layers:
            self.forward(L, torch.cuda.current_stream(dev).cuda_stream)
            st = fq.fq_check(self.ws)
            if st != 0:
                raise RuntimeError(f"{L['name']}: {fq.fq_status_str(st)}")
        for grp in self.groups:
            self.forward_group(grp, torch.cuda.current_stream(dev).cuda_stream)
            st = fq.fq_check(self.ws)
            if st != 0:
                raise RuntimeError(f"group {[L['name'] for L in grp]}: {fq.fq_status_str(st)}")
        torch.cuda.synchronize()

    def group_layers(self, grp):
        fq = self.fq
        t = self.use_tiles
        return [fq.Layer(L["x"], L["d_in"], L["T_in"], L["C"], L["T_out_t"], L["d_out"],
                         L["gamma"] if self.use_gamma else None, L["y"],
                         L["T_in_tiles"] if t else None, L["T_out_tiles"] if t else None)
                for L in grp]

    def forward_group(self, grp, stream, prefetch=None):
        """One launch for the group's layers (fq_linear_forward_group, which takes the tiled
        frames; a single layer on row-major frames through fq_linear_forward_ex), naming
        `prefetch` as the L2 hint."""
        if len(grp) == 1 and not self.use_tiles:
            self.forward(grp[0], stream, prefetch)
            return
        self.fq.fq_linear_forward_group(self.M, self.group_layers(grp), self.ws, self.ws_bytes,
                                        0, prefetch, stream)

    def capture_groups(self, stream, host=False):
        """One graph: the block as its launches (groups in order), each naming the next
        launch's first T_in as its L2 prefetch hint; with host=True the step's inputs come
        from pinned host memory first and its results go back at the end."""
        torch = self.torch
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            if host:
                self.x_all.copy_(self.x_host_all, non_blocking=True)
            self.launch_groups(stream)
            if host:
                self.y_host_all.copy_(self.y_all, non_blocking=True)
        return g

    def launch_groups(self, stream, only=None):
        n = len(self.groups)
        for i, grp in enumerate(self.groups):
            if only is not None and i != only:
                continue
            nxt = self.groups[(i + 1) % n][0]
            self.forward_group(grp, stream.cuda_stream,
                               nxt["T_in_tiles"] if self.use_tiles else nxt["T_in"])

    def forward(self, L, stream, prefetch=None):
        fq = self.fq
        if prefetch is None:
            fq.fq_linear_forward(L["x"], self.M, L["d_in"], L["T_in"], L["C"], L["T_out_t"],
                                 L["d_out"], L["gamma"] if self.use_gamma else None, L["y"],
                                 self.ws, self.ws_bytes, fq.FQ_BF16, stream)
        else:
            fq.fq_linear_forward_ex(L["x"], self.M, L["d_in"], L["T_in"], L["C"], L["T_out_t"],
                                    L["d_out"], L["gamma"] if self.use_gamma else None, L["y"],
                                    self.ws, self.ws_bytes, fq.FQ_BF16, 0, prefetch, stream)

    def capture(self, layers, stream, host=False, chain=False):
        """One graph: the layers' forwards in order; with host=True (all layers) the step's
        inputs come from pinned host memory first and its results go back at the end.  With
        chain=True each forward names the next layer's T_in (the first layer's after the last)
        as its L2 prefetch hint."""
        torch = self.torch
        assert not host or layers is self.layers
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            if host:
                self.x_all.copy_(self.x_host_all, non_blocking=True)
            for i, L in enumerate(layers):
                nxt = layers[(i + 1) % len(layers)]["T_in"] if chain else None
                self.forward(L, stream.cuda_stream, nxt)
            if host:
                self.y_host_all.copy_(self.y_all, non_blocking=True)
        return g

    def host_bytes(self):
        """Bytes one host-backed step copies in and out."""
        return self.x_all.numel() * 2, self.y_all.numel() * 2

    def bytes_flops(self, L):
        args = (L["d_in"], L["d_out"], L["n_in"], L["n_out"], self.M)
        return layer_bytes(*args), layer_flops(*args)


def eager_e2e(torch, dec, stream, steps, warmup):
    """Total ms of `steps` end-to-end steps issued as plain API calls on `stream`: the H2D
    copy of the step's inputs from pinned memory, the block's 4 launches (q|k|v and gate|up
    through fq_linear_forward_group, o and down through fq_linear_forward_ex, each naming the
    next launch's T_in as its L2 prefetch hint), the D2H copy of the outputs."""
    def step():
        dec.x_all.copy_(dec.x_host_all, non_blocking=True)
        dec.launch_groups(stream)
        dec.y_host_all.copy_(dec.y_all, non_blocking=True)

    with torch.cuda.stream(stream):
        for _ in range(warmup):
            step()
    torch.cuda.synchronize()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        start.record(stream)
        for _ in range(steps):
            step()
        end.record(stream)
    torch.cuda.synchronize()
    if dec.fq.fq_check(dec.ws) != 0:
        raise RuntimeError("eager end-to-end step: device status")
    return start.elapsed_time(end)


def timed_replays(torch, graphs, stream, steps, warmup, events_between=False):
    """Replay the graphs (one step = all of them in order) `steps` times after `warmup`
    untimed steps; returns total ms and, with events_between, per-graph mean ms."""
    with torch.cuda.stream(stream):
        for _ in range(warmup):
            for g in graphs:
                g.replay()
    torch.cuda.synchronize()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    marks = []
    with torch.cuda.stream(stream):
        start.record(stream)
        for _ in range(steps):
            if events_between:
                row = []
                for g in graphs:
                    e = torch.cuda.Event(enable_timing=True)
                    e.record(stream)
                    row.append(e)
                    g.replay()
                marks.append(row)
            else:
                for g in graphs:
                    g.replay()
        end.record(stream)
    torch.cuda.synchronize()
    total = start.elapsed_time(end)
    per = None
    if events_between:
        per = [0.0] * len(graphs)
        for i, row in enumerate(marks):
            nxt = marks[i + 1][0] if i + 1 < len(marks) else end
            for j, e in enumerate(row):
                per[j] += e.elapsed_time(row[j + 1] if j + 1 < len(row) else nxt)
        per = [p / steps for p in per]
    return total, per


# --------------------------------------------------------------------------- CPU oracle
def cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo), or the machine type."""
    import platform
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        fields = dict(l.split(":", 1) for l in out.splitlines() if ":" in l)
        name = " ".join(fields.get(k, "").strip() for k in ("Vendor ID", "Model name")).strip()
        if name:
            return f"{name} ({platform.machine()})"
    except (OSError, subprocess.SubprocessError, ValueError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith(("model name", "cpu part")):
                    return f"{line.split(':', 1)[1].strip()} ({platform.machine()})"
    except OSError:
        pass
    return platform.machine()


def cpu_baseline(seconds=12.0):
    """The fp64 oracle's layer forward on this host's cores, on a bounded sample of the
    decode workload: the q (4096x4096) and down (4096x11008) layer shapes at M = 16, repeated
    until `seconds` have passed; reported per layer with the block's 4 : 3 mix of small and
    large layers (gate, up and down have the same cost)."""
    import numpy as np

    import workloads as wl
    from oracle import forward, frames

    wk = wl.WORKLOADS["llama2_7b_decode"]
    r = wk.redundancy[0]
    shapes = {"q": wk.layers[0], "down": wk.layers[6]}
    built = {}
    for key, layer in shapes.items():
        k_in, k_out = wl.k_for(r, layer.d_in), wl.k_for(r, layer.d_out)
        T_in = frames.frame(k_in, RHO, layer.d_in,
                            wl.rotation_draws(wk.seed, wk.key, layer.name, "in", d=layer.d_in))
        T_out = frames.frame(k_out, RHO, layer.d_out,
                             wl.rotation_draws(wk.seed, wk.key, layer.name, "out", d=layer.d_out))
        n_in, n_out = T_in.shape[0], T_out.shape[0]
        codes = wl.random_codes(wk.seed, wk.key, layer.name, n_out=n_out, n_in=n_in)
        scale, zero = wl.random_scale_zero(wk.seed, wk.key, layer.name, n_out=n_out, mag=0.01)
        X = wl.activations(wk, layer, 16)
        built[key] = (X, T_in, codes, scale, zero, T_out)
    times = {k: [] for k in built}
    t_end = time.perf_counter() + seconds
    while time.perf_counter() < t_end or any(len(v) < 2 for v in times.values()):
        for k, args in built.items():
            t0 = time.perf_counter()
            forward.layer_forward(*args)
            times[k].append(time.perf_counter() - t0)
    tq = statistics.median(times["q"])
    tl = statistics.median(times["down"])
    per_layer_us = (4 * tq + 3 * tl) / 7 * 1e6
    n = sum(len(v) for v in times.values())
    return {"value": round(per_layer_us, 1), "unit": UNIT, "cores": os.cpu_count(),
            "tokens_per_s": round(16 / (per_layer_us * 1e-6), 1),
            "cpu": cpu_model(), "kind": "oracle",
            "sample": (f"fp64 numpy oracle forward, M=16, {n} layer calls over "
                       f"{seconds:.0f}+ s: q-shape median {tq * 1e3:.1f} ms, "
                       f"down-shape median {tl * 1e3:.1f} ms, weighted 4:3 as in the block; "
                       "seeded random 2-bit codes")}


def reference_arm(args, rank):
    """--impl reference: the fp64 oracle as it stands, on this host's cores, one decode
    layer forward (M = 16, cycling through the block's layer shapes) per step, within a time
    budget so the whole run stays within a few minutes."""
    if rank:
        return
    budget = float(os.environ.get("FQ_REFERENCE_BUDGET_S", "150"))
    import numpy as np  # noqa: F401

    import workloads as wl
    from oracle import forward, frames

    wk = wl.WORKLOADS["llama2_7b_decode"]
    r = wk.redundancy[0]
    cache = {}

    def operands(layer):
        key = (layer.d_in, layer.d_out)
        if key not in cache:
            k_in, k_out = wl.k_for(r, layer.d_in), wl.k_for(r, layer.d_out)
            T_in = frames.frame(k_in, RHO, layer.d_in, wl.rotation_draws(
                wk.seed, wk.key, layer.name, "in", d=layer.d_in))
            T_out = frames.frame(k_out, RHO, layer.d_out, wl.rotation_draws(
                wk.seed, wk.key, layer.name, "out", d=layer.d_out))
            n_in, n_out = T_in.shape[0], T_out.shape[0]
            codes = wl.random_codes(wk.seed, wk.key, layer.name, n_out=n_out, n_in=n_in)
            s, z = wl.random_scale_zero(wk.seed, wk.key, layer.name, n_out=n_out, mag=0.01)
            cache[key] = (T_in, codes, s, z, T_out)
        T_in, codes, s, z, T_out = cache[key]
        return (wl.activations(wk, layer, 16), T_in, codes, s, z, T_out)

    layers = list(wk.layers)
    for i in range(args.warmup):
        forward.layer_forward(*operands(layers[i % len(layers)]))
    done, elapsed = 0, 0.0
    t_stop = time.perf_counter() + budget
    for i in range(args.steps):
        ops = operands(layers[i % len(layers)])
        t0 = time.perf_counter()
        forward.layer_forward(*ops)
        elapsed += time.perf_counter() - t0
        done += 1
        if time.perf_counter() > t_stop:
            break
    us = elapsed / done * 1e6
    sample = (f"fp64 numpy oracle, decode M=16, {done} layer forwards cycling q,k,v,o,gate,up,"
              f"down (of {args.steps} requested; {budget:.0f} s budget), seeded random codes")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": round(us, 1), "unit": UNIT,
        "n_gpus": args.gpus, "steps": done, "warmup": args.warmup,
        "ms_per_step": round(us / 1e3, 3), "higher_is_better": False, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": "llama2_7b_block_decode", "M": 16, "r": "1.1", "rho": RHO},
        "cpu_baseline": {"value": round(us, 1), "unit": UNIT, "cores": os.cpu_count(),
                         "cpu": cpu_model(), "kind": "oracle", "sample": sample},
        "e2e": {"value": round(us, 1), "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


def measure_prefill(args, fq, wl, torch, dev, rank, world, dist, stream, peaks):
    """Prefill regime: the same block at M = 2048 with the de-noising filter on."""
    pre = Regime(fq, wl, torch, "llama2_7b_prefill", 2048, dev, rank, use_gamma=True)
    pg = pre.capture(pre.layers, stream)
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    p_ms, _ = timed_replays(torch, [pg], stream, args.prefill_steps, 3)
    p_ms = max_over_ranks(p_ms, dist, dev)
    lgs = [pre.capture([L], stream) for L in pre.layers]
    _, p_per = timed_replays(torch, lgs, stream, max(5, args.prefill_steps // 2), 3,
                             events_between=True)
    fl = [pre.bytes_flops(L)[1] for L in pre.layers]
    step_fl = sum(fl)
    tflops = step_fl / (p_ms / args.prefill_steps * 1e-3) / 1e12
    pdom = max(range(len(fl)), key=lambda i: p_per[i])
    out = {
        "M": 2048, "gamma": True, "steps": args.prefill_steps,
        "us_per_layer": round(aggregate(p_ms, args.prefill_steps, len(fl), world), 2),
        "tflops": round(tflops * world, 1),
        # each layer is a graph of 0.2-0.7 ms and the step a few ms: the burst peak applies
        "tensor_frac": round(tflops / peaks["bf16_tflops"], 3),
        "peak_tflops": peaks["bf16_tflops"],
        "peak_kind": "burst (cuBLAS bf16, timed alone)",
        "tensor_frac_of_sustained": round(tflops / peaks["bf16_tflops_sustained"], 3),
        "per_layer_us": {L["name"]: round(p_per[i] * 1e3, 1) for i, L in enumerate(pre.layers)},
        "dominant": {"kernel": f"fq_linear_forward[{pre.layers[pdom]['name']}]",
                     "achieved_tflops": round(fl[pdom] / (p_per[pdom] * 1e-3) / 1e12, 1),
                     "frac": round(fl[pdom] / (p_per[pdom] * 1e-3) / 1e12
                                   / peaks["bf16_tflops"], 3)},
    }
    del pg, lgs, pre
    torch.cuda.empty_cache()
    return out


def prefill_only(args, fq, wl, torch, dev, rank, world, dist, stream, peaks):
    """--regime prefill: one JSON line for the prefill regime alone (value in us/layer)."""
    pf = measure_prefill(args, fq, wl, torch, dev, rank, world, dist, stream, peaks)
    if rank == 0:
        print(json.dumps({"metric": METRIC, "value": pf["us_per_layer"], "unit": UNIT,
                          "n_gpus": world, "steps": args.prefill_steps, "warmup": 3,
                          "higher_is_better": False, "scaling": "weak", "dtype": "bf16",
                          "config": {"workload": "llama2_7b_block_prefill", "M": 2048},
                          "prefill": pf}), flush=True)
    if dist is not None:
        dist.destroy_process_group()


# --------------------------------------------------------------------------- structured frames
def measure_implicit(args, fq, wl, torch, dec, stream, peaks):
    """The decode block with T_in and T_out in structured form: one CUDA graph of the seven
    fq_linear_forward_implicit calls on the regime's tokens, codes and workspace."""
    wk, dev, M = dec.wk, dec.dev, dec.M
    frames, bytes_ = [], 0
    for L, layer in zip(dec.layers, wk.layers):
        def fr(side, d, k):
            dr = wl.rotation_draws(wk.seed, wk.key, layer.name, side, d=d)
            return fq.fq_frame_implicit(k, RHO, d, (dr.a, dr.b, dr.ga, dr.gb, dr.perm, dr.signs),
                                        dev)
        Fi, Fo = fr("in", L["d_in"], L["k_in"]), fr("out", L["d_out"], L["k_out"])
        frames.append((Fi, Fo))
        # what one forward reads: codes, scale and zero, tokens in and out, the input frame's
        # analysis tiles and the output frame's synthesis tiles, and both rotations' factors
        rot = lambda F: 4 * (F.c.a * F.c.a * 2 + F.c.b * F.c.b * 2) + 12 * F.c.d
        bytes_ += (L["n_out"] * L["n_in"] // 4 + 4 * L["n_out"] + 2 * M * (L["d_in"] + L["d_out"])
                   + 16384 * (Fi.c.ana_count + Fo.c.syn_count) + rot(Fi) + rot(Fo))
    nb = max(fq.fq_implicit_workspace_bytes(M, L["d_in"], L["n_in"], L["n_out"], L["d_out"])
             for L in dec.layers)

    by = {L["name"]: (L, F) for L, F in zip(dec.layers, frames)}
    groups = [[by[n] for n in names] for names in GROUPS if all(n in by for n in names)]
    glayers = [[fq.ImplicitLayer(L["x"], Fi, L["C"], Fo, None, L["y"]) for L, (Fi, Fo) in grp]
               for grp in groups]
    nb = max([nb] + [fq.fq_implicit_group_workspace_bytes(M, g) for g in glayers])

    def step(st):
        # the block's launches as in the headline: q|k|v and gate|up one group call each
        for g in glayers:
            if len(g) == 1:
                Ly = g[0]
                fq.fq_linear_forward_implicit(Ly.x, M, Ly.F_in, Ly.C, Ly.F_out, None, Ly.y, ws,
                                              nb, 0, st.cuda_stream)
            else:
                fq.fq_linear_forward_implicit_group(M, g, ws, nb, 0, st.cuda_stream)

    ws = torch.zeros(nb, dtype=torch.uint8, device=dev)
    step(stream)
    torch.cuda.synchronize()
    if fq.fq_check(ws) != 0:
        raise RuntimeError("implicit block: device status")
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        step(stream)
    steps = max(50, args.steps // 4)
    ms, _ = timed_replays(torch, [g], stream, steps, args.warmup)
    if fq.fq_check(ws) != 0:
        raise RuntimeError("implicit block: device status after timing")
    us = ms * 1e3 / (steps * len(dec.layers))
    roof_us = bytes_ / (peaks["hbm_gbs"] * 1e9) * 1e6 / len(dec.layers)
    del g
    return {
        "value": round(us, 3), "unit": UNIT, "steps": steps,
        "bytes_per_layer": round(bytes_ / len(dec.layers)),
        "hbm_frac": round(roof_us / us, 3),
        "launches_per_step": 3 * len(groups),
        "how": ("the block's 4 launches as in the headline, frames in structured form: per "
                "launch the input rotations (fp32, CUDA cores, one kernel for the group), the "
                "fused decode kernel with block-sparse frame operands (analysis, code product "
                "and synthesis on the tensor cores), the output rotations; "
                "fq_linear_forward_implicit_group for q|k|v and gate|up"),
    }


# --------------------------------------------------------------------------- sweep
def prepare_layer_random_codes(fq, wl, torch, wk, layer, r, dev):
    """Like prepare_layer, with seeded uniform codes and scale/zero in place of the real frame
    coefficients (the kernels' work does not depend on the code values; computing C for the
    70B shapes takes seconds of fp32 GEMM per layer)."""
    import numpy as np
    k_in, k_out = wl.k_for(r, layer.d_in), wl.k_for(r, layer.d_out)
    n_in, n_out = k_in * RHO, k_out * RHO

    def frame(k, d, side):
        dr = wl.rotation_draws(wk.seed, wk.key, layer.name, side, d=d)
        nb = fq.fq_frame_workspace_bytes(k, RHO, d, dr.a, dr.b)
        ws = torch.empty(nb, dtype=torch.uint8, device=dev)
        T = torch.empty(k * RHO, d, dtype=torch.float32, device=dev)
        fq.fq_frame_build(k, RHO, d, (dr.a, dr.b, dr.ga, dr.gb, dr.perm, dr.signs), T, ws, nb)
        return T

    T_in = frame(k_in, layer.d_in, "in").to(torch.bfloat16)
    T_out_t = frame(k_out, layer.d_out, "out").t().contiguous().to(torch.bfloat16)
    torch.cuda.empty_cache()
    codes = torch.from_numpy(wl.random_codes(wk.seed, wk.key, layer.name, str(r), n_out=n_out,
                                             n_in=n_in)).to(dev)
    words = torch.empty(fq.fq_packed_words(n_out, n_in), dtype=torch.int32, device=dev)
    sc, ze = wl.random_scale_zero(wk.seed, wk.key, layer.name, n_out=n_out, mag=0.01)
    scale = torch.from_numpy(sc.view(np.int16)).to(dev)
    zero = torch.from_numpy(ze.view(np.int16)).to(dev)
    C_packed = fq.fq_pack(codes, scale, zero, n_out, n_in, words)
    del codes
    gamma = torch.ones(n_out, dtype=torch.float32, device=dev)
    return {
        "name": layer.name, "d_in": layer.d_in, "d_out": layer.d_out, "n_in": n_in,
        "n_out": n_out, "k_in": k_in, "k_out": k_out, "T_in": T_in, "T_out_t": T_out_t,
        "C": C_packed, "gamma": gamma,
    }


def time_layer(fq, torch, L, X, use_gamma, dev, stream, flush, reps=30, warm_calls=20):
    """Cold time (median over `reps` calls, each after writing a buffer twice the size of L2,
    CUDA events around the call alone) and warm time (`warm_calls` calls back to back in one
    CUDA graph, total / calls) of one layer forward, in microseconds."""
    M = X.shape[0]
    x = X if X.is_cuda else X.to(dev)
    y = torch.empty(M, L["d_out"], dtype=torch.bfloat16, device=dev)
    nb = fq.fq_workspace_bytes(M, L["d_in"], L["n_in"], L["n_out"], L["d_out"], 0)
    ws = torch.zeros(nb, dtype=torch.uint8, device=dev)
    g = L["gamma"] if use_gamma else None

    def call():
        fq.fq_linear_forward(x, M, L["d_in"], L["T_in"], L["C"], L["T_out_t"], L["d_out"], g,
                             y, ws, nb, fq.FQ_BF16, stream.cuda_stream)

    with torch.cuda.stream(stream):
        for _ in range(3):
            call()
    torch.cuda.synchronize()
    st = fq.fq_check(ws)
    if st != 0:
        raise RuntimeError(f"{L['name']} M={M}: {fq.fq_status_str(st)}")
    cold = []
    with torch.cuda.stream(stream):
        for _ in range(reps):
            flush.add_(1)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            call()
            e1.record(stream)
            cold.append((e0, e1))
    torch.cuda.synchronize()
    cold_us = statistics.median(a.elapsed_time(b) for a, b in cold) * 1e3
    gr = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gr, stream=stream):
        for _ in range(warm_calls):
            call()
    warm_ms, _ = timed_replays(torch, [gr], stream, 3, 3)
    warm_us = warm_ms * 1e3 / (3 * warm_calls)
    if fq.fq_check(ws) != 0:
        raise RuntimeError(f"{L['name']} M={M}: device status after timing")
    del gr
    return cold_us, warm_us


def sweep(args, fq, wl, torch, dev, stream, peaks):
    """--sweep: every configuration of the workload set, one layer shape at a time: cold and
    warm microseconds per layer, tokens/s and the fraction of the roofline
    max(bytes / HBM peak, FLOPs / bf16 peak)."""
    flush = torch.zeros(2 * 129 * 2**20 // 4, dtype=torch.float32, device=dev)
    rows = []
    plan = [("single256", None, False), ("vit_b16_mlp", None, False),
            ("llama2_7b_decode", ("q", "gate", "down"), False),
            ("llama2_7b_prefill", ("q", "gate", "down"), False),
            ("llama2_70b", ("q", "gate", "down"), True)]
    for key, names, random_codes in plan:
        wk = wl.WORKLOADS[key]
        layers = [l for l in wk.layers if names is None or l.name in names]
        for layer in layers:
            acts = {}
            for r in wk.redundancy:
                prep = prepare_layer_random_codes if random_codes else prepare_layer
                L = prep(fq, wl, torch, wk, layer, r, dev)
                for M in wk.tokens:
                    if M not in acts:
                        acts[M] = torch.from_numpy(wl.activations(wk, layer, M)).to(
                            dev, torch.bfloat16)
                    for use_gamma in wk.gamma:
                        cold, warm = time_layer(fq, torch, L, acts[M], use_gamma, dev, stream,
                                                flush)
                        args_ = (L["d_in"], L["d_out"], L["n_in"], L["n_out"], M)
                        by, fl = layer_bytes(*args_), layer_flops(*args_)
                        t_hbm = by / (peaks["hbm_gbs"] * 1e9) * 1e6
                        t_tc = fl / (peaks["bf16_tflops"] * 1e12) * 1e6
                        bound = "hbm" if t_hbm >= t_tc else "tensor"
                        rows.append({
                            "workload": key, "layer": f"{layer.name} {layer.d_out}x{layer.d_in}",
                            "r": str(r), "k_in": L["k_in"], "k_out": L["k_out"], "M": M,
                            "gamma": use_gamma, "us_cold": round(cold, 2),
                            "us_warm": round(warm, 2), "tokens_per_s": round(M / cold * 1e6),
                            "bytes": by, "flops": fl, "bound": bound,
                            "roof_us": round(max(t_hbm, t_tc), 2),
                            "frac_cold": round(max(t_hbm, t_tc) / cold, 3),
                            "frac_warm": round(max(t_hbm, t_tc) / warm, 3),
                            "codes": "seeded uniform" if random_codes else "RTN of C",
                        })
                        print(json.dumps(rows[-1]), file=sys.stderr, flush=True)
                del L
                torch.cuda.empty_cache()
            del acts
    print(json.dumps({
        "metric": METRIC, "unit": UNIT, "n_gpus": 1, "dtype": "bf16", "data": "synthetic",
        "peaks": {"hbm_gbs": peaks["hbm_gbs"], "bf16_tflops": peaks["bf16_tflops"]},
        "timing": ("cold: median of 30 calls, each after writing a 258 MB buffer (2 x L2), CUDA "
                   "events around the call; warm: 20 calls back to back in a CUDA graph"),
        "sweep": rows}), flush=True)


# --------------------------------------------------------------------------- summaries
SUMMARY_PLAN = (
    # (configuration, workload, layer, r, M, gamma, seeded codes)
    ("cfg1 single 256x256", "single256", "single", None, 8, False, False),
    ("cfg2 ViT-B/16 fc1 3072x768", "vit_b16_mlp", "fc1", None, 12608, False, False),
    ("cfg2 ViT-B/16 fc2 768x3072", "vit_b16_mlp", "fc2", None, 12608, False, False),
    ("cfg4 7B gate 11008x4096", "llama2_7b_prefill", "gate", None, 4096, True, False),
    ("cfg5 70B q 8192x8192", "llama2_70b", "q", "11/10", 16, False, True),
    ("cfg5 70B gate 28672x8192", "llama2_70b", "gate", "11/10", 16, False, True),
    ("cfg5 70B down 8192x28672", "llama2_70b", "down", "11/10", 128, False, True),
    ("cfg5 70B q 8192x8192 M=4096", "llama2_70b", "q", "11/10", 4096, False, True),
)


def config_summary(fq, wl, torch, dev, stream, peaks):
    """One representative layer of the configurations the headline block does not cover,
    timed cold (a 258 MB L2 flush before each call, CUDA events around the call): us/layer,
    tokens/s and the fraction of max(bytes / HBM peak, FLOPs / burst bf16 peak)."""
    from fractions import Fraction
    flush = torch.zeros(2 * 129 * 2**20 // 4, dtype=torch.float32, device=dev)
    out = {}
    for label, key, name, r, M, use_gamma, seeded in SUMMARY_PLAN:
        wk = wl.WORKLOADS[key]
        layer = next(l for l in wk.layers if l.name == name)
        rr = wk.redundancy[0] if r is None else Fraction(r)
        prep = prepare_layer_random_codes if seeded else prepare_layer
        L = prep(fq, wl, torch, wk, layer, rr, dev)
        X = torch.from_numpy(wl.activations(wk, layer, M)).to(dev, torch.bfloat16)
        cold, warm = time_layer(fq, torch, L, X, use_gamma, dev, stream, flush, reps=20,
                                warm_calls=10)
        args_ = (L["d_in"], L["d_out"], L["n_in"], L["n_out"], M)
        by, fl = layer_bytes(*args_), layer_flops(*args_)
        t_hbm = by / (peaks["hbm_gbs"] * 1e9) * 1e6
        t_tc = fl / (peaks["bf16_tflops"] * 1e12) * 1e6
        out[label] = {"M": M, "r": str(rr), "gamma": use_gamma, "us_cold": round(cold, 2),
                      "us_warm": round(warm, 2), "tokens_per_s": round(M / cold * 1e6),
                      "bound": "hbm" if t_hbm >= t_tc else "tensor",
                      "roof_us": round(max(t_hbm, t_tc), 2),
                      "frac_cold": round(max(t_hbm, t_tc) / cold, 3),
                      "codes": "seeded uniform" if seeded else "RTN of C"}
        del L, X
        torch.cuda.empty_cache()
    del flush
    torch.cuda.empty_cache()
    return out


def reconstruction_crossover(fq, wl, torch, dev, stream, peaks):
    """The weight-reconstruction path against the frame forward on the 7B q and gate shapes
    at 2048 and 4096 tokens: the one-off fq_reconstruct_weight, then fq_dense_forward per batch,
    against fq_linear_forward per batch (cold, median of 10).  The crossover is the number of
    batches after which reconstructing once and running dense products is cheaper."""
    wk = wl.WORKLOADS["llama2_7b_prefill"]
    flush = torch.zeros(2 * 129 * 2**20 // 4, dtype=torch.float32, device=dev)

    def cold_us(fn, reps=10):
        with torch.cuda.stream(stream):
            fn()
            fn()
        torch.cuda.synchronize()
        evs = []
        with torch.cuda.stream(stream):
            for _ in range(reps):
                flush.add_(1)
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                fn()
                e1.record(stream)
                evs.append((e0, e1))
        torch.cuda.synchronize()
        return statistics.median(a.elapsed_time(b) for a, b in evs) * 1e3

    out = {}
    for name in ("q", "gate"):
        layer = next(l for l in wk.layers if l.name == name)
        L = prepare_layer(fq, wl, torch, wk, layer, wk.redundancy[0], dev)
        d_in, d_out = L["d_in"], L["d_out"]
        W = torch.empty(d_out, d_in, dtype=torch.bfloat16, device=dev)
        nr = fq.fq_reconstruct_workspace_bytes(d_in, L["n_in"], L["n_out"], d_out)
        wsr = torch.zeros(nr, dtype=torch.uint8, device=dev)
        rec = cold_us(lambda: fq.fq_reconstruct_weight(
            L["T_in"], L["C"], L["T_out_t"], d_in, d_out, None, W, wsr, nr, stream.cuda_stream),
            reps=3)
        if fq.fq_check(wsr) != 0:
            raise RuntimeError(f"reconstruct {name}: device status")
        del wsr
        torch.cuda.empty_cache()
        for M in (2048, 4096):
            x = torch.from_numpy(wl.activations(wk, layer, M)).to(dev, torch.bfloat16)
            y = torch.empty(M, d_out, dtype=torch.bfloat16, device=dev)
            nf = fq.fq_workspace_bytes(M, d_in, L["n_in"], L["n_out"], d_out, 0)
            wsf = torch.zeros(nf, dtype=torch.uint8, device=dev)
            nd = fq.fq_dense_workspace_bytes(M, d_in, d_out)
            wsd = torch.zeros(nd, dtype=torch.uint8, device=dev)
            fwd = cold_us(lambda: fq.fq_linear_forward(
                x, M, d_in, L["T_in"], L["C"], L["T_out_t"], d_out, None, y, wsf, nf, 0,
                stream.cuda_stream))
            dense = cold_us(lambda: fq.fq_dense_forward(x, M, d_in, W, d_out, y, wsd, nd,
                                                        stream.cuda_stream))
            fl_dense = 2 * M * d_in * d_out
            out[f"{name} {d_out}x{d_in} M={M}"] = {
                "forward_us": round(fwd, 1), "dense_us": round(dense, 1),
                "reconstruct_us": round(rec, 1),
                "dense_tflops": round(fl_dense / (dense * 1e-6) / 1e12, 1),
                "dense_frac": round(fl_dense / (dense * 1e-6) / 1e12 / peaks["bf16_tflops"], 3),
                "crossover_batches": (round(rec / (fwd - dense), 2) if fwd > dense else None),
            }
            del x, y, wsf, wsd
            torch.cuda.empty_cache()
        del L, W
        torch.cuda.empty_cache()
    del flush
    return out


# --------------------------------------------------------------------------- main
def aggregate(elapsed_ms, steps, layers_per_step, world):
    """Whole-job microseconds per layer from the slowest rank's elapsed time: every rank
    runs its own batch, so the job processes steps * layers_per_step * world layer calls."""
    return elapsed_ms * 1e3 / (steps * layers_per_step * world)


def max_over_ranks(value, dist=None, device="cpu"):
    """Largest value over the ranks of the default process group (the value itself alone)."""
    if dist is None:
        return value
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--prefill-steps", type=int, default=20)
    ap.add_argument("--no-prefill", action="store_true")
    ap.add_argument("--regime", default="both", choices=["both", "decode", "prefill"],
                    help="decode (the headline), prefill, or both (default)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-summary", action="store_true",
                    help="skip the per-configuration summary and the reconstruction crossover")
    ap.add_argument("--sweep", action="store_true",
                    help="time every configuration's layer shapes (one JSON line) and exit")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world != args.gpus:
        if world == 1 and args.gpus > 1:
            ap.error("--gpus N > 1 runs under torchrun (one process per GPU)")
    if args.impl == "reference":
        reference_arm(args, rank)
        return

    import torch

    import paper_2403_06082_gb300 as fq
    import workloads as wl

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    fq.lib()
    peaks, peak_src = load_peaks()
    stream = torch.cuda.Stream(device=dev)

    def barrier():
        torch.cuda.synchronize()
        if dist is not None:
            dist.barrier()

    if args.sweep:
        if rank == 0:
            sweep(args, fq, wl, torch, dev, stream, peaks)
        return
    if args.regime == "prefill":
        prefill_only(args, fq, wl, torch, dev, rank, world, dist, stream, peaks)
        return
    if args.regime == "decode":
        args.no_prefill = True

    # ---------------- decode: Llama-2-7B block, M = 16
    dec = Regime(fq, wl, torch, "llama2_7b_decode", 16, dev, rank)
    nL = len(dec.layers)
    nG = len(dec.groups)
    step_graph = dec.capture_groups(stream)
    launch_graphs = []
    for gi in range(nG):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            dec.launch_groups(stream, only=gi)
        launch_graphs.append(g)
    # the same 4 launches reading the row-major frames through 2-D tensor-map boxes
    dec.use_tiles = False
    rm_graph = dec.capture_groups(stream)
    dec.use_tiles = True
    seq_graph = dec.capture(dec.layers, stream, chain=True)
    layer_graphs = [dec.capture([L], stream) for L in dec.layers]
    e2e_graph = dec.capture_groups(stream, host=True)

    uuid = None
    try:
        uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:  # noqa: BLE001 - older torch without uuid
        uuid = None
    barrier()
    with ClockSampler(uuid) as clk:
        total_ms, _ = timed_replays(torch, [step_graph], stream, args.steps, args.warmup)
    barrier()
    total_ms = max_over_ranks(total_ms, dist, dev)
    us_layer = aggregate(total_ms, args.steps, nL, world)
    if fq.fq_check(dec.ws) != 0:
        raise RuntimeError("decode block: device status after timing")

    # per-launch durations (events between per-launch graphs) for the roofline
    rl_steps = max(50, args.steps // 4)
    _, per_launch = timed_replays(torch, launch_graphs, stream, rl_steps, args.warmup,
                                  events_between=True)
    bytes_fl = {L["name"]: dec.bytes_flops(L) for L in dec.layers}
    launch_bytes = [sum(bytes_fl[L["name"]][0] for L in grp) for grp in dec.groups]
    dom = max(range(nG), key=lambda i: per_launch[i])
    achieved = launch_bytes[dom] / (per_launch[dom] * 1e-3) / 1e9
    step_bytes = sum(launch_bytes)
    dom_names = "|".join(L["name"] for L in dec.groups[dom])

    # the same block as 7 single-layer launches (each naming the next layer's T_in as its
    # L2 hint), and each layer alone
    barrier()
    seq_ms, _ = timed_replays(torch, [seq_graph], stream, args.steps, args.warmup)
    seq_ms = max_over_ranks(seq_ms, dist, dev)
    seq_us = aggregate(seq_ms, args.steps, nL, world)
    _, per_ms = timed_replays(torch, layer_graphs, stream, rl_steps, args.warmup,
                              events_between=True)
    sequential = {
        "value": round(seq_us, 3), "unit": UNIT, "ms_per_step": round(seq_ms / args.steps, 4),
        "how": "one fq_linear_forward_ex launch per layer (7 per step), one CUDA graph per step",
        "per_layer": {L["name"]: {"us": round(per_ms[i] * 1e3, 2),
                                  "GBps": round(bytes_fl[L["name"]][0] / (per_ms[i] * 1e-3) / 1e9,
                                                1),
                                  "hbm_frac": round(bytes_fl[L["name"]][0] / (per_ms[i] * 1e-3)
                                                    / 1e9 / peaks["hbm_gbs"], 3)}
                      for i, L in enumerate(dec.layers)},
    }
    del seq_graph, layer_graphs
    barrier()
    rm_ms, _ = timed_replays(torch, [rm_graph], stream, args.steps, args.warmup)
    rm_ms = max_over_ranks(rm_ms, dist, dev)
    row_major = {
        "value": round(aggregate(rm_ms, args.steps, nL, world), 3), "unit": UNIT,
        "ms_per_step": round(rm_ms / args.steps, 4),
        "how": ("the headline's 4 launches with the frames read row-major (T_in, T_out_t "
                "through 2-D tensor-map boxes of 128 rows x 128 bytes) instead of as tiles"),
    }
    del rm_graph

    # the same block with the frames in structured form (fq_linear_forward_implicit)
    implicit = measure_implicit(args, fq, wl, torch, dec, stream, peaks)

    # end to end through the C ABI with host buffers: plain calls (the API's host work inside
    # the timed region), and the same step captured once as a CUDA graph
    barrier()
    e2e_steps = max(100, args.steps // 4)
    e2e_ms = eager_e2e(torch, dec, stream, e2e_steps, args.warmup)
    e2e_ms = max_over_ranks(e2e_ms, dist, dev)
    e2e_us = aggregate(e2e_ms, e2e_steps, nL, world)
    e2eg_ms, _ = timed_replays(torch, [e2e_graph], stream, e2e_steps, args.warmup)
    e2eg_ms = max_over_ranks(e2eg_ms, dist, dev)
    e2eg_us = aggregate(e2eg_ms, e2e_steps, nL, world)
    h2d, d2h = dec.host_bytes()

    per_launch_out = {
        "|".join(L["name"] for L in grp): {
            "us": round(per_launch[i] * 1e3, 2),
            "GBps": round(launch_bytes[i] / (per_launch[i] * 1e-3) / 1e9, 1),
            "hbm_frac": round(launch_bytes[i] / (per_launch[i] * 1e-3) / 1e9 / peaks["hbm_gbs"],
                              3)}
        for i, grp in enumerate(dec.groups)}
    roof_us = step_bytes / (peaks["hbm_gbs"] * 1e9) * 1e6 / nL
    del step_graph, launch_graphs, e2e_graph
    dec_layers = [(L["name"], L["d_out"], L["d_in"], L["k_in"], L["k_out"]) for L in dec.layers]
    group_names = " ; ".join("|".join(L["name"] for L in grp) for grp in dec.groups)
    del dec
    torch.cuda.empty_cache()

    # ---------------- prefill: same block, M = 2048, de-noising filter on
    prefill = None if args.no_prefill else measure_prefill(args, fq, wl, torch, dev, rank, world,
                                                            dist, stream, peaks)
    summary = crossover = None
    if world == 1 and not args.no_summary:
        summary = config_summary(fq, wl, torch, dev, stream, peaks)
        crossover = reconstruction_crossover(fq, wl, torch, dev, stream, peaks)

    if dist is not None:
        dist.barrier()
    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return

    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline()

    clocks = clk.summary()
    line = {
        "metric": METRIC, "value": round(us_layer, 3), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(total_ms / args.steps, 4), "higher_is_better": False,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": ("synthetic: W ~ N(0, 0.02^2), tokens ~ N(0,1) bf16 with 1% channels x30; "
                 "frames, coefficients and 2-bit codes built on the GPU from seeded draws"),
        "config": {
            "workload": "llama2_7b_block_decode", "M": 16, "r": "1.1", "rho": RHO,
            "layers": {n: f"{o}x{i} k_in={ki} k_out={ko}" for n, o, i, ki, ko in dec_layers},
            "l2": ("no flush: each step streams 1.2 GB of distinct layer operands (> 126 MB "
                   "L2), so every layer's operands were last touched one step earlier"),
            "timing": ("one CUDA graph per step: the block's 4 launches (" + group_names +
                       "; q|k|v and gate|up each one fq_linear_forward_group call), each naming "
                       "the next launch's T_in as its L2 prefetch hint; CUDA events around K "
                       "replays"),
            "parallelism": f"replicas x{world}, no data-path collective",
        },
        "roofline": {
            "bound": "hbm", "kernel": (f"decode_layer_kernel[{dom_names}] (analysis, code "
                                       "product and synthesis fused, one launch)"),
            "achieved": round(achieved, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": round(achieved / peaks["hbm_gbs"], 3),
            "traffic": recorded_traffic(f"decode_{dom_names}"),
            "peak_source": f"{peak_src} (STREAM-style copy)",
            "step_frac": round(roof_us / us_layer, 3),
            "per_launch": per_launch_out,
        },
        "sequential": sequential,
        "row_major": row_major,
        "implicit": implicit,
        "e2e": {"value": round(e2e_us, 3), "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h,
                "copies": ("per step: one host-to-device copy of the 7 layers' inputs from pinned "
                           "memory, the block's 4 launches, one device-to-host copy of their "
                           "outputs"),
                "how": ("plain calls: each step issues the copies and the 4 forward calls through "
                        "the C ABI (argument checks, tensor-map encoding and plan lookup on the "
                        "host inside the timed region); CUDA events around K steps"),
                "graph_value": round(e2eg_us, 3),
                "graph_how": "the same step captured once in a CUDA graph and replayed"},
        "gpu_launches": nG * args.steps,      # one fused kernel per launch (M <= 64)
        "clocks": clocks,
        "prefill": prefill,
        "configs": summary,
        "reconstruction": crossover,
        "cpu_baseline": cpu,
    }
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
