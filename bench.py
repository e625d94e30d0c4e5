#!/usr/bin/env python3
"""Throughput of one QUASAR reconstruction step on GB300.

A step is one pass of the whole hot path -- saliency EMA, clip-range search,
code assignment, weighted least-squares fit and the write of r, v', a, b and
the kept candidate -- over every linear weight of a 32-layer
Llama-3.1-8B-shaped model (224 tensors, 6.98e9 weights, ~84 GB resident:
fp32 w and v, bf16 g and r), with inputs already resident in HBM.  The
headline format is INT3 with group 128 and 8 clip candidates; the other
formats of the sweep (INT2, INT4, NVFP4, one AdamW step fused with the INT3
reconstruction, and the Rubin INT3 lookup-table format) are timed after it
and reported in "sweep".  Each step
streams ~70 GB of inputs, far more than the 129 MB L2.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
With N > 1 it runs under torchrun, one rank per GPU; every rank processes the
whole model (independent replicas, weak scaling) and the slowest rank's time
counts.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_13966_gb300 import quasar as Q  # noqa: E402
from paper_2608_13966_gb300 import workloads as WL  # noqa: E402

METRIC = "reconstructed weights/sec and achieved HBM GB/s (fraction of ~8 TB/s) per QUASAR step"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


# ------------------------------------------------------------------ setup --

def dist_setup(n_gpus):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        torch.distributed.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    if torch.cuda.is_available():
        torch.cuda.set_device(local)
    return world, rank


def barrier(world):
    if world > 1:
        torch.distributed.barrier()


def max_over_ranks(x, world):
    if world == 1:
        return x
    dev = "cuda" if torch.distributed.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


DTYPE_NAME = {torch.bfloat16: "bf16", torch.float32: "f32"}


def bytes_per_step(wlo, elements, amax_supplied=False):
    """Algorithmic HBM bytes of one step: read w (4) + g (2 bf16, 4 fp32) +
    v (4), write v (4) + r (2 bf16, 4 fp32) and the codes (1, where the
    workload writes them) per weight; per group a, b (fp32) and the kept
    index (u8) for integer codes; per 16-block the E4M3 scale and index for
    NVFP4, plus the tensor-absmax pre-pass (one more read of w) unless the
    caller supplies the amax; per 512-block 8 table bytes and the index for
    the lookup table.  The fused AdamW step also reads m and writes w' and m'
    (12 more bytes a weight)."""
    gb = 2 if wlo.g_dtype == torch.bfloat16 else 4
    rb = 2 if wlo.r_dtype == torch.bfloat16 else 4
    cb = 1 if wlo.with_codes else 0
    core = 4 + gb + 4 + 4 + rb + cb
    if wlo.fmt == "int" and wlo.adamw:
        return elements * (core + 12) + (elements // wlo.group) * 9
    if wlo.fmt == "nvfp4" and wlo.adamw:  # AdamW + absmax pass, then w', v' -> r
        return elements * (12 + gb + 12) + elements * (8 + rb + cb) + (elements // 16) * 2
    if wlo.fmt == "lut":
        return elements * core + (elements // 512) * 9
    if wlo.fmt == "int":
        return elements * core + (elements // wlo.group) * 9
    return elements * core + (elements // 16) * 2 + (0 if amax_supplied else elements * 4)


class Model:
    """All tensors of a workload, resident on the device, with outputs."""

    def __init__(self, wlo, device, shard=0):
        """``shard``: the rank's shard of a weak-scaled job -- every rank holds
        a full model's worth of distinct tensors (seed = shard)."""
        self.wlo = wlo
        self.seed = shard
        self.tensors = []
        for spec in wlo.tensors:
            d = WL.make_tensor(wlo, spec, device=device, seed=shard)
            n = spec.numel
            d["r"] = torch.empty((spec.rows, spec.cols), dtype=wlo.r_dtype, device=device)
            if wlo.with_codes:
                d["codes"] = torch.empty(n, dtype=torch.uint8, device=device)
            gsz = min(wlo.group, 128) if wlo.fmt == "int" else 128
            d["a"] = torch.empty(n // gsz, dtype=torch.float32, device=device)
            d["b"] = torch.empty(n // gsz, dtype=torch.float32, device=device)
            d["idx"] = torch.empty(n // 16, dtype=torch.uint8, device=device)
            d["scale"] = torch.empty(n // 16, dtype=torch.uint8, device=device)
            d["ts"] = torch.empty(1, dtype=torch.float32, device=device)
            d["spec"] = spec
            self.tensors.append(d)
        self.elements = sum(t["spec"].numel for t in self.tensors)


class Step:
    """Pre-marshalled C-ABI calls of one step for one format."""

    def __init__(self, model, wlo, stream, amax_supplied=False):
        """amax_supplied (NVFP4): every tensor's absmax is handed to the call
        (taken once here, outside any timing), so the absmax pass is skipped."""
        import ctypes
        self.lib = Q.load()
        self.wlo = wlo
        self.stream = stream.cuda_stream
        GD = Q.BF16 if wlo.g_dtype == torch.bfloat16 else Q.F32
        RD = Q.BF16 if wlo.r_dtype == torch.bfloat16 else Q.F32
        if amax_supplied:
            for d in model.tensors:
                d["amax"] = d["w"].abs().max().reshape(1).float()
        self.clip = (ctypes.c_float * len(wlo.clip))(*wlo.clip)
        self.calls = []
        if wlo.adamw and wlo.fmt == "nvfp4":
            # AdamW step taking the absmax of w', then the NVFP4 batch
            for d in model.tensors:
                if "m" not in d:
                    spec = d["spec"]
                    d["m"] = WL.first_moment((spec.rows, spec.cols), model.seed * 1000 + spec.index,
                                             d["w"].device)
            hp = wlo.adamw
            self.descs = Q.adamw_nvfp4_tensor_array([
                {"w": d["w"], "g": d["g"], "m": d["m"], "v": d["v"], "r": d["r"], "codes": d.get("codes"),
                 "block_scale": d["scale"], "tensor_scale": d["ts"], "cand_idx": d["idx"],
                 "rows": d["spec"].rows, "cols": d["spec"].cols}
                for d in model.tensors])
            args = (ctypes.cast(self.descs, ctypes.c_void_p), len(self.descs), GD, hp["lr"],
                    hp["beta1"], wlo.beta2, hp["eps"], hp["weight_decay"], hp["step"], self.clip,
                    len(wlo.clip), RD, None, self.stream)
            self.calls.append((self.lib.quasar_adamw_recon_nvfp4_batch, args, model.elements))
        elif wlo.adamw:
            # AdamW step + reconstruction of every tensor in one launch
            # (quasar_adamw_recon_int_batch); m is drawn here if the model
            # was built for a workload without an optimizer step
            for d in model.tensors:
                if "m" not in d:
                    spec = d["spec"]
                    d["m"] = WL.first_moment((spec.rows, spec.cols), model.seed * 1000 + spec.index,
                                             d["w"].device)
            hp = wlo.adamw
            self.descs = Q.adamw_tensor_array([
                {"w": d["w"], "g": d["g"], "m": d["m"], "v": d["v"], "r": d["r"], "codes": d.get("codes"),
                 "a": d["a"], "b": d["b"], "cand_idx": d["idx"], "rows": d["spec"].rows,
                 "cols": d["spec"].cols}
                for d in model.tensors])
            args = (ctypes.cast(self.descs, ctypes.c_void_p), len(self.descs), GD, hp["lr"],
                    hp["beta1"], wlo.beta2, hp["eps"], hp["weight_decay"], hp["step"], wlo.bits,
                    wlo.group, self.clip, len(wlo.clip), RD, None, self.stream)
            self.calls.append((self.lib.quasar_adamw_recon_int_batch, args, model.elements))
        elif wlo.fmt == "lut":
            # every tensor in one launch (quasar_recon_lut_batch)
            for d in model.tensors:
                if "book" not in d:
                    d["book"] = torch.empty((d["spec"].numel // 512, 8), dtype=torch.uint8,
                                            device=d["w"].device)
            self.descs = Q.lut_tensor_array([
                {"w": d["w"], "g": d["g"], "v": d["v"], "r": d["r"], "codes": d.get("codes"), "book": d["book"],
                 "cand_idx": d["idx"], "rows": d["spec"].rows, "cols": d["spec"].cols}
                for d in model.tensors])
            args = (ctypes.cast(self.descs, ctypes.c_void_p), len(self.descs), GD, wlo.beta2,
                    self.clip, len(wlo.clip), RD, None, self.stream)
            self.calls.append((self.lib.quasar_recon_lut_batch, args, model.elements))
        elif wlo.fmt == "int":
            # every tensor of the model in one launch (quasar_recon_int_batch)
            self.descs = Q.int_tensor_array([
                {"w": d["w"], "g": d["g"], "v": d["v"], "r": d["r"], "codes": d.get("codes"),
                 "a": d["a"], "b": d["b"], "cand_idx": d["idx"], "rows": d["spec"].rows,
                 "cols": d["spec"].cols}
                for d in model.tensors])
            if wlo.symmetric:
                self.opt = Q.options(symmetric=True)
                args = (ctypes.cast(self.descs, ctypes.c_void_p), len(self.descs), GD,
                        wlo.beta2, wlo.bits, wlo.group, self.clip, len(wlo.clip), RD,
                        ctypes.cast(ctypes.pointer(self.opt), ctypes.c_void_p), self.stream)
                self.calls.append((self.lib.quasar_recon_int_batch_ex, args, model.elements))
            else:
                args = (ctypes.cast(self.descs, ctypes.c_void_p), len(self.descs), GD,
                        wlo.beta2, wlo.bits, wlo.group, self.clip, len(wlo.clip), RD,
                        self.stream)
                self.calls.append((self.lib.quasar_recon_int_batch, args, model.elements))
        else:
            # every tensor in one call (quasar_recon_nvfp4_batch): absmax of
            # every tensor, their scales, one reconstruction launch
            self.descs = Q.nvfp4_tensor_array([
                {"w": d["w"], "g": d["g"], "v": d["v"], "tensor_amax": d.get("amax"), "r": d["r"],
                 "codes": d.get("codes"), "block_scale": d["scale"], "tensor_scale": d["ts"],
                 "cand_idx": d["idx"], "rows": d["spec"].rows, "cols": d["spec"].cols}
                for d in model.tensors])
            args = (ctypes.cast(self.descs, ctypes.c_void_p), len(self.descs), GD, wlo.beta2,
                    self.clip, len(wlo.clip), RD, self.stream)
            self.calls.append((self.lib.quasar_recon_nvfp4_batch, args, model.elements))
        # INT: one launch; NVFP4: absmax, scale and reconstruction launches
        # (plus one small memset of the scale slot per tensor)
        self.launches_per_call = (2 if amax_supplied else 3) if wlo.fmt == "nvfp4" else 1

    def run(self, events=None):
        for i, (fn, args, _) in enumerate(self.calls):
            if events is not None:
                events[i][0].record()
            st = fn(*args)
            if st != 0:
                raise Q.QuasarError(st)
            if events is not None:
                events[i][1].record()


# ----------------------------------------------------------------- clocks --

class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.dev = device_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.dev), f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        smax = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[j] for r in rows for j in range(4)
                          if r[5 + j].lower() in ("active", "1")})
        power = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": reasons, "samples": len(rows),
                "power_w_max": max(power) if power else None}


# ------------------------------------------------------------- CPU oracle --

def cpu_oracle_rate(wlo, budget_s=12.0, seed=0):
    """The fp64 oracle as it stands, on this host's cores, over a bounded
    sample of the workload: the leading groups of each tensor of layer 0,
    sized to take about budget_s seconds.  Returns (weights/s, cores, desc)."""
    import oracle
    oracle.build()
    cores = oracle.get_threads()
    specs = wlo.tensors[:7]
    gsize = wlo.group if wlo.fmt in ("int", "lut") else 16

    def run(n_per_tensor):
        total, t_run = 0, 0.0
        for j, spec in enumerate(specs):
            n = min(spec.numel, n_per_tensor) // gsize * gsize
            d = WL.random_groups(n // gsize, gsize, seed=seed * 1000 + j, dist=wlo.w_dist,
                                 g_dtype=wlo.g_dtype)
            w = d["w"].numpy()
            g = d["g"].float().numpy()
            v = d["v"].numpy()
            t0 = time.perf_counter()
            h = oracle.ema(v, g, wlo.beta2)
            if wlo.fmt == "int":
                oracle.recon_int(w, h, wlo.group, wlo.bits, list(wlo.clip))
            elif wlo.fmt == "lut":  # the sample as 8-row strips of 8x64 blocks
                oracle.recon_lut(w.reshape(8, -1), h.reshape(8, -1), list(wlo.clip))
            else:
                _, sT = oracle.tensor_scale(w)
                oracle.recon_nvfp4(w, h, sT, list(wlo.clip))
            t_run += time.perf_counter() - t0
            total += n
        return total, t_run

    n0 = 1 << 15
    total, t = run(n0)
    per = max(t / total, 1e-12)
    n1 = int(min(budget_s / per / len(specs), 1 << 24))
    n1 = max(n1, n0)
    total, t = run(n1)
    desc = (f"{n1 // gsize} groups per tensor shape of one layer, same value distributions, "
            f"{total} weights in {t:.1f} s")
    return total / t, cores, desc


# ------------------------------------------------------------------- main --

def kernel_source_hash():
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2608_13966_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode())
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(kernel_tag):
    """From the committed summary of one ncu capture, if it was taken on the
    current kernel sources (else None): DRAM bytes per weight
    (dram__bytes_read.sum + dram__bytes_write.sum over the weights that launch
    processed) and, where recorded, the issue-slot and FMA-pipe utilisation
    (smsp__issue_active and sm__pipe_fma_cycles_active, % of peak)."""
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(path):
        return None
    want = kernel_source_hash()
    with open(path) as f:
        for line in f:
            parts = line.split()
            if len(parts) >= 3 and parts[0] == kernel_tag and parts[1] == want:
                out = {"bytes_per_weight": float(parts[2])}
                if len(parts) >= 5:
                    out["issue_active_pct"] = float(parts[3])
                    out["fma_pipe_pct"] = float(parts[4])
                return out
    return None


def timed_steps(step, n_launch_calls, steps, warmup, world):
    for _ in range(warmup):
        step.run()
    torch.cuda.synchronize()
    barrier(world)
    events = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(n_launch_calls)] for _ in range(steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    start.record()
    for k in range(steps):
        step.run(events[k])
    end.record()
    torch.cuda.synchronize()
    barrier(world)
    # a kernel that gave up on a wait leaves its outputs incomplete: such a
    # run has measured nothing
    st = Q.quasar_get_device_status(None)
    if st != Q.QuasarStatus.OK:
        raise Q.QuasarError(st)
    total_ms = start.elapsed_time(end)
    kernel_ms = sum(s.elapsed_time(e) for ev in events for (s, e) in ev)
    return total_ms, kernel_ms


def clamp_set_size(bits, clip):
    """The clamp-set size the library's integer kernel runs with for this
    candidate list (the largest of 4, 2, 1 consecutive slots whose sets all
    admit one code clamp; the library's own rule, restated to name the
    kernel in the report)."""
    if os.environ.get("QUASAR_HOIST", "1") == "0":
        return 1
    f = [float(np.float32(clip[min(k, len(clip) - 1)])) for k in range(32)]
    J = ((1 << bits) - 1) >> 1
    for size in (4, 2):
        if all(J * max(f[s:s + size]) * 1.001 < (J + 1) * min(f[s:s + size]) * 0.999
               for s in range(0, 32, size)):
            return size
    return 1


def host_link(host, dev, s_in, s_out, reps=5):
    """Pinned-copy rates of this machine's host link on one layer's e2e buffers:
    host-to-device (w, g, v into slot 0), device-to-host (r, v', a, b, index
    out of slot 1), and both at once on two streams, as the pipeline overlaps
    them (GB/s; the best of `reps` runs, since other tenants of the host can
    slow a single run)."""
    def run(inb, outb):
        return min(run1(inb, outb) for _ in range(reps))

    def run1(inb, outb):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        if inb:
            with torch.cuda.stream(s_in):
                for h, d in zip(host[0], dev[0]):
                    for k in ("w", "g", "v"):
                        d[k].copy_(h[k], non_blocking=True)
        if outb:
            with torch.cuda.stream(s_out):
                for h, d in zip(host[1], dev[1]):
                    for k in ("r", "v", "a", "b", "idx"):
                        h[k].copy_(d[k], non_blocking=True)
        torch.cuda.synchronize()
        return time.perf_counter() - t0

    nin = sum(h[k].numel() * h[k].element_size() for h in host[0] for k in ("w", "g", "v"))
    nout = sum(h[k].numel() * h[k].element_size() for h in host[1] for k in ("r", "v", "a", "b", "idx"))
    run1(True, True)
    t_in, t_out, t_both = run(True, False), run(False, True), run(True, True)
    return {"h2d_gbs": nin / t_in / 1e9, "d2h_gbs": nout / t_out / 1e9,
            "both_gbs": (nin + nout) / t_both / 1e9}


def e2e_rate(wlo, steps, device, stream, n_slots=2):
    """Same metric through the C ABI with HOST buffers: every step copies each
    tensor's w, g, v from pinned host memory, reconstructs, and reads r, v',
    a, b and the kept index back.  Layers are pipelined over three streams
    (host-to-device copies of layer L+1, the batched reconstruction of layer
    L, device-to-host copies of layer L-1) with two device slots and two
    pinned host buffer sets, each reused every other layer (the bytes moved
    are those of all 32 layers)."""
    import ctypes
    lib = Q.load()
    n_layers = len(wlo.tensors) // 7
    specs = wlo.tensors[:7]
    host, dev = [[] for _ in range(n_slots)], [[] for _ in range(n_slots)]
    for spec in specs:
        d = WL.make_tensor(wlo, spec, device=device)
        n = spec.numel
        for slot in range(n_slots):
            h = {k: v.cpu().pin_memory() for k, v in d.items()}
            h["r"] = torch.empty((spec.rows, spec.cols), dtype=torch.bfloat16).pin_memory()
            h["a"] = torch.empty(n // wlo.group, dtype=torch.float32).pin_memory()
            h["b"] = torch.empty(n // wlo.group, dtype=torch.float32).pin_memory()
            h["idx"] = torch.empty(n // wlo.group, dtype=torch.uint8).pin_memory()
            host[slot].append(h)
            dev[slot].append({k: torch.empty_like(v, device=device) for k, v in h.items()})
        del d
    h2d = sum(h[k].numel() * h[k].element_size() for h in host[0] for k in ("w", "g", "v")) * n_layers
    d2h = sum(h[k].numel() * h[k].element_size() for h in host[0]
              for k in ("r", "v", "a", "b", "idx")) * n_layers
    elements = sum(s.numel for s in wlo.tensors)
    clip = (ctypes.c_float * len(wlo.clip))(*wlo.clip)
    descs = [Q.int_tensor_array([
        {"w": d["w"], "g": d["g"], "v": d["v"], "r": d["r"], "codes": None, "a": d["a"],
         "b": d["b"], "cand_idx": d["idx"], "rows": sp.rows, "cols": sp.cols}
        for d, sp in zip(dev[slot], specs)]) for slot in range(n_slots)]
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    ev = {name: [torch.cuda.Event() for _ in range(n_slots)] for name in ("in", "comp", "out")}
    started = [False] * n_slots

    def one_step():
        for layer in range(n_layers):
            slot = layer % n_slots
            with torch.cuda.stream(s_in):
                if started[slot]:
                    s_in.wait_event(ev["out"][slot])  # the slot's previous layer is out
                for h, d in zip(host[slot], dev[slot]):
                    for k in ("w", "g", "v"):
                        d[k].copy_(h[k], non_blocking=True)
                ev["in"][slot].record(s_in)
            stream.wait_event(ev["in"][slot])
            st = lib.quasar_recon_int_batch(ctypes.cast(descs[slot], ctypes.c_void_p), 7, Q.BF16,
                                            wlo.beta2, wlo.bits, wlo.group, clip, len(wlo.clip),
                                            Q.BF16, stream.cuda_stream)
            if st != 0:
                raise Q.QuasarError(st)
            ev["comp"][slot].record(stream)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev["comp"][slot])
                for h, d in zip(host[slot], dev[slot]):
                    for k in ("r", "v", "a", "b", "idx"):
                        h[k].copy_(d[k], non_blocking=True)
                ev["out"][slot].record(s_out)
            started[slot] = True
        torch.cuda.synchronize()

    one_step()
    t0 = time.perf_counter()
    for _ in range(steps):
        one_step()
    dt = (time.perf_counter() - t0) / steps
    link = host_link(host, dev, s_in, s_out)
    # the copies alone need at least this long: in at the one-way rate, out
    # at its rate, and both over the link's two-way rate
    bound = max(h2d / link["h2d_gbs"], d2h / link["d2h_gbs"], (h2d + d2h) / link["both_gbs"]) / 1e9
    link["copy_bound_ms"] = bound * 1e3
    link["frac_of_copy_bound"] = bound / dt
    return {"value": elements / dt, "unit": "weights/s", "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "ms_per_step": dt * 1e3, "host_link": link,
            "how": "one quasar_recon_int_batch call per layer on pinned host buffers: H2D of "
                   "w/g/v, the call, D2H of r/v/a/b/idx, pipelined over three streams with two "
                   "device slots, all inside the timed region"}


def reference_arm(args, world, rank):
    """The oracle, as it stands, on the host cores (rank 0 only)."""
    if rank != 0:
        return
    wlo = WL.workload(args.workload)
    rates = []
    desc = cores = None
    for i in range(args.warmup + args.steps):
        rate, cores, desc = cpu_oracle_rate(wlo, budget_s=args.ref_budget)
        if i >= args.warmup:
            rates.append(rate)
    value = statistics.median(rates)
    n = sum(s.numel for s in wlo.tensors)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "weights/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": n / value * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": wlo.notes, "elements": n,
                       "timing": "sampled and extrapolated: each step times the oracle on a "
                                 "bounded sample of every tensor shape of layer 0 (%s); "
                                 "ms_per_step is the whole workload at that rate" % desc},
            "cpu_baseline": {"value": value, "unit": "weights/s", "cores": cores, "kind": "oracle",
                             "sample": desc},
            "e2e": {"value": value, "unit": "weights/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# What limits each kernel (from its ncu profiles): the integer kernel is bound
# by instruction issue -- the candidate loop by the FP32 (FMA) pipe, the
# per-group selection, fit and output work by dependent latency -- with DRAM
# well short of its peak; the HBM roofline above is the target's measure.
LIMITER = {"int": "instruction issue: FMA pipe in the candidate loop, dependent latency in the "
                  "per-group work; DRAM below its peak (profiles/)",
           "nvfp4": "instruction issue (E2M1/E4M3 conversions and direct error sums)",
           "lut": "instruction issue (per-index table sums)"}


def alu_roofline(wlo, weights, launch_ms, clk):
    """The FP32-pipe view of an integer launch: algorithmic FP32 operations
    (8 per weight and candidate -- code, its clamp, three moment products and
    their sums -- plus 25 per weight for the EMA, the range, the fixed sums,
    the output code and r; an FMA counts once) over the launch time, against
    the SMs' FP32 lanes (128 an SM) at the median SM clock under load."""
    if wlo.fmt != "int" or launch_ms <= 0:
        return None
    props = torch.cuda.get_device_properties(torch.cuda.current_device())
    mhz = (clk or {}).get("sm_mhz") or 2070.0
    peak = props.multi_processor_count * 128 * mhz * 1e6 / 1e12
    ops = 8 * len(wlo.clip) + 25
    achieved = ops * weights / (launch_ms / 1e3) / 1e12
    return {"achieved": achieved, "peak": peak, "unit": "T FP32 ops/s", "frac": achieved / peak,
            "ops_per_weight": ops}


# The paper-shaped configurations other than the 32-layer step, each timed
# on its own: one 256x1024 fp32 matrix (INT4; launch-bound, reported in us,
# L2 flushed between calls), one Llama-3.1-8B-shaped layer (INT3), one
# Qwen3-8B-shaped layer (INT2 group 64, 16 candidates), one Llama layer
# (NVFP4).  Codes are written, as these configurations specify.
CONFIGS = (("config1_single_int4", "single_int4"), ("config2_llama_layer_int3", "llama_layer_int3"),
           ("config3_qwen_layer_int2", "qwen_layer_int2"), ("config4_llama_layer_nvfp4", "llama_layer_nvfp4"))


def config_entries(device, stream, hbm_peak, reps=20, warm=10):
    out = {}
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=device)  # twice the L2
    for key, name in CONFIGS:
        wlo = WL.workload(name)
        model = Model(wlo, device)
        st = Step(model, wlo, stream)
        small = model.elements * 10 < (1 << 28)
        times = []
        with torch.cuda.stream(stream):
            for i in range(warm + reps):
                if small:
                    flush.zero_()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                st.run()
                e1.record()
                torch.cuda.synchronize()
                if i >= warm:
                    times.append(e0.elapsed_time(e1))
        status = Q.quasar_get_device_status(None)
        if status != Q.QuasarStatus.OK:
            raise Q.QuasarError(status)
        ms = statistics.median(times)
        b = bytes_per_step(wlo, model.elements)
        out[key] = {"workload": wlo.notes, "elements": model.elements, "ms_per_call": ms,
                    "us_per_call": ms * 1e3, "weights_per_s": model.elements / (ms / 1e3),
                    "hbm_gbs": b / (ms / 1e3) / 1e9, "frac_of_8tbs": b / (ms / 1e3) / 1e9 / NOMINAL_HBM_GBS,
                    "frac_of_measured": b / (ms / 1e3) / 1e9 / hbm_peak,
                    "bytes_per_weight": b / model.elements, "calls": reps,
                    "l2": "flushed between calls" if small else "inputs larger than L2",
                    "launch_bound": small}
        del st, model
        torch.cuda.empty_cache()
    del flush
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llama_int3")
    ap.add_argument("--sweep", default="llama_int2,llama_int4,llama_nvfp4,llama_nvfp4_amax,"
                                       "llama_int3_adamw,llama_nvfp4_adamw,llama_lut,llama_int4_sym")
    ap.add_argument("--configs", type=int, default=1, help="time the per-config entries (0: skip)")
    ap.add_argument("--layers", type=int, default=0,
                    help="keep only the first N layers of the workload (0: all)")
    ap.add_argument("--sweep-steps", type=int, default=10)
    ap.add_argument("--e2e-steps", type=int, default=2)
    ap.add_argument("--e2e-slots", type=int, default=2)
    ap.add_argument("--cpu-budget", type=float, default=12.0)
    ap.add_argument("--ref-budget", type=float, default=8.0)
    args = ap.parse_args()

    world, rank = dist_setup(args.gpus)
    if args.impl == "reference":
        reference_arm(args, world, rank)
        return

    device = torch.device("cuda", torch.cuda.current_device())
    stream = torch.cuda.Stream()
    hbm_peak, peak_kind = peaks()
    wlo = WL.workload(args.workload)
    if args.layers > 0:
        # the first N layers of the workload (small cases for the profiler)
        wlo = dataclasses.replace(wlo, tensors=tuple(t for t in wlo.tensors if t.layer < args.layers))
    model = Model(wlo, device, shard=rank)
    torch.cuda.synchronize()
    n_el = model.elements

    clocks = ClockSampler(torch.cuda.current_device())
    step = Step(model, wlo, stream)
    with torch.cuda.stream(stream):
        clocks.start()
        total_ms, kernel_ms = timed_steps(step, len(step.calls), args.steps, args.warmup, world)
        clk = clocks.stop()
    total_ms = max_over_ranks(total_ms, world)
    ms_per_step = total_ms / args.steps
    step_bytes = bytes_per_step(wlo, n_el)
    value = world * n_el / (ms_per_step / 1e3)
    achieved = step_bytes * args.steps / (kernel_ms / 1e3) / 1e9
    hbm_gbs = step_bytes / (ms_per_step / 1e3) / 1e9

    sweep = {}
    for name in [s for s in args.sweep.split(",") if s]:
        # llama_nvfp4_amax: the NVFP4 step with every tensor's absmax supplied
        # (no absmax pass: 16.125 bytes a weight instead of 20.125)
        amax_supplied = name == "llama_nvfp4_amax"
        sw = WL.workload("llama_nvfp4" if amax_supplied else name)
        st = Step(model, sw, stream, amax_supplied=amax_supplied)
        with torch.cuda.stream(stream):
            t_ms, k_ms = timed_steps(st, len(st.calls), args.sweep_steps, 2, world)
        t_ms = max_over_ranks(t_ms, world)
        b = bytes_per_step(sw, n_el, amax_supplied)
        sweep[name] = {"ms_per_step": t_ms / args.sweep_steps,
                       "weights_per_s": world * n_el / (t_ms / args.sweep_steps / 1e3),
                       "hbm_gbs": b / (t_ms / args.sweep_steps / 1e3) / 1e9,
                       "kernel_gbs": b * args.sweep_steps / (k_ms / 1e3) / 1e9,
                       "frac_of_measured": b / (t_ms / args.sweep_steps / 1e3) / 1e9 / hbm_peak,
                       "bytes_per_weight": b / n_el}

    e2e = None
    configs = None
    if args.e2e_steps > 0 and rank == 0 or args.configs:
        del model
        torch.cuda.empty_cache()
    if args.configs and rank == 0:
        # the paper-shaped configurations beside the sweep's formats (the
        # 32-layer INT3 step itself is this line's headline)
        configs = config_entries(device, stream, hbm_peak)
        sweep.update(configs)
    if args.e2e_steps > 0 and rank == 0:
        torch.cuda.empty_cache()
        e2e = e2e_rate(wlo, args.e2e_steps, device, stream, args.e2e_slots)
        e2e["value"] *= world

    cpu = None
    if rank == 0 and world == 1 and args.cpu_budget > 0:
        rate, cores, desc = cpu_oracle_rate(wlo, budget_s=args.cpu_budget)
        cpu = {"value": rate, "unit": "weights/s", "cores": cores, "kind": "oracle", "sample": desc}

    if rank != 0:
        return
    # per-launch figures: the average launch of the step (the step's tensors
    # differ in size; bytes and time both scale with the weights processed)
    if wlo.fmt == "int":
        tag = "k_recon_int_g%d_k%d%s" % (wlo.group, len(wlo.clip), "_adamw" if wlo.adamw else "")
        ss = clamp_set_size(wlo.bits, wlo.clip)
        if wlo.adamw and ss == 2:
            ss = 1
        kname = "k_recon_int<%d,%d,256,%s,false,%d> (one launch per step)" % (
            wlo.group // 4, (len(wlo.clip) + 7) // 8, "true" if wlo.adamw else "false", ss)
    else:
        tag = ("k_recon_lut_k%d" if wlo.fmt == "lut" else "k_recon_nvfp4_k%d") % len(wlo.clip)
        kname = ("k_recon_lut<256>" if wlo.fmt == "lut" else "k_recon_nvfp4<1,256>") + \
            " (one launch per step)"
    prof = profiled_traffic(tag)
    traffic = None if prof is None else prof["bytes_per_weight"] * n_el / len(step.calls)
    line = {
        "metric": METRIC, "value": value, "unit": "weights/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic",
        "config": {"workload": wlo.notes, "elements": n_el, "tensors": len(wlo.tensors),
                   "bits": wlo.bits, "group": wlo.group, "clip_candidates": len(wlo.clip),
                   "g_dtype": DTYPE_NAME[wlo.g_dtype], "r_dtype": DTYPE_NAME[wlo.r_dtype],
                   "codes": "written" if wlo.with_codes else "not written",
                   "l2": "inputs larger than L2 (%.0f GB read per step)" % (n_el * 10 / 1e9),
                   "parallelism": "replicas" if world > 1 else "single GPU"},
        "hbm_gbs": hbm_gbs, "frac_of_8tbs": hbm_gbs / NOMINAL_HBM_GBS,
        "frac_of_measured_copy": hbm_gbs / hbm_peak,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
                     "frac": achieved / hbm_peak, "traffic": traffic,
                     "peak_kind": peak_kind,
                     "kernel": kname,
                     "bytes_per_weight": step_bytes / n_el,
                     "launch_bytes": step_bytes / len(step.calls),
                     "launch_ms": kernel_ms / args.steps / len(step.calls),
                     "traffic_tag": tag,
                     "limiter": LIMITER.get(wlo.fmt),
                     "ncu_pipes": None if prof is None or "fma_pipe_pct" not in prof else
                     {"issue_active": prof["issue_active_pct"] / 100,
                      "fma_pipe": prof["fma_pipe_pct"] / 100,
                      "source": "profiles/traffic.txt (one ncu capture of one layer)"},
                     "alu": alu_roofline(wlo, n_el / len(step.calls),
                                         kernel_ms / args.steps / len(step.calls), clk)},
        "cpu_baseline": cpu, "e2e": e2e,
        "gpu_launches": len(step.calls) * step.launches_per_call * args.steps,
        "clocks": clk, "sweep": sweep,
    }
    print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
