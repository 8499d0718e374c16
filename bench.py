#!/usr/bin/env python3
"""Benchmark of the OffQ W4A4 linear path on GB300.

One step = one pass of the whole hot path over one batch of synthetic input of
the workload: the activation quantizer (online block Hadamard where the site
has one, offsets, 4-bit codes) on every layer input, the seven W4A4 GEMMs with
the fused dequant + offset epilogue (q, k, v, o, gate, up, down), and the KV4
quantizer on the K and V projections. Weights are prepared once, offline.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl reference]

Prints one JSON line (rank 0). ``value`` is the whole-job W4A4 linear
throughput in TOPS (2*T*N*K integer multiply-adds per layer) with inputs
resident in HBM; ``e2e`` is the same metric through the public API with the
inputs copied from pinned host memory and the final output read back inside
the timed region. ``--impl reference`` times the CPU oracle instead.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import platform
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import workloads as W  # noqa: E402

METRIC = "W4A4 OffQ linear TOPS (% dense INT8 peak); act-quant GB/s (% of HBM BW)"
UNIT = "TOPS"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
FP8_PER_BF16 = 2.0   # nominal dense fp8 / bf16 tensor ratio (4.5 / 2.25 PFLOP/s)
L2_FLUSH_BYTES = 512 << 20


def _env_int(name, default):
    try:
        return int(os.environ.get(name, default))
    except ValueError:
        return default


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                "source": "measured"}
    except (OSError, KeyError, ValueError):
        return dict(FALLBACK_PEAKS, source="fallback")


def workload_by_name(name: str) -> W.Workload:
    if name in W.WORKLOADS:
        return W.WORKLOADS[name]
    if name.startswith("decode_t"):
        return W.decode_workload(int(name[len("decode_t"):]))
    raise SystemExit(f"unknown workload {name}")


def gemm_ops(w: W.Workload, T: int) -> float:
    return float(sum(2.0 * T * l.N * l.K for l in w.layers))


def rank_seed_base(rank: int) -> int:
    """Seed offset of a rank's token batch: each rank quantizes and multiplies its own
    synthetic batch (weak scaling, no exchange between ranks in the data path)."""
    return rank * 1000


def reduce_over_ranks(values, dist=None, device=None):
    """Each value's maximum over all ranks: the slowest rank sets the job's time."""
    if dist is None:
        return [float(v) for v in values]
    import torch
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.tolist()]


def job_tops(ops_per_rank: float, world: int, ms: float) -> float:
    """Whole-job TOPS: the operations all ranks performed over the slowest rank's time."""
    return ops_per_rank * world / (ms * 1e-3) / 1e12


def sites(w: W.Workload):
    """Distinct layer inputs: (site name, K, rotate, [layers fed])."""
    out = []
    seen = {}
    for l in w.layers:
        key = {"q": "attn_in", "k": "attn_in", "v": "attn_in", "o": "attn_out", "gate": "mlp_in",
               "up": "mlp_in", "down": "down_in"}.get(l.name, l.name)
        if key not in seen:
            seen[key] = len(out)
            out.append([key, l.K, l.rotate, []])
        out[seen[key]][3].append(l)
    return out


# ---------------------------------------------------------------------------
# Clock sampling during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        self.lines = []
        self.error = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "20",
                 "-i", str(self.dev)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.first = threading.Event()
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            # nvidia-smi needs a moment to start; its first sample predates the timed region.
            self.first.wait(timeout=5.0)
            self.lines = []
        except OSError as e:
            self.error = str(e)
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.perf_counter(), line.strip()))
            self.first.set()

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.thread.join(timeout=5)

    def summary(self, t0=None, t1=None):
        """Median SM clock, maximum clock, power and throttle reasons of the
        samples taken between host times t0 and t1 (all samples by default)."""
        lines = [ln for t, ln in self.lines if (t0 is None or t >= t0) and (t1 is None or t <= t1)]
        if self.error or not lines:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0,
                    "note": self.error or "no nvidia-smi samples"}
        sm, smax, power, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
                power.append(float(parts[3]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm), "power_w_max": max(power)}


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------

class GpuStep:
    """Device buffers of one layer step and the library calls that make the step."""

    def __init__(self, w: W.Workload, T: int, device, seed_base: int = 0):
        import torch
        from paper_2606_07116_gb300 import offq as Q
        self.torch, self.Q, self.w, self.T, self.device = torch, Q, w, T, device
        dt = torch.bfloat16 if w.x_dtype == "bf16" else torch.float32
        self.sites = []
        for i, (name, K, rotate, layers) in enumerate(sites(w)):
            dev = device_activations(T, K, w, seed=seed_base + 10 + i, device=device).to(dt)
            host = dev.cpu().pin_memory()
            dev_alt = dev.clone()  # end-to-end steps alternate between two input buffers
            g = W.block_for(K)
            codes = torch.empty((Q.padded_rows(T), K // 2), dtype=torch.uint8, device=device)
            scale = torch.empty((T,), dtype=torch.float32, device=device)
            off = torch.empty((T, K // g), dtype=torch.float32, device=device)
            flags = (Q.OFFQ_ROTATE if rotate else 0) | Q.OFFQ_OFFSET
            gemms = []
            for l in layers:
                wt = device_weights(l.N, l.K, seed=seed_base + 100 + len(self.sites) * 10 + len(gemms), device=device)
                wc, ws, wr = Q.prepare_weight(wt, g, rotate=l.rotate)
                del wt
                out = torch.empty((T, l.N), dtype=torch.bfloat16, device=device)
                gemms.append({"layer": l, "codes": wc, "scale": ws, "rowsum": wr, "out": out})
            self.sites.append({"name": name, "K": K, "g": g, "flags": flags, "host": host, "dev": dev,
                               "dev_alt": dev_alt, "consumed": [None, None],
                               "codes": codes, "scale": scale, "off": off, "gemms": gemms,
                               "in_bytes": dev.element_size()})
        self.kv = []
        if w.kv_heads:
            H, hd = w.kv_heads, w.head_dim
            for site in self.sites:
                for gm in site["gemms"]:
                    if gm["layer"].name in ("k", "v"):
                        rot = gm["layer"].name == "k"    # K takes the per-head online Hadamard H3
                        flags = (Q.OFFQ_ROTATE if rot else 0) | Q.OFFQ_OFFSET
                        self.kv.append({"src": gm["out"], "H": H, "hd": hd, "flags": flags,
                                        "codes": torch.empty((T, H, hd // 2), dtype=torch.uint8, device=device),
                                        "scale": torch.empty((T, H), dtype=torch.float32, device=device),
                                        "off": torch.empty((T, H), dtype=torch.float32, device=device)})
        last = self.sites[-1]["gemms"][-1]["out"]
        self.result = last
        self.result_host = torch.empty(last.shape, dtype=last.dtype).pin_memory()
        self.copy_stream = torch.cuda.Stream(device)
        self.parity = 0
        torch.cuda.synchronize(device)

    def launches_per_step(self):
        return len(self.sites) + sum(len(s["gemms"]) for s in self.sites) + len(self.kv)

    def quant_bytes(self):
        T = self.T
        return sum(T * s["K"] * s["in_bytes"] + T * s["K"] // 2 + 4 * T + 4 * T * (s["K"] // s["g"])
                   for s in self.sites)

    def kv_bytes(self):
        T = self.T
        return sum(T * k["H"] * k["hd"] * 2 + T * k["H"] * (k["hd"] // 2) + 8 * T * k["H"] for k in self.kv)

    def run(self, stream, timers=None, h2d=False, d2h=False):
        Q, torch = self.Q, self.torch
        T = self.T

        def rec(kind):
            if timers is None:
                return None
            e = torch.cuda.Event(enable_timing=True)
            e.record(stream)
            timers.setdefault(kind, []).append(e)
            return e

        kv_done = False
        ready = {}
        if h2d:
            # All of the step's inputs are on the host at its start: copy them on a
            # side stream, each into the buffer its last use has finished reading.
            par = self.parity
            for s in self.sites:
                dst = s["dev_alt"] if par else s["dev"]
                if s["consumed"][par] is not None:
                    self.copy_stream.wait_event(s["consumed"][par])
                with torch.cuda.stream(self.copy_stream):
                    dst.copy_(s["host"], non_blocking=True)
                    ev = torch.cuda.Event()
                    ev.record(self.copy_stream)
                ready[s["name"]] = (dst, ev)
            self.parity ^= 1
        for s in self.sites:
            x = s["dev"]
            if h2d:
                x, ev = ready[s["name"]]
                stream.wait_event(ev)
            rec("quant")
            Q.offq_quantize_act(x, T, s["K"], x.stride(0), s["g"], s["flags"], s["codes"],
                                s["scale"], s["off"], stream)
            rec("quant")
            if h2d:
                done = torch.cuda.Event()
                done.record(stream)
                s["consumed"][par] = done
            for gm in s["gemms"]:
                l = gm["layer"]
                rec("gemm")
                Q.offq_w4a4_linear(s["codes"], s["scale"], s["off"], T, l.N, l.K, s["g"], gm["codes"],
                                   gm["scale"], gm["rowsum"], gm["out"], gm["out"].stride(0), None, stream)
                rec("gemm")
            if not kv_done and any(g["layer"].name == "v" for g in s["gemms"]):
                for k in self.kv:
                    rec("kv4")
                    Q.offq_kv4_quantize(k["src"], T, k["H"], k["hd"], k["src"].stride(0), k["flags"], k["codes"],
                                        k["scale"], k["off"], stream)
                    rec("kv4")
                kv_done = True
        if d2h:
            self.result_host.copy_(self.result, non_blocking=True)


class GroupStep:
    """The same layers through the per-group asymmetric path (the paper's
    evaluated activation setting: groups of 128 with zero-points): per site the
    group quantizer (with the site's rotation), then its layers' group GEMMs."""

    def __init__(self, w: W.Workload, T: int, device, seed_base: int = 0):
        import torch
        from paper_2606_07116_gb300 import offq as Q
        self.torch, self.Q, self.T = torch, Q, T
        dt = torch.bfloat16 if w.x_dtype == "bf16" else torch.float32
        self.sites = []
        for i, (name, K, rotate, layers) in enumerate(sites(w)):
            x = device_activations(T, K, w, seed=seed_base + 10 + i, device=device).to(dt)
            g = W.block_for(K)
            G = K // Q.GROUP
            gemms = []
            for l in layers:
                wt = device_weights(l.N, l.K, seed=seed_base + 100 + len(self.sites) * 10 + len(gemms), device=device)
                wc, ws, _ = Q.prepare_weight(wt, g, rotate=l.rotate)
                del wt
                gemms.append({"layer": l, "codes": wc, "scale": ws, "gsum": Q.weight_group_sums(wc, l.N, l.K),
                              "out": torch.empty((T, l.N), dtype=torch.bfloat16, device=device)})
            self.sites.append({"K": K, "g": g, "flags": Q.OFFQ_ROTATE if rotate else 0, "x": x,
                               "codes": torch.empty((Q.padded_rows(T), K // 2), dtype=torch.uint8, device=device),
                               "scale": torch.empty((T, G), dtype=torch.float32, device=device),
                               "zero": torch.empty((T, G), dtype=torch.float32, device=device),
                               "gemms": gemms})
        torch.cuda.synchronize(device)

    def launches_per_step(self):
        return len(self.sites) + sum(len(s["gemms"]) for s in self.sites)

    def quant_bytes(self):
        T = self.T
        return sum(T * s["K"] * s["x"].element_size() + T * s["K"] // 2 + 8 * T * (s["K"] // self.Q.GROUP)
                   for s in self.sites)

    def run(self, stream, timers=None):
        Q, torch, T = self.Q, self.torch, self.T

        def rec(kind):
            if timers is not None:
                e = torch.cuda.Event(enable_timing=True)
                e.record(stream)
                timers.setdefault(kind, []).append(e)

        for s in self.sites:
            rec("quant")
            Q.offq_quantize_act_group(s["x"], T, s["K"], s["x"].stride(0), s["g"], Q.GROUP, s["flags"],
                                      s["codes"], s["scale"], s["zero"], stream)
            rec("quant")
            for gm in s["gemms"]:
                l = gm["layer"]
                rec("gemm")
                Q.offq_w4a4_linear_group(s["codes"], s["scale"], s["zero"], T, l.N, l.K, Q.GROUP, gm["codes"],
                                         gm["scale"], gm["gsum"], gm["out"], gm["out"].stride(0), stream)
                rec("gemm")


class MxStep:
    """The same layers in MXFP4 with the offsets as zero-points (Sec. 3.4's
    extension to micro-scaled formats): per site the MX quantizer (rotation and
    offsets as the main path), then its layers' MX GEMMs (E2M1 codes widened to
    exact E4M3 with their 32-channel shifts, the offsets' rank-G epilogue)."""

    def __init__(self, w: W.Workload, T: int, device, seed_base: int = 0):
        import torch
        from paper_2606_07116_gb300 import offq as Q
        self.torch, self.Q, self.T = torch, Q, T
        dt = torch.bfloat16 if w.x_dtype == "bf16" else torch.float32
        self.sites = []
        for i, (name, K, rotate, layers) in enumerate(sites(w)):
            x = device_activations(T, K, w, seed=seed_base + 10 + i, device=device).to(dt)
            g = W.block_for(K)
            gemms = []
            for l in layers:
                wt = device_weights(l.N, l.K, seed=seed_base + 100 + len(self.sites) * 10 + len(gemms), device=device)
                wc, wsh, wsc, wsum = Q.prepare_weight_mx(wt, g, rotate=l.rotate)
                del wt
                gemms.append({"layer": l, "codes": wc, "shifts": wsh, "scale": wsc, "offsum": wsum,
                              "out": torch.empty((T, l.N), dtype=torch.bfloat16, device=device)})
            self.sites.append({"K": K, "g": g, "flags": (Q.OFFQ_ROTATE if rotate else 0) | Q.OFFQ_OFFSET, "x": x,
                               "codes": torch.empty((Q.padded_rows(T), K // 2), dtype=torch.uint8, device=device),
                               "shifts": torch.empty((Q.mx_shift_bytes(T, K),), dtype=torch.uint8, device=device),
                               "scale": torch.empty((T,), dtype=torch.float32, device=device),
                               "off": torch.empty((T, K // g), dtype=torch.float32, device=device),
                               "gemms": gemms})
        torch.cuda.synchronize(device)

    def launches_per_step(self):
        return len(self.sites) + sum(len(s["gemms"]) for s in self.sites)

    def quant_bytes(self):
        T = self.T
        return sum(T * s["K"] * s["x"].element_size() + T * s["K"] // 2 + T * s["K"] // 32 + 4 * T
                   + 4 * T * (s["K"] // s["g"]) for s in self.sites)

    def run(self, stream, timers=None):
        Q, torch, T = self.Q, self.torch, self.T

        def rec(kind):
            if timers is not None:
                e = torch.cuda.Event(enable_timing=True)
                e.record(stream)
                timers.setdefault(kind, []).append(e)

        for s in self.sites:
            rec("quant")
            Q.offq_quantize_act_mx(s["x"], T, s["K"], s["x"].stride(0), s["g"], s["flags"], s["codes"],
                                   s["shifts"], s["scale"], s["off"], stream)
            rec("quant")
            for gm in s["gemms"]:
                l = gm["layer"]
                rec("gemm")
                Q.offq_mx_linear(s["codes"], s["shifts"], s["scale"], s["off"], T, l.N, l.K, s["g"], gm["codes"],
                                 gm["shifts"], gm["scale"], gm["offsum"], gm["out"], gm["out"].stride(0), stream)
                rec("gemm")


def time_variant_path(step_cls, w, T, device, args, rank, flush_l2, barrier, stream):
    """Step time and per-kernel rates of a variant path (same protocol as the main step)."""
    import torch
    from paper_2606_07116_gb300 import offq as Q
    gstep = step_cls(w, T, device, seed_base=rank_seed_base(rank))
    for _ in range(args.warmup):
        flush_l2()
        gstep.run(stream)
    steps = args.steps
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    barrier()
    torch.cuda.synchronize(device)
    for i in range(steps):
        flush_l2()
        starts[i].record(stream)
        gstep.run(stream)
        ends[i].record(stream)
    torch.cuda.synchronize(device)
    dev_ms = sum(s.elapsed_time(e) for s, e in zip(starts, ends))
    timers = {}
    kb = max(1, min(steps, 50))
    for _ in range(kb):
        flush_l2()
        gstep.run(stream, timers=timers)
    torch.cuda.synchronize(device)
    st = Q.offq_get_device_status(stream)
    if st != Q.OFFQ_OK:
        raise RuntimeError(f"device status after {step_cls.__name__}: {Q.status_string(st)}")
    gemm_ms = sum(_pair_times(timers["gemm"])) / kb
    quant_ms = sum(_pair_times(timers["quant"])) / kb
    return gstep, dev_ms / steps, gemm_ms, quant_ms


def time_key_rotation(w, T, device, args, flush_l2, stream):
    """The key cache under a dense per-head rotation M (U3 P3 H3 in place of H3)
    and the query-side rotation, on the workload's key / query shapes."""
    import torch
    from paper_2606_07116_gb300 import offq as Q
    H, hd = w.kv_heads, w.head_dim
    g = torch.Generator(device="cpu").manual_seed(7)
    # Any orthonormal M exercises the kernel identically: a seeded random one.
    rot = torch.linalg.qr(torch.randn((H, hd, hd), generator=g, dtype=torch.float64))[0].to(torch.float32)
    rot = rot.to(device).contiguous()
    k = torch.randn((T, H, hd), generator=g).to(torch.bfloat16).to(device)
    q = torch.randn((T, H, hd), generator=g).to(torch.bfloat16).to(device)
    codes = torch.empty((T, H, hd // 2), dtype=torch.uint8, device=device)
    scale = torch.empty((T, H), dtype=torch.float32, device=device)
    off = torch.empty((T, H), dtype=torch.float32, device=device)
    qo = torch.empty((T, H, hd), dtype=torch.bfloat16, device=device)
    # M is fixed per model: its three bf16 parts are prepared once, offline.
    prep = torch.empty((H, Q.KEY_ROTATION_BYTES), dtype=torch.uint8, device=device)
    Q.offq_prepare_key_rotation(rot, H, hd, prep, stream)
    # The structured form of the method's M = U3 P3 H3: a seeded top-1 direction
    # and a permutation keeping channel 0 first per head.
    v = torch.randn((H, hd), generator=g)
    perm = torch.stack([torch.cat([torch.zeros(1, dtype=torch.int64), 1 + torch.randperm(hd - 1, generator=g)])
                        for _ in range(H)]).to(torch.int32)
    refl = Q.prepare_key_reflection(v, perm, device=device)
    ts = {"k": [], "q": [], "k_split": [], "k_refl": []}
    for i in range(3 + max(1, min(args.steps, 50))):
        e = [torch.cuda.Event(enable_timing=True) for _ in range(8)]
        flush_l2()
        e[0].record(stream)
        Q.offq_kv4_quantize_prepared(k, T, H, hd, k.stride(0), prep, Q.OFFQ_OFFSET, codes, scale, off, stream)
        e[1].record(stream)
        flush_l2()
        e[2].record(stream)
        Q.offq_rotate_heads_prepared(q, T, H, hd, q.stride(0), prep, qo, qo.stride(0), stream)
        e[3].record(stream)
        flush_l2()
        e[4].record(stream)
        Q.offq_kv4_quantize_rotated(k, T, H, hd, k.stride(0), rot, Q.OFFQ_OFFSET, codes, scale, off, stream)
        e[5].record(stream)
        flush_l2()
        e[6].record(stream)
        Q.offq_kv4_quantize_reflected(k, T, H, hd, k.stride(0), refl, Q.OFFQ_OFFSET, codes, scale, off, stream)
        e[7].record(stream)
        torch.cuda.synchronize(device)
        if i >= 3:
            ts["k"].append(e[0].elapsed_time(e[1]))
            ts["q"].append(e[2].elapsed_time(e[3]))
            ts["k_split"].append(e[4].elapsed_time(e[5]))
            ts["k_refl"].append(e[6].elapsed_time(e[7]))
    st = Q.offq_get_device_status(stream)
    if st != Q.OFFQ_OK:
        raise RuntimeError(f"device status after the key rotation: {Q.status_string(st)}")
    k_ms = sum(ts["k"]) / len(ts["k"])
    q_ms = sum(ts["q"]) / len(ts["q"])
    ks_ms = sum(ts["k_split"]) / len(ts["k_split"])
    kr_ms = sum(ts["k_refl"]) / len(ts["k_refl"])
    flops = 2.0 * T * H * hd * hd
    # Algorithmic bytes: bf16 keys in, 4-bit codes and fp32 scale / offset out, M read once.
    kb = T * H * (hd * 2 + hd // 2 + 8) + H * hd * hd * 4
    peaks = load_peaks()
    gbs = kb / (k_ms * 1e-3) / 1e9
    return {
        "what": "key cache under a dense per-head rotation M = U3 P3 H3 (offq_kv4_quantize_prepared: bf16 keys on "
                "the tensor cores, M's three bf16 parts prepared offline) and the query rotation "
                "(offq_rotate_heads_prepared), "
                f"{T} tokens x {H} heads x {hd}; per-call events, L2 flushed before each call; "
                "kv4_rotated_split_us: offq_kv4_quantize_rotated, which splits M in every CTA; "
                "kv4_reflected_us: offq_kv4_quantize_reflected, M in structured form (one +-1 product of N = 144)",
        "kv4_rotated_us": round(k_ms * 1e3, 2), "rotate_q_us": round(q_ms * 1e3, 2),
        "kv4_rotated_split_us": round(ks_ms * 1e3, 2), "kv4_reflected_us": round(kr_ms * 1e3, 2),
        "rotation_tflops": round(flops / (k_ms * 1e-3) / 1e12, 2),
        "roofline": {"bound": "hbm", "kernel": "rotate_heads_mma_kernel (tcgen05.mma kind::f16)",
                     "achieved": round(gbs, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
                     "frac": round(gbs / peaks["hbm_gbs"], 4), "bytes": kb},
    }


def time_builder(device, args, flush_l2, stream):
    """The offline transform builder on a calibration set of 64 sequences x 512
    tokens x 4096 channels (bf16), fusing a 11008 x 4096 weight."""
    import torch
    from paper_2606_07116_gb300 import offq as Q
    S, L, D, N, G, iters = 64, 512, 4096, 11008, 1, 100
    g = torch.Generator(device="cpu").manual_seed(11)
    x = torch.randn((S, L, D), generator=g).to(torch.bfloat16).to(device)
    W = (torch.randn((N, D), generator=g) * 0.02).to(device)
    peaks = load_peaks()

    def timed(fn, reps):
        ts = []
        for i in range(2 + reps):
            flush_l2()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            out = fn()
            e1.record(stream)
            torch.cuda.synchronize(device)
            if i >= 2:
                ts.append(e0.elapsed_time(e1))
        return sum(ts) / len(ts), out

    reps = max(1, min(args.steps, 20))
    tok_ms, (_, rows) = timed(lambda: Q.top1_tokens(x, stream), reps)
    dir_ms, (v, _) = timed(lambda: Q.top1_direction(rows, iters=iters, stream=stream), max(1, reps // 4))
    mag = Q.column_absmax(Q.reflect_rows(rows, v, stream), stream)
    perm = Q.sorted_grouping(mag, G)
    fuse_ms, _ = timed(lambda: Q.fuse_rotation(W, v, perm, D // G, stream), reps)
    st = Q.offq_get_device_status(stream)
    if st != Q.OFFQ_OK:
        raise RuntimeError(f"device status after the builder: {Q.status_string(st)}")
    tok_bytes = S * L * D * 2 + S * D * 4
    fuse_bytes = 2 * N * D * 4
    tok_gbs = tok_bytes / (tok_ms * 1e-3) / 1e9
    return {
        "what": f"offline transform builder: top-1 L-inf tokens of {S} x {L} x {D} bf16, {iters} power-iteration "
                f"steps on the {S} x {D} selection, fusion of U1 P1 H1 (g = {D // G}) into a {N} x {D} fp32 weight; "
                "per-call events",
        "top1_tokens_us": round(tok_ms * 1e3, 2), "top1_tokens_gbs": round(tok_gbs, 1),
        "direction_us": round(dir_ms * 1e3, 2),
        "fuse_us": round(fuse_ms * 1e3, 2), "fuse_gbs": round(fuse_bytes / (fuse_ms * 1e-3) / 1e9, 1),
        "roofline": {"bound": "hbm", "kernel": "top1_scan_kernel", "achieved": round(tok_gbs, 1),
                     "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": round(tok_gbs / peaks["hbm_gbs"], 4)},
    }


def device_weights(N: int, K: int, seed: int, device, std: float = 0.02):
    """Weights W [N, K] ~ N(0, std^2) in fp32, drawn on the device (seeded): the
    recipe of workloads.weights, for timing (the 70B layers hold 0.86 G weights)."""
    import torch
    gen = torch.Generator(device=device).manual_seed(seed)
    return torch.randn((N, K), generator=gen, device=device) * std


def device_activations(T: int, K: int, w: W.Workload, seed: int, device):
    """The workload's activation recipe drawn on the device (seeded): N(0, 1) or
    Student-t(3) entries, plus the outlier channels with per-token jitter, in bf16.
    For timing only: rows this large take too long to draw on the host."""
    import torch
    gen = torch.Generator(device=device).manual_seed(seed)
    x = torch.randn((T, K), generator=gen, device=device)
    if w.dist == "student_t3":
        chi2 = sum(torch.randn((T, K), generator=gen, device=device) ** 2 for _ in range(3))
        x /= torch.sqrt(chi2 / 3.0)
    if w.n_out > 0 and w.mult != 0.0:
        amp = w.mult * (1.0 + 0.1 * torch.randn((T,), generator=gen, device=device))
        for c in W.outlier_channels(K, w.n_out):
            x[:, c] = amp
    return x.to(torch.bfloat16)


def time_quant_sites(device, args, flush_l2, stream):
    """The activation quantizer alone on the prefill inputs of the larger Llama
    shapes (Llama-3-8B MLP at 4096 tokens, Llama-2-70B at 8192 tokens): rows
    long enough that the launch cost no longer hides the kernel's streaming
    rate. Per-call events, L2 flushed before each call."""
    import torch
    from paper_2606_07116_gb300 import offq as Q
    peaks = load_peaks()
    out = {"what": "offq_quantize_act alone on the prefill layer inputs of the Llama-3-8B MLP and Llama-2-70B "
                   "shapes (bf16 in; offsets on; the block Hadamard on the down-proj inputs); per-call events, "
                   "L2 flushed before each call", "sites": []}
    best = None
    reps = max(1, min(args.steps, 20))
    for wname in ("llama3_8b_mlp", "llama2_70b"):
        w = workload_by_name(wname)
        T = w.T
        shapes = set()
        for i, (name, K, rotate, _) in enumerate(sites(w)):
            if (K, rotate) in shapes:
                continue  # a site of the same shape was timed already
            shapes.add((K, rotate))
            g = W.block_for(K)
            x = device_activations(T, K, w, seed=1000 + i, device=device)
            codes = torch.empty((Q.padded_rows(T), K // 2), dtype=torch.uint8, device=device)
            scale = torch.empty((T,), dtype=torch.float32, device=device)
            off = torch.empty((T, K // g), dtype=torch.float32, device=device)
            flags = (Q.OFFQ_ROTATE if rotate else 0) | Q.OFFQ_OFFSET
            ts = []
            for r in range(2 + reps):
                flush_l2()
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                Q.offq_quantize_act(x, T, K, x.stride(0), g, flags, codes, scale, off, stream)
                e1.record(stream)
                torch.cuda.synchronize(device)
                if r >= 2:
                    ts.append(e0.elapsed_time(e1))
            ms = sum(ts) / len(ts)
            nbytes = T * K * 2 + T * K // 2 + 4 * T + 4 * T * (K // g)
            gbs = nbytes / (ms * 1e-3) / 1e9
            site = {"workload": wname, "site": name, "T": T, "K": K, "g": g, "rotate": bool(rotate),
                    "us": round(ms * 1e3, 2), "bytes": nbytes, "gbs": round(gbs, 1),
                    "frac": round(gbs / peaks["hbm_gbs"], 4)}
            out["sites"].append(site)
            if best is None or nbytes > best["bytes"]:
                best = site
            del x, codes, scale, off
    st = Q.offq_get_device_status(stream)
    if st != Q.OFFQ_OK:
        raise RuntimeError(f"device status after the quantizer sites: {Q.status_string(st)}")
    torch.cuda.empty_cache()
    out["roofline"] = {"bound": "hbm", "kernel": "offq_quantize_act on the largest site "
                                                 f"({best['workload']} {best['site']}, {best['T']} x {best['K']})",
                       "achieved": best["gbs"], "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": best["frac"]}
    return out


def time_decode(device, args, flush_l2, stream):
    """The decode sweep on Llama-2-7B shapes: T = 1, 8, 32, 64 tokens through the
    activation quantizer, one 4096 -> 11008 W4A4 linear and the KV4 quantizer of
    32 heads x 128 per token (keys with the per-head Hadamard, values offset
    only). Per-call events, L2 flushed before each call, so every GEMM streams
    its 22.5 MB of weight codes from HBM."""
    import torch
    from paper_2606_07116_gb300 import offq as Q
    peaks = load_peaks()
    K, N, H, hd = 4096, 11008, 32, 128
    g = W.block_for(K)
    wt = torch.from_numpy(W.weights(N, K, seed=501)).to(device)
    wc, ws, wr = Q.prepare_weight(wt, g, rotate=False)
    del wt
    w_bytes = wc.numel() + 4 * N + 4 * N * (K // g)
    # The GEMM is timed back to back over copies of the weight codes that together
    # hold more than twice the L2, so each call streams its weights from HBM.
    l2 = torch.cuda.get_device_properties(device).L2_cache_size
    n_sets = max(2, -(-2 * l2 // w_bytes) + 1)
    sets = [(wc.clone(), ws.clone(), wr.clone()) for _ in range(n_sets)]
    reps = max(1, min(args.steps, 50))
    calls = n_sets * max(4, reps // n_sets + 1)
    out = {"what": "decode on Llama-2-7B shapes: offq_quantize_act + offq_w4a4_linear 4096 -> 11008 + "
                   "offq_kv4_quantize of the keys (rotated) and values. GEMM: back-to-back calls (queued behind a spin kernel) cycling over "
                   f"{n_sets} copies of the weights ({n_sets * w_bytes / 1e6:.0f} MB, over twice the L2), events "
                   "around the batch; quantizer and KV4: per-call events, L2 flushed before each call; "
                   "weight_gbs = weight codes, scales and row sums read by the GEMM / its time",
           "points": []}
    best = None
    for T in W.DECODE_BATCHES:
        x = W.to_bf16(W.activations(T, K, seed=600 + T, n_out=4, mult=100.0)).to(device)
        kv = W.to_bf16(W.kv_heads(T, H, hd, seed=700 + T)).to(device).reshape(T, H * hd)
        codes = torch.empty((Q.padded_rows(T), K // 2), dtype=torch.uint8, device=device)
        scale = torch.empty((T,), dtype=torch.float32, device=device)
        off = torch.empty((T, K // g), dtype=torch.float32, device=device)
        y = torch.empty((T, N), dtype=torch.bfloat16, device=device)
        kc = torch.empty((T, H, hd // 2), dtype=torch.uint8, device=device)
        ks = torch.empty((T, H), dtype=torch.float32, device=device)
        ko = torch.empty((T, H), dtype=torch.float32, device=device)
        ts = {"quant": [], "kv4": []}
        for r in range(3 + reps):
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
            flush_l2()
            ev[0].record(stream)
            Q.offq_quantize_act(x, T, K, x.stride(0), g, Q.OFFQ_OFFSET, codes, scale, off, stream)
            ev[1].record(stream)
            flush_l2()
            ev[2].record(stream)
            Q.offq_kv4_quantize(kv, T, H, hd, kv.stride(0), Q.OFFQ_ROTATE | Q.OFFQ_OFFSET, kc, ks, ko, stream)
            Q.offq_kv4_quantize(kv, T, H, hd, kv.stride(0), Q.OFFQ_OFFSET, kc, ks, ko, stream)
            ev[3].record(stream)
            torch.cuda.synchronize(device)
            if r >= 3:
                ts["quant"].append(ev[0].elapsed_time(ev[1]))
                ts["kv4"].append(ev[2].elapsed_time(ev[3]))
        for i in range(2 * n_sets):  # warm-up
            wci, wsi, wri = sets[i % n_sets]
            Q.offq_w4a4_linear(codes, scale, off, T, N, K, g, wci, wsi, wri, y, y.stride(0), None, stream)
        flush_l2()
        # The stream waits on a spin kernel while the host enqueues the whole batch,
        # so the events time the GPU's back-to-back execution, not the launch rate.
        torch.cuda._sleep(int(2e6 + 1e5 * calls))
        g0 = torch.cuda.Event(enable_timing=True)
        g1 = torch.cuda.Event(enable_timing=True)
        g0.record(stream)
        for i in range(calls):
            wci, wsi, wri = sets[i % n_sets]
            Q.offq_w4a4_linear(codes, scale, off, T, N, K, g, wci, wsi, wri, y, y.stride(0), None, stream)
        g1.record(stream)
        torch.cuda.synchronize(device)
        qm, km = (sum(ts[k]) / len(ts[k]) for k in ("quant", "kv4"))
        gm = g0.elapsed_time(g1) / calls
        gbs = w_bytes / (gm * 1e-3) / 1e9
        pt = {"T": T, "quant_us": round(qm * 1e3, 2), "gemm_us": round(gm * 1e3, 2), "kv4_us": round(km * 1e3, 2),
              "gemm_tops": round(2.0 * T * N * K / (gm * 1e-3) / 1e12, 3), "weight_gbs": round(gbs, 1),
              "weight_frac": round(gbs / peaks["hbm_gbs"], 4)}
        out["points"].append(pt)
        if best is None or pt["weight_gbs"] > best["weight_gbs"]:
            best = pt
    st = Q.offq_get_device_status(stream)
    if st != Q.OFFQ_OK:
        raise RuntimeError(f"device status after the decode sweep: {Q.status_string(st)}")
    del sets
    kern = "w4a4_gemv_kernel (dp4a, T <= 4)" if best["T"] <= 4 else "w4a4_decode_kernel (tcgen05, 4 < T <= 64)"
    out["roofline"] = {"bound": "hbm", "kernel": f"{kern} weight stream (T = {best['T']})",
                       "achieved": best["weight_gbs"], "peak": peaks["hbm_gbs"], "unit": "GB/s",
                       "frac": best["weight_frac"], "bytes": w_bytes}
    return out


def time_gemm_shape(device, args, flush_l2, stream):
    """One offq_w4a4_linear shape alone (T, K -> N, block g; codes made without
    the rotation unless g < K), per-call events after an L2 flush: a side
    measurement for profiling, not the bench line."""
    import torch
    from paper_2606_07116_gb300 import offq as Q
    T, K, N = (int(v) for v in args.gemm.split(",")[:3])
    g = W.block_for(K)
    w = workload_by_name(args.workload)
    x = device_activations(T, K, w, seed=900, device=device)
    codes, scale, off = Q.quantize_act(x, g, rotate=g < K, offset=True)
    del x
    wc, ws, wr = Q.prepare_weight(device_weights(N, K, seed=901, device=device), g, rotate=g < K)
    y = torch.empty((T, N), dtype=torch.bfloat16, device=device)
    reps = max(1, min(args.steps, 50))
    ts = []
    for r in range(args.warmup + reps):
        flush_l2()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        Q.offq_w4a4_linear(codes, scale, off, T, N, K, g, wc, ws, wr, y, N, None, stream)
        e1.record(stream)
        torch.cuda.synchronize(device)
        if r >= args.warmup:
            ts.append(e0.elapsed_time(e1))
    st = Q.offq_get_device_status(stream)
    if st != Q.OFFQ_OK:
        raise RuntimeError(f"device status after the GEMM: {Q.status_string(st)}")
    ms = sum(ts) / len(ts)
    peaks = load_peaks()
    tflops = 2.0 * T * N * K / (ms * 1e-3) / 1e12
    peak = peaks["bf16_tflops"] * FP8_PER_BF16
    return {"gemm": {"T": T, "K": K, "N": N, "g": g}, "us": round(ms * 1e3, 2), "tflops": round(tflops, 1),
            "peak": peak, "frac": round(tflops / peak, 4), "reps": reps}


def _pair_times(events):
    return [events[i].elapsed_time(events[i + 1]) for i in range(0, len(events), 2)]


def load_traffic_record():
    path = os.path.join(ROOT, "profiles", "gemm_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except (OSError, ValueError):
        return None
    if rec.get("gemm_src_sha256") != gemm_source_digest():
        return None
    return rec


def gemm_source_digest() -> str:
    """sha256 over the per-token GEMM's sources (gemm.cu, then pair_common.cuh)."""
    h = hashlib.sha256()
    for name in ("gemm.cu", "pair_common.cuh"):
        with open(os.path.join(ROOT, "paper_2606_07116_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def run_gpu(args, rank, world, local_rank):
    import torch
    import __graft_entry__ as G
    G.build()
    from paper_2606_07116_gb300 import offq as Q

    device = torch.device("cuda", local_rank)
    torch.cuda.set_device(device)
    w = workload_by_name(args.workload)
    T = w.T
    step = GpuStep(w, T, device, seed_base=rank_seed_base(rank))
    stream = torch.cuda.current_stream(device)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=device)

    def flush_l2():
        # Write a buffer four times the L2, then read its first half back, so
        # the step starts with no workload data and no dirty lines in L2.
        flush.zero_()
        flush[:L2_FLUSH_BYTES // 2].view(torch.int32).amax()  # a read with no temporary

    dist = None
    if world > 1:
        import torch.distributed as dist_mod
        dist = dist_mod

    def barrier():
        if dist is not None:
            dist.barrier()

    for _ in range(args.warmup):
        flush_l2()
        step.run(stream)
    torch.cuda.synchronize(device)
    st = Q.offq_get_device_status(stream)
    if st != Q.OFFQ_OK:
        raise RuntimeError(f"device status after warm-up: {Q.status_string(st)}")

    # ---- timed region: K steps, inputs resident, L2 flushed between steps ----
    # Events bracket whole steps only: an event recorded between two launches
    # would keep the second from being scheduled during the first one's tail.
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    barrier()
    torch.cuda.synchronize(device)
    # The sampler runs through the timed region and the per-call phase that the
    # roofline's kernel times come from; each window is summarised on its own.
    clk = ClockSampler(device.index if device.index is not None else 0).__enter__()
    wall0 = time.perf_counter()
    for i in range(args.steps):
        flush_l2()
        starts[i].record(stream)
        step.run(stream)
        ends[i].record(stream)
    torch.cuda.synchronize(device)
    wall1 = time.perf_counter()
    barrier()
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    dev_ms = sum(step_ms)

    # ---- per-kernel durations: the same steps again, an event pair around every call ----
    timers = {}
    kb = max(1, min(args.steps, 50))
    wall2 = time.perf_counter()
    for _ in range(kb):
        flush_l2()
        step.run(stream, timers=timers)
    torch.cuda.synchronize(device)
    wall3 = time.perf_counter()
    clk.__exit__(None, None, None)
    gemm_ms = sum(_pair_times(timers["gemm"])) * args.steps / kb
    quant_ms = sum(_pair_times(timers["quant"])) * args.steps / kb
    kv_ms = sum(_pair_times(timers.get("kv4", []))) * args.steps / kb if timers.get("kv4") else 0.0
    st = Q.offq_get_device_status(stream)
    if st != Q.OFFQ_OK:
        raise RuntimeError(f"device status after the timed region: {Q.status_string(st)}")

    # ---- end to end through the public API: pinned H2D inputs, D2H result ----
    e2e_steps = max(1, args.steps)
    barrier()
    torch.cuda.synchronize(device)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    step.copy_stream.wait_event(e0)  # no copy starts before the timed region does
    for _ in range(e2e_steps):
        step.run(stream, h2d=True, d2h=True)
    e1.record(stream)
    torch.cuda.synchronize(device)
    barrier()
    e2e_ms = e0.elapsed_time(e1) / e2e_steps

    ms_per_step, e2e_ms = reduce_over_ranks([dev_ms / args.steps, e2e_ms], dist, device)
    ops = gemm_ops(w, T)
    value = job_tops(ops, world, ms_per_step)
    e2e_value = job_tops(ops, world, e2e_ms)

    peaks = load_peaks()
    # The GEMMs are timed per call (an event pair around each launch), so the
    # burst rate is their denominator.
    fp8_peak = peaks["bf16_tflops"] * FP8_PER_BF16
    group = mxfp4 = None
    if not args.no_group:
        gstep, g_ms, g_gemm_ms, g_quant_ms = time_variant_path(GroupStep, w, T, device, args, rank, flush_l2,
                                                               barrier, stream)
        (g_ms,) = reduce_over_ranks([g_ms], dist, device)
        g_gemm_tflops = ops / (g_gemm_ms * 1e-3) / 1e12
        g_quant_gbs = gstep.quant_bytes() / (g_quant_ms * 1e-3) / 1e9
        group = {
            "what": "the paper's evaluated activation setting on the same layers: per-group (128) asymmetric "
                    "activations with zero-points (offq_quantize_act_group + offq_w4a4_linear_group), no KV4",
            "value": round(job_tops(ops, world, g_ms), 3), "unit": UNIT, "ms_per_step": round(g_ms, 4),
            "roofline": {"bound": "tensor", "kernel": "w4a4_group_gemm_kernel (tcgen05.mma kind::f8f6f4, "
                                                      "per-group scaling in the scaler warps)",
                         "achieved": round(g_gemm_tflops, 2), "peak": round(fp8_peak, 1), "unit": "TFLOP/s",
                         "frac": round(g_gemm_tflops / fp8_peak, 4), "gemm_ms_per_step": round(g_gemm_ms, 4)},
            "act_quant": {"value": round(g_quant_gbs, 1), "unit": "GB/s", "peak": peaks["hbm_gbs"],
                          "frac": round(g_quant_gbs / peaks["hbm_gbs"], 4), "ms_per_step": round(g_quant_ms, 4),
                          "bytes_per_step": gstep.quant_bytes()},
            "gpu_launches": gstep.launches_per_step() * args.steps,
        }
        del gstep
        mstep, m_ms, m_gemm_ms, m_quant_ms = time_variant_path(MxStep, w, T, device, args, rank, flush_l2,
                                                               barrier, stream)
        (m_ms,) = reduce_over_ranks([m_ms], dist, device)
        m_gemm_tflops = ops / (m_gemm_ms * 1e-3) / 1e12
        m_quant_gbs = mstep.quant_bytes() / (m_quant_ms * 1e-3) / 1e9
        mxfp4 = {
            "what": "the same layers in MXFP4 (E2M1 codes, a power-of-two scale per 32 channels) with the offsets "
                    "as zero-points: offq_quantize_act_mx + offq_mx_linear, no KV4",
            "value": round(job_tops(ops, world, m_ms), 3), "unit": UNIT, "ms_per_step": round(m_ms, 4),
            "roofline": {"bound": "tensor", "kernel": "w4a4_gemm_kernel<MX> (tcgen05.mma kind::f8f6f4, codes "
                                                      "widened with their block shifts in the converter warps)",
                         "achieved": round(m_gemm_tflops, 2), "peak": round(fp8_peak, 1), "unit": "TFLOP/s",
                         "frac": round(m_gemm_tflops / fp8_peak, 4), "gemm_ms_per_step": round(m_gemm_ms, 4)},
            "act_quant": {"value": round(m_quant_gbs, 1), "unit": "GB/s", "peak": peaks["hbm_gbs"],
                          "frac": round(m_quant_gbs / peaks["hbm_gbs"], 4), "ms_per_step": round(m_quant_ms, 4),
                          "bytes_per_step": mstep.quant_bytes()},
            "gpu_launches": mstep.launches_per_step() * args.steps,
        }
        del mstep
    gemm_tflops = ops * args.steps / (gemm_ms * 1e-3) / 1e12
    quant_gbs = step.quant_bytes() * args.steps / (quant_ms * 1e-3) / 1e9
    kv_gbs = step.kv_bytes() * args.steps / (kv_ms * 1e-3) / 1e9 if kv_ms > 0 else None
    traffic = load_traffic_record()
    if rank != 0:
        return None
    line = {
        "metric": METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int4",
        "data": "synthetic (seeded Llama-shaped activations with outlier channels, N(0,0.02) weights)",
        "config": {"workload": w.name, "description": w.description, "tokens": T,
                   "layers": [f"{l.name}:{l.K}->{l.N}" for l in w.layers],
                   "kv4_heads": w.kv_heads, "block_sizes": {str(s['K']): s['g'] for s in step.sites},
                   "out_dtype": "bf16",
                   "l2": "flushed between timed steps (512 MiB write, then 256 MiB of it read back)",
                   "parallelism": f"dp{world} (token batches, no collective in the data path)"},
        "roofline": {"bound": "tensor", "kernel": "w4a4_gemm_kernel (tcgen05.mma kind::f8f6f4)",
                     "achieved": round(gemm_tflops, 2), "peak": round(fp8_peak, 1), "unit": "TFLOP/s",
                     "frac": round(gemm_tflops / fp8_peak, 4),
                     "peak_source": f"{peaks['source']}: bf16 burst {peaks['bf16_tflops']} "
                                    f"x nominal fp8/bf16 ratio {FP8_PER_BF16} (the GEMMs are timed per call)",
                     "traffic": traffic["bytes_per_launch"] if traffic else None,
                     "traffic_note": traffic.get("note") if traffic else "no ncu record for this gemm.cu",
                     "gemm_ms_per_step": round(gemm_ms / args.steps, 4)},
        "act_quant": {"value": round(quant_gbs, 1), "unit": "GB/s", "peak": peaks["hbm_gbs"],
                      "frac": round(quant_gbs / peaks["hbm_gbs"], 4),
                      "ms_per_step": round(quant_ms / args.steps, 4), "bytes_per_step": step.quant_bytes()},
        "kv4": {"value": round(kv_gbs, 1) if kv_gbs else None, "unit": "GB/s",
                "ms_per_step": round(kv_ms / args.steps, 4), "bytes_per_step": step.kv_bytes()},
        "e2e": {"value": round(e2e_value, 3), "unit": UNIT,
                "h2d_bytes_per_step": int(sum(s["host"].numel() * s["host"].element_size() for s in step.sites)),
                "d2h_bytes_per_step": int(step.result.numel() * step.result.element_size()),
                "ms_per_step": round(e2e_ms, 4)},
        "gpu_launches": step.launches_per_step() * args.steps,
        "kernel_timing": f"per-launch durations from {kb} more flushed steps with an event pair around every call",
        "wall_s_timed_region": round(wall1 - wall0, 4),
        "clocks": clk.summary(wall0, wall1),
        "clocks_kernel_timing": clk.summary(wall2, wall3),
    }
    if group is not None:
        line["group_asym"] = group
    if mxfp4 is not None:
        line["mxfp4"] = mxfp4
    if not args.no_group and w.kv_heads and w.head_dim == 128:
        line["kv4_rotated"] = time_key_rotation(w, T, device, args, flush_l2, stream)
    if not args.no_group:
        line["builder"] = time_builder(device, args, flush_l2, stream)
    if not args.no_group and world == 1:
        line["act_quant_prefill"] = time_quant_sites(device, args, flush_l2, stream)
        line["decode"] = time_decode(device, args, flush_l2, stream)
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w, budget_s=args.cpu_budget)
    return line


# ---------------------------------------------------------------------------
# CPU oracle (baseline leg and the reference arm)
# ---------------------------------------------------------------------------

class OracleStep:
    """The same step computed by the float64 oracle on a sample of tokens."""

    def __init__(self, w: W.Workload, T_full: int):
        import oracle as O
        self.O, self.w = O, w
        dt = w.x_dtype
        self.inputs = []
        self.weights = []
        for i, (name, K, rotate, layers) in enumerate(sites(w)):
            x = W.activations(T_full, K, seed=10 + i, dist=w.dist, n_out=w.n_out, mult=w.mult)
            if dt == "bf16":
                x = W.bf16_to_f64(W.to_bf16(x))
            g = W.block_for(K)
            wl = []
            for j, l in enumerate(layers):
                wp = O.prepare_weight(W.weights(l.N, l.K, seed=100 + i * 10 + j).astype(np.float64), g,
                                      rotate=l.rotate)
                wl.append((l, wp))
            self.inputs.append((name, K, g, rotate, x.astype(np.float64)))
            self.weights.append(wl)

    def run(self, rows: np.ndarray):
        O = self.O
        outs = {}
        for (name, K, g, rotate, x), wl in zip(self.inputs, self.weights):
            a = O.quantize_act(x[rows], g, rotate=rotate, offset=True)
            for l, wp in wl:
                y = O.w4a4_linear(a["q"], a["scale"], a["offset"], wp["q"], wp["scale"], wp["offsum"])["y"]
                outs[l.name] = y
        if self.w.kv_heads:
            H, hd = self.w.kv_heads, self.w.head_dim
            for nm, rot in (("k", True), ("v", False)):
                if nm in outs:
                    O.kv4_quantize(outs[nm].reshape(len(rows), H, hd), rotate=rot, offset=True)
        return outs


def _cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_baseline(w: W.Workload, budget_s: float = 15.0):
    ostep = OracleStep(w, w.T)
    rows = W.unit_index_sample(w.T, 8, seed=1)
    ostep.run(rows)  # the first pass warms BLAS threads and the Hadamard cache
    t0 = time.perf_counter()
    ostep.run(rows)
    per_tok = (time.perf_counter() - t0) / len(rows)
    n = int(max(8, min(w.T, budget_s / max(per_tok, 1e-9))))
    rows = W.unit_index_sample(w.T, n, seed=2)
    t0 = time.perf_counter()
    ostep.run(rows)
    dt = time.perf_counter() - t0
    value = gemm_ops(w, len(rows)) / dt / 1e12
    return {"value": value, "unit": UNIT, "cores": _cores(), "kind": "oracle",
            "sample": f"{len(rows)} of {w.T} tokens through every layer (float64 oracle: explicit Hadamard, "
                      f"exact integer GEMM via float64 BLAS, float64 epilogue, KV4), {dt:.1f} s",
            "cpu": platform.processor() or platform.machine()}


def run_reference(args, rank, world):
    if rank != 0:
        return None
    w = workload_by_name(args.workload)
    ostep = OracleStep(w, w.T)
    probe = W.unit_index_sample(w.T, 4, seed=1)
    t0 = time.perf_counter()
    ostep.run(probe)
    per_tok = (time.perf_counter() - t0) / len(probe)
    t0 = time.perf_counter()
    ostep.run(probe)  # a second probe, with BLAS threads and the Hadamard cache warm
    per_tok = min(per_tok, (time.perf_counter() - t0) / len(probe))
    per_step_budget = max(1.0, args.ref_budget / max(1, args.steps + args.warmup))
    n = int(max(4, min(w.T, per_step_budget / max(per_tok, 1e-9))))
    rows = W.unit_index_sample(w.T, n, seed=2)
    for _ in range(args.warmup):
        ostep.run(rows)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        ostep.run(rows)
    dt = (time.perf_counter() - t0) / args.steps
    value = gemm_ops(w, n) / dt / 1e12
    sample = f"{n} of {w.T} tokens per step through every layer and KV4 (float64 oracle)"
    return {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": w.name, "description": w.description, "tokens_per_step": n},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": _cores(), "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--workload", default="llama2_70b")
    ap.add_argument("--impl", default="offq", choices=["offq", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-group", action="store_true", help="skip the per-group asymmetric path's timing")
    ap.add_argument("--cpu-budget", type=float, default=15.0, help="seconds of oracle work for cpu_baseline")
    ap.add_argument("--ref-budget", type=float, default=120.0, help="seconds of oracle work for --impl reference")
    ap.add_argument("--key-rotation-tokens", type=int, default=0,
                    help="time only the key-cache rotation calls, at this many tokens, and print that object "
                         "(a side measurement for profiling, not the bench line)")
    ap.add_argument("--decode", action="store_true",
                    help="time only the decode sweep (1/8/32/64 tokens) and print that object")
    ap.add_argument("--gemm", default="",
                    help="T,K,N: time only offq_w4a4_linear at this shape (bf16 out) and print that object "
                         "(a side measurement for profiling, not the bench line)")
    ap.add_argument("--quant-sites", action="store_true",
                    help="time only the activation quantizer on the larger prefill inputs and print that object "
                         "(a side measurement for profiling, not the bench line)")
    args = ap.parse_args()
    if args.warmup < 3:
        raise SystemExit("--warmup must be at least 3")
    if args.decode:
        import torch
        import __graft_entry__ as G
        G.build()
        device = torch.device("cuda", 0)
        torch.cuda.set_device(device)
        flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=device)

        def flush_l2():
            flush.zero_()
            flush[:L2_FLUSH_BYTES // 2].view(torch.int32).amax()

        print(json.dumps(time_decode(device, args, flush_l2, torch.cuda.current_stream(device))), flush=True)
        return
    if args.gemm:
        import torch
        import __graft_entry__ as G
        G.build()
        device = torch.device("cuda", 0)
        torch.cuda.set_device(device)
        flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=device)

        def flush_l2():
            flush.zero_()
            flush[:L2_FLUSH_BYTES // 2].view(torch.int32).amax()

        print(json.dumps(time_gemm_shape(device, args, flush_l2, torch.cuda.current_stream(device))), flush=True)
        return
    if args.quant_sites:
        import torch
        import __graft_entry__ as G
        G.build()
        device = torch.device("cuda", 0)
        torch.cuda.set_device(device)
        flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=device)

        def flush_l2():
            flush.zero_()
            flush[:L2_FLUSH_BYTES // 2].view(torch.int32).amax()

        print(json.dumps(time_quant_sites(device, args, flush_l2, torch.cuda.current_stream(device))), flush=True)
        return
    if args.key_rotation_tokens > 0:
        import torch
        device = torch.device("cuda", 0)
        torch.cuda.set_device(device)
        w = workload_by_name(args.workload)
        flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=device)

        def flush_l2():
            flush.zero_()
            flush[:L2_FLUSH_BYTES // 2].view(torch.int32).amax()

        print(json.dumps(time_key_rotation(w, args.key_rotation_tokens, device, args, flush_l2,
                                           torch.cuda.current_stream(device))), flush=True)
        return

    world = _env_int("WORLD_SIZE", 1)
    rank = _env_int("RANK", 0)
    local_rank = _env_int("LOCAL_RANK", 0)
    if args.impl == "reference":
        line = run_reference(args, rank, world)
    else:
        if world > 1:
            import torch
            import torch.distributed as dist
            torch.cuda.set_device(local_rank)
            dist.init_process_group("nccl")
        line = run_gpu(args, rank, world, local_rank)
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
    if line is not None and rank == 0:
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
