#!/usr/bin/env python
"""Throughput of the EOGP hot path on GB300.

Headline: one step compresses one batch of B = 32 training examples through all
224 modules of the OLMo-2-7B-shaped stack (32 layers x {q, k, v, o 4096 x
4096; gate, up 4096 -> 11008; down 11008 -> 4096}, T = 2048 tokens, m = 8192
retained first-stage coordinates, k = 2048 PCA coordinates per module) into
one-bit codes: Kronecker rotations, per-example contraction with the
scale-and-gather epilogue, PCA projection, sign packing (Alg. 1 "Storing one
training example"). The retained eigenvector rows of every layer live in
page-locked host memory and are copied one layer ahead of its compute on a side
stream. Inputs are synthetic (Gaussian a and s, Haar eigenbases, power-law
spectra with exponent 1.0), drawn on the device before timing; one input buffer
per module type serves the 32 layers, and each module's inputs (0.5-2 GB) exceed
L2, so no flush is needed.

Consecutive modules alternate between two streams with a workspace each (the
modules are independent), so one module's contraction, projection and pack run
beside the next module's rotations. `value` is examples compressed per second
per layer stack (whole job, all ranks). `e2e` repeats the step through the C-ABI's host-input call
(eogp_compress_layer_host) with a, s and the eigenbases in page-locked host
memory: the call's host-to-device copies and the device-to-host read of the
codes are inside the timed region; the plain host-to-device copy rate of the
same run is reported beside it. `roofline` is that of the rotation kernels,
timed launch by launch with CUDA events in a few profiled steps of the same
configuration after the timed ones (every module on one stream, so that no
launch overlaps another), and `roofline.others` carries the other timed
kernels' rooflines, the
query x train scoring rates included. The GPT-2, OLMo-1B, 32B-gate and fp32
stacks, the scoring workloads and the PCA fit follow in the same line.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--batch B] [--workload NAME]
    python bench.py --impl reference ...   # the CPU oracle on the host cores
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

HEADLINE = "olmo2_7b_bf16"
METRIC = "training examples compressed/sec per layer stack"
PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# Examples per compression call (one step) of each workload's throughput line.
CONFIG_BATCH = {"gpt2_small_bf16": 512, "tiny_f32": 4096, "olmo2_1b_bf16": 128, "olmo2_7b_bf16": 32,
                "olmo2_32b_gate_bf16": 64}
# dram__bytes_read.sum + dram__bytes_write.sum per rotation launch from the committed
# ncu captures (profiles/), as (bytes per launch, examples per launch at capture), or
# None when the kernel changed after the capture. Traffic grows with the examples
# per launch, so it is scaled to the bench's batch.
ROTATE_TRAFFIC = {"gpt2_small_bf16": (1415.1e6, 512), "olmo2_7b_bf16": (267.2e6, 8)}
E2E_BATCH = {"olmo2_7b_bf16": 8, "gpt2_small_bf16": 128}


def score_peak(ks, probes, bf16_burst, peaks_src):
    """Denominator of a one-bit tensor-core scoring rate: the measured rate of the
    MMA the library issues for these module sizes (e2m1 kind::mxf4 when every
    module is a multiple of 256 bits, else e4m3 kind::f8f6f4), as (TFLOP/s,
    source, mode label). Without the probes: the bf16 burst peak times the
    nominal dense ratio (fp8 2x, fp4 6x)."""
    f4 = all(k % 256 == 0 for k in ks)
    if f4:
        mode = "tcgen05 kind::mxf4, +-1 e2m1 operands, unit ue8m0 scales"
        if probes:
            return probes["e2m1_tflops"], "eogp_measure_peaks e2m1", mode
        return 6.0 * bf16_burst, f"6 x {peaks_src} bf16_tflops (nominal fp4 ratio)", mode
    mode = "tcgen05 kind::f8f6f4, +-1 e4m3 operands"
    if probes:
        return probes["e4m3_tflops"], "eogp_measure_peaks e4m3", mode
    return 2.0 * bf16_burst, f"2 x {peaks_src} bf16_tflops (nominal fp8 ratio)", mode


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    except Exception:
        return PEAKS_FALLBACK, "fallback"


# --------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi clock / throttle-reason samples every 200 ms while running."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.idx = None
        try:
            import torch
            self.idx = "GPU-" + str(torch.cuda.get_device_properties(device_index).uuid)
        except Exception:
            vis = os.environ.get("CUDA_VISIBLE_DEVICES")
            self.idx = vis.split(",")[device_index] if vis else str(device_index)
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        rows = []
        with open(self.path) as f:
            for ln in f:
                parts = [x.strip() for x in ln.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i] == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows)}


# ----------------------------------------------------------- workload
def build_stack(w, B, dev, seed):
    """Per-module plans, retained eigenvector rows, PCA directions and inputs
    (one input buffer per module)."""
    import torch
    from paper_2609_37842_gb300 import eogp as E
    from paper_2609_37842_gb300 import synth
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    gh = torch.Generator()
    gh.manual_seed(seed)
    mods = []
    plans = {}
    bases = {}
    Pt = synth.torch_eigvec_rows(w.m, w.k, dev, gh, torch.bfloat16)
    for u, mod in enumerate(w.modules):
        key = (mod.d_in, mod.d_out)
        if key not in plans:
            plans[key] = E.Plan.from_factors(synth.power_spectrum(mod.d_out, w.alpha),
                                             synth.power_spectrum(mod.d_in, w.alpha), w.m,
                                             w.damping_rel)
            inf = plans[key].info()
            # The spectra are sorted, so C and R are index prefixes: the retained rows are
            # the leading eigenvectors of Haar bases (shared by modules of one shape; the
            # work per module does not depend on their values).
            R, C = plans[key].sets()
            assert (C == range(inf.nC)).all() and (R == range(inf.nR)).all()
            bases[key] = (synth.torch_eigvec_rows(mod.d_in, inf.nC, dev, gh, torch.bfloat16),
                          synth.torch_eigvec_rows(mod.d_out, inf.nR, dev, gh, torch.bfloat16))
        plan = plans[key]
        inf = plan.info()
        VA, VS = bases[key]
        a, s = synth.torch_layer_inputs(w, u, B, dev, g)
        desc = E.layer_desc(plan, w.T, w.k, VA, VS, Pt)
        mods.append(dict(desc=desc, a=a, s=s, d_in=mod.d_in, d_out=mod.d_out, nC=inf.nC,
                         nR=inf.nR))
    return mods


def compress_step(mods, E, codes, scales, ws, words):
    for u, md in enumerate(mods):
        E.compress_layer(md["desc"], md["a"], md["s"], E.OUT_CODES,
                         codes=codes[:, u * words:(u + 1) * words], scales=scales[:, u], ws=ws)


def rotate_flops(mods, B, T):
    return sum(2.0 * B * T * (md["d_in"] * md["nC"] + md["d_out"] * md["nR"]) for md in mods)


def _config_stack(name, B, dev, gh, g):
    """Plans, retained eigenvector rows and inputs for one layer's module types of a
    workload; the per-layer inputs are reused by every layer (the work per layer is
    identical, and each module's inputs still exceed L2)."""
    import torch
    from paper_2609_37842_gb300 import eogp as E
    from paper_2609_37842_gb300 import synth
    w = synth.WORKLOADS[name]
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    per_layer = {}
    for u, mod in enumerate(w.modules):
        key = (mod.d_in, mod.d_out, mod.gelu_input, u % 7 if name.startswith("olmo") else u % 4)
        if key in per_layer:
            continue
        if w.spectrum == "channel":
            spec = synth.layer_spec(w, u, 1, 1)
            lamA, lamS = spec.lam_A, spec.lam_S
        else:
            lamA = synth.power_spectrum(mod.d_in, w.alpha)
            lamS = synth.power_spectrum(mod.d_out, w.alpha)
        plan = E.Plan.from_factors(lamS, lamA, w.m, w.damping_rel)
        inf = plan.info()
        R, C = plan.sets()
        if w.spectrum == "channel":
            # permutation eigenbasis: row r of V_A[C] is the unit vector at the channel
            # holding the C[r]-th largest variance
            pa = np.argsort(-spec.chan_A ** 2, kind="stable")
            ps = np.argsort(-spec.chan_S ** 2, kind="stable")
            VA = torch.zeros((inf.nC, mod.d_in), dtype=dt, device=dev)
            VA[torch.arange(inf.nC), torch.from_numpy(pa[C]).long()] = 1
            VS = torch.zeros((inf.nR, mod.d_out), dtype=dt, device=dev)
            VS[torch.arange(inf.nR), torch.from_numpy(ps[R]).long()] = 1
            sa = torch.from_numpy(spec.chan_A).float().to(dev)
            ss = torch.from_numpy(spec.chan_S).float().to(dev)
        else:
            VA = synth.torch_eigvec_rows(mod.d_in, inf.nC, dev, gh, dt)
            VS = synth.torch_eigvec_rows(mod.d_out, inf.nR, dev, gh, dt)
            sa = ss = None
        a, s = synth.torch_layer_inputs(w, u, B, dev, g)
        if sa is not None:
            a = (a.float() * sa).to(dt)
            s = (s.float() * ss).to(dt)
        per_layer[key] = dict(plan=plan, VA=VA, VS=VS, a=a, s=s, d_in=mod.d_in, d_out=mod.d_out,
                              nC=inf.nC, nR=inf.nR)
    keys = []
    for u, mod in enumerate(w.modules):
        keys.append((mod.d_in, mod.d_out, mod.gelu_input, u % 7 if name.startswith("olmo") else u % 4))
    return w, per_layer, keys


def config_setup(name, B, dev):
    """Everything one step of a workload's throughput line launches with: the
    workload, per-module-type plans, retained eigenvector rows and inputs
    (`per_layer`), the module-type key of every module of the stack (`keys`),
    the PCA directions `Pt`, one layer descriptor per module type (`descs`) and
    a workspace for B examples (`ws`). The tests call this too, so that they
    check the launches the bench times."""
    import torch
    from paper_2609_37842_gb300 import eogp as E
    from paper_2609_37842_gb300 import synth
    g = torch.Generator(device=dev)
    g.manual_seed(7)
    gh = torch.Generator()
    gh.manual_seed(7)
    w, per_layer, keys = _config_stack(name, B, dev, gh, g)
    Pt = synth.torch_eigvec_rows(w.m, w.k, dev, gh,
                                 torch.bfloat16 if w.dtype == "bf16" else torch.float32)
    descs = {key: E.layer_desc(L["plan"], w.T, w.k, L["VA"], L["VS"], Pt) for key, L in per_layer.items()}
    ws = E.workspace(max(E.compress_workspace_size(d, B, E.OUT_CODES) for d in descs.values()), dev)
    return dict(w=w, per_layer=per_layer, keys=keys, Pt=Pt, descs=descs, ws=ws)


class Stack:
    """One workload's compression step: B examples through every module of the
    stack into one-bit codes. Consecutive modules alternate between two streams,
    each with its own workspace (the modules are independent), so that one
    module's contraction, projection and pack overlap the next module's
    rotations. With stream_bases the retained eigenvector rows of every layer
    live in page-locked host memory and are copied to the device one layer ahead
    of its compute on a side stream (two device slots)."""

    def __init__(self, name, B, dev, stream_bases=False, modules=0):
        import dataclasses
        import torch
        from paper_2609_37842_gb300 import eogp as E
        self.E = E
        self.name, self.B, self.dev = name, B, dev
        cs = config_setup(name, B, dev)
        self.w, self.per_layer, self.keys, self.Pt, self.descs, self.ws = (
            cs[x] for x in ("w", "per_layer", "keys", "Pt", "descs", "ws"))
        if modules:
            self.keys = self.keys[:modules]
            self.w = dataclasses.replace(self.w, modules=self.w.modules[:modules])
        w = self.w
        self.words = (w.k + 31) // 32
        self.U = len(self.keys)
        self.codes = torch.empty((B, self.U * self.words), dtype=torch.int32, device=dev)
        self.scales = torch.empty((B, self.U), dtype=torch.float32, device=dev)
        self.stream = torch.cuda.current_stream()
        self.streams = [self.stream, torch.cuda.Stream()]
        self.wss = [self.ws, E.workspace(self.ws.numel(), dev)]
        self.nmod_layer = len(set(self.keys))
        self.layers = max(1, self.U // self.nmod_layer) if name.startswith("olmo") else 1
        self.stream_bases = stream_bases and self.layers > 1
        if self.stream_bases:
            pl = self.per_layer
            # page-locked through the library's allocator (huge-page backed): the
            # same memory class the e2e inputs use, which copies at the link rate
            def pinned(t):
                h = E.host_empty(tuple(t.shape), t.dtype)
                h.copy_(t)
                return h
            self.host_one = {k: (pinned(L["VA"]), pinned(L["VS"])) for k, L in pl.items()}
            self.dev_bases = [{k: (torch.empty_like(L["VA"]), torch.empty_like(L["VS"])) for k, L in pl.items()}
                              for _ in range(2)]
            self.slot_descs = [{k: E.layer_desc(pl[k]["plan"], w.T, w.k, self.dev_bases[sl][k][0],
                                                self.dev_bases[sl][k][1], self.Pt) for k in pl} for sl in range(2)]
            self.cstream = torch.cuda.Stream()
            self.landed = [torch.cuda.Event() for _ in range(2)]
            self.freed = [None, None]

    def _module(self, u, desc, single=False):
        L = self.per_layer[self.keys[u]]
        wd = self.words
        i = 0 if single else u % 2
        self.E.compress_layer(desc, L["a"], L["s"], self.E.OUT_CODES, codes=self.codes[:, u * wd:(u + 1) * wd],
                              scales=self.scales[:, u], ws=self.wss[i], stream=self.streams[i])

    def step(self, single=False):
        """One step; `single` keeps every module on the main stream (the profiled
        steps that time each kernel on its own)."""
        import torch
        s0, s1 = self.streams
        s1.wait_stream(s0)  # the step starts after everything before it on the main stream
        if not self.stream_bases:
            for u, key in enumerate(self.keys):
                self._module(u, self.descs[key], single)
            s0.wait_stream(s1)  # and ends after both streams' work
            return

        def issue_copy(layer):
            sl = layer % 2
            if self.freed[sl] is not None:
                for ev in self.freed[sl]:
                    self.cstream.wait_event(ev)
            with torch.cuda.stream(self.cstream):
                for k in self.per_layer:
                    self.dev_bases[sl][k][0].copy_(self.host_one[k][0], non_blocking=True)
                    self.dev_bases[sl][k][1].copy_(self.host_one[k][1], non_blocking=True)
                self.landed[sl].record(self.cstream)
        issue_copy(0)
        for layer in range(self.layers):
            sl = layer % 2
            if layer + 1 < self.layers:
                issue_copy(layer + 1)
            s0.wait_event(self.landed[sl])
            s1.wait_event(self.landed[sl])
            for j in range(self.nmod_layer):
                u = layer * self.nmod_layer + j
                self._module(u, self.slot_descs[sl][self.keys[u]], single)
            evs = (torch.cuda.Event(), torch.cuda.Event())  # the slot is free once both streams are done with it
            evs[0].record(s0)
            evs[1].record(s1)
            self.freed[sl] = evs
        s0.wait_stream(s1)

    def timed(self, steps, warmup, clocks=None, barrier=None, prof_steps=0):
        """Warm-up, then `steps` steps between CUDA events on the main stream
        (modules alternating between the two streams); then `prof_steps` (default:
        min(steps, 3)) steps with every module on the main stream and every library
        launch bracketed by CUDA events, which time each kernel on its own. Returns
        (ms of the timed steps, per-kind kernel times of the profiled steps, clocks,
        profiled steps)."""
        import torch
        E = self.E
        for _ in range(warmup):
            self.step()
        torch.cuda.synchronize()
        E.sync_status()
        if barrier:
            barrier()
        torch.cuda.synchronize()
        if clocks:
            clocks.start()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(self.stream)
        for _ in range(steps):
            self.step()
        e1.record(self.stream)
        torch.cuda.synchronize()
        if barrier:
            barrier()
        clk = clocks.stop() if clocks else None
        E.sync_status()
        prof_steps = prof_steps or min(steps, 3)
        for kk in E.KERNEL_KINDS:
            E.profile_read(kk, reset=True)
        E.profile_enable(True)
        for _ in range(prof_steps):
            self.step(single=True)
        torch.cuda.synchronize()
        E.profile_enable(False)
        E.sync_status()
        kern = {}
        for kk, nm in E.KERNEL_KINDS.items():
            n, kms = E.profile_read(kk, reset=True)
            if n:
                kern[nm] = {"launches": n, "ms": kms}
        ktot = sum(v["ms"] for v in kern.values())
        for v in kern.values():
            v["share"] = v["ms"] / ktot if ktot else None
        return e0.elapsed_time(e1), kern, clk, prof_steps

    def rot_flops(self):
        pl = self.per_layer
        return sum(2.0 * self.B * self.w.T * (pl[k]["d_in"] * pl[k]["nC"] + pl[k]["d_out"] * pl[k]["nR"])
                   for k in self.keys)

    def in_bytes(self):
        pl = self.per_layer
        return sum(2.0 * self.B * self.w.T * (pl[k]["d_in"] + pl[k]["d_out"]) * (2 if self.w.dtype == "f32" else 1)
                   for k in self.keys)

    def summary(self, ms, steps, kern, peaks, prof_steps):
        """examples/s, stack and rotation TFLOP/s, input GB/s (timed steps) and the
        rotation roofline (profiled steps)."""
        w, B = self.w, self.B
        sec = ms / 1000.0
        rot = kern.get("rotate", {"launches": 0, "ms": 0.0})
        rf = self.rot_flops()
        out = {"examples_per_s": B * steps / sec, "ms_per_step": ms / steps, "batch": B,
               "modules": self.U, "T": w.T, "m": w.m, "k": w.k,
               "stack_TFLOPs": rf * steps / sec / 1e12,
               "input_GBps": self.in_bytes() * steps / sec / 1e9,
               "alg_GFLOP_per_example": rf / B / 1e9,
               "input_MB_per_example": self.in_bytes() / B / 1e6,
               "kernels": kern}
        hbm = peaks.get("hbm_gbs") or PEAKS_FALLBACK["hbm_gbs"]
        out["input_frac_of_hbm"] = out["input_GBps"] / hbm
        if rot["launches"]:
            per_launch = rf * prof_steps / rot["launches"]
            avg_ms = rot["ms"] / rot["launches"]
            ach = per_launch / (avg_ms / 1000.0) / 1e12
            peak = peaks.get("bf16_tflops_sustained") or PEAKS_FALLBACK["bf16_tflops_sustained"]
            tr = ROTATE_TRAFFIC.get(self.name)
            out["roofline"] = {"bound": "tensor", "achieved": ach, "peak": peak, "unit": "TFLOP/s",
                               "frac": ach / peak,
                               "traffic": tr[0] * B / tr[1] if tr and self.U == len(self.w.modules) else None,
                               "kernel": "k_tc_rotate / k_tc_rotate2 (Kronecker rotations)",
                               "flops_per_launch": per_launch,
                               "timing": f"CUDA events around each launch in {prof_steps} profiled steps of the same "
                                         "configuration after the timed ones, every module on one stream (the "
                                         "timed steps alternate two streams, so launches overlap there)"}
        if self.stream_bases:
            out["eigenbases"] = "host-pinned, one layer ahead on a side stream"
            out["h2d_bytes_per_step"] = self.layers * sum(2 * (L["VA"].numel() + L["VS"].numel())
                                                          for L in self.per_layer.values())
        if self.layers > 1:
            out["inputs"] = f"one buffer per module type, shared by the {self.layers} layers"
        return out

    def release(self):
        import torch
        for k in list(vars(self)):
            if k not in ("name", "B", "w", "U", "keys", "layers"):
                setattr(self, k, None)
        torch.cuda.empty_cache()


def h2d_link_rate(h, dev, reps=3):
    """Plain host-to-device copy rate of the page-locked host tensor `h` (one of the
    e2e run's own input buffers) with one cudaMemcpyAsync per repetition, GB/s."""
    import torch
    nbytes = h.numel() * h.element_size()
    d = torch.empty(h.shape, dtype=h.dtype, device=dev)
    d.copy_(h, non_blocking=True)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        d.copy_(h, non_blocking=True)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    del d
    return nbytes * reps / (ms / 1000.0) / 1e9


def e2e_run(st, Be, steps, chunk, dev, world, barrier):
    """The step through the public host-input call for several modules
    (eogp_compress_layers_host), all modules of the stack in one call: per module,
    a and s in page-locked host memory (one buffer per module type) and, for
    streamed-eigenbasis stacks, the retained eigenvector rows too (descriptor
    bases_on_host); the call copies each module's inputs chunk by chunk into
    staging sets that alternate between modules, so one module's copies overlap
    the previous module's compute; the step ends with the device-to-host read of
    the stack's codes and scales."""
    import torch
    E = st.E
    w = st.w
    hdt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    host = {}
    hdesc = {}
    bases_bytes = 0
    for key, L in st.per_layer.items():
        ha = E.host_empty((Be, w.T, L["d_in"]), hdt)
        hs = E.host_empty((Be, w.T, L["d_out"]), hdt)
        ha.copy_(L["a"][:Be])
        hs.copy_(L["s"][:Be])
        host[key] = (ha, hs)
        if st.stream_bases:
            hva, hvs = st.host_one[key]
            hdesc[key] = E.layer_desc(L["plan"], w.T, w.k, hva, hvs, st.Pt)
        else:
            hdesc[key] = st.descs[key]
    if st.stream_bases:
        bases_bytes = sum(2 * (st.per_layer[k]["VA"].numel() + st.per_layer[k]["VS"].numel()) for k in st.keys)
    wd = st.words
    ecodes, escales = st.codes[:Be], st.scales[:Be]
    sdescs = [hdesc[key] for key in st.keys]
    sa = [host[key][0] for key in st.keys]
    ss = [host[key][1] for key in st.keys]
    scodes = [ecodes[:, u * wd:(u + 1) * wd] for u in range(len(st.keys))]
    sscales = [escales[:, u] for u in range(len(st.keys))]
    hws = E.workspace(E.compress_layers_host_workspace_size(sdescs, Be, E.OUT_CODES, chunk), dev)
    hcodes = torch.empty(ecodes.shape, dtype=ecodes.dtype, pin_memory=True)
    hscales = torch.empty(escales.shape, dtype=escales.dtype, pin_memory=True)
    h2d = sum(host[k][0].numel() * host[k][0].element_size() + host[k][1].numel() * host[k][1].element_size()
              for k in st.keys) + bases_bytes
    d2h = hcodes.numel() * 4 + hscales.numel() * 4

    def e2e_step():
        E.compress_layers_host(sdescs, sa, ss, E.OUT_CODES, dev, chunk=chunk, codes=scodes, scales=sscales,
                               ws=hws, stream=st.stream)
        hcodes.copy_(ecodes, non_blocking=True)
        hscales.copy_(escales, non_blocking=True)

    e2e_step()
    torch.cuda.synchronize()
    barrier()
    t0 = time.perf_counter()
    for _ in range(steps):
        e2e_step()
    torch.cuda.synchronize()
    ems = (time.perf_counter() - t0) * 1000.0
    E.sync_status()
    if world > 1:
        import torch.distributed as dist
        tt = torch.tensor([ems], device=dev)
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        ems = float(tt.item())
    big = max((t for pair in host.values() for t in pair), key=lambda t: t.numel() * t.element_size())
    link = h2d_link_rate(big, dev)
    rate = h2d * steps / (ems / 1000.0) / 1e9
    out = {"value": world * Be * steps / (ems / 1000.0), "unit": "examples/s", "batch": Be,
           "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": steps,
           "h2d_GBps": rate, "link_GBps": link, "frac_of_link": rate / link if link else None,
           "link": "one cudaMemcpyAsync of the run's largest input buffer (the same page-locked memory), "
                   "3 copies",
           "api": "eogp_compress_layers_host (the stack's modules in one call: host inputs, chunked copies "
                  "inside the call, one module's copies overlapping the previous module's compute)",
           "chunk": chunk or "library default (about 64 MB of inputs)"}
    if st.stream_bases:
        out["eigenbases"] = "page-locked host memory, copied by each call (bases_on_host)"
    del host, hdesc, hws
    torch.cuda.empty_cache()
    return out


def bench_ekfac(dev, d_in, d_out, T, B, reps=3):
    """EK-FAC eigenvalue correction over the full coordinate block of one module:
    examples/s and TFLOP/s (algorithmic: full rotations 2 B T (d_in^2 + d_out^2)
    plus the contraction 2 B T d_in d_out)."""
    import torch
    from paper_2609_37842_gb300 import eogp as E
    from paper_2609_37842_gb300 import synth
    g = torch.Generator(device=dev)
    g.manual_seed(13)
    gh = torch.Generator()
    gh.manual_seed(13)
    VA = synth.torch_eigvec_rows(d_in, d_in, dev, gh, torch.bfloat16)
    VS = synth.torch_eigvec_rows(d_out, d_out, dev, gh, torch.bfloat16)
    a = torch.randn((B, T, d_in), generator=g, device=dev).to(torch.bfloat16)
    s = (0.1 * torch.randn((B, T, d_out), generator=g, device=dev)).to(torch.bfloat16)
    desc = E.ekfac_desc(T, VA, VS)
    sumsq = torch.zeros((d_out, d_in), dtype=torch.float64, device=dev)
    ws = E.workspace(E.ekfac_workspace_size(desc, B), dev)
    E.ekfac_accumulate(desc, a, s, sumsq=sumsq, ws=ws)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        E.ekfac_accumulate(desc, a, s, sumsq=sumsq, accumulate=True, ws=ws)
    e1.record()
    torch.cuda.synchronize()
    E.sync_status()
    ms = e0.elapsed_time(e1) / reps
    flops = 2.0 * B * T * (d_in * d_in + d_out * d_out + d_in * d_out)
    return {"shape": f"{d_in}->{d_out}", "T": T, "batch": B, "ms_per_call": ms,
            "examples_per_s": B / (ms / 1000.0), "alg_TFLOPs": flops / (ms / 1000.0) / 1e12}


def bench_fit(dev, n=10000, m=4096, k=1024):
    """Seconds for the one-time PCA fit (App. B.2) of n fitting rows of m
    first-stage coordinates to k directions (Z drawn on the device with a
    decaying column spectrum)."""
    import torch
    from paper_2609_37842_gb300 import eogp as E
    g = torch.Generator(device=dev)
    g.manual_seed(11)
    col = torch.arange(1, m + 1, device=dev, dtype=torch.float32) ** -0.7
    Z = torch.randn((n, m), generator=g, device=dev) * col
    E.fit_pca(Z[:2048, :1536], 128)   # warm-up (module load, both solvers' kernels)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    Pt, eig = E.fit_pca(Z, k)
    torch.cuda.synchronize()
    E.sync_status()
    sec = time.perf_counter() - t0
    del Z, Pt, eig
    torch.cuda.empty_cache()
    return {"n": n, "m": m, "k": k, "seconds": sec,
            "route": "covariance; tensor-core Gram, subspace iteration with Rayleigh-Ritz"}


# ------------------------------------------------------------ CPU oracle
def _shapes(w):
    shapes = {}
    for u, mod in enumerate(w.modules):
        shapes.setdefault((mod.d_in, mod.d_out), []).append(u)
    return shapes


def _dense_orthogonal(d, rng):
    """A dense orthogonal d x d matrix (I - 2 u u^T)(I - 2 v v^T) for random unit
    u, v: cheap to form at d = 11008, where a Haar draw (QR of a Gaussian) takes
    minutes on the host cores. The oracle's cost does not depend on the values
    of the eigenbases, only on their (dense) shape."""
    u = rng.standard_normal(d)
    v = rng.standard_normal(d)
    u /= np.linalg.norm(u)
    v /= np.linalg.norm(v)
    H = np.eye(d) - 2.0 * np.outer(u, u)
    return H - 2.0 * np.outer(H @ v, v)


class OracleSample:
    """The oracle compressing one example through one module of each distinct shape
    of a workload (inputs prepared once, not timed): dense orthogonal eigenbases
    and P rounded to the workload dtype, the workload's spectra and inputs."""

    def __init__(self, w, seed=1):
        from paper_2609_37842_gb300 import synth
        from oracle import eogp_oracle as O
        self.O, self.w = O, w
        rng = np.random.default_rng(seed)
        qcache = {}

        def q(d):
            if d not in qcache:
                qcache[d] = synth.round_to(_dense_orthogonal(d, rng), w.dtype)
            return qcache[d]
        self.P = synth.round_to(_dense_orthogonal(w.m, rng)[:, :w.k], w.dtype)
        self.cases = []
        for (d_in, d_out), us in _shapes(w).items():
            u = us[0]
            if w.spectrum == "channel":
                sp = synth.layer_spec(w, u, 1, 1)
                lamA, lamS = sp.lam_A, sp.lam_S
            else:
                lamA, lamS = synth.power_spectrum(d_in, w.alpha), synth.power_spectrum(d_out, w.alpha)
            a, s = synth.layer_inputs(w, u, 1)
            self.cases.append(dict(shape=f"{d_in}->{d_out}", count=len(us), QA=q(d_in), QS=q(d_out),
                                   lamA=lamA, lamS=lamS, a=a, s=s, d_in=d_in, d_out=d_out))

    def run(self, i):
        """Seconds for the oracle on case i (one example, one module)."""
        c, O, w = self.cases[i], self.O, self.w
        t0 = time.perf_counter()
        Lam = O.kfac_eigenvalues(c["lamS"], c["lamA"])
        lam = O.damping(Lam, w.damping_rel)
        O.compress_layer(c["a"], c["s"], c["QA"], c["QS"], Lam, lam, w.m, self.P)
        return time.perf_counter() - t0

    def flops(self, i):
        # the oracle's dense work per example: G (2 T d_out d_in), Q_S^T G Q_A
        # (2 d_out d_in (d_in + d_out)), P^T z (2 m k)
        c, w = self.cases[i], self.w
        return (2.0 * w.T * c["d_out"] * c["d_in"] + 2.0 * c["d_out"] * c["d_in"] * (c["d_in"] + c["d_out"]) +
                2.0 * w.m * w.k)


def _cores():
    return len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()


def cpu_baseline(w):
    """Examples/s per stack of the oracle, from one example through one module of
    each distinct shape, scaled by the shape counts (1 / sum_s count_s t_s)."""
    smp = OracleSample(w)
    total, per_shape, flops = 0.0, {}, 0.0
    for i, c in enumerate(smp.cases):
        t = smp.run(i)
        total += c["count"] * t
        per_shape[c["shape"]] = 1.0 / t
        flops += c["count"] * smp.flops(i)
    desc = (f"1 example x one module of each of the {len(smp.cases)} distinct shapes, "
            f"scaled by the shape counts to the {len(w.modules)}-module stack")
    return {"value": 1.0 / total, "unit": "examples/s", "cores": _cores(), "kind": "oracle",
            "sample": desc, "examples_per_s_per_shape": per_shape,
            "oracle_GFLOPs": flops / total / 1e9}


def cpu_score_sample(ks, seconds=3.0):
    """Oracle one-bit scores/s (float32 evaluation order) for stored codes of the
    given modules: repeated batches of 16 stored rows x 4 queries for about
    `seconds` of scoring (input generation not timed)."""
    from oracle import eogp_oracle as O
    rng = np.random.default_rng(3)
    Q, n = 4, 16
    qc = O.pack_concat([rng.integers(0, 2, (Q, k)).astype(bool) for k in ks])
    qs = rng.lognormal(0, 0.5, (Q, len(ks))).astype(np.float32)
    done, busy = 0, 0.0
    while busy < seconds:
        tc = O.pack_concat([rng.integers(0, 2, (n, k)).astype(bool) for k in ks])
        ts = rng.lognormal(0, 0.5, (n, len(ks))).astype(np.float32)
        t1 = time.perf_counter()
        O.score_codes_f32(tc, ts, ks, qc, qs)
        busy += time.perf_counter() - t1
        done += n * Q
    return done / busy


def headline_config(w, B, world, name):
    cfg = {"workload": name, "batch_per_gpu": B, "seq_len": w.T, "m": w.m, "k": w.k,
           "modules": len(w.modules), "parallelism": f"replicas x{world}",
           "l2": "inputs > L2 (each module's inputs exceed 129 MB every step)",
           "streams": "consecutive modules alternate between two streams, one workspace each"}
    if name == "olmo2_7b_bf16":
        cfg["eigenbases"] = "page-locked host memory, streamed one layer ahead"
    return cfg


def run_reference(args):
    """The reference arm: the oracle on the host cores, on the headline workload.
    A step is the oracle compressing one example through one module, the
    distinct module shapes taken in turn; the timed steps give each shape's mean
    time t_s, and value = 1 / sum_s count_s t_s examples/s per stack."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    from paper_2609_37842_gb300 import synth
    name = args.workload
    w = synth.WORKLOADS[name]
    B = args.batch or CONFIG_BATCH[name]
    smp = OracleSample(w)
    nc = len(smp.cases)
    for i in range(args.warmup):
        smp.run(i % nc)
    times = [[] for _ in range(nc)]
    wall0 = time.perf_counter()
    for i in range(args.steps):
        times[i % nc].append(smp.run(i % nc))
    wall = time.perf_counter() - wall0
    mean = [statistics.mean(t) if t else smp.run(i) for i, t in enumerate(times)]
    value = 1.0 / sum(c["count"] * t for c, t in zip(smp.cases, mean))
    world = int(os.environ.get("WORLD_SIZE", str(args.gpus)))
    sample = (f"each step: 1 example through one module, the {nc} distinct module shapes in turn; value = 1 / "
              f"sum over shapes of (modules of that shape x mean step time of that shape)")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "examples/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1000.0 * wall / max(1, args.steps), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": headline_config(w, B, world, name),
            "value_basis": "per-shape step times scaled to the stack (a step is one module, not one stack)",
            "cpu_baseline": {"value": value, "unit": "examples/s", "cores": _cores(), "kind": "oracle",
                             "sample": sample,
                             "seconds_per_shape": {c["shape"]: t for c, t in zip(smp.cases, mean)}},
            "e2e": {"value": value, "unit": "examples/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


# ------------------------------------------------------------- scoring
def timed_call(fn, stream, reps=3):
    import torch
    from paper_2609_37842_gb300 import eogp as E
    fn()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(reps):
        fn()
    b.record(stream)
    torch.cuda.synchronize()
    E.sync_status()
    return a.elapsed_time(b) / reps


def bench_query_scoring(w, N, Q, dev, stream, probes, bf16_burst, peaks_src, seed, paper=True):
    """CODES scores (dense and with the top 20 fused) of Q one-bit queries against N
    stored codes of the workload's modules; PAPER mode (unquantised queries) too."""
    import torch
    from paper_2609_37842_gb300 import eogp as E
    U, words = len(w.modules), (w.k + 31) // 32
    ks = [w.k] * U
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    tc = torch.randint(-2 ** 31, 2 ** 31 - 1, (N, U * words), generator=g, device=dev, dtype=torch.int32)
    qc = torch.randint(-2 ** 31, 2 ** 31 - 1, (Q, U * words), generator=g, device=dev, dtype=torch.int32)
    tsc = torch.exp(0.5 * torch.randn((N, U), generator=g, device=dev))
    qsc = torch.exp(0.5 * torch.randn((Q, U), generator=g, device=dev))
    out = torch.empty((Q, N), dtype=torch.float32, device=dev)
    sms = timed_call(lambda: E.score(tc, tsc, ks, E.SCORE_CODES, qc, qsc, out=out), stream)
    D = U * w.k
    pk, pk_src, pk_mode = score_peak(ks, probes, bf16_burst, peaks_src)
    alg = 2.0 * N * Q * D               # +-1 multiply-adds of the inner products
    res = {"metric": "query x train scores/sec", "value": N * Q / (sms / 1000.0), "unit": "scores/s",
           "ms_per_call": sms, "N": N, "Q": Q, "modules": U, "bits": D, "mode": f"CODES ({pk_mode})",
           "tensor_TFLOPs": alg / (sms / 1000.0) / 1e12,
           "tensor_frac": alg / (sms / 1000.0) / 1e12 / pk,
           "tensor_peak": pk, "tensor_peak_source": pk_src}
    del out
    K = 20
    wtc = E.workspace(E.score_topk_workspace_size(N, ks, E.SCORE_CODES, Q, K), dev)
    cms = timed_call(lambda: E.score_topk(tc, tsc, ks, E.SCORE_CODES, qc, K, query_scales=qsc, ws=wtc), stream)
    res["codes_top20"] = {"ms_per_call": cms, "scores_per_s": N * Q / (cms / 1000.0)}
    del wtc
    if paper:
        y = torch.randn((Q, D), generator=g, device=dev)
        out = torch.empty((Q, N), dtype=torch.float32, device=dev)
        wsp = E.workspace(E.score_workspace_size(N, ks, E.SCORE_PAPER, Q), dev)
        pms = timed_call(lambda: E.score(tc, tsc, ks, E.SCORE_PAPER, y, out=out, ws=wsp), stream)
        res["paper_dense"] = {"ms_per_call": pms, "scores_per_s": N * Q / (pms / 1000.0),
                              "tensor_TFLOPs_issued": 2 * alg / (pms / 1000.0) / 1e12,
                              "tensor_frac_issued": 2 * alg / (pms / 1000.0) / 1e12 / bf16_burst,
                              "note": "bf16 hi + lo query split: 2 MMAs per algorithmic one"}
        del out, wsp
        wtp = E.workspace(E.score_topk_workspace_size(N, ks, E.SCORE_PAPER, Q, K), dev)
        tms = timed_call(lambda: E.score_topk(tc, tsc, ks, E.SCORE_PAPER, y, K, ws=wtp), stream)
        res["paper_top20"] = {"ms_per_call": tms, "scores_per_s": N * Q / (tms / 1000.0)}
        del y, wtp
    del tc, qc, tsc, qsc
    torch.cuda.empty_cache()
    return res


def bench_scan(dev, stream, probes, bf16_burst, peaks_src, hbm, rows=0, qs_arg=""):
    """The scoring-bound sweep: 4,194,304 stored 16,384-bit codes, Q in {1, 64, 1024,
    8192} (chunks of 1024 queries), top 20 fused for Q >= 1024."""
    import torch
    from paper_2609_37842_gb300 import eogp as E
    from paper_2609_37842_gb300 import synth
    g = torch.Generator(device=dev)
    g.manual_seed(99)
    sc = synth.SCAN
    N, ksc = (rows or sc["N"]), sc["k"]
    scan_qs = [int(q) for q in qs_arg.split(",")] if qs_arg else list(sc["Qs"])
    Wsc = ksc // 32
    tr = torch.randint(-2 ** 31, 2 ** 31 - 1, (N, Wsc), generator=g, device=dev, dtype=torch.int32)
    tsc = torch.exp(sc["scale_sigma"] * torch.randn((N, 1), generator=g, device=dev))
    qmax = 1024
    out = torch.empty((qmax, N), dtype=torch.float32, device=dev)
    scan = {"N": N, "bits": ksc, "mode": "CODES", "per_Q": {}}
    for Q in scan_qs:
        qc = torch.randint(-2 ** 31, 2 ** 31 - 1, (Q, Wsc), generator=g, device=dev, dtype=torch.int32)
        qs = torch.exp(sc["scale_sigma"] * torch.randn((Q, 1), generator=g, device=dev))
        chunks = [(q0, min(Q, q0 + qmax)) for q0 in range(0, Q, qmax)]

        def run():
            for q0, q1 in chunks:
                E.score(tr, tsc, [ksc], E.SCORE_CODES, qc[q0:q1], qs[q0:q1], out=out[:q1 - q0])
        qms = timed_call(run, stream, reps=1)
        byts = len(chunks) * (N * Wsc * 4 + N * 4) + Q * N * 4
        ent = {"ms": qms, "scores_per_s": N * Q / (qms / 1000.0), "GBps": byts / (qms / 1000.0) / 1e9,
               "frac_of_hbm": byts / (qms / 1000.0) / 1e9 / hbm}
        if Q >= 64:   # tensor-core kernel: +-1 multiply-adds against the rate of the MMA it issues
            tfl = 2.0 * N * ksc * Q / (qms / 1000.0) / 1e12
            pk, pk_src, pk_mode = score_peak([ksc], probes, bf16_burst, peaks_src)
            kern = ("k_score_pair_ks" if Q <= 64 else "k_score_pair") if "mxf4" in pk_mode else "k_score_tc"
            ent.update({"kernel": f"{kern} ({pk_mode})", "tensor_TFLOPs": tfl,
                        "tensor_frac": tfl / pk, "tensor_peak_source": pk_src})
        else:
            wops = N * Q * Wsc / (qms / 1000.0)
            ent.update({"kernel": "k_score_codes_smallq (popcount)", "word_ops_per_s": wops})
            if probes:
                ent["popc_frac"] = wops / probes["popc_words_per_s"]
        if Q >= 1024:  # per-query top 20 in the scoring epilogue: no Q x N output
            K = 20
            wt = E.workspace(E.score_topk_workspace_size(N, [ksc], E.SCORE_CODES, Q, K), dev)
            kms = timed_call(lambda: E.score_topk(tr, tsc, [ksc], E.SCORE_CODES, qc, K, query_scales=qs, ws=wt),
                             stream, reps=1)
            ent["top20"] = {"ms": kms, "scores_per_s": N * Q / (kms / 1000.0), "output_bytes_avoided": Q * N * 4}
            del wt
        scan["per_Q"][str(Q)] = ent
        del qc, qs
    del tr, out
    torch.cuda.empty_cache()
    return scan


def bench_pack(dev, stream, hbm):
    import torch
    from paper_2609_37842_gb300 import eogp as E
    g = torch.Generator(device=dev)
    g.manual_seed(98)
    xs = torch.randn((262144, 1024), generator=g, device=dev)
    pc = torch.empty((262144, 32), dtype=torch.int32, device=dev)
    psc = torch.empty((262144,), dtype=torch.float32, device=dev)
    pms = timed_call(lambda: E.pack_sign(xs, pc, psc), stream, reps=5)
    pbytes = xs.numel() * 4 + pc.numel() * 4 + psc.numel() * 4
    del xs, pc, psc
    torch.cuda.empty_cache()
    return {"rows": 262144, "k": 1024, "ms": pms, "GBps": pbytes / (pms / 1000.0) / 1e9,
            "frac_of_hbm": pbytes / (pms / 1000.0) / 1e9 / hbm}


def compact_rooflines(scoring, scan, pack, others, fit):
    """Other kernels' roofline fractions and rates, for the record's `roofline`."""
    r = {}
    for nm, sc in (scoring or {}).items():
        r[f"score_codes_{nm}"] = {"bound": "tensor (+-1 MMA)", "scores_per_s": sc["value"],
                                  "achieved": sc["tensor_TFLOPs"], "peak": sc["tensor_peak"], "unit": "TFLOP/s",
                                  "frac": sc["tensor_frac"], "peak_source": sc["tensor_peak_source"],
                                  "ms": sc["ms_per_call"], "N": sc["N"], "Q": sc["Q"], "bits": sc["bits"]}
        if "codes_top20" in sc:
            r[f"score_codes_{nm}"]["top20_scores_per_s"] = sc["codes_top20"]["scores_per_s"]
        if "paper_dense" in sc:
            r[f"score_paper_{nm}"] = {"bound": "tensor (bf16, hi/lo issued)",
                                      "scores_per_s": sc["paper_dense"]["scores_per_s"],
                                      "frac": sc["paper_dense"]["tensor_frac_issued"]}
    for q, ent in ((scan or {}).get("per_Q") or {}).items():
        e = {"scores_per_s": ent["scores_per_s"], "ms": ent["ms"], "hbm_frac": ent["frac_of_hbm"]}
        if "tensor_frac" in ent:
            e.update({"bound": "tensor (+-1 MMA)" if int(q) >= 1024 else "hbm or tensor", "tensor_frac": ent["tensor_frac"]})
        else:
            e.update({"bound": "hbm", "popc_frac": ent.get("popc_frac")})
        if "top20" in ent:
            e["top20_scores_per_s"] = ent["top20"]["scores_per_s"]
        r[f"scan_4M_q{q}"] = e
    if pack:
        r["pack_sign"] = {"bound": "hbm", "achieved": pack["GBps"], "unit": "GB/s", "frac": pack["frac_of_hbm"]}
    for nm, o in (others or {}).items():
        if isinstance(o, dict) and "roofline" in o:
            rf = o["roofline"]
            r[f"rotate_{nm}"] = {"bound": "tensor", "achieved": rf["achieved"], "peak": rf["peak"],
                                 "unit": "TFLOP/s", "frac": rf["frac"], "traffic": rf["traffic"],
                                 "examples_per_s": o["examples_per_s"]}
        if isinstance(o, dict) and nm == "olmo2_1b_bf16":
            r["olmo2_1b_input_hbm"] = {"bound": "hbm", "frac": o["input_frac_of_hbm"],
                                      "achieved": o["input_GBps"], "unit": "GB/s"}
    if fit:
        r["fit_pca_seconds"] = {f"m{f['m']}_k{f['k']}": f["seconds"] for f in fit}
    return r


# ------------------------------------------------------------------ main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default=HEADLINE,
                    help="headline stack (default: the OLMo-2-7B-shaped stack)")
    ap.add_argument("--batch", type=int, default=0, help="examples per step (default: the workload's)")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-score", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--e2e-chunk", type=int, default=0,
                    help="examples per host-to-device chunk inside the call (0: about 64 MB)")
    ap.add_argument("--e2e-batch", type=int, default=0, help="examples per e2e step (default: the workload's)")
    ap.add_argument("--no-scan", action="store_true")
    ap.add_argument("--scan-rows", type=int, default=0,
                    help="stored codes in the scan (default: the 4,194,304 of the scan workload)")
    ap.add_argument("--scan-qs", default="",
                    help="comma-separated query counts of the scan (default: 1,64,1024,8192)")
    ap.add_argument("--only-ekfac", action="store_true",
                    help="time only the EK-FAC correction (GPT-2 c_fc and OLMo-1B gate modules); "
                         "the case profiles/ captures for k_tc_ekfac")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the other stacks and the PCA-fit timing")
    ap.add_argument("--modules", type=int, default=0,
                    help="use only the first N modules of the headline stack (small profiling cases)")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)

    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_37842_gb300 import eogp as E
    from paper_2609_37842_gb300 import synth

    if args.only_ekfac:
        ek = [bench_ekfac(dev, 768, 3072, 512, 32), bench_ekfac(dev, 2048, 8192, 2048, 4)]
        if rank == 0:
            print(json.dumps({"ekfac_correction": ek}))
        return
    name = args.workload
    B = args.batch or CONFIG_BATCH[name]
    peaks, peaks_src = load_peaks()
    bf16_burst = peaks.get("bf16_tflops") or PEAKS_FALLBACK["bf16_tflops"]
    hbm = peaks.get("hbm_gbs") or PEAKS_FALLBACK["hbm_gbs"]

    def barrier():
        if world > 1:
            dist.barrier()

    # ---- headline: K compression steps of the stack, kernel events on ----
    st = Stack(name, B, dev, stream_bases=(name == "olmo2_7b_bf16"), modules=args.modules)
    w = st.w
    clocks = ClockSampler(local)
    ms, kern, clk, psteps = st.timed(args.steps, args.warmup, clocks=clocks, barrier=barrier)
    t_max = ms
    if world > 1:
        tt = torch.tensor([ms], device=dev)
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        t_max = float(tt.item())
    value = world * B * args.steps / (t_max / 1000.0)
    # library launches inside the timed region: per step as counted in the profiled steps
    launches = round(sum(v["launches"] for v in kern.values()) / psteps * args.steps)
    head = st.summary(ms, args.steps, kern, peaks, psteps)
    roofline = dict(head.get("roofline") or {"bound": "tensor", "achieved": None, "peak": None,
                                             "unit": "TFLOP/s", "frac": None, "traffic": None})
    roofline["peak_source"] = f"{peaks_src} bf16_tflops_sustained"

    # ---- end to end through the public host-input call ----
    e2e = None
    if not args.no_e2e:
        Be = min(B, args.e2e_batch or E2E_BATCH.get(name, B))
        e2e = e2e_run(st, Be, args.e2e_steps, args.e2e_chunk, dev, world, barrier)
    st.release()
    del st
    torch.cuda.empty_cache()

    # ---- measured +-1 MMA and popcount rates (scoring rooflines) ----
    probes = None
    if rank == 0 and not args.no_score:
        f8, f4, pc = E.measure_peaks()
        probes = {"e4m3_tflops": f8, "e2m1_tflops": f4, "popc_words_per_s": pc,
                  "what": "eogp_measure_peaks: back-to-back kind::f8f6f4 (e4m3) and kind::mxf4 (e2m1, unit "
                          "scales) MMAs; XOR + popcount chains on every core"}

    # ---- query x train scoring: the headline's query workload and GPT-2's ----
    stream = torch.cuda.current_stream()
    scoring = None
    if rank == 0 and not args.no_score:
        scoring = {}
        if w.Q and len(w.modules) > 1:
            scoring[name] = bench_query_scoring(w, w.N, w.Q, dev, stream, probes, bf16_burst, peaks_src, 77,
                                                paper=False)
        g2 = synth.WORKLOADS["gpt2_small_bf16"]
        if name != "gpt2_small_bf16" or not scoring:
            scoring["gpt2_small_bf16"] = bench_query_scoring(g2, g2.N, g2.Q, dev, stream, probes, bf16_burst,
                                                             peaks_src, 78)

    # ---- standalone sign-pack and the scoring sweep ----
    pack = scan = None
    if rank == 0 and not args.no_scan:
        pack = bench_pack(dev, stream, hbm)
        scan = bench_scan(dev, stream, probes, bf16_burst, peaks_src, hbm, args.scan_rows, args.scan_qs)

    # ---- the other stacks, the EK-FAC correction and the PCA fit ----
    configs = fit = None
    if rank == 0 and not args.no_configs:
        configs = {}
        for nm in ("gpt2_small_bf16", "olmo2_1b_bf16", "olmo2_7b_bf16", "olmo2_32b_gate_bf16", "tiny_f32"):
            if nm == name:
                continue
            o = Stack(nm, CONFIG_BATCH[nm], dev, stream_bases=(nm == "olmo2_7b_bf16"))
            steps = 3 if nm.startswith("olmo2_") and nm != "olmo2_32b_gate_bf16" else 5
            oms, okern, _, opsteps = o.timed(steps, 3)
            configs[nm] = o.summary(oms, steps, okern, peaks, opsteps)
            o.release()
            del o
            torch.cuda.empty_cache()
        configs["ekfac_correction"] = [bench_ekfac(dev, 768, 3072, 512, 32),
                                       bench_ekfac(dev, 2048, 8192, 2048, 4)]
        fit = [bench_fit(dev, 10000, 4096, 1024), bench_fit(dev, 10000, 8192, 2048)]

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w)
        ks = [w.k] * len(w.modules)
        cpu["oracle_scores_per_s"] = cpu_score_sample(ks)
        cpu["scores_sample"] = (f"16 stored rows x 4 one-bit queries of {len(ks)} x {w.k} bits, "
                                f"repeated for ~3 s")

    if rank == 0:
        roofline["others"] = compact_rooflines(scoring, scan, pack, configs, fit)
        line = {"metric": METRIC, "value": value, "unit": "examples/s", "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": t_max / args.steps, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "bf16" if w.dtype == "bf16" else "f32", "data": "synthetic",
                "config": headline_config(w, B, world, name if not args.modules else
                                          f"{name} (first {len(w.modules)} modules)"),
                "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e,
                "headline": {k: v for k, v in head.items() if k != "roofline"},
                "scoring": scoring, "pack_sign": pack, "scan": scan,
                "measured_rates": probes, "other_workloads": configs, "fit_pca": fit,
                "gpu_launches": launches, "kernels": kern, "clocks": clk}
        print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
