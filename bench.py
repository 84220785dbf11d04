#!/usr/bin/env python3
"""Benchmark of the GradLev token scans on GB300.

One step = the forward scan (Sec. 3 step 2, Eq. 3) and the costate scan
(Sec. 3 step 3, Eq. 4) over one batch of the workload, through the library's
C ABI.  Default workload: the model-shaped layer sweep (12 independent layers
x 12 heads of 64x64 fast weights, B=8, T=8192, bf16), all layers' forward and
costate scans per step.  `--workload c3` runs the two-layer MLP of Appendix A
(512 -> 2048 -> 512, GELU): forward through both layers, then costates back
through both.

Prints ONE JSON line on rank 0.  `value` is tokens/s of the whole step
(L*B*T tokens per step, both scans) with inputs resident in HBM; `scans`
breaks it down per scan with each scan's roofline; `roofline` is the dominant
(slowest) kernel's; `e2e` is the same metric through the public API with
pinned host buffers copied in and results copied out inside the timed region;
`cpu_baseline` is the fp64 oracle timed on this host's cores on a bounded
sample of the same workload.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload c5] [--impl reference]
"""
from __future__ import annotations

import argparse
import ctypes
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import torch  # noqa: E402

import workloads as W  # noqa: E402

METRIC = "tokens/s per scan (fwd, costate) at 1 GB300; % of scan roofline"
UNIT = "tokens/s"
COUNT_CHUNK = 64  # chunk size fixed for counting flops (scan roofline convention)
L2_BYTES = 129 * 1024 * 1024


def nvtx(name):
    """An NVTX range around one library call of the timed step (for ncu --nvtx and
    timeline tools); host-side markers only."""
    return torch.cuda.nvtx.range(name)


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16_tflops": float(p["bf16_tflops"]),
                "bf16_tflops_sustained": float(p.get("bf16_tflops_sustained", p["bf16_tflops"])),
                "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "source": "fallback"}


def roofline_entry(flops, nbytes, seconds, pk):
    t_hbm = nbytes / (pk["hbm_gbs"] * 1e9)
    t_tc = flops / (pk["bf16_tflops"] * 1e12)
    if t_hbm >= t_tc:
        ach = nbytes / seconds / 1e9
        return {"bound": "hbm", "achieved": round(ach, 1), "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": round(ach / pk["hbm_gbs"], 4), "algorithmic_bytes": nbytes,
                "peak_source": pk["source"]}
    ach = flops / seconds / 1e12
    return {"bound": "tensor", "achieved": round(ach, 2), "peak": pk["bf16_tflops"],
            "unit": "TFLOP/s", "frac": round(ach / pk["bf16_tflops"], 4),
            "algorithmic_flops": flops, "peak_source": pk["source"]}


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi clock / throttle sampling while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.marks = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def mark(self):
        self.marks.append(time.time())

    def stop(self):
        if self.proc is None:
            return
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()

    def summary(self):
        if not self.lines:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        t0, t1 = (self.marks[0], self.marks[-1]) if len(self.marks) >= 2 else (0, 1e30)
        inside = [ln for (t, ln) in self.lines if t0 <= t <= t1]
        rows = inside if inside else [ln for _, ln in self.lines]
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in rows:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        out = {"sm_mhz": statistics.median(sm) if sm else None,
               "sm_max_mhz": max(smax) if smax else None, "reasons": sorted(reasons),
               "samples": len(sm), "window": "timed region" if inside else "whole run"}
        return out


# ------------------------------------------------------------------ workloads
def _bytes(*ts):
    return sum(t.numel() * t.element_size() for t in ts)


def make_gates(wl, gates, device):
    """Synthetic gates of the gated modes, drawn once: per-token eta_t in [0, 2 eta]
    and, for "alpha", retention alpha_t in [0.9, 1] (fp32 [L, B, T, H]); for "docs",
    document starts per batch row (uint8 [B, T]) with documents of 512 to 1535 tokens
    and the scalar eta."""
    gen = torch.Generator()
    gen.manual_seed(wl.seed * 1000 + 17)
    out = {}
    shape = (wl.L, wl.B, wl.T, wl.H)
    if gates in ("eta", "alpha"):
        out["eta_t"] = (torch.rand(shape, generator=gen) * (2 * wl.eta)).to(device)
        if gates == "alpha":
            out["alpha_t"] = (0.9 + 0.1 * torch.rand(shape, generator=gen)).to(device)
    elif gates == "docs":
        ds = torch.zeros(wl.B, wl.T, dtype=torch.uint8)
        for b in range(wl.B):
            t = int(torch.randint(512, 1536, (1,), generator=gen))
            while t < wl.T:
                ds[b, t] = 1
                t += int(torch.randint(512, 1536, (1,), generator=gen))
        out["doc_start"] = ds.to(device)
    return out


class LinearJob:
    """One fast-weight linear map per (layer, batch, head) unit: the forward scan
    (Eq. 3) and the costate scan (Eq. 4), one library call each."""

    kind = "linear"

    def __init__(self, gl, wl, device, rank, gates=None):
        self.gl, self.wl = gl, wl
        self.inp = W.make_linear(wl.resized(seed=wl.seed + 1000 * rank), device=device)
        self.outs = {"y": torch.empty_like(self.inp["g_hat"]),
                     "g_in": torch.empty_like(self.inp["x"])}
        # Gated scans (Eq. 2) and document resets, inputs from make_gates; the
        # library folds document starts into the gates on every call.
        self.gates = gates
        code = 1 if wl.dtype == "bf16" else 0
        nb = gl.workspace_bytes(wl.L, wl.B, wl.T, wl.H, wl.d_in, wl.d_out, code)
        self.inp.update(make_gates(wl, gates, device))
        self.eta_t, self.alpha_t = self.inp.get("eta_t"), self.inp.get("alpha_t")
        if gates:
            from paper_2609_34174_gb300 import _binding as _B
            d = _B._Desc(wl.L, wl.B, wl.T, wl.H, wl.d_in, wl.d_out, code, 0)
            nb = int(_B.load_library().gradlev_workspace_bytes_gated(ctypes.byref(d)))
        self.ws = torch.empty(max(256, nb), dtype=torch.uint8, device=device)
        self.tokens = wl.tokens
        # one chunk-kernel launch per scan; eta_t adds the prescale launch to each,
        # documents the gate-folding launch.  The retention kernel cuts few long units
        # (fewer than two per SM, more than 1024 tokens) into segments: an aggregate
        # launch and a carry launch precede its scan.
        units = wl.L * wl.B * wl.H
        sms = torch.cuda.get_device_properties(device).multi_processor_count if str(device).startswith("cuda") else 152
        segmented = gates in ("alpha", "docs") and units < 2 * sms and wl.T > 1024
        per_scan = (3 if segmented else 1) + (1 if gates in ("eta", "docs") else 0)
        self.launches_per_step = 2 * per_scan
        self.in_keys = ("x", "g_hat", "g_out", "W0") + (
            ("eta_t",) if gates in ("eta", "alpha") else ()) + (
            ("alpha_t",) if gates == "alpha" else ()) + (("doc_start",) if gates == "docs" else ())
        self.out_keys = ("y", "g_in")
        self.kernel = {"fwd": "tc_scan_kernel<64, false> (forward scan)",
                       "costate": "tc_scan_kernel<64, true> (costate scan)"}
        if gates in ("alpha", "docs"):
            self.kernel = {"fwd": "decay_scan_kernel<false, false> (forward scan, retention)",
                           "costate": "decay_scan_kernel<true, false> (costate scan, retention)"}

    def input_bytes(self):
        return _bytes(self.inp["x"], self.inp["g_hat"], self.inp["g_out"])

    def step(self, inp=None, events=None):
        gl, wl, o = self.gl, self.wl, self.outs
        inp = inp or self.inp
        if events is not None:
            events[0].record()
        eta = inp["eta_t"] if self.gates in ("eta", "alpha") else wl.eta
        alpha = inp.get("alpha_t")
        ds = inp.get("doc_start")
        with nvtx("gradlev forward scan"):
            gl.forward_scan(inp["x"], inp["g_hat"], inp["W0"], eta, y=o["y"], workspace=self.ws,
                            alpha=alpha, doc_start=ds)
        if events is not None:
            events[1].record()
        with nvtx("gradlev costate scan"):
            gl.costate_scan(inp["x"], inp["g_hat"], inp["W0"], eta, inp["g_out"], g_in=o["g_in"],
                            workspace=self.ws, alpha=alpha, doc_start=ds)
        if events is not None:
            events[2].record()

    # --- pipelined end-to-end step: chunks along layers (or batch rows when L = 1)
    def e2e_chunks(self):
        wl = self.wl
        if wl.L > 1:
            return [("L", l, l + 1) for l in range(wl.L)]
        if wl.B > 1:
            return [("B", b, b + 1) for b in range(wl.B)]
        return [("L", 0, 1)]

    @staticmethod
    def _cut(t, sl, lead_w0=False):
        axis, a, b = sl
        if axis == "L" or lead_w0:
            return t[a:b] if axis == "L" else t
        return t[:, a:b]

    def e2e_inputs(self, host, dev, sl, first):
        out = []
        for k in self.in_keys:
            if k == "doc_start":  # [B, T]: whole with layer chunks, rows with batch chunks
                if sl[0] == "B":
                    out.append((k, host[k][sl[1]:sl[2]], dev[k][sl[1]:sl[2]]))
                elif first:
                    out.append((k, host[k], dev[k]))
            elif k == "W0":
                if sl[0] == "L":
                    out.append((k, host[k][sl[1]:sl[2]], dev[k][sl[1]:sl[2]]))
                elif first:
                    out.append((k, host[k], dev[k]))
            else:
                out.append((k, self._cut(host[k], sl), self._cut(dev[k], sl)))
        return out

    def e2e_outputs(self, hout, sl):
        return [(self._cut(self.outs[k], sl), self._cut(hout[k], sl)) for k in self.out_keys]

    def e2e_step(self, dev, sl, ws):
        gl, wl = self.gl, self.wl
        cut = lambda t: self._cut(t, sl)
        w0 = dev["W0"][sl[1]:sl[2]] if sl[0] == "L" else dev["W0"]
        eta = cut(dev["eta_t"]) if self.gates in ("eta", "alpha") else wl.eta
        alpha = cut(dev["alpha_t"]) if self.gates == "alpha" else None
        ds = None
        if self.gates == "docs":
            ds = dev["doc_start"][sl[1]:sl[2]] if sl[0] == "B" else dev["doc_start"]
        gl.forward_scan(cut(dev["x"]), cut(dev["g_hat"]), w0, eta, y=cut(self.outs["y"]),
                        workspace=ws, alpha=alpha, doc_start=ds)
        gl.costate_scan(cut(dev["x"]), cut(dev["g_hat"]), w0, eta, cut(dev["g_out"]),
                        g_in=cut(self.outs["g_in"]), workspace=ws, alpha=alpha, doc_start=ds)

    def e2e_workspace_bytes(self):
        wl = self.wl
        sl = self.e2e_chunks()[0]
        L = 1 if sl[0] == "L" else wl.L
        B = wl.B if sl[0] == "L" else 1
        code = 1 if wl.dtype == "bf16" else 0
        from paper_2609_34174_gb300 import _binding as _B
        d = _B._Desc(L, B, wl.T, wl.H, wl.d_in, wl.d_out, code, 0)
        lib = _B.load_library()
        return int(max(lib.gradlev_workspace_bytes(ctypes.byref(d)),
                       lib.gradlev_workspace_bytes_gated(ctypes.byref(d))))

    def counts(self, scan):
        """Algorithmic flops and compulsory bytes of one scan call.

        Per token and unit: flops 4*d*m + C*(d+m) with C = 64 (state read 2dm,
        state update 2dm, causal halves of the two CxC products); bytes
        e*(d + 2m) forward (x, ghat in; y out), e*(2d + 2m) costate (x, ghat,
        g_out in; g_in out), plus 4*d*m per slow matrix W0.
        """
        wl = self.wl
        e = 2 if wl.dtype == "bf16" else 4
        d, m = wl.d_in, wl.d_out
        tu = wl.L * wl.B * wl.T * wl.H
        flops = tu * (4 * d * m + COUNT_CHUNK * (d + m))
        per_tok = e * (d + 2 * m) if scan == "fwd" else e * (2 * d + 2 * m)
        return flops, tu * per_tok + 4 * d * m * wl.L * wl.H

    def config(self):
        wl = self.wl
        c = {"L": wl.L, "B": wl.B, "T": wl.T, "H": wl.H, "d_in": wl.d_in, "d_out": wl.d_out,
             "eta": wl.eta}
        if self.gates:
            c["gates"] = {"eta": "per-token eta_t",
                          "alpha": "per-token eta_t and retention alpha_t (tensor-core retention kernel)",
                          "docs": "document resets, documents of 512-1535 tokens, scalar eta "
                                  "(gate folding + tensor-core retention kernel)"}[self.gates]
        return c

    def oracle_run(self, inp, n_units, cores, t_tokens=None):
        """Time the fp64 oracle on the first n_units units (forward and costate
        reads in one sequential walk per unit); returns (seconds, metric tokens)."""
        import oracle
        wl = self.wl
        units = [(l, b, h) for l in range(wl.L) for b in range(wl.B) for h in range(wl.H)]
        units = units[:n_units]
        x = W.units_fp64(inp["x"], units)
        g = W.units_fp64(inp["g_hat"], units)
        w0 = W.w0_fp64(inp["W0"], units)
        go = W.units_fp64(inp["g_out"], units)
        gates = getattr(self, "gates", None)
        if not gates:
            t = time.perf_counter()
            oracle.linear_scan(x, g, w0, wl.eta, gout=go, nthreads=cores)
        else:
            # every unit with its own gate sequences: one oracle call per unit, the
            # calls spread over the cores (the C oracle releases the interpreter)
            import concurrent.futures as cf
            f64 = lambda t_: t_.detach().to("cpu", torch.float64).numpy()
            if gates == "docs":
                ds = inp["doc_start"].cpu().numpy() != 0
                calls = [(oracle.linear_scan_docs, (x[i:i + 1], g[i:i + 1], w0[i], wl.eta,
                                                    ds[b][None]), {"gout": go[i:i + 1]})
                         for i, (l, b, h) in enumerate(units)]
            else:
                calls = [(oracle.linear_scan,
                          (x[i:i + 1], g[i:i + 1], w0[i], f64(inp["eta_t"][l, b, :, h])),
                          {"gout": go[i:i + 1], "nthreads": 1,
                           "alpha": (f64(inp["alpha_t"][l, b, :, h]) if "alpha_t" in inp
                                     else None)})
                         for i, (l, b, h) in enumerate(units)]
            t = time.perf_counter()
            with cf.ThreadPoolExecutor(max_workers=cores) as ex:
                list(ex.map(lambda c: c[0](*c[1], **c[2]), calls))
        # one metric token spans all H heads of a layer
        return time.perf_counter() - t, len(units) * wl.T / wl.H

    def n_units(self):
        return self.wl.L * self.wl.B * self.wl.H

    def sample_text(self, n):
        gates = getattr(self, "gates", None)
        with_gates = {None: "", "eta": ", with their eta_t", "alpha": ", with their eta_t and alpha_t",
                      "docs": ", one learner per document"}[gates]
        return (f"{n} of {self.n_units()} (layer, batch, head) units at full T={self.wl.T}, "
                f"forward and costate reads in one sequential walk per unit{with_gates}, fp64")


class FusedJob(LinearJob):
    """Both reads of one linear map per unit in one pass (gradlev_fused_scan, Sec. 3
    steps 2 and 3): x, ghat and g_out are read once and one running state serves the
    forward and the costate read.  The step computes what LinearJob's two scans do."""

    kind = "fused"

    def __init__(self, gl, wl, device, rank):
        super().__init__(gl, wl, device, rank)
        self.launches_per_step = 1
        self.kernel = {"fused": "tc_scan_kernel<64, fused> (forward and costate reads, one pass)"}

    def step(self, inp=None, events=None):
        gl, wl, o = self.gl, self.wl, self.outs
        inp = inp or self.inp
        if events is not None:
            events[0].record()
        with nvtx("gradlev fused scan"):
            gl.fused_scan(inp["x"], inp["g_hat"], inp["W0"], wl.eta, inp["g_out"], y=o["y"],
                          g_in=o["g_in"], workspace=self.ws)
        if events is not None:
            events[1].record()
            events[2].record()

    def e2e_step(self, dev, sl, ws):
        cut = lambda t: self._cut(t, sl)
        w0 = dev["W0"][sl[1]:sl[2]] if sl[0] == "L" else dev["W0"]
        self.gl.fused_scan(cut(dev["x"]), cut(dev["g_hat"]), w0, self.wl.eta, cut(dev["g_out"]),
                           y=cut(self.outs["y"]), g_in=cut(self.outs["g_in"]), workspace=ws)

    def counts(self, scan):
        """Algorithmic flops and compulsory bytes of one fused call.

        Per token and unit: flops 6*d*m + 2*C*(d+m) (two state reads, one state
        update, the causal halves of both reads' CxC products, C = 64); bytes
        e*(2d + 3m): x, ghat, g_out in, y and g_in out; plus 4*d*m per W0.
        """
        wl = self.wl
        e = 2 if wl.dtype == "bf16" else 4
        d, m = wl.d_in, wl.d_out
        tu = wl.L * wl.B * wl.T * wl.H
        flops = tu * (6 * d * m + 2 * COUNT_CHUNK * (d + m))
        return flops, tu * e * (2 * d + 3 * m) + 4 * d * m * wl.L * wl.H


class GradsJob(LinearJob):
    """Step-size gradients of both reads of one linear map per unit, writes
    detached (Sec. 3, practical architecture and training): dL/deta_t of the
    forward read for an upstream u = dL/dy, and of the costate read for
    w = dL/dg_in.  Each is the anti-causal suffix read of the same writes,
    reduced per token by a dot in the reverse kernel's epilogue."""

    kind = "grads"

    def __init__(self, gl, wl, device, rank):
        super().__init__(gl, wl, device, rank)
        gen = torch.Generator(device=device)
        gen.manual_seed(wl.seed * 1000 + 29)
        dt = self.inp["x"].dtype
        self.inp["u"] = torch.randn(self.inp["g_hat"].shape, generator=gen, device=device).to(dt)
        self.inp["w"] = torch.randn(self.inp["x"].shape, generator=gen, device=device).to(dt)
        shape = (wl.L, wl.B, wl.T, wl.H)
        self.outs = {"deta_f": torch.empty(shape, device=device),
                     "deta_c": torch.empty(shape, device=device)}
        from paper_2609_34174_gb300 import _binding as _B
        code = 1 if wl.dtype == "bf16" else 0
        d = _B._Desc(wl.L, wl.B, wl.T, wl.H, wl.d_in, wl.d_out, code, 0)
        lib = _B.load_library()
        nb = max(lib.gradlev_eta_grad_workspace_bytes(ctypes.byref(d), 0),
                 lib.gradlev_eta_grad_workspace_bytes(ctypes.byref(d), 1))
        self.ws = torch.empty(max(256, int(nb)), dtype=torch.uint8, device=device)
        self.in_keys = ("x", "g_hat", "g_out", "u", "w")
        self.out_keys = ("deta_f", "deta_c")
        self.kernel = {"fwd": "tc_scan_kernel<64, false, REV, DOT> (suffix read, q = k = x, dot with ghat)",
                       "costate": "tc_scan_kernel<64, true, REV, DOT> (suffix read, q = ghat, k = g_out, dot with x)"}

    def input_bytes(self):
        return _bytes(*(self.inp[k] for k in self.in_keys))

    def _run(self, src, cut, ws):
        gl = self.gl
        with nvtx("gradlev eta_grad forward read"):
            gl.eta_grad(cut(src["x"]), cut(src["g_hat"]), cut(src["u"]),
                        deta=cut(self.outs["deta_f"]), workspace=ws)
        yield
        with nvtx("gradlev eta_grad costate read"):
            gl.eta_grad(cut(src["x"]), cut(src["g_hat"]), cut(src["w"]), read="costate",
                        g_out=cut(src["g_out"]), deta=cut(self.outs["deta_c"]), workspace=ws)
        yield

    def step(self, inp=None, events=None):
        inp = inp or self.inp
        if events is not None:
            events[0].record()
        for i, _ in enumerate(self._run(inp, lambda t: t, self.ws)):
            if events is not None:
                events[i + 1].record()

    def e2e_inputs(self, host, dev, sl, first):
        return [(k, self._cut(host[k], sl), self._cut(dev[k], sl)) for k in self.in_keys]

    def e2e_step(self, dev, sl, ws):
        for _ in self._run(dev, lambda t: self._cut(t, sl), ws):
            pass

    def e2e_workspace_bytes(self):
        return self.ws.numel()

    def counts(self, scan):
        """Per token and unit: the suffix read's flops 4*d*m + C*(d+m) (C = 64) plus
        the dot; compulsory bytes e*(2d + m) + 4 for the forward read's gradient
        (x, u, ghat in; deta out) and e*(2m + 2d) + 4 for the costate read's
        (ghat, g_out, w, x in; deta out)."""
        wl = self.wl
        e = 2 if wl.dtype == "bf16" else 4
        d, m = wl.d_in, wl.d_out
        tu = wl.L * wl.B * wl.T * wl.H
        if scan == "fwd":
            return tu * (4 * d * m + COUNT_CHUNK * (d + m) + 2 * m), tu * (e * (d + 2 * m) + 4)
        return tu * (4 * d * m + COUNT_CHUNK * (d + m) + 2 * d), tu * (e * (2 * d + 2 * m) + 4)

    def config(self):
        c = super().config()
        c["computes"] = "dL/deta_t of the forward and costate reads (suffix read + dot)"
        return c

    def oracle_run(self, inp, n_units, cores, t_tokens=None):
        """The fp64 oracle's suffix reads and dots for the first n_units units."""
        import numpy as np
        import oracle
        wl = self.wl
        units = [(l, b, h) for l in range(wl.L) for b in range(wl.B) for h in range(wl.H)]
        units = units[:n_units]
        f = lambda k: W.units_fp64(inp[k], units)
        x, g, go, u, w = f("x"), f("g_hat"), f("g_out"), f("u"), f("w")
        t = time.perf_counter()
        np.sum(g * oracle.suffix_scan(x, x, u, nthreads=cores), axis=2)
        np.sum(x * oracle.suffix_scan(g, go, w, nthreads=cores), axis=2)
        return time.perf_counter() - t, len(units) * wl.T / wl.H

    def sample_text(self, n):
        return (f"{n} of {self.n_units()} (layer, batch, head) units at full T={self.wl.T}, "
                f"suffix reads and dots of both reads, fp64")


class MLPJob:
    """The two-layer fast-weight MLP of Appendix A: forward through both layers
    (sigma fused in the layer-1 epilogue), then costates back through both
    (sigma' fused in the layer-2 costate epilogue)."""

    kind = "mlp"

    def __init__(self, gl, wl, device, rank):
        self.gl, self.wl = gl, wl
        self.inp = W.make_mlp(wl.resized(seed=wl.seed + 1000 * rank), device=device)
        B, T, d, m, k = wl.B, wl.T, wl.d, wl.m, wl.k
        dt = self.inp["x"].dtype
        mk = lambda w: torch.empty((B, T, w), dtype=dt, device=device)
        self.outs = {"z": mk(m), "h": mk(m), "y": mk(k), "gz": mk(m), "gx": mk(d)}
        code = 1 if wl.dtype == "bf16" else 0
        nb = max(gl.workspace_bytes(1, B, T, 1, d, m, code), gl.workspace_bytes(1, B, T, 1, m, k, code))
        self.ws = torch.empty(max(256, nb), dtype=torch.uint8, device=device)
        self.tokens = wl.tokens
        # forward: two layers x (state, score, output pass); the same for the costate
        self.launches_per_step = 12
        self.in_keys = ("x", "g_hat_z", "g_hat_y", "g_out", "W1", "W2")
        self.out_keys = ("y", "gx")
        self.kernel = {"fwd": "seg_gemm_kernel state/score/output passes (forward, both layers)",
                       "costate": "seg_gemm_kernel state/score/output passes (costate, both layers)"}

    def input_bytes(self):
        return _bytes(self.inp["x"], self.inp["g_hat_z"], self.inp["g_hat_y"], self.inp["g_out"])

    def step(self, inp=None, events=None):
        gl, wl, o = self.gl, self.wl, self.outs
        inp = inp or self.inp
        if events is not None:
            events[0].record()
        with nvtx("gradlev MLP forward"):
            gl.forward_scan(inp["x"], inp["g_hat_z"], inp["W1"], wl.eta1, act=wl.act, y=o["z"],
                            act_out=o["h"], workspace=self.ws)
            gl.forward_scan(o["h"], inp["g_hat_y"], inp["W2"], wl.eta2, y=o["y"],
                            workspace=self.ws)
        if events is not None:
            events[1].record()
        with nvtx("gradlev MLP costate"):
            gl.costate_scan(o["h"], inp["g_hat_y"], inp["W2"], wl.eta2, inp["g_out"], act=wl.act,
                            z=o["z"], g_in=o["gz"], workspace=self.ws)
            gl.costate_scan(inp["x"], inp["g_hat_z"], inp["W1"], wl.eta1, o["gz"], g_in=o["gx"],
                            workspace=self.ws)
        if events is not None:
            events[2].record()

    # --- pipelined end-to-end step: two chunks of batch rows (a single row leaves the
    # wide passes too few tiles to fill the GPU)
    def e2e_chunks(self):
        B = self.wl.B
        half = (B + 1) // 2
        return [(0, half), (half, B)] if B > 1 else [(0, 1)]

    def e2e_inputs(self, host, dev, sl, first):
        out = []
        for k in self.in_keys:
            if k in ("W1", "W2"):
                if first:
                    out.append((k, host[k], dev[k]))
            else:
                out.append((k, host[k][sl[0]:sl[1]], dev[k][sl[0]:sl[1]]))
        return out

    def e2e_outputs(self, hout, sl):
        return [(self.outs[k][sl[0]:sl[1]], hout[k][sl[0]:sl[1]]) for k in self.out_keys]

    def e2e_step(self, dev, sl, ws):
        gl, wl, o = self.gl, self.wl, self.outs
        c = lambda t: t[sl[0]:sl[1]]
        gl.forward_scan(c(dev["x"]), c(dev["g_hat_z"]), dev["W1"], wl.eta1, act=wl.act, y=c(o["z"]),
                        act_out=c(o["h"]), workspace=ws)
        gl.forward_scan(c(o["h"]), c(dev["g_hat_y"]), dev["W2"], wl.eta2, y=c(o["y"]), workspace=ws)
        gl.costate_scan(c(o["h"]), c(dev["g_hat_y"]), dev["W2"], wl.eta2, c(dev["g_out"]), act=wl.act,
                        z=c(o["z"]), g_in=c(o["gz"]), workspace=ws)
        gl.costate_scan(c(dev["x"]), c(dev["g_hat_z"]), dev["W1"], wl.eta1, c(o["gz"]), g_in=c(o["gx"]),
                        workspace=ws)

    def e2e_workspace_bytes(self):
        return self.ws.numel()

    def counts(self, scan):
        """Both layers: flops 4*d_i*m_i + C*(d_i+m_i) per token and layer (C = 64).
        Compulsory bytes with sigma fused (h is never needed from HBM): forward
        x, ghat_z in, z out; z, ghat_y in, y out.  Costate g_out, ghat_y, z in,
        g_z out; g_z, ghat_z, x in, g_x out.  Plus 4*d*m per slow matrix."""
        wl = self.wl
        e = 2 if wl.dtype == "bf16" else 4
        d, m, k = wl.d, wl.m, wl.k
        n = wl.B * wl.T
        flops = n * (4 * d * m + COUNT_CHUNK * (d + m) + 4 * m * k + COUNT_CHUNK * (m + k))
        if scan == "fwd":
            per_tok = e * ((d + m + m) + (m + k + k))
        else:
            per_tok = e * ((k + k + m + m) + (m + m + d + d))
        return flops, n * per_tok + 4 * (d * m + m * k)

    def config(self):
        wl = self.wl
        return {"B": wl.B, "T": wl.T, "widths": [wl.d, wl.m, wl.k], "act": wl.act,
                "eta": [wl.eta1, wl.eta2]}

    def oracle_run(self, inp, n_units, cores, t_tokens=None):
        """Time the fp64 MLP oracle on the first n_units sequences, truncated to
        t_tokens tokens (all reads and writes of both layers in one walk)."""
        import oracle
        wl = self.wl
        T = t_tokens or wl.T
        f = lambda t: t[:n_units, :T].to(torch.float64).cpu().numpy()
        args = (f(inp["x"]), f(inp["g_hat_z"]), f(inp["g_hat_y"]),
                inp["W1"].double().cpu().numpy(), inp["W2"].double().cpu().numpy())
        t = time.perf_counter()
        oracle.mlp_scan(*args, wl.eta1, wl.eta2, act=oracle.ACT_GELU_TANH, gout=f(inp["g_out"]),
                        nthreads=min(cores, n_units))
        return time.perf_counter() - t, n_units * T

    def n_units(self):
        return self.wl.B

    def sample_text(self, n, t_tokens=None):
        return (f"{n} of {self.wl.B} sequences, first {t_tokens or self.wl.T} of {self.wl.T} "
                f"tokens, both layers forward and costate in one sequential walk, fp64")


class GateGradsJob(GradsJob):
    """Derivatives with respect to the per-token gates (eta_t and retention alpha_t)
    of both reads of one linear map per unit, writes detached (Sec. 3, practical
    architecture and training; Eq. 2): alpha_t dL/dalpha_t and dL/deta_t of the
    forward read for an upstream u = dL/dy and of the costate read for w = dL/dg_in.
    Each call runs the retention scan twice (the state at every chunk start,
    forwards and over reversed inputs) and one per-chunk kernel."""

    kind = "gate_grads"

    def __init__(self, gl, wl, device, rank):
        LinearJob.__init__(self, gl, wl, device, rank, "alpha")
        gen = torch.Generator(device=device)
        gen.manual_seed(wl.seed * 1000 + 31)
        dt = self.inp["x"].dtype
        self.inp["u"] = torch.randn(self.inp["g_hat"].shape, generator=gen, device=device).to(dt)
        self.inp["w"] = torch.randn(self.inp["x"].shape, generator=gen, device=device).to(dt)
        shape = (wl.L, wl.B, wl.T, wl.H)
        self.outs = {k: torch.empty(shape, device=device) for k in ("dla_f", "deta_f", "dla_c", "deta_c")}
        from paper_2609_34174_gb300 import _binding as _B
        d = _B._Desc(wl.L, wl.B, wl.T, wl.H, wl.d_in, wl.d_out, 1 if wl.dtype == "bf16" else 0, 0)
        lib = _B.load_library()
        nb = max(lib.gradlev_gate_grads_workspace_bytes(ctypes.byref(d), 0),
                 lib.gradlev_gate_grads_workspace_bytes(ctypes.byref(d), 1))
        self.ws = torch.empty(max(256, int(nb)), dtype=torch.uint8, device=device)
        self.in_keys = ("x", "g_hat", "g_out", "u", "w", "eta_t", "alpha_t")
        self.out_keys = ("dla_f", "deta_f", "dla_c", "deta_c")
        # per read: the chunk aggregates, the carried chunk states, the per-chunk expansion
        self.launches_per_step = 2 * 3
        self.kernel = {"fwd": "gate_agg_tc_kernel + gate_state_scan_kernel + gate_chunk_tc_kernel, forward read",
                       "costate": "gate_agg_tc_kernel + gate_state_scan_kernel + gate_chunk_tc_kernel, costate read"}

    def _run(self, src, cut, ws):
        gl, o = self.gl, self.outs
        with nvtx("gradlev gate_grads forward read"):
            gl.gate_grads(cut(src["x"]), cut(src["g_hat"]), cut(src["eta_t"]), cut(src["u"]),
                          alpha=cut(src["alpha_t"]), dlog_alpha=cut(o["dla_f"]), deta=cut(o["deta_f"]),
                          workspace=ws)
        yield
        with nvtx("gradlev gate_grads costate read"):
            gl.gate_grads(cut(src["x"]), cut(src["g_hat"]), cut(src["eta_t"]), cut(src["w"]),
                          alpha=cut(src["alpha_t"]), read="costate", g_out=cut(src["g_out"]),
                          dlog_alpha=cut(o["dla_c"]), deta=cut(o["deta_c"]), workspace=ws)
        yield

    def counts(self, scan):
        """Per token and unit: two retention scans (each that of the chunk kernel) and the
        per-chunk kernel's C*(d+m) + 4*d*m flops; compulsory bytes e*(d + 2m) + 16 for the
        forward read's derivatives (x, ghat, u, eta_t, alpha_t in; two fp32 outputs) and
        e*(2d + 2m) + 16 for the costate read's (g_out too)."""
        wl = self.wl
        e = 2 if wl.dtype == "bf16" else 4
        d, m = wl.d_in, wl.d_out
        tu = wl.L * wl.B * wl.T * wl.H
        flops = tu * (2 * (4 * d * m + COUNT_CHUNK * (d + m)) + 2 * COUNT_CHUNK * (d + m) + 4 * d * m)
        if scan == "fwd":
            return flops, tu * (e * (d + 2 * m) + 16)
        return flops, tu * (e * (2 * d + 2 * m) + 16)

    def config(self):
        c = LinearJob.config(self)
        c["computes"] = ("alpha_t dL/dalpha_t and dL/deta_t of the forward and costate reads "
                         "(state dumps of the retention scan + per-chunk expansion)")
        return c

    def oracle_run(self, inp, n_units, cores, t_tokens=None):
        """The fp64 oracle's gate derivatives of both reads for the first n_units units."""
        import numpy as np
        import oracle
        wl = self.wl
        units = [(l, b, h) for l in range(wl.L) for b in range(wl.B) for h in range(wl.H)]
        units = units[:n_units]
        f = lambda k: W.units_fp64(inp[k], units)
        x, g, go, u, w = f("x"), f("g_hat"), f("g_out"), f("u"), f("w")
        gates = lambda k: np.stack([inp[k][l, b, :, h].double().cpu().numpy() for (l, b, h) in units])
        et, al = gates("eta_t"), gates("alpha_t")
        t = time.perf_counter()
        oracle.gate_grads(x, g, et, al, u, x, nthreads=cores)
        oracle.gate_grads(x, g, et, al, go, w, nthreads=cores)
        return time.perf_counter() - t, len(units) * wl.T / wl.H

    def sample_text(self, n, t_tokens=None):
        return (f"{n} of {self.n_units()} (layer, batch, head) units at full T={self.wl.T}: "
                f"gate derivatives of both reads, fp64")


def make_job(gl, wl, device, rank, gates=None, grads=False, fused=False):
    if fused:
        if isinstance(wl, W.MLPWorkload) or gates or grads:
            raise SystemExit("--fused applies to the ungated linear workloads")
        return FusedJob(gl, wl, device, rank)
    if grads:
        if isinstance(wl, W.MLPWorkload) or gates not in (None, "alpha"):
            raise SystemExit("--grads applies to the linear workloads, ungated or with --gates alpha")
        if gates == "alpha":
            return GateGradsJob(gl, wl, device, rank)
        return GradsJob(gl, wl, device, rank)
    if isinstance(wl, W.MLPWorkload):
        if gates:
            raise SystemExit("--gates applies to the linear workloads")
        return MLPJob(gl, wl, device, rank)
    return LinearJob(gl, wl, device, rank, gates)


def cpu_baseline(job, inp, target_s=12.0):
    """The fp64 oracle (as it stands) on a bounded sample of the workload, all host cores."""
    cores = len(os.sched_getaffinity(0))
    if job.kind == "mlp":
        # calibrate on a short prefix of one sequence per core, then grow the prefix
        n = min(job.n_units(), cores)
        t_try = 128
        dt0, _ = job.oracle_run(inp, n, cores, t_try)
        t_tok = int(min(job.wl.T, max(t_try, t_try * target_s / max(dt0, 1e-9))))
        dt, tokens = job.oracle_run(inp, n, cores, t_tok)
        sample = job.sample_text(n, t_tok)
    else:
        n0 = min(job.n_units(), cores)
        dt0, _ = job.oracle_run(inp, n0, cores)
        per_unit = dt0 / n0
        n = int(max(n0, min(job.n_units(), target_s / max(per_unit, 1e-9))))
        n = max(cores, n // cores * cores) if n >= cores else n
        n = min(n, job.n_units())
        dt, tokens = job.oracle_run(inp, n, cores)
        sample = job.sample_text(n)
    return {"value": round(tokens / dt, 1), "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": sample, "seconds": round(dt, 2)}


def e2e_measure(job, steps, stream):
    """The same step through the public API from pinned host buffers, copies inside.

    The step is cut into chunks along its leading independent dimension (layers,
    or batch rows) and pipelined over three streams: the host-to-device copy of
    chunk c+1 and the device-to-host copy of chunk c-1 overlap the scans of chunk
    c.  Every input byte is copied in and every result byte out on every step."""
    dev_id = job.ws.device
    host = {k: job.inp[k].cpu().pin_memory() for k in job.in_keys}
    # two sets of device inputs and outputs, used by alternate steps: a step's copies
    # in do not wait for the previous step's scans of the same chunk, nor its scans
    # for the previous step's copies out
    devs = [{k: torch.empty_like(job.inp[k]) for k in job.in_keys} for _ in range(2)]
    outs = [job.outs, {k: torch.empty_like(v) for k, v in job.outs.items()}]
    dev = devs[0]
    hout = {k: torch.empty(job.outs[k].shape, dtype=job.outs[k].dtype, pin_memory=True)
            for k in job.out_keys}
    bi = _bytes(*host.values())
    bo = _bytes(*hout.values())
    chunks = job.e2e_chunks()
    ws = torch.empty(max(job.ws.numel(), job.e2e_workspace_bytes()), dtype=torch.uint8,
                     device=dev_id)
    s_in = torch.cuda.Stream(dev_id)
    s_run = torch.cuda.Stream(dev_id)
    s_out = torch.cuda.Stream(dev_id)
    n = len(chunks)
    ev_in = [[torch.cuda.Event() for _ in range(n)] for _ in range(2)]
    ev_run = [[torch.cuda.Event() for _ in range(n)] for _ in range(2)]
    ev_out = [[torch.cuda.Event() for _ in range(n)] for _ in range(2)]
    started = [[False] * n for _ in range(2)]
    par = [0]

    def one():
        b = par[0]
        dv_set = devs[b]
        job.outs = outs[b]
        for c, sl in enumerate(chunks):
            with torch.cuda.stream(s_in):
                if started[b][c]:
                    s_in.wait_event(ev_run[b][c])  # this set's last scans of chunk c are done
                for k, hv, dv in job.e2e_inputs(host, dv_set, sl, c == 0):
                    dv.copy_(hv, non_blocking=True)
                ev_in[b][c].record(s_in)
            with torch.cuda.stream(s_run):
                s_run.wait_event(ev_in[b][c])
                if started[b][c]:
                    s_run.wait_event(ev_out[b][c])  # this set's last results have been read out
                job.e2e_step(dv_set, sl, ws)
                ev_run[b][c].record(s_run)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_run[b][c])
                for dv, hv in job.e2e_outputs(hout, sl):
                    hv.copy_(dv, non_blocking=True)
                ev_out[b][c].record(s_out)
            started[b][c] = True
        par[0] = b ^ 1

    one()
    one()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(s_in)
    for _ in range(steps):
        one()
    s_out.wait_stream(s_in)
    s_out.wait_stream(s_run)
    e1.record(s_out)
    torch.cuda.synchronize()
    sec = e0.elapsed_time(e1) / 1e3
    # the results that came back agree with the whole-step call on resident inputs
    job.outs = outs[0]
    job.step()
    torch.cuda.synchronize()
    worst = 0.0
    for k in job.out_keys:
        ref = job.outs[k].double().cpu()
        got = hout[k].double()
        worst = max(worst, float((got - ref).norm() / max(float(ref.norm()), 1e-30)))
    if not worst <= 2e-2:
        raise RuntimeError(f"pipelined end-to-end results differ from the resident step: {worst:.3e}")
    ms = sec / steps * 1e3
    return {"value": round(job.tokens * steps / sec, 1), "unit": UNIT, "h2d_bytes_per_step": bi,
            "d2h_bytes_per_step": bo, "steps": steps, "ms_per_step": round(ms, 3),
            "pipeline": (f"{n} chunks, copies overlapped with the scans on three streams, "
                         "two sets of device buffers"),
            "rel_l2_vs_resident_step": worst}


# ---------------------------------------------------------- DRAM traffic
TRAFFIC_RECORD = os.path.join(ROOT, "profiles", "dram_traffic.txt")
KERNEL_SOURCES = ("paper_2609_34174_gb300/csrc/scan_tc.cu", "paper_2609_34174_gb300/csrc/sm103_ptx.cuh",
                  "paper_2609_34174_gb300/csrc/scan_common.cuh",
                  "paper_2609_34174_gb300/csrc/gradlev_host.cu")


def kernel_source_digest():
    import hashlib
    h = hashlib.sha1()
    for rel in KERNEL_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def recorded_traffic(workload_key, scan):
    """DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) of the
    dominant kernel from the committed ncu record, or None when no record exists
    for this workload and scan or the kernel sources changed since it was taken."""
    try:
        with open(TRAFFIC_RECORD) as f:
            rec = json.load(f)
    except Exception:
        return None
    if rec.get("kernel_source_sha1") != kernel_source_digest():
        return None
    ent = rec.get("entries", {}).get(f"{workload_key}:{scan}")
    return None if ent is None else int(ent["bytes_per_launch"])


# ------------------------------------------------------------- multi-rank
def combine_ranks(step_ms, tokens_per_rank, world, device):
    """Whole-job step time and throughput over N replicas: every rank processes
    its own copy of the workload, the step time is the maximum over ranks, and
    the value counts all ranks' tokens.  Returns (step_ms, tokens/s)."""
    if world > 1:
        t = torch.tensor([float(step_ms)], dtype=torch.float64, device=device)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        step_ms = float(t.item())
    return step_ms, world * tokens_per_rank / (step_ms / 1e3)


# ------------------------------------------------------------------- arms
def run_reference(args, wl, rank, world):
    """The oracle as the reference arm, on this host's cores (rank 0 only)."""
    if rank != 0:
        return None
    import oracle

    oracle.build()
    cores = len(os.sched_getaffinity(0))
    metric = METRIC
    job_cfg = {}
    if args.workload == "decode_mlp":
        inp = W.make_mlp(wl, device="cpu")
        f = lambda t, T: t[:, :T].to(torch.float64).numpy()
        W1, W2 = inp["W1"].double().numpy(), inp["W2"].double().numpy()
        t_tok = 16

        def run():
            t0 = time.perf_counter()
            oracle.mlp_deploy(f(inp["x"], t_tok), W1, W2, wl.eta1, wl.eta2,
                              gout=f(inp["g_out"], t_tok), act=oracle.ACT_GELU_TANH,
                              nthreads=min(cores, wl.B))
            return time.perf_counter() - t0, wl.B * t_tok

        sample = f"{wl.B} sequences x {t_tok} tokens of the deployed MLP per step, fp64"
        metric = DECODE_METRIC
    elif args.grads and args.gates == "alpha":
        job = GateGradsJob.__new__(GateGradsJob)
        job.wl = wl
        inp = W.make_linear(wl, device="cpu")
        inp.update(make_gates(wl, "alpha", "cpu"))
        gen = torch.Generator()
        gen.manual_seed(wl.seed * 1000 + 31)
        dt = inp["x"].dtype
        inp["u"] = torch.randn(inp["g_hat"].shape, generator=gen).to(dt)
        inp["w"] = torch.randn(inp["x"].shape, generator=gen).to(dt)
        n = min(job.n_units(), cores)
        run = lambda: job.oracle_run(inp, n, cores)
        sample = job.sample_text(n) + " per step"
        metric = GATE_GRADS_METRIC
    elif args.grads:
        job = GradsJob.__new__(GradsJob)
        job.wl = wl
        inp = W.make_linear(wl, device="cpu")
        gen = torch.Generator()
        gen.manual_seed(wl.seed * 1000 + 29)
        dt = inp["x"].dtype
        inp["u"] = torch.randn(inp["g_hat"].shape, generator=gen).to(dt)
        inp["w"] = torch.randn(inp["x"].shape, generator=gen).to(dt)
        n = min(job.n_units(), max(cores, 2 * cores))
        run = lambda: job.oracle_run(inp, n, cores)
        sample = (f"{n} of {job.n_units()} (layer, batch, head) units at full T={wl.T} per step, "
                  f"suffix reads and dots of both reads, fp64")
        metric = GRADS_METRIC
    elif isinstance(wl, W.MLPWorkload):
        inp = W.make_mlp(wl, device="cpu")
        job = MLPJob.__new__(MLPJob)
        job.wl = wl
        n = min(wl.B, cores)
        t_tok = min(wl.T, 256)
        run = lambda: job.oracle_run(inp, n, cores, t_tok)
        sample = job.sample_text(n, t_tok) + " per step"
    else:
        inp = W.make_linear(wl, device="cpu")
        job = LinearJob.__new__(LinearJob)
        job.wl = wl
        job.gates = args.gates
        inp.update(make_gates(wl, args.gates, "cpu"))
        n = min(job.n_units(), max(cores, 2 * cores))
        run = lambda: job.oracle_run(inp, n, cores)
        sample = job.sample_text(n) + " per step"
        job_cfg = job.config()
    for _ in range(args.warmup):
        run()
    sec = 0.0
    tokens = 0.0
    for _ in range(args.steps):
        dt, tk = run()
        sec += dt
        tokens += tk
    value = tokens / sec
    return {"impl": "reference", "metric": metric, "value": round(value, 1), "unit": UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(sec / args.steps * 1e3, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": f"{args.workload}: {wl.name}", **job_cfg, "sample": sample},
            "cpu_baseline": {"value": round(value, 1), "unit": UNIT, "cores": cores,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 1), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


GRADS_METRIC = ("tokens/s of dL/deta_t per read (forward read, costate read) at 1 GB300; "
                "% of roofline")
GATE_GRADS_METRIC = ("tokens/s of the gate derivatives (alpha_t dL/dalpha_t, dL/deta_t) per read "
                     "(forward read, costate read) at 1 GB300; % of HBM roofline")
DECODE_METRIC = "deployment tokens/s (one token per sequence per step) at 1 GB300; % of HBM roofline"


class DecodeMLPJob:
    """Deployment of the two-layer MLP (Sec. 3; Appendix A): every step each of the
    B sequences advances one token.  Layer 1 is read (sigma fused), then layer 2;
    with the scored token's costate, layer 2 is written together with its costate
    read (sigma' fused, giving gz) and layer 1 is written with gz.  The fast
    weights live on the device as Delta = W - W0 in fp32 between steps."""

    kernels = ("read L1", "read L2", "write L2 + g_in", "write L1")

    def __init__(self, gl, wl, device, rank):
        self.gl, self.wl = gl, wl
        inp = W.make_mlp(wl.resized(seed=wl.seed + 1000 * rank), device=device)
        self.inp = inp
        B, d, m, k = wl.B, wl.d, wl.m, wl.k
        dt = inp["x"].dtype
        self.W1 = inp["W1"].reshape(1, 1, m, d)
        self.W2 = inp["W2"].reshape(1, 1, k, m)
        self.D1 = torch.zeros(1, B, 1, m, d, device=device)
        self.D2 = torch.zeros(1, B, 1, k, m, device=device)
        mk = lambda w: torch.empty(1, B, 1, w, dtype=dt, device=device)
        self.x, self.g = mk(d), mk(k)           # the token's input and scored costate
        self.z, self.h, self.y, self.gz = mk(m), mk(m), mk(k), mk(m)
        self.eta1 = torch.full((1, B, 1), wl.eta1, device=device)
        self.eta2 = torch.full((1, B, 1), wl.eta2, device=device)
        self.ws = torch.empty(max(256, gl.decode_workspace_bytes(1, B, 1, m, k)), dtype=torch.uint8,
                              device=device)
        self.t = 0

    def load_token(self, t):
        T = self.wl.T
        self.x.copy_(self.inp["x"][:, t % T].reshape(self.x.shape))
        self.g.copy_(self.inp["g_out"][:, t % T].reshape(self.g.shape))

    def launch(self, i):
        gl, wl = self.gl, self.wl
        if i == 0:
            gl.decode_read(self.x, self.W1, self.D1, act=wl.act, y=self.z, act_out=self.h)
        elif i == 1:
            gl.decode_read(self.h, self.W2, self.D2, y=self.y)
        elif i == 2:
            gl.decode_write(self.h, self.g, self.W2, self.D2, self.eta2, act=wl.act, z=self.z,
                            g_in=self.gz, workspace=self.ws)
        else:
            gl.decode_write(self.x, self.gz, self.W1, self.D1, self.eta1, want_g_in=False)

    def step(self):
        for i in range(4):
            self.launch(i)

    def kernel_bytes(self, i):
        """Algorithmic HBM bytes of kernel i: Delta once per sequence (read, or read
        and written), W0 once (shared by the B sequences), token vectors."""
        wl = self.wl
        B, d, m, k = wl.B, wl.d, wl.m, wl.k
        e = 2 if wl.dtype == "bf16" else 4
        if i == 0:
            return 4 * m * d * (B + 1) + e * B * (d + 2 * m)
        if i == 1:
            return 4 * k * m * (B + 1) + e * B * (m + k)
        if i == 2:
            return 4 * k * m * (2 * B + 1) + e * B * (m + k + m + m)
        return 4 * m * d * 2 * B + e * B * (d + m)

    def step_bytes(self):
        return sum(self.kernel_bytes(i) for i in range(4))


def _graph(fn, stream):
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        fn()
    return g


def run_decode(args, wl, rank, world, local_rank):
    """Deployment steps of the paper-shaped final MLP, replayed as one CUDA graph per
    step (the four kernels back to back, no host in between)."""
    import paper_2609_34174_gb300 as gl

    device = torch.device("cuda", local_rank)
    torch.cuda.set_device(device)
    gl.load_library()
    job = DecodeMLPJob(gl, wl, device, rank)
    cap = torch.cuda.Stream(device)
    job.load_token(0)
    with torch.cuda.stream(cap):
        job.step()  # warm the binding before capture
    torch.cuda.synchronize()
    g_step = _graph(job.step, cap)
    g_kern = [_graph(lambda i=i: job.launch(i), cap) for i in range(4)]
    # L2 flush between steps: write a buffer larger than L2, then read another one,
    # so that no dirty lines are left for the timed step to write back
    fw = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device=device)
    fr = torch.ones(2 * L2_BYTES // 4, dtype=torch.float32, device=device)

    def flush():
        fw.zero_()
        fr.sum()

    stream = torch.cuda.current_stream(device)
    for t in range(args.warmup):
        job.load_token(t)
        g_step.replay()
    torch.cuda.synchronize()
    sampler = ClockSampler(local_rank)
    sampler.start()
    time.sleep(0.3)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    sampler.mark()
    for i in range(args.steps):
        job.load_token(args.warmup + i)
        flush()
        ev[i][0].record(stream)
        g_step.replay()
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    sampler.mark()
    # per-kernel times (each kernel alone after a flush), for the roofline of each
    kev = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            for _ in range(args.steps)] for _ in range(4)]
    for j in range(args.steps):
        for i in range(4):
            flush()
            kev[i][j][0].record(stream)
            g_kern[i].replay()
            kev[i][j][1].record(stream)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    time.sleep(0.25)
    sampler.stop()
    step_ms = statistics.median(a.elapsed_time(b) for a, b in ev)
    step_ms, value = combine_ranks(step_ms, wl.B, world, device)
    pk = peaks()
    kern = {}
    for i, name in enumerate(job.kernels):
        ms = statistics.median(a.elapsed_time(b) for a, b in kev[i])
        nb = job.kernel_bytes(i)
        ach = nb / (ms / 1e3) / 1e9
        kern[name] = {"ms": round(ms, 4), "bytes": nb, "achieved_gbs": round(ach, 1),
                      "frac": round(ach / pk["hbm_gbs"], 4)}
    dom = max(kern, key=lambda n: kern[n]["ms"])
    rl = {"bound": "hbm", "achieved": kern[dom]["achieved_gbs"], "peak": pk["hbm_gbs"],
          "unit": "GB/s", "frac": kern[dom]["frac"], "traffic": None,
          "kernel": f"decode {dom} ({'write_kernel' if 'write' in dom else 'read_kernel'})",
          "peak_source": pk.get("source", "MEASURED_PEAKS.json"),
          "step_frac": round(job.step_bytes() / (step_ms / 1e3) / 1e9 / pk["hbm_gbs"], 4)}
    cfg = {"workload": f"{args.workload}: deployment of {wl.name}", "B": wl.B,
           "widths": [wl.d, wl.m, wl.k], "act": wl.act, "eta": [wl.eta1, wl.eta2],
           "state": "Delta fp32 on the device", "tokens_per_step": wl.B,
           "parallelism": f"replicas x{world}", "l2": "L2 flushed between steps",
           "launch": "CUDA graph per step"}
    line = {"metric": DECODE_METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(step_ms, 4),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype,
            "data": "synthetic", "config": cfg, "kernels": kern, "roofline": rl,
            "clocks": sampler.summary(), "gpu_launches": 4 * args.steps}
    if rank == 0 and world == 1 and not args.no_e2e:
        line["e2e"] = decode_e2e(job, g_step, max(20, min(args.steps, 200)), stream)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle

        oracle.build()
        line["cpu_baseline"] = decode_cpu_baseline(wl, job.inp)
    return line


def decode_e2e(job, g_step, steps, stream):
    """Deployment steps through the public API from pinned host memory: each step
    copies the token's x and scored costate in and reads y back."""
    B = job.wl.B
    hx = job.inp["x"].cpu().pin_memory()
    hg = job.inp["g_out"].cpu().pin_memory()
    hy = torch.empty(job.y.shape, dtype=job.y.dtype, pin_memory=True)
    T = job.wl.T
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    for t in range(steps):
        job.x.copy_(hx[:, t % T].reshape(job.x.shape), non_blocking=True)
        job.g.copy_(hg[:, t % T].reshape(job.g.shape), non_blocking=True)
        g_step.replay()
        hy.copy_(job.y, non_blocking=True)
    e1.record(stream)
    torch.cuda.synchronize()
    sec = e0.elapsed_time(e1) / 1e3
    return {"value": round(steps * B / sec, 1), "unit": UNIT,
            "h2d_bytes_per_step": _bytes(job.x, job.g), "d2h_bytes_per_step": _bytes(hy),
            "note": "L2 not flushed: consecutive tokens, as in deployment"}


def decode_cpu_baseline(wl, inp, target_s=12.0):
    """The fp64 oracle's deployed MLP on a bounded number of tokens per sequence."""
    import oracle
    cores = len(os.sched_getaffinity(0))
    f = lambda t, T: t[:, :T].to(torch.float64).cpu().numpy()
    W1 = inp["W1"].double().cpu().numpy()
    W2 = inp["W2"].double().cpu().numpy()

    def run(T):
        t0 = time.perf_counter()
        oracle.mlp_deploy(f(inp["x"], T), W1, W2, wl.eta1, wl.eta2, gout=f(inp["g_out"], T),
                          act=oracle.ACT_GELU_TANH, nthreads=min(cores, wl.B))
        return time.perf_counter() - t0

    dt0 = run(4)
    T = int(min(wl.T, max(4, 4 * target_s / max(dt0, 1e-9))))
    dt = run(T)
    return {"value": round(wl.B * T / dt, 1), "unit": UNIT, "cores": min(cores, wl.B),
            "kind": "oracle", "seconds": round(dt, 2),
            "sample": f"{wl.B} sequences x first {T} tokens of the deployed MLP, fp64"}


def side_scans(gl, key, device, steps=20, warmup=3):
    """Per-scan times and rooflines of another linear workload at its full size,
    timed like the headline (CUDA events on the launching stream, inputs larger
    than L2), so that one default run also records it."""
    job = make_job(gl, W.workload(key), device, 0)
    for _ in range(warmup):
        job.step()
    torch.cuda.synchronize()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    for i in range(steps):
        job.step(events=ev[i])
    torch.cuda.synchronize()
    if gl.workspace_status(job.ws) != 0:
        raise RuntimeError("device-side timeout reported by the scan kernels")
    pk = peaks()
    out = {"workload": f"{key}: {job.wl.name}", "steps": steps}
    for name, a, b in (("fwd", 0, 1), ("costate", 1, 2)):
        ms = sum(e[a].elapsed_time(e[b]) for e in ev) / steps
        fl, nb = job.counts(name)
        out[name] = {"ms": round(ms, 4), "tokens_per_s": round(job.tokens / (ms / 1e3), 1),
                     "roofline": roofline_entry(fl, nb, ms / 1e3, pk)}
    del job
    torch.cuda.empty_cache()
    return out


def side_fused(gl, key, device, steps=20, warmup=3):
    """The fused pass (both reads in one call) on a linear workload at full size, timed
    like the headline; its roofline counts its own compulsory bytes."""
    job = FusedJob(gl, W.workload(key), device, 0)
    for _ in range(warmup):
        job.step()
    torch.cuda.synchronize()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    for i in range(steps):
        job.step(events=ev[i])
    torch.cuda.synchronize()
    if gl.workspace_status(job.ws) != 0:
        raise RuntimeError("device-side timeout reported by the fused kernel")
    ms = sum(e[0].elapsed_time(e[1]) for e in ev) / steps
    fl, nb = job.counts("fused")
    out = {"workload": f"{key}: {job.wl.name}", "steps": steps, "ms": round(ms, 4),
           "tokens_per_s": round(job.tokens / (ms / 1e3), 1),
           "roofline": roofline_entry(fl, nb, ms / 1e3, peaks())}
    del job
    torch.cuda.empty_cache()
    return out


def run_gradlev(args, wl, rank, world, local_rank):
    import paper_2609_34174_gb300 as gl

    device = torch.device("cuda", local_rank)
    torch.cuda.set_device(device)
    gl.load_library()
    job = make_job(gl, wl, device, rank, args.gates, args.grads, args.fused)
    flush = None
    if job.input_bytes() < 2 * L2_BYTES:
        flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device=device)
    stream = torch.cuda.current_stream(device)

    for _ in range(args.warmup):
        job.step()
    torch.cuda.synchronize()
    if gl.workspace_status(job.ws) != 0:
        raise RuntimeError("device-side timeout reported by the scan kernels")

    sampler = ClockSampler(local_rank)
    sampler.start()
    # let the sampler produce a first line before the timed region
    time.sleep(0.3)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    sampler.mark()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for i in range(args.steps):
        if flush is not None:
            flush.zero_()
        job.step(events=ev[i])
    t_end.record(stream)
    torch.cuda.synchronize()
    sampler.mark()
    if world > 1:
        torch.distributed.barrier()
    time.sleep(0.25)
    sampler.stop()
    if gl.workspace_status(job.ws) != 0:
        raise RuntimeError("device-side timeout reported by the scan kernels")

    total_ms = t_start.elapsed_time(t_end)
    fwd_ms = sum(e[0].elapsed_time(e[1]) for e in ev) / args.steps
    cos_ms = sum(e[1].elapsed_time(e[2]) for e in ev) / args.steps
    step_ms = total_ms / args.steps
    if flush is not None:
        # the flush is not part of the step: take the scans' own time
        step_ms = max(fwd_ms + cos_ms, 1e-9)
    step_ms, value = combine_ranks(step_ms, job.tokens, world, device)
    pk = peaks()
    scans = {}
    reads = (("fused", fwd_ms),) if job.kind == "fused" else (("fwd", fwd_ms), ("costate", cos_ms))
    for name, ms in reads:
        fl, nb = job.counts(name)
        scans[name] = {"ms": round(ms, 4), "tokens_per_s": round(job.tokens / (ms / 1e3), 1),
                       "roofline": roofline_entry(fl, nb, ms / 1e3, pk)}
    dominant = "fused" if job.kind == "fused" else ("costate" if cos_ms >= fwd_ms else "fwd")
    rl = dict(scans[dominant]["roofline"])
    rl["kernel"] = job.kernel[dominant]
    rl["traffic"] = (None if (args.resize or args.gates or args.grads)
                     else recorded_traffic(args.workload, dominant))
    cfg = {"workload": f"{args.workload}: {wl.name}", **job.config(),
           "tokens_per_step": job.tokens, "parallelism": f"replicas x{world}",
           "l2": "inputs larger than L2" if flush is None else "L2 flushed between steps"}
    if job.kind == "fused":
        cfg["step"] = "forward and costate reads in one pass (gradlev_fused_scan)"
    line = {"metric": (GATE_GRADS_METRIC if args.gates == "alpha" else GRADS_METRIC) if args.grads else METRIC,
            "value": round(value, 1),
            "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(step_ms, 4),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype,
            "data": "synthetic", "config": cfg, "scans": scans, "roofline": rl,
            "clocks": sampler.summary(), "gpu_launches": job.launches_per_step * args.steps}
    if rank == 0 and world == 1 and not args.no_e2e:
        line["e2e"] = e2e_measure(job, max(3, min(args.steps, 20)), stream)
    if (rank == 0 and world == 1 and args.workload == "c5" and not
            (args.gates or args.grads or args.fused or args.no_side)):
        # the long-context workload, the other one with a roofline target, and both
        # workloads' reads in one fused pass
        line["also"] = {"c4": side_scans(gl, "c4", device),
                        "fused": {k: side_fused(gl, k, device) for k in ("c5", "c4")}}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle

        oracle.build()
        line["cpu_baseline"] = cpu_baseline(job, job.inp)
    return line


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default="c5",
                    choices=["c1", "c2", "c3", "c4", "c5", "paper_mlp", "decode_mlp"])
    ap.add_argument("--impl", default="gradlev", choices=["gradlev", "reference"])
    ap.add_argument("--resize", default="",
                    help="comma-separated K=V overrides of the workload's sizes (e.g. L=2), "
                         "for small profiling captures; the headline uses the full workload")
    ap.add_argument("--gates", default=None, choices=["eta", "alpha", "docs"],
                    help="time the gated scans of Eq. 2: per-token eta_t, eta_t with retention, "
                         "or document resets of packed sequences")
    ap.add_argument("--grads", action="store_true",
                    help="time the step-size gradients of both reads (suffix reads) instead")
    ap.add_argument("--fused", action="store_true",
                    help="time both reads of each map in one pass (gradlev_fused_scan) as the step")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-side", action="store_true",
                    help="skip the long-context (c4) scans added to the default line")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        args.warmup = 3

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    decode = args.workload == "decode_mlp"
    wl = W.workload("paper_mlp" if decode else args.workload)
    if args.resize:
        kw = {}
        for item in args.resize.split(","):
            k, v = item.split("=")
            kw[k.strip()] = int(v) if v.strip().lstrip("-").isdigit() else float(v)
        wl = wl.resized(**kw)
        args.workload = f"{args.workload}[{args.resize}]"

    if args.impl == "reference":
        line = run_reference(args, wl, rank, world)
        if line is not None:
            print(json.dumps(line), flush=True)
        return 0

    if world > 1:
        torch.cuda.set_device(local_rank)
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    try:
        if decode:
            line = run_decode(args, wl, rank, world, local_rank)
        else:
            line = run_gradlev(args, wl, rank, world, local_rank)
        if rank == 0:
            print(json.dumps(line), flush=True)
    finally:
        if world > 1:
            torch.distributed.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
