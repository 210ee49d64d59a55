"""Benchmark of checkpoint-aligned restore-and-resume on GB300.

One step = the nine-length serial hybrid workload for one seed: for each
prompt length L in 512..4608 (step 512) of a 12-layer synthetic stack
(9 linear-attention layers, 16 heads, d=128; 3 full-attention layers,
4 KV heads, head_dim 128, page 16) with state checkpoints every 256 tokens:
strict-prefix alignment (c = L-256), KV page restore for [0,c), state
restore at c, the 256-token tail prefill emitting the checkpoint at L, then
64 single-token decode steps of the linear recurrence.  Seeds 0..3 rotate
across steps, so consecutive steps touch different inputs (the per-step
working set is larger than L2).

Reported ``value``: resumed tokens per second = (tail tokens + decode
tokens) of the step's nine requests / step time, summed over ranks.
Also reported: the prefill kernel's roofline, KV restore GB/s on the
KV-stress workload (48 layers x 256 pages x 64 KiB, 64 serial requests
into a paged cache of up to 180 GB), resumed vs recomputed TTFT per length,
an end-to-end figure through host (pinned) buffers, and the float64 oracle
timed on the host cores as a CPU baseline.

``--impl reference`` times the oracle itself (CPU) on a bounded sample of
the same workload.

``--case decode|prefill|kv|ckpt|sweep`` runs one small piece of the workload
and prints its CUDA-event times: the cases the committed ncu captures under
profiles/ were taken on (``--source-hashes`` prints the source hash each
profiles/*.txt row is keyed on).  ``--case long`` prints resumed vs
recomputed TTFT for the long-context stack (L = 16k/32k/64k, batch 4).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

from hs_inputs import HYBRID12, KVSTRESS, SWEEP_LENGTHS, DECODE_STEPS  # noqa: E402

METRIC = ("resumed-tail tokens/s & restore GB/s on 1 GB300 (% roofline); TTFT vs recompute")
WORKLOAD = ("hybrid-12L serial sweep: 9 linear layers (16 heads, d=128, fp32 state) + 3 full layers "
            "(4 KV heads, head_dim 128, bf16, page 16); L=512..4608 step 512, checkpoints every 256, "
            "complete hit -> tail 256 + 64 decode steps; seeds 0..3 rotating")
TAIL = 256
N_REQ = len(SWEEP_LENGTHS)
TOKENS_PER_STEP = N_REQ * (TAIL + DECODE_STEPS)


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


# ---------------------------------------------------------------------------
# algorithmic bytes (the roofline numerators)
# ---------------------------------------------------------------------------

def gla_bytes(n_problems, n_heads, d, tokens_per_problem, ckpts_per_problem):
    """q,k,v bf16 + log-gates f32 + o f32 per token-head, plus the state read
    and written once per head, plus each emitted checkpoint."""
    per_tok = d * (2 + 2 + 2 + 4 + 4)
    state = d * d * 4
    return n_problems * n_heads * (tokens_per_problem * per_tok + 2 * state
                                   + ckpts_per_problem * state)


def kv_bytes(n_layers, n_pages, page_bytes):
    return 2 * n_layers * n_pages * page_bytes


KERNEL_OF = {"decode": "gla_decode_kernel<128>", "prefill": "gla_chunked_tc_kernel",
             "restore": "restore_request_kernel"}

# the source file of each kernel named in profiles/*.txt (a "kernel@workload" key names the
# kernel before the "@")
KERNEL_SRC = {"gla_decode_kernel": "gla_decode.cu", "gla_chunked_tc_kernel": "gla_chunked_tc.cu",
              "gla_recurrent_kernel": "gla_recurrent.cu", "restore_request_kernel": "restore_request.cu",
              "kv_scatter_kernel": "kv_scatter.cu", "kv_gather_kernel": "kv_scatter.cu",
              "kv_slices_kernel": "kv_scatter.cu", "slot_copy_kernel": "slot_copy.cu",
              "gla_scan_kernel": "gla_scan.cu", "gla_dstate_kernel": "gla_dstate.cu"}
DTYPE = "bf16 q/k/v, fp32 log-gates; fp16 (fast) or tf32 (exact) MMA operands, fp32 accumulate, state and outputs"


def source_files(kernel: str) -> list:
    """The kernel's source file and every local header it includes, directly or through
    other headers (in breadth-first order)."""
    import re
    name = kernel.split("@")[0].split("<")[0]
    dirs = [os.path.join(ROOT, "paper_2609_15030_gb300", "csrc"), os.path.join(ROOT, "include")]
    files, todo = [], [os.path.join(dirs[0], KERNEL_SRC[name])]
    while todo:
        f = todo.pop(0)
        if f in files:
            continue
        files.append(f)
        for inc in re.findall(r'^\s*#\s*include\s+"([^"]+)"', open(f).read(), re.M):
            for d in dirs:
                cand = os.path.join(d, inc)
                if os.path.exists(cand):
                    todo.append(cand)
                    break
    return files


def _strip_comments(src: str) -> str:
    """C/C++ source without its comments (string literals in these files hold no comment
    markers) and with every run of whitespace made one space, so that a documentation or
    layout edit does not count as a kernel change."""
    import re
    return re.sub(r"\s+", " ", re.sub(r"/\*.*?\*/|//[^\n]*", "", src, flags=re.S)).strip()


def source_hash(kernel: str) -> str:
    """First 12 hex digits of the SHA-256 of the kernel's source files (`source_files`: what
    its machine code depends on), comments left out: a profile row captured under another
    hash describes another kernel."""
    import hashlib
    h = hashlib.sha256()
    for f in source_files(kernel):
        h.update(_strip_comments(open(f).read()).encode())
    return h.hexdigest()[:12]


PROFILES = os.path.join(ROOT, "profiles")


def _profile_rows(fname, ncols):
    """Rows `kernel v1 .. v_ncols source_hash capture ...` of a profiles/ table whose source
    hash still matches the kernel's source; stale rows map to None."""
    p = os.path.join(PROFILES, fname)
    out = {}
    if os.path.exists(p):
        for line in open(p):
            f = line.split()
            if len(f) < ncols + 2 or line.startswith("#"):
                continue
            kern, vals, hsh = f[0], f[1:1 + ncols], f[1 + ncols]
            try:
                fresh = source_hash(kern) == hsh
            except (KeyError, OSError):
                fresh = False
            out[kern] = (vals, f[2 + ncols] if len(f) > 2 + ncols else "") if fresh else None
    return out


def _nvtx(name: str):
    """An NVTX range around one section of the run (visible to ncu --nvtx and nsys);
    a no-op context where torch has no NVTX support."""
    import contextlib
    try:
        import torch
        return torch.cuda.nvtx.range(name)
    except Exception:
        return contextlib.nullcontext()


def _traffic():
    """DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) from the
    committed ncu captures listed in profiles/dram_traffic.txt; None for a kernel whose
    source changed since its capture (the row's source hash no longer matches)."""
    return {k: (int(float(v[0][0])) if v else None) for k, v in _profile_rows("dram_traffic.txt", 1).items()}


def _tensor_pipe():
    """Tensor-pipe utilisation (of active, of elapsed cycles) from the committed ncu captures
    listed in profiles/tensor_pipe.txt; None for a kernel changed since its capture."""
    return {k: ({"active": float(v[0][0]), "elapsed": float(v[0][1]), "source": "ncu " + v[1]}
                if v else None) for k, v in _profile_rows("tensor_pipe.txt", 2).items()}


# ---------------------------------------------------------------------------
# clocks sampler
# ---------------------------------------------------------------------------

class Clocks:
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        import tempfile
        self.path = tempfile.mktemp(prefix="hs_clocks_", suffix=".csv")
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sms, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sms.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for nm, val in zip(names, f[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(nm)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sms) if sms else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sms)}


# ---------------------------------------------------------------------------
# the workload on the device
# ---------------------------------------------------------------------------

def _arena(torch, dev, fields):
    """One device byte buffer holding typed views [(name, dtype, shape)], each view
    starting on a 256-byte boundary."""
    offs, off = [], 0
    for _, dt, shp in fields:
        n = 1
        for x in shp:
            n *= x
        offs.append(off)
        off += -(-(n * torch.empty((), dtype=dt).element_size()) // 256) * 256
    arena = torch.empty(off, dtype=torch.uint8, device=dev)
    views = {}
    for (name, dt, shp), o in zip(fields, offs):
        n = 1
        for x in shp:
            n *= x
        nb = n * torch.empty((), dtype=dt).element_size()
        views[name] = arena[o:o + nb].view(dt).view(shp)
    return arena, views


class Hybrid12:
    """Device-resident buffers for the nine-length serial hybrid workload."""

    def __init__(self, dev, seeds=4, num_blocks=8192):
        import torch
        import paper_2609_15030_gb300 as hs
        from hs_inputs import torch_gen_linear, torch_fill_bf16_normal, gen_block_table
        self.hs, self.torch, self.dev = hs, torch, dev
        S = HYBRID12
        self.S = S
        self.nL, self.nF, self.nH, self.d = S.n_lin, S.n_full, S.n_heads, S.d
        self.T = TAIL + DECODE_STEPS
        self.state_floats = self.nH * self.d * self.d
        self.page_bytes = S.page_bytes
        self.NB = num_blocks
        self.seeds = seeds
        self.stream = torch.cuda.current_stream(dev)
        # paged KV cache: n_full layers x NB blocks
        self.cache = torch.empty((self.nF, num_blocks * self.page_bytes), dtype=torch.uint8, device=dev)
        self.cache_ptrs = hs.ptr_array([self.cache[l] for l in range(self.nF)], dev)
        self.req = []
        for r, L in enumerate(SWEEP_LENGTHS):
            c, n_pages, tail = hs.hs_align_prefix(L, L, list(range(S.ckpt, L + 1, S.ckpt)), S.page)
            assert tail == TAIL
            self.req.append(dict(L=L, c=c, n_pages=n_pages))
        # per (seed, request) inputs, all of a request's in one contiguous arena (so that
        # the end-to-end run moves them with one host-to-device copy)
        self.inp = {}
        tok = (self.nL, self.T, self.nH, self.d)
        for s in range(seeds):
            for r, R in enumerate(self.req):
                q, k, v, a = torch_gen_linear(100 * s + r, 0, self.nL, self.T, self.nH, self.d, dev)
                arena, views = _arena(torch, dev, [
                    ("q", torch.bfloat16, tok), ("k", torch.bfloat16, tok),
                    ("v", torch.bfloat16, tok), ("a", torch.float32, tok),
                    ("staging", torch.uint8, (self.nF, max(R["n_pages"], 1) * self.page_bytes)),
                    ("ck", torch.float32, (self.nL, self.state_floats))])
                views["q"].copy_(q)
                views["k"].copy_(k)
                views["v"].copy_(v)
                views["a"].copy_(a)
                del q, k, v, a
                q, k, v, a, staging, ck = (views[x] for x in ("q", "k", "v", "a", "staging", "ck"))
                torch_fill_bf16_normal(staging, 1000 * s + r)
                ck.copy_(torch.randn((self.nL, self.state_floats), device=dev,
                                     generator=torch.Generator(device=dev).manual_seed(7 * s + r)) * 0.5)
                bt = torch.from_numpy(gen_block_table(s, r, max(R["n_pages"], 1), num_blocks)).to(dev)
                self.inp[(s, r)] = dict(
                    arena=arena, q=q, k=k, v=v, a=a, staging=staging, ck=ck, bt=bt,
                    staging_ptrs=hs.ptr_array([staging[l] for l in range(self.nF)], dev),
                    ck_ptrs=hs.ptr_array([ck[l] for l in range(self.nL)], dev))
        # per-request outputs (reused across seeds)
        self.out = []
        for r, R in enumerate(self.req):
            arena, views = _arena(torch, dev, [
                ("o", torch.float32, tok), ("live", torch.float32, (self.nL, self.state_floats)),
                ("emit", torch.float32, (self.nL, self.state_floats))])
            live, o, emit = views["live"], views["o"], views["emit"]
            self.out.append(dict(arena=arena, live=live, o=o, emit=emit,
                                 live_ptrs=hs.ptr_array([live[l] for l in range(self.nL)], dev),
                                 emit_ptrs=hs.ptr_array([emit[l] for l in range(self.nL)], dev)))
        self.shape = hs.make_shape(self.nL, self.nH, self.d, self.d, self.T, hs.HS_LINATTN_AUTO)
        self.tok_bytes = self.nH * self.d * 2        # one token of one problem, bf16
        self.tok_bytes_f = self.nH * self.d * 4
        torch.cuda.synchronize(dev)

    # -- the three phases of one resumed request (enqueued on stream handle st) --
    def phase_restore(self, s, r, st):
        """KV page restore of [0,c) for the full layers + state restore at c."""
        hs, R, I, O = self.hs, self.req[r], self.inp[(s, r)], self.out[r]
        hs.hs_restore_request(I["staging_ptrs"], self.cache_ptrs, self.nF, I["bt"], R["n_pages"],
                              self.page_bytes, self.NB, I["ck_ptrs"], O["live_ptrs"], self.nL,
                              self.state_floats, None, st)
        return 1

    def phase_prefill(self, s, r, st):
        """Tail prefill of [c,L) for all linear layers, emitting the checkpoint at L."""
        hs, R, I, O = self.hs, self.req[r], self.inp[(s, r)], self.out[r]
        B = self.nL
        hs.hs_linattn_prefill_from_state(self.shape, I["q"], I["k"], I["v"], I["a"], O["o"],
                                         O["live"], [R["c"]] * B, [TAIL] * B, self.S.ckpt,
                                         O["emit_ptrs"], None, st)
        return 1

    def phase_decode(self, s, r, st):
        """64 single-token steps of the recurrence after the prompt."""
        hs, R, I, O = self.hs, self.req[r], self.inp[(s, r)], self.out[r]
        B, L = self.nL, R["L"]
        for j in range(DECODE_STEPS):
            t0 = TAIL + j
            hs.hs_linattn_prefill_from_state(
                self.shape, I["q"].data_ptr() + t0 * self.tok_bytes,
                I["k"].data_ptr() + t0 * self.tok_bytes, I["v"].data_ptr() + t0 * self.tok_bytes,
                I["a"].data_ptr() + t0 * self.tok_bytes_f, O["o"].data_ptr() + t0 * self.tok_bytes_f,
                O["live"], [L + j] * B, [1] * B, 0, None, None, st)
        return DECODE_STEPS

    PHASES = ("restore", "prefill", "decode")

    def capture(self):
        """One CUDA graph per (seed, request, phase): the step replays them, so the
        576 single-token launches of a step are not bound by host launch latency."""
        torch = self.torch
        self.graphs = {}
        self.n_launch = {}
        side = torch.cuda.Stream(self.dev)
        for key in self.inp:
            for ph in self.PHASES:
                fn = getattr(self, "phase_" + ph)
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=side, capture_error_mode="relaxed"):
                    n = fn(key[0], key[1], torch.cuda.current_stream(self.dev).cuda_stream)
                self.graphs[key + (ph,)] = g
                self.n_launch[key + (ph,)] = n
            # the three phases of the request in one graph (one launch chain)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=side, capture_error_mode="relaxed"):
                for ph in self.PHASES:
                    getattr(self, "phase_" + ph)(key[0], key[1],
                                                 torch.cuda.current_stream(self.dev).cuda_stream)
            self.graphs[key] = g
        torch.cuda.synchronize(self.dev)

    def capture_steps(self, n, events):
        """One CUDA graph per timed step (seed = step index mod seeds) holding the
        phases of all nine requests, so a step is one graph launch.  With `events`,
        timing events are recorded between phases inside the graph, so the per-phase
        times are device times of the kernels themselves; each such event also ends
        the programmatic launch chain across its phase boundary (~5 us per boundary),
        so the headline step time is taken on the graphs without them.  Without events
        only one graph per seed is captured (steps replay them in rotation); with events
        every step has its own graph, whose events keep that step's times.  Returns False
        (nothing captured) where this PyTorch cannot record events inside a graph."""
        torch = self.torch
        if events:
            try:
                torch.cuda.Event(enable_timing=True, external=True)
            except TypeError:
                return False
        side = torch.cuda.Stream(self.dev)
        graphs = []
        for i in range(n if events else min(n, self.seeds)):
            s = i % self.seeds
            g = torch.cuda.CUDAGraph()
            marks, launches = [], 0
            with torch.cuda.graph(g, stream=side, capture_error_mode="relaxed"):
                cur = torch.cuda.current_stream(self.dev)
                if events:
                    prev = torch.cuda.Event(enable_timing=True, external=True)
                    prev.record(cur)
                for r in range(N_REQ):
                    for ph in self.PHASES:
                        nl = getattr(self, "phase_" + ph)(s, r, cur.cuda_stream)
                        if events:
                            e = torch.cuda.Event(enable_timing=True, external=True)
                            e.record(cur)
                            marks.append((ph, self.bytes_of(r, ph), nl, prev, e))
                            prev = e
                        launches += nl
            graphs.append((s, g, marks, launches))
        torch.cuda.synchronize(self.dev)
        if events:
            self.step_graphs = graphs
        else:
            self.plain_graphs = graphs
        return True

    def replay_step(self, i, events=True):
        """Step i from its graph: host alignment of the nine requests, then one
        graph launch.  Returns the number of kernel launches."""
        graphs = self.step_graphs if events else self.plain_graphs
        s, g, _, launches = graphs[i % len(graphs)]
        for R in self.req:
            L = R["L"]
            c, n_pages, tail = self.hs.hs_align_prefix(
                L, L, list(range(self.S.ckpt, L + 1, self.S.ckpt)), self.S.page)
            assert (c, n_pages, tail) == (R["c"], R["n_pages"], TAIL)
        g.replay()
        return launches

    def step_phase_times(self):
        """{phase: [bytes, ms, launches]} from the events inside every step graph
        (each holds the times of its latest replay)."""
        out = {}
        for _, _, marks, _ in self.step_graphs:
            for ph, nb, nl, e0, e1 in marks:
                t = out.setdefault(ph, [0, 0.0, 0])
                t[0] += nb
                t[1] += e0.elapsed_time(e1)
                t[2] += nl
        return out

    def bytes_of(self, r, ph):
        R = self.req[r]
        if ph == "restore":
            return kv_bytes(self.nF, R["n_pages"], self.page_bytes) + 2 * self.nL * self.state_floats * 4
        if ph == "prefill":
            return gla_bytes(self.nL, self.nH, self.d, TAIL, 1)
        return DECODE_STEPS * gla_bytes(self.nL, self.nH, self.d, 1, 0)

    def request(self, s, r, timer=None):
        """Replay one resumed request; returns the number of kernel launches."""
        hs, R = self.hs, self.req[r]
        L = R["L"]
        c, n_pages, tail = hs.hs_align_prefix(L, L, list(range(self.S.ckpt, L + 1, self.S.ckpt)),
                                              self.S.page)
        assert (c, n_pages, tail) == (R["c"], R["n_pages"], TAIL)
        if timer is None:
            self.graphs[(s, r)].replay()
            return sum(self.n_launch[(s, r, ph)] for ph in self.PHASES)
        n = 0
        for ph in self.PHASES:
            key = (s, r, ph)
            if timer:
                timer.begin(ph, self.bytes_of(r, ph), self.n_launch[key])
            self.graphs[key].replay()
            if timer:
                timer.end()
            n += self.n_launch[key]
        return n

    def step(self, s, timer=None):
        n = 0
        for r in range(N_REQ):
            n += self.request(s % self.seeds, r, timer)
        return n


class LaunchTimer:
    """CUDA events around individual launches inside the timed region."""

    def __init__(self, torch, stream):
        self.torch, self.stream = torch, stream
        self.rec = []
        self._cur = None

    def begin(self, name, nbytes, launches=1):
        e0 = self.torch.cuda.Event(enable_timing=True)
        e0.record(self.stream)
        self._cur = (name, nbytes, launches, e0)

    def end(self):
        e1 = self.torch.cuda.Event(enable_timing=True)
        e1.record(self.stream)
        self.rec.append(self._cur + (e1,))

    def summary(self):
        g = {}
        for name, nb, n, e0, e1 in self.rec:
            ms = e0.elapsed_time(e1)
            t = g.setdefault(name, [0, 0.0, 0])
            t[0] += nb
            t[1] += ms
            t[2] += n
        return g


# ---------------------------------------------------------------------------
# secondary measurements
# ---------------------------------------------------------------------------

def ttft_arms(wl, reps=10):
    """Resumed TTFT (align + KV restore + state restore + tail prefill) vs
    recomputation (prefill of [0,L) from the zero state emitting every
    checkpoint + KV write of all L tokens), per length, median of reps.
    Both arms replay CUDA graphs between CUDA events on one stream."""
    torch, hs = wl.torch, wl.hs
    dev = wl.dev
    Lmax = SWEEP_LENGTHS[-1]
    from hs_inputs import torch_gen_linear, torch_fill_bf16_normal
    q, k, v, a = torch_gen_linear(999, 0, wl.nL, Lmax, wl.nH, wl.d, dev)
    o = torch.empty((wl.nL, Lmax, wl.nH, wl.d), device=dev)
    state = torch.zeros((wl.nL, wl.state_floats), device=dev)
    n_ck = Lmax // wl.S.ckpt
    slots = torch.empty((wl.nL * n_ck, wl.state_floats), device=dev)
    kv_src = torch.empty((wl.nF, (Lmax // wl.S.page) * wl.page_bytes), dtype=torch.uint8, device=dev)
    torch_fill_bf16_normal(kv_src, 5)
    kv_src_ptrs = hs.ptr_array([kv_src[l] for l in range(wl.nF)], dev)
    bt_all = torch.randperm(wl.NB, device=dev)[:Lmax // wl.S.page].to(torch.int32)
    shape = hs.make_shape(wl.nL, wl.nH, wl.d, wl.d, Lmax, hs.HS_LINATTN_AUTO)
    side = torch.cuda.Stream(dev)
    stream = torch.cuda.current_stream(dev)
    out = {}
    for r, L in enumerate(SWEEP_LENGTHS):
        slot_ptrs = hs.ptr_array([slots[l * n_ck + m] for l in range(wl.nL)
                                  for m in range(L // wl.S.ckpt)], dev)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=side, capture_error_mode="relaxed"):
            st = torch.cuda.current_stream(dev).cuda_stream
            hs.hs_linattn_prefill_from_state(shape, q, k, v, a, o, state, [0] * wl.nL,
                                             [L] * wl.nL, wl.S.ckpt, slot_ptrs, None, st)
            hs.hs_restore_kv_pages(kv_src_ptrs, wl.cache_ptrs, wl.nF, bt_all, L // wl.S.page,
                                   wl.page_bytes, wl.NB, None, st)

        def recompute():
            state.zero_()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            g.replay()
            e1.record(stream)
            return e0, e1

        def resume():
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            c, n_pages, tail = hs.hs_align_prefix(L, L, list(range(wl.S.ckpt, L + 1, wl.S.ckpt)),
                                                  wl.S.page)
            wl.graphs[(0, r, "restore")].replay()
            wl.graphs[(0, r, "prefill")].replay()
            e1.record(stream)
            return e0, e1

        res = {}
        for name, fn in (("resume", resume), ("recompute", recompute)):
            for _ in range(3):
                fn()
            evs = [fn() for _ in range(reps)]
            torch.cuda.synchronize(dev)
            res[name] = statistics.median(e0.elapsed_time(e1) * 1e3 for e0, e1 in evs)
        out[str(L)] = {"resume_us": round(res["resume"], 2),
                       "recompute_us": round(res["recompute"], 2),
                       "ratio": round(res["recompute"] / res["resume"], 3)}
        del g
    del q, k, v, a, o, slots, kv_src
    return out


def kv_stress(dev, n_requests=64, staging_pool=4):
    """48 full layers x 256 pages x 64 KiB per request into a paged cache of
    min(180 GB, free - 8 GB); block tables uniform over the pool; staging
    pool rotating over 4 requests (3 GiB >> L2)."""
    import torch
    import paper_2609_15030_gb300 as hs
    from hs_inputs import gen_block_table
    S = KVSTRESS
    nL, n_pages, P = S.n_full, 4096 // S.page, S.page_bytes
    free, _ = torch.cuda.mem_get_info(dev)
    cache_bytes = min(180 * 10 ** 9, free - 8 * 2 ** 30 - staging_pool * nL * n_pages * P)
    NB = int(cache_bytes // (nL * P))
    cache = torch.empty((nL, NB * P), dtype=torch.uint8, device=dev)
    cache_ptrs = hs.ptr_array([cache[l] for l in range(nL)], dev)
    pool = torch.empty((staging_pool, nL, n_pages * P), dtype=torch.uint8, device=dev)
    pool.view(torch.int32).random_(generator=torch.Generator(device=dev).manual_seed(3))
    pool_ptrs = [hs.ptr_array([pool[i, l] for l in range(nL)], dev) for i in range(staging_pool)]
    bts = [torch.from_numpy(gen_block_table(40, i, n_pages, NB)).to(dev) for i in range(n_requests)]
    stream = torch.cuda.current_stream(dev)
    for i in range(3):
        hs.hs_restore_kv_pages(pool_ptrs[i % staging_pool], cache_ptrs, nL, bts[i], n_pages, P, NB,
                               None, stream.cuda_stream)
    evs = []
    torch.cuda.synchronize(dev)
    for i in range(n_requests):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        hs.hs_restore_kv_pages(pool_ptrs[i % staging_pool], cache_ptrs, nL, bts[i], n_pages, P, NB,
                               None, stream.cuda_stream)
        e1.record(stream)
        evs.append((e0, e1))
    torch.cuda.synchronize(dev)
    ts = [e0.elapsed_time(e1) * 1e-3 for e0, e1 in evs]
    nbytes = kv_bytes(nL, n_pages, P)
    del cache, pool
    torch.cuda.empty_cache()
    return {"cache_gb": round(NB * nL * P / 1e9, 1), "num_blocks": NB,
            "bytes_per_request": nbytes, "median_us": round(statistics.median(ts) * 1e6, 2),
            "gbs_median": round(nbytes / statistics.median(ts) / 1e9, 1),
            "gbs_aggregate": round(nbytes * len(ts) / sum(ts) / 1e9, 1)}


def kv_host(dev, save=False, n_requests=8, pool=2):
    """KV-stress requests (48 layers x 256 pages x 64 KiB) between the paged cache in HBM
    and a pinned host staging pool, with no separate copy: restored straight from host
    memory (the scatter kernel reads it over the host link, the paper's CPU cache tier,
    Section 5.5), or saved to it (the gather kernel writes it, the save path of
    Section 3.1)."""
    import torch
    import paper_2609_15030_gb300 as hs
    from hs_inputs import gen_block_table
    S = KVSTRESS
    nL, n_pages, P = S.n_full, 4096 // S.page, S.page_bytes
    NB = 4 * n_pages
    cache = torch.empty((nL, NB * P), dtype=torch.uint8, device=dev)
    cache.view(torch.int32).random_(generator=torch.Generator(device=dev).manual_seed(6))
    cache_ptrs = hs.ptr_array([cache[l] for l in range(nL)], dev)
    host = torch.empty((pool, nL, n_pages * P), dtype=torch.uint8).pin_memory()
    host.view(torch.int32).random_(generator=torch.Generator().manual_seed(5))
    ptrs = [hs.ptr_array([host[i, l] for l in range(nL)], dev) for i in range(pool)]
    bts = [torch.from_numpy(gen_block_table(41, i, n_pages, NB)).to(dev) for i in range(n_requests)]
    stream = torch.cuda.current_stream(dev)

    def move(i):
        if save:
            hs.hs_save_kv_pages(cache_ptrs, ptrs[i % pool], nL, bts[i], n_pages, P, NB, None,
                                stream.cuda_stream)
        else:
            hs.hs_restore_kv_pages(ptrs[i % pool], cache_ptrs, nL, bts[i], n_pages, P, NB, None,
                                   stream.cuda_stream)
    move(0)
    torch.cuda.synchronize(dev)
    evs = []
    for i in range(n_requests):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        move(i)
        e1.record(stream)
        evs.append((e0, e1))
    torch.cuda.synchronize(dev)
    ts = [e0.elapsed_time(e1) * 1e-3 for e0, e1 in evs]
    payload = nL * n_pages * P
    # context: the same bytes as one contiguous copy-engine transfer in the same direction
    dev_buf = cache[:, :n_pages * P]
    ce = []
    for _ in range(3):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        if save:
            host[0].copy_(dev_buf, non_blocking=True)
        else:
            dev_buf.copy_(host[0], non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        ce.append(e0.elapsed_time(e1) * 1e-3)
    del cache, host, dev_buf
    torch.cuda.empty_cache()
    out = {"bytes_per_request": payload, "median_us": round(statistics.median(ts) * 1e6, 1),
           "copy_engine_gbs": round(payload / statistics.median(ce) / 1e9, 1)}
    if save:
        out["host_write_gbs"] = round(payload / statistics.median(ts) / 1e9, 1)
        out["target"] = "pinned host memory (device-accessible), written by the gather kernel"
    else:
        out["host_read_gbs"] = round(payload / statistics.median(ts) / 1e9, 1)
        out["source"] = "pinned host memory (device-accessible), read by the scatter kernel"
    return out


def host_link(dev, nbytes=1 << 30, reps=5):
    """The host link's copy rate (NVLink-C2C between Grace memory and HBM) with the copy
    engines: one 1 GiB transfer between pinned host memory and the device in each direction,
    the same bytes as four concurrent 256 MiB transfers on four streams, and both directions
    at once (1 GiB each way on two streams); medians of `reps`, CUDA events."""
    import torch
    host = [torch.empty(nbytes, dtype=torch.uint8).pin_memory() for _ in range(2)]
    devb = [torch.empty(nbytes, dtype=torch.uint8, device=dev) for _ in range(2)]
    host[0].fill_(1)
    devb[0].fill_(2)
    main = torch.cuda.current_stream(dev)
    streams = [torch.cuda.Stream(dev) for _ in range(4)]

    def timed(fn):
        ts = []
        for _ in range(reps + 1):
            torch.cuda.synchronize(dev)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(main)
            fn()
            e1.record(main)
            torch.cuda.synchronize(dev)
            ts.append(e0.elapsed_time(e1) * 1e-3)
        return statistics.median(ts[1:])

    def split(dst, src):
        q = nbytes // 4
        for i, st in enumerate(streams):
            st.wait_stream(main)
            with torch.cuda.stream(st):
                dst[i * q:(i + 1) * q].copy_(src[i * q:(i + 1) * q], non_blocking=True)
        for st in streams:
            main.wait_stream(st)

    def both():
        for st in streams[:2]:
            st.wait_stream(main)
        with torch.cuda.stream(streams[0]):
            devb[1].copy_(host[0], non_blocking=True)
        with torch.cuda.stream(streams[1]):
            host[1].copy_(devb[0], non_blocking=True)
        for st in streams[:2]:
            main.wait_stream(st)
    h2d = nbytes / timed(lambda: devb[1].copy_(host[0], non_blocking=True)) / 1e9
    d2h = nbytes / timed(lambda: host[1].copy_(devb[0], non_blocking=True)) / 1e9
    h2d4 = nbytes / timed(lambda: split(devb[1], host[0])) / 1e9
    d2h4 = nbytes / timed(lambda: split(host[1], devb[0])) / 1e9
    bi = 2 * nbytes / timed(both) / 1e9
    del host, devb
    torch.cuda.empty_cache()
    return {"h2d_gbs": round(max(h2d, h2d4), 1), "d2h_gbs": round(max(d2h, d2h4), 1),
            "bidirectional_gbs": round(bi, 1),
            "h2d_one_copy_gbs": round(h2d, 1), "h2d_four_streams_gbs": round(h2d4, 1),
            "d2h_one_copy_gbs": round(d2h, 1), "d2h_four_streams_gbs": round(d2h4, 1),
            "method": "copy-engine transfers between 1 GiB pinned host buffers and HBM: one copy, "
                      "four concurrent 256 MiB copies on four streams (the better of the two is the "
                      "direction's peak), and 1 GiB each way at once; medians of 5, CUDA events"}


def state_copy(dev, reps=20, pool=8):
    """The standalone checkpoint writer (hs_checkpoint_states; hs_restore_state is the same
    copy the other way) on the long-context stack's live states: 4 requests x 18 linear
    layers, 32 heads x 128 x 128 float32 each (2 MiB per layer, 144 MiB per snapshot), into
    checkpoint slots rotating over `pool` snapshots (1.2 GB) from two rotating live sets, so
    neither side stays in L2."""
    import torch
    import paper_2609_15030_gb300 as hs
    from hs_inputs import LONG24
    S = LONG24
    n = S.batch * S.n_lin
    floats = S.n_heads * S.d * S.d
    live = torch.randn((2, n, floats), device=dev)
    slots = torch.empty((pool, n, floats), device=dev)
    live_ptrs = [hs.ptr_array([live[j, i] for i in range(n)], dev) for j in range(2)]
    slot_ptrs = [hs.ptr_array([slots[j, i] for i in range(n)], dev) for j in range(pool)]
    stream = torch.cuda.current_stream(dev)
    for i in range(3):
        hs.hs_checkpoint_states(live_ptrs[i % 2], slot_ptrs[i % pool], n, floats, None, stream.cuda_stream)
    torch.cuda.synchronize(dev)
    evs = []
    for i in range(reps):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        hs.hs_checkpoint_states(live_ptrs[i % 2], slot_ptrs[(i + 3) % pool], n, floats, None,
                                stream.cuda_stream)
        e1.record(stream)
        evs.append((e0, e1))
    torch.cuda.synchronize(dev)
    ok = torch.equal(slots[(reps - 1 + 3) % pool], live[(reps - 1) % 2])
    t = statistics.median(e0.elapsed_time(e1) for e0, e1 in evs) * 1e-3
    nb = 2 * n * floats * 4
    del live, slots
    return {"bytes_per_call": nb, "median_us": round(t * 1e6, 2), "gbs": round(nb / t / 1e9, 1),
            "states": f"{n} x {floats * 4 // 2 ** 20} MiB (4 requests x 18 layers x 32 heads)",
            "copy_checked": bool(ok)}


def kv_rank_slices(dev, n_requests=16):
    """One tensor-parallel rank's restore of FP8 KV pages (Table 1: TP=4, FP8 KV): 48
    layers x 256 pages of 16 tokens x 8 KV heads x 128 (one byte each, 32 KiB pages);
    the rank moves its 2 heads of every page row (8 KiB per page) from a device staging
    pool into a paged cache."""
    import torch
    import paper_2609_15030_gb300 as hs
    from hs_inputs import gen_block_table
    nL, n_pages, tokens, kvh, hd, TP = 48, 256, 16, 8, 128, 4
    rows, row_bytes = 2 * tokens, kvh * hd
    P, cb = rows * row_bytes, row_bytes // TP
    NB = 4 * n_pages
    cache = torch.zeros((nL, NB * P), dtype=torch.uint8, device=dev)
    stg = torch.empty((2, nL, n_pages * rows * cb), dtype=torch.uint8, device=dev)
    stg.view(torch.int32).random_(generator=torch.Generator(device=dev).manual_seed(8))
    cache_ptrs = hs.ptr_array([cache[l] for l in range(nL)], dev)
    sps = [hs.ptr_array([stg[i, l] for l in range(nL)], dev) for i in range(2)]
    bts = [torch.from_numpy(gen_block_table(44, i, n_pages, NB)).to(dev) for i in range(n_requests)]
    stream = torch.cuda.current_stream(dev)

    def move(i):
        hs.hs_restore_kv_page_slices(sps[i % 2], cache_ptrs, nL, bts[i], n_pages, P, rows, 0, cb,
                                     NB, None, stream.cuda_stream)
    move(0)
    torch.cuda.synchronize(dev)
    evs = []
    for i in range(n_requests):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        move(i)
        e1.record(stream)
        evs.append((e0, e1))
    torch.cuda.synchronize(dev)
    ts = [e0.elapsed_time(e1) * 1e-3 for e0, e1 in evs]
    moved = 2 * nL * n_pages * rows * cb            # read + write
    del cache, stg
    torch.cuda.empty_cache()
    t = statistics.median(ts)
    return {"bytes_per_request": moved, "median_us": round(t * 1e6, 1),
            "gbs": round(moved / t / 1e9, 1), "slice": f"{cb} of {row_bytes} bytes per row, "
            f"{rows} rows per {P}-byte page"}


def e2e_run(wl, steps, warmup):
    """Same step with every request's inputs in pinned host memory (KV staging
    pages, checkpoint state, q/k/v/log-gates) copied to the device inside the
    timed region, and its outputs (o, final state, emitted checkpoint) copied
    back.  Copies run on their own streams, so request r+1's inputs arrive and
    request r-1's outputs leave while request r computes; events order every
    reuse of a device buffer.  Host buffers exist for seed 0; every step uses
    them."""
    torch = wl.torch
    dev, stream = wl.dev, wl.stream
    host = []
    h2d = d2h = 0
    for r in range(N_REQ):
        I, O = wl.inp[(0, r)], wl.out[r]
        # one pinned buffer per request each way, mirroring the device arenas: every
        # request's inputs (q, k, v, log-gates, KV staging pages, checkpoint state) arrive
        # in one copy and its outputs (o, live state, emitted checkpoint) leave in one
        hb = {"arena": I["arena"].cpu().pin_memory()}
        ob = {"arena": torch.empty(O["arena"].shape, dtype=torch.uint8).pin_memory()}
        host.append((hb, ob))
        h2d += sum(t.numel() * t.element_size() for t in hb.values())
        d2h += sum(t.numel() * t.element_size() for t in ob.values())
    s_in = torch.cuda.Stream(dev)
    s_out = torch.cuda.Stream(dev)
    ev = lambda: torch.cuda.Event()
    consumed = [None] * N_REQ     # compute of request r done with its device inputs
    read = [None] * N_REQ         # device outputs of request r copied to the host

    def step():
        ready = []
        for r in range(N_REQ):
            hb, _ = host[r]
            I = wl.inp[(0, r)]
            if consumed[r] is not None:
                s_in.wait_event(consumed[r])
            with torch.cuda.stream(s_in):
                for k in hb:
                    I[k].copy_(hb[k], non_blocking=True)
            e = ev()
            e.record(s_in)
            ready.append(e)
        for r in range(N_REQ):
            _, ob = host[r]
            O = wl.out[r]
            stream.wait_event(ready[r])
            if read[r] is not None:
                stream.wait_event(read[r])
            wl.request(0, r, None)
            consumed[r] = ev()
            consumed[r].record(stream)
            s_out.wait_event(consumed[r])
            with torch.cuda.stream(s_out):
                for k in ob:
                    ob[k].copy_(O[k], non_blocking=True)
            read[r] = ev()
            read[r].record(s_out)

    for _ in range(warmup):
        step()
    torch.cuda.synchronize(dev)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    s_in.wait_stream(stream)        # no copy starts before the timed region
    for _ in range(steps):
        step()
    stream.wait_stream(s_out)       # ... and the last one ends inside it
    e1.record(stream)
    torch.cuda.synchronize(dev)
    t = e0.elapsed_time(e1) * 1e-3
    return {"value": round(TOKENS_PER_STEP * steps / t, 1), "unit": "tokens/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "ms_per_step": round(t * 1e3 / steps, 3)}


def _l2_flush(torch, dev, buf=[]):
    """Write 512 MiB (more than the 129 MB L2) so the next call reads its inputs from HBM."""
    if not buf:
        buf.append(torch.empty(512 * 2 ** 20, dtype=torch.uint8, device=dev))
    buf[0].fill_(1)


def sweep_run(dev, reps=10, scan=True, seq=True, lengths=None):
    """Single-layer kernel sweep: one linear layer, 16 heads, d = 128, checkpoints every 512,
    batch 1.  For each L in 512..4608: the resumed tail prefill (c = C floor((L-1)/C), 512
    tokens from the state at c, emitting the checkpoint at L; the hit L-37 aligns to the same
    c) and the recomputation of [0,L) from the zero state emitting every checkpoint; with
    `scan`, both also through the segment-parallel prefill (`seq=False`: only there).  Each
    call is timed alone between CUDA events with L2 flushed before it; median of `reps`."""
    import torch
    import paper_2609_15030_gb300 as hs
    from hs_inputs import SWEEP, torch_gen_linear
    S = SWEEP
    nH, d, C, Lmax = S.n_heads, S.d, S.ckpt, max(SWEEP_LENGTHS)
    q, k, v, a = torch_gen_linear(11, 0, 1, Lmax, nH, d, dev)
    o = torch.empty((1, Lmax, nH, d), device=dev)
    state = torch.empty((1, nH, d, d), device=dev)
    ck = torch.randn((1, nH, d, d), device=dev,
                     generator=torch.Generator(device=dev).manual_seed(12)) * 0.5
    slots = torch.empty((Lmax // C, nH, d, d), device=dev)
    shape = hs.make_shape(1, nH, d, d, Lmax, hs.HS_LINATTN_AUTO)
    stream = torch.cuda.current_stream(dev)
    tb, tbf = nH * d * 2, nH * d * 4
    peak = _peaks()[0]
    tensor = _tensor_pipe()
    ws_bytes = hs.hs_linattn_scan_workspace_bytes(shape, [0], [Lmax])
    ws = torch.empty((ws_bytes // 4,), device=dev)
    rows = []
    for L in (lengths or SWEEP_LENGTHS):
        c, _, tail = hs.hs_align_prefix(L, L, list(range(C, L + 1, C)), S.page)
        c37, _, _ = hs.hs_align_prefix(L, L - 37, list(range(C, L + 1, C)), S.page)
        nck_t = hs.hs_linattn_num_checkpoints([c], [tail], C)
        tail_ptrs = hs.ptr_array([slots[i] for i in range(nck_t)], dev) if nck_t else None
        rec_ptrs = hs.ptr_array([slots[i] for i in range(L // C)], dev)

        def resume():
            hs.hs_linattn_prefill_from_state(
                shape, q.data_ptr() + c * tb, k.data_ptr() + c * tb, v.data_ptr() + c * tb,
                a.data_ptr() + c * tbf, o.data_ptr() + c * tbf, state, [c], [tail], C, tail_ptrs,
                None, stream.cuda_stream)

        def recompute():
            hs.hs_linattn_prefill_from_state(shape, q, k, v, a, o, state, [0], [L], C, rec_ptrs,
                                             None, stream.cuda_stream)

        # the same two calls through the segment-parallel prefill (its own workspace)
        def resume_scan():
            hs.hs_linattn_prefill_scan(
                shape, q.data_ptr() + c * tb, k.data_ptr() + c * tb, v.data_ptr() + c * tb,
                a.data_ptr() + c * tbf, o.data_ptr() + c * tbf, state, [c], [tail], C, tail_ptrs,
                ws, ws_bytes, None, stream.cuda_stream)

        def recompute_scan():
            hs.hs_linattn_prefill_scan(shape, q, k, v, a, o, state, [0], [L], C, rec_ptrs, ws,
                                       ws_bytes, None, stream.cuda_stream)
        res = {}
        arms = [("tail", resume, lambda: state.copy_(ck)),
                ("recompute", recompute, lambda: state.zero_())] if seq else []
        if scan:
            arms += [("tail_scan", resume_scan, lambda: state.copy_(ck)),
                     ("recompute_scan", recompute_scan, lambda: state.zero_())]
        for nm, fn, init in arms:
            ts = []
            for i in range(reps + 2):
                init()
                _l2_flush(torch, dev)
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                fn()
                e1.record(stream)
                torch.cuda.synchronize(dev)
                if i >= 2:
                    ts.append(e0.elapsed_time(e1) * 1e-3)
            res[nm] = statistics.median(ts)
        b_tail = gla_bytes(1, nH, d, tail, nck_t)
        b_rec = gla_bytes(1, nH, d, L, L // C)
        tp_t = tensor.get(f"gla_chunked_tc_kernel@sweep_tail_{L}")
        tp_r = tensor.get(f"gla_chunked_tc_kernel@sweep_recompute_{L}")
        rows.append({"L": L, "c": c, "c_hit_L-37": c37, "tail": tail})
        if seq:
            rows[-1].update({
                "tail_us": round(res["tail"] * 1e6, 2),
                "tail_tokens_per_s": round(tail / res["tail"], 1),
                "tail_hbm_frac": round(b_tail / res["tail"] / 1e9 / peak, 4),
                "tail_tensor_pipe": tp_t["active"] if tp_t else None,
                "recompute_us": round(res["recompute"] * 1e6, 2),
                "recompute_tokens_per_s": round(L / res["recompute"], 1),
                "recompute_hbm_frac": round(b_rec / res["recompute"] / 1e9 / peak, 4),
                "recompute_tensor_pipe": tp_r["active"] if tp_r else None})
        if scan:
            rows[-1].update({
                "tail_scan_us": round(res["tail_scan"] * 1e6, 2),
                "tail_scan_hbm_frac": round(b_tail / res["tail_scan"] / 1e9 / peak, 4),
                "recompute_scan_us": round(res["recompute_scan"] * 1e6, 2),
                "recompute_scan_hbm_frac": round(b_rec / res["recompute_scan"] / 1e9 / peak, 4)})
    del q, k, v, a, o, slots, ws
    return {"workload": "single-layer sweep: 16 heads, d = 128, C = 512, batch 1, tails of 512 "
                        "(complete hit and hit L-37 align to the same c)",
            "scan": "*_scan_*: the same calls through hs_linattn_prefill_scan (every 64-token "
                    "segment its own tensor-core problem from the zero state, an elementwise "
                    "state scan, every segment again from its start state; algorithmic bytes "
                    "as the sequential call's)",
            "timing": f"each call alone, L2 flushed before it, median of {reps}",
            "tensor_pipe": "sm__pipe_tensor_cycles_active, % of active cycles, from the committed "
                           "ncu capture of `bench.py --case sweep` (null when the kernel changed since)",
            "rows": rows}


def packed_run(dev, reps=10):
    """Packed varlen tails: the tails of one engine batch back to back without padding, each
    problem with its own resume point, in one launch (hs_linattn_prefill_packed).  The batch
    is the hybrid workload's nine requests x nine linear layers (81 problems, 16 heads, d = 128,
    C = 256) with seeded tail lengths in [65, 512] and resume points on the 256-token grid in
    [0, 4352]; the checkpoints each tail crosses are emitted.  Timed alone between CUDA events
    with L2 flushed before each call, median of `reps`; against the same problems in the padded
    layout (rows of 512 tokens)."""
    import numpy as np
    import torch
    import paper_2609_15030_gb300 as hs
    from hs_inputs import torch_gen_linear
    nP, nH, d, C, Tmax = HYBRID12.n_lin * N_REQ, HYBRID12.n_heads, HYBRID12.d, HYBRID12.ckpt, 512
    rng = np.random.default_rng(21)
    n_tok = [int(x) for x in rng.integers(65, Tmax + 1, nP)]
    pos0 = [int(x) * C for x in rng.integers(0, 18, nP)]
    cu = np.concatenate([[0], np.cumsum(n_tok)]).astype(np.int64)
    rows = int(cu[-1])
    q, k, v, a = torch_gen_linear(13, 0, 1, rows, nH, d, dev)
    o = torch.empty((rows, nH, d), device=dev)
    qp, kp, vp, ap = (torch_gen_linear(13, 0, nP, Tmax, nH, d, dev))
    op = torch.empty((nP, Tmax, nH, d), device=dev)
    st0 = torch.randn((nP, nH, d, d), device=dev,
                      generator=torch.Generator(device=dev).manual_seed(14)) * 0.5
    state = torch.empty_like(st0)
    nck = hs.hs_linattn_num_checkpoints(pos0, n_tok, C)
    slots = torch.empty((max(nck, 1), nH, d, d), device=dev)
    sp = hs.ptr_array([slots[i] for i in range(nck)], dev) if nck else None
    stream = torch.cuda.current_stream(dev)
    shape_p = hs.make_shape(nP, nH, d, d, 0)
    shape_d = hs.make_shape(nP, nH, d, d, Tmax)

    def packed():
        hs.hs_linattn_prefill_packed(shape_p, q, k, v, a, o, state, pos0, n_tok, cu.tolist(), C, sp,
                                     None, stream.cuda_stream)

    def padded():
        hs.hs_linattn_prefill_from_state(shape_d, qp, kp, vp, ap, op, state, pos0, n_tok, C, sp, None,
                                         stream.cuda_stream)
    res = {}
    for nm, fn in (("packed", packed), ("padded", padded)):
        ts = []
        for i in range(reps + 2):
            state.copy_(st0)
            _l2_flush(torch, dev)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            torch.cuda.synchronize(dev)
            if i >= 2:
                ts.append(e0.elapsed_time(e1) * 1e3)
        res[nm] = statistics.median(ts)
    nb = sum(gla_bytes(1, nH, d, n, (p0 + n) // C - p0 // C) for p0, n in zip(pos0, n_tok))
    peak = _peaks()[0]
    return {"problems": nP, "tokens": rows, "tail_min": min(n_tok), "tail_max": max(n_tok),
            "checkpoints": nck, "packed_us": round(res["packed"], 2),
            "packed_tokens_per_s": round(rows / (res["packed"] * 1e-6), 1),
            "packed_hbm_frac": round(nb / (res["packed"] * 1e-6) / 1e9 / peak, 4),
            "padded_us": round(res["padded"], 2),
            "timing": "each call alone, L2 flushed before it, median of %d" % reps}


def tiny_run(dev, reps=20):
    """Tiny hybrid stack (1 linear layer: 2 heads, d = 64, C = 64; 1 full layer: 2 KV heads,
    head_dim 64, page 16), seed 0, N = 256, complete hit -> c = 192: the resumed request
    (alignment, restore of 12 KV pages and the state at 192, the 64-token tail) against the
    recomputation of [0,256) (prefill from the zero state emitting every checkpoint and the KV
    write of 16 pages).  Latency of each arm, host-launched, median of `reps`; the resumed
    outputs and final state must equal the recomputation's bit for bit."""
    import torch
    import paper_2609_15030_gb300 as hs
    from hs_inputs import TINY, gen_linear, gen_kv_pages, gen_block_table
    S = TINY
    N, C, P, nH, d = 256, S.ckpt, S.page, S.n_heads, S.d
    c, n_pages, tail = hs.hs_align_prefix(N, N, list(range(C, N + 1, C)), P)
    x = gen_linear(0, 0, 1, N, nH, d, d, gates=S.gates)
    dv = lambda arr: torch.from_numpy(arr.view(np.int16) if arr.dtype == np.uint16 else arr).to(dev)
    q, k, v, a = dv(x.q), dv(x.k), dv(x.v), dv(x.a)
    pb = S.page_bytes
    NB = 64
    staging = torch.from_numpy(gen_kv_pages(0, 0, N // P, pb).reshape(-1)).to(dev)
    cache = torch.zeros(NB * pb, dtype=torch.uint8, device=dev)
    bt = torch.from_numpy(gen_block_table(0, 0, N // P, NB)).to(dev)
    sp, cp = hs.ptr_array([staging], dev), hs.ptr_array([cache], dev)
    o_rec = torch.empty((1, N, nH, d), device=dev)
    o_res = torch.empty((1, N, nH, d), device=dev)
    st_rec = torch.zeros((1, nH, d, d), device=dev)
    live = torch.zeros((1, nH, d, d), device=dev)
    slots = torch.empty((N // C, nH, d, d), device=dev)
    slot_ptrs = hs.ptr_array([slots[i] for i in range(N // C)], dev)
    last_ptr = hs.ptr_array([slots[N // C - 1]], dev)
    src = hs.ptr_array([slots[c // C - 1]], dev)
    dst = hs.ptr_array([live], dev)
    shape = hs.make_shape(1, nH, d, d, N, hs.HS_LINATTN_AUTO)
    tb, tbf = nH * d * 2, nH * d * 4
    stream = torch.cuda.current_stream(dev)

    def recompute():
        st_rec.zero_()
        hs.hs_linattn_prefill_from_state(shape, q, k, v, a, o_rec, st_rec, [0], [N], C, slot_ptrs,
                                         None, stream.cuda_stream)
        hs.hs_restore_kv_pages(sp, cp, 1, bt, N // P, pb, NB, None, stream.cuda_stream)

    def resume():
        cc, npg, tl = hs.hs_align_prefix(N, N, list(range(C, N + 1, C)), P)
        hs.hs_restore_request(sp, cp, 1, bt, npg, pb, NB, src, dst, 1, nH * d * d, None,
                              stream.cuda_stream)
        hs.hs_linattn_prefill_from_state(
            shape, q.data_ptr() + cc * tb, k.data_ptr() + cc * tb, v.data_ptr() + cc * tb,
            a.data_ptr() + cc * tbf, o_res.data_ptr() + cc * tbf, live, [cc], [tl], C, last_ptr,
            None, stream.cuda_stream)
    out = {}
    for nm, fn in (("recompute", recompute), ("resume", resume)):
        ts = []
        for i in range(reps + 3):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            torch.cuda.synchronize(dev)
            if i >= 3:
                ts.append(e0.elapsed_time(e1) * 1e3)
        out[nm + "_us"] = round(statistics.median(ts), 2)
    same = (torch.equal(o_res[:, c:].view(torch.int32), o_rec[:, c:].view(torch.int32))
            and torch.equal(live.view(torch.int32), st_rec.view(torch.int32)))
    out.update({"N": N, "c": c, "pages": n_pages, "tail": tail, "resume_equals_recompute": bool(same),
                "timing": f"host-launched calls between CUDA events, median of {reps}"})
    return out


# ---------------------------------------------------------------------------
# the oracle on the host cores (CPU baseline / reference arm)
# ---------------------------------------------------------------------------

class OracleSample:
    """One resumed request of the workload run by the float64 oracle: alignment,
    page scatter, state copy, then the 256-token tail and 64 decode tokens of
    all nine linear layers (token by token; decode is the same recurrence)."""

    def __init__(self, r, seed=0):
        import oracle
        from hs_inputs import gen_linear, gen_kv_pages, gen_block_table
        self.oracle = oracle
        S = HYBRID12
        self.S = S
        self.L = SWEEP_LENGTHS[r]
        self.T = TAIL + DECODE_STEPS
        c, n_pages, tail = oracle.align_prefix(self.L, self.L, list(range(S.ckpt, self.L + 1, S.ckpt)),
                                               S.page)
        self.c, self.n_pages = c, n_pages
        self.inp = gen_linear(seed, r, S.n_lin, self.T, S.n_heads, S.d, S.d, gates=S.gates)
        self.staging = [gen_kv_pages(seed, l, max(n_pages, 1), S.page_bytes).reshape(-1)
                        for l in range(S.n_full)]
        self.NB = 2 * max(n_pages, 1)
        self.cache = [np.zeros(self.NB * S.page_bytes, np.uint8) for _ in range(S.n_full)]
        self.bt = gen_block_table(seed, r, max(n_pages, 1), self.NB)
        self.ck = [np.random.default_rng(r).standard_normal(S.n_heads * S.d * S.d).astype(np.float32)
                   for _ in range(S.n_lin)]
        self.live = [np.zeros_like(x) for x in self.ck]

    def run(self, threads):
        o, S = self.oracle, self.S
        c, n_pages, tail = o.align_prefix(self.L, self.L, list(range(S.ckpt, self.L + 1, S.ckpt)),
                                          S.page)
        o.scatter_pages(self.staging, self.cache, self.bt, n_pages, S.page_bytes)
        o.copy_slots(self.ck, self.live, S.n_heads * S.d * S.d)
        S0 = np.stack(self.live).reshape(S.n_lin, S.n_heads, S.d, S.d)
        n = self.T
        o.gla(self.inp.q, self.inp.k, self.inp.v, self.inp.a, [c] * S.n_lin, [n] * S.n_lin,
              S0=S0, C_=S.ckpt, threads=threads)
        return TAIL + DECODE_STEPS


def _cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_baseline():
    cores = _cores()
    samples = [OracleSample(r) for r in range(N_REQ)]
    t0 = time.perf_counter()
    toks = sum(s.run(cores) for s in samples)
    t = time.perf_counter() - t0
    # the same oracle on one thread, for the first request only
    t1 = time.perf_counter()
    toks1 = samples[0].run(1)
    t1 = time.perf_counter() - t1
    return {"value": round(toks / t, 2), "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"one step (the 9 requests of seed 0): align + page scatter + state copy + "
                      "256-token tail and 64 decode tokens of all 9 linear layers x 16 heads, "
                      f"float64 token by token; {t:.1f} s wall on {cores} threads",
            "one_thread": {"value": round(toks1 / t1, 2), "unit": "tokens/s", "cores": 1,
                           "sample": f"request 0 of the same step (L = 512) on one thread, {t1:.1f} s wall"}}


def cpu_baseline_configs():
    """The float64 oracle as it stands on the host cores, on the other configurations:
    the tiny stack's resumed request (in full), the sweep's nine tails and nine
    recomputations (in full), one KV-stress request's page scatter (in full), and one
    long-context request at L = 65,536: its page scatter and state copy in full, its
    linear-attention work on one (layer, head) and scaled to all 18 x 32 heads of one request
    (labelled extrapolated)."""
    import oracle
    from hs_inputs import SWEEP, TINY, LONG24, LONG_LENGTHS, gen_linear, gen_kv_pages, gen_block_table
    cores = _cores()
    out = {"cores": cores, "kind": "oracle"}
    # tiny stack, one resumed request
    S = TINY
    N, C = 256, S.ckpt
    x = gen_linear(0, 0, 1, N, S.n_heads, S.d, S.d, gates=S.gates)
    stg = [gen_kv_pages(0, 0, N // S.page, S.page_bytes).reshape(-1)]
    cache = [np.zeros(64 * S.page_bytes, np.uint8)]
    bt = gen_block_table(0, 0, N // S.page, 64)
    ck = [np.random.default_rng(1).standard_normal(S.n_heads * S.d * S.d).astype(np.float32)]
    live = [np.zeros_like(ck[0])]
    reps = 20
    t0 = time.perf_counter()
    for _ in range(reps):
        c, npg, tail = oracle.align_prefix(N, N, list(range(C, N + 1, C)), S.page)
        oracle.scatter_pages(stg, cache, bt, npg, S.page_bytes)
        oracle.copy_slots(ck, live, S.n_heads * S.d * S.d)
        oracle.gla(x.q[:, c:], x.k[:, c:], x.v[:, c:], x.a[:, c:], [c], [tail],
                   S0=live[0].reshape(1, S.n_heads, S.d, S.d), C_=C, threads=1)
    t = (time.perf_counter() - t0) / reps
    out["tiny"] = {"resume_us": round(t * 1e6, 1), "cores": 1,
                   "sample": f"align + 12-page scatter + state copy + 64-token tail (2 heads, d = 64), "
                             f"one thread, mean of {reps}"}
    # sweep: the nine tails and recomputations, 16 heads in parallel
    S = SWEEP
    Lmax = max(SWEEP_LENGTHS)
    x = gen_linear(11, 0, 1, Lmax, S.n_heads, S.d, S.d)
    S0 = np.random.default_rng(12).standard_normal((1, S.n_heads, S.d, S.d)).astype(np.float32)
    t_tail = t_rec = 0.0
    for L in SWEEP_LENGTHS:
        c = S.ckpt * ((L - 1) // S.ckpt)
        t0 = time.perf_counter()
        oracle.gla(x.q[:, c:L], x.k[:, c:L], x.v[:, c:L], x.a[:, c:L], [c], [L - c], S0=S0,
                   C_=S.ckpt, threads=cores)
        t_tail += time.perf_counter() - t0
        t0 = time.perf_counter()
        oracle.gla(x.q[:, :L], x.k[:, :L], x.v[:, :L], x.a[:, :L], [0], [L], C_=S.ckpt, threads=cores)
        t_rec += time.perf_counter() - t0
    n_tail = sum(L - S.ckpt * ((L - 1) // S.ckpt) for L in SWEEP_LENGTHS)
    out["sweep"] = {"tail_tokens_per_s": round(n_tail / t_tail, 1),
                    "recompute_tokens_per_s": round(sum(SWEEP_LENGTHS) / t_rec, 1), "cores": cores,
                    "sample": f"all nine 512-token tails and recomputations of [0,L), 16 heads on "
                              f"{cores} threads, {t_tail + t_rec:.1f} s wall"}
    # KV stress: one request's scatter (48 layers x 256 pages x 64 KiB)
    P = KVSTRESS.page_bytes
    nL, npg = KVSTRESS.n_full, 4096 // KVSTRESS.page
    stg = [np.ones(npg * P, np.uint8) for _ in range(nL)]
    cache = [np.full(2 * npg * P, 0, np.uint8) for _ in range(nL)]   # touched before timing
    bt = gen_block_table(40, 0, npg, 2 * npg)
    oracle.scatter_pages(stg, cache, bt, npg, P)
    t0 = time.perf_counter()
    oracle.scatter_pages(stg, cache, bt, npg, P)
    t = time.perf_counter() - t0
    out["kv_stress"] = {"gbs": round(kv_bytes(nL, npg, P) / t / 1e9, 2), "cores": 1,
                        "sample": "one request: 48 layers x 256 pages x 64 KiB (read + write bytes), "
                                  f"one thread, {t:.2f} s"}
    del stg, cache
    # long context: one request at L = 65,536 (complete hit, c = 65,024)
    S = LONG24
    L = max(LONG_LENGTHS)
    c = S.ckpt * ((L - 1) // S.ckpt)
    npg = c // S.page
    stg = [np.ones(npg * S.page_bytes, np.uint8) for _ in range(S.n_full)]
    cache = [np.full(npg * S.page_bytes, 0, np.uint8) for _ in range(S.n_full)]
    bt = np.arange(npg, dtype=np.int32)[::-1].copy()
    ckl = [np.ones(S.n_heads * S.d * S.d, np.float32) for _ in range(S.n_lin)]
    livel = [np.zeros_like(z) for z in ckl]
    t0 = time.perf_counter()
    oracle.scatter_pages(stg, cache, bt, npg, S.page_bytes)
    oracle.copy_slots(ckl, livel, S.n_heads * S.d * S.d)
    t_copy = time.perf_counter() - t0
    del stg, cache
    xl = gen_linear(13, 0, 1, 4096, 1, S.d, S.d)
    t0 = time.perf_counter()
    oracle.gla(xl.q[:, :L - c], xl.k[:, :L - c], xl.v[:, :L - c], xl.a[:, :L - c], [c], [L - c],
               S0=None, C_=S.ckpt, threads=1)
    t_head_tail = time.perf_counter() - t0
    t0 = time.perf_counter()
    oracle.gla(xl.q, xl.k, xl.v, xl.a, [0], [4096], C_=S.ckpt, threads=1)
    t_head_4k = time.perf_counter() - t0
    heads = S.n_lin * S.n_heads
    out["long"] = {
        "L": L, "c": c, "extrapolated": True, "cores": 1,
        "ttft_resume_s": round(t_copy + heads * t_head_tail, 2),
        "ttft_recompute_s": round(heads * t_head_4k * L / 4096, 1),
        "sample": f"one request of the batch of 4: page scatter of 6 layers x {npg} pages x 128 KiB and "
                  f"18 state copies in full ({t_copy:.2f} s); the 512-token tail of one (layer, head) "
                  f"({t_head_tail:.2f} s) x 576 heads; the recomputation from one head's first 4,096 "
                  f"tokens ({t_head_4k:.2f} s) x 576 heads x L/4096; one thread"}
    return out


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    cores = _cores()
    samples = [OracleSample(r) for r in range(N_REQ)]
    for i in range(args.warmup):
        samples[i % N_REQ].run(cores)
    toks = 0
    t0 = time.perf_counter()
    for i in range(args.steps):
        toks += samples[i % N_REQ].run(cores)
    t = time.perf_counter() - t0
    val = toks / t
    sample = ("each step: one of the 9 requests (rotating L) of the hybrid workload run by the float64 "
              "oracle: align + page scatter + state copy + 256-token tail and 64 decode tokens of 9 "
              "linear layers x 16 heads")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": round(val, 2), "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(t * 1e3 / max(args.steps, 1), 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD},
        "cpu_baseline": {"value": round(val, 2), "unit": "tokens/s", "cores": cores,
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": round(val, 2), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0}}))
    return 0


# ---------------------------------------------------------------------------
# small standalone cases for profiler captures
# ---------------------------------------------------------------------------

def run_case(name: str, iters: int = 5):
    """decode: 64 single-token calls over 9 problems x 16 heads (d = 128);
    prefill: one 256-token tail over 9 problems x 16 heads from pos0 = 4096 with
    checkpoints every 256; kv: 12 layers x 256 pages x 64 KiB scattered into a
    2,048-block cache; ckpt: the standalone checkpoint writer on the long-context stack's
    live states (72 x 2 MiB).  Each repeated `iters` times on the current stream."""
    import torch
    import paper_2609_15030_gb300 as hs
    from hs_inputs import torch_gen_linear, gen_block_table
    from paper_2609_15030_gb300 import build
    build.build()
    dev = torch.device("cuda:0")
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    if name in ("decode", "prefill"):
        B, nH, d = HYBRID12.n_lin, HYBRID12.n_heads, HYBRID12.d
        T = DECODE_STEPS if name == "decode" else TAIL
        q, k, v, a = torch_gen_linear(2, 0, B, T, nH, d, dev)
        o = torch.empty((B, T, nH, d), device=dev)
        st = torch.randn((B, nH, d, d), device=dev) * 0.5
        slots = torch.empty((B, nH, d, d), device=dev)
        ptrs = hs.ptr_array([slots[i] for i in range(B)], dev)
        shape = hs.make_shape(B, nH, d, d, T)
        tb, tbf = nH * d * 2, nH * d * 4
        for it in range(iters):
            ev[0].record()
            if name == "decode":
                for j in range(T):
                    hs.hs_linattn_prefill_from_state(
                        shape, q.data_ptr() + j * tb, k.data_ptr() + j * tb, v.data_ptr() + j * tb,
                        a.data_ptr() + j * tbf, o.data_ptr() + j * tbf, st, [4096 + j] * B, [1] * B,
                        0, None, None)
            else:
                hs.hs_linattn_prefill_from_state(shape, q, k, v, a, o, st, [4096] * B, [T] * B,
                                                 HYBRID12.ckpt, ptrs, None)
            ev[1].record()
            torch.cuda.synchronize()
            per = ev[0].elapsed_time(ev[1]) * 1e3 / (T if name == "decode" else 1)
            print(f"{name} iter {it}: {per:.2f} us per call (host-launched)", flush=True)
    elif name == "kv":
        nL, n_pages, P, NB = 12, 256, KVSTRESS.page_bytes, 2048
        st = torch.empty((nL, n_pages * P), dtype=torch.uint8, device=dev)
        st.view(torch.int32).random_(generator=torch.Generator(device=dev).manual_seed(1))
        cache = torch.empty((nL, NB * P), dtype=torch.uint8, device=dev)
        sp = hs.ptr_array([st[l] for l in range(nL)], dev)
        cp = hs.ptr_array([cache[l] for l in range(nL)], dev)
        bt = torch.from_numpy(gen_block_table(9, 0, n_pages, NB)).to(dev)
        for it in range(iters):
            ev[0].record()
            hs.hs_restore_kv_pages(sp, cp, nL, bt, n_pages, P, NB, None)
            ev[1].record()
            torch.cuda.synchronize()
            t = ev[0].elapsed_time(ev[1]) * 1e-3
            print(f"kv iter {it}: {t * 1e6:.1f} us, {kv_bytes(nL, n_pages, P) / t / 1e9:.0f} GB/s",
                  flush=True)
    elif name == "ckpt":
        for it in range(iters):
            r = state_copy(dev, reps=4)
            print(f"ckpt iter {it}: {r['median_us']:.1f} us, {r['gbs']:.0f} GB/s", flush=True)
    elif name == "long":
        run_long(dev)
        return 0
    elif name == "sweep":
        # single-layer sweep: each L's 512-token tail from c, then its recomputation of [0,L),
        # one call each with L2 flushed before it (18 prefill launches, L = 512 .. 4608)
        r = sweep_run(dev, reps=1, scan=False)
        for row in r["rows"]:
            print(json.dumps({k: row[k] for k in ("L", "tail_us", "recompute_us")}), flush=True)
    elif name == "sweep_scan":
        # the same sweep's tail at L = 512 and recomputation at L = 4608 through the
        # segment-parallel prefill only (3 calls each: both tensor-core passes and the scan)
        r = sweep_run(dev, reps=1, seq=False, lengths=[512, 4608])
        for row in r["rows"]:
            print(json.dumps({k: row[k] for k in ("L", "tail_scan_us", "recompute_scan_us")}),
                  flush=True)
    else:
        raise SystemExit(f"unknown case {name}")
    return 0


def run_long(dev, reps=3, quiet=False):
    """Long-context hybrid stack: 24 layers (18 linear: 32 heads, d = 128, C = 512;
    6 full: 8 KV heads, head_dim 128, page 32), batch 4, L in {16k, 32k, 64k},
    complete hit (c = L - 512) and partial hit L - 37 (same c).  Resumed TTFT =
    align + KV restore of [0,c) for 6 layers + state restore of 18 layers + the
    512-token tail prefill of every linear layer; recomputation = prefill of
    [0,L) from the zero state emitting every checkpoint + the KV write of L
    tokens.  One q/k/v/gate set per request is shared by the 18 linear layers
    (18 distinct sets at L = 64k would need ~190 GB), so each layer is one call.
    Medians of `reps` timed runs after one warm-up; returns one row per case."""
    import torch
    import paper_2609_15030_gb300 as hs
    from hs_inputs import LONG24, LONG_LENGTHS, torch_gen_linear, torch_fill_bf16_normal
    S = LONG24
    B, nH, d, nL, nF, P, C = S.batch, S.n_heads, S.d, S.n_lin, S.n_full, S.page, S.ckpt
    Lmax = max(LONG_LENGTHS)
    q, k, v, a = torch_gen_linear(7, 0, B, Lmax, nH, d, dev)
    o = torch.empty((B, Lmax, nH, d), device=dev)
    states = torch.zeros((nL, B, nH, d, d), device=dev)
    nck = Lmax // C
    slots = torch.empty((B * nck, nH, d, d), device=dev)
    pb = S.page_bytes
    n_pages_max = Lmax // P
    NB = B * n_pages_max + 64
    cache = torch.empty((nF, NB * pb), dtype=torch.uint8, device=dev)
    staging = torch.empty((B, nF, n_pages_max * pb), dtype=torch.uint8, device=dev)
    torch_fill_bf16_normal(staging, 3)
    cache_ptrs = hs.ptr_array([cache[l] for l in range(nF)], dev)
    stg_ptrs = [hs.ptr_array([staging[b, l] for l in range(nF)], dev) for b in range(B)]
    perm = torch.randperm(NB, device=dev).to(torch.int32)
    bts = [perm[b * n_pages_max:(b + 1) * n_pages_max].contiguous() for b in range(B)]
    ck_src = torch.randn((nL, B, nH, d, d), device=dev) * 0.5
    src_ptrs = hs.ptr_array([ck_src[l] for l in range(nL)], dev)
    dst_ptrs = hs.ptr_array([states[l] for l in range(nL)], dev)
    ev = lambda: torch.cuda.Event(enable_timing=True)
    rows = []
    if not quiet:
        print(json.dumps({"case": "long", "workload": "long-24L (18 linear 32h d128 C512 + 6 full 8kv hd128 P32), batch 4"}))
    for Lc in LONG_LENGTHS:
        # complete hit; cached prefix L-37 of an L-token prompt; an (L-37)-token prompt
        # fully cached (ragged tail inside the last chunk)
        for L, hit in ((Lc, Lc), (Lc, Lc - 37), (Lc - 37, Lc - 37)):
            c, n_pages, tail = hs.hs_align_prefix(L, hit, list(range(C, L + 1, C)), P)
            # resumed
            shape_t = hs.make_shape(B, nH, d, d, Lmax)
            slot_ptrs = hs.ptr_array([slots[b] for b in range(B)], dev) if L % C == 0 else None
            tok = c * nH * d
            def resume(mid=None):
                for b in range(B):      # the batch's states ride with the first request's pages
                    hs.hs_restore_request(stg_ptrs[b], cache_ptrs, nF, bts[b], n_pages, pb, NB,
                                          src_ptrs, dst_ptrs, nL if b == 0 else 0, B * nH * d * d)
                if mid is not None:
                    mid.record()
                for l in range(nL):
                    hs.hs_linattn_prefill_from_state(
                        shape_t, q.data_ptr() + 2 * tok, k.data_ptr() + 2 * tok, v.data_ptr() + 2 * tok,
                        a.data_ptr() + 4 * tok, o.data_ptr() + 4 * tok, states[l], [c] * B, [tail] * B, C,
                        slot_ptrs)
            per = L // C
            ckp = hs.ptr_array([slots[b * nck + m] for b in range(B) for m in range(per)], dev)
            if hs.hs_linattn_num_checkpoints([c] * B, [tail] * B, C) != (B if L % C == 0 else 0):
                raise SystemExit("unexpected checkpoint count")
            def recompute(mid=None):
                for l in range(nL):
                    states[l].zero_()
                    hs.hs_linattn_prefill_from_state(shape_t, q, k, v, a, o, states[l], [0] * B, [L] * B, C, ckp)
                if mid is not None:
                    mid.record()
                for b in range(B):
                    hs.hs_restore_kv_pages(stg_ptrs[b], cache_ptrs, nF, bts[b], L // P, pb, NB)
            res, part = {}, {}
            for nm, fn in (("resume", resume), ("recompute", recompute)):
                fn()
                torch.cuda.synchronize(dev)
                ts, t1s = [], []
                for _ in range(reps):
                    e0, em, e1 = ev(), ev(), ev()
                    e0.record()
                    fn(em)       # an event between the arm's two parts (restore | prefills,
                    e1.record()  # prefills | KV write)
                    torch.cuda.synchronize(dev)
                    ts.append(e0.elapsed_time(e1))
                    t1s.append(e0.elapsed_time(em))
                res[nm] = statistics.median(ts)
                part[nm] = statistics.median(t1s)
            # algorithmic bytes of each arm: resume = KV restore of [0,c) + state restore +
            # the tail prefill of every linear layer; recompute = the prefill of [0,L) of every
            # linear layer emitting every checkpoint + the KV write of L tokens
            b_restore = B * kv_bytes(nF, n_pages, pb) + 2 * nL * B * nH * d * d * 4
            b_tail = nL * gla_bytes(B, nH, d, tail, 1 if L % C == 0 else 0)
            b_res = b_restore + b_tail
            b_k2 = nL * gla_bytes(B, nH, d, L, L // C)
            b_rec = b_k2 + B * kv_bytes(nF, L // P, pb)
            peak = _peaks()[0]
            frac = lambda nb, ms: round(nb / (ms * 1e-3) / 1e9 / peak, 3)
            row = {"L": L, "hit": hit, "c": c, "tail": tail, "ttft_resume_ms": round(res["resume"], 3),
                   "ttft_recompute_ms": round(res["recompute"], 3),
                   "ratio": round(res["recompute"] / res["resume"], 1),
                   "resume_hbm_frac": round(b_res / (res["resume"] * 1e-3) / 1e9 / peak, 3),
                   "recompute_hbm_frac": round(b_rec / (res["recompute"] * 1e-3) / 1e9 / peak, 3),
                   # the arms' parts (events between them): K1 + K2a, the restore of 6
                   # attention layers' pages and 18 states for the batch; K2, the 512-token
                   # tails of the 18 linear layers; K2 over [0,L) emitting every checkpoint
                   "restore_ms": round(part["resume"], 3),
                   "restore_hbm_frac": frac(b_restore, part["resume"]),
                   "k2_tail_ms": round(res["resume"] - part["resume"], 3),
                   "k2_tail_hbm_frac": frac(b_tail, res["resume"] - part["resume"]),
                   "k2_recompute_ms": round(part["recompute"], 3),
                   "k2_recompute_hbm_frac": frac(b_k2, part["recompute"])}
            rows.append(row)
            if not quiet:
                print(json.dumps(row), flush=True)
    del q, k, v, a, o, states, slots, cache, staging, ck_src
    return rows


# ---------------------------------------------------------------------------
# multi-rank helpers (host logic, tested on CPU with gloo)
# ---------------------------------------------------------------------------

def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", str(rank)))
    return ws, rank, local


def max_over_ranks(x: float, world_size: int, device=None) -> float:
    if world_size <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world_size: int):
    if world_size > 1:
        import torch.distributed as dist
        dist.barrier()


def aggregate_value(tokens_per_rank_step: int, steps: int, world_size: int, t_max: float) -> float:
    """Whole-job throughput: every rank runs the full step on its own requests."""
    return tokens_per_rank_step * steps * world_size / t_max


# ---------------------------------------------------------------------------

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-extras", action="store_true",
                    help="skip TTFT arms, KV stress, e2e and CPU baseline")
    ap.add_argument("--case", choices=["decode", "prefill", "kv", "ckpt", "long", "sweep",
                                       "sweep_scan"],
                    help="run one small standalone case for a profiler capture")
    ap.add_argument("--source-hashes", action="store_true",
                    help="print each profiled kernel's source hash (the key of profiles/*.txt rows)")
    args = ap.parse_args()
    if args.source_hashes:
        for k in sorted(KERNEL_SRC):
            print(k, source_hash(k))
        return 0
    if args.case:
        return run_case(args.case)
    if args.impl == "reference":
        return run_reference(args)
    args.warmup = max(args.warmup, 3)

    import torch
    ws, rank, local = dist_env()
    if ws > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    from paper_2609_15030_gb300 import build
    build.build()

    wl = Hybrid12(dev)
    wl.capture()
    # one graph per timed step (all phases of the nine requests): the headline run on
    # graphs without events, then the same steps again on graphs with timing events
    # between phases for the per-kernel times; per-phase graphs with events around each
    # replay where events inside graphs are unavailable
    whole = wl.capture_steps(args.steps, events=True)
    if whole:
        wl.capture_steps(args.steps, events=False)
    for i in range(args.warmup):
        if whole:
            wl.replay_step(i, events=False)
            wl.replay_step(i, events=True)
        else:
            wl.step(i)
    torch.cuda.synchronize(dev)

    def timed(events, timer=None):
        barrier(ws)
        torch.cuda.synchronize(dev)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(wl.stream)
        n = 0
        for i in range(args.steps):
            n += wl.replay_step(i, events) if whole else wl.step(i, timer)
        e1.record(wl.stream)
        torch.cuda.synchronize(dev)
        barrier(ws)
        return e0.elapsed_time(e1) * 1e-3, n

    clocks = Clocks(local)
    clocks.start()
    timer = LaunchTimer(torch, wl.stream)
    if whole:
        with _nvtx("hybrid12 timed steps"):
            t_local, launches = timed(False)
        with _nvtx("hybrid12 timed steps with phase events"):
            t_phases, _ = timed(True)
    else:
        t_local, launches = timed(False, timer)
        t_phases = t_local
    clk = clocks.stop()
    t = max_over_ranks(t_local, ws, dev)
    value = aggregate_value(TOKENS_PER_STEP, args.steps, ws, t)

    peak, peak_kind = _peaks()
    groups = wl.step_phase_times() if whole else timer.summary()
    traffic = _traffic()

    tensor = _tensor_pipe()

    def roofline(phase):
        nb, ms, n = groups[phase]
        ach = nb / (ms * 1e-3) / 1e9
        kern = KERNEL_OF[phase]
        r = {"bound": "hbm", "kernel": kern, "phase": phase, "achieved": round(ach, 1),
             "peak": peak, "unit": "GB/s", "frac": round(ach / peak, 4), "peak_kind": peak_kind,
             "traffic": traffic.get(kern), "bytes_per_launch": int(nb / n),
             "avg_launch_us": round(ms * 1e3 / n, 3), "launches": n,
             "share_of_step": round(ms * 1e-3 / t_phases, 3)}
        if kern in tensor:
            r["tensor_pipe_frac"] = tensor[kern]
        r["source_hash"] = source_hash(kern)
        return r

    dominant = max(groups, key=lambda k: groups[k][1])
    out = {
        "metric": METRIC, "value": round(value, 1), "unit": "tokens/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(t * 1e3 / args.steps, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": DTYPE,
        "data": "synthetic",
        "config": {"workload": WORKLOAD, "tokens_per_step": TOKENS_PER_STEP,
                   "l2": "inputs larger than L2: four seeds x nine requests rotate "
                         "(~2.7 GB of inputs), each step touches ~0.7 GB"},
        "roofline": roofline(dominant),
        "roofline_by_phase": {k: roofline(k) for k in groups},
        "gpu_launches": launches,
        "launch": ("one CUDA graph per step (value); per-kernel times from a second timed run "
                   f"of the same steps with phase events inside the graphs "
                   f"({t_phases * 1e3 / args.steps:.3f} ms per step with the events)") if whole
                  else "one CUDA graph per request phase, events around each replay",
        "clocks": clk,
    }
    if rank == 0 and not args.no_extras:
        with _nvtx("e2e through host buffers"):
            wl_e2e = e2e_run(wl, args.steps, args.warmup)
        out["e2e"] = {k: wl_e2e[k] for k in ("value", "unit", "h2d_bytes_per_step", "d2h_bytes_per_step")}
        out["e2e"]["ms_per_step"] = wl_e2e["ms_per_step"]
        with _nvtx("ttft resume vs recompute"):
            out["ttft_us"] = ttft_arms(wl)
        with _nvtx("tiny stack latency"):
            out["tiny_latency"] = tiny_run(dev)
        with _nvtx("packed varlen tails"):
            out["packed_tails"] = packed_run(dev)
        with _nvtx("single-layer sweep"):
            out["sweep"] = sweep_run(dev)
        red = [1.0 - r["resume_us"] / r["recompute_us"] for r in out["ttft_us"].values()]
        out["paper_context"] = {
            "ttft_reduction": "46-64 %", "total_time_reduction": "1.9-7.0 %",
            "hardware": "4x RTX PRO 6000 Blackwell Server Edition, TP=4, vLLM + LMCache reload "
                        "from the CPU cache over PCIe, GLM-5.3-Flash NVFP4, C = 1,792 "
                        "(abstract; Section 5.5, Table 7, Fig. 3)",
            "kind": "end-to-end serving latency of whole requests: context, not the target",
            "ours_component_ttft_reduction": f"{100 * min(red):.0f}-{100 * max(red):.0f} %",
            "ours_kind": "restore + tail prefill vs recompute of the linear-attention layers and "
                         "the KV write, L = 512..4608 (no projections, MLP or attention compute)"}
        del wl
        torch.cuda.empty_cache()
        with _nvtx("kv stress"):
            kv = kv_stress(dev)
        kv["frac"] = round(kv["gbs_aggregate"] / peak, 4)
        kv["traffic"] = _traffic().get("kv_scatter_kernel@kvstress")
        out["kv_restore"] = kv
        with _nvtx("kv host staging"):
            link = host_link(dev)
            out["host_link"] = link
            out["kv_restore_from_host"] = kv_host(dev)
            out["kv_save_to_host"] = kv_host(dev, save=True)
            out["kv_restore_from_host"]["frac_of_link_h2d"] = round(
                out["kv_restore_from_host"]["host_read_gbs"] / link["h2d_gbs"], 3)
            out["kv_save_to_host"]["frac_of_link_d2h"] = round(
                out["kv_save_to_host"]["host_write_gbs"] / link["d2h_gbs"], 3)
        with _nvtx("kv rank slices"):
            sl = kv_rank_slices(dev)
        sl["frac"] = round(sl["gbs"] / peak, 4)
        out["kv_restore_rank_slice_fp8"] = sl
        with _nvtx("checkpoint writer"):
            sc = state_copy(dev)
        sc["frac"] = round(sc["gbs"] / peak, 4)
        sc["traffic"] = _traffic().get("slot_copy_kernel@long24")
        out["checkpoint_writer"] = sc
        torch.cuda.empty_cache()
        with _nvtx("long context"):
            out["ttft_long_ms"] = run_long(dev, quiet=True)
        with _nvtx("oracle baseline"):
            out["cpu_baseline"] = cpu_baseline()
            out["cpu_baseline_configs"] = cpu_baseline_configs()
    if rank == 0:
        print(json.dumps(out))
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
