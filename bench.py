#!/usr/bin/env python
"""Benchmark of one Early-Bird decoding step (window attention, LM head with
fused softmax statistics, EB decision) on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config llada8b]
                    [--state select|inblock] [--impl ours|reference]

Prints ONE JSON line.  The default workload is the LLaDA-8B-shaped step
(batch 1, hidden 4096, vocab 126464, 32x128 MHA, cached prefix 512, window
32 with 24 masked rows, no active block so the LBS router runs).  `value` is
window positions scored per second; `ms_per_step` the device time of one
step (CUDA events around a CUDA-graph replay of ebd_step; before every timed
step L2 is flushed by a 256 MB write followed by a 256 MB read, which leaves
no dirty lines to be written back inside the timed region; decode state
restored outside the timed interval).  Multi-GPU runs are independent replicas (one process per
GPU, no collective on the data path): value = rows of all ranks / max time.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "µs/step & positions/s at LLaDA-8B shape; % of HBM/tensor roofline"
UNIT = "positions/s"
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0


# ----------------------------------------------------------------------------- helpers
def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return (float(d["hbm_gbs"]), float(d["bf16_tflops"]),
                float(d.get("bf16_tflops_sustained", d["bf16_tflops"])), "measured")
    except Exception:
        return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS, 1700.0, "fallback"


def shape_for(name):
    import synth
    if name in synth.SHAPES:
        return synth.SHAPES[name]
    if name.startswith("sweep_"):
        for s in synth.sweep_points():
            if s.name == name:
                return s
    raise SystemExit(f"unknown config {name}")


def full_sequence(sh):
    """The full-sequence setting: windows of more than 64 rows (every
    position of the response), decided by the grid-wide kernels, without
    the window attention."""
    import synth
    return int(np.max(synth.window_sizes(sh))) > 64


def workload_text(sh, state):
    import synth
    w = synth.window_sizes(sh)
    if full_sequence(sh):
        return (f"{sh.name} full-sequence step: batch {sh.batch}, hidden {sh.d_model}, vocab {sh.vocab}, "
                f"every position of a {int(w.max())}-token response is a row ({int(w.sum())} rows), "
                f"LBS over all masked positions ({'no active block: LBS runs' if state == 'select' else 'active block'}); "
                f"no window attention")
    return (f"{sh.name} decoding step: batch {sh.batch}, hidden {sh.d_model}, vocab {sh.vocab}, "
            f"{sh.n_heads_q}q/{sh.n_heads_kv}kv heads x {sh.head_dim}, cached prefix {sh.prefix}, "
            f"window rows {int(w.sum())} ({'no active block: LBS runs' if state == 'select' else 'active block'})")


def strip_comments(src: str) -> str:
    """C/C++ source without its comments and blank lines (string literals in
    these files hold no comment markers)."""
    import re
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    src = re.sub(r"//[^\n]*", "", src)
    return "\n".join(l.rstrip() for l in src.splitlines() if l.strip())


def lm_kernel_hash(read=None):
    """Hash of the LM head's sources (k_lmhead.cu, ptx.cuh, lm_params.h)
    without comments: the kernel a profile was captured on."""
    h = hashlib.sha256()
    for f in ("k_lmhead.cu", "ptx.cuh", "lm_params.h"):
        if read is None:
            with open(os.path.join(ROOT, "paper_2609_16450_gb300", "csrc", f)) as fh:
                text = fh.read()
        else:
            text = read(f)
        h.update(strip_comments(text).encode())
    return h.hexdigest()[:16]


def profiled_traffic(workload):
    """DRAM bytes per LM-head launch from the committed ncu summary
    (profiles/lm_head_<workload>.md: lines "kernel_sha: ..." and
    "dram_bytes_per_launch: ..."), or None if the kernel changed since the
    counters were taken."""
    p = os.path.join(ROOT, "profiles", f"lm_head_{workload}.md")
    try:
        kv = {}
        with open(p) as f:
            for line in f:
                if ":" in line and not line.startswith(("|", " ", "#")):
                    k, v = line.split(":", 1)
                    kv[k.strip()] = v.strip()
        if kv.get("kernel_sha") != lm_kernel_hash():
            return None
        return float(kv["dram_bytes_per_launch"])
    except Exception:
        return None


class ClockSampler:
    """Samples SM clock, power and clock-event reasons through NVML while the
    timed region runs (read-only queries)."""

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown", 0x1: "gpu_idle",
               0x2: "applications_clocks_setting", 0x10: "sync_boost"}

    def __init__(self, uuid: str, period_s: float = 0.002):
        self.samples = []
        self.max_mhz = None
        self.err = None
        self.period = period_s
        self._stop = threading.Event()
        self._t = None
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() != 0:
                raise RuntimeError("nvmlInit failed")
            h = ctypes.c_void_p()
            if nv.nvmlDeviceGetHandleByUUID(("GPU-" + uuid).encode(), ctypes.byref(h)) != 0:
                raise RuntimeError("nvmlDeviceGetHandleByUUID failed")
            mx = ctypes.c_uint()
            nv.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx))
            self.max_mhz = int(mx.value)
            self.nv, self.h = nv, h
        except Exception as e:  # no NVML: no clock record
            self.nv = None
            self.err = str(e)

    def _run(self):
        nv, h = self.nv, self.h
        mhz, reasons, mw = ctypes.c_uint(), ctypes.c_ulonglong(), ctypes.c_uint()
        while not self._stop.is_set():
            nv.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(mhz))
            r = nv.nvmlDeviceGetCurrentClocksEventReasons(h, ctypes.byref(reasons))
            if r != 0:
                nv.nvmlDeviceGetCurrentClocksThrottleReasons(h, ctypes.byref(reasons))
            nv.nvmlDeviceGetPowerUsage(h, ctypes.byref(mw))
            self.samples.append((int(mhz.value), int(reasons.value), mw.value / 1000.0))
            time.sleep(self.period)

    def start(self):
        if self.nv is not None:
            self._t = threading.Thread(target=self._run, daemon=True)
            self._t.start()

    def stop(self):
        if self._t is not None:
            self._stop.set()
            self._t.join()

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": [],
                    "samples": 0, "note": self.err or "no samples"}
        mhz = [s[0] for s in self.samples]
        bits = 0
        for s in self.samples:
            bits |= s[1]
        reasons = sorted(v for k, v in self.REASONS.items() if bits & k and k != 0x1)
        return {"sm_mhz": statistics.median(mhz), "sm_max_mhz": self.max_mhz,
                "reasons": reasons, "samples": len(mhz),
                "power_w_max": round(max(s[2] for s in self.samples), 1)}


# ----------------------------------------------------------------------------- work model
def suffix_len(sh):
    """Cached positions after the window in dual-cache mode: the rest of a
    gen_len response whose first positions form the largest window."""
    import synth
    return int(sh.gen_len - int(np.max(synth.window_sizes(sh))))


def lm_grid(num_sms, n_units):
    """CTAs of the library's unpaired LM-head launch, hence partial states
    per row (the same rule as the library's lm_grid): the fewest CTAs that
    take at most one 64-row vocabulary unit more each than an even split over
    every SM, if that keeps 90 % of the SMs."""
    num_sms = max(1, num_sms)
    if n_units <= num_sms:
        return max(1, n_units)
    per = -(-n_units // num_sms) + 1
    g = -(-n_units // per)
    return g if 10 * g >= 9 * num_sms else num_sms


PAIR_MIN_ROWS = 65  # LM-head launches of at least this many rows run in CTA pairs


def lm_pair_grid(num_sms, n_units):
    """CTAs of the library's paired (cta_group::2) LM-head launch: one pair
    per two SMs, at most one per 4-unit chunk of the vocabulary."""
    return 2 * max(1, min(num_sms // 2, -(-n_units // 4)))


def partials_per_row(num_sms, n_units, max_rows):
    """LM-head partial states per row that a handle with max_rows rows per
    step keeps (the library's rule): room for the paired launch when a step
    may take it."""
    g = lm_grid(num_sms, n_units)
    return max(g, lm_pair_grid(num_sms, n_units)) if max_rows >= PAIR_MIN_ROWS else g


def step_work(sh, rows, masked, grid_lm, lbs_runs, suffix=0, append=False):
    """Algorithmic bytes and flops of one step (each input read once); suffix:
    cached keys after each window (dual cache); append: committed rows'
    K/V written to the cache (counted for every row, an upper bound)."""
    d, V, Hq, Hkv, D = sh.d_model, sh.vocab, sh.n_heads_q, sh.n_heads_kv, sh.head_dim
    import synth
    w = synth.window_sizes(sh)
    keys = int(sum(sh.prefix + int(x) + suffix for x in w))
    attn = not full_sequence(sh)
    lm_bytes = V * d * 2 + rows * d * 2 + rows * grid_lm * 20
    lm_flops = 2 * rows * d * V
    attn_bytes = keys * Hkv * D * 2 * 2 + rows * Hq * D * 2 + rows * Hq * D * 4
    attn_flops = 4 * sum(int(x) * (sh.prefix + int(x) + suffix) for x in w) * Hq * D
    if append:
        attn_bytes += rows * Hkv * D * 2 * 2 * 2
    if not attn:
        attn_bytes = attn_flops = 0
    dec_bytes = rows * grid_lm * 20 + rows * 40
    if lbs_runs:
        dec_bytes += 2 * (613761 - 262208) + masked * 64 * 4
    return dict(lm_bytes=lm_bytes, lm_flops=lm_flops, attn_bytes=attn_bytes,
                attn_flops=attn_flops, step_bytes=lm_bytes + attn_bytes + dec_bytes,
                step_flops=lm_flops + attn_flops)


# ----------------------------------------------------------------------------- our arm
class L2Flush:
    """Evicts L2 between timed steps: writes a 256 MB buffer (twice the
    129 MB L2), then reads a second 256 MB buffer so that the dirty lines of
    the write are written back to HBM before the timed region starts (a real
    step is preceded by the backbone's weight reads, not by dirty data)."""

    def __init__(self, torch):
        n = 256 * 1024 * 1024 // 4
        self.w = torch.empty(n, dtype=torch.float32, device="cuda")
        self.r = torch.zeros(n, dtype=torch.float32, device="cuda")
        self.mode = os.environ.get("EBD_BENCH_FLUSH", "write+read")

    def __call__(self, i):
        if "write" in self.mode:
            self.w.fill_(float(i))
        if "read" in self.mode:
            self.r.sum()


def max_over_ranks(x: float, world: int, device: str) -> float:
    """The maximum of x over the ranks of the process group (x itself for one
    rank): the step time of N independent replicas is the slowest one's."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replicas_value(rows_per_rank: int, world: int, t_step_s: float) -> float:
    """Whole-job throughput of N replicas: positions of all ranks per second
    of the slowest rank's step."""
    return rows_per_rank * world / t_step_s


def run_ours(args, rank, world, local_rank):
    import torch
    torch.cuda.set_device(local_rank)
    from paper_2609_16450_gb300 import build as B
    if rank == 0 or world == 1:
        B.build()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    B.build()
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    import synth

    sh = shape_for(args.config)
    inp = synth.make_step_inputs(sh)
    if args.state == "inblock":
        synth.preset_in_block(inp, 20)
    sfx = None
    if args.cache == "dual":  # the rest of a gen_len response after the window
        inp, sfx = synth.with_suffix_cache(inp, suffix_len(sh))
    w = rt.upload_weights(inp)
    h = rt.Handle(rt.config_for(sh, max_prefix=inp.k_cache.shape[1]), w.w_emb)
    if args.w_layout == "packed":
        w = rt.pack_weights(h, w)  # one-time tiling of W_lm (model load)
    ds = rt.DeviceStep(inp, w, attention=not full_sequence(sh))
    stream = torch.cuda.Stream()
    sid = stream.cuda_stream
    args_c = ds.args()
    sfx_d = None
    if sfx is not None:
        sfx_d = torch.from_numpy(sfx).cuda()
        args_c.suffix = sfx_d.data_ptr()
    args_c.kv_append = 1 if args.append else 0
    flush = L2Flush(torch)
    torch.cuda.synchronize()

    def make_step(mode):
        """ebd_step in profile mode `mode` (0: production, no interior events;
        2: events around the LM head, the rest as in production), replayed
        from a CUDA graph unless --no-graph."""
        E.check(E.ebd_profile_enable(h.h, mode), h.h)
        if args.no_graph:
            def run():
                E.check(E.ebd_profile_enable(h.h, mode), h.h)
                E.check(E.ebd_step(h.h, args_c, sid), h.h)
            return run
        with torch.cuda.stream(stream):
            E.check(E.ebd_step(h.h, args_c, sid), h.h)  # warm once outside capture
        torch.cuda.synchronize()
        ds.restore_state()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            E.check(E.ebd_step(h.h, args_c, stream.cuda_stream), h.h)
        torch.cuda.synchronize()
        return g.replay

    one_step = make_step(0)       # the timed steps: production order and overlap
    lm_step = make_step(2)        # the live LM-head timing pass
    E.check(E.ebd_profile_enable(h.h, 0), h.h)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            ds.restore_state()
            one_step()
    torch.cuda.synchronize()
    if h.sync_status(sid) != 0:
        raise SystemExit(f"device status after warm-up: {E.ebd_last_error(h.h)}")

    sampler = ClockSampler(str(torch.cuda.get_device_properties(local_rank).uuid))
    ev0 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ev1 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    sampler.start()
    t_wall = time.perf_counter()
    with torch.cuda.stream(stream):
        for i in range(args.steps):
            ds.restore_state()
            flush(i)
            ev0[i].record(stream)
            one_step()
            ev1[i].record(stream)
    torch.cuda.synchronize()
    t_wall = time.perf_counter() - t_wall
    if world > 1:
        dist.barrier()
    sampler.stop()
    status = h.sync_status(sid)
    if status != 0:
        raise SystemExit(f"device status {status}: {E.ebd_last_error(h.h)}")
    step_ms = [a.elapsed_time(b) for a, b in zip(ev0, ev1)]
    mean_ms = max_over_ranks(float(np.mean(step_ms)), world, "cuda")
    # the LM head timed live with CUDA events on its stream (same inputs,
    # same flush); the events around it keep the decision from starting in
    # the LM head's tail, so these steps are not the timed ones
    kern = []
    with torch.cuda.stream(stream):
        for i in range(max(20, min(args.steps, 100))):
            ds.restore_state()
            flush(i)
            lm_step()
            stream.synchronize()
            s, ms = E.ebd_profile_read(h.h)
            if s != 0:
                raise SystemExit(f"ebd_profile_read: {E.ebd_last_error(h.h)}")
            kern.append(ms)
    kern = np.array(kern)
    k_lm, k_tail = float(np.mean(kern[:, 1])), float(np.mean(kern[:, 2]))
    # per-kernel breakdown outside the timed region: mode 1 runs the three
    # kernels one after the other, each bracketed by events
    E.check(E.ebd_profile_enable(h.h, 1), h.h)
    brk = []
    with torch.cuda.stream(stream):
        for i in range(max(5, min(args.steps, 30))):
            ds.restore_state()
            flush(i)
            E.check(E.ebd_step(h.h, args_c, sid), h.h)
            stream.synchronize()
            s, ms = E.ebd_profile_read(h.h)
            if s != 0:
                raise SystemExit(f"ebd_profile_read: {E.ebd_last_error(h.h)}")
            brk.append(ms)
    brk = np.array(brk)
    k_attn, k_dec = float(np.mean(brk[:, 0])), float(np.mean(brk[:, 2]))

    # end to end through ebd_step_host: pinned host inputs in, results out
    e2e = None
    if not args.skip_e2e:
        e2e = run_e2e(args, h, ds, inp, sh, stream, world, sfx)
    out = dict(sh=sh, inp=inp, rows=inp.rows, masked=int(inp.mask.sum()), mean_ms=mean_ms,
               step_ms=step_ms, k_attn=k_attn, k_lm=k_lm, k_dec=k_dec, k_tail=k_tail,
               grid_lm=None,
               clocks=sampler.summary(), e2e=e2e, t_wall=t_wall,
               lbs_runs=args.state == "select")
    out["launches_per_step"] = 2 + (inp.rows + 511) // 512 + (1 if args.append else 0)
    if full_sequence(sh):  # LM head groups, merge, memsets and the decision chain
        out["launches_per_step"] = (inp.rows + 511) // 512 + 1 + (2 + 12 + 8 if args.state == "select" else 2 + 12)
    out["suffix"] = None if sfx is None else sfx
    out["fetch"] = ds.fetch()
    h_sms = torch.cuda.get_device_properties(local_rank).multi_processor_count
    out["grid_lm"] = partials_per_row(h_sms, (sh.vocab + 63) // 64, h.cfg.max_rows)
    out["num_sms"] = h_sms
    h.close()
    return out


def run_e2e(args, h, ds, inp, sh, stream, world, sfx=None):
    """Same step through ebd_step_host: every step copies its inputs from
    pinned host memory and its results back inside the timed interval."""
    import torch
    from paper_2609_16450_gb300 import _ebd as E
    R, Hq, Hkv, D = inp.rows, sh.n_heads_q, sh.n_heads_kv, sh.head_dim
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()  # noqa: E731
    host_in = dict(cu_rows=pin(inp.cu_rows.astype(np.int32)),
                   prefix_len=pin(inp.prefix_len.astype(np.int32)),
                   row_pos=pin(inp.row_pos.astype(np.int32)),
                   hidden=pin(inp.hidden.view(np.int16)), q=pin(inp.q.view(np.int16)),
                   k_win=pin(inp.k_win.view(np.int16)), v_win=pin(inp.v_win.view(np.int16)))
    if ds.attn_out is None:  # no window attention: its inputs are not copied
        for k in ("q", "k_win", "v_win"):
            del host_in[k]
    st0 = dict(tokens=inp.tokens.astype(np.int32), mask=inp.mask.astype(np.uint8),
               in_block=inp.in_block.astype(np.uint8), blk_meta=inp.blk_meta.astype(np.int32))
    host_state = {k: pin(v) for k, v in st0.items()}
    host_out = dict(attn_out=torch.empty((R, Hq, D), dtype=torch.float32).pin_memory()) \
        if ds.attn_out is not None else {}
    for k in ("conf", "entropy", "ent_norm", "gap", "lbs_logit", "lps_prob"):
        host_out[k] = torch.empty(R, dtype=torch.float32).pin_memory()
    host_out["argmax"] = torch.empty(R, dtype=torch.int32).pin_memory()
    host_out["accepted"] = torch.empty(R, dtype=torch.uint8).pin_memory()
    a = E.ebd_step_args()
    a.batch, a.rows = sh.batch, R
    for k, t in {**host_in, **host_state, **host_out}.items():
        setattr(a, k, t.data_ptr())
    a.k_cache, a.v_cache, a.w_lm = ds.k_cache.data_ptr(), ds.v_cache.data_ptr(), \
        ds.weights.w_lm.data_ptr()
    a.w_lm_layout = ds.weights.layout
    if sfx is not None:
        host_in["suffix"] = pin(sfx)
        a.suffix = host_in["suffix"].data_ptr()
    a.kv_append = 1 if args.append else 0
    h2d = sum(t.numel() * t.element_size() for t in host_in.values()) + \
        sum(t.numel() * t.element_size() for t in host_state.values())
    d2h = sum(t.numel() * t.element_size() for t in host_state.values()) + \
        sum(t.numel() * t.element_size() for t in host_out.values())
    sid = stream.cuda_stream
    E.check(E.ebd_profile_enable(h.h, False), h.h)

    def reset():
        for k, v in st0.items():
            host_state[k].numpy()[...] = v

    for _ in range(max(1, args.warmup)):
        reset()
        E.check(E.ebd_step_host(h.h, a, sid), h.h)
        stream.synchronize()
    flush = L2Flush(torch)
    times = []
    with torch.cuda.stream(stream):
        for i in range(args.steps):
            reset()
            flush(i)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            E.check(E.ebd_step_host(h.h, a, sid), h.h)
            e1.record(stream)
            stream.synchronize()
            times.append(e0.elapsed_time(e1))
    if h.sync_status(sid) != 0:
        raise SystemExit("device status after e2e")
    mean_ms = max_over_ranks(float(np.mean(times)), world, "cuda")
    return dict(mean_ms=mean_ms, h2d=int(h2d), d2h=int(d2h))


# ----------------------------------------------------------------------------- oracle arm
def oracle_step_sample(sh, inp, budget_s, suffix=None):
    """Times the CPU oracle on the step's inputs: full steps until budget_s
    has passed (at least one).  Returns (positions/s, steps, seconds, the
    oracle's result of the step)."""
    from oracle import ebd_oracle as o
    import synth
    W = o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))
    prm = o.DecisionParams(tau=sh.tau, tau_psi=sh.tau_psi, l_min=sh.l_min, l_b=sh.l_b,
                           g_max=sh.g_max, eos_id=sh.eos_id, lps_enabled=bool(sh.lps_enabled))
    n, t0 = 0, time.perf_counter()
    while True:
        res = o.step(inp, W, prm, suffix=suffix)
        n += 1
        el = time.perf_counter() - t0
        if el >= budget_s:
            break
    return inp.rows * n / el, n, el, res


def parity_summary(sh, inp, res, gpu, tol=2e-3):
    """The GPU step's outputs (one step from the same state) against the
    oracle's: near-ties counted (a top-2 logit gap, or a decision margin,
    below 1e-3), argmax mismatches outside near-ties,
    decision mismatches in sequences the oracle does not flag, and the
    largest differences of the floating-point outputs."""
    NT = 1e-3
    st = res.stats
    masked = inp.mask.astype(bool)
    scored = ~np.isnan(res.lps_prob)
    routed = ~np.isnan(res.lbs_logit)
    nt = st.logit_gap < NT
    out = {"against": "the CPU oracle (float64) on the same inputs, one step",
           "tolerance_abs": tol,
           "near_ties": {"top2_logit_gap": int(nt.sum()),
                         "kappa_vs_tau": int((masked & (np.abs(st.conf - sh.tau) < NT)).sum()),
                         "p_psi_vs_tau_psi": int((scored & (np.abs(res.lps_prob - sh.tau_psi) < NT)).sum()),
                         "lbs_logit_vs_0": int((routed & (np.abs(res.lbs_logit) < NT)).sum())},
           "argmax_mismatch": int(((gpu["argmax"].astype(np.int64) != st.argmax) & ~nt).sum())}
    B = len(inp.cu_rows) - 1
    flagged = 0
    mism = {"accepted": 0, "tokens": 0, "mask": 0, "in_block": 0, "blk_meta": 0}
    for b in range(B):
        if res.flag_accept[b] or res.flag_lbs[b]:
            flagged += 1
            continue
        sl = slice(int(inp.cu_rows[b]), int(inp.cu_rows[b + 1]))
        for k in ("accepted", "tokens", "mask", "in_block"):
            mism[k] += int((np.asarray(gpu[k][sl]).astype(np.int64) !=
                            np.asarray(getattr(res, k)[sl]).astype(np.int64)).sum())
        mism["blk_meta"] += int(not np.array_equal(gpu["blk_meta"][b], res.blk_meta[b]))
    out["flagged_sequences"] = flagged
    out["sequences"] = B
    out["decision_mismatch"] = mism
    diff = {}
    for k, ref in (("conf", st.conf), ("entropy", st.entropy), ("ent_norm", st.ent_norm),
                   ("gap", st.gap)):
        diff[k] = float(np.abs(gpu[k].astype(np.float64) - ref).max())
    if "attn_out" in gpu and res.attn_out is not None:
        diff["attn_out"] = float(np.abs(gpu["attn_out"].astype(np.float64) - res.attn_out).max())
    out["max_abs_diff"] = {k: float(f"{v:.3g}") for k, v in diff.items()}
    out["within_tolerance"] = bool(max(diff.values()) <= tol and out["argmax_mismatch"] == 0 and
                                   not any(mism.values()))
    return out


def run_loop_bench(args):
    """The generation loop (configs loop_*): one untimed loop, then
    max(1, steps // 100) timed loops to completion; reports the number of
    steps, the device time of all steps (CUDA events around every ebd_step)
    and the wall time including the per-step host work (synthetic backbone
    outputs, window rule, state read-back)."""
    import torch
    from paper_2609_16450_gb300 import build as B
    B.build()
    from paper_2609_16450_gb300 import loop as lp
    from paper_2609_16450_gb300 import runtime as rt
    import synth
    sh = shape_for(args.config)
    inp = synth.make_step_inputs(sh)
    w = rt.upload_weights(inp)
    mode = {"eb": 0, "threshold": 1, "topm": 2}[args.decode]
    full = full_sequence(sh)
    h = rt.Handle(lp.config_for_loop(sh, max_window=sh.gen_len if full else 64, decode_mode=mode,
                                     top_m=args.top_m), w.w_emb)
    if args.w_layout == "packed":
        w = rt.pack_weights(h, w)
    win = lambda s, p: synth.loop_window_inputs(sh, s, p)
    kv = lambda p: synth.loop_kv(sh, p)
    opts = dict(keep=False, block=sh.l_b, cache=args.cache, append=args.append)
    if full:
        opts.update(window="full", attention=False)
    lp.run_loop(h, sh, w, win, kv, **opts)  # warm-up loop
    runs = []
    for _ in range(max(1, args.steps // 100)):
        t0 = time.perf_counter()
        res = lp.run_loop(h, sh, w, win, kv, **opts)
        runs.append((res.steps, res.device_us, time.perf_counter() - t0))
    steps = runs[0][0]
    dev_us = float(np.mean([r[1] for r in runs]))
    wall_s = float(np.mean([r[2] for r in runs]))
    wk_rows = sh.gen_len
    line = {"metric": "generation loop: steps and total time (LLaDA-8B shape)",
            "value": round(wk_rows / (dev_us * 1e-6), 1), "unit": "positions/s",
            "n_gpus": 1, "steps": len(runs), "warmup": 1, "ms_per_step": round(dev_us / steps / 1000, 5),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded per step and position)",
            "config": {"workload": (f"{sh.name}: prompt {sh.prefix}, gen {sh.gen_len}, every step's "
                                    f"window is the whole response (full-sequence setting), no "
                                    f"window attention") if full else
                                   (f"{sh.name}: prompt {sh.prefix}, gen {sh.gen_len}, windows of "
                                    f"at most 64 rows, attention over the committed prefix"),
                       "decode": args.decode + (f" (m={args.top_m})" if args.decode == "topm" else ""),
                       "fixed_block": sh.l_b if args.decode != "eb" else None,
                       "kv_cache": ("dual: the window also attends to the positions after it"
                                    if args.cache == "dual" else "prefix") +
                                   ("; committed rows appended to the cache by each step, which "
                                    "starts with the prompt only" if args.append and args.cache == "prefix"
                                    else "; committed rows appended by each step" if args.append else ""),
                       "loop_steps": steps, "device_us_total": round(dev_us, 1),
                       "wall_s_total": round(wall_s, 3),
                       "l2": "not flushed between steps (consecutive steps of one loop)"}}
    h.close()
    print(json.dumps(line))


def config_dict(sh, args, rows, masked, world):
    """The workload of a bench line, the same for both arms."""
    return {"workload": workload_text(sh, args.state), "state": args.state,
            "rows": rows, "masked": masked,
            "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
            "l2": "flushed before every timed step: 256 MB write, then 256 MB read (write-back "
                  "done outside the timed region); W_lm (1 GB) > L2",
            "launch": "cuda_graph" if not args.no_graph else "stream",
            "kv_cache": (f"dual: prefix + window + {suffix_len(sh)} cached positions after "
                         f"the window" if args.cache == "dual" else "prefix") +
                        ("; committed rows appended every step" if args.append else ""),
            "w_lm": ("64x64 tiles, unit-major (ebd_pack_lm_head, once at load)"
                     if args.w_layout == "packed" else "row-major [V][d]")}


def run_reference(args, rank, world):
    """The CPU oracle as the reference arm: rank 0 only."""
    if rank != 0:
        return
    import synth
    sh = shape_for(args.config)
    inp = synth.make_step_inputs(sh)
    if args.state == "inblock":
        synth.preset_in_block(inp, 20)
    from oracle import ebd_oracle as o
    W = o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))
    prm = o.DecisionParams(tau=sh.tau, tau_psi=sh.tau_psi, l_min=sh.l_min, l_b=sh.l_b,
                           g_max=sh.g_max, eos_id=sh.eos_id, lps_enabled=bool(sh.lps_enabled))
    # size each step's sample so that warm-up + timed steps fit in ~150 s
    t0 = time.perf_counter()
    o.step(inp, W, prm)
    t_full = time.perf_counter() - t0
    budget = 150.0 / max(1, args.steps + args.warmup)
    rows = inp.rows
    if t_full > budget:
        rows = max(1, int(inp.rows * budget / t_full))
    sub = inp if rows == inp.rows else _row_sample(inp, rows)
    for _ in range(args.warmup):
        o.step(sub, W, prm)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        o.step(sub, W, prm)
        times.append(time.perf_counter() - t0)
    ms = 1000.0 * float(np.mean(times))
    value = rows / (ms / 1000.0)
    cores = os.cpu_count()
    sample = (f"oracle step on {rows} of {inp.rows} window rows of {sh.name} per timed step"
              if rows != inp.rows else f"full oracle step of {sh.name} ({inp.rows} rows)")
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 3), "unit": UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(ms, 3), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_dict(sh, args, inp.rows, int(inp.mask.sum()), world),
            "cpu_baseline": {"value": round(value, 3), "unit": UNIT, "cores": cores,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 3), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def _row_sample(inp, rows):
    """First `rows` window rows of the single-sequence step (bounded sample)."""
    import copy
    s = copy.copy(inp)
    s.cu_rows = np.array([0, rows], np.int32)
    s.row_pos = inp.row_pos[:rows]
    for k in ("hidden", "q", "k_win", "v_win", "tokens", "mask", "in_block"):
        setattr(s, k, getattr(inp, k)[:rows])
    return s


# ----------------------------------------------------------------------------- main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--config", default="llada8b")
    ap.add_argument("--state", choices=["select", "inblock"], default="select")
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--skip-cpu", action="store_true", help="omit the cpu_baseline leg")
    ap.add_argument("--skip-e2e", action="store_true", help="omit the end-to-end leg")
    ap.add_argument("--no-graph", action="store_true", help="launch ebd_step without a graph")
    ap.add_argument("--cpu-budget", type=float, default=12.0)
    ap.add_argument("--decode", choices=["eb", "threshold", "topm"], default="eb",
                    help="decision of the loop configs: EB, or a baseline's fixed-block rule")
    ap.add_argument("--top-m", type=int, default=1, help="commits per step of --decode topm")
    ap.add_argument("--cache", choices=["prefix", "dual"], default="prefix",
                    help="dual: each window also attends to the cached rest of its response")
    ap.add_argument("--append", action="store_true",
                    help="write committed rows' K/V into the cache every step")
    ap.add_argument("--w-layout", choices=["packed", "rowmajor"], default="packed",
                    help="W_lm tiled once by ebd_pack_lm_head (default) or row-major")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if args.config.startswith("loop_"):
        if rank == 0:
            run_loop_bench(args)
        return
    import torch
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    r = run_ours(args, rank, world, local_rank)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    sh = r["sh"]
    hbm, bf16, bf16_sus, peak_src = load_peaks()
    wk = step_work(sh, r["rows"], r["masked"], r["grid_lm"], r["lbs_runs"],
                   suffix=suffix_len(sh) if args.cache == "dual" else 0, append=args.append)
    t_lm = r["k_lm"] / 1000.0
    lm_hbm_t = wk["lm_bytes"] / (hbm * 1e9)
    lm_tc_t = wk["lm_flops"] / (bf16 * 1e12)
    if lm_hbm_t >= lm_tc_t:
        roof = {"bound": "hbm", "achieved": round(wk["lm_bytes"] / t_lm / 1e9, 1),
                "peak": hbm, "unit": "GB/s"}
    else:
        roof = {"bound": "tensor", "achieved": round(wk["lm_flops"] / t_lm / 1e12, 1),
                "peak": bf16, "unit": "TFLOP/s"}
    roof["frac"] = round(roof["achieved"] / roof["peak"], 4)
    roof["traffic"] = profiled_traffic(sh.name)
    roof["kernel"] = "lm_stats_kernel (LM head + online softmax statistics)"
    roof["algorithmic"] = {"bytes": wk["lm_bytes"], "flops": wk["lm_flops"]}
    roof["peak_source"] = f"{peak_src} (MEASURED_PEAKS.json)" if peak_src == "measured" else "fallback"
    t_step = r["mean_ms"] / 1000.0
    t_roof = max(wk["step_bytes"] / (hbm * 1e9), wk["step_flops"] / (bf16 * 1e12))
    value = replicas_value(r["rows"], world, t_step)
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(r["mean_ms"], 5),
        "us_per_step": round(r["mean_ms"] * 1000, 2),
        "us_per_step_p10_p50_p90": [round(float(np.percentile(r["step_ms"], q)) * 1000, 2)
                                    for q in (10, 50, 90)],
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded; LLaDA-8B/Dream-7B shapes, random-init routers)",
        "config": config_dict(sh, args, r["rows"], r["masked"], world),
        "roofline": roof,
        "step_roofline": {"bytes": wk["step_bytes"], "flops": wk["step_flops"],
                          "t_roofline_us": round(t_roof * 1e6, 2),
                          "frac": round(t_roof / t_step, 4),
                          "peak_hbm_gbs": hbm, "peak_bf16_tflops": bf16},
        "kernels_us": {"attention": round(r["k_attn"] * 1000, 2),
                       "lm_head": round(r["k_lm"] * 1000, 2),
                       "decision": round(r["k_dec"] * 1000, 2),
                       "decision_with_attention_overlapped": round(r["k_tail"] * 1000, 2),
                       "note": "timed steps carry no interior events; lm_head and the "
                               "overlapped tail come from a pass with events around the LM "
                               "head, attention and decision alone from a serial pass"},
        "kernels_achieved": {
            "lm_head": {"GB/s": round(wk["lm_bytes"] / t_lm / 1e9, 1),
                        "TFLOP/s": round(wk["lm_flops"] / t_lm / 1e12, 1)},
            "attention": ({"GB/s": round(wk["attn_bytes"] / (r["k_attn"] / 1000.0) / 1e9, 1),
                           "TFLOP/s": round(wk["attn_flops"] / (r["k_attn"] / 1000.0) / 1e12, 2)}
                          if wk["attn_bytes"] and r["k_attn"] > 0 else None),
            "note": "algorithmic bytes and flops over each kernel's measured time"},
        "vs_spec": {"hbm_gbs_spec": 8000.0,
                    "lm_head_frac_of_spec_hbm": round(wk["lm_bytes"] / t_lm / 1e9 / 8000.0, 4),
                    "bf16_tflops_sustained": bf16_sus,
                    "step_frac_with_sustained_bf16": round(max(wk["step_bytes"] / (hbm * 1e9),
                                                               wk["step_flops"] / (bf16_sus * 1e12)) / t_step, 4)},
        "decision_share": round(r["k_dec"] / max(1e-9, r["mean_ms"]), 4),
        "decision_share_paper": "6.21 % (LBS 3.80 % + LPS 2.41 % of the backbone forward, A100)",
        "gpu_launches": int(r["launches_per_step"] * args.steps),
        "clocks": r["clocks"],
    }
    if r["e2e"] is not None:
        e = r["e2e"]
        line["e2e"] = {"value": round(replicas_value(r["rows"], world, e["mean_ms"] / 1000.0), 1),
                       "unit": UNIT, "h2d_bytes_per_step": e["h2d"],
                       "d2h_bytes_per_step": e["d2h"], "ms_per_step": round(e["mean_ms"], 4),
                       "api": "ebd_step_host"}
    if not args.skip_cpu and world == 1:
        v, n, el, res = oracle_step_sample(sh, r["inp"], args.cpu_budget, r["suffix"])
        line["cpu_baseline"] = {"value": round(v, 3), "unit": UNIT, "cores": os.cpu_count(),
                                "kind": "oracle",
                                "sample": f"{n} full oracle steps of {sh.name} "
                                          f"({r['rows']} rows each) in {el:.1f} s"}
        line["parity"] = parity_summary(sh, r["inp"], res, r["fetch"])
    print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
