"""Decode-step benchmark: paged decode attention (+ fused K/V append) on GB300.

A step is one pass of the whole hot path over one batch: the step's lazy page
allocation, page-table update and split plan (kv_begin_step_device, all on the
device) and, for each of the L layers, the fused K/V append + decode attention
(decode_attention_append; the merge pass follows when a row is split).  By
default the step is captured once into CUDA graphs and replayed; --host-steps
plans on the host (kv_begin_step) and launches from Python, --unfused launches
kv_append and decode_attention separately.  The default workload is the
LLaVA-1.5-7B-shaped batch (32 layers, 32/32 heads, d 128, batch 64, 576 vision
tokens + U[64,512] prompt + U{0..256} generated tokens, page 16, shuffled page
table).  Inputs are seeded synthetic draws (paper_2603_12707_gb300.workloads).

value = algorithmic bytes of K timed steps / their device time (GB/s): per
layer and sequence, K and V of every attended token, the Q read, the O write
and the appended K/V write, all bf16.  The timed region is R consecutive
blocks of exactly K steps (R from 3 to 10, for about half a second of timed
work, so that the clock samples taken every 20 ms cover it); the line reports
the median block and lists every block's time.  The roofline object reports
the decode_attention kernel alone (KV + Q + O bytes per launch over its
CUDA-event duration on the launch stream) against the measured HBM copy
bandwidth.  At one GPU the line also carries, under "configs", the same
measurement of every other workload (qwen, long, ragged, tiny), each run in
its own cache with the same steps and warm-up.

Multi-GPU: the path has no exchange step, so N GPUs run N independent replicas
(weak scaling); ranks meet only for the barrier and the max of their times.
--impl reference times the float64 CPU oracle on the host cores instead.
"""
from __future__ import annotations

import argparse
import hashlib
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
sys.path.insert(0, ROOT)

METRIC = "decode-attention achieved HBM GB/s (% of GB300 peak) and decode steps/sec"
ALL_WORKLOADS = ("llava", "qwen", "long", "ragged", "tiny")
NOMINAL_HBM_GBS = 8000.0


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def layer_bytes(cfg, attended):
    """(attention bytes, append bytes) of one layer: KV of every attended
    token + Q read + O write; appended K and V written."""
    Hq, Hkv, d = cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim
    B = len(attended)
    attn = int(sum(attended)) * 2 * Hkv * d * 2 + B * Hq * d * 2 * 2
    app = B * 2 * Hkv * d * 2
    return attn, app


def kv_bytes(cfg, attended):
    """KV bytes one layer reads for the attended lengths."""
    return int(sum(attended)) * 2 * cfg.num_kv_heads * cfg.head_dim * 2


def describe(cfg):
    return {"workload": cfg.name + ": " + cfg.description, "batch": cfg.batch, "layers": cfg.num_layers,
            "layer_pools": cfg.phys_layers, "q_heads": cfg.num_q_heads, "kv_heads": cfg.num_kv_heads,
            "head_dim": cfg.head_dim, "page_size": cfg.page_size, "page_order": cfg.page_order,
            "seed": cfg.seed}


def workload_config(args):
    """The named workload with the command line's overrides (layer pools held, page order)."""
    import dataclasses
    from paper_2603_12707_gb300 import workloads as wl
    cfg = wl.CONFIGS[args.config]
    if args.phys_layers:
        cfg = dataclasses.replace(cfg, phys_layers=args.phys_layers)
    if args.page_order:
        cfg = dataclasses.replace(cfg, page_order=args.page_order)
    return cfg


# ------------------------------------------------------------------ clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id, interval_ms=20):
        self.gpu_id = gpu_id
        self.interval_ms = int(interval_ms)
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu_id}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", str(self.interval_ms)],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception as e:  # no nvidia-smi: report no samples
            log("clock sampling unavailable:", e)
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if self.proc is None or not self.path:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(n)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def clocks_slowed(summary):
    """A clock record that the timing rules reject: hardware or thermal
    slowdown active, or SM clocks far below their maximum with no reason."""
    if set(summary.get("reasons", [])) & {"hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"}:
        return True
    sm, smax = summary.get("sm_mhz"), summary.get("sm_max_mhz")
    return bool(sm and smax and sm < 0.85 * smax and not summary.get("reasons"))


def gpu_smi_id(torch, dev):
    try:
        p = torch.cuda.get_device_properties(dev)
        return f"{p.pci_domain_id:08X}:{p.pci_bus_id:02X}:{p.pci_device_id:02X}.0"
    except Exception:
        return str(dev)


# --------------------------------------------------------- kernel traffic
KERNEL_SOURCES = [os.path.join(ROOT, "paper_2603_12707_gb300", "csrc", f)
                  for f in ("kvd_decode_kernel.cuh", "kvd_ptx.cuh")]


def kernel_code_hash(paths):
    """sha256 (16 hex digits) of the split-pass kernel's device code: line
    comments, blank lines and surrounding whitespace removed, so a comment
    edit keeps a capture valid and any code edit voids it."""
    import re
    lines = []
    for path in paths:
        with open(path) as f:
            lines += [re.sub(r"//.*$", "", l).strip() for l in f]
    return hashlib.sha256("\n".join(l for l in lines if l).encode()).hexdigest()[:16]


def committed_traffic(kernel_srcs, workload, algorithmic_bytes):
    """DRAM bytes per launch of the decode kernel: the committed ncu capture's
    traffic / algorithmic ratio for this workload times this launch's
    algorithmic bytes; None unless the capture was taken on the current
    kernel source."""
    p = os.path.join(ROOT, "profiles", "decode_kernel_traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    h = kernel_code_hash(kernel_srcs)
    cap = d.get("captures", {}).get(workload)
    if d.get("source_sha256_16") != h or cap is None:
        return None
    return int(round(cap["traffic_over_algorithmic"] * algorithmic_bytes))


# ------------------------------------------------------------- CPU oracle
def oracle_sample(cfg, budget_s):
    """Time the float64 oracle on one layer of the workload (all sequences and
    heads, one decode step), repeated until about budget_s seconds of oracle
    time or one full step's worth of layers.  Returns (bytes, seconds,
    description, threads)."""
    import oracle
    from paper_2603_12707_gb300 import workloads as wl
    import torch
    lens = [int(n) + 1 for n in wl.context_lengths(cfg)]
    k = torch.cat([wl.kv_block(cfg, 0, b, n, "k", "cpu") for b, n in enumerate(lens)])
    v = torch.cat([wl.kv_block(cfg, 0, b, n, "v", "cpu") for b, n in enumerate(lens)])
    q = wl.step_inputs(cfg, 0, 0, "cpu")[0]
    attn, _ = layer_bytes(cfg, lens)
    done_bytes, spent, layers = 0, 0.0, 0
    while spent < budget_s and layers < cfg.num_layers:
        t0 = time.perf_counter()
        oracle.decode_attention(q, lens, k, v)
        spent += time.perf_counter() - t0
        done_bytes += attn
        layers += 1
    threads = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    desc = (f"{layers} of {cfg.num_layers} layers of one decode step of the {cfg.name} workload "
            f"({cfg.batch} sequences x {cfg.num_q_heads} heads each; every layer repeats layer 0's K/V), "
            f"float64 oracle, OpenMP over (sequence, head)")
    return done_bytes, spent, desc, threads


# -------------------------------------------------------------- GPU run
def block_count(first_block_ms, args):
    """Timed blocks of K steps: enough for about args.block_target_s seconds of
    timed work (so the clock samples cover it), within [args.min_blocks,
    args.max_blocks]."""
    want = math.ceil(args.block_target_s * 1e3 / max(first_block_ms, 1e-6))
    return int(min(args.max_blocks, max(args.min_blocks, want)))


def median_block(block_ms):
    """Index of the median block (the lower median for an even count)."""
    order = sorted(range(len(block_ms)), key=lambda i: block_ms[i])
    return order[(len(order) - 1) // 2]


def run_gpu(args, rank, world, cfg):
    import torch
    from paper_2603_12707_gb300 import kvdecode as kd, workloads as wl
    from paper_2603_12707_gb300.harness import DecodeSession

    dev = int(os.environ.get("LOCAL_RANK", 0))
    torch.cuda.set_device(dev)
    stream = torch.cuda.Stream()
    # room for the warm-up, the timed blocks (twice: they are taken again
    # once if the clocks show a slowdown), the end-to-end steps and slack
    total_steps = (args.warmup + 2 * args.max_blocks * args.steps + (args.steps if not args.no_e2e else 0) + 2)
    t_setup = time.perf_counter()
    with torch.cuda.stream(stream):
        sess = DecodeSession(cfg, extra_tokens=total_steps + 1, device="cuda", stream=stream,
                             split_pages=args.split_pages)
        sess.fill_prefix()
        L, B = cfg.num_layers, cfg.batch
        # Every layer's q, k_new, v_new live in one device buffer and every
        # layer's output in another, so the end-to-end leg moves a step's
        # inputs and outputs in one copy each way.
        Hq, Hkv, d = cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim
        per_layer = B * (Hq + 2 * Hkv) * d
        d_in = torch.empty(L * per_layer, dtype=torch.bfloat16, device="cuda")
        d_out = torch.empty((L, B, Hq, d), dtype=torch.bfloat16, device="cuda")

        def views(d_in, d_out):
            qs, ks, vs = [], [], []
            for l in range(L):
                x = d_in[l * per_layer:(l + 1) * per_layer]
                qs.append(x[:B * Hq * d].view(B, Hq, d))
                ks.append(x[B * Hq * d:B * (Hq + Hkv) * d].view(B, Hkv, d))
                vs.append(x[B * (Hq + Hkv) * d:].view(B, Hkv, d))
            return qs, ks, vs, [d_out[l] for l in range(L)]

        qs, ks, vs, outs = views(d_in, d_out)
        for l in range(L):
            q, k, v = wl.step_inputs(cfg, 0, l, "cuda")
            qs[l].copy_(q), ks[l].copy_(k), vs[l].copy_(v)
    stream.synchronize()
    log(f"[rank {rank}] setup {time.perf_counter() - t_setup:.1f} s; pool "
        f"{sess.query().pool_bytes / 2**30:.1f} GiB")

    graphs = None
    if args.graph:
        # The whole step as two CUDA graphs: the device-side kv_begin_step
        # (page pops, lengths, split plan) and the L fused layers.  Replays
        # need no host work; an event between the two times the layers.
        ids_dev = torch.tensor(sess.seq_ids, dtype=torch.int32, device="cuda")
        kd.kv_cache_device_steps(sess.h, B, True, stream)

        def layers(v):
            for l in range(L):
                sess.append_attend(l, v[0][l], v[1][l], v[2][l], v[3][l])

        with torch.cuda.stream(stream):
            kd.kv_begin_step_device(sess.h, B, ids_dev, stream)   # eager step: nothing lazy in the capture
            layers((qs, ks, vs, outs))
        sess.lens += 1
        stream.synchronize()
        n0 = sess.query().kernel_launches
        g_begin, g_layers = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_begin, stream=stream):
            kd.kv_begin_step_device(sess.h, B, ids_dev, stream)
        with torch.cuda.graph(g_layers, stream=stream):
            layers((qs, ks, vs, outs))
        graphs = (g_begin, g_layers, sess.query().kernel_launches - n0)
        # a second input/output set, so the end-to-end leg can move one step's
        # inputs and outputs while another step runs
        d_in2, d_out2 = d_in.clone(), torch.empty_like(d_out)
        g_layers2 = torch.cuda.CUDAGraph()
        if not args.no_e2e:
            with torch.cuda.graph(g_layers2, stream=stream):
                layers(views(d_in2, d_out2))

    def step(events=None):
        """One decode step.  events: per-step event list to time the attention
        launches.  Unfused: a pair around every decode_attention.  Fused: one
        event after kv_begin_step and one after the last layer (the fused
        launches are PDL-chained, and an event between two of them would cut
        the overlap), so a launch's time is the span over L."""
        if graphs is not None:
            graphs[0].replay()
            if events is not None:
                events[0].record(stream)
            graphs[1].replay()
            if events is not None:
                events[1].record(stream)
            sess.lens += 1
            return
        sess.begin_step()
        if events is not None and not args.unfused:
            events[0].record(stream)
        for l in range(L):
            if args.unfused:
                sess.append(l, ks[l], vs[l])
                if events is not None:
                    events[2 * l].record(stream)
                sess.attend(l, qs[l], outs[l])
                if events is not None:
                    events[2 * l + 1].record(stream)
            else:
                sess.append_attend(l, qs[l], ks[l], vs[l], outs[l])
        if events is not None and not args.unfused:
            events[1].record(stream)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step()
    stream.synchronize()

    # ---- device-timed region: R blocks of exactly K steps each, the whole
    # region under the clock sampler; the median block is reported.  It is
    # taken again once if the clock samples show a thermal or hardware
    # slowdown, or SM clocks far below their maximum with no reason given
    # (the second run is the one reported).
    n_ev = 2 * L if args.unfused else 2

    def timed_block():
        attended = []
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(n_ev)] for _ in range(args.steps)]
        step_ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
        with torch.cuda.stream(stream):
            step_ev[0].record(stream)
            for s in range(args.steps):
                attended.append([int(n) + 1 for n in sess.lens])
                step(ev[s])
                step_ev[s + 1].record(stream)
        return attended, ev, step_ev

    def block_result(attended, ev, step_ev):
        step_ms = [step_ev[i].elapsed_time(step_ev[i + 1]) for i in range(args.steps)]
        if args.unfused:
            attn_ms = [evs[2 * l].elapsed_time(evs[2 * l + 1]) for evs in ev for l in range(L)]
        else:
            attn_ms = [evs[0].elapsed_time(evs[1]) / L for evs in ev]
        step_bytes, attn_bytes = [], []
        for att in attended:
            a, p = layer_bytes(cfg, att)
            step_bytes.append(L * (a + p))
            attn_bytes.append(a if args.unfused else a + p)   # the fused kernel also writes the new K/V
        return {"ms": step_ev[0].elapsed_time(step_ev[-1]), "step_ms": step_ms, "attn_ms": attn_ms,
                "step_bytes": step_bytes, "attn_bytes": attn_bytes,
                "attended": [statistics.mean(att) for att in attended],
                "kv_bytes": [L * kv_bytes(cfg, att) for att in attended]}

    for attempt in range(2):
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()
        launches0 = sess.query().kernel_launches
        blocks = []
        with ClockSampler(gpu_smi_id(torch, dev), args.clock_ms) as clocks:
            recorded = [timed_block()]
            stream.synchronize()
            first = reduce_max(torch, recorded[0][2][0].elapsed_time(recorded[0][2][-1]), world)
            n_blocks = block_count(first, args)
            for _ in range(n_blocks - 1):
                recorded.append(timed_block())
            stream.synchronize()
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()
        blocks = [block_result(*r) for r in recorded]
        for b in blocks:
            b["ms"] = reduce_max(torch, b["ms"], world)
        clock_summary = clocks.summary()
        slowed = reduce_max(torch, 1.0 if clocks_slowed(clock_summary) else 0.0, world) > 0
        if not slowed or attempt == 1:
            break
        log("clock samples show a slowdown during the timed steps:", clock_summary, "- timing them again")
    clock_summary["retimed"] = attempt == 1
    st = sess.query()
    assert st.device_error == 0, st.device_error
    # graph replays do not pass through the library: count the captured launches
    total_launches = (graphs[2] * args.steps * len(blocks) if graphs is not None
                      else st.kernel_launches - launches0)
    timed_launches = total_launches // len(blocks)

    # ---- end to end: host inputs -> device -> host outputs, every step: a
    # step's q, k_new, v_new of all layers go over from pinned host memory in
    # one copy and all layers' outputs come back in one copy.  With replayed
    # graphs the copies run on a second stream, double-buffered: step s+1's
    # inputs move while step s runs, and step s's outputs once it is done.
    # With --host-steps / --unfused, or under 1 MB a step, they are serial.
    e2e = None
    if not args.no_e2e:
        h_in = d_in.cpu().pin_memory()
        h_out = torch.empty_like(d_out, device="cpu").pin_memory()
        e_bytes = 0
        h2d = h_in.numel() * 2
        d2h = h_out.numel() * 2
        s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        # (device steps stay enabled from the capture on: re-enabling them
        # could move the scratch buffers the captured graphs point at)
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()
        w0 = time.perf_counter()
        # (a step that moves under 1 MB is launch-bound: the extra stream
        # operations of double buffering would cost more than they hide)
        if graphs is not None and h2d + d2h >= 2**20:
            copy = torch.cuda.Stream()
            sets = [(d_in, d_out, graphs[1]), (d_in2, d_out2, g_layers2)]
            ev_in = [torch.cuda.Event() for _ in range(2)]
            ev_done = [torch.cuda.Event() for _ in range(2)]
            ev_out = [torch.cuda.Event() for _ in range(2)]
            s0.record(stream)
            copy.wait_event(s0)
            with torch.cuda.stream(copy):
                d_in.copy_(h_in, non_blocking=True)
                ev_in[0].record(copy)
            for s in range(args.steps):
                i = s % 2
                att = [int(n) + 1 for n in sess.lens]
                a, p = layer_bytes(cfg, att)
                e_bytes += L * (a + p)
                with torch.cuda.stream(stream):
                    stream.wait_event(ev_in[i])
                    if s >= 2:
                        stream.wait_event(ev_out[i])   # step s-2's outputs have left this set
                    graphs[0].replay()
                    sets[i][2].replay()
                    ev_done[i].record(stream)
                sess.lens += 1
                with torch.cuda.stream(copy):
                    if s + 1 < args.steps:
                        j = 1 - i
                        if s >= 1:
                            copy.wait_event(ev_done[j])   # step s-1 has read this set's inputs
                        sets[j][0].copy_(h_in, non_blocking=True)
                        ev_in[j].record(copy)
                    copy.wait_event(ev_done[i])
                    h_out.copy_(sets[i][1], non_blocking=True)
                    ev_out[i].record(copy)
            stream.wait_stream(copy)
            s1.record(stream)
        else:
            with torch.cuda.stream(stream):
                s0.record(stream)
                for s in range(args.steps):
                    att = [int(n) + 1 for n in sess.lens]
                    a, p = layer_bytes(cfg, att)
                    e_bytes += L * (a + p)
                    d_in.copy_(h_in, non_blocking=True)
                    step()
                    h_out.copy_(d_out, non_blocking=True)
                s1.record(stream)
        stream.synchronize()
        wall = time.perf_counter() - w0
        e_ms = s0.elapsed_time(s1)
        e2e = {"ms": e_ms, "wall_s": wall, "bytes": e_bytes, "h2d": h2d, "d2h": d2h}
        st = sess.query()
        assert st.device_error == 0

    start_attended = statistics.mean(int(n) for n in sess.lens0) + 1   # the first step's contexts
    sess.close()
    del sess
    torch.cuda.synchronize()
    return {"blocks": blocks, "launches": timed_launches, "clocks": clock_summary, "e2e": e2e, "cfg": cfg, "L": L,
            "start_attended": start_attended}


def run_varlen_write(args, rank, world):
    """Time kv_write_varlen: the workload's whole batch of cached prefixes
    (vision tokens + prompt + generated), packed, written into every layer
    pool in one call per step.  Bytes = packed K/V read + pool pages written."""
    import torch
    from paper_2603_12707_gb300 import _build, kvdecode as kd, workloads as wl
    from paper_2603_12707_gb300.harness import DecodeSession

    dev = int(os.environ.get("LOCAL_RANK", 0))
    torch.cuda.set_device(dev)
    if rank == 0:
        _build.build_library()
    if world > 1:
        torch.distributed.barrier()
    cfg = workload_config(args)
    stream = torch.cuda.Stream()
    sess = DecodeSession(cfg, extra_tokens=1, device="cuda", stream=stream)
    lens = [int(n) for n in sess.lens0]
    L = cfg.phys_layers
    src_bytes = 2 * sum(lens) * cfg.num_kv_heads * cfg.head_dim * 2 * L
    if src_bytes > 64 * 2**30:
        raise SystemExit(f"packed source of {src_bytes / 2**30:.0f} GiB: pass --phys-layers")
    k, v, cu = wl.packed_prefix(cfg, range(L), lens, "cuda")
    torch.cuda.synchronize()

    def step():
        kd.kv_write_varlen(sess.h, 0, L, sess.seq_ids, cu, k, v, stream=stream)

    for _ in range(args.warmup):
        step()
    stream.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    n0 = sess.query().kernel_launches
    with ClockSampler(gpu_smi_id(torch, dev), args.clock_ms) as clocks:
        for a, b in ev:
            a.record(stream)
            step()
            b.record(stream)
        stream.synchronize()
    torch.cuda.synchronize()
    st = sess.query()
    assert st.device_error == 0
    launches = st.kernel_launches - n0
    ms = sum(a.elapsed_time(b) for a, b in ev)
    sess.close()
    return {"ms": ms, "bytes": 2 * src_bytes, "launches": launches, "clocks": clocks.summary(), "cfg": cfg,
            "blocks": len(lens), "rows": cu[-1]}


def varlen_main(args, rank, world):
    import torch
    r = run_varlen_write(args, rank, world)
    ms = reduce_max(torch, r["ms"], world)
    gbs = r["bytes"] * args.steps * world / (ms / 1e3) / 1e9
    peak, peak_kind = measured_peaks()
    cfg = r["cfg"]
    out = {
        "metric": "paged varlen K/V bulk write (prefix handoff), HBM GB/s read + write", "value": round(gbs, 2),
        "unit": "GB/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms / args.steps, 4), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {**describe(cfg), "blocks": r["blocks"], "packed_rows": r["rows"],
                   "l2": "each step reads and writes the whole prefix batch (far larger than the 129 MB L2)"
                         if r["bytes"] > 2**30 else "fits in L2: launch-bound, not a roofline number",
                   "parallelism": f"replicas x{world}"},
        "roofline": {"bound": "hbm", "kernel": "kv_write_varlen", "achieved": round(gbs / world, 2), "peak": peak,
                     "peak_kind": peak_kind, "unit": "GB/s", "frac": round(gbs / world / peak, 4), "traffic": None,
                     "algorithmic_bytes_per_launch": int(r["bytes"] / max(1, r["launches"] // args.steps)),
                     "avg_launch_ms": round(ms / max(1, r["launches"]), 4)},
        "clocks": r["clocks"], "gpu_launches": r["launches"],
    }
    if world > 1:
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()
    if rank == 0:
        print(json.dumps(out))


def reduce_max(torch, x, world):
    """Max of x over the ranks (the job's time is its slowest rank's)."""
    if world == 1:
        return x
    dev = "cpu" if torch.distributed.get_backend() == "gloo" else "cuda"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def whole_job_gbs(bytes_per_rank, max_ms, world):
    """Whole-job throughput: every rank's bytes over the slowest rank's time."""
    return bytes_per_rank * world / (max_ms / 1e3) / 1e9


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default="llava", choices=["tiny", "llava", "qwen", "ragged", "long"])
    ap.add_argument("--phys-layers", type=int, default=0, help="layer pools held (profiling on a smaller cache)")
    ap.add_argument("--page-order", choices=["sequential", "shuffled", "interleaved"], default=None,
                    help="physical page order of the pool (default: the workload's own)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--split-pages", type=int, default=0,
                    help="target pages per work item (0: the library's automatic choice)")
    ap.add_argument("--unfused", action="store_true",
                    help="kv_append and decode_attention as two launches per layer (default: one fused launch)")
    ap.add_argument("--host-steps", action="store_true",
                    help="plan each step on the host (kv_begin_step) and launch the layers from Python "
                         "(default: replay CUDA graphs of kv_begin_step_device and the fused layers)")
    ap.add_argument("--varlen-write", action="store_true",
                    help="time the packed varlen bulk K/V write of the workload's prefixes instead of decode")
    ap.add_argument("--configs", default=None,
                    help="comma-separated workloads measured after the headline one, in the same run "
                         "(default: every other workload at one GPU, none on several)")
    ap.add_argument("--min-blocks", type=int, default=3, help="timed blocks of --steps steps, at least")
    ap.add_argument("--max-blocks", type=int, default=10, help="timed blocks of --steps steps, at most")
    ap.add_argument("--block-target-s", type=float, default=0.5,
                    help="timed blocks are added up to about this many seconds of timed work")
    ap.add_argument("--clock-ms", type=int, default=20, help="clock sampling interval (nvidia-smi -lms)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget-s", type=float, default=12.0)
    args = ap.parse_args()
    args.graph = not (args.host_steps or args.unfused)
    if args.warmup < 3:
        log("warning: fewer than 3 warm-up steps")

    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    if args.configs is None:
        args.configs = "" if world > 1 else ",".join(ALL_WORKLOADS)
    if args.min_blocks < 1 or args.max_blocks < args.min_blocks:
        raise SystemExit("need 1 <= --min-blocks <= --max-blocks")
    from paper_2603_12707_gb300 import workloads as wl

    if args.impl == "reference":
        if rank != 0:
            return
        cfg = wl.CONFIGS[args.config]
        # each step: one layer of the workload through the float64 oracle
        import torch
        import oracle
        lens = [int(n) + 1 for n in wl.context_lengths(cfg)]
        k = torch.cat([wl.kv_block(cfg, 0, b, n, "k", "cpu") for b, n in enumerate(lens)])
        v = torch.cat([wl.kv_block(cfg, 0, b, n, "v", "cpu") for b, n in enumerate(lens)])
        q = wl.step_inputs(cfg, 0, 0, "cpu")[0]
        for _ in range(args.warmup):
            oracle.decode_attention(q, lens, k, v)
        t0 = time.perf_counter()
        for _ in range(args.steps):
            oracle.decode_attention(q, lens, k, v)
        dt = time.perf_counter() - t0
        attn, _ = layer_bytes(cfg, lens)
        val = attn * args.steps / dt / 1e9
        threads = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
        sample = (f"per step: 1 of {cfg.num_layers} layers ({cfg.batch} sequences x {cfg.num_q_heads} heads) "
                  f"of the {cfg.name} workload")
        print(json.dumps({
            "impl": "reference", "metric": METRIC, "value": round(val, 4), "unit": "GB/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(dt / args.steps * 1e3, 3), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": describe(cfg),
            "cpu_baseline": {"value": round(val, 4), "unit": "GB/s", "cores": threads, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": round(val, 4), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }))
        return

    import torch
    if world > 1:
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0))))
    if args.varlen_write:
        varlen_main(args, rank, world)
        return
    from paper_2603_12707_gb300 import _build
    if rank == 0:
        _build.build_library()
    if world > 1:
        torch.distributed.barrier()
    head_cfg = workload_config(args)
    r = run_gpu(args, rank, world, head_cfg)
    out = summarize(args, world, r)
    out.update({"metric": METRIC, "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
                "data": "synthetic"})
    # every other workload, measured in the same run with the same steps and
    # warm-up (each in its own cache, freed before the next one is set up)
    extra = [c for c in args.configs.split(",") if c and c != head_cfg.name] if args.configs else []
    if extra:
        out["configs"] = {}
        for name in extra:
            ns = argparse.Namespace(**{**vars(args), "config": name, "phys_layers": 0, "page_order": None})
            rc = run_gpu(ns, rank, world, workload_config(ns))
            out["configs"][name] = summarize(ns, world, rc)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        nbytes, secs, desc, threads = oracle_sample(head_cfg, args.cpu_budget_s)
        out["cpu_baseline"] = {"value": round(nbytes / secs / 1e9, 4), "unit": "GB/s", "cores": threads,
                               "kind": "oracle", "sample": desc}
    if world > 1:
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()
    if rank == 0:
        print(json.dumps(out))


def summarize(args, world, r):
    """The bench line's measurement keys for one workload's run: the median
    timed block (K steps) for value / ms_per_step / steps/s and the roofline
    object, the clock record of the whole timed region, the end-to-end leg."""
    import torch
    from paper_2603_12707_gb300 import workloads as wl
    cfg, L = r["cfg"], r["L"]
    blocks = r["blocks"]
    mid = blocks[median_block([b["ms"] for b in blocks])]
    ms = mid["ms"]
    gbs = whole_job_gbs(sum(mid["step_bytes"]), ms, world)
    attn_ms = statistics.mean(mid["attn_ms"])
    attn_bytes = statistics.mean(mid["attn_bytes"])
    peak, peak_kind = measured_peaks()
    achieved = attn_bytes / (attn_ms / 1e3) / 1e9
    # the committed captures were taken with each workload's own page order
    default_order = args.page_order in (None, wl.CONFIGS[args.config].page_order)
    traffic = (committed_traffic(KERNEL_SOURCES, cfg.name, attn_bytes)
               if not args.unfused and default_order else None)
    step_ms = [x for b in blocks for x in b["step_ms"]]
    all_ms = sum(b["ms"] for b in blocks)
    all_bytes = sum(sum(b["step_bytes"]) for b in blocks)
    small = sum(mid["step_bytes"]) / args.steps < 2 * 129e6
    out = {
        "value": round(gbs, 2), "unit": "GB/s", "ms_per_step": round(ms / args.steps, 4),
        "config": {**describe(cfg),
                   "l2": ("each step streams the whole cache (far larger than the 129 MB L2)" if not small
                          else "a step's cache fits in the 129 MB L2: launch-bound, not a roofline number"),
                   "split_pages": args.split_pages or "auto",
                   "step_driver": "cuda_graph" if args.graph else "host",
                   "parallelism": f"replicas x{world}"},
        "steps_per_s": round(args.steps / (ms / 1e3), 3),
        "timed_blocks": len(blocks),
        # every step appends a token, so the blocks attend longer contexts as the
        # run goes on: the median block's workload, for reading the numbers above
        "median_block_context": {"mean_attended_tokens": round(statistics.mean(mid["attended"]), 1),
                                 "kv_gb_per_step": round(statistics.mean(mid["kv_bytes"]) / 1e9, 4),
                                 "tokens_appended_before_it": int(round(statistics.mean(mid["attended"])
                                                                        - r["start_attended"]))},
        "block_statistic": f"median of {len(blocks)} consecutive timed blocks of {args.steps} steps each "
                           "(contexts grow by one token per step across the blocks)",
        "block_ms": [round(b["ms"], 4) for b in blocks],
        "all_blocks_gbs": round(whole_job_gbs(all_bytes, all_ms, world), 2),
        "step_ms_median": round(statistics.median(step_ms), 4),
        "step_ms_min": round(min(step_ms), 4),
        "pct_of_measured_hbm": round(100 * gbs / world / peak, 2),
        "pct_of_nominal_8tbs": round(100 * gbs / world / NOMINAL_HBM_GBS, 2),
        "roofline": {"bound": "hbm", "kernel": "decode_attention" if args.unfused else "decode_attention_append",
                     "achieved": round(achieved, 2),
                     "peak": peak, "peak_kind": peak_kind, "unit": "GB/s", "frac": round(achieved / peak, 4),
                     "traffic": traffic,
                     "algorithmic_bytes_per_launch": int(attn_bytes), "avg_launch_ms": round(attn_ms, 4)},
        "clocks": r["clocks"],
        "gpu_launches": r["launches"],
        "step_kernels": ("kv_begin_step" + ("_device (CUDA-graph replay)" if args.graph else "") + " + per layer "
                         + ("kv_append, decode_attention" if args.unfused else "decode_attention_append (fused, PDL)")),
    }
    if r["e2e"]:
        e = r["e2e"]
        e_ms = reduce_max(torch, e["ms"], world)
        out["e2e"] = {"value": round(e["bytes"] * world / (e_ms / 1e3) / 1e9, 2), "unit": "GB/s",
                      "h2d_bytes_per_step": e["h2d"], "d2h_bytes_per_step": e["d2h"],
                      "steps_per_s": round(args.steps / (e_ms / 1e3), 3)}
    return out


if __name__ == "__main__":
    main()
