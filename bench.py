#!/usr/bin/env python3
"""Throughput of the GF(2) encoder-learning hot path on GB300.

Default workload (one "step"): learn the joint-Blackwell-scale synthetic
store -- 77,926 contexts, n log-normal (median 64) in [16, 256], ~80M
observations with 85% duplicates and 49,566 two-variant-stream contexts --
from scratch (reset + f2_learn_batched), solve every affine map
(f2_solve_affine), then encode 10M Zipf(1.1) queries with the span check
(f2_encode_batched).  Inputs are resident in HBM when the timed region starts
and are larger than L2 (2+ GB), so no L2 flush is needed.

Prints one JSON line.  ``value`` = observations eliminated per second over
the whole step; the encode throughput and per-phase times are reported
beside it.  ``--impl reference`` times the plain CPU oracle on the host
cores on a bounded sample of the same workload.

Other workloads: ``--config 1|2|5`` (learn + solve, plus encode for 1).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "GF(2) rows eliminated/sec and words encoded/sec at 1 GB300; % HBM/INT roofline"
HBM_FALLBACK_GBS = 6800.0
SMS = 152
INT_LANES_PER_SM = 64      # 32-bit logic lanes per SM per clock (4 SMSPs x 16)
SMEM_BYTES_PER_CLK = 128   # shared-memory bandwidth per SM per clock (32 banks x 4 bytes)
SM_MAX_MHZ_FALLBACK = 2070.0


# ----------------------------------------------------------------- helpers

def measured_peaks() -> dict:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": float(d["hbm_gbs"]), "sm_max_mhz": float(d.get("sm_max_mhz", SM_MAX_MHZ_FALLBACK)),
                "source": "measured (MEASURED_PEAKS.json)"}
    return {"hbm_gbs": HBM_FALLBACK_GBS, "sm_max_mhz": SM_MAX_MHZ_FALLBACK, "source": "fallback"}


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.samples = []
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-i",
                 str(gpu_index), "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None
            return
        self.t = threading.Thread(target=self._read, daemon=True)
        self.t.start()

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 9:
                self.samples.append((time.time(), parts))

    def stop(self, t0: float, t1: float) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        inside = [p for t, p in self.samples if t0 <= t <= t1]
        if not inside and self.samples:  # region shorter than the sampling period: nearest samples
            inside = [p for t, p in sorted(self.samples, key=lambda s: abs(s[0] - (t0 + t1) / 2))[:2]]
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}

        def num(v):
            try:
                return float(v)
            except ValueError:
                return None

        mhz = [num(p[1]) for p in inside if num(p[1]) is not None]
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for p in inside:
            for name, v in zip(names, p[5:9]):
                if v.strip().lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(mhz) if mhz else None, "sm_max_mhz": num(inside[0][2]),
                "power_w_max": max((num(p[3]) or 0.0) for p in inside), "reasons": sorted(reasons),
                "samples": len(inside)}


class NvmlSampler:
    """SM clock, power and clock-event reasons read through NVML (read-only
    queries, ctypes) every few milliseconds while the timed region runs, so
    that a region of a few tens of milliseconds still holds several samples.
    Falls back to ClockSampler (nvidia-smi) where NVML cannot be loaded."""

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown",
               0x80: "hw_power_brake_slowdown"}

    def __init__(self, device_index: int, period_s: float = 0.005):
        import ctypes

        self.samples = []
        self.ok = False
        try:
            lib = ctypes.CDLL("libnvidia-ml.so.1")
            if lib.nvmlInit_v2() != 0:
                return
            h = ctypes.c_void_p()
            bus = None
            try:
                import torch

                pr = torch.cuda.get_device_properties(device_index)
                bus = f"{pr.pci_domain_id:08x}:{pr.pci_bus_id:02x}:{pr.pci_device_id:02x}.0".encode()
            except Exception:
                bus = None
            rc = lib.nvmlDeviceGetHandleByPciBusId_v2(bus, ctypes.byref(h)) if bus else 1
            if rc != 0 and lib.nvmlDeviceGetHandleByIndex_v2(device_index, ctypes.byref(h)) != 0:
                return
            self.lib, self.h, self.ct = lib, h, ctypes
            self.reasons_fn = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or getattr(
                lib, "nvmlDeviceGetCurrentClocksThrottleReasons")
            mx = ctypes.c_uint(0)
            lib.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx))  # NVML_CLOCK_SM
            self.max_mhz = float(mx.value) or None
        except (OSError, AttributeError):
            return
        self.ok = True
        self.period = period_s
        self.stop_flag = False
        self.t = threading.Thread(target=self._run, daemon=True)
        self.t.start()

    def _run(self):
        ct, lib, h = self.ct, self.lib, self.h
        clk, pw, rs = ct.c_uint(0), ct.c_uint(0), ct.c_ulonglong(0)
        while not self.stop_flag:
            lib.nvmlDeviceGetClockInfo(h, 1, ct.byref(clk))
            lib.nvmlDeviceGetPowerUsage(h, ct.byref(pw))
            self.reasons_fn(h, ct.byref(rs))
            self.samples.append((time.time(), float(clk.value), pw.value / 1000.0, int(rs.value)))
            time.sleep(self.period)

    def stop(self, t0: float, t1: float) -> dict:
        self.stop_flag = True
        self.t.join(timeout=2)
        inside = [s for s in self.samples if t0 <= s[0] <= t1]
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": ["no samples"], "samples": 0,
                    "source": "nvml"}
        reasons = sorted({name for _, _, _, r in inside for bit, name in self.REASONS.items() if r & bit})
        return {"sm_mhz": statistics.median([c for _, c, _, _ in inside]), "sm_max_mhz": self.max_mhz,
                "power_w_max": max(p for _, _, p, _ in inside), "reasons": reasons, "samples": len(inside),
                "source": "nvml, 5 ms period"}


def clock_sampler(device_index: int):
    s = NvmlSampler(device_index)
    return s if s.ok else ClockSampler(device_index)


def cpu_model() -> str:
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform

    return platform.processor() or platform.machine()


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def reduce_across_ranks(value: float, op: str, device=None) -> float:
    """MAX or SUM of a per-rank number over all ranks (identity without a
    process group).  Ranks run independent problems, so this reduction of
    timings and unit counts is the only communication."""
    import torch
    import torch.distributed as dist

    if not (dist.is_available() and dist.is_initialized()):
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX if op == "max" else dist.ReduceOp.SUM)
    return float(t.item())


def workload_for(cfg_id: int, rank: int, query_count=None, num_ctx=None):
    from paper_2608_20532_gb300 import workloads as W

    if cfg_id == 6:  # parsed-value contexts with the paper's low exact-context ranks
        over = {"num_ctx": num_ctx} if num_ctx else {}
        return W.parsed_lowrank(seed=W.seed_for(6) + 1000 * rank, **over)
    cfg = dict(W.CONFIGS[cfg_id]) if not num_ctx else W.scaled(cfg_id, num_ctx)
    if num_ctx and query_count is None and cfg.get("queries", {}).get("count"):
        query_count = int(cfg["queries"]["count"] * num_ctx / W.CONFIGS[cfg_id]["num_ctx"])
    seed = W.seed_for(cfg_id) + 1000 * rank
    return W.generate(cfg, seed, name=f"config{cfg_id}", query_count=query_count)


def describe(cfg_id: int, wl) -> dict:
    scaled_note = "" if wl.num_ctx == {1: 256, 2: 4096, 3: 77926, 5: 64, 6: 10000}[cfg_id] else " [SCALED DOWN]"
    d = {"workload": scaled_note + {1: "config-1 parity case: 256 contexts, n=48, 260 rows each, 100 queries/context",
                      2: "4,096 contexts, n in [32,128], ~2.6M rows",
                      3: "joint-Blackwell-scale learn (77,926 contexts, ~80M rows, 85% duplicates) + 10M Zipf(1.1) encode queries",
                      5: "64 contexts, n=1024, 2^20 rows each in 16 incremental 65,536-row batches",
                      6: "parsed-value contexts: 10,000 contexts of k in [2,8] int64 values (n = 64k), exact-context "
                         "rank median 3 / p95 21, ~200 rows per rank (13.6M rows)"}[cfg_id],
         "contexts": wl.num_ctx, "rows": wl.total_rows, "n_median": float(np.median(wl.n_bits)),
         "queries": int(len(wl.queries.ctx_id)) if wl.queries is not None else 0,
         "input_bytes": int(wl.x.nbytes + wl.y.nbytes),
         "l2": "inputs larger than L2 (no flush)" if wl.x.nbytes + wl.y.nbytes >= 129e6 * 2
         else "L2 flushed between steps (256 MB write, outside the per-step events)"}
    return d


def algorithmic_bytes_learn(wl) -> int:
    """Packed x (ceil(n/8) bytes, constant implicit) + 16 bytes of y per row."""
    return int((wl.rows * ((wl.n_bits.astype(np.int64) + 7) // 8 + 16)).sum())


def algorithmic_bytes_encode(wl, basis_bytes_touched: int) -> int:
    q = wl.queries
    n = wl.n_bits.astype(np.int64)[q.ctx_id]
    return int((4 + (n + 7) // 8 + 16 + 1).sum()) + int(basis_bytes_touched)


def _popcount(t):
    t = t - ((t >> 1) & 0x55555555)
    t = (t & 0x33333333) + ((t >> 2) & 0x33333333)
    t = (t + (t >> 4)) & 0x0F0F0F0F
    return ((t * 0x01010101) & 0xFFFFFFFF) >> 24


def _q_words(xw_rows, g, dev):
    """[1 || x] words (int64 holding 32-bit values) of rows with g x-words."""
    import torch

    X = xw_rows & 0xFFFFFFFF
    Q = torch.zeros((X.shape[0], g + 1), dtype=torch.int64, device=dev)
    Q[:, :g] = (X << 1) & 0xFFFFFFFF
    Q[:, 1:] |= X >> 31
    Q[:, 0] |= 1
    return Q


def algorithmic_ops(wl, pivot_words, pw_off, dev, queries=False) -> int:
    """Sum over rows (or queries) of |q AND P| * (wd + 4): the 32-bit word
    XORs of step (1) against the final reduced basis."""
    import torch

    n = wl.n_bits.astype(np.int64)
    xw = (n + 31) // 32
    wd = (n + 1 + 31) // 32
    wdmax = int(wd.max())
    C = wl.num_ctx
    P = np.zeros((C, wdmax + 1), np.int64)
    for c_w in range(wdmax):
        has = wd > c_w
        P[has, c_w] = pivot_words[pw_off[:-1][has] + c_w].astype(np.int64) & 0xFFFFFFFF
    Pt = torch.from_numpy(P).to(dev)
    total = 0
    if queries:
        q = wl.queries
        ctx = torch.from_numpy(q.ctx_id.astype(np.int64)).to(dev)
        X = torch.from_numpy(q.x.view(np.int32).astype(np.int64)).to(dev)
        wd4 = torch.from_numpy(wd + 4).to(dev)
        for g in np.unique(xw):
            sel = torch.from_numpy(np.flatnonzero(xw[q.ctx_id] == g)).to(dev)
            if sel.numel() == 0:
                continue
            Q = _q_words(X[sel][:, :g], int(g), dev)
            cnt = _popcount(Q & Pt[ctx[sel]][:, :g + 1]).sum(dim=1)
            total += int((cnt * wd4[ctx[sel]]).sum())
        return total
    xs = torch.from_numpy(wl.x.view(np.int32).astype(np.int64)).to(dev)
    for g in np.unique(xw):
        cs = np.flatnonzero(xw == g)
        for chunk in np.array_split(cs, max(1, len(cs) // 8000)):
            rows = wl.rows[chunk]
            R = int(rows.sum())
            if R == 0:
                continue
            starts = np.repeat(wl.x_off[chunk], rows) + (np.arange(R) - np.repeat(np.cumsum(rows) - rows, rows)) * g
            idx = torch.from_numpy(starts).to(dev)[:, None] + torch.arange(int(g), device=dev)[None, :]
            Q = _q_words(xs[idx], int(g), dev)
            ctx = torch.from_numpy(np.repeat(chunk, rows)).to(dev)
            cnt = _popcount(Q & Pt[ctx][:, :g + 1]).sum(dim=1)
            total += int((cnt * torch.from_numpy(wd + 4).to(dev)[ctx]).sum())
    return total


# --------------------------------------------------------------- our arm

def run_ours(args):
    import torch

    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    import __graft_entry__

    if rank == 0:
        __graft_entry__.build()
    if world > 1:
        torch.distributed.barrier()
    from paper_2608_20532_gb300 import binding

    binding.load_library()
    cfg_id = args.config
    wl = workload_for(cfg_id, rank, num_ctx=args.ctx)
    t = lambda a: binding.to_device(a, dev)
    x_t, y_t = t(wl.x), t(wl.y)
    batches = [(t(ro), t(xo)) for ro, xo in wl.batches]
    has_q = wl.queries is not None
    if has_q:
        ctx_t, qx_t = t(wl.queries.ctx_id), t(wl.queries.x)
        Q = int(ctx_t.numel())
        y_out = torch.empty((Q, 4), dtype=torch.int32, device=dev)
        span = torch.empty(Q, dtype=torch.uint8, device=dev)
    store = binding.Store(wl.n_bits, device=dev)
    W_out = torch.empty((int(store.slot_off[-1]), 4), dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()
    nev = 4

    def step(evs=None):
        if evs is not None:
            evs[0].record(stream)
        store.reset()
        for ro, xo in batches:
            store.learn(ro, x_t, xo, y_t)
        if evs is not None:
            evs[1].record(stream)
        store.solve(out=W_out)
        if evs is not None:
            evs[2].record(stream)
        if has_q:
            store.encode(ctx_t, qx_t, y_out, span)
        if evs is not None:
            evs[3].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    status = store.device_status()
    if status != 0:
        raise RuntimeError(f"device status {status} after warm-up")

    # --graph: each phase of the step (reset + learn, solve, encode) captured
    # once as a CUDA graph and replayed every step -- the same kernels and
    # work, without the host launch overhead of the small configurations.
    # The calls allocate nothing after the warm-up and never synchronize, so
    # they capture; if capture fails the step runs eagerly (said on the line).
    graphs, launch_mode = None, "eager launches"
    if args.graph:
        try:
            def learn_phase():
                store.reset()
                for ro, xo in batches:
                    store.learn(ro, x_t, xo, y_t)

            parts = [learn_phase, lambda: store.solve(out=W_out)]
            if has_q:
                parts.append(lambda: store.encode(ctx_t, qx_t, y_out, span))
            graphs = []
            for fn in parts:
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, capture_error_mode="thread_local"):
                    fn()
                graphs.append(g)
            for g in graphs:  # one replay of each before timing
                g.replay()
            torch.cuda.synchronize()
            if store.device_status() != 0:
                raise RuntimeError("device status after graph replay")
            launch_mode = "CUDA graphs (one per phase), replayed"
        except Exception as exc:  # noqa: BLE001 - reported on the line
            graphs, launch_mode = None, f"eager launches (graph capture failed: {exc})"
            torch.cuda.synchronize()

    def step_graph(evs):
        evs[0].record(stream)
        graphs[0].replay()
        evs[1].record(stream)
        graphs[1].replay()
        evs[2].record(stream)
        if has_q:
            graphs[2].replay()
        evs[3].record(stream)

    K = args.steps
    # inputs smaller than L2 are timed with an L2 flush (a 256 MB write)
    # between steps, outside the per-step event pairs
    flush = None
    if wl.x.nbytes + wl.y.nbytes < 129e6 * 2:
        flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    events = [[torch.cuda.Event(enable_timing=True) for _ in range(nev)] for _ in range(K)]
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    sampler = clock_sampler(local)
    time.sleep(0.3)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    t0 = time.time()
    start.record(stream)
    for k in range(K):
        if flush is not None:
            flush.zero_()
        if graphs is not None:
            step_graph(events[k])
        else:
            step(events[k])
    end.record(stream)
    torch.cuda.synchronize()
    t1 = time.time()
    if world > 1:
        torch.distributed.barrier()
    clocks = sampler.stop(t0, t1)
    total_ms = start.elapsed_time(end)
    if flush is not None:
        total_ms = sum(e[0].elapsed_time(e[3]) for e in events)
    learn_ms = [e[0].elapsed_time(e[1]) for e in events]
    solve_ms = [e[1].elapsed_time(e[2]) for e in events]
    enc_ms = [e[2].elapsed_time(e[3]) for e in events]
    each_ms = [e[0].elapsed_time(e[3]) for e in events]  # one step, bracketed by its own events
    total_ms = reduce_across_ranks(total_ms, "max", dev)
    ms_step = total_ms / K

    # results (for accounting) and a sanity check of the final state
    b = store.basis()
    torch.cuda.synchronize()
    pivots = binding.to_numpy(b["pivot_mask"]).view(np.uint32)
    contra = int(binding.to_numpy(b["contra"]).sum())
    rows_total = reduce_across_ranks(wl.total_rows, "sum", dev)
    value = rows_total / (ms_step / 1e3)

    # ---- full-rank verification (config 5 after saturation): one more
    # incremental call on the saturated store, timed alone -- every row is a
    # check y = T(phi(x)) by verify_full_kernel (ceil(d/4) 16-byte lookups a
    # row from a table in shared memory; the plan kernels are the rest)
    verify = None
    if cfg_id == 5:
        ro1, xo1 = batches[1]
        v0 = torch.cuda.Event(enable_timing=True)
        v1 = torch.cuda.Event(enable_timing=True)
        store.learn(ro1, x_t, xo1, y_t)  # warm
        torch.cuda.synchronize()
        v0.record(stream)
        for _ in range(K):
            store.learn(ro1, x_t, xo1, y_t)
        v1.record(stream)
        torch.cuda.synchronize()
        v_ms = v0.elapsed_time(v1) / K
        rows1 = int(wl.batches[1][0][-1] - wl.batches[1][0][0])
        d = int(wl.n_bits.max()) + 1
        lookups = rows1 * ((d + 3) // 4)
        smem_bytes = lookups * 16
        verify = {"ms_per_call": v_ms, "rows_per_call": rows1, "rows_per_s": rows1 / (v_ms / 1e3),
                  "lookups_per_row": (d + 3) // 4, "smem_bytes_per_call": smem_bytes,
                  "kernel": "verify_full_kernel (+ plan kernels), one incremental call on full-rank contexts"}

    # ---- encode epilogue (Appendix C/D): scheduler control merged at bit 105,
    # opaque-mask bits restored from recorded state; timed on its own, after
    # the step, on the step's encoded words (seeded synthetic control/state)
    epilogue = None
    if has_q:
        g = torch.Generator(device=dev)
        g.manual_seed(20260004)
        Qn = int(ctx_t.numel())
        sched_t = torch.randint(0, 1 << 17, (Qn,), dtype=torch.int32, device=dev, generator=g)
        state_t = torch.randint(-(1 << 31), (1 << 31) - 1, (Qn, 4), dtype=torch.int32, device=dev, generator=g)
        mask_t = torch.zeros((wl.num_ctx, 4), dtype=torch.int32, device=dev)
        mask_t[::7, 3] = (1 << (122 - 96)) | (1 << (124 - 96))  # the Appendix D bits in some contexts
        y_epi = y_out.clone()
        for _ in range(3):
            store.encode_epilogue(ctx_t, span, y_epi, sched=sched_t, state=state_t, opaque_mask=mask_t)
        torch.cuda.synchronize()
        p0 = torch.cuda.Event(enable_timing=True)
        p1 = torch.cuda.Event(enable_timing=True)
        p0.record(stream)
        for _ in range(K):
            store.encode_epilogue(ctx_t, span, y_epi, sched=sched_t, state=state_t, opaque_mask=mask_t)
        p1.record(stream)
        torch.cuda.synchronize()
        e_ms = p0.elapsed_time(p1) / K
        # y read + written, control word, recorded state, in-span flag, context id
        ebytes = Qn * (16 + 16 + 4 + 16 + 1 + 4) + 16 * wl.num_ctx
        epilogue = {"ms": e_ms, "bytes_per_call": ebytes, "achieved_gbs": ebytes / (e_ms / 1e3) / 1e9,
                    "kernel": "epilogue_kernel (f2_encode_epilogue)"}
        del y_epi, state_t, sched_t

    # ---- map pooling (Sec. 3): the exact contexts of each (f, m) group of the
    # parsed-value workload merged into one store; the call synchronizes, so
    # it is timed on the host clock, after the step
    pooling = None
    gs = int(wl.params.get("group_size", 0) or 0)
    if gs > 0:
        group_of = (np.arange(wl.num_ctx) // gs).astype(np.int32)
        G = int(group_of[-1]) + 1
        for _ in range(2):
            store.merge(group_of, G)[0].close()
        torch.cuda.synchronize()
        t_m = time.perf_counter()
        for _ in range(K):
            merged, _ok = store.merge(group_of, G)
            if _ < K - 1:
                merged.close()
        m_ms = (time.perf_counter() - t_m) * 1e3 / K
        mb = merged.basis()
        torch.cuda.synchronize()
        pooling = {"ms": m_ms, "groups": G, "group_size": gs,
                   "merged_rows": int(binding.to_numpy(b["rank"]).astype(np.int64).sum()),
                   "shared_maps": int((binding.to_numpy(mb["contra"]) == 0).sum()),
                   "call": "f2_merge_bases (merge_gather_kernel + learn kernels; host clock)"}
        merged.close()

    # ---- e2e through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        pin = lambda a: torch.from_numpy(np.ascontiguousarray(a.view(np.int32) if a.dtype == np.uint32 else a)).pin_memory()
        hx, hy = pin(wl.x), pin(wl.y)
        hb = [(pin(ro), pin(xo)) for ro, xo in wl.batches]
        h_in = [hx, hy] + [a for pair in hb for a in pair]
        d_in = [x_t, y_t] + [a for pair in batches for a in pair]
        if has_q:
            h_in += [pin(wl.queries.ctx_id), pin(wl.queries.x)]
            d_in += [ctx_t, qx_t]
        outs = {k: v for k, v in store.basis().items()}
        outs["W"] = W_out
        if has_q:
            outs["y"] = y_out
            outs["span"] = span
        h_out = {k: torch.empty(v.shape, dtype=v.dtype, pin_memory=True) for k, v in outs.items()}
        bi = sum(h.numel() * h.element_size() for h in h_in)
        bo = sum(h.numel() * h.element_size() for h in h_out.values())

        side = torch.cuda.Stream(device=dev)
        basis_ready = torch.cuda.Event()
        outs_done = torch.cuda.Event()

        def e2e_step():
            # learn and encode straight from pinned host memory (the library
            # overlaps the chunked copies with its kernels); the basis and the
            # map go to the host on a side stream while the queries are encoded
            store.reset()
            for hro, hxo in hb:
                store.learn_host(hro, hx, hxo, hy)
            store.solve(out=W_out)
            bb = store.basis()
            basis_ready.record(stream)
            side.wait_event(basis_ready)
            with torch.cuda.stream(side):
                for k in ("rank", "pivot_mask", "basis_x", "basis_z", "contra", "first_contra", "n_contra",
                          "rows_seen"):
                    h_out[k].copy_(bb[k], non_blocking=True)
                h_out["W"].copy_(W_out, non_blocking=True)
                outs_done.record(side)
            if has_q:
                store.encode_host(h_in[-2], h_in[-1], h_out["y"], h_out["span"])
            stream.wait_event(outs_done)

        Ke = max(1, min(K, args.e2e_steps))
        for _ in range(min(2, args.warmup)):
            e2e_step()
        torch.cuda.synchronize()
        # an event between steps: the per-step times, their mean and median
        # (the host link is shared on the box: a step now and then stalls for
        # tens of ms outside this process, and the median is the steady rate)
        sev = [torch.cuda.Event(enable_timing=True) for _ in range(Ke + 1)]
        sev[0].record(stream)
        for k in range(Ke):
            e2e_step()
            sev[k + 1].record(stream)
        torch.cuda.synchronize()
        per = [sev[k].elapsed_time(sev[k + 1]) for k in range(Ke)]
        e_mean = reduce_across_ranks(sum(per) / Ke, "max", dev)
        e_ms = reduce_across_ranks(float(np.median(per)), "max", dev)
        e2e = {"value": rows_total / (e_ms / 1e3), "unit": "rows/s", "ms_per_step": e_ms, "steps": Ke,
               "timing": "median of the per-step event times", "mean_ms_per_step": e_mean,
               "per_step_ms": [round(v, 3) for v in per],
               "h2d_bytes_per_step": int(bi), "d2h_bytes_per_step": int(bo),
               "path": "f2_learn_host + f2_solve_affine + f2_encode_host from pinned host memory; basis and map "
                       "copied out on a side stream during the encode"}

    if rank != 0:
        if world > 1:
            torch.distributed.destroy_process_group()
        return

    peaks = measured_peaks()
    # ALU peak: derived from unit counts and the max clock; the probe checks it
    alu_peak = SMS * INT_LANES_PER_SM * peaks["sm_max_mhz"] * 1e6
    probe = None
    if not args.no_probe:
        out = torch.zeros(4096, dtype=torch.int32, device=dev)
        iters = 4096
        blocks = SMS * 8
        binding.peak_lop3(blocks, 64, out)
        torch.cuda.synchronize()
        p0 = torch.cuda.Event(enable_timing=True)
        p1 = torch.cuda.Event(enable_timing=True)
        p0.record(stream)
        nops = binding.peak_lop3(blocks, iters, out)
        p1.record(stream)
        torch.cuda.synchronize()
        probe = nops / (p0.elapsed_time(p1) / 1e3)

    learn_mean = statistics.mean(learn_ms) / 1e3
    bytes_learn = algorithmic_bytes_learn(wl)
    ops_learn = algorithmic_ops(wl, pivots, store.pw_off, dev)
    hbm_peak = peaks["hbm_gbs"] * 1e9
    # The learn pass eliminates only the first occurrence of each distinct row
    # (exact dedup), so its arithmetic is a fraction of ops_learn (which counts
    # every row reduced) and reading the input once is the binding floor: the
    # learn roofline is HBM.  ops_learn is kept as the naive-method reference.
    learn_bound = "hbm"
    rl_learn = {
        "kernel": "f2_learn_batched (fill, plan kernels, dedup_kernel, elim_narrow_kernel<true/false>, "
                  "elim_wide_kernel, verify_full_kernel)",
        "hbm": {"achieved": bytes_learn / learn_mean / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": (bytes_learn / learn_mean) / hbm_peak, "bytes_per_launch": bytes_learn},
        # The naive method's word-XOR count (every row reduced against the
        # final basis, one pivot row at a time) per second of the learn: a
        # reference rate, not a fraction of work done -- the library does not
        # reduce duplicates, and checks the rows of full-rank contexts with
        # 4-bit tables (about d/4 lookups a row), so it can exceed the peak.
        "naive_alu_reference": {"ops_per_launch": ops_learn, "naive_ops_per_s": ops_learn / learn_mean,
                                "alu_peak_ops_per_s": alu_peak,
                                "peak_probe_lop3_ops_per_s": probe if probe else None},
    }
    traffic = profile_traffic("f2_learn_batched")
    dom = rl_learn[learn_bound]
    roofline = {"bound": learn_bound, "achieved": dom["achieved"], "peak": dom["peak"], "unit": dom["unit"],
                "frac": dom["frac"], "traffic": traffic,
                "peak_source": peaks["source"] if learn_bound == "hbm" else
                "derived: 152 SMs x 64 INT32 lanes x max SM clock"}
    result = {
        "metric": METRIC, "value": value, "unit": "rows/s", "n_gpus": world, "steps": K, "warmup": args.warmup,
        "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "u32", "data": "synthetic (seeded planted affine maps)",
        "config": dict(describe(cfg_id, wl), parallelism=f"replicas x{world}" if world > 1 else "single GPU"),
        "launch": launch_mode,
        "phases_ms": {"learn": statistics.mean(learn_ms), "solve": statistics.mean(solve_ms),
                      "encode": statistics.mean(enc_ms)},
        "step_stats_ms": {"mean": statistics.mean(each_ms), "median": statistics.median(each_ms),
                          "best": min(each_ms),
                          "learn": {"median": statistics.median(learn_ms), "best": min(learn_ms)},
                          "encode": {"median": statistics.median(enc_ms), "best": min(enc_ms)}},
        "learn_rows_per_s": wl.total_rows / learn_mean,
        "roofline": roofline,
        "roofline_learn": rl_learn,
        "clocks": clocks,
        "gpu_launches": K * launches_per_step(wl, has_q),
        "contradiction_contexts": contra,
    }
    if has_q:
        enc_mean = statistics.mean(enc_ms) / 1e3
        span_np = binding.to_numpy(span)
        ops_enc = algorithmic_ops(wl, pivots, store.pw_off, dev, queries=True)
        bytes_enc = algorithmic_bytes_encode(wl, basis_bytes_touched(wl, store))
        result["encode_words_per_s"] = Q / enc_mean
        result["encode_in_span_frac"] = float((span_np == 1).mean())
        result["roofline_encode"] = {
            "kernel": ("f2_encode_batched (fill, enc_count, enc_table, enc_build, enc_scan, enc_scatter, "
                       "enc_runs, enc_short kernels; enc_direct alone for a pass of at most 65,536 queries)"),
            "hbm": {"achieved": bytes_enc / enc_mean / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                    "frac": bytes_enc / enc_mean / hbm_peak, "bytes_per_launch": bytes_enc},
            # per query the naive pivot walk's word XORs (|q AND P| x (wd + 4)):
            # a reference rate; long runs are encoded with 4-bit tables instead
            "naive_alu_reference": {"ops_per_launch": ops_enc, "naive_ops_per_s": ops_enc / enc_mean,
                                    "alu_peak_ops_per_s": alu_peak},
            "traffic": profile_traffic("f2_encode_batched"),
        }
    if verify is not None:
        # the shared-memory pipe: 128 bytes a clock per SM (32 banks x 4 bytes)
        smem_peak = SMS * SMEM_BYTES_PER_CLK * peaks["sm_max_mhz"] * 1e6
        ach = verify["smem_bytes_per_call"] / (verify["ms_per_call"] / 1e3)
        result["roofline_verify"] = {
            "bound": "smem", "achieved": ach / 1e9, "peak": smem_peak / 1e9, "unit": "GB/s (shared memory)",
            "frac": ach / smem_peak, "peak_source": "derived: 152 SMs x 128 B/clock x max SM clock",
            "hbm_frac": (verify["rows_per_call"] * (16 + 4 * int(wl.n_bits.max() // 32)) /
                         (verify["ms_per_call"] / 1e3)) / (peaks["hbm_gbs"] * 1e9), **verify}
    if epilogue is not None:
        epilogue["frac_of_measured_hbm"] = epilogue["achieved_gbs"] / peaks["hbm_gbs"]
        result["encode_epilogue"] = epilogue
    if pooling is not None:
        result["map_pooling"] = pooling
    if e2e is not None:
        result["e2e"] = e2e
    if world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(wl, args.cpu_seconds)
    print(json.dumps(result), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def launches_per_step(wl, has_q: bool) -> int:
    """Kernels one step enqueues (the host logic of the library): the reset's
    fill; per learn call the fill of its counters, a plan (one kernel for at
    most 8,192 contexts, else three) and dedup_kernel (a second instance when
    some feature row has more than 9 words) for the duplicate pass, a plan,
    the elimination kernel of each width class present (d <= 96, 96 < d <=
    288, 288 < d <= 544, wider) and the full-rank check; solve_kernel; per
    2^25 queries the encode's fill and its seven kernels (count, table,
    build, scan, scatter, runs, short), or one kernel for a pass of at most
    65,536 queries."""
    wd = (wl.n_bits.astype(np.int64) + 1 + 31) // 32
    xw = (wl.n_bits.astype(np.int64) + 31) // 32
    plan = 1 if wl.num_ctx <= 8192 else 3
    elim = (int((wd <= 3).any()) + int(((wd > 3) & (wd <= 9)).any()) + int(((wd > 9) & (wd <= 17)).any())
            + int((wd > 17).any()))
    learn = 1 + plan + 1 + int((xw > 9).any()) + plan + elim + 1
    nq = len(wl.queries.ctx_id) if has_q else 0
    enc = (1 if nq <= 65536 else 8 * ((nq + (1 << 25) - 1) >> 25)) if has_q else 0
    return 1 + len(wl.batches) * learn + 1 + enc


def basis_bytes_touched(wl, store) -> int:
    """Basis bytes of the distinct contexts the queries name, each read once."""
    used = np.unique(wl.queries.ctx_id)
    d = wl.n_bits.astype(np.int64)[used] + 1
    wd = (d + 31) // 32
    return int((d * (16 + 4 * wd) + 4 * wd).sum())


# the translation units of each library call's kernels
KERNEL_SOURCES = {"f2_learn_batched": ("learn.cu", "f2_internal.cuh"),
                  "f2_encode_batched": ("encode.cu", "f2_internal.cuh")}


def kernel_source_hash(call: str) -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2608_20532_gb300", "csrc")
    for f in KERNEL_SOURCES[call]:
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def profile_traffic(call: str):
    """DRAM bytes per call from a committed ncu summary, if it was taken on
    the current sources of that call's kernels (null otherwise)."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(call)
    if not e or e.get("source_hash") != kernel_source_hash(call):
        return None
    return e.get("dram_bytes_per_launch")


# ------------------------------------------------------------ CPU oracle

def _sample(wl, target_rows: int, seed: int = 7):
    rng = np.random.default_rng(seed)
    perm = rng.permutation(wl.num_ctx)
    acc = np.cumsum(wl.rows[perm])
    k = int(np.searchsorted(acc, target_rows)) + 1
    return np.sort(perm[:max(1, min(k, wl.num_ctx))])


def _subset(wl, ctxs, qsel):
    """Compact copy of the rows (and queries) of the sampled contexts."""
    n = wl.n_bits[ctxs]
    W = (n.astype(np.int64) + 31) // 32
    batches, xs, ys = [], [], []
    xbase = ybase = 0
    for ro, xo in wl.batches:
        cnt = ro[ctxs + 1] - ro[ctxs]
        r_off = np.zeros(len(ctxs) + 1, np.int64)
        r_off[1:] = ybase + np.cumsum(cnt)
        r_off[0] = ybase
        x_off = xbase + np.concatenate([[0], np.cumsum(cnt * W)[:-1]])
        yi = np.concatenate([np.arange(ro[c], ro[c + 1]) for c in ctxs])
        xi = np.concatenate([np.arange(xo[c], xo[c] + k * w) for c, k, w in zip(ctxs, cnt, W)])
        ys.append(wl.y[yi])
        xs.append(wl.x[xi])
        batches.append((r_off, x_off))
        ybase += len(yi)
        xbase += len(xi)
    x = np.concatenate(xs)
    y = np.concatenate(ys)
    q = None
    if qsel is not None and len(qsel):
        remap = np.full(wl.num_ctx, -1, np.int32)
        remap[ctxs] = np.arange(len(ctxs), dtype=np.int32)
        q = (remap[wl.queries.ctx_id[qsel]], np.ascontiguousarray(wl.queries.x[qsel]))
    return n, batches, x, y, q


def _oracle_step(sub, threads):
    """One oracle step on a prepared subset: learn, solve, encode (timed)."""
    import oracle

    n, batches, x, y, q = sub
    t0 = time.perf_counter()
    O = oracle.Oracle(n, threads=threads)
    for ro, xo in batches:
        O.learn(ro, xo, x, y)
    O.solve()
    if q is not None:
        O.encode(q[0], q[1])
    t = time.perf_counter() - t0
    O.close()
    return t


def _queries_for(wl, ctxs, frac):
    if wl.queries is None:
        return None
    ins = np.flatnonzero(np.isin(wl.queries.ctx_id, ctxs))
    return ins[: int(len(wl.queries.ctx_id) * frac)]


def cpu_baseline(wl, seconds: float) -> dict:
    """The oracle as it stands, on the host cores, on a bounded sample."""
    threads = os.cpu_count() or 1
    probe = _sample(wl, 300_000, seed=1)
    t = _oracle_step(_subset(wl, probe, None), threads)
    rate = wl.rows[probe].sum() / max(t, 1e-6)
    target = int(min(wl.total_rows, max(100_000, rate * seconds)))
    ctxs = _sample(wl, target, seed=2)
    frac = wl.rows[ctxs].sum() / wl.total_rows
    qsel = _queries_for(wl, ctxs, frac)
    t = _oracle_step(_subset(wl, ctxs, qsel), threads)
    rows = int(wl.rows[ctxs].sum())
    # one thread, on a sample a sixth the size (a few seconds)
    ctx1 = _sample(wl, max(20_000, target // 6), seed=4)
    frac1 = wl.rows[ctx1].sum() / wl.total_rows
    t1 = _oracle_step(_subset(wl, ctx1, _queries_for(wl, ctx1, frac1)), 1)
    rows1 = int(wl.rows[ctx1].sum())
    return {"value": rows / t, "unit": "rows/s", "cores": threads, "kind": "oracle", "cpu_model": cpu_model(),
            "sample": f"{len(ctxs)} of {wl.num_ctx} contexts ({rows} rows, {0 if qsel is None else len(qsel)} "
                      f"queries, {100 * frac:.1f}% of the step), learn + solve + encode, {t:.1f} s",
            "single_thread": {"value": rows1 / t1, "unit": "rows/s", "cores": 1,
                              "sample": f"{len(ctx1)} contexts ({rows1} rows), {t1:.1f} s"}}


def _phase_summary(T, wl, b, e, smcol, ctx_ids):
    has = T[:, e] > 0
    if not has.any():
        return None
    beg, end, sm = T[has, b].astype(np.int64), T[has, e].astype(np.int64), T[has, smcol].astype(np.int64)
    ids = ctx_ids[has]
    t0 = int(beg.min())
    span = int(end.max()) - t0
    last = np.array([end[sm == k].max() - t0 for k in np.unique(sm)])
    dur = end - beg
    top = np.argsort(-dur)[:8]
    return {
        "contexts": int(has.sum()), "span_us": span / 1e3, "sms": int(len(last)),
        "sm_finish_us": {"min": float(last.min()) / 1e3, "median": float(np.median(last)) / 1e3,
                         "p90": float(np.percentile(last, 90)) / 1e3, "max": float(last.max()) / 1e3},
        "tail_past_median_sm_frac": float((span - np.median(last)) / span),
        "longest": [{"ctx": int(ids[k]), "rows": int(wl.rows[ids[k]]), "n": int(wl.n_bits[ids[k]]),
                     "us": float(dur[k]) / 1e3, "start_us": float(beg[k] - t0) / 1e3,
                     "end_us": float(end[k] - t0) / 1e3} for k in top],
        "context_us_total": float(dur.sum()) / 1e3,
    }


def run_timing(args):
    """Diagnostic (not the bench line): per-context timestamps of one learn
    call (F2_OPT_TIMING) summarised per pass: how long the last context runs
    past the median SM's last context, and the longest contexts."""
    import torch
    import __graft_entry__

    __graft_entry__.build()
    from paper_2608_20532_gb300 import binding

    dev = torch.device("cuda", 0)
    wl = workload_for(args.config, 0, num_ctx=args.ctx)
    t = lambda a: binding.to_device(a, dev)
    x_t, y_t = t(wl.x), t(wl.y)
    batches = [(t(ro), t(xo)) for ro, xo in wl.batches]
    store = binding.Store(wl.n_bits, device=dev)
    store.set_option(binding.F2_OPT_TIMING, 1)
    for _ in range(args.warmup):
        store.reset()
        for ro, xo in batches:
            store.learn(ro, x_t, xo, y_t)
    torch.cuda.synchronize()
    store.reset()
    for ro, xo in batches[:-1]:
        store.learn(ro, x_t, xo, y_t)
    ro, xo = batches[-1]
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    ev[0].record()
    store.learn(ro, x_t, xo, y_t)
    ev[1].record()
    torch.cuda.synchronize()
    T = store.learn_timing()
    ids = np.arange(wl.num_ctx)
    out = {"config": describe(args.config, wl), "learn_call_ms": ev[0].elapsed_time(ev[1]),
           "dedup": _phase_summary(T, wl, 0, 1, 4, ids), "elimination": _phase_summary(T, wl, 2, 3, 5, ids)}
    if out["dedup"] and out["elimination"]:
        out["dedup_end_to_elim_start_us"] = (int(T[T[:, 2] > 0, 2].min()) - int(T[T[:, 1] > 0, 1].max())) / 1e3
    print(json.dumps(out), flush=True)


def run_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return
    import oracle

    oracle.build()
    wl = workload_for(args.config, 0, num_ctx=args.ctx)
    threads = os.cpu_count() or 1
    ctxs = _sample(wl, args.ref_rows, seed=3)
    frac = wl.rows[ctxs].sum() / wl.total_rows
    qsel = _queries_for(wl, ctxs, frac)
    sub = _subset(wl, ctxs, qsel)
    for _ in range(args.warmup):
        _oracle_step(sub, threads)
    times = [_oracle_step(sub, threads) for _ in range(args.steps)]
    rows = int(wl.rows[ctxs].sum())
    ms = 1e3 * statistics.mean(times)
    value = rows / (ms / 1e3)
    sample = (f"{len(ctxs)} of {wl.num_ctx} contexts ({rows} rows, {0 if qsel is None else len(qsel)} queries, "
              f"{100 * frac:.1f}% of the step) per step")
    out = {"impl": "reference", "metric": METRIC, "value": value, "unit": "rows/s", "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "u64", "data": "synthetic (seeded planted affine maps)",
           "config": dict(describe(args.config, wl),
                         parallelism=f"replicas x{world}" if world > 1 else "single GPU"),
           "cpu_baseline": {"value": value, "unit": "rows/s", "cores": threads, "kind": "oracle", "sample": sample,
                            "cpu_model": cpu_model()},
           "e2e": {"value": value, "unit": "rows/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", type=int, choices=[1, 2, 3, 5, 6], default=3)
    ap.add_argument("--ctx", type=int, default=0,
                    help="scaled-down workload with this many contexts (profiling); 0 = full size")
    ap.add_argument("--e2e-steps", type=int, default=7)
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--ref-rows", type=int, default=4_000_000)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-probe", action="store_true")
    ap.add_argument("--graph", action="store_true",
                    help="replay each phase of the step as a captured CUDA graph (the small configurations are "
                         "launch-heavy); default: eager launches")
    ap.add_argument("--timing", action="store_true",
                    help="diagnostic: per-context timestamps of one learn call, summarised (not the bench line)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    if args.impl == "reference":
        run_reference(args)
    elif args.timing:
        run_timing(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
