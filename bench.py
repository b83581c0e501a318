"""Benchmark: forced-weight subset evaluation on GB300.

Headline workload: exact enumeration at measurement scale -- 168,192 rows in
five groups (d = 64,128,128,128,64), n = 24 keys, k = 6 (134,596 subsets per
row), logits Gumbel*tau + sink, V fp32.  One step runs the whole path on every
row: softmax, top-k kept set, dense and forced-weight outputs, gap and dropped
mass (fw_dense_and_topk_gap), the swap rule over all keys (fw_swap_refine) and
the exact best subset ES(k) (fw_best_subset).  Metric: rows/s (every row gets
its exact ES(k)); the subsets the search covers per second are reported beside
it as a derived figure, with the subsets its walk actually visits.

Also timed in the same run (reported under "sections"), one line per config:
  exact_toy       256 rows, n=20, k=5, d=64: the whole path
  adversarial     512 rows each of flat, near-duplicate and planted-tie rows
  long_rows       4,096 rows x 32,768 keys, d=128, three budgets: gap, swap, vote
  contour         ContourKV allocation + ragged compaction, 256 cells x 32,768 tokens;
                  the capped (enforced) allocation, the window score, decode appends
  mixed_profiles  168,192 ragged rows (n 1,024..16,384, GQA-4, bf16 V): gap + swap
  pool            ES_pool (Definition 2.2) at s = 4/8/16/32 on mixed-profile rows
  audit           the deployed selectors' es against ES_pool and top-mass (App. C)

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
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

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

import workloads  # noqa: E402

N_KEYS, K_SEL = 24, 6
SUBSETS_PER_ROW = math.comb(N_KEYS, K_SEL)
POOL_SCHED = ((4, 24), (8, 12), (16, 6), (32, 4))  # (s, E): the candidate-set schedule of App. B

# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum, ncu, one pass,
# cold caches per kernel) per unit of each line, from kernel-filtered captures
# of reduced cases of the same workloads (the commands are listed with the
# summaries under profiles/), scaled to a full launch by the units it
# processes; None where a kernel changed after its capture:
#   fw_best_subset  the headline path's kernels at --rows-scale 0.1, per row
#   long_gap        8 heads x 128 rows: per-row logit bytes of k_long_select_reg
#                   and k_long_pv_tma scaled to 4,096 rows, plus each head's
#                   value block once (8 x 8.4 MB), per row
#   group_vote      the same for k_vote_mass + k_vote_select + k_long_pv_tma
#   contour         64 cells: k_c_* of one allocation + k_compact, per kept row
#   compact         k_compact alone, per kept row
#   window_score    k_wscore, per key (it reads K twice)
#   mixed_gap       --mixed-rows-scale 0.1, one gap call per profile, per row
TRAFFIC_PER_UNIT = {
    # line: (bytes per unit, unit)
    "fw_best_subset": (40328.0, "row"),
    "long_gap": (282648.0, "row"),
    "group_vote": (280709.0, "row"),
    "contour": (1023.2, "kept row"),
    "compact": (830.1, "kept row"),
    "window_score": (519.4, "key"),
    "mixed_gap": (322689.0, "row"),
}


def read_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return dict(hbm_gbs=p.get("hbm_gbs", 6800.0), bf16=p.get("bf16_tflops", 1900.0),
                    bf16_sust=p.get("bf16_tflops_sustained", 1700.0), sm_max=p.get("sm_max_mhz", 2070.0),
                    source="measured")
    return dict(hbm_gbs=6800.0, bf16=1900.0, bf16_sust=1700.0, sm_max=2070.0, source="fallback")


def fp32_peak_tflops(device, sm_mhz):
    """FP32 FMA peak: SMs x 128 lanes x 2 flops x the SM clock sampled under load."""
    sms = torch.cuda.get_device_properties(device).multi_processor_count
    return sms * 128 * 2 * sm_mhz * 1e6 / 1e12, sms


def fp32_fma_measured(fw, device, iters=1 << 15, reps=3):
    """The fp32 FMA throughput of the library's probe kernel (16 independent
    chains per thread, 8 CTAs of 256 threads per SM), TFLOP/s: a check of the
    nominal peak above."""
    sms = torch.cuda.get_device_properties(device).multi_processor_count
    blocks = sms * 8
    out = torch.empty(blocks * 256, dtype=torch.float32, device=device)
    for _ in range(2):
        fw.fp32_fma_probe(blocks, iters, out)
    torch.cuda.synchronize()
    best = float("inf")
    for _ in range(reps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        fw.fp32_fma_probe(blocks, iters, out)
        e1.record()
        e1.synchronize()
        best = min(best, e0.elapsed_time(e1))
    return 2.0 * blocks * 256 * 16 * iters / (best * 1e-3) / 1e12


class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons during a region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.f = None

    def __enter__(self):
        try:
            self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if self.proc is None or self.f is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.f.flush()
        rows = []
        with open(self.f.name) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.f.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


class L2Flush:
    """Writes a buffer larger than L2 between timed iterations."""

    def __init__(self, device):
        self.buf = torch.empty(256 << 20, dtype=torch.uint8, device=device)

    def __call__(self):
        self.buf.fill_(1)


class Events:
    """CUDA events recorded on the current stream around calls, read later."""

    def __init__(self):
        self.ev = []

    def start(self):
        e = torch.cuda.Event(enable_timing=True)
        e.record()
        return e

    def stop(self, e0, tag=None):
        e1 = torch.cuda.Event(enable_timing=True)
        e1.record()
        self.ev.append((e0, e1, tag))

    def take(self):
        torch.cuda.synchronize()
        r = [(a.elapsed_time(b), t) for a, b, t in self.ev]
        self.ev = []
        return r


# ---------------------------------------------------------------- workloads

class EnumWorkload:
    """168,192 rows, n=24, k=6: the whole a1..a6 path per step."""

    def __init__(self, fw, seed, device, rows_scale=1.0, batches=None, E=N_KEYS):
        self.fw = fw
        self.batches = batches if batches is not None else workloads.exact_enum(
            seed=seed, rows_scale=rows_scale, backend="torch", device=device)
        self.rows = [fw.rows_from_batch(b, device) for b in self.batches]
        self.k2 = [torch.as_tensor(np.asarray(b.k)).to(device) if not isinstance(b.k, torch.Tensor) else b.k
                   for b in self.batches]
        self.k1 = [k[:, 0].contiguous() for k in self.k2]
        self.kmax = [int(k.max().item()) for k in self.k1]
        self.num_rows = sum(r.num_rows for r in self.rows)
        self.subsets = sum(r.num_rows * math.comb(int(b.n_host[0]), int(np.asarray(b.k if not isinstance(
            b.k, torch.Tensor) else b.k.cpu())[0, 0])) for r, b in zip(self.rows, self.batches))
        self.E = E
        self.ev = Events()
        self.last = None
        # one stream per group: the groups are independent, so one group's
        # kernels fill the SMs another group's launch tails leave idle
        self.streams = [torch.cuda.Stream() for _ in self.rows]

    def step(self, time_enum=False):
        fw = self.fw
        main = torch.cuda.current_stream()
        for st in self.streams:
            st.wait_stream(main)
        outs = []
        for st, rows, k2, k1, kmax in zip(self.streams, self.rows, self.k2, self.k1, self.kmax):
            with torch.cuda.stream(st):
                top = fw.dense_and_topk_gap(rows, k2, kept_bits=False)
                sw = fw.swap_refine(rows, k2, top, E=self.E, max_swaps=32)
                e0 = self.ev.start() if time_enum else None
                bs = fw.best_subset(rows, k1, k_max=kmax)
                if time_enum:
                    self.ev.stop(e0, rows.num_rows)
            outs.append((top, sw, bs))
        for st in self.streams:
            main.wait_stream(st)
        self.last = outs
        return outs

    def stats(self):
        """Work counters of the last step's fw_best_subset calls, summed."""
        tot = {}
        for rows, (_, _, bs) in zip(self.rows, self.last):
            for key, v in self.fw.best_subset_stats(rows, bs).items():
                tot[key] = tot.get(key, 0) + v
        return tot

    def gram_flops(self):
        """The prep kernel's Gram products per step: (n+1)(n+2)/2 dot products of
        length d per row (the n keys and g of the top-k set), 2 flops per FMA."""
        f = 0
        for r, b in zip(self.rows, self.batches):
            n = int(b.n_host[0])
            f += r.num_rows * 2 * b.d * (n + 1) * (n + 2) // 2
        return f


class EnumE2E:
    """The same step through the public API from pinned host buffers: inputs are
    copied to the device, results copied back, inside the timed region.  The
    five groups are pipelined: a copy stream uploads group g + 1 while group
    g computes on its own stream (each group's compute waits for its own
    upload; the uploads of a step wait for the previous step's compute)."""

    def __init__(self, wl: EnumWorkload):
        self.wl = wl
        self.host = []
        self.h2d = 0
        self.d2h = 0
        self.copy_stream = torch.cuda.Stream()
        self.upload_ev = []  # (start, end) of each step's uploads on the copy stream
        for rows in wl.rows:
            hl = rows.logits.cpu().pin_memory()
            hv = rows.v.cpu().pin_memory()
            self.host.append((hl, hv))
            self.h2d += hl.numel() * hl.element_size() + hv.numel() * hv.element_size()
        for rows in wl.rows:
            # per row: topk gap, dropped, refined gap, best gap, best rank (8 B), best idx (k * 4 B)
            self.d2h += rows.num_rows * (4 * 4 + 8 + 4 * K_SEL)
        # pinned host buffers for the results, so every download is asynchronous
        self.out_host = []
        for rows in wl.rows:
            R = rows.num_rows
            self.out_host.append([torch.empty(R, 1, dtype=torch.float32).pin_memory(),
                                  torch.empty(R, 1, dtype=torch.float32).pin_memory(),
                                  torch.empty(R, 1, dtype=torch.float32).pin_memory(),
                                  torch.empty(R, dtype=torch.float32).pin_memory(),
                                  torch.empty(R, dtype=torch.int64).pin_memory(),
                                  torch.empty(R, K_SEL, dtype=torch.int32).pin_memory()])

    def step(self):
        wl, fw = self.wl, self.wl.fw
        main, cs = torch.cuda.current_stream(), self.copy_stream
        cs.wait_stream(main)
        ready = []
        with torch.cuda.stream(cs):
            u0 = torch.cuda.Event(enable_timing=True)
            u0.record(cs)
            for (hl, hv), rows in zip(self.host, wl.rows):
                rows.logits.copy_(hl, non_blocking=True)
                rows.v.copy_(hv, non_blocking=True)
                ev = torch.cuda.Event(enable_timing=True)
                ev.record(cs)
                ready.append(ev)
        self.upload_ev.append((u0, ready[-1]))
        for st in wl.streams:
            st.wait_stream(main)
        for st, ev, rows, k2, k1, hout in zip(wl.streams, ready, wl.rows, wl.k2, wl.k1, self.out_host):
            with torch.cuda.stream(st):
                st.wait_event(ev)
                top = fw.dense_and_topk_gap(rows, k2, kept_bits=False)
                sw = fw.swap_refine(rows, k2, top, E=N_KEYS, max_swaps=32)
                bs = fw.best_subset(rows, k1, k_max=K_SEL)
                for h, t in zip(hout, (top["gap"], top["dropped"], sw["refined_gap"], bs["best_gap"],
                                       bs["best_rank"], bs["best_idx"][:, :K_SEL])):
                    h.copy_(t.reshape(h.shape), non_blocking=True)
        for st in wl.streams:
            main.wait_stream(st)
        return self.out_host

    def upload_ms(self, last):
        """Copy-stream time of the uploads of the last `last` steps (ms each)."""
        torch.cuda.synchronize()
        r = [a.elapsed_time(b) for a, b in self.upload_ev[-last:]]
        self.upload_ev = []
        return r


def combine_ranks(ms, units_per_rank, dist=None, device=None):
    """Whole-job throughput of weak-scaling replicas: every rank processed
    units_per_rank in its own ms; the job took the slowest rank's time.
    Returns (units per second over all ranks, max ms)."""
    world = 1
    if dist is not None and dist.is_initialized():
        import torch as _t

        world = dist.get_world_size()
        dev = device if dist.get_backend() == "nccl" else "cpu"
        t = _t.tensor([float(ms)], dtype=_t.float64, device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
    return units_per_rank * world / (ms * 1e-3), ms


def time_steps(step, K, W, flush, barrier):
    for _ in range(W):
        step()
    torch.cuda.synchronize()
    barrier()
    torch.cuda.synchronize()
    times = []
    total = 0.0
    for _ in range(K):
        flush()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        step()
        e1.record()
        e1.synchronize()
        t = e0.elapsed_time(e1)
        times.append(t)
        total += t
    torch.cuda.synchronize()
    barrier()
    return total, times


def roofline(bound, achieved, peak, unit, traffic=None, **extra):
    return dict(bound=bound, achieved=achieved, peak=peak, unit=unit, frac=achieved / peak, traffic=traffic, **extra)


def traffic_of(name, units):
    t = TRAFFIC_PER_UNIT.get(name)
    return None if t is None else t[0] * units


# ------------------------------------------------------------- CPU oracle

def cpu_baseline(seed, rows_per_group=40):
    """The fp64 oracle on a bounded sample of the headline workload: the first
    rows_per_group rows of each of the five groups, the whole path."""
    import oracle

    oracle.build()
    bs = workloads.exact_enum(seed=seed, rows_scale=1.0,
                              groups=tuple((rows_per_group, d) for _, d in workloads.ENUM_GROUPS))
    Hs = [oracle.HostRows(b) for b in bs]
    t0 = time.perf_counter()
    for H in Hs:
        oracle.dense_and_topk_gap(H)
        oracle.swap_refine(H, E=N_KEYS, max_swaps=32)
        oracle.best_subset(H)
    dt = time.perf_counter() - t0
    rows = sum(H.num_rows for H in Hs)
    return dict(value=rows / dt, unit="rows/s", cores=oracle.num_threads(), kind="oracle",
                sample=f"first {rows_per_group} rows of each of the 5 groups ({rows} rows, "
                       f"{rows * SUBSETS_PER_ROW:,} subsets), whole path (gap, swap, best subset), fp64",
                seconds=dt)


# ----------------------------------------------------------------- sections

def section_exact_toy(fw, device, K, W, flush, peaks):
    """cfg 1: 256 rows, n=20, k=5, d=64, the whole path (latency-bound, too small
    for a roofline claim)."""
    b = workloads.exact_toy(seed=0)
    wl = EnumWorkload(fw, 0, device, batches=[b], E=20)
    total, _ = time_steps(lambda: wl.step(), K, W, flush, lambda: None)
    ms = total / K
    st = wl.stats()
    return dict(workload="exact_toy: 256 rows, n=20, k=5, d=64, fp32 V", metric="rows/s",
                value=wl.num_rows / (ms * 1e-3), ms_per_step=ms,
                subsets_covered_per_s=wl.subsets / (ms * 1e-3), walk_leaves=st["inner_leaves"],
                rows_exhaustive=st["rows_exhaustive"])


def section_adversarial(fw, device, K, W, flush, peaks):
    """The exact search alone on 512 rows of each adversarial kind: rows/s and
    the rows that overflow to the exhaustive fp64 path."""
    out = {}
    for kind in workloads.ADVERSARIAL_KINDS:
        b = workloads.exact_adversarial(kind, rows=512, seed=0)
        rows = fw.rows_from_batch(b, device)
        k1 = torch.as_tensor(np.asarray(b.k)[:, 0].copy()).to(device)
        kk = int(np.asarray(b.k)[0, 0])
        holder = {}

        def step():
            holder["bs"] = fw.best_subset(rows, k1, k_max=kk)

        total, _ = time_steps(step, K, W, flush, lambda: None)
        ms = total / K
        st = fw.best_subset_stats(rows, holder["bs"])
        n = int(b.n_host[0])
        out[kind] = dict(n=n, k=kk, d=b.d, rows=rows.num_rows, ms_per_call=ms, rows_per_s=rows.num_rows / (ms * 1e-3),
                         subsets_covered_per_s=rows.num_rows * math.comb(n, kk) / (ms * 1e-3),
                         rows_exhaustive=st["rows_exhaustive"],
                         exhaustive_frac=st["rows_exhaustive"] / rows.num_rows, candidates=st["candidates"],
                         walk_leaves=st["inner_leaves"])
    return out


def section_long_rows(fw, device, K, W, flush, peaks, rows_per_head=512):
    """a1-a4 (top-k gap) and a5 (swap rule, E=32) on 8 heads x rows_per_head rows
    x 32,768 keys (4,096 rows at the default), and the group vote."""
    b = workloads.long_rows(seed=0, rows_per_head=rows_per_head, backend="torch", device=device)
    rows = fw.rows_from_batch(b, device)
    rows_k = b.k
    holder = {}

    def gap_step():
        holder["top"] = fw.dense_and_topk_gap(rows, rows_k, kept_bits=True)

    total, _ = time_steps(gap_step, K, W, flush, lambda: None)
    ms_gap = total / K
    top = holder["top"]

    def swap_step():
        holder["sw"] = fw.swap_refine(rows, rows_k, top, E=32, max_swaps=64)

    ks = max(2, K // 2)
    total, _ = time_steps(swap_step, ks, 1, flush, lambda: None)
    ms_swap = total / ks
    ns = holder["sw"]["n_swaps"].float()
    R, n, d, nb = rows.num_rows, int(b.n_host[0]), b.d, rows_k.shape[1]

    # the group vote: one set per KV head (its rows_per_head query rows) at the
    # same three budgets, every row scored against it
    s_vote = rows_k[::rows.rows_per_group].contiguous()

    def vote_step():
        holder["vote"] = fw.group_vote(rows, s_vote, top)

    total, _ = time_steps(vote_step, K, W, flush, lambda: None)
    ms_vote = total / K
    G = rows.num_groups
    # algorithmic bytes: the logits twice (the set needs every row's logits, each
    # row's score needs the set), the value blocks once, the summed masses
    # written and read, outputs (gap, dropped, status, bits)
    vbytes = (2 * rows.logits.numel() * 4 + rows.v.numel() * 2 + 2 * G * n * 4
              + R * (nb * 8 + 4) + G * nb * (n // 8))
    vach = vbytes / (ms_vote * 1e-3) / 1e9
    # algorithmic bytes of the gap call: logits once, the value blocks once,
    # outputs (o, three o_A, gap / dropped / phi, thresholds, kept bits)
    nbytes = (rows.logits.numel() * 4 + rows.v.numel() * 2
              + R * (d * 4 * (1 + nb) + nb * 3 * 4 + nb * 8 + nb * (n // 8)))
    ach = nbytes / (ms_gap * 1e-3) / 1e9
    rounds = float((ns + 1).sum().item())
    return dict(workload=f"long_rows: 8 heads x {rows_per_head} rows, n=32768, d=128, bf16 V, k in {{2048,4096,8192}}",
                path="a1-a4 (fw_dense_and_topk_gap) then a5 (fw_swap_refine, E=32)", metric="rows/s",
                value=R / ((ms_gap + ms_swap) * 1e-3), gap_rows_per_s=R / (ms_gap * 1e-3),
                swap_rows_per_s=R / (ms_swap * 1e-3), ms_gap=ms_gap, ms_swap=ms_swap,
                swaps_per_row_budget=float(ns.mean().item()), swap_rounds=rounds,
                roofline=roofline("hbm", ach, peaks["hbm_gbs"], "GB/s", traffic_of("long_gap", R),
                                  kernel="fw_dense_and_topk_gap (select + P.V)", algorithmic_bytes=nbytes,
                                  launch_ms=ms_gap),
                group_vote=dict(path="fw_group_vote: one set per KV head by summed mass, all rows scored",
                                ms_per_call=ms_vote, rows_per_s=R / (ms_vote * 1e-3),
                                roofline=roofline("hbm", vach, peaks["hbm_gbs"], "GB/s", traffic_of("group_vote", R),
                                                  kernel="k_vote_mass + k_vote_select + k_long_pv_tma (vote mode: tcgen05 band-masked P.V)",
                                                  algorithmic_bytes=vbytes)))


def section_contour(fw, device, K, W, flush, peaks, cells=256):
    cb = workloads.contour_cache(seed=0, cells=cells, backend="torch", device=device)
    Kc, Vc = cb.K.view(torch.int16), cb.V.view(torch.int16)
    Ko = torch.empty(cb.total_budget, cb.d, dtype=torch.int16, device=device)
    Vo = torch.empty_like(Ko)
    ev = Events()
    # outputs and workspace allocated once, as a serving loop would hold them
    ca = fw.contour_alloc(cb.scores, floor=cb.floor, total_budget=cb.total_budget, uniform_s=cb.uniform_s)
    cc = fw.contour_alloc_capped(cb.scores, floor=cb.floor, total_budget=cb.total_budget, uniform_s=cb.uniform_s,
                                 cap=cb.uniform_s)

    def step():
        e0 = ev.start()
        a = fw.contour_alloc(cb.scores, floor=cb.floor, total_budget=cb.total_budget, uniform_s=cb.uniform_s,
                             out=ca, workspace=ca["_ws"])
        ev.stop(e0, "alloc")
        e1 = ev.start()
        fw.ragged_compact(Kc, Vc, a["offsets"], a["kept_pos"], cb.total_budget, out=(Ko, Vo))
        ev.stop(e1, "compact")

    total, times = time_steps(step, K, W, flush, lambda: None)
    ms = total / K
    parts = ev.take()[-2 * K:]
    # the enforced mode: every cell capped at the uniform count
    holder = {}

    def capped_step():
        holder["c"] = fw.contour_alloc_capped(cb.scores, floor=cb.floor, total_budget=cb.total_budget,
                                              uniform_s=cb.uniform_s, cap=cb.uniform_s, out=cc, workspace=cc["_ws"])

    tc_, _ = time_steps(capped_step, K, W, flush, lambda: None)
    ms_capped = tc_ / K
    kept_capped = int(holder["c"]["offsets"][-1].item())
    # the observation-window score (32 window queries per cell) on the cache's keys
    Qw = workloads.window_queries(seed=0, cells=cb.cells, w=32, d=cb.d, backend="torch", device=device)
    Qi = Qw.view(torch.int16)
    wsc = torch.empty(cb.cells, cb.T, dtype=torch.float32, device=device)

    def wscore_step():
        fw.window_score(Qi, Kc, pool=7, out=wsc)

    tw, _ = time_steps(wscore_step, K, W, flush, lambda: None)
    ms_ws = tw / K
    wbytes = cb.cells * cb.T * cb.d * 2 + cb.cells * 32 * cb.d * 2 + 2 * cb.cells * cb.T * 4
    wflops = 2 * 2 * cb.cells * 32 * cb.T * cb.d  # two passes of the window products
    # decode-time appends: one new row per cell into storage with 64 rows of room per cell
    cnt = holder["c"]["counts"].to(torch.int32)
    cap = (cnt + 64).to(torch.int32)
    base = torch.cumsum(cap.to(torch.int64), 0) - cap.to(torch.int64)
    rows_store = int((base[-1] + cap[-1]).item())
    Ks = torch.empty(rows_store, cb.d, dtype=torch.int16, device=device)
    Vs = torch.empty_like(Ks)
    nK = torch.zeros(cb.cells, 1, cb.d, dtype=torch.int16, device=device)
    nV = torch.zeros_like(nK)
    fill = torch.zeros_like(cnt)
    st_app = torch.empty_like(cnt)

    def append_step():
        fill.zero_()
        fw.ragged_append(Ks, Vs, base, cap, fill, nK, nV, st_app)

    ta, _ = time_steps(append_step, K, W, flush, lambda: None)
    ms_app = ta / K
    ms_alloc = sum(t for t, tag in parts if tag == "alloc") / K
    ms_comp = sum(t for t, tag in parts if tag == "compact") / K
    nbytes = cb.cells * cb.T * 4 + 2 * 2 * cb.total_budget * cb.d * 2 + cb.total_budget * 4 + (cb.cells + 1) * 8
    ach = nbytes / (ms * 1e-3) / 1e9
    cbytes = 2 * 2 * cb.total_budget * cb.d * 2
    return dict(workload=f"contour_cache: {cb.cells} cells x 32768 tokens, d=128 bf16 K/V, budget 1/8, floor 32",
                path="a7-a8 (fw_contour_alloc + fw_ragged_compact)", metric="kept KV rows/s",
                value=cb.total_budget / (ms * 1e-3), ms_per_step=ms, ms_alloc=ms_alloc, ms_compact=ms_comp,
                roofline=roofline("hbm", ach, peaks["hbm_gbs"], "GB/s", traffic_of("contour", cb.total_budget),
                                  algorithmic_bytes=nbytes, kernel="k_c_* + k_compact"),
                compact_roofline=roofline("hbm", cbytes / (ms_comp * 1e-3) / 1e9, peaks["hbm_gbs"], "GB/s",
                                          traffic_of("compact", cb.total_budget), kernel="k_compact",
                                          algorithmic_bytes=cbytes),
                capped=dict(path="fw_contour_alloc_capped, cap = uniform count (4,096): the enforced mode",
                            ms_per_call=ms_capped, kept_rows=kept_capped),
                window_score=dict(path=f"fw_window_score: 32 window queries x {cb.cells} cells x 32,768 keys, d=128, "
                                       "pool 7 (TMA + tcgen05, two passes over K)",
                                  ms_per_call=ms_ws, keys_per_s=cb.cells * cb.T / (ms_ws * 1e-3),
                                  roofline=roofline("hbm", wbytes / (ms_ws * 1e-3) / 1e9, peaks["hbm_gbs"], "GB/s",
                                                    traffic_of("window_score", cb.cells * cb.T),
                                                    kernel="k_wscore", algorithmic_bytes=wbytes,
                                                    bytes_basis="K once, the window queries, votes and scores "
                                                                "written; the kernel reads K twice"),
                                  tensor_tflops=wflops / (ms_ws * 1e-3) / 1e12),
                decode_append=dict(path=f"fw_ragged_append: one new K/V row per cell ({cb.cells} cells, d=128)",
                                   ms_per_call=ms_app, rows_per_s=cb.cells / (ms_app * 1e-3)))


def section_mixed(fw, device, K, W, flush, peaks, rows_scale=1.0):
    """cfg 5: 168,192 rows from five profiles, GQA groups of 4 sharing bf16 V,
    one budget per row: the gap call and the swap rule (E = 32), one profile
    per call (each profile is generated, timed and freed in turn)."""
    tot_rows, ms_gap, ms_swap, nbytes, swaps = 0, 0.0, 0.0, 0, []
    per = {}
    for prof in workloads.MIXED_PROFILES:
        b = workloads.mixed_profiles(seed=0, backend="torch", device=device, profiles=(prof,),
                                     rows_scale=rows_scale)[0]
        rows = fw.rows_from_batch(b, device)
        holder = {}

        def gap_step():
            holder["top"] = fw.dense_and_topk_gap(rows, b.k, kept_bits=False)

        t, _ = time_steps(gap_step, K, W, flush, lambda: None)
        g = t / K

        def swap_step():
            holder["sw"] = fw.swap_refine(rows, b.k, holder["top"], E=32, max_swaps=64)

        t, _ = time_steps(swap_step, 2, 1, flush, lambda: None)
        s = t / 2
        R, n, d = rows.num_rows, int(b.n_host[0]), b.d
        by = rows.logits.numel() * 4 + rows.v.numel() * 2 + R * (d * 4 * 2 + 4 * 4 + 8)
        per[prof[0]] = dict(rows=R, n=n, d=d, ms_gap=g, ms_swap=s, gap_gbs=by / (g * 1e-3) / 1e9,
                            swaps_per_row=float(holder["sw"]["n_swaps"].float().mean().item()))
        tot_rows += R
        ms_gap += g
        ms_swap += s
        nbytes += by
        del rows, holder, b
        torch.cuda.empty_cache()
    ach = nbytes / (ms_gap * 1e-3) / 1e9
    return dict(workload="mixed_profiles: 168,192 rows, 5 profiles (d 64/128, n 1,024..16,384), GQA-4 bf16 V, "
                         "k/n in {1/32,1/16,1/8,1/4}", metric="rows/s", value=tot_rows / ((ms_gap + ms_swap) * 1e-3),
                gap_rows_per_s=tot_rows / (ms_gap * 1e-3), swap_rows_per_s=tot_rows / (ms_swap * 1e-3),
                ms_gap=ms_gap, ms_swap=ms_swap, profiles=per,
                roofline=roofline("hbm", ach, peaks["hbm_gbs"], "GB/s", traffic_of("mixed_gap", tot_rows),
                                  kernel="fw_dense_and_topk_gap, one call per profile", algorithmic_bytes=nbytes,
                                  bytes_basis="logits once, each GQA group's value block once, outputs"))


def section_pool(fw, device, K, W, flush, peaks, groups=256):
    """f2: ES_pool at the candidate-set schedule s = 4/8/16/32 (E = 24/12/6/4)
    on the first `groups` GQA groups of mixed profiles B (n = 4,096, d = 128)
    and E (n = 16,384, d = 128): rows/s, subsets/s, and the share of the top-mass
    gap that the best candidate subset closes."""
    out = {}
    for prof in (workloads.MIXED_PROFILES[1], workloads.MIXED_PROFILES[4]):
        name, rows_full, d, n = prof
        b = workloads.mixed_profiles(seed=0, backend="torch", device=device, profiles=(prof,),
                                     rows_scale=groups * 4 / rows_full)[0]
        rows = fw.rows_from_batch(b, device)
        R = rows.num_rows
        k = torch.tensor([s for s, _ in POOL_SCHED], dtype=torch.int32, device=device).repeat(R, 1)
        E = [e for _, e in POOL_SCHED]
        top = fw.dense_and_topk_gap(rows, k, kept_bits=False, o_kept=False)
        holder = {}

        def step():
            holder["p"] = fw.pool_best_subset(rows, k, top, E=E)

        t, _ = time_steps(step, max(1, K // 2), 1, flush, lambda: None)
        ms = t / max(1, K // 2)
        p = holder["p"]
        bg, tg = p["best_gap"].double(), p["topk_gap"].double()
        c_hat = torch.where(tg > 0, 1.0 - bg / tg, torch.zeros_like(tg)).cpu().numpy()
        subsets = sum(math.comb(s + e, min(s, e)) for s, e in POOL_SCHED) * R
        out[name] = dict(rows=R, n=n, d=d, ms_per_call=ms, rows_per_s=R / (ms * 1e-3), subsets_per_s=subsets / (ms * 1e-3),
                         c_hat_quartiles={f"s={s}": [float(np.percentile(c_hat[:, j], q)) for q in (25, 50, 75)]
                                          for j, (s, _) in enumerate(POOL_SCHED)},
                         rescored_per_item=float(p["n_cand"].double().mean().item()))
        del rows, top, holder, b
        torch.cuda.empty_cache()
    return out


def section_audit(fw, device, K, W, flush, peaks, groups=256):
    """f4: the deployed selectors' es against ES_pool and top-mass at s = 4/8/16/32
    on the first `groups` GQA groups of mixed profile B (n = 4,096, d = 128): the
    audit call's time and the median of each rule's es / ES_pool."""
    prof = workloads.MIXED_PROFILES[1]
    b = workloads.mixed_profiles(seed=1, backend="torch", device=device, profiles=(prof,),
                                 rows_scale=groups * 4 / prof[1])[0]
    rows = fw.rows_from_batch(b, device)
    R = rows.num_rows
    sched = [s for s, _ in POOL_SCHED]
    k = torch.tensor(sched, dtype=torch.int32, device=device).repeat(R, 1)
    top = fw.dense_and_topk_gap(rows, k, kept_bits=False, o_kept=False)
    holder = {}

    def step():
        holder["a"] = fw.selector_audit(rows, sched, top)

    t, _ = time_steps(step, K, W, flush, lambda: None)
    ms = t / K
    pool = fw.pool_best_subset(rows, k, top, E=[e for _, e in POOL_SCHED])
    es = holder["a"]["es"].double()
    esp = pool["best_gap"].double()
    ratios = {}
    for j, s in enumerate(sched):
        r = {name: float(torch.nanmedian(es[:, i, j] / esp[:, j]).item()) for i, name in enumerate(fw.SELECTORS)}
        r["top_mass"] = float(torch.median(top["gap"].double()[:, j] / esp[:, j]).item())
        ratios[f"s={s}"] = r
    return dict(workload=f"mixed profile B, first {groups} GQA groups ({R} rows, n=4096, d=128)",
                ms_per_call=ms, rows_per_s=R / (ms * 1e-3), median_es_over_ES_pool=ratios)


# --------------------------------------------------------------------- main

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-sections", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--rows-scale", type=float, default=1.0,
                    help="fraction of the headline rows (profiling captures of a smaller case)")
    ap.add_argument("--only", default="all",
                    choices=["all", "exact_toy", "adversarial", "long_rows", "contour", "mixed", "pool", "audit"],
                    help="run one section alone and print its line (profiling captures)")
    ap.add_argument("--long-rows-per-head", type=int, default=512,
                    help="rows per head of the long-row section (profiling captures of a smaller case)")
    ap.add_argument("--mixed-rows-scale", type=float, default=1.0,
                    help="fraction of the mixed-profile rows (profiling captures of a smaller case)")
    ap.add_argument("--contour-cells", type=int, default=256,
                    help="cells of the contour workload (profiling captures of a smaller case)")
    args = ap.parse_args()
    K, W = args.steps, max(3, args.warmup)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist_mod

        dist = dist_mod
        dist.init_process_group("nccl" if args.impl == "ours" else "gloo")

    if args.impl == "reference":
        # the reference arm is the fp64 CPU oracle, on rank 0 only
        if rank == 0:
            steps = []
            for _ in range(W):
                cpu_baseline(seed=0, rows_per_group=8)
            for _ in range(K):
                steps.append(cpu_baseline(seed=0, rows_per_group=8))
            v = statistics.median(s["value"] for s in steps)
            sec = sum(s["seconds"] for s in steps) / K
            line = dict(impl="reference", metric="rows/s", value=v, unit="rows/s", n_gpus=args.gpus,
                        steps=K, warmup=W, ms_per_step=sec * 1e3, higher_is_better=True, scaling="weak",
                        vs_baseline=None, dtype="f64", data="synthetic",
                        config=dict(workload="exact_enum: 168,192 rows (5 groups, d=64/128), n=24, k=6; "
                                             "step = gap + swap + exact best subset",
                                    sample="first 8 rows of each group per step"),
                        cpu_baseline=dict(value=v, unit="rows/s", cores=steps[0]["cores"], kind="oracle",
                                          sample=steps[0]["sample"]),
                        e2e=dict(value=v, unit="rows/s", h2d_bytes_per_step=0, d2h_bytes_per_step=0))
            print(json.dumps(line), flush=True)
        if dist:
            dist.destroy_process_group()
        return

    device = f"cuda:{local}"
    torch.cuda.set_device(local)
    from paper_2608_25230_gb300 import fw

    peaks = read_peaks()
    flush = L2Flush(device)
    sections_fn = dict(
        exact_toy=lambda k, w: section_exact_toy(fw, device, k, w, flush, peaks),
        adversarial=lambda k, w: section_adversarial(fw, device, k, w, flush, peaks),
        long_rows=lambda k, w: section_long_rows(fw, device, k, w, flush, peaks, rows_per_head=args.long_rows_per_head),
        contour=lambda k, w: section_contour(fw, device, k, w, flush, peaks, cells=args.contour_cells),
        mixed=lambda k, w: section_mixed(fw, device, k, w, flush, peaks, rows_scale=args.mixed_rows_scale),
        pool=lambda k, w: section_pool(fw, device, k, w, flush, peaks),
        audit=lambda k, w: section_audit(fw, device, k, w, flush, peaks))
    if args.only != "all":
        if rank == 0:
            print(json.dumps(dict(section=args.only, **{"result": sections_fn[args.only](K, W)})), flush=True)
        if dist:
            dist.destroy_process_group()
        return
    barrier = (lambda: dist.barrier()) if dist else (lambda: None)

    wl = EnumWorkload(fw, seed=rank, device=device, rows_scale=args.rows_scale)
    torch.cuda.synchronize()
    l0 = fw.launch_count()
    with ClockSampler(local) as clk:
        total_ms, times = time_steps(lambda: wl.step(time_enum=True), K, W, flush, barrier)
    launches = (fw.launch_count() - l0) // (K + W)
    launches_timed = launches * K
    enum_ev = wl.ev.take()[-5 * K:]
    clocks = clk.summary()
    value, ms = combine_ranks(total_ms / K, wl.num_rows, dist, device)
    stats = wl.stats()

    # roofline of the dominant call (fw_best_subset: prep, walk, rescore, exhaustive)
    enum_ms = sum(t for t, _ in enum_ev) / K  # per step, all five groups
    enum_launch_ms = sum(t for t, _ in enum_ev) / len(enum_ev)
    sm_mhz = clocks.get("sm_mhz") or peaks["sm_max"]
    fma_peak, sms = fp32_peak_tflops(device, sm_mhz)
    fma_probe = fp32_fma_measured(fw, device)
    gram = wl.gram_flops()
    work = gram + stats["inner_ops"]
    alu_ach = work / (enum_ms * 1e-3) / 1e12

    # end to end through the public API with host buffers
    e2e = EnumE2E(wl)
    K2 = max(3, K // 2)
    e2e_total, e2e_times = time_steps(e2e.step, K2, W, flush, barrier)
    e2e_value, e2e_ms = combine_ranks(e2e_total / K2, wl.num_rows, dist, device)
    up_ms = e2e.upload_ms(K2)

    sections = {}
    if not args.no_sections and rank == 0:
        for name in ("exact_toy", "adversarial", "long_rows", "contour", "mixed", "pool", "audit"):
            sections[name] = sections_fn[name](5, 3)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        cpu = cpu_baseline(seed=0)
        cpu.pop("seconds", None)

    line = dict(metric="rows/s", value=value, unit="rows/s", n_gpus=world, steps=K, warmup=W,
                ms_per_step=ms, higher_is_better=True, scaling="weak", vs_baseline=None,
                dtype="f32 (screening), double-float (every decision and reported gap)", data="synthetic",
                config=dict(workload="exact_enum: 168,192 rows in 5 groups (d=64,128,128,128,64), n=24, k=6, "
                                     "134,596 subsets/row; step = gap + swap (E=all) + exact best subset",
                            rows_per_gpu=wl.num_rows, subsets_per_step_per_gpu=wl.subsets,
                            l2="inputs larger than L2 (1.6 GB) and a 256 MiB L2 flush between steps",
                            parallelism=f"rows sharded, {world} independent replica(s)"),
                derived=dict(subsets_covered_per_s=wl.subsets * world / (ms * 1e-3),
                             walk_leaves_per_s=stats["inner_leaves"] * world / (ms * 1e-3),
                             walk_leaves_per_row=stats["inner_leaves"] / wl.num_rows,
                             rows_exhaustive=stats["rows_exhaustive"], candidates=stats["candidates"],
                             note="the search covers every subset; its bounds exclude most of them without a "
                                  "visit, and walk_leaves counts the subsets its inner enumeration visits"),
                roofline=roofline("alu", alu_ach, fma_peak, "TFLOP/s", traffic_of("fw_best_subset", wl.num_rows),
                                  kernel="fw_best_subset (k_enum_prep + k_enum_walk + k_enum_rescore + "
                                         "k_enum_exhaustive)", launch_ms=enum_launch_ms,
                                  work_basis="fp32 flops the call is known to execute: the prep kernel's Gram "
                                             "products (2 d (n+1)(n+2)/2 per row) plus the walk's counted "
                                             "inner-enumeration operations; per step "
                                             f"{gram:.3e} + {stats['inner_ops']:.3e}",
                                  peak_basis=f"{sms} SMs x 128 fp32 lanes x 2 x {sm_mhz:.0f} MHz (median SM clock "
                                             f"under load)",
                                  peak_check=dict(fma_probe_tflops=fma_probe, of_nominal=fma_probe / fma_peak,
                                                  kernel="fw_fp32_fma_probe: 16 independent FMA chains per "
                                                         "thread, 8 CTAs of 256 threads per SM")),
                e2e=dict(value=e2e_value, unit="rows/s",
                         h2d_bytes_per_step=e2e.h2d, d2h_bytes_per_step=e2e.d2h,
                         step_ms=[round(t, 2) for t in e2e_times],
                         upload_ms=[round(t, 2) for t in up_ms],
                         upload_gbs=e2e.h2d / (statistics.median(up_ms) * 1e-3) / 1e9 if up_ms else None,
                         note="uploads overlap compute within a step (group g + 1 uploads while group g "
                              "computes); upload_ms is the copy stream's time from the first to the last "
                              "upload of a step"),
                gpu_launches=int(launches_timed), clocks=clocks, peaks_source=peaks["source"])
    if cpu:
        line["cpu_baseline"] = cpu
    if sections:
        line["sections"] = sections
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
