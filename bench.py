#!/usr/bin/env python3
"""Benchmark of the restoration sweep (fingerprint, pack, unpack+verify, diff).

One step is one restoration of a rank's state from a data-parallel replica
(FlashRecovery, arXiv 2509.03047, Sec. III-E), with every sweep call once:
  fingerprint(replica) -> pack(replica -> transfer buffer) -> inject the
  workload's bit flips -> unpack_verify(buffer -> restored rank)
  -> fingerprint(restored) -> diff(tables).
The default workload is the largest one that fits one GPU: a Llama-3-70B
rank at TP=8/PP=4 (20 layers + embedding, bf16 weight + fp32 master/m/v,
31.8 GB), 16 MiB chunks, 50 NaNs in the state and 1,000 bit flips in the
buffer.  Inputs are synthetic and seeded, and far larger than L2.

value = state bytes swept per step (4 sweeps of S) / step time, in GB/s,
summed over ranks (replicas only: every rank restores its own state; no
collective is on the data path).

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl flashrec|reference]
"""
from __future__ import annotations

import argparse
import gc
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

METRIC = "state GB/s per call (fingerprint, pack, unpack+verify) and fraction of HBM peak"
SWEEPS_PER_STEP = 4  # fingerprint x2, pack, unpack_verify each touch every state byte
DEFAULT_CONFIG = "l70b_tp8pp4"


# ---------------------------------------------------------------- distributed plumbing

def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def dist_setup(backend: str):
    import torch.distributed as dist

    ws, rank, _ = dist_env()
    if ws > 1 and not dist.is_initialized():
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        os.environ.setdefault("MASTER_PORT", "29511")
        dist.init_process_group(backend=backend, rank=rank, world_size=ws)
    return ws, rank


def barrier():
    import torch.distributed as dist

    if dist.is_initialized():
        dist.barrier()


def max_over_ranks(x: float, device=None) -> float:
    import torch
    import torch.distributed as dist

    if not dist.is_initialized():
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x: float, device=None) -> float:
    import torch
    import torch.distributed as dist

    if not dist.is_initialized():
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


# ---------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi samples every 100 ms while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        return self.summary()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------- helpers

def repo_libraries_loaded():
    """Shared objects of this repository mapped into the process."""
    found = set()
    try:
        with open("/proc/self/maps") as f:
            for line in f:
                path = line.split()[-1] if line.strip() else ""
                if path.startswith(ROOT) and ".so" in path:
                    found.add(os.path.relpath(path, ROOT))
    except OSError:
        pass
    return sorted(found)


def measured_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


def profiled_traffic(kernel_key: str, workload: str):
    """DRAM bytes per launch of `kernel_key` from a committed ncu summary, if
    it was taken on the current kernel sources; else None."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except (OSError, ValueError):
        return None
    from paper_2509_03047_gb300 import build as _b

    ent = rec.get(kernel_key)
    if not ent or ent.get("workload") != workload or ent.get("kernel_sources") != _b.source_digest(kernels_only=True):
        return None
    return ent.get("bytes_per_launch")


def sweep_classes(tensors):
    """Sweep kernels a call launches: one per (element type, 16-byte aligned)
    class that has a chunk body (the library's own planning rule)."""
    from paper_2509_03047_gb300 import flashrec as fr

    cls = set()
    for t in tensors:
        if t.numel() * t.element_size() >= 512:
            cls.add((fr.fr_dtype_of(t), t.data_ptr() % 16 == 0))
    return len(cls)


# ---------------------------------------------------------------- the flashrec arm

def run_flashrec(args):
    import numpy as np
    import torch

    from paper_2509_03047_gb300 import flashrec as fr
    from paper_2509_03047_gb300 import synth

    ws, rank = dist_setup("nccl")
    _, _, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    cfg = synth.get_config(args.config)
    src = synth.make_state(cfg, dev)
    nan_pos = synth.inject_nonfinite(cfg, src)
    dst = [torch.empty_like(t) for t in src]
    plan_s = fr.Plan(src, cfg.chunk_bytes)
    plan_d = fr.Plan(dst, cfg.chunk_bytes)
    S, C, P = plan_s.state_bytes, plan_s.n_chunks, plan_s.packed_bytes
    packed = plan_s.new_packed()
    tab_s, tab_d = plan_s.new_table(), plan_d.new_table()
    mism = torch.empty(C, dtype=torch.int32, device=dev)
    nmis = torch.empty(1, dtype=torch.int64, device=dev)
    div = torch.empty(C, dtype=torch.int32, device=dev)
    ndiv = torch.empty(1, dtype=torch.int64, device=dev)
    flips = synth.flip_positions(P, cfg.flips, cfg.seed)
    fb = np.unique(flips // 8)
    fmask = np.zeros(fb.size, dtype=np.uint8)
    for p in flips:
        fmask[np.searchsorted(fb, p // 8)] ^= np.uint8(1 << (p % 8))
    flip_idx = torch.as_tensor(fb, dtype=torch.int64, device=dev)
    flip_mask = torch.as_tensor(fmask, device=dev)
    flip_idx_h = torch.as_tensor(fb, dtype=torch.int64)
    flip_mask_h = torch.as_tensor(fmask)
    stream = torch.cuda.current_stream()
    n_cls = sweep_classes(src)

    def step(ev=None, buf=None, sync_counts=False):
        if buf is None:
            buf = packed
        if ev:
            ev[0].record(stream)
        fr.fr_fingerprint(plan_s.handle, tab_s, stream)
        if ev:
            ev[1].record(stream)
        fr.fr_pack(plan_s.handle, buf, stream)
        if ev:
            ev[2].record(stream)
        if flip_idx.numel():  # the workload's faults in the transfer buffer
            if buf.is_cuda:
                buf[flip_idx] ^= flip_mask
            else:
                stream.synchronize()
                buf[flip_idx_h] ^= flip_mask_h
        if ev:
            ev[3].record(stream)
        fr.fr_unpack_verify(plan_d.handle, buf, mism, nmis, stream)
        if ev:
            ev[4].record(stream)
        fr.fr_fingerprint(plan_d.handle, tab_d, stream)
        if ev:
            ev[5].record(stream)
        fr.fr_diff(tab_s, tab_d, C, div, ndiv, stream)
        if ev:
            ev[6].record(stream)
        if sync_counts:
            return int(nmis.item()), int(ndiv.item())
        return None

    # every call: one sweep launch for all classes + finalize; fingerprint
    # twice, unpack with its compaction; diff
    sweeps = min(n_cls, 1)
    launches_per_step = (sweeps + 1) * 2 + (sweeps + 1) + (sweeps + 2) + 1

    # correctness of the timed configuration: the injected flips are found
    for _ in range(args.warmup):
        step()
    n_mis, n_div = step(sync_counts=True)
    torch.cuda.synchronize()

    clocks = ClockSampler(local)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(7)] for _ in range(args.steps)]
    barrier()
    torch.cuda.synchronize()
    clocks.start()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for k in range(args.steps):
        step(evs[k])
    t_end.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    barrier()
    total_ms = t_start.elapsed_time(t_end)
    names = ["fingerprint_replica", "pack", "inject_flips", "unpack_verify", "fingerprint_restored", "diff"]
    per = {n: sum(e[i].elapsed_time(e[i + 1]) for e in evs) / args.steps for i, n in enumerate(names)}
    samples = {n: sorted(e[i].elapsed_time(e[i + 1]) for e in evs) for i, n in enumerate(names)}
    samples["fingerprint"] = sorted(samples["fingerprint_replica"] + samples["fingerprint_restored"])
    ms_step = max_over_ranks(total_ms / args.steps, dev)
    value = sum_over_ranks(SWEEPS_PER_STEP * S / (ms_step * 1e-3) / 1e9, dev)

    # ---- roofline of the dominant kernel pair (sweep + finalize of one call)
    peak, peak_kind = measured_peak()
    H = P - S  # header table, gap and padding bytes
    alg = {"fingerprint": S + 16 * C, "pack": S + P, "unpack_verify": P + S + 4 * C}
    t_call = {"fingerprint": (per["fingerprint_replica"] + per["fingerprint_restored"]) / 2,
              "pack": per["pack"], "unpack_verify": per["unpack_verify"]}
    share = {"fingerprint": 2 * t_call["fingerprint"], "pack": t_call["pack"],
             "unpack_verify": t_call["unpack_verify"]}
    dom = max(share, key=share.get)
    calls = {}
    for k in alg:
        gbs = alg[k] / (t_call[k] * 1e-3) / 1e9
        xs = samples[k]
        calls[k] = {"ms": round(t_call[k], 4), "ms_median": round(xs[len(xs) // 2], 4), "ms_best": round(xs[0], 4),
                    "state_gbs": round(S / (t_call[k] * 1e-3) / 1e9, 1),
                    "alg_bytes": alg[k], "achieved_gbs": round(gbs, 1), "frac": round(gbs / peak, 4),
                    "frac_of_8tbs": round(gbs / 8000.0, 4)}
    calls["diff"] = {"us": round(per["diff"] * 1e3, 2), "alg_bytes": 32 * C}
    calls["inject_flips_us"] = round(per["inject_flips"] * 1e3, 2)
    ach = alg[dom] / (t_call[dom] * 1e-3) / 1e9
    roofline = {"kernel": "fr_%s (sweep + finalize kernels)" % dom, "bound": "hbm", "achieved": round(ach, 1),
                "peak": peak, "unit": "GB/s", "frac": round(ach / peak, 4),
                "peak_source": "%s HBM copy bandwidth (MEASURED_PEAKS.json hbm_gbs)" % peak_kind
                if peak_kind == "measured" else "fallback 6.8 TB/s",
                "traffic": profiled_traffic("fr_" + dom, args.config),
                "alg_bytes_per_launch": alg[dom]}

    # ---- the same step with the fingerprints fused into pack and unpack: the
    # replica's table comes out of fr_pack_fp, the restored state's out of
    # fr_unpack_verify_fp, so the step makes two state sweeps instead of four
    def fused_step(ev=None):
        if ev:
            ev[0].record(stream)
        fr.fr_pack_fp(plan_s.handle, packed, tab_s, stream)
        if ev:
            ev[1].record(stream)
        if flip_idx.numel():
            packed[flip_idx] ^= flip_mask
        if ev:
            ev[2].record(stream)
        fr.fr_unpack_verify_fp(plan_d.handle, packed, mism, nmis, tab_d, stream)
        if ev:
            ev[3].record(stream)
        fr.fr_diff(tab_s, tab_d, C, div, ndiv, stream)
        if ev:
            ev[4].record(stream)

    for _ in range(args.warmup):
        fused_step()
    torch.cuda.synchronize()
    f_mis, f_div = int(nmis.item()), int(ndiv.item())
    fev = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(args.steps)]
    barrier()
    torch.cuda.synchronize()
    for k in range(args.steps):
        fused_step(fev[k])
    torch.cuda.synchronize()
    barrier()
    f_ms = sum(e[0].elapsed_time(e[4]) for e in fev) / args.steps
    f_pack = sum(e[0].elapsed_time(e[1]) for e in fev) / args.steps
    f_unpack = sum(e[2].elapsed_time(e[3]) for e in fev) / args.steps
    fused = {"ms_per_step": round(f_ms, 3),
             "state_gbs_4_sweeps_equiv": round(SWEEPS_PER_STEP * S / (f_ms * 1e-3) / 1e9, 1),
             "pack_fp": {"ms": round(f_pack, 4), "alg_bytes": alg["pack"] + 16 * C,
                         "frac": round((alg["pack"] + 16 * C) / (f_pack * 1e-3) / 1e9 / peak, 4)},
             "unpack_verify_fp": {"ms": round(f_unpack, 4), "alg_bytes": alg["unpack_verify"] + 16 * C,
                                  "frac": round((alg["unpack_verify"] + 16 * C) / (f_unpack * 1e-3) / 1e9 / peak, 4)},
             "found": {"mismatching_chunks": f_mis, "diverged_chunks": f_div},
             "how": "fr_pack_fp -> flips -> fr_unpack_verify_fp -> fr_diff: both fingerprint tables come out of "
                    "the pack and unpack sweeps; same outputs as the step above"}

    # ---- optionally, the fused step captured once in a CUDA graph and replayed
    # (the calls only enqueue kernels, so small states can shed launch overhead)
    graph = None
    if args.graph:
        gs = torch.cuda.Stream(device=dev)

        def graph_body():
            fr.fr_pack_fp(plan_s.handle, packed, tab_s, gs)
            fr.fr_unpack_verify_fp(plan_d.handle, packed, mism, nmis, tab_d, gs)
            fr.fr_diff(tab_s, tab_d, C, div, ndiv, gs)

        gs.wait_stream(stream)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=gs):
            graph_body()
        for _ in range(args.warmup):
            g.replay()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            g.replay()
        e1.record(stream)
        torch.cuda.synchronize()
        g_ms = e0.elapsed_time(e1) / args.steps
        e0.record(stream)
        for _ in range(args.steps):
            fr.fr_pack_fp(plan_s.handle, packed, tab_s, stream)
            fr.fr_unpack_verify_fp(plan_d.handle, packed, mism, nmis, tab_d, stream)
            fr.fr_diff(tab_s, tab_d, C, div, ndiv, stream)
        e1.record(stream)
        torch.cuda.synchronize()
        eager_ms = e0.elapsed_time(e1) / args.steps
        graph = {"ms_per_step": round(g_ms, 4), "eager_ms_per_step": round(eager_ms, 4),
                 "how": "fr_pack_fp -> fr_unpack_verify_fp -> fr_diff captured once in a CUDA graph and "
                        "replayed back to back (no flips), against the same calls launched eagerly"}
        del g

    # ---- end to end through the C ABI with the transfer buffer in pinned host memory
    e2e = None
    if not args.no_e2e:
        try:
            host_buf = plan_s.new_packed(pinned=True)
        except RuntimeError as exc:  # pinning P bytes per rank can fail on a crowded host
            host_buf = None
            e2e = {"unavailable": "pinned host buffer of %d bytes: %s" % (P, str(exc).splitlines()[0])}
        # every rank takes the leg (it has collectives) only if every rank could pin
        if max_over_ranks(0.0 if host_buf is not None else 1.0, dev) > 0.0 and host_buf is not None:
            e2e = {"unavailable": "another rank could not pin its host buffer"}
            host_buf = None
    if not args.no_e2e and host_buf is not None:
        # (a) the pipelined restore: batches packed on the replica's stream and
        # unpacked on the receiver's stream as soon as each is packed, so both
        # directions of the host link work at once; one re-send round
        bs = fr.Plan(src, cfg.chunk_bytes, n_batches=args.batches)
        bd = fr.Plan(dst, cfg.chunk_bytes, n_batches=args.batches)
        s_src, s_dst = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)

        def restore_step():
            # both fingerprint tables come out of the restore's own sweeps
            fr.fr_restore_fp(bs.handle, bd.handle, host_buf, 1, mism, nmis, tab_s, tab_d, s_src, s_dst)
            fr.fr_diff(tab_s, tab_d, C, div, ndiv, s_dst)
            s_dst.synchronize()
            return int(nmis.item()), int(ndiv.item())  # the step's result, read on the host

        def restore_step_unfused():
            fr.fr_fingerprint(bs.handle, tab_s, s_src)
            fr.fr_restore(bs.handle, bd.handle, host_buf, 1, mism, nmis, s_src, s_dst)
            fr.fr_fingerprint(bd.handle, tab_d, s_dst)
            fr.fr_diff(tab_s, tab_d, C, div, ndiv, s_dst)
            s_dst.synchronize()
            return int(nmis.item()), int(ndiv.item())

        def sample(fn):
            """Per-step wall times of `fn` (each step ends by reading its result on
            the host): (mean, median, best, the last step's result)."""
            fn()
            barrier()
            torch.cuda.synchronize()
            ts, res = [], None
            for _ in range(args.e2e_steps):
                t0 = time.perf_counter()
                res = fn()
                ts.append(time.perf_counter() - t0)
            torch.cuda.synchronize()
            return (max_over_ranks(sum(ts) / len(ts), dev), max_over_ranks(statistics.median(ts), dev),
                    max_over_ranks(min(ts), dev), res)

        t_e2e, med_e2e, best_e2e, e2e_found = sample(restore_step)
        # (b) for comparison: the same restore with separate fingerprint sweeps
        t_unfused, med_unfused, best_unfused, _ = sample(restore_step_unfused)
        # (c) for comparison: whole-buffer pack, then whole-buffer unpack
        t_serial, med_serial, best_serial, _ = sample(lambda: step(buf=host_buf, sync_counts=True))
        # (d) the bound: the host link's copy engines moving P/2 bytes each way
        # at once (64 MiB pieces, two streams, disjoint halves of the buffers)
        half, piece = P // 2, 64 << 20

        def link_step():
            for o in range(0, half, piece):
                n = min(piece, half - o)
                with torch.cuda.stream(s_src):
                    host_buf[o:o + n].copy_(packed[o:o + n], non_blocking=True)
                with torch.cuda.stream(s_dst):
                    packed[half + o:half + o + n].copy_(host_buf[half + o:half + o + n], non_blocking=True)
            torch.cuda.synchronize()

        link_step()
        t_links = []
        for _ in range(5):  # the host link's rate varies from call to call
            t0 = time.perf_counter()
            link_step()
            t_links.append(time.perf_counter() - t0)
        t_link = min(t_links)
        link_gbs = half / t_link / 1e9
        restore_gbs = P / t_e2e / 1e9

        def ms(x):
            return round(x * 1e3, 2)
        e2e = {"value": round(sum_over_ranks(SWEEPS_PER_STEP * S / t_e2e / 1e9, dev), 2), "unit": "GB/s",
               "h2d_bytes_per_step": P, "d2h_bytes_per_step": P + 16, "ms_per_step": ms(t_e2e),
               "ms_median": ms(med_e2e), "ms_best": ms(best_e2e), "steps": args.e2e_steps,
               "value_median": round(sum_over_ranks(SWEEPS_PER_STEP * S / med_e2e / 1e9, dev), 2),
               "transfer": "pinned host buffer over NVLink-C2C; fr_restore_fp with %d batches, pack and unpack "
                           "on two streams, both fingerprint tables from the same sweeps, 1 re-send round, then "
                           "fr_diff; no injected flips" % bs.n_batches,
               "unfused": {"value": round(sum_over_ranks(SWEEPS_PER_STEP * S / t_unfused / 1e9, dev), 2),
                           "ms_per_step": ms(t_unfused), "ms_median": ms(med_unfused), "ms_best": ms(best_unfused),
                           "how": "fr_fingerprint, fr_restore, fr_fingerprint, fr_diff"},
               "found": {"mismatching_chunks": e2e_found[0], "diverged_chunks": e2e_found[1]},
               "link": {"copy_engines_each_way_gbs": round(link_gbs, 1),
                        "copy_engines_median_gbs": round(half / statistics.median(t_links) / 1e9, 1),
                        "restore_each_way_gbs": round(restore_gbs, 1), "frac": round(restore_gbs / link_gbs, 4),
                        "frac_median": round((P / med_e2e) / (half / statistics.median(t_links)), 4),
                        "how": "cudaMemcpyAsync of P/2 bytes device->host and P/2 host->device at once, 64 MiB "
                               "pieces on two streams, pinned host memory, best and median of 5; the restore "
                               "moves P each way with the sweep kernels' own loads and stores over the same "
                               "link, which is not bound to the copy engines' rate (frac > 1 when they are "
                               "slower)"},
               "serial": {"value": round(sum_over_ranks(SWEEPS_PER_STEP * S / t_serial / 1e9, dev), 2),
                          "ms_per_step": ms(t_serial), "ms_median": ms(med_serial), "ms_best": ms(best_serial),
                          "how": "fr_pack to the host buffer, then fr_unpack_verify from it, with the flips"}}
        bs.close()
        bd.close()
        del host_buf, bs, bd

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(cfg, src, args.cpu_sample_gb)

    # the other workloads, one at a time, with this state's buffers freed first
    workloads = None
    if ws == 1 and args.workloads:
        plan_s.close()
        plan_d.close()
        del src, dst, packed, tab_s, tab_d, plan_s, plan_d, step, fused_step
        gc.collect()
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
        held = torch.cuda.memory_allocated(dev)
        if held > (1 << 30):
            raise RuntimeError("%d bytes of the headline workload are still held" % held)
        workloads = time_workloads([w for w in args.workloads.split(",") if w], dev, args.workload_reps, local)

    if rank == 0:
        out = {"metric": METRIC, "value": round(value, 1), "unit": "GB/s", "n_gpus": ws, "steps": args.steps,
               "warmup": args.warmup, "ms_per_step": round(ms_step, 3), "higher_is_better": True,
               "scaling": "weak", "vs_baseline": None, "dtype": "u8",
               "data": "synthetic (seeded; shapes of the named model shard)",
               "config": {"workload": args.config, "state_bytes": S, "chunk_bytes": cfg.chunk_bytes,
                          "n_chunks": C, "packed_bytes": P, "header_pad_bytes": H,
                          "faults": {"nan": int(nan_pos.size), "bit_flips": int(flips.size)},
                          "found": {"mismatching_chunks": n_mis, "diverged_chunks": n_div},
                          "l2": "inputs larger than L2 (state %.1f GB vs 129 MB L2); no flush" % (S / 1e9),
                          "parallelism": "replicas only (%d independent rank%s)" % (ws, "s" if ws > 1 else ""),
                          "value_def": "4 sweeps x state bytes / step time"},
               "calls": calls, "roofline": roofline, "fused_step": fused, "graph_step": graph, "e2e": e2e,
               "cpu_baseline": cpu, "workloads": workloads,
               "gpu_launches": launches_per_step * args.steps, "clocks": clk}
        print(json.dumps(out))
    if workloads is None:
        plan_s.close()
        plan_d.close()


def time_workloads(names, dev, reps, gpu_index, warmup=3):
    """Per-call times of fingerprint, pack, unpack_verify and diff on each named
    workload: the state is generated, its faults injected, every call timed
    `reps` times with CUDA events on the launching stream after `warmup`
    untimed calls, and everything freed before the next workload.  States
    smaller than 1 GiB have L2 (129 MB) flushed before every timed call (a
    256 MiB write, then a 256 MiB read that evicts the written lines); larger
    ones stream far more than L2 holds."""
    import torch

    from paper_2509_03047_gb300 import flashrec as fr
    from paper_2509_03047_gb300 import synth

    peak, peak_kind = measured_peak()
    stream = torch.cuda.current_stream()
    flush_buf = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    flush_read = torch.zeros(256 << 20, dtype=torch.uint8, device=dev)
    flush_out = torch.empty(1, dtype=torch.uint8, device=dev)

    def flush_l2(i):
        # write 256 MiB (twice the L2), then read another 256 MiB: the read
        # evicts the written lines, so their write-back to HBM is done before
        # the timed call starts and the call finds an L2 of clean, unrelated
        # lines
        flush_buf.fill_(i & 0xFF)
        torch.amax(flush_read, dim=0, keepdim=True, out=flush_out)
    clocks = ClockSampler(gpu_index)
    clocks.start()
    out = {"peak_gbs": peak, "peak_source": peak_kind, "reps": reps, "warmup": warmup}
    for name in names:
        t_setup = time.perf_counter()
        cfg = synth.get_config(name)
        src = synth.make_state(cfg, dev)
        nan_pos = synth.inject_nonfinite(cfg, src)
        dst = [torch.empty_like(t) for t in src]
        ps, pd = fr.Plan(src, cfg.chunk_bytes), fr.Plan(dst, cfg.chunk_bytes)
        S, C, P = ps.state_bytes, ps.n_chunks, ps.packed_bytes
        packed, tab_s, tab_d = ps.new_packed(), ps.new_table(), pd.new_table()
        mism = torch.empty(max(C, 1), dtype=torch.int32, device=dev)
        nmis = torch.empty(1, dtype=torch.int64, device=dev)
        div = torch.empty(max(C, 1), dtype=torch.int32, device=dev)
        ndiv = torch.empty(1, dtype=torch.int64, device=dev)
        flush = S < (1 << 30)
        torch.cuda.synchronize()
        t_setup = time.perf_counter() - t_setup

        def timed(fn, cold=flush):
            for _ in range(warmup):
                fn()
            evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                   for _ in range(reps)]
            for i, (a, b) in enumerate(evs):
                if cold:
                    flush_l2(i)
                a.record(stream)
                fn()
                b.record(stream)
            torch.cuda.synchronize()
            return sorted(a.elapsed_time(b) for a, b in evs)

        def f_fp(s=stream):
            fr.fr_fingerprint(ps.handle, tab_s, s)

        def f_pack(s=stream):
            fr.fr_pack(ps.handle, packed, s)

        def f_unpack(s=stream):
            fr.fr_unpack_verify(pd.handle, packed, mism, nmis, s)

        def graph_ms(fn, n=10):
            """Per-call device time of n back-to-back calls captured in one CUDA
            graph and replayed: no host time between the kernels."""
            gs = torch.cuda.Stream(device=dev)
            gs.wait_stream(stream)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=gs):
                for _ in range(n):
                    fn(gs)
            for _ in range(warmup):
                g.replay()
            ts = []
            for _ in range(reps):
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(stream)
                g.replay()
                b.record(stream)
                torch.cuda.synchronize()
                ts.append(a.elapsed_time(b) / n)
            del g
            return statistics.median(ts)

        t_fp = timed(f_fp)
        t_pack = timed(f_pack)
        flips = synth.flip_positions(P, cfg.flips, cfg.seed)
        synth.apply_flips(packed, flips)
        t_unpack = timed(f_unpack)
        # small states: also back to back with L2 left as the previous call
        # left it (the state, or most of it, then stays in the 129 MB L2), as
        # launched from Python and as replayed from a CUDA graph
        warm = {k: (statistics.median(timed(f, cold=False)), graph_ms(f))
                for k, f in (("fingerprint", f_fp), ("pack", f_pack), ("unpack_verify", f_unpack))} if flush else {}
        fr.fr_fingerprint(pd.handle, tab_d, stream)
        t_diff = timed(lambda: fr.fr_diff(tab_s, tab_d, C, div, ndiv, stream))
        found = {"mismatching_chunks": int(nmis.item()), "diverged_chunks": int(ndiv.item())}
        alg = {"fingerprint": S + 16 * C, "pack": S + P, "unpack_verify": P + S + 4 * C}
        calls = {}
        for k, ts in (("fingerprint", t_fp), ("pack", t_pack), ("unpack_verify", t_unpack)):
            med, best = statistics.median(ts), ts[0]
            calls[k] = {"ms_median": round(med, 4), "ms_best": round(best, 4),
                        "ms_mean": round(sum(ts) / len(ts), 4),
                        "state_gbs": round(S / (med * 1e-3) / 1e9, 1), "alg_bytes": alg[k],
                        "achieved_gbs": round(alg[k] / (med * 1e-3) / 1e9, 1),
                        "frac": round(alg[k] / (med * 1e-3) / 1e9 / peak, 4),
                        "frac_best": round(alg[k] / (best * 1e-3) / 1e9 / peak, 4)}
            if k in warm:
                calls[k]["ms_median_l2_resident"] = round(warm[k][0], 4)
                calls[k]["ms_l2_resident_graph"] = round(warm[k][1], 4)
        calls["diff"] = {"us_median": round(statistics.median(t_diff) * 1e3, 2), "alg_bytes": 32 * C}
        out[name] = {"state_bytes": S, "chunk_bytes": cfg.chunk_bytes, "n_chunks": C, "packed_bytes": P,
                     "tensors": len(src), "faults": {"nonfinite": int(nan_pos.size), "bit_flips": int(flips.size)},
                     "found": found, "calls": calls, "setup_s": round(t_setup, 1),
                     "l2": ("L2 flushed (256 MiB write, then 256 MiB read) before every timed call" if flush else
                            "state %.1f GB streams far more than the 129 MB L2; no flush" % (S / 1e9))}
        ps.close()
        pd.close()
        del src, dst, packed, tab_s, tab_d, mism, div, ps, pd
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
    out["clocks"] = clocks.stop()
    return out


# ---------------------------------------------------------------- the oracle

def oracle_sample(cfg, tensors_host, dtypes, steps=1):
    """Time the CPU oracle doing one restoration step on a host sample."""
    import oracle

    oracle.build()
    t0 = time.perf_counter()
    for _ in range(steps):
        fa = oracle.fingerprint(tensors_host, dtypes, cfg.chunk_bytes)
        pk = oracle.pack(tensors_host, dtypes, cfg.chunk_bytes)
        dst = [h.copy() for h in tensors_host]
        oracle.unpack_verify(dst, dtypes, cfg.chunk_bytes, pk)
        fb = oracle.fingerprint(dst, dtypes, cfg.chunk_bytes)
        oracle.diff(fa, fb)
    return (time.perf_counter() - t0) / steps


def sample_buffers(cfg, sample_gb):
    """Indices of a bounded, representative slice of the state's buffers:
    whole parameter groups (weight, master, m, v) in order, skipping any single
    parameter larger than the budget (the embedding), so the bf16/fp32 mix is
    the workload's; for the fragmented state, its first buffers."""
    limit = int(sample_gb * 1e9)
    specs = cfg.buffer_specs()
    idx, tot = [], 0
    group = 4 if cfg.kind == "adam" else 1
    for g in range(0, len(specs), group):
        nb = sum(b for _, _, b in specs[g:g + group])
        if nb > limit and not idx:
            continue
        if idx and tot + nb > limit:
            break
        idx += list(range(g, g + group))
        tot += nb
    return idx, tot


def cpu_baseline(cfg, tensors, sample_gb):
    import torch

    from paper_2509_03047_gb300 import flashrec as fr

    idx, tot = sample_buffers(cfg, sample_gb)
    host = [tensors[i].view(torch.uint8).reshape(-1).cpu().numpy() for i in idx]
    dts = [fr.fr_dtype_of(tensors[i]) for i in idx]
    dt = oracle_sample(cfg, host, dts)
    return {"value": round(SWEEPS_PER_STEP * tot / dt / 1e9, 4), "unit": "GB/s", "cores": 1,
            "host_cores": os.cpu_count(), "kind": "oracle",
            "sample": "%d buffers (%.2f GB) of the %s state, one restoration step (fingerprint, pack, "
                      "unpack_verify, fingerprint, diff), single thread, %.1f s" % (len(host), tot / 1e9,
                                                                                    cfg.name, dt)}


def run_reference(args):
    """The reference arm: the CPU oracle as it stands, on the host cores, on a
    bounded slice of the same workload generated on the host."""
    import torch

    import oracle
    from paper_2509_03047_gb300 import synth

    ws, rank, _ = dist_env()
    if rank != 0:
        return
    cfg = synth.get_config(args.config)
    # size each step's sample so that the W + K steps take about 100 s: the
    # oracle does one restoration step at roughly 0.1 GB of state per second
    per_step_s = max(1.0, 100.0 / max(1, args.steps + args.warmup))
    idx, tot = sample_buffers(cfg, min(args.cpu_sample_gb, 0.1 * per_step_s))
    if cfg.kind == "adam":
        sub = synth.Config(cfg.name, cfg.chunk_bytes, "adam", [cfg.shapes[i // 4] for i in idx[::4]],
                           seed=cfg.seed)
        state = synth.make_state(sub, "cpu")
    else:
        specs = cfg.buffer_specs()
        state = [torch.randn(specs[i][2] // 4, generator=synth._gen("cpu", cfg.seed, i, 9)) for i in idx]
    host = [t.view(torch.uint8).reshape(-1).numpy() for t in state]
    dts = [oracle.DT_BF16 if t.dtype == torch.bfloat16 else oracle.DT_F32 for t in state]
    for _ in range(args.warmup):
        oracle_sample(cfg, host, dts)
    times = [oracle_sample(cfg, host, dts) for _ in range(args.steps)]
    dt = sum(times) / len(times)
    value = SWEEPS_PER_STEP * tot / dt / 1e9
    cpu = {"value": round(value, 4), "unit": "GB/s", "cores": 1, "host_cores": os.cpu_count(), "kind": "oracle",
           "sample": "%d buffers (%.2f GB) of the %s state per step, single thread" % (len(host), tot / 1e9,
                                                                                     cfg.name)}
    out = {"impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": "GB/s", "n_gpus": ws,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(dt * 1e3, 1),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u8",
           "data": "synthetic (seeded; shapes of the named model shard)",
           "config": {"workload": args.config, "sample_bytes": tot, "chunk_bytes": cfg.chunk_bytes,
                      "value_def": "4 sweeps x state bytes / step time"},
           "cpu_baseline": cpu,
           "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
           "native_libraries": repo_libraries_loaded()}
    if any("libflashrec" in x for x in out["native_libraries"]):
        raise RuntimeError("the reference arm must not load the product library")
    print(json.dumps(out))


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["flashrec", "reference"], default="flashrec")
    ap.add_argument("--config", default=DEFAULT_CONFIG)
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--batches", type=int, default=16)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-sample-gb", type=float, default=1.0)
    ap.add_argument("--graph", action="store_true", help="also time the fused step replayed from a CUDA graph")
    ap.add_argument("--workloads", default="tiny,gpt2s,l8b_tp8,zero_frag,zero_frag4g",
                    help="comma-separated workloads timed per call after the headline step ('' for none)")
    ap.add_argument("--workload-reps", type=int, default=10)
    args = ap.parse_args(argv)
    if args.warmup < 3 and args.impl == "flashrec":
        ap.error("at least 3 warm-up steps")
    if args.impl == "reference":
        run_reference(args)
    else:
        run_flashrec(args)


if __name__ == "__main__":
    main()
