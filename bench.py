#!/usr/bin/env python3
"""Benchmark of the per-step logit path (plan + replay + verify) on one GB300 per rank.

Workload (batched serving): B=16 trees, V=151,936, draft block L=16, N=64 planned nodes,
top-k 8, T=1, bf16 logits; target rows [16, 65, V] = the node's depth row + N(0, 0.7^2).
A step = tsb_plan_rows + tsb_replay_verify on one batch (4 kernel launches: the planner
streams each draft row once for its chunk statistics and top-K, then runs the frontier
kernel; then one grid holds the replay draws beside the verifier's target-row pre-pass, and
the verifier's walk follows). The same step as three calls (tsb_replay, then tsb_verify with
its own pre-pass) is timed among the ``variants``.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl tsb|reference]

Prints one JSON line (rank 0). ``value`` is the mean device time per step in microseconds
(lower is better), timed with CUDA events over exactly K steps after W warm-up steps, with
the inputs resident in HBM. Per-call durations (``per_kernel_us``, the roofline's kernel
time) come from a second pass over the first min(K, 300) of the same prepared steps with an
event between calls; events inside the timed region would serialise the kernels'
programmatic launches. Inputs rotate over several independent sets whose per-step
footprint together exceeds the L2 several times, so no step finds its rows in L2 from an
earlier step. ``e2e`` repeats the measurement through the same C ABI with host (pinned)
inputs: every step copies its draft and target rows to the device and its outputs back.
``timing`` adds per-step percentiles (a pass with an event between steps) and the same steps
replayed from one CUDA graph; ``other_workloads`` times the single-stream, corrected-drafter
(T = 0.6 and 1.0) and V = 128,256 workloads the same way; ``variants`` the paper's other
sampling and verification schemes. ``cpu_baseline`` and ``--impl reference`` time the CPU
oracle as it stands on the host's cores: whole steps (the B trees of a set) over a process
pool with one process per usable core, rank 0 only.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = dict(name="batched", B=16, V=151936, L=16, N=64, K=8, T=1.0, dtype="bf16", target_noise=0.7)
METRIC = "plan+replay+verify us/step and HBM GB/s (% of GB300 peak), V=151,936, N=64"
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 8000.0
L2_BYTES = 129 * 1024 * 1024
KERNELS = ("tsb_plan_rows", "tsb_replay_verify")
LAUNCHES_PER_STEP = {"tsb_plan_rows": 2, "tsb_replay_verify": 2}
KERNEL_SOURCES = {"tsb_plan_rows": ("k_plan.cu",), "tsb_replay_verify": ("k_verify.cu", "replay_body.cuh")}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=None)
    ap.add_argument("--impl", choices=("tsb", "reference"), default="tsb")
    ap.add_argument("--sets", type=int, default=8, help="independent input sets rotated across steps")
    ap.add_argument("--e2e-steps", type=int, default=40)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-variants", action="store_true", help="skip the other sampling / verification schemes")
    ap.add_argument("--variant-steps", type=int, default=300)
    ap.add_argument("--no-planners", action="store_true", help="skip the first-pass-only timings at N = 64 and 256")
    ap.add_argument("--no-pooled", action="store_true", help="skip the pooled-law step")
    ap.add_argument("--no-graph", action="store_true", help="skip the CUDA-graph replay timing")
    ap.add_argument("--no-presets", action="store_true",
                    help="skip the other workloads (single stream, corrected drafter at T 0.6 / 1.0, V = 128,256)")
    ap.add_argument("--sweep", action="store_true",
                    help="instead of the headline step: the budget sweep at scale (B=64, V=151,936, L=16, "
                         "N in --budgets, bf16 and fp32), one JSON line with us/step and HBM GB/s per (dtype, N)")
    ap.add_argument("--budgets", default="16,32,64,128,256")
    ap.add_argument("--workload", default="batched", choices=("batched", "batched128k"))
    args = ap.parse_args()
    if args.steps is None:
        args.steps = 2000 if args.impl == "tsb" else 8
    if args.warmup is None:
        args.warmup = 20 if args.impl == "tsb" else 1
    if args.warmup < 3 and args.impl == "tsb":
        args.warmup = 3
    return args


def workload(args):
    w = dict(WORKLOAD)
    if args.workload == "batched128k":
        w.update(name="batched128k", V=128256)
    return w


def config_of(w, args):
    """The workload as both arms state it (identical dicts for the same arguments)."""
    es = 2 if w["dtype"] == "bf16" else 4
    set_mb = (w["B"] * w["L"] + w["B"] * (w["N"] + 1)) * w["V"] * es / 1e6
    return {"workload": f"batched serving: B={w['B']}, V={w['V']}, L={w['L']}, N={w['N']}, K={w['K']}, "
                        f"T={w['T']}, {w['dtype']} logits, target = depth row + N(0,{w['target_noise']}^2)",
            "B": w["B"], "V": w["V"], "L": w["L"], "N": w["N"], "K": w["K"], "temperature": w["T"],
            "parallelism": f"replicas only, {args.gpus} x 1 GPU",
            "l2": f"inputs larger than L2: {args.sets} input sets rotated, {set_mb:.0f} MB of draft and target rows "
                  f"each ({args.sets * set_mb * 1e6 / L2_BYTES:.0f}x L2)"}


def measured_peak_hbm():
    try:
        with open(PEAKS_FILE) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def source_hash(names):
    h = hashlib.sha256()
    for name in names:
        with open(os.path.join(ROOT, "paper_2609_33652_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(kernel, workload_name):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on the current
    source of that kernel (profiles/ncu_traffic.txt lines: kernel workload src_hash bytes)."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.txt")
    if not os.path.exists(path):
        return None
    want = source_hash(KERNEL_SOURCES[kernel])
    with open(path) as f:
        for line in f:
            p = line.split()
            if len(p) >= 4 and not line.startswith("#") and p[0] == kernel and p[1] == workload_name and p[2] == want:
                return float(p[3])
    return None


class ClockSampler:
    """nvidia-smi clock / throttle-reason sampling while the timed region runs."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            time.sleep(0.15)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.06)
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()
                out = ""
            self.lines = [ln for ln in out.splitlines() if ln.strip()]

    def summary(self):
        sm, smax, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for ln in self.lines:
            p = [x.strip() for x in ln.split(",")]
            if len(p) < 9:
                continue
            try:
                sm.append(float(p[1]))
                smax.append(float(p[2]))
            except ValueError:
                continue
            for n, v in zip(names, p[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------------------
def build_sets(w, S, device, rank):
    import torch

    from paper_2609_33652_gb300 import synth, tsb

    sets = []
    for s in range(S):
        seed = 1003 + 100 * s + 10000 * rank
        draft = synth.draft_logits(w["B"], w["L"], w["V"], "planted", w["dtype"], seed, device=device)
        buf = tsb.TsbBuffers.allocate(w["B"], w["L"], w["N"], w["K"], w["V"], w["T"], device=device)
        tsb.tsb_row_stats(draft, w["T"], buf.stats, buf.ws)
        tsb.tsb_plan(buf.cfg, draft, buf.stats, buf.tree, buf.ws)
        target = synth.rows_from_depth(draft, buf.tree["depth"], w["target_noise"], seed + 1)
        torch.cuda.synchronize()
        if tsb.tsb_device_status(buf.ws) != 0:
            raise RuntimeError("device status set while preparing inputs")
        sets.append(dict(draft=draft, target=target, buf=buf,
                         child_off=buf.tree["child_off"].cpu().numpy()))
    return sets


def algorithmic_bytes(w, sets, out_len, out_nodes):
    """Per step: draft rows once (B*L*V*s) + target rows of the visited nodes; plus the q rows
    the verifier stages (visited nodes with children), reported separately."""
    es = 2 if w["dtype"] == "bf16" else 4
    row = w["V"] * es
    K = out_len.shape[0]
    S = len(sets)
    visited = out_len.sum(axis=1).astype(np.int64)  # root + accepted nodes per tree
    staged_q = np.zeros(K, dtype=np.int64)
    for k in range(K):
        off = sets[k % S]["child_off"]
        for b in range(out_len.shape[1]):
            n = int(out_len[k, b])
            nodes = [0] + [int(x) for x in out_nodes[k, b, :n - 1]]
            staged_q[k] += sum(1 for u in nodes if off[b, u + 1] > off[b, u])
    draft_bytes = w["B"] * w["L"] * row
    return draft_bytes, visited * row, staged_q * row, visited


# Other sampling / verification schemes of the paper on the same workload (Table 2 and Sec.
# 3.1): each runs eagerly like the headline step and is timed the same way (start and end
# events only), followed by an event-separated pass for its per-call times.
VARIANTS = (
    ("wor_rrs_three_calls", dict(together=False), False),
    ("mixed_replay_naive_verify", dict(replay="mixed", mode=2), False),
    ("first_pass_tokens_naive_verify", dict(replay="plan", mode=2), False),
    ("expand_prune_w10_wor_rrs", dict(width=10), False),
    ("top1_chain_naive_verify", dict(replay="plan", mode=2), True),
    ("sampled_chain_block_verify", dict(mode=1), True),
    ("wor_traversal_verify", dict(mode=3), False),
)


def run_variants(w, sets, device, steps=300, warmup=10):
    import torch

    from paper_2609_33652_gb300 import synth, tsb

    B, L, S = w["B"], w["L"], len(sets)
    chain_sets = []
    for i, st in enumerate(sets):  # K = 1 chains of min(N, L) nodes on the same draft rows
        buf = tsb.TsbBuffers.allocate(B, L, min(w["N"], L), 1, w["V"], w["T"], device=device)
        tsb.tsb_row_stats(st["draft"], w["T"], buf.stats, buf.ws)
        tsb.tsb_plan(buf.cfg, st["draft"], buf.stats, buf.tree, buf.ws)
        target = synth.rows_from_depth(st["draft"], buf.tree["depth"], w["target_noise"], 5000 + i)
        chain_sets.append(dict(draft=st["draft"], target=target, buf=buf))
    torch.cuda.synchronize()
    out = {}
    for name, opts, chain in VARIANTS:
        src = chain_sets if chain else sets
        olen = torch.empty(steps, B, dtype=torch.int32, device=device)
        otok = torch.empty(steps, B, L + 1, dtype=torch.int32, device=device)
        onod = torch.empty(steps, B, L, dtype=torch.int32, device=device)
        prep = [tsb.PreparedStep(src[k % S]["buf"], src[k % S]["draft"], src[k % S]["target"], 7_000_000 + k,
                                 out_tokens=otok[k], out_nodes=onod[k], out_len=olen[k], **opts)
                for k in range(steps)]
        for k in range(min(warmup, steps)):
            prep[k].run()
        torch.cuda.synchronize()
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0.record()
        for p in prep:
            p.run()
        t1.record()
        torch.cuda.synchronize()
        us = t0.elapsed_time(t1) * 1e3 / steps
        KA = min(steps, 100)
        names = [c[0] for c in prep[0].calls]
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(len(names) + 1)] for _ in range(KA)]
        for k in range(KA):
            prep[k].run(ev[k])
        torch.cuda.synchronize()
        for st in src:
            if tsb.tsb_device_status(st["buf"].ws) != 0:
                raise RuntimeError(f"device status bits set in variant {name}")
        calls = {n: round(statistics.mean(ev[k][i].elapsed_time(ev[k][i + 1]) * 1e3 for k in range(KA)), 3)
                 for i, n in enumerate(names)}
        out[name] = {"us_per_step": round(us, 3), "per_call_us": calls,
                     "mean_emitted_len": round(float(olen.float().mean().item()), 4), "steps": steps}
    return out


def run_planners(w, sets, device, steps=300, warmup=10, budgets=(64, 256), width=10):
    """The first pass alone (draft statistics + top-K + expansion) at two budgets: the max-heap
    planner against expand-then-prune with the given frontier width (App. B.3)."""
    import torch

    from paper_2609_33652_gb300 import tsb

    B, L, S = w["B"], w["L"], len(sets)
    out = {}
    for N in budgets:
        bufs = [tsb.TsbBuffers.allocate(B, L, N, w["K"], w["V"], w["T"], device=device) for _ in range(S)]
        for name, wd in (("max_heap", None), (f"expand_prune_w{width}", width)):
            prep = [tsb.PreparedStep(bufs[k % S], sets[k % S]["draft"], sets[k % S]["target"], 1, width=wd,
                                     plan_only=True) for k in range(steps)]
            for k in range(min(warmup, steps)):
                prep[k].run()
            torch.cuda.synchronize()
            t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            t0.record()
            for p in prep:
                p.run()
            t1.record()
            torch.cuda.synchronize()
            for bf in bufs:
                if tsb.tsb_device_status(bf.ws) != 0:
                    raise RuntimeError(f"device status bits set in planner {name}, N={N}")
            out[f"{name}_N{N}"] = round(t0.elapsed_time(t1) * 1e3 / steps, 3)
    return out


def run_pooled(w, sets, device, steps=300, warmup=10, P=16):
    """A step with pooled draft laws (pools of P tokens, as DFlash2's 16): tsb_row_stats +
    tsb_plan_pooled, tsb_replay_pooled, tsb_verify_pooled, on the same inputs."""
    import ctypes

    import torch

    from paper_2609_33652_gb300 import tsb

    lib = tsb.load()
    B, L, S = w["B"], w["L"], len(sets)
    bufs = [tsb.TsbBuffers.allocate(B, L, w["N"], w["K"], w["V"], w["T"], device=device) for _ in range(S)]
    pools = [torch.empty(B, L, P, dtype=torch.int32, device=device) for _ in range(S)]
    s = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    keep, steps_calls = [], []
    for k in range(steps):
        st, bf, pl = sets[k % S], bufs[k % S], pools[k % S]
        dd, dt, tr = tsb.logits_desc(st["draft"]), tsb.logits_desc(st["target"]), tsb.tree_struct(bf.tree)
        keep += [dd, dt, tr]
        sb, wb = bf.stats.numel() * 4, bf.ws.numel()
        seed = 9_000_000 + k
        steps_calls.append([
            (lib.tsb_row_stats, (ctypes.byref(dd), ctypes.c_float(w["T"]), ctypes.c_void_p(bf.stats.data_ptr()), sb,
                                 ctypes.c_void_p(bf.ws.data_ptr()), wb, s)),
            (lib.tsb_plan_pooled, (ctypes.byref(bf.cfg), P, ctypes.byref(dd), ctypes.c_void_p(bf.stats.data_ptr()), sb,
                                   ctypes.c_void_p(pl.data_ptr()), ctypes.byref(tr), ctypes.c_void_p(bf.ws.data_ptr()),
                                   wb, s)),
            (lib.tsb_replay_pooled, (ctypes.byref(bf.cfg), P, ctypes.byref(dd), None, ctypes.c_void_p(pl.data_ptr()),
                                     ctypes.byref(tr), seed, ctypes.c_void_p(bf.token.data_ptr()),
                                     ctypes.c_void_p(bf.ws.data_ptr()), wb, s)),
            (lib.tsb_verify_pooled, (ctypes.byref(bf.cfg), P, ctypes.byref(dt), ctypes.byref(dd), None,
                                     ctypes.c_void_p(pl.data_ptr()), ctypes.byref(tr),
                                     ctypes.c_void_p(bf.token.data_ptr()), seed,
                                     ctypes.c_void_p(bf.out_tokens.data_ptr()), ctypes.c_void_p(bf.out_nodes.data_ptr()),
                                     ctypes.c_void_p(bf.out_len.data_ptr()), ctypes.c_void_p(bf.ws.data_ptr()), wb,
                                     s)),
        ])

    def run(calls):
        for fn, args in calls:
            rc = fn(*args)
            if rc != 0:
                raise RuntimeError(f"pooled step failed with status {rc}")

    for k in range(min(warmup, steps)):
        run(steps_calls[k])
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record()
    for c in steps_calls:
        run(c)
    t1.record()
    torch.cuda.synchronize()
    for bf in bufs:
        if tsb.tsb_device_status(bf.ws) != 0:
            raise RuntimeError("device status bits set in the pooled step")
    lens = torch.stack([bf.out_len for bf in bufs]).float().mean().item()
    return {"us_per_step": round(t0.elapsed_time(t1) * 1e3 / steps, 3), "pool": P, "steps": steps,
            "mean_emitted_len_last_steps": round(lens, 4)}


PRESETS = (
    # name, workload, per-node q rows
    ("single_stream_B1_N32", dict(name="single", B=1, V=151936, L=16, N=32, K=8, T=1.0, dtype="bf16",
                                  target_noise=0.7), False),
    ("corrected_B1_N64_T0.6", dict(name="corrected", B=1, V=151936, L=16, N=64, K=8, T=0.6, dtype="bf16",
                                   target_noise=0.7), True),
    ("corrected_B1_N64_T1.0", dict(name="corrected", B=1, V=151936, L=16, N=64, K=8, T=1.0, dtype="bf16",
                                   target_noise=0.7), True),
    ("batched_B16_N64_V128256", dict(name="batched128k", B=16, V=128256, L=16, N=64, K=8, T=1.0, dtype="bf16",
                                     target_noise=0.7), False),
)


def run_presets(device, steps=300, warmup=10):
    """The other workloads of the benchmark (not bench lines): each rotates enough input sets
    that their rows exceed L2 three times, and is timed like the headline step (start and end
    events around the steps), with per-step percentiles. Algorithmic bytes: draft rows once,
    per-node q rows once, target rows of the visited nodes."""
    import torch

    from paper_2609_33652_gb300 import synth, tsb

    peak, _ = measured_peak_hbm()
    out = {}
    for name, w, per_node in PRESETS:
        es = 2 if w["dtype"] == "bf16" else 4
        row = w["V"] * es
        NN = w["N"] + 1
        set_bytes = (w["B"] * w["L"] + w["B"] * NN * (2 if per_node else 1)) * row
        S = max(2, int(np.ceil(3 * L2_BYTES / set_bytes)))
        sets = build_sets(w, S, device, 0)
        olen = torch.empty(steps, w["B"], dtype=torch.int32, device=device)
        prep = []
        for st_i, st in enumerate(sets):
            if per_node:
                st["qrows"] = synth.rows_from_depth(st["draft"], st["buf"].tree["depth"], 0.3, 7000 + st_i)
                st["qstats"] = torch.empty(tsb.tsb_stats_bytes(w["B"], NN, w["V"]) // 4, dtype=torch.float32,
                                           device=device)
                st["qidx"] = torch.arange(NN, dtype=torch.int32, device=device).repeat(w["B"], 1).contiguous()
        for k in range(steps + warmup):
            st = sets[k % S]
            extra = dict(qrows=st["qrows"], qstats=st["qstats"], qrow_of_node=st["qidx"]) if per_node else {}
            prep.append(tsb.PreparedStep(st["buf"], st["draft"], st["target"], 6_000_000 + k,
                                         out_len=olen[k - warmup] if k >= warmup else None, **extra))
        for p in prep[:warmup]:
            p.run()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for p in prep[warmup:]:
            p.run()
        b.record()
        torch.cuda.synchronize()
        us = a.elapsed_time(b) * 1e3 / steps
        pct = step_percentiles(prep[warmup:warmup + min(steps, 200)])
        for st in sets:
            if tsb.tsb_device_status(st["buf"].ws) != 0:
                raise RuntimeError(f"device status bits set in preset {name}")
        visited = float(olen.float().sum(dim=1).mean().item())
        nbytes = w["B"] * w["L"] * row + (w["B"] * NN * row if per_node else 0) + visited * row
        out[name] = {"us_per_step": round(us, 3), "per_step_us": pct, "hbm_gbs": round(nbytes / (us * 1e-6) / 1e9, 1),
                     "hbm_frac_of_measured": round(nbytes / (us * 1e-6) / 1e9 / peak, 4),
                     "algorithmic_bytes_per_step": round(nbytes),
                     "mean_emitted_len": round(float(olen.float().mean().item()), 4), "input_sets": S,
                     "steps": steps}
        del sets, prep
        torch.cuda.empty_cache()
    return out


def max_over_ranks(value: float, dist, device) -> float:
    """The largest of the ranks' values (every rank gets it): a job's time is its slowest
    replica's. ``device`` is where the process group's backend reduces (cuda for nccl)."""
    import torch

    t = torch.tensor([float(value)], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def run_tsb(args):
    import torch

    from paper_2609_33652_gb300 import tsb

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    w = workload(args)
    from paper_2609_33652_gb300 import build as libbuild

    libbuild.build()
    tsb.load()
    S = args.sets
    sets = build_sets(w, S, device, rank)
    K, W = args.steps, args.warmup
    B, L = w["B"], w["L"]
    out_tokens = torch.empty(K, B, L + 1, dtype=torch.int32, device=device)
    out_nodes = torch.empty(K, B, L, dtype=torch.int32, device=device)
    out_len = torch.empty(K, B, dtype=torch.int32, device=device)

    def prepared(k, seed, tgt_slot=True):
        st = sets[k % S]
        if tgt_slot:
            return tsb.PreparedStep(st["buf"], st["draft"], st["target"], seed, out_tokens=out_tokens[k],
                                    out_nodes=out_nodes[k], out_len=out_len[k])
        return tsb.PreparedStep(st["buf"], st["draft"], st["target"], seed)

    warm = [prepared(k, 900_000 + k, tgt_slot=False) for k in range(W)]
    steps = [prepared(k, 1 + k + 1_000_000 * rank) for k in range(K)]
    for p in warm:
        p.run()
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    # Timed region: only its start and end events, so consecutive kernels keep their
    # programmatic launch overlap (an event between two calls would serialise them).
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clocks:
        torch.cuda.synchronize()
        if dist is not None:
            dist.barrier()
        start.record()
        for k in range(K):
            steps[k].run()
        end.record()
        torch.cuda.synchronize()
        if dist is not None:
            dist.barrier()
    total_ms = start.elapsed_time(end)
    # Per-call durations: a second pass over the same prepared steps with an event before the
    # first call and after each call (on the launching stream).
    KA = min(K, 300)
    events = [[torch.cuda.Event(enable_timing=True) for _ in range(len(KERNELS) + 1)] for _ in range(KA)]
    for k in range(KA):
        steps[k].run(events[k])
    torch.cuda.synchronize()
    if dist is not None:
        total_ms = max_over_ranks(total_ms, dist, device)
    for st in sets:
        if tsb.tsb_device_status(st["buf"].ws) != 0:
            raise RuntimeError("device status bits set during the timed region")
    per_kernel = {n: [] for n in KERNELS}
    for k in range(KA):
        for i, n in enumerate(KERNELS):
            per_kernel[n].append(events[k][i].elapsed_time(events[k][i + 1]) * 1e3)
    kern_us = {n: statistics.mean(v) for n, v in per_kernel.items()}
    us_step = total_ms * 1e3 / K
    dist_us = step_percentiles(steps[:KA])
    graph_us = graph_step_us(w, sets, device) if not args.no_graph else None

    h_len = out_len.cpu().numpy()
    h_nodes = out_nodes.cpu().numpy()
    draft_bytes, target_bytes, q_bytes, visited = algorithmic_bytes(w, sets, h_len, h_nodes)
    step_bytes = draft_bytes + float(target_bytes.mean())
    hbm_gbs = step_bytes / (us_step * 1e-6) / 1e9
    peak, peak_kind = measured_peak_hbm()

    # roofline of the dominant kernel (largest share of the step)
    dom = max(kern_us, key=kern_us.get)
    C = (w["V"] + 255) // 256
    es = 2 if w["dtype"] == "bf16" else 4
    kernel_bytes = {
        "tsb_plan_rows": B * L * w["V"] * es + B * L * C * 8,
        "tsb_replay_verify": B * w["N"] * (C * 8) + float(target_bytes.mean()),
    }
    achieved = kernel_bytes[dom] / (kern_us[dom] * 1e-6) / 1e9
    roofline = {"bound": "hbm", "kernel": dom, "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4), "peak_source": f"{peak_kind} (MEASURED_PEAKS hbm_gbs copy)",
                "traffic": profiled_traffic(dom, w["name"]),
                "bytes_per_launch": float(kernel_bytes[dom])}
    per_kernel_gbs = {n: round(kernel_bytes[n] / (kern_us[n] * 1e-6) / 1e9, 1) for n in KERNELS}

    # end to end through the C ABI with pinned host buffers
    e2e = run_e2e(args, w, sets, device) if args.e2e_steps > 0 else None
    variants = run_variants(w, sets, device, steps=args.variant_steps) if not args.no_variants else None
    if variants is not None and not args.no_planners:
        variants["first_pass_us_per_call"] = run_planners(w, sets, device, steps=args.variant_steps)
    if variants is not None and not args.no_pooled:
        for P in (16, 64):  # DFlash2's pools of 16 and Domino's sparse pools of 64 (App. B.7)
            variants[f"pooled{P}_wor_rrs"] = run_pooled(w, sets, device, steps=args.variant_steps, P=P)

    presets = run_presets(device) if not args.no_presets else None

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, sets, seconds=12.0)

    rows_per_s = world * (B * L + float(visited.mean())) / (us_step * 1e-6)
    line = {
        "metric": METRIC, "value": round(us_step, 3), "unit": "us/step", "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": round(us_step / 1e3, 6), "higher_is_better": False, "scaling": "weak", "vs_baseline": None,
        "dtype": w["dtype"], "data": "synthetic (seeded; shapes and value distributions of the batched serving "
                                     "workload; no datasets or model weights)",
        "config": config_of(w, args),
        "timing": {"launch": "eager C-ABI calls with programmatic dependent launch, inputs resident in HBM; "
                             "start and end events only in the timed region",
                   "per_step_us": dist_us, "cuda_graph_us_per_step": graph_us,
                   "algorithmic_footprint_per_step_mb": round(step_bytes / 1e6, 1)},
        "hbm_gbs": round(hbm_gbs, 1), "hbm_frac_of_measured": round(hbm_gbs / peak, 4),
        "hbm_frac_of_nominal_8tbs": round(hbm_gbs / NOMINAL_HBM_GBS, 4),
        "algorithmic_bytes_per_step": round(step_bytes), "rows_per_s": round(rows_per_s, 1),
        "mean_emitted_len": round(float(h_len.mean()), 4),
        "per_kernel_us": {n: round(v, 3) for n, v in kern_us.items()},
        "per_kernel_gbs": per_kernel_gbs,
        "roofline": roofline,
        "gpu_launches": sum(LAUNCHES_PER_STEP.values()) * K,
        "clocks": clocks.summary(),
        "e2e": e2e,
        "variants": variants,
        "other_workloads": presets,
        "cpu_baseline": cpu,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()


def step_percentiles(prep):
    """Per-step device times (an event between consecutive steps, which serialises only the
    step boundary): p10, median and p90 in microseconds."""
    import torch

    ev = [torch.cuda.Event(enable_timing=True) for _ in range(len(prep) + 1)]
    ev[0].record()
    for k, p in enumerate(prep):
        p.run()
        ev[k + 1].record()
    torch.cuda.synchronize()
    d = np.array([ev[k].elapsed_time(ev[k + 1]) * 1e3 for k in range(len(prep))])
    return {"p10": round(float(np.percentile(d, 10)), 3), "median": round(float(np.median(d)), 3),
            "p90": round(float(np.percentile(d, 90)), 3), "steps": len(prep)}


def graph_step_us(w, sets, device, steps_per_graph=16, replays=20):
    """The same steps captured in one CUDA graph (steps_per_graph steps over the rotating input
    sets) and replayed: mean device time per step. None (with the reason) if capture fails."""
    import torch

    from paper_2609_33652_gb300 import tsb

    S = len(sets)
    stream = torch.cuda.Stream(device)
    try:
        prep = [tsb.PreparedStep(sets[k % S]["buf"], sets[k % S]["draft"], sets[k % S]["target"], 3_000_000 + k,
                                 stream=stream) for k in range(steps_per_graph)]
        with torch.cuda.stream(stream):
            for p in prep:  # warm-up on the capture stream (cluster choices cached, modules loaded)
                p.run()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream, capture_error_mode="relaxed"):
            for p in prep:
                p.run()
        torch.cuda.synchronize()
        g.replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            a.record()
            for _ in range(replays):
                g.replay()
            b.record()
        torch.cuda.synchronize()
        for st in sets:
            if tsb.tsb_device_status(st["buf"].ws) != 0:
                raise RuntimeError("device status bits set in the graph replays")
        return round(a.elapsed_time(b) * 1e3 / (replays * steps_per_graph), 3)
    except Exception as e:  # capture not possible here: report why
        torch.cuda.synchronize()
        return {"error": f"{type(e).__name__}: {e}"[:300]}


def bind_near_gpu(device):
    """Run the host side on the CPUs local to the GPU (as the kernel reports them for its PCI
    function), so that pinned buffers allocated afterwards sit in the near memory: a buffer
    on the far socket slows every host-to-device copy. Returns the CPU list, or None where
    the topology is not exposed (the affinity is then left alone)."""
    import torch

    try:
        pr = torch.cuda.get_device_properties(device)
        addr = f"{pr.pci_domain_id:04x}:{pr.pci_bus_id:02x}:{pr.pci_device_id:02x}.0"
        with open(f"/sys/bus/pci/devices/{addr}/local_cpulist") as f:
            spec = f.read().strip()
        cpus = set()
        for part in spec.split(","):
            lo, _, hi = part.partition("-")
            cpus.update(range(int(lo), int(hi or lo) + 1))
        cpus &= os.sched_getaffinity(0)
        if not cpus:
            return None
        os.sched_setaffinity(0, cpus)
        return spec
    except (AttributeError, OSError, ValueError):
        return None


def run_e2e(args, w, sets, device):
    import torch

    from paper_2609_33652_gb300 import tsb

    near = bind_near_gpu(device)
    S = len(sets)
    E = args.e2e_steps
    h_draft = [st["draft"].cpu().pin_memory() for st in sets]
    h_target = [st["target"].cpu().pin_memory() for st in sets]
    d_draft = torch.empty_like(sets[0]["draft"])
    d_target = torch.empty_like(sets[0]["target"])
    bufs = [st["buf"] for st in sets]
    B, L = w["B"], w["L"]
    h_tok = torch.empty(B, L + 1, dtype=torch.int32).pin_memory()
    h_len = torch.empty(B, dtype=torch.int32).pin_memory()
    preps = [tsb.PreparedStep(bufs[k % S], d_draft, d_target, 5_000_000 + k) for k in range(E + 3)]

    def one(k):
        d_draft.copy_(h_draft[k % S], non_blocking=True)
        d_target.copy_(h_target[k % S], non_blocking=True)
        preps[k].run()
        h_tok.copy_(bufs[k % S].out_tokens, non_blocking=True)
        h_len.copy_(bufs[k % S].out_len, non_blocking=True)

    for k in range(3):
        one(k)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for k in range(3, 3 + E):
        one(k)
    b.record()
    torch.cuda.synchronize()
    us = a.elapsed_time(b) * 1e3 / E
    es = sets[0]["draft"].element_size()
    h2d = (sets[0]["draft"].numel() + sets[0]["target"].numel()) * es
    d2h = h_tok.numel() * 4 + h_len.numel() * 4
    return {"value": round(us, 3), "unit": "us/step", "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "steps": E, "host_cpus": near}


# ---------------------------------------------------------------------------------------
_SHARED = {}  # worker side: set index -> (draft [B, L, V], target [B, N+1, V]) views of shared memory


def _pool_init(descs):
    """Worker start-up: attach the shared input sets and load the oracle."""
    from multiprocessing import shared_memory

    import oracle

    oracle.build()
    oracle._load()
    for i, (dn, ds, dd, tn, ts_, td) in enumerate(descs):
        a = shared_memory.SharedMemory(name=dn)
        b = shared_memory.SharedMemory(name=tn)
        _SHARED[i] = (np.ndarray(ds, dtype=dd, buffer=a.buf), np.ndarray(ts_, dtype=td, buffer=b.buf), a, b)


def _pool_tree(task):
    """One tree of the oracle in a worker: (workload, set, tree, seed) -> (seconds, flags)."""
    w, si, b, seed = task
    d, t = _SHARED[si][0], _SHARED[si][1]
    sec, _, flags = oracle_tree_step(w, d[b:b + 1], t[b:b + 1], seed)
    return sec, flags


def _pool_pid(_):
    return os.getpid()


class OraclePool:
    """Input sets in shared memory (draft rows and target rows, as the oracle reads them) and a
    spawn pool of n oracle processes attached to them (spawn: the parent may hold a CUDA
    context)."""

    def __init__(self, n, host_sets):
        import multiprocessing as mp
        from multiprocessing import shared_memory

        self.blocks, descs = [], []
        for d, t in host_sets:
            entry = []
            for arr in (d, t):
                shm = shared_memory.SharedMemory(create=True, size=arr.nbytes)
                np.ndarray(arr.shape, dtype=arr.dtype, buffer=shm.buf)[...] = arr
                self.blocks.append(shm)
                entry += [shm.name, arr.shape, arr.dtype.str]
            descs.append(tuple(entry))
        self.nsets = len(host_sets)
        self.pool = mp.get_context("spawn").Pool(n, initializer=_pool_init, initargs=(descs,))
        self.pool.map(_pool_pid, range(n))  # every worker has started and attached

    def steps(self, w, steps, seed0):
        """Whole steps: each runs the B trees of one set across the pool; returns the wall
        seconds of every step and the summed near-tie flags."""
        times, flags = [], {"trees": 0, "plan": 0, "replay_parents": 0, "replay_flagged": 0, "verify": 0}
        for k in range(steps):
            tasks = [(w, k % self.nsets, b, seed0 + k * w["B"] + b) for b in range(w["B"])]
            t0 = time.perf_counter()
            res = self.pool.map(_pool_tree, tasks, chunksize=1)
            times.append(time.perf_counter() - t0)
            for _, f in res:
                for key in flags:
                    flags[key] += f[key]
        return times, flags

    def close(self):
        self.pool.close()
        self.pool.join()
        for shm in self.blocks:
            shm.close()
            shm.unlink()


def host_sets(sets):
    """(draft, target) host arrays of each input set, in the oracle's layout."""
    from paper_2609_33652_gb300 import synth

    return [(synth.to_host(st["draft"].contiguous()), synth.to_host(st["target"].contiguous())) for st in sets]


def oracle_tree_step(w, draft_h, target_h, seed):
    """The CPU oracle on one tree: plan, replay, verify (RRS); returns its seconds, outputs and
    the near-tie flags of its decisions."""
    import oracle

    t0 = time.perf_counter()
    ref = oracle.plan(draft_h, w["T"], w["N"], w["K"], w["L"])
    tok, rex = oracle.replay(draft_h, w["T"], ref, seed)
    out = oracle.verify_rrs(target_h, draft_h, w["T"], ref, tok, seed, w["L"])
    t1 = time.perf_counter()
    # decisions the oracle flags as near ties (where a GPU result may differ, reading of the
    # 1e-6 band): planner pops per tree, Gumbel selections per parent, walk decisions per tree
    parents = int((np.diff(ref["child_off"], axis=1) > 0).sum())
    flags = {"trees": int(draft_h.shape[0]), "plan": int(ref["exempt"].sum()), "replay_parents": parents,
             "replay_flagged": int(rex.sum()), "verify": int(out["exempt"].sum())}
    return t1 - t0, out, flags


def cpu_baseline(w, sets, seconds=12.0):
    """The oracle as it stands on the host cores: whole steps (the B trees of a set across a
    pool of one process per usable core) for about ``seconds``, and single trees on one core."""
    cores = len(os.sched_getaffinity(0))
    hs = host_sets(sets[:2])
    pool = OraclePool(cores, hs)
    try:
        pool.steps(w, 1, 50)  # warm-up step
        t0 = time.perf_counter()
        times, flags = [], None
        while time.perf_counter() - t0 < seconds or not times:
            tt, ff = pool.steps(w, 1, 100 + len(times) * w["B"])
            times += tt
            flags = ff if flags is None else {k: flags[k] + ff[k] for k in flags}
    finally:
        pool.close()
    one = []
    t1 = time.perf_counter()
    while time.perf_counter() - t1 < seconds / 3 or not one:
        b = len(one) % w["B"]
        one.append(oracle_tree_step(w, hs[0][0][b:b + 1], hs[0][1][b:b + 1], 9000 + len(one))[0])
    return {"value": round(statistics.mean(times) * 1e6, 1), "unit": "us/step", "cores": cores, "kind": "oracle",
            "sample": f"{len(times)} whole steps (B={w['B']} trees of plan + replay + verify, spread over {cores} "
                      f"processes, one per usable core; inputs in shared memory); one core: {len(one)} single "
                      f"trees, {statistics.mean(one) * 1e6:.0f} us per tree",
            "one_core_us_per_tree": round(statistics.mean(one) * 1e6, 1),
            "near_tie_flags": flags}


def run_reference(args):
    """The CPU oracle as the reference arm: K timed steps of the B trees of the workload on the
    host's cores (a spawn pool, one process per usable core), after W warm-up steps; the number
    of timed steps is capped so the arm ends within a few minutes (``steps_run``)."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import torch

    import oracle
    from paper_2609_33652_gb300 import synth

    w = workload(args)
    K, W = args.steps, args.warmup
    cores = len(os.sched_getaffinity(0))
    sets = []
    for s_ in range(2):  # the bench's first two input sets, targets from the oracle's own plan
        seed = 1003 + 100 * s_
        draft = synth.draft_logits(w["B"], w["L"], w["V"], "planted", w["dtype"], seed, device="cpu")
        ref = oracle.plan(synth.to_host(draft), w["T"], w["N"], w["K"], w["L"])
        target = synth.rows_from_depth(draft, torch.from_numpy(ref["depth"]), w["target_noise"], seed + 1)
        sets.append({"draft": draft, "target": target})
    pool = OraclePool(cores, host_sets(sets))
    try:
        pool.steps(w, max(W, 1), 10)
        t_one = pool.steps(w, 1, 20)[0][0]
        budget = 150.0
        run_k = K if K * t_one <= budget else max(3, int(budget / t_one))
        times, _ = pool.steps(w, run_k, 1000)
    finally:
        pool.close()
    us = statistics.mean(times) * 1e6
    sample_txt = (f"{run_k} of the {K} requested steps, each the B={w['B']} trees of one input set (plan + replay + "
                  f"verify) over {cores} processes, one per usable core")
    line = {"impl": "reference", "metric": METRIC, "value": round(us, 1), "unit": "us/step", "n_gpus": args.gpus,
            "steps": K, "steps_run": run_k, "warmup": W, "ms_per_step": round(us / 1e3, 4), "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": config_of(w, args),
            "cpu_baseline": {"value": round(us, 1), "unit": "us/step", "cores": cores, "kind": "oracle",
                             "sample": sample_txt},
            "e2e": {"value": round(us, 1), "unit": "us/step", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_sweep(args):
    """Budget sweep at scale: B=64 trees, V=151,936, L=16, K=8, T=1, one plan + replay + verify
    (RRS) step per batch, for each dtype and budget N; each (dtype, N) rotates two input sets and
    is timed like the headline step (start and end events around K steps after W warm-up
    steps). Algorithmic bytes: draft rows once + the visited target rows."""
    import torch

    from paper_2609_33652_gb300 import build as libbuild
    from paper_2609_33652_gb300 import synth, tsb

    device = torch.device("cuda", 0)
    torch.cuda.set_device(device)
    libbuild.build()
    tsb.load()
    B, V, L, K, T = 64, 151936, 16, 8, 1.0
    peak, peak_kind = measured_peak_hbm()
    out = {}
    sampler = ClockSampler(0)
    sampler.__enter__()
    for dtype in ("bf16", "f32"):
        es = 2 if dtype == "bf16" else 4
        for N in [int(x) for x in args.budgets.split(",")]:
            sets = []
            for s_ in range(2):
                seed = 1004 + 100 * s_
                draft = synth.draft_logits(B, L, V, "planted", dtype, seed, device=device)
                buf = tsb.TsbBuffers.allocate(B, L, N, K, V, T, device=device)
                tsb.tsb_row_stats(draft, T, buf.stats, buf.ws)
                tsb.tsb_plan(buf.cfg, draft, buf.stats, buf.tree, buf.ws)
                target = synth.rows_from_depth(draft, buf.tree["depth"], 0.7, seed + 1)
                sets.append((draft, target, buf))
            torch.cuda.synchronize()
            olen = torch.empty(args.steps, B, dtype=torch.int32, device=device)
            prep = [tsb.PreparedStep(sets[k % 2][2], sets[k % 2][0], sets[k % 2][1], 1 + k, out_len=olen[k])
                    for k in range(args.steps)]
            warm = [tsb.PreparedStep(sets[k % 2][2], sets[k % 2][0], sets[k % 2][1], 500_000 + k)
                    for k in range(args.warmup)]
            for p_ in warm:
                p_.run()
            torch.cuda.synchronize()
            t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            t0.record()
            for p_ in prep:
                p_.run()
            t1.record()
            torch.cuda.synchronize()
            for _, _, bf in sets:
                if tsb.tsb_device_status(bf.ws) != 0:
                    raise RuntimeError(f"device status bits set in the sweep at {dtype}, N={N}")
            us = t0.elapsed_time(t1) * 1e3 / args.steps
            pct = step_percentiles(prep[:min(args.steps, 100)])
            visited = float(olen.float().sum(dim=1).mean().item())
            nbytes = B * L * V * es + visited * V * es
            out[f"{dtype}_N{N}"] = {"us_per_step": round(us, 3), "hbm_gbs": round(nbytes / (us * 1e-6) / 1e9, 1),
                                    "hbm_frac_of_measured": round(nbytes / (us * 1e-6) / 1e9 / peak, 4),
                                    "algorithmic_bytes_per_step": round(nbytes), "per_step_us": pct,
                                    "mean_emitted_len": round(float(olen.float().mean().item()), 4)}
            del sets, prep, warm
            torch.cuda.empty_cache()
    sampler.__exit__(None, None, None)
    print(json.dumps({"clocks": sampler.summary(), "metric": "budget sweep: plan+replay+verify us/step and HBM GB/s per N", "n_gpus": 1,
                      "steps": args.steps, "warmup": args.warmup, "higher_is_better": False,
                      "config": {"workload": "budget sweep at scale: B=64, V=151936, L=16, K=8, T=1.0, depth cap 16, "
                                             "target = depth row + N(0,0.7^2)", "B": B, "V": V, "L": L, "K": K,
                                 "l2": "two input sets rotated (every set is above the L2 size)",
                                 "peak_source": f"{peak_kind} (MEASURED_PEAKS hbm_gbs copy)"},
                      "data": "synthetic", "sweep": out}), flush=True)


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    elif args.sweep:
        run_sweep(args)
    else:
        run_tsb(args)


if __name__ == "__main__":
    main()
