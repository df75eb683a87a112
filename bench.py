#!/usr/bin/env python3
"""Throughput of the GB300 routing engine: requests routed/s and (request, peer) lookups/s.

A step is one pass of the whole hot path over one batch: for the scale workload the anti-entropy delta on
every replica (device INSERT/DELETE) followed by the route of the batch (longest-prefix match against all
P trees + route decision); for the other workloads the route alone.  Inputs are seeded synthetic
stand-ins for the paper's few-shot-prompt workloads (see workload/wl.h), resident in HBM when the timed
region starts.  The JSON line also carries:
  kernels       every kernel launched in the timed region: launches, device ms per step (the library's kernel
                clock, CUDA events on the router stream), share, and its DRAM traffic per launch where an ncu
                capture of the same kernel source gave one;
  roofline      the delta kernel when it is the kernel with the most device time, else the route step's launches
                taken together, against the measured HBM copy bandwidth: achieved = algorithmic bytes per launch /
                device time.
                The delta kernel's algorithmic bytes are the oracle's per-op counters (input, walk, writes);
                the route step's are its compulsory bytes (request tokens and offsets read once, the match
                matrix and peers written once).  `traffic` is ncu's DRAM bytes for that kernel;
  route         the route step's compulsory-byte rate and its touched-byte rate (the oracle's per-(request,
                tree) walk bytes, which shared-prefix groups and L2 hits let the device exceed);
  e2e           the same metric through the host-pointer C-ABI calls (copies in the timed region);
  cpu_baseline  the CPU oracle on the host cores over a bounded sample of the same workload, on all cores and
                on one thread, with the CPU model.
--impl reference times that oracle as the reference arm.

Multi-GPU (torchrun): every rank holds all P trees and routes its own batch (requests [rank*B, (rank+1)*B)
of the request stream); no data-path collective.  Timing is max over ranks.
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
from concurrent.futures import ThreadPoolExecutor

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "requests routed/sec and (req,peer) lookups/sec at 1 GB300; % of HBM roofline"
WORKLOADS = {
    "cfg0": (0, "P=4 trees x 1,000 seqs (57 shared prefixes of 256-1,024 tokens), 4,096 requests/batch"),
    "cfg1": (1, "P=16 trees x 20,000 seqs (512 prefixes of 128-2,048 tokens), 65,536 requests/batch"),
    "cfg2": (2, "stale replicas: P=64 trees x 20,000 seqs (trees 1-63: -10%/+5%), 262,144 requests/batch"),
    "cfg3": (3, "long context: P=32 trees x 5,000 seqs (prefixes 4,096-32,768), 16,384 requests/batch"),
    "cfg4": (4, "scale + anti-entropy: P=256 trees x 100,000 seqs (10,000 prefixes of 128-4,096), "
                "1,048,576 requests/batch, 5% DELETE + 5% INSERT per replica per batch"),
}
L2_BYTES = 126 * 2**20
CSRC = os.path.join(ROOT, "paper_2606_17059_gb300", "csrc")
# Source file of each kernel (with internal.h, the layout they share): a DRAM-traffic figure holds only for
# the source it was captured on.
KERNEL_SOURCE = {
    "group_hash_kernel": "group_kernel.cu", "group_resolve_kernel": "group_kernel.cu",
    "group_resolve32_kernel": "group_kernel.cu", "route_kernel": "route_kernel.cu",
    "lane_kernel<true>": "route_kernel.cu", "lane_kernel<false>": "route_kernel.cu", "decide_kernel": "route_kernel.cu",
    "validate_kernel": "delta_kernel.cu", "init_ranges_kernel": "delta_kernel.cu", "delta_kernel": "delta_kernel.cu",
    "compact_kernel": "delta_kernel.cu", "compact_labels_kernel": "delta_kernel.cu",
    "refresh_views_kernel": "delta_kernel.cu", "set_tree_kernel": "delta_kernel.cu",
    "update_count_kernel": "update_kernel.cu", "update_scan_kernel": "update_kernel.cu",
    "update_scatter_kernel": "update_kernel.cu", "group_ranges_kernel": "group_kernel.cu",
    "group_place_kernel": "group_kernel.cu", "lru_walk_kernel": "lru_kernel.cu", "lru_stamp_kernel": "lru_kernel.cu",
    "lru_order_kernels": "lru_kernel.cu", "lru_count_kernel": "lru_kernel.cu", "lru_evict_kernel": "lru_kernel.cu",
    "lru_ops_kernel": "lru_kernel.cu", "hit_rate_kernel": "lru_kernel.cu", "room_kernel": "delta_kernel.cu",
}
# DRAM bytes per launch (ncu dram__bytes_read.sum + dram__bytes_write.sum) per workload and kernel, with the
# source hash of the capture and the profile summary that holds the command.  A figure whose source hash
# differs from the current source is not reported (the kernel changed since it was taken).
TRAFFIC: dict = {
    "cfg4": {k: dict(v, profile="profiles/traffic_workload4.md") for k, v in {
        "delta_kernel": {"bytes": 6722955162, "source": "e2ef36bc7089a1f9"},
        "validate_kernel": {"bytes": 99170202, "source": "e2ef36bc7089a1f9"},
        "compact_kernel": {"bytes": 10286514944, "source": "e2ef36bc7089a1f9"},
        "compact_labels_kernel": {"bytes": 24298933760, "source": "e2ef36bc7089a1f9"},
        "group_hash_kernel": {"bytes": 491484160, "source": "5dbd6a2a3cb8351d"},
        "group_resolve32_kernel": {"bytes": 9457201050, "source": "5dbd6a2a3cb8351d"},
        "group_ranges_kernel": {"bytes": 4005018, "source": "5dbd6a2a3cb8351d"},
        "group_place_kernel": {"bytes": 8143744, "source": "5dbd6a2a3cb8351d"},
        "lane_kernel<true>": {"bytes": 6151677824, "source": "73d5d75a48fec1cc"},
        "lane_kernel<false>": {"bytes": 16206268134, "source": "73d5d75a48fec1cc"},
    }.items()},
}


def source_hash(kernel: str) -> str | None:
    f = KERNEL_SOURCE.get(kernel)
    if f is None or not os.path.exists(os.path.join(CSRC, f)):
        return None
    h = hashlib.sha256()
    for name in (f, "internal.h"):
        with open(os.path.join(CSRC, name), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def traffic_of(workload: str, kernel: str):
    t = TRAFFIC.get(workload, {}).get(kernel)
    if t is None or t["source"] != source_hash(kernel):
        return None
    return t


def cpu_model() -> str:
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.strip().startswith("Model name:"):
                return ln.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for ln in f:
                if ln.lower().startswith("model name"):
                    return ln.split(":", 1)[1].strip()
    except Exception:
        pass
    return platform.processor() or platform.machine()


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi clock/throttle samples while the timed region runs."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu: int):
        self.gpu = gpu
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def dist_info():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def rank_requests(rank: int, B: int) -> tuple[int, int]:
    """Weak scaling: rank r routes requests [r*B, (r+1)*B) of the request stream (every rank holds all P
    trees and applies every delta; no data-path collective)."""
    return rank * B, (rank + 1) * B


def max_over_ranks(ms: float, dist, device=None) -> float:
    """Slowest rank's time: the job is done when every rank is."""
    if dist is None:
        return ms
    import torch
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---- workload setup ---------------------------------------------------------------------------------

def make_workload(cfg: int, trees: int = 0, batch: int = 0, seqs: int = 0):
    """The preset workload; trees/batch/seqs > 0 scale P, B and the sequences per tree down (smaller variants
    for profiling only)."""
    import workload as wl
    if not trees and not batch and not seqs:
        return wl.Workload(cfg)
    prm = wl.preset(cfg)
    if trees:
        prm["P"] = trees
    if batch:
        prm["B"] = batch
    if seqs:
        prm["n_seq"] = seqs
    return wl.Workload(params=prm, seed=wl.default_seed(cfg))


def build_trees(W, router, with_oracle: bool, n_threads: int):
    """Snapshots (and oracle trees) built on host threads, uploads in order on this thread."""
    import paper_2606_17059_gb300 as g
    import oracle as orc  # the oracle is used only by the CPU-baseline leg and the byte accounting
    P = W.P
    otrees = [None] * P

    def make(p):
        sl = W.tree(p)
        snap = g.p2p_snapshot_build(sl)
        if with_oracle:
            t = orc.OTree()
            t.insert_seqlist(sl)
            otrees[p] = t
        return snap

    with ThreadPoolExecutor(max_workers=n_threads) as ex:
        futs = [ex.submit(make, p) for p in range(P)]
        for p, f in enumerate(futs):
            snap = f.result()
            flat = g.FlatTree()
            g._load().p2p_snapshot_view(snap, flat)
            g._check(g._load().p2p_tree_upload(router.handle, p, flat), router.handle)
            g.p2p_snapshot_free(snap)
    router.sync()
    return otrees


def delta_to_device(d):
    import torch
    import workload as wl
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    return (dev(d.op), wl.SeqList(dev(d.seqs.seg_begin), dev(d.seqs.seg_off), dev(d.seqs.seg_len), dev(d.seqs.pool)),
            dev(d.peer_begin))


def delta_bytes(d) -> int:
    s = d.seqs
    return d.op.nbytes + s.seg_begin.nbytes + s.seg_off.nbytes + s.seg_len.nbytes + s.pool.nbytes + d.peer_begin.nbytes


# ---- the CPU oracle leg ------------------------------------------------------------------------------------

def oracle_sample(W, otrees, tok, off, load, alpha, target_s: float, n_threads: int, delta=None, B_total=None,
                  min_route_s: float = 3.0):
    """Times the oracle on a bounded prefix of the batch: n requests (and, with a delta, the matching share
    of every tree's ops).  Returns (requests/s, seconds, n, counters, description)."""
    import oracle as orc
    B = len(off) - 1
    pilot = min(B, 256)
    t0 = time.perf_counter()
    orc.route(otrees, tok, off[: pilot + 1], load, alpha, n_threads=n_threads)
    per_req = (time.perf_counter() - t0) / pilot
    n = int(min(B, max(pilot, target_s / max(per_req, 1e-9))))
    frac = n / float(B_total or B)
    t_delta = 0.0
    n_ops = 0
    if delta is not None:
        pb = delta.peer_begin
        t0 = time.perf_counter()

        def apply(p):
            lo = int(pb[p])
            k = int(math.ceil(frac * (int(pb[p + 1]) - lo)))
            otrees[p].apply_ops(delta.op, delta.seqs, lo, lo + k)
            return k

        with ThreadPoolExecutor(max_workers=n_threads) as ex:
            n_ops = sum(ex.map(apply, range(len(otrees))))
        t_delta = time.perf_counter() - t0
    # Route the sample; repeat passes over it until the route leg has run for min_route_s (stable timing).
    passes, t_route = 0, 0.0
    while True:
        t0 = time.perf_counter()
        m, peer, ctr = orc.route(otrees, tok, off[: n + 1], load, alpha, n_threads=n_threads)
        t_route += time.perf_counter() - t0
        passes += 1
        if t_route >= min(min_route_s, target_s) or passes >= 1000:
            break
    t_route /= passes
    secs = t_delta + t_route
    desc = f"first {n} of {B} requests of the batch x all {len(otrees)} trees (route timed over {passes} passes)"
    if delta is not None:
        desc += f", plus {n_ops} delta ops (the same {frac:.4%} share of every replica's delta)"
    return n / secs, secs, n, ctr, desc, (m, peer)


def oracle_single_thread(otrees, tok, off, load, alpha, target_s: float):
    """The oracle's route on one host thread over the first requests of the batch (about target_s of CPU
    work).  Returns (requests/s, requests)."""
    import oracle as orc
    B = len(off) - 1
    pilot = min(B, 16)
    t0 = time.perf_counter()
    orc.route(otrees, tok, off[: pilot + 1], load, alpha, n_threads=1)
    per_req = (time.perf_counter() - t0) / pilot
    n = int(min(B, max(pilot, target_s / max(per_req, 1e-9))))
    t0 = time.perf_counter()
    orc.route(otrees, tok, off[: n + 1], load, alpha, n_threads=1)
    return n / (time.perf_counter() - t0), n


def delta_op_bytes(otrees, delta, share: float, n_threads: int):
    """Mean algorithmic bytes per op of a delta (oracle counters: input, walk, writes) over the ops that
    follow the timed share in every tree (those trees have applied the ops before them).  Returns (bytes per
    op, ops counted)."""
    import oracle as orc
    pb = delta.peer_begin

    def count(p):
        lo, hi = int(pb[p]), int(pb[p + 1])
        a = lo + int(math.ceil(share * (hi - lo)))
        b = min(hi, a + max(1, (hi - lo) // 50))
        c = np.zeros(8, np.int64)
        if a < b:
            otrees[p].apply_ops_counted(delta.op, delta.seqs, c, a, b)
        return c

    with ThreadPoolExecutor(max_workers=n_threads) as ex:
        tot = sum(ex.map(count, range(len(otrees))))
    n_ops = int(tot[5] + tot[7])
    return (orc.delta_touched_bytes(tot) / n_ops if n_ops else 0.0), n_ops


# ---- our arm --------------------------------------------------------------------------------------------

def run_ours(args):
    import torch
    import paper_2606_17059_gb300 as g
    import oracle as orc

    ws, rank, local = dist_info()
    torch.cuda.set_device(local)
    dist = None
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    cfg, wdesc = WORKLOADS[args.workload]
    n_cpu = os.cpu_count() or 1
    t_setup = time.perf_counter()
    W = make_workload(cfg, args.trees, args.batch, args.seqs)
    P, B, alpha = W.P, W.B, W.alpha
    if args.trees or args.batch or args.seqs:
        wdesc += f" [scaled down: P={P}, B={B}, {W.params['n_seq']} sequences per tree]"
    router = g.Router(P)
    want_oracle = rank == 0 and not args.no_cpu_baseline
    otrees = build_trees(W, router, want_oracle, n_cpu)
    log(f"[rank {rank}] trees built in {time.perf_counter() - t_setup:.1f}s")
    # Requests of this rank, pinned on the host (for the end-to-end leg) and resident on the device.
    b0, b1 = rank_requests(rank, B)
    n_tok = W._lib.wl_requests_size(W._h, b0, b1, n_cpu)
    h_tok = torch.empty(n_tok, dtype=torch.int32, pin_memory=True)
    tok_np, off_np = W.requests(b0, b1, n_threads=n_cpu, out_tokens=h_tok.numpy())
    h_off = torch.from_numpy(off_np).pin_memory()
    d_tok = h_tok.cuda()
    d_off = h_off.cuda()
    load = W.load()
    out_match = torch.empty((B, P), dtype=torch.int32, device="cuda")
    out_peer = torch.empty(B, dtype=torch.int32, device="cuda")
    has_delta = W.params["delta_frac"] > 0
    n_steps = args.warmup + args.steps
    deltas = []
    if has_delta:
        t0 = time.perf_counter()
        for s in range(n_steps):
            W.delta_make(s, W.params["delta_frac"], W.params["delta_frac"], n_threads=n_cpu)
            d = W.delta(n_threads=n_cpu)
            deltas.append(delta_to_device(d))
            if s == 0:
                host_delta0 = d
        log(f"[rank {rank}] {n_steps} deltas staged in {time.perf_counter() - t0:.1f}s "
            f"({len(host_delta0.op)} ops, {delta_bytes(host_delta0) / 1e6:.0f} MB each)")
    flush = None
    if (n_tok * 4 + B * P * 4) < 2 * L2_BYTES:
        flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream()

    def step(s, ev):
        if has_delta:
            op, sl, pb = deltas[s]
            ev[0].record(stream)
            # The batch's grouping (it reads only the requests) runs alongside the delta kernel.
            g.p2p_route_prepare(router.handle, d_tok, n_tok, d_off, B)
            router.apply_delta(-1, op, sl, pb, on_device=True)
        ev[1].record(stream)
        g.p2p_route_batch(router.handle, d_tok, n_tok, d_off, B, load, alpha, out_match, out_peer)
        ev[2].record(stream)

    mk = lambda: [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    for s in range(args.warmup):
        step(s, mk())
        if flush is not None:
            flush.zero_()
    router.sync()
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.start()
    router.kernel_clock(True)  # per-kernel device time over the timed steps
    launches0 = router.launch_count()
    evs = []
    t_begin = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_begin.record(stream)
    for k in range(args.steps):
        ev = mk()
        step(args.warmup + k, ev)
        evs.append(ev)
        if flush is not None:
            # L2 flush between steps, outside the per-step events below.
            flush.zero_()
    t_end.record(stream)
    torch.cuda.synchronize()
    launches = router.launch_count() - launches0
    ktimes = router.kernel_times()
    router.kernel_clock(False)
    clk = clocks.stop()
    if dist:
        dist.barrier()
    router.sync()
    route_ms = [ev[1].elapsed_time(ev[2]) for ev in evs]
    delta_ms = [ev[0].elapsed_time(ev[1]) for ev in evs] if has_delta else [0.0] * len(evs)
    step_ms = [a + b for a, b in zip(route_ms, delta_ms)]
    total_ms = sum(step_ms) if flush is not None else t_begin.elapsed_time(t_end)
    total_ms = max_over_ranks(total_ms, dist, device="cuda")
    ms_per_step = total_ms / args.steps
    value = ws * B / (ms_per_step / 1e3)
    res = {}
    if rank == 0:
        gm = out_match.cpu().numpy()
        gp = out_peer.cpu().numpy()
        # ---- CPU oracle leg: baseline timing, touched-byte accounting and a parity spot check ----
        # (For the delta workload the oracle trees are the initial replicas, before the GPU's deltas: they
        # differ from the device trees by a few percent of their edges, so they give the byte accounting
        # but no parity check; the tests check that workload's parity.)
        ctr, n_acc, cpu, counted_share = None, 0, None, 0.0
        if want_oracle:
            rate, secs, n_acc, ctr, desc, (om, op) = oracle_sample(
                W, otrees, tok_np, off_np, load, alpha, args.cpu_seconds, n_cpu,
                delta=host_delta0 if has_delta else None, B_total=B)
            counted_share = n_acc / B
            rate1, n1 = oracle_single_thread(otrees, tok_np, off_np, load, alpha, args.cpu1_seconds)
            cpu = {"value": rate, "unit": "requests/s", "cores": n_cpu, "kind": "oracle",
                   "sample": desc + f" ({secs:.1f} s on {n_cpu} host threads)", "cpu_model": cpu_model(),
                   "single_thread": {"value": rate1, "unit": "requests/s", "cores": 1,
                                     "sample": f"route of the first {n1} requests x all {P} trees on one thread"}}
            if not has_delta:
                same = bool(np.array_equal(gm[:n_acc], om) and np.array_equal(gp[:n_acc], op))
                res["parity_spot_check"] = {"requests": n_acc, "bit_exact": same}
        hbm, src = peaks()
        peak_source = f"{src} (MEASURED_PEAKS.json hbm_gbs, STREAM-style copy)"
        route_avg_ms = statistics.mean(route_ms)
        tkey = None if (args.trees or args.batch or args.seqs) else args.workload
        # ---- every kernel of the timed region (the library's kernel clock) ----
        k_total = sum(ms for _, ms in ktimes.values()) or 1.0
        kernels = []
        for name, (n, ms) in sorted(ktimes.items(), key=lambda kv: -kv[1][1]):
            t = traffic_of(tkey, name) if tkey else None
            row = {"kernel": name, "launches_per_step": n / args.steps, "ms_per_step": ms / args.steps,
                   "ms_per_launch": ms / n, "share": ms / k_total, "traffic_per_launch": t["bytes"] if t else None}
            if t:
                row["dram_gbs"] = t["bytes"] / (ms / n / 1e3) / 1e9
                row["dram_frac"] = row["dram_gbs"] / hbm
                row["traffic_profile"] = t["profile"]
            kernels.append(row)
        kt = {k["kernel"]: k for k in kernels}
        # ---- the route step: compulsory bytes, and the oracle's touched bytes ----
        compulsory = 4 * int(n_tok) + 8 * (B + 1) + 4 * B * P + 4 * B
        route = {"kernels": [k for k in ("group_hash_kernel", "group_resolve_kernel", "group_resolve32_kernel",
                                         "group_ranges_kernel", "group_place_kernel", "route_kernel",
                                         "lane_kernel<true>", "lane_kernel<false>") if k in kt],
                 "ms": route_avg_ms, "compulsory_bytes": compulsory}
        # Device time of the route kernels (with p2p_route_prepare the grouping runs alongside the delta kernel,
        # outside the route span), the time the route's bytes are measured against.
        route_k_ms = sum(kt[k]["ms_per_step"] for k in route["kernels"]) or route_avg_ms
        route["kernel_ms"] = route_k_ms
        route["compulsory_gbs"] = compulsory / (route_k_ms / 1e3) / 1e9
        route["compulsory_frac"] = route["compulsory_gbs"] / hbm
        tr = [traffic_of(tkey, k) if tkey else None for k in route["kernels"]]
        route["traffic"] = sum(t["bytes"] for t in tr) if tr and all(tr) else None
        if route["traffic"]:
            route["dram_gbs"] = route["traffic"] / (route_k_ms / 1e3) / 1e9
        if ctr is not None:
            touched = orc.touched_bytes(ctr) / n_acc * B
            route.update({"touched_bytes": touched, "effective_gbs": touched / (route_k_ms / 1e3) / 1e9,
                          "touched_basis": f"oracle per-(request, tree) walk counters over {n_acc} requests x {P} "
                                           f"trees, scaled to {B} requests; groups and L2 hits let the device "
                                           "exceed HBM by this measure"})
        # ---- the roofline of the stage that takes the most time ----
        roof = None
        delta_k = kt.get("delta_kernel")
        # The kernel with the most device time per step.  With the grouping running alongside the delta kernel
        # (scale workload), the route kernels' device times overlap it and are not summed against it.
        dominant = max(kernels, key=lambda k: k["ms_per_step"])["kernel"] if kernels else None
        if delta_k and has_delta and dominant == "delta_kernel":
            n_ops_step = len(host_delta0.op)
            per_op, counted = delta_op_bytes(otrees, host_delta0, counted_share, n_cpu) if want_oracle else (0.0, 0)
            if counted:
                alg = per_op * n_ops_step / delta_k["launches_per_step"]
                achieved = alg / (delta_k["ms_per_launch"] / 1e3) / 1e9
                t = traffic_of(tkey, "delta_kernel") if tkey else None
                roof = {"bound": "hbm", "kernel": "delta_kernel", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                        "frac": achieved / hbm, "traffic": t["bytes"] if t else None, "peak_source": peak_source,
                        "bytes_per_launch": alg, "ms_per_launch": delta_k["ms_per_launch"],
                        "bytes_basis": f"oracle per-op counters (input, PrefixMatch walk, writes) over {counted} ops, "
                                       f"{per_op:.0f} B per op x {n_ops_step} ops per step"}
                if t:
                    roof["dram_gbs"] = t["bytes"] / (delta_k["ms_per_launch"] / 1e3) / 1e9
                    roof["dram_frac"] = roof["dram_gbs"] / hbm
        if roof is None:
            roof = {"bound": "hbm", "kernel": "route step: " + " + ".join(route["kernels"]),
                    "achieved": route["compulsory_gbs"], "peak": hbm, "unit": "GB/s", "frac": route["compulsory_frac"],
                    "traffic": route["traffic"], "peak_source": peak_source, "bytes_per_launch": compulsory,
                    "ms_per_launch": route_k_ms,
                    "bytes_basis": "compulsory bytes: request tokens and offsets read once, match matrix and peers "
                                   "written once (tree bytes left out: a lower bound)"}
            if route["traffic"]:
                roof["dram_gbs"] = route["dram_gbs"]
                roof["dram_frac"] = route["dram_gbs"] / hbm
        # ---- optional: the route decision with excluded peers on this batch's match matrix ----
        if not args.no_decide:
            res["decide"] = time_decide(router, out_match, load, alpha, P, B, hbm, src)
            res["route_decide"] = time_route_decide(router, d_tok, n_tok, d_off, B, load, alpha, P, route_avg_ms)
        # ---- end to end through the host-pointer C-ABI call ----
        e2e = run_e2e(args, W, router, tok_np, h_off.numpy(), load, alpha, has_delta, n_cpu)
        # ---- UpdateTrieEstimate / UpdateTrie of Algorithm 1 on the last timed batch (changes the trees) ----
        if not args.no_update:
            res["update_estimates"] = time_update(router, d_tok, d_off, out_peer, route_avg_ms)
        # ---- the own tree as an LRU cache trie (last: an LRU tree takes no more deltas) ----
        if not args.no_lru:
            res["lru"] = time_lru(router, d_tok, n_tok, d_off, B, out_match, out_peer)
        res.update({
            "metric": METRIC, "value": value, "unit": "requests/s", "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int32", "data": "synthetic",
            "config": {"workload": f"{args.workload}: {wdesc}", "P": P, "B_per_gpu": B, "alpha": alpha,
                       "tokens_per_batch": int(n_tok), "l2": "L2 flushed between steps" if flush is not None
                       else "inputs larger than L2 (request tokens stream from HBM each step)",
                       "step": "delta on every replica + route" if has_delta else "route"},
            "lookups_per_s": value * P, "route_ms": route_avg_ms,
            "delta_ms": statistics.mean(delta_ms) if has_delta else None,
            "roofline": roof, "route": route, "kernels": kernels, "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": int(launches), "clocks": clk,
        })
        print(json.dumps(res), flush=True)
    router.close()
    if dist:
        dist.destroy_process_group()


def time_update(router, d_tok, d_off, out_peer, route_ms):
    """One p2p_update_estimates call on the last timed batch (every request inserted into the tree it was routed
    to): CUDA events on the router stream around the call (the call waits for its work, so host-side steps
    between its launches count too), and the device time of its kernels from the kernel clock."""
    import torch
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    router.kernel_clock(True)
    t0 = time.perf_counter()
    e0.record(stream)
    n = router.update_estimates(d_tok, d_off, out_peer)
    e1.record(stream)
    torch.cuda.synchronize()
    wall = (time.perf_counter() - t0) * 1e3
    kt = router.kernel_times()
    router.kernel_clock(False)
    ms = e0.elapsed_time(e1)
    return {"inserted": n, "ms": ms, "wall_ms": wall, "kernel_ms": {k: v[1] for k, v in kt.items()},
            "route_plus_update_ms": route_ms + ms,
            "note": "one call after the timed steps on the last routed batch; the first call on fresh trees also "
                    "grows their arenas"}


def time_lru(router, d_tok, n_tok, d_off, B, out_match, out_peer):
    """The own tree (tree 0) as Section 2's LRU cache trie, after every other leg (an LRU tree takes no deltas):
    p2p_lru_enable (not timed), one p2p_lru_access of the whole batch at time 1 (each request's matched tokens
    stamped: Algorithm 1's cache hits), one p2p_lru_evict of 1% of the tree's own label tokens (EvictLRUTrie),
    and p2p_hit_rate of the routed batch (Section 5's expected hit rate).  Wall time around each call, which
    waits for its work (the hit rate is synchronized)."""
    import paper_2606_17059_gb300 as g
    import torch
    g.p2p_lru_enable(router.handle, 0)
    n_ev = max(1, router.stats(0)["label_tokens"] // 100)

    def timed(fn):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        out = fn()
        torch.cuda.synchronize()
        return out, (time.perf_counter() - t0) * 1e3

    m0 = torch.empty(B, dtype=torch.int32, device="cuda")
    _, acc_ms = timed(lambda: g.p2p_lru_access(router.handle, 0, d_tok, n_tok, d_off, B, 1, m0))
    evicted, ev_ms = timed(lambda: g.p2p_lru_evict(router.handle, 0, n_ev))
    hr = torch.empty(B, dtype=torch.float32, device="cuda")
    _, hr_ms = timed(lambda: g.p2p_hit_rate(router.handle, out_match, d_off, B, out_peer, hr))
    return {"tree": 0, "access_ms": acc_ms, "access_requests": B, "matched_tokens": int(m0.sum().item()),
            "evict_ms": ev_ms, "evicted_tokens": evicted, "hit_rate_ms": hr_ms,
            "mean_expected_hit_rate": float(hr.mean().item())}


def time_route_decide(router, d_tok, n_tok, d_off, B, load, alpha, P, route_ms, reps: int = 5):
    """p2p_route_batch_decide (the route with 5% of the trees excluded and the next-best target, decided in the
    walk kernels) against p2p_route_batch on the same batch: mean route time of `reps` calls of each, after
    one warm-up call, CUDA events on the router stream."""
    import torch
    import paper_2606_17059_gb300 as g
    ex = (np.random.default_rng(5).random(P) < 0.05).astype(np.uint8)
    m = torch.empty((B, P), dtype=torch.int32, device="cuda")
    peer = torch.empty(B, dtype=torch.int32, device="cuda")
    nxt = torch.empty(B, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream()

    def timed(fn):
        fn()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps

    plain = timed(lambda: g.p2p_route_batch(router.handle, d_tok, n_tok, d_off, B, load, alpha, m, peer))
    fused = timed(lambda: g.p2p_route_batch_decide(router.handle, d_tok, n_tok, d_off, B, load, alpha, ex, m, peer, nxt))
    return {"call": "p2p_route_batch_decide", "excluded": int(ex.sum()), "ms": fused, "plain_route_ms": plain,
            "cost": fused / plain - 1.0, "timed_step_route_ms": route_ms,
            "note": "back-to-back calls on the timed batch (no L2 flush between them)"}


def time_decide(router, out_match, load, alpha, P, B, hbm, src, reps: int = 10):
    """p2p_route_decide on the routed batch's match matrix with 5% of the trees excluded (seeded): mean
    time of `reps` calls after 3 warm-up calls (CUDA events on the router stream), and the read rate of
    the B x P int32 matrix against the HBM copy bandwidth."""
    import torch
    ex = (np.random.default_rng(5).random(P) < 0.05).astype(np.uint8)
    peer = torch.empty(B, dtype=torch.int32, device="cuda")
    nxt = torch.empty(B, dtype=torch.int32, device="cuda")
    for _ in range(3):
        router.decide(out_match, load, alpha, ex, peer, nxt)
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(reps):
        router.decide(out_match, load, alpha, ex, peer, nxt)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    gbs = B * P * 4 / (ms / 1e3) / 1e9
    return {"kernel": "decide_kernel", "ms": ms, "excluded": int(ex.sum()), "bytes_per_launch": B * P * 4,
            "achieved_gbs": gbs, "peak_gbs": hbm, "frac": gbs / hbm, "peak_source": f"{src} (MEASURED_PEAKS.json hbm_gbs)",
            "note": "the match matrix is read once per call; it may partly sit in L2 from the route step"}


def run_e2e(args, W, router, tok_np, off_np, load, alpha, has_delta, n_cpu):
    """The same metric through the host-pointer calls: request tokens/offsets copied in and match/peer
    copied out every step (and, for the delta workload, each step's delta from host memory)."""
    import torch
    import paper_2606_17059_gb300 as g
    B, P = len(off_np) - 1, W.P
    h_match = torch.empty((B, P), dtype=torch.int32, pin_memory=True).numpy()
    h_peer = torch.empty(B, dtype=torch.int32, pin_memory=True).numpy()
    k = max(1, min(args.steps, args.e2e_steps))
    hds = []
    if has_delta:
        import workload as wl
        base = args.warmup + args.steps

        def pinned(a):  # the delta's host arrays in pinned memory, as a serving process would keep them
            t = torch.empty(a.shape, dtype=getattr(torch, a.dtype.name), pin_memory=True).numpy()
            t[...] = a
            return t

        for s in range(k + 1):
            W.delta_make(base + s, W.params["delta_frac"], W.params["delta_frac"], n_threads=n_cpu)
            d = W.delta(n_threads=n_cpu)
            sl = d.seqs
            hds.append(type(d)(pinned(d.op), wl.SeqList(pinned(sl.seg_begin), pinned(sl.seg_off), pinned(sl.seg_len),
                                                        pinned(sl.pool)), pinned(d.peer_begin)))

    def one(i):
        if has_delta:
            d = hds[i]
            router.apply_delta(-1, d.op, d.seqs, d.peer_begin)
        g.p2p_route_batch_host(router.handle, tok_np, off_np, B, load, alpha, h_match, h_peer)

    one(0)  # warm
    t0 = time.perf_counter()
    for i in range(1, k + 1):
        one(i)
    secs = time.perf_counter() - t0
    h2d = tok_np.nbytes + off_np.nbytes + 4 * P
    if has_delta:
        h2d += delta_bytes(hds[1])
    d2h = h_match.nbytes + h_peer.nbytes
    return {"value": k * B / secs, "unit": "requests/s", "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "steps": k, "host_link_gbs": (h2d + d2h) * k / secs / 1e9,
            "host_buffers": "pinned",
            "call": "p2p_tree_apply_delta (host arrays) + p2p_route_batch_host" if has_delta else "p2p_route_batch_host"}


# ---- reference arm: the CPU oracle as it stands -------------------------------------------------------------

def run_reference(args):
    ws, rank, _ = dist_info()
    if rank != 0:
        return
    import oracle as orc
    cfg, wdesc = WORKLOADS[args.workload]
    n_cpu = os.cpu_count() or 1
    W = make_workload(cfg, args.trees, args.batch, args.seqs)
    P, B, alpha = W.P, W.B, W.alpha
    otrees = orc.build_trees([W.tree(p) for p in range(P)], n_threads=n_cpu)
    has_delta = W.params["delta_frac"] > 0
    b_sample = min(B, args.ref_requests)
    tok, off = W.requests(0, b_sample, n_threads=n_cpu)
    load = W.load()
    times = []
    desc = ""
    for s in range(args.warmup + args.steps):
        d = None
        if has_delta:
            W.delta_make(s, W.params["delta_frac"], W.params["delta_frac"], n_threads=n_cpu)
            d = W.delta(n_threads=n_cpu)
        rate, secs, n, _, desc, _ = oracle_sample(W, otrees, tok, off, load, alpha, args.ref_seconds, n_cpu,
                                                  delta=d, B_total=B)
        if s >= args.warmup:
            times.append((n, secs))
    n_req = sum(n for n, _ in times)
    secs = sum(t for _, t in times)
    value = n_req / secs
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "requests/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * secs / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int32", "data": "synthetic",
        "config": {"workload": f"{args.workload}: {wdesc}", "P": P, "B_per_gpu": B, "alpha": alpha},
        "cpu_baseline": {"value": value, "unit": "requests/s", "cores": n_cpu, "kind": "oracle",
                         "sample": "per step: " + desc},
        "e2e": {"value": value, "unit": "requests/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default="cfg4", choices=sorted(WORKLOADS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="target CPU time of the oracle sample")
    ap.add_argument("--cpu1-seconds", type=float, default=4.0, help="target time of the single-thread oracle sample")
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--no-update", action="store_true",
                    help="skip the timing of p2p_update_estimates (UpdateTrieEstimate) on the last routed batch")
    ap.add_argument("--no-lru", action="store_true",
                    help="skip the timing of the LRU calls on the own tree (p2p_lru_access, p2p_lru_evict) and of "
                         "p2p_hit_rate after the other legs")
    ap.add_argument("--no-decide", action="store_true",
                    help="skip the timing of p2p_route_decide and p2p_route_batch_decide (excluded peers, next-best "
                         "target) on the routed batch")
    ap.add_argument("--ref-requests", type=int, default=65536)
    ap.add_argument("--ref-seconds", type=float, default=4.0, help="oracle time per reference step")
    ap.add_argument("--trees", type=int, default=0, help="override P (a scaled-down variant, not a bench line)")
    ap.add_argument("--batch", type=int, default=0, help="override B (a scaled-down variant, not a bench line)")
    ap.add_argument("--seqs", type=int, default=0,
                    help="override the sequences per tree (a scaled-down variant, not a bench line)")
    args = ap.parse_args()
    if args.warmup < 3:
        log("warmup < 3 is below the timing rules; using 3")
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
