#!/usr/bin/env python3
"""Benchmark of the DensityKV hot path on GB300: bank update + bank-reading attention.

Default workload: the Wan-14B-shaped stack (40 layers x 40 heads, d = 128, bf16,
4,680-token blocks, per-head budgets drawn from {2,340, 4,680, 9,360, 18,720}, window =
previous block, 4,680 queries).  One step = one generated block through the whole
model: in every layer, attention of the block's queries over [bank | window], then
admit, evict and commit of the block leaving the window (Sec. 3.4, Alg. 1 per layer,
each layer with its own prefix r*, Eq. 11), all through one handle of the C ABI
(libdkv.so) whose calls are single launches over all 1,600 heads.  Every layer and head
draws its own synthetic stream (synth.device, generated on the GPU before each step's
start event).  W warm-up steps start from empty banks; K steps are timed one by one with
CUDA events on the launching stream, a 256 MiB buffer written between them.

Metric: bank keys scored per second = sum over heads of (m_h + N) per update (every
bank key's projected growth and every candidate are scored) / step time; blocks/s =
model steps per second.

A one-layer workload (--workload wan13b_layer_h12 and the like) runs the single-layer
step with its ablation flags (policies, descriptor, RoPE re-zeroing, sequential
admission, repeated attention passes), CUDA graphs and the numpy input generator.

``--impl reference`` times the CPU oracle (oracle/, numpy float64) on the host cores,
each step a bounded sample of the same workload (one head at steady state).

Multi-GPU (torchrun): every rank runs its own independent rollout (an independent video
on a stack workload, an independent layer on a one-layer workload), so no collective
is on the data path; ranks meet only at the barriers around the timed region and in a
reduction of the elapsed time and the keys.
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

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "bank keys scored/s (update+attention)"
UNIT = "keys/s"
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "traffic.json")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# GB300's nominal dense bf16 tensor rate and HBM3e bandwidth: fractions are also given
# against these, beside the measured peaks above
NOMINAL_BF16_TFLOPS, NOMINAL_HBM_GBS = 2250.0, 8000.0


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="wan14b_headwise_l40h40",
                    help="a stack workload (L > 1) runs the whole model step on one handle; a one-layer "
                         "workload runs the single-layer step")
    ap.add_argument("--sync-heads", type=int, choices=[0, 1], default=1,
                    help="1: shared prefix per layer (Eq. 11, the method's default); 0: independent per-head "
                         "prefixes (App. E ablation)")
    ap.add_argument("--profile-steps", type=int, default=2,
                    help="stack run: steps after the timed region with every kernel timed (per-kernel roofline)")
    ap.add_argument("--score-mode", choices=["tensor", "fp32"], default="tensor")
    ap.add_argument("--order", choices=["score", "source"], default="score",
                    help="candidate order (policy ablation of Table 2(b); default: the method's)")
    ap.add_argument("--eviction", choices=["mandatory_densest", "densest", "mandatory_source"],
                    default="mandatory_densest", help="eviction rule (policy ablation)")
    ap.add_argument("--refresh-baselines", action="store_true", help="refresh b after every update (ablation)")
    ap.add_argument("--within-block", choices=["batch", "sequential"], default="batch",
                    help="sequential: within-block competition, one candidate per head at a time (ablation; "
                         "no graphs, no overlap, no e2e leg)")
    ap.add_argument("--attn-passes", type=int, default=1,
                    help="bank-reading attention passes per update (denoising passes; the update runs once)")
    ap.add_argument("--stack", action="store_true",
                    help="run a one-layer workload through the stack path (per-kernel roofline pass, "
                         "device-generated inputs)")
    ap.add_argument("--layers", type=int, default=0,
                    help="stack run: number of layers (default: the workload's; fewer for small profiling cases)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-schedule", choices=["overlap", "serial"], default="overlap",
                    help="stack run, end-to-end leg: copies beside the compute of the neighbouring steps, or "
                         "each step's copies before its compute")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--no-flush", action="store_true", help="do not flush L2 between steps")
    ap.add_argument("--heads", type=int, default=0, help="override the head count (profiling runs)")
    ap.add_argument("--no-overlap", action="store_true",
                    help="run attention and the update on one stream instead of overlapping them")
    ap.add_argument("--no-graphs", action="store_true",
                    help="launch every step directly instead of replaying a captured CUDA graph")
    ap.add_argument("--descriptor", choices=["k", "kv"], default="k",
                    help="retention descriptor: keys, or [K; V] (App. E ablation)")
    ap.add_argument("--rope", choices=["off", "interleaved", "half"], default="off",
                    help="blocks arrive rotated to their frames' temporal RoPE coordinates and admit "
                         "rotates them back to coordinate 0 (dkv_bank_admit_rope)")
    args = ap.parse_args()
    if args.within_block == "sequential":
        # the sequential path synchronises with its stream once per block: no graph capture
        args.no_graphs = args.no_overlap = args.no_e2e = True
        if args.rope != "off":
            ap.error("--rope applies to the batch admission path")
    return args


def update_pairs(hs, N, rmax):
    """Key-pair interactions the update's pair passes evaluate, summed over heads: scores
    m N (Eq. 6), crossings m rmax (Eqs. 8-9), the projection resumed from the last
    128-column snapshot m (r* mod 128) (Eq. C.2), survivor maintenance (m - e) e
    (Eq. C.4) and new baselines r* m' (Eq. 5); an empty bank only the last."""
    tot = 0
    for h in hs:
        m, r, e, m2 = h.occupancy_before, h.admitted, h.evicted, h.occupancy_after
        if m == 0:
            tot += r * m2
        else:
            tot += m * N + m * rmax + m * (r % 128) + (m - e) * e + r * m2
    return tot


def rotate_to_frames(K, t, theta, layout):
    """Input synthesis for --rope: keys as a backbone's local window holds them, each
    rotation pair turned by its token's temporal coordinate (z -> z e^{i t theta}),
    rounded to the key type.  Runs once before timing, with torch on the host."""
    import torch
    Kf = K.to(torch.float64)
    d = Kf.shape[-1]
    xi, yi = (slice(0, d, 2), slice(1, d, 2)) if layout == "interleaved" else (slice(0, d // 2), slice(d // 2, d))
    a = torch.as_tensor(t, dtype=torch.float64)[:, None] * torch.as_tensor(theta).to(torch.float64)[None, :]
    c, s_ = torch.cos(a), torch.sin(a)
    x, y = Kf[..., xi], Kf[..., yi]
    out = Kf.clone()
    out[..., xi] = x * c - y * s_
    out[..., yi] = x * s_ + y * c
    return out.to(K.dtype)


def dist_env():
    return int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("LOCAL_RANK", "0"))


def layer_of_rank(rank: int) -> int:
    """Weak scaling: each rank updates its own layer (layers are independent: separate
    banks, r* per layer), so ranks exchange nothing on the data path."""
    return rank


def reduce_over_ranks(total_ms: float, keys: float, world: int, device=None):
    """Whole-job figures: the slowest rank's time and the keys of all ranks."""
    if world <= 1:
        return total_ms, float(keys)
    import torch
    import torch.distributed as dist
    tt = torch.tensor([total_ms, keys], dtype=torch.float64, device=device)
    mx = tt.clone()
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    sm = tt.clone()
    dist.all_reduce(sm, op=dist.ReduceOp.SUM)
    return float(mx[0]), float(sm[1])


def reference_runs_on(rank: int) -> bool:
    """The reference arm (the oracle on the host) runs and prints on rank 0 only."""
    return rank == 0


# --------------------------------------------------------------------------- clocks
class ClockSampler:
    """Samples nvidia-smi clocks and throttle reasons while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, enabled: bool = True):
        self.proc = None
        self.path = os.path.join(tempfile.gettempdir(), f"dkv_clocks_{os.getpid()}.csv")
        self.idx = gpu_index
        if not enabled:
            return
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-i", str(gpu_index), "-lms", "200"], stdout=self.fh,
                                         stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        sm, mx, reasons = [], [], set()
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for name, v in zip(("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"),
                               parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        try:
            os.remove(self.path)
        except OSError:
            pass
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


# --------------------------------------------------------------------------- helpers
def numa_info(gpu_index: int):
    """NUMA nodes of this host and the GPU's own node (where the pinned buffers can live)."""
    info = {"host_nodes": None, "gpu_node": None}
    try:
        info["host_nodes"] = len([n for n in os.listdir("/sys/devices/system/node") if n.startswith("node")])
        bus = subprocess.run(["nvidia-smi", "--query-gpu=pci.bus_id", "--format=csv,noheader", "-i", str(gpu_index)],
                             capture_output=True, text=True, timeout=30).stdout.strip().lower()
        if bus.startswith("00000000:"):
            bus = "0000:" + bus[9:]
        with open(f"/sys/bus/pci/devices/{bus}/numa_node") as f:
            info["gpu_node"] = int(f.read().strip())
    except Exception:
        pass
    return info


def peaks():
    if os.path.exists(PEAKS_FILE):
        p = json.load(open(PEAKS_FILE))
        return p, "measured"
    return FALLBACK_PEAKS, "fallback"


def source_sha1(*names):
    h = hashlib.sha1()
    for n in names:
        with open(os.path.join(ROOT, "paper_2608_27922_gb300", "csrc", n), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def traffic_for(kernel: str, src_files, workload: str, heads: int):
    """DRAM bytes per launch of `kernel` on `workload` from the committed ncu summary, if
    the kernel's source is unchanged since the capture; a capture on fewer heads of the
    same workload is scaled to `heads` (each head's operands are read once per launch)."""
    if not os.path.exists(TRAFFIC_FILE):
        return None
    t = json.load(open(TRAFFIC_FILE)).get(f"{kernel}@{workload}")
    if not t or t.get("source_sha1") != source_sha1(*src_files):
        return None
    return t["bytes_per_launch"] * heads / t["heads_captured"]


def make_workload(name, world, heads=0):
    import synth
    over = {}
    if heads:
        over["H"] = heads
    wl = synth.get_workload(name, **over)
    if world > wl.L:
        wl = synth.get_workload(name, L=world, **over)
    return wl


class Inputs:
    """Host copies of the blocks and queries of steps [0, n) of one layer's rollout."""

    def __init__(self, wl, layer, n_steps):
        import synth
        self.wl = wl
        ro = synth.LayerRollout(wl, layer)
        need = set()
        for t in range(n_steps):
            for blk, _, _ in wl.window_parts(t):
                need.add(blk)
            b = wl.admitted_block(t)
            if b is not None:
                need.add(b)
        self.blocks = {b: ro.block(b) for b in sorted(need)}
        self.queries = [ro.queries(t) for t in range(n_steps)]

    def window(self, t, blocks, cat):
        """Window K/V of step t from the given block tensors (whole block: no copy)."""
        parts = self.wl.window_parts(t)
        if len(parts) == 1 and parts[0][1] == 0 and parts[0][2] == self.wl.N:
            return blocks[parts[0][0]]
        return (cat([blocks[b][0][:, s0:e0] for b, s0, e0 in parts]),
                cat([blocks[b][1][:, s0:e0] for b, s0, e0 in parts]))

    def window_is_block(self, t, b):
        parts = self.wl.window_parts(t)
        return len(parts) == 1 and parts[0] == (b, 0, self.wl.N)


# --------------------------------------------------------------------------- our arm
def run_ours(args):
    import torch

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    import __graft_entry__
    if rank == 0 or world == 1:
        __graft_entry__.build()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    from paper_2608_27922_gb300 import dkv

    wl = make_workload(args.workload, world, args.heads)
    layer = layer_of_rank(rank)
    W, K = args.warmup, args.steps
    n_total = W + K + (0 if args.no_e2e else K)
    inp = Inputs(wl, layer, n_total)
    bf = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    if args.rope != "off":
        import synth
        theta = synth.temporal_rope_theta(wl.d, layout_first=args.rope == "interleaved")
        inp.blocks = {b: (rotate_to_frames(torch.from_numpy(k).to(bf), wl.frame_coords(b), theta, args.rope).float()
                          .numpy(), v) for b, (k, v) in inp.blocks.items()}
        theta_d = torch.from_numpy(theta).to(dev)
        tco = {b: torch.from_numpy(wl.frame_coords(b)).to(dev) for b in inp.blocks}
        rope_kw = lambda b, tbuf=None: dict(
            t_coord=tco[b] if tbuf is None else tbuf, theta=theta_d,
            rope_layout={"interleaved": dkv.DKV_ROPE_INTERLEAVED, "half": dkv.DKV_ROPE_HALF}[args.rope])
    else:
        rope_kw = lambda b, tbuf=None: {}
    dblocks = {b: (torch.from_numpy(k).to(dev, bf), torch.from_numpy(v).to(dev, bf)) for b, (k, v) in inp.blocks.items()}
    dq = [torch.from_numpy(q).to(dev, bf) for q in inp.queries[:W + K]]
    cat1 = lambda xs: torch.cat(xs, dim=1).contiguous()
    dwin = [inp.window(t, dblocks, cat1) for t in range(W + K)]
    P = max(1, args.attn_passes)
    mode = dkv.DKV_SCORE_TENSOR if args.score_mode == "tensor" else dkv.DKV_SCORE_FP32
    policy = dict(order={"score": dkv.DKV_ORDER_SCORE, "source": dkv.DKV_ORDER_SOURCE}[args.order],
                  eviction={"mandatory_densest": dkv.DKV_EVICT_MANDATORY_DENSEST, "densest": dkv.DKV_EVICT_DENSEST,
                            "mandatory_source": dkv.DKV_EVICT_MANDATORY_SOURCE}[args.eviction],
                  refresh_baselines=int(args.refresh_baselines))
    if args.descriptor == "kv":   # [K; V] rows, sigma = sqrt(2d / 2)
        policy.update(descriptor=dkv.DKV_DESC_KV, sigma=float(wl.d) ** 0.5)
    bank = dkv.BankLayer(wl.H, wl.d, wl.budgets_of_layer(layer), wl.N, bf, score_mode=mode, device=dev,
                         **policy)
    bank.reset()
    out = torch.empty(wl.H, wl.Nq, wl.d, dtype=bf, device=dev)
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    side = torch.cuda.Stream(dev)

    def step(t, Q, KW, VW, KC, VC):
        b = wl.admitted_block(t)
        if args.no_overlap:
            for _ in range(P):
                bank.attend(Q, KW, VW, out=out)
            if b is not None:
                if args.within_block == "sequential":
                    bank.update_sequential(KC, VC, b)
                else:
                    bank.admit(KC, VC, b, **rope_kw(b))
                    bank.compress()
            return
        # attention, admit and evict only read the bank (the update is atomic from the
        # reader's side); with one attention pass per update attention starts once admit has
        # run, so the tensor-heavy score and crossing passes have the GPU to themselves and
        # attention fills the latency-bound evict phase (several passes: attention dominates
        # and starts at once); only the commit waits for attention
        cur = torch.cuda.current_stream(dev)
        late = P == 1
        if b is not None and late:
            bank.admit(KC, VC, b, stream=cur, **rope_kw(b))
        go = torch.cuda.Event()
        go.record(cur)
        side.wait_event(go)
        for _ in range(P):   # every denoising pass reads the bank; the update runs once
            bank.attend(Q, KW, VW, out=out, stream=side)
        done = torch.cuda.Event()
        done.record(side)
        if b is not None:
            if not late:
                bank.admit(KC, VC, b, stream=cur, **rope_kw(b))
            bank.evict(stream=cur)
        cur.wait_event(done)
        if b is not None:
            bank.commit(stream=cur)

    def device_step(t):
        kw, vw = dwin[t]
        b = wl.admitted_block(t)
        kc, vc = dblocks[b] if b is not None else (None, None)
        step(t, dq[t], kw, vw, kc, vc)

    for t in range(W):
        device_step(t)
    bank.sync()

    # ---- optional CUDA graphs: one per timed step, captured before the timed region
    # (each step reads its own input buffers; the bank state stays on the device, so the
    # graphs replay the exact same work in order)
    graphs = None
    if not args.no_graphs:
        # the attention launches' timing events are captured into the graphs (the other
        # kernels are only counted: events between them would cost the step ~1.5%)
        bank.set_timing(True, attention_only=True)
        graphs = []
        cap = torch.cuda.Stream(dev)
        cap.wait_stream(stream)
        with torch.cuda.stream(cap):
            for i in range(K):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=cap):
                    device_step(W + i)
                graphs.append(g)
        stream.wait_stream(cap)
        torch.cuda.synchronize()

    # ---- timed region: K steps, CUDA events on the launching stream, L2 flushed between steps
    clocks = ClockSampler(local, enabled=(not args.no_clocks) and rank == 0)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    if graphs is None:
        bank.set_timing(True)   # with graphs, the timing events were captured into them
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    keys = 0
    pairs = 0
    stats = []
    wall0 = time.perf_counter()
    for i in range(K):
        t = W + i
        if not args.no_flush:
            flush.fill_(float(i))
        ev[i][0].record(stream)
        if graphs is not None:
            graphs[i].replay()
        else:
            device_step(t)
        ev[i][1].record(stream)
        ev[i][1].synchronize()
        L, hs = bank.stats()
        if wl.admitted_block(t) is not None:
            keys += sum(h.occupancy_before + wl.N for h in hs)
            pairs += update_pairs(hs, wl.N, L.rmax)
        # occupancy_before is the bank this step's attention read
        stats.append((L.r_star, sum(h.evicted for h in hs), sum(h.mandatory for h in hs),
                      sum(h.occupancy_before for h in hs)))
    torch.cuda.synchronize()
    wall = time.perf_counter() - wall0
    ktimes = bank.kernel_times()
    bank.set_timing(False)
    step_ms = [a.elapsed_time(b) for a, b in ev]
    clk = clocks.stop()
    bank.sync()
    total_ms = sum(step_ms)
    total_ms_max, keys_all = reduce_over_ranks(total_ms, keys, world, dev)
    _, pairs_all = reduce_over_ranks(total_ms, pairs, world, dev)
    value = keys_all / (total_ms_max / 1e3)

    # ---- end to end through the C ABI with host buffers: H2D inputs, compute, D2H output.
    # Every step's queries and window K/V come from pinned host memory and its attention
    # output goes back to it.  The inputs are double-buffered: step i computes from one
    # device set while a second copy stream uploads step i + 1's inputs into the other
    # (the step's graph completes only once that upload has landed), as a serving loop
    # would; the first timed step uploads its own inputs first, the last prefetches
    # nothing, so every timed step's uploads fall inside the timed regions exactly once.
    # O is downloaded while the commit runs.
    e2e = None
    if not args.no_e2e:
        host_blocks = {b: (torch.from_numpy(k).to(bf).pin_memory(), torch.from_numpy(v).to(bf).pin_memory())
                       for b, (k, v) in inp.blocks.items()}
        host_q = [torch.from_numpy(q).to(bf).pin_memory() for q in inp.queries[W + K:]]
        cat_pin = lambda xs: torch.cat(xs, dim=1).contiguous().pin_memory()
        host_win = [inp.window(W + K + i, host_blocks, cat_pin) for i in range(K)]
        host_out = torch.empty(wl.H, wl.Nq, wl.d, dtype=bf).pin_memory()
        host_tco = {b: torch.from_numpy(wl.frame_coords(b)).pin_memory() for b in inp.blocks}
        win_lens = sorted({hw[0].shape[1] for hw in host_win})
        # two device input sets (allocated before any capture)
        sets = []
        for _ in range(2):
            kb = torch.empty(wl.H, wl.N, wl.d, dtype=bf, device=dev)
            sets.append({"q": torch.empty(wl.H, wl.Nq, wl.d, dtype=bf, device=dev), "k": kb, "v": torch.empty_like(kb),
                         "t": torch.empty(wl.N, dtype=torch.int32, device=dev),
                         "win": {n: (torch.empty(wl.H, n, wl.d, dtype=bf, device=dev),
                                     torch.empty(wl.H, n, wl.d, dtype=bf, device=dev)) for n in win_lens}})
        # input uploads and the O download: one copy stream (on this host a download beside
        # an upload slows the upload several-fold)
        pre_s = torch.cuda.Stream(dev)
        bank.set_timing(False)

        def inputs_of(i):
            """Device buffers of step i (set i % 2) and the host tensors that fill them."""
            t = W + K + i
            ab = wl.admitted_block(t)
            st = sets[i % 2]
            kw_h, vw_h = host_win[i]
            kw, vw = st["win"][kw_h.shape[1]]
            pairs = [(st["q"], host_q[i]), (kw, kw_h), (vw, vw_h)]
            if ab is not None and not inp.window_is_block(t, ab):
                pairs += [(st["k"], host_blocks[ab][0]), (st["v"], host_blocks[ab][1])]
                kc, vc = st["k"], st["v"]
            else:
                kc, vc = kw, vw   # the block leaving the window is the window block
            if ab is not None and args.rope != "off":   # the block's temporal coordinates
                pairs.append((st["t"], host_tco[ab]))
            return ab, st["q"], kw, vw, kc, vc, st["t"], pairs

        def upload(pairs, after):
            """Copies host -> device on the upload stream after event `after`; returns its
            completion event and the bytes copied."""
            pre_s.wait_event(after)
            with torch.cuda.stream(pre_s):
                for d_, h_ in pairs:
                    d_.copy_(h_, non_blocking=True)
            ev = torch.cuda.Event()
            ev.record(pre_s)
            return ev, sum(h_.numel() * h_.element_size() for _, h_ in pairs)

        def e2e_step(i):
            cur = torch.cuda.current_stream(dev)
            start = torch.cuda.Event()
            start.record(cur)
            ab, qbuf, kw, vw, kc, vc, tbuf, pairs = inputs_of(i)
            nbytes = 0
            if i == 0:   # nothing was prefetched for the first timed step
                ready, nbytes = upload(pairs, start)
                cur.wait_event(ready)
            pre_done = None
            if i + 1 < K:   # the next step's inputs, beside this step's compute
                pre_done, nb = upload(inputs_of(i + 1)[-1], start)
                nbytes += nb
            if args.no_overlap:
                for _ in range(P):
                    bank.attend(qbuf, kw, vw, out=out)
                host_out.copy_(out, non_blocking=True)
                if ab is not None:
                    bank.admit(kc, vc, ab, **rope_kw(ab, tbuf))
                    bank.compress()
            else:
                late = P == 1
                if ab is not None and late:
                    bank.admit(kc, vc, ab, stream=cur, **rope_kw(ab, tbuf))
                go = torch.cuda.Event()
                go.record(cur)
                side.wait_event(go)
                for _ in range(P):
                    bank.attend(qbuf, kw, vw, out=out, stream=side)
                att_done = torch.cuda.Event()
                att_done.record(side)
                if ab is not None:
                    if not late:
                        bank.admit(kc, vc, ab, stream=cur, **rope_kw(ab, tbuf))
                    bank.evict(stream=cur)
                pre_s.wait_event(att_done)   # same stream as the uploads: the copies take turns
                with torch.cuda.stream(pre_s):
                    host_out.copy_(out, non_blocking=True)
                o_done = torch.cuda.Event()
                o_done.record(pre_s)
                cur.wait_event(att_done)
                if ab is not None:
                    bank.commit(stream=cur)
                cur.wait_event(o_done)
            if pre_done is not None:
                cur.wait_event(pre_done)
            return nbytes

        e2e_graphs = None
        h2d_step = []
        if not args.no_graphs:
            # capture before the timed region (the bank state stays on the device, so the
            # graphs replay the exact same uploads, kernels and download in order)
            e2e_graphs = []
            cap = torch.cuda.Stream(dev)
            cap.wait_stream(stream)
            with torch.cuda.stream(cap):
                for i in range(K):
                    g = torch.cuda.CUDAGraph()
                    with torch.cuda.graph(g, stream=cap):
                        h2d_step.append(e2e_step(i))
                    e2e_graphs.append(g)
            stream.wait_stream(cap)
            torch.cuda.synchronize()
        e2e_keys = 0
        e2e_ms = 0.0
        e2e_step_ms = []
        h2d = d2h = 0
        for i in range(K):
            t = W + K + i
            if not args.no_flush:
                flush.fill_(float(i))
            s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            # as in the device leg, the step is enqueued behind the L2 flush, so the host's
            # graph launch overlaps the flush and the events bracket the step's own work
            s0.record(stream)
            if e2e_graphs is not None:
                e2e_graphs[i].replay()
                h2d_i = h2d_step[i]
            else:
                h2d_i = e2e_step(i)
            s1.record(stream)
            s1.synchronize()
            e2e_step_ms.append(s0.elapsed_time(s1))
            e2e_ms += e2e_step_ms[-1]
            L, hs = bank.stats()
            if wl.admitted_block(t) is not None:
                e2e_keys += sum(h.occupancy_before + wl.N for h in hs)
            h2d += h2d_i
            d2h += host_out.numel() * host_out.element_size()
        e2e_ms, e2e_keys = reduce_over_ranks(e2e_ms, e2e_keys, world, dev)
        e2e = {"value": e2e_keys / (e2e_ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d // K,
               "d2h_bytes_per_step": d2h // K, "ms_per_step": e2e_ms / K,
               "step_ms": {"min": min(e2e_step_ms), "median": statistics.median(e2e_step_ms),
                           "max": max(e2e_step_ms), "first": e2e_step_ms[0]},
               "copies": "pinned host buffers; inputs double-buffered and uploaded one step ahead on a copy "
                         "stream (every timed step's uploads inside the timed regions), O downloaded on the same "
                         "stream",
               "cuda_graphs": e2e_graphs is not None}

    # ---- roofline of the dominant kernel (largest share of the timed region)
    pk, pk_src = peaks()
    launches = sum(v[0] for v in ktimes.values())
    dom = max(ktimes.items(), key=lambda kv: kv[1][1])
    dom_name, (dom_n, dom_ms) = dom
    roof = None
    m_bank = statistics.mean([s[3] / wl.H for s in stats]) if stats else 0
    if dom_name.startswith("attend"):
        # 2 flops per multiply-add in Q K^T and in P V over (m + W) keys per query
        flops = 4.0 * wl.H * wl.Nq * (m_bank + wl.W) * wl.d
        achieved = flops / (dom_ms / dom_n / 1e3) / 1e12
        peak = float(pk["bf16_tflops"])
        roof = {"kernel": dom_name, "bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": achieved / peak, "peak_source": f"{pk_src} bf16 dense (burst)",
                "frac_of_nominal": achieved / NOMINAL_BF16_TFLOPS,
                "algorithmic_per_launch": {"flops": flops, "keys_per_query": m_bank + wl.W},
                "traffic": traffic_for(dom_name, ["k_tc_attn.cu", "tc_ptx.cuh"], wl.name, wl.H)}
    else:
        roof = {"kernel": dom_name, "bound": "tensor", "achieved": None, "peak": float(pk["bf16_tflops"]),
                "unit": "TFLOP/s", "frac": None, "traffic": None}
    # with graphs only the attention launches are timed (the others are counted): list timed kernels
    per_kernel = {k: {"launches": n, "avg_ms": ms / max(n, 1), "share": ms / max(sum(v[1] for v in ktimes.values()), 1e-9)}
                  for k, (n, ms) in sorted(ktimes.items(), key=lambda kv: -kv[1][1]) if ms > 0}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline_sample(wl, layer)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": W,
            "ms_per_step": total_ms_max / K, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16" if wl.dtype == "bf16" else "f32", "data": "synthetic",
            "config": {"workload": f"{wl.name}: {wl.L if world > 1 else 1} layer(s) x {wl.H} heads, d={wl.d}, "
                                   f"N={wl.N}, M={max(wl.budgets)}, W={wl.W}, Nq={wl.Nq}",
                       "score_mode": args.score_mode, "layers_per_gpu": 1,
                       "attn_passes_per_update": max(1, args.attn_passes),
                       "policy": {"order": args.order, "eviction": args.eviction,
                                  "refresh_baselines": bool(args.refresh_baselines),
                                  "within_block": args.within_block,
                                  "rope_rezero": args.rope, "descriptor": args.descriptor},
                       "streams": (("admit, then attention || evict" if P == 1 else "attention || admit + evict") + ", then commit")
                       if not args.no_overlap else "one stream",
                       "cuda_graphs": graphs is not None,
                       "l2": "flushed between timed steps (256 MiB write)" if not args.no_flush else "not flushed",
                       "parallelism": f"{world} independent layers, no collective" if world > 1 else "single layer"},
            "blocks_per_s": world * K / (total_ms_max / 1e3),
            "interaction_pairs_per_s": pairs_all / (total_ms_max / 1e3),
            "wall_s_timed": wall,
            "e2e": e2e, "gpu_launches": launches * world, "roofline": roof, "cpu_baseline": cpu,
            "clocks": clk, "per_kernel": per_kernel,
            "update": {"r_star": [s[0] for s in stats], "evicted": [s[1] for s in stats],
                       "mandatory": [s[2] for s in stats]},
        }
        print(json.dumps(line), flush=True)
    bank.close()
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


# --------------------------------------------------------------------------- oracle timing
def oracle_threads():
    for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
        if os.environ.get(k):
            return int(os.environ[k])
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def _oracle_head_setup(wl, layer, head):
    """Oracle bank of one head brought to steady state (untimed): updates until the bank
    reaches its budget."""
    import oracle
    import synth
    ro = synth.LayerRollout(wl, layer, heads=[head])
    ob = oracle.LayerBank.empty([wl.budgets[layer * wl.H + head]], wl.d)
    t = 0
    while True:
        b = wl.admitted_block(t)
        if b is not None:
            K, V = ro.block(b)
            oracle.update_layer(ob, K, V, b)
            if ob.heads[0].m >= ob.heads[0].M:
                return ro, ob, t + 1
        t += 1
        if t > 8:
            return ro, ob, t


def _oracle_step(wl, ro, ob, t):
    """One step of one head in the oracle: attention of all queries, then the update."""
    import oracle
    Q = ro.queries(t)
    Kw, Vw = ro.window(t)
    b = wl.admitted_block(t)
    K, V = ro.block(b)
    t0 = time.perf_counter()
    oracle.attend(ob.heads[0], Q[0], Kw[0], Vw[0])
    m = ob.heads[0].m
    oracle.update_layer(ob, K, V, b)
    return time.perf_counter() - t0, m + wl.N


def _oracle_steps(wl, ro, ob, t, n):
    """n consecutive steady-state steps of one head in the oracle: (seconds, keys scored)."""
    tot_s, tot_k = 0.0, 0
    for i in range(n):
        dt, k = _oracle_step(wl, ro, ob, t + i)
        tot_s += dt
        tot_k += k
    return tot_s, tot_k


CPU_SAMPLE_STEPS = 4         # single-layer workloads: steady-state steps of one head
CPU_SAMPLE_STACK = (3, 2)    # stacks: heads of layer 0, steady-state steps each


def cpu_baseline_sample(wl, layer):
    ro, ob, t = _oracle_head_setup(wl, layer, 0)
    dt, keys = _oracle_steps(wl, ro, ob, t, CPU_SAMPLE_STEPS)
    return {"value": keys / dt, "unit": UNIT, "cores": oracle_threads(), "kind": "oracle",
            "sample": f"1 head (of {wl.H}), {CPU_SAMPLE_STEPS} steady-state steps of {wl.name}: attention of "
                      f"{wl.Nq} queries + bank update each, {keys} keys scored in {dt:.2f} s (numpy float64)"}


def run_reference(args):
    rank, world, _ = dist_env()
    if not reference_runs_on(rank):
        return
    wl = make_workload(args.workload, 1)
    head = _stack_sample_heads(wl, 1)[0] if wl.L > 1 else 0
    ro, ob, t = _oracle_head_setup(wl, 0, head)
    for i in range(args.warmup):
        _oracle_step(wl, ro, ob, t)
        t += 1
    tot, keys = 0.0, 0
    for i in range(args.steps):
        dt, k = _oracle_step(wl, ro, ob, t)
        tot += dt
        keys += k
        t += 1
    value = keys / tot
    cpu = {"value": value, "unit": UNIT, "cores": oracle_threads(), "kind": "oracle",
           "sample": f"each step: head {head} of layer 0 (budget {wl.budgets[head]}; {wl.L} x {wl.H} heads in the "
                     f"workload) of {wl.name} at steady state, attention of {wl.Nq} queries + bank update "
                     f"(numpy float64)"}
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": f"{wl.name} (one head per step on the host CPU)"},
            "cpu_baseline": cpu,
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------- whole stacks
TENSOR_KERNELS = ("attend_tc", "score_tc", "cross_tc", "project_tc", "subtract_tc", "newbase_tc")
HBM_KERNELS = ("cand_norms", "sort_runs", "sort_rank", "rstar", "select", "commit")


def kernel_roofs(per_kernel, steps):
    """The per-kernel pass against its kernels' roofs: the timed kernels' time per step,
    the time they would take at their roofs (tensor kernels' algorithmic flops at the bf16
    peak, memory-bound kernels' algorithmic bytes at the HBM peak), and the ratio."""
    if not per_kernel or steps <= 0:
        return None
    per_step = lambda r: r["avg_ms"] * r["launches"] / steps
    t = sum(per_step(r) for r in per_kernel.values())
    at = sum(per_step(r) * r.get("frac_of_bf16_peak", r.get("frac_of_hbm_alg", 0.0)) for r in per_kernel.values())
    return {"ms_per_step": t, "at_roofs_ms": at, "frac": at / t if t > 0 else None}


def kernel_work(name, d, esize, N, Nq, W, layer_of_head, Ls, hs):
    """Algorithmic work of one launch of kernel `name` over every head of a handle in one
    update step, from the step's statistics (Ls per layer, hs per head).

    Tensor-core passes: flops, 2d per key pair (Eq. 2 through the MMA) and 4d per
    query-key pair of the attention:
      scores m N (Eq. 6), crossings m rmax (Eqs. 8-9), projection m (r* mod 128)
      (Eq. C.2 resumed from the last 128-column snapshot), survivor maintenance (m - e) e
      (Eq. C.4), new baselines r* m' (Eq. 5), attention Nq (m + W).
    Memory-bound kernels: (algorithmic bytes, bytes the kernel moves by design):
      candidate norms: read the candidate keys, write norms and extension rows;
      sort runs: read scores 4N, write run keys 8N; sort rank: read run keys 8N, write
      pi 4N (algorithmic: 12N per head over both phases, the sort's read of s and write of
      pi plus the key exchange), and by design also the copy of the candidates into pi
      order (key, norm, extension row read and written);
      r*: the crossing histogram (N + 2) and the feasibility bits;
      select: rho~, crossing index and mask, 12 m (algorithmic), plus the provenance
      read for ties and the slot lists written, 32 m (moved);
      commit: the admitted K and V rows read and written plus 20 B of metadata per
      admitted state (algorithmic); by design also the evicted keys copied out, the
      survivors' keys copied beside them (operands of Eq. C.4) and the extension rows."""
    rowb = d * esize
    tot_a = tot_m = 0.0
    for h, st in enumerate(hs):
        m, m2, r, e = st.occupancy_before, st.occupancy_after, st.admitted, st.evicted
        rmax = Ls[layer_of_head(h)].rmax
        live = m > 0
        if name == "attend_tc":
            tot_a += 4.0 * d * Nq * (m + W)
        elif name == "score_tc":
            tot_a += 2.0 * d * m * N if live else 0
        elif name == "cross_tc":
            tot_a += 2.0 * d * m * rmax if live else 0
        elif name == "project_tc":
            tot_a += 2.0 * d * m * (r % 128) if live else 0
        elif name == "subtract_tc":
            tot_a += 2.0 * d * (m - e) * e if live else 0
        elif name == "newbase_tc":
            tot_a += 2.0 * d * r * m2
        elif name == "cand_norms":
            tot_a += N * (rowb + 4 + 64)
            tot_m += N * (rowb + 4 + 64)
        elif name == "sort_runs":
            tot_a += 6.0 * N if live else 0
            tot_m += 12.0 * N if live else 0
        elif name == "sort_rank":
            tot_a += 6.0 * N if live else 0
            tot_m += (12.0 * N + 2.0 * N * (rowb + 68)) if live else 4.0 * N + 2.0 * N * (rowb + 68)
        elif name == "rstar":
            tot_a += 4.0 * (rmax + 2) + (rmax + 1) / 8.0 if live else 0
            tot_m += 4.0 * (rmax + 2) + (rmax + 1) / 8.0 if live else 0
        elif name == "select":
            tot_a += 12.0 * m if live and e > 0 else 0
            tot_m += 32.0 * m if live and e > 0 else 0
        elif name == "commit":
            tot_a += r * (4.0 * rowb + 20.0)
            ng = (m - e) if e > 0 else 0
            tot_m += r * (4.0 * rowb + 20.0 + 128.0) + e * (2.0 * rowb + 136.0) + ng * (2.0 * rowb + 136.0)
    if name in TENSOR_KERNELS:
        return tot_a
    return tot_a, tot_m


def run_stack(args):
    """Whole-stack throughput: every step is one generated block passing through all L
    layers of the model (L x H heads, per-head budgets): attention of the block's queries
    over [bank | window] in every layer, then admit, evict and commit of the block leaving
    the window (Alg. 1 per layer, each layer with its own prefix r*, Eq. 11), all through
    one handle whose calls are single launches over all L x H heads.  Every layer and
    head draws its own synthetic stream (synth.device, generated on the GPU between
    timed steps, outside the events)."""
    import torch
    from synth.device import StackRollout

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    import __graft_entry__
    if rank == 0 or world == 1:
        __graft_entry__.build()
    if world > 1:
        dist.barrier()
    from paper_2608_27922_gb300 import dkv

    over = {"H": args.heads} if args.heads else {}
    if args.layers:
        over["L"] = args.layers
    wl = synth_workload(args.workload, **over)
    if wl.window not in ("prev", "own"):
        raise SystemExit("the stack run takes whole-block windows (prev / own)")
    L, H, d, N, Nq = wl.L, wl.H, wl.d, wl.N, wl.Nq
    LH = L * H
    W_, K = args.warmup, args.steps
    bf = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    esize = 2 if wl.dtype == "bf16" else 4
    mode = dkv.DKV_SCORE_TENSOR if args.score_mode == "tensor" else dkv.DKV_SCORE_FP32
    sync = 0 if args.sync_heads == 0 else 1
    # weak scaling: each rank runs its own rollout (an independent video) of the whole stack
    gen = StackRollout(wl, device=dev, rank_seed=rank)
    bank = dkv.BankLayer(LH, d, list(wl.budgets), N, bf, score_mode=mode, device=dev, layer_heads=H,
                         sync_heads=sync)
    bank.reset()
    lay = lambda h: h // H
    out = torch.empty(LH, Nq, d, dtype=bf, device=dev)
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    side = torch.cuda.Stream(dev)
    stream = torch.cuda.current_stream(dev)

    def new_set():
        return {"q": torch.empty(LH, Nq, d, dtype=bf, device=dev), "k": torch.empty(LH, N, d, dtype=bf, device=dev),
                "v": torch.empty(LH, N, d, dtype=bf, device=dev)}

    gset = new_set()   # generated inputs of the device leg (and staging of the end-to-end leg)

    def generate(t, st):
        gen.queries(t, st["q"])
        gen.block(wl.window_block(t), st["k"], st["v"])

    def step(t, st, cur, serial=False, o=None):
        """Attention of step t over [bank | window] in every layer, then the update with
        the block leaving the window (= the window block for these workloads).  serial:
        everything on one stream (per-kernel timing).  o: the attention output buffer."""
        o = out if o is None else o
        b = wl.admitted_block(t)
        if b is not None:   # admit first: the score and crossing passes have the GPU alone
            bank.admit(st["k"], st["v"], b, stream=cur)
        att = cur if serial else side
        go = torch.cuda.Event()
        go.record(cur)
        att.wait_event(go)
        bank.attend(st["q"], st["k"], st["v"], out=o, stream=att)
        done = torch.cuda.Event()
        done.record(att)
        if b is not None:
            bank.evict(stream=cur)
        cur.wait_event(done)   # commit changes the bank attention reads
        if b is not None:
            bank.commit(stream=cur)
        return done

    def step_stats(t):
        if wl.admitted_block(t) is None:
            return None
        Ls = bank.layer_stats()
        _, hs = bank.stats()
        return Ls, hs

    for t in range(W_):
        generate(t, gset)
        step(t, gset, stream)
    torch.cuda.synchronize()
    bank.sync()

    # ---- timed region: K steps, each bracketed by CUDA events on the launching stream;
    # the step's inputs are generated on the device and the L2 flushed before the start event
    clocks = ClockSampler(local, enabled=(not args.no_clocks) and rank == 0)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    bank.set_timing(True, attention_only=True)   # live events around the attention launches only
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    keys = pairs = 0
    per_step = []
    wall0 = time.perf_counter()
    for i in range(K):
        t = W_ + i
        generate(t, gset)
        if not args.no_flush:
            flush.fill_(float(i))
        ev[i][0].record(stream)
        step(t, gset, stream)
        ev[i][1].record(stream)
        ev[i][1].synchronize()
        st = step_stats(t)
        if st is not None:
            Ls, hs = st
            keys += sum(h.occupancy_before + N for h in hs)
            pairs += sum(kernel_work(k, d, esize, N, Nq, wl.W, lay, Ls, hs) for k in TENSOR_KERNELS[1:]) / (2 * d)
            per_step.append({"r_star": [x.r_star for x in Ls], "evicted": sum(h.evicted for h in hs),
                             "admitted": sum(h.admitted for h in hs), "mandatory": sum(h.mandatory for h in hs),
                             "bank_keys": sum(h.occupancy_before for h in hs)})
    torch.cuda.synchronize()
    wall = time.perf_counter() - wall0
    clk = clocks.stop()
    ktimes = bank.kernel_times()
    bank.set_timing(False)
    bank.sync()
    step_ms = [a.elapsed_time(b) for a, b in ev]
    total_ms = sum(step_ms)
    total_ms_max, keys_all = reduce_over_ranks(total_ms, keys, world, dev)
    _, pairs_all = reduce_over_ranks(total_ms, pairs, world, dev)
    value = keys_all / (total_ms_max / 1e3)
    launches = sum(n for n, _ in ktimes.values())
    att_n, att_ms = ktimes.get("attend_tc", (0, 0.0))
    att_flops = statistics.mean(
        [4.0 * d * Nq * (s["bank_keys"] + LH * wl.W) for s in per_step]) if per_step else 0.0

    # ---- per-kernel pass (not part of the value): a few more steps with every kernel timed
    # by CUDA events on its stream, against its algorithmic work
    P = max(0, args.profile_steps)
    prof = {}
    bank.set_timing(True)
    t_next = W_ + K
    for i in range(P):
        t = t_next + i
        generate(t, gset)
        if not args.no_flush:
            flush.fill_(float(i))
        step(t, gset, stream, serial=True)
        torch.cuda.synchronize()
        st = step_stats(t)
        kt = bank.kernel_times()
        bank.set_timing(False)
        bank.set_timing(True)
        if st is None:
            continue
        Ls, hs = st
        for name, (n, ms) in kt.items():
            if n == 0 or ms <= 0:
                continue
            e = prof.setdefault(name, {"launches": 0, "ms": 0.0, "work": 0.0, "moved": 0.0})
            e["launches"] += n
            e["ms"] += ms
            if name in TENSOR_KERNELS:
                e["work"] += kernel_work(name, d, esize, N, Nq, wl.W, lay, Ls, hs)
            elif name in HBM_KERNELS:
                a, m_ = kernel_work(name, d, esize, N, Nq, wl.W, lay, Ls, hs)
                e["work"] += a
                e["moved"] += m_
    bank.set_timing(False)
    t_next += P
    pk, pk_src = peaks()
    tpeak, hpeak = float(pk["bf16_tflops"]), float(pk["hbm_gbs"])
    tot_prof = sum(e["ms"] for e in prof.values()) or 1.0
    per_kernel = {}
    for name, e in sorted(prof.items(), key=lambda kv: -kv[1]["ms"]):
        row = {"launches": e["launches"], "avg_ms": e["ms"] / e["launches"], "share": e["ms"] / tot_prof}
        if name in TENSOR_KERNELS:
            tf = e["work"] / (e["ms"] / 1e3) / 1e12
            row.update(tflops=tf, frac_of_bf16_peak=tf / tpeak, frac_of_bf16_nominal=tf / NOMINAL_BF16_TFLOPS)
        elif name in HBM_KERNELS:
            gbs = e["work"] / (e["ms"] / 1e3) / 1e9
            row.update(alg_gbs=gbs, frac_of_hbm_alg=gbs / hpeak, frac_of_hbm_alg_nominal=gbs / NOMINAL_HBM_GBS,
                       moved_gbs=e["moved"] / (e["ms"] / 1e3) / 1e9, frac_of_hbm_moved=e["moved"] / (e["ms"] / 1e3) / 1e9 / hpeak)
        per_kernel[name] = row

    # ---- end to end through the C ABI with host buffers: every step's queries and block K/V
    # come from pinned host memory and its attention output goes back to it.  Inputs and
    # outputs are double-buffered on the device, as a serving loop would pipeline them:
    # step i computes from one input set while a copy stream uploads step i + 1's inputs
    # into the other and a second copy stream downloads step i - 1's output; the step
    # completes only once both copies have landed.  The first timed step uploads its own
    # inputs first, the last one also downloads its own output after its attention, so
    # every step's uploads and its download fall inside the timed regions exactly once.
    # The host buffers of step i + 1 are written (generated on the device, copied down)
    # before step i starts.
    e2e = None
    if not args.no_e2e:
        hsets = [{k: torch.empty(v.shape, dtype=bf, pin_memory=True) for k, v in gset.items()} for _ in range(2)]
        dsets = [new_set(), new_set()]
        douts = [out, torch.empty_like(out)]
        host_outs = [torch.empty(LH, Nq, d, dtype=bf, pin_memory=True) for _ in range(2)]
        # one copy stream for both directions: on this host a download running beside an
        # upload slows the upload several-fold, so the copies take turns
        pre_s = torch.cuda.Stream(dev)
        in_bytes = sum(x.numel() * x.element_size() for x in hsets[0].values())
        out_bytes = out.numel() * out.element_size()

        # serial schedule: the download beside the upload (both directions at once, with the
        # GPU otherwise idle, move more bytes per second than one direction)
        dn_s = torch.cuda.Stream(dev) if args.e2e_schedule == "serial" else pre_s

        def download(i, after):
            dn_s.wait_event(after)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(dn_s)
            with torch.cuda.stream(dn_s):
                host_outs[i % 2].copy_(douts[i % 2], non_blocking=True)
            e1.record(dn_s)
            return e0, e1

        def fill_host(t, hs_):
            generate(t, gset)
            for k_ in hs_:
                hs_[k_].copy_(gset[k_], non_blocking=True)
            torch.cuda.synchronize()

        def upload(hs_, ds_, after):
            pre_s.wait_event(after)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(pre_s)
            with torch.cuda.stream(pre_s):
                for k_ in ds_:
                    ds_[k_].copy_(hs_[k_], non_blocking=True)
            e1.record(pre_s)
            return e0, e1

        base_t = t_next
        fill_host(base_t, hsets[0])
        e2e_ms, e2e_keys, up_ms, down_ms, up_b, down_b = 0.0, 0, [], [], 0, 0
        for i in range(K):
            t = base_t + i
            if i + 1 < K:
                fill_host(t + 1, hsets[(i + 1) % 2])
            if not args.no_flush:
                flush.fill_(float(i))
            s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            s0.record(stream)
            ups, downs = [], []
            serial = args.e2e_schedule == "serial"
            if i == 0 or serial:   # this step's own inputs first
                ups.append(upload(hsets[i % 2], dsets[i % 2], s0))
                up_b += in_bytes
            if i > 0:   # the previous step's output
                downs.append(download(i - 1, s0))
            if serial:   # copies first, then the compute with the GPU to itself
                for _, e1 in ups + downs:
                    stream.wait_event(e1)
            else:
                if i == 0:
                    stream.wait_event(ups[-1][1])
                if i + 1 < K:   # the next step's inputs, beside this step's compute
                    ups.append(upload(hsets[(i + 1) % 2], dsets[(i + 1) % 2], s0))
                    up_b += in_bytes
            att_done = step(t, dsets[i % 2], stream, o=douts[i % 2])
            if i + 1 == K:   # the last step's own output
                downs.append(download(i, att_done))
            down_b += out_bytes * len(downs)
            for _, e1 in downs:
                stream.wait_event(e1)
            if ups:
                stream.wait_event(ups[-1][1])
            s1.record(stream)
            s1.synchronize()
            e2e_ms += s0.elapsed_time(s1)
            up_ms.append(sum(a.elapsed_time(b) for a, b in ups))
            down_ms.append(sum(a.elapsed_time(b) for a, b in downs))
            stt = step_stats(t)
            if stt is not None:
                e2e_keys += sum(h.occupancy_before + N for h in stt[1])
        e2e_ms_max, e2e_keys = reduce_over_ranks(e2e_ms, e2e_keys, world, dev)
        e2e = {"value": e2e_keys / (e2e_ms_max / 1e3), "unit": UNIT, "h2d_bytes_per_step": up_b // K,
               "d2h_bytes_per_step": down_b // K, "ms_per_step": e2e_ms_max / K,
               "blocks_per_s": world * K / (e2e_ms_max / 1e3),
               "upload_ms_per_step": sum(up_ms) / K, "download_ms_per_step": sum(down_ms) / K,
               "upload_gbs": up_b / (sum(up_ms) / 1e3) / 1e9 if sum(up_ms) > 0 else None,
               "download_gbs": down_b / (sum(down_ms) / 1e3) / 1e9 if sum(down_ms) > 0 else None,
               "schedule": args.e2e_schedule, "numa": numa_info(local),
               "copies": ("pinned host buffers (one NUMA node on this host); each step uploads its own inputs "
                          "while the previous step's output downloads, then computes" if args.e2e_schedule == "serial"
                          else "pinned host buffers (one NUMA node on this host); inputs and outputs double-buffered "
                          "on the device: the previous step's output downloads, then the next step's inputs upload, "
                          "on one copy stream beside each step's compute") + "; no CUDA graphs"}
        del hsets, dsets, douts, host_outs

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline_stack(wl, keys_all / max(K, 1) / world)

    if rank == 0:
        roof = {"kernel": "attend_tc", "bound": "tensor", "achieved": None, "peak": tpeak, "unit": "TFLOP/s",
                "frac": None, "peak_source": f"{pk_src} bf16 dense (burst)",
                "algorithmic_per_launch": {"flops": att_flops}, "traffic": None}
        if att_n:
            ach = att_flops / (att_ms / att_n / 1e3) / 1e12
            roof.update(achieved=ach, frac=ach / tpeak, frac_of_nominal=ach / NOMINAL_BF16_TFLOPS,
                        launches=att_n, avg_ms=att_ms / att_n,
                        traffic=traffic_for("attend_tc", ["k_tc_attn.cu", "tc_ptx.cuh"], wl.name, LH))
        admitting = [sum(1 for r in s["r_star"] if r > 0) for s in per_step]
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": W_,
            "ms_per_step": total_ms_max / K, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16" if wl.dtype == "bf16" else "f32", "data": "synthetic",
            "config": {"workload": f"{wl.name}: {L} layers x {H} heads per block step (one model step), d={d}, "
                                   f"N={N}, M_h in {sorted(set(wl.budgets))}, W={wl.W}, Nq={Nq}",
                       "score_mode": args.score_mode, "prefix": "shared per layer (Eq. 11)" if sync
                       else "independent per head (App. E)",
                       "inputs": "every layer and head an independent synthetic stream, generated on the device "
                                 "before each step's start event",
                       "streams": "admit, then attention || evict, then commit; one handle over all layers "
                                  "(single launches over all L x H heads)",
                       "cuda_graphs": False,
                       "l2": "flushed between timed steps (256 MiB write); inputs larger than L2",
                       "parallelism": f"{world} independent rollouts (one per GPU), no collective" if world > 1
                       else "one GPU"},
            "blocks_per_s": world * K / (total_ms_max / 1e3),
            "interaction_pairs_per_s": pairs_all / (total_ms_max / 1e3),
            "wall_s_timed": wall, "step_ms": {"min": min(step_ms), "median": statistics.median(step_ms),
                                              "max": max(step_ms)},
            "e2e": e2e, "gpu_launches": launches * world, "roofline": roof, "cpu_baseline": cpu, "clocks": clk,
            "per_kernel": per_kernel, "per_kernel_roofs": kernel_roofs(per_kernel, P),
            "per_kernel_note": f"{P} further steps on one stream with every launch timed by CUDA events (not "
                               "in value; the survivor and new-baseline passes then run one after the other); "
                               "tensor kernels against the bf16 peak, memory-bound kernels' algorithmic (and "
                               "moved-by-design) bytes against the HBM peak",
            "update": {"layers_admitting_per_step": admitting,
                       "admitted_per_step": [s["admitted"] for s in per_step],
                       "evicted_per_step": [s["evicted"] for s in per_step],
                       "mandatory_per_step": [s["mandatory"] for s in per_step],
                       "last_step_r_star_per_layer": per_step[-1]["r_star"] if per_step else [],
                       "note": "a layer with r* = 0 admits nothing (under the shared prefix one saturated head "
                               "holds its layer at 0, Eq. 11); its admit pass still scores every bank key"},
        }
        print(json.dumps(line), flush=True)
    bank.close()
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


def synth_workload(name, **over):
    import synth
    return synth.get_workload(name, **over)


def _stack_sample_heads(wl, n):
    """Heads of layer 0 for the oracle sample: the first head of each of the n distinct
    budgets nearest the workload's mean budget."""
    mean = sum(wl.budgets) / len(wl.budgets)
    first = {}
    for h in range(wl.H):
        first.setdefault(wl.budgets[h], h)
    return [first[b] for b in sorted(first, key=lambda b: (abs(b - mean), b))[:n]]


def cpu_baseline_stack(wl, keys_per_block):
    """The oracle on a bounded sample of the stack workload: heads of layer 0 brought to
    steady state (untimed), then one step each (attention + update) timed; the rate is
    keys scored per second, and the model step's time is extrapolated from it."""
    n_heads, n_steps = CPU_SAMPLE_STACK
    heads = _stack_sample_heads(wl, n_heads)
    tot_s, tot_k = 0.0, 0
    for h in heads:
        ro, ob, t = _oracle_head_setup(wl, 0, h)
        dt, k = _oracle_steps(wl, ro, ob, t, n_steps)
        tot_s += dt
        tot_k += k
    rate = tot_k / tot_s
    return {"value": rate, "unit": UNIT, "cores": oracle_threads(), "kind": "oracle",
            "sample": f"{len(heads)} head(s) of layer 0 (budgets {[wl.budgets[h] for h in heads]}) of {wl.name}, "
                      f"{n_steps} steady-state steps each (attention of {wl.Nq} queries + bank update), {tot_k} "
                      f"keys scored in {tot_s:.1f} s (numpy float64)",
            "blocks_per_s_extrapolated": rate / keys_per_block if keys_per_block else None}


def main():
    args = parse_args()
    if args.warmup < 3:
        print("warning: --warmup < 3 does not reach the steady state of the bank", file=sys.stderr)
    if args.impl == "reference":
        run_reference(args)
    elif synth_workload(args.workload).L > 1 or args.stack:
        if args.within_block != "batch" or args.rope != "off" or args.descriptor != "k" or args.attn_passes != 1 \
                or args.order != "score" or args.eviction != "mandatory_densest" or args.refresh_baselines:
            raise SystemExit("policy, descriptor, RoPE and sequential ablations are measured on one-layer workloads")
        run_stack(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
