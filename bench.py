#!/usr/bin/env python3
"""Benchmark of the DensityKV hot path on GB300: bank update + bank-reading attention.

One step = one rollout step of one layer (all H heads): attention of the current
block's queries over [bank | window], then admit + compress of the block leaving
the window (Sec. 3.4, Alg. 1), all through the C ABI (libdkv.so).

Default workload: the Wan-1.3B-shaped single layer (12 heads, d = 128, bf16,
4,680-token blocks, 9,360-token bank, window = previous block, 4,680 queries),
synthetic clustered keys from ``synth``.  W warm-up steps start from an empty bank
(the first two fill it, eviction starts at the third), then K steps are timed one
by one with CUDA events on the launching stream; a 256 MiB buffer is written
between timed steps to flush the 129 MB L2.

Metric: bank keys scored per second = sum over heads of (m_h + N) per update
(every bank key's projected growth and every candidate are scored) / step time.

``--impl reference`` times the CPU oracle (oracle/, numpy float64) on the host
cores, each step a bounded sample of the same workload (one head).

Multi-GPU (torchrun): every rank runs an independent layer of the same shape (the
bank update and attention are per layer and head, with no exchange), so no
collective is on the data path; ranks meet only at the barriers around the timed
region and in a max-reduction of the elapsed time.
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


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=17)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="wan13b_layer_h12")
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
    ap.add_argument("--layers", type=int, default=1,
                    help="layers updated per step on this GPU (whole-stack throughput; > 1 selects the stack run)")
    ap.add_argument("--streams", type=int, default=4, help="stream pairs the layers of a stack step spread over "
                    "(--stack-mode streams)")
    ap.add_argument("--stack-mode", choices=["grouped", "streams"], default="grouped",
                    help="grouped: one handle over all layers, single launches; streams: one handle per layer")
    ap.add_argument("--distinct-layers", type=int, default=2,
                    help="stack run: layers with their own synthetic input stream (the rest reuse them)")
    ap.add_argument("--no-e2e", action="store_true")
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
    if args.rope != "off" and args.layers > 1:
        ap.error("--rope is measured on the single-layer step")
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


def traffic_for(kernel: str, src_files):
    """DRAM bytes per launch from the committed ncu summary, if the kernel is unchanged since."""
    if not os.path.exists(TRAFFIC_FILE):
        return None
    t = json.load(open(TRAFFIC_FILE)).get(kernel)
    if not t or t.get("source_sha1") != source_sha1(*src_files):
        return None
    return t.get("bytes_per_launch")


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
        copy_s = torch.cuda.Stream(dev)   # O download
        pre_s = torch.cuda.Stream(dev)    # input uploads
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
                copy_s.wait_event(att_done)
                with torch.cuda.stream(copy_s):
                    host_out.copy_(out, non_blocking=True)
                o_done = torch.cuda.Event()
                o_done.record(copy_s)
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
            e2e_ms += s0.elapsed_time(s1)
            L, hs = bank.stats()
            if wl.admitted_block(t) is not None:
                e2e_keys += sum(h.occupancy_before + wl.N for h in hs)
            h2d += h2d_i
            d2h += host_out.numel() * host_out.element_size()
        e2e_ms, e2e_keys = reduce_over_ranks(e2e_ms, e2e_keys, world, dev)
        e2e = {"value": e2e_keys / (e2e_ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d // K,
               "d2h_bytes_per_step": d2h // K, "ms_per_step": e2e_ms / K,
               "copies": "pinned host buffers; inputs double-buffered and uploaded one step ahead on a copy "
                         "stream (every timed step's uploads inside the timed regions), O downloaded on another",
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
                "algorithmic_per_launch": {"flops": flops, "keys_per_query": m_bank + wl.W},
                "traffic": traffic_for(dom_name, ["k_tc_attn.cu", "tc_ptx.cuh"])}
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
    """Oracle bank of one head brought to steady state (untimed): first two updates."""
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


def cpu_baseline_sample(wl, layer):
    ro, ob, t = _oracle_head_setup(wl, layer, 0)
    dt, keys = _oracle_step(wl, ro, ob, t)
    return {"value": keys / dt, "unit": UNIT, "cores": oracle_threads(), "kind": "oracle",
            "sample": f"1 head (of {wl.H}), 1 steady-state step of {wl.name}: attention of {wl.Nq} queries "
                      f"+ bank update, {keys} keys scored in {dt:.2f} s (numpy float64)"}


def run_reference(args):
    rank, world, _ = dist_env()
    if not reference_runs_on(rank):
        return
    wl = make_workload(args.workload, 1)
    ro, ob, t = _oracle_head_setup(wl, 0, 0)
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
           "sample": f"each step: 1 head (of {wl.H}) of {wl.name} at steady state, attention of {wl.Nq} "
                     f"queries + bank update (numpy float64)"}
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": f"{wl.name} (one head per step on the host CPU)"},
            "cpu_baseline": cpu,
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_stack(args):
    """Whole-stack throughput on one GPU: every step updates `--layers` independent layer
    banks (attention || admit + evict, then commit), the whole step captured as one CUDA
    graph.  `--stack-mode grouped` (default): one handle holds all layers and every call
    is a single launch per kernel over all L x H heads (each layer keeps its own r*);
    `streams`: one handle per layer, the layers spread over `--streams` stream pairs.
    Inputs of `--distinct-layers` synthetic layer streams are reused round-robin by the
    others (each layer still has its own bank)."""
    import torch

    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_27922_gb300 import dkv

    wl = make_workload(args.workload, 1, args.heads)
    L, S = args.layers, max(1, args.streams)
    D = max(1, min(args.distinct_layers, L))
    W, K = args.warmup, args.steps
    bf = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    inputs = []
    cat1 = lambda xs: torch.cat(xs, dim=1).contiguous()
    for l in range(D):
        inp = Inputs(wl, l, W + K)
        blocks = {b: (torch.from_numpy(k).to(dev, bf), torch.from_numpy(v).to(dev, bf)) for b, (k, v) in inp.blocks.items()}
        inputs.append((blocks, [torch.from_numpy(q).to(dev, bf) for q in inp.queries],
                       [inp.window(t, blocks, cat1) for t in range(W + K)]))
    P = max(1, args.attn_passes)
    mode = dkv.DKV_SCORE_TENSOR if args.score_mode == "tensor" else dkv.DKV_SCORE_FP32
    grouped = args.stack_mode == "grouped"
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    if grouped:
        # one handle holds all L layers (L x H heads, params.layer_heads = H): every call
        # is one launch per kernel over all layers; the inputs are stacked along heads
        budgets = [b for l in range(L) for b in wl.budgets_of_layer(l)]
        banks = [dkv.BankLayer(L * wl.H, wl.d, budgets, wl.N, bf, score_mode=mode, device=dev, layer_heads=wl.H)]
        banks[0].reset()
        stack0 = lambda xs: torch.cat(xs, dim=0).contiguous()
        admitted = sorted({wl.admitted_block(t) for t in range(W + K)} - {None})
        s_blocks = {b: (stack0([inputs[l % D][0][b][0] for l in range(L)]),
                        stack0([inputs[l % D][0][b][1] for l in range(L)])) for b in admitted}
        s_queries = [stack0([inputs[l % D][1][t] for l in range(L)]) for t in range(W + K)]
        def s_window(t):   # a window that is exactly an admitted block shares its tensors
            parts = wl.window_parts(t)
            if len(parts) == 1 and parts[0][1] == 0 and parts[0][2] == wl.N and parts[0][0] in s_blocks:
                return s_blocks[parts[0][0]]
            return (stack0([inputs[l % D][2][t][0] for l in range(L)]),
                    stack0([inputs[l % D][2][t][1] for l in range(L)]))
        s_windows = [s_window(t) for t in range(W + K)]
        del inputs
        out_all = torch.empty(L * wl.H, wl.Nq, wl.d, dtype=bf, device=dev)
        side = torch.cuda.Stream(dev)

        def stack_step(t):
            cur = torch.cuda.current_stream(dev)
            b = wl.admitted_block(t)
            kw, vw = s_windows[t]
            late = P == 1
            if b is not None and late:
                banks[0].admit(s_blocks[b][0], s_blocks[b][1], b, stream=cur)
            go = torch.cuda.Event()
            go.record(cur)
            side.wait_event(go)
            for _ in range(P):
                banks[0].attend(s_queries[t], kw, vw, out=out_all, stream=side)
            done = torch.cuda.Event()
            done.record(side)
            if b is not None:
                if not late:
                    banks[0].admit(s_blocks[b][0], s_blocks[b][1], b, stream=cur)
                banks[0].evict(stream=cur)
            cur.wait_event(done)
            if b is not None:
                banks[0].commit(stream=cur)
    else:
        banks = [dkv.BankLayer(wl.H, wl.d, wl.budgets_of_layer(l), wl.N, bf, score_mode=mode, device=dev)
                 for l in range(L)]
        for bk in banks:
            bk.reset()
        outs = [torch.empty(wl.H, wl.Nq, wl.d, dtype=bf, device=dev) for _ in range(L)]
        mains = [torch.cuda.Stream(dev) for _ in range(S)]
        sides = [torch.cuda.Stream(dev) for _ in range(S)]

    def stack_step_streams(t):
        cur = torch.cuda.current_stream(dev)
        fork = torch.cuda.Event()
        fork.record(cur)
        joins = []
        for l in range(L):
            ms, ss = mains[l % S], sides[l % S]
            blocks, queries, windows = inputs[l % D]
            kw, vw = windows[t]
            b = wl.admitted_block(t)
            ms.wait_event(fork)
            go = torch.cuda.Event()
            go.record(ms)
            ss.wait_event(go)
            for _ in range(P):
                banks[l].attend(queries[t], kw, vw, out=outs[l], stream=ss)
            done = torch.cuda.Event()
            done.record(ss)
            if b is not None:
                kc, vc = blocks[b]
                banks[l].admit(kc, vc, b, stream=ms)
                banks[l].evict(stream=ms)
            ms.wait_event(done)
            if b is not None:
                banks[l].commit(stream=ms)
            j = torch.cuda.Event()
            j.record(ms)
            joins.append(j)
        for j in joins:
            cur.wait_event(j)

    if not grouped:
        stack_step = stack_step_streams
    stream = torch.cuda.current_stream(dev)
    for t in range(W):
        stack_step(t)
    torch.cuda.synchronize()
    graphs = []
    cap = torch.cuda.Stream(dev)
    cap.wait_stream(stream)
    with torch.cuda.stream(cap):
        for i in range(K):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=cap):
                stack_step(W + i)
            graphs.append(g)
    stream.wait_stream(cap)
    torch.cuda.synchronize()
    clocks = ClockSampler(0, enabled=not args.no_clocks)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    keys = 0
    total_ms = 0.0
    rstars = []
    for i in range(K):
        t = W + i
        if not args.no_flush:
            flush.fill_(float(i))
        ev[i][0].record(stream)
        graphs[i].replay()
        ev[i][1].record(stream)
        ev[i][1].synchronize()
        total_ms += ev[i][0].elapsed_time(ev[i][1])
        if wl.admitted_block(t) is not None:
            per_layer = []
            for bk in banks:
                _, hs = bk.stats()
                keys += sum(h.occupancy_before + wl.N for h in hs)
                for l, Ls in enumerate(bk.layer_stats()):
                    per_layer.append((Ls.r_star, sum(h.evicted for h in hs[l * wl.H:(l + 1) * wl.H])))
            rstars.append(per_layer)
    clk = clocks.stop()
    for bk in banks:
        bk.sync()
    line = {
        "metric": METRIC, "value": keys / (total_ms / 1e3), "unit": UNIT, "n_gpus": 1, "steps": K, "warmup": W,
        "ms_per_step": total_ms / K, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16" if wl.dtype == "bf16" else "f32", "data": "synthetic",
        "config": {"workload": f"{wl.name}: {L} layer(s) x {wl.H} heads per step, d={wl.d}, N={wl.N}, "
                               f"M={max(wl.budgets)}, W={wl.W}, Nq={wl.Nq}",
                   "score_mode": args.score_mode, "layers_per_gpu": L,
                   "streams": ("one handle over all layers (single launches), admit, then attention || "
                               "evict, then commit" if grouped else f"one handle per layer on {S} stream pairs"),
                   "cuda_graphs": True, "inputs": f"{D} distinct synthetic layer streams, reused round-robin",
                   "l2": "flushed between timed steps (256 MiB write)" if not args.no_flush else "not flushed",
                   "parallelism": "layers of one GPU, grouped launches" if grouped
                   else "layers of one GPU on concurrent streams"},
        "blocks_per_s": K / (total_ms / 1e3),
        "e2e": None, "gpu_launches": None, "roofline": None, "cpu_baseline": None, "clocks": clk,
        "update": {"last_step_r_star_per_layer": [r for r, _ in rstars[-1]] if rstars else [],
                   "last_step_evicted_per_layer": [e for _, e in rstars[-1]] if rstars else [],
                   "layers_admitting_per_step": [sum(1 for r, _ in st if r > 0) for st in rstars]},
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    if args.warmup < 3:
        print("warning: --warmup < 3 does not reach the steady state of the bank", file=sys.stderr)
    if args.impl == "reference":
        run_reference(args)
    elif args.layers > 1:
        run_stack(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
