"""Seeded synthetic rollouts shaped like the DensityKV workloads.

This module only produces inputs: candidate keys/values for each finalized
block, queries, and local-window contents.  It holds none of the method's
arithmetic (no kernel, density, ordering or eviction logic), so both the CPU
oracle (``oracle/``) and the CUDA path may use it without sharing any of the
method between them.

Workload shapes follow the paper's evaluated setting: Wan2.1-T2V-1.3B heads
with d_k = d_v = 128, 1,560 latent tokens per frame, finalized blocks of three
frames (N = 4,680 candidates per head), and a nonlocal budget of six frames
(M = 9,360) (Sec. 4.1 "Implementation Details"; App. D "Memory budget and
temporal alignment").  Real post-RoPE key traces, MovieGenBench prompts and
VBench are not available, so keys are drawn from a mixture of von Mises-Fisher
clusters with recurrence across blocks (and optional slow drift of the
cluster centres), which gives the redundant / recurrent coverage the bank
update is designed for.

Key directions are sampled with Wood's (1994) rejection algorithm ("Simulation
of the von Mises Fisher distribution", Commun. Stat. Simul. Comput. 23(1)).
Directions are unit vectors; they are scaled by ``key_scale`` (default
sqrt(d_k)), so that two keys at angle theta have ||k_i - k_j||^2 / sigma^2 =
4 (1 - cos theta) with the calibrated bandwidth sigma = sqrt(d_k / 2)
(App. B, Eq. "supp-bandwidth" and its intuition equation).

The configured concentration kappa is read per key dimension: the sampler
uses kappa_vMF = kappa * d_k (``kappa_per_dim=True``).  On S^{d-1} the mean
cosine to the centre is about kappa / d for kappa << d, so a literal
kappa = 20 in 128 dimensions gives nearly isotropic keys (mean cosine 0.15 to
the centre, 0.02 between cluster mates): every pairwise interaction is about
1/25 and there are no clusters, no redundancy and, after the bank fills, no
admissions at all.  With kappa * d_k the angular radius of a cluster,
1 - E[cos] ~ 1 / (2 kappa), does not depend on d_k (about 13 degrees at
kappa = 20).  ``kappa_per_dim=False`` keeps the literal reading.

Every random draw comes from ``numpy.random.Generator(PCG64)`` seeded by a
``SeedSequence`` keyed on (workload seed, layer, head, step, stream), so a
block can be regenerated in isolation, in any order, on any machine.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

__all__ = [
    "Workload",
    "WORKLOADS",
    "get_workload",
    "LayerRollout",
    "round_to_bf16",
    "temporal_rope_theta",
    "sample_vmf",
    "make_workload",
]

# stream ids inside a (layer, head, step) seed key
_S_CENTRES, _S_ASSIGN, _S_KEYS, _S_VALUES, _S_QUERIES, _S_QASSIGN, _S_HEADPARAMS = range(7)


def temporal_rope_theta(d: int, band_pairs: Optional[int] = None, base: float = 10000.0,
                        layout_first: bool = True) -> np.ndarray:
    """Angular frequencies [d/2] (float32) of a 3-D rotary layout whose temporal band is
    band_pairs rotation pairs (default: a third of the pairs, rounded down, 21 of 64 at
    d = 128) with RoFormer frequencies base^(-j / band_pairs); the spatial pairs get 0
    (their rotations are not touched by temporal re-zeroing).  The band is the first
    pairs (layout_first) or the last ones."""
    P = d // 2
    n = P // 3 if band_pairs is None else band_pairs
    th = np.zeros(P, dtype=np.float32)
    band = (base ** (-np.arange(n, dtype=np.float64) / n)).astype(np.float32)
    if layout_first:
        th[:n] = band
    else:
        th[P - n:] = band
    return th


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even), returned as float32.

    The result is exactly representable in bfloat16, so converting it to a
    torch.bfloat16 tensor is lossless and both sides see identical inputs.
    """
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    bias = 0x7FFF + ((u >> 16) & 1)
    r = ((u + bias) & 0xFFFF0000).astype(np.uint32)
    out = r.view(np.float32).copy()
    nan = np.isnan(x)
    if nan.any():
        out[nan] = np.nan
    return out.reshape(x.shape)


def sample_vmf(rng: np.random.Generator, mu: np.ndarray, kappa: float, n: int) -> np.ndarray:
    """Draw ``n`` unit vectors from vMF(mu, kappa) on S^{d-1} (Wood 1994).

    Step 1 samples the cosine ``w`` to the mean direction by rejection from a
    transformed Beta((d-1)/2, (d-1)/2) proposal; step 2 draws a uniform
    direction ``v`` orthogonal to ``mu``; the sample is ``w mu + sqrt(1-w^2) v``.
    """
    mu = np.asarray(mu, dtype=np.float64)
    d = mu.shape[0]
    if n == 0:
        return np.zeros((0, d), dtype=np.float64)
    dm1 = d - 1.0
    b = (-2.0 * kappa + math.sqrt(4.0 * kappa * kappa + dm1 * dm1)) / dm1
    x0 = (1.0 - b) / (1.0 + b)
    c = kappa * x0 + dm1 * math.log(1.0 - x0 * x0)
    ws: List[np.ndarray] = []
    need = n
    while need > 0:
        m = max(2 * need, 64)
        z = rng.beta(dm1 / 2.0, dm1 / 2.0, size=m)
        w = (1.0 - (1.0 + b) * z) / (1.0 - (1.0 - b) * z)
        u = rng.uniform(size=m)
        ok = kappa * w + dm1 * np.log(1.0 - x0 * w) - c >= np.log(u)
        acc = w[ok][:need]
        ws.append(acc)
        need -= acc.shape[0]
    w = np.concatenate(ws)
    g = rng.standard_normal(size=(n, d))
    g -= np.outer(g @ mu, mu)
    g /= np.linalg.norm(g, axis=1, keepdims=True)
    return w[:, None] * mu[None, :] + np.sqrt(np.maximum(0.0, 1.0 - w * w))[:, None] * g


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic rollout configuration.

    Per-head quantities (budget, cluster count, concentration, recurrence) are
    tuples of length ``L * H`` indexed ``layer * H + head``.
    """

    name: str
    L: int
    H: int
    d: int
    N: int                      # candidates per finalized block (per head)
    W: int                      # local-window tokens read by attention
    Nq: int                     # queries per step (per head)
    steps: int                  # rollout length
    dtype: str                  # "fp32" or "bf16"
    window: str                 # "own": window = block t; "prev": window = block t-1;
                                # "sink5": first frame of block 0 + the 5 most recent frames
    budgets: Tuple[int, ...]    # M_h per (layer, head)
    clusters: Tuple[int, ...]
    kappa: Tuple[float, ...]
    recurrence: Tuple[float, ...]
    drift: float = 0.0          # radians per step that each cluster centre rotates
    key_scale: Optional[float] = None  # None -> sqrt(d)
    kappa_per_dim: bool = True  # vMF concentration used = kappa * d (see module docstring)
    seed: int = 0
    frames_per_block: int = 3   # a block is this many latent frames of N / frames_per_block tokens

    def kappa_vmf(self, idx: int) -> float:
        return self.kappa[idx] * (self.d if self.kappa_per_dim else 1)

    @property
    def scale(self) -> float:
        return math.sqrt(self.d) if self.key_scale is None else float(self.key_scale)

    def budgets_of_layer(self, layer: int) -> Tuple[int, ...]:
        return tuple(self.budgets[layer * self.H:(layer + 1) * self.H])

    def admitted_block(self, t: int) -> Optional[int]:
        """Index of the block that leaves the window (is offered to the bank) at step t."""
        if self.window == "own":
            return t
        if self.window == "sink5":
            # after step t the 5-frame window starts at frame 3t - 2: block t - 2 has left it
            return t - 2 if t >= 2 else None
        return t - 1 if t >= 1 else None

    def frame_coords(self, b: int) -> np.ndarray:
        """Temporal coordinate (latent frame index) of each token of block b, int32 [N]:
        block b holds frames frames_per_block * b ... in raster order of N / frames_per_block
        tokens each."""
        per = self.N // self.frames_per_block
        return (self.frames_per_block * b + np.minimum(np.arange(self.N) // per,
                                                       self.frames_per_block - 1)).astype(np.int32)

    def window_block(self, t: int) -> int:
        """Index of the block whose K/V form the local window read at step t (whole-block
        windows only; see window_parts)."""
        if self.window == "sink5":
            raise ValueError("the sink5 window is not one block; use window_parts")
        if self.window == "own":
            return t
        return t - 1 if t >= 1 else 0

    def window_parts(self, t: int) -> List[Tuple[int, int, int]]:
        """The local window read at step t as (block, first token, end token) pieces, in order.
        sink5: the first frame of block 0 (the first-frame sink) followed by the five most
        recent finalized frames (Sec. 4.1 / App. D); at t = 0 nothing is finalized and the
        block attends to itself."""
        if self.window != "sink5":
            return [(self.window_block(t), 0, self.N)]
        F = self.N // self.frames_per_block
        if t == 0:
            return [(0, 0, self.N)]
        parts = [(0, 0, F)]
        for f in range(max(1, self.frames_per_block * t - 5), self.frames_per_block * t):
            b, o = divmod(f, self.frames_per_block)
            if parts[-1][0] == b and parts[-1][2] == o * F and len(parts) > 1:
                parts[-1] = (b, parts[-1][1], (o + 1) * F)
            else:
                parts.append((b, o * F, (o + 1) * F))
        return parts

    def window_len(self, t: int) -> int:
        return sum(e - s for _, s, e in self.window_parts(t))


def _per_head(rng: np.random.Generator, n: int, choices=None, lo=None, hi=None, const=None):
    if const is not None:
        return tuple([const] * n)
    if choices is not None:
        return tuple(choices[i] for i in rng.integers(0, len(choices), size=n))
    return tuple(float(v) for v in rng.uniform(lo, hi, size=n))


def make_workload(name: str, **over) -> Workload:
    """Build a named workload; keyword overrides replace fields (and re-derive per-head tuples)."""
    base = dict(_SPECS[name])
    base.update(over)
    L, H = base["L"], base["H"]
    n = L * H
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([base.get("seed", 0), 9999, _S_HEADPARAMS])))
    per = {}
    for key in ("budgets", "clusters", "kappa", "recurrence"):
        spec = base.pop(key)
        if isinstance(spec, dict):
            vals = _per_head(rng, n, **spec)
        elif isinstance(spec, (list, tuple)) and len(spec) == n:
            vals = tuple(spec)
        else:
            vals = tuple([spec] * n)
        if key in ("budgets", "clusters"):
            vals = tuple(int(v) for v in vals)
        else:
            vals = tuple(float(v) for v in vals)
        per[key] = vals
    return Workload(name=name, **base, **per)


# The five workload shapes (names say what they are).
_SPECS: Dict[str, dict] = {
    # 1 layer x 2 heads, d=64, fp32; 256-token blocks into a 512-token bank; 6 steps;
    # 16 clusters, kappa 20, 50% recurrence; window = the current block.
    "tiny_fp32_l1h2_d64": dict(L=1, H=2, d=64, N=256, W=256, Nq=256, steps=6, dtype="fp32",
                               window="own", budgets=512, clusters=16, kappa=20.0,
                               recurrence=0.5, seed=0),
    # Wan-1.3B-shaped single layer: 12 heads, d=128, bf16; 4680-token blocks (3 x 1560),
    # 9360-token bank (6 frames), window = previous block (3 frames); 20 steps;
    # 64 clusters, 60% recurrence.
    "wan13b_layer_h12": dict(L=1, H=12, d=128, N=4680, W=4680, Nq=4680, steps=20, dtype="bf16",
                             window="prev", budgets=9360, clusters=64, kappa=20.0,
                             recurrence=0.6, seed=0),
    # The Wan-1.3B layer with the paper's visible context: a first-frame sink plus a 5-frame
    # local window (9,360 window tokens) next to the bank; the block offered at step t is the
    # one that has left the 5-frame window (t - 2).
    "wan13b_layer_h12_sink5": dict(L=1, H=12, d=128, N=4680, W=9360, Nq=4680, steps=20, dtype="bf16",
                                   window="sink5", budgets=9360, clusters=64, kappa=20.0,
                                   recurrence=0.6, seed=0),
    # Full Wan-1.3B-shaped stack: 30 x 12 heads; 64-256 clusters and 40-80% recurrence per head.
    "wan13b_stack_l30h12": dict(L=30, H=12, d=128, N=4680, W=4680, Nq=4680, steps=40, dtype="bf16",
                                window="prev", budgets=9360,
                                clusters=dict(choices=(64, 128, 192, 256)),
                                kappa=20.0, recurrence=dict(lo=0.4, hi=0.8), seed=0),
    # Large-bank stress: 30 x 12 heads, 32760-token bank (21 frames), 120 steps,
    # drifting centres (0.02 rad / step), 70% recurrence.
    "largebank_l30h12_m32760": dict(L=30, H=12, d=128, N=4680, W=4680, Nq=4680, steps=120,
                                    dtype="bf16", window="prev", budgets=32760, clusters=64,
                                    kappa=20.0, recurrence=0.7, drift=0.02, seed=0),
    # Wan-14B-shaped head-wise budgets: 40 x 40 heads, budgets U{2340,4680,9360,18720},
    # clusters U{8,32,128,512}, kappa U[5,50].
    "wan14b_headwise_l40h40": dict(L=40, H=40, d=128, N=4680, W=4680, Nq=4680, steps=60,
                                   dtype="bf16", window="prev",
                                   budgets=dict(choices=(2340, 4680, 9360, 18720)),
                                   clusters=dict(choices=(8, 32, 128, 512)),
                                   kappa=dict(lo=5.0, hi=50.0), recurrence=0.6, seed=0),
}

WORKLOADS = tuple(_SPECS)


def get_workload(name: str, **over) -> Workload:
    return make_workload(name, **over)


class LayerRollout:
    """Deterministic per-layer stream of candidate blocks, queries and windows."""

    def __init__(self, wl: Workload, layer: int = 0, heads: Optional[Sequence[int]] = None):
        self.wl = wl
        self.layer = layer
        self.heads = list(range(wl.H)) if heads is None else list(heads)
        self._centres = {}
        for h in self.heads:
            idx = layer * wl.H + h
            rng = self._rng(h, 0, _S_CENTRES)
            K = wl.clusters[idx]
            mu = rng.standard_normal(size=(K, wl.d))
            mu /= np.linalg.norm(mu, axis=1, keepdims=True)
            nu = rng.standard_normal(size=(K, wl.d))
            nu -= np.sum(nu * mu, axis=1, keepdims=True) * mu
            nu /= np.linalg.norm(nu, axis=1, keepdims=True)
            self._centres[h] = (mu, nu)

    def _rng(self, head: int, t: int, stream: int) -> np.random.Generator:
        ss = np.random.SeedSequence([self.wl.seed, self.layer, head, t, stream])
        return np.random.Generator(np.random.PCG64(ss))

    def _fresh_group(self, K: int) -> int:
        return max(1, K // 8)

    def _centre(self, h: int, c: np.ndarray, t: int) -> np.ndarray:
        mu, nu = self._centres[h]
        if self.wl.drift == 0.0:
            return mu[c]
        a = self.wl.drift * t
        return math.cos(a) * mu[c] + math.sin(a) * nu[c]

    def _assign(self, h: int, t: int, n: int, stream: int) -> np.ndarray:
        """Cluster index per token of block t: recurrent tokens reuse clusters of blocks < t."""
        idx = self.layer * self.wl.H + h
        K = self.wl.clusters[idx]
        rec = self.wl.recurrence[idx]
        g = self._fresh_group(K)
        rng = self._rng(h, t, stream)
        used = min(t * g, K)
        fresh_lo = (t * g) % K if t * g < K else None
        is_rec = rng.uniform(size=n) < rec if used > 0 else np.zeros(n, dtype=bool)
        out = np.empty(n, dtype=np.int64)
        nrec = int(is_rec.sum())
        out[is_rec] = rng.integers(0, used, size=nrec) if nrec else out[is_rec]
        nfresh = n - nrec
        if fresh_lo is not None:
            grp = (fresh_lo + np.arange(g)) % K
            out[~is_rec] = grp[rng.integers(0, g, size=nfresh)]
        else:
            out[~is_rec] = rng.integers(0, K, size=nfresh)
        return out

    def _directions(self, h: int, t: int, assign: np.ndarray, stream: int) -> np.ndarray:
        idx = self.layer * self.wl.H + h
        kappa = self.wl.kappa_vmf(idx)
        rng = self._rng(h, t, stream)
        out = np.empty((assign.shape[0], self.wl.d), dtype=np.float64)
        for c in np.unique(assign):
            sel = np.nonzero(assign == c)[0]
            mu = self._centre(h, np.asarray(c), t)
            mu = mu / np.linalg.norm(mu)
            out[sel] = sample_vmf(rng, mu, kappa, sel.shape[0])
        return out

    def _finish(self, x: np.ndarray) -> np.ndarray:
        x = x.astype(np.float32)
        return round_to_bf16(x) if self.wl.dtype == "bf16" else x

    def block(self, t: int) -> Tuple[np.ndarray, np.ndarray]:
        """Candidate keys and values of block t, each float32 [len(heads)][N][d]."""
        wl = self.wl
        K = np.empty((len(self.heads), wl.N, wl.d), dtype=np.float32)
        V = np.empty_like(K)
        for i, h in enumerate(self.heads):
            a = self._assign(h, t, wl.N, _S_ASSIGN)
            K[i] = self._finish(self._directions(h, t, a, _S_KEYS) * wl.scale)
            V[i] = self._finish(self._rng(h, t, _S_VALUES).standard_normal(size=(wl.N, wl.d)))
        return K, V

    def queries(self, t: int) -> np.ndarray:
        """Queries of step t, drawn like the keys of block t: float32 [len(heads)][Nq][d]."""
        wl = self.wl
        Q = np.empty((len(self.heads), wl.Nq, wl.d), dtype=np.float32)
        for i, h in enumerate(self.heads):
            a = self._assign(h, t, wl.Nq, _S_QASSIGN)
            Q[i] = self._finish(self._directions(h, t, a, _S_QUERIES) * wl.scale)
        return Q

    def window(self, t: int) -> Tuple[np.ndarray, np.ndarray]:
        """Local-window K/V read at step t, float32 [len(heads)][window_len(t)][d]."""
        parts = self.wl.window_parts(t)
        if len(parts) == 1 and parts[0][1] == 0 and parts[0][2] == self.wl.N:
            return self.block(parts[0][0])
        ks, vs = [], []
        for b, s0, e0 in parts:
            K, V = self.block(b)
            ks.append(K[:, s0:e0])
            vs.append(V[:, s0:e0])
        return np.concatenate(ks, axis=1), np.concatenate(vs, axis=1)
