"""Seeded synthetic rollouts of whole layer stacks, drawn on the GPU with torch.

Input synthesis only (no method arithmetic).  The recipe is the one of
``synth.LayerRollout``, vectorised over every (layer, head) of a stack so that the
stack workloads (up to 40 x 40 heads x 4,680 tokens x 128 dimensions per step, with
per-head budgets, cluster counts and concentrations) take milliseconds per step
instead of minutes:

- per (layer, head): K cluster centres uniform on S^{d-1} (plus a unit tangent
  direction for drift), K, the concentration and the recurrence rate of that head
  from the workload's per-head tuples, so every layer and head is an independent
  stream;
- per block: each token is recurrent with the head's recurrence rate (a cluster drawn
  uniformly among those used by earlier blocks) or fresh (the block's group of
  max(1, K // 8) next unused clusters, uniform over all once every cluster is used);
- directions from vMF(centre, kappa * d_k) by Wood's (1994) rejection algorithm,
  scaled by sqrt(d_k); values N(0, 1); queries drawn like the keys of their step with
  their own cluster assignment; bf16 workloads rounded to bf16 (nearest, ties to even).

Random numbers come from torch's device generator, seeded per (workload seed, rank
seed, step, stream, head chunk) by a splitmix64 mix, so a step can be regenerated in
isolation.  The samples follow the same distribution as ``LayerRollout``'s numpy
streams but are different draws.
"""
from __future__ import annotations

import math
from typing import Optional, Sequence

import torch

_S_CENTRES, _S_ASSIGN, _S_KEYS, _S_VALUES, _S_QUERIES, _S_QASSIGN = range(6)
_M64 = (1 << 64) - 1


def _splitmix64(x: int) -> int:
    x = (x + 0x9E3779B97F4A7C15) & _M64
    x = ((x ^ (x >> 30)) * 0xBF58476D1CE4E5B9) & _M64
    x = ((x ^ (x >> 27)) * 0x94D049BB133111EB) & _M64
    return x ^ (x >> 31)


def _seed(*parts: int) -> int:
    h = 0
    for p in parts:
        h = _splitmix64(h ^ (p & _M64))
    return h & ((1 << 63) - 1)


class StackRollout:
    """Blocks and queries of every head of ``layers`` (stacked along heads, layer-major)."""

    def __init__(self, wl, layers: Optional[Sequence[int]] = None, device="cuda", rank_seed: int = 0,
                 chunk_heads: int = 160):
        self.wl = wl
        self.layers = list(range(wl.L)) if layers is None else list(layers)
        self.dev = torch.device(device)
        self.rank_seed = rank_seed
        idx = [l * wl.H + h for l in self.layers for h in range(wl.H)]
        self.n_heads = len(idx)
        self.chunk = max(1, chunk_heads)
        self.dtype = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
        self.Kc = torch.tensor([wl.clusters[i] for i in idx], dtype=torch.int64, device=self.dev)
        self.kappa = torch.tensor([wl.kappa_vmf(i) for i in idx], dtype=torch.float64, device=self.dev)
        self.rec = torch.tensor([wl.recurrence[i] for i in idx], dtype=torch.float64, device=self.dev)
        self.g = torch.clamp(self.Kc // 8, min=1)
        kmax = int(self.Kc.max())
        d = wl.d
        gen = self._gen(0, _S_CENTRES, 0)
        mu = torch.randn(self.n_heads, kmax, d, generator=gen, device=self.dev, dtype=torch.float32)
        mu /= mu.norm(dim=-1, keepdim=True)
        self.mu = mu
        self.nu = None
        if wl.drift != 0.0:
            nu = torch.randn(self.n_heads, kmax, d, generator=gen, device=self.dev, dtype=torch.float32)
            nu -= (nu * mu).sum(-1, keepdim=True) * mu
            nu /= nu.norm(dim=-1, keepdim=True)
            self.nu = nu

    def _gen(self, t: int, stream: int, chunk: int) -> torch.Generator:
        g = torch.Generator(device=self.dev)
        g.manual_seed(_seed(self.wl.seed, self.rank_seed, t, stream, chunk))
        return g

    def _assign(self, h0: int, h1: int, t: int, n: int, stream: int) -> torch.Tensor:
        """Cluster index [h1 - h0][n] of every token of step t."""
        gen = self._gen(t, stream, h0)
        K = self.Kc[h0:h1, None]
        g = self.g[h0:h1, None]
        used = torch.clamp(t * g, max=K)
        u = torch.rand(h1 - h0, n, generator=gen, device=self.dev, dtype=torch.float64)
        is_rec = (u < self.rec[h0:h1, None]) & (used > 0)
        u_rec = torch.rand(h1 - h0, n, generator=gen, device=self.dev, dtype=torch.float64)
        u_fr = torch.rand(h1 - h0, n, generator=gen, device=self.dev, dtype=torch.float64)
        rec_c = torch.clamp((u_rec * used).long(), max=used - 1).clamp(min=0)
        fresh_avail = t * g < K
        fresh_c = torch.where(fresh_avail, (t * g + torch.clamp((u_fr * g).long(), max=g - 1)) % K,
                              torch.clamp((u_fr * K).long(), max=K - 1))
        return torch.where(is_rec, rec_c, fresh_c)

    def _wood_cosines(self, kappa: torch.Tensor, gen: torch.Generator) -> torch.Tensor:
        """Cosine to the mean direction of one vMF draw per entry of kappa (float64), by
        Wood's rejection step with a Beta((d-1)/2, (d-1)/2) proposal."""
        dm1 = self.wl.d - 1.0
        b = (-2.0 * kappa + torch.sqrt(4.0 * kappa * kappa + dm1 * dm1)) / dm1
        x0 = (1.0 - b) / (1.0 + b)
        c = kappa * x0 + dm1 * torch.log1p(-x0 * x0)
        w = torch.empty_like(kappa)
        todo = torch.arange(kappa.numel(), device=self.dev)
        a = torch.full((1,), dm1 / 2.0, dtype=torch.float64, device=self.dev)
        for _ in range(64):
            if todo.numel() == 0:
                break
            n = todo.numel()
            g1 = torch._standard_gamma(a.expand(n).contiguous(), generator=gen)
            g2 = torch._standard_gamma(a.expand(n).contiguous(), generator=gen)
            z = g1 / (g1 + g2)
            bb, xx, cc, kk = b[todo], x0[todo], c[todo], kappa[todo]
            ww = (1.0 - (1.0 + bb) * z) / (1.0 - (1.0 - bb) * z)
            u = torch.rand(n, generator=gen, device=self.dev, dtype=torch.float64)
            ok = kk * ww + dm1 * torch.log1p(-xx * ww) - cc >= torch.log(u)
            w[todo[ok]] = ww[ok]
            todo = todo[~ok]
        if todo.numel():
            raise RuntimeError("vMF rejection sampler did not converge")
        return w

    def _directions(self, h0: int, h1: int, t: int, assign: torch.Tensor, stream: int) -> torch.Tensor:
        """Unit vMF draws [h1 - h0][n][d] (float32) around each token's cluster centre."""
        gen = self._gen(t, stream, h0)
        nh, n = assign.shape
        d = self.wl.d
        hix = torch.arange(h0, h1, device=self.dev)[:, None].expand(nh, n)
        mu = self.mu[hix, assign]
        if self.nu is not None:
            a = self.wl.drift * t
            mu = math.cos(a) * mu + math.sin(a) * self.nu[hix, assign]
            mu = mu / mu.norm(dim=-1, keepdim=True)
        kap = self.kappa[h0:h1, None].expand(nh, n).reshape(-1)
        w = self._wood_cosines(kap, gen).view(nh, n, 1).float()
        v = torch.randn(nh, n, d, generator=gen, device=self.dev, dtype=torch.float32)
        v -= (v * mu).sum(-1, keepdim=True) * mu
        v /= v.norm(dim=-1, keepdim=True)
        return w * mu + torch.sqrt(torch.clamp(1.0 - w * w, min=0.0)) * v

    def block(self, t: int, out_k: torch.Tensor, out_v: torch.Tensor) -> None:
        """Candidate keys and values of block t into out_k, out_v [n_heads][N][d]."""
        wl = self.wl
        for h0 in range(0, self.n_heads, self.chunk):
            h1 = min(self.n_heads, h0 + self.chunk)
            a = self._assign(h0, h1, t, wl.N, _S_ASSIGN)
            out_k[h0:h1].copy_(self._directions(h0, h1, t, a, _S_KEYS) * wl.scale)
            gen = self._gen(t, _S_VALUES, h0)
            out_v[h0:h1].copy_(torch.randn(h1 - h0, wl.N, wl.d, generator=gen, device=self.dev))

    def queries(self, t: int, out_q: torch.Tensor) -> None:
        """Queries of step t into out_q [n_heads][Nq][d], drawn like the keys of block t."""
        wl = self.wl
        for h0 in range(0, self.n_heads, self.chunk):
            h1 = min(self.n_heads, h0 + self.chunk)
            a = self._assign(h0, h1, t, wl.Nq, _S_QASSIGN)
            out_q[h0:h1].copy_(self._directions(h0, h1, t, a, _S_QUERIES) * wl.scale)
