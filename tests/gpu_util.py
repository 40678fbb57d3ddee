"""Helpers of the GPU parity tests: teacher forcing and oracle-vs-CUDA comparison.

The CUDA path is driven only through the C ABI binding (paper_2608_27922_gb300.dkv);
expected values come only from the CPU oracle (oracle/) on the same seeded inputs.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional, Tuple

import numpy as np
import torch

import oracle
import synth
from paper_2608_27922_gb300 import dkv

INT_MAX = 2 ** 31 - 1

# fp32 score mode: every w within a few ulp, sums of up to ~1e4 positive fp32 terms;
# decisions may differ only within the probabilistic rounding bound of such sums,
# lambda sqrt(n) u = 3.5 * sqrt(9360) * 2^-24 = 2.0e-5, and the retained sets must be
# identical
FP32_TOL, FP32_DENS = 2e-5, 2e-5
# tensor-core mode: bf16 inputs exact, products exact, fp32 accumulation (spec bounds)
TC_TOL, TC_DENS = 1e-3, 1e-2


def tols(mode: str) -> Tuple[float, float]:
    """(decision window, density tolerance) of a score mode ("fp32" or "tc")."""
    return (FP32_TOL, FP32_DENS) if mode == "fp32" else (TC_TOL, TC_DENS)


def check_report(rep: "Report", mode: str, where=None) -> None:
    """The parity bar of one teacher-forced update (see tols)."""
    _, dens = tols(mode)
    assert rep.ok(), (where, rep)
    assert rep.rstar_gpu == rep.rstar_oracle, (where, rep)
    assert rep.score_max_rel <= dens and rep.rho_tilde_max_rel <= dens, (where, rep)
    assert rep.rho_max_rel <= dens and rep.base_max_rel <= dens, (where, rep)
    if mode == "fp32":   # the exactness mode: identical retained sets
        assert rep.set_mismatch == 0, (where, rep)


def to_dev(x: np.ndarray, dtype: torch.dtype) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to("cuda", dtype)


ORDER_NAMES = {dkv.DKV_ORDER_SCORE: "score", dkv.DKV_ORDER_SOURCE: "source"}
EVICT_NAMES = {dkv.DKV_EVICT_MANDATORY_DENSEST: "mandatory_densest", dkv.DKV_EVICT_DENSEST: "densest",
               dkv.DKV_EVICT_MANDATORY_SOURCE: "mandatory_source"}


def oracle_params(bank: dkv.BankLayer) -> oracle.Params:
    p = bank.params
    return oracle.Params(tau=float(p.tau), sigma=float(p.sigma), p=float(p.p), eps=float(p.eps),
                         delta=float(np.float32(p.delta)), sync_heads=bool(p.sync_heads),
                         order=ORDER_NAMES[p.order], evict=EVICT_NAMES[p.eviction],
                         refresh_baselines=bool(p.refresh_baselines))


def load_state(bank: dkv.BankLayer, ob, head0: int = 0, imp: bool = True) -> None:
    """Writes the oracle's bank of one layer (or a list of layers, stacked along heads)
    into the GPU bank buffers (slots 0..m-1) from head head0 on, and imports it."""
    obs = ob if isinstance(ob, (list, tuple)) else [ob]
    h = head0
    for lb in obs:
        for hb in lb.heads:
            m = hb.m
            if m:
                bank.k[h, :m] = to_dev(hb.K[:, :bank.d], bank.dtype)   # a [K; V] bank: its key part
                bank.v[h, :m] = to_dev(hb.V, bank.dtype)
                bank.rho[h, :m] = torch.from_numpy(hb.rho.astype(np.float32)).cuda()
                bank.base[h, :m] = torch.from_numpy(hb.base.astype(np.float32)).cuda()
                bank.prov_step[h, :m] = torch.from_numpy(hb.step.astype(np.int64)).cuda()
                bank.prov_src[h, :m] = torch.from_numpy(hb.src.astype(np.int32)).cuda()
            h += 1
    if imp:
        bank.import_state([hb.m for lb in obs for hb in lb.heads])


def gpu_heads(bank: dkv.BankLayer) -> List[Dict[Tuple[int, int], tuple]]:
    occ = bank.occupancy_host()
    out = []
    K = bank.k.float().cpu().numpy()
    V = bank.v.float().cpu().numpy()
    rho = bank.rho.cpu().numpy()
    base = bank.base.cpu().numpy()
    st = bank.prov_step.cpu().numpy()
    sr = bank.prov_src.cpu().numpy()
    kn = bank.knorm.cpu().numpy()
    for h in range(bank.H):
        d = {}
        for i in range(occ[h]):
            key = (int(st[h, i]), int(sr[h, i]))
            assert key not in d, f"duplicate provenance {key} in head {h}"
            d[key] = (K[h, i], V[h, i], float(rho[h, i]), float(base[h, i]), float(kn[h, i]), i)
        out.append(d)
    return out


def oracle_heads(ob: oracle.LayerBank) -> List[Dict[Tuple[int, int], tuple]]:
    out = []
    for hb in ob.heads:
        out.append({(int(a), int(b)): (hb.K[i], hb.V[i], float(hb.rho[i]), float(hb.base[i]))
                    for i, (a, b) in enumerate(zip(hb.step, hb.src))})
    return out


@dataclasses.dataclass
class Report:
    rstar_gpu: int = 0
    rstar_oracle: int = 0
    score_max_rel: float = 0.0
    perm_mismatch: int = 0
    perm_unexplained: int = 0
    cross_mismatch: int = 0
    cross_unexplained: int = 0
    set_mismatch: int = 0
    set_unexplained: int = 0
    rho_max_rel: float = 0.0
    base_max_rel: float = 0.0
    # |rho_gpu - rho_oracle| over the magnitude of the terms that formed rho: rho~ + sum_R w
    # for a survivor (Eq. C.4 subtracts the evicted neighbours from rho~), rho otherwise
    rho_term_rel: float = 0.0
    base_term_rel: float = 0.0
    rho_tilde_max_rel: float = 0.0
    rho_tilde_checked: int = 0          # heads whose crossings and rho~(r*) were compared
    # largest relative distance to its cut-off of any decision that differed (s for the
    # order, g vs tau for crossings, g vs tau or rho~ vs the fill cut-off for the sets)
    perm_gap_max: float = 0.0
    cross_gap_max: float = 0.0
    set_gap_max: float = 0.0
    kv_bit_exact: bool = True
    heads_set_differs: int = 0          # heads whose final banks differ by explained decisions
    notes: List[str] = dataclasses.field(default_factory=list)

    def ok(self) -> bool:
        return (self.perm_unexplained == 0 and self.cross_unexplained == 0 and self.set_unexplained == 0
                and self.kv_bit_exact)


def _g_row(hb: oracle.HeadBank, i: int, Kpi: np.ndarray, r: int, prm: oracle.Params) -> float:
    """Oracle g_i(r) for one bank row and a given candidate order (Eq. C.3)."""
    if r == 0:
        return float(hb.rho[i]) / float(hb.base[i])
    w = oracle.soft_riesz(oracle.sq_dist(hb.K[i:i + 1], Kpi[:r]), prm, hb.d)[0]
    return (float(hb.rho[i]) + float(w.sum())) / float(hb.base[i])


def update_and_compare(bank: dkv.BankLayer, ob: oracle.LayerBank, K: np.ndarray, V: np.ndarray, step: int,
                       tol: float, dens_tol: float, rope=None) -> Tuple[Report, oracle.UpdateRecord]:
    """Teacher-forced update of a one-layer handle: the GPU starts from the oracle's bank;
    both apply one update.

    tol: relative window within which a decision may differ (near-tie of s, g vs tau,
    rho~ vs the fill cutoff).  dens_tol: relative tolerance of s, rho~, rho and b.
    ``ob`` is advanced by the oracle's update.  rope = (t_coord, theta, layout): K carries
    the temporal rotation; the GPU re-zeroes it in admit, the oracle updates with
    ``oracle.rope_rezero`` of it.
    """
    reps, recs = update_and_compare_layers(bank, [ob], [K], [V], step, tol, dens_tol, rope)
    return reps[0], recs[0]


def update_and_compare_layers(bank: dkv.BankLayer, obs: List[oracle.LayerBank], Ks: List[np.ndarray],
                              Vs: List[np.ndarray], step: int, tol: float, dens_tol: float,
                              rope=None) -> Tuple[List[Report], List[oracle.UpdateRecord]]:
    """Teacher-forced update of a handle holding len(obs) layers of H heads each (stacked
    along heads, params.layer_heads = H): the GPU starts from the oracle banks, applies one
    update with the stacked candidates (each layer its own prefix r*, Eq. 11), the oracle
    updates every layer on its own; one report per layer."""
    prm = oracle_params(bank)
    before = [ob.copy() for ob in obs]
    load_state(bank, before)
    Kd = to_dev(np.concatenate(Ks, axis=0), bank.dtype)
    Vd = to_dev(np.concatenate(Vs, axis=0), bank.dtype)
    Ko = list(Ks)
    if rope is not None:
        t_coord, theta, layout = rope
        bank.admit(Kd, Vd, step, t_coord=torch.from_numpy(np.asarray(t_coord, np.int32)).to(bank.device),
                   theta=torch.from_numpy(np.asarray(theta, np.float32)).to(bank.device),
                   rope_layout={"interleaved": 0, "half": 1}[layout])
        kt = "bf16" if bank.dtype == torch.bfloat16 else "fp32"
        Ko = [oracle.rope_rezero(K, t_coord, theta, layout, kt) for K in Ko]
    else:
        bank.admit(Kd, Vd, step)
    if bank.params.descriptor == dkv.DKV_DESC_KV:   # the oracle bank holds [K; V] rows (App. E)
        Ko = [oracle.kv_descriptor(K, V) for K, V in zip(Ko, Vs)]
    bank.compress()
    bank.sync()
    recs = [oracle.update_layer(ob, K, V, step, prm) for ob, K, V in zip(obs, Ko, Vs)]
    Ls = bank.layer_stats()
    _, hs = bank.stats()
    inter = {k: v.cpu().numpy().copy() for k, v in bank.intermediates().items()}
    G = gpu_heads(bank)
    reps = []
    h0 = 0
    for l, (ob, bef, rec, K) in enumerate(zip(obs, before, recs, Ko)):
        H = len(ob.heads)
        sl = slice(h0, h0 + H)
        rep = Report(rstar_gpu=Ls[l].r_star, rstar_oracle=rec.r_star)
        _compare_layer(rep, prm, bef, ob, rec, {k: v[sl] for k, v in inter.items()}, hs[sl], G[sl], K, tol)
        reps.append(rep)
        h0 += H
    return reps, recs


def _compare_layer(rep: Report, prm: oracle.Params, before: oracle.LayerBank, ob: oracle.LayerBank,
                   rec: oracle.UpdateRecord, inter, hs, G, K: np.ndarray, tol: float) -> None:
    """Fills rep for one layer: s, pi, cross, rho~ against the oracle's record of the
    update from ``before``; admitted / evicted counts; the committed banks (``G``, read
    back from the GPU) against the oracle's ``ob`` as provenance-keyed sets."""
    N = K.shape[1]
    Kq = K.astype(np.float64)
    for h, (hb, hr) in enumerate(zip(before.heads, rec.heads)):
        if hr.empty_init:
            continue
        if prm.order == "score":   # the source-order policy computes no scores
            s_g = inter["score"][h, :N]
            rel = np.abs(s_g - hr.s) / np.maximum(np.abs(hr.s), 1e-30)
            rep.score_max_rel = max(rep.score_max_rel, float(rel.max()))
        pg = inter["perm"][h, :N]
        diff = np.nonzero(pg != hr.pi)[0]
        rep.perm_mismatch += len(diff)
        for j in diff:
            a, b = hr.s[pg[j]], hr.s[hr.pi[j]]
            gap = abs(a - b) / max(abs(a), abs(b), 1e-300)
            rep.perm_gap_max = max(rep.perm_gap_max, gap)
            if gap > tol:
                rep.perm_unexplained += 1
        # crossing index of every bank row and rho~(r) of the head's prefix: under the
        # oracle's order when both orders agree; otherwise the orders differ only by swaps
        # of near-tied scores (checked above), the GPU's order is an equally valid order of
        # the oracle's scores, and Eq. C.2 is evaluated by the oracle under that order
        if rep.perm_unexplained == 0:
            cg = inter["cross"][h, :hb.m].astype(np.int64)
            if len(diff) == 0:
                Kpi = Kq[h][hr.pi]
                co = np.where(hr.cross < 0, INT_MAX, hr.cross)
                rt_ref = hr.rho_tilde
            else:
                Kpi = Kq[h][pg]
                w = oracle.soft_riesz(oracle.sq_dist(hb.K, Kpi[:rec.rmax]), prm, hb.d)
                tab = np.empty((hb.m, rec.rmax + 1))
                tab[:, 0] = hb.rho.astype(np.float64)
                np.cumsum(w, axis=1, out=tab[:, 1:])
                tab[:, 1:] += tab[:, :1]
                del w
                viol = tab / hb.base.astype(np.float64)[:, None] >= prm.tau
                co = np.where(viol.any(axis=1), np.argmax(viol, axis=1), INT_MAX)
                rt_ref = tab[:, hr.r_used] if hr.rho_tilde is not None else None
                del tab, viol
            bad = np.nonzero(cg != co)[0]
            rep.cross_mismatch += len(bad)
            for i in bad:
                rs = [int(x) for x in (cg[i], co[i]) if x != INT_MAX]
                gaps = [abs(_g_row(hb, i, Kpi, r, prm) - prm.tau) / prm.tau for r in rs]
                gaps += [abs(_g_row(hb, i, Kpi, r - 1, prm) - prm.tau) / prm.tau for r in rs if r > 0]
                gap = min(gaps) if gaps else float("inf")
                rep.cross_gap_max = max(rep.cross_gap_max, gap)
                if gap > tol:
                    rep.cross_unexplained += 1
            if rec.r_star == rep.rstar_gpu and rt_ref is not None:
                rt = inter["rho_tilde"][h, :hb.m]
                rel = np.abs(rt - rt_ref) / np.maximum(np.abs(rt_ref), 1e-30)
                rep.rho_tilde_max_rel = max(rep.rho_tilde_max_rel, float(rel.max()))
                rep.rho_tilde_checked += 1
    if rep.rstar_gpu != rep.rstar_oracle:
        rep.notes.append(f"r* gpu {rep.rstar_gpu} oracle {rep.rstar_oracle}")
    else:
        for h, (st, hr) in enumerate(zip(hs, rec.heads)):
            if st.admitted != hr.r_used or st.evicted != len(hr.evicted):
                rep.set_unexplained += 1
                rep.notes.append(f"head {h}: admitted/evicted gpu {st.admitted}/{st.evicted} "
                                 f"oracle {hr.r_used}/{len(hr.evicted)}")
            if not hr.empty_init and st.mandatory != int(hr.mandatory.sum()):
                rep.notes.append(f"head {h}: mandatory gpu {st.mandatory} oracle {int(hr.mandatory.sum())}")
    # committed banks, compared as sets keyed by provenance
    Oh = oracle_heads(ob)
    for h in range(len(ob.heads)):
        g, o = G[h], Oh[h]
        hr, hb = rec.heads[h], before.heads[h]
        pre = {(int(a), int(b)): i for i, (a, b) in enumerate(zip(hb.step, hb.src))}
        only_g = set(g) - set(o)
        only_o = set(o) - set(g)
        rep.set_mismatch += len(only_g) + len(only_o)
        if only_g or only_o:
            ok = rep.rstar_gpu == rep.rstar_oracle and hr.rho_tilde is not None
            if ok:
                # an eviction decision within `tol` of its cutoff explains the difference
                fill = [i for i in hr.evicted if not hr.mandatory[i]]
                cut = min(hr.rho_tilde[fill]) if fill else None
                for key in only_g | only_o:
                    i = pre.get(key)
                    if i is None:
                        # a candidate admitted on one side only: explained when its score is
                        # within `tol` of the admission cut-off (the scores of the last
                        # admitted and the first refused candidate in the oracle's order)
                        r = hr.r_used
                        src = key[1]
                        if prm.order != "score" or r <= 0 or r >= N or not 0 <= src < N:
                            ok = False
                            break
                        cuts = [hr.s[hr.pi[r - 1]], hr.s[hr.pi[r]]]
                        gap = min(abs(hr.s[src] - c) / max(abs(c), 1e-300) for c in cuts)
                        rep.set_gap_max = max(rep.set_gap_max, gap)
                        if gap > tol:
                            ok = False
                            break
                        continue
                    gap = abs(hr.g_star[i] - prm.tau) / prm.tau
                    if cut is not None:
                        gap = min(gap, abs(hr.rho_tilde[i] - cut) / abs(cut))
                    rep.set_gap_max = max(rep.set_gap_max, gap)
                    if gap > tol:
                        ok = False
                        break
            if not ok:
                rep.set_unexplained += len(only_g) + len(only_o)
            else:
                rep.heads_set_differs += 1
        # an equally valid but different final bank (explained decisions): the densities of
        # Eq. 5 / C.4 are sums over it, so they are compared only in heads whose banks agree
        same_bank = not (only_g or only_o)
        for key in set(g) & set(o):
            kg, vg, rg, bg, kn, _ = g[key]
            ko, vo, ro, bo = o[key]
            if not (np.array_equal(kg, ko[:kg.shape[0]].astype(np.float32)) and np.array_equal(vg, vo.astype(np.float32))):
                rep.kv_bit_exact = False
            if not same_bank:
                continue
            rep.rho_max_rel = max(rep.rho_max_rel, abs(rg - ro) / max(abs(ro), 1e-30))
            rep.base_max_rel = max(rep.base_max_rel, abs(bg - bo) / max(abs(bo), 1e-30))
            i = pre.get(key)
            scale = abs(ro)
            if i is not None and hr.rho_tilde is not None:   # a survivor: rho~ - sum_R w (Eq. C.4)
                rt = float(hr.rho_tilde[i])
                scale = max(scale, rt + max(rt - ro, 0.0))
            rep.rho_term_rel = max(rep.rho_term_rel, abs(rg - ro) / max(scale, 1e-30))
            rep.base_term_rel = max(rep.base_term_rel, abs(bg - bo) / max(scale, abs(bo), 1e-30))


def attention_error(bank: dkv.BankLayer, ob: oracle.LayerBank, Q: np.ndarray, Kw: Optional[np.ndarray],
                    Vw: Optional[np.ndarray]) -> float:
    """Max abs error of the CUDA attention against the oracle on the GPU bank's current contents."""
    O = bank.attend(to_dev(Q, bank.dtype), None if Kw is None else to_dev(Kw, bank.dtype),
                    None if Vw is None else to_dev(Vw, bank.dtype)).float().cpu().numpy()
    H = Q.shape[0]
    err = 0.0
    for h in range(H):
        kw = np.zeros((0, Q.shape[2])) if Kw is None else Kw[h]
        vw = np.zeros((0, Q.shape[2])) if Vw is None else Vw[h]
        ref = oracle.attend(ob.heads[h], Q[h], kw, vw)
        err = max(err, float(np.abs(O[h] - ref).max()))
    return err
