"""Plain CPU oracle of the DensityKV bank update and of bank-reading attention.

TEST INFRASTRUCTURE ONLY.  This module is the slow, obviously-correct
reference that the CUDA path is checked against.  It may be imported only by
``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py``; the product path never calls it, and it shares no code with the
CUDA library (it imports numpy only).

Arithmetic is float64 throughout.  The paper fixes the storage precision of
the two per-state density scalars as FP32 (App. D "Persistent-storage
accounting"), so the cached density rho and the frozen baseline b are rounded
to float32 when they are stored in the bank; every sum and comparison is
evaluated in float64.  Keys and values are taken exactly as given (bf16 inputs
arrive as their exactly-representable float32 values).

What each function follows (paper sections / equations):

* ``soft_riesz``         Eq. 2 (Soft-Riesz interaction), App. B Eq. B.2.
* ``sq_dist``            squared Euclidean key distance (Sec. 3.2; the
                         expansion ||a||^2 + ||b||^2 - 2 a.b is the one written
                         out in App. A, Eq. "supp-unitnorm-equivalence").
* ``density``            Eq. 3, Soft-Riesz density over an indexed multiset,
                         self excluded by index.
* ``update_layer``       Algorithm 1 (App. C) with Eqs. 5-12 and C.1-C.4:
                         empty-bank initialisation, mean-normalised candidate
                         score, stable sort, projected growth ratios for every
                         prefix length, shared cross-head prefix r*,
                         mandatory-then-densest eviction, commit, exact density
                         maintenance and frozen insertion baselines.
* ``update_layer_sequential``  App. E "Within-block competition": the block's
                         candidates offered one at a time (reading below).
* ``attend``             softmax attention of queries over [bank | window]
                         with scale 1/sqrt(d_k) (Sec. 3.2 logit definition,
                         App. A Eq. "supp-logit"; Fig. 2 caption).
* ``storage_bytes``      App. D persistent-storage accounting.
* ``rope_rezero``        App. A: memory keys carry temporal RoPE coordinate 0
                         (spatial coordinates kept); offered keys that carry
                         their frame's temporal rotation are rotated back.
* ``round_nearest_bf16`` the storage rounding of rotated bf16 keys (nearest,
                         ties to even), from its definition.
* ``kv_descriptor``      App. E "Retention geometry": the [K; V] descriptor, run
                         through the same update in place of the keys.

Readings taken where the paper is silent or ambiguous (each is restated in
the design notes of the repository):

* Ties in the "decreasing projected density" fill are broken by provenance:
  the older state (smaller (step, src)) is evicted first (the paper allows any
  tie rule, Alg. 1).
* ``g >= tau`` is inclusive and evaluated as a float64 ratio rho~ / b.
* r = 0 is always treated as feasible, and R is empty when r* = 0, even if
  rounding made some g(0) reach tau (the invariant that makes r = 0 feasible
  holds in exact arithmetic; Sec. 3.4 Step 2).
* Per-head budgets M_h generalise e_r = max(0, m + r - M) to
  e_r^h = max(0, m_h + r - M_h) with r <= min(N, min_h M_h); a head whose bank
  is empty takes the empty-bank path (first min(N, M_h) candidates in source
  order) and does not take part in the shared prefix search.
* sync_heads=False gives the "independent per-head prefix" ablation
  (App. E "Cross-head synchronization").
* The other policy ablations of Table 2(b) / App. E, all on the same steps:
  order="source" takes candidates in source order (pi = identity) instead of
  ascending Eq. 6 scores; evict="densest" evicts the e_{r*} states of largest
  rho~(r*) with no mandatory-first step; evict="mandatory_source" evicts the
  threshold crossers first and fills the remaining slots in source order of
  the bank, read as provenance order (oldest (step, src) first);
  refresh_baselines=True sets b = max(rho, delta) for every retained state
  after each update instead of keeping the insertion-time baseline.  In every
  variant r* is still the largest prefix feasible under Eqs. 9-11 for the
  candidates in the variant's order.
* Within-block competition (App. E) is read as: the block's order fixed once
  against the bank at block start, then one one-candidate update per position
  of that order (the j-th candidate of every head together, so the shared prefix
  of Eq. 11 is taken over the heads for each offer), provenance keeping the
  candidate's source index; an all-empty bank is initialised by the whole block
  as in the default.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence

import numpy as np

__all__ = [
    "Params", "HeadBank", "LayerBank", "HeadRecord", "UpdateRecord",
    "soft_riesz", "sq_dist", "density", "potential_against",
    "update_layer", "update_layer_sequential", "block_order", "attend", "storage_bytes", "GIB",
    "rope_rezero", "round_nearest_bf16", "kv_descriptor",
]

GIB = float(1 << 30)


@dataclasses.dataclass(frozen=True)
class Params:
    """Method parameters; defaults from Sec. 4.1 and App. D ("Default DensityKV configuration")."""

    tau: float = 2.0          # allowed density-growth factor, tau > 1
    sigma: Optional[float] = None  # None -> sqrt(d_k / 2) (App. B, Eq. "supp-bandwidth")
    p: float = 2.0            # decay exponent
    eps: float = 1.0          # regulariser
    delta: float = 1e-6       # baseline floor
    sync_heads: bool = True   # shared cross-head prefix (default policy)
    order: str = "score"      # "score" (Eq. 6 ascending, default) or "source"
    evict: str = "mandatory_densest"   # or "densest", "mandatory_source"
    refresh_baselines: bool = False    # default: baselines frozen at insertion (Eq. 5)

    def sigma_for(self, d: int) -> float:
        return math.sqrt(d / 2.0) if self.sigma is None else float(self.sigma)


def sq_dist(A: np.ndarray, B: np.ndarray) -> np.ndarray:
    """||a_i - b_j||^2 for all rows of A against all rows of B, float64 [len(A), len(B)].

    Uses ||a||^2 + ||b||^2 - 2 a.b (App. A) with a library matmul, then clamps
    at zero because a squared distance is non-negative.
    """
    A = np.asarray(A, dtype=np.float64)
    B = np.asarray(B, dtype=np.float64)
    na = np.einsum("ij,ij->i", A, A)
    nb = np.einsum("ij,ij->i", B, B)
    d2 = na[:, None] + nb[None, :] - 2.0 * (A @ B.T)
    return np.maximum(d2, 0.0)


def soft_riesz(d2: np.ndarray, prm: Params, d: int) -> np.ndarray:
    """Eq. 2: w = (eps + ||k_i - k_j||^2 / sigma^2)^(-p)."""
    s = prm.sigma_for(d)
    return np.power(prm.eps + np.asarray(d2, dtype=np.float64) / (s * s), -prm.p)


def density(K: np.ndarray, prm: Params) -> np.ndarray:
    """Eq. 3: Phi_A(i) = sum_{j != i} w(k_i, k_j) over the indexed multiset K (rows)."""
    K = np.asarray(K, dtype=np.float64)
    n = K.shape[0]
    if n == 0:
        return np.zeros(0)
    W = soft_riesz(sq_dist(K, K), prm, K.shape[1])
    W[np.arange(n), np.arange(n)] = 0.0        # j != i, by index (duplicates still count)
    return W.sum(axis=1)


def potential_against(x: np.ndarray, A: np.ndarray, prm: Params) -> np.ndarray:
    """App. B Eq. "supp-insertion-energy": Phi_A(k_x) = sum_j w(k_x, k_j) for each row x."""
    x = np.atleast_2d(np.asarray(x, dtype=np.float64))
    A = np.asarray(A, dtype=np.float64)
    if A.shape[0] == 0:
        return np.zeros(x.shape[0])
    return soft_riesz(sq_dist(x, A), prm, x.shape[1]).sum(axis=1)


@dataclasses.dataclass
class HeadBank:
    """Bank of one (layer, head): Eq. 4 plus the cached density and provenance (App. C, App. D)."""

    M: int                      # per-head budget
    d: int
    dv: int
    K: np.ndarray = None        # [m, d] float64 (exact copies of the admitted keys)
    V: np.ndarray = None        # [m, dv]
    rho: np.ndarray = None      # [m] float32, cached current density Phi_{K(B)}(i)
    base: np.ndarray = None     # [m] float32, frozen insertion baseline b_i
    step: np.ndarray = None     # [m] int64, update step that admitted the state
    src: np.ndarray = None      # [m] int64, source index of the state within its block
    store: type = np.float32    # storage type of rho and b (FP32 per App. D; float64 for pins)

    def __post_init__(self):
        if self.K is None:
            self.K = np.zeros((0, self.d))
            self.V = np.zeros((0, self.dv))
            self.rho = np.zeros(0, self.store)
            self.base = np.zeros(0, self.store)
            self.step = np.zeros(0, np.int64)
            self.src = np.zeros(0, np.int64)

    @property
    def m(self) -> int:
        return int(self.K.shape[0])

    def copy(self) -> "HeadBank":
        return HeadBank(self.M, self.d, self.dv, self.K.copy(), self.V.copy(), self.rho.copy(),
                        self.base.copy(), self.step.copy(), self.src.copy(), self.store)


@dataclasses.dataclass
class LayerBank:
    heads: List[HeadBank]

    @staticmethod
    def empty(budgets: Sequence[int], d: int, dv: Optional[int] = None, store=np.float32) -> "LayerBank":
        return LayerBank([HeadBank(int(M), d, d if dv is None else dv, store=store) for M in budgets])

    def copy(self) -> "LayerBank":
        return LayerBank([h.copy() for h in self.heads])


@dataclasses.dataclass
class HeadRecord:
    """Intermediate quantities of one head's update, exposed for parity checks."""

    empty_init: bool
    s: Optional[np.ndarray] = None          # [N] Eq. 6 / C.1 scores
    pi: Optional[np.ndarray] = None         # [N] stable ascending order of s
    counts: Optional[np.ndarray] = None     # [rmax+1] c_r^h for every tested prefix
    e: Optional[np.ndarray] = None          # [rmax+1] e_r^h
    cross: Optional[np.ndarray] = None      # [m] min{r : g_i(r) >= tau}, or -1 if none <= rmax
    r_used: int = 0                         # number of candidates admitted in this head
    rho_tilde: Optional[np.ndarray] = None  # [m] rho~_i(r*) (float64)
    g_star: Optional[np.ndarray] = None     # [m] g_i(r*)
    mandatory: Optional[np.ndarray] = None  # [m] bool, g_i(r*) >= tau (and r* > 0)
    evicted: Optional[np.ndarray] = None    # indices (pre-update bank order) of R, mandatory first
    admitted: Optional[np.ndarray] = None   # candidate indices admitted, in admission order


@dataclasses.dataclass
class UpdateRecord:
    r_star: int
    rmax: int
    heads: List[HeadRecord]


def _prefix_rho_tilde(hb: HeadBank, Kc_pi: np.ndarray, prm: Params, rmax: int) -> np.ndarray:
    """Eq. C.2 for every prefix length r = 0..rmax: rho~_i(r) = rho_i + sum_{j<=r} w(kbar_i, k_pi(j)).

    Returns float64 [m, rmax+1].  Column-wise cumulative sums over the
    pi-ordered candidate interactions give all prefix contributions (App. C,
    "Decision granularity versus computational tiling").
    """
    Wmat = soft_riesz(sq_dist(hb.K, Kc_pi[:rmax]), prm, hb.d)          # [m, rmax]
    out = np.empty((hb.m, rmax + 1))
    out[:, 0] = hb.rho.astype(np.float64)
    out[:, 1:] = hb.rho.astype(np.float64)[:, None] + np.cumsum(Wmat, axis=1)
    return out


def _prefix_rho_tilde_literal(hb: HeadBank, Kc_pi: np.ndarray, prm: Params, rmax: int) -> np.ndarray:
    """Same quantity as ``_prefix_rho_tilde``, recomputed from scratch for each r with plain loops.

    Tiny inputs only; used to pin the cumulative-sum form (Alg. 1 tests every prefix length).
    """
    s = prm.sigma_for(hb.d)
    out = np.empty((hb.m, rmax + 1))
    for i in range(hb.m):
        for r in range(rmax + 1):
            acc = float(hb.rho[i])
            for j in range(r):
                diff = hb.K[i] - Kc_pi[j]
                d2 = float(np.dot(diff, diff))
                acc += (prm.eps + d2 / (s * s)) ** (-prm.p)
            out[i, r] = acc
    return out


def _empty_init(hb: HeadBank, Kc: np.ndarray, Vc: np.ndarray, step: int, prm: Params,
                src: Optional[np.ndarray] = None) -> HeadRecord:
    """Alg. 1, m = 0 branch: admit the first min(N, M) source-ordered candidates, then set
    rho_i = Phi over the resulting bank and b_i = max(rho_i, delta)."""
    N = Kc.shape[0]
    r = min(N, hb.M)
    hb.K = np.asarray(Kc[:r], dtype=np.float64).copy()
    hb.V = np.asarray(Vc[:r], dtype=np.float64).copy()
    rho = density(hb.K, prm)
    hb.rho = rho.astype(hb.store)
    hb.base = np.maximum(rho, prm.delta).astype(hb.store)
    hb.step = np.full(r, step, np.int64)
    hb.src = (np.arange(r) if src is None else np.asarray(src[:r])).astype(np.int64)
    return HeadRecord(empty_init=True, r_used=r, admitted=np.arange(r), evicted=np.zeros(0, np.int64))


def update_layer(bank: LayerBank, Kc: np.ndarray, Vc: np.ndarray, step: int,
                 prm: Params = Params(), literal: bool = False,
                 src_index: Optional[np.ndarray] = None) -> UpdateRecord:
    """One DensityKV update of one layer (Algorithm 1, App. C), in place on ``bank``.

    Kc, Vc: candidate keys/values of the finalized block, [H][N][d] and [H][N][dv],
    in source order.  ``step`` is recorded as the provenance of admitted states, with
    the candidate's row as its source index, or src_index[h][row] when given.
    ``literal=True`` recomputes every prefix sum from scratch (tiny inputs).
    """
    assert prm.order in ("score", "source")
    assert prm.evict in ("mandatory_densest", "densest", "mandatory_source")
    H = len(bank.heads)
    Kc = np.asarray(Kc, dtype=np.float64)
    Vc = np.asarray(Vc, dtype=np.float64)
    assert Kc.shape[0] == H and Vc.shape[0] == H
    N = Kc.shape[1]
    recs: List[Optional[HeadRecord]] = [None] * H

    live = [h for h in range(H) if bank.heads[h].m > 0]
    for h in range(H):
        if bank.heads[h].m == 0:
            recs[h] = _empty_init(bank.heads[h], Kc[h], Vc[h], step, prm,
                                  None if src_index is None else src_index[h])

    rmax = min([N] + [bank.heads[h].M for h in live]) if live else 0
    if not live:
        return UpdateRecord(r_star=min(N, min(hb.M for hb in bank.heads)) if H else 0,
                            rmax=rmax, heads=recs)

    # Steps 1-2 per head: score, stable sort, projected growth for every prefix length.
    tables = {}
    for h in live:
        hb = bank.heads[h]
        m = hb.m
        # Eq. 6 / C.1: s_h(x) = (1/m) sum_i w(kbar_i, k_x) / b_i
        Wxb = soft_riesz(sq_dist(Kc[h], hb.K), prm, hb.d)              # [N, m]
        s = (Wxb / hb.base.astype(np.float64)[None, :]).sum(axis=1) / m
        # stable ascending sort, ties broken by source order (or source order itself)
        pi = np.argsort(s, kind="stable") if prm.order == "score" else np.arange(N)
        Kc_pi = Kc[h][pi]
        if literal:
            rt = _prefix_rho_tilde_literal(hb, Kc_pi, prm, rmax)
        else:
            rt = _prefix_rho_tilde(hb, Kc_pi, prm, rmax)
        g = rt / hb.base.astype(np.float64)[:, None]                    # Eq. C.3
        viol = g >= prm.tau
        counts = viol.sum(axis=0)                                        # c_r^h, Eq. 9
        r_all = np.arange(rmax + 1)
        e = np.maximum(0, m + r_all - hb.M)                              # e_r^h, Eq. 10
        feasible = counts <= e
        feasible[0] = True                                               # r = 0 always feasible
        anyv = viol.any(axis=1)
        cross = np.where(anyv, np.argmax(viol, axis=1), -1)
        tables[h] = (s, pi, rt, g, counts, e, feasible, cross)

    # Eq. 11: largest prefix length feasible for every head (or per head when not synchronised).
    if prm.sync_heads:
        allf = np.logical_and.reduce([tables[h][6] for h in live])
        r_star = int(np.nonzero(allf)[0].max())
        r_of = {h: r_star for h in live}
    else:
        r_of = {h: int(np.nonzero(tables[h][6])[0].max()) for h in live}
        r_star = max(r_of.values())

    # Step 3 per head: evict, commit, maintain densities.
    for h in live:
        hb = bank.heads[h]
        s, pi, rt, g, counts, e, feasible, cross = tables[h]
        r = r_of[h]
        m = hb.m
        e_r = int(e[r])
        rho_t = rt[:, r]
        g_r = g[:, r]
        mand = (g_r >= prm.tau) if r > 0 else np.zeros(m, bool)
        mand_idx = np.nonzero(mand)[0]
        assert mand_idx.shape[0] <= e_r, "feasibility violated"
        if prm.evict == "densest":
            # the e_r largest rho~(r*) over the whole bank; ties: older provenance first
            order = np.lexsort((hb.src, hb.step, -rho_t))
            R = order[:e_r].astype(np.int64)
        else:
            rest = np.nonzero(~mand)[0]
            if prm.evict == "mandatory_source":
                # fill in source (provenance) order: oldest (step, src) first
                order = np.lexsort((hb.src[rest], hb.step[rest]))
            else:
                # decreasing rho~(r*); ties: older provenance (smaller step, then src) first
                order = np.lexsort((hb.src[rest], hb.step[rest], -rho_t[rest]))
            fill = rest[order[:e_r - mand_idx.shape[0]]]
            R = np.concatenate([mand_idx, fill]).astype(np.int64)
        keep = np.ones(m, bool)
        keep[R] = False
        adm = pi[:r]

        # Eq. C.4: survivors' cached density, exactly: rho~(r*) minus interactions with R.
        if R.shape[0] > 0 and keep.any():
            sub = soft_riesz(sq_dist(hb.K[keep], hb.K[R]), prm, hb.d).sum(axis=1)
        else:
            sub = np.zeros(int(keep.sum()))
        rho_surv = rho_t[keep] - sub

        # Eq. 12 commit: (B \ R) followed by the admitted prefix in pi order.
        K_new = np.concatenate([hb.K[keep], Kc[h][adm]], axis=0)
        V_new = np.concatenate([hb.V[keep], Vc[h][adm]], axis=0)
        # Eq. 5 / C.4: new states' density over the final bank (co-admitted included), frozen as b.
        n_surv = int(keep.sum())
        if r > 0:
            W_new = soft_riesz(sq_dist(K_new[n_surv:], K_new), prm, hb.d)    # [r, m']
            W_new[np.arange(r), n_surv + np.arange(r)] = 0.0                  # exclude self by index
            rho_new = W_new.sum(axis=1)
        else:
            rho_new = np.zeros(0)
        hb.K, hb.V = K_new, V_new
        hb.rho = np.concatenate([rho_surv, rho_new]).astype(hb.store)
        if prm.refresh_baselines:
            # every retained state's baseline follows its current (stored) density
            hb.base = np.maximum(hb.rho.astype(np.float64), prm.delta).astype(hb.store)
        else:
            hb.base = np.concatenate([hb.base[keep], np.maximum(rho_new, prm.delta)]).astype(hb.store)
        hb.step = np.concatenate([hb.step[keep], np.full(r, step, np.int64)])
        adm_src = adm if src_index is None else np.asarray(src_index[h])[adm]
        hb.src = np.concatenate([hb.src[keep], adm_src.astype(np.int64)])
        recs[h] = HeadRecord(empty_init=False, s=s, pi=pi, counts=counts, e=e, cross=cross,
                             r_used=r, rho_tilde=rho_t, g_star=g_r, mandatory=mand,
                             evicted=R, admitted=adm)
    return UpdateRecord(r_star=r_star, rmax=rmax, heads=recs)


def block_order(bank: LayerBank, Kc: np.ndarray, prm: Params = Params()) -> np.ndarray:
    """pi_h of every head against the bank as it is now ([H][N]): ascending Eq. 6 score
    (ties in source order), or source order under the source-order policy; the order
    update_layer takes for a non-empty head (an empty head: source order)."""
    Kc = np.asarray(Kc, dtype=np.float64)
    H, N = Kc.shape[0], Kc.shape[1]
    out = np.tile(np.arange(N), (H, 1))
    for h, hb in enumerate(bank.heads):
        if hb.m == 0 or prm.order == "source":
            continue
        Wxb = soft_riesz(sq_dist(Kc[h], hb.K), prm, hb.d)
        s = (Wxb / hb.base.astype(np.float64)[None, :]).sum(axis=1) / hb.m
        out[h] = np.argsort(s, kind="stable")
    return out


def update_layer_sequential(bank: LayerBank, Kc: np.ndarray, Vc: np.ndarray, step: int,
                            prm: Params = Params()) -> List[UpdateRecord]:
    """Within-block competition (App. E "Within-block competition"; Sec. 4 ablations):
    sequential density-gated admission, so that earlier candidates of the block act on
    later ones.  Reading: the block's order is fixed once, as the default order against
    the bank at block start (block_order); the candidates are then offered one per head
    at a time (the j-th of every head's order, for j = 0 .. N-1), each offer a complete
    one-candidate update (Eqs. 6-12 with N = 1: the growth gate, eviction, commit and the
    frozen baseline of the admitted state), the candidate keeping its source index in the
    block as provenance.  A bank whose heads are all empty is initialised by the whole
    block (Alg. 1, m = 0 branch) exactly as in the default; a partly empty bank is not
    accepted (an empty head would otherwise start from a single state whose baseline is
    delta, and then reject every later candidate)."""
    empty = [hb.m == 0 for hb in bank.heads]
    if all(empty):
        return [update_layer(bank, Kc, Vc, step, prm)]
    if any(empty):
        raise ValueError("sequential admission needs every head empty or every head non-empty")
    Kc = np.asarray(Kc, dtype=np.float64)
    Vc = np.asarray(Vc, dtype=np.float64)
    H, N = Kc.shape[0], Kc.shape[1]
    pi = block_order(bank, Kc, prm)
    rows = np.arange(H)
    recs = []
    for j in range(N):
        c = pi[:, j]
        recs.append(update_layer(bank, Kc[rows, c][:, None], Vc[rows, c][:, None], step, prm,
                                 src_index=c[:, None]))
    return recs


def attend(hb: HeadBank, Q: np.ndarray, Kw: np.ndarray, Vw: np.ndarray) -> np.ndarray:
    """Softmax attention of Q over [bank keys | window keys], logits q.k / sqrt(d_k), no mask."""
    Q = np.asarray(Q, dtype=np.float64)
    Kall = np.concatenate([hb.K, np.asarray(Kw, dtype=np.float64)], axis=0)
    Vall = np.concatenate([hb.V, np.asarray(Vw, dtype=np.float64)], axis=0)
    if Kall.shape[0] == 0:
        return np.zeros((Q.shape[0], hb.dv))
    S = (Q @ Kall.T) / math.sqrt(Q.shape[1])
    S -= S.max(axis=1, keepdims=True)
    P = np.exp(S)
    P /= P.sum(axis=1, keepdims=True)
    return P @ Vall


def kv_descriptor(K: np.ndarray, V: np.ndarray) -> np.ndarray:
    """App. E "Retention geometry": the [K; V] descriptor of each state, its key and value
    concatenated (2 d_k values), float64.

    The [K; V] policy is the same algorithm with these rows in place of the keys: a
    LayerBank of dimension 2 d_k updated by ``update_layer(bank, kv_descriptor(Kc, Vc),
    Vc, ...)``; sigma defaults to sqrt(2 d_k / 2) = sqrt(d_k) (the App. B rule for the
    descriptor dimension), and a stored row's first d_k values are its key.
    """
    return np.concatenate([np.asarray(K, dtype=np.float64), np.asarray(V, dtype=np.float64)], axis=-1)


def round_nearest_bf16(x: np.ndarray) -> np.ndarray:
    """Nearest bfloat16 value (8 significant bits, ties to even) of float64 values, as float64.

    Written from the definition: x = m 2^e with 1/2 <= |m| < 1 (frexp, exact), the
    significand scaled to 8 integer bits, rounded to the nearest integer with ties to even
    (rint), and scaled back.  One rounding from float64, so no double rounding through
    float32.  Normal range only (keys and values are O(1)); zeros stay zeros.
    """
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)
    out = np.ldexp(np.rint(m * 256.0), e - 8)
    nz = out[x != 0]
    assert np.all(np.isfinite(out)) and np.all(np.abs(nz) >= 2.0 ** -126), "outside the bf16 normal range"
    return out


def rope_rezero(K: np.ndarray, t_coord: np.ndarray, theta: np.ndarray, layout: str = "interleaved",
                storage: Optional[str] = "bf16") -> np.ndarray:
    """Offered keys moved to temporal rotary coordinate 0 (App. A: the backbones attend to
    nonlocal memory keys with the temporal RoPE coordinate set to 0 and the spatial ones
    kept, and the bank stores exactly those keys).

    K [H][N][d] carries, in every rotation pair j with theta_j != 0, the rotation by the
    angle a = t_x theta_j of its token's temporal coordinate t_x (t_coord [N], shared by
    the heads): a pair (x, y) of the unrotated key appears as
    (x cos a - y sin a, x sin a + y cos a).  Setting the coordinate to 0 rotates it back
    by -a:  x0 = x cos a + y sin a,  y0 = y cos a - x sin a.  Pairs with theta_j = 0
    (the spatial bands) are left as they are.  layout "interleaved": pair j is elements
    (2j, 2j+1); "half": (j, j + d/2).  theta is float32 [d/2]; the angle t theta is
    formed exactly in float64 and the rotation evaluated in float64, then rounded once
    to the storage precision ("bf16": nearest bfloat16, ties to even; "fp32": nearest
    float32; None: the float64 values).
    """
    K = np.asarray(K, dtype=np.float64)
    H, N, d = K.shape
    th = np.asarray(theta, dtype=np.float32).astype(np.float64)
    assert th.shape == (d // 2,)
    t = np.asarray(t_coord, dtype=np.int64).astype(np.float64)
    assert t.shape == (N,)
    if layout == "interleaved":
        xi, yi = np.arange(0, d, 2), np.arange(1, d, 2)
    elif layout == "half":
        xi, yi = np.arange(d // 2), np.arange(d // 2, d)
    else:
        raise ValueError(layout)
    a = t[:, None] * th[None, :]                  # [N][d/2], exact in float64
    c, s = np.cos(a), np.sin(a)
    x, y = K[:, :, xi], K[:, :, yi]
    out = K.copy()
    out[:, :, xi] = x * c + y * s
    out[:, :, yi] = y * c - x * s
    keep = th == 0.0                              # unrotated pairs stay bit for bit
    out[:, :, xi[keep]] = K[:, :, xi[keep]]
    out[:, :, yi[keep]] = K[:, :, yi[keep]]
    if storage is None:
        return out
    if storage == "bf16":
        return round_nearest_bf16(out)
    if storage == "fp32":
        return out.astype(np.float32).astype(np.float64)
    raise ValueError(storage)


def storage_bytes(L: int, H: int, n: int, dk: int = 128, dv: int = 128,
                  kv_bytes: int = 2, meta_bytes: int = 4 + 4 + 8 + 4) -> dict:
    """App. D accounting: S_KV(n) = L H n (d_k + d_v) x 2 bytes, plus per-state metadata
    (two FP32 density scalars, int64 + int32 provenance = 20 bytes)."""
    kv = L * H * n * (dk + dv) * kv_bytes
    meta = L * H * n * meta_bytes
    return {"kv": kv, "meta": meta, "total": kv + meta}
