"""Pins of the CPU oracle against what the paper and the mathematics fix.

Every check takes the oracle module ``O`` as its argument, so the same checks
run against the real oracle (``test_oracle_pins.py``, all must pass) and
against copies of it with a planted mistake (``test_oracle_mutants.py``, each
mutant must fail at least one check).  Nothing here calls the CUDA library,
and no expected value comes from it.

Sources of truth used:
  * closed forms of Eq. 2 and App. B (w(k, k) = eps^-p, far-field Riesz decay);
  * identities of App. A (unit-norm cosine equivalence, (gamma - 1)^2 ||k||^2);
  * the energy insertion identity of App. B;
  * brute force on tiny inputs (explicit loops, literal per-r enumeration);
  * the invariants of App. C ("Invariant after commit", Eq. C.4, Alg. 1);
  * a worked example derived by hand with exact rational arithmetic;
  * the (eps, sigma) scale equivalence of App. B "Parameterization";
  * storage figures printed in App. D (golden file);
  * textbook softmax attention (torch scaled_dot_product_attention in fp64);
  * brute-force nearest-value enumeration and torch's float32 -> bfloat16
    conversion for the storage rounding; the rotary embedding written as complex
    multiplication (RoFormer) for the temporal re-zeroing of App. A.
"""
from __future__ import annotations

import json
import math
import os
from fractions import Fraction as F

import numpy as np

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _prm(O, **kw):
    return O.Params(**kw)


# --------------------------------------------------------------------------- P1: Eq. 2
def check_kernel_closed_forms(O):
    d = 128
    prm = _prm(O)                                # eps = 1, sigma = sqrt(64) = 8, p = 2
    # w(k, k) = eps^-p (App. B, coincident keys)
    for eps, p in ((1.0, 2.0), (0.5, 1.0), (2.0, 4.0)):
        w0 = O.soft_riesz(np.array([0.0]), _prm(O, eps=eps, p=p), d)[0]
        assert abs(w0 - eps ** (-p)) < 1e-15 * max(1.0, eps ** (-p)), (eps, p, w0)
    # hand values at sigma = 8, eps = 1, p = 2: d^2 = 64 -> (1+1)^-2 = 1/4; d^2 = 192 -> 1/16
    w = O.soft_riesz(np.array([64.0, 192.0, 0.0, 576.0]), prm, d)
    assert np.allclose(w, [0.25, 1.0 / 16, 1.0, 0.01], rtol=0, atol=1e-15), w
    # sigma is sqrt(d/2) by default: d = 64 -> sigma^2 = 32, d^2 = 32 -> 1/4
    assert abs(O.soft_riesz(np.array([32.0]), prm, 64)[0] - 0.25) < 1e-15
    # explicit sigma and p = 1: (1 + 9/9)^-1 = 1/2
    assert abs(O.soft_riesz(np.array([9.0]), _prm(O, sigma=3.0, p=1.0), d)[0] - 0.5) < 1e-15
    # strictly decreasing in the distance
    r2 = np.linspace(0.0, 1000.0, 101)
    assert np.all(np.diff(O.soft_riesz(r2, prm, d)) < 0)
    # far field: w ~ sigma^{2p} r^{-2p} (App. B, asymptotic form)
    for p in (1.0, 2.0, 4.0):
        big = np.array([1e8])
        ratio = O.soft_riesz(big, _prm(O, p=p), d)[0] / (64.0 ** p * big[0] ** (-p))
        assert abs(ratio - 1.0) < 1e-5, (p, ratio)


# --------------------------------------------------------------------------- P2: distances
def check_distance_identities(O):
    rng = np.random.default_rng(1)
    A = rng.standard_normal((7, 16))
    B = rng.standard_normal((5, 16))
    direct = np.array([[np.sum((a - b) ** 2) for b in B] for a in A])
    assert np.allclose(O.sq_dist(A, B), direct, rtol=1e-12, atol=1e-12)
    # unit keys: ||ki - kj||^2 = 2 d_cos (App. A)
    U = A / np.linalg.norm(A, axis=1, keepdims=True)
    dcos = 1.0 - U @ U.T
    assert np.allclose(O.sq_dist(U, U), 2.0 * dcos, atol=1e-12)
    # ||k - gamma k||^2 = (gamma - 1)^2 ||k||^2
    k = A[:1]
    for g in (0.5, 2.0, 3.0):
        assert abs(O.sq_dist(k, g * k)[0, 0] - (g - 1) ** 2 * np.sum(k * k)) < 1e-10
    # asymmetric shapes keep row/column roles (a transposed operand fails here)
    D = O.sq_dist(A[:3], B)
    assert D.shape == (3, 5) and np.allclose(D, direct[:3], atol=1e-12)


# --------------------------------------------------------------------------- P3: Eq. 3
def check_density_brute_force(O):
    rng = np.random.default_rng(2)
    prm = _prm(O, sigma=1.5, p=2.0)
    K = rng.standard_normal((9, 4))
    K[5] = K[2]                                  # a duplicate key counts eps^-p, not zero
    s2 = 1.5 ** 2
    brute = np.zeros(9)
    for i in range(9):
        for j in range(9):
            if j != i:
                brute[i] += (1.0 + np.sum((K[i] - K[j]) ** 2) / s2) ** -2.0
    phi = O.density(K, prm)
    assert np.allclose(phi, brute, rtol=1e-12), (phi, brute)
    # energy insertion identity (App. B): E(A + x) - E(A) = Phi_A(x), E = 1/2 sum Phi
    A, x = K[:6], K[6:7]
    E = lambda X: 0.5 * O.density(X, prm).sum()
    lhs = E(np.concatenate([A, x])) - E(A)
    rhs = O.potential_against(x, A, prm)[0]
    assert abs(lhs - rhs) < 1e-12 * max(1.0, abs(rhs)), (lhs, rhs)


# --------------------------------------------------------------------------- worked example
def _w1(a, b):
    """Exact w for 1-D keys with eps = 1, sigma = 1, p = 1: w = 1 / (1 + (a - b)^2)."""
    return F(1, 1 + (a - b) ** 2)


def check_worked_example(O):
    """Three updates of one head, derived by hand (1-D keys, eps = 1, sigma = 1, p = 1,
    tau = 2, delta = 1e-6, M = 4).  Expected decisions and densities follow Alg. 1:

    update 0 (empty bank), candidates [0, 1, 4]: all admitted in source order;
        rho(0) = w(0,1) + w(0,4) = 1/2 + 1/17 = 19/34, rho(1) = 1/2 + 1/10 = 3/5,
        rho(4) = 1/17 + 1/10 = 27/170; b = rho.
    update 1, candidates [4, 100, 1] (src 0, 1, 2), m = 3, e_r = max(0, r - 1):
        s(4)   = (1/3)(2/19 + 1/6 + 170/27)              ~ 2.1894
        s(100) = (1/3)(34/190019 + 5/29406 + 170/248859) ~ 3.44e-4
        s(1)   = (1/3)(17/19 + 5/3 + 17/27)              ~ 1.0637
        pi = [1, 2, 0] (sources of 100, 1, 4).
        r = 1: no violator (c = 0 <= 0).
        r = 2: bank key 1 gets + w(1,1) = 1 -> g = (3/5 + 1/9802 + 1)/(3/5) ~ 2.667 >= 2;
               c_2 = 1 <= e_2 = 1 -> feasible.
        r = 3: key 0 reaches g = 2 + 34/190019 (>= 2), keys 1 and 4 violate too:
               c_3 = 3 > e_3 = 2 -> infeasible.   So r* = 2.
        R = {key 1} (mandatory; e = 1, no fill).  Final bank {0, 4, 100, 1'}.
        survivors: rho(0) = 19/34 + 1/10001, rho(4) = 27/170 + 1/9217, b unchanged;
        new: rho(100) = b(100) = 1/10001 + 1/9217 + 1/9802, rho(1') = b(1') = 1/2 + 1/10 + 1/9802.
    update 2, candidate [-30]: e_1 = 1, no violator at r = 1 -> r* = 1;
        fill evicts the largest rho~(1): key 1' (3/5 + 1/9802 + 1/962).
        survivors: rho(0) = 1/17 + 1/10001 + 1/901, rho(4) = 1/17 + 1/9217 + 1/1157,
                   rho(100) = 1/10001 + 1/9217 + 1/16901;
        new: rho(-30) = 1/901 + 1/1157 + 1/16901.
    """
    prm = _prm(O, sigma=1.0, p=1.0, eps=1.0, tau=2.0, delta=1e-6)
    bank = O.LayerBank.empty([4], d=1, store=np.float64)
    kv = lambda xs: (np.array(xs, float).reshape(1, -1, 1), np.array(xs, float).reshape(1, -1, 1) * 10)

    def state(hb):
        return {(int(st), int(sr)): (float(k[0]), float(r), float(b))
                for k, r, b, st, sr in zip(hb.K, hb.rho, hb.base, hb.step, hb.src)}

    def close(a, b):
        assert abs(a - float(b)) < 1e-13, (a, float(b))

    K, V = kv([0, 1, 4])
    rec = O.update_layer(bank, K, V, step=0, prm=prm)
    st = state(bank.heads[0])
    assert sorted(st) == [(0, 0), (0, 1), (0, 2)]
    close(st[(0, 0)][1], F(19, 34)); close(st[(0, 1)][1], F(3, 5)); close(st[(0, 2)][1], F(27, 170))
    for v in st.values():
        close(v[2], v[1])

    K, V = kv([4, 100, 1])
    rec = O.update_layer(bank, K, V, step=1, prm=prm)
    hr = rec.heads[0]
    s_exp = [F(1, 3) * (F(2, 19) + F(1, 6) + F(170, 27)),
             F(1, 3) * (F(34, 190019) + F(5, 29406) + F(170, 248859)),
             F(1, 3) * (F(17, 19) + F(5, 3) + F(17, 27))]
    for a, b in zip(hr.s, s_exp):
        assert abs(a - float(b)) < 1e-13 * float(b), (a, b)
    assert list(hr.pi) == [1, 2, 0]
    assert list(hr.counts) == [0, 0, 1, 3] and list(hr.e) == [0, 0, 1, 2]
    assert rec.r_star == 2
    st = state(bank.heads[0])
    assert sorted(st) == [(0, 0), (0, 2), (1, 1), (1, 2)]      # key 1 (0, 1) evicted
    close(st[(0, 0)][1], F(19, 34) + F(1, 10001)); close(st[(0, 0)][2], F(19, 34))
    close(st[(0, 2)][1], F(27, 170) + F(1, 9217)); close(st[(0, 2)][2], F(27, 170))
    close(st[(1, 1)][1], F(1, 10001) + F(1, 9217) + F(1, 9802)); close(st[(1, 1)][2], st[(1, 1)][1])
    close(st[(1, 2)][1], F(1, 2) + F(1, 10) + F(1, 9802)); close(st[(1, 2)][2], st[(1, 2)][1])
    assert st[(1, 1)][0] == 100.0 and st[(1, 2)][0] == 1.0

    K, V = kv([-30])
    rec = O.update_layer(bank, K, V, step=2, prm=prm)
    assert rec.r_star == 1
    st = state(bank.heads[0])
    assert sorted(st) == [(0, 0), (0, 2), (1, 1), (2, 0)]      # (1, 2) = key 1' evicted by fill
    close(st[(0, 0)][1], F(1, 17) + F(1, 10001) + F(1, 901))
    close(st[(0, 2)][1], F(1, 17) + F(1, 9217) + F(1, 1157))
    close(st[(1, 1)][1], F(1, 10001) + F(1, 9217) + F(1, 16901))
    close(st[(2, 0)][1], F(1, 901) + F(1, 1157) + F(1, 16901)); close(st[(2, 0)][2], st[(2, 0)][1])
    close(st[(0, 0)][2], F(19, 34)); close(st[(1, 1)][2], F(1, 10001) + F(1, 9217) + F(1, 9802))


# --------------------------------------------------------------------------- helpers
def _random_bank_rollout(O, seed, H=2, d=3, N=6, M=9, steps=5, prm=None, literal=False,
                         store=np.float64, ties=False):
    rng = np.random.default_rng(seed)
    prm = prm or _prm(O, sigma=1.0, p=2.0)
    bank = O.LayerBank.empty([M] * H, d, store=store)
    out = []
    for t in range(steps):
        K = rng.standard_normal((H, N, d)) * (1.0 + 0.3 * t)
        if ties:
            K[:, N // 2:] = K[:, :N - N // 2]
        V = rng.standard_normal((H, N, d))
        before = bank.copy()
        rec = O.update_layer(bank, K, V, step=t, prm=prm, literal=literal)
        out.append((before, K, V, rec, bank.copy()))
    return out


# --------------------------------------------------------------------------- P4: Alg. 1 per-r
def check_literal_prefix_enumeration(O):
    """The cumulative-sum prefix table equals a from-scratch recomputation for every r."""
    for seed in range(6):
        prm = _prm(O, sigma=1.0, p=2.0, tau=1.6)
        a = _random_bank_rollout(O, seed, prm=prm, literal=False)
        b = _random_bank_rollout(O, seed, prm=prm, literal=True)
        for (_, _, _, ra, ba), (_, _, _, rb, bb) in zip(a, b):
            assert ra.r_star == rb.r_star
            for ha, hb_ in zip(ra.heads, rb.heads):
                if ha.counts is not None:
                    assert np.array_equal(ha.counts, hb_.counts)
                    assert np.all(np.diff(ha.counts) >= 0)          # c_r non-decreasing
            for xa, xb in zip(ba.heads, bb.heads):
                assert np.array_equal(xa.K, xb.K) and np.allclose(xa.rho, xb.rho, rtol=1e-12)


def _brute_update_decision(O, before, K, prm):
    """r* by brute force from the definitions (explicit loops over r, i, j)."""
    H = len(before.heads)
    N = K.shape[1]
    live = [h for h in range(H) if before.heads[h].m > 0]
    if not live:
        return None
    rmax = min([N] + [before.heads[h].M for h in live])
    feas_all = [True] * (rmax + 1)
    for h in live:
        hb = before.heads[h]
        s = prm.sigma_for(hb.d)
        w = lambda a, b: (prm.eps + float(np.sum((a - b) ** 2)) / (s * s)) ** (-prm.p)
        if getattr(prm, "order", "score") == "source":
            pi = list(range(N))
        else:
            score = [sum(w(hb.K[i], K[h][x]) / float(hb.base[i]) for i in range(hb.m)) / hb.m for x in range(N)]
            pi = sorted(range(N), key=lambda x: (score[x], x))
        for r in range(rmax + 1):
            c = 0
            for i in range(hb.m):
                rt = float(hb.rho[i]) + sum(w(hb.K[i], K[h][pi[j]]) for j in range(r))
                if rt / float(hb.base[i]) >= prm.tau:
                    c += 1
            if r > 0 and c > max(0, hb.m + r - hb.M):
                feas_all[r] = False
    return max(r for r in range(rmax + 1) if feas_all[r])


def check_rstar_brute_force(O):
    for seed in range(5):
        prm = _prm(O, sigma=1.0, p=2.0, tau=1.5)
        for before, K, V, rec, after in _random_bank_rollout(O, 100 + seed, prm=prm, steps=4):
            r_bf = _brute_update_decision(O, before, K, prm)
            if r_bf is not None:
                assert rec.r_star == r_bf, (seed, rec.r_star, r_bf)


# --------------------------------------------------------------------------- P5-P7: invariants
def check_invariants(O):
    for seed in range(4):
        for tau in (1.3, 2.0):
            prm = _prm(O, sigma=1.0, p=2.0, tau=tau)
            for t, (before, K, V, rec, after) in enumerate(
                    _random_bank_rollout(O, 200 + seed, prm=prm, steps=6, M=10, N=7)):
                N = K.shape[1]
                for h, (hb0, hb1, hr) in enumerate(zip(before.heads, after.heads, rec.heads)):
                    assert hb1.m <= hb1.M                                   # budget
                    assert hb1.m == hb0.m + hr.r_used - len(hr.evicted)
                    if hb0.m == 0:
                        # empty bank: first min(N, M) candidates in source order
                        assert hr.r_used == min(N, hb0.M)
                        assert list(hb1.src) == list(range(hr.r_used))
                    else:
                        assert hr.r_used == rec.r_star                      # all heads admit r*
                        e = max(0, hb0.m + rec.r_star - hb0.M)
                        assert len(hr.evicted) == e                         # |R| = e_{r*}
                        if hb0.m + rec.r_star <= hb0.M:
                            assert len(hr.evicted) == 0                     # under budget: no eviction
                        # mandatory states are all in R; they are exactly g(r*) >= tau
                        assert set(np.nonzero(hr.mandatory)[0]) <= set(hr.evicted.tolist())
                        if rec.r_star > 0:
                            assert np.array_equal(hr.mandatory, hr.g_star >= tau)
                        # fill picks the largest rho~ among the non-mandatory
                        fill = [i for i in hr.evicted if not hr.mandatory[i]]
                        rest = [i for i in range(hb0.m) if i not in set(hr.evicted.tolist())]
                        if fill and rest:
                            assert min(hr.rho_tilde[fill]) >= max(hr.rho_tilde[i] for i in rest
                                                                  if not hr.mandatory[i])
                        # survivors keep b; admitted candidates are the pi prefix
                        prov0 = {(int(a), int(b)): float(x) for a, b, x in zip(hb0.step, hb0.src, hb0.base)}
                        for a, b, x in zip(hb1.step, hb1.src, hb1.base):
                            if (int(a), int(b)) in prov0:
                                assert float(x) == prov0[(int(a), int(b))]
                        assert sorted(hr.admitted.tolist()) == sorted(hr.pi[:rec.r_star].tolist())
                    # P6: every retained (k, v) equals its source bit for bit
                    src_rows = {}
                    for i in range(hb0.m):
                        src_rows[(int(hb0.step[i]), int(hb0.src[i]))] = (hb0.K[i], hb0.V[i])
                    for i in range(hb1.m):
                        key = (int(hb1.step[i]), int(hb1.src[i]))
                        if key in src_rows:
                            k, v = src_rows[key]
                        else:
                            k, v = K[h][key[1]], V[h][key[1]]
                        assert np.array_equal(hb1.K[i], k) and np.array_equal(hb1.V[i], v)
                    # P7: cached rho equals the from-scratch density (fp64 storage)
                    phi = O.density(hb1.K, prm)
                    assert np.allclose(hb1.rho, phi, rtol=1e-9, atol=1e-12)
                    # App. C invariant: every retained state has g < tau; new states g <= 1
                    g = phi / hb1.base
                    assert np.all(g < tau)
                    assert np.all(g[hb1.step == t] <= 1.0 + 1e-12)


# --------------------------------------------------------------------------- P8: special cases
def check_special_cases(O):
    prm = _prm(O)
    rng = np.random.default_rng(3)
    d = 16
    # (ii) candidates far from the bank: no violators -> r* = min(N, M), eviction by densest fill
    bank = O.LayerBank.empty([12], d, store=np.float64)
    O.update_layer(bank, rng.standard_normal((1, 12, d)), rng.standard_normal((1, 12, d)), 0, prm)
    far = rng.standard_normal((1, 5, d)) + 1e4
    rho_before = bank.heads[0].rho.copy()
    rec = O.update_layer(bank, far, rng.standard_normal((1, 5, d)), 1, prm)
    hr = rec.heads[0]
    assert rec.r_star == 5 and not hr.mandatory.any() and len(hr.evicted) == 5
    assert set(hr.evicted.tolist()) == set(np.argsort(-rho_before, kind="stable")[:5].tolist())
    # (iii) identical candidate keys -> equal scores -> source order
    bank = O.LayerBank.empty([6], d, store=np.float64)
    O.update_layer(bank, rng.standard_normal((1, 6, d)), rng.standard_normal((1, 6, d)), 0, prm)
    dup = np.repeat(rng.standard_normal((1, 1, d)), 4, axis=1)
    rec = O.update_layer(bank, dup, rng.standard_normal((1, 4, d)), 1, prm)
    assert list(rec.heads[0].pi) == [0, 1, 2, 3]
    # fill ties are broken by provenance: older first.  Bank of 4 identical keys, far candidate.
    bank = O.LayerBank.empty([4], d, store=np.float64)
    same = np.repeat(rng.standard_normal((1, 1, d)), 4, axis=1)
    O.update_layer(bank, same, rng.standard_normal((1, 4, d)), 0, prm)
    rec = O.update_layer(bank, rng.standard_normal((1, 2, d)) + 1e4, rng.standard_normal((1, 2, d)),
                         1, prm)
    assert sorted(rec.heads[0].evicted.tolist()) == [0, 1]
    # (iv) scale equivalence (App. B): eps sigma^2 fixed -> same decisions, rho scaled by (eps'/eps)^-p
    rng = np.random.default_rng(4)
    stream = [(rng.standard_normal((2, 8, 4)) * 2, rng.standard_normal((2, 8, 4))) for _ in range(5)]
    pa = _prm(O, eps=1.0, sigma=2.0, delta=1e-30, tau=1.5)
    pb = _prm(O, eps=4.0, sigma=1.0, delta=1e-30, tau=1.5)
    ba = O.LayerBank.empty([11, 11], 4, store=np.float64)
    bb = O.LayerBank.empty([11, 11], 4, store=np.float64)
    for t, (K, V) in enumerate(stream):
        ra = O.update_layer(ba, K, V, t, pa)
        rb = O.update_layer(bb, K, V, t, pb)
        assert ra.r_star == rb.r_star
        for xa, xb in zip(ba.heads, bb.heads):
            assert np.array_equal(xa.src, xb.src) and np.array_equal(xa.step, xb.step)
            assert np.allclose(xb.rho, xa.rho * 4.0 ** -2, rtol=1e-9)
    # (i) empty bank with N > M: the first M candidates in source order, keys and values exact
    bank = O.LayerBank.empty([3], d, store=np.float64)
    Kc, Vc = rng.standard_normal((1, 5, d)), rng.standard_normal((1, 5, d))
    rec = O.update_layer(bank, Kc, Vc, 7, prm)
    hb = bank.heads[0]
    assert rec.heads[0].r_used == 3 and list(hb.src) == [0, 1, 2] and list(hb.step) == [7, 7, 7]
    assert np.array_equal(hb.K, Kc[0, :3]) and np.array_equal(hb.V, Vc[0, :3])
    # g = tau exactly counts as a violation (inclusive comparison, Eq. 9).  Two coincident keys:
    # rho = b = 1; a third coincident candidate gives g(1) = 2 = tau for both, c_1 = 2 > e_1 = 1.
    p2 = _prm(O, sigma=1.0, tau=2.0)
    bank = O.LayerBank.empty([2], 2, store=np.float64)
    O.update_layer(bank, np.ones((1, 2, 2)), np.ones((1, 2, 2)), 0, p2)
    rec = O.update_layer(bank, np.ones((1, 1, 2)), np.ones((1, 1, 2)), 1, p2)
    assert list(rec.heads[0].counts) == [0, 2] and rec.r_star == 0
    # r* = 0 leaves the bank unchanged.  Three coincident keys: rho = b = 2 (w = 1 each).
    # One more coincident candidate gives g = 3/2 >= tau = 1.4 for all three: c_1 = 3 > e_1 = 1.
    p14 = _prm(O, sigma=1.0, tau=1.4)
    bank = O.LayerBank.empty([3], 2, store=np.float64)
    O.update_layer(bank, np.zeros((1, 3, 2)), np.ones((1, 3, 2)), 0, p14)
    snap = bank.copy()
    rec = O.update_layer(bank, np.zeros((1, 2, 2)), np.ones((1, 2, 2)), 1, p14)
    assert rec.r_star == 0 and list(rec.heads[0].counts) == [0, 3, 3]
    assert np.array_equal(snap.heads[0].K, bank.heads[0].K) and np.array_equal(snap.heads[0].rho, bank.heads[0].rho)


def check_shared_prefix_across_heads(O):
    """One head whose candidates sit on top of its bank limits r* for both heads (Eq. 11);
    with sync_heads=False each head takes its own largest feasible prefix (App. E)."""
    rng = np.random.default_rng(5)
    d = 8
    Kb = rng.standard_normal((2, 6, d)) * 3
    for sync in (True, False):
        prm = _prm(O, sigma=1.0, sync_heads=sync)
        bank = O.LayerBank.empty([8, 8], d, store=np.float64)
        O.update_layer(bank, Kb, rng.standard_normal((2, 6, d)), 0, prm)
        Kc = np.empty((2, 4, d))
        Kc[0] = rng.standard_normal((4, d)) * 3 + 100.0     # head 0: far -> wants r = 4
        Kc[1] = Kb[1, :4]                                  # head 1: duplicates -> violators
        rec = O.update_layer(bank, Kc, rng.standard_normal((2, 4, d)), 1, prm)
        r0, r1 = rec.heads[0].r_used, rec.heads[1].r_used
        if sync:
            assert r0 == r1 == rec.r_star < 4
        else:
            assert r0 == 4 and r1 < 4


# --------------------------------------------------------------------------- P9: App. D storage
def check_storage_accounting(O):
    g = json.load(open(os.path.join(GOLDEN, "storage_app_d.json")))
    for case in g["cases"]:
        sb = O.storage_bytes(case["L"], case["H"], case["n"], case["dk"], case["dv"])
        assert round(sb["kv"] / O.GIB, 2) == case["kv_gib"], (sb, case)
        assert round(sb["total"] / O.GIB, 2) == case["bank_total_gib"], (sb, case)
        if "with_window_gib" in case:
            win = O.storage_bytes(case["L"], case["H"], case["window_states"], case["dk"], case["dv"])
            assert round((sb["total"] + win["kv"]) / O.GIB, 2) == case["with_window_gib"]


# --------------------------------------------------------------------------- P10: attention
def check_attention_textbook(O):
    import torch
    rng = np.random.default_rng(6)
    d = 16
    bank = O.LayerBank.empty([20], d, store=np.float64)
    O.update_layer(bank, rng.standard_normal((1, 13, d)), rng.standard_normal((1, 13, d)), 0, _prm(O))
    hb = bank.heads[0]
    Q = rng.standard_normal((9, d)) * 2
    Kw, Vw = rng.standard_normal((7, d)), rng.standard_normal((7, d))
    out = O.attend(hb, Q, Kw, Vw)
    Kall = np.concatenate([hb.K, Kw])
    Vall = np.concatenate([hb.V, Vw])
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(Q)[None], torch.from_numpy(Kall)[None], torch.from_numpy(Vall)[None]
    )[0].numpy()
    assert np.allclose(out, ref, atol=1e-12), np.abs(out - ref).max()
    # invariant to a permutation of the bank slots
    perm = rng.permutation(hb.m)
    hp = hb.copy()
    hp.K, hp.V = hb.K[perm], hb.V[perm]
    assert np.allclose(O.attend(hp, Q, Kw, Vw), out, atol=1e-12)
    # empty bank -> window-only attention
    eb = O.LayerBank.empty([4], d).heads[0]
    ref2 = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(Q)[None], torch.from_numpy(Kw)[None], torch.from_numpy(Vw)[None])[0].numpy()
    assert np.allclose(O.attend(eb, Q, Kw, Vw), ref2, atol=1e-12)


# --------------------------------------------------------------------------- P9: policy ablations
def _expected_eviction(hr, hb0, e, evict):
    """R re-derived with explicit sorts from rho~, the mandatory flags and provenance."""
    idx = list(range(hb0.m))
    prov = lambda i: (int(hb0.step[i]), int(hb0.src[i]))
    if evict == "densest":
        return sorted(idx, key=lambda i: (-float(hr.rho_tilde[i]), prov(i)))[:e]
    mand = [i for i in idx if hr.mandatory[i]]
    rest = [i for i in idx if not hr.mandatory[i]]
    if evict == "mandatory_source":
        rest = sorted(rest, key=prov)
    else:
        rest = sorted(rest, key=lambda i: (-float(hr.rho_tilde[i]), prov(i)))
    return mand + rest[:e - len(mand)]


def check_policy_variants(O):
    """Table 2(b) / App. E ablations: source-order candidates, densest-only and
    mandatory + source eviction, refreshed baselines (each alone and combined)."""
    variants = [dict(order="source"), dict(evict="densest"), dict(evict="mandatory_source"),
                dict(refresh_baselines=True), dict(order="source", evict="densest", refresh_baselines=True)]
    for vi, kw in enumerate(variants):
        for seed in range(3):
            prm = _prm(O, sigma=1.0, p=2.0, tau=1.5, **kw)
            for t, (before, K, V, rec, after) in enumerate(
                    _random_bank_rollout(O, 500 + 10 * vi + seed, prm=prm, steps=5, M=10, N=7)):
                r_bf = _brute_update_decision(O, before, K, prm)
                if r_bf is not None:
                    assert rec.r_star == r_bf, (kw, seed, t, rec.r_star, r_bf)
                for h, (hb0, hb1, hr) in enumerate(zip(before.heads, after.heads, rec.heads)):
                    assert hb1.m <= hb1.M
                    if hb0.m == 0:
                        continue
                    if prm.order == "source":
                        assert np.array_equal(hr.pi, np.arange(K.shape[1]))
                    assert hr.admitted.tolist() == hr.pi[:rec.r_star].tolist()
                    e = max(0, hb0.m + rec.r_star - hb0.M)
                    assert sorted(hr.evicted.tolist()) == sorted(_expected_eviction(hr, hb0, e, prm.evict))
                    phi = O.density(hb1.K, prm)
                    assert np.allclose(hb1.rho, phi, rtol=1e-9, atol=1e-12)
                    prov0 = {(int(a), int(b)): float(x) for a, b, x in zip(hb0.step, hb0.src, hb0.base)}
                    for i, (a, b) in enumerate(zip(hb1.step, hb1.src)):
                        if prm.refresh_baselines:
                            assert float(hb1.base[i]) == max(float(hb1.rho[i]), prm.delta)
                        elif (int(a), int(b)) in prov0:
                            assert float(hb1.base[i]) == prov0[(int(a), int(b))]

    # Densest-only eviction can keep a threshold crosser that the default evicts: an isolated
    # state with a tiny baseline (g >= tau) next to a dense pair, one candidate far away.
    d = 2
    Kb = np.array([[10.0, 0.0], [0.0, 0.0], [0.1, 0.0]])
    prm0 = _prm(O, sigma=1.0, p=2.0, tau=2.0)
    rho = O.density(Kb, prm0)
    base = rho.copy()
    base[0] = rho[0] / 4.0                         # g_0(0) = 4 >= tau
    Kc = np.array([[[-50.0, 0.0]]])
    Vc = np.zeros((1, 1, d))
    outs = {}
    for ev in ("mandatory_densest", "densest"):
        prm = _prm(O, sigma=1.0, p=2.0, tau=2.0, evict=ev)
        bank = O.LayerBank.empty([3], d, store=np.float64)
        hb = bank.heads[0]
        hb.K, hb.V = Kb.copy(), np.zeros((3, d))
        hb.rho, hb.base = rho.copy(), base.copy()
        hb.step, hb.src = np.zeros(3, np.int64), np.arange(3, dtype=np.int64)
        rec = O.update_layer(bank, Kc, Vc, step=1, prm=prm)
        assert rec.r_star == 1
        outs[ev] = sorted(rec.heads[0].evicted.tolist())
    assert outs["mandatory_densest"] == [0]        # the crosser goes first
    assert outs["densest"] in ([1], [2])           # the densest of the pair instead



def check_sequential_admission(O):
    """Within-block competition (App. E), read as one-candidate updates in the order fixed
    at block start.  Pinned independently of the oracle's code: (1) after every block the
    cached densities equal the exact Soft-Riesz density over the bank (Eq. 3, self
    excluded) and states of earlier blocks keep their frozen baselines and provenance;
    (2) two identical candidates offered to a bank that is not full and lies far from them
    are both admitted by the default update (their mutual interaction only enters their
    new baselines), but sequentially the second is gated out: once the first is in, the
    duplicate would raise its density by w(0) = eps^-p, far beyond tau times its baseline,
    and a bank with free room has no eviction budget for it (e_1 = 0); (3) the offers follow
    the ascending Eq. 6 order of block start: with every bank state on the +e0 side,
    x' = +0.25 e0 (source index 0) scores above x = -0.25 e0 (index 1), so x is offered and
    admitted first and x' is gated out; (4) an all-empty bank is initialised by the whole
    block as in the default, and a partly empty bank is refused."""
    rng = np.random.default_rng(3)
    for sync in (True, False):
        prm = _prm(O, sync_heads=sync)
        ob = O.LayerBank.empty([24, 30], 8)
        O.update_layer_sequential(ob, rng.standard_normal((2, 16, 8)) * 2, rng.standard_normal((2, 16, 8)), 0, prm)
        for t in range(1, 4):
            before = [dict(zip(zip(hb.step.tolist(), hb.src.tolist()), hb.base.tolist())) for hb in ob.heads]
            O.update_layer_sequential(ob, rng.standard_normal((2, 12, 8)) * 2, rng.standard_normal((2, 12, 8)), t, prm)
            for h, hb in enumerate(ob.heads):
                assert hb.m <= hb.M
                K = hb.K.astype(np.float64)
                d2 = ((K[:, None, :] - K[None, :, :]) ** 2).sum(-1)
                W = (prm.eps + d2 / prm.sigma_for(8) ** 2) ** (-prm.p)
                np.fill_diagonal(W, 0.0)
                np.testing.assert_allclose(hb.rho.astype(np.float64), W.sum(axis=1), rtol=2e-6, atol=1e-30)
                keys = list(zip(hb.step.tolist(), hb.src.tolist()))
                assert len(set(keys)) == len(keys)
                for k, b in zip(keys, hb.base.tolist()):
                    if k[0] < t:
                        assert before[h][k] == b
                    else:
                        assert k[0] == t and 0 <= k[1] < 12

    prm = _prm(O)
    e0 = np.eye(8)[0]

    def far_bank():
        r = np.random.default_rng(5)
        K0 = r.standard_normal((1, 20, 8))
        K0 = K0 / np.linalg.norm(K0, axis=2, keepdims=True) * 6.0
        ob = O.LayerBank.empty([40], 8)
        O.update_layer(ob, K0, K0, 0, prm)
        return ob

    block = np.stack([0.25 * e0, 0.25 * e0])[None]
    default = far_bank()
    assert O.update_layer(default, block, block, 1, prm).r_star == 2 and default.heads[0].m == 22
    seq = far_bank()
    assert [r.r_star for r in O.update_layer_sequential(seq, block, block, 1, prm)] == [1, 0]
    hb = seq.heads[0]
    assert hb.m == 21 and [s for st, s in zip(hb.step.tolist(), hb.src.tolist()) if st == 1] == [0]

    u = np.random.default_rng(11).standard_normal((20, 8))
    K0 = 6.0 * e0 + 3.0 * u / np.linalg.norm(u, axis=1, keepdims=True)   # first coordinate >= 3
    ob = O.LayerBank.empty([40], 8)
    O.update_layer(ob, K0[None], K0[None], 0, prm)
    block = np.stack([0.25 * e0, -0.25 * e0])[None]
    assert [r.r_star for r in O.update_layer_sequential(ob, block, block, 1, prm)] == [1, 0]
    hb = ob.heads[0]
    assert [s for st, s in zip(hb.step.tolist(), hb.src.tolist()) if st == 1] == [1]

    K = np.random.default_rng(9).standard_normal((2, 10, 8))
    a, b = O.LayerBank.empty([6, 8], 8), O.LayerBank.empty([6, 8], 8)
    O.update_layer_sequential(a, K, K, 0, prm)
    O.update_layer(b, K, K, 0, prm)
    for ha, hb in zip(a.heads, b.heads):
        assert np.array_equal(ha.K, hb.K) and np.array_equal(ha.base, hb.base)
    b.heads[1] = O.HeadBank(M=8, d=8, dv=8)
    try:
        O.update_layer_sequential(b, K, K, 1, prm)
    except ValueError:
        pass
    else:
        raise AssertionError("a partly empty bank was accepted")


# --------------------------------------------------------------------------- storage rounding
def _bf16_neighbours(v):
    """Brute force: every bf16 value within two bf16 steps of v (8 significant bits)."""
    if v == 0.0:
        return [0.0]
    e = math.floor(math.log2(abs(v)))
    out = set()
    for ee in (e - 1, e, e + 1):
        step = 2.0 ** (ee - 7)
        base = math.floor(abs(v) / step)
        for k in range(base - 2, base + 3):
            if 128 <= k < 256:
                out.add(math.copysign(k * step, v))
    return sorted(out)


def check_round_nearest_bf16(O):
    rng = np.random.default_rng(41)
    # brute force: the nearest of the enumerated bf16 values, ties to the even significand
    xs = np.concatenate([rng.normal(size=400) * 4.0, rng.uniform(-1e3, 1e3, size=100)])
    got = O.round_nearest_bf16(xs)
    for x, g in zip(xs, got):
        cand = _bf16_neighbours(float(x))
        best = min(abs(c - x) for c in cand)
        near = [c for c in cand if abs(c - x) == best]
        if len(near) == 2:       # tie: the one whose 8-bit significand is even
            near = [c for c in near if int(abs(c) / 2.0 ** (math.floor(math.log2(abs(c))) - 7)) % 2 == 0]
        assert g == near[0], (x, g, near)
    # hand cases: ties to even around 1, and one float64 value just above a tie, which
    # rounds up here but to the even neighbour 1 if it went through float32 first
    hand = np.array([1 + 2.0 ** -8, 1 + 3 * 2.0 ** -8, 1 + 2.0 ** -8 + 2.0 ** -30, -(1 + 2.0 ** -8 + 2.0 ** -30),
                     0.0, 255.0, 257.0, 259.0])
    want = np.array([1.0, 1 + 2.0 ** -6, 1 + 2.0 ** -7, -(1 + 2.0 ** -7), 0.0, 255.0, 256.0, 260.0])
    assert np.array_equal(O.round_nearest_bf16(hand), want), O.round_nearest_bf16(hand)
    # float32 inputs: the library conversion (torch float32 -> bfloat16 rounds to nearest even)
    import torch
    f = (rng.normal(size=2000) * 3.0).astype(np.float32)
    lib = torch.from_numpy(f).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(O.round_nearest_bf16(f.astype(np.float64)), lib)


# --------------------------------------------------------------------------- App. A: temporal RoPE coordinate 0
def _rope_forward(K0, t, theta, layout):
    """Rotary embedding of temporal coordinate t written as complex multiplication:
    pair j as z = x + i y, rotated to z e^{i t theta_j} (RoFormer convention)."""
    K0 = np.asarray(K0, dtype=np.float64)
    d = K0.shape[-1]
    xi, yi = (np.arange(0, d, 2), np.arange(1, d, 2)) if layout == "interleaved" else \
        (np.arange(d // 2), np.arange(d // 2, d))
    z = K0[..., xi] + 1j * K0[..., yi]
    z = z * np.exp(1j * np.asarray(t, dtype=np.float64)[:, None] * np.asarray(theta, np.float32).astype(np.float64))
    out = K0.copy()
    out[..., xi], out[..., yi] = z.real, z.imag
    return out


def check_rope_rezero(O):
    rng = np.random.default_rng(43)
    H, N, d = 2, 7, 16
    theta = np.zeros(d // 2, dtype=np.float32)
    theta[:3] = 10000.0 ** (-np.arange(3) / 3.0)      # a temporal band of three pairs; the rest spatial
    t = np.array([0, 1, 1, 2, 5, 37, -4])
    K0 = rng.normal(size=(H, N, d))
    for layout in ("interleaved", "half"):
        # rotating back undoes the forward embedding (the sign and direction of the angle)
        Kt = _rope_forward(K0, t, theta, layout)
        back = O.rope_rezero(Kt, t, theta, layout, storage=None)
        assert np.allclose(back, K0, rtol=0, atol=1e-12), layout
        # rotations keep norms and, at a common coordinate, inner products
        assert np.allclose(np.linalg.norm(back, axis=-1), np.linalg.norm(Kt, axis=-1), rtol=1e-13)
        same = t == 1
        g1 = np.einsum("hnd,hmd->hnm", Kt[:, same], Kt[:, same])
        g0 = np.einsum("hnd,hmd->hnm", back[:, same], back[:, same])
        assert np.allclose(g0, g1, rtol=1e-12, atol=1e-12)
        # coordinate 0 and the spatial pairs come back bit for bit
        Kb = O.round_nearest_bf16(rng.normal(size=(H, N, d)))
        out = O.rope_rezero(Kb, t, theta, layout)
        assert np.array_equal(out[:, t == 0], Kb[:, t == 0])
        sp = np.nonzero(theta == 0)[0]
        idx = np.concatenate([2 * sp, 2 * sp + 1]) if layout == "interleaved" else np.concatenate([sp, sp + d // 2])
        assert np.array_equal(out[..., idx], Kb[..., idx])
        # the stored keys are the nearest bf16 values of the exact rotation
        exact = O.rope_rezero(Kb, t, theta, layout, storage=None)
        assert np.array_equal(out, O.round_nearest_bf16(exact))
        assert np.array_equal(O.rope_rezero(Kb, t, theta, layout, storage="fp32"),
                              exact.astype(np.float32).astype(np.float64))
    # a quarter turn by hand: theta = pi/2 (as float32), t = 1: (x, y) -> (y, -x)
    th = np.zeros(2, dtype=np.float32)
    th[0] = np.float32(np.pi / 2)
    k = np.array([[[3.0, 5.0, 7.0, 11.0]]])
    q = O.rope_rezero(k, np.array([1]), th, "interleaved", storage=None)
    assert np.allclose(q, [[[5.0, -3.0, 7.0, 11.0]]], rtol=0, atol=1e-6), q
    q = O.rope_rezero(k, np.array([1]), th, "half", storage=None)     # pair 0 = elements (0, 2)
    assert np.allclose(q, [[[7.0, 5.0, -3.0, 11.0]]], rtol=0, atol=1e-6), q
    # two quarter turns are a half turn: t = 2 -> (-x, -y)
    q = O.rope_rezero(k, np.array([2]), th, "interleaved", storage=None)
    assert np.allclose(q, [[[-3.0, -5.0, 7.0, 11.0]]], rtol=0, atol=1e-6), q
    # half layout is interleaved layout on the channel-permuted key
    perm = np.empty(d, dtype=np.int64)
    perm[0::2], perm[1::2] = np.arange(d // 2), np.arange(d // 2, d)
    Kt = rng.normal(size=(H, N, d))
    a = O.rope_rezero(Kt, t, theta, "half", storage=None)[..., perm]
    b = O.rope_rezero(Kt[..., perm], t, theta, "interleaved", storage=None)
    assert np.array_equal(a, b)


# --------------------------------------------------------------------------- App. E: [K; V] descriptor
def check_kv_descriptor(O):
    rng = np.random.default_rng(47)
    H, d, N, M, steps = 2, 3, 6, 9, 4
    prm = _prm(O, sigma=2.0)

    def rollout(make):
        bank = O.LayerBank.empty([M] * H, 2 * d)
        out = []
        for t in range(steps):
            K = rng_k[t]
            V = rng_v[t]
            rec = O.update_layer(bank, make(K, V), V, t, prm)
            out.append((rec.r_star, [sorted(zip(hb.step.tolist(), hb.src.tolist())) for hb in bank.heads],
                        [np.sort(hb.rho) for hb in bank.heads]))
        return bank, out

    rng_k = [rng.normal(size=(H, N, d)) for _ in range(steps)]
    rng_v = [rng.normal(size=(H, N, d)) for _ in range(steps)]
    # the descriptor is the key followed by the value; stored rows keep both
    D = O.kv_descriptor(rng_k[0], rng_v[0])
    assert D.shape == (H, N, 2 * d) and np.array_equal(D[..., :d], rng_k[0]) and np.array_equal(D[..., d:], rng_v[0])
    # distances are permutation-invariant over coordinates: [V; K] decides exactly as [K; V]
    _, a = rollout(O.kv_descriptor)
    _, b = rollout(lambda K, V: O.kv_descriptor(V, K))
    for (ra, pa, qa), (rb, pb, qb) in zip(a, b):
        assert ra == rb and pa == pb
        assert all(np.allclose(x, y, rtol=1e-12, atol=0) for x, y in zip(qa, qb))
    # with all values equal the descriptor geometry is that of the keys (same sigma)
    bank_k = O.LayerBank.empty([M] * H, d)
    bank_kv = O.LayerBank.empty([M] * H, 2 * d)
    for t in range(steps):
        V1 = np.ones((H, N, d))
        rk = O.update_layer(bank_k, rng_k[t], V1, t, prm)
        rkv = O.update_layer(bank_kv, O.kv_descriptor(rng_k[t], V1), V1, t, prm)
        assert rk.r_star == rkv.r_star
        for hk, hkv in zip(bank_k.heads, bank_kv.heads):
            assert np.array_equal(hk.step, hkv.step) and np.array_equal(hk.src, hkv.src)
            assert np.allclose(hk.rho, hkv.rho, rtol=1e-12) and np.array_equal(hk.K, hkv.K[:, :d])
    # the descriptor default bandwidth is sqrt(2 d / 2) = sqrt(d) (App. B rule at dimension 2 d)
    assert abs(O.Params().sigma_for(2 * 64) - 8.0) < 1e-15


ALL_CHECKS = [
    check_kernel_closed_forms,
    check_distance_identities,
    check_density_brute_force,
    check_worked_example,
    check_literal_prefix_enumeration,
    check_rstar_brute_force,
    check_invariants,
    check_special_cases,
    check_shared_prefix_across_heads,
    check_storage_accounting,
    check_attention_textbook,
    check_policy_variants,
    check_sequential_admission,
    check_round_nearest_bf16,
    check_rope_rezero,
    check_kv_descriptor,
]
