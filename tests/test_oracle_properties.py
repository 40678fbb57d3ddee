"""Randomised properties of the oracle's bank update (Alg. 1, App. C), beside the
fixed-seed pins: random sizes, exponents p in {1, 2, 4} (Table 2a), tau, sigma, eps,
and both prefix rules (shared across heads, Eq. 11; independent per head, App. E).

After every update, for every head:
  * the bank never exceeds its budget; m' = m + r - |R|;
  * an empty bank admits its first min(N, M) candidates in source order;
  * otherwise its Eq. 6 scores equal explicit loops over the definition, the head
    admits r* (its own r*_h without the shared prefix), and r* is the
    largest prefix r <= min(N, min_h M_h) (over the heads with a bank; the layer's
    prefix range under either rule) that is feasible for every head (for the head) by
    brute force from the definitions: c_r = #{i : (rho_i + sum_{j < r} w(k_i, x_pi(j))) / b_i >= tau} against
    e_r = max(0, m + r - M) (Eqs. 8-11), pi the stable ascending Eq. 6 order;
  * |R| = e_{r*}; no eviction under budget; every mandatory state is evicted and the
    fill takes the largest rho~(r*) (Step 3); the admitted states are the pi prefix;
  * survivors keep their baselines; every retained (k, v) is its source bit for bit;
  * cached rho equals the from-scratch density Phi over the bank (Eq. C.4; float64
    storage here, as in the fixed-seed pin), and every retained state has g < tau, new
    states g <= 1 (App. C, "Invariant after commit").
"""
import numpy as np
import pytest

pytest.importorskip("hypothesis")
from hypothesis import HealthCheck, given, settings, strategies as st  # noqa: E402

import oracle  # noqa: E402


def _w(prm, d, a, b):
    s = prm.sigma_for(d)
    return (prm.eps + float(np.sum((a - b) ** 2)) / (s * s)) ** (-prm.p)


def _scores(hb, Kh, prm):
    """Eq. 6 for every candidate, as explicit loops."""
    return [sum(_w(prm, hb.d, hb.K[i], Kh[x]) / float(hb.base[i]) for i in range(hb.m)) / hb.m
            for x in range(Kh.shape[0])]


def _order(hb, Kh, prm):
    """pi: stable ascending Eq. 6 order, or source order under the source-order policy."""
    N = Kh.shape[0]
    if prm.order == "source":
        return list(range(N))
    score = _scores(hb, Kh, prm)
    return sorted(range(N), key=lambda x: (score[x], x))


def _feasible(hb, Kh, prm, r_hi):
    """Feasibility of every prefix length r <= r_hi for one head, from the definitions."""
    pi = _order(hb, Kh, prm)
    feas = []
    for r in range(r_hi + 1):
        c = 0
        for i in range(hb.m):
            rt = float(hb.rho[i]) + sum(_w(prm, hb.d, hb.K[i], Kh[pi[j]]) for j in range(r))
            c += rt / float(hb.base[i]) >= prm.tau
        feas.append(r == 0 or c <= max(0, hb.m + r - hb.M))
    return feas


def update_properties(O, seed, H, d, N, M, p, tau, sigma, eps, sync, steps, order="score",
                      evict="mandatory_densest", refresh=False):
    """Every property above on one random rollout of oracle module O, under the given
    policy (Table 2(b), App. E)."""
    rng = np.random.default_rng(seed)
    prm = O.Params(tau=tau, sigma=sigma, p=p, eps=eps, sync_heads=sync, order=order, evict=evict,
                   refresh_baselines=refresh)
    budgets = [int(x) for x in rng.integers(max(1, M // 2), M + 1, size=H)]
    bank = O.LayerBank.empty(budgets, d, store=np.float64)   # fp64 storage: Eq. C.4 exact
    for t in range(steps):
        K = rng.standard_normal((H, N, d)) * (0.5 + 0.5 * t)
        V = rng.standard_normal((H, N, d))
        before = bank.copy()
        rec = O.update_layer(bank, K, V, step=t, prm=prm)
        live = [h for h in range(H) if before.heads[h].m > 0]
        if live:
            # the layer's prefix range r <= min(N, min_h M_h) over the heads with a bank,
            # with either prefix rule
            rmax = min([N] + [before.heads[h].M for h in live])
            feas = {h: np.array(_feasible(before.heads[h], K[h], prm, rmax)) for h in live}
            if sync:
                allf = np.logical_and.reduce([feas[h] for h in live])
                want = {h: int(np.nonzero(allf)[0].max()) for h in live}
            else:
                want = {h: int(np.nonzero(feas[h])[0].max()) for h in live}
        for h, (hb0, hb1, hr) in enumerate(zip(before.heads, bank.heads, rec.heads)):
            assert hb1.m <= hb1.M
            assert hb1.m == hb0.m + hr.r_used - len(hr.evicted)
            if hb0.m == 0:
                assert hr.r_used == min(N, hb0.M)
                assert list(hb1.src) == list(range(hr.r_used))
            else:
                r = hr.r_used
                sc = np.array(_scores(hb0, K[h], prm))
                assert np.allclose(hr.s, sc, rtol=1e-10, atol=0.0)
                gaps = np.diff(np.sort(sc))
                if order == "source" or (len(gaps) == 0 or gaps.min() > 1e-9 * np.abs(sc).max()):
                    assert list(hr.pi) == _order(hb0, K[h], prm)   # no near-tie: the order is unique
                assert r == want[h], (h, r, want[h])
                if sync:
                    assert r == rec.r_star
                e = max(0, hb0.m + r - hb0.M)
                assert len(hr.evicted) == e
                ev = set(hr.evicted.tolist())
                kept = [i for i in range(hb0.m) if i not in ev]
                prov = [(int(hb0.step[i]), int(hb0.src[i])) for i in range(hb0.m)]
                if evict == "densest":   # the e largest rho~(r*) of the whole bank
                    if ev and kept:
                        assert min(hr.rho_tilde[list(ev)]) >= max(hr.rho_tilde[kept])
                else:                    # mandatory first, then the fill rule
                    assert set(np.nonzero(hr.mandatory)[0]) <= ev
                    fill = [i for i in ev if not hr.mandatory[i]]
                    rest = [i for i in kept if not hr.mandatory[i]]
                    if fill and rest and evict == "mandatory_source":   # oldest provenance first
                        assert max(prov[i] for i in fill) < min(prov[i] for i in rest)
                    elif fill and rest:                                 # largest rho~(r*) first
                        assert min(hr.rho_tilde[fill]) >= max(hr.rho_tilde[rest])
                assert sorted(hr.admitted.tolist()) == sorted(hr.pi[:r].tolist())
                if not refresh:   # survivors keep their frozen baselines
                    prov0 = {(int(a), int(b)): float(x) for a, b, x in zip(hb0.step, hb0.src, hb0.base)}
                    for a, b, x in zip(hb1.step, hb1.src, hb1.base):
                        if (int(a), int(b)) in prov0:
                            assert float(x) == prov0[(int(a), int(b))]
            rows = {(int(hb0.step[i]), int(hb0.src[i])): (hb0.K[i], hb0.V[i]) for i in range(hb0.m)}
            for i in range(hb1.m):
                key = (int(hb1.step[i]), int(hb1.src[i]))
                k, v = rows[key] if key in rows else (K[h][key[1]], V[h][key[1]])
                assert np.array_equal(hb1.K[i], k) and np.array_equal(hb1.V[i], v)
            if hb1.m:
                phi = O.density(hb1.K, prm)
                assert np.allclose(hb1.rho, phi, rtol=1e-9, atol=1e-300)
                if refresh:       # every retained baseline follows its density
                    assert np.array_equal(hb1.base, np.maximum(hb1.rho, prm.delta))
                else:             # new states: b = max(Phi, delta)
                    new = hb1.step == t
                    assert np.allclose(hb1.base[new], np.maximum(phi[new], prm.delta), rtol=1e-12, atol=0.0)
                g = phi / hb1.base
                if evict != "densest":   # every threshold crosser was evicted
                    assert np.all(g[hb1.step != t] < tau)
                assert np.all(g[hb1.step == t] <= 1.0 + 1e-12)


PROPERTY_ARGS = dict(seed=st.integers(0, 2 ** 31 - 1), H=st.integers(1, 3), d=st.sampled_from([2, 3, 5]),
                     N=st.integers(1, 8), M=st.integers(1, 11), p=st.sampled_from([1.0, 2.0, 4.0]),
                     tau=st.floats(1.1, 3.0), sigma=st.floats(0.5, 3.0), eps=st.floats(0.2, 2.0),
                     sync=st.booleans(), steps=st.integers(1, 4))


@settings(max_examples=80, deadline=None, suppress_health_check=[HealthCheck.too_slow])
@given(**PROPERTY_ARGS)
def test_update_properties(seed, H, d, N, M, p, tau, sigma, eps, sync, steps):
    update_properties(oracle, seed, H, d, N, M, p, tau, sigma, eps, sync, steps)


@settings(max_examples=80, deadline=None, suppress_health_check=[HealthCheck.too_slow])
@given(order=st.sampled_from(["score", "source"]),
       evict=st.sampled_from(["mandatory_densest", "densest", "mandatory_source"]),
       refresh=st.booleans(), **PROPERTY_ARGS)
def test_policy_properties(order, evict, refresh, seed, H, d, N, M, p, tau, sigma, eps, sync, steps):
    """The ablation policies of Table 2(b) / App. E, each with its own eviction rule."""
    update_properties(oracle, seed, H, d, N, M, p, tau, sigma, eps, sync, steps, order, evict, refresh)
