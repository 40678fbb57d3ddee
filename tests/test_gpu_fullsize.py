"""Full-size parity in the launch configuration bench.py times (tensor-core mode).

At these sizes the oracle cannot replay whole updates, so every step is checked on
sampled outputs that the oracle computes one by one from the pre-update bank (read
back from the GPU), plus properties that must hold exactly at any size:
  * Eq. 6 score of sampled candidates (1e-2 relative);
  * pi is a permutation sorted by the GPU's own scores, ties in source order;
  * first crossing of sampled bank rows under the GPU's pi (equal, or g within 1e-3
    of tau at the boundary), and rho~(r*) of sampled rows (1e-2);
  * r* recomputed exactly from the GPU's crossing indices and budgets (Eq. 9-11);
  * the eviction set: |R| = e_{r*}, every mandatory state evicted, the fill takes the
    largest rho~ (Step 3);
  * the committed bank = (old bank minus R) plus pi[:r*], keys/values bit-exact;
  * cached densities of sampled survivors and new states vs Phi over the final bank
    (1e-2), b = max(rho, delta) for new states;
  * attention of sampled queries over [bank | window] (2e-2 absolute).
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import INT_MAX, to_dev

pytestmark = pytest.mark.gpu

TOL_DEC = 1e-3
TOL_DENS = 1e-2
TOL_ATTN = 2e-2


@pytest.fixture(scope="module")
def dkv():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_27922_gb300 import dkv as d
    return d


def _snapshot(bank):
    occ = bank.occupancy_host()
    return {
        "occ": occ,
        "K": bank.k.float().cpu().numpy().astype(np.float64),
        "V": bank.v.float().cpu().numpy(),
        "rho": bank.rho.cpu().numpy().copy(),
        "base": bank.base.cpu().numpy().copy(),
        "step": bank.prov_step.cpu().numpy().copy(),
        "src": bank.prov_src.cpu().numpy().copy(),
    }


def _w(prm, d, A, B):
    return oracle.soft_riesz(oracle.sq_dist(A, B), prm, d)


def _check_attention(bank, snap, prm, Q, Kw, Vw, rng, nsample=24):
    O = bank.attend(to_dev(Q, bank.dtype), to_dev(Kw, bank.dtype), to_dev(Vw, bank.dtype)).float().cpu().numpy()
    err = 0.0
    for h in rng.choice(bank.H, size=min(3, bank.H), replace=False):
        m = snap["occ"][h]
        hb = oracle.HeadBank(bank.budgets[h], bank.d, bank.d, snap["K"][h, :m], snap["V"][h, :m].astype(np.float64))
        qs = rng.choice(Q.shape[1], size=nsample, replace=False)
        ref = oracle.attend(hb, Q[h][qs], Kw[h], Vw[h])
        err = max(err, float(np.abs(O[h][qs] - ref).max()))
    assert err < TOL_ATTN, err


def _rstar_from_cross(cross_all, occ, budgets, rmax, sync):
    feas_all = np.ones(rmax + 1, bool)
    per_head = []
    for h, cr in enumerate(cross_all):
        m, M = occ[h], budgets[h]
        if m == 0:
            per_head.append(None)
            continue
        c = np.bincount(np.minimum(cr[cr != INT_MAX], rmax + 1), minlength=rmax + 2)[:rmax + 1].cumsum()
        e = np.maximum(0, m + np.arange(rmax + 1) - M)
        f = c <= e
        f[0] = True
        per_head.append(f)
        feas_all &= f
    if sync:
        return int(np.nonzero(feas_all)[0].max()), None
    return None, [None if f is None else int(np.nonzero(f)[0].max()) for f in per_head]


def _run(dkv, wl, steps, sync_heads=1, rows=40, cands=40, seed=0, kv=False):
    """kv: the [K; V] descriptor (App. E); every interaction below is then taken between
    [k; v] rows."""
    rng = np.random.default_rng(seed)
    extra = dict(descriptor=dkv.DKV_DESC_KV, sigma=float(np.sqrt(wl.d))) if kv else {}
    bank = dkv.BankLayer(wl.H, wl.d, wl.budgets_of_layer(0), wl.N, torch.bfloat16,
                         score_mode=dkv.DKV_SCORE_TENSOR, sync_heads=sync_heads, **extra)
    desc = (lambda K, V: oracle.kv_descriptor(K, V)) if kv else (lambda K, V: np.asarray(K, dtype=np.float64))
    bank.reset()
    prm = oracle.Params(tau=float(bank.params.tau), sigma=float(bank.params.sigma), p=float(bank.params.p),
                        eps=float(bank.params.eps), delta=float(np.float32(bank.params.delta)),
                        sync_heads=bool(sync_heads))
    ro = synth.LayerRollout(wl, 0)
    d = wl.d
    evicted_total = 0
    for t in range(steps):
        snap = _snapshot(bank)
        if t % 2 == 1:
            Kw, Vw = ro.window(t)
            _check_attention(bank, snap, prm, ro.queries(t), Kw, Vw, rng)
        b = wl.admitted_block(t)
        if b is None:
            continue
        Kc, Vc = ro.block(b)
        Kd, Vd = to_dev(Kc, torch.bfloat16), to_dev(Vc, torch.bfloat16)
        bank.admit(Kd, Vd, b)
        bank.compress()
        bank.sync()
        # score, pi and cross are set by admit, rho~ by compress; none is overwritten later
        inter = {k: v.cpu().numpy().copy() for k, v in bank.intermediates().items()}
        L, hs = bank.stats()
        after = _snapshot(bank)
        N = wl.N
        occ0 = snap["occ"]
        live = [h for h in range(wl.H) if occ0[h] > 0]
        # ---- r* from the GPU's own crossing indices (exact, integer)
        if live:
            rmax = min([N] + [bank.budgets[h] for h in live])
            assert L.rmax == rmax
            cross_all = [inter["cross"][h, :occ0[h]] for h in range(wl.H)]
            rs, rh = _rstar_from_cross(cross_all, occ0, bank.budgets, rmax, sync_heads)
            for h in live:
                assert hs[h].admitted == (rs if sync_heads else rh[h]), (t, h)
            if sync_heads:
                assert L.r_star == rs
        for h in range(wl.H):
            m, M = occ0[h], bank.budgets[h]
            r = hs[h].admitted
            if m == 0:
                assert r == min(N, M)
                assert sorted(after["src"][h, :r].tolist()) == list(range(r))
                continue
            Kb = desc(snap["K"][h, :m], snap["V"][h, :m])
            rho0, b0 = snap["rho"][h, :m].astype(np.float64), snap["base"][h, :m].astype(np.float64)
            s_gpu = inter["score"][h, :N]
            pi = inter["perm"][h, :N]
            # pi: permutation sorted by the GPU's own scores, ties in source order
            assert np.array_equal(np.sort(pi), np.arange(N))
            sp = s_gpu[pi]
            assert np.all((sp[1:] > sp[:-1]) | ((sp[1:] == sp[:-1]) & (pi[1:] > pi[:-1])))
            # Eq. 6 on sampled candidates
            xs = rng.choice(N, size=min(cands, N), replace=False)
            s_ref = (_w(prm, d, desc(Kc[h][xs], Vc[h][xs]), Kb) / b0[None, :]).sum(1) / m
            assert np.max(np.abs(s_gpu[xs] - s_ref) / s_ref) < TOL_DENS, (t, h)
            # crossing and rho~(r) of sampled rows under the GPU's pi
            Kpi = desc(Kc[h][pi], Vc[h][pi])
            rowsel = rng.choice(m, size=min(rows, m), replace=False)
            rmax = L.rmax
            Wr = _w(prm, d, Kb[rowsel], Kpi[:rmax])                       # [rows, rmax]
            run = rho0[rowsel][:, None] + np.concatenate([np.zeros((len(rowsel), 1)), np.cumsum(Wr, 1)], 1)
            g = run / b0[rowsel][:, None]
            for k, i in enumerate(rowsel):
                hit = np.nonzero(g[k] >= prm.tau)[0]
                c_ref = int(hit[0]) if len(hit) else INT_MAX
                c_gpu = int(inter["cross"][h, i])
                if c_gpu != c_ref:
                    near = [cc for cc in (c_gpu, c_ref) if cc != INT_MAX]
                    assert any(abs(g[k][cc] - prm.tau) <= TOL_DEC * prm.tau or
                               (cc > 0 and abs(g[k][cc - 1] - prm.tau) <= TOL_DEC * prm.tau) for cc in near), \
                        (t, h, i, c_gpu, c_ref)
            rt_gpu = inter["rho_tilde"][h, :m]
            rt_ref = run[:, r]
            assert np.max(np.abs(rt_gpu[rowsel] - rt_ref) / rt_ref) < TOL_DENS, (t, h)
            # eviction set (Step 3) from the GPU's own cross and rho~
            e = max(0, m + r - M)
            assert hs[h].evicted == e
            before_keys = {(int(a), int(c)): i for i, (a, c) in enumerate(zip(snap["step"][h, :m], snap["src"][h, :m]))}
            mnew = after["occ"][h]
            assert mnew == m - e + r and mnew <= M
            after_keys = {(int(a), int(c)): i for i, (a, c) in enumerate(zip(after["step"][h, :mnew], after["src"][h, :mnew]))}
            evicted = [i for k_, i in before_keys.items() if k_ not in after_keys]
            assert len(evicted) == e
            cr = inter["cross"][h, :m]
            mand = (cr <= r) if r > 0 else np.zeros(m, bool)
            ev = np.zeros(m, bool)
            ev[evicted] = True
            assert np.all(ev[mand])
            fill = ev & ~mand
            rest = ~ev & ~mand
            if fill.any() and rest.any():
                assert rt_gpu[fill].min() >= rt_gpu[rest].max()
            # commit: survivors unchanged, admitted = pi[:r], keys/values bit-exact
            new = [k_ for k_ in after_keys if k_ not in before_keys]
            assert sorted(k_[1] for k_ in new) == sorted(pi[:r].tolist()) and all(k_[0] == b for k_ in new)
            for k_, i in list(after_keys.items())[:2000]:
                if k_ in before_keys:
                    j = before_keys[k_]
                    assert np.array_equal(after["K"][h, i], snap["K"][h, j]) and \
                        np.array_equal(after["V"][h, i], snap["V"][h, j])
                    assert after["base"][h, i] == snap["base"][h, j]
                else:
                    assert np.array_equal(after["K"][h, i], Kc[h][k_[1]]) and \
                        np.array_equal(after["V"][h, i], Vc[h][k_[1]])
            # cached densities vs Phi over the final bank (sampled)
            Kf = desc(after["K"][h, :mnew], after["V"][h, :mnew])
            sel = rng.choice(mnew, size=min(rows, mnew), replace=False)
            phi = _w(prm, d, Kf[sel], Kf).sum(1) - prm.eps ** (-prm.p)     # Eq. 3: self excluded by index
            rho_f = after["rho"][h, sel]
            assert np.max(np.abs(rho_f - phi) / phi) < TOL_DENS, (t, h)
            isnew = np.array([(int(after["step"][h, i]), int(after["src"][h, i])) not in before_keys for i in sel])
            assert np.all(after["base"][h, sel][isnew] == np.maximum(rho_f[isnew], np.float32(prm.delta)))
            evicted_total += e
    occ_final = bank.occupancy_host()
    bank.close()
    return evicted_total, occ_final


def test_fullsize_wan13b_layer_kv_descriptor(dkv):
    """The [K; V] descriptor at the bench size (12 heads, N = 4,680, M = 9,360), tensor
    mode, the first four steps (fill, saturation, eviction)."""
    wl = synth.get_workload("wan13b_layer_h12")
    evicted, _ = _run(dkv, wl, steps=4, kv=True)
    assert evicted > 0


def test_fullsize_wan13b_layer(dkv):
    """12 heads, N = 4,680, M = 9,360, window = previous block: the bench workload."""
    wl = synth.get_workload("wan13b_layer_h12")
    evicted, _ = _run(dkv, wl, steps=5)
    assert evicted > 0


def test_fullsize_large_bank(dkv):
    """One layer of the 32,760-token-bank stress workload (drifting centres); three heads.
    On this data the growth bound stops admission near 11k states, below the budget, so
    r* = 0 from then on (Sec. 3.4: the bank may remain below M); every step is checked."""
    wl = synth.get_workload("largebank_l30h12_m32760", H=3)
    _, occ = _run(dkv, wl, steps=8, rows=24, cands=24)
    assert min(occ) > 2 * wl.N


def test_fullsize_sink5_context(dkv):
    """The paper's visible context: first-frame sink + 5-frame window (9,360 window tokens)
    next to the bank; the block offered at step t is the one that left the window."""
    wl = synth.get_workload("wan13b_layer_h12_sink5")
    evicted, _ = _run(dkv, wl, steps=6)
    assert evicted > 0


@pytest.mark.parametrize("sync", [1, 0])
def test_fullsize_headwise_budgets(dkv, sync):
    """Wan-14B-shaped layer: 40 heads with budgets drawn from {2340, 4680, 9360, 18720}."""
    wl = synth.get_workload("wan14b_headwise_l40h40", L=1)
    _run(dkv, wl, steps=4, sync_heads=sync, rows=12, cands=12)


def test_fullsize_headwise_wide_score_pass(dkv):
    """80 Wan-14B-shaped heads (budgets drawn from {2340, 4680, 9360, 18720}, N = 4,680):
    2,960 candidate row tiles, so the score pass takes the persistent 256-column form
    that the config-4 model step runs."""
    wl = synth.get_workload("wan14b_headwise_l40h40", L=1, H=80)
    assert wl.H * ((wl.N + 127) // 128) >= 16 * 152
    _run(dkv, wl, steps=3, rows=8, cands=8)
