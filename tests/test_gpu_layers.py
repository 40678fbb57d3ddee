"""Several layers in one handle (params.layer_heads): every call updates or reads all
layers with single launches, each layer keeping its own shared prefix r* (Eq. 11).

The grouped handle is compared bit for bit with one handle per layer fed the same
per-layer streams (those are themselves parity-tested against the oracle): bank
contents, occupancy, provenance, densities, baselines and each layer's r* must be
identical, and so must attention outputs whenever both handles take the same attention
schedule (the grids of the small cases); the grouped handle is also teacher-forced
against the oracle layer by layer.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import check_report, to_dev, tols, update_and_compare_layers

pytestmark = pytest.mark.gpu

BUFFERS = ("k", "v", "rho", "base", "knorm", "prov_step", "prov_src", "occupancy")


@pytest.fixture(scope="module")
def dkv():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_27922_gb300 import dkv as d
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return d


def _cat_heads(parts, dtype):
    return torch.cat([to_dev(p, dtype) for p in parts], dim=0).contiguous()


@pytest.mark.parametrize("mode,sync,desc", [("tc", 1, 0), ("tc", 0, 0), ("fp32", 1, 0), ("fp32", 0, 0),
                                             ("tc", 1, 1), ("fp32", 1, 1)])
def test_grouped_layers_match_one_handle_per_layer(dkv, mode, sync, desc):
    """desc = 1: the [K; V] descriptor (App. E)."""
    L, H = 3, 2
    # per-layer budgets differ, so the layers fill, saturate and freeze at different steps
    budgets = [300, 300, 190, 250, 420, 420]
    wl = synth.get_workload("wan13b_layer_h12", L=L, H=H, N=96, W=96, Nq=64, budgets=budgets, steps=9)
    sm = dkv.DKV_SCORE_TENSOR if mode == "tc" else dkv.DKV_SCORE_FP32
    dt = torch.bfloat16
    kw = dict(score_mode=sm, sync_heads=sync, descriptor=desc)
    sep = [dkv.BankLayer(H, wl.d, wl.budgets_of_layer(l), wl.N, dt, **kw) for l in range(L)]
    grp = dkv.BankLayer(L * H, wl.d, list(wl.budgets), wl.N, dt, layer_heads=H, **kw)
    assert grp.n_layers == L
    for b in sep + [grp]:
        b.reset()
    ro = [synth.LayerRollout(wl, l) for l in range(L)]
    rstars = []
    for t in range(wl.steps):
        qs = [ro[l].queries(t) for l in range(L)]
        wins = [ro[l].window(t) for l in range(L)]
        o_sep = [sep[l].attend(to_dev(qs[l], dt), to_dev(wins[l][0], dt), to_dev(wins[l][1], dt)) for l in range(L)]
        o_grp = grp.attend(_cat_heads(qs, dt), _cat_heads([w[0] for w in wins], dt),
                           _cat_heads([w[1] for w in wins], dt))
        b = wl.admitted_block(t)
        if b is not None:
            blocks = [ro[l].block(b) for l in range(L)]
            for l in range(L):
                sep[l].admit(to_dev(blocks[l][0], dt), to_dev(blocks[l][1], dt), b)
                sep[l].compress()
            grp.admit(_cat_heads([x[0] for x in blocks], dt), _cat_heads([x[1] for x in blocks], dt), b)
            grp.compress()
        torch.cuda.synchronize()
        for bk in sep + [grp]:
            bk.sync()
        assert torch.equal(torch.cat(o_sep, 0), o_grp), t
        for name in BUFFERS:
            g = getattr(grp, name)
            for l in range(L):
                want = getattr(sep[l], name)   # [H] or [H][M_l(, d)]; the grouped rows are longer
                got = g[l * H:(l + 1) * H]
                if want.dim() > 1:
                    got = got[:, :want.shape[1]]
                assert torch.equal(want, got), (t, name, l)
        if b is not None:
            ls = grp.layer_stats()
            assert [x.r_star for x in ls] == [sep[l].stats()[0].r_star for l in range(L)], t
            assert [x.rmax for x in ls] == [sep[l].stats()[0].rmax for l in range(L)], t
            rstars.append(tuple(x.r_star for x in ls))
    # the layers really did take different prefixes at some step
    assert any(len(set(r)) > 1 for r in rstars), rstars
    for bk in sep + [grp]:
        bk.close()


@pytest.mark.parametrize("mode,sync", [("tc", 1), ("tc", 0), ("fp32", 1), ("fp32", 0)])
def test_grouped_layers_match_oracle(dkv, mode, sync):
    """A three-layer handle (ragged sizes, per-layer budgets) teacher-forced against
    oracle.update_layer run on every layer by itself: each layer's r* (Eq. 11 per layer),
    scores, order, crossings, retained set, K/V bits and densities at the mode's bar."""
    L, H = 3, 3
    budgets = [700, 700, 700, 420, 520, 600, 900, 900, 650]
    wl = synth.get_workload("wan13b_layer_h12", L=L, H=H, N=300, W=64, Nq=64, budgets=budgets, steps=7)
    sm = dkv.DKV_SCORE_TENSOR if mode == "tc" else dkv.DKV_SCORE_FP32
    grp = dkv.BankLayer(L * H, wl.d, list(wl.budgets), wl.N, torch.bfloat16, layer_heads=H, score_mode=sm,
                        sync_heads=sync)
    grp.reset()
    tol, dens = tols(mode)
    ro = [synth.LayerRollout(wl, l) for l in range(L)]
    obs = [oracle.LayerBank.empty(wl.budgets_of_layer(l), wl.d) for l in range(L)]
    rstars, evicted = [], 0
    for t in range(wl.steps):
        b = wl.admitted_block(t)
        if b is None:
            continue
        blocks = [ro[l].block(b) for l in range(L)]
        reps, recs = update_and_compare_layers(grp, obs, [x[0] for x in blocks], [x[1] for x in blocks], b,
                                               tol, dens)
        for l, rep in enumerate(reps):
            check_report(rep, mode, (t, l))
        rstars.append(tuple(r.rstar_oracle for r in reps))
        evicted += sum(len(hr.evicted) for rec in recs for hr in rec.heads)
    assert evicted > 0
    assert any(len(set(r)) > 1 for r in rstars), rstars   # the layers took different prefixes
    grp.close()


def test_grouped_layers_rope(dkv):
    """Temporal re-zeroing (dkv_bank_admit_rope) in a three-layer handle: one coordinate
    array for all layers' heads, bit-identical to one handle per layer."""
    L, H = 3, 2
    wl = synth.get_workload("wan13b_layer_h12", L=L, H=H, N=96, W=96, Nq=64, budgets=[300, 190, 420] * 2, steps=6)
    dt = torch.bfloat16
    sep = [dkv.BankLayer(H, wl.d, wl.budgets_of_layer(l), wl.N, dt) for l in range(L)]
    grp = dkv.BankLayer(L * H, wl.d, list(wl.budgets), wl.N, dt, layer_heads=H)
    for b in sep + [grp]:
        b.reset()
    theta = torch.from_numpy(synth.temporal_rope_theta(wl.d)).cuda()
    ro = [synth.LayerRollout(wl, l) for l in range(L)]
    for t in range(wl.steps):
        b = wl.admitted_block(t)
        if b is None:
            continue
        tc = torch.from_numpy(wl.frame_coords(b) + 500).cuda()
        blocks = [ro[l].block(b) for l in range(L)]
        for l in range(L):
            sep[l].update(to_dev(blocks[l][0], dt), to_dev(blocks[l][1], dt), b, t_coord=tc, theta=theta)
        grp.update(_cat_heads([x[0] for x in blocks], dt), _cat_heads([x[1] for x in blocks], dt), b,
                   t_coord=tc, theta=theta)
        torch.cuda.synchronize()
        for bk in sep + [grp]:
            bk.sync()
        for name in BUFFERS:
            g = getattr(grp, name)
            for l in range(L):
                want = getattr(sep[l], name)
                got = g[l * H:(l + 1) * H]
                if want.dim() > 1:
                    got = got[:, :want.shape[1]]
                assert torch.equal(want, got), (t, name, l)
    for bk in sep + [grp]:
        bk.close()


def test_layer_heads_must_divide_heads(dkv):
    wl = synth.get_workload("wan13b_layer_h12", H=6, N=16, budgets=32)
    for bad in (4, 7, -1):
        with pytest.raises(dkv.DkvError) as e:
            dkv.BankLayer(6, wl.d, wl.budgets_of_layer(0), 16, torch.bfloat16, layer_heads=bad)
        assert e.value.status == 1


def test_grouped_layers_fullsize(dkv):
    """Three Wan-1.3B-shaped layers (12 heads, N = 4,680, M = 9,360) in one handle against
    three one-layer handles over the first five steps (fill and eviction): bank contents
    bit for bit, attention within its bound."""
    L = 3
    wl = synth.get_workload("wan13b_stack_l30h12", L=L)
    H, dt = wl.H, torch.bfloat16
    sep = [dkv.BankLayer(H, wl.d, wl.budgets_of_layer(l), wl.N, dt) for l in range(L)]
    grp = dkv.BankLayer(L * H, wl.d, list(wl.budgets), wl.N, dt, layer_heads=H)
    for b in sep + [grp]:
        b.reset()
    ro = [synth.LayerRollout(wl, l) for l in range(L)]
    evicted = 0
    for t in range(5):
        wins = [ro[l].window(t) for l in range(L)]
        qs = [ro[l].queries(t) for l in range(L)]
        o_sep = [sep[l].attend(to_dev(qs[l], dt), to_dev(wins[l][0], dt), to_dev(wins[l][1], dt)) for l in range(L)]
        o_grp = grp.attend(_cat_heads(qs, dt), _cat_heads([w[0] for w in wins], dt), _cat_heads([w[1] for w in wins], dt))
        b = wl.admitted_block(t)
        if b is not None:
            blocks = [ro[l].block(b) for l in range(L)]
            for l in range(L):
                sep[l].update(to_dev(blocks[l][0], dt), to_dev(blocks[l][1], dt), b)
            grp.update(_cat_heads([x[0] for x in blocks], dt), _cat_heads([x[1] for x in blocks], dt), b)
        torch.cuda.synchronize()
        for bk in sep + [grp]:
            bk.sync()
        # 36 heads take the two-query-tile attention schedule, 12 the key-split one: the
        # outputs agree within the attention bound (each schedule is checked against the
        # oracle elsewhere); the banks stay bit-identical
        assert (torch.cat(o_sep, 0).float() - o_grp.float()).abs().max().item() < 2e-2, t
        for name in BUFFERS:
            assert torch.equal(torch.cat([getattr(sep[l], name) for l in range(L)], 0), getattr(grp, name)), (t, name)
        if b is not None:
            assert [x.r_star for x in grp.layer_stats()] == [sep[l].stats()[0].r_star for l in range(L)], t
            evicted += sum(h.evicted for h in grp.stats()[1])
    assert evicted > 0
    for bk in sep + [grp]:
        bk.close()
