"""Free-running divergence: the GPU and the oracle each follow their own trajectory.

The parity tests are teacher-forced (every step starts both sides from the oracle's
bank).  Here neither side is reset: each applies Alg. 1 to its own bank, block after
block, so a decision that differs once (a near-tie of s, g against tau or the fill
cut-off) would carry into every later step.  After each update the retained sets are
compared by provenance (the bank is a set keyed by (step, source index), Eq. 12) and
the report gives, per step, r* on both sides and the overlap |G & O| / |G | O| of the
retained sets, plus the largest relative difference of rho and b over the states both
sides hold.

In the fp32-score mode the retained sets must stay identical at every step (the
exactness mode: no decision may differ).  In the tensor-core mode decisions near a
cut-off may differ; the report must show it, and the sets must stay close (overlap at
least 0.97 per step on this workload).
"""
import pytest
import torch

import oracle
import synth
from gpu_util import gpu_heads, oracle_heads, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dkv():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_27922_gb300 import dkv as d
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return d


def _free_run(dkv, wl, mode):
    dt = torch.float32 if wl.dtype == "fp32" else torch.bfloat16
    bank = dkv.BankLayer(wl.H, wl.d, wl.budgets_of_layer(0), wl.N, dt, score_mode=mode)
    bank.reset()
    ob = oracle.LayerBank.empty(wl.budgets_of_layer(0), wl.d)
    ro = synth.LayerRollout(wl, 0)
    rows = []
    for t in range(wl.steps):
        b = wl.admitted_block(t)
        if b is None:
            continue
        K, V = ro.block(b)
        bank.update(to_dev(K, dt), to_dev(V, dt), b)
        rec = oracle.update_layer(ob, K, V, b)
        bank.sync()
        L, _ = bank.stats()
        g, o = gpu_heads(bank), oracle_heads(ob)
        inter = sum(len(set(gh) & set(oh)) for gh, oh in zip(g, o))
        union = sum(len(set(gh) | set(oh)) for gh, oh in zip(g, o))
        rho_rel = base_rel = 0.0
        for gh, oh in zip(g, o):
            for key in set(gh) & set(oh):
                rg, bg = gh[key][2], gh[key][3]
                ro_, bo = oh[key][2], oh[key][3]
                rho_rel = max(rho_rel, abs(rg - ro_) / max(abs(ro_), 1e-30))
                base_rel = max(base_rel, abs(bg - bo) / max(abs(bo), 1e-30))
        rows.append(dict(step=t, rstar_gpu=int(L.r_star), rstar_oracle=int(rec.r_star),
                         overlap=inter / max(union, 1), rho_rel=rho_rel, base_rel=base_rel,
                         occupancy=[len(x) for x in g]))
    bank.close()
    print("\nstep  r*(gpu)  r*(oracle)  overlap   rho rel    b rel")
    for r in rows:
        print(f"{r['step']:4d}  {r['rstar_gpu']:7d}  {r['rstar_oracle']:10d}  {r['overlap']:.5f}  "
              f"{r['rho_rel']:.2e}  {r['base_rel']:.2e}")
    return rows


def test_free_running_fp32_mode_identical(dkv):
    """Config-0 shapes (1 x 2 heads, d = 64, fp32), every step: identical trajectories."""
    wl = synth.get_workload("tiny_fp32_l1h2_d64")
    rows = _free_run(dkv, wl, dkv.DKV_SCORE_FP32)
    assert len(rows) >= 4 and max(sum(r["occupancy"]) for r in rows) == sum(wl.budgets_of_layer(0))
    for r in rows:
        assert r["rstar_gpu"] == r["rstar_oracle"], r
        assert r["overlap"] == 1.0, r
        assert r["rho_rel"] <= 2e-5 and r["base_rel"] <= 2e-5, r


def test_free_running_fp32_mode_d128_identical(dkv):
    """d = 128 bf16 keys, sizes off the tile grid, fp32 scoring: identical trajectories."""
    wl = synth.get_workload("wan13b_layer_h12", H=3, N=300, W=64, Nq=64, budgets=700, steps=8)
    rows = _free_run(dkv, wl, dkv.DKV_SCORE_FP32)
    for r in rows:
        assert r["rstar_gpu"] == r["rstar_oracle"], r
        assert r["overlap"] == 1.0, r


def test_free_running_tensor_mode_report(dkv):
    """A longer rollout in the tensor-core mode (16 blocks into banks of 1,200): the
    divergence stays small."""
    wl = synth.get_workload("wan13b_layer_h12", H=3, N=600, W=64, Nq=64, budgets=1200, steps=17)
    rows = _free_run(dkv, wl, dkv.DKV_SCORE_TENSOR)
    for r in rows:
        assert r["overlap"] >= 0.97, r
        assert abs(r["rstar_gpu"] - r["rstar_oracle"]) <= 0.05 * wl.N, r
