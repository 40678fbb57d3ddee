"""Whole-update parity at full size against the oracle: one Wan-1.3B-shaped layer
(12 heads, d = 128, bf16, N = 4,680 candidates, budget M = 9,360, tensor-core mode,
the launch configuration bench.py times for this layer).

The oracle builds its bank itself from the seeded blocks (the empty-bank branch of
Alg. 1 with block 0); the GPU bank is loaded from the oracle's before every compared
update (teacher forcing), and both apply the same update.  Compared on every head of
block 1 (the bank grows to its budget) and blocks 2 and 3 (steady state: N admitted and
N evicted per head): r*, admitted / evicted / mandatory counts, the whole retained set
by provenance, the K/V bits of every state, every cached density and baseline, every
candidate's score, the order, every crossing index and rho~(r*).  About two minutes of
host time in the oracle.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import check_report, tols, update_and_compare

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dkv():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_27922_gb300 import dkv as d
    return d


def test_wan13b_layer_whole_update_teacher_forced(dkv):
    wl = synth.get_workload("wan13b_layer_h12")
    bank = dkv.BankLayer(wl.H, wl.d, wl.budgets_of_layer(0), wl.N, torch.bfloat16,
                         score_mode=dkv.DKV_SCORE_TENSOR)
    bank.reset()
    tol, dens = tols("tc")
    ro = synth.LayerRollout(wl, 0)
    ob = oracle.LayerBank.empty(wl.budgets_of_layer(0), wl.d)
    K, V = ro.block(0)
    oracle.update_layer(ob, K, V, 0)          # the oracle's own empty-bank initialisation
    steady = 0
    for b in (1, 2, 3):
        K, V = ro.block(b)
        rep, rec = update_and_compare(bank, ob, K, V, b, tol, dens)
        check_report(rep, "tc", b)
        assert rep.kv_bit_exact
        assert rep.rho_tilde_checked == wl.H   # every head's crossings and rho~(r*) compared
        evicted = sum(len(hr.evicted) for hr in rec.heads)
        assert all(hb.m <= hb.M for hb in ob.heads)
        steady += evicted > 0
        print(f"block {b}: r* {rec.r_star}, evicted {evicted}, set mismatches {rep.set_mismatch}, "
              f"perm mismatches {rep.perm_mismatch} (largest gap {rep.perm_gap_max:.1e}), "
              f"cross mismatches {rep.cross_mismatch}, "
              f"max rel: s {rep.score_max_rel:.2e} rho~ {rep.rho_tilde_max_rel:.2e} rho {rep.rho_max_rel:.2e} "
              f"b {rep.base_max_rel:.2e}")
    assert steady == 2, "blocks 2 and 3 must evict (steady state)"
    bank.close()
