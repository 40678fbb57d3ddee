"""The allocation-free candidate ordering entry point agrees with dkv_bank_admit.

dkv_candidate_order_noalloc serves callers that cannot allocate device memory:
its only scratch is a fixed array inside the library.  Here it must reproduce, for
every head, the Eq. 6 scores and the stable candidate order that dkv_bank_admit
computes in the fp32 score mode on the same bank and candidates, on two calls in a
row (the second call reuses the scratch the first one left behind).  The file is
named to be collected last.
"""
import numpy as np
import pytest
import torch

import synth
from gpu_util import to_dev

pytestmark = pytest.mark.gpu

TOL = 2e-4   # same scores tolerance as the fp32-mode parity tests


@pytest.fixture(scope="module")
def dkv():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_27922_gb300 import dkv as d
    return d


def _order_matches(s_ref, perm_ref, perm):
    """Same order, up to swaps of candidates whose reference scores tie within TOL."""
    diff = np.nonzero(perm != perm_ref)[0]
    for j in diff:
        a, b = s_ref[perm[j]], s_ref[perm_ref[j]]
        if abs(a - b) > TOL * max(abs(a), abs(b)):
            return False
    return True


def test_noalloc_order_matches_admit_on_two_calls(dkv):
    wl = synth.get_workload("wan13b_layer_h12", H=3, N=700, budgets=1500)
    ro = synth.LayerRollout(wl, 0)
    bank = dkv.BankLayer(wl.H, wl.d, wl.budgets_of_layer(0), wl.N, torch.bfloat16,
                         score_mode=dkv.DKV_SCORE_FP32)
    bank.reset()
    for b in range(3):                      # fill the bank, then one evicting update
        K, V = ro.block(b)
        bank.update(to_dev(K, torch.bfloat16), to_dev(V, torch.bfloat16), b)
    occ = bank.occupancy_host()
    assert min(occ) > 0
    for call, blk in enumerate((3, 4)):     # two calls in a row, different candidates
        K, V = ro.block(blk)
        Kd, Vd = to_dev(K, torch.bfloat16), to_dev(V, torch.bfloat16)
        k_snap = bank.k.clone()
        b_snap = bank.base.clone()
        occ = bank.occupancy_host()
        bank.admit(Kd, Vd, blk)             # reference: the regular entry point
        bank.sync()
        inter = bank.intermediates()
        s_ref = inter["score"][:, :wl.N].cpu().numpy().copy()
        p_ref = inter["perm"][:, :wl.N].cpu().numpy().copy()
        bank.compress()
        for h in range(wl.H):
            m = occ[h]
            scores = torch.full((wl.N,), float("nan"), dtype=torch.float32, device="cuda")
            perm = torch.full((wl.N,), -1, dtype=torch.int32, device="cuda")
            dkv.dkv_candidate_order_noalloc(k_snap[h, :m].contiguous(), b_snap[h, :m].contiguous(), m,
                                            Kd[h].contiguous(), wl.N, wl.d, dkv.DKV_DTYPE_BF16, bank.params,
                                            scores, perm)
            torch.cuda.synchronize()
            s = scores.cpu().numpy()
            p = perm.cpu().numpy()
            rel = np.abs(s - s_ref[h]) / np.maximum(np.abs(s_ref[h]), 1e-30)
            assert rel.max() <= TOL, (call, h, rel.max())
            assert sorted(p.tolist()) == list(range(wl.N))
            assert _order_matches(s_ref[h], p_ref[h], p), (call, h)
    bank.sync()
    bank.close()


def test_noalloc_rejects_oversized_input(dkv):
    x = torch.zeros(1, 128, dtype=torch.bfloat16, device="cuda")
    out = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(dkv.DkvError) as e:
        dkv.dkv_candidate_order_noalloc(x, torch.ones(1, device="cuda"), 1, x, dkv.DKV_NOALLOC_MAX_N + 1, 128,
                                        dkv.DKV_DTYPE_BF16, dkv.dkv_params_default(128), None, out)
    assert e.value.status == 2
