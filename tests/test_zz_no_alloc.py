"""The allocation-free candidate ordering entry point, checked against the oracle.

dkv_candidate_order_noalloc serves callers that cannot allocate device memory (a
framework whose pool owns every device byte, hosts that forbid allocation after
start-up, plugins handed only fixed buffers): its only scratch is a fixed array
inside the library.  Here, on banks written from the oracle's own rollout, it must
give every head the Eq. 6 scores and the stable ascending candidate order of the
oracle (within the fp32 bound, near-ties only), and exactly what dkv_bank_admit
computes in the fp32 score mode, whose arithmetic it shares; on two calls in a row
(the second call finds the first call's scores in the scratch), on an empty bank,
with fp32 keys at d = 64, and at the largest accepted candidate count.  The file is
named to be collected last.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import load_state, oracle_params, to_dev

pytestmark = pytest.mark.gpu

# fp32 scores against the float64 oracle: relative bound of the fp32 score mode
TOL = 2e-4


@pytest.fixture(scope="module")
def dkv():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_27922_gb300 import dkv as d
    return d


def _dt(wl):
    return torch.float32 if wl.dtype == "fp32" else torch.bfloat16


def _oracle_bank(wl, blocks):
    """The oracle's bank after updates with the given blocks (teacher state)."""
    ro = synth.LayerRollout(wl, 0)
    ob = oracle.LayerBank.empty(wl.budgets_of_layer(0), wl.d)
    for b in blocks:
        K, V = ro.block(b)
        oracle.update_layer(ob, K, V, b)
    return ob, ro


def _check_against_oracle(s, p, s_ref, pi_ref, what):
    rel = np.abs(s - s_ref) / np.maximum(np.abs(s_ref), 1e-30)
    assert rel.max() <= TOL, (what, float(rel.max()))
    assert sorted(p.tolist()) == list(range(len(p))), what
    for j in np.nonzero(p != pi_ref)[0]:    # an inversion only between oracle near-ties
        a, b = s_ref[p[j]], s_ref[pi_ref[j]]
        assert abs(a - b) <= TOL * max(abs(a), abs(b)), (what, int(j), a, b)


def _noalloc(dkv, bank, h, m, Kd, N, dtype):
    scores = torch.full((N,), float("nan"), dtype=torch.float32, device="cuda")
    perm = torch.full((N,), -1, dtype=torch.int32, device="cuda")
    kb = bank.k[h, :max(m, 1)].contiguous()
    bb = bank.base[h, :max(m, 1)].contiguous()
    dkv.dkv_candidate_order_noalloc(kb, bb, m, Kd[h].contiguous(), N, bank.d, dtype, bank.params, scores, perm)
    torch.cuda.synchronize()
    return scores.cpu().numpy(), perm.cpu().numpy()


def _compare_case(dkv, wl, fill_blocks, cand_blocks):
    """Teacher bank from the oracle; per candidate block and head: no-alloc vs the oracle's
    Eq. 6 scores and order, and vs dkv_bank_admit (fp32 score mode) bit for bit."""
    dt = _dt(wl)
    code = dkv.DKV_DTYPE_FP32 if dt == torch.float32 else dkv.DKV_DTYPE_BF16
    bank = dkv.BankLayer(wl.H, wl.d, wl.budgets_of_layer(0), wl.N, dt, score_mode=dkv.DKV_SCORE_FP32)
    ob, ro = _oracle_bank(wl, fill_blocks)
    prm = oracle_params(bank)
    for call, blk in enumerate(cand_blocks):     # calls in a row, different candidates
        K, V = ro.block(blk)
        rec = oracle.update_layer(ob.copy(), K, V, blk, prm)
        load_state(bank, ob)
        Kd, Vd = to_dev(K, dt), to_dev(V, dt)
        got = [_noalloc(dkv, bank, h, hb.m, Kd, wl.N, code) for h, hb in enumerate(ob.heads)]
        bank.admit(Kd, Vd, blk)                  # the regular entry point on the same bank
        bank.sync()
        inter = bank.intermediates()
        s_adm = inter["score"][:, :wl.N].cpu().numpy()
        p_adm = inter["perm"][:, :wl.N].cpu().numpy()
        bank.compress()
        bank.sync()
        for h, (s, p) in enumerate(got):
            hr = rec.heads[h]
            assert ob.heads[h].m > 0 and not hr.empty_init
            _check_against_oracle(s, p, hr.s, hr.pi, (call, h))
            assert np.array_equal(s.view(np.uint32), s_adm[h].view(np.uint32)), (call, h)
            assert np.array_equal(p, p_adm[h]), (call, h)
    bank.close()


def test_noalloc_matches_oracle_and_admit_on_two_calls(dkv):
    wl = synth.get_workload("wan13b_layer_h12", H=3, N=700, budgets=1500)
    _compare_case(dkv, wl, fill_blocks=(0, 1, 2), cand_blocks=(3, 4))


def test_noalloc_fp32_keys_d64(dkv):
    wl = synth.get_workload("tiny_fp32_l1h2_d64")
    _compare_case(dkv, wl, fill_blocks=(0, 1, 2), cand_blocks=(3, 4))


def test_noalloc_largest_candidate_count(dkv):
    """N = DKV_NOALLOC_MAX_N: the ordering kernel's shared memory needs the opt-in the
    first call on the device makes."""
    N = dkv.DKV_NOALLOC_MAX_N
    wl = synth.get_workload("wan13b_layer_h12", H=1, N=N, budgets=1200)
    ro = synth.LayerRollout(wl, 0)
    ob = oracle.LayerBank.empty(wl.budgets_of_layer(0), wl.d)
    K0, V0 = ro.block(0)
    oracle.update_layer(ob, K0[:, :1200], V0[:, :1200], 0)       # a full bank of 1,200 states
    bank = dkv.BankLayer(1, wl.d, (1200,), N, torch.bfloat16, score_mode=dkv.DKV_SCORE_FP32)
    load_state(bank, ob)
    K, _ = ro.block(1)
    rec = oracle.update_layer(ob.copy(), K, K, 1, oracle_params(bank))
    for _ in range(2):
        s, p = _noalloc(dkv, bank, 0, ob.heads[0].m, to_dev(K, torch.bfloat16), N, dkv.DKV_DTYPE_BF16)
        _check_against_oracle(s, p, rec.heads[0].s, rec.heads[0].pi, "max N")
    bank.close()


def test_noalloc_empty_bank_gives_source_order(dkv):
    """m = 0 (Alg. 1's empty-bank branch): source order and zero scores, also right after
    a call that left nonzero scores in the scratch."""
    wl = synth.get_workload("wan13b_layer_h12", H=1, N=300, budgets=600)
    ob, ro = _oracle_bank(wl, (0,))
    bank = dkv.BankLayer(1, wl.d, (600,), wl.N, torch.bfloat16, score_mode=dkv.DKV_SCORE_FP32)
    load_state(bank, ob)
    Kd = to_dev(ro.block(1)[0], torch.bfloat16)
    s, _ = _noalloc(dkv, bank, 0, ob.heads[0].m, Kd, wl.N, dkv.DKV_DTYPE_BF16)
    assert np.all(s > 0)
    s, p = _noalloc(dkv, bank, 0, 0, Kd, wl.N, dkv.DKV_DTYPE_BF16)
    assert np.array_equal(p, np.arange(wl.N)) and np.all(s == 0)
    bank.close()


def test_noalloc_rejects_oversized_input(dkv):
    x = torch.zeros(1, 128, dtype=torch.bfloat16, device="cuda")
    out = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(dkv.DkvError) as e:
        dkv.dkv_candidate_order_noalloc(x, torch.ones(1, device="cuda"), 1, x, dkv.DKV_NOALLOC_MAX_N + 1, 128,
                                        dkv.DKV_DTYPE_BF16, dkv.dkv_params_default(128), None, out)
    assert e.value.status == 2
