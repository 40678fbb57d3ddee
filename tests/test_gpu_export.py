"""Checkpoint read (dkv_bank_export) and resume (dkv_bank_import) through the C ABI.

The bank that Alg. 1 carries from one update to the next is (K, V, rho, b, provenance,
occupancy) per head (Sec. 3.4, App. C).  A free-running GPU rollout is exported to host
and to device memory; the export must equal the handle's buffers bit for bit.  A second
handle resumed from the export and the original handle then take the same next update:
their banks must agree bit for bit, and the resumed one must match the oracle started
from the same checkpoint (the update parity bar of the rollout tests).
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import check_report, to_dev, tols, update_and_compare

pytestmark = pytest.mark.gpu

FIELDS = ("k", "v", "rho", "base", "prov_step", "prov_src")


@pytest.fixture(scope="module")
def dkv():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_27922_gb300 import dkv as d
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return d


def _bank(dkv, wl, mode):
    b = dkv.BankLayer(wl.H, wl.d, wl.budgets_of_layer(0), wl.N, torch.bfloat16, score_mode=mode)
    b.reset()
    return b


def _rows(x, occ):
    """Meaningful rows of every head: [(head, rows 0..occ_h)]."""
    return [x[h, :occ[h]] for h in range(len(occ))]


def _same(a, b, occ):
    return all(torch.equal(x.cpu(), y.cpu()) for x, y in zip(_rows(a, occ), _rows(b, occ)))


def _oracle_from(ck, budgets, d):
    ob = oracle.LayerBank.empty(budgets, d)
    occ = ck["occupancy"].tolist()
    for h, hb in enumerate(ob.heads):
        m = occ[h]
        hb.K = ck["k"][h, :m].float().numpy().astype(np.float64)
        hb.V = ck["v"][h, :m].float().numpy().astype(np.float64)
        hb.rho = ck["rho"][h, :m].numpy().astype(np.float32)
        hb.base = ck["base"][h, :m].numpy().astype(np.float32)
        hb.step = ck["prov_step"][h, :m].numpy().astype(np.int64)
        hb.src = ck["prov_src"][h, :m].numpy().astype(np.int64)
    return ob


@pytest.mark.parametrize("mode_name", ["tc", "fp32"])
def test_export_resume_matches_original_and_oracle(dkv, mode_name):
    mode = {"fp32": dkv.DKV_SCORE_FP32, "tc": dkv.DKV_SCORE_TENSOR}[mode_name]
    wl = synth.get_workload("wan13b_layer_h12", H=3, N=300, W=64, Nq=64, budgets=700, steps=6)
    ro = synth.LayerRollout(wl, 0)
    a = _bank(dkv, wl, mode)
    dev = torch.device("cuda")
    for t in range(4):   # free running: blocks 0..3, eviction from the third on
        K, V = ro.block(t)
        a.update(to_dev(K, torch.bfloat16), to_dev(V, torch.bfloat16), t)
    a.sync()
    occ = a.occupancy_host()
    assert min(occ) > 0 and max(occ) <= 700
    ck = a.export_state("cpu")
    ck_dev = a.export_state(dev)
    assert ck["occupancy"].tolist() == occ and ck_dev["occupancy"].cpu().tolist() == occ
    for f in FIELDS:
        assert _same(ck[f], getattr(a, f), occ), f
        assert _same(ck_dev[f], getattr(a, f), occ), f

    # resume: a fresh handle's buffers take the checkpoint, import recomputes the norms
    b = _bank(dkv, wl, mode)
    for f in FIELDS:
        getattr(b, f).copy_(ck[f])
    b.import_state(occ)
    a.import_state(occ)   # the control recomputes its norms the same way
    assert _same(a.knorm, b.knorm, occ)
    K, V = ro.block(4)
    a.update(to_dev(K, torch.bfloat16), to_dev(V, torch.bfloat16), 4)
    b.update(to_dev(K, torch.bfloat16), to_dev(V, torch.bfloat16), 4)
    a.sync()
    b.sync()
    occ_a, occ_b = a.occupancy_host(), b.occupancy_host()
    assert occ_a == occ_b
    for f in FIELDS + ("knorm",):
        assert _same(getattr(a, f), getattr(b, f), occ_a), f

    # the same checkpoint through the oracle: the resumed handle meets the parity bar
    ob = _oracle_from(ck, wl.budgets_of_layer(0), wl.d)
    c = _bank(dkv, wl, mode)
    tol, dens = tols(mode_name)
    rep, _ = update_and_compare(c, ob, K, V, 4, tol, dens)
    check_report(rep, mode_name, "resumed step")
    if mode_name == "fp32":   # identical decisions: the same occupancy as the resumed handle
        assert [hb.m for hb in ob.heads] == occ_b
    for x in (a, b, c):
        x.close()


def test_export_refused_between_admit_and_compress(dkv):
    wl = synth.get_workload("wan13b_layer_h12", H=2, N=160, W=64, Nq=64, budgets=300, steps=3)
    ro = synth.LayerRollout(wl, 0)
    a = _bank(dkv, wl, dkv.DKV_SCORE_TENSOR)
    K, V = ro.block(0)
    a.admit(to_dev(K, torch.bfloat16), to_dev(V, torch.bfloat16), 0)
    with pytest.raises(dkv.DkvError) as e:
        a.export_state("cpu")
    assert e.value.status == 3   # DKV_ERR_STATE
    a.compress()
    a.sync()
    ck = a.export_state("cpu")
    assert ck["occupancy"].tolist() == a.occupancy_host()
    a.close()
