"""Temporal rotary re-zeroing of offered keys (App. A) through the C ABI, against the oracle.

The backbones attend to memory keys whose temporal RoPE coordinate is 0, and the bank
stores those keys.  dkv_bank_admit_rope takes keys that still carry their frame's
temporal rotation and rotates them back before the update.  The stored keys must be
bit-identical to ``oracle.rope_rezero`` (the nearest bf16 / fp32 value of the exact
rotation), and a teacher-forced rollout on rotated keys must pass the same parity bar
as the plain admit.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import check_report, to_dev, tols, update_and_compare
from oracle_pins import _rope_forward

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dkv():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_27922_gb300 import dkv as d
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return d


LAYOUTS = {"interleaved": 0, "half": 1}


def _rotated(K, t, theta, layout, dtype):
    """Keys as a backbone's window holds them: rotated to their frame's coordinate and
    stored in the key type (inputs only; any rounding will do)."""
    Kt = _rope_forward(K, t, theta, layout).astype(np.float32)
    return synth.round_to_bf16(Kt) if dtype == torch.bfloat16 else Kt


def _admit_empty(dkv, K, V, t, theta, layout, dtype, score_mode=None):
    H, N, d = K.shape
    kw = {} if score_mode is None else dict(score_mode=score_mode)
    bank = dkv.BankLayer(H, d, [max(N, 16)] * H, N, dtype, **kw)
    bank.reset()
    bank.admit(to_dev(K, dtype), to_dev(V, dtype), 3,
               t_coord=torch.from_numpy(np.asarray(t, np.int32)).cuda(),
               theta=torch.from_numpy(np.asarray(theta, np.float32)).cuda(), rope_layout=LAYOUTS[layout])
    bank.compress()
    bank.sync()
    return bank


def _stored_in_source_order(bank, N):
    """Bank keys and values of the empty-bank initialisation, indexed by source position."""
    occ = bank.occupancy.cpu().numpy()
    src = bank.prov_src.cpu().numpy()
    k = bank.k.float().cpu().numpy()
    v = bank.v.float().cpu().numpy()
    H = k.shape[0]
    Ks = np.zeros((H, N, k.shape[2]), np.float64)
    Vs = np.zeros_like(Ks)
    for h in range(H):
        assert occ[h] == N
        assert sorted(src[h, :N].tolist()) == list(range(N))
        Ks[h, src[h, :N]] = k[h, :N]
        Vs[h, src[h, :N]] = v[h, :N]
    return Ks, Vs


@pytest.mark.parametrize("layout", sorted(LAYOUTS))
def test_rezeroed_keys_bit_exact_fullsize(dkv, layout):
    """12 heads x 4,680 keys, d = 128, bf16, frames 1,200-1,202 (angles up to 1,202 rad),
    into an empty bank: every stored key bit-identical to the oracle's."""
    wl = synth.get_workload("wan13b_layer_h12")
    ro = synth.LayerRollout(wl, 0)
    K, V = ro.block(0)
    t = wl.frame_coords(400)
    theta = synth.temporal_rope_theta(wl.d, layout_first=(layout == "interleaved"))
    Kt = _rotated(K, t, theta, layout, torch.bfloat16)
    bank = _admit_empty(dkv, Kt, V, t, theta, layout, torch.bfloat16)
    Ks, Vs = _stored_in_source_order(bank, wl.N)
    want = oracle.rope_rezero(Kt, t, theta, layout, "bf16")
    bad = np.argwhere(Ks != want)
    assert len(bad) == 0, (len(bad), bad[:5])
    assert np.array_equal(Vs, V.astype(np.float64))          # values are not rotated
    assert not np.array_equal(Ks, Kt.astype(np.float64))     # something did rotate
    # stored norms are those of the stored keys
    kn = bank.knorm.cpu().numpy()[:, :wl.N]
    src = bank.prov_src.cpu().numpy()[:, :wl.N]
    ref = np.stack([(Ks[h][src[h]] ** 2).sum(-1) for h in range(wl.H)])
    assert np.allclose(kn, ref, rtol=2e-6, atol=0)
    bank.close()


@pytest.mark.parametrize("d", [128, 64])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("layout", sorted(LAYOUTS))
def test_rezeroed_keys_wide_angles(dkv, dtype, layout, d):
    """Random coordinates in [-70,000, 70,000] (negative too, many distinct ones per row
    strip), random frequencies up to 3 in most pairs: angles from 0 to 2e5 rad; both
    head dimensions (at d = 64 a lane holds one pair, or half a split pair)."""
    rng = np.random.default_rng(7)
    H, N = 3, 1000
    K = synth.round_to_bf16(rng.normal(size=(H, N, d)).astype(np.float32) * 4.0)
    V = synth.round_to_bf16(rng.normal(size=(H, N, d)).astype(np.float32))
    t = rng.integers(-70000, 70000, size=N).astype(np.int32)
    t[:50] = 0
    t[50:100] = rng.integers(-3, 4, size=50)
    theta = (rng.uniform(0, 3, size=d // 2) * (rng.uniform(size=d // 2) < 0.9)).astype(np.float32)
    theta[:4] = np.float32([1e-6, 1.0, 2.5e-3, 0.0])
    bank = _admit_empty(dkv, K, V, t, theta, layout, dtype,
                        score_mode=dkv.DKV_SCORE_FP32 if dtype == torch.float32 or d != 128 else None)
    Ks, _ = _stored_in_source_order(bank, N)
    want = oracle.rope_rezero(K, t, theta, layout, "bf16" if dtype == torch.bfloat16 else "fp32")
    bad = np.argwhere(Ks != want)
    assert len(bad) == 0, (len(bad), bad[:5])
    assert np.array_equal(Ks[:, :50], K[:, :50].astype(np.float64))   # coordinate 0 is the identity
    bank.close()


@pytest.mark.parametrize("mode,layout,desc", [("fp32", "interleaved", 0), ("fp32", "half", 0),
                                              ("tc", "interleaved", 0), ("tc", "half", 0), ("tc", "interleaved", 1)])
def test_rope_rollout_matches_oracle(dkv, mode, layout, desc):
    """Teacher-forced rollout (d = 128 bf16, N = 300, M = 700, 3 heads) whose blocks arrive
    rotated to their frames' coordinates: decisions, r*, retained sets, K/V bits and
    densities against the oracle updating with rope_rezero of the same keys (desc = 1:
    with the [K; V] descriptor, re-zeroed key then value)."""
    wl = synth.get_workload("wan13b_layer_h12", H=3, N=300, W=200, Nq=130, budgets=700, steps=7)
    sm = dkv.DKV_SCORE_TENSOR if mode == "tc" else dkv.DKV_SCORE_FP32
    tol, dens = tols(mode)
    kw = dict(descriptor=desc, sigma=float(np.sqrt(wl.d))) if desc else {}
    bank = dkv.BankLayer(wl.H, wl.d, wl.budgets_of_layer(0), wl.N, torch.bfloat16, score_mode=sm, **kw)
    bank.reset()
    ro = synth.LayerRollout(wl, 0)
    ob = oracle.LayerBank.empty(wl.budgets_of_layer(0), wl.d * (2 if desc else 1))
    theta = synth.temporal_rope_theta(wl.d, layout_first=(layout == "interleaved"))
    for t in range(wl.steps):
        b = wl.admitted_block(t)
        if b is None:
            continue
        K, V = ro.block(b)
        tc = wl.frame_coords(b)
        Kt = _rotated(K, tc, theta, layout, torch.bfloat16)
        rep, _ = update_and_compare(bank, ob, Kt, V, b, tol, dens, rope=(tc, theta, layout))
        check_report(rep, mode, t)
    bank.close()


def test_admit_rope_argument_errors(dkv):
    wl = synth.get_workload("wan13b_layer_h12", H=2, N=64, budgets=128)
    bank = dkv.BankLayer(wl.H, wl.d, wl.budgets_of_layer(0), wl.N, torch.bfloat16)
    bank.reset()
    K = torch.zeros(wl.H, wl.N, wl.d, dtype=torch.bfloat16, device="cuda")
    t = torch.zeros(wl.N, dtype=torch.int32, device="cuda")
    th = torch.zeros(wl.d // 2, dtype=torch.float32, device="cuda")
    L = dkv.lib()
    for args in ((K, K, None, th, 0), (K, K, t, None, 0), (K, K, t, th, 2), (K, K, t, th, -1)):
        Kc, Vc, tc, thc, lay = args
        st = L.dkv_bank_admit_rope(bank.handle, Kc.data_ptr(), Vc.data_ptr(), wl.N, 1,
                                   tc.data_ptr() if tc is not None else None,
                                   thc.data_ptr() if thc is not None else None, lay, None)
        assert st == 1, args
    # misaligned t_coord
    st = L.dkv_bank_admit_rope(bank.handle, K.data_ptr(), K.data_ptr(), wl.N, 1, t.data_ptr() + 2,
                               th.data_ptr(), 0, None)
    assert st == 1
    # the call errors left the handle usable: a plain admit + compress still works
    bank.admit(K, K, 1)
    bank.compress()
    bank.sync()
    bank.close()
