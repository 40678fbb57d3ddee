"""Bank-reading attention (Sec. 3.2) on grids that take the two-query-tile kernel.

The tensor-core attention has two schedules: one CTA per 128 queries with the key
range split between its two softmax groups (small grids), and one CTA per 256 queries
whose two query tiles share every key tile (grids of at least two CTAs per SM).  These
cases have enough heads to take the second one.  They use ragged bank occupancies and
window lengths, query counts that leave a partial second tile or none, and heads with
no keys.  Every output is compared with the oracle's softmax attention over
[bank | window] in float64, within 2e-2 absolute.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import load_state, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dkv():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_27922_gb300 import dkv as d
    return d


def _bf16(rng, shape, scale):
    return synth.round_to_bf16((rng.standard_normal(shape) * scale).astype(np.float32))


def _bank_with(dkv, occ, M, d=128, seed=0):
    """A bank whose head h holds occ[h] random bf16 states (the oracle's copy alongside)."""
    rng = np.random.default_rng(seed)
    H = len(occ)
    ob = oracle.LayerBank.empty([M] * H, d)
    for h, m in enumerate(occ):
        hb = ob.heads[h]
        hb.K = _bf16(rng, (m, d), 1.5).astype(np.float64)
        hb.V = _bf16(rng, (m, d), 1.0).astype(np.float64)
        hb.rho = np.ones(m, np.float32)
        hb.base = np.ones(m, np.float32)
        hb.step = np.zeros(m, np.int64)
        hb.src = np.arange(m, dtype=np.int64)
    bank = dkv.BankLayer(H, d, [M] * H, 64, torch.bfloat16, score_mode=dkv.DKV_SCORE_TENSOR)
    load_state(bank, ob)
    return bank, ob


@pytest.mark.parametrize("Nq,W", [(300, 200), (256, 0), (129, 77), (520, 128)])
def test_two_tile_attention_matches_oracle(dkv, Nq, W):
    H, M, d = 320, 400, 128   # >= 2 CTAs per SM in every case
    occ = [(37 * h) % (M + 1) for h in range(H)]   # 0 .. 400, ragged
    occ[5] = 0
    bank, ob = _bank_with(dkv, occ, M, seed=Nq + W)
    rng = np.random.default_rng(Nq)
    Q = _bf16(rng, (H, Nq, d), 1.5)
    Kw = _bf16(rng, (H, W, d), 1.5) if W else None
    Vw = _bf16(rng, (H, W, d), 1.0) if W else None
    O = bank.attend(to_dev(Q, torch.bfloat16), None if Kw is None else to_dev(Kw, torch.bfloat16),
                    None if Vw is None else to_dev(Vw, torch.bfloat16)).float().cpu().numpy()
    bank.sync()
    err = 0.0
    for h in range(H):
        kw = np.zeros((0, d)) if Kw is None else Kw[h]
        vw = np.zeros((0, d)) if Vw is None else Vw[h]
        if occ[h] + kw.shape[0] == 0:
            assert np.all(O[h] == 0), h            # no keys at all: zero output
            continue
        ref = oracle.attend(ob.heads[h], Q[h], kw, vw)
        err = max(err, float(np.abs(O[h] - ref).max()))
    assert err < 2e-2, err
    bank.close()


def test_two_tile_attention_reads_a_long_bank(dkv):
    """Many key tiles (bank 4,000 states + window 700) on the two-tile grid: the key and
    value slots are reused many times over."""
    H, M, d, Nq, W = 152, 4000, 128, 300, 700
    occ = [M - (h % 3) * 61 for h in range(H)]
    bank, ob = _bank_with(dkv, occ, M, seed=7)
    rng = np.random.default_rng(8)
    Q = _bf16(rng, (H, Nq, d), 1.5)
    Kw, Vw = _bf16(rng, (H, W, d), 1.5), _bf16(rng, (H, W, d), 1.0)
    O = bank.attend(to_dev(Q, torch.bfloat16), to_dev(Kw, torch.bfloat16), to_dev(Vw, torch.bfloat16))
    O = O.float().cpu().numpy()
    bank.sync()
    err = 0.0
    for h in range(0, H, 7):
        err = max(err, float(np.abs(O[h] - oracle.attend(ob.heads[h], Q[h], Kw[h], Vw[h])).max()))
    assert err < 2e-2, err
    bank.close()
