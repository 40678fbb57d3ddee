"""The seeded input generator: determinism, shapes, bf16 exactness and the vMF law."""
import numpy as np
from scipy.special import ive

import synth


def test_vmf_mean_resultant_length_matches_theory():
    # E[mu . x] = A_d(kappa) = I_{d/2}(kappa) / I_{d/2-1}(kappa) for x ~ vMF(mu, kappa) on S^{d-1}
    rng = np.random.default_rng(0)
    for d, kappa in ((64, 20.0), (128, 2560.0), (16, 5.0)):
        mu = np.zeros(d)
        mu[3] = 1.0
        x = synth.sample_vmf(rng, mu, kappa, 20000)
        assert np.allclose(np.linalg.norm(x, axis=1), 1.0, atol=1e-12)
        theory = ive(d / 2, kappa) / ive(d / 2 - 1, kappa)
        assert abs(x[:, 3].mean() - theory) < 4 * x[:, 3].std() / np.sqrt(len(x)) + 1e-4


def test_blocks_are_deterministic_and_bf16_exact():
    wl = synth.get_workload("wan13b_layer_h12", N=64, Nq=32, H=3)
    a = synth.LayerRollout(wl, 0)
    b = synth.LayerRollout(wl, 0, heads=[2])
    K, V = a.block(5)
    K2, V2 = b.block(5)
    assert K.shape == (3, 64, 128) and np.array_equal(K[2], K2[0]) and np.array_equal(V[2], V2[0])
    assert np.array_equal(synth.round_to_bf16(K), K)
    assert not np.array_equal(a.block(6)[0], K)
    assert abs(np.linalg.norm(K, axis=-1).mean() - np.sqrt(128)) < 0.2


def test_round_to_bf16_ties_to_even():
    x = np.array([1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -1.5, 3.0e38], np.float32)
    r = synth.round_to_bf16(x)
    assert r[0] == 1.0 and r[1] == 1.0 + 2 ** -6 and r[2] == -1.5


def test_workload_shapes():
    wl = synth.get_workload("wan14b_headwise_l40h40")
    assert len(wl.budgets) == 1600 and set(wl.budgets) <= {2340, 4680, 9360, 18720}
    assert set(wl.clusters) <= {8, 32, 128, 512} and 5.0 <= min(wl.kappa) and max(wl.kappa) <= 50.0
    wl0 = synth.get_workload("tiny_fp32_l1h2_d64")
    assert (wl0.L, wl0.H, wl0.d, wl0.N, wl0.budgets, wl0.dtype) == (1, 2, 64, 256, (512, 512), "fp32")
    assert wl0.admitted_block(0) == 0 and synth.get_workload("wan13b_layer_h12").admitted_block(0) is None


def test_sink5_window_parts_and_contents():
    """First-frame sink + five most recent frames (Sec. 4.1, App. D): 9,360 window tokens
    from step 2 on, the sink first; the block offered at step t is t - 2."""
    wl = synth.get_workload("wan13b_layer_h12_sink5", H=2, N=12, W=24, Nq=4)
    F = wl.N // wl.frames_per_block
    assert wl.window_len(0) == wl.N and wl.window_len(1) == wl.N
    for t in range(2, 6):
        parts = wl.window_parts(t)
        assert parts[0] == (0, 0, F)                                   # the sink
        frames = []
        for b, s0, e0 in parts[1:]:
            assert s0 % F == 0 and e0 % F == 0
            frames += [b * wl.frames_per_block + f for f in range(s0 // F, e0 // F)]
        assert frames == list(range(3 * t - 5, 3 * t))                # the 5 most recent frames
        assert wl.window_len(t) == 6 * F
        assert wl.admitted_block(t) == t - 2
    assert wl.admitted_block(0) is None and wl.admitted_block(1) is None
    ro = synth.LayerRollout(wl, 0)
    Kw, Vw = ro.window(3)
    K0, _ = ro.block(0)
    K1, V1 = ro.block(1)
    K2, V2 = ro.block(2)
    assert np.array_equal(Kw[:, :F], K0[:, :F])
    assert np.array_equal(Kw[:, F:3 * F], K1[:, F:]) and np.array_equal(Vw[:, 3 * F:], V2)


def test_device_stack_generator_follows_the_recipe():
    """synth.device (run on the CPU here): determinism per step, bf16 exactness, key norms
    sqrt(d), the vMF law per head (mean cosine to the assigned centre = A_d(kappa d)),
    the recurrence rule (block t uses clusters [0, (t + 1) g) while fresh ones remain),
    and independent streams for different heads and rank seeds."""
    import torch
    from synth.device import StackRollout

    wl = synth.get_workload("wan14b_headwise_l40h40", L=2, H=3, N=600, Nq=200)
    gen = StackRollout(wl, device="cpu", chunk_heads=6)
    K = torch.empty(6, 600, 128, dtype=torch.bfloat16)
    V = torch.empty_like(K)
    Q = torch.empty(6, 200, 128, dtype=torch.bfloat16)
    gen.block(2, K, V)
    gen.queries(2, Q)
    K2, V2 = torch.empty_like(K), torch.empty_like(V)
    StackRollout(wl, device="cpu", chunk_heads=6).block(2, K2, V2)
    assert torch.equal(K, K2) and torch.equal(V, V2)
    assert not torch.equal(K[0], K[1])
    K3, V3 = torch.empty_like(K), torch.empty_like(V)
    StackRollout(wl, device="cpu", chunk_heads=6, rank_seed=1).block(2, K3, V3)
    assert not torch.equal(K, K3)
    Kf = K.float()
    assert abs(Kf.norm(dim=-1).mean().item() - np.sqrt(128)) < 0.05
    assert abs(V.float().std().item() - 1.0) < 0.02
    a = gen._assign(0, 6, 2, 600, 1)   # the block's own assignment stream (_S_ASSIGN)
    mu = gen.mu[torch.arange(6)[:, None].expand(6, 600), a]
    cos = (Kf / np.sqrt(128) * mu).sum(-1)
    for h in range(6):
        kap = wl.kappa_vmf(h)
        theory = ive(64, kap) / ive(63, kap)
        assert abs(cos[h].mean().item() - theory) < 2e-3, (h, cos[h].mean().item(), theory)
        Kc, g = wl.clusters[h], max(1, wl.clusters[h] // 8)
        if 3 * g <= Kc:
            assert int(a[h].max()) < 3 * g
        assert int(a[h].min()) >= 0 and int(a[h].max()) < Kc
