"""Host-side helpers of bench.py on the CPU: the interaction-pair count behind
`interaction_pairs_per_s` and the input synthesis of `--rope`."""
import os
import sys
import types

import numpy as np
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
import oracle  # noqa: E402
import synth  # noqa: E402


def _head(m, r, e, m2):
    return types.SimpleNamespace(occupancy_before=m, admitted=r, evicted=e, occupancy_after=m2)


def test_update_pairs_counts_each_pass():
    N = 4680
    # steady state of the single-layer workload: m = M = 9,360, r* = e = N
    steady = _head(9360, N, N, 9360)
    want = 9360 * N + 9360 * N + 9360 * (N % 128) + (9360 - N) * N + N * 9360
    assert bench.update_pairs([steady], N, N) == want == 153990720
    # an empty bank only computes the new baselines of the admitted block
    assert bench.update_pairs([_head(0, N, 0, N)], N, N) == N * N
    # no eviction: no survivor pass; r* a multiple of 128: no projection columns
    assert bench.update_pairs([_head(1000, 256, 0, 1256)], N, 300) == 1000 * N + 1000 * 300 + 0 + 0 + 256 * 1256
    # heads add up
    assert bench.update_pairs([steady, steady], N, N) == 2 * want


def test_rope_input_synthesis_is_undone_by_the_oracle():
    """Keys rotated to their frames by bench.rotate_to_frames come back to the generated
    keys (up to the storage rounding) under the oracle's re-zeroing, in both layouts."""
    rng = np.random.default_rng(5)
    K = synth.round_to_bf16(rng.normal(size=(2, 40, 128)).astype(np.float32) * 3.0)
    t = (np.arange(40) // 8 + 11).astype(np.int32)
    for layout in ("interleaved", "half"):
        theta = synth.temporal_rope_theta(128, layout_first=layout == "interleaved")
        Kt = bench.rotate_to_frames(torch.from_numpy(K).to(torch.bfloat16), t, theta, layout).float().numpy()
        assert not np.allclose(Kt, K)
        back = oracle.rope_rezero(Kt, t, theta, layout, storage=None)
        assert np.max(np.abs(back - K)) <= 2.0 ** -7 * np.max(np.abs(K))


def test_kernel_work_of_a_stack_step():
    """Per-kernel algorithmic work behind the bench's per-kernel roofline, for two layers
    of two heads: flops of the tensor-core passes, bytes of the memory-bound kernels."""
    N, Nq, W, d = 4680, 4680, 4680, 128
    Ls = [types.SimpleNamespace(rmax=N, r_star=N), types.SimpleNamespace(rmax=2340, r_star=0)]
    hs = [_head(9360, N, N, 9360), _head(0, N, 0, N), _head(2340, 0, 0, 2340), _head(4680, 0, 0, 4680)]
    lay = lambda h: h // 2
    kw = lambda name: bench.kernel_work(name, d, 2, N, Nq, W, lay, Ls, hs)
    assert kw("score_tc") == 2 * d * N * (9360 + 2340 + 4680)
    assert kw("cross_tc") == 2 * d * (9360 * N + (2340 + 4680) * 2340)
    assert kw("project_tc") == 2 * d * 9360 * (N % 128)
    assert kw("subtract_tc") == 2 * d * (9360 - N) * N
    assert kw("newbase_tc") == 2 * d * (N * 9360 + N * N)
    assert kw("attend_tc") == 4 * d * Nq * (9360 + 0 + 2340 + 4680 + 4 * W)
    alg, moved = kw("commit")
    assert alg == 2 * N * (4 * d * 2 + 20) and moved > alg
    alg, moved = kw("select")
    assert alg == 12 * 9360 and moved == 32 * 9360      # only the evicting head selects


def test_stack_sample_heads_near_the_mean_budget():
    wl = synth.get_workload("wan14b_headwise_l40h40")
    heads = bench._stack_sample_heads(wl, 2)
    mean = sum(wl.budgets) / len(wl.budgets)
    assert len(heads) == 2 and all(h < wl.H for h in heads)
    assert sorted(abs(wl.budgets[h] - mean) for h in heads) == sorted(
        abs(b - mean) for b in set(wl.budgets))[:2]


def test_kernel_roofs_of_the_per_kernel_pass():
    """The per-kernel pass against the sum of its kernels' roofs (time per step at each
    kernel's measured fraction of its roof)."""
    import pytest
    pk = {"attend_tc": {"launches": 2, "avg_ms": 28.0, "share": 0.6, "frac_of_bf16_peak": 0.8},
          "cand_norms": {"launches": 2, "avg_ms": 1.0, "share": 0.1, "frac_of_hbm_alg": 0.5},
          "sort_runs": {"launches": 4, "avg_ms": 0.25, "share": 0.0}}
    r = bench.kernel_roofs(pk, 2)
    assert r["ms_per_step"] == pytest.approx(28.0 + 1.0 + 0.5)
    assert r["at_roofs_ms"] == pytest.approx(28.0 * 0.8 + 0.5)
    assert r["frac"] == pytest.approx((28.0 * 0.8 + 0.5) / 29.5)
    assert bench.kernel_roofs({}, 2) is None and bench.kernel_roofs(pk, 0) is None
