"""CPU emulation of the candidate sort's index arithmetic (k_update.cu: k_sort_runs,
k_sort_rank).

The kernels sort (score bits << 32 | source index) keys.  Phase 1: each warp sorts a
run of 256 keys (8 per lane) with a bitonic network in registers and warp shuffles,
direction bits taken from the run-local index.  Phase 2: each key goes to its index in
its own run plus its rank (number of smaller keys) in every other run.  This test
replays both phases step by step in Python and checks that every output position is
written exactly once and that the result is the stable ascending order, for sizes
around the run and padding boundaries and with many tied scores.
"""
import numpy as np
import pytest

SKPT = 8
RUN = 32 * SKPT
PAD = (1 << 64) - 1


def sort_run(keys):
    """Phase 1 on one run (list of 256 ints): lane t holds keys [8 t, 8 t + 8)."""
    x = [keys[t * SKPT:(t + 1) * SKPT] for t in range(32)]

    def cas_regs(k, j):
        for t in range(32):
            for r in range(SKPT):
                pr = r ^ j
                if pr > r:
                    up = ((t * SKPT + r) & k) == 0
                    a, c = x[t][r], x[t][pr]
                    if (a > c) == up:
                        x[t][r], x[t][pr] = c, a

    def cas_shfl(k, j):
        ld = j // SKPT
        new = [row[:] for row in x]
        for t in range(32):
            lower = (t & ld) == 0
            for r in range(SKPT):
                o = x[t ^ ld][r]
                up = ((t * SKPT + r) & k) == 0
                lo, hi = min(x[t][r], o), max(x[t][r], o)
                new[t][r] = lo if lower == up else hi
        x[:] = new

    k = 2
    while k <= RUN:
        j = k >> 1
        while j > 0:
            (cas_regs if j < SKPT else cas_shfl)(k, j)
            j >>= 1
        k <<= 1
    return [v for row in x for v in row]


def run_rank(r, x):
    """Branchless lower bound of x in the sorted run r (9 probes)."""
    pos, s = 0, RUN // 2
    while s > 0:
        if r[pos + s - 1] < x:
            pos += s
        s >>= 1
    return pos + (1 if r[pos] < x else 0)


def emulate(bits, N):
    nruns = (N + RUN - 1) // RUN
    runs = []
    for a in range(nruns):
        keys = [((int(bits[i]) << 32) | i) if i < N else PAD for i in range(a * RUN, (a + 1) * RUN)]
        runs.append(sort_run(keys))
    perm = [None] * N
    for a in range(nruns):
        for t in range(RUN):
            x = runs[a][t]
            if x == PAD:
                continue
            pos = t + sum(run_rank(runs[b], x) for b in range(nruns) if b != a)
            assert 0 <= pos < N and perm[pos] is None
            perm[pos] = x & 0xffffffff
    assert all(p is not None for p in perm)
    return np.array(perm)


@pytest.mark.parametrize("N", [1, 2, 255, 256, 257, 511, 1000, 1537])
@pytest.mark.parametrize("ties", [False, True])
def test_sort_matches_stable_order(N, ties):
    rng = np.random.default_rng(N * 2 + ties)
    if ties:
        bits = rng.integers(0, 5, size=N).astype(np.uint32)   # heavy ties: order by index
    else:
        bits = rng.permutation(1 << 20)[:N].astype(np.uint32)
    perm = emulate(bits, N)
    ref = np.lexsort((np.arange(N), bits))
    assert np.array_equal(perm, ref)


def test_each_run_ascending():
    rng = np.random.default_rng(7)
    keys = [int(v) for v in rng.integers(0, 1 << 40, size=RUN)]
    assert sort_run(keys) == sorted(keys)
