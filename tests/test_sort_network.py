"""CPU emulation of the candidate-sort kernel's index arithmetic (k_update.cu: k_sort).

The kernel sorts (score bits << 32 | source index) keys: 8 keys per thread, a bitonic
network in registers and warp shuffles for runs of 256 keys, then pairwise merges of
runs by rank.  This test replays that exact sequence of compare-exchanges and rank
computations in Python and checks the result is the stable ascending order, for sizes
around the run and padding boundaries.  (The merges need every run ascending; an
earlier version left runs in alternating bitonic directions.)
"""
import numpy as np
import pytest

KPT = 8
PAD = (1 << 64) - 1


def emulate(bits, N):
    n = 32 * KPT
    while n < N:
        n <<= 1
    nthr = n // KPT
    x = [[PAD] * KPT for _ in range(nthr)]
    for t in range(nthr):
        for r in range(KPT):
            i = t * KPT + r
            if i < N:
                x[t][r] = (int(bits[i]) << 32) | i

    def cas_regs(k, j):
        for t in range(nthr):
            for r in range(KPT):
                pr = r ^ j
                if pr > r:
                    up = ((t * KPT + r) & k) == 0
                    a, c = x[t][r], x[t][pr]
                    if (a > c) == up:
                        x[t][r], x[t][pr] = c, a

    def cas_shfl(k, j):
        ld = j // KPT
        new = [row[:] for row in x]
        for t in range(nthr):
            lower = (t & ld) == 0
            for r in range(KPT):
                o = x[t ^ ld][r]
                up = ((t * KPT + r) & k) == 0
                lo, hi = min(x[t][r], o), max(x[t][r], o)
                new[t][r] = lo if lower == up else hi
        x[:] = new

    k = 2
    while k <= 32 * KPT and k <= n:
        kd = (1 << 30) if k == 32 * KPT else k
        j = k >> 1
        while j > 0:
            (cas_regs if j < KPT else cas_shfl)(kd, j)
            j >>= 1
        k <<= 1
    src = [x[t][r] for t in range(nthr) for r in range(KPT)]
    length = 32 * KPT
    while length < n:
        dst = [None] * n
        for i in range(n):
            key = src[i]
            pair0 = i & ~(2 * length - 1)
            in_a = (i & length) == 0
            own = i - (pair0 if in_a else pair0 + length)
            other = src[pair0 + length:pair0 + 2 * length] if in_a else src[pair0:pair0 + length]
            lo, hi = 0, length
            while lo < hi:
                mid = (lo + hi) >> 1
                if other[mid] < key or (not in_a and other[mid] == key):
                    lo = mid + 1
                else:
                    hi = mid
            assert dst[pair0 + own + lo] is None
            dst[pair0 + own + lo] = key
        assert all(v is not None for v in dst)
        src = dst
        length <<= 1
    return [src[i] & 0xFFFFFFFF for i in range(N)]


@pytest.mark.parametrize("N", [1, 5, 256, 257, 511, 700, 1025])
def test_sort_network_is_stable_ascending(N):
    rng = np.random.default_rng(N)
    s = rng.uniform(0, 3, N).astype(np.float32)
    if N > 10:
        s[3] = s[8] = s[N - 1]          # ties resolved by source index
    perm = emulate(s.view(np.uint32), N)
    assert perm == np.lexsort((np.arange(N), s)).tolist()
