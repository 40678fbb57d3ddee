"""Host model of the mbarrier protocol of the persistent tensor-core passes.

The persistent score pass (one 128-row candidate tile per unit, 256-column bank tiles)
and the persistent crossing pass (two 128-row bank tiles per unit, 128-column candidate
tiles) each run one TMA-producer thread, one MMA-issuing thread and 16 epilogue warps
that meet only at mbarriers, whose phases run on across units.  The persistent
projection, survivor and new-baseline passes initialise their barriers again for every
unit, so each unit must end with nothing in flight.  Both attention schedules (two query
tiles per CTA; one query tile with its key tiles split over two groups) run a producer,
the issuing thread and two softmax groups whose S, P and O live in TMEM.  A mistake
there shows up
on the GPU as a hang or an exception, not as a wrong number, so the protocol is replayed
here on the host:

- every barrier keeps its completed-phase count, pending arrivals and transaction bytes
  (a phase completes when both reach zero), and every arrival and every landed copy
  names the phase it is meant for: one that lands in an earlier, still open phase would
  complete that phase early;
- a waiter waits for the completion of one phase (the kernels' parity waits) and must
  not find the barrier two phases on;
- the producer, the issuer and the epilogue warps are generator actors interleaved at
  random; copies land at random later points, in any order; MMAs and tcgen05 commits
  complete at random later points, in issue order;
- no shared-memory stage, row-tile buffer, weight slot or TMEM accumulator is written
  while a reader still needs it, and every reader finds the tile it expects;
- every run ends (no deadlock), and every epilogue warp sees every tile in order.

Five planted variants must be caught: four column stages with the combined "tile
landed and accumulator free" barrier still indexed by accumulator (the form that raised
a GPU exception: the producer arms the barrier for tile T + 2 while tile T's phase is
open), an epilogue that releases its accumulator before its TMEM loads are done, in the
re-initialising passes a tile's two MMA commits issued in the other order (the stage
barrier's commit then outlives the unit), attention with one group-0 barrier instead of
one per tile parity, and key-split attention reloading a group's value slot without
waiting for the previous tile's P.V products.
"""
import random

import pytest


class ProtocolError(AssertionError):
    pass


class Bar:
    """One mbarrier: `count` arrivals and the expected transaction bytes per phase."""

    def __init__(self, name, count):
        self.name, self.count = name, count
        self.pending, self.tx, self.phase = count, 0, 0

    def _own(self, idx, what):
        if idx != self.phase:
            raise ProtocolError(f"{what} on {self.name} meant for phase {idx} while phase {self.phase} is open")

    def _settle(self):
        if self.pending == 0 and self.tx == 0:
            self.phase += 1
            self.pending = self.count

    def arrive(self, idx, tx=0):
        self._own(idx, "arrival")
        self.tx += tx
        self.pending -= 1
        self._settle()

    def land(self, idx, nbytes):
        self._own(idx, "copy")
        self.tx -= nbytes
        if self.tx < 0:
            raise ProtocolError(f"{self.name}: more bytes landed than expected")
        self._settle()

    def passed(self, idx):
        """A parity wait for the completion of phase idx (-1: the phase before the first)."""
        if self.phase > idx + 1:
            raise ProtocolError(f"{self.name} completed phase {self.phase - 1} before its waiter for phase {idx}")
        return self.phase == idx + 1


class Sim:
    """Random interleaving of actors (generators yielding None, or (bar, phase) to wait)
    with the asynchronous copies and the in-order tensor-core queue."""

    def __init__(self, rng):
        self.rng = rng
        self.copies = []   # (bar, phase, bytes, on_land)
        self.tc = []       # ("mma", fn) / ("commit", bar, phase), in issue order

    def copy(self, bar, idx, nbytes, on_land):
        self.copies.append((bar, idx, nbytes, on_land))

    def run(self, actors, max_events=2_000_000, drain=True):
        """drain=False: return once every actor has finished (a CTA-wide barrier), with
        whatever copies and commits are still in flight."""
        cond = {i: None for i in range(len(actors))}
        live = set(range(len(actors)))
        for _ in range(max_events):
            if not live and (not drain or (not self.copies and not self.tc)):
                return
            ready = [i for i in sorted(live) if cond[i] is None or cond[i][0].passed(cond[i][1])]
            n = len(ready) + len(self.copies) + (1 if self.tc else 0)
            if n == 0:
                waits = {i: (cond[i][0].name, cond[i][1]) for i in live}
                raise ProtocolError(f"deadlock: {waits}")
            pick = self.rng.randrange(n)
            if pick < len(ready):
                i = ready[pick]
                try:
                    cond[i] = next(actors[i])
                except StopIteration:
                    live.discard(i)
            elif pick < len(ready) + len(self.copies):
                bar, idx, nbytes, on_land = self.copies.pop(pick - len(ready))
                on_land()
                bar.land(idx, nbytes)
            else:
                op = self.tc.pop(0)
                if op[0] == "mma":
                    op[1]()
                else:
                    op[1].arrive(op[2])
        raise ProtocolError("no end after the event limit")


EPI = 16   # epilogue warps of both persistent kernels


def score_wide_model(sim, units, stages=2, meta_slots=5, release_early=False):
    """The score pass with 256-column bank tiles: units = bank tiles per candidate row
    tile (0 for an empty bank; the row tile is still loaded and its buffer released)."""
    A, B, M = 36864, 73728, 1024          # row tile + extension, bank tile + extension, 1/b weights
    a_full = [Bar(f"a_full{i}", 1) for i in range(2)]
    a_free = [Bar(f"a_free{i}", 1) for i in range(2)]
    empty = [Bar(f"empty{s}", 1) for s in range(stages)]
    rdy = [Bar(f"rdy{b}", EPI + 1) for b in range(2)]     # indexed by accumulator T & 1
    accf = [Bar(f"accf{b}", 1) for b in range(2)]
    meta = [Bar(f"meta{q}", 1) for q in range(meta_slots)]
    st = dict(a_loaded=[-1, -1], a_reads=[0, 0], b_loaded=[-1] * stages, b_reads=[0] * stages,
              acc_tile=[-1, -1], acc_reading=[0, 0], meta_loaded=[-1] * meta_slots,
              meta_reading=[0] * meta_slots, released=[-1] * EPI, seen=[[] for _ in range(EPI)])

    def setter(key, i, v):
        return lambda: st[key].__setitem__(i, v)

    def producer():
        k = T = 0
        for nt in units:
            a = k & 1
            yield (a_free[a], (k >> 1) - 1)
            if st["a_reads"][a]:
                raise ProtocolError("row-tile buffer reloaded while MMAs read it")
            a_full[a].arrive(k >> 1, tx=A)
            sim.copy(a_full[a], k >> 1, A, setter("a_loaded", a, k))
            for _ in range(nt):
                s = T % stages
                yield (empty[s], T // stages - 1)
                if st["b_reads"][s]:
                    raise ProtocolError("bank-tile stage reloaded while MMAs read it")
                rdy[T & 1].arrive(T >> 1, tx=B)
                sim.copy(rdy[T & 1], T >> 1, B, setter("b_loaded", s, T))
                q = T % meta_slots
                if st["meta_reading"][q]:
                    raise ProtocolError("weight slot reloaded while an epilogue warp reads it")
                meta[q].arrive(T // meta_slots, tx=M)
                sim.copy(meta[q], T // meta_slots, M, setter("meta_loaded", q, T))
                T += 1
                yield None
            k += 1

    def mma(a, s, b, T):
        def run():
            if st["acc_reading"][b]:
                raise ProtocolError("accumulator overwritten while an epilogue warp reads it")
            st["acc_tile"][b] = T
            st["a_reads"][a] -= 1
            st["b_reads"][s] -= 1
        return run

    def issuer():
        k = T = 0
        issued = False
        for nt in units:
            a = k & 1
            yield (a_full[a], k >> 1)
            if st["a_loaded"][a] != k:
                raise ProtocolError("MMAs issued on a row tile that has not landed")
            for _ in range(nt):
                b, s = T & 1, T % stages
                yield (rdy[b], T >> 1)
                if st["b_loaded"][s] != T:
                    raise ProtocolError(f"MMAs of tile {T} issued before its bank tile landed")
                if T >= 2 and min(st["released"]) < T - 2:
                    raise ProtocolError("accumulator reused before every epilogue warp released it")
                st["a_reads"][a] += 1
                st["b_reads"][s] += 1
                sim.tc.append(("mma", mma(a, s, b, T)))
                sim.tc.append(("commit", accf[b], T >> 1))
                sim.tc.append(("commit", empty[s], T // stages))
                issued = True
                T += 1
                yield None
            sim.tc.append(("commit", a_free[a], k >> 1))
            k += 1
        if issued:   # every MMA complete before TMEM is freed
            sim.tc.append(("commit", a_free[k & 1], k >> 1))
            yield (a_free[k & 1], k >> 1)

    def epilogue(w):
        rdy[0].arrive(0)
        rdy[1].arrive(0)
        T = 0
        for nt in units:
            for _ in range(nt):
                b, q = T & 1, T % meta_slots
                yield (accf[b], T >> 1)
                yield (meta[q], T // meta_slots)
                if st["acc_tile"][b] != T:
                    raise ProtocolError(f"warp {w} finds tile {st['acc_tile'][b]} in the accumulator of tile {T}")
                if release_early:
                    st["released"][w] = T
                    rdy[b].arrive((T >> 1) + 1)
                st["acc_reading"][b] += 1
                yield None                               # TMEM loads in flight
                st["acc_reading"][b] -= 1
                if not release_early:
                    st["released"][w] = T
                    rdy[b].arrive((T >> 1) + 1)          # accumulator b free for tile T + 2
                if st["meta_loaded"][q] != T:
                    raise ProtocolError(f"warp {w} reads the weights of tile {st['meta_loaded'][q]} for tile {T}")
                st["meta_reading"][q] += 1
                yield None
                st["meta_reading"][q] -= 1
                st["seen"][w].append(T)
                T += 1

    actors = [producer(), issuer()] + [epilogue(w) for w in range(EPI)]
    sim.run(actors)
    total = sum(units)
    assert all(s == list(range(total)) for s in st["seen"])


def cross_dual_model(sim, units, stages=2):
    """The crossing pass, two row tiles per unit: units = (candidate tiles, second row
    tile present) (0 tiles: no column, the producer and issuer skip the unit)."""
    TILE, EXT = 32768, 4096
    a_full = [Bar(f"a_full{i}", 1) for i in range(2)]
    a_free = [Bar(f"a_free{i}", 1) for i in range(2)]
    empty = [Bar(f"empty{s}", 1) for s in range(stages)]
    rdy = [Bar(f"rdy{b}", EPI + 1) for b in range(2)]      # indexed by accumulator T & 1
    accf = [[Bar(f"accf{r}{b}", 1) for b in range(2)] for r in range(2)]
    st = dict(a_loaded=[-1, -1], a_reads=[0, 0], b_loaded=[-1] * stages, b_reads=[0] * stages,
              acc_tile=[[-1, -1], [-1, -1]], acc_reading=[[0, 0], [0, 0]], released=[-1] * EPI,
              seen=[[] for _ in range(EPI)])

    def setter(key, i, v):
        return lambda: st[key].__setitem__(i, v)

    def producer():
        k = T = 0
        for nt, two in units:
            if nt == 0:
                continue
            a = k & 1
            yield (a_free[a], (k >> 1) - 1)
            if st["a_reads"][a]:
                raise ProtocolError("row-tile buffer reloaded while MMAs read it")
            nb = (2 if two else 1) * (TILE + EXT)
            a_full[a].arrive(k >> 1, tx=nb)
            sim.copy(a_full[a], k >> 1, nb, setter("a_loaded", a, k))
            for _ in range(nt):
                s = T % stages
                yield (empty[s], T // stages - 1)
                if st["b_reads"][s]:
                    raise ProtocolError("column-tile stage reloaded while MMAs read it")
                rdy[T & 1].arrive(T >> 1, tx=TILE + EXT)
                sim.copy(rdy[T & 1], T >> 1, TILE + EXT, setter("b_loaded", s, T))
                T += 1
                yield None
            k += 1

    def mma(a, s, r, b, T):
        def run():
            if st["acc_reading"][r][b]:
                raise ProtocolError("accumulator overwritten while an epilogue warp reads it")
            st["acc_tile"][r][b] = T
            st["a_reads"][a] -= 1
            st["b_reads"][s] -= 1
        return run

    def issuer():
        k = T = 0
        issued = False
        for nt, two in units:
            if nt == 0:
                continue
            a = k & 1
            yield (a_full[a], k >> 1)
            if st["a_loaded"][a] != k:
                raise ProtocolError("MMAs issued on row tiles that have not landed")
            for _ in range(nt):
                b, s = T & 1, T % stages
                yield (rdy[b], T >> 1)
                if st["b_loaded"][s] != T:
                    raise ProtocolError(f"MMAs of tile {T} issued before its column tile landed")
                if T >= 2 and min(st["released"]) < T - 2:
                    raise ProtocolError("accumulator reused before every epilogue warp released it")
                for r in range(2):
                    if r == 0 or two:
                        st["a_reads"][a] += 1
                        st["b_reads"][s] += 1
                        sim.tc.append(("mma", mma(a, s, r, b, T)))
                    sim.tc.append(("commit", accf[r][b], T >> 1))   # an absent row tile: at once
                sim.tc.append(("commit", empty[s], T // stages))
                issued = True
                T += 1
                yield None
            sim.tc.append(("commit", a_free[a], k >> 1))
            k += 1
        if issued:
            sim.tc.append(("commit", a_free[k & 1], k >> 1))
            yield (a_free[k & 1], k >> 1)

    def epilogue(w):
        r = w // 8   # row tile of the unit
        rdy[0].arrive(0)
        rdy[1].arrive(0)
        T = 0
        for nt, two in units:
            live = r == 0 or two
            for _ in range(nt):
                b = T & 1
                yield (accf[r][b], T >> 1)
                if live:
                    if st["acc_tile"][r][b] != T:
                        raise ProtocolError(f"warp {w} finds tile {st['acc_tile'][r][b]} for tile {T}")
                    st["acc_reading"][r][b] += 1
                    yield None                           # TMEM loads, chunk sums, exchange
                    st["acc_reading"][r][b] -= 1
                st["released"][w] = T
                rdy[b].arrive((T >> 1) + 1)
                st["seen"][w].append(T)
                T += 1

    actors = [producer(), issuer()] + [epilogue(w) for w in range(EPI)]
    sim.run(actors)
    total = sum(nt for nt, _ in units)
    assert all(s == list(range(total)) for s in st["seen"])


def pairs_loop_model(sim, units, stages=2, accf_first=False):
    """The persistent projection / survivor / new-baseline passes: a CTA takes units (one
    128-row tile, `nt` column tiles) one after the other and initialises its barriers
    again for every unit, after a CTA-wide barrier; so when every thread has left a unit,
    no copy and no MMA commit may still be in flight (it would land in a barrier of the
    next unit).  Eight epilogue warps; the row-sum passes free an accumulator after their
    last TMEM load of the tile."""
    LOAD = 36864
    warps = 8
    for u, nt in enumerate(units):
        bar_a = Bar(f"u{u}.a", 1)
        empty = [Bar(f"u{u}.empty{s}", 1) for s in range(stages)]
        rdy = [Bar(f"u{u}.rdy{b}", warps + 1) for b in range(2)]
        accf = [Bar(f"u{u}.accf{b}", 1) for b in range(2)]
        st = dict(b_loaded=[-1] * stages, b_reads=[0] * stages, acc_tile=[-1, -1], acc_reading=[0, 0],
                  released=[-1] * warps, seen=[[] for _ in range(warps)], a_loaded=False)

        def setter(i, v, st=st):
            return lambda: st["b_loaded"].__setitem__(i, v)

        def producer(nt=nt, st=st, bar_a=bar_a, empty=empty, rdy=rdy):
            bar_a.arrive(0, tx=LOAD)
            sim.copy(bar_a, 0, LOAD, lambda: st.__setitem__("a_loaded", True))
            for t in range(nt):
                s = t % stages
                yield (empty[s], t // stages - 1)
                if st["b_reads"][s]:
                    raise ProtocolError("column-tile stage reloaded while MMAs read it")
                rdy[t & 1].arrive(t >> 1, tx=LOAD)
                sim.copy(rdy[t & 1], t >> 1, LOAD, setter(s, t))
                yield None
            # never leave with copies in flight: the row tile, then the last stages' tiles
            yield (bar_a, 0)
            for t in range(max(0, nt - stages), nt):
                yield (rdy[t & 1], t >> 1)

        def mma(s, b, t, st=st):
            def run():
                if st["acc_reading"][b]:
                    raise ProtocolError("accumulator overwritten while an epilogue warp reads it")
                st["acc_tile"][b] = t
                st["b_reads"][s] -= 1
            return run

        def issuer(nt=nt, st=st, bar_a=bar_a, empty=empty, rdy=rdy, accf=accf):
            yield (bar_a, 0)
            if not st["a_loaded"]:
                raise ProtocolError("MMAs issued on a row tile that has not landed")
            for t in range(nt):
                s, b = t % stages, t & 1
                yield (rdy[b], t >> 1)
                if st["b_loaded"][s] != t:
                    raise ProtocolError(f"MMAs of tile {t} issued before its column tile landed")
                if t >= 2 and min(st["released"]) < t - 2:
                    raise ProtocolError("accumulator reused before every epilogue warp released it")
                st["b_reads"][s] += 1
                sim.tc.append(("mma", mma(s, b, t)))
                commits = [("commit", empty[s], t // stages), ("commit", accf[b], t >> 1)]
                sim.tc.extend(commits[::-1] if accf_first else commits)
                yield None
            if nt > 0:   # every MMA complete before the unit ends
                yield (accf[(nt - 1) & 1], (nt - 1) >> 1)

        def epilogue(w, nt=nt, st=st, rdy=rdy, accf=accf):
            rdy[0].arrive(0)
            rdy[1].arrive(0)
            for t in range(nt):
                b = t & 1
                yield (accf[b], t >> 1)
                if st["acc_tile"][b] != t:
                    raise ProtocolError(f"warp {w} finds tile {st['acc_tile'][b]} for tile {t}")
                st["acc_reading"][b] += 1
                yield None                               # the tile's TMEM loads
                st["acc_reading"][b] -= 1
                st["released"][w] = t
                rdy[b].arrive((t >> 1) + 1)              # then the chunk arithmetic
                yield None
                st["seen"][w].append(t)

        actors = [producer(), issuer()] + [epilogue(w) for w in range(warps)]
        sim.run(actors, drain=False)
        if sim.copies or sim.tc:
            raise ProtocolError(f"unit {u} ends with {len(sim.copies)} copies and {len(sim.tc)} "
                                f"tensor-core operations in flight; its barriers are initialised again")
        assert all(x == list(range(nt)) for x in st["seen"])


def attend2_model(sim, nt, G, pf0_single=False):
    """Attention with two query tiles per CTA: a producer, the MMA-issuing thread and two
    softmax groups of four warps (group g over query tile g; G = 1 when only one query
    tile is valid).  Per key tile i the issuer, after group 0's barrier, issues
    PV_0(i) and S_0(i + 1), then after group 1's barrier PV_1(i) and S_1(i + 1).  Group g's
    S and P share one TMEM region (P(i) overwrites S(i), S(i + 1) overwrites P(i)); O is
    rescaled in place by the softmax warps.  Key slots: 2 (K(0) through its own barrier,
    K(i + 1) with tile i); value slots: 3.  pf0 is one barrier per tile parity (group 0's
    softmax warps + the producer with V(i), K(i + 1)); pf1 one barrier (group 1)."""
    TB = 32768
    npf = 1 if pf0_single else 2
    q_full, k0_full = Bar("q_full", 1), Bar("k0_full", 1)
    pf0 = [Bar(f"pf0_{p}", 5) for p in range(npf)]
    pf1 = Bar("pf1", 4)
    k_empty = [Bar(f"k_empty{s}", 1) for s in range(2)]
    v_empty = [Bar(f"v_empty{s}", 1) for s in range(3)]
    s_full = [Bar(f"s_full{g}", 1) for g in range(2)]
    pv_done = [Bar(f"pv_done{g}", 1) for g in range(2)]
    st = dict(q=False, k=[-1, -1], k_reads=[0, 0], v=[-1, -1, -1], v_reads=[0, 0, 0],
              region=[("none", -1)] * 8, busy=[0] * 8, o_through=[-1, -1],
              pv_pending=[0, 0], seen=[[] for _ in range(8)])

    def pf(i):   # the barrier and phase of group 0 for tile i
        return (pf0[0], i) if pf0_single else (pf0[i & 1], i >> 1)

    def setter(key, i, v):
        return lambda: st[key].__setitem__(i, v)

    def producer():
        q_full.arrive(0, tx=G * TB)
        sim.copy(q_full, 0, G * TB, lambda: st.__setitem__("q", True))
        k0_full.arrive(0, tx=TB)
        sim.copy(k0_full, 0, TB, setter("k", 0, 0))
        for i in range(nt):
            if i >= 2:   # the phase two tiles back is over (the same parity's barrier)
                yield pf(i - 2)
            if i >= 3:
                yield (v_empty[i % 3], (i - 3) // 3)
            knext = i + 1 < nt
            if knext and i >= 1:
                yield (k_empty[(i + 1) & 1], (i - 1) >> 1)
            if st["v_reads"][i % 3]:
                raise ProtocolError("value slot reloaded while P.V products read it")
            if knext and st["k_reads"][(i + 1) & 1]:
                raise ProtocolError("key slot reloaded while score products read it")
            bar, idx = pf(i)
            bar.arrive(idx, tx=(2 if knext else 1) * TB)
            sim.copy(bar, idx, TB, setter("v", i % 3, i))
            if knext:
                sim.copy(bar, idx, TB, setter("k", (i + 1) & 1, i + 1))
            yield None
        yield (q_full, 0)
        yield (k0_full, 0)
        for i in range(max(0, nt - 2), nt):
            yield pf(i)

    quarter = lambda g: range(4 * g, 4 * g + 4)   # a group's warps: TMEM lane quarters

    def s_mma(g, i):
        def run():
            if any(st["busy"][w] for w in quarter(g)):
                raise ProtocolError(f"S_{g}({i}) written while a softmax warp of group {g} works on its lanes")
            for w in quarter(g):
                st["region"][w] = ("S", i)
            st["k_reads"][i & 1] -= 1
        return run

    def pv_mma(g, i):
        def run():
            if any(st["region"][w] != ("P", i) for w in quarter(g)):
                raise ProtocolError(f"PV_{g}({i}) reads {[st['region'][w] for w in quarter(g)]} instead of P({i})")
            if any(st["busy"][w] for w in quarter(g)):
                raise ProtocolError(f"PV_{g}({i}) while a softmax warp of group {g} works on O")
            st["o_through"][g] = i
            st["v_reads"][i % 3] -= 1
            st["pv_pending"][g] -= 1
        return run

    def issue_s(g, i):
        if st["k"][i & 1] != i:
            raise ProtocolError(f"S_{g}({i}) issued before K({i}) landed")
        st["k_reads"][i & 1] += 1
        sim.tc.append(("mma", s_mma(g, i)))
        sim.tc.append(("commit", s_full[g], i))
        if g == G - 1:
            sim.tc.append(("commit", k_empty[i & 1], i >> 1))

    def issue_pv(g, i):
        if st["v"][i % 3] != i:
            raise ProtocolError(f"PV_{g}({i}) issued before V({i}) landed")
        st["v_reads"][i % 3] += 1
        st["pv_pending"][g] += 1
        sim.tc.append(("mma", pv_mma(g, i)))
        sim.tc.append(("commit", pv_done[g], i))
        if g == G - 1:
            sim.tc.append(("commit", v_empty[i % 3], i // 3))

    def issuer():
        yield (q_full, 0)
        yield (k0_full, 0)
        if not st["q"]:
            raise ProtocolError("score products issued before the query tiles landed")
        for g in range(G):
            issue_s(g, 0)
        for i in range(nt):
            yield pf(i)
            issue_pv(0, i)
            if i + 1 < nt:
                issue_s(0, i + 1)
            if G == 2:
                yield (pf1, i)
                issue_pv(1, i)
                if i + 1 < nt:
                    issue_s(1, i + 1)
            yield None
        yield (pv_done[0], nt - 1)
        if G == 2:
            yield (pv_done[1], nt - 1)

    def softmax(w):
        g = w // 4
        ng = nt if g < G else 0
        for i in range(ng):
            yield (s_full[g], i)
            if st["region"][w] != ("S", i):
                raise ProtocolError(f"warp {w} finds {st['region'][w]} for S({i})")
            st["busy"][w] += 1
            yield None                               # S loads, P stores, O rescale
            if st["pv_pending"][g] or st["o_through"][g] != i - 1:
                raise ProtocolError(f"group {g} rescales O with P.V products of earlier tiles in flight")
            st["busy"][w] -= 1
            st["region"][w] = ("P", i)
            if g == 0:
                bar, idx = pf(i)
                bar.arrive(idx)
            else:
                pf1.arrive(i)
            st["seen"][w].append(i)
            yield None
        if ng:
            yield (pv_done[g], ng - 1)
            if st["o_through"][g] != ng - 1:
                raise ProtocolError(f"group {g} reads O before the last P.V product")

    actors = [producer(), issuer()] + [softmax(w) for w in range(8)]
    sim.run(actors)
    assert all(st["seen"][w] == (list(range(nt)) if w // 4 < G else []) for w in range(8))


def attend_split_model(sim, nt, skip_v_wait=False):
    """Attention with the key tiles of one query tile split over two softmax groups
    (group 0 the first (nt + 1) / 2 tiles, group 1 the rest).  Per group: its first key
    tile through its own barrier, two key slots, one value slot; p_full_g (four softmax
    warps + the producer with V(i) and K(i + 1)) has one phase per tile; the producer
    reloads the group's value slot only after PV_g(i - 1) is complete."""
    TB = 32768
    n = [(nt + 1) // 2, nt - (nt + 1) // 2]
    q_full = Bar("q_full", 1)
    k0_full = [Bar(f"k0_full{g}", 1) for g in range(2)]
    k_empty = [[Bar(f"k_empty{g}{s}", 1) for s in range(2)] for g in range(2)]
    v_empty = [Bar(f"v_empty{g}", 1) for g in range(2)]
    s_full = [Bar(f"s_full{g}", 1) for g in range(2)]
    p_full = [Bar(f"p_full{g}", 5) for g in range(2)]
    pv_done = [Bar(f"pv_done{g}", 1) for g in range(2)]
    st = dict(q=False, k=[[-1, -1], [-1, -1]], k_reads=[[0, 0], [0, 0]], v=[-1, -1], v_reads=[0, 0],
              region=[("none", -1)] * 8, busy=[0] * 8, o_through=[-1, -1], pv_pending=[0, 0],
              seen=[[] for _ in range(8)])
    quarter = lambda g: range(4 * g, 4 * g + 4)

    def set_k(g, slot, i):
        return lambda: st["k"][g].__setitem__(slot, i)

    def set_v(g, i):
        return lambda: st["v"].__setitem__(g, i)

    def producer():
        q_full.arrive(0, tx=TB)
        sim.copy(q_full, 0, TB, lambda: st.__setitem__("q", True))
        for g in range(2):
            if n[g] > 0:
                k0_full[g].arrive(0, tx=TB)
                sim.copy(k0_full[g], 0, TB, set_k(g, 0, 0))
        for i in range(n[0]):
            for g in range(2):
                if i >= n[g]:
                    continue
                if i > 0 and not skip_v_wait:
                    yield (v_empty[g], i - 1)
                knext = i + 1 < n[g]
                if knext and i > 0:
                    yield (k_empty[g][(i + 1) & 1], (i - 1) >> 1)
                if st["v_reads"][g]:
                    raise ProtocolError(f"value slot of group {g} reloaded while P.V products read it")
                if knext and st["k_reads"][g][(i + 1) & 1]:
                    raise ProtocolError(f"key slot of group {g} reloaded while score products read it")
                p_full[g].arrive(i, tx=(2 if knext else 1) * TB)
                sim.copy(p_full[g], i, TB, set_v(g, i))
                if knext:
                    sim.copy(p_full[g], i, TB, set_k(g, (i + 1) & 1, i + 1))
                yield None
        yield (q_full, 0)
        for g in range(2):
            if n[g] > 0:
                yield (k0_full[g], 0)
                yield (p_full[g], n[g] - 1)

    def s_mma(g, i):
        def run():
            if any(st["busy"][w] for w in quarter(g)):
                raise ProtocolError(f"S_{g}({i}) written while a softmax warp of group {g} works on its lanes")
            for w in quarter(g):
                st["region"][w] = ("S", i)
            st["k_reads"][g][i & 1] -= 1
        return run

    def pv_mma(g, i):
        def run():
            if any(st["region"][w] != ("P", i) for w in quarter(g)):
                raise ProtocolError(f"PV_{g}({i}) does not read P({i})")
            if any(st["busy"][w] for w in quarter(g)):
                raise ProtocolError(f"PV_{g}({i}) while a softmax warp of group {g} works on O")
            st["o_through"][g] = i
            st["v_reads"][g] -= 1
            st["pv_pending"][g] -= 1
        return run

    def issue_s(g, i):
        if st["k"][g][i & 1] != i:
            raise ProtocolError(f"S_{g}({i}) issued before its key tile landed")
        st["k_reads"][g][i & 1] += 1
        sim.tc.append(("mma", s_mma(g, i)))
        sim.tc.append(("commit", k_empty[g][i & 1], i >> 1))
        sim.tc.append(("commit", s_full[g], i))

    def issuer():
        yield (q_full, 0)
        if not st["q"]:
            raise ProtocolError("score products issued before the query tile landed")
        for g in range(2):
            if n[g] > 0:
                yield (k0_full[g], 0)
                issue_s(g, 0)
        for i in range(n[0]):
            for g in range(2):
                if i >= n[g]:
                    continue
                yield (p_full[g], i)
                if st["v"][g] != i:
                    raise ProtocolError(f"PV_{g}({i}) issued before V({i}) landed")
                st["v_reads"][g] += 1
                st["pv_pending"][g] += 1
                sim.tc.append(("mma", pv_mma(g, i)))
                sim.tc.append(("commit", v_empty[g], i))
                sim.tc.append(("commit", pv_done[g], i))
                if i + 1 < n[g]:
                    issue_s(g, i + 1)
                yield None
        for g in range(2):
            if n[g] > 0:
                yield (pv_done[g], n[g] - 1)

    def softmax(w):
        g = w // 4
        for i in range(n[g]):
            yield (s_full[g], i)
            if st["region"][w] != ("S", i):
                raise ProtocolError(f"warp {w} finds {st['region'][w]} for S({i})")
            st["busy"][w] += 1
            yield None
            if st["pv_pending"][g] or st["o_through"][g] != i - 1:
                raise ProtocolError(f"group {g} rescales O with P.V products of earlier tiles in flight")
            st["busy"][w] -= 1
            st["region"][w] = ("P", i)
            p_full[g].arrive(i)
            st["seen"][w].append(i)
            yield None
        if n[g]:
            yield (pv_done[g], n[g] - 1)
            if st["o_through"][g] != n[g] - 1:
                raise ProtocolError(f"group {g} reads O before the last P.V product")

    actors = [producer(), issuer()] + [softmax(w) for w in range(8)]
    sim.run(actors)
    assert all(st["seen"][w] == list(range(n[w // 4])) for w in range(8))


def _score_units(rng):
    return [rng.choice([0, 1, 1, 2, 3, 5]) for _ in range(rng.randrange(1, 8))]


def _cross_units(rng):
    return [(rng.choice([0, 1, 2, 3, 4, 7]), rng.random() < 0.7) for _ in range(rng.randrange(1, 7))]


@pytest.mark.parametrize("seed", range(60))
def test_score_pass_protocol(seed):
    rng = random.Random(seed)
    score_wide_model(Sim(rng), _score_units(rng))


@pytest.mark.parametrize("seed", range(60))
def test_crossing_pass_protocol(seed):
    rng = random.Random(1000 + seed)
    cross_dual_model(Sim(rng), _cross_units(rng))


@pytest.mark.parametrize("seed", range(40))
def test_persistent_row_passes_protocol(seed):
    rng = random.Random(2000 + seed)
    pairs_loop_model(Sim(rng), [rng.randrange(1, 7) for _ in range(rng.randrange(1, 6))])


@pytest.mark.parametrize("seed", range(60))
def test_attention_protocol(seed):
    rng = random.Random(3000 + seed)
    attend2_model(Sim(rng), rng.randrange(1, 9), rng.choice([1, 2, 2]))


@pytest.mark.parametrize("seed", range(60))
def test_split_attention_protocol(seed):
    rng = random.Random(4000 + seed)
    attend_split_model(Sim(rng), rng.randrange(1, 12))


def test_long_units_both_passes():
    rng = random.Random(7)
    score_wide_model(Sim(rng), [0, 9, 1, 0, 12, 2])
    cross_dual_model(Sim(rng), [(9, True), (0, True), (1, False), (12, True), (2, False)])


def _caught(fn, seeds):
    for seed in seeds:
        try:
            fn(seed)
        except ProtocolError:
            return True
    return False


def test_planted_four_stages_with_accumulator_barrier_is_caught():
    """Four column stages, the combined barrier still one per accumulator: the producer,
    up to four tiles ahead, arms the barrier of tile T + 2 while tile T's phase is open."""
    assert _caught(lambda s: cross_dual_model(Sim(random.Random(s)), [(8, True), (6, False)], stages=4),
                   range(40))
    assert _caught(lambda s: score_wide_model(Sim(random.Random(s)), [8, 6], stages=4), range(40))


def test_planted_commit_order_is_caught():
    """The last waits of a unit are on the accumulator barrier of its last tile (the
    epilogue's and the issuer's); with that tile's two commits issued accumulator first,
    the stage barrier's commit can still be in flight when the next unit initialises it."""
    assert _caught(lambda s: pairs_loop_model(Sim(random.Random(s)), [3, 2], accf_first=True), range(300))


def test_planted_single_attention_barrier_is_caught():
    """Attention with one group-0 barrier for all tiles instead of one per tile parity:
    the producer arms tile i + 1 while tile i's phase is still open."""
    assert _caught(lambda s: attend2_model(Sim(random.Random(s)), 6, 2, pf0_single=True), range(40))


def test_planted_missing_value_slot_wait_is_caught():
    """Key-split attention whose producer reloads a group's one value slot without
    waiting for the previous tile's P.V products."""
    assert _caught(lambda s: attend_split_model(Sim(random.Random(s)), 8, skip_v_wait=True), range(40))


def test_planted_early_release_is_caught():
    """An epilogue warp that frees its accumulator before its TMEM loads are done lets
    the MMAs of tile T + 2 overwrite what it still reads."""
    assert _caught(lambda s: score_wide_model(Sim(random.Random(s)), [6, 5], release_early=True), range(60))
