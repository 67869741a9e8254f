"""A host model of the pipeline protocol of the binary tcgen05 contractions:
the ring of shared-memory stages between the TMA producer warps and the MMA
warps, and the ring of TMEM accumulator buffers between the MMA warps and the
epilogue, each guarded by mbarriers that are waited on by phase parity.

The model runs the roles as coroutines under a random scheduler, with the
mbarrier semantics (a wait on parity P passes while the barrier's completed
phase count has the other parity) and tcgen05.commit arrivals that complete
later, in issue order per thread.  It checks what the kernels rely on:

* a stage is refilled only after its previous fill was released (a producer
  never passes an empty-barrier wait a phase early);
* every segment's pairs reach the epilogue in the buffer it reads, split over
  the MMA warps' halves;
* no schedule deadlocks.

The plain kernel deals fills round-robin to its two producers and, with two
MMA warps, to the MMA warps; it takes two MMA warps only on an even ring.  The
windowed kernel has one MMA warp that may hold a stage (the loader of an A
tile shared by later pairs) for up to ns - 2 further fills and releases it
after the stage of that fill, so stages are released out of fill order; its
producers own stages (fill f to producer (f mod ns) mod kProducers).  The
tests cover both, and show the model catching the two unsafe combinations:
two MMA warps on an odd ring with round-robin producers, and held stages with
round-robin producers."""
import random

import pytest

K_PRODUCERS = 2


class Barrier:
    def __init__(self, count):
        self.count = count
        self.pending = count
        self.phase = 0

    def arrive(self):
        self.pending -= 1
        assert self.pending >= 0, "more arrivals than the barrier's count"
        if self.pending == 0:
            self.phase += 1
            self.pending = self.count

    def passed(self, parity):
        return (self.phase & 1) != parity


class ProtocolError(AssertionError):
    pass


def simulate(seed, n, seg_start, ns, nacc, nmma, pps, producer_of, max_hold=0):
    """One random schedule of one unit: n pair positions, segments given by
    seg_start (0 = first, n = last), ns stages of pps pairs, nacc accumulator
    buffers, nmma MMA warps.  producer_of(f) names the producer of fill f.
    With max_hold > 0 (one MMA warp) a fill's stage may be held and released
    only after up to max_hold later fills.  Returns normally or raises
    ProtocolError."""
    rng = random.Random(seed)
    full = [Barrier(1) for _ in range(ns)]
    empty = [Barrier(1) for _ in range(ns)]
    accf = [Barrier(nmma) for _ in range(nacc)]
    acce = [Barrier(1) for _ in range(nacc)]
    held = [None] * ns            # fill a stage holds
    acc = {}                      # (buffer, warp) -> positions accumulated
    commits = {w: [] for w in range(nmma)}   # in flight, per issuing thread
    nfills = (n + pps - 1) // pps
    S = len(seg_start) - 1

    def producer(p):
        for f in range(nfills):
            if producer_of(f) != p:
                continue
            st, ph = f % ns, (f // ns) & 1
            yield lambda st=st, ph=ph: empty[st].passed(ph ^ 1)
            if held[st] is not None:
                raise ProtocolError(f"fill {f} refills stage {st} still holding fill {held[st]}")
            held[st] = f
            full[st].arrive()

    def mma(w):
        state = {"b": 0, "aph": 0, "s": 0, "fresh": True,
                 "seg_end": seg_start[1] if n > 0 else 0}

        def open_seg():
            b, aph = state["b"], state["aph"]
            yield lambda: acce[b].passed(aph ^ 1)
            if acc.get((b, w)):
                raise ProtocolError(f"warp {w} opens buffer {b} before the epilogue drained it")
            state["fresh"] = False

        def close_seg(pos):
            commits[w].append(("accf", state["b"]))
            state["b"] += 1
            if state["b"] == nacc:
                state["b"] = 0
                state["aph"] ^= 1
            state["s"] += 1
            if pos < n:
                state["seg_end"] = seg_start[state["s"] + 1]
            state["fresh"] = True

        owns = lambda f: (f % ns) % nmma == w
        held_until = []
        f = 0
        while f * pps < n and not owns(f):
            f += 1
        while f * pps < n:
            st, ph = f % ns, (f // ns) & 1
            start = f * pps
            np_ = min(pps, n - start)
            while state["seg_end"] <= start:
                if state["fresh"]:
                    yield from open_seg()
                close_seg(state["seg_end"])
            yield lambda st=st, ph=ph: full[st].passed(ph)
            if held[st] != f:
                raise ProtocolError(f"warp {w} consumes fill {f} but stage {st} holds {held[st]}")
            if not state["fresh"] and start + np_ <= state["seg_end"]:
                acc.setdefault((state["b"], w), []).extend(range(start, start + np_))
            else:
                for j in range(np_):
                    if state["fresh"]:
                        yield from open_seg()
                    acc.setdefault((state["b"], w), []).append(start + j)
                    if start + j + 1 == state["seg_end"]:
                        close_seg(start + j + 1)
            if max_hold and rng.random() < 0.5:
                held_until.append((f + rng.randint(1, max_hold), st))
            else:
                commits[w].append(("empty", st))
            for h in [h for h in held_until if h[0] <= f]:
                held_until.remove(h)
                commits[w].append(("empty", h[1]))
            if not state["fresh"] and start + np_ == state["seg_end"]:
                close_seg(state["seg_end"])
            f += 1
            while f * pps < n and not owns(f):
                f += 1
        for h in held_until:
            commits[w].append(("empty", h[1]))
        while state["s"] < S:
            if state["fresh"]:
                yield from open_seg()
            close_seg(state["seg_end"])

    def epilogue():
        b, ph = 0, 0
        for s in range(S):
            yield lambda b=b, ph=ph: accf[b].passed(ph)
            got = sorted(sum((acc.get((b, w), []) for w in range(nmma)), []))
            want = list(range(seg_start[s], seg_start[s + 1]))
            if got != want:
                raise ProtocolError(f"segment {s}: buffer {b} holds {got}, want {want}")
            for w in range(nmma):
                acc[(b, w)] = []
            acce[b].arrive()
            b += 1
            if b == nacc:
                b, ph = 0, ph ^ 1

    roles = [producer(p) for p in range(K_PRODUCERS)] + [mma(w) for w in range(nmma)] + [epilogue()]
    waits = [None] * len(roles)
    alive = list(range(len(roles)))
    while alive or any(commits.values()):
        runnable = [i for i in alive if waits[i] is None or waits[i]()]
        landing = [w for w in commits if commits[w]]
        choices = runnable + [-1 - w for w in landing]
        if not choices:
            raise ProtocolError("deadlock")
        c = rng.choice(choices)
        if c < 0:
            kind, i = commits[-1 - c].pop(0)
            if kind == "empty":
                held[i] = None
                empty[i].arrive()
            else:
                accf[i].arrive()
            continue
        try:
            waits[c] = next(roles[c])
        except StopIteration:
            alive.remove(c)


def random_segments(rng, n, mode):
    b = [0]
    while b[-1] < n:
        step = (rng.randint(1, 3), rng.choice([1, 1, 1, 2, 7, 20]), rng.randint(1, 40))[mode]
        b.append(min(n, b[-1] + step))
    return b


def cases(count, ns_choices, nmma_choices):
    for t in range(count):
        rng = random.Random(t)
        n = rng.randint(1, 80)
        yield dict(seed=t, n=n, seg_start=random_segments(rng, n, t % 3), ns=rng.choice(ns_choices),
                   nacc=rng.choice([1, 2, 3, 4]), nmma=rng.choice(nmma_choices), pps=rng.choice([1, 1, 2, 3, 4]))


def round_robin(f):
    return f % K_PRODUCERS


def stage_owned(ns):
    return lambda f: (f % ns) % K_PRODUCERS


def test_plain_kernel_one_mma_warp_any_ring():
    """One MMA warp releases stages in fill order: round-robin producers are
    safe with any ring size."""
    for c in cases(600, [2, 3, 4, 5, 6, 7, 8], [1]):
        simulate(producer_of=round_robin, **c)


@pytest.mark.parametrize("ns", [2, 4, 6, 8])
def test_plain_kernel_two_mma_warps_even_ring(ns):
    """Two MMA warps on an even ring: every fill of a stage comes from one
    producer and goes to one MMA warp."""
    for c in cases(250, [ns], [2]):
        simulate(producer_of=round_robin, **c)


@pytest.mark.parametrize("ns", [3, 4, 5, 6, 7, 8])
def test_windowed_kernel_held_stages(ns):
    """One MMA warp holding stages for up to ns - 2 fills, stage-owned
    producers."""
    for c in cases(250, [ns], [1]):
        simulate(producer_of=stage_owned(ns), max_hold=ns - 2, **c)


@pytest.mark.parametrize("ns", [2, 3, 4, 5, 6, 7, 8])
def test_stage_owned_producers_any_ring_any_warps(ns):
    for c in cases(250, [ns], [1, 2]):
        simulate(producer_of=stage_owned(ns), **c)


def _failures(count, ns_choices, nmma_choices, producer_of, max_hold=lambda ns: 0):
    failures = 0
    for c in cases(count, ns_choices, nmma_choices):
        try:
            simulate(producer_of=producer_of, max_hold=max_hold(c["ns"]), **c)
        except ProtocolError as e:
            assert "refills stage" in str(e)
            failures += 1
    return failures


def test_round_robin_producers_break_odd_rings_with_two_mma_warps():
    """Two MMA warps on an odd ring release stages out of fill order while
    consecutive fills of a stage come from different producers: a producer
    refills a stage still in use."""
    assert _failures(400, [3, 5, 7], [2], round_robin) > 0


def test_round_robin_producers_break_held_stages():
    """Held stages released after a later fill's stage, with round-robin
    producers: the same early pass is reachable."""
    assert _failures(600, [3, 4, 5, 6, 7], [1], round_robin, max_hold=lambda ns: ns - 2) > 0
