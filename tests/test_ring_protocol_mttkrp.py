"""A host model of the tcgen05 MTTKRP kernel's pipeline protocol, in the
style of test_ring_protocol.py: four roles as coroutines under a random
scheduler, mbarriers waited on by phase parity, TMA copies and
tcgen05.commit arrivals that complete later (commits in issue order).

Roles and barriers, as in the kernel:

* producer: per fill (a stage of up to four triples) waits the stage's
  empty barrier, then its copies land on the stage's full barrier;
* group warp: per fill waits the stage's empty barrier (its plan word is
  then free); for each triple that opens a group waits until the epilogue
  released the group's accumulator buffer (acce), then requests the group's
  E tile into that buffer's E slot (ef lands later); for each triple that
  closes a group posts whether the group ends its output key (info,
  infoc); then posts the stage's plan (planned);
* MMA thread: per fill waits full and planned, accumulates each triple
  into its group's buffer, commits a buffer at its group's end (accf) and
  the stage after its last triple (empty);
* epilogue: per group waits ef, reads E, waits infoc, reads the info, waits
  accf, drains the buffer, releases it (acce).

It checks that every wait passes only for the phase it means, that no plan
word, E slot, info word or accumulator buffer is overwritten before it was
read, that every group's triples reach the epilogue in its buffer, and that
no schedule deadlocks."""
import random

import pytest

from tests.test_ring_protocol import Barrier, ProtocolError

STAGES = 4
PER_STAGE = 4
ACC = 4


def simulate(seed, groups_of, keys_of, skip_buffer_wait=False):
    """groups_of[t] / keys_of[t]: group and output key of triple t (groups
    are runs of equal group ids, never spanning two keys).
    skip_buffer_wait plants a mistake: the group warp opens groups without
    waiting for the epilogue's release of their buffer."""
    rng = random.Random(seed)
    n = len(groups_of)
    nfills = (n + PER_STAGE - 1) // PER_STAGE
    full = [Barrier(1) for _ in range(STAGES)]
    empty = [Barrier(1) for _ in range(STAGES)]
    planned = [Barrier(1) for _ in range(STAGES)]
    accf = [Barrier(1) for _ in range(ACC)]
    acce = [Barrier(1) for _ in range(ACC)]
    ef = [Barrier(1) for _ in range(ACC)]
    infoc = [Barrier(1) for _ in range(ACC)]
    stage_fill = [None] * STAGES     # fill whose copies a stage holds
    plan_word = [None] * STAGES      # fill whose plan a stage's word holds
    e_slot = [None] * ACC            # group whose E tile a slot holds (landed)
    e_read = [True] * ACC            # slot's E read by the epilogue
    info_word = [None] * ACC
    info_read = [True] * ACC
    acc = [None] * ACC               # (group, triples) a buffer holds
    released = [True] * ACC          # buffer drained and released
    pending = []                     # async events: TMA landings (any order)
    commits = []                     # tcgen05.commit arrivals, in issue order
    opens = [t == 0 or groups_of[t] != groups_of[t - 1] for t in range(n)]
    closes = [t == n - 1 or groups_of[t + 1] != groups_of[t] for t in range(n)]
    group_list = [groups_of[t] for t in range(n) if opens[t]]

    def producer():
        for f in range(nfills):
            st, ph = f % STAGES, (f // STAGES) & 1
            yield lambda st=st, ph=ph: empty[st].passed(ph ^ 1)
            if stage_fill[st] is not None:
                raise ProtocolError(f"fill {f} refills stage {st} still holding fill {stage_fill[st]}")
            pending.append(("full", st, f))

    def group_warp():
        gb = gph = cb = 0
        for f in range(nfills):
            st, ph = f % STAGES, (f // STAGES) & 1
            yield lambda st=st, ph=ph: empty[st].passed(ph ^ 1)
            if plan_word[st] is not None:
                raise ProtocolError(f"plan of fill {f} overwrites the unread plan of fill {plan_word[st]}")
            for t in range(f * PER_STAGE, min(n, (f + 1) * PER_STAGE)):
                if opens[t]:
                    b, p = gb, gph
                    if not skip_buffer_wait:
                        yield lambda b=b, p=p: acce[b].passed(p ^ 1)
                    if not e_read[b] or not released[b]:
                        raise ProtocolError(f"group {groups_of[t]} takes buffer {b} before the epilogue freed it")
                    e_read[b] = False
                    pending.append(("ef", b, groups_of[t]))
                    gb += 1
                    if gb == ACC:
                        gb, gph = 0, gph ^ 1
                if closes[t]:
                    if not info_read[cb]:
                        raise ProtocolError(f"info of group {groups_of[t]} overwrites an unread info word")
                    info_word[cb] = (groups_of[t], t == n - 1 or keys_of[t + 1] != keys_of[t])
                    info_read[cb] = False
                    infoc[cb].arrive()
                    cb = (cb + 1) % ACC
            plan_word[st] = f
            planned[st].arrive()

    def mma():
        b = 0
        for f in range(nfills):
            st, ph = f % STAGES, (f // STAGES) & 1
            yield lambda st=st, ph=ph: full[st].passed(ph) and planned[st].passed(ph)
            if stage_fill[st] != f or plan_word[st] != f:
                raise ProtocolError(f"fill {f}: stage holds {stage_fill[st]}, plan {plan_word[st]}")
            plan_word[st] = None   # the plan word is read
            for t in range(f * PER_STAGE, min(n, (f + 1) * PER_STAGE)):
                if opens[t]:
                    if not released[b]:
                        raise ProtocolError(f"group {groups_of[t]} overwrites buffer {b} before it was drained")
                    released[b] = False
                    acc[b] = (groups_of[t], [])
                if acc[b] is None or acc[b][0] != groups_of[t]:
                    raise ProtocolError(f"triple {t} accumulates into buffer {b} holding {acc[b]}")
                acc[b][1].append(t)
                if closes[t]:
                    commits.append(("accf", b))
                    b = (b + 1) % ACC
            commits.append(("empty", st))

    def epilogue():
        b = ph = 0
        for g in group_list:
            yield lambda b=b, ph=ph: ef[b].passed(ph)
            if e_slot[b] != g:
                raise ProtocolError(f"epilogue of group {g} reads the E tile of group {e_slot[b]}")
            e_read[b] = True
            yield lambda b=b, ph=ph: infoc[b].passed(ph)
            if info_word[b] is None or info_word[b][0] != g:
                raise ProtocolError(f"epilogue of group {g} reads info {info_word[b]}")
            info_read[b] = True
            yield lambda b=b, ph=ph: accf[b].passed(ph)
            want = [t for t in range(n) if groups_of[t] == g]
            if acc[b] is None or acc[b][0] != g or acc[b][1] != want:
                raise ProtocolError(f"group {g}: buffer {b} holds {acc[b]}, want triples {want}")
            released[b] = True
            acce[b].arrive()
            b += 1
            if b == ACC:
                b, ph = 0, ph ^ 1

    def land(ev):
        kind, i, x = ev
        if kind == "full":
            stage_fill[i] = x
            full[i].arrive()
        else:
            e_slot[i] = x
            ef[i].arrive()

    roles = [producer(), group_warp(), mma(), epilogue()]
    waits = [None] * len(roles)
    alive = list(range(len(roles)))
    while alive or pending or commits:
        runnable = [i for i in alive if waits[i] is None or waits[i]()]
        choices = runnable + (["tma"] if pending else []) + (["commit"] if commits else [])
        if not choices:
            raise ProtocolError("deadlock")
        c = rng.choice(choices)
        if c == "tma":
            land(pending.pop(rng.randrange(len(pending))))
        elif c == "commit":
            kind, i = commits.pop(0)
            if kind == "empty":
                stage_fill[i] = None
                empty[i].arrive()
            else:
                accf[i].arrive()
        else:
            try:
                waits[c] = next(roles[c])
            except StopIteration:
                alive.remove(c)


def random_triples(rng, n, mode):
    """Group and key ids for n triples: groups are runs of equal E tuples
    inside a key (mean 3.5 triples at full size; here from 1 to long)."""
    groups, keys = [], []
    g = k = 0
    t = 0
    while t < n:
        key_len = rng.randint(1, (6, 20, 60)[mode])
        end = min(n, t + key_len)
        while t < end:
            run = min(end - t, rng.choice((1, 1, 2, 3, 4, 5, 9)))
            groups += [g] * run
            keys += [k] * run
            g += 1
            t += run
        k += 1
    return groups, keys


@pytest.mark.parametrize("mode", [0, 1, 2])
def test_mttkrp_protocol(mode):
    for seed in range(600):
        rng = random.Random(seed * 3 + mode)
        groups, keys = random_triples(rng, rng.randint(1, 70), mode)
        simulate(seed, groups, keys)


def test_mttkrp_protocol_one_triple_groups():
    """Every triple its own group (E changes every triple, as when the
    first join is on K): four groups a stage, the buffer ring's tightest use."""
    for seed in range(300):
        n = random.Random(seed).randint(1, 60)
        simulate(seed, list(range(n)), [t // 3 for t in range(n)])


def test_model_catches_a_missing_buffer_wait():
    """The mistake planted in the model (a group warp that reuses a buffer
    without waiting for its release) is caught."""
    caught = 0
    for seed in range(200):
        n = random.Random(seed).randint(20, 60)
        try:
            simulate(seed, list(range(n)), [t // 3 for t in range(n)], skip_buffer_wait=True)
        except ProtocolError:
            caught += 1
    assert caught > 0
