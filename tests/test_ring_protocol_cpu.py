"""A model of the weight ring of the persistent decode-chain kernel, on the CPU.

The kernel streams every weight chunk of every stage through `nslots`
shared-memory slots.  Chunk c (numbered across the whole token) lives in slot
c % nslots and lands on full barrier c % nbars; a consumer waits for it with
the barrier's phase parity (c // nbars) & 1.  A parity wait only tells the
wanted phase from the one before it, so it passes wrongly ("aliases") when the
barrier is still one whole cycle behind: chunk c - nbars has not landed yet.
Consumer warps take the items of a stage round-robin and skip the chunks that
hold none of their items, so within a stage a warp can run ahead of the
oldest unconsumed chunk (all warps meet at a barrier at every stage start).
The planner's rule, nslots + ceil(NW / items per slot) <= nbars, bounds how
far ahead, and this model (random copy and compute latencies) checks that no
wait aliases under the rule, and that waits do alias without it.
"""
import heapq
import math
import random

import pytest


def simulate(stages, nslots, nbars, nw, rng):
    """Discrete-event run of one token.  stages: list of (items, items per
    chunk).  Returns the number of aliased waits (0 means the protocol held);
    raises if the run deadlocks."""
    chunks = []            # per global chunk: (stage, first item, end item)
    for si, (items, ips) in enumerate(stages):
        for a in range(0, items, ips):
            chunks.append((si, a, min(items, a + ips)))
    nch = len(chunks)
    landed = [False] * nch
    completed = [0] * nbars            # completed phases per full barrier
    consumed = [0] * nch               # items consumed per chunk
    released = [False] * nch
    aliased = 0

    # warp programs: (stage, chunk) visits in order, stage after stage
    progs = []
    for w in range(nw):
        seq = []
        base = 0
        for si, (items, ips) in enumerate(stages):
            for it in range(w, items, nw):
                seq.append((si, base + it // ips))
            base += math.ceil(items / ips)
        progs.append(seq)
    pos = [0] * nw
    stage_left = [0] * len(stages)   # items of each stage not yet consumed
    for si, (items, _) in enumerate(stages):
        stage_left[si] = items
    at_barrier = set()               # warps waiting for the previous stage to finish

    t = 0.0
    events = []            # (time, kind, payload)
    next_issue = 0         # producer: next chunk to issue

    def try_issue(now):
        nonlocal next_issue
        while next_issue < nch:
            c = next_issue
            if c >= nslots and not released[c - nslots]:
                return
            heapq.heappush(events, (now + rng.uniform(0.5, 3.0), 0, c))   # copy lands later
            next_issue += 1

    waiting = {}           # warp -> chunk it waits for

    def stage_done(si):
        return all(stage_left[j] == 0 for j in range(si))

    def step_warp(w, now):
        nonlocal aliased
        while pos[w] < len(progs[w]):
            si, c = progs[w][pos[w]]
            if not stage_done(si):                   # the stage-start barrier
                at_barrier.add(w)
                return
            b, k = c % nbars, c // nbars
            want = k & 1
            cur = completed[b]
            if cur % 2 != want:                      # the parity wait passes
                if cur != k + 1:                     # ... but not on chunk c's phase
                    aliased += 1
                heapq.heappush(events, (now + rng.uniform(0.2, 1.5), 1, (w, si, c)))
                pos[w] += 1
                return
            waiting[w] = c
            return

    try_issue(t)
    for w in range(nw):
        step_warp(w, t)
    while events:
        t, kind, payload = heapq.heappop(events)
        if kind == 0:                                # chunk c landed
            c = payload
            landed[c] = True
            completed[c % nbars] += 1
            for w, wc in list(waiting.items()):
                if wc % nbars == c % nbars:
                    del waiting[w]
                    step_warp(w, t)
        else:                                        # warp w consumed an item of chunk c
            w, si, c = payload
            consumed[c] += 1
            stage_left[si] -= 1
            _, a, e = chunks[c]
            if consumed[c] == e - a:
                released[c] = True
                try_issue(t)
            step_warp(w, t)
            if stage_left[si] == 0:
                for v in sorted(at_barrier):
                    at_barrier.discard(v)
                    step_warp(v, t)
    if any(pos[w] < len(progs[w]) for w in range(nw)):
        raise RuntimeError("deadlock")
    return aliased


def plan_nbars(nslots, stages, nw, max_bars=48):
    """The planner's choice: the largest multiple of nslots up to 48 barriers,
    accepted only if nslots + ceil(nw / ips) <= nbars for every stage."""
    nbars = (max_bars // nslots) * nslots
    ok = all(nslots + math.ceil(nw / ips) <= nbars for _, ips in stages)
    return nbars, ok


# stage mixes shaped like the chain (items per CTA, items per chunk)
LAYER_3B = [(17, 5), (10, 5), (27, 2), (10, 2)]
LAYER_8B = [(21, 4), (14, 4), (48, 2), (14, 1)]
NARROW = [(3, 1), (2, 1), (5, 1), (1, 1)]


@pytest.mark.parametrize("layer", [LAYER_3B, LAYER_8B, NARROW])
@pytest.mark.parametrize("nslots", [3, 6, 9, 12, 16])
def test_no_aliased_wait_under_the_planner_rule(layer, nslots):
    stages = layer * 4 + [(211, 4)]
    nbars, ok = plan_nbars(nslots, stages, 15)
    if not ok:
        pytest.skip("the planner rejects this ring")
    rng = random.Random(nslots * 1000 + len(layer))
    for _ in range(30):
        assert simulate(stages, nslots, nbars, 15, rng) == 0


def test_waits_alias_when_barriers_equal_slots():
    """With one full barrier per slot (the rule broken for one-item chunks),
    some wait passes on the previous cycle's phase."""
    stages = NARROW * 6
    rng = random.Random(7)
    total = sum(simulate(stages, 4, 4, 15, rng) for _ in range(40))
    assert total > 0


def test_model_has_no_false_alarms_in_lockstep():
    """One warp, one item per chunk: every wait is on the chunk it wants."""
    rng = random.Random(3)
    assert simulate([(50, 1)], 4, 4, 1, rng) == 0
