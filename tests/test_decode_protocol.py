"""The split-KV decode kernel's K/V ring protocol, modelled on the CPU.

fav_decode_kernel streams a split's key tiles through a ring of shared-memory stages: the K
producer and the V producer (one issuing lane each) arm the stage's full barrier (count 2, one
expect_tx each) once the stage's previous tile has been released, and consumer warp
lt % kConsumers takes tile lt from stage lt % kStages, waits for its full phase lt / kStages and
releases the stage with one arrival on its empty barrier.  The ring is sound only because every
stage is owned by a single consumer warp (kStages a multiple of kConsumers): a warp that reached
a stage whose previous tile belonged to another warp could find the barrier a phase behind and
pass its parity wait on the old phase.  Every parity wait here must pass exactly when the phase
it stands for has completed, and no role may be left waiting.
"""
import random

import pytest

CONSUMERS = 6
STAGES = 12
TILE_BYTES = 32 * 128 * 2      # one K (or V) tile of 32 keys at D = 128, fp16


class Bar:
    def __init__(self, name, count):
        self.name, self.count, self.pending, self.tx, self.phase = name, count, count, 0, 0

    def _complete(self):
        if self.pending == 0 and self.tx == 0:
            self.phase += 1
            self.pending = self.count

    def arrive(self):
        self.pending -= 1
        assert self.pending >= 0, "%s: more arrivals than its count in phase %d" % (self.name, self.phase)
        self._complete()

    def expect_tx(self, nbytes):
        self.tx += nbytes
        self.arrive()

    def complete_tx(self, nbytes):
        self.tx -= nbytes
        assert self.tx >= 0, "%s: more bytes than expected in phase %d" % (self.name, self.phase)
        self._complete()

    def passed(self, parity):
        return (self.phase & 1) != parity


def simulate(n_tiles, rng, consumers=CONSUMERS, stages=STAGES):
    """Runs one block's split of n_tiles key tiles; returns the roles left waiting."""
    bars = {}
    for s in range(stages):
        bars["full%d" % s] = Bar("full%d" % s, 2)
        bars["empty%d" % s] = Bar("empty%d" % s, 1)
    events, now, seq = [], [0.0], [0]

    def at(t, fn):
        seq[0] += 1
        events.append((t, seq[0], fn))

    def producer():
        for lt in range(n_tiles):
            st = lt % stages
            if lt >= stages:
                yield ("wait", "empty%d" % st, lt // stages - 1)
            bars["full%d" % st].expect_tx(TILE_BYTES)
            at(now[0] + rng.uniform(0.5, 8.0), lambda st=st: bars["full%d" % st].complete_tx(TILE_BYTES))
            yield None

    def consumer(w):
        for lt in range(w, n_tiles, consumers):
            st = lt % stages
            yield ("wait", "full%d" % st, lt // stages)
            yield None                                   # the tile's scores and P.V
            bars["empty%d" % st].arrive()

    procs = {"k_producer": producer(), "v_producer": producer()}
    procs.update({"consumer%d" % w: consumer(w) for w in range(consumers)})
    waiting = dict.fromkeys(procs)
    done = set()

    def ready(p):
        w = waiting[p]
        return w is None or bars[w[1]].passed(w[2] & 1)

    while True:
        runnable = [p for p in procs if p not in done and ready(p)]
        if runnable:
            p = rng.choice(runnable)
            w = waiting[p]
            if w is not None:
                assert bars[w[1]].phase == w[2] + 1, "%s passed %s for phase %d at phase %d" % (
                    p, w[1], w[2], bars[w[1]].phase)
            try:
                waiting[p] = next(procs[p])
            except StopIteration:
                done.add(p)
        elif events:
            events.sort()
            now[0], _, fn = events.pop(0)
            fn()
        else:
            return {p: waiting[p] for p in procs if p not in done}


@pytest.mark.parametrize("n_tiles", [0, 1, 5, 6, 7, 11, 12, 13, 24, 25, 64, 97])
def test_decode_ring_never_stalls(n_tiles):
    for trial in range(8):
        stuck = simulate(n_tiles, random.Random(100 * n_tiles + trial))
        assert not stuck, (n_tiles, stuck)


def test_decode_ring_random_splits():
    rng = random.Random(7)
    for _ in range(60):
        n = rng.randint(0, 200)
        stuck = simulate(n, random.Random(rng.random()))
        assert not stuck, (n, stuck)


def test_decode_ring_needs_stages_owned_by_one_warp():
    """With a stage count that is not a multiple of the consumer warps (8 stages, 6 warps), a warp
    can reach a stage before the previous tile of that stage has landed and pass its parity wait
    on the older phase; the exact-phase check catches that."""
    caught = 0
    for trial in range(40):
        try:
            simulate(64, random.Random(trial), stages=8)
        except AssertionError as e:
            caught += "passed" in str(e)
    assert caught > 0
