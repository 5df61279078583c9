"""The D = 64 two-tile prefill kernel's barrier protocol, modelled on the CPU.

fav_prefill_pair_kernel's roles as processes that wait on and arrive at mbarriers exactly as the
source does: the TMA producer (both Q tiles of a unit once the previous unit's last S has
completed; K and V through a three-stage ring with per-stage empty barriers), the MMA warp
(S_i(j+1) as soon as tile i's softmax has read S_i(j), tile 1's first S after tile 0's softmax
has read its first scores, P_i(j).V once P_i(j) is stored, the last tile's commits releasing
K and V stages, one Q release per unit) and the two four-warp softmax groups with their
epilogues.  Units pair tile t of two heads of an even GQA group, or tiles 2p and 2p+1 of one
head (the second possibly beyond the sequence).  Every parity wait must pass exactly when the
phase it stands for has completed, and no process may be left waiting.
"""
import random

import pytest

BM = BN = 128
S = 3                      # K/V ring stages
QB = KVB = 128 * 64 * 2


class Bar:
    def __init__(self, name, count):
        self.name, self.count, self.pending, self.tx, self.phase = name, count, count, 0, 0

    def _complete(self):
        if self.pending == 0 and self.tx == 0:
            self.phase += 1
            self.pending = self.count

    def arrive(self, n=1):
        self.pending -= n
        assert self.pending >= 0, "%s: more arrivals than its count in phase %d" % (self.name, self.phase)
        self._complete()

    def expect_tx(self, nbytes):
        self.tx += nbytes
        self.arrive()

    def complete_tx(self, nbytes):
        self.tx -= nbytes
        self._complete()

    def passed(self, parity):
        return (self.phase & 1) != parity


def units_of(B, Hq, Hkv, Nq, Nkv, P, c, causal=True):
    n_qtiles = (Nq + BM - 1) // BM
    G = Hq // Hkv
    pair_heads = G % 2 == 0
    n_units = n_qtiles * B * (Hq // 2) if pair_heads else ((n_qtiles + 1) // 2) * B * Hq
    out, k = [], 0
    while True:
        u = k * P + ((P - 1 - c) if k & 1 else c)
        if u >= n_units:
            return out
        if pair_heads:
            t0 = t1 = n_qtiles - 1 - u // (B * (Hq // 2))
        else:
            pr = (n_qtiles + 1) // 2 - 1 - u // (B * Hq)
            t0, t1 = 2 * pr, 2 * pr + 1
        tiles = []
        for t in (t0, t1):
            if t >= n_qtiles:
                tiles.append(0)
            else:
                kv_end = min(Nkv, t * BM + BM + Nkv - Nq) if causal else Nkv
                tiles.append((kv_end + BN - 1) // BN)
        out.append(tiles)
        k += 1


def simulate(units, rng, mistake=None):
    bars = {}
    for name, count in [("q_full0", 1), ("q_full1", 1), ("q_empty", 1), ("s_full0", 1), ("s_full1", 1),
                        ("p_full0", 4), ("p_full1", 4), ("o_done0", 1), ("o_done1", 1),
                        ("s_free0", 4), ("s_free1", 4), ("p_free0", 1), ("p_free1", 1)]:
        bars[name] = Bar(name, count)
    for s in range(S):
        for name in ("k_full", "k_empty", "v_full", "v_empty"):
            bars["%s%d" % (name, s)] = Bar("%s%d" % (name, s), 1)
    events, now, pipe_free, seq = [], [0.0], [0.0], [0]

    def at(t, fn):
        seq[0] += 1
        events.append((t, seq[0], fn))

    def tma(bar, nbytes):
        at(now[0] + rng.uniform(0.2, 5.0), lambda: bars[bar].complete_tx(nbytes))

    def mma(commits):
        pipe_free[0] = max(now[0], pipe_free[0]) + rng.uniform(0.3, 1.0)
        at(pipe_free[0], lambda: [bars[c].arrive() for c in commits if c])

    def producer():
        g = 0
        for k, U in enumerate(units):
            if k > 0:
                yield ("wait", "q_empty", k - 1)
            for i in range(2):
                bars["q_full%d" % i].expect_tx(QB)
                tma("q_full%d" % i, QB)
            for _ in range(max(U)):
                st = g % S
                if g >= S:
                    yield ("wait", "k_empty%d" % st, g // S - 1)
                bars["k_full%d" % st].expect_tx(KVB)
                tma("k_full%d" % st, KVB)
                if g >= S:
                    yield ("wait", "v_empty%d" % st, g // S - 1)
                bars["v_full%d" % st].expect_tx(KVB)
                tma("v_full%d" % st, KVB)
                g += 1
                yield None

    def mma_warp():
        g, np_, nsi = 0, [0, 0], [0, 0]
        for k, U in enumerate(units):
            n_kv = max(U)
            g0 = g
            last0 = 1 if U[1] > 0 else 0
            yield ("wait", "k_full%d" % (g0 % S), g0 // S)
            for i in range(2):
                # both Q tiles have landed (an unused one too: its barrier is re-armed by the next
                # unit's load once q_empty says the buffers are free)
                if not (mistake == "skip_unused_q" and U[i] == 0):
                    yield ("wait", "q_full%d" % i, k)
                if U[i] == 0:
                    continue
                if i == 1 and mistake != "no_stagger":
                    yield ("wait", "s_free0", nsi[0] - 1)
                if nsi[i] > 0:
                    yield ("wait", "s_free%d" % i, nsi[i] - 1)
                mma(["s_full%d" % i, "k_empty%d" % (g0 % S) if i == last0 else None])
                nsi[i] += 1
            if n_kv == 1:
                mma(["q_empty"])
            for j in range(n_kv):
                gj = g0 + j
                st, st1 = gj % S, (gj + 1) % S
                last1 = 1 if j + 1 < U[1] else 0
                last = 1 if j < U[1] else 0
                k_ok = v_ok = False
                for i in range(2):
                    if j + 1 < U[i]:
                        if not k_ok:
                            yield ("wait", "k_full%d" % st1, (gj + 1) // S)
                            k_ok = True
                        yield ("wait", "s_free%d" % i, nsi[i] - 1)
                        mma(["s_full%d" % i, "k_empty%d" % st1 if i == last1 else None])
                        nsi[i] += 1
                    if j < U[i]:
                        if not v_ok:
                            yield ("wait", "v_full%d" % st, gj // S)
                            v_ok = True
                        yield ("wait", "p_full%d" % i, np_[i])
                        np_[i] += 1
                        mma(["p_free%d" % i, "v_empty%d" % st if i == last else None])
                        if j + 1 == U[i]:
                            mma(["o_done%d" % i])
                if j + 2 == n_kv:
                    mma(["q_empty"])
            g += n_kv

    def softmax_warp(i):
        ns = no = npst = 0
        for U in units:
            for _ in range(U[i]):
                yield ("wait", "s_full%d" % i, ns)
                ns += 1
                bars["s_free%d" % i].arrive()
                if npst > 0:
                    yield ("wait", "p_free%d" % i, npst - 1)
                npst += 1
                bars["p_full%d" % i].arrive()
                yield None
            if U[i]:
                yield ("wait", "o_done%d" % i, no)
                no += 1

    procs = {"producer": producer(), "mma": mma_warp()}
    procs.update({"softmax%d_%d" % (i, w): softmax_warp(i) for i in range(2) for w in range(4)})
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


SHAPES = [   # B, Hq, Hkv, Nq, Nkv, grid
    (1, 8, 2, 200, 200, 7), (1, 6, 3, 520, 520, 2), (1, 4, 1, 520, 520, 1), (1, 2, 2, 300, 300, 3),
    (2, 8, 2, 260, 260, 5), (1, 3, 1, 129, 700, 1), (4, 32, 8, 1024, 1024, 152),
]


@pytest.mark.parametrize("B,Hq,Hkv,Nq,Nkv,P", SHAPES)
def test_pair_protocol_never_stalls(B, Hq, Hkv, Nq, Nkv, P):
    for c in range(0, P, max(1, P // 8)):
        units = units_of(B, Hq, Hkv, Nq, Nkv, P, c)
        for trial in range(6):
            stuck = simulate(units, random.Random(1000 * trial + c))
            assert not stuck, "CTA %d of %d, units %s: %s" % (c, P, units, stuck)


def test_pair_protocol_unused_q_tile_must_be_waited():
    """Without waiting for the Q copy of a pair's second tile when that tile lies beyond the
    sequence, the next unit can re-arm its barrier while the copy is still in flight (a second
    arrival in one phase)."""
    # 3 query tiles (the first pair is (2, 3), tile 3 beyond the sequence) and one K/V tile, so
    # q_empty is committed right after the first S
    units = units_of(1, 3, 1, 300, 64, 1, 0, causal=False)
    assert any(U[1] == 0 for U in units) and len(units) > 1
    caught = 0
    for trial in range(40):
        try:
            simulate(units, random.Random(trial), mistake="skip_unused_q")
        except AssertionError as e:
            caught += "q_full1" in str(e)
    assert caught > 0


def test_pair_protocol_random_shapes_and_grids():
    rng = random.Random(64)
    for _ in range(40):
        B, Hkv = rng.randint(1, 2), rng.choice([1, 2])
        Hq = Hkv * rng.choice([1, 2, 3, 4])
        Nq = rng.randint(1, 700)
        Nkv = Nq if rng.random() < 0.5 else rng.randint(Nq, 1200)
        causal = rng.random() < 0.7
        n_qtiles = (Nq + BM - 1) // BM
        n_units = n_qtiles * B * (Hq // 2) if (Hq // Hkv) % 2 == 0 else ((n_qtiles + 1) // 2) * B * Hq
        P = rng.randint(1, n_units)
        for c in rng.sample(range(P), min(P, 3)):
            units = units_of(B, Hq, Hkv, Nq, Nkv, P, c, causal)
            stuck = simulate(units, random.Random(rng.random()))
            assert not stuck, ((B, Hq, Hkv, Nq, Nkv, causal, P, c), stuck)


def test_pair_protocol_packed_batch_unit_orders():
    """A packed variable-length batch gives a block any mix of units: pairs of heads (equal key
    tiles), pairs of tiles of one sequence (the second with fewer or no key tiles), from short
    and long sequences in the host's heaviest-first order."""
    rng = random.Random(2608)
    for _ in range(60):
        units = []
        for _ in range(rng.randint(1, 12)):
            n0 = rng.randint(1, 9)
            kind = rng.random()
            n1 = n0 if kind < 0.4 else (0 if kind < 0.7 else rng.randint(1, n0 + 1))
            units.append([n0, n1])
        units.sort(key=lambda U: -max(U))
        stuck = simulate(units, random.Random(rng.random()))
        assert not stuck, (units, stuck)
