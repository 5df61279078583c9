"""The D = 128 prefill kernel's barrier protocol, modelled on the CPU.

Every role of fav_prefill_split_kernel (the Q/K and V producers, the MMA warp with its scores two
key tiles ahead of the P.V products, eight softmax warps, four epilogue warps, the O store warp) is
a process that waits on and arrives at mbarriers exactly as the kernel source does: the same
per-CTA unit lists (snake order, heaviest query tile first), the same stage indices and phase
parities, arrival counts, expected transaction bytes and tcgen05 commits.  TMA copies and MMA
bursts complete after random delays and the processes run in random order.  A run must finish
with no process left waiting and no barrier receiving more arrivals than its count in a phase
(also in the packed-batch variant: O rows written by the epilogue, Q buffers released by the last
S, back-pressure on the (m, l) exchange slots, whose removal the model catches);
every parity wait must pass exactly when the phase it stands for has completed (not before it,
and not after a later phase of the same barrier); a deliberately wrong parity must be caught.  (The GPU tests check the results; this checks
the orderings that a GPU run only samples.)
"""
import random

import pytest

BM = BN = 128
KS = VS = 2
QB = KVB = 128 * 128 * 2


class Bar:
    """mbarrier: arrival count, transaction bytes, phase number; a wait on parity p passes while
    the current phase's parity differs from p."""

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


def units_of(B, Hq, Nq, Nkv, P, c, causal=True):
    """The units of CTA c of P: one 128-row query tile each, {t, key tiles}."""
    n_qtiles = (Nq + BM - 1) // BM
    BH = B * Hq
    out, k = [], 0
    while True:
        u = k * P + ((P - 1 - c) if k & 1 else c)
        if u >= n_qtiles * BH:
            return out
        t = n_qtiles - 1 - u // BH
        kv_end = min(Nkv, t * BM + BM + Nkv - Nq) if causal else Nkv
        out.append({"t": t, "n_kv": (kv_end + BN - 1) // BN})
        k += 1


def simulate(units, rng, mistake=None, packed=False):
    """packed: the packed-batch variant (the epilogue writes O rows itself, so a Q buffer is
    released by its unit's last S alone, and the (m, l) exchange slot k % 2 has a back-pressure
    barrier: the softmax waits for the epilogue to have read unit k - 2's slot)."""
    bars = {}
    for name, count in [("q_full", 1), ("q_empty", 1 if packed else 2), ("o_staged", 128),
                        ("xch_bar", 256), ("xch_free", 128), ("s_full", 1), ("p_full", 8)]:
        for i in range(2):
            bars["%s%d" % (name, i)] = Bar("%s%d" % (name, i), count)
    for i in range(KS):
        bars["k_full%d" % i] = Bar("k_full%d" % i, 1)
        bars["k_empty%d" % i] = Bar("k_empty%d" % i, 1)
    for i in range(VS):
        bars["v_full%d" % i] = Bar("v_full%d" % i, 1)
        bars["v_empty%d" % i] = Bar("v_empty%d" % i, 1)
    for name, count in [("pv_done", 1), ("o_done", 1), ("o_free", 128)]:
        bars[name] = Bar(name, count)
    events, now, pipe_free, seq = [], [0.0], [0.0], [0]

    def at(t, fn):
        seq[0] += 1
        events.append((t, seq[0], fn))

    def tma(bar, nbytes):                      # a TMA copy: its bytes land later
        at(now[0] + rng.uniform(0.2, 5.0), lambda: bars[bar].complete_tx(nbytes))

    def mma(commits):                          # an MMA burst: in order, then its commits arrive
        pipe_free[0] = max(now[0], pipe_free[0]) + rng.uniform(0.5, 1.5)
        at(pipe_free[0], lambda: [bars[c].arrive() for c in commits])

    n = len(units)
    # prologue (the Q/K producer lane, before the block-wide barrier)
    bars["q_full0"].expect_tx(QB)
    tma("q_full0", QB)
    for g in range(min(KS, units[0]["n_kv"])):
        bars["k_full%d" % g].expect_tx(KVB)
        tma("k_full%d" % g, KVB)

    def k_producer():
        g, early = 0, min(KS, units[0]["n_kv"])
        for k, U in enumerate(units):
            if k >= 2:
                yield ("wait", "q_empty%d" % (k & 1), (k >> 1) - 1)
            if k > 0:
                bars["q_full%d" % (k & 1)].expect_tx(QB)
                tma("q_full%d" % (k & 1), QB)
            for _ in range(U["n_kv"]):
                st = g % KS
                if g >= early:
                    if g >= KS:
                        yield ("wait", "k_empty%d" % st, (g // KS) - 1)
                    bars["k_full%d" % st].expect_tx(KVB)
                    tma("k_full%d" % st, KVB)
                g += 1
                yield None

    def v_producer():
        g = 0
        for U in units:
            for _ in range(U["n_kv"]):
                st = g % VS
                if g >= VS:
                    yield ("wait", "v_empty%d" % st, (g // VS) - 1)
                bars["v_full%d" % st].expect_tx(KVB)
                tma("v_full%d" % st, KVB)
                g += 1
                yield None

    def mma_warp():
        s = {"ks": 0, "js": 0, "Gs": 0}

        def next_s_ready():
            if s["ks"] >= n:
                return
            if s["js"] == 0:
                yield ("wait", "q_full%d" % (s["ks"] & 1), s["ks"] >> 1,
                       (s["ks"] & 1) if mistake == "q_parity" else None)
            yield ("wait", "k_full%d" % (s["Gs"] % KS), s["Gs"] // KS)

        def issue_s():
            if s["ks"] >= n:
                return
            commits = ["s_full%d" % (s["Gs"] & 1), "k_empty%d" % (s["Gs"] % KS)]
            if s["js"] + 1 == units[s["ks"]]["n_kv"]:
                commits.append("q_empty%d" % (s["ks"] & 1))     # the unit's last S
            mma(commits)
            s["Gs"] += 1
            s["js"] += 1
            if s["js"] == units[s["ks"]]["n_kv"]:
                s["js"], s["ks"] = 0, s["ks"] + 1

        for _ in range(2):                     # S(0), S(1) before the loop
            yield from next_s_ready()
            issue_s()
        Gp = 0
        for k, U in enumerate(units):
            for j in range(U["n_kv"]):
                yield ("wait", "p_full%d" % (Gp & 1), Gp >> 1)
                yield ("wait", "v_full%d" % (Gp % VS), Gp // VS)
                if j == 0 and k > 0:
                    yield ("wait", "o_free", k - 1)
                commits = ["v_empty%d" % (Gp % VS), "pv_done"]
                if j + 1 == U["n_kv"]:
                    commits.append("o_done")
                mma(commits)
                yield from next_s_ready()      # then S(G + 2)
                issue_s()
                Gp += 1

    def softmax_warp():
        Gt = 0
        for k, U in enumerate(units):
            for j in range(U["n_kv"]):
                yield ("wait", "s_full%d" % (Gt & 1), Gt >> 1)
                if j > 0 and rng.random() < 0.3:           # lazy rescale of O
                    yield ("wait", "pv_done", Gt - 1)
                bars["p_full%d" % (Gt & 1)].arrive()
                Gt += 1
                yield None
            if packed and packed != "no_backpressure" and k >= 2:   # unit k - 2's (m, l) read
                yield ("wait", "xch_free%d" % (k & 1), (k >> 1) - 1)
            bars["xch_bar%d" % (k & 1)].arrive(32)
            yield None

    def epilogue_warp():
        for k in range(n):
            yield ("wait", "o_done", k)
            yield ("wait", "xch_bar%d" % (k & 1), k >> 1)
            if packed:                             # (m, l) read: the slot is free again
                bars["xch_free%d" % (k & 1)].arrive(32)
                yield None
            bars["o_free"].arrive(32)
            yield None
            if packed:                             # the O rows' stores to global memory take a while
                stored = [False]
                at(now[0] + rng.uniform(0.1, 4.0), lambda: stored.__setitem__(0, True))
                yield ("until", stored)
            if not packed:                         # O staged for the store warp's TMA store
                bars["o_staged%d" % (k & 1)].arrive(32)
                yield None

    def store_warp():
        if packed:                                 # the epilogue writes O itself
            return
            yield
        for k in range(n):
            yield ("wait", "o_staged%d" % (k & 1), k >> 1)
            read = [False]
            at(now[0] + rng.uniform(0.1, 2.0), lambda: read.__setitem__(0, True))
            yield ("until", read)
            bars["q_empty%d" % (k & 1)].arrive()

    procs = {"k_producer": k_producer(), "v_producer": v_producer(), "mma": mma_warp(),
             "store": store_warp()}
    procs.update({"softmax%d" % w: softmax_warp() for w in range(8)})
    procs.update({"epilogue%d" % w: epilogue_warp() for w in range(4)})
    waiting = dict.fromkeys(procs)
    done = set()

    def parity(w):                             # the kernel waits on idx % 2 (or a planted value)
        return w[3] if len(w) > 3 and w[3] is not None else w[2] & 1

    def ready(name):
        w = waiting[name]
        return (w is None or (w[0] == "wait" and bars[w[1]].passed(parity(w)))
                or (w[0] == "until" and w[1][0]))

    while True:
        runnable = [p for p in procs if p not in done and ready(p)]
        if runnable:
            p = rng.choice(runnable)
            w = waiting[p]
            if w is not None and w[0] == "wait":
                # the parity wait passed: the phase it stands for, and no later one, completed
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


SHAPES = [   # B, Hq, Nq, Nkv, grid
    (1, 8, 200, 200, 7), (1, 8, 200, 200, 3), (1, 8, 200, 200, 1), (1, 6, 300, 300, 5),
    (2, 4, 700, 700, 3), (1, 3, 257, 257, 2), (1, 2, 255, 1000, 1), (1, 32, 2048, 2048, 152),
]


@pytest.mark.parametrize("B,Hq,Nq,Nkv,P", SHAPES)
def test_protocol_never_stalls(B, Hq, Nq, Nkv, P):
    for c in range(0, P, max(1, P // 8)):
        units = units_of(B, Hq, Nq, Nkv, P, c)
        for trial in range(6):
            stuck = simulate(units, random.Random(1000 * trial + c))
            assert not stuck, "CTA %d of %d, units %s: %s" % (c, P, units, stuck)


def test_protocol_random_shapes_and_grids():
    """Random batch, head count, ragged lengths, causal or not, and grids from one block to one
    block per query tile."""
    rng = random.Random(2026)
    for _ in range(40):
        B, Hq = rng.randint(1, 3), rng.choice([1, 2, 3, 4, 8])
        Nq = rng.randint(1, 700)
        Nkv = Nq if rng.random() < 0.5 else rng.randint(Nq, 1200)
        causal = rng.random() < 0.7
        n_units = ((Nq + BM - 1) // BM) * B * Hq
        P = rng.randint(1, n_units)
        for c in rng.sample(range(P), min(P, 3)):
            units = units_of(B, Hq, Nq, Nkv, P, c, causal)
            stuck = simulate(units, random.Random(rng.random()))
            assert not stuck, ((B, Hq, Nq, Nkv, causal, P, c), stuck)


def test_planted_parity_mistake_is_caught():
    """The Q buffer's phase parity taken as ks % 2 instead of (ks / 2) % 2: in every run the MMA
    warp's wait for a unit's Q tile either passes before that tile has landed or, once it has,
    never passes."""
    units = units_of(1, 8, 200, 200, 3, 0)
    assert len(units) >= 3
    for trial in range(8):
        try:
            stuck = simulate(units, random.Random(trial), mistake="q_parity")
        except AssertionError as e:
            assert "passed q_full" in str(e)
        else:
            assert stuck and stuck["mma"][1].startswith("q_full")


@pytest.mark.parametrize("packed", [False, True])
def test_protocol_packed_batch_unit_mixes(packed):
    """A packed variable-length batch gives a block units of any key-tile count (sequences of
    different lengths, ragged last tiles) in the host's heaviest-first order; run with the dense
    kernel's O staging and with the packed variant's own protocol (direct O rows, Q buffer
    released by the last S, back-pressure on the (m, l) exchange slots)."""
    rng = random.Random(18656)
    for _ in range(60):
        units = [{"t": 0, "n_kv": rng.randint(1, 10)} for _ in range(rng.randint(1, 12))]
        units.sort(key=lambda U: -U["n_kv"])
        stuck = simulate(units, random.Random(rng.random()), packed=packed)
        assert not stuck, (units, stuck)


def test_packed_exchange_without_back_pressure_is_caught():
    """Planted in the model: the packed variant without the exchange slot's back-pressure wait
    lets the softmax complete a second phase of xch_bar (unit k + 2) before the epilogue has
    waited for the first (unit k): the epilogue then either passes a later phase (the exact-phase
    check) or never sees its phase (left waiting), on units of one key tile."""
    units = [{"t": 0, "n_kv": 1} for _ in range(8)]
    caught = 0
    for trial in range(40):
        try:
            stuck = simulate(units, random.Random(trial), packed="no_backpressure")
        except AssertionError as e:
            caught += "xch_bar" in str(e) or "more arrivals" in str(e)
        else:
            caught += any(w and w[0] == "wait" and w[1].startswith("xch_bar") for w in stuck.values())
    assert caught > 0
