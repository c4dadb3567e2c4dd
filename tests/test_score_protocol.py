"""Host models of the two tensor-core score passes' synchronisation
(score_lse_tc_kernel and score_colsum_tc_kernel, csrc/score_tc.cu).

As for the fusion (test_fusion_protocol.py): each role of a CTA pair is a
coroutine doing the kernel's waits and arrivals in the kernel's order, the
tensor pipe completes MMAs in issue order with their commits, copies land in
any order, and a random scheduler interleaves them.  Every run must end, no
waiter may find its barrier two phases ahead, and every buffer must be written
only after its readers are done and read only after its writer:

* pass 1 (row log-sum-exp): the key ring (4 stages), the two tensor-memory
  slots (tile i in slot i % 2, drained by warpgroup i % 2), the query rows;
* pass 2 (column sums): the key double buffer (one per layer), the window-row
  ring with its row normalisers (4 stages, freed by the MMA and by the
  warpgroup that read the normalisers), the two tensor-memory slots (chunk q
  in slot q % 2, drained by warpgroup q % 2), and the warpgroups' per-layer
  exchange of column sums in the per-layer ranking mode.

Planted mistakes (a missing wait) must be caught.  No arithmetic is modelled.
"""
import random

import pytest


class Bar:
    def __init__(self, count):
        self.count, self.pending, self.done = count, 0, 0

    def arrive(self, n=1):
        self.pending += n
        while self.pending >= self.count:
            self.pending -= self.count
            self.done += 1


class ProtocolError(AssertionError):
    pass


class Engine:
    """Barriers, an in-order MMA pipe, unordered copies, events and a random scheduler."""

    def __init__(self, seed):
        self.rnd = random.Random(seed)
        self.bars = {}
        self.pipe = []
        self.copies = []
        self.ev = set()

    def bar(self, name, count=1):
        self.bars.setdefault(name, Bar(count))

    def at(self, name):
        self.ev.add(name)

    def done(self, name):
        return name in self.ev

    @staticmethod
    def need(cond, what):
        if not cond:
            raise ProtocolError(what)

    def run(self, roles, execute, land):
        waiting = {r: None for r in roles}
        finished = set()
        for _ in range(10 ** 6):
            ready = []
            for r in roles:
                if r in finished:
                    continue
                w = waiting[r]
                if w is None:
                    ready.append(r)
                    continue
                name, phase = w
                got = self.bars[name].done
                if phase < 0 or got >= phase + 1:
                    if phase >= 0 and got >= phase + 2:
                        raise ProtocolError("%s fell two phases behind on %s" % (r, name))
                    ready.append(r)
            if self.pipe:
                ready.append("pipe")
            if self.copies:
                ready.append("copy")
            if not ready:
                if len(finished) == len(roles):
                    return "ok"
                raise ProtocolError("deadlock: " + ", ".join(
                    "%s waits %s" % (r, waiting[r]) for r in roles if r not in finished))
            r = self.rnd.choice(ready)
            if r == "pipe":
                item = self.pipe.pop(0)
                execute(*item[:-1])
                for a in item[-1]:
                    self.bars[a].arrive()
            elif r == "copy":
                item = self.copies.pop(self.rnd.randrange(len(self.copies)))
                land(*item[:-1])
                for a in item[-1]:
                    self.bars[a].arrive()
            else:
                try:
                    waiting[r] = next(roles[r])
                except StopIteration:
                    waiting[r] = None
                    finished.add(r)
        raise ProtocolError("no end")


def run_pass1(ntiles, seed, mistake=None):
    """One CTA pair of the row log-sum-exp pass over `ntiles` key tiles."""
    E = Engine(seed)
    S = 4                                          # key ring stages
    E.bar("q_full")
    for i in range(S):
        E.bar(("k_full", i)); E.bar(("k_empty", i))
    for i in range(2):
        E.bar(("tm_full", i)); E.bar(("tm_empty", i))

    def producer():
        E.copies.append(("q", 0, ["q_full"]))
        for i in range(ntiles):
            st = i % S
            if mistake != "k_empty":
                yield ("k_empty", st), i // S - 1
            E.copies.append(("k", i, [("k_full", st)]))

    def mma():
        yield "q_full", 0
        for i in range(ntiles):
            yield ("k_full", i % S), i // S
            if mistake != "tm_empty":
                yield ("tm_empty", i & 1), (i >> 1) - 1
            E.pipe.append(("mma", i, [("tm_full", i & 1), ("k_empty", i % S)]))

    def consumer(wg):
        def role():
            for i in range(wg, ntiles, 2):
                if mistake != "tm_full":
                    yield ("tm_full", wg), i >> 1
                E.need(E.done(("mma", i)), "warpgroup %d reads tile %d before its MMA" % (wg, i))
                E.at(("read", i))
                E.bars[("tm_empty", wg)].arrive()
        return role()

    def execute(kind, i):
        E.need(E.done(("q", 0)), "MMA %d before the query rows landed" % i)
        E.need(E.done(("k", i)), "MMA %d before its key tile landed" % i)
        if i >= 2:
            E.need(E.done(("read", i - 2)), "MMA %d overwrites slot %d before tile %d was read" % (i, i & 1, i - 2))
        E.at(("mma", i))

    def land(kind, i):
        if kind == "k" and i >= S:
            E.need(E.done(("mma", i - S)), "key tile %d lands in the stage tile %d is read from" % (i, i - S))
        E.at((kind, i))

    return E.run({"producer": producer(), "mma": mma(), "wg0": consumer(0), "wg1": consumer(1)}, execute, land)


def run_pass2(L, C, seed, per_layer=False, mistake=None):
    """One CTA pair of the column-sum pass over L layers of C row chunks each."""
    E = Engine(seed)
    QS = 4                                         # window-row ring stages
    for i in range(2):
        E.bar(("k_full", i)); E.bar(("k_empty", i)); E.bar(("tm_full", i)); E.bar(("tm_empty", i))
    for i in range(QS):
        E.bar(("q_full", i)); E.bar(("nl_full", i)); E.bar(("q_empty", i), 2)   # MMA commit + warpgroup
    E.bar("red", 2)                                # the two warpgroups meet (named barrier)

    def producer():
        for l in range(L):
            ks = l & 1
            if mistake != "k_empty":
                yield ("k_empty", ks), (l >> 1) - 1
            E.copies.append(("k", l, [("k_full", ks)]))
            for c in range(C):
                q = l * C + c
                qs = q % QS
                if mistake != "q_empty":
                    yield ("q_empty", qs), q // QS - 1
                E.copies.append(("q", q, [("q_full", qs)]))
                E.copies.append(("nl", q, [("nl_full", qs)]))

    def mma():
        for l in range(L):
            ks = l & 1
            yield ("k_full", ks), l >> 1
            for c in range(C):
                q = l * C + c
                yield ("q_full", q % QS), q // QS
                if mistake != "tm_empty":
                    yield ("tm_empty", q & 1), (q >> 1) - 1
                E.pipe.append(("mma", q, [("tm_full", q & 1), ("q_empty", q % QS)]))
            E.pipe.append(("layer", l, [("k_empty", ks)]))

    red_round = [0, 0]

    def consumer(wg):
        def role():
            for l in range(L):
                for c in range(C):
                    q = l * C + c
                    if q & 1 != wg:
                        continue
                    if mistake != "tm_full":
                        yield ("tm_full", wg), q >> 1
                    if mistake != "nl_full":
                        yield ("nl_full", q % QS), q // QS
                    E.need(E.done(("mma", q)), "warpgroup %d reads chunk %d before its MMA" % (wg, q))
                    E.need(E.done(("nl", q)), "warpgroup %d reads chunk %d's normalisers early" % (wg, q))
                    E.at(("read", q))
                    E.bars[("tm_empty", wg)].arrive()
                    E.at(("nl_read", q))
                    E.bars[("q_empty", q % QS)].arrive()
                if per_layer:
                    # both warpgroups' column sums of layer l meet in shared memory
                    n = red_round[wg]
                    red_round[wg] += 1
                    E.bars["red"].arrive()
                    yield "red", n
        return role()

    def execute(kind, i):
        if kind == "mma":
            q = i
            l = q // C
            E.need(E.done(("k", l)), "MMA of chunk %d before layer %d's keys landed" % (q, l))
            E.need(E.done(("q", q)), "MMA of chunk %d before its rows landed" % q)
            if q >= 2:
                E.need(E.done(("read", q - 2)), "MMA %d overwrites slot %d before chunk %d was read"
                       % (q, q & 1, q - 2))
        E.at((kind, i))

    def land(kind, i):
        if kind == "k" and i >= 2:
            E.need(E.done(("layer", i - 2)), "keys of layer %d land over layer %d's before its MMAs" % (i, i - 2))
        if kind in ("q", "nl") and i >= QS:
            E.need(E.done(("mma", i - QS)), "rows of chunk %d land in the stage chunk %d is read from" % (i, i - QS))
            E.need(E.done(("nl_read", i - QS)),
                   "normalisers of chunk %d land before chunk %d's were read" % (i, i - QS))
        E.at((kind, i))

    return E.run({"producer": producer(), "mma": mma(), "wg0": consumer(0), "wg1": consumer(1)}, execute, land)


def test_pass1_protocol():
    for n in list(range(0, 12)) + [49, 128]:
        for seed in range(40):
            assert run_pass1(n, 100 * n + seed) == "ok", n


@pytest.mark.parametrize("per_layer", [False, True])
def test_pass2_protocol(per_layer):
    for L in (1, 2, 3, 5, 28):
        for C in (1, 2, 3, 4):
            for seed in range(8):
                assert run_pass2(L, C, 1000 * L + 10 * C + seed, per_layer) == "ok", (L, C)


@pytest.mark.parametrize("mistake", ["k_empty", "tm_empty", "tm_full"])
def test_pass1_planted_mistakes_are_caught(mistake):
    caught = 0
    for seed in range(200):
        try:
            run_pass1(9, seed, mistake)
        except ProtocolError:
            caught += 1
    assert caught > 0


@pytest.mark.parametrize("mistake", ["k_empty", "q_empty", "tm_empty", "tm_full", "nl_full"])
def test_pass2_planted_mistakes_are_caught(mistake):
    caught = 0
    for seed in range(200):
        try:
            run_pass2(5, 2, seed, mistake=mistake)
        except ProtocolError:
            caught += 1
    assert caught > 0
