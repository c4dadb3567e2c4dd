"""Host model of the persistent fusion's synchronisation (fuse_v_tcp_kernel, csrc/fuse_tc.cu).

compute-sanitizer is not available for these kernels, so the CTA pair's barrier
protocol is checked here instead, as a model: each role of the kernel (loader,
kept-row relay, MMA issuer, softmax warps, epilogue warps) is a coroutine that
performs the kernel's waits and arrivals in the kernel's order; the tensor pipe
completes the issuer's MMA batches in issue order, each batch's commit arriving
on its barriers; TMA copies land in any order; a random scheduler interleaves
everything.  For units of 0 to 9 dropped tiles (a unit with none still runs
every handshake) and many schedules, the model checks that

* the run ends (no deadlock) and no waiter ever finds its barrier two phases
  ahead of the phase it waits for (a parity wait would then be ambiguous);
* every buffer is written only after its last reader is done, and read only
  after its writer: O[k % 2] (first O product of unit k after the epilogue of
  unit k - 2 read it), S[t % 2] (S(t) after the softmax read S(t - 2) and O(t - 2)
  read P(t - 2)), the ring stage of tile t (its copy after S(t - 3) and O(t - 3)),
  vk[k % 2] (unit k's kept rows after unit k - 2's S products and epilogue), the
  row sums lsum[k % 2], and the rare rescale of O by the softmax (after O(t - 1),
  before O(t)).

Planted mistakes in the model (a missing wait) must be caught.  One wait is
found redundant: the issuer's wait for the epilogue to free O before a unit's
first O product is implied by the loader's wait for it to free the kept rows
(the epilogue frees both at once, and the unit's first O needs its kept rows),
so dropping it breaks nothing; the kernel keeps it.  The model has no
arithmetic; it is the protocol the kernel's comments state, written out.
"""
import random

import pytest

STAGES = 3          # dropped-tile ring


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


def run(units, seed, mistake=None, rescale_p=0.2):
    """One schedule of the pair over `units` (dropped tiles per unit); returns 'ok'
    or raises ProtocolError.  `mistake` removes one wait from the model."""
    rnd = random.Random(seed)
    bars = {}

    def bar(name, count=1):
        bars.setdefault(name, Bar(count))
        return bars[name]

    for b in range(2):
        bar(("vk_full", b)); bar(("vk_pair", b)); bar(("vk_empty", b))
        bar(("s_full", b)); bar(("p_full", b)); bar(("o_full", b)); bar(("o_empty", b))
        bar(("lsum_full", b)); bar(("lsum_empty", b))
    for i in range(STAGES):
        bar(("vd_full", i)); bar(("vd_empty", i))

    # global tile index of unit k's first tile
    first = [0]
    for nt in units:
        first.append(first[-1] + nt)
    unit_of = {}
    for k, nt in enumerate(units):
        for j in range(nt):
            unit_of[first[k] + j] = k

    now = [0]
    ev = {}                  # event name -> time it happened

    def at(name):
        ev[name] = now[0]

    def done(name):
        return name in ev

    def need(cond, what):
        if not cond:
            raise ProtocolError(what)

    pipe = []                # MMA batches in issue order: (kind, t or k, barriers to arrive)
    copies = []              # copies in flight: (kind, index)

    def wait(name, phase):   # phase: 0-based completion the waiter needs (-1: none)
        return name, phase

    # ---- roles, in the kernel's order
    def loader():
        t = 0
        for k, nt in enumerate(units):
            b = k & 1
            if mistake != "vk_empty":
                yield wait(("vk_empty", b), (k >> 1) - 1)
            copies.append(("vk", k))
            for _ in range(nt):
                st = t % STAGES
                if mistake != "loader_ring":
                    yield wait(("vd_empty", st), t // STAGES - 1)
                copies.append(("vd", t))
                t += 1

    def relay():
        for k in range(len(units)):
            yield wait(("vk_full", k & 1), k >> 1)
            bars[("vk_pair", k & 1)].arrive()

    def issuer():
        pend = None

        def issue_o(q):
            t, k, is_first, is_last = q
            b = k & 1
            if is_first and mistake != "o_empty":
                yield wait(("o_empty", b), (k >> 1) - 1)
            if mistake != "p_full":
                yield wait(("p_full", t & 1), t >> 1)
            arr = [("vd_empty", t % STAGES)] + ([("o_full", b)] if is_last else [])
            pipe.append(("O", t, arr))

        t = 0
        for k, nt in enumerate(units):
            b = k & 1
            yield wait(("vk_pair", b), k >> 1)
            if nt == 0:
                if pend is not None:
                    yield from issue_o(pend)
                    pend = None
                yield wait(("o_empty", b), (k >> 1) - 1)
                pipe.append(("Onone", k, [("o_full", b)]))
                continue
            for j in range(nt):
                yield wait(("vd_full", t % STAGES), t // STAGES)
                pipe.append(("S", t, [("s_full", t & 1)]))
                if pend is not None:
                    yield from issue_o(pend)
                pend = (t, k, j == 0, j == nt - 1)
                t += 1
        if pend is not None:
            yield from issue_o(pend)

    def softmax():
        t = 0
        for k, nt in enumerate(units):
            b = k & 1
            for j in range(nt):
                if mistake != "s_full":
                    yield wait(("s_full", t & 1), t >> 1)
                need(done(("S", t)), "softmax reads S(%d) before it is written" % t)
                at(("smx_read", t))
                if j > 0 and rnd.random() < rescale_p:
                    # rescale O[b] once O(t - 1) is done (its commit frees its stage)
                    if mistake != "rescale":
                        yield wait(("vd_empty", (t - 1) % STAGES), (t - 1) // STAGES)
                    need(done(("O", t - 1)), "rescale of O before O(%d) is done" % (t - 1))
                    at(("rescale", t))
                at(("P", t))
                bars[("p_full", t & 1)].arrive()
                t += 1
            if mistake != "lsum_empty":
                yield wait(("lsum_empty", b), (k >> 1) - 1)
            need(k < 2 or done(("epi_lsum", k - 2)), "row sums of unit %d over unread ones" % k)
            at(("lsum", k))
            bars[("lsum_full", b)].arrive()

    def epilogue():
        for k in range(len(units)):
            b = k & 1
            yield wait(("vk_full", b), k >> 1)
            yield wait(("lsum_full", b), k >> 1)
            if mistake != "o_full":
                yield wait(("o_full", b), k >> 1)
            need(done(("lsum", k)), "epilogue reads unit %d's row sums early" % k)
            need(units[k] == 0 or done(("O", first[k] + units[k] - 1)),
                 "epilogue reads O of unit %d before its last product" % k)
            at(("epi_lsum", k))
            bars[("lsum_empty", b)].arrive()
            at(("epi_O", k))
            bars[("o_empty", b)].arrive()
            at(("epi_vk", k))
            bars[("vk_empty", b)].arrive()

    # ---- the tensor pipe and the copies
    def execute(kind, idx, arr):
        if kind == "S":
            t = idx
            k = unit_of[t]
            need(done(("vd", t)), "S(%d) reads a stage before its copy landed" % t)
            need(done(("vk", k)), "S(%d) reads kept rows before they landed" % t)
            if t >= 2:
                need(done(("smx_read", t - 2)), "S(%d) overwrites S(%d) before the softmax read it" % (t, t - 2))
                need(done(("O", t - 2)), "S(%d) overwrites P(%d) before O read it" % (t, t - 2))
        elif kind == "O":
            t = idx
            k = unit_of[t]
            need(done(("P", t)), "O(%d) reads P before the softmax wrote it" % t)
            need(done(("vd", t)), "O(%d) reads a stage before its copy landed" % t)
            if t == first[k] and k >= 2:
                need(done(("epi_O", k - 2)), "first O of unit %d overwrites O[%d] before the epilogue read it"
                     % (k, k & 1))
        else:  # Onone: unit idx has no dropped rows
            k = idx
            if k >= 2:
                need(done(("epi_O", k - 2)), "O[%d] handshake of unit %d before the epilogue read it" % (k & 1, k))
        at((kind if kind != "Onone" else "Onone", idx))
        for a in arr:
            bars[a].arrive()

    def land(kind, idx):
        if kind == "vk":
            k = idx
            if k >= 2:
                need(done(("epi_vk", k - 2)), "kept rows of unit %d land before the epilogue of unit %d read vk"
                     % (k, k - 2))
                prev = units[k - 2]
                if prev:
                    need(done(("S", first[k - 2] + prev - 1)),
                         "kept rows of unit %d land before unit %d's S products" % (k, k - 2))
            at(("vk", k))
            bars[("vk_full", k & 1)].arrive()
        else:
            t = idx
            if t >= STAGES:
                need(done(("S", t - STAGES)) and done(("O", t - STAGES)),
                     "tile %d lands in the stage of tile %d while it is read" % (t, t - STAGES))
            at(("vd", t))
            bars[("vd_full", t % STAGES)].arrive()

    roles = {"loader": loader(), "relay": relay(), "issuer": issuer(), "softmax": softmax(),
             "epilogue": epilogue()}
    waiting = {r: None for r in roles}
    finished = set()
    for _ in range(10 ** 6):
        now[0] += 1
        ready = []
        for r in roles:
            if r in finished:
                continue
            w = waiting[r]
            if w is None:
                ready.append(r)
                continue
            name, phase = w
            got = bars[name].done
            if phase < 0 or got >= phase + 1:
                if phase >= 0 and got >= phase + 2:
                    raise ProtocolError("%s fell two phases behind on %s" % (r, name))
                ready.append(r)
        if pipe:
            ready.append("pipe")
        if copies:
            ready.append("copy")
        if not ready:
            if len(finished) == len(roles):
                return "ok"
            raise ProtocolError("deadlock: " + ", ".join(
                "%s waits %s" % (r, waiting[r]) for r in roles if r not in finished))
        r = rnd.choice(ready)
        if r == "pipe":
            execute(*pipe.pop(0))
        elif r == "copy":
            land(*copies.pop(rnd.randrange(len(copies))))
        else:
            try:
                waiting[r] = next(roles[r])
            except StopIteration:
                waiting[r] = None
                finished.add(r)
    raise ProtocolError("no end")


def _unit_lists(n, seed):
    rnd = random.Random(seed)
    for _ in range(n):
        yield [rnd.choice([0, 0, 1, 1, 2, 3, 4, 6, 9]) for _ in range(rnd.randint(1, 8))]


def test_protocol_ends_and_orders_every_access():
    runs = 0
    for i, units in enumerate(_unit_lists(400, 2608)):
        for seed in range(3):
            assert run(units, 1000 * i + seed) == "ok", units
            runs += 1
    assert runs == 1200


@pytest.mark.parametrize("mistake", ["p_full", "s_full", "o_full", "vk_empty", "loader_ring", "rescale",
                                     "lsum_empty"])
def test_planted_protocol_mistakes_are_caught(mistake):
    caught = 0
    for i, units in enumerate(_unit_lists(300, 99)):
        try:
            run(units, i, mistake=mistake, rescale_p=0.5)
        except ProtocolError:
            caught += 1
    assert caught > 0, mistake


def test_o_empty_wait_is_implied_by_the_kept_rows():
    for i, units in enumerate(_unit_lists(200, 7)):
        assert run(units, i, mistake="o_empty", rescale_p=0.5) == "ok", units
