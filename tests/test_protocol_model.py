"""A host model of the tensor-core chain kernel's barrier protocol, run under random schedules.

compute-sanitizer is closed on this machine, so the synchronisation design of `tc_chain_kernel`
(csrc/tc_kernels.cu) is checked here as a model: the producer, the four MMA warps and the four
softmax warpgroups of one CTA follow the kernel's waits, arrivals and commits step for step,
while the asynchronous parts run at random times: TMA copies complete in any order, and each
MMA warp's products and commits complete in its issue order (`tcgen05.commit` arrives once every
product the thread issued before it is complete).

mbarrier waits are modelled as the hardware takes them, by phase parity: a wait for phase k of
a barrier that has completed P phases passes when P and k differ in parity. The model knows
which phase each wait means, and fails when P is not k or k + 1 at any look at the barrier (the
barrier ran two phases ahead of the waiter, or the waiter names a phase not yet begun), when the
agents stop with work left (deadlock), and when a product or a softmax read finds a buffer
holding the wrong data: a ring stage, an A buffer, a score tile or an O accumulator overwritten
before its last reader, or read before its writer completed.

Configurations are the kernel's: the decode (four token tiles per unit, every stream takes every
item, two A buffers; two O accumulators with the unit's last PV carried into the next unit's
first issue and its end run after that item, or one at D = 64) and the encode (units of one, two
or four route tiles, streams splitting items by token parity, one A buffer, 8 to 16 ring
stages). Each MMA warp waits on the full barrier of every ring item and on every unit's a_full,
in order, so each parity test names one phase; the producer frees each stage on behalf of the
streams that skip its item. a_free takes one arrival per stream, made when the stream sees its
last S of the unit; stream 0 also arrives for the streams with no item in the unit (short encode
chunks), which do not arrive themselves: arriving at once, such a stream could arrive for the
next unit too before a slower stream arrived for this one.

Assumption, shown by test_observer_lag_limit: an MMA warp keeps up with the barriers of the
items its stream skips, as a warp does on the GPU when all it does for such an item is wait; it
would have to fall a whole ring (8 to 16 items) or A-buffer cycle behind to find a barrier two
phases ahead. The scheduler lets a runnable warp move before a pending copy or product
completes nine times in ten (warps issue far faster than those complete), and the agents
slowed on purpose are the producer and the softmax warpgroups. Planted mistakes must be caught:
an A buffer freed at the unit's first S, a deferred end run before the next unit's first item,
a no-item stream arriving on a_free at once, and a ring of one stage.
"""
import random

import pytest

NS = 4  # TMEM streams


class ProtocolError(AssertionError):
    pass


class Barrier:
    def __init__(self, name, count):
        self.name, self.count, self.pending, self.phases = name, count, count, 0

    def arrive(self, n=1):
        self.pending -= n
        if self.pending < 0:
            raise ProtocolError(f"{self.name}: more arrivals than its count")
        if self.pending == 0:
            self.phases += 1
            self.pending = self.count

    def check(self, k, who):
        """Whether a wait for phase k passes now (k = -1: the phase before the first)."""
        p = self.phases
        if p != k and p != k + 1:
            raise ProtocolError(f"{who}: waits for phase {k} of {self.name}, which has "
                                f"completed {p} phases")
        return (p & 1) != (k & 1)


class Model:
    def __init__(self, units, n_items, stages, abufs, obufs, rng, plant=None, slow=None):
        self.U, self.units, self.n_items = len(units), units, n_items
        self.S, self.AB, self.OB = stages, abufs, obufs
        self.ahead = abufs - 1 if abufs > 1 else 1
        self.rng, self.plant, self.slow = rng, plant, slow  # slow: an agent run 1 step in 50
        self.full = [Barrier(f"full[{i}]", 1) for i in range(stages)]
        self.empty = [Barrier(f"empty[{i}]", NS) for i in range(stages)]
        self.afull = [Barrier(f"a_full[{b}]", 1) for b in range(abufs)]
        self.afree = [Barrier(f"a_free[{b}]", NS) for b in range(abufs)]
        self.sready = [Barrier(f"s_ready[{s}]", 1) for s in range(NS)]
        self.odone = [Barrier(f"o_done[{s}]", 1) for s in range(NS)]
        self.pready = [Barrier(f"p_ready[{s}]", 1) for s in range(NS)]
        # buffer contents
        self.stage = [None] * stages          # ring item held: (unit, item)
        self.abuf = [None] * abufs            # unit whose A tiles a buffer holds
        self.sbuf = [None] * NS               # ('S' | 'P', unit, item) in a stream's score tile
        self.obuf = [[None] * obufs for _ in range(NS)]  # [unit, PVs applied] per O accumulator
        self.tma = []                         # pending copies: (kind, index, content)
        self.fifo = [[] for _ in range(NS)]   # each MMA warp's products and commits in order

    # ---------------------------------------------------------------- the kernel's geometry
    def n_par(self, k):
        return NS // self.units[k]

    def stream_items(self, k, s):
        """Items of unit k that stream s takes (their indices within the unit)."""
        n_a, n_par = self.units[k], self.n_par(k)
        par = s // n_a
        return [i for i in range(self.n_items[k]) if i % n_par == par]

    def no_item_streams(self, k):
        if self.plant == "afree_unguarded":
            return 0
        n_a, n_par = self.units[k], self.n_par(k)
        return n_a * max(0, n_par - self.n_items[k])

    def carried(self, k):
        return self.OB == 2 and k + 1 < self.U

    # ---------------------------------------------------------------- agents
    def producer(self):
        it = 0

        def issue_a(k):
            b = k % self.AB
            yield ("wait", self.afree[b], k // self.AB - 1, "producer")
            self.tma.append(("A", b, k))

        for k in range(min(self.ahead, self.U)):
            yield from issue_a(k)
        for k in range(self.U):
            for i in range(self.n_items[k]):
                st = it % self.S
                yield ("wait", self.empty[st], it // self.S - 1, "producer")
                self.tma.append(("ring", st, (k, i)))
                self.empty[st].arrive(NS - self.units[k])  # for the streams that skip it
                it += 1
                yield ("step",)
            if k + self.ahead < self.U:
                yield from issue_a(k + self.ahead)

    def mma(self, s):
        it, pc, pv = 0, 0, None  # pv: the owed PV (stage, item, O accumulator, unit)
        for k in range(self.U):
            n_a, n_par = self.units[k], self.n_par(k)
            par = s // n_a
            ab = k % self.AB
            ob = k % 2 if self.OB == 2 else 0
            yield ("wait", self.afull[ab], k // self.AB, f"mma{s}")
            for i in range(self.n_items[k]):
                st = it % self.S
                it += 1
                # every item's full barrier, in order, so each parity test names one phase
                yield ("wait", self.full[st], (it - 1) // self.S, f"mma{s}")
                if i % n_par != par:
                    continue
                if pv is not None:
                    yield ("wait", self.pready[s], pc, f"mma{s}")
                    pc += 1
                    self.fifo[s].append(("PV", s) + pv)
                self.fifo[s].append(("S", s, st, (k, i), ab))
                self.fifo[s].append(("commit", self.sready[s]))
                pv = (st, (k, i), ob, k)
                yield ("step",)
            if self.carried(k):
                continue
            if pv is not None:
                yield ("wait", self.pready[s], pc, f"mma{s}")
                pc += 1
                self.fifo[s].append(("PV", s) + pv)
                self.fifo[s].append(("commit", self.odone[s]))
            pv = None

    def softmax(self, s):
        ph0, od, it0, owed = 0, 0, 0, None
        for k in range(self.U):
            mine = self.stream_items(k, s)
            cnt = len(mine)
            ab = k % self.AB
            ob = k % 2 if self.OB == 2 else 0
            if self.plant == "early_end" and owed is not None:
                yield from self.finish(s, owed, True, od)
                owed = None
            for j, i in enumerate(mine):
                yield ("wait", self.sready[s], ph0 + j, f"softmax{s}")
                if j >= 1:  # S of item j: the PV of item j - 1 is complete
                    self.release(it0 + mine[j - 1])
                last = j == cnt - 1
                if (self.plant == "afree_first" and j == 0) or (self.plant != "afree_first" and last):
                    # stream 0 also arrives for the streams with no item in the unit
                    self.afree[ab].arrive(1 + (self.no_item_streams(k) if s == 0 else 0))
                if self.sbuf[s] != ("S", k, i):
                    raise ProtocolError(f"softmax{s} reads {self.sbuf[s]} for the S of {(k, i)}")
                self.sbuf[s] = ("P", k, i)
                self.pready[s].arrive()
                yield ("step",)
                if owed is not None:
                    od = yield from self.finish(s, owed, True, od)
                    owed = None
            end = (k, mine, it0, ob, ab)
            if self.carried(k):
                owed = end
            else:
                od = yield from self.finish(s, end, False, od)
            ph0 += cnt
            it0 += self.n_items[k]

    def finish(self, s, end, deferred, od):
        k, mine, it0, ob, ab = end
        if mine:
            if not deferred:
                yield ("wait", self.odone[s], od, f"softmax{s} end")
                od += 1
            self.release(it0 + mine[-1])
            o = self.obuf[s][ob]
            if o != [k, len(mine)]:
                raise ProtocolError(f"softmax{s} reads O[{ob}] = {o} as unit {k} with "
                                    f"{len(mine)} PVs")
        elif self.plant == "afree_unguarded":
            self.afree[ab].arrive()  # at once: may count toward an earlier unit's phase
        return od

    def release(self, it):
        self.empty[it % self.S].arrive()

    # ---------------------------------------------------------------- asynchronous parts
    def complete_tma(self, idx):
        kind, where, what = self.tma.pop(idx)
        if kind == "ring":
            self.stage[where] = what
            self.full[where].arrive()
        else:
            self.abuf[where] = what
            self.afull[where].arrive()

    def complete_mma(self, s):
        op = self.fifo[s].pop(0)
        if op[0] == "commit":
            op[1].arrive()
        elif op[0] == "S":
            _, s_, st, item, ab = op
            if self.stage[st] != item:
                raise ProtocolError(f"S of {item} finds stage {st} holding {self.stage[st]}")
            if self.abuf[ab] != item[0]:
                raise ProtocolError(f"S of {item} finds A buffer {ab} holding unit {self.abuf[ab]}")
            self.sbuf[s_] = ("S",) + item
        else:
            _, s_, st, item, ob, k = op
            if self.stage[st] != item:
                raise ProtocolError(f"PV of {item} finds stage {st} holding {self.stage[st]}")
            if self.sbuf[s_] != ("P",) + item:
                raise ProtocolError(f"PV of {item} finds {self.sbuf[s_]} in the score tile")
            o = self.obuf[s_][ob]
            if o is None or o[0] != k:
                o = [k, 0]  # the unit's first PV starts the accumulator
            o[1] += 1
            self.obuf[s_][ob] = o

    # ---------------------------------------------------------------- scheduler
    def run(self, max_steps=200000):
        agents = {"producer": self.producer()}
        for s in range(NS):
            agents[f"mma{s}"] = self.mma(s)
            agents[f"softmax{s}"] = self.softmax(s)
        waiting = {name: None for name in agents}
        for _ in range(max_steps):
            runnable = []
            for name, w in waiting.items():
                if w is None or w[1].check(w[2], w[3]):
                    runnable.append(("agent", name))
            runnable += [("tma", i) for i in range(len(self.tma))]
            runnable += [("mma", s) for s in range(NS) if self.fifo[s]]
            if not runnable:
                if agents:
                    raise ProtocolError(f"deadlock: {sorted(agents)} wait on "
                                        f"{[(n, w[1].name, w[2]) for n, w in waiting.items()]}")
                return
            # warps issue their next instruction far sooner than a copy or a product completes:
            # a runnable agent moves first nine times in ten
            agents_ready = [r for r in runnable if r[0] == "agent"]
            if agents_ready and (len(agents_ready) == len(runnable) or self.rng.random() < 0.9):
                kind, x = self.rng.choice(agents_ready)
            else:
                kind, x = self.rng.choice([r for r in runnable if r[0] != "agent"])
            if x == self.slow and len(runnable) > 1 and self.rng.random() < 0.98:
                continue
            if kind == "tma":
                self.complete_tma(x)
            elif kind == "mma":
                self.complete_mma(x)
            else:
                try:
                    req = next(agents[x])
                except StopIteration:
                    del agents[x], waiting[x]
                    continue
                waiting[x] = req if req[0] == "wait" else None
        raise ProtocolError("step bound reached")


def decode_case(n_units, n_items, obufs):
    return dict(units=[4] * n_units, n_items=[n_items] * n_units, stages=8, abufs=2, obufs=obufs)


def encode_case(rng):
    n = rng.randint(1, 4)
    return dict(units=[rng.choice([1, 2, 4]) for _ in range(n)],
                n_items=[rng.randint(1, 12) for _ in range(n)],
                stages=rng.choice([8, 10, 13, 16]), abufs=1, obufs=1)


@pytest.mark.parametrize("obufs", [1, 2])
@pytest.mark.parametrize("n_units,n_items", [(1, 1), (2, 1), (5, 1), (3, 2), (4, 3), (6, 8),
                                             (3, 11)])
def test_decode_protocol(n_units, n_items, obufs):
    for seed in range(25):
        Model(rng=random.Random(seed), **decode_case(n_units, n_items, obufs)).run()


def test_encode_protocol():
    rng = random.Random(7)
    for seed in range(150):
        Model(rng=random.Random(seed), **encode_case(rng)).run()


def short_units_case():
    # consecutive units of one route tile whose chunks have fewer items than token parities:
    # three streams take no item of any of them
    return dict(units=[1] * 4, n_items=[1, 2, 1, 1], stages=16, abufs=1, obufs=1)


def test_encode_short_units():
    for seed in range(300):
        Model(rng=random.Random(seed), **short_units_case()).run()


def lagging_cases():
    """The protocol must hold however slow the producer or any one softmax warpgroup is: each in
    turn runs one step in fifty. (MMA warps issue a handful of instructions per item and keep up
    with the ring; the last test shows what the design assumes there.)"""
    names = ["producer"] + [f"softmax{s}" for s in range(NS)]
    cases = [decode_case(5, 2, 2), decode_case(3, 3, 1), short_units_case(),
             dict(units=[1, 2, 4], n_items=[20, 9, 20], stages=8, abufs=1, obufs=1)]
    return [(n, c) for n in names for c in cases]


@pytest.mark.parametrize("slow,case", lagging_cases())
def test_protocol_with_a_lagging_agent(slow, case):
    for seed in range(8):
        Model(rng=random.Random(seed), slow=slow, **case).run()


def test_observer_lag_limit():
    """The stated assumption: an MMA warp watches the full barrier of every item, its stream's or
    not, and the stages of items it skips are freed without it; slowed to one step in fifty
    over a ring of 8 stages it can find full two phases ahead. On the GPU it keeps up: per item
    it skips it only waits, and per item of its own it spends far less than the item takes."""
    case = dict(units=[1] * 3, n_items=[20] * 3, stages=8, abufs=1, obufs=1)
    with pytest.raises(ProtocolError):
        for seed in range(200):
            Model(rng=random.Random(seed), slow="mma3", **case).run()


@pytest.mark.parametrize("plant,case,slow", [
    ("afree_first", decode_case(4, 3, 2), None),
    ("early_end", decode_case(4, 3, 2), None),
    ("afree_unguarded", short_units_case(), "softmax0"),
])
def test_planted_mistakes_are_caught(plant, case, slow):
    with pytest.raises(ProtocolError):
        for seed in range(200):
            Model(rng=random.Random(seed), plant=plant, slow=slow, **case).run()


def test_one_stage_ring_is_caught():
    """One ring stage: the next item cannot land before the stream's own S frees the stage,
    which needs that item. (The kernel keeps at least 2 NS stages.)"""
    case = dict(units=[4] * 3, n_items=[6] * 3, stages=1, abufs=2, obufs=2)
    with pytest.raises(ProtocolError):
        Model(rng=random.Random(0), **case).run()
