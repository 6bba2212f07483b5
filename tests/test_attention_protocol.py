"""A randomised model of the forward attention kernel's synchronisation
protocol (paper_2602_12529_gb300/csrc/attention.cu, persistent variant),
run on the CPU.

The kernel has four agents sharing shared-memory slots, two query tiles and
TMEM, ordered only by mbarrier phases:
  * the TMA producer: the two query tiles of each work item, then K_0, V_0,
    K_1, V_1, ... into a ring of S slots.  Ring item n sits in slot n % S
    and belongs to operand group (n + 1) // 2 (group 0 = K_0; group g =
    V_g-1 and K_g; the last group = the last V), whose barrier (one of four,
    g % 4) expects two arrivals (one for a one-operand group) and the
    copies' bytes.  Before reusing slot n % S it waits until S_1 of step
    (n - S + 1) // 2 is done (the last reader of the slot's previous item
    precedes it in the tensor pipe).  A new item's query tile t is loaded
    once S_t of the previous item's last step is done.
  * the MMA-issuing thread: S_t,0 for both tiles, then per step g and tile
    t: wait P_t,g, issue O_t += P_t,g V_g, then S_t,g+1 (after the next
    item's query tile when g ends an item), committing S_0 to a two-phase
    barrier and S_1 to a ring of four; the item's last O += P V is
    committed to o_last[t].
  * the tensor pipe: executes MMAs and commits in issue order.
  * two softmax warpgroups: per step wait S_t,g, turn it into P_t,g (tile
    0's warps also check operand group g + 1 first), arrive on P_t; per
    item wait o_last[t] and read O_t.
A split launch gives a CTA one half item after its whole items: steps
[0, h) or [h, T) of an item of T steps.

The model executes random interleavings and checks every hazard: a slot,
query tile or TMEM region overwritten while a reader is pending, an operand
read before its copy landed, a barrier receiving more arrivals than its
count, a parity wait passing on an older phase, and deadlock.  The kernel
caps its ring at seven slots; with eight, ring item 7 can arrive on the
barrier group 0 still uses, the defect the last test plants.
"""
import random

import pytest


class _Bar:
    def __init__(self, name, count):
        self.name, self.count = name, count
        self.arrivals, self.tx, self.phases = 0, 0, 0

    def arrive(self, tx=0):
        self.arrivals += 1
        self.tx += tx
        self._settle()

    def complete_tx(self, nbytes):
        self.tx -= nbytes
        self._settle()

    def _settle(self):
        if self.arrivals > self.count:
            raise _Hazard(f"{self.name}: more arrivals than its count")
        if self.arrivals == self.count and self.tx == 0:
            self.arrivals = self.tx = 0
            self.phases += 1

    def passes(self, parity):
        # mbarrier.try_wait.parity: true once the phase with this parity completed
        return (self.phases & 1) != parity


class _Hazard(Exception):
    pass


def _simulate(S, steps, items, seed, half=None, defect=None, max_events=10 ** 6):
    """One random interleaving.  S slots; `items` work items of `steps` K/V
    steps each; half = 0 / 1 makes the last item that half of its steps.
    defect plants a mistake: "no_slot_wait" (the producer reuses a slot
    without waiting for its readers) or "early_query" (a new item's query
    tiles load without waiting for the previous item's last S MMAs)."""
    rng = random.Random(seed)
    segs = [(0, steps)] * items
    if half is not None:
        h = steps // 2
        segs[-1] = (0, h) if half == 0 else (h, steps)
    gmap = [(k, j) for k, (j0, j1) in enumerate(segs) for j in range(j0, j1)]   # global step -> (item, step)
    nsteps = len(gmap)
    bars = {"q0": _Bar("q0", 1), "q1": _Bar("q1", 1), "s0": _Bar("s0", 1), "p0": _Bar("p0", 1),
            "p1": _Bar("p1", 1), "ol0": _Bar("ol0", 1), "ol1": _Bar("ol1", 1), "drain": _Bar("drain", 1)}
    for i in range(4):
        bars[f"grp{i}"] = _Bar(f"grp{i}", 2)
        bars[f"s1_{i}"] = _Bar(f"s1_{i}", 1)
    slot = [None] * S                      # ring item held
    landed = [False] * S
    readers = [set() for _ in range(S)]    # MMAs that still have to read the slot's item
    qtile, q_landed = [None, None], [False, False]
    tma = []                               # copies in flight: (kind, index, owner, barrier)
    pipe = []                              # issued MMAs and commits, in order
    tm_s = [None, None]                    # ("S", g) or ("P", g) in tile t's S/P columns
    tm_o = [None, None]                    # (item, local step) accumulated in O_t
    o_read = [-1, -1]                      # last item whose O_t the epilogue read
    pv_done = [-1, -1]

    def wait(name, parity, need_phases):
        while not bars[name].passes(parity):
            yield "blocked"
        if bars[name].phases < need_phases:
            raise _Hazard(f"{name}: parity wait passed on an older phase")

    def producer():
        seen = [-1]

        def s1_done_upto(c):
            while seen[0] < c:
                e = seen[0] + 1
                yield from wait(f"s1_{e & 3}", (e >> 2) & 1, (e >> 2) + 1)
                seen[0] += 1

        def load_q(t, k):
            if any(op[0] == "S" and op[1] == t for op in pipe):
                raise _Hazard(f"query tile {t} reloaded with an S MMA pending")
            bars[f"q{t}"].arrive(tx=1)
            qtile[t], q_landed[t] = k, False
            tma.append(("q", t, k, f"q{t}"))

        load_q(0, 0)
        load_q(1, 0)
        for n in range(2 * nsteps):
            s, g = n % S, n >> 1
            k, j = gmap[g]
            if n >= S and defect != "no_slot_wait":
                yield from s1_done_upto((n - S + 1) >> 1)
            if readers[s]:
                raise _Hazard(f"slot {s} reused with reads pending")
            grp = (n + 1) >> 1
            bars[f"grp{grp & 3}"].arrive(tx=1)
            slot[s], landed[s] = n, False
            readers[s] = {("S", 0, g), ("S", 1, g)} if n % 2 == 0 else {("PV", 0, g), ("PV", 1, g)}
            tma.append(("kv", s, n, f"grp{grp & 3}"))
            if n == 0 or n == 2 * nsteps - 1:
                bars[f"grp{grp & 3}"].arrive()          # one-operand groups
            if n % 2 == 0 and k > 0 and j == segs[k][0]:
                if defect != "early_query":
                    yield from s1_done_upto(g - 2)
                    yield from wait("s0", (g - 1) & 1, g)
                load_q(0, k)
                if defect != "early_query":
                    yield from s1_done_upto(g - 1)
                load_q(1, k)
            yield "step"

    def mma():
        def issue_s(t, g):
            pipe.append(("S", t, g))
            pipe.append(("commit", "s0" if t == 0 else f"s1_{g & 3}"))

        yield from wait("q0", 0, 1)
        yield from wait("q1", 0, 1)
        yield from wait("grp0", 0, 1)
        issue_s(0, 0)
        issue_s(1, 0)
        for g in range(nsteps):
            k, j = gmap[g]
            j0, j1 = segs[k]
            last = j == j1 - 1
            for t in range(2):
                yield from wait(f"p{t}", g & 1, g + 1)
                pipe.append(("PV", t, g, j - j0, k))
                if last:
                    pipe.append(("commit", f"ol{t}"))
                if g + 1 < nsteps:
                    if last:
                        yield from wait(f"q{t}", (k + 1) & 1, k + 2)
                    issue_s(t, g + 1)
                yield "step"
        pipe.append(("commit", "drain"))
        yield from wait("drain", 0, 1)

    def softmax(t):
        g = -1
        for k, (j0, j1) in enumerate(segs):
            for _ in range(j0, j1):
                g += 1
                if t == 0:
                    yield from wait("s0", g & 1, g + 1)
                else:
                    yield from wait(f"s1_{g & 3}", (g >> 2) & 1, (g >> 2) + 1)
                if tm_s[t] != ("S", g):
                    raise _Hazard(f"softmax {t} read {tm_s[t]} for S of step {g}")
                yield "step"
                tm_s[t] = ("P", g)
                if t == 0:
                    yield from wait(f"grp{(g + 1) & 3}", ((g + 1) >> 2) & 1, ((g + 1) >> 2) + 1)
                bars[f"p{t}"].arrive()
                yield "step"
            yield from wait(f"ol{t}", k & 1, k + 1)
            for _ in range(2):   # the epilogue's loads span two events
                if tm_o[t] != (k, j1 - j0 - 1):
                    raise _Hazard(f"epilogue {t} of item {k} read O {tm_o[t]}")
                yield "step"
            o_read[t] = k

    def execute(op):
        if op[0] == "S":
            _, t, g = op
            ks = (2 * g) % S
            if slot[ks] != 2 * g or not landed[ks]:
                raise _Hazard(f"S{t},{g} read slot {ks} before K_{g} landed")
            if qtile[t] != gmap[g][0] or not q_landed[t]:
                raise _Hazard(f"S{t},{g} read query tile {t} before it landed")
            if tm_s[t] is not None and not (tm_s[t] == ("P", g - 1) and pv_done[t] >= g - 1):
                raise _Hazard(f"S{t},{g} overwrote {tm_s[t]}")
            tm_s[t] = ("S", g)
            readers[ks].discard(("S", t, g))
        elif op[0] == "PV":
            _, t, g, j, k = op
            vs = (2 * g + 1) % S
            if slot[vs] != 2 * g + 1 or not landed[vs]:
                raise _Hazard(f"PV{t},{g} read slot {vs} before V_{g} landed")
            if tm_s[t] != ("P", g):
                raise _Hazard(f"PV{t},{g} read {tm_s[t]} as P")
            if j == 0:
                if k > 0 and o_read[t] != k - 1:
                    raise _Hazard(f"PV{t},{g} overwrote O of item {k - 1} before its epilogue")
                tm_o[t] = (k, 0)
            else:
                if tm_o[t] != (k, j - 1):
                    raise _Hazard(f"PV{t},{g} accumulated onto {tm_o[t]}")
                tm_o[t] = (k, j)
            pv_done[t] = g
            readers[vs].discard(("PV", t, g))
        else:
            bars[op[1]].arrive()

    agents = {"producer": producer(), "mma": mma(), "softmax0": softmax(0), "softmax1": softmax(1)}
    done = set()
    for _ in range(max_events):
        live = [a for a in agents if a not in done]
        hardware = (["pipe"] if pipe else []) + (["tma"] if tma else [])
        if not live and not hardware:
            return
        choice = rng.choice(live + hardware * 2)
        if choice == "pipe":
            execute(pipe.pop(0))
        elif choice == "tma":
            kind, idx, owner, bar = tma.pop(rng.randrange(len(tma)))
            if kind == "kv" and slot[idx] == owner:
                landed[idx] = True
            if kind == "q" and qtile[idx] == owner:
                q_landed[idx] = True
            bars[bar].complete_tx(1)
        else:
            try:
                next(agents[choice])
            except StopIteration:
                done.add(choice)
    raise _Hazard("no progress: deadlock")


CASES = [(7, 4, 4, None), (7, 4, 3, 0), (7, 4, 3, 1), (5, 2, 3, 0), (5, 2, 3, 1), (5, 2, 1, 0), (5, 2, 1, 1),
         (7, 3, 2, 1), (7, 3, 2, 0), (5, 36, 3, 1), (5, 36, 1, 0), (5, 5, 4, 1), (5, 1, 6, None), (3, 4, 3, None),
         (6, 4, 3, None)]


@pytest.mark.parametrize("S,steps,items,half", CASES)
def test_protocol_is_hazard_free(S, steps, items, half):
    """Rings of 3 to 7 slots (the kernel uses 5 at d = 128 and 7 at d = 64),
    items of 1 to 36 K/V steps, several items per CTA, and a split launch's
    half item (either half) as the CTA's only or last item."""
    for seed in range(150):
        _simulate(S, steps, items, seed, half)


@pytest.mark.parametrize("defect,match", [("no_slot_wait", "slot|landed|more arrivals"),
                                          ("early_query", "query tile")])
def test_planted_protocol_mistakes_are_caught(defect, match):
    """Each wait the producer makes is needed: without it some interleaving
    overwrites an operand that an MMA has yet to read."""
    with pytest.raises(_Hazard, match=match):
        for seed in range(400):
            _simulate(5, 4, 3, seed, defect=defect)


def test_eight_slots_overfill_an_operand_group_barrier():
    """The planted defect: with eight slots ring item 7 (V_3, group 4) needs
    no slot wait and can arrive on barrier 0 while group 0 still waits for
    K_0's bytes.  Some interleaving must show it."""
    with pytest.raises(_Hazard, match="more arrivals"):
        for seed in range(400):
            _simulate(8, 4, 3, seed)
