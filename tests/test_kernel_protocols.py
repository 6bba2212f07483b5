"""Randomised models of the tcgen05 kernels' synchronisation protocols, run
on the CPU: the forward attention kernel (paper_2602_12529_gb300/csrc/
attention.cu, persistent variant) first, then the attention backward's two
kernels, the pair GEMM's main pipeline and its gated-residual epilogue.

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

The backward's two kernels (csrc/attention_bwd.cu: dQ over key tiles, dK / dV
over query tiles, each with a ring of three and a ring of two operand slots)
get models of the same kind below.

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


def _run(agents, pipe, tma, execute, land, rng, max_events=10 ** 6):
    """Random interleaving of the agents (generators), the in-order tensor
    pipe and the TMA engine (copies land in any order) until all finish."""
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
            land(tma.pop(rng.randrange(len(tma))))
        else:
            try:
                next(agents[choice])
            except StopIteration:
                done.add(choice)
    raise _Hazard("no progress: deadlock")


def _waiter(bars):
    def wait(name, parity, need_phases):
        while not bars[name].passes(parity):
            yield "blocked"
        if bars[name].phases < need_phases:
            raise _Hazard(f"{name}: parity wait passed on an older phase")
    return wait


def _ring_wait(wait, name, j):
    """Wait for phase j of a four-entry barrier ring (entry j % 4)."""
    return wait(f"{name}{j & 3}", (j >> 2) & 1, (j >> 2) + 1)


def _simulate_dq(T, seed, defect=None):
    """The backward's dQ kernel (csrc/attention_bwd.cu) for one 128-row query
    tile against T key tiles: K_j into K slot j % 3 once dQ_j-3 is done
    (rel ring), V_j into V slot j % 2 once S / dP of tile j - 2 are done
    (s0 ring), both on operand barrier j % 4 (two arrivals); the MMA thread
    issues S_j+1 / dP_j+1 once both elementwise warps hold S_j / dP_j, and
    dQ += dS_j K_j once both have written dS_j; an elementwise warp writes
    dS_j only after dQ_j-1 (rel ring).  defect: "no_v_wait" drops the
    producer's wait before reusing a V slot; "no_ds_wait" drops the
    elementwise warps' wait before writing dS."""
    rng = random.Random(seed)
    bars = {"p0": _Bar("p0", 2), "p1": _Bar("p1", 2), "done": _Bar("done", 1)}
    for i in range(4):
        bars[f"grp{i}"] = _Bar(f"grp{i}", 2)
        bars[f"rel{i}"] = _Bar(f"rel{i}", 1)
        bars[f"sring{i}"] = _Bar(f"sring{i}", 1)
    wait = _waiter(bars)
    kslot, vslot = [[None, False] for _ in range(3)], [[None, False] for _ in range(2)]
    kread, vread = [set() for _ in range(3)], [set() for _ in range(2)]
    tma, pipe = [], []
    st = {"sp": None, "sp_read": [-1, -1], "ds": [-1, -1], "dq": -1}

    def producer():
        for j in range(T):
            if j >= 3:
                yield from _ring_wait(wait, "rel", j - 3)
            if kread[j % 3]:
                raise _Hazard(f"K slot {j % 3} reused with reads pending")
            bars[f"grp{j & 3}"].arrive(tx=1)
            kslot[j % 3][:] = [j, False]
            kread[j % 3] |= {("SDP", j), ("DQ", j)}
            tma.append(("k", j % 3, j, f"grp{j & 3}"))
            if j >= 2 and defect != "no_v_wait":
                yield from _ring_wait(wait, "sring", j - 2)
            if vread[j % 2]:
                raise _Hazard(f"V slot {j % 2} reused with reads pending")
            bars[f"grp{j & 3}"].arrive(tx=1)
            vslot[j % 2][:] = [j, False]
            vread[j % 2] |= {("SDP", j)}
            tma.append(("v", j % 2, j, f"grp{j & 3}"))
            yield "step"

    def mma():
        yield from _ring_wait(wait, "grp", 0)
        pipe.extend([("SDP", 0), ("commit", "sring0")])
        for j in range(T):
            yield from wait("p0", j & 1, j + 1)
            if j + 1 < T:
                pipe.extend([("SDP", j + 1), ("commit", f"sring{(j + 1) & 3}")])
            yield from wait("p1", j & 1, j + 1)
            pipe.extend([("DQ", j), ("commit", f"rel{j & 3}")])
            yield "step"
        pipe.append(("commit", "done"))

    def elementwise(cg):
        for j in range(T):
            yield from _ring_wait(wait, "sring", j)
            for _ in range(2):   # the TMEM loads span two events
                if st["sp"] != j:
                    raise _Hazard(f"warp {cg} read S / dP {st['sp']} for tile {j}")
                yield "step"
            st["sp_read"][cg] = j
            if j + 1 < T:
                yield from _ring_wait(wait, "grp", j + 1)
            bars["p0"].arrive()
            yield "step"
            if j > 0 and defect != "no_ds_wait":
                yield from _ring_wait(wait, "rel", j - 1)
            if st["dq"] < j - 1:
                raise _Hazard(f"warp {cg} wrote dS_{j} before dQ_{j - 1} read dS_{j - 1}")
            st["ds"][cg] = j
            bars["p1"].arrive()
            yield "step"
        yield from wait("done", 0, 1)
        if st["dq"] != T - 1:
            raise _Hazard("dQ read before its last product")

    def execute(op):
        if op[0] == "SDP":
            j = op[1]
            if kslot[j % 3] != [j, True] or vslot[j % 2] != [j, True]:
                raise _Hazard(f"S / dP of tile {j} read K or V before it landed")
            if j > 0 and min(st["sp_read"]) < j - 1:
                raise _Hazard(f"S / dP of tile {j} overwrote tile {j - 1}'s before both warps read them")
            st["sp"] = j
            kread[j % 3].discard(("SDP", j))
            vread[j % 2].discard(("SDP", j))
        elif op[0] == "DQ":
            j = op[1]
            if st["ds"] != [j, j]:
                raise _Hazard(f"dQ_{j} read dS {st['ds']}")
            if kslot[j % 3] != [j, True] or st["dq"] != j - 1:
                raise _Hazard(f"dQ_{j} out of order or before K_{j} landed")
            st["dq"] = j
            kread[j % 3].discard(("DQ", j))
        else:
            bars[op[1]].arrive()

    def land(copy):
        kind, idx, owner, bar = copy
        ring = kslot if kind == "k" else vslot
        if ring[idx][0] == owner:
            ring[idx][1] = True
        bars[bar].complete_tx(1)

    agents = {"producer": producer(), "mma": mma(), "ew0": elementwise(0), "ew1": elementwise(1)}
    _run(agents, pipe, tma, execute, land, rng)


def _simulate_dkdv(T, seed, defect=None):
    """The backward's dK / dV kernel for one 128-key tile against T query
    tiles: Q_i (with lse_i) into Q slot i % 3 on barrier ring grp, dO_i (with
    D_i) into dO slot i % 2 on ring do; before step n the producer waits for
    step n - 2's last MMA (rel ring), then loads Q_n+1 and dO_n.  The MMA
    thread: dV += P^T_i dO_i once both elementwise warps wrote P^T_i, S^T_i+1
    over it, dK += dS^T_i Q_i once both wrote dS^T_i, release, dP^T_i+1 over
    it.  The elementwise warps check Q_i+1 (dO_i+1) before publishing P^T_i
    (dS^T_i).  defect: "no_release_wait" drops the producer's wait."""
    rng = random.Random(seed)
    bars = {"s0": _Bar("s0", 1), "s1": _Bar("s1", 1), "p0": _Bar("p0", 2), "p1": _Bar("p1", 2),
            "done": _Bar("done", 1)}
    for i in range(4):
        bars[f"grp{i}"] = _Bar(f"grp{i}", 1)
        bars[f"do{i}"] = _Bar(f"do{i}", 1)
        bars[f"rel{i}"] = _Bar(f"rel{i}", 1)
    wait = _waiter(bars)
    qslot, doslot = [[None, False] for _ in range(3)], [[None, False] for _ in range(2)]
    qread, doread = [set() for _ in range(3)], [set() for _ in range(2)]
    tma, pipe = [], []
    st = {"a": None, "pt": [-1, -1], "b": None, "dst": [-1, -1], "dv": -1, "dk": -1}

    def producer():
        def load(ring, reads, i, tag, bar, slots):
            if reads[i % slots]:
                raise _Hazard(f"{tag} slot {i % slots} reused with reads pending")
            bars[bar].arrive(tx=1)
            ring[i % slots][:] = [i, False]
            reads[i % slots] |= {(tag, i, "mma"), (tag, i, 0), (tag, i, 1), (tag, i, "acc")}
            tma.append((tag, i % slots, i, bar))

        load(qslot, qread, 0, "q", "grp0", 3)
        for n in range(T):
            if n >= 2 and defect != "no_release_wait":
                yield from _ring_wait(wait, "rel", n - 2)
            if n + 1 < T:
                load(qslot, qread, n + 1, "q", f"grp{(n + 1) & 3}", 3)
            load(doslot, doread, n, "do", f"do{n & 3}", 2)
            yield "step"

    def mma():
        yield from _ring_wait(wait, "grp", 0)
        pipe.extend([("ST", 0), ("commit", "s0")])
        yield from _ring_wait(wait, "do", 0)
        pipe.extend([("DPT", 0), ("commit", "s1")])
        for i in range(T):
            yield from wait("p0", i & 1, i + 1)
            pipe.append(("DV", i))
            if i + 1 < T:
                pipe.extend([("ST", i + 1), ("commit", "s0")])
            yield from wait("p1", i & 1, i + 1)
            pipe.extend([("DK", i), ("commit", f"rel{i & 3}")])
            if i + 1 < T:
                pipe.extend([("DPT", i + 1), ("commit", "s1")])
            yield "step"
        pipe.append(("commit", "done"))

    def elementwise(cg):
        for i in range(T):
            yield from wait("s0", i & 1, i + 1)
            if st["a"] != i or qslot[i % 3] != [i, True]:
                raise _Hazard(f"warp {cg} read S^T {st['a']} / lse of Q slot {qslot[i % 3]} for tile {i}")
            yield "step"
            if st["a"] != i:
                raise _Hazard(f"S^T_{i} overwritten while warp {cg} read it")
            st["pt"][cg] = i
            qread[i % 3].discard(("q", i, cg))
            if i + 1 < T:
                yield from _ring_wait(wait, "grp", i + 1)
            bars["p0"].arrive()
            yield from wait("s1", i & 1, i + 1)
            if st["b"] != i or doslot[i % 2] != [i, True]:
                raise _Hazard(f"warp {cg} read dP^T {st['b']} / D of dO slot {doslot[i % 2]} for tile {i}")
            yield "step"
            st["dst"][cg] = i
            doread[i % 2].discard(("do", i, cg))
            if i + 1 < T:
                yield from _ring_wait(wait, "do", i + 1)
            bars["p1"].arrive()
            yield "step"
        yield from wait("done", 0, 1)
        if st["dv"] != T - 1 or st["dk"] != T - 1:
            raise _Hazard("dK / dV read before their last products")

    def execute(op):
        kind, i = op
        if kind == "ST":
            if qslot[i % 3] != [i, True]:
                raise _Hazard(f"S^T_{i} read Q_{i} before it landed")
            if i > 0 and st["dv"] < i - 1:
                raise _Hazard(f"S^T_{i} overwrote P^T_{i - 1} before dV read it")
            st["a"] = i
            qread[i % 3].discard(("q", i, "mma"))
        elif kind == "DPT":
            if doslot[i % 2] != [i, True]:
                raise _Hazard(f"dP^T_{i} read dO_{i} before it landed")
            if i > 0 and st["dk"] < i - 1:
                raise _Hazard(f"dP^T_{i} overwrote dS^T_{i - 1} before dK read it")
            st["b"] = i
            doread[i % 2].discard(("do", i, "mma"))
        elif kind == "DV":
            if st["pt"] != [i, i] or st["a"] != i or doslot[i % 2] != [i, True] or st["dv"] != i - 1:
                raise _Hazard(f"dV_{i} read P^T {st['pt']} / dO slot {doslot[i % 2]}")
            st["dv"] = i
            doread[i % 2].discard(("do", i, "acc"))
        elif kind == "DK":
            if st["dst"] != [i, i] or st["b"] != i or qslot[i % 3] != [i, True] or st["dk"] != i - 1:
                raise _Hazard(f"dK_{i} read dS^T {st['dst']} / Q slot {qslot[i % 3]}")
            st["dk"] = i
            qread[i % 3].discard(("q", i, "acc"))
        else:
            bars[i].arrive()

    def land(copy):
        tag, idx, owner, bar = copy
        ring = qslot if tag == "q" else doslot
        if ring[idx][0] == owner:
            ring[idx][1] = True
        bars[bar].complete_tx(1)

    agents = {"producer": producer(), "mma": mma(), "ew0": elementwise(0), "ew1": elementwise(1)}
    _run(agents, pipe, tma, execute, land, rng)


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


@pytest.mark.parametrize("T", [1, 2, 3, 5, 9])
def test_backward_protocols_are_hazard_free(T):
    """The backward's dQ kernel (K ring of 3, V ring of 2) and dK / dV
    kernel (Q ring of 3, dO ring of 2) over 1 to 9 tiles."""
    for seed in range(120):
        _simulate_dq(T, seed)
        _simulate_dkdv(T, seed)


@pytest.mark.parametrize("sim,defect", [(_simulate_dq, "no_v_wait"), (_simulate_dq, "no_ds_wait"),
                                        (_simulate_dkdv, "no_release_wait")])
def test_backward_planted_mistakes_are_caught(sim, defect):
    with pytest.raises(_Hazard):
        for seed in range(400):
            sim(6, seed, defect=defect)


def _simulate_gemm_pair(tiles, kblocks, seed, stages=5, defect=None):
    """The pair GEMM's main pipeline (csrc/gemm.cu, gemm_pair_kernel): two
    CTAs each load their half of a K block's A and B into stage s of a ring;
    both halves complete on the leader's full[s] (the leader alone announces
    the bytes); the leader's MMA thread consumes the stage and its commit
    arrives on both CTAs' empty[s]; after a tile's last K block it commits
    tfull[a] to both CTAs for accumulator a (two, alternating); each CTA's
    epilogue reads its half and arrives on the leader's tempty[a] (one
    arrival per CTA here, eight warps each in the kernel).  defect:
    "no_tempty_wait" drops the MMA thread's wait for a free accumulator,
    "no_empty_wait" the producers' wait for a free stage."""
    rng = random.Random(seed)
    bars = {}
    for s in range(stages):
        bars[f"full{s}"] = _Bar(f"full{s}", 1)
        for r in range(2):
            bars[f"empty{s}.{r}"] = _Bar(f"empty{s}.{r}", 1)
    for a in range(2):
        bars[f"tempty{a}"] = _Bar(f"tempty{a}", 2)
        for r in range(2):
            bars[f"tfull{a}.{r}"] = _Bar(f"tfull{a}.{r}", 1)
    wait = _waiter(bars)
    stage = [[None, [False, False]] for _ in range(stages)]   # (round, both halves landed)
    pending_reads = [None] * stages                           # round an MMA has yet to read
    tma, pipe = [], []
    acc = [{"tile": None, "k": -1, "read": [True, True]} for _ in range(2)]

    def producer(rank):
        n = 0
        for _ in range(tiles):
            for _ in range(kblocks):
                s, rnd = n % stages, n // stages
                if defect != "no_empty_wait":
                    yield from wait(f"empty{s}.{rank}", (rnd & 1) ^ 1, rnd)
                if pending_reads[s] is not None and pending_reads[s] != rnd:
                    raise _Hazard(f"stage {s} refilled before the MMA read round {pending_reads[s]}")
                if rank == 0:
                    bars[f"full{s}"].arrive(tx=2)
                if stage[s][0] != rnd:
                    stage[s][0], stage[s][1] = rnd, [False, False]
                    pending_reads[s] = rnd
                tma.append((s, rnd, rank))
                n += 1
                yield "step"

    def mma():
        n = 0
        for t in range(tiles):
            a, use = t & 1, t >> 1
            if defect != "no_tempty_wait":
                yield from wait(f"tempty{a}", (use & 1) ^ 1, use)
            for kb in range(kblocks):
                s, rnd = n % stages, n // stages
                yield from wait(f"full{s}", rnd & 1, rnd + 1)
                pipe.append(("MMA", s, rnd, t, kb, a))
                pipe.append(("commit", [f"empty{s}.0", f"empty{s}.1"]))
                n += 1
                yield "step"
            pipe.append(("commit", [f"tfull{a}.0", f"tfull{a}.1"]))

    def epilogue(rank):
        for t in range(tiles):
            a, use = t & 1, t >> 1
            yield from wait(f"tfull{a}.{rank}", use & 1, use + 1)
            for _ in range(2):
                if acc[a]["tile"] != t or acc[a]["k"] != kblocks - 1:
                    raise _Hazard(f"epilogue {rank} read accumulator {a} holding {acc[a]} for tile {t}")
                yield "step"
            acc[a]["read"][rank] = True
            bars[f"tempty{a}"].arrive()

    def execute(op):
        if op[0] == "commit":
            for name in op[1]:
                bars[name].arrive()
            return
        _, s, rnd, t, kb, a = op
        if stage[s][0] != rnd or stage[s][1] != [True, True]:
            raise _Hazard(f"MMA of tile {t} block {kb} read stage {s} before both halves landed")
        pending_reads[s] = None
        if kb == 0:
            if not all(acc[a]["read"]):
                raise _Hazard(f"tile {t} overwrote accumulator {a} before both epilogues read it")
            acc[a].update(tile=t, k=0, read=[False, False])
        else:
            if acc[a]["tile"] != t or acc[a]["k"] != kb - 1:
                raise _Hazard(f"MMA of tile {t} block {kb} accumulated onto {acc[a]}")
            acc[a]["k"] = kb

    def land(copy):
        s, rnd, rank = copy
        if stage[s][0] == rnd:
            stage[s][1][rank] = True
        bars[f"full{s}"].complete_tx(1)

    agents = {"prod0": producer(0), "prod1": producer(1), "mma": mma(), "epi0": epilogue(0), "epi1": epilogue(1)}
    _run(agents, pipe, tma, execute, land, rng)


@pytest.mark.parametrize("tiles,kblocks", [(1, 1), (3, 2), (5, 7), (4, 48), (9, 3)])
def test_gemm_pair_pipeline_is_hazard_free(tiles, kblocks):
    """Five stages, two accumulators, K blocks from 1 to 48 (K = 3072 at
    BK 64), several tiles per CTA pair."""
    for seed in range(100):
        _simulate_gemm_pair(tiles, kblocks, seed)


@pytest.mark.parametrize("defect,match", [("no_tempty_wait", "accumulator"),
                                          ("no_empty_wait", "stage|landed|more arrivals")])
def test_gemm_pair_planted_mistakes_are_caught(defect, match):
    with pytest.raises(_Hazard, match=match):
        for seed in range(400):
            _simulate_gemm_pair(6, 4, seed, defect=defect)


def _simulate_gated_epilogue(tiles, chunks, seed, workers=3, defect=None):
    """The gated-residual epilogue's chunk ring (csrc/gemm.cu, epilogue_tile):
    per column group two shared-memory buffers; chunk c of a tile uses
    buffer c % 2.  The group's leader loads the fp32 residual chunk by TMA
    (rfull[b]: its own arrival plus the bytes), every thread waits for it,
    updates its row, arrives on rdone[b]; the leader waits for all arrivals,
    stores the chunk by TMA and, before reloading the buffer with chunk
    c + 2 (or the next tile's first chunks), waits until its stores have
    read shared memory (bulk_wait_read).  Worker 0 is the leader.  defect:
    "no_store_wait" drops the bulk_wait_read, "no_rdone_wait" the leader's
    wait for every thread's update."""
    rng = random.Random(seed)
    bars = {}
    for b in range(2):
        bars[f"rfull{b}"] = _Bar(f"rfull{b}", 1)
        bars[f"rdone{b}"] = _Bar(f"rdone{b}", workers)
    wait = _waiter(bars)
    buf = [{"chunk": None, "landed": False, "updated": set()} for _ in range(2)]
    stores, loads = [], []   # the TMA engine: stores reading a buffer, loads filling one

    def store_free():
        while stores:
            yield "blocked"

    def load(b, chunk):
        if any(sb == b for sb, _ in stores):
            raise _Hazard(f"buffer {b} reloaded while a store still reads it")
        if buf[b]["chunk"] is not None and len(buf[b]["updated"]) < workers:
            raise _Hazard(f"buffer {b} reloaded before every thread updated chunk {buf[b]['chunk']}")
        bars[f"rfull{b}"].arrive(tx=1)
        buf[b].update(chunk=chunk, landed=False, updated=set())
        loads.append((b, chunk))

    def worker(w):
        ruse = [0, 0]
        for t in range(tiles):
            if w == 0:
                for c in range(min(2, chunks)):
                    if defect != "no_store_wait":
                        yield from store_free()
                    load(c, (t, c))
            for c in range(chunks):
                b = c & 1
                yield from wait(f"rfull{b}", ruse[b] & 1, ruse[b] + 1)
                for _ in range(2):   # the row update spans two events
                    if buf[b]["chunk"] != (t, c) or not buf[b]["landed"]:
                        raise _Hazard(f"thread {w} updated buffer {b} holding {buf[b]['chunk']} for {(t, c)}")
                    yield "step"
                buf[b]["updated"].add(w)
                bars[f"rdone{b}"].arrive()
                if w == 0 and defect != "no_rdone_wait":
                    yield from wait(f"rdone{b}", ruse[b] & 1, ruse[b] + 1)
                ruse[b] += 1
                if w == 0:
                    if len(buf[b]["updated"]) < workers:
                        raise _Hazard(f"chunk {(t, c)} stored before every thread updated it")
                    stores.append((b, (t, c)))
                    if c + 2 < chunks:
                        if defect != "no_store_wait":
                            yield from store_free()
                        load(b, (t, c + 2))
                yield "step"

    agents = {f"w{w}": worker(w) for w in range(workers)}
    done = set()
    for _ in range(10 ** 6):
        live = [a for a in agents if a not in done]
        hw = (["store"] if stores else []) + (["load"] if loads else [])
        if not live and not hw:
            return
        choice = rng.choice(live + hw * 2)
        if choice == "store":
            stores.pop(rng.randrange(len(stores)))
        elif choice == "load":
            b, chunk = loads.pop(rng.randrange(len(loads)))
            if buf[b]["chunk"] == chunk:
                buf[b]["landed"] = True
            bars[f"rfull{b}"].complete_tx(1)
        else:
            try:
                next(agents[choice])
            except StopIteration:
                done.add(choice)
    raise _Hazard("no progress: deadlock")


@pytest.mark.parametrize("tiles,chunks", [(1, 1), (1, 2), (3, 4), (4, 3), (2, 8)])
def test_gated_epilogue_ring_is_hazard_free(tiles, chunks):
    """Four chunks per column group (256-column pair tiles, eight epilogue
    warps), and other counts; several tiles in a row."""
    for seed in range(100):
        _simulate_gated_epilogue(tiles, chunks, seed)


@pytest.mark.parametrize("defect,match", [("no_store_wait", "store still reads"),
                                          ("no_rdone_wait", "every thread")])
def test_gated_epilogue_planted_mistakes_are_caught(defect, match):
    with pytest.raises(_Hazard, match=match):
        for seed in range(400):
            _simulate_gated_epilogue(3, 4, seed, defect=defect)
