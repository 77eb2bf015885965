"""CPU model of the forward kernel's per-item barrier protocol (csrc/attn_fwd.cu): one
work item (two query tiles) on its own. tests/test_fwd_walk_protocol.py models the walk
over many items that the kernel runs; this file keeps the single-item cases exhaustive
and the negative control of the first design.

A K producer, a V producer, the MMA issuer and two softmax groups synchronise through
mbarriers with parity waits, and the K / V ring stages are handed back to the producers
by the softmax thread that last read a key tile (k_empty / v_empty arrivals relayed after
it has seen the s_full commit of the S that followed the tile's last use). The model runs
those agents as coroutines against barrier objects with the hardware's parity
semantics, an in-order tensor pipe and copies that land after random delays,
and checks, for every query-tile pair and document-start placement up to 17
query tiles, that:
  * nothing deadlocks (every agent finishes),
  * no barrier phase is over-arrived (a re-arm before the phase completed),
  * a copy never lands in a ring stage an unfinished MMA still reads.
A negative control runs the first design, in which the producers waited on
s_full themselves: it over-arrives v_full, which a GPU run of that design
answered with a fault.
"""
import random

import pytest


class OverArrival(Exception):
    pass


class Deadlock(Exception):
    pass


class Barrier:
    """mbarrier: `count` arrivals plus expected transaction bytes complete a phase."""

    def __init__(self, count=1):
        self.count, self.pending, self.tx, self.done = count, count, 0, 0

    def _check(self):
        if self.pending < 0 or self.tx < 0:
            raise OverArrival()
        if self.pending == 0 and self.tx == 0:
            self.done += 1
            self.pending = self.count

    def arrive(self):
        self.pending -= 1
        self._check()

    def expect_tx(self, nbytes):
        self.tx += nbytes
        self.pending -= 1
        self._check()

    def complete_tx(self, nbytes):
        self.tx -= nbytes
        self._check()

    def test(self, parity):
        """try_wait.parity: true once the phase of that parity has completed."""
        return (self.done & 1) != parity


def simulate(nqt, u, lo0, lo1, seed, relay=True):
    rnd = random.Random(seed)
    has1 = 2 * u + 1 < nqt
    hi0, hi1 = 2 * u, 2 * u + 1
    J0 = lo0
    NJ = (hi1 if has1 else hi0) - J0 + 1
    bars = {n: Barrier() for n in ("q0", "q1", "k0", "k1", "v0", "v1", "s0", "s1", "pv0", "pv1", "drain",
                                   "ke0", "ke1", "ve0", "ve1", "p0", "p1")}
    now = [0]
    events = []                 # (time, callback)
    pipe = []                   # queued tensor-pipe items
    busy_until = [0]
    readers = {("k", 0): 0, ("k", 1): 0, ("v", 0): 0, ("v", 1): 0}

    def copy(bar, stage):
        if stage is not None and readers[stage]:
            raise AssertionError("copy into a stage an MMA still reads: %s" % (stage,))
        events.append((now[0] + rnd.randint(50, 3000), lambda: bars[bar].complete_tx(1)))

    def run_pipe():
        while pipe and busy_until[0] <= now[0]:
            kind, arg = pipe.pop(0)
            if kind == "mma":
                for st in arg:
                    readers[st] += 1
                busy_until[0] = max(now[0], busy_until[0]) + rnd.randint(300, 700)

                def finish(sts=arg):
                    for st in sts:
                        readers[st] -= 1
                events.append((busy_until[0], finish))
            else:   # a commit arrives once every earlier MMA has completed
                events.append((busy_until[0] + 1, lambda b=arg: bars[b].arrive()))

    def k_producer():
        for t in range(2 if has1 else 1):
            bars["q%d" % t].expect_tx(1)
            copy("q%d" % t, None)
        for j in range(NJ):
            s = j % 2
            if j >= 2:
                if relay:
                    yield ("wait", "ke%d" % s, ((j // 2) - 1) & 1)
                else:
                    kt = J0 + j - 2
                    t1 = has1 and kt >= lo1
                    yield ("wait", "s1" if t1 else "s0", (kt - (lo1 if t1 else lo0)) & 1)
            bars["k%d" % s].expect_tx(1)
            copy("k%d" % s, ("k", s))

    def v_producer():
        for j in range(NJ):
            s = j % 2
            if j >= 2:
                if relay:
                    yield ("wait", "ve%d" % s, ((j // 2) - 1) & 1)
                else:
                    kt = J0 + j - 1
                    t1 = has1 and kt - 1 >= lo1
                    yield ("wait", "s1" if t1 else "s0", (kt - (lo1 if t1 else lo0)) & 1)
            bars["v%d" % s].expect_tx(1)
            copy("v%d" % s, ("v", s))

    def mma():
        ns, npv = [0, 0], [0, 0]
        for j in range(NJ + 1):
            kt = J0 + j
            for t in range(2):
                if not (t == 0 or has1):
                    continue
                lo_t, hi_t = (lo1, hi1) if t else (lo0, hi0)
                if j >= 1 and lo_t <= kt - 1 <= hi_t:       # O_t += P_t V_{j-1}
                    yield ("wait", "v%d" % ((j - 1) % 2), ((j - 1) // 2) & 1)
                    yield ("wait", "p%d" % t, npv[t] & 1)
                    pipe.append(("mma", [("v", (j - 1) % 2)]))
                    if kt - 1 == hi_t:
                        pipe.append(("commit", "pv%d" % t))
                    npv[t] += 1
                if j < NJ and lo_t <= kt <= hi_t:           # S_t = Q_t K_j^T
                    yield ("wait", "k%d" % (j % 2), (j // 2) & 1)
                    if ns[t] == 0:
                        yield ("wait", "q%d" % t, 0)
                    pipe.append(("mma", [("k", j % 2)]))
                    pipe.append(("commit", "s%d" % t))
                    ns[t] += 1
        pipe.append(("commit", "drain"))
        yield ("wait", "drain", 0)

    def softmax(t):
        lo_t = lo1 if t else lo0
        nt = ((hi1 if t else hi0) - lo_t + 1) if (t == 0 or has1) else 0
        for i in range(nt):
            yield ("wait", "s%d" % t, i & 1)
            kt = lo_t + i
            if relay:
                if t == 1 or not (has1 and kt >= lo1):
                    bars["ke%d" % ((kt - J0) % 2)].arrive()
                if i >= 1 and (t == 1 or not (has1 and kt - 1 >= lo1)):
                    bars["ve%d" % ((kt - 1 - J0) % 2)].arrive()
            yield ("delay", rnd.randint(200, 1500))
            bars["p%d" % t].arrive()
        if nt:
            yield ("wait", "pv%d" % t, 0)

    agents = {"kp": k_producer(), "vp": v_producer(), "mma": mma(), "sm0": softmax(0), "sm1": softmax(1)}
    state = {n: None for n in agents}
    alive = set(agents)

    def step(name):
        while True:
            req = state[name]
            if req is None:
                try:
                    req = next(agents[name])
                except StopIteration:
                    alive.discard(name)
                    return
                state[name] = req
            if req[0] == "wait" and bars[req[1]].test(req[2]):
                state[name] = None
                continue
            if req[0] == "delay":
                state[name] = ("until", now[0] + req[1])
                return
            if req[0] == "until" and now[0] >= req[1]:
                state[name] = None
                continue
            return

    def snapshot():
        return (tuple(sorted(alive)), tuple(state[n] for n in sorted(agents)),
                tuple((b.done, b.pending, b.tx) for b in bars.values()), len(pipe))

    for _ in range(200000):
        if not alive:
            return
        while True:                  # every agent to a fixpoint at this time
            before = snapshot()
            for n in list(alive):
                step(n)
            run_pipe()
            if snapshot() == before:
                break
        times = [e[0] for e in events] + [state[n][1] for n in alive if state[n] and state[n][0] == "until"]
        if pipe:
            times.append(max(busy_until[0], now[0] + 1))
        if not times:
            if alive:
                raise Deadlock(str({n: state[n] for n in alive}))
            return
        now[0] = max(now[0] + 1, min(times))
        due = sorted((e for e in events if e[0] <= now[0]), key=lambda e: e[0])
        events[:] = [e for e in events if e[0] > now[0]]
        for _, cb in due:
            cb()
    raise AssertionError("no progress")


def _layouts(nqts):
    for nqt in nqts:
        for u in range((nqt + 1) // 2):
            for lo0 in range(0, 2 * u + 1):
                for lo1 in range(lo0, 2 * u + 2):
                    yield nqt, u, lo0, lo1


@pytest.mark.parametrize("nqt", [1, 2, 3, 4, 5, 8, 17])
def test_relay_protocol_completes_for_every_layout(nqt):
    """Every query-tile pair of an nqt-tile sequence, every pair of document-start key
    tiles (lo0 <= lo1 <= the pair's diagonal), three timing seeds."""
    n = 0
    for case in _layouts([nqt]):
        for seed in range(3):
            simulate(*case, seed=seed, relay=True)
            n += 1
    assert n > 0


def test_producers_waiting_on_s_full_over_arrive():
    """Negative control: with two ring stages the tensor core can complete two s_full
    phases before a producer looks, so a parity wait on s_full passes early and the
    producer re-arms a stage whose previous copy has not landed."""
    failures = 0
    for case in _layouts([3, 4, 8]):
        try:
            simulate(*case, seed=0, relay=False)
        except (OverArrival, AssertionError, Deadlock):
            failures += 1
    assert failures > 0
