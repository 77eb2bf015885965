"""CPU model of the walking backward kernel's barrier protocol (csrc/attn_bwd_d128_persist.cu,
which shares its per-step protocol with csrc/attn_bwd_d128.cu).

A CTA walks items (one 128-key tile and its nq query tiles). Per step g (running over the
CTA's items) the producer loads Q, dO, LSE, D into stage g % 2, and K, V once per item; the
MMA issuer runs S^T, dP^T, dV += P^T dO, dK += dS^T Q and dQ^T = K^T dS^T; two P / dS
groups read S^T and dP^T from TMEM, write P^T and dS^T back to TMEM and dS^T into the dO
buffer of the stage; the drain group reads dQ^T out of TMEM. Two TMEM regions swap roles
every step (S^T -> P^T -> dQ^T, and dP^T -> the next S^T). At the end of an item the P / dS
and drain groups write dV / dK from TMEM (after mma_done) and hand the accumulators back
(dv_free / dk_free); the producer replaces K, V after kv_empty.

Checked under random timings for walks of random items: nothing deadlocks, no barrier
phase is over-arrived, no copy lands in a shared-memory buffer an MMA or a P / dS group
still reads, no MMA writes a TMEM region or accumulator that a group still reads, and no
P / dS group writes dS^T into a dO buffer an MMA still reads. Negative controls: without
the dp_read wait the next S^T overwrites dP^T while it is being read, and without
dk_free the next item's first dK overwrites dK while the drain group's epilogue reads it.
(The kernel's dv_free wait is implied by p_full: the next item's first dV waits for the
P / dS groups' first p_full of that item, which they arrive only after their dV
epilogue; the model finds no hazard without it.)
"""
import random

import pytest


class OverArrival(Exception):
    pass


class Deadlock(Exception):
    pass


class Hazard(Exception):
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
        return (self.done & 1) != parity


def simulate(items, seed, dp_read_wait=True, dv_free_wait=True, dk_free_wait=True):
    """items: the nq (query tiles) of each item of one CTA's walk."""
    rnd = random.Random(seed)
    bars = {n: Barrier() for n in ("kv_full", "kv_empty", "q_full0", "q_full1", "q_empty0", "q_empty1",
                                    "s_full", "dp_full", "dv_done", "dq_full", "mma_done", "drain")}
    for n in ("p_full", "dp_read", "dss_full", "dv_free"):
        bars[n] = Barrier(2)          # both P / dS groups arrive
    bars["r_free"], bars["dk_free"] = Barrier(1), Barrier(1)
    now = [0]
    events = []
    pipe = []
    busy_until = [0]
    # readers of shared-memory buffers (MMAs and groups) and of TMEM regions / accumulators
    smem_readers = {b: 0 for b in ("K", "V", "Q0", "Q1", "dO0", "dO1")}
    tmem_readers = {b: 0 for b in ("R0", "R1", "dV", "dK")}

    def copy(bar, bufs):
        for b in bufs:
            if smem_readers[b]:
                raise Hazard("copy into %s while it is read" % b)
        events.append((now[0] + rnd.randint(50, 3000), lambda: bars[bar].complete_tx(1)))

    def run_pipe():
        while pipe and busy_until[0] <= now[0]:
            kind, arg = pipe.pop(0)
            if kind == "mma":
                reads, writes = arg
                for b in writes:
                    if tmem_readers.get(b, 0):
                        raise Hazard("MMA writes %s while a group reads it" % b)
                for b in reads:
                    smem_readers[b] += 1
                busy_until[0] = max(now[0], busy_until[0]) + rnd.randint(200, 600)

                def finish(rs=reads):
                    for b in rs:
                        smem_readers[b] -= 1
                events.append((busy_until[0], finish))
            else:
                events.append((busy_until[0] + 1, lambda b=arg: bars[b].arrive()))

    def producer():
        g = 0
        for ic, nq in enumerate(items):
            for i in range(nq):
                s = g & 1
                if g >= 2:
                    yield ("wait", "q_empty%d" % s, ((g >> 1) - 1) & 1)
                bars["q_full%d" % s].expect_tx(1)
                copy("q_full%d" % s, ["Q%d" % s, "dO%d" % s])
                if i == 0:
                    if ic > 0:
                        yield ("wait", "kv_empty", (ic - 1) & 1)
                    bars["kv_full"].expect_tx(1)
                    copy("kv_full", ["K", "V"])
                g += 1

    def mma():
        g0 = 0
        for ic, nq in enumerate(items):
            yield ("wait", "kv_full", ic & 1)
            yield ("wait", "q_full%d" % (g0 & 1), (g0 >> 1) & 1)
            if g0 > 0:
                if dp_read_wait:
                    yield ("wait", "dp_read", (g0 - 1) & 1)
                yield ("wait", "r_free", (g0 - 1) & 1)
            pipe.append(("mma", (["K", "Q%d" % (g0 & 1)], ["R%d" % (g0 & 1)])))          # S^T
            pipe.append(("commit", "s_full"))
            pipe.append(("mma", (["V", "dO%d" % (g0 & 1)], ["R%d" % ((g0 + 1) & 1)])))    # dP^T
            pipe.append(("commit", "dp_full"))
            for i in range(nq):
                g = g0 + i
                s = g & 1
                rA, rB = "R%d" % (g & 1), "R%d" % ((g + 1) & 1)
                yield ("wait", "p_full", g & 1)
                if i == 0 and ic > 0 and dv_free_wait:
                    yield ("wait", "dv_free", (ic - 1) & 1)
                pipe.append(("mma", (["dO%d" % s], ["dV"])))                               # dV += P^T dO
                pipe.append(("commit", "dv_done"))
                if i + 1 < nq:
                    yield ("wait", "q_full%d" % ((g + 1) & 1), ((g + 1) >> 1) & 1)
                    if dp_read_wait:
                        yield ("wait", "dp_read", g & 1)
                    pipe.append(("mma", (["K", "Q%d" % ((g + 1) & 1)], [rB])))             # S^T_{i+1}
                    pipe.append(("commit", "s_full"))
                yield ("wait", "dss_full", g & 1)
                if i == 0 and ic > 0 and dk_free_wait:
                    yield ("wait", "dk_free", (ic - 1) & 1)
                pipe.append(("mma", (["Q%d" % s], ["dK"])))                                # dK += dS^T Q
                pipe.append(("mma", (["K", "dO%d" % s], [rA])))                            # dQ^T (dS^T in dO)
                pipe.append(("commit", "dq_full"))
                pipe.append(("commit", "q_empty%d" % s))
                if i + 1 < nq:
                    yield ("wait", "r_free", g & 1)
                    pipe.append(("mma", (["V", "dO%d" % ((g + 1) & 1)], [rA])))            # dP^T_{i+1}
                    pipe.append(("commit", "dp_full"))
            pipe.append(("commit", "kv_empty"))
            pipe.append(("commit", "mma_done"))
            g0 += nq
        pipe.append(("commit", "drain"))
        yield ("wait", "drain", 0)

    def pds(wg):
        g0 = 0
        for ic, nq in enumerate(items):
            for i in range(nq):
                g = g0 + i
                s = g & 1
                rA, rB = "R%d" % (g & 1), "R%d" % ((g + 1) & 1)
                yield ("wait", "q_full%d" % s, (g >> 1) & 1)
                smem_readers["Q%d" % s] += 1            # LSE / D of the stage
                yield ("wait", "s_full", g & 1)
                tmem_readers[rA] += 1
                yield ("delay", rnd.randint(300, 1500))    # P from S^T, P^T back to TMEM
                tmem_readers[rA] -= 1
                bars["p_full"].arrive()
                yield ("wait", "dp_full", g & 1)
                tmem_readers[rB] += 1
                yield ("delay", rnd.randint(100, 600))
                tmem_readers[rB] -= 1
                bars["dp_read"].arrive()
                yield ("delay", rnd.randint(100, 800))     # dS, dS^T to TMEM
                yield ("wait", "dv_done", g & 1)
                if smem_readers["dO%d" % s]:
                    raise Hazard("dS^T written into dO%d while an MMA reads it" % s)
                yield ("delay", rnd.randint(50, 300))
                smem_readers["Q%d" % s] -= 1
                bars["dss_full"].arrive()
            yield ("wait", "mma_done", ic & 1)
            tmem_readers["dV"] += 1
            yield ("delay", rnd.randint(200, 1500))
            tmem_readers["dV"] -= 1
            bars["dv_free"].arrive()
            g0 += nq

    def drain():
        g0 = 0
        for ic, nq in enumerate(items):
            for i in range(nq):
                g = g0 + i
                rA = "R%d" % (g & 1)
                yield ("wait", "dq_full", g & 1)
                tmem_readers[rA] += 1
                yield ("delay", rnd.randint(100, 500))
                tmem_readers[rA] -= 1
                bars["r_free"].arrive()
                yield ("delay", rnd.randint(200, 2500))    # the bulk reductions
            yield ("wait", "mma_done", ic & 1)
            tmem_readers["dK"] += 1
            yield ("delay", rnd.randint(200, 1500))
            tmem_readers["dK"] -= 1
            bars["dk_free"].arrive()
            g0 += nq

    agents = {"prod": producer(), "mma": mma(), "pds0": pds(0), "pds1": pds(1), "drain": drain()}
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

    for _ in range(400000):
        if not alive:
            return
        while True:
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


@pytest.mark.parametrize("walk_seed", range(8))
def test_backward_walk_random_items(walk_seed):
    """Walks of 1-6 items of 1-16 query tiles each (one-tile items, odd and even step
    counts, so the Q / dO stage and TMEM region of an item's first step take both
    parities), three timing seeds each."""
    rnd = random.Random(2000 + walk_seed)
    for _ in range(5):
        items = [rnd.randint(1, 16) for _ in range(rnd.randint(1, 6))]
        for seed in range(3):
            simulate(items, seed)


def test_backward_walk_short_items():
    """Runs of one- and two-step items, where the item hand-offs (kv_empty, dv_free,
    dk_free, the first S^T / dP^T into the regions the previous step left) follow each
    other most closely."""
    for items in ([1] * 8, [2, 1, 2, 1, 2], [1, 16, 1, 1], [3, 1, 1, 2]):
        for seed in range(5):
            simulate(items, seed)


def test_backward_walk_negative_controls():
    """Without the dp_read wait the next S^T can overwrite dP^T while the P / dS groups
    read it; without dk_free the next item's first dK can overwrite dK during the drain
    group's epilogue. Without dv_free nothing breaks (implied by p_full)."""
    rnd = random.Random(9)
    caught = {"dp_read": 0, "dk_free": 0, "dv_free": 0}
    for _ in range(40):
        items = [rnd.randint(1, 4) for _ in range(4)]
        for seed in range(2):
            for key, kw in (("dp_read", dict(dp_read_wait=False)), ("dk_free", dict(dk_free_wait=False)),
                            ("dv_free", dict(dv_free_wait=False))):
                try:
                    simulate(items, seed, **kw)
                except (Hazard, OverArrival, Deadlock):
                    caught[key] += 1
    assert caught["dp_read"] > 0 and caught["dk_free"] > 0, caught
    assert caught["dv_free"] == 0, caught
