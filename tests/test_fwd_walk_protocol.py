"""CPU model of the walking forward kernel's barrier protocol (csrc/attn_fwd.cu, the form
in which one CTA per SM computes several query-tile pairs in turn).

Per CTA: a Q producer, a K producer, a V producer, the MMA issuer and two softmax
groups, synchronised by mbarriers with parity waits; copies land after random delays
and the tensor core runs MMAs in issue order, each commit arriving once everything
issued before it has completed. The Q producer claims the CTA's items one at a time and
publishes each through a 4-slot ring in shared memory (item_full, item_empty with one
arrival per reading role), closed by an end marker; every other role takes its items
from that ring. Across the items (query-tile pairs of any sequence) a CTA walks:
  * the K / V rings continue with a running ring index;
  * Q of tile t is reloaded once the last S of tile t of the previous item has completed:
    the softmax thread that sees that S's commit relays it (q_empty);
  * a value tile whose last reader no later S commit of the item covers (the item's
    last one, and tile 0's last one when tile 1's document starts at tile 1) is relayed
    after that tile's pv_done;
  * the first O += P V of tile t of an item overwrites O_t; it needs no barrier of its
    own: it waits for that item's first P of tile t, which the tile's softmax group
    writes only after its epilogue of the previous item has read O_t out.
Checked, for random walks of items with random document starts and timing seeds:
nothing deadlocks, no barrier phase is over-arrived, no copy lands in a buffer an
unfinished MMA still reads, no S MMA overwrites S / P of a tile while its softmax still
reads it, and no PV writes O_t while an epilogue still reads it. Negative controls: the
walk deadlocks without tile 0's end-of-item value relay, and a Q copy lands on a Q
still being read without the q_empty wait.
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

    def arrive(self, n=1):
        self.pending -= n
        self._check()

    def expect_tx(self, nbytes):
        self.tx += nbytes
        self.pending -= 1
        self._check()

    def complete_tx(self, nbytes):
        self.tx -= nbytes
        self._check()

    def test(self, parity):
        """try_wait.parity: true once the phase of that parity has completed (valid while
        the completed-phase count is parity's phase or one more)."""
        return (self.done & 1) != parity


def make_item(nqt, u, lo0, lo1):
    has1 = 2 * u + 1 < nqt
    hi0, hi1 = 2 * u, 2 * u + 1
    return dict(has1=has1, lo0=lo0, lo1=lo1, hi0=hi0, hi1=hi1, J0=lo0,
                NJ=(hi1 if has1 else hi0) - lo0 + 1)


def tiles(it):
    return (0, 1) if it["has1"] else (0,)


N_READERS = 5     # K producer, V producer, MMA issuer, two softmax groups
RING = 4


def simulate_walk(items, seed, tile0_v_relay=True, q_empty_wait=True):
    rnd = random.Random(seed)
    names = ["q0", "q1", "k0", "k1", "v0", "v1", "s0", "s1", "pv0", "pv1", "drain",
             "qe0", "qe1", "ke0", "ke1", "ve0", "ve1"]
    bars = {n: Barrier() for n in names}
    for i in range(RING):
        bars["if%d" % i] = Barrier()
        bars["ie%d" % i] = Barrier(N_READERS)
    ring = [None] * RING
    bars["p0"], bars["p1"] = Barrier(), Barrier()       # one arrival per softmax group in the model
    now = [0]
    events = []
    pipe = []
    busy_until = [0]
    readers = {("q", 0): 0, ("q", 1): 0, ("k", 0): 0, ("k", 1): 0, ("v", 0): 0, ("v", 1): 0}
    in_p_phase = [False, False]     # softmax t between its s_full wait and its p_full arrive
    o_reading = [False, False]      # epilogue t between its pv_done wait and its o_free arrive

    def copy(bar, stage):
        if readers[stage]:
            raise Hazard("copy into %s while an MMA reads it" % (stage,))
        events.append((now[0] + rnd.randint(50, 3000), lambda: bars[bar].complete_tx(1)))

    def run_pipe():
        while pipe and busy_until[0] <= now[0]:
            kind, arg = pipe.pop(0)
            if kind == "mma":
                stages, writes = arg
                for st in stages:
                    readers[st] += 1
                if writes[0] == "S" and in_p_phase[writes[1]]:
                    raise Hazard("S_%d overwritten while its softmax reads it" % writes[1])
                if writes[0] == "O" and o_reading[writes[1]]:
                    raise Hazard("O_%d written while its epilogue reads it" % writes[1])
                busy_until[0] = max(now[0], busy_until[0]) + rnd.randint(300, 700)

                def finish(sts=stages):
                    for st in sts:
                        readers[st] -= 1
                events.append((busy_until[0], finish))
            else:
                events.append((busy_until[0] + 1, lambda b=arg: bars[b].arrive()))

    def publish(n, value):
        slot = n % RING
        if n >= RING:
            yield ("wait", "ie%d" % slot, ((n // RING) - 1) & 1)
        ring[slot] = value
        bars["if%d" % slot].arrive()

    def take(n):
        """A reading role's n-th item from the ring (None: the end marker)."""
        slot = n % RING
        yield ("wait", "if%d" % slot, (n // RING) & 1)
        value = ring[slot]
        bars["ie%d" % slot].arrive()
        return value

    def q_producer():
        n_t = [0, 0]
        for n, it in enumerate(items):
            yield from publish(n, it)
            for t in tiles(it):
                if n_t[t] > 0 and q_empty_wait:
                    yield ("wait", "qe%d" % t, (n_t[t] - 1) & 1)
                bars["q%d" % t].expect_tx(1)
                copy("q%d" % t, ("q", t))
                n_t[t] += 1
        yield from publish(len(items), None)

    def ring_producer(kind):
        jg = 0
        n_item = 0
        while True:
            it = yield from take(n_item)
            if it is None:
                break
            n_item += 1
            for j in range(it["NJ"]):
                s = jg & 1
                if jg >= 2:
                    yield ("wait", "%se%d" % (kind, s), ((jg >> 1) - 1) & 1)
                bars["%s%d" % (kind, s)].expect_tx(1)
                copy("%s%d" % (kind, s), (kind, s))
                jg += 1

    def mma():
        jg0 = 0
        n_t = [0, 0]            # items with tile t so far
        ns, npv = [0, 0], [0, 0]
        n_item = 0
        while True:
            it = yield from take(n_item)
            if it is None:
                break
            n_item += 1
            first_pv, first_s = [True, True], [True, True]
            for j in range(it["NJ"] + 1):
                kt = it["J0"] + j
                for t in tiles(it):
                    lo_t, hi_t = (it["lo1"], it["hi1"]) if t else (it["lo0"], it["hi0"])
                    if j >= 1 and lo_t <= kt - 1 <= hi_t:            # O_t += P_t V
                        jv = jg0 + j - 1
                        yield ("wait", "v%d" % (jv & 1), (jv >> 1) & 1)
                        yield ("wait", "p%d" % t, npv[t] & 1)
                        pipe.append(("mma", ([("v", jv & 1)], ("O", t))))
                        if kt - 1 == hi_t:
                            pipe.append(("commit", "pv%d" % t))
                        first_pv[t] = False
                        npv[t] += 1
                    if j < it["NJ"] and lo_t <= kt <= hi_t:           # S_t = Q_t K^T
                        jk = jg0 + j
                        yield ("wait", "k%d" % (jk & 1), (jk >> 1) & 1)
                        if first_s[t]:
                            yield ("wait", "q%d" % t, n_t[t] & 1)
                        pipe.append(("mma", ([("k", jk & 1), ("q", t)], ("S", t))))
                        pipe.append(("commit", "s%d" % t))
                        first_s[t] = False
                        ns[t] += 1
            for t in tiles(it):
                n_t[t] += 1
            jg0 += it["NJ"]
        pipe.append(("commit", "drain"))
        yield ("wait", "drain", 0)

    def softmax(t):
        jg0 = 0
        n_t = 0
        ns = 0
        n_item = 0
        while True:
            it = yield from take(n_item)
            if it is None:
                break
            n_item += 1
            if t in tiles(it):
                lo_t, hi_t = (it["lo1"], it["hi1"]) if t else (it["lo0"], it["hi0"])
                nt = hi_t - lo_t + 1
                last_t = 1 if it["has1"] else 0
                for i in range(nt):
                    yield ("wait", "s%d" % t, ns & 1)
                    ns += 1
                    in_p_phase[t] = True
                    kt = lo_t + i
                    jk = jg0 + kt - it["J0"]
                    if t == 1 or not (it["has1"] and kt >= it["lo1"]):
                        bars["ke%d" % (jk & 1)].arrive()
                    if i >= 1 and (t == 1 or not (it["has1"] and kt - 1 >= it["lo1"])):
                        bars["ve%d" % ((jk - 1) & 1)].arrive()
                    if i == nt - 1:
                        bars["qe%d" % t].arrive()
                    yield ("delay", rnd.randint(200, 1500))
                    in_p_phase[t] = False
                    bars["p%d" % t].arrive()
                yield ("wait", "pv%d" % t, n_t & 1)
                o_reading[t] = True
                # Value tile hi_t when no S commit of the item covers its last reader: the
                # item's last value tile, and tile 0's last one when tile 1 reads none of it.
                if t == last_t or (tile0_v_relay and t == 0 and it["has1"] and it["lo1"] > it["hi0"]):
                    bars["ve%d" % ((jg0 + hi_t - it["J0"]) & 1)].arrive()
                yield ("delay", rnd.randint(100, 2000))
                o_reading[t] = False
                yield ("delay", rnd.randint(100, 1500))   # the O / LSE stores
                n_t += 1
            jg0 += it["NJ"]

    agents = {"qp": q_producer(), "kp": ring_producer("k"), "vp": ring_producer("v"), "mma": mma(),
              "sm0": softmax(0), "sm1": softmax(1)}
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


def random_item(rnd, max_nqt=16):
    nqt = rnd.randint(1, max_nqt)
    u = rnd.randint(0, (nqt + 1) // 2 - 1)
    lo0 = rnd.randint(0, 2 * u) if rnd.random() < 0.5 else 0
    lo1 = rnd.randint(lo0, 2 * u + 1) if rnd.random() < 0.5 else lo0
    return make_item(nqt, u, lo0, lo1)


@pytest.mark.parametrize("walk_seed", range(12))
def test_walk_protocol_random_walks(walk_seed):
    """Walks of 1-7 items drawn from sequences of 1-16 query tiles, with random document
    starts, each under three timing seeds."""
    rnd = random.Random(1000 + walk_seed)
    for _ in range(6):
        items = [random_item(rnd) for _ in range(rnd.randint(1, 7))]
        for seed in range(3):
            simulate_walk(items, seed)


def test_walk_protocol_single_tiles_and_odd_counts():
    """Items with tile 1 absent (odd tile counts) next to full pairs, and one-key-tile
    pairs, in every order."""
    a = make_item(1, 0, 0, 0)          # one tile, one key tile
    b = make_item(3, 1, 0, 0)          # tile 2 alone, key tiles 0..2
    c = make_item(4, 1, 2, 3)          # documents start at both tiles: one key tile each
    d = make_item(16, 7, 0, 0)         # the longest pair
    for items in ([a, a, a], [b, d, a], [c, c, b, a], [d, c, d], [a, d, a, d]):
        for seed in range(4):
            simulate_walk(items, seed)


def test_walk_protocol_negative_controls():
    """Without tile 0's end-of-item relay of its last value tile (when tile 1's document
    starts at tile 1) the next item's V loads never get that ring stage back; without
    the q_empty wait a Q copy overwrites Q while the previous item's S still reads it."""
    a = make_item(4, 1, 0, 3)      # tile 1's document starts at tile 1: value tile 2 read by tile 0 only
    b = make_item(4, 1, 0, 0)
    with pytest.raises(Deadlock):
        simulate_walk([a, b, b], 0, tile0_v_relay=False)
    simulate_walk([a, b, b], 0)
    rnd = random.Random(3)
    caught = 0
    for _ in range(20):
        items = [random_item(rnd, 16) for _ in range(4)]
        for seed in range(3):
            try:
                simulate_walk(items, seed, q_empty_wait=False)
            except (Hazard, OverArrival):
                caught += 1
    assert caught > 0



def items_from_offsets(offsets, B, L):
    """The forward's work items of a document-masked batch: per sequence b and pair u, the
    key-tile ranges from the document starts of the pair's first rows (as the kernel
    derives them from cu_doc_offsets)."""
    import bisect
    nqt = (L + 127) // 128
    out = []
    for b in range(B):
        seq0 = b * L

        def doc_start(row):
            t = seq0 + row
            i = bisect.bisect_right(offsets, t) - 1
            return max(offsets[i], seq0) - seq0 if i >= 0 else 0

        for u in range((nqt + 1) // 2 - 1, -1, -1):
            r1 = min((2 * u + 1) * 128, L - 1)
            out.append(make_item(nqt, u, doc_start(2 * u * 128) // 128, doc_start(r1) // 128))
    return out


@pytest.mark.parametrize("kind", ["dm", "pack"])
def test_walk_protocol_on_document_masked_batches(kind):
    """Items of the DM and Pack-8k steps the benchmark times (8 x 8192), walked in the
    orders a CTA meets them: runs of consecutive claims and strided picks."""
    from paper_2405_13226_gb300 import workloads as wl
    for seed in range(2):
        off = (wl.concat_and_chunk_offsets(seed) if kind == "dm" else wl.packed_dm_offsets(seed)).tolist()
        items = items_from_offsets(off, 8, 8192)
        rnd = random.Random(seed)
        for start in rnd.sample(range(len(items) - 6), 4):
            simulate_walk(items[start:start + 6], seed)
        simulate_walk(items[seed::37][:6], seed + 1)
