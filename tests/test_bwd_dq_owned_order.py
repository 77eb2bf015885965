"""CPU model of the dQ-owned walk of the short-sequence backward kernel
(csrc/attn_bwd_d128_persist.cu with dq_owned; order in csrc/bwd_d128.cuh, bwd_walk_item).

A CTA owns whole (sequence, head) pairs and walks each one's key tiles from the last to
the first; key tile n's item has a step per live query tile n .. hi(n). Each drain warp
issues one bulk group per 32-row block of a step into the CTA's own fp32 slot: a plain
store on the item's first step (the diagonal query tile), a reduce-add on the others,
each add preceded by `cp.async.bulk.wait_group 7`. After an item it waits for all its
groups (`wait_group 0`) and converts the query tiles whose last contributor is that key
tile (the tile holding the document start of the query tile's first row).

The model runs one drain warp's issue sequence with random bulk-group latencies
(completion in any order; `wait_group N` blocks until all but the N most recent groups
are complete) and checks, for random sequence lengths, document layouts and pair
counts: a query tile's first partial is the store of its diagonal step; no add is
issued before the store of the same block has completed; a converted tile has received
every partial of its pair and all of them have completed; no store into the slot is
issued while a group of the previous pair on the same block is still pending. Negative
control: without the wait before an add, adds overtake their store.
The barrier protocol of the same walks runs through the discrete-event model of
tests/test_bwd_walk_protocol.py.
"""
import random

import pytest

from test_bwd_walk_protocol import simulate

BQ = 128


def doc_start(starts, t):
    return max(s for s in starts if s <= t)


def doc_end(starts, t, L):
    later = [s for s in starts if s > t]
    return min(later) if later else L


def walk_items(L, starts):
    """Items of one (sequence, head) pair in the dQ-owned order: (key tile n, [query tiles])."""
    nkt = (L + BQ - 1) // BQ
    items = []
    for n in range(nkt - 1, -1, -1):
        kv_last = min(n * BQ + BQ - 1, L - 1)
        hi = (doc_end(starts, kv_last, L) - 1) // BQ
        items.append((n, list(range(n, hi + 1))))
    return items


def last_contributor(L, starts, qt):
    return doc_start(starts, qt * BQ) // BQ


def random_docs(rnd, L):
    k = rnd.choice([0, 0, 1, 2, 5, 12])
    return sorted({0} | {rnd.randrange(1, L) for _ in range(k)}) if L > 1 else [0]


class Hazard(Exception):
    pass


def run_drain(pairs, seed, wait_before_add=7):
    """pairs: list of (L, doc starts) owned one after the other by one CTA (one slot)."""
    rnd = random.Random(seed)
    now = 0
    groups = []            # dicts: key, kind, pair, done_at
    received = {}          # (pair, qt) -> partials issued

    def wait_group(n):
        nonlocal now
        pending = groups[:-n] if n else groups[:]
        for g in pending:
            now = max(now, g["done_at"])

    def issue(kind, key, pair):
        nonlocal now
        now += rnd.randint(1, 30)
        for g in groups:
            if g["key"] == key and g["done_at"] > now:
                if kind == "store" and g["pair"] != pair:
                    raise Hazard("store into the slot over a pending group of the previous pair")
                if kind == "add" and g["kind"] == "store":
                    raise Hazard("add issued before the store of %s completed" % (key,))
        groups.append({"key": key, "kind": kind, "pair": pair, "done_at": now + rnd.randint(50, 4000)})

    for pi, (L, starts) in enumerate(pairs):
        items = walk_items(L, starts)
        seen = set()
        touches = {}
        for n, qts in items:
            for qt in qts:
                touches[qt] = touches.get(qt, 0) + 1
        for n, qts in items:
            for i, qt in enumerate(qts):
                if qt not in seen:
                    assert i == 0 and qt == n, "first partial of tile %d is not its diagonal step" % qt
                    seen.add(qt)
                for c in range(4):
                    key = (qt, c)
                    if i == 0:
                        issue("store", key, pi)
                    else:
                        if wait_before_add is not None:
                            wait_group(wait_before_add)
                        issue("add", key, pi)
                    received[(pi, qt)] = received.get((pi, qt), 0) + 1
            done = [qt for qt in qts if last_contributor(L, starts, qt) == n]
            if done:
                wait_group(0)
                for qt in done:
                    if received[(pi, qt)] != 4 * touches[qt]:
                        raise Hazard("tile %d converted before all its partials were issued" % qt)
                    for g in groups:
                        if g["key"][0] == qt and g["pair"] == pi and g["done_at"] > now:
                            raise Hazard("tile %d converted with a pending group" % qt)
                now += rnd.randint(100, 2000)      # the conversion reads
        for qt in touches:
            assert any(last_contributor(L, starts, qt) == n for n, qts in items if qt in qts)


@pytest.mark.parametrize("seed", range(6))
def test_dq_owned_order_random_pairs(seed):
    """Random sequence lengths (1 .. 1024 tokens: 1 .. 8 key tiles, ragged ends), random
    document layouts and several owned pairs per slot."""
    rnd = random.Random(500 + seed)
    for _ in range(30):
        pairs = []
        for _ in range(rnd.randint(1, 4)):
            L = rnd.choice([1, 7, 128, 200, 256, 384, 512, 700, 1000, 1024])
            pairs.append((L, random_docs(rnd, L)))
        for s in range(3):
            run_drain(pairs, seed * 100 + s)


def test_dq_owned_order_negative_control():
    """Issuing the adds without waiting lets an add overtake its tile's store."""
    rnd = random.Random(7)
    caught = 0
    for s in range(40):
        L = rnd.choice([256, 512, 1024])
        try:
            run_drain([(L, [0]), (L, random_docs(rnd, L))], s, wait_before_add=None)
        except Hazard:
            caught += 1
    assert caught > 0


def test_dq_owned_walks_barrier_protocol():
    """The barrier protocol of the walking kernel over dQ-owned item sequences (key tiles
    last to first, so step counts 1, 2, ..., nkt per pair without documents)."""
    rnd = random.Random(3)
    shapes = [[1, 2] * 4, list(range(1, 9)) * 2, [1, 2, 3, 4] * 3]
    for _ in range(4):
        L = rnd.choice([300, 640, 1024])
        shapes.append([len(q) for _, q in walk_items(L, random_docs(rnd, L))] * 2)
    for items in shapes:
        for seed in range(3):
            simulate(items, seed)
