"""A host model of the persistent kernel's in-CTA barrier protocol, run under
random interleavings (no GPU).

The model follows the kernel's roles and mbarriers: the claimer's
descriptor ring and publish ring, the producer's Q buffers and K stages, two
UMMA warps (one per epilogue warpgroup, tile t of a chunk to warp t % 2) with
their TMEM buffers, and eight epilogue warps with their warpgroup and
all-warp syncs.  Barriers keep an arrival count, a transaction count and a
phase; a wait on parity P passes when P differs from the parity of the
current phase (the PTX rule), so a waiter that falls two phases behind -- or
runs two ahead -- is misled.  TMA copies and UMMA completions are
asynchronous events.  The model checks that no barrier gets more arrivals
than its count allows and that every role finishes.

It pins the K-ring layout: with one shared ring (stage = tile % stages), a
UMMA warp that skipped the other warp's tiles at an odd-sized chunk can wait
on a stage whose previous fill has not landed and take that older phase for
its own -- which the model finds; with one sub-ring per UMMA warp (the
kernel's layout) it finds nothing.
"""
import random

import pytest


class _Bar:
    def __init__(self, name, count):
        self.name, self.count = name, count
        self.pending, self.tx, self.phase = count, 0, 0

    def arrive(self, tx=0):
        self.pending -= 1
        self.tx += tx
        if self.pending < 0:
            raise AssertionError(f"{self.name}: more arrivals than its count")
        self._complete()

    def land(self):
        self.tx -= 1
        if self.tx < 0:
            raise AssertionError(f"{self.name}: more bytes than expected")
        self._complete()

    def _complete(self):
        if self.pending == 0 and self.tx == 0:
            self.phase += 1
            self.pending = self.count

    def passes(self, parity):
        return parity != (self.phase & 1)


def _simulate(seed, stages, q_bufs, bufs_per_wg, sub_rings, n_chunks=30, pub=6, descs=4):
    rng = random.Random(seed)
    bars = {}

    def mk(name, count):
        bars[name] = _Bar(name, count)

    for i in range(stages):
        mk(f"full{i}", 1)
        mk(f"empty{i}", 1)
    for b in range(2 * bufs_per_wg):
        mk(f"tfull{b}", 1)
        mk(f"tempty{b}", 4)
    for i in range(descs):
        mk(f"dfull{i}", 1)
        mk(f"dempty{i}", 3 + 8)
    for i in range(q_bufs):
        mk(f"qfull{i}", 1)
        mk(f"qempty{i}", 2)
    for w in range(2):
        mk(f"wg{w}", 4)
    mk("epi", 8)
    for i in range(pub):
        mk(f"pubfull{i}", 8)
        mk(f"pubempty{i}", 1)
    # chunks: (pass, tiles), with the short and odd-sized ones of ragged units
    chunks = [(rng.choice((1, 2)), rng.choice((1, 1, 2, 3, 5, 7, 16, 16))) for _ in range(n_chunks)]
    ring = [None] * descs
    events = []
    clock = [0]

    def after(fn, lo=1, hi=30, at=None):
        events.append((clock[0] + rng.randint(lo, hi) if at is None else at, fn))

    def wait(name, parity):
        return ("wait", name, parity)

    def claimer():
        issued = nxt = 0

        def pump():
            nonlocal nxt
            while nxt < issued and bars[f"pubfull{nxt % pub}"].passes((nxt // pub) & 1):
                bars[f"pubempty{nxt % pub}"].arrive()
                nxt += 1

        for c in range(n_chunks + 1):
            ds = c % descs
            while not bars[f"dempty{ds}"].passes(((c // descs) & 1) ^ 1):
                pump()
                yield ("spin",)
            while issued - nxt > pub - 1:
                pump()
                yield ("spin",)
            ring[ds] = None if c == n_chunks else chunks[c]
            issued += c < n_chunks
            bars[f"dfull{ds}"].arrive()
            yield ("spin",)
        while nxt < issued:
            pump()
            yield ("spin",)

    def stage_of(w, slot):
        return w + 2 * slot if sub_rings else slot

    def producer():
        slot, ph = [0, 0], [0, 0]
        shared_slot, shared_ph = 0, 0
        qb = qph = 0
        for c in range(n_chunks + 1):
            ds = c % descs
            yield wait(f"dfull{ds}", (c // descs) & 1)
            d = ring[ds]
            bars[f"dempty{ds}"].arrive()
            if d is None:
                return
            yield wait(f"qempty{qb}", qph ^ 1)
            bars[f"qfull{qb}"].arrive(tx=1)
            after(lambda q=qb: bars[f"qfull{q}"].land())
            qb, qph = (0, qph ^ 1) if qb + 1 == q_bufs else (qb + 1, qph)
            for t in range(d[1]):
                w = t & 1
                if sub_rings:
                    st, p = stage_of(w, slot[w]), ph[w]
                else:
                    st, p = shared_slot, shared_ph
                yield wait(f"empty{st}", p ^ 1)
                bars[f"full{st}"].arrive(tx=1)
                after(lambda s=st: bars[f"full{s}"].land())
                if sub_rings:
                    slot[w] += 1
                    if slot[w] == stages // 2:
                        slot[w], ph[w] = 0, ph[w] ^ 1
                else:
                    shared_slot += 1
                    if shared_slot == stages:
                        shared_slot, shared_ph = 0, shared_ph ^ 1

    def mma(mw):
        slot = ph = qb = qph = used = 0
        busy_until = 0
        for c in range(n_chunks + 1):
            ds = c % descs
            yield wait(f"dfull{ds}", (c // descs) & 1)
            d = ring[ds]
            bars[f"dempty{ds}"].arrive()
            if d is None:
                return
            yield wait(f"qfull{qb}", qph)
            for t in range(d[1]):
                if (t & 1) != mw:
                    if not sub_rings:  # the shared ring advances for every tile
                        slot += 1
                        if slot == stages:
                            slot, ph = 0, ph ^ 1
                    continue
                b = mw + 2 * (used % bufs_per_wg)
                yield wait(f"tempty{b}", ((used // bufs_per_wg) & 1) ^ 1)
                used += 1
                st = stage_of(mw, slot)
                yield wait(f"full{st}", ph)
                busy_until = max(clock[0], busy_until) + rng.randint(1, 10)
                after(lambda s=st: bars[f"empty{s}"].arrive(), at=busy_until)
                after(lambda x=b: bars[f"tfull{x}"].arrive(), at=busy_until)
                slot += 1
                if slot == (stages // 2 if sub_rings else stages):
                    slot, ph = 0, ph ^ 1
            after(lambda q=qb: bars[f"qempty{q}"].arrive(), at=max(clock[0], busy_until) + 1)
            qb, qph = (0, qph ^ 1) if qb + 1 == q_bufs else (qb + 1, qph)

    def epilogue(wg):
        used = syncs = syncs8 = 0
        for ci in range(n_chunks + 1):
            ds = ci % descs
            yield wait(f"dfull{ds}", (ci // descs) & 1)
            d = ring[ds]
            bars[f"dempty{ds}"].arrive()
            if d is None:
                return
            for _ in range(wg, d[1], 2):
                b = wg + 2 * (used % bufs_per_wg)
                yield wait(f"tfull{b}", (used // bufs_per_wg) & 1)
                used += 1
                yield ("spin",)
                bars[f"tempty{b}"].arrive()
            if d[0] == 1:  # pass 1: two warpgroup syncs
                for _ in range(2):
                    bars[f"wg{wg}"].arrive()
                    yield wait(f"wg{wg}", syncs & 1)
                    syncs += 1
            else:  # pass 2: one all-epilogue sync
                bars["epi"].arrive()
                yield wait("epi", syncs8 & 1)
                syncs8 += 1
            if ci >= pub:
                yield wait(f"pubempty{ci % pub}", (ci // pub - 1) & 1)
            bars[f"pubfull{ci % pub}"].arrive()

    roles = {"claimer": claimer(), "producer": producer(), "mma0": mma(0), "mma1": mma(1)}
    for wg in range(2):
        for w in range(4):
            roles[f"epi{wg}.{w}"] = epilogue(wg)
    state = dict.fromkeys(roles)
    alive = set(roles)
    for _ in range(400_000):
        if not alive and not events:
            return True
        runnable = [n for n in alive if state[n] is None or state[n][0] == "spin" or
                    bars[state[n][1]].passes(state[n][2])]
        if runnable and (not events or rng.random() < 0.7):
            n = rng.choice(sorted(runnable))
            try:
                state[n] = next(roles[n])
            except StopIteration:
                alive.discard(n)
        elif events:
            events.sort(key=lambda e: e[0])
            t, fn = events.pop(0)
            clock[0] = max(clock[0], t)
            fn()
        else:
            raise AssertionError(f"deadlock: {sorted((n, state[n]) for n in alive)}")
    raise AssertionError("no progress (spinning roles only)")


@pytest.mark.parametrize("stages,q_bufs,bufs_per_wg,descs", [(2, 2, 4, 2), (4, 2, 4, 2), (4, 3, 2, 2),
                                                             (8, 2, 1, 2), (6, 3, 4, 2), (4, 2, 4, 4),
                                                             (2, 3, 2, 4)])
def test_sub_rings_survive_random_interleavings(stages, q_bufs, bufs_per_wg, descs):
    for seed in range(25):
        assert _simulate(seed, stages, q_bufs, bufs_per_wg, sub_rings=True, descs=descs)


def test_shared_ring_with_two_issuers_is_caught():
    """The layout the kernel does not use: one ring shared by the two UMMA
    warps.  Some interleaving breaks it (an over-arrived barrier, a deadlock
    or a role spinning for ever)."""
    for seed in range(200):
        try:
            _simulate(seed, 3, 2, 4, sub_rings=False)
        except AssertionError:
            return
    raise AssertionError("the shared ring survived every interleaving")
