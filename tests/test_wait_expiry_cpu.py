"""Model checks of the kernels' wind-down when a bounded wait gives up.

Every wait between two roles of a ring kernel (a consumer waiting for a
filled stage or accumulator, a producer waiting for a released stage) polls a
bounded number of times (the option ``wait_polls``; < 0 means none).  A wait
that gives up sets the timeout bit, and the role stops taking part: it issues
no more copies or MMAs, and a consumer that gave up does not release the
stage it was waiting for (its copy may still be in flight).  The producer
still waits, with the built-in bound, for every copy it has issued, and the
MMA lane for every MMA it has issued, before the CTA's threads leave.

These tests run those control flows (restated from csrc/gemv_tc.cu,
csrc/gemv.cu and csrc/attention.cu) as host state machines in which any
role-to-role wait may give up at any moment -- when its phase is not yet
complete, or always (``wait_polls`` < 0) -- and check under random
interleavings that

  * a copy is issued into a ring slot only when no earlier copy into that
    slot is still in flight and nobody reads it, and no mbarrier receives
    more arrivals than it expects in a phase;
  * a consumer reads a stage or an accumulator only after its wait saw the
    data land;
  * when every role has finished, no copy and no MMA is in flight (the CTA
    can exit and free its shared and tensor memory);
  * every schedule terminates.
"""
from __future__ import annotations

import random

import pytest

from tests.test_ring_protocol_cpu import Barrier, Group


class StrictBarrier(Barrier):
    """An mbarrier that also rejects an over-arrival by expect_tx."""

    def arrive_expect_tx(self, nbytes: int):
        assert self.pending > 0, "arrive.expect_tx on a barrier with no pending arrival (over-arrival)"
        super().arrive_expect_tx(nbytes)


class ExpirySim:
    """Agents are generators yielding ('wait', pred) -- a wait that always
    completes (a drain) -- or ('twait', pred) -- a bounded wait that may give
    up, which the generator receives as False -- or ('step',).  Async events
    are callables."""

    def __init__(self, rng: random.Random, event_bias: float, p_expire: float, always: bool):
        self.rng, self.event_bias, self.p_expire, self.always = rng, event_bias, p_expire, always
        self.agents, self.req, self.events = {}, {}, []

    def add(self, name, gen):
        self.agents[name] = gen
        self.req[name] = ("step",)

    def post(self, fn):
        self.events.append(fn)

    def _choices(self):
        out = []
        for n, r in self.req.items():
            if r[0] == "step":
                out.append((n, None))
            elif r[0] == "wait":
                if r[1]():
                    out.append((n, True))
            else:                                 # twait
                ready = r[1]()
                if self.always:
                    out.append((n, False))        # no polls at all: it gives up at once
                elif ready:
                    out.append((n, True))
                elif self.rng.random() < self.p_expire:
                    out.append((n, False))        # the bound runs out before the phase completes
        return out

    def run(self, limit=2_000_000):
        for _ in range(limit):
            choices = self._choices()
            if not choices and not self.events:
                if not self.agents:
                    return
                # only unready bounded waits left: one of them runs out
                tw = [n for n, r in self.req.items() if r[0] == "twait"]
                assert tw, f"deadlock: {sorted(self.agents)} blocked on drains"
                choices = [(self.rng.choice(tw), False)]
            if self.events and (not choices or self.rng.random() < self.event_bias):
                self.events.pop(self.rng.randrange(len(self.events)))()
                continue
            name, val = self.rng.choice(choices)
            try:
                self.req[name] = self.agents[name].send(val)
            except StopIteration:
                del self.agents[name]
                del self.req[name]
        raise AssertionError("schedule did not terminate")


# ------------------------------------------------- gemv_tc_kernel / gemv_tcs_kernel

def run_tc_expiry(S, my_tiles, n_kst, seed, event_bias, p_expire, always, streamed):
    rng = random.Random(seed)
    sim = ExpirySim(rng, event_bias, p_expire, always)
    full = [StrictBarrier(1) for _ in range(S)]
    empty = [StrictBarrier(1) for _ in range(S)]
    acc_full = [StrictBarrier(1), StrictBarrier(1)]
    acc_empty = [StrictBarrier(4), StrictBarrier(4)]
    mma_done = StrictBarrier(1)
    inflight = [0] * S             # copy parts in flight into each slot
    content = [None] * S
    parts = [set() for _ in range(S)]
    readers = [0] * S
    acc_tile = [None, None]
    queue = []
    total = my_tiles * n_kst
    nparts = 2 if streamed else 1
    gate = {"open": not streamed}
    if streamed:
        sim.post(lambda: gate.update(open=True))

    def pump():
        queue.pop(0)()
        if queue:
            sim.post(pump)

    def push(op):
        queue.append(op)
        if len(queue) == 1:
            sim.post(pump)

    def request(s, j, part):
        assert inflight[s] < nparts, f"slot {s}: a copy issued while an earlier one is in flight"
        inflight[s] += 1

        def land(s=s, j=j, part=part):
            inflight[s] -= 1
            parts[s].add((j, part))
            if len([p for p in parts[s] if p[0] == j]) == nparts:
                content[s] = j
            full[s].complete_tx(1)
        sim.post(land)

    def arm(s):
        assert readers[s] == 0 and inflight[s] == 0, f"slot {s} rearmed while in use"
        full[s].arrive_expect_tx(nparts)
        content[s] = None
        parts[s] = set()

    def producer():
        s, ph, issued = 0, 0, 0
        pre = min(total, S) if streamed else 0
        for j in range(pre):                       # fresh slots: no wait
            arm(j)
            request(j, j, "w")
            yield ("step",)
        if streamed:
            yield ("wait", lambda: gate["open"])
            for j in range(pre):
                request(j, j, "x")
            issued, s, ph = pre, pre % S, 1 if pre == S else 0
        for j in range(pre, total):
            ok = yield ("twait", lambda s=s, ph=ph: empty[s].ready(ph ^ 1))
            if not ok:
                break
            arm(s)
            request(s, j, "w")
            if streamed:
                request(s, j, "x")
            issued += 1
            s += 1
            if s == S:
                s, ph = 0, ph ^ 1
            yield ("step",)
        for j in range(max(0, issued - S), issued):   # drain: the built-in bound
            yield ("wait", lambda j=j: full[j % S].ready((j // S) & 1))

    def mma():
        if streamed:
            yield ("wait", lambda: gate["open"])
        s, ph, j, dead = 0, 0, 0, False
        for i in range(my_tiles):
            ab = i & 1
            ok = yield ("twait", lambda ab=ab, p=((i >> 1) & 1) ^ 1: acc_empty[ab].ready(p))
            if not ok:
                break
            acc_tile[ab] = None
            for q in range(n_kst):
                ok = yield ("twait", lambda s=s, ph=ph: full[s].ready(ph))
                if not ok:
                    dead = True
                    break
                assert content[s] == j, f"MMA reads slot {s} before item {j} landed"
                readers[s] += 1

                def op(s=s, j=j):
                    assert content[s] == j, "slot changed under an MMA"
                    readers[s] -= 1
                push(op)
                push(lambda s=s: empty[s].arrive())
                j += 1
                s += 1
                if s == S:
                    s, ph = 0, ph ^ 1
                yield ("step",)
            if dead:
                break

            def tile_done(ab=ab, i=i):
                acc_tile[ab] = i
                acc_full[ab].arrive()
            push(tile_done)
        push(lambda: mma_done.arrive())
        yield ("wait", lambda: mma_done.ready(0))     # drain: every MMA issued has completed

    def epilogue(w):
        if streamed:
            yield ("wait", lambda: gate["open"])
        dead = False
        for i in range(my_tiles):
            ab = i & 1
            if not dead:
                ok = yield ("twait", lambda ab=ab, p=(i >> 1) & 1: acc_full[ab].ready(p))
                dead = not ok
            if not dead:
                assert acc_tile[ab] == i, f"epilogue reads buffer {ab} before tile {i} is done"
                yield ("step",)
                acc_empty[ab].arrive()

    sim.add("producer", producer())
    sim.add("mma", mma())
    for w in range(4):
        sim.add(f"epi{w}", epilogue(w))
    sim.run()
    assert not queue, "MMAs in flight when the CTA exits"
    assert sum(inflight) == 0 and not sim.events, "copies in flight when the CTA exits"


TC_CASES = [(S, tiles, kst, streamed) for S in (1, 2, 3, 4, 8) for tiles in (1, 2, 5) for kst in (1, 3, 7)
            for streamed in (False, True)]


@pytest.mark.parametrize("S,tiles,kst,streamed", TC_CASES)
def test_tcgen05_kernels_wind_down_when_a_wait_gives_up(S, tiles, kst, streamed):
    for trial in range(16):
        run_tc_expiry(S, tiles, kst, seed=3 * S + 17 * tiles + 101 * kst + 7919 * trial + streamed,
                      event_bias=[0.2, 0.5, 0.8][trial % 3], p_expire=[0.02, 0.1, 0.4, 0.9][trial % 4],
                      always=trial % 8 == 7, streamed=streamed)


# ------------------------------------------------------------------ gemv_kernel

def run_ring_expiry(S, G, n_chunks, n_pass, seed, event_bias, p_expire, always, release_when_dead=False):
    """The CUDA-core ring: consumer warps of group g take items g, g + G, ...;
    a warp whose wait gave up keeps the barrier sequence (group barriers
    between passes) but neither reads nor releases stages.
    release_when_dead=True plants the earlier mistake (a warp that gave up
    still released its stage)."""
    consumers = 16
    Wg = consumers // G
    rng = random.Random(seed)
    sim = ExpirySim(rng, event_bias, p_expire, always)
    full = [StrictBarrier(1) for _ in range(S)]
    empty = [StrictBarrier(Wg) for _ in range(S)]
    inflight = [0] * S
    content = [None] * S
    readers = [set() for _ in range(S)]
    total = n_pass * n_chunks
    all_sync = Group(consumers)

    def producer():
        s, ph, issued = 0, 0, 0
        for i in range(total):
            ok = yield ("twait", lambda s=s, ph=ph: empty[s].ready(ph ^ 1))
            if not ok:
                break
            assert inflight[s] == 0, f"slot {s}: a copy issued while the previous one is in flight"
            assert not readers[s], f"slot {s} overwritten while read"
            full[s].arrive_expect_tx(1)
            content[s] = None
            inflight[s] += 1

            def land(s=s, i=i):
                inflight[s] -= 1
                content[s] = i
                full[s].complete_tx(1)
            sim.post(land)
            issued = i + 1
            s += 1
            if s == S:
                s, ph = 0, ph ^ 1
            yield ("step",)
        for i in range(max(0, issued - S), issued):
            yield ("wait", lambda i=i: full[i % S].ready((i // S) & 1))

    def consumer(w):
        grp = w // Wg
        item, s, ph, dead = grp, grp, 0, False
        for p in range(n_pass):
            yield from all_sync.sync()
            while item < (p + 1) * n_chunks:
                if not dead:
                    ok = yield ("twait", lambda s=s, ph=ph: full[s].ready(ph))
                    dead = not ok
                if not dead:
                    assert content[s] == item, f"warp {w} reads slot {s} before item {item} landed"
                    readers[s].add(w)
                    yield ("step",)
                    readers[s].discard(w)
                if not dead or release_when_dead:
                    empty[s].arrive()
                item += G
                s += G
                if s >= S:
                    s, ph = s - S, ph ^ 1
            yield from all_sync.sync()

    def consumer_twait_adapter(w):
        # Group.sync yields plain waits; the consumer's own waits are bounded
        yield from consumer(w)

    sim.add("producer", producer())
    for w in range(consumers):
        sim.add(f"warp{w}", consumer_twait_adapter(w))
    sim.run()
    assert sum(inflight) == 0 and not sim.events, "copies in flight when the CTA exits"


RING_CASES = [(S, G) for G in (1, 2, 4, 16) for S in range(max(2, G), 17, G) if S <= 8 or S == 16]


@pytest.mark.parametrize("S,G", RING_CASES)
def test_cuda_core_ring_winds_down_when_a_wait_gives_up(S, G):
    for trial in range(12):
        run_ring_expiry(S, G, max(1, [1, S - 1, S + 1, 2 * S + 3][trial % 4]), 1 + trial % 2,
                        seed=1000 * S + 10 * G + trial, event_bias=[0.2, 0.5, 0.8][trial % 3],
                        p_expire=[0.05, 0.3, 0.9][trial % 3], always=trial % 6 == 5)


def test_the_checks_catch_a_stage_released_by_a_warp_that_gave_up():
    """The earlier rule (a warp that gave up still released its stage) lets
    the producer issue into a slot whose copy is still in flight."""
    bad = 0
    for seed in range(200):
        try:
            run_ring_expiry(2, 1, 6, 1, seed=seed, event_bias=0.05, p_expire=0.5, always=False,
                            release_when_dead=True)
        except AssertionError:
            bad += 1
    assert bad > 0


# --------------------------------------------------- fused_attention_tc_kernel

def run_attention_expiry(S, nst, pre, seed, event_bias, p_expire, always):
    """Producer: stages [0, pre) before the block barrier, then [pre, nst),
    each i >= S after a bounded wait for slot i % S; compute warps: a bounded
    wait per stage; a warp that gave up neither reads nor releases; after the
    loop, a block barrier (the ring is then reused for the warps' states)."""
    warps = 8
    rng = random.Random(seed)
    sim = ExpirySim(rng, event_bias, p_expire, always)
    full = [StrictBarrier(1) for _ in range(S)]
    empty = [StrictBarrier(warps) for _ in range(S)]
    inflight = [0] * S
    content = [None] * S
    readers = [set() for _ in range(S)]
    block = Group(warps + 1)
    end = Group(warps + 1)
    state = {"reused": False}

    def load(i):
        s = i % S
        assert inflight[s] == 0 and not readers[s], f"slot {s} reloaded while in use"
        full[s].arrive_expect_tx(1)
        content[s] = None
        inflight[s] += 1

        def land(s=s, i=i):
            assert not state["reused"], "a copy lands after the ring was reused"
            inflight[s] -= 1
            content[s] = i
            full[s].complete_tx(1)
        sim.post(land)

    def producer():
        for i in range(pre):
            load(i)
            yield ("step",)
        yield from block.sync()
        issued = pre
        for i in range(pre, nst):
            if i >= S:
                ok = yield ("twait", lambda i=i: empty[i % S].ready((i // S - 1) & 1))
                if not ok:
                    break
            load(i)
            issued = i + 1
            yield ("step",)
        for i in range(max(0, issued - S), issued):
            yield ("wait", lambda i=i: full[i % S].ready((i // S) & 1))
        yield from end.sync()

    def compute(w):
        yield from block.sync()
        dead = False
        for i in range(nst):
            s = i % S
            if not dead:
                ok = yield ("twait", lambda s=s, i=i: full[s].ready((i // S) & 1))
                dead = not ok
            if not dead:
                assert content[s] == i, f"warp {w} reads slot {s} before stage {i} landed"
                readers[s].add(w)
                yield ("step",)
                readers[s].discard(w)
                empty[s].arrive()
        yield from end.sync()
        # after the block barrier the ring holds the warps' states
        assert sum(inflight) == 0, "the ring is reused while a copy is in flight"
        state["reused"] = True

    sim.add("producer", producer())
    for w in range(warps):
        sim.add(f"warp{w}", compute(w))
    sim.run()
    assert sum(inflight) == 0 and not sim.events


ATTN_CASES = [(S, nst, pre) for S in (2, 3) for nst in (1, 3, 4, 9) for pre in range(0, min(S, nst) + 1)]


@pytest.mark.parametrize("S,nst,pre", ATTN_CASES)
def test_attention_ring_winds_down_when_a_wait_gives_up(S, nst, pre):
    for trial in range(16):
        run_attention_expiry(S, nst, pre, seed=104729 * S + 101 * nst + 7 * pre + trial,
                             event_bias=[0.2, 0.5, 0.8][trial % 3], p_expire=[0.05, 0.3, 0.9][trial % 3],
                             always=trial % 8 == 7)
