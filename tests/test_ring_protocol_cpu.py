"""Model checks of the shared-memory ring protocols of the projection kernels.

The weight-streaming kernels hand ring stages between a TMA producer and
their consumers with mbarriers that are waited on by phase parity only.  A
parity wait is correct only if the waiter is never two phases away from the
phase it means; otherwise a stale phase of the same parity satisfies it and a
stage is read before its data lands or overwritten while still in use.  These
tests run the kernels' barrier sequences as host-side state machines under
many random interleavings (asynchronous copies, MMAs and commits complete at
random times) and check at every step that

  * a wait succeeds only when exactly the intended phase has completed (the
    barrier is exactly one phase past it, never two),
  * a copy writes a stage only after every reader of its previous contents
    has finished, and a reader finds its own item's data there,
  * a tensor-memory accumulator is overwritten only after all epilogue warps
    have read the previous tile, and read only after that tile's MMAs are done,
  * every schedule terminates (no deadlock) with every item consumed.

The models restate the control flow of ``gemv_kernel`` (csrc/gemv.cu: one
producer lane, 16 consumer warps in G groups, group g taking stages s = g mod
G), of ``gemv_tc_kernel`` / ``gemv_tcs_kernel`` (csrc/gemv_tc.cu: producer
lane, MMA lane committing to the stage and accumulator barriers, four
epilogue warps over two accumulator buffers) and of
``fused_attention_tc_kernel`` (csrc/attention.cu: stages of committed rows
requested before the block-wide barrier, eight compute warps releasing every
stage), with the plans the host code can choose (S stages a multiple of G,
2 <= S <= 16; 1..8 stages; any stage and tile counts)."""
from __future__ import annotations

import random

import pytest


class Barrier:
    """mbarrier: expected arrival count, pending arrivals, transaction bytes
    and the number of completed phases.  try_wait.parity(p) succeeds while the
    current phase's parity differs from p."""

    def __init__(self, count: int):
        self.count = count
        self.pending = count
        self.tx = 0
        self.phase = 0

    def _maybe_complete(self):
        if self.pending == 0 and self.tx == 0:
            self.phase += 1
            self.pending = self.count

    def arrive(self):
        assert self.pending > 0
        self.pending -= 1
        self._maybe_complete()

    def arrive_expect_tx(self, nbytes: int):
        self.tx += nbytes
        self.pending -= 1
        self._maybe_complete()

    def complete_tx(self, nbytes: int):
        self.tx -= nbytes
        assert self.tx >= 0
        self._maybe_complete()

    def ready(self, parity: int) -> bool:
        return self.phase % 2 != parity


def check_wait(bar: Barrier, parity: int, intended_phase: int, what: str):
    """A successful wait for the completion of phase `intended_phase` (0-based)
    must find exactly that phase completed and no later one."""
    assert parity == intended_phase % 2, what
    assert bar.phase == intended_phase + 1, f"{what}: barrier at phase {bar.phase}, wanted {intended_phase + 1}"


class Sim:
    """Agents are generators yielding either ('wait', predicate) or ('step',);
    async events are callables.  The scheduler picks uniformly among runnable
    agents and pending events (optionally biased to delay events)."""

    def __init__(self, rng: random.Random, event_bias: float):
        self.rng = rng
        self.agents = {}
        self.blocked = {}
        self.events = []
        self.event_bias = event_bias

    def add(self, name, gen):
        self.agents[name] = gen
        self.blocked[name] = None

    def post(self, fn):
        self.events.append(fn)

    def run(self, limit=2_000_000):
        for _ in range(limit):
            runnable = [n for n, pred in self.blocked.items() if pred is None or pred()]
            if not runnable and not self.events:
                assert not self.agents, f"deadlock: {sorted(self.agents)} blocked"
                return
            take_event = self.events and (not runnable or self.rng.random() < self.event_bias)
            if take_event:
                fn = self.events.pop(self.rng.randrange(len(self.events)))
                fn()
                continue
            name = self.rng.choice(runnable)
            try:
                req = next(self.agents[name])
            except StopIteration:
                del self.agents[name]
                del self.blocked[name]
                continue
            self.blocked[name] = req[1] if req[0] == "wait" else None
        raise AssertionError("schedule did not terminate")


class Group:
    """A named barrier (bar.sync) among a fixed set of agents."""

    def __init__(self, n):
        self.n, self.arrived, self.gen = n, 0, 0

    def sync(self):
        g = self.gen
        self.arrived += 1
        if self.arrived == self.n:
            self.arrived, self.gen = 0, self.gen + 1
        yield ("wait", lambda: self.gen > g)


# --------------------------------------------------------------- gemv_kernel

def run_cuda_core_ring(S, G, n_chunks, n_pass, R, seed, event_bias, empty_count=None):
    """gemv_kernel: producer waits empty[s] (parity ph ^ 1), expects the
    stage's bytes on full[s] and issues the copies; consumer warps of group g
    take items g, g + G, ... across all passes, wait full[s] (parity ph),
    read, and arrive on empty[s] (count = warps per group)."""
    consumers = 16
    Wg = consumers // G
    SEG = 1 if R >= Wg else Wg // R
    if SEG > 1:
        assert 2 + G - 1 <= 15, "group barriers must fit the 16 named barriers"
    rng = random.Random(seed)
    sim = Sim(rng, event_bias)
    full = [Barrier(1) for _ in range(S)]
    empty = [Barrier(empty_count or Wg) for _ in range(S)]
    content = [None] * S          # item whose data has landed in the stage
    readers = [set() for _ in range(S)]    # warps still to release the stage's current item
    consumed = {}
    total = n_pass * n_chunks
    all_sync = Group(consumers)
    grp_sync = [Group(Wg) for _ in range(G)]

    def producer():
        issued = 0
        s, ph = 0, 0
        for i in range(total):
            yield ("wait", lambda s=s, ph=ph: empty[s].ready(ph ^ 1))
            if i >= S:
                check_wait(empty[s], ph ^ 1, i // S - 1, "producer empty")
            assert not readers[s], f"stage {s} overwritten while item {content[s]} is being read"
            full[s].arrive_expect_tx(1)
            content[s] = None

            def land(s=s, i=i):
                content[s] = i
                readers[s] = {w for w in range(consumers) if w // Wg == i % G}
                full[s].complete_tx(1)
            sim.post(land)
            issued = i + 1
            s += 1
            if s == S:
                s, ph = 0, ph ^ 1
            yield ("step",)
        for i in range(max(0, issued - S), issued):
            yield ("wait", lambda i=i: full[i % S].ready((i // S) & 1))
            check_wait(full[i % S], (i // S) & 1, i // S, "producer drain")

    def consumer(w):
        grp = w // Wg
        item, s, ph = grp, grp, 0
        for p in range(n_pass):
            yield from all_sync.sync()           # activation rows staged
            while item < (p + 1) * n_chunks:
                yield ("wait", lambda s=s, ph=ph: full[s].ready(ph))
                check_wait(full[s], ph, item // S, f"warp {w} full")
                assert content[s] == item, f"warp {w} reads stage {s}: {content[s]} instead of {item}"
                consumed.setdefault(item, set()).add(w)
                yield ("step",)
                if SEG > 1:
                    yield from grp_sync[grp].sync()
                assert content[s] == item
                readers[s].discard(w)
                empty[s].arrive()
                item += G
                s += G
                if s >= S:
                    s, ph = s - S, ph ^ 1
            yield from all_sync.sync()           # end of pass

    sim.add("producer", producer())
    for w in range(consumers):
        sim.add(f"warp{w}", consumer(w))
    sim.run()
    for i in range(total):
        assert consumed[i] == {w for w in range(consumers) if w // Wg == i % G}, i


CUDA_CORE_PLANS = [(S, G) for G in (1, 2, 4, 8, 16) for S in range(max(2, G), 17, G)]


@pytest.mark.parametrize("S,G", CUDA_CORE_PLANS)
def test_cuda_core_ring_parity_waits_are_unambiguous(S, G):
    for trial in range(24):
        n_chunks = max(1, [1, 2, S - 1, S, S + 1, 3 * S + 2][trial % 6])
        n_pass = 1 if trial % 2 == 0 else 3
        R = [1, 2, 8][trial % 3]
        run_cuda_core_ring(S, G, n_chunks, n_pass, R, seed=1000 * S + 10 * G + trial,
                           event_bias=[0.1, 0.5, 0.9, 0.3][trial % 4])


# ------------------------------------------------------------ gemv_tc_kernel

def run_tc_ring(S, my_tiles, n_kst, seed, event_bias, mma_lag, acc_empty_count=4, streamed=False,
                early_x=False):
    """gemv_tc_kernel: producer as above (empty[s] has one arrival: the MMA
    lane's tcgen05.commit); the MMA lane waits acc_empty[ab] (parity
    ((i >> 1) & 1) ^ 1), then full[s] per stage, issues MMAs into accumulator
    buffer ab = i & 1 and commits them to empty[s], then commits the tile to
    acc_full[ab]; four epilogue warps wait acc_full[ab] (parity (i >> 1) & 1),
    read the buffer and arrive on acc_empty[ab] (count 4).  Commits arrive
    when every MMA issued before them has completed (in issue order).

    streamed=True: gemv_tcs_kernel, whose stages hold weight boxes and
    activation (X) boxes, X being the previous kernel's output.  The producer
    arms each of the first min(total, S) stages for both parts and requests
    their weight boxes, waits for the previous kernel (griddepcontrol.wait,
    here a gate that opens at a random time), then requests those stages' X
    boxes; later stages get both parts together.  A stage's data is complete
    only when both parts have landed.  early_x=True requests the first X boxes
    before the gate (a planted mistake the checks must catch)."""
    rng = random.Random(seed)
    sim = Sim(rng, event_bias)
    gate = {"open": not streamed}
    if streamed:
        sim.post(lambda: gate.update(open=True))
    full = [Barrier(1) for _ in range(S)]
    empty = [Barrier(1) for _ in range(S)]
    acc_full = [Barrier(1), Barrier(1)]
    acc_empty = [Barrier(acc_empty_count), Barrier(acc_empty_count)]
    mma_done = Barrier(1)
    content = [None] * S
    stage_readers = [0] * S       # MMAs issued on the stage's current item and not yet complete
    acc_tile = [None, None]       # tile whose MMAs have all completed in the buffer
    acc_readers = [set(), set()]
    queue = []                    # the MMA lane's async tcgen05 operations, in issue order
    read = {}
    total = my_tiles * n_kst

    def pump():
        # the head of the MMA queue completes
        op = queue.pop(0)
        op()
        if queue:
            sim.post(pump)

    def push(op):
        queue.append(op)
        if len(queue) == 1:
            sim.post(pump)

    parts = [set() for _ in range(S)]

    def request(s, j, part):
        if part == "x":
            assert gate["open"], f"X box of item {j} requested before the previous kernel completed"

        def land(s=s, j=j, part=part):
            parts[s].add((j, part))
            if {(j, "w"), (j, "x")} <= parts[s] or not streamed:
                content[s] = j
            full[s].complete_tx(1)
        sim.post(land)

    def producer():
        s, ph, issued = 0, 0, 0
        nparts = 2 if streamed else 1
        pre = min(total, S) if streamed else 0
        for j in range(pre):                  # first pass: arm, weight boxes only
            assert stage_readers[j] == 0
            full[j].arrive_expect_tx(nparts)
            content[j] = None
            parts[j] = set()
            request(j, j, "w")
            if early_x:
                request(j, j, "x")
            yield ("step",)
        if streamed:
            yield ("wait", lambda: gate["open"])        # griddepcontrol.wait
            for j in range(pre):
                if not early_x:
                    request(j, j, "x")
                yield ("step",)
            issued = pre
            s, ph = pre % S, 1 if pre == S else 0
        for j in range(pre, total):
            yield ("wait", lambda s=s, ph=ph: empty[s].ready(ph ^ 1))
            if j >= S:
                check_wait(empty[s], ph ^ 1, j // S - 1, "producer empty")
            assert stage_readers[s] == 0, f"stage {s} overwritten while MMAs read it"
            full[s].arrive_expect_tx(nparts)
            content[s] = None
            parts[s] = set()
            request(s, j, "w")
            if streamed:
                request(s, j, "x")
            issued += 1
            s += 1
            if s == S:
                s, ph = 0, ph ^ 1
            yield ("step",)
        for j in range(max(0, issued - S), issued):
            yield ("wait", lambda j=j: full[j % S].ready((j // S) & 1))
            check_wait(full[j % S], (j // S) & 1, j // S, "producer drain")

    def mma():
        s, ph, j = 0, 0, 0
        if streamed:
            yield ("wait", lambda: gate["open"])        # griddepcontrol.wait
        for i in range(my_tiles):
            ab = i & 1
            par = ((i >> 1) & 1) ^ 1
            yield ("wait", lambda ab=ab, par=par: acc_empty[ab].ready(par))
            if i >= 2:
                check_wait(acc_empty[ab], par, (i >> 1) - 1, "mma acc_empty")
            assert not acc_readers[ab], f"accumulator {ab} overwritten while tile {acc_tile[ab]} is read"
            acc_tile[ab] = None
            for q in range(n_kst):
                yield ("wait", lambda s=s, ph=ph: full[s].ready(ph))
                check_wait(full[s], ph, j // S, "mma full")
                assert content[s] == j, f"MMA reads stage {s}: {content[s]} instead of {j}"
                stage_readers[s] += 1

                def mma_op(s=s, j=j):
                    assert content[s] == j, "stage changed under an MMA"
                    stage_readers[s] -= 1
                for _ in range(mma_lag):
                    push(lambda: None)
                push(mma_op)
                push(lambda s=s: empty[s].arrive())          # tcgen05.commit -> empty[s]
                j += 1
                s += 1
                if s == S:
                    s, ph = 0, ph ^ 1
                yield ("step",)

            def tile_done(ab=ab, i=i):
                acc_tile[ab] = i
                acc_readers[ab] = {0, 1, 2, 3}
                acc_full[ab].arrive()
            push(tile_done)                                   # tcgen05.commit -> acc_full[ab]
        push(lambda: mma_done.arrive())
        yield ("wait", lambda: mma_done.ready(0))

    def epilogue(w):
        for i in range(my_tiles):
            ab = i & 1
            par = (i >> 1) & 1
            yield ("wait", lambda ab=ab, par=par: acc_full[ab].ready(par))
            check_wait(acc_full[ab], par, i >> 1, f"epilogue {w} acc_full")
            assert acc_tile[ab] == i, f"epilogue {w} reads buffer {ab}: tile {acc_tile[ab]} instead of {i}"
            read.setdefault(i, set()).add(w)
            yield ("step",)
            acc_readers[ab].discard(w)
            acc_empty[ab].arrive()

    sim.add("producer", producer())
    sim.add("mma", mma())
    for w in range(4):
        sim.add(f"epi{w}", epilogue(w))
    sim.run()
    assert all(read.get(i) == {0, 1, 2, 3} for i in range(my_tiles))
    assert not queue


TC_PLANS = [(S, tiles, kst) for S in (1, 2, 3, 4, 5, 8) for tiles in (1, 2, 3, 7) for kst in (1, 2, 5, 11)]


@pytest.mark.parametrize("S,tiles,kst", TC_PLANS)
@pytest.mark.parametrize("streamed", [False, True], ids=["staged", "streamed"])
def test_tcgen05_ring_and_accumulator_handoff(S, tiles, kst, streamed):
    for trial in range(12):
        run_tc_ring(S, tiles, kst, seed=7919 * S + 31 * tiles + kst + trial,
                    event_bias=[0.15, 0.5, 0.85][trial % 3], mma_lag=trial % 4, streamed=streamed)


# ------------------------------------------------- fused_attention_tc_kernel

def run_attention_ring(S, nst, pre, seed, event_bias, empty_count=8):
    """fused_attention_tc_kernel: the producer requests stages [0, pre)
    (committed rows only) before the block-wide barrier, then stages
    [pre, nst), each i >= S after waiting empty[i % S] for the release of
    stage i - S (parity (i / S - 1) & 1); eight compute warps wait full[i % S]
    (parity (i / S) & 1) for every stage and arrive on empty[i % S] (count 8)."""
    warps = 8
    rng = random.Random(seed)
    sim = Sim(rng, event_bias)
    full = [Barrier(1) for _ in range(S)]
    empty = [Barrier(empty_count) for _ in range(S)]
    content = [None] * S
    readers = [set() for _ in range(S)]
    block = Group(warps + 1)
    read = {}

    def load(i):
        s = i % S
        assert not readers[s], f"slot {s} overwritten while stage {content[s]} is read"
        full[s].arrive_expect_tx(1)
        content[s] = None

        def land(s=s, i=i):
            content[s] = i
            readers[s] = set(range(warps))
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
                par = (i // S - 1) & 1
                yield ("wait", lambda i=i, par=par: empty[i % S].ready(par))
                check_wait(empty[i % S], par, i // S - 1, "attention producer empty")
            load(i)
            issued = i + 1
            yield ("step",)
        for i in range(max(0, issued - S), issued):
            yield ("wait", lambda i=i: full[i % S].ready((i // S) & 1))
            check_wait(full[i % S], (i // S) & 1, i // S, "attention producer drain")

    def compute(w):
        yield from block.sync()
        for i in range(nst):
            s = i % S
            yield ("wait", lambda s=s, i=i: full[s].ready((i // S) & 1))
            check_wait(full[s], (i // S) & 1, i // S, f"attention warp {w} full")
            assert content[s] == i, f"warp {w} reads slot {s}: stage {content[s]} instead of {i}"
            read.setdefault(i, set()).add(w)
            yield ("step",)
            assert content[s] == i
            readers[s].discard(w)
            empty[s].arrive()

    sim.add("producer", producer())
    for w in range(warps):
        sim.add(f"warp{w}", compute(w))
    sim.run()
    assert all(read.get(i) == set(range(warps)) for i in range(nst))


ATTN_CASES = [(S, nst, pre) for S in (2, 3, 4) for nst in (1, 2, 3, 4, 7, 12) for pre in range(0, min(S, nst) + 1)]


@pytest.mark.parametrize("S,nst,pre", ATTN_CASES)
def test_attention_ring_parity_waits_are_unambiguous(S, nst, pre):
    for trial in range(12):
        run_attention_ring(S, nst, pre, seed=104729 * S + 101 * nst + 7 * pre + trial,
                           event_bias=[0.1, 0.5, 0.9][trial % 3])


def _fails(run, n=40):
    bad = 0
    for seed in range(n):
        try:
            run(seed)
        except AssertionError:
            bad += 1
    return bad


def test_the_checks_catch_an_early_stage_release():
    """The checks have teeth: a stage barrier expecting one arrival instead of
    one per warp of the group releases the stage while other warps still read
    it, and some schedule shows it."""
    assert _fails(lambda seed: run_cuda_core_ring(4, 2, 9, 1, 8, seed=seed, event_bias=0.5, empty_count=1)) > 0


def test_the_checks_catch_an_early_accumulator_release():
    """Likewise for the accumulator: released after the first epilogue warp
    instead of all four, the MMA lane overwrites a buffer still being read."""
    assert _fails(lambda seed: run_tc_ring(2, 5, 2, seed=seed, event_bias=0.5, mma_lag=0, acc_empty_count=1)) > 0


def test_the_checks_catch_x_boxes_requested_before_the_dependency_wait():
    """The streamed producer requests its first weight boxes early; its X
    boxes (the previous kernel's output) must wait, and the checks see it."""
    assert _fails(lambda seed: run_tc_ring(3, 2, 4, seed=seed, event_bias=0.5, mma_lag=1, streamed=True,
                                           early_x=True)) > 0


def test_the_checks_catch_an_early_attention_stage_release():
    assert _fails(lambda seed: run_attention_ring(3, 9, 2, seed=seed, event_bias=0.5, empty_count=1)) > 0
