"""A discrete-event model of the attention kernel's synchronisation protocol
(paper_2609_09768_gb300/csrc/attn.cu), run on the CPU under many random schedules.

The kernel has one wait without a time limit: the named barrier through which the four
softmax warps hand P_j to the P.V issuer (bar.sync, five warps, once per key tile).  Its
safety rests on every warp passing it exactly once per tile on every path, including
after a bounded mbarrier wait has run out.  The model replays the kernel's warps as
cooperative actors:

  producer   : for tile j, wait pv_done[j % 3] (P.V of tile j - 3 done), issue the TMA load
               of K_j and V_j onto kv_full[j % 3]; it may stall between any two steps
  S issuer   : wait q_ready; per j: wait kv_full (tile j), then for j >= 2 pv_done of tile
               j - 2 (P.V_{j-2} read the buffer S_j overwrites), issue S_j, commit s_full[j % 2]
  P.V issuer : per j: wait kv_full (tile j), pass the P barrier for tile j, issue P.V_j,
               commit pv_done[j % 3]
  softmax x4 : arrive q_ready; per j: wait s_full, compute, optionally wait pv_done of tile
               j - 1 and rescale O, write P_j over S_j's buffer, pass the P barrier; finally
               wait pv_done of the last tile

Each issuer's MMAs run in its own issue order; the two issuers' MMAs are either not
ordered with each other at all (two pipes running concurrently, the general case) or
interleaved in one pipe.  TMA loads land after random delays, and mbarrier waits have
parity semantics and a time limit that, when it runs out, sets the CTA's abort flag
(every later incomplete wait then returns at once).

Each run checks: every actor finishes (no deadlock, in particular at the P barrier); no
warp arrives twice in one phase of the named barrier; no parity wait ever finds its
barrier two phases ahead, nor asks for a phase while the one before it is still open
(either would make the hardware answer wrongly: a parity wait cannot tell phase k from
k - 2); and, in runs where no wait runs out, the data hazards are ordered: a slot is
reloaded only after the P.V that read it, S_j runs only after K_j landed and P.V_j only
after V_j landed, P.V_j only after all four warps wrote P_j, S_{j+2} only after P.V_j read
P_j from the same buffer, and O is rescaled only when no P.V into it is outstanding.
After a wait has run out the kernel still finishes but may compute on stale data in
shared and tensor memory; it stays in bounds and the status word reports the timeout.
"""
import random

import pytest

STAGES = 3
N_SOFTMAX = 4
BAR_COUNT = N_SOFTMAX + 1


class Protocol:
    def __init__(self, n_tiles, seed, abort_at=None, limit=400, shared_pipe=False):
        self.rng = random.Random(seed)
        self.shared = shared_pipe        # one pipe for both issuers' MMAs, or one each
        self.n = n_tiles
        self.t = 0
        self.limit = limit               # ticks a bounded wait may last before it gives up
        self.abort_at = abort_at         # tick at which some wait is made to run out
        self.abort = False
        self.mbar = {}                   # (name, index) -> completed phases
        self.arrivals = {}               # (name, index) -> arrivals in the current phase
        self.expected = {("q_ready", 0): N_SOFTMAX}
        self.events = []                 # (tick, callable) for TMA completions
        self.pipes = {"s": [], "pv": []}   # issued tensor-pipe work per issuer, in order
        self.busy = {"s": 0, "pv": 0}
        self.bar_phase = 0
        self.bar_arrived = set()
        self.bar_waiting = set()
        self.done = {"kv": set(), "S": set(), "PV": set()}
        self.p_written = {}
        self.errors = []

    def hazard(self, msg):
        # after a wait has run out the kernel computes on stale data (in bounds; the status
        # word reports the timeout and the result is discarded), so only runs without an
        # abort must keep the data order
        if not self.abort:
            self.errors.append(msg)

    # ------------------------------------------------------------------ primitives
    def phases(self, name, idx):
        return self.mbar.get((name, idx), 0)

    def complete(self, name, idx):
        self.mbar[(name, idx)] = self.phases(name, idx) + 1

    def arrive(self, name, idx):
        key = (name, idx)
        self.arrivals[key] = self.arrivals.get(key, 0) + 1
        if self.arrivals[key] == self.expected.get(key, 1):
            self.arrivals[key] = 0
            self.complete(name, idx)

    def check_parity(self, name, idx, parity, phase):
        """try_wait.parity: true iff the barrier's current phase parity differs from `parity`."""
        c = self.phases(name, idx)
        if c - phase >= 2:
            self.errors.append(f"{name}[{idx}] two phases past the awaited phase {phase} (c = {c})")
        if c < phase:
            self.errors.append(f"{name}[{idx}] asked for phase {phase} while phase {c} is still open")
        return (c & 1) != parity

    def issue(self, who, kind, j=None, commit=None):
        self.pipes["s" if self.shared else who].append((kind, j, commit))

    def stall(self):
        """the producer may be slow to get to its next step"""
        if self.rng.random() < 0.3:
            yield ("delay", self.rng.randint(1, 80))

    # ------------------------------------------------------------------ actors
    def producer(self):
        for j in range(self.n):
            st = j % STAGES
            ok = yield ("wait", "pv_done", st, ((j // STAGES) & 1) ^ 1, j // STAGES - 1)
            if not ok:
                break
            if j >= STAGES and (j - STAGES) not in self.done["PV"]:
                self.hazard(f"slot {st} reloaded for tile {j} before P.V of tile {j - STAGES}")
            yield from self.stall()
            delay = self.rng.randint(5, 60)

            def land(j=j, st=st):
                self.done["kv"].add(j)
                self.complete("kv_full", st)
            self.events.append((self.t + delay, land))

    def s_issuer(self):
        ok = yield ("wait", "q_ready", 0, 0, 0)
        for j in range(self.n):
            if not ok:
                break
            ok = yield ("wait", "kv_full", j % STAGES, (j // STAGES) & 1, j // STAGES)
            if ok and j >= 2:
                ok = yield ("wait", "pv_done", (j - 2) % STAGES, ((j - 2) // STAGES) & 1, (j - 2) // STAGES)
            if not ok:
                break
            self.issue("s", "S", j, ("s_full", j % 2))
        self.issue("s", "drain", None, ("drain_s", 0))
        yield ("wait", "drain_s", 0, 0, 0)

    def pv_issuer(self):
        ok = True
        for j in range(self.n):
            if ok:
                ok = yield ("wait", "kv_full", j % STAGES, (j // STAGES) & 1, j // STAGES)
            yield ("bar",)
            if ok:
                self.issue("pv", "PV", j, ("pv_done", j % STAGES))
        self.issue("pv", "drain", None, ("drain", 0))
        yield ("wait", "drain", 0, 0, 0)

    def softmax(self, w):
        self.arrive("q_ready", 0)
        ok = True
        for j in range(self.n):
            if ok:
                ok = yield ("wait", "s_full", j % 2, (j >> 1) & 1, j // 2)
            if not ok:
                yield ("bar",)
                continue
            if j not in self.done["S"]:
                self.hazard(f"softmax {w} read S_{j} before it was done")
            yield ("delay", self.rng.randint(3, 30))
            if j >= 1 and self.rng.random() < 0.15:      # the running max grew: rescale O
                ok2 = yield ("wait", "pv_done", (j - 1) % STAGES, ((j - 1) // STAGES) & 1, (j - 1) // STAGES)
                if not ok2:
                    ok = False
                    yield ("bar",)
                    continue
                if (j - 1) not in self.done["PV"]:
                    self.hazard(f"O rescaled at tile {j} while P.V_{j - 1} is outstanding")
            yield ("delay", self.rng.randint(1, 5))
            self.p_written.setdefault(j, set()).add(w)
            yield ("bar",)
        if ok:
            yield ("wait", "pv_done", (self.n - 1) % STAGES, ((self.n - 1) // STAGES) & 1, (self.n - 1) // STAGES)

    # ------------------------------------------------------------------ tensor pipe
    def step_one(self, key):
        q = self.pipes[key]
        if not q or self.t < self.busy[key]:
            return False
        kind, j, commit = q.pop(0)
        if kind in ("S", "PV") and j not in self.done["kv"]:
            self.hazard(f"{kind}_{j} ran before K_{j} and V_{j} landed")
        if kind == "S" and j >= 2 and (j - 2) not in self.done["PV"]:
            self.hazard(f"S_{j} overwrote P_{j - 2} before P.V_{j - 2} read it")
        if kind == "PV" and self.p_written.get(j, set()) != set(range(N_SOFTMAX)):
            self.hazard(f"P.V_{j} ran before all warps wrote P_{j}")
        self.busy[key] = self.t + (self.rng.randint(4, 12) if kind != "drain" else 0)

        def finish(kind=kind, j=j, commit=commit):
            if kind in ("S", "PV"):
                self.done[kind].add(j)
            if commit:
                self.complete(*commit)
        self.events.append((self.busy[key], finish))
        return True

    def step_pipe(self):
        a = self.step_one("s")
        b = self.step_one("pv")
        return a or b

    # ------------------------------------------------------------------ scheduler
    def run(self, max_ticks=200000):
        actors = {"producer": self.producer(), "s_issuer": self.s_issuer(), "pv_issuer": self.pv_issuer()}
        for w in range(N_SOFTMAX):
            actors[f"softmax{w}"] = self.softmax(w)
        state = {}                       # actor -> (request, start tick)
        values = {a: None for a in actors}
        finished = set()
        bar_members = {"pv_issuer"} | {f"softmax{w}" for w in range(N_SOFTMAX)}
        while len(finished) < len(actors):
            if self.t > max_ticks:
                raise AssertionError(f"deadlock: waiting {sorted(set(actors) - finished)} at tick {self.t}")
            if self.abort_at is not None and self.t >= self.abort_at:
                self.abort = True
            progressed = False
            for tick, fn in [e for e in self.events if e[0] <= self.t]:
                fn()
                progressed = True
            self.events = [e for e in self.events if e[0] > self.t]
            progressed |= self.step_pipe()
            for a, gen in actors.items():
                if a in finished:
                    continue
                if a in state:
                    req, t0 = state[a]
                    if req[0] == "wait":
                        _, name, idx, parity, phase = req
                        if self.check_parity(name, idx, parity, phase):
                            values[a] = True
                        elif self.abort:
                            values[a] = False
                        elif self.t - t0 > self.limit:
                            self.abort = True
                            values[a] = False
                        else:
                            continue
                    elif req[0] == "delay":
                        if self.t < t0 + req[1]:
                            continue
                        values[a] = None
                    elif req[0] == "bar":
                        if a in self.bar_waiting:
                            continue
                        values[a] = None
                    del state[a]
                try:
                    req = gen.send(values[a])
                except StopIteration:
                    finished.add(a)
                    progressed = True
                    continue
                progressed = True
                if req[0] == "bar":
                    assert a in bar_members
                    if a in self.bar_arrived:
                        self.errors.append(f"{a} arrived twice in phase {self.bar_phase} of the P barrier")
                    self.bar_arrived.add(a)
                    self.bar_waiting.add(a)
                    if len(self.bar_arrived) == BAR_COUNT:
                        self.bar_arrived, self.bar_waiting = set(), set()
                        self.bar_phase += 1
                state[a] = (req, self.t)
            self.t += 1
        assert not self.errors, self.errors[:5]
        return self.bar_phase


@pytest.mark.parametrize("shared_pipe", [False, True])
@pytest.mark.parametrize("n_tiles", [1, 2, 3, 4, 7, 20])
def test_protocol_completes_and_orders_every_hazard(n_tiles, shared_pipe):
    for seed in range(40):
        phases = Protocol(n_tiles, seed, shared_pipe=shared_pipe).run()
        assert phases == n_tiles                      # one P-barrier phase per key tile


@pytest.mark.parametrize("shared_pipe", [False, True])
@pytest.mark.parametrize("n_tiles", [1, 3, 6, 20])
def test_protocol_completes_after_a_wait_runs_out(n_tiles, shared_pipe):
    """Some wait gives up at a random tick: every warp still passes every tile's P
    barrier once, so the barrier cannot block the kernel's exit."""
    for seed in range(60):
        rng = random.Random(1000 + seed)
        phases = Protocol(n_tiles, seed, abort_at=rng.randint(0, 40 * n_tiles), shared_pipe=shared_pipe).run()
        assert phases == n_tiles


def test_model_catches_a_warp_that_skips_the_barrier():
    """The check has teeth: a softmax warp that leaves its loop after a failed wait leaves
    the P.V issuer blocked at the barrier."""
    class Skipping(Protocol):
        def softmax(self, w):
            self.arrive("q_ready", 0)
            for j in range(self.n):
                ok = yield ("wait", "s_full", j % 2, (j >> 1) & 1, j // 2)
                if not ok:
                    return
                yield ("delay", 3)
                self.p_written.setdefault(j, set()).add(w)
                yield ("bar",)
    with pytest.raises(AssertionError, match="deadlock"):
        Skipping(6, 0, abort_at=20).run(max_ticks=20000)


def test_model_catches_a_slot_reloaded_too_early():
    """A producer that reuses a K/V slot without waiting for the P.V that reads it is
    flagged as a hazard."""
    class Eager(Protocol):
        def producer(self):
            for j in range(self.n):
                st = j % STAGES
                yield ("delay", 1)
                if j >= STAGES and (j - STAGES) not in self.done["PV"]:
                    self.hazard(f"slot {st} reloaded for tile {j} before P.V of tile {j - STAGES}")

                def land(j=j, st=st):
                    self.done["kv"].add(j)
                    self.complete("kv_full", st)
                self.events.append((self.t + 5, land))
    with pytest.raises(AssertionError, match="reloaded|two phases past"):
        Eager(12, 0).run()


def test_model_catches_s_issued_before_the_pv_that_reads_its_buffer():
    """The two issuers' MMAs are not ordered with each other, so an S issuer that does not
    wait for P.V_{j-2} can overwrite P_{j-2} before it is read."""
    class NoPvWait(Protocol):
        def s_issuer(self):
            yield ("wait", "q_ready", 0, 0, 0)
            for j in range(self.n):
                yield ("wait", "kv_full", j % STAGES, (j // STAGES) & 1, j // STAGES)
                self.issue("s", "S", j, ("s_full", j % 2))
            self.issue("s", "drain", None, ("drain_s", 0))
            yield ("wait", "drain_s", 0, 0, 0)
    caught = 0
    for seed in range(10):
        try:
            NoPvWait(12, seed).run()
        except AssertionError as e:
            assert "overwrote" in str(e) or "two phases" in str(e) or "still open" in str(e), e
            caught += 1
    assert caught >= 8


def test_model_catches_a_wait_on_a_phase_not_yet_reached():
    """A producer that frees slot j % 3 by waiting for S_{j-1} on the double-buffered
    s_full barrier asks, at tiles 3 and 4, for a phase the barrier has not reached while
    the one before is still open; the hardware answers such a parity wait at once.  The
    model flags it."""
    class WaitsOnS(Protocol):
        def producer(self):
            for j in range(self.n):
                st = j % STAGES
                if j >= STAGES:
                    ok = yield ("wait", "s_full", (j - 1) & 1, ((j - 1) >> 1) & 1, (j - 1) >> 1)
                    if not ok:
                        break

                def land(j=j, st=st):
                    self.done["kv"].add(j)
                    self.complete("kv_full", st)
                self.events.append((self.t + 5, land))
    with pytest.raises(AssertionError, match="still open"):
        WaitsOnS(12, 0).run()

