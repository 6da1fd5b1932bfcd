"""A CPU model of decode_main's synchronisation (csrc/decode.cu): the eight
worker warps and the four MMA-issuing threads of one CTA, for the packed
caches, written as the sequence of barrier, buffer and MMA operations each of
them performs per tile, in program order. A scheduler runs them under random
interleavings; tensor-core work (MMAs, commits, per issuer in order) and the
query's bulk copy complete asynchronously at random later points.

Checked at every step:
- a parity wait for phase i starts only once phase i - 1 has completed (else
  the hardware's parity test would pass at once, on the phase two back) and
  its barrier never completes phase i + 1 while it still waits (else the
  waiter would miss its phase);
- a generic write (dequantised chunk, P, TMEM rescale) never overlaps an MMA
  or copy still in flight that reads or writes the same buffer;
- an MMA reads only buffers completely written for its tile, and a worker
  reads an accumulator (S, O, row sums) only when no MMA is writing it and it
  holds the tile the worker expects.
Mutations (each wait taken out in turn, among them the P slot reused without
waiting for the row-sum MMAs, the race a full-size two-token GPU test
exposed) must be caught, except two that the model shows implied by other
waits, kept as explicit guards: the rescale's row-sum wait (the P hand-off
comes after every worker's, or on the BF16 cache every parity-0 worker's,
row-sum wait before the RoPE chunk's store) and the issuers' o_free wait (the
issuers wait for every worker's P, written after its epilogue). On the BF16
cache, where one parity stores the RoPE chunk, the epilogue's row-sum wait is
needed."""
import random

import pytest


class Bar:
    def __init__(self, count):
        self.count, self.arrived, self.done = count, 0, 0
        self.waiting = []  # intended phases of blocked waiters


class Hazard(AssertionError):
    pass


class Sim:
    def __init__(self, n_tiles, last, resc, seed, drop=None, bf16=False):
        self.rng = random.Random(seed)
        # how often the tensor core and the copy engine get to finish work,
        # against the threads' steps: some runs have a very slow tensor core
        self.async_weight = self.rng.choice([1.0, 0.3, 0.05])
        self.n = n_tiles
        self.last = last  # last[t]: tile t ends a segment
        self.first = [t == 0 or last[t - 1] for t in range(n_tiles)]
        self.unit = []
        u = 0
        for t in range(n_tiles):
            self.unit.append(u)
            if last[t]:
                u += 1
        self.resc = resc  # resc[t]: the softmax of tile t raises the reference
        self.drop = drop  # the name of one wait to leave out (a mutation), or None
        # bf16: the BF16-cache path, whose workers store chunks 2 kc + parity for
        # kc = 0..4 (the RoPE chunk 8 by parity 0 only), each after a PV wait
        self.bf16 = bf16
        self.bars = {"pv_done": Bar(4), "rs_done": Bar(1), "s_full": Bar(2), "p_full": Bar(8),
                     "p_fixed": Bar(8), "o_free": Bar(8), "q_full": Bar(1), "grp": Bar(8)}
        for k in range(9):
            self.bars["chunk%d" % k] = Bar(8 if k == 8 and not bf16 else 4)
        self.parts = {}  # (buffer, version) -> set of writer parts
        self.state = {}  # accumulator / copied buffer -> completed version
        self.fifo = {j: [] for j in range(4)}  # per issuer: in-order async ops
        self.copies = []
        self.actors = {("w", w): self.worker(w) for w in range(8)}
        self.actors.update({("i", j): self.issuer(j) for j in range(4)})
        self.cur = {a: None for a in self.actors}

    # ---------------------------------------------------------------- programs
    def worker(self, w):
        par, q4 = w >> 2, w & 3
        gph = 0

        def sync():
            nonlocal gph
            yield ("arrive", "grp")
            yield ("wait", "grp", gph)
            gph += 1

        pending = None
        for t in range(self.n):
            if self.drop != "worker_pv":
                yield ("wait", "pv_done", t - 1)  # the previous tile's PV has released every slot
            if self.bf16:
                for kc in range(5):
                    k = 2 * kc + par
                    if k > 8:
                        break
                    if k == 8 and self.drop != "rope_rs":
                        yield ("wait", "rs_done", t - 1)
                    if kc > 0 and self.drop != "worker_pv":
                        yield ("wait", "pv_done", t - 1)
                    if k == 8:
                        yield ("write", "slot8", ("rope", t), q4)
                    else:
                        yield ("write", "slot%d" % k, t, q4)
                    yield ("arrive", "chunk%d" % k)
            else:
                for kc in range(4):
                    k = 2 * kc + par
                    yield ("write", "slot%d" % k, t, q4)
                    yield ("arrive", "chunk%d" % k)
                if self.drop != "rope_rs":
                    yield ("wait", "rs_done", t - 1)  # the slot held P, read by the row-sum MMAs
                yield ("write", "slot8", ("rope", t), w)
                yield ("arrive", "chunk8")
            if pending is not None:  # the previous segment's results
                e = pending
                if q4 == 0:
                    if self.drop != "epi_rs":
                        yield ("wait", "rs_done", e)
                    yield ("read", "L", e)
                yield from sync()
                yield from sync()
                for i in range(4):
                    yield ("read", "O%d" % i, e)
                yield ("arrive", "o_free")
                pending = None
            if self.drop != "s_full":
                yield ("wait", "s_full", t)
            yield ("read", "S0", t)
            yield ("read", "S1", t)
            if self.first[t]:
                yield from sync()
                yield from sync()
            yield ("write", "slot8", ("p", t), w)
            yield ("arrive", "p_full")
            yield ("wait", "p_full", t)
            if self.resc[t]:
                yield from sync()
                yield from sync()
                if not self.first[t]:
                    if self.drop != "resc_rs":
                        yield ("wait", "rs_done", t - 1)
                    for b in ("O0", "O1", "O2", "O3", "L"):
                        yield ("tmem_rw", b, t - 1)
                yield ("write", "slot8", ("p", t), w)
                yield ("arrive", "p_fixed")
            if self.last[t]:
                pending = t
        if pending is not None:
            yield ("wait", "pv_done", self.n - 1)
            e = pending
            if q4 == 0:
                if self.drop != "epi_rs":
                    yield ("wait", "rs_done", e)
                yield ("read", "L", e)
            yield from sync()
            yield from sync()
            for i in range(4):
                yield ("read", "O%d" % i, e)
            yield ("arrive", "o_free")

    def issuer(self, j):
        seg = nresc = 0
        if j == 0:
            yield ("copy", "Q", self.unit[0], "q_full")
        for t in range(self.n):
            if self.first[t] and self.drop != "q_full":
                yield ("wait", "q_full", seg)
            if j < 2:
                for k in range(9):
                    if self.drop != "chunk":
                        yield ("wait", "chunk%d" % k, t)
                    src = ("slot8", ("rope", t), 4 if self.bf16 else 8) if k == 8 else ("slot%d" % k, t, 4)
                    yield ("mma", j, [src, ("Q", self.unit[t], None)], ["S%d" % j], t)
                yield ("commit", j, "s_full")
            if self.drop != "issuer_p_full":
                yield ("wait", "p_full", t)
            if self.resc[t]:
                if self.drop != "p_fixed":
                    yield ("wait", "p_fixed", nresc)
                nresc += 1
            if j == 0 and self.last[t] and t + 1 < self.n:
                yield ("copy", "Q", self.unit[t + 1], "q_full")
            if self.first[t] and seg > 0 and self.drop != "o_free":
                yield ("wait", "o_free", seg - 1)
            yield ("mma", j, [("slot%d" % (2 * j), t, 4), ("slot%d" % (2 * j + 1), t, 4), ("slot8", ("p", t), 8)],
                   ["O%d" % j], t)
            yield ("commit", j, "pv_done")
            if j == 3:
                yield ("mma", j, [("slot8", ("p", t), 8)], ["L"], t)
                yield ("commit", j, "rs_done")
            if self.last[t]:
                seg += 1

    # ---------------------------------------------------------------- semantics
    def inflight(self):
        for j in range(4):
            for op in self.fifo[j]:
                if op[0] == "mma":
                    yield op
        for c in self.copies:
            yield ("mma", None, [], [c[0]], None)

    def touching(self, buf, writes_only=False):
        for op in self.inflight():
            if buf in op[3] or (not writes_only and any(r[0] == buf for r in op[2])):
                return True
        return False

    def complete_phase(self, name):
        b = self.bars[name]
        b.done += 1
        for i in b.waiting:
            if b.done > i + 1:
                raise Hazard(f"{name}: a waiter for phase {i} missed it ({b.done} phases done)")

    def arrive(self, name):
        b = self.bars[name]
        b.arrived += 1
        if b.arrived == b.count:
            b.arrived = 0
            self.complete_phase(name)

    def enabled(self, op):
        return op[0] != "wait" or self.bars[op[1]].done >= op[2] + 1

    def start(self, actor, op):
        if op[0] == "wait":
            b = self.bars[op[1]]
            if b.done < op[2]:
                raise Hazard(f"{actor} waits for {op[1]} phase {op[2]} with only {b.done} done: "
                             "the parity test would pass on an older phase")
            b.waiting.append(op[2])

    def execute(self, actor, op):
        kind = op[0]
        if kind == "wait":
            self.bars[op[1]].waiting.remove(op[2])
        elif kind == "arrive":
            self.arrive(op[1])
        elif kind == "write":
            _, buf, ver, part = op
            if self.touching(buf):
                raise Hazard(f"{actor} writes {buf} {ver} while an MMA or copy on it is in flight")
            self.parts.setdefault((buf, ver), set()).add(part)
        elif kind in ("read", "tmem_rw"):
            _, buf, ver = op
            if self.touching(buf, writes_only=kind == "read"):
                raise Hazard(f"{actor} accesses {buf} while an MMA writes it")
            if self.state.get(buf) != ver:
                raise Hazard(f"{actor} expects {buf} of tile {ver}, holds {self.state.get(buf)}")
        elif kind == "mma":
            _, j, reads, writes, t = op
            for buf, ver, nparts in reads:
                if nparts is None:
                    if self.state.get(buf) != ver:
                        raise Hazard(f"issuer {j} reads {buf} {ver} before its copy landed")
                elif len(self.parts.get((buf, ver), ())) != nparts:
                    raise Hazard(f"issuer {j} reads {buf} {ver} before it is written")
            for buf in writes:
                for other in range(4):
                    if other != j and any(buf in o[3] for o in self.fifo[other] if o[0] == "mma"):
                        raise Hazard(f"issuers {j} and {other} write {buf} at once")
            self.fifo[j].append(("mma", j, reads, writes, t))
        elif kind == "commit":
            self.fifo[op[1]].append(("commit", op[2]))
        elif kind == "copy":
            _, buf, ver, bar = op
            if self.touching(buf):
                raise Hazard(f"copy into {buf} while an MMA reads it")
            self.copies.append((buf, ver, bar))

    def async_step(self, src):
        if src == "copy":
            buf, ver, bar = self.copies.pop(0)
            self.state[buf] = ver
            self.arrive(bar)
            return
        op = self.fifo[src].pop(0)
        if op[0] == "mma":
            for buf in op[3]:
                self.state[buf] = op[4]
        else:
            self.arrive(op[1])

    def run(self, max_steps=200000):
        for _ in range(max_steps):
            for a, g in self.actors.items():
                if self.cur[a] is None and g is not None:
                    try:
                        self.cur[a] = next(g)
                        self.start(a, self.cur[a])
                    except StopIteration:
                        self.actors[a] = None
            threads = [("a", a) for a, op in self.cur.items() if op is not None and self.enabled(op)]
            engines = [("q", j) for j in range(4) if self.fifo[j]]
            if self.copies:
                engines.append(("q", "copy"))
            if not threads and not engines:
                if any(op is not None for op in self.cur.values()):
                    raise Hazard(f"deadlock: {[(a, op) for a, op in self.cur.items() if op is not None]}")
                return
            if engines and (not threads or self.rng.random() < self.async_weight * len(engines) /
                            (len(engines) + len(threads))):
                kind, who = self.rng.choice(engines)
            else:
                kind, who = self.rng.choice(threads)
            if kind == "a":
                op, self.cur[who] = self.cur[who], None
                self.execute(who, op)
            else:
                self.async_step(who)
        raise Hazard("step limit")


def _patterns():
    yield 6, [False] * 5 + [True], [False] * 6                      # one segment
    yield 7, [False, True, False, False, True, False, True], [False, False, True, False, False, True, True]
    yield 5, [True] * 5, [True] * 5                                 # a segment per tile, every tile rescales
    yield 8, [False, False, True, False, False, False, False, True], [False, True, False, True, True, False, False,
                                                                      True]


@pytest.mark.parametrize("pattern", list(range(4)))
def test_protocol_has_no_hazard(pattern):
    n, last, resc = list(_patterns())[pattern]
    for seed in range(150):
        Sim(n, last, resc, seed).run()


@pytest.mark.parametrize("drop", ["rope_rs", "worker_pv", "epi_rs", "s_full", "chunk", "issuer_p_full",
                                  "p_fixed", "q_full"])
def test_model_catches_each_missing_wait(drop):
    # "rope_rs" is the P-slot race: without the row-sum wait before the RoPE
    # chunk's store, some interleaving overwrites P while the row-sum MMAs may
    # still read it.
    caught = 0
    for pattern in range(4):
        n, last, resc = list(_patterns())[pattern]
        for seed in range(60):
            try:
                Sim(n, last, resc, seed, drop=drop).run()
            except Hazard:
                caught += 1
    assert caught > 0, drop


@pytest.mark.parametrize("drop", ["resc_rs", "o_free"])
def test_waits_implied_on_the_packed_path(drop):
    # The rescale's row-sum wait follows the RoPE store's wait for the same
    # phase; the issuers' o_free wait follows their wait for every worker's P,
    # which each worker writes after its epilogue. Without either the packed
    # path stays hazard-free.
    for pattern in range(4):
        n, last, resc = list(_patterns())[pattern]
        for seed in range(60):
            Sim(n, last, resc, seed, drop=drop).run()


@pytest.mark.parametrize("pattern", list(range(4)))
def test_bf16_path_has_no_hazard(pattern):
    n, last, resc = list(_patterns())[pattern]
    for seed in range(100):
        Sim(n, last, resc, seed, bf16=True).run()


@pytest.mark.parametrize("drop", ["rope_rs", "epi_rs", "worker_pv", "s_full", "chunk"])
def test_bf16_path_needs_its_waits(drop):
    # On the BF16 cache the RoPE chunk is stored by parity 0 only, so the
    # parity-1 warps reach the epilogue without having waited for the row-sum
    # MMAs: the epilogue's wait is needed there.
    caught = 0
    for pattern in range(4):
        n, last, resc = list(_patterns())[pattern]
        for seed in range(60):
            try:
                Sim(n, last, resc, seed, drop=drop, bf16=True).run()
            except Hazard:
                caught += 1
    assert caught > 0, drop


def test_rescale_wait_implied_on_the_bf16_path():
    for pattern in range(4):
        n, last, resc = list(_patterns())[pattern]
        for seed in range(60):
            Sim(n, last, resc, seed, drop="resc_rs", bf16=True).run()
