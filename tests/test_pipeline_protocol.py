"""Model of the window kernels' synchronisation, run on the CPU.

One CTA of a window pass has a producer (TMA loads of K tiles into a ring of
stages and of the window rows into one or two slots), an MMA thread (waits
for the operands and for free TMEM buffers, commits its MMAs to mbarriers)
and sixteen epilogue warps (wait for accumulators, free the buffers, and hand
partial results to a rotating merging group through shared-memory slots
guarded by x_full / x_empty barriers).  mbarrier waits test a phase parity,
so each wait is correct only while the barrier is exactly one phase past the
one the waiter expects when the wait returns.  The model replays the
kernels' sequence of waits and arrivals (TMA completions and MMA commits
arrive asynchronously, commits in issue order) under random interleavings,
on work lists cut the way the kernels cut them (each CTA a contiguous range
of 1024-token chunks over (request, layer, kv-head) units), and checks that
every schedule finishes and every wait returns in its own phase.  The
variant in which the merging group does not first wait for the slot's
previous read (the kernels' earlier protocol) fails the check.  The one-pass
kernel (logits resident in TMEM, two CTA-wide syncs per unit) is modelled
the same way, and so is the abort path: with one K-tile load withheld (the
failure-detection test's injected missing arrival), every role's bounded
wait gives up, the CTA drains the copies it issued and every role finishes.
"""

import random

import pytest


class Bar:
    """An mbarrier: `count` arrivals complete a phase."""

    def __init__(self, count, name):
        self.count, self.pending, self.phase, self.name = count, count, 0, name

    def arrive(self):
        self.pending -= 1
        assert self.pending >= 0, self.name
        if self.pending == 0:
            self.phase += 1
            self.pending = self.count


class Fault(Exception):
    pass


def wait(bar, k):
    """Generator: wait for completion of phase k with a parity test; checks the
    barrier is exactly one phase past k when the wait returns."""
    while (bar.phase & 1) == (k & 1):
        yield
    if bar.phase != k + 1:
        raise Fault(f"{bar.name}: waited for phase {k}, barrier at phase {bar.phase}")


def simulate(chunks, n_tiles, tpc, jobs_per_tile, nbuf, stages, q_slots, pass2, guard, seed):
    """chunks: the CTA's list of (unit, chunk index); n_tiles: tiles per unit."""
    rnd = random.Random(seed)
    t_full = [Bar(1, f"t_full{i}") for i in range(nbuf)]
    t_empty = [Bar(16, f"t_empty{i}") for i in range(nbuf)]
    k_full = [Bar(1, f"k_full{i}") for i in range(stages)]
    k_empty = [Bar(1, f"k_empty{i}") for i in range(stages)]
    q_full = [Bar(2 if pass2 else 1, f"q_full{i}") for i in range(q_slots)]
    q_empty = [Bar(1, f"q_empty{i}") for i in range(q_slots)]
    x_full = {(p, q): Bar(3, f"x_full{p}{q}") for p in range(2) for q in range(4)}
    x_empty = {(p, q): Bar(1, f"x_empty{p}{q}") for p in range(2) for q in range(4)}
    drain = Bar(1, "drain")
    tma = []       # pending TMA completions (any order)
    commits = []   # pending MMA-commit arrivals (in issue order)

    def tiles_of(ci):
        return range(ci * tpc, min(n_tiles, (ci + 1) * tpc))

    def producer():
        cur, qloads, kt = -1, 0, 0
        for u, ci in chunks:
            if u != cur:
                slot, use = qloads % q_slots, qloads // q_slots
                yield from wait(q_empty[slot], use - 1)
                tma.append(q_full[slot])
                if pass2:
                    yield
                    q_full[slot].arrive()
                qloads += 1
                cur = u
            for _ in tiles_of(ci):
                st, n = kt % stages, kt // stages
                yield from wait(k_empty[st], n - 1)
                tma.append(k_full[st])
                kt += 1
                yield
        for st in range(min(stages, kt)):
            last = kt - 1 - ((kt - 1 - st) % stages)
            yield from wait(k_full[st], last // stages)
        for slot in range(min(q_slots, qloads)):
            last = qloads - 1 - ((qloads - 1 - slot) % q_slots)
            yield from wait(q_full[slot], last // q_slots)

    def mma():
        cur, cur_slot, qwaits, kt, job = -1, 0, 0, 0, 0
        for u, ci in chunks:
            if u != cur:
                if cur >= 0:
                    commits.append(q_empty[cur_slot])
                slot, use = qwaits % q_slots, qwaits // q_slots
                yield from wait(q_full[slot], use)
                qwaits += 1
                cur, cur_slot = u, slot
            for _ in tiles_of(ci):
                st, n = kt % stages, kt // stages
                yield from wait(k_full[st], n)
                kt += 1
                for _ in range(jobs_per_tile):
                    buf, nb = job % nbuf, job // nbuf
                    job += 1
                    yield from wait(t_empty[buf], nb - 1)
                    commits.append(t_full[buf])
                    yield
                commits.append(k_empty[st])
        commits.append(drain)
        yield from wait(drain, 0)

    def epilogue(q, g):
        job = n = 0
        for u, ci in chunks:
            ts = list(tiles_of(ci))
            for i, _ in enumerate(ts):
                for _ in range(jobs_per_tile):
                    buf, nb = job % nbuf, job // nbuf
                    job += 1
                    yield from wait(t_full[buf], nb)
                    yield
                    t_empty[buf].arrive()
                last_of_chunk = i == len(ts) - 1
                if not pass2 and not last_of_chunk:
                    continue
                slots = 2 if pass2 else 1
                par, use, merger = n % slots, n // slots, n & 3
                n += 1
                if g != merger or guard:
                    yield from wait(x_empty[(par, q)], use - 1)
                if g != merger:
                    yield
                    x_full[(par, q)].arrive()
                else:
                    yield from wait(x_full[(par, q)], use)
                    yield
                    x_empty[(par, q)].arrive()

    procs = [producer(), mma()] + [epilogue(q, g) for q in range(4) for g in range(4)]
    live = list(range(len(procs)))
    for _ in range(500000):
        if not live and not tma and not commits:
            return None
        r = rnd.random()
        if tma and r < 0.25:
            tma.pop(rnd.randrange(len(tma))).arrive()
            continue
        if commits and r < 0.5:
            commits.pop(0).arrive()
            continue
        if not live:
            continue
        i = rnd.choice(live)
        try:
            next(procs[i])
        except StopIteration:
            live.remove(i)
        except Fault as f:
            return str(f)
    return "deadlock"

def cta_range(units, chunks_per_unit, total_ctas, cta):
    total = units * chunks_per_unit
    c0, c1 = cta * total // total_ctas, (cta + 1) * total // total_ctas
    return [(g // chunks_per_unit, g % chunks_per_unit) for g in range(c0, c1)]


def _cases(n=40, seed=3):
    rng = random.Random(seed)
    out = []
    while len(out) < n:
        n_tiles = rng.choice([1, 3, 8, 9, 11, 16, 51, 128])
        cpu = -(-n_tiles // 8)
        units = rng.randint(1, 12)
        ctas = rng.randint(1, max(1, units * cpu))
        chunks = cta_range(units, cpu, ctas, rng.randrange(ctas))
        if not chunks or len(chunks) > 24:
            continue
        pass2 = rng.random() < 0.5
        if pass2:
            jobs, nbuf = rng.choice([(1, 4), (2, 2), (2, 4), (1, 2)])
        else:
            jobs, nbuf = rng.choice([1, 2, 3, 4]), 4
        out.append((chunks, n_tiles, jobs, nbuf, rng.choice([2, 3, 4]), rng.choice([1, 2]), pass2))
    return out


@pytest.mark.parametrize("chunks,n_tiles,jobs,nbuf,stages,q_slots,pass2", _cases())
def test_pipeline_finishes_and_waits_in_phase(chunks, n_tiles, jobs, nbuf, stages, q_slots, pass2):
    for seed in range(6):
        fault = simulate(chunks, n_tiles, 8, jobs, nbuf, stages, q_slots, pass2, True, seed)
        assert fault is None, (seed, fault)


def test_model_catches_the_unguarded_merger():
    # one job per tile and four TMEM buffers let an epilogue group run two
    # tiles ahead of another; without the extra wait the merging group's
    # x_full wait passes on the slot's previous phase
    chunks = cta_range(3, 2, 1, 0)
    faults = [simulate(chunks, 11, 8, 1, 4, 4, 1, True, False, s) for s in range(8)]
    assert any(f is not None for f in faults)


# ------------------------------------------------ one-pass kernel

def simulate_onepass(n_units, ntiles, stages, epi_warps, seed):
    """The one-pass kernel: a unit's logits occupy one of two TMEM halves;
    the epilogue warps meet twice per unit at a CTA-wide mbarrier and reuse
    two shared-memory buffers of partials (row maxima, row sums)."""
    rnd = random.Random(seed)
    k_full = [Bar(1, f"k_full{i}") for i in range(stages)]
    k_empty = [Bar(1, f"k_empty{i}") for i in range(stages)]
    q_full = [Bar(1, f"q_full{i}") for i in range(2)]
    q_empty = [Bar(1, f"q_empty{i}") for i in range(2)]
    t_full = [Bar(1, f"t_full{i}") for i in range(2)]
    t_empty = [Bar(epi_warps, f"t_empty{i}") for i in range(2)]
    e_sync = Bar(epi_warps, "e_sync")
    drain = Bar(1, "drain")
    tma, commits = [], []
    xr, xs = {}, {}

    def producer():
        kt = 0
        for n in range(n_units):
            yield from wait(q_empty[n & 1], (n >> 1) - 1)
            tma.append(q_full[n & 1])
            for _ in range(ntiles):
                st, m = kt % stages, kt // stages
                yield from wait(k_empty[st], m - 1)
                tma.append(k_full[st])
                kt += 1
                yield

    def mma():
        kt = 0
        for n in range(n_units):
            yield from wait(q_full[n & 1], n >> 1)
            yield from wait(t_empty[n & 1], (n >> 1) - 1)
            for _ in range(ntiles):
                st, m = kt % stages, kt // stages
                yield from wait(k_full[st], m)
                kt += 1
                yield
                commits.append(k_empty[st])
            commits.append(t_full[n & 1])
            commits.append(q_empty[n & 1])
        commits.append(drain)
        yield from wait(drain, 0)

    def epilogue(w):
        nsync = 0
        for n in range(n_units):
            yield from wait(t_full[n & 1], n >> 1)
            xr[w] = n
            yield
            e_sync.arrive()
            yield from wait(e_sync, nsync)
            nsync += 1
            if any(xr[v] != n for v in range(epi_warps)):
                raise Fault(f"row maxima of unit {n} overwritten before they were read")
            xs[w] = n
            yield
            e_sync.arrive()
            yield from wait(e_sync, nsync)
            nsync += 1
            if any(xs[v] != n for v in range(epi_warps)):
                raise Fault(f"row sums of unit {n} overwritten before they were read")
            yield
            t_empty[n & 1].arrive()

    procs = [producer(), mma()] + [epilogue(w) for w in range(epi_warps)]
    live = list(range(len(procs)))
    for _ in range(300000):
        if not live and not tma and not commits:
            return None
        r = rnd.random()
        if tma and r < 0.25:
            tma.pop(rnd.randrange(len(tma))).arrive()
            continue
        if commits and r < 0.5:
            commits.pop(0).arrive()
            continue
        if not live:
            continue
        i = rnd.choice(live)
        try:
            next(procs[i])
        except StopIteration:
            live.remove(i)
        except Fault as f:
            return str(f)
    return "deadlock"


@pytest.mark.parametrize("n_units,ntiles,stages", [(1, 1, 4), (3, 5, 2), (7, 8, 4), (9, 8, 3),
                                                   (6, 1, 4), (4, 7, 3)])
def test_onepass_protocol(n_units, ntiles, stages):
    for seed in range(6):
        fault = simulate_onepass(n_units, ntiles, stages, 8, seed)
        assert fault is None, (seed, fault)


# ------------------------------------------------ abort path (missing arrival)

def simulate_abort(chunks, n_tiles, tpc, jobs_per_tile, nbuf, stages, q_slots, pass2, seed,
                   limit=400):
    """The two-pass kernel with the first K-tile load withheld.  Waits are
    bounded (`limit` polls stand for the clock limit) and also give up once
    the CTA's abort flag is set, except the drains, which only have the
    clock; a role whose wait gives up raises the flag and leaves its loops,
    as the kernels do.  Returns None when every role finishes with no copy
    still in flight, else what went wrong."""
    rnd = random.Random(seed)
    t_full = [Bar(1, f"t_full{i}") for i in range(nbuf)]
    t_empty = [Bar(16, f"t_empty{i}") for i in range(nbuf)]
    k_full = [Bar(1, f"k_full{i}") for i in range(stages)]
    k_empty = [Bar(1, f"k_empty{i}") for i in range(stages)]
    q_full = [Bar(2 if pass2 else 1, f"q_full{i}") for i in range(q_slots)]
    q_empty = [Bar(1, f"q_empty{i}") for i in range(q_slots)]
    x_full = {(p, q): Bar(3, f"x_full{p}{q}") for p in range(2) for q in range(4)}
    x_empty = {(p, q): Bar(1, f"x_empty{p}{q}") for p in range(2) for q in range(4)}
    drain = Bar(1, "drain")
    tma, commits = [], []
    abort = [False]
    ok = {}

    def bwait(bar, k, key, flag=True):
        """Bounded wait; its outcome lands in ok[key]."""
        polls = 0
        while (bar.phase & 1) == (k & 1):
            if (flag and abort[0]) or polls > limit:
                ok[key] = False
                return
            polls += 1
            yield
        ok[key] = True

    def tiles_of(ci):
        return range(ci * tpc, min(n_tiles, (ci + 1) * tpc))

    def producer():
        cur, qloads, kt = -1, 0, 0
        good = True
        for u, ci in chunks:
            if u != cur:
                slot, use = qloads % q_slots, qloads // q_slots
                yield from bwait(q_empty[slot], use - 1, "p")
                if not ok["p"]:
                    good = False
                    break
                tma.append(q_full[slot])
                if pass2:
                    yield
                    q_full[slot].arrive()
                qloads += 1
                cur = u
            for _ in tiles_of(ci):
                st, n = kt % stages, kt // stages
                yield from bwait(k_empty[st], n - 1, "p")
                if not ok["p"]:
                    good = False
                    break
                if kt > 0:          # the first load is withheld
                    tma.append(k_full[st])
                kt += 1
                yield
            if not good:
                break
        if not good:
            abort[0] = True
        for st in range(min(stages, kt)):
            last = kt - 1 - ((kt - 1 - st) % stages)
            yield from bwait(k_full[st], last // stages, "pd", flag=False)
        for slot in range(min(q_slots, qloads)):
            last = qloads - 1 - ((qloads - 1 - slot) % q_slots)
            yield from bwait(q_full[slot], last // q_slots, "pd", flag=False)

    def mma():
        cur, cur_slot, qwaits, kt, job = -1, 0, 0, 0, 0
        good = True
        for u, ci in chunks:
            if u != cur:
                if cur >= 0:
                    commits.append(q_empty[cur_slot])
                slot, use = qwaits % q_slots, qwaits // q_slots
                yield from bwait(q_full[slot], use, "m")
                if not ok["m"]:
                    good = False
                    break
                qwaits += 1
                cur, cur_slot = u, slot
            for _ in tiles_of(ci):
                st, n = kt % stages, kt // stages
                yield from bwait(k_full[st], n, "m")
                if not ok["m"]:
                    good = False
                    break
                if st == 0 and n == 0:
                    raise Fault("an MMA read the K stage whose load never arrived")
                kt += 1
                for _ in range(jobs_per_tile):
                    buf, nb = job % nbuf, job // nbuf
                    job += 1
                    yield from bwait(t_empty[buf], nb - 1, "m")
                    if not ok["m"]:
                        good = False
                        break
                    commits.append(t_full[buf])
                    yield
                if not good:
                    break
                commits.append(k_empty[st])
            if not good:
                break
        if not good:
            abort[0] = True
        commits.append(drain)
        yield from bwait(drain, 0, "md", flag=False)
        if not ok["md"]:
            raise Fault("the MMA drain did not complete")

    def epilogue(q, g):
        job = n = 0
        key = f"e{q}{g}"
        for u, ci in chunks:
            ts = list(tiles_of(ci))
            for i, _ in enumerate(ts):
                for _ in range(jobs_per_tile):
                    buf, nb = job % nbuf, job // nbuf
                    job += 1
                    yield from bwait(t_full[buf], nb, key)
                    if not ok[key]:
                        abort[0] = True
                        return
                    yield
                    t_empty[buf].arrive()
                if not pass2 and i != len(ts) - 1:
                    continue
                slots = 2 if pass2 else 1
                par, use, merger = n % slots, n // slots, n & 3
                n += 1
                yield from bwait(x_empty[(par, q)], use - 1, key)
                if not ok[key]:
                    abort[0] = True
                    return
                if g != merger:
                    yield
                    x_full[(par, q)].arrive()
                else:
                    yield from bwait(x_full[(par, q)], use, key)
                    if not ok[key]:
                        abort[0] = True
                        return
                    yield
                    x_empty[(par, q)].arrive()

    procs = [producer(), mma()] + [epilogue(q, g) for q in range(4) for g in range(4)]
    live = list(range(len(procs)))
    for _ in range(2000000):
        if not live:
            if tma:
                return "a copy was still in flight when the CTA finished"
            return None if abort[0] else "no role noticed the missing arrival"
        r = rnd.random()
        if tma and r < 0.25:
            tma.pop(rnd.randrange(len(tma))).arrive()
            continue
        if commits and r < 0.5:
            commits.pop(0).arrive()
            continue
        i = rnd.choice(live)
        try:
            next(procs[i])
        except StopIteration:
            live.remove(i)
        except Fault as f:
            return str(f)
    return "deadlock"


@pytest.mark.parametrize("chunks,n_tiles,jobs,nbuf,stages,q_slots,pass2", _cases(12, seed=11))
def test_missing_arrival_ends_every_role(chunks, n_tiles, jobs, nbuf, stages, q_slots, pass2):
    for seed in range(3):
        fault = simulate_abort(chunks, n_tiles, 8, jobs, nbuf, stages, q_slots, pass2, seed)
        assert fault is None, (seed, fault)
