"""Model of the window kernels' epilogue exchange protocol, run on the CPU.

The epilogue groups of a lane quarter hand partial results to a rotating
merging group through shared-memory slots guarded by two mbarriers per slot
(x_full: the three other groups have written; x_empty: the merging group has
read), while all sixteen epilogue warps and the MMA thread share a ring of
TMEM buffers (t_full / t_empty).  mbarrier waits test a phase parity, so a
wait is unambiguous only when the barrier's previous phase has completed.
The model runs the same sequence of waits and arrivals as the kernels, with
mbarrier parity semantics and random interleavings, and checks that every
schedule finishes and that a merging group only reads a slot in the phase it
expects.  The variant in which the merging group does not first wait for the
slot's previous read (the kernels' earlier protocol) fails the same check.
"""

import random

import pytest


class Barrier:
    def __init__(self, count):
        self.count, self.pending, self.phase = count, count, 0

    def arrive(self):
        self.pending -= 1
        assert self.pending >= 0
        if self.pending == 0:
            self.phase += 1
            self.pending = self.count

    def passes(self, parity):
        # mbarrier.try_wait.parity: true unless the current phase has that parity
        return (self.phase & 1) != parity


def simulate(items, jobs_per_tile, nbuf, slots, per_chunk, merger_waits_empty, seed):
    """items: tiles of each work item of one CTA; per_chunk: merge once per
    item (pass 1) instead of once per tile (pass 2).  Returns None or a fault."""
    rnd = random.Random(seed)
    t_full = [Barrier(1) for _ in range(nbuf)]
    t_empty = [Barrier(16) for _ in range(nbuf)]
    x_full = {(p, q): Barrier(3) for p in range(slots) for q in range(4)}
    x_empty = {(p, q): Barrier(1) for p in range(slots) for q in range(4)}
    commits = []  # MMA completions land later than their issue
    reads = []

    def mma():
        for job in range(sum(items) * jobs_per_tile):
            buf, use = job % nbuf, job // nbuf
            while not t_empty[buf].passes((use & 1) ^ 1):
                yield
            commits.append(t_full[buf])
            yield

    def epilogue(q, g):
        job = n = 0
        for tiles in items:
            for t in range(tiles):
                for _ in range(jobs_per_tile):
                    buf, use = job % nbuf, job // nbuf
                    job += 1
                    while not t_full[buf].passes(use & 1):
                        yield
                    yield
                    t_empty[buf].arrive()
                if per_chunk and t != tiles - 1:
                    continue
                par, use, merger = n % slots, n // slots, n & 3
                n += 1
                ph = use & 1
                if g != merger or merger_waits_empty:
                    while not x_empty[(par, q)].passes(ph ^ 1):
                        yield
                if g != merger:
                    yield
                    x_full[(par, q)].arrive()
                else:
                    while not x_full[(par, q)].passes(ph):
                        yield
                    reads.append((use, x_full[(par, q)].phase))
                    yield
                    x_empty[(par, q)].arrive()

    procs = [mma()] + [epilogue(q, g) for q in range(4) for g in range(4)]
    live = list(range(len(procs)))
    for _ in range(200000):
        if not live:
            break
        if commits and rnd.random() < 0.3:
            commits.pop(0).arrive()
        i = rnd.choice(live)
        try:
            next(procs[i])
        except StopIteration:
            live.remove(i)
    else:
        return "deadlock"
    for use, phase in reads:
        if phase != use + 1:
            return f"read of use {use} while x_full is in phase {phase}"
    return None


def _cases():
    rng = random.Random(7)
    out = []
    for _ in range(12):
        items = [rng.choice([1, 2, 3, 8, 8]) for _ in range(rng.randint(1, 5))]
        out.append(("pass2_one_job_four_buffers", items, 1, 4, 2, False))
        out.append(("pass2_two_jobs_two_buffers", items, 2, 2, 2, False))
        out.append(("pass1", items, rng.choice([1, 2, 3, 4]), 4, 1, True))
    return out


@pytest.mark.parametrize("name,items,jobs,nbuf,slots,per_chunk", _cases())
def test_protocol_finishes_and_reads_in_phase(name, items, jobs, nbuf, slots, per_chunk):
    for seed in range(6):
        fault = simulate(items, jobs, nbuf, slots, per_chunk, True, seed)
        assert fault is None, (name, items, seed, fault)


def test_model_catches_the_unguarded_merger():
    # one job per tile and four TMEM buffers let a group run two tiles ahead;
    # without the extra wait the merging group's x_full wait passes early
    faults = [simulate([8, 1], 1, 4, 2, False, False, seed) for seed in range(6)]
    assert any(f is not None for f in faults)
