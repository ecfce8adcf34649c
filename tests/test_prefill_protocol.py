"""Model check of the chunked-prefill kernel's mbarrier protocol (host only).

`ps_prefill.cu` runs one CTA pair per persistent cluster with these roles per
CTA: a K producer (which also loads Q, double-buffered per unit), a V
producer, the MMA issuer (leader CTA only), and two softmax groups (even and
odd key tiles); at the end of a unit the group that ran its last tile merges
the two halves, after the other group has handed over its (m, l).
Every wait is a parity wait on an mbarrier, which is sound only while the
barrier has completed exactly the awaited phase's predecessor or the awaited
phase itself: one phase further behind and the wait passes at once, one phase
further ahead and it never passes.  A kernel cannot assert that on the
device, so this model replays the protocol with random timings and checks, at
every poll, that the barrier is within that window, and at every step the
data hazards the barriers exist for (a K/V stage reloaded before its tile's
Q K^T and P V finished, P written over an S buffer before the P V reading it
finished, O rescaled or read out before the P V into it finished).

The model follows the kernel's order of operations: tcgen05 MMAs of the one
issuing thread complete in issue order, and a commit completes its barrier
once every MMA issued before it has completed.  Variants with a known
mistake must be caught, which shows the check has teeth: producers gated on
S-full with a phase-0 wait at the first reuse of each stage (an unsound
parity wait), and a dropped O-free or Q-free wait (a data race).
"""
import random

import pytest

STAGES = 4  # K/V ring depth (PS_PREFILL_STAGES)


class _Bar:
    def __init__(self, count):
        self.count, self.pending, self.done = count, 0, 0

    def arrive(self, n=1):
        for _ in range(n):
            self.pending += 1
            if self.pending == self.count:
                self.pending = 0
                self.done += 1


class _Model:
    def __init__(self, units, seed, protocol):
        self.rng = random.Random(seed)
        self.units, self.protocol = units, protocol
        self.errors = []
        self.mma = []       # issued, not yet complete: ('op', key) or ('commit', barrier)
        self.finished = set()
        self.o_read = set()  # (rank, unit): the merging group has read O_0 and O_1 of the unit
        self.xs = {}         # rank -> ('written', unit) or the last unit read
        self.last_qk = {}    # unit -> global index of its last tile
        b = {}
        for st in range(STAGES):
            b['kvfull', st] = _Bar(4)  # K and V arrival of each CTA
            b['kvfree', st] = _Bar(1)
        for i in range(2):
            b['q', i] = _Bar(2)        # one Q arrival per CTA
            b['qfree', i] = _Bar(1)
            b['sfull', i] = _Bar(1)
            b['pfull', i] = _Bar(8)    # the group's four warps in each CTA
        b['ofree'] = _Bar(8)           # the merging group's four warps in each CTA
        for r in range(2):
            b['xfull', r] = _Bar(1)    # per CTA: (m, l) hand-off to the merging group
            b['xempty', r] = _Bar(1)
        self.b = b

    def ready(self, name, k):
        """One poll of a parity wait for phase k of barrier `name`."""
        c = self.b[name].done
        if not (k <= c <= k + 1):
            self.errors.append('parity wait on %s for phase %d while %d phases are complete' % (name, k, c))
            return True
        return c == k + 1

    def pause(self, hi):
        for _ in range(self.rng.randint(0, hi)):
            yield

    # ----------------------------------------------------------- roles --
    def producer(self, rank, is_k):
        issued = 0
        for ui, nt in enumerate(self.units):
            if is_k:
                qb = ui & 1
                if ui >= 2 and self.protocol != 'no_qfree_wait':
                    while not self.ready(('qfree', qb), (ui - 2) >> 1):
                        yield
                if ui >= 2 and ('QK', self.last_qk[ui - 2]) not in self.finished:
                    self.errors.append('Q buffer %d reloaded before the last Q K^T of unit %d' % (qb, ui - 2))
                yield from self.pause(3)
                self.b['q', qb].arrive()
            for _ in range(nt):
                i, st = issued, issued % STAGES
                if self.protocol != 'sfull_gate':
                    if i >= STAGES:
                        while not self.ready(('kvfree', st), i // STAGES - 1):
                            yield
                else:  # S-full gate with a phase-0 wait at each S buffer's first reuse
                    if STAGES <= i < STAGES + 2:
                        while not self.ready(('sfull', (i - STAGES) & 1), 0):
                            yield
                    if i >= STAGES:
                        while not self.ready(('sfull', (i - 2) & 1), (i - 2) >> 1):
                            yield
                old = i - STAGES
                if old >= 0 and not {('QK', old), ('PV', old)} <= self.finished:
                    self.errors.append('stage %d reloaded for tile %d before tile %d was consumed' % (st, i, old))
                yield from self.pause(4)
                self.b['kvfull', st].arrive()
                issued += 1
                yield

    def issuer(self):
        t0 = 0
        for ui, nt in enumerate(self.units):
            qb = ui & 1
            while not self.ready(('q', qb), ui >> 1):
                yield
            for n in range(nt + 1):
                if n < nt:
                    t = t0 + n
                    while not self.ready(('kvfull', t % STAGES), t // STAGES):
                        yield
                    self.mma += [('op', ('QK', t)), ('commit', ('sfull', t & 1))]
                    if n == nt - 1:
                        self.mma.append(('commit', ('qfree', qb)))
                    yield
                if n >= 1:
                    t = t0 + n - 1
                    while not self.ready(('pfull', t & 1), t >> 1):
                        yield
                    if n == 1 and ui > 0:
                        if self.protocol != 'no_ofree_wait':
                            while not self.ready('ofree', ui - 1):
                                yield
                        if not {(0, ui - 1), (1, ui - 1)} <= self.o_read:
                            self.errors.append('P V of unit %d overwrites O before unit %d was read out' % (ui, ui - 1))
                    self.mma += [('op', ('PV', t)), ('commit', ('kvfree', t % STAGES))]
                    yield
            t0 += nt

    def softmax(self, rank, G):
        t0 = 0
        for ui, nt in enumerate(self.units):
            for n in range(0 if (t0 & 1) == G else 1, nt, 2):
                t = t0 + n
                while not self.ready(('sfull', G), t >> 1):
                    yield
                if n >= 2 and self.rng.random() < 0.5:  # the lazy rescale of O_G
                    while not self.ready(('kvfree', (t - 2) % STAGES), (t - 2) // STAGES):
                        yield
                    if ('PV', t - 2) not in self.finished:
                        self.errors.append('O rescaled before the P V of tile %d' % (t - 2))
                if t >= 2 and ('PV', t - 2) not in self.finished:
                    self.errors.append('P of tile %d written over S before the P V of tile %d' % (t, t - 2))
                yield from self.pause(6)
                self.b['pfull', G].arrive(4)
            last = t0 + nt - 1
            merger = last & 1  # the group of the unit's last tile merges
            if G != merger:
                if ui > 0:
                    while not self.ready(('xempty', rank), ui - 1):
                        yield
                if self.xs.get(rank, -1) != ui - 1:
                    self.errors.append('hand-off of unit %d overwrites one not yet read' % ui)
                self.xs[rank] = ('written', ui)
                self.b['xfull', rank].arrive()
            else:
                while not self.ready(('xfull', rank), ui):
                    yield
                # After the hand-off group 1's last softmax has passed its S-full
                # wait, so every P V up to tile last - 3 is complete: the
                # barrier of the unit's last P V is at most one phase behind.
                while not self.ready(('kvfree', last % STAGES), last // STAGES):
                    yield
                missing = [t for t in range(t0, t0 + nt) if ('PV', t) not in self.finished]
                if missing:
                    self.errors.append('O read out before the P V of tiles %s' % missing)
                if self.xs.get(rank) != ('written', ui):
                    self.errors.append('merge of unit %d read a hand-off that is not its own' % ui)
                self.xs[rank] = ui
                self.b['xempty', rank].arrive()
                yield from self.pause(3)
                self.o_read.add((rank, ui))
                self.b['ofree'].arrive(4)
            t0 += nt

    def run(self, max_steps=200000):
        t = 0
        for ui, nt in enumerate(self.units):
            t += nt
            self.last_qk[ui] = t - 1
        roles = [self.producer(r, k) for r in range(2) for k in (True, False)]
        roles += [self.issuer()] + [self.softmax(r, G) for r in range(2) for G in range(2)]
        for _ in range(max_steps):
            if not roles and not self.mma:
                return self.errors
            if self.mma and self.rng.random() < 0.3:  # the oldest MMA completes
                kind, what = self.mma.pop(0)
                if kind == 'op':
                    self.finished.add(what)
                else:
                    self.b[what].arrive()
                while self.mma and self.mma[0][0] == 'commit':
                    self.b[self.mma.pop(0)[1]].arrive()
            self.rng.shuffle(roles)
            for r in list(roles):
                try:
                    next(r)
                except StopIteration:
                    roles.remove(r)
            if self.errors:
                return self.errors
        return self.errors + ['no progress: a wait never passed']


def _schedules(n, seed):
    rng = random.Random(seed)
    for k in range(n):
        # a cluster's list of units, each 1..7 key tiles (one-tile units included)
        yield k, [rng.randint(1, 7) for _ in range(rng.randint(1, 9))]


@pytest.mark.parametrize('block', range(4))
def test_kernel_protocol_waits_stay_in_their_parity_window(block):
    for k, units in _schedules(150, 1000 + block):
        errors = _Model(units, seed=block * 1000 + k, protocol='kernel').run()
        assert not errors, (units, errors[:3])


def test_long_unit_lists_complete():
    rng = random.Random(5)
    units = [rng.randint(1, 30) for _ in range(16)]
    for seed in range(10):
        assert not _Model(units, seed, 'kernel').run(), seed


def test_model_catches_an_unsound_first_reuse_wait():
    # Gating the stage reload on S-full with a phase-0 wait at the first reuse
    # lets that wait find S-full two phases ahead (tiles 0 and 2 done): the
    # parity wait would then never pass.  The model must see it.
    caught = sum(1 for k, units in _schedules(300, 77) if _Model(units, k, 'sfull_gate').run())
    assert caught > 0



@pytest.mark.parametrize('protocol', ['no_ofree_wait', 'no_qfree_wait'])
def test_model_catches_a_dropped_wait(protocol):
    # A unit's first P V overwrites both O accumulators, and a Q buffer is
    # reused two units later: without their waits some schedules must race.
    caught = sum(1 for k, units in _schedules(300, 78) if _Model(units, k, protocol).run())
    assert caught > 0
