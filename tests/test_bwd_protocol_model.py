"""A host-side model of the backward tile kernel's barrier protocol (relation_tc_bwd.cu;
the persistent d_h = 64 form and the one-unit d_h = 128 form with its per-step dQ^T): the
TMA, MMA, elementwise and dQ roles as sequences of mbarrier
waits and arrivals with the phase arithmetic the kernel uses, run under many random
interleavings and unit sequences.  Checks that every role finishes (no deadlock) and that
no wait polls a barrier that has already run two phases past the one it waits for (an
mbarrier parity wait cannot tell those apart).  CPU only; the model mirrors the kernel's
code, it does not run it."""
import random

import pytest

NBUF, NQS, SPT, NKV = 2, 2, 2, 2  # d_h = 64 configuration


class Ambiguous(Exception):
    pass


class Barriers:
    def __init__(self):
        self.done = {}

    def completed(self, name):
        return self.done.get(name, 0)

    def arrive(self, name):  # one arrival completes a phase (each role is one agent here)
        self.done[name] = self.completed(name) + 1

    def ready(self, name, k):
        """A wait for completion k (0-based), as mbarrier parity k & 1 sees it: exact only
        while the barrier has completed k or k + 1 phases.  Two phases ahead the parity
        test would never pass; one phase short (k - 1 completed) it passes at once, as if
        phase k had completed."""
        c = self.completed(name)
        if c >= k + 2:
            raise Ambiguous(f"{name}: waiting for phase {k}, already {c} completed")
        if c <= k - 1:
            raise Ambiguous(f"{name}: waiting for phase {k} with only {c} completed: the "
                            "parity test passes early")
        return c >= k + 1


def tma(units):
    ul, gq0 = 0, 0
    for n_i in units:
        kvb = ul % NKV
        if ul >= NKV:
            yield ("wait", f"KVE{kvb}", (ul - NKV) // NKV)
        yield ("arrive", f"KV{kvb}")
        for u in range(n_i):
            g = gq0 + u
            s, r = g % NQS, g // NQS
            if r > 0:
                yield ("wait", f"QE{s}", r - 1)
            yield ("arrive", f"QF{s}")
        gq0 += n_i
        ul += 1


def mma(units):
    gs0 = gq0 = gt0 = 0
    pre = 0

    def issue_u(ctx_gs0, ctx_gq0, s):
        g = ctx_gq0 + s // SPT
        if s % SPT == 0:
            yield ("wait", f"QF{g % NQS}", g // NQS)

    def issue_dp(ctx_gs0, s):
        yield ("arrive", f"S{(ctx_gs0 + s) % NBUF}")

    for ul, n_i in enumerate(units):
        total = n_i * SPT
        kvb = ul % NKV
        if pre == 0:
            yield ("wait", f"KV{kvb}", ul // NKV)
        sn, pre, units_done = pre, 0, 0
        while sn < total and sn < NBUF:
            yield from issue_u(gs0, gq0, sn)
            yield from issue_dp(gs0, sn)
            sn += 1
        for s in range(total):
            t, hh, g = s // SPT, s % SPT, gs0 + s
            st = (gq0 + s // SPT) % NQS
            yield ("wait", f"P{g % NBUF}", g // NBUF)
            if s == total - 1:
                yield ("arrive", "ACC")
                if ul + 1 < len(units):  # the next unit's first steps, ahead of the last dQ
                    yield ("wait", f"KV{(ul + 1) % NKV}", (ul + 1) // NKV)
                    n_next = units[ul + 1] * SPT
                    while pre < n_next and pre < NBUF:
                        yield from issue_u(gs0 + total, gq0 + n_i, pre)
                        yield from issue_dp(gs0 + total, pre)
                        pre += 1
            if hh == SPT - 1:
                gt = gt0 + t
                if gt > 0:
                    yield ("wait", "DQE", gt - 1)
                yield ("arrive", "DQF")
                yield ("arrive", f"QE{st}")
                units_done += 1
            while sn < total and sn <= s + NBUF and sn // SPT - NQS < units_done:
                yield from issue_u(gs0, gq0, sn)
                yield from issue_dp(gs0, sn)
                sn += 1
        yield ("arrive", f"KVE{kvb}")
        gs0 += total
        gq0 += n_i
        gt0 += n_i


def ew(units):
    gs0 = gq0 = 0
    for ul, n_i in enumerate(units):
        total = n_i * SPT
        for s in range(total):
            g, gu = gs0 + s, gq0 + s // SPT
            yield ("wait", f"S{g % NBUF}", g // NBUF)
            yield ("wait", f"QF{gu % NQS}", gu // NQS)
            if s == 0 and ul > 0:
                yield ("arrive", "STG")
                yield ("wait", "STG", ul - 1)
            yield ("arrive", f"P{g % NBUF}")
        yield ("wait", "ACC", ul)
        gs0 += total
        gq0 += n_i


def dq(units):
    gt0 = 0
    for n_i in units:
        for i in range(n_i):
            yield ("wait", "DQF", gt0 + i)
            yield ("arrive", "DQE")
        gt0 += n_i


def run(units, seed):
    rng = random.Random(seed)
    bars = Barriers()
    roles = {name: fn(units) for name, fn in (("tma", tma), ("mma", mma), ("ew", ew), ("dq", dq))}
    pending = {name: next(gen, None) for name, gen in roles.items()}
    while any(ev is not None for ev in pending.values()):
        runnable = []
        for name, ev in pending.items():
            if ev is None:
                continue
            if ev[0] == "arrive" or bars.ready(ev[1], ev[2]):
                runnable.append(name)
        if not runnable:
            stuck = {n: e for n, e in pending.items() if e is not None}
            raise AssertionError(f"deadlock with units {units}: {stuck}")
        name = rng.choice(runnable)
        ev = pending[name]
        if ev[0] == "arrive":
            bars.arrive(ev[1])
        pending[name] = next(roles[name], None)


def head_groups(n_t, BH, slots):
    """Number of head groups of the kernels' work order (at least ceil(2.5 slots / (n_t + 1))
    heads per group)."""
    g = max(1, -(-5 * slots // (2 * (n_t + 1))))
    return max(1, BH // g)


def grouped_unit(w, n_t, BH, n_groups):
    """(t, bh) of unit w: heads in n_groups equal groups (the first BH % n_groups one head
    larger), heaviest tiles (t = 0) of a group first."""
    q, r = divmod(BH, n_groups)
    big = r * (q + 1) * n_t
    if w < big:
        g, rem = divmod(w, (q + 1) * n_t)
        base, gs = g * (q + 1), q + 1
    else:
        g, rem = divmod(w - big, q * n_t)
        base, gs = r * (q + 1) + g * q, q
    return rem // gs, base + rem % gs


def cta_units(n_t, BH, grid, c):
    """Units (query tiles per key tile) of CTA c under the zigzag order of the persistent
    kernel (one head group)."""
    n_work, out, r = n_t * BH, [], 0
    while True:
        j = (grid - 1 - c) if (r & 1) else c
        w = r * grid + j
        if w >= n_work:
            return out
        out.append(n_t - grouped_unit(w, n_t, BH, 1)[0])
        r += 1


@pytest.mark.parametrize("n_t,BH,ng", [(128, 32, 10), (128, 32, 3), (16, 96, 4), (5, 7, 2),
                                       (1, 3, 3), (4, 10, 3), (16, 96, 1)])
def test_grouped_order_is_a_permutation(n_t, BH, ng):
    """The grouped work order visits every (key tile, head) unit exactly once, within a group
    the tiles come heaviest first, and the groups' sizes differ by at most one head."""
    seen = [grouped_unit(w, n_t, BH, ng) for w in range(n_t * BH)]
    assert sorted(seen) == sorted((t, bh) for t in range(n_t) for bh in range(BH))
    sizes = [BH // ng + (1 if g < BH % ng else 0) for g in range(ng)]
    w0, h0 = 0, 0
    for gs in sizes:
        chunk = seen[w0:w0 + gs * n_t]
        assert {bh for _, bh in chunk} == set(range(h0, h0 + gs))
        assert [t for t, _ in chunk] == sorted(t for t, _ in chunk)
        w0, h0 = w0 + gs * n_t, h0 + gs
    assert max(sizes) - min(sizes) <= 1 and w0 == n_t * BH


def test_head_groups_cover_the_heaviest_unit():
    for n_t, BH, slots in [(128, 32, 152), (128, 32, 304), (16, 96, 304), (8, 128, 304),
                           (1, 5, 304)]:
        ng = head_groups(n_t, BH, slots)
        smallest = BH // ng
        work_per_slot = smallest * n_t * (n_t + 1) / 2 / slots
        assert ng == 1 or work_per_slot >= 1.25 * n_t


@pytest.mark.parametrize("n_t,BH,grid", [(1, 400, 152), (2, 400, 152), (3, 320, 152),
                                         (8, 128, 152), (16, 96, 152), (5, 7, 3)])
def test_protocol_of_real_unit_sequences(n_t, BH, grid):
    for c in sorted({0, 1, grid // 2, grid - 1}):
        units = cta_units(n_t, BH, grid, c)
        for seed in range(25):
            run(units, seed)


def test_protocol_of_random_unit_sequences():
    rng = random.Random(7)
    for trial in range(150):
        units = [rng.randint(1, 6) for _ in range(rng.randint(1, 5))]
        run(units, trial)


def test_model_detects_a_broken_protocol():
    """The checker itself: without the stage release the TMA waits forever."""
    global mma
    saved = mma

    def mma_without_stage_release(units):
        for ev in saved(units):
            if ev == ("arrive", "QE0") or ev == ("arrive", "QE1"):
                continue
            yield ev
    try:
        mma = mma_without_stage_release
        with pytest.raises(AssertionError, match="deadlock"):
            run([3, 2], 0)
    finally:
        mma = saved


# --- d_h = 128: one unit per CTA, Q/dO staged per 64-query step (three stages), and
# --- dQ^T per step into the step's dP^T columns, read out before the next dP^T

NQS_H = 3


def tma_half(n_i):
    yield ("arrive", "KV0")
    for g in range(n_i * SPT):
        s, r = g % NQS_H, g // NQS_H
        if r > 0:
            yield ("wait", f"QE{s}", r - 1)
        yield ("arrive", f"QF{s}")


def mma_half(n_i):
    total = n_i * SPT

    def issue_u(s):
        yield ("wait", f"QF{s % NQS_H}", s // NQS_H)

    yield ("wait", "KV0", 0)
    for sn in range(min(total, NBUF)):
        yield from issue_u(sn)
        yield ("arrive", f"S{sn % NBUF}")
    for s in range(total):
        bb = s % NBUF
        yield ("wait", f"P{bb}", s // NBUF)
        if s == total - 1:
            yield ("arrive", "ACC")
        yield ("arrive", f"QE{s % NQS_H}")
        yield ("arrive", f"DQF{bb}")           # dQ^T of step s into the buffer's dP^T columns
        s2 = s + NBUF
        if s2 < total:
            yield from issue_u(s2)              # U^T of step s + 2 over P, which dV has read
            yield ("wait", f"DQE{bb}", s // NBUF)  # dQ^T read out before the next dP^T
            yield ("arrive", f"S{bb}")
    yield ("arrive", "KVE0")


def ew_half(n_i):
    for s in range(n_i * SPT):
        yield ("wait", f"S{s % NBUF}", s // NBUF)
        yield ("wait", f"QF{s % NQS_H}", s // NQS_H)
        yield ("arrive", f"P{s % NBUF}")
    yield ("wait", "ACC", 0)


def dq_half(n_i):
    for s in range(n_i * SPT):
        yield ("wait", f"DQF{s % NBUF}", s // NBUF)
        yield ("arrive", f"DQE{s % NBUF}")


def run_half(n_i, seed):
    rng = random.Random(seed)
    bars = Barriers()
    roles = {"tma": tma_half(n_i), "mma": mma_half(n_i), "ew": ew_half(n_i), "dq": dq_half(n_i)}
    pending = {name: next(gen, None) for name, gen in roles.items()}
    while any(ev is not None for ev in pending.values()):
        runnable = [n for n, ev in pending.items()
                    if ev is not None and (ev[0] == "arrive" or bars.ready(ev[1], ev[2]))]
        if not runnable:
            raise AssertionError(f"deadlock at n_i = {n_i}: "
                                 f"{ {n: e for n, e in pending.items() if e is not None} }")
        name = rng.choice(runnable)
        if pending[name][0] == "arrive":
            bars.arrive(pending[name][1])
        pending[name] = next(roles[name], None)


@pytest.mark.parametrize("n_i", [1, 2, 3, 4, 7, 16])
def test_protocol_d128(n_i):
    for seed in range(40):
        run_half(n_i, seed)
