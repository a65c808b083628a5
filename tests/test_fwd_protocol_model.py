"""A host-side model of the forward tile kernel's barrier protocol (relation_tc_fwd.cu):
TMA (Q once, K and V through a ring of stages), MMA (U of step s + NBUF after the z update
of step s, 64-key steps on one or two TMEM buffers) and the scan warps (with the
data-dependent wait for the previous z update before a rescale), run under random
interleavings for every layout of the kernel.  Checks for deadlock and for parity waits on a barrier two phases
ahead or one phase short of the awaited completion.  CPU only; the model mirrors the kernel's code, it does not run it."""
import random

import pytest

from tests.test_bwd_protocol_model import Ambiguous, Barriers


# Layouts of the kernel (FwdCfg): U/P buffers, scan steps per K/V load unit, stages, scan
# steps per 128-key tile.
LAYOUTS = {
    "two buffers of 64 keys, one stage (d_h = 128)": (2, 2, 1, 2),
    "two buffers of 32 keys, 64-key units, two stages (d_h = 64)": (2, 2, 2, 4),
    "one buffer of 64 keys, two stages": (1, 1, 2, 2),
    "four buffers of 32 keys, one stage": (4, 4, 1, 4),
}


def tma(n_ld, stages):
    yield ("arrive", "Q")
    for j in range(n_ld):
        s, u = j % stages, j // stages
        if u > 0:
            yield ("wait", f"KE{s}", u - 1)
        yield ("arrive", f"KF{s}")
        if u > 0:
            yield ("wait", f"VE{s}", u - 1)
        yield ("arrive", f"VF{s}")


def mma(total, spl, nbuf, stages, shared_od=False):
    def issue_u(s):
        j, hh = s // spl, s % spl
        st, bf = j % stages, s % nbuf
        if hh == 0:
            yield ("wait", f"KF{st}", j // stages)
        yield ("arrive", f"S{bf}")
        if hh == spl - 1:
            yield ("arrive", f"KE{st}")

    yield ("wait", "Q", 0)
    for s0 in range(min(nbuf, total)):  # every buffer's first step ahead
        yield from issue_u(s0)
    for s in range(total):
        j, hh = s // spl, s % spl
        st, bf = j % stages, s % nbuf
        if hh == 0:
            yield ("wait", f"VF{st}", j // stages)
        yield ("wait", f"P{bf}", s // nbuf)
        yield ("arrive", "OD" if shared_od else f"OD{bf}")
        if hh == spl - 1:
            yield ("arrive", f"VE{st}")
        if s + nbuf < total:
            yield from issue_u(s + nbuf)
    yield ("arrive", "O")


def scan(total, nbuf, rescale_rng, rescale_first=False, shared_od=False):
    """The scan warps' waits: U of step s, then (data-dependent) the z update of step
    s - 1 before a rescale: the scale raised at step s - 1, applied at step s, and the
    rarer redo of a step whose bound jumped.  rescale_first puts the first of them
    before the wait for U (an order the kernel must not use)."""
    def od(k):  # the z update of step k: that step's buffer's barrier (or one shared)
        return ("wait", "OD", k) if shared_od else ("wait", f"OD{k % nbuf}", k // nbuf)

    for s in range(total):
        bf = s % nbuf
        pending = s > 0 and rescale_rng.random() < 0.3
        if rescale_first and pending:
            yield od(s - 1)
        yield ("wait", f"S{bf}", s // nbuf)
        if pending and not rescale_first:
            yield od(s - 1)
        if s > 0 and rescale_rng.random() < 0.1:  # the step's bound jumped: redo it
            yield od(s - 1)
        yield ("arrive", f"P{bf}")
    yield ("wait", "O", 0)


def run(n_kv, layout, seed, rescale_first=False, shared_od=False):
    nbuf, spl, stages, spt = LAYOUTS[layout]
    total = spt * n_kv
    rng = random.Random(seed)
    bars = Barriers()
    roles = {"tma": tma(total // spl, stages), "mma": mma(total, spl, nbuf, stages, shared_od),
             "scan": scan(total, nbuf, random.Random(seed + 1000), rescale_first, shared_od)}
    pending = {name: next(gen, None) for name, gen in roles.items()}
    while any(ev is not None for ev in pending.values()):
        runnable = [n for n, ev in pending.items()
                    if ev is not None and (ev[0] == "arrive" or bars.ready(ev[1], ev[2]))]
        if not runnable:
            raise AssertionError(f"deadlock at n_kv = {n_kv}, layout {layout}: "
                                 f"{ {n: e for n, e in pending.items() if e is not None} }")
        name = rng.choice(runnable)
        if pending[name][0] == "arrive":
            bars.arrive(pending[name][1])
        pending[name] = next(roles[name], None)


@pytest.mark.parametrize("layout", sorted(LAYOUTS))
@pytest.mark.parametrize("n_kv", [1, 2, 3, 5, 16])
def test_forward_protocol(n_kv, layout):
    for seed in range(40):
        run(n_kv, layout, seed)


def test_rescale_wait_before_the_step_is_caught():
    """With one z-update barrier shared by the buffers, waiting for the update of step
    s - 1 before U of step s can meet the barrier one phase short, where its parity test
    passes at once (z rescaled under an update still in flight): the model flags that
    order.  With a barrier per buffer (the kernel), U of step s - 1 already implies the
    buffer's previous update, so the wait is exact in either order."""
    layout = "two buffers of 64 keys, one stage (d_h = 128)"
    caught = 0
    for seed in range(200):
        try:
            run(16, layout, seed, rescale_first=True, shared_od=True)
        except Ambiguous:
            caught += 1
    assert caught > 0
    for lay in LAYOUTS:
        for seed in range(40):
            run(16, lay, seed, rescale_first=True)
