"""A host-side model of the forward tile kernel's barrier protocol (relation_tc_fwd.cu):
TMA (Q once, K and V through a ring of stages), MMA (U of step s + NBUF after the z update
of step s, 64-key steps on one or two TMEM buffers) and the scan warps (with the
data-dependent wait for the previous z update before a rescale), run under random
interleavings for every layout of the kernel.  Checks for deadlock and for parity waits on a barrier two phases
ahead or one phase short of the awaited completion.  CPU only; the model mirrors the kernel's code, it does not run it."""
import random

import pytest

from tests.test_bwd_protocol_model import Ambiguous, Barriers


# Layouts of the kernel (FwdCfg): U/P buffers, 64-key scan steps per K/V load unit, stages.
LAYOUTS = {
    "two buffers, one stage (d_h = 128)": (2, 2, 1),
    "two buffers, two stages": (2, 2, 2),
    "one buffer, 64-key units, two stages (d_h = 64, four CTAs per SM)": (1, 1, 2),
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


def mma(total, spl, nbuf, stages):
    def issue_u(s):
        j, hh = s // spl, s % spl
        st, bf = j % stages, s % nbuf
        if hh == 0:
            yield ("wait", f"KF{st}", j // stages)
        yield ("arrive", f"S{bf}")
        if hh == spl - 1:
            yield ("arrive", f"KE{st}")

    yield ("wait", "Q", 0)
    yield from issue_u(0)
    if total > 1 and nbuf == 2:
        yield from issue_u(1)
    for s in range(total):
        j, hh = s // spl, s % spl
        st, bf = j % stages, s % nbuf
        if hh == 0:
            yield ("wait", f"VF{st}", j // stages)
        yield ("wait", f"P{bf}", s // nbuf)
        yield ("arrive", "OD")
        if hh == spl - 1:
            yield ("arrive", f"VE{st}")
        if s + nbuf < total:
            yield from issue_u(s + nbuf)
    yield ("arrive", "O")


def scan(total, nbuf, rescale_rng, rescale_first=False):
    """The scan warps' waits: U of step s, then (data-dependent) the z update of step
    s - 1 before a rescale: the scale raised at step s - 1, applied at step s, and the
    rarer redo of a step whose bound jumped.  rescale_first puts the first of them
    before the wait for U (an order the kernel must not use)."""
    for s in range(total):
        bf = s % nbuf
        pending = s > 0 and rescale_rng.random() < 0.3
        if rescale_first and pending:
            yield ("wait", "OD", s - 1)
        yield ("wait", f"S{bf}", s // nbuf)
        if pending and not rescale_first:
            yield ("wait", "OD", s - 1)
        if s > 0 and rescale_rng.random() < 0.1:  # the step's bound jumped: redo it
            yield ("wait", "OD", s - 1)
        yield ("arrive", f"P{bf}")
    yield ("wait", "O", 0)


def run(n_kv, layout, seed, rescale_first=False):
    nbuf, spl, stages = LAYOUTS[layout]
    total = 2 * n_kv
    rng = random.Random(seed)
    bars = Barriers()
    roles = {"tma": tma(total // spl, stages), "mma": mma(total, spl, nbuf, stages),
             "scan": scan(total, nbuf, random.Random(seed + 1000), rescale_first)}
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
    """Waiting for the z update of step s - 1 before U of step s can meet the barrier one
    phase short, where its parity test passes at once (z rescaled under an update still in
    flight): the model flags that order."""
    caught = 0
    for seed in range(200):
        try:
            run(16, "two buffers, one stage (d_h = 128)", seed, rescale_first=True)
        except Ambiguous:
            caught += 1
    assert caught > 0
