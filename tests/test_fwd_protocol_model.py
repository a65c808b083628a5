"""A host-side model of the forward tile kernel's barrier protocol (relation_tc_fwd.cu):
TMA (Q once, K and V through a ring of stages), MMA (U of step s + 2 after the z update of
step s, 64-key steps on two TMEM buffers) and the scan warps (with the data-dependent
wait for the previous z update before a rescale), run under random interleavings for
both stage counts.  Checks for deadlock and for parity waits on a barrier two phases
ahead or one phase short of the awaited completion.  CPU only; the model mirrors the kernel's code, it does not run it."""
import random

import pytest

from tests.test_bwd_protocol_model import Ambiguous, Barriers


def tma(n_kv, stages):
    yield ("arrive", "Q")
    for j in range(n_kv):
        s, u = j % stages, j // stages
        if u > 0:
            yield ("wait", f"KE{s}", u - 1)
        yield ("arrive", f"KF{s}")
        if u > 0:
            yield ("wait", f"VE{s}", u - 1)
        yield ("arrive", f"VF{s}")


def mma(n_kv, stages):
    total = 2 * n_kv

    def issue_u(s):
        j, hh = s >> 1, s & 1
        st = j % stages
        if hh == 0:
            yield ("wait", f"KF{st}", j // stages)
        yield ("arrive", f"S{hh}")
        if hh == 1:
            yield ("arrive", f"KE{st}")

    yield ("wait", "Q", 0)
    yield from issue_u(0)
    if total > 1:
        yield from issue_u(1)
    for s in range(total):
        j, hh = s >> 1, s & 1
        st = j % stages
        if hh == 0:
            yield ("wait", f"VF{st}", j // stages)
        yield ("wait", f"P{hh}", s >> 1)
        yield ("arrive", "OD")
        if hh == 1:
            yield ("arrive", f"VE{st}")
        if s + 2 < total:
            yield from issue_u(s + 2)
    yield ("arrive", "O")


def scan(n_kv, rescale_rng, rescale_first=False):
    """The scan warps' waits: U of step s, then (data-dependent) the z update of step
    s - 1 before a rescale: the scale raised at step s - 1, applied at step s, and the
    rarer redo of a step whose bound jumped.  rescale_first puts the first of them
    before the wait for U (an order the kernel must not use)."""
    for s in range(2 * n_kv):
        pending = s > 0 and rescale_rng.random() < 0.3
        if rescale_first and pending:
            yield ("wait", "OD", s - 1)
        yield ("wait", f"S{s & 1}", s >> 1)
        if pending and not rescale_first:
            yield ("wait", "OD", s - 1)
        if s > 0 and rescale_rng.random() < 0.1:  # the step's bound jumped: redo it
            yield ("wait", "OD", s - 1)
        yield ("arrive", f"P{s & 1}")
    yield ("wait", "O", 0)


def run(n_kv, stages, seed, rescale_first=False):
    rng = random.Random(seed)
    bars = Barriers()
    roles = {"tma": tma(n_kv, stages), "mma": mma(n_kv, stages),
             "scan": scan(n_kv, random.Random(seed + 1000), rescale_first)}
    pending = {name: next(gen, None) for name, gen in roles.items()}
    while any(ev is not None for ev in pending.values()):
        runnable = [n for n, ev in pending.items()
                    if ev is not None and (ev[0] == "arrive" or bars.ready(ev[1], ev[2]))]
        if not runnable:
            raise AssertionError(f"deadlock at n_kv = {n_kv}, stages = {stages}: "
                                 f"{ {n: e for n, e in pending.items() if e is not None} }")
        name = rng.choice(runnable)
        if pending[name][0] == "arrive":
            bars.arrive(pending[name][1])
        pending[name] = next(roles[name], None)


@pytest.mark.parametrize("stages", [1, 2])
@pytest.mark.parametrize("n_kv", [1, 2, 3, 5, 16])
def test_forward_protocol(n_kv, stages):
    for seed in range(40):
        run(n_kv, stages, seed)


def test_rescale_wait_before_the_step_is_caught():
    """Waiting for the z update of step s - 1 before U of step s can meet the barrier one
    phase short, where its parity test passes at once (z rescaled under an update still in
    flight): the model flags that order."""
    caught = 0
    for seed in range(200):
        try:
            run(16, 2, seed, rescale_first=True)
        except Ambiguous:
            caught += 1
    assert caught > 0
