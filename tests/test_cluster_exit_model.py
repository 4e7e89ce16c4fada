"""A model, on the CPU, of how the persistent decode grid's clusters end (decode_stream).

Each CTA of a cluster of ks CTAs walks its tiles: it pushes partial sums into every owner's
shared memory, arrives remotely on the owners' "ready" barriers, waits (bounded) until its own
receive buffer is complete, reads it and releases it with remote arrivals on the sources' "free"
barriers. Any wait may run out (a timeout); the CTA then skips its later waits but still runs its
remaining pushes and arrivals, then retires.

The safety property: no CTA ever writes into, or arrives on, the shared memory of a CTA that has
already retired. The kernel gets it from a hardware cluster barrier at the very end, which every
thread of every CTA reaches after its last remote access (all earlier waits are bounded, so every
CTA does reach it) and which nobody leaves before all have arrived. The model checks that the
property holds under that rule for random schedules and timeouts, and that the rule it replaced
(retire after a bounded wait on a "done" barrier) can break it.
"""
import random

import pytest


def simulate(ks, tiles, rng, closing, timeout_prob):
    """One random schedule of a cluster; returns the number of remote accesses that hit a retired
    CTA. `closing` is 'cluster_barrier' (the kernel's rule) or 'bounded_done' (the old rule)."""
    # every CTA's program: per tile, pushes to all owners, then (maybe) a bounded wait, then
    # releases to all sources; then the closing step
    events = []                        # (time, cta, kind, target)
    finish = []                        # time each CTA reaches its closing step
    for c in range(ks):
        t = rng.uniform(0, 5)
        dead = False
        for _ in range(tiles):
            t += rng.expovariate(1.0)                      # compute the tile
            for o in range(ks):                            # pushes + ready arrivals
                t += rng.uniform(0, 0.05)
                events.append((t, c, "remote", o))
            if not dead and rng.random() < timeout_prob:   # the bounded wait gave up
                dead = True
            t += rng.uniform(0, 0.5) if not dead else 0.0
            for o in range(ks):                            # release to the sources
                t += rng.uniform(0, 0.05)
                events.append((t, c, "remote", o))
            if rng.random() < 0.1:                         # a CTA held up (preemption, slow SM)
                t += rng.uniform(0, 50)
        finish.append(t)
    if closing == "cluster_barrier":
        # nobody leaves before the last CTA has arrived
        leave = [max(finish)] * ks
    else:
        # each CTA waits at most `limit` for the others' "done" arrivals, then leaves anyway
        limit = 1.0
        leave = []
        for c in range(ks):
            others = max(finish)
            leave.append(min(max(finish[c], others), finish[c] + limit))
    return sum(1 for (t, c, kind, o) in events if o != c and t > leave[o])


@pytest.mark.parametrize("ks", [2, 4, 8])
def test_cluster_barrier_exit_never_lets_a_peer_write_into_a_retired_cta(ks):
    rng = random.Random(1234 + ks)
    for _ in range(400):
        assert simulate(ks, tiles=rng.randint(1, 6), rng=rng, closing="cluster_barrier",
                        timeout_prob=0.2) == 0


def test_bounded_done_wait_exit_can_let_a_peer_write_into_a_retired_cta():
    """The replaced rule: with a held-up peer, a CTA whose bounded wait ran out retires while the
    peer still pushes into it -- the exposure the closing cluster barrier removes."""
    rng = random.Random(99)
    hits = sum(simulate(8, tiles=4, rng=rng, closing="bounded_done", timeout_prob=0.2) for _ in range(400))
    assert hits > 0
