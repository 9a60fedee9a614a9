"""The lookahead kernel's worker protocol, checked on a host model under random interleavings.

The worker CTAs of the lookahead kernel take the layers in groups. Per group g a CTA loads the
group's plan, computes its gate/up rows (writing the group's u vectors; a miss CTA first waits for
every worker's arrival for g - 1, then streams the group's misses into their slots), arrives on
the counter of g's parity, waits until every worker arrived for the group whose down rows come
next (g unskewed, g - 1 skewed), stages that group's u and computes its down rows. This model
runs the same sequence of actions for W CTAs, one action at a time in a random order, with the
waits satisfied only when their counter says so, and checks what the kernel relies on:

  - a CTA stages a group's u only after every CTA has really arrived for that group (written its
    gate/up rows); per-parity counters keep that exact, a single counter does not once the CTAs
    are skewed (a CTA's early arrival for g + 1 stands in for a late one of g);
  - u of group g may share a buffer with g - 4 (four sets skewed, two unskewed): no CTA writes
    u of g while another has yet to stage a group in the same buffer; three sets are not enough;
  - when a miss of group g lands, no CTA still reads a group older than g - 2 skewed (g - 1
    unskewed): with P layers a group that is 3 P - 1 (2 P - 1) layer-steps before the miss's,
    the window the LRU slot bound of the kernel is sized for.
"""
import random

import pytest


def _run(W, G, skew, seed, counters="parity", nu=None, miss_ctas=1, miss_wait=True):
    """One random interleaving; returns the set of violated properties (empty if none)."""
    nu = nu if nu is not None else (4 if skew else 2)
    rng = random.Random(seed)
    cnt = [0, 0] if counters == "parity" else [0]
    arrived = [[False] * G for _ in range(W)]   # real arrivals
    staged = [[False] * G for _ in range(W)]    # u of group staged by the CTA
    down_done = [[False] * G for _ in range(W)]
    bad = set()

    def all_arrived_counter(g):
        if counters == "parity":
            return cnt[g & 1] >= (g // 2 + 1) * W
        return cnt[0] >= (g + 1) * W

    def program(c):
        for g in range(G + skew):
            if g < G:
                miss = c >= W - miss_ctas
                if miss and g > 0:
                    if miss_wait:
                        yield ("wait", g - 1)
                    # a miss of group g lands: every reader must be within the window
                    oldest = min((h for w in range(W) for h in range(G) if not down_done[w][h]), default=G)
                    if g - oldest > (2 if skew else 1):
                        bad.add("slot window")
                # gate/up rows write u of g into buffer g % nu
                for w in range(W):
                    for h in range(g):
                        if h % nu == g % nu and not staged[w][h]:
                            bad.add("u buffer")
                yield ("act", None)
                arrived[c][g] = True
                cnt[g & 1 if counters == "parity" else 0] += 1
                yield ("act", None)
            dg = g - skew
            if dg < 0:
                continue
            yield ("wait", dg)
            if not all(arrived[w][dg] for w in range(W)):
                bad.add("early down")
            staged[c][dg] = True
            yield ("act", None)
            down_done[c][dg] = True
            yield ("act", None)

    progs = [program(c) for c in range(W)]
    pending = [next(p) for p in progs]
    live = set(range(W))
    while live:
        ready = [c for c in live if pending[c][0] == "act" or all_arrived_counter(pending[c][1])]
        assert ready, "the protocol deadlocked"
        c = rng.choice(ready)
        try:
            pending[c] = next(progs[c])
        except StopIteration:
            live.discard(c)
    return bad


@pytest.mark.parametrize("skew", [0, 1])
def test_parity_counters_keep_every_property(skew):
    for seed in range(300):
        rng = random.Random(seed)
        W, G = rng.randint(2, 5), rng.randint(2, 9)
        assert not _run(W, G, skew, seed, miss_ctas=rng.randint(0, W - 1)), (skew, seed)


def test_a_single_counter_lets_skewed_down_rows_start_early():
    hits = sum("early down" in _run(4, 8, 1, seed, counters="single") for seed in range(300))
    assert hits > 0


def test_a_single_counter_is_exact_unskewed():
    for seed in range(200):
        assert not _run(4, 8, 0, seed, counters="single"), seed


def test_three_u_sets_are_too_few_when_skewed():
    hits = sum("u buffer" in _run(4, 10, 1, seed, nu=3) for seed in range(400))
    assert hits > 0


def test_miss_ctas_that_do_not_wait_widen_the_window():
    # without the wait for g - 1 a skewed miss CTA can land group g's misses while a CTA still
    # reads a group older than g - 2
    hits = sum("slot window" in _run(4, 10, 1, seed, miss_ctas=2, miss_wait=False) for seed in range(400))
    assert hits > 0
