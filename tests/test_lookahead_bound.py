"""The bound the device schedule's exact layer lookahead rests on, checked on the oracle's LRU.

In that kernel CTA 0 decides the lookup of layer-step m ahead of the other CTAs, and the missed
experts' bytes go into their slots during layer-step m's gate-up rows. At that moment every row of
layer-steps before m - 1 has been read (a barrier separates them), but the down rows of m - 1 may
still be reading. So the slot a miss takes must not hold an expert of layer-step m - 1. Under LRU
with lower-id ties that holds whenever the pool has at least 2 k slots: the experts of m - 1 carry
the newest timestamp apart from m's own, and at least k older residents remain for the at most k
misses. Here the oracle's LRU checks the claim at the tightest cap on random routings (single
sequence and batched unions, cold and preloaded pools), and shows that one slot fewer breaks it.
The kernel's two refinements widen the window of layer-steps that may still read when a miss
lands, and the same check covers them: layers in groups of P per arrival (2 P - 1 layer-steps,
2 P k slots) and workers skewed by one group (3 P - 1 layer-steps, 3 P k slots).
"""
import random

import oracle


def _victims_avoid_previous_step(L, E, k, cap, steps, seed, batch=1, preload=False):
    """Run random layer-steps through the oracle's LRU; True if no miss evicted an expert that the
    layer-step just before it used."""
    rng = random.Random(seed)
    tbl = oracle.LRUTable(L * E, cap, E)
    if preload:
        tbl.preload()
    clock = 0
    prev = set()
    for t in range(steps):
        for l in range(L):
            needed = set()
            for _ in range(batch):
                needed.update(l * E + e for e in rng.sample(range(E), k))
            for r in tbl.step(clock, sorted(needed), t):
                if r["evicted"] >= 0 and int(r["evicted"]) in prev:
                    return False
            prev = needed
            clock += 1
    return True


def test_no_victim_from_the_previous_layer_step_at_the_tightest_cap():
    checked = 0
    for seed in range(80):
        rng = random.Random(1000 + seed)
        L, E = rng.randint(1, 6), rng.randint(4, 24)
        k = rng.randint(1, min(8, E // 2))
        cap = 2 * k
        if cap >= L * E:
            continue
        checked += 1
        assert _victims_avoid_previous_step(L, E, k, cap, steps=12, seed=seed, preload=seed % 2 == 0), seed
    assert checked > 50


def test_batched_unions_need_the_bound_on_distinct_experts():
    # with a batch, k is replaced by the most distinct experts one layer-step can need
    for seed in range(30):
        rng = random.Random(2000 + seed)
        L, E, k, B = rng.randint(1, 4), rng.randint(8, 20), rng.randint(1, 3), rng.randint(2, 3)
        cap = 2 * min(E, k * B)
        if cap >= L * E:
            continue
        assert _victims_avoid_previous_step(L, E, k, cap, steps=10, seed=seed, batch=B), seed


def test_one_slot_fewer_can_evict_from_the_previous_layer_step():
    broken = 0
    for seed in range(100):
        rng = random.Random(3000 + seed)
        k = rng.randint(2, 4)
        broken += not _victims_avoid_previous_step(3, 16, k, 2 * k - 1, steps=10, seed=seed)
    assert broken > 0


def _victims_avoid_recent_steps(L, E, k, cap, steps, seed, depth):
    """Like _victims_avoid_previous_step for the `depth` layer-steps before each one."""
    rng = random.Random(seed)
    tbl = oracle.LRUTable(L * E, cap, E)
    clock = 0
    recent = []
    for t in range(steps):
        for l in range(L):
            needed = set(l * E + e for e in rng.sample(range(E), k))
            used = set().union(*recent) if recent else set()
            for r in tbl.step(clock, sorted(needed), t):
                if r["evicted"] >= 0 and int(r["evicted"]) in used:
                    return False
            recent = (recent + [needed])[-depth:]
            clock += 1
    return True


def test_layer_groups_need_2_p_k_slots():
    # The lookahead kernel with groups of P layers per worker barrier writes a miss of a layer while
    # the down rows of the previous group and the gate/up rows of its own group may still read: the
    # 2 P - 1 layer-steps before it. LRU keeps their experts from (2 P - 1 + 1) k = 2 P k slots on.
    for P in (2, 3):
        depth = 2 * P - 1
        checked = 0
        for seed in range(60):
            rng = random.Random(4000 + 100 * P + seed)
            L, E = rng.randint(2, 6), rng.randint(8, 32)
            k = rng.randint(1, min(4, E // (2 * P)))
            cap = 2 * P * k
            if cap >= L * E:
                continue
            checked += 1
            assert _victims_avoid_recent_steps(L, E, k, cap, steps=10, seed=seed, depth=depth), (P, seed)
        assert checked > 30
        broken = sum(not _victims_avoid_recent_steps(4, 24, 3, 2 * P * 3 - 1, steps=10, seed=s, depth=depth)
                     for s in range(60))
        assert broken > 0


def test_skewed_workers_need_3_p_k_slots():
    # Skewed, a worker CTA runs the down rows of group g - 1 after the gate/up rows of group g, and
    # the miss CTAs of a group start once every worker has arrived for the group before. A miss of a
    # layer then lands while the down rows of the two groups before its own and the gate/up rows of
    # its own group may still read: the 3 P - 1 layer-steps before it, which LRU keeps from
    # (3 P - 1 + 1) k = 3 P k slots on.
    for P in (1, 2, 3):
        depth = 3 * P - 1
        checked = 0
        for seed in range(60):
            rng = random.Random(5000 + 100 * P + seed)
            L, E = rng.randint(2, 6), rng.randint(6 * P, 40)
            k = rng.randint(1, min(4, E // (3 * P)))
            cap = 3 * P * k
            if cap >= L * E:
                continue
            checked += 1
            assert _victims_avoid_recent_steps(L, E, k, cap, steps=10, seed=seed, depth=depth), (P, seed)
        assert checked > 30
        broken = sum(not _victims_avoid_recent_steps(4, 30, 3, 3 * P * 3 - 1, steps=10, seed=s, depth=depth)
                     for s in range(60))
        assert broken > 0
