"""The library's host slot table, through the residency planner (moe_planner_*), against the
oracle on the CPU: the same records, bit for bit, for the LRU, rotary and router-guided policies,
with preload, batched unions and prefetch admission, and the planner's argument and capacity errors. The host
copy-engine decode schedule runs this same table, so this checks its decisions without a GPU."""
import numpy as np
import pytest

import oracle
import synth
from paper_2605_29135_gb300 import MoEError, Planner
from paper_2605_29135_gb300.buildsys import build


@pytest.fixture(scope="module", autouse=True)
def _built():
    build()


def _tuples(recs, E):
    return [(int(r["step"]), int(r["layer"]) * E + int(r["expert"]), int(r["kind"]), int(r["slot"]),
             int(r["evicted"])) for r in recs]


def _drive(policy, n_layers, E, cap, seqs, preload=False):
    """seqs: per (token, layer) the used and prefetch global-id lists. Returns both record lists."""
    table = oracle.TABLES[policy](n_layers * E, cap, E)
    if preload:
        table.preload()
    got, want = [], []
    with Planner(n_layers, E, cap, policy) as p:
        if preload:
            assert p.preload() == min(cap, n_layers * E)
        for (tok, l), (used, pf) in seqs:
            clock = tok * n_layers + l
            r = table.step(clock, used, tok)
            if pf:
                r = np.concatenate([r, table.admit(clock, used, pf, tok)])
            want += _tuples(r, E)
            got += _tuples(p.step(tok, l, [g - l * E for g in used], [g - l * E for g in pf]), E)
    return got, want


def _random_seqs(rng, tokens, n_layers, E, k, B=1, m=0):
    seqs = []
    for tok in range(tokens):
        for l in range(n_layers):
            used, pf = set(), set()
            for _ in range(B):
                order = [l * E + int(e) for e in rng.permutation(E)]
                used.update(order[:k])
                pf.update(order[k:k + m])
            seqs.append(((tok, l), (sorted(used), sorted(pf - used))))
    return seqs


@pytest.mark.parametrize("policy", ["lru", "rotary"])
@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("n_layers,E,k,cap,B", [(1, 8, 2, 4, 1), (3, 8, 2, 5, 1), (4, 16, 4, 9, 1),
                                                (2, 32, 8, 8, 1), (3, 16, 3, 14, 4), (2, 64, 8, 200, 1)])
def test_matches_the_oracle_on_random_sequences(policy, seed, n_layers, E, k, cap, B):
    rng = np.random.default_rng(seed)
    got, want = _drive(policy, n_layers, E, cap, _random_seqs(rng, 40, n_layers, E, k, B))
    assert got == want


@pytest.mark.parametrize("policy", ["lru", "rotary"])
@pytest.mark.parametrize("seed", range(3))
def test_matches_the_oracle_after_preload(policy, seed):
    rng = np.random.default_rng(50 + seed)
    n_layers, E, k, cap = 3, 16, 4, 20
    got, want = _drive(policy, n_layers, E, cap, _random_seqs(rng, 40, n_layers, E, k), preload=True)
    assert got == want


@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("n_layers,E,k,m,cap,B", [(1, 8, 2, 1, 4, 1), (3, 8, 2, 2, 5, 1), (4, 16, 4, 3, 9, 1),
                                                  (2, 32, 8, 8, 12, 1), (3, 16, 3, 2, 15, 4)])
def test_prefetch_admission_matches_the_oracle(seed, n_layers, E, k, m, cap, B):
    rng = np.random.default_rng(200 + seed)
    got, want = _drive("lru", n_layers, E, cap, _random_seqs(rng, 40, n_layers, E, k, B, m))
    assert got == want
    assert any(t[2] == 2 for t in got)


def test_prefetch_on_the_oracle_routing_of_a_stack():
    # the planner fed the oracle's own routing reproduces the oracle's full decode-step trace
    wl = synth.WORKLOADS["tiny_fp32"].replace(n_layers=3, tokens=20)
    hidden = synth.hidden_all(wl)
    m, cap, E, L = 2, 6, wl.n_experts, wl.n_layers
    orc = oracle.Oracle.for_workload(wl, cap_slots=cap, keep_slot_copies=False, prefetch=m)
    with Planner(L, E, cap) as p:
        for t in range(wl.tokens):
            st = orc.decode_step(hidden[t], compute_out=False)
            got = []
            for l in range(L):
                pf = oracle.prefetch_candidates(st.z[l, 0], st.idx[l, 0], m)
                got += _tuples(p.step(t, l, st.idx[l, 0], pf), E)
            assert got == _tuples(st.records, E), f"token {t}"


def test_golden_hand_trace_with_prefetch():
    import os

    path = os.path.join(os.path.dirname(__file__), "golden", "lru_prefetch_hand_trace_4slot.txt")
    expect, steps = {}, {}
    for line in open(path):
        line = line.split("#")[0].strip()
        if not line:
            continue
        lhs, rhs = line.split("|")
        s, a, b, c = (int(v) for v in lhs.split())
        steps[s] = ((a, b), c)
        expect.setdefault(s, []).append(tuple(int(v) for v in rhs.split()))
    with Planner(1, 8, 4) as p:
        for s in sorted(steps):
            (a, b), c = steps[s]
            recs = p.step(s, 0, [b, a], [c])
            assert [(int(r["expert"]), int(r["kind"]), int(r["slot"]), int(r["evicted"])) for r in recs] == expect[s]


def test_duplicates_are_merged_and_records_are_ascending():
    with Planner(2, 8, 16) as p:
        recs = p.step(0, 1, [5, 2, 5, 7, 2])
        assert [int(r["expert"]) for r in recs] == [2, 5, 7]
        assert all(int(r["layer"]) == 1 and int(r["kind"]) == 1 for r in recs)
        assert [int(r["kind"]) for r in p.step(1, 1, [7, 2])] == [0, 0]


def test_cap_is_clipped_to_the_number_of_experts():
    with Planner(2, 4, 100) as p:
        assert p.preload() == 8
        assert [int(r["kind"]) for r in p.step(0, 0, [0, 1, 2, 3])] == [0, 0, 0, 0]


@pytest.mark.parametrize("policy", ["lru", "rotary"])
def test_capacity_error_writes_the_decided_records_then_refuses(policy):
    with Planner(1, 8, 2, policy) as p:
        with pytest.raises(MoEError) as ei:
            p.step(0, 0, [1, 3, 6])
        assert ei.value.status == -4
        assert [int(r["expert"]) for r in ei.value.records] == [1, 3]
        with pytest.raises(MoEError) as ei:
            p.step(1, 0, [1])
        assert ei.value.status == -1


def test_argument_errors_change_nothing():
    with Planner(2, 8, 4) as p:
        p.step(0, 1, [1, 2])
        for args in [(0, 1, [3]), (0, 0, [3]), (1, 2, [3]), (-1, 0, [3]), (1, 0, [8]), (1, 0, [-1])]:
            with pytest.raises(MoEError) as ei:
                p.step(*args)
            assert ei.value.status == -1
        # the table is as it was: 1 and 2 still hit, at their slots
        recs = p.step(1, 1, [1, 2])
        assert [(int(r["kind"]), int(r["slot"])) for r in recs] == [(0, 0), (0, 1)]


def test_prefetch_needs_the_lru_policy():
    with Planner(1, 8, 4, "rotary") as p:
        with pytest.raises(MoEError) as ei:
            p.step(0, 0, [1], [2])
        assert ei.value.status == -1
        p.step(0, 0, [1])


@pytest.mark.parametrize("args", [(0, 8, 4, "lru"), (2, 0, 4, "lru"), (2, 8, 0, "lru"), (65536, 65536, 4, "lru")])
def test_create_rejects_bad_sizes(args):
    with pytest.raises(MoEError) as ei:
        Planner(*args)
    assert ei.value.status == -1
    assert str(ei.value)


def test_empty_layer_step_is_allowed():
    with Planner(1, 8, 4) as p:
        assert len(p.step(0, 0, [])) == 0
        assert len(p.step(1, 0, [3])) == 1


def _ranks_of(order):
    r = np.empty(len(order), dtype=np.int32)
    r[list(order)] = np.arange(len(order))
    return r


@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("n_layers,E,k,cap,B,preload", [(1, 8, 2, 4, 1, False), (3, 8, 2, 5, 1, False),
                                                        (4, 16, 4, 9, 1, False), (3, 4, 1, 5, 1, False),
                                                        (3, 16, 3, 14, 4, False), (3, 4, 1, 7, 1, True)])
def test_guided_policy_matches_the_oracle(seed, n_layers, E, k, cap, B, preload):
    rng = np.random.default_rng(400 + seed)
    table = oracle.GuidedTable(n_layers * E, cap, E)
    with Planner(n_layers, E, cap, "guided") as p:
        if preload:
            table.preload()
            p.preload()
        for tok in range(40):
            for l in range(n_layers):
                used, best = set(), np.full(E, E, dtype=np.int32)
                for _ in range(B):
                    order = [int(e) for e in rng.permutation(E)]
                    used.update(order[:k])
                    best = np.minimum(best, _ranks_of(order))
                table.set_layer_ranks(l, best)
                want = _tuples(table.step(tok * n_layers + l, [l * E + e for e in used], tok), E)
                got = _tuples(p.step(tok, l, sorted(used), ranks=best), E)
                assert got == want, f"token {tok} layer {l}"


def test_guided_golden_traces():
    from tests.test_oracle_guided import read_guided_golden

    for name, (E, L, k, cap, preload, steps) in read_guided_golden().items():
        with Planner(L, E, cap, "guided") as p:
            if preload:
                p.preload()
            for (tok, l, order), expect in steps:
                recs = p.step(tok, l, order[:k], ranks=_ranks_of(order))
                got = [(int(r["expert"]), int(r["kind"]), int(r["slot"]), int(r["evicted"])) for r in recs]
                assert got == expect, f"case {name} token {tok} layer {l}"


def test_guided_policy_on_the_oracle_routing_of_a_stack():
    wl = synth.WORKLOADS["tiny_fp32"].replace(n_layers=3, tokens=20)
    hidden = synth.hidden_all(wl)
    cap, E, L = 8, wl.n_experts, wl.n_layers
    orc = oracle.Oracle.for_workload(wl, cap_slots=cap, keep_slot_copies=False, policy="guided")
    with Planner(L, E, cap, "guided") as p:
        for t in range(wl.tokens):
            st = orc.decode_step(hidden[t], compute_out=False)
            got = []
            for l in range(L):
                got += _tuples(p.step(t, l, st.idx[l, 0], ranks=oracle.route_ranks(st.z[l, 0])), E)
            assert got == _tuples(st.records, E), f"token {t}"


def test_guided_rank_arguments_are_checked():
    with Planner(1, 8, 4, "guided") as p:
        for kw in ({}, {"ranks": [0, 1, 2, 3, 4, 5, 6, 9]}, {"ranks": [-1, 1, 2, 3, 4, 5, 6, 7]}):
            with pytest.raises(MoEError) as ei:
                p.step(0, 0, [1, 2], **kw)
            assert ei.value.status == -1
        with pytest.raises(ValueError):
            p.step(0, 0, [1, 2], ranks=[0, 1])
        assert len(p.step(0, 0, [1, 2], ranks=np.arange(8))) == 2
    with Planner(1, 8, 4, "lru") as p:
        with pytest.raises(MoEError):
            p.step(0, 0, [1, 2], ranks=np.arange(8))


def test_random_configurations_match_the_oracle():
    # property check over random shapes, caps, policies, batches and prefetch depths
    hyp = pytest.importorskip("hypothesis")
    st = hyp.strategies

    @hyp.settings(max_examples=60, deadline=None, derandomize=True)
    @hyp.given(L=st.integers(1, 4), E=st.integers(2, 24), data=st.data(), policy=st.sampled_from(["lru", "rotary", "guided"]),
               seed=st.integers(0, 2 ** 31 - 1))
    def check(L, E, data, policy, seed):
        k = data.draw(st.integers(1, E))
        B = data.draw(st.integers(1, 3))
        need_max = min(E, k * B)
        cap = data.draw(st.integers(need_max, L * E + 2))
        m = data.draw(st.integers(0, E - k)) if policy == "lru" else 0
        preload = data.draw(st.booleans())
        rng = np.random.default_rng(seed)
        table = oracle.TABLES[policy](L * E, min(cap, L * E), E)
        with Planner(L, E, cap, policy) as p:
            if preload:
                table.preload()
                p.preload()
            for tok in range(6):
                for l in range(L):
                    used, pf, best = set(), set(), np.full(E, E, dtype=np.int32)
                    for _ in range(B):
                        order = [int(e) for e in rng.permutation(E)]
                        used.update(order[:k])
                        pf.update(order[k:k + m])
                        best = np.minimum(best, _ranks_of(order))
                    pf -= used
                    clock = tok * L + l
                    if policy == "guided":
                        table.set_layer_ranks(l, best)
                    want = table.step(clock, [l * E + e for e in used], tok)
                    if pf:
                        want = np.concatenate([want, table.admit(clock, [l * E + e for e in used],
                                                                 [l * E + e for e in pf], tok)])
                    got = p.step(tok, l, sorted(used), sorted(pf), ranks=best if policy == "guided" else None)
                    assert _tuples(got, E) == _tuples(want, E)

    check()


def test_run_replays_a_recorded_routing_like_the_oracle():
    # the oracle's routing of a small stack, replayed in one call: same records, counts from them
    wl = synth.WORKLOADS["tiny_fp32"].replace(n_layers=3, tokens=16)
    hidden = synth.hidden_all(wl)
    orc = oracle.Oracle.for_workload(wl, cap_slots=6, keep_slot_copies=False, policy="guided")
    steps = [orc.decode_step(hidden[t], compute_out=False) for t in range(wl.tokens)]
    idx = np.stack([s.idx for s in steps])  # [T x L x B x k]
    ranks = np.stack([[oracle.route_ranks(s.z[l, 0]) for l in range(wl.n_layers)] for s in steps])
    with Planner(wl.n_layers, wl.n_experts, 6, "guided") as p:
        res = p.run(idx, ranks=ranks)
    want = np.concatenate([s.records for s in steps])
    assert _tuples(res["records"], wl.n_experts) == _tuples(want, wl.n_experts)
    assert res["hits"] == int((want["kind"] == 0).sum()) and res["misses"] == int((want["kind"] == 1).sum())
    assert 0.0 < res["hit_rate"] < 1.0 and res["prefetches"] == 0
    with Planner(wl.n_layers, wl.n_experts, 6) as p:
        with pytest.raises(ValueError):
            p.run(idx[:, :2])


def test_cap_sweep_counts_match_the_oracle_and_the_full_cap_misses_once_per_expert():
    from paper_2605_29135_gb300 import plan_caps

    rng = np.random.default_rng(7)
    L, E, k, T = 3, 12, 3, 20
    idx = np.stack([[rng.permutation(E)[:k] for _ in range(L)] for _ in range(T)])  # [T x L x k]
    caps = [k, 2 * k, 10, L * E]
    rows = plan_caps(L, E, caps, idx, expert_bytes=1000)
    assert [r["cap"] for r in rows] == caps
    for cap, row in zip(caps, rows):
        table = oracle.LRUTable(L * E, cap, E)
        kinds, ev = [], 0
        for t in range(T):
            for l in range(L):
                r = table.step(t * L + l, sorted(l * E + int(e) for e in idx[t, l]), t)
                kinds += list(r["kind"])
                ev += int((r["evicted"] >= 0).sum())
        kinds = np.array(kinds)
        assert row["misses"] == int((kinds == 1).sum()) and row["evictions"] == ev
        assert row["hit_rate"] == pytest.approx((kinds == 0).sum() / len(kinds))
        assert row["link_bytes_per_step"] == pytest.approx(row["misses"] * 1000 / T)
    full = rows[-1]
    assert full["evictions"] == 0 and full["misses"] == len({(l, int(e)) for t in range(T) for l in range(L)
                                                            for e in idx[t, l]})
    assert plan_caps(L, E, [L * E], idx, preload=True)[0]["misses"] == 0  # every expert resident up front
