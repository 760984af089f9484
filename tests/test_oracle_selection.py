"""Pins of the oracle's context selection (Eq. 2-3), pipeline rounds (Eq. 6)
and availability rule (Eq. 7) against facts the paper states and against a
round-by-round simulation of the pipeline that does not use those formulas."""
import json
import os

import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def test_worked_example_k3(oracle_mod):
    o = oracle_mod
    ex = _load("worked_example_k3.json")
    K, n, B = ex["K"], ex["round"], ex["B"]
    assert o.pipeline_round(K, B, n) == [tuple(s) for s in ex["active_states"]]
    b, j = ex["node"]
    for name, pid in o.POLICY_IDS.items():
        sel = o.select(pid, ex["W"], b, j)
        assert sel == [tuple(s) for s in ex["selection"][name]], name
        ok = all(o.available(j, b - c, lvl) for (c, lvl) in sel)
        assert ok == ex["available"][name], name


def test_policy_closed_forms(oracle_mod):
    o = oracle_mod
    # Eq. 3 at a few hand-evaluated points.
    assert o.phi(o.POLICY_CLEAN, 4, 1) == 0
    assert o.phi(o.POLICY_SAME, 4, 3) == 4
    assert o.phi(o.POLICY_PROG, 4, 1) == 3
    assert o.phi(o.POLICY_PROG, 4, 4) == 0
    assert o.phi(o.POLICY_PROG, 2, 5) == 0
    assert o.phi(o.POLICY_PROG, 0, 1) == 0
    assert o.phi(7, 1, 1) == -1


def test_window_shape(oracle_mod):
    """Eq. 2: offsets run over {1..min(W, b-1)}, the chunk b-r for offset r."""
    o = oracle_mod
    for pid in (0, 1, 2):
        for W in range(0, 9):
            for b in range(1, 21):
                for j in range(0, 5):
                    sel = o.select(pid, W, b, j)
                    assert len(sel) == max(0, min(W, b - 1))
                    assert [c for c, _ in sel] == [b - r for r in range(1, len(sel) + 1)]
                    assert all(0 <= lvl <= j for _, lvl in sel)


def test_progressive_prefill_of_prog4(oracle_mod):
    """Node (20, 4) of the prog4 workload reads (19,3), (18,2), (17,1), then clean 16, 15, 14."""
    o = oracle_mod
    assert o.select(o.POLICY_PROG, 6, 20, 4) == [(19, 3), (18, 2), (17, 1), (16, 0), (15, 0), (14, 0)]
    assert o.select(o.POLICY_PROG, 6, 17, 1) == [(16, 0), (15, 0), (14, 0), (13, 0), (12, 0), (11, 0)]


@pytest.mark.parametrize("case", _load("pipeline_counts.json")["cases"])
def test_pipeline_counting_facts(oracle_mod, case):
    o = oracle_mod
    K, B = case["K"], case["B"]
    rounds = [o.pipeline_round(K, B, n) for n in range(1, K + B + 3)]
    nonempty = [n + 1 for n, r in enumerate(rounds) if r]
    assert len(nonempty) == case["rounds"]
    assert nonempty == list(range(1, case["rounds"] + 1))
    assert sum(len(r) for r in rounds) == case["updates"]
    # first output: the round in which chunk 1 takes its last update (level 1)
    first = next(n + 1 for n, r in enumerate(rounds) if (1, 1) in r)
    assert first == case["first_output_round"]
    # a filled pipeline finishes exactly one chunk per round
    for n in range(K, B + 1):
        assert sum(1 for (_, lvl) in rounds[n - 1] if lvl == 1) == 1
    # every chunk gets each level 1..K exactly once
    seen = {}
    for r in rounds:
        for (c, lvl) in r:
            seen.setdefault(c, []).append(lvl)
    assert sorted(seen) == list(range(1, B + 1))
    assert all(v == list(range(K, 0, -1)) for v in seen.values())


def _simulate(K, B, rounds):
    """Round-by-round state machine of the Eq. 6 pipeline, written without the
    Eq. 6 formula: each round, every active chunk drops one level and one new
    chunk enters at level K.  Yields {chunk: level at the start of round n}
    for all chunks that have started (finished chunks stay at 0)."""
    level = {}
    next_chunk = 1
    for n in range(1, rounds + 1):
        if next_chunk <= B:
            level[next_chunk] = K
            next_chunk += 1
        yield n, dict(level)
        for c in list(level):
            if level[c] > 0:
                level[c] -= 1


def test_rounds_match_simulation(oracle_mod):
    o = oracle_mod
    for K in range(1, 7):
        for B in range(1, 12):
            for n, lv in _simulate(K, B, K + B + 1):
                active = sorted(((c, l) for c, l in lv.items() if l > 0), key=lambda s: -s[1])
                assert o.pipeline_round(K, B, n) == active, (K, B, n)


def test_progressive_equals_states_current_in_round(oracle_mod):
    """Section 3.3: in the Eq. 6 pipeline, when chunk b is at level j, chunk
    b-r has reached level max(j-r, 0): the progressive policy reads exactly
    the states current in the same round."""
    o = oracle_mod
    for K in range(1, 6):
        B = 12
        for n, lv in _simulate(K, B, K + B - 1):
            for (b, j) in o.pipeline_round(K, B, n):
                for (c, lvl) in o.select(o.POLICY_PROG, 8, b, j):
                    assert lv[c] == lvl, (K, n, b, j, c)


def test_eq7_holds_for_same_and_prog_not_clean(oracle_mod):
    o = oracle_mod
    for K in range(1, 6):
        for W in range(1, 7):
            B = 10
            for n in range(1, K + B):
                for (b, j) in o.pipeline_round(K, B, n):
                    for pid in (o.POLICY_SAME, o.POLICY_PROG):
                        assert all(o.available(j, b - c, l) for c, l in o.select(pid, W, b, j))
                    clean = o.select(o.POLICY_CLEAN, W, b, j)
                    expect_ok = all(j - (b - c) <= 0 for c, _ in clean)
                    assert all(o.available(j, b - c, l) for c, l in clean) == expect_ok


def test_available_examples(oracle_mod):
    o = oracle_mod
    assert o.available(3, 1, 2)
    assert not o.available(3, 1, 1)
    assert o.available(3, 1, 3)
    assert o.available(3, 3, 0)
    assert not o.available(2, 1, 0)
