"""The C-ABI library without a GPU: it loads, exports every function that
include/sva.h declares, and its host-side integer logic (context selection,
pipeline rounds, availability) agrees bit-exactly with the oracle."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            text = open(os.path.join(ROOT, "include", fn)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names |= set(re.findall(r"\b(sva_[a-z_0-9]+)\s*\(", text))
    return names


def test_exports_every_declared_symbol(sva_mod):
    lib = sva_mod.load()
    declared = _declared()
    assert len(declared) >= 14
    for name in sorted(declared):
        assert hasattr(lib, name), name
    assert declared == set(sva_mod.EXPORTED)


def test_select_context_matches_oracle(sva_mod, oracle_mod):
    for pid in (0, 1, 2):
        for K in range(1, 9):
            for W in range(0, 9):
                for b in range(1, 21):
                    for j in range(0, K + 1):
                        assert sva_mod.select_context(pid, K, W, b, j) == oracle_mod.select(pid, W, b, j)


def test_pipeline_round_matches_oracle(sva_mod, oracle_mod):
    for K in range(1, 9):
        for B in range(0, 15):
            for n in range(-2, K + B + 3):
                assert sva_mod.pipeline_round(K, B, n) == oracle_mod.pipeline_round(K, B, n)


def test_check_pipeline_matches_oracle(sva_mod, oracle_mod):
    rng = np.random.default_rng(0)
    for _ in range(3000):
        K = int(rng.integers(1, 7))
        j = int(rng.integers(0, K + 1))
        b = int(rng.integers(2, 30))
        n = int(rng.integers(0, 6))
        states = []
        for _ in range(n):
            r = int(rng.integers(1, b))
            states.append((b - r, int(rng.integers(0, K + 1))))
        expect = all(oracle_mod.available(j, b - c, l) for c, l in states)
        st = sva_mod.check_pipeline(K, j, b, states)
        assert st == (sva_mod.OK if expect else sva_mod.ERR_UNAVAILABLE)


def test_check_pipeline_worked_example(sva_mod):
    # K = 3, node (2, 3): level 3 and level 2 of chunk 1 are available, level 0 is not
    assert sva_mod.check_pipeline(3, 3, 2, [(1, 3)]) == sva_mod.OK
    assert sva_mod.check_pipeline(3, 3, 2, [(1, 2)]) == sva_mod.OK
    assert sva_mod.check_pipeline(3, 3, 2, [(1, 0)]) == sva_mod.ERR_UNAVAILABLE
    assert sva_mod.check_pipeline(3, 3, 2, [(2, 3)]) == sva_mod.ERR_CAUSALITY


def test_selection_errors(sva_mod):
    with pytest.raises(sva_mod.SvaError) as e:
        sva_mod.select_context(3, 4, 3, 10, 2)
    assert e.value.status == sva_mod.ERR_INVALID_ARGUMENT
    with pytest.raises(sva_mod.SvaError) as e:
        sva_mod.select_context(2, 4, 3, 10, 5)
    assert e.value.status == sva_mod.ERR_INVALID_ARGUMENT
    with pytest.raises(sva_mod.SvaError) as e:
        sva_mod.select_context(2, 4, 6, 10, 2, cap=3)
    assert e.value.status == sva_mod.ERR_CAPACITY
    with pytest.raises(sva_mod.SvaError) as e:
        sva_mod.pipeline_round(4, 40, 20, cap=2)
    assert e.value.status == sva_mod.ERR_CAPACITY


def test_cache_bytes(sva_mod):
    g = sva_mod.make_geometry(12, 128, 3, 30, 52, num_slots=10, pairs=(22, 21, 21), max_frames=66)
    T, Tpad = 4680, 4736
    pool = 10 * 2 * 12 * Tpad * 128 * 2
    tabs = [66 * 22 * 8, 30 * 21 * 8, 52 * 21 * 8, 30 * 21 * 8, 52 * 21 * 8]  # + pair-major h, w
    expect = -(-pool // 256) * 256
    for t in tabs:
        expect = -(-(expect + t) // 256) * 256
    expect += 256
    assert sva_mod.cache_bytes(g) == expect
    bad = [
        sva_mod.make_geometry(12, 96, 3, 30, 52, 10, (16, 16, 16), 66),      # head_dim
        sva_mod.make_geometry(12, 128, 3, 30, 52, 10, (22, 21, 20), 66),     # pairs sum
        sva_mod.make_geometry(0, 128, 3, 30, 52, 10, (22, 21, 21), 66),      # heads
        sva_mod.make_geometry(12, 128, 3, 30, 52, 0, (22, 21, 21), 66),      # slots
        sva_mod.make_geometry(12, 128, 3, 30, 52, 10, (22, 21, 21), 0),      # max_frames
        sva_mod.make_geometry(128, 128, 3, 30, 52, 4000, (22, 21, 21), 66),  # TMA row range
    ]
    for g in bad:
        assert sva_mod.cache_bytes(g) == 0


def test_workload_rounds_are_pipeline_rounds(sva_mod):
    from paper_2609_22283_gb300 import inputs as I
    for name in I.ORDER + I.EXTRA:
        w = I.WORKLOADS[name]
        if w.round is None:
            continue
        seqs = sorted({s for s, _, _ in w.nodes})
        for s in seqs:
            # level-0 nodes are clean-state refreshes batched into the round
            mine = [(c, l) for (q, c, l) in w.nodes if q == s and l > 0]
            assert mine == sva_mod.pipeline_round(w.K, w.B, w.round)
            for (q, c, l) in w.nodes:
                if q == s and l == 0:
                    assert c == w.round - w.K   # the chunk that left the pipeline last round
