"""bench.py's algorithmic FLOP counts (CPU): the dense count is 4*T*Lkv*d*H
per node written out from the workload's geometry, and the block-sparse
count keeps only the mask's (query tile, key tile) pairs: an all-ones mask
gives the dense count, the own-chunk-only mask gives a node without history."""
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

import bench  # noqa: E402
from paper_2609_22283_gb300 import inputs as I  # noqa: E402


def test_dense_counts():
    w = I.WORKLOADS["clean1"]
    assert bench.attn_flops(w) == 4.0 * 4680 * (4 * 4680) * 128 * 12
    w = I.WORKLOADS["prog4"]
    assert bench.attn_flops(w) == 4 * 4.0 * 4680 * (7 * 4680) * 128 * 12


def test_sparse_counts():
    dense = I.WORKLOADS["tinys"]
    ones = I.Workload(**{**dense.__dict__, "sparse": 1.0})
    none = I.Workload(**{**dense.__dict__, "sparse": 0.0})
    base = I.Workload(**{**dense.__dict__, "sparse": None})
    assert bench.attn_flops(ones) == bench.attn_flops(base)
    own_only = sum(4.0 * dense.T * dense.T * dense.d * dense.H for _ in dense.nodes)
    assert bench.attn_flops(none) == own_only
    assert own_only < bench.attn_flops(dense) < bench.attn_flops(base)


def test_frame_causal_counts():
    # prog4fc: 3 frames of 1560 tokens; a query of frame f sees 1560 (f + 1)
    # own keys, so the own chunk holds 1560^2 (1 + 2 + 3) visible pairs
    w = I.WORKLOADS["prog4fc"]
    own = 1560.0 * 1560 * 6
    assert bench.attn_flops(w) == 4 * 4.0 * (own + 4680.0 * 6 * 4680) * 128 * 12
    # frame boundaries inside a 128-token tile are counted at token precision
    t = I.WORKLOADS["tinyfc"]                   # 3 frames of 32 tokens, T = 96
    per_node = [4.0 * (32 * (32 + 64 + 96) + 96 * max(0, min(t.W, b - 1)) * 96) * t.d * t.H
                for (_, b, _) in t.nodes]
    assert bench.attn_flops(t) == sum(per_node)


def test_attention_algorithmic_bytes():
    # distinct states read x (K + V) x heads x T x d x 2 B, plus Q read and O written
    slot = 2 * 4680 * 128 * 2
    assert bench.attn_bytes(I.WORKLOADS["clean1"]) == 4 * 12 * slot + 2 * 1 * 12 * 4680 * 128 * 2
    # prog4: the 4 nodes' own states and the clean chunks 11..16 (10 states)
    assert bench.attn_bytes(I.WORKLOADS["prog4"]) == 10 * 12 * slot + 2 * 4 * 12 * 4680 * 128 * 2
    # stress14b: two streams of prog4's states, 40 heads
    assert bench.attn_bytes(I.WORKLOADS["stress14b"]) == 20 * 40 * slot + 2 * 8 * 40 * 4680 * 128 * 2
    # same4: each node's own state and its three same-level predecessors
    assert bench.attn_bytes(I.WORKLOADS["same4"]) == 16 * 12 * slot + 2 * 4 * 12 * 4680 * 128 * 2
