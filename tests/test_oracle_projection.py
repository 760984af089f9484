"""Pins of the oracle's QKV projection (the linear layer in front of the
attention, y = x W^T + b split into q, k, v): brute force on tiny inputs,
exact special cases (identity-like weights, bias alone) and the output order
(q's rows of W first, then k's, then v's; heads contiguous inside each)."""
import numpy as np

from paper_2609_22283_gb300 import inputs as I


def test_brute_force_tiny(oracle_mod):
    rng = np.random.default_rng(3)
    rows, C, heads, dh = 5, 7, 2, 3
    n = heads * dh
    x = rng.standard_normal((rows, C))
    w = rng.standard_normal((3 * n, C))
    b = rng.standard_normal(3 * n)
    q, k, v = oracle_mod.qkv_project(x, w, b, heads=heads)
    for t, out in enumerate((q, k, v)):
        for r in range(rows):
            for h in range(heads):
                for j in range(dh):
                    o = t * n + h * dh + j
                    want = sum(x[r, c] * w[o, c] for c in range(C)) + b[o]
                    assert abs(out[r, h, j] - want) < 1e-12


def test_identity_blocks_and_bias_alone(oracle_mod):
    rng = np.random.default_rng(4)
    rows, n = 6, 8
    x = rng.standard_normal((rows, n))
    eye = np.eye(n)
    q, k, v = oracle_mod.qkv_project(x, np.concatenate([eye, 2 * eye, -eye]), heads=2)
    np.testing.assert_array_equal(q.reshape(rows, n), x)
    np.testing.assert_array_equal(k.reshape(rows, n), 2 * x)
    np.testing.assert_array_equal(v.reshape(rows, n), -x)
    b = np.arange(3 * n, dtype=np.float64)
    q, k, v = oracle_mod.qkv_project(np.zeros((rows, n)), rng.standard_normal((3 * n, n)), b, heads=4)
    for t, out in enumerate((q, k, v)):
        np.testing.assert_array_equal(out, np.broadcast_to(b[t * n:(t + 1) * n].reshape(4, 2), (rows, 4, 2)))


def test_output_order_tags(oracle_mod):
    # weight row o picks input feature o % C with value o + 1: output (t, h, j)
    # must carry the tag of row t * n + h * dh + j
    rows, C, heads, dh = 3, 64, 4, 4
    n = heads * dh
    w = np.zeros((3 * n, C))
    for o in range(3 * n):
        w[o, o % C] = o + 1
    x = np.ones((rows, C))
    q, k, v = oracle_mod.qkv_project(x, w, heads=heads)
    for t, out in enumerate((q, k, v)):
        assert np.array_equal(out[0].reshape(-1), np.arange(t * n, (t + 1) * n) + 1.0)


def test_projection_inputs_are_seeded():
    w = I.WORKLOADS["tiny"]
    a = I.projection_inputs(w, 128)
    b = I.projection_inputs(w, 128)
    assert all(np.array_equal(u.float().numpy(), v.float().numpy()) for u, v in zip(a, b))
    x, wt, bias = a
    assert x.shape == (w.n_nodes, w.T, 128) and wt.shape == (3 * w.H * w.d, 128)
    assert abs(float(wt.float().std()) - 128 ** -0.5) < 0.01
