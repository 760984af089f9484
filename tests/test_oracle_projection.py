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


# ---------------------------------------------------------------- projection + RoPE (fused)

def _geom(oracle_mod):
    # d = 8: pairs (t, h, w) = (2, 1, 1); 2 frames of 2 x 3 patches per chunk
    return oracle_mod.Geometry(F=2, Hp=2, Wp=3, H=2, d=8, pairs=(2, 1, 1))


def _proj_inputs(g, n, C, seed):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((n * g.T, C))
    w = rng.standard_normal((3 * g.H * g.d, C))
    b = rng.standard_normal(3 * g.H * g.d)
    return x, w, b


def test_fused_rope_at_position_zero_is_the_projection(oracle_mod):
    g = _geom(oracle_mod)
    x, w, b = _proj_inputs(g, 1, 5, 11)
    q, k, v = oracle_mod.qkv_project(x, w, b, heads=g.H)
    qr, kr, vr = oracle_mod.qkv_project_rope(x, w, b, g, [0])
    # chunk 0, frame 0, patch (0, 0): every angle is 0
    np.testing.assert_array_equal(qr[0, 0], q[0])
    np.testing.assert_array_equal(kr[0, 0], k[0])
    # other tokens of the chunk are rotated
    assert np.abs(qr[0, 1:] - q.reshape(qr.shape)[0, 1:]).max() > 1e-3


def test_fused_rope_keeps_pair_norms_and_v(oracle_mod):
    g = _geom(oracle_mod)
    x, w, b = _proj_inputs(g, 2, 6, 12)
    q, k, v = (t.reshape(2, g.T, g.H, g.d) for t in oracle_mod.qkv_project(x, w, b, heads=g.H))
    qr, kr, vr = oracle_mod.qkv_project_rope(x, w, b, g, [3, 7])
    np.testing.assert_array_equal(vr, v)
    for a, r in ((q, qr), (k, kr)):
        na = np.hypot(a[..., 0::2], a[..., 1::2])
        nr = np.hypot(r[..., 0::2], r[..., 1::2])
        np.testing.assert_allclose(nr, na, rtol=1e-12, atol=0)


def test_fused_rope_rotates_after_the_bias(oracle_mod):
    # W = 0: q = k = the bias for every token, so only the rotation varies
    g = _geom(oracle_mod)
    C = 4
    b = np.random.default_rng(13).standard_normal(3 * g.H * g.d)
    qr, kr, _ = oracle_mod.qkv_project_rope(np.zeros((g.T, C)), np.zeros((3 * g.H * g.d, C)), b, g, [0])
    bq = b[: g.H * g.d].reshape(g.H, g.d)
    np.testing.assert_array_equal(qr[0, 0], bq)
    assert np.abs(qr[0, 1:] - bq[None]).max() > 1e-3


def test_fused_rope_chunk_moves_only_the_time_pairs(oracle_mod):
    # the same token features in two nodes of different chunks: the pairs
    # rotated by patch row and column agree, those rotated by frame differ
    g = _geom(oracle_mod)
    x1, w, b = _proj_inputs(g, 1, 5, 14)
    qr, kr, _ = oracle_mod.qkv_project_rope(np.concatenate([x1, x1]), w, b, g, [1, 4])
    Pt = g.pairs[0]
    for r in (qr, kr):
        np.testing.assert_array_equal(r[0, :, :, 2 * Pt:], r[1, :, :, 2 * Pt:])
        assert np.abs(r[0, :, :, : 2 * Pt] - r[1, :, :, : 2 * Pt]).max() > 1e-3


def test_fused_rope_nodes_are_independent(oracle_mod):
    g = _geom(oracle_mod)
    x, w, b = _proj_inputs(g, 2, 5, 15)
    both = oracle_mod.qkv_project_rope(x, w, b, g, [2, 5])
    for i, c in enumerate((2, 5)):
        one = oracle_mod.qkv_project_rope(x[i * g.T:(i + 1) * g.T], w, b, g, [c])
        for t in range(3):
            np.testing.assert_array_equal(both[t][i], one[t][0])
