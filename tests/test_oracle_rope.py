"""Pins of the oracle's 3D RoPE reading and bf16 store rounding against closed
forms and a library conversion."""
import math

import numpy as np
import pytest
import torch


def _geom(oracle_mod, d=64, F=2, Hp=3, Wp=5):
    from paper_2609_22283_gb300.inputs import rope_pairs_for
    return oracle_mod.Geometry(F=F, Hp=Hp, Wp=Wp, H=1, d=d, pairs=rope_pairs_for(d))


def _token(g, f, h, w):
    return (f * g.Hp + h) * g.Wp + w


def test_pairs_convention():
    from paper_2609_22283_gb300.inputs import rope_pairs_for
    assert rope_pairs_for(128) == (22, 21, 21)
    assert rope_pairs_for(64) == (12, 10, 10)


def test_identity_at_origin(oracle_mod):
    g = _geom(oracle_mod)
    rng = np.random.default_rng(0)
    x = rng.standard_normal((g.T, g.d))
    y = oracle_mod.rope_head(x, 0, g)
    assert np.array_equal(y[0], x[0])          # chunk 0, frame 0, (0, 0): every angle is 0
    assert not np.allclose(y[1], x[1])


def test_pair_norms_preserved(oracle_mod):
    g = _geom(oracle_mod, d=128)
    rng = np.random.default_rng(1)
    x = rng.standard_normal((g.T, g.d))
    y = oracle_mod.rope_head(x, 7, g)
    nx = np.hypot(x[:, 0::2], x[:, 1::2])
    ny = np.hypot(y[:, 0::2], y[:, 1::2])
    np.testing.assert_allclose(ny, nx, rtol=1e-13, atol=0)


def test_direction_and_unit_frequency(oracle_mod):
    """Pair 0 of every axis has frequency theta^0 = 1, so a unit vector turns
    counter-clockwise by exactly the axis position."""
    g = _geom(oracle_mod)
    P0, P1, _ = g.pairs
    x = np.zeros((g.T, g.d))
    x[:, 0] = 1.0                 # t-axis pair 0
    x[:, 2 * P0] = 1.0            # h-axis pair 0
    x[:, 2 * (P0 + P1)] = 1.0     # w-axis pair 0
    b = 3
    u = _token(g, 1, 2, 4)
    y = oracle_mod.rope_head(x, b, g)
    t = g.F * b + 1
    assert y[u, 0] == pytest.approx(math.cos(t), abs=1e-15)
    assert y[u, 1] == pytest.approx(math.sin(t), abs=1e-15)
    assert y[u, 2 * P0] == pytest.approx(math.cos(2), abs=1e-15)
    assert y[u, 2 * P0 + 1] == pytest.approx(math.sin(2), abs=1e-15)
    assert y[u, 2 * (P0 + P1)] == pytest.approx(math.cos(4), abs=1e-15)
    assert y[u, 2 * (P0 + P1) + 1] == pytest.approx(math.sin(4), abs=1e-15)


def test_frequency_ladder(oracle_mod):
    """Pair i of an axis with D_a = 2 P_a dimensions turns at theta^(-2i/D_a)."""
    g = _geom(oracle_mod, d=128, F=1, Hp=1, Wp=2)
    P0, P1, P2 = g.pairs
    x = np.zeros((g.T, g.d))
    x[:, 0::2] = 1.0
    y = oracle_mod.rope_head(x, 0, g)
    # token 1 sits at w = 1 (t = 0, h = 0): only w pairs turn, by their frequency
    w_ang = np.arctan2(y[1, 2 * (P0 + P1) + 1::2], y[1, 2 * (P0 + P1)::2])
    expect = np.array([10000.0 ** (-2.0 * i / (2 * P2)) for i in range(P2)])
    np.testing.assert_allclose(w_ang, expect, rtol=1e-12)
    assert np.array_equal(y[1, : 2 * (P0 + P1)], x[1, : 2 * (P0 + P1)])


def test_axis_partition(oracle_mod):
    """Tokens differing only in w agree on the t and h pairs; only in h, on t and w pairs."""
    g = _geom(oracle_mod, d=128)
    P0, P1, _ = g.pairs
    rng = np.random.default_rng(2)
    row = rng.standard_normal(g.d)
    x = np.tile(row, (g.T, 1))
    y = oracle_mod.rope_head(x, 5, g)
    a, b_ = _token(g, 1, 2, 0), _token(g, 1, 2, 3)
    np.testing.assert_array_equal(y[a, : 2 * (P0 + P1)], y[b_, : 2 * (P0 + P1)])
    assert not np.allclose(y[a, 2 * (P0 + P1):], y[b_, 2 * (P0 + P1):])
    c = _token(g, 1, 0, 3)
    np.testing.assert_array_equal(y[c, : 2 * P0], y[b_, : 2 * P0])
    np.testing.assert_array_equal(y[c, 2 * (P0 + P1):], y[b_, 2 * (P0 + P1):])
    assert not np.allclose(y[c, 2 * P0: 2 * (P0 + P1)], y[b_, 2 * P0: 2 * (P0 + P1)])


def test_relative_position_dot_products(oracle_mod):
    """<R_m q, R_n k> depends only on m - n: shifting both chunks by the same
    amount leaves every query-key dot product unchanged."""
    g = _geom(oracle_mod, d=128)
    rng = np.random.default_rng(3)
    q = rng.standard_normal((g.T, g.d))
    k = rng.standard_normal((g.T, g.d))
    d1 = oracle_mod.rope_head(q, 9, g) @ oracle_mod.rope_head(k, 6, g).T
    d2 = oracle_mod.rope_head(q, 40, g) @ oracle_mod.rope_head(k, 37, g).T
    np.testing.assert_allclose(d1, d2, rtol=1e-9, atol=1e-9)
    d3 = oracle_mod.rope_head(q, 40, g) @ oracle_mod.rope_head(k, 36, g).T
    assert not np.allclose(d1, d3, atol=1e-3)


def test_composition(oracle_mod):
    """With one token per chunk (h = w = 0) a rotation at chunk 3 followed by
    one at chunk 4 equals a single rotation at chunk 7."""
    g = _geom(oracle_mod, d=64, F=1, Hp=1, Wp=1)
    rng = np.random.default_rng(4)
    x = rng.standard_normal((g.T, g.d))
    two = oracle_mod.rope_head(oracle_mod.rope_head(x, 3, g), 4, g)
    one = oracle_mod.rope_head(x, 7, g)
    np.testing.assert_allclose(two, one, rtol=1e-12, atol=1e-12)


def test_bf16_rounding_matches_library(oracle_mod):
    rng = np.random.default_rng(5)
    x32 = np.concatenate([
        rng.standard_normal(20000).astype(np.float32),
        (rng.standard_normal(2000) * 1e-38).astype(np.float32),     # subnormal range
        (rng.standard_normal(2000) * 1e30).astype(np.float32),
    ])
    # exact ties: the 16 bits below the bf16 grid are 0x8000
    base = rng.standard_normal(4000).astype(np.float32).view(np.uint32)
    ties = (base & np.uint32(0xFFFF0000)) | np.uint32(0x8000)
    x32 = np.concatenate([x32, ties.view(np.float32)])
    x32 = x32[np.isfinite(x32)]
    lib = torch.from_numpy(x32).to(torch.bfloat16).to(torch.float64).numpy()
    mine = oracle_mod.bf16(x32.astype(np.float64))
    np.testing.assert_array_equal(mine, lib)


def test_rms_norm_matches_library(oracle_mod):
    rng = np.random.default_rng(21)
    x = rng.standard_normal((40, 3, 16)) * rng.uniform(0.1, 10.0, (40, 1, 1))
    gamma = rng.uniform(0.5, 1.5, 48)
    y = oracle_mod.rms_norm(x, gamma, 1e-6)
    ref = torch.nn.functional.rms_norm(torch.from_numpy(x.reshape(40, 48)), (48,),
                                       torch.from_numpy(gamma), eps=1e-6).numpy()
    np.testing.assert_allclose(y.reshape(40, 48), ref, rtol=1e-13, atol=1e-14)
    # scale invariance (up to eps) and unit RMS with unit gamma
    y2 = oracle_mod.rms_norm(x * 7.0, np.ones(48), 1e-12)
    np.testing.assert_allclose(np.sqrt(np.mean(y2.reshape(40, 48) ** 2, axis=1)), 1.0, rtol=1e-9)
