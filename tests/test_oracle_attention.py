"""Pins of the oracle's masked softmax attention (Eq. 4) and of its per-node
pipeline (selection + RoPE + bf16 store + attention): against the dense-mask
brute force over the whole (chunk, level) grid, softmax invariants, library
routines (scipy softmax / logsumexp, torch SDPA in fp64) and row
independence."""
import math

import numpy as np
import pytest
import scipy.special
import torch

from paper_2609_22283_gb300 import inputs as I


def _tiny(oracle_mod):
    w = I.WORKLOADS["tiny"]
    inp = I.generate(w)
    g = oracle_mod.Geometry(F=w.F, Hp=w.Hp, Wp=w.Wp, H=w.H, d=w.d, pairs=w.pairs, theta=w.theta)
    return w, inp, g


def _f64(t):
    return t.to(torch.float64).numpy()


def test_tiny_against_dense_brute_force(oracle_mod):
    from oracle import brute
    w, inp, g = _tiny(oracle_mod)
    states = {k: (_f64(a), _f64(b)) for k, (a, b) in I.all_states(w, inp).items()}
    # distractors the policy must NOT select: other levels of past chunks, a
    # future chunk, and the same chunks of another sequence
    rng = np.random.default_rng(7)
    grid = dict(states)
    for s in [(0, 1, 1), (0, 1, 2), (0, 2, 0), (0, 2, 2), (0, 4, 0), (1, 1, 0), (1, 2, 1)]:
        grid[s] = (rng.standard_normal((w.T, w.H, w.d)), rng.standard_normal((w.T, w.H, w.d)))
    scale = 1.0 / math.sqrt(w.d)
    for i, node in enumerate(w.nodes):
        q = _f64(inp.q[i])
        out, lse, _ = oracle_mod.node_forward(g, oracle_mod.POLICY_IDS[w.policy], w.W, node,
                                              states, q, range(w.H), range(w.T), scale)
        bo, bl = brute.brute_forward(w.policy, w.W, w.F, w.Hp, w.Wp, w.pairs, w.theta, node,
                                     grid, q, range(w.H), scale)
        np.testing.assert_allclose(out, bo, rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse, bl, rtol=0, atol=1e-12)


def test_hidden_state_matches_brute_force(oracle_mod):
    from oracle import brute
    w, inp, g = _tiny(oracle_mod)
    states = {k: (_f64(a), _f64(b)) for k, (a, b) in I.all_states(w, inp).items()}
    node = w.nodes[0]                      # (3, 2) reads (2, 1) and (1, 0)
    hidden = frozenset({(2, 1)})
    q = _f64(inp.q[0])
    scale = 0.2
    out, lse, _ = oracle_mod.node_forward(g, oracle_mod.POLICY_IDS[w.policy], w.W, node, states, q,
                                          [1], range(w.T), scale, hidden=hidden)
    bo, bl = brute.brute_forward(w.policy, w.W, w.F, w.Hp, w.Wp, w.pairs, w.theta, node, states, q,
                                 [1], scale, hidden=hidden)
    np.testing.assert_allclose(out, bo, rtol=0, atol=1e-12)
    full, _, _ = oracle_mod.node_forward(g, oracle_mod.POLICY_IDS[w.policy], w.W, node, states, q,
                                         [1], range(w.T), scale)
    assert not np.allclose(out, full)


def test_rows_are_the_library_softmax(oracle_mod):
    rng = np.random.default_rng(0)
    L, d = 48, 64
    q = rng.standard_normal((10, d))
    k = rng.standard_normal((L, d))
    v = np.eye(L, d)                        # one-hot values: out = attention weights
    mask = np.where(rng.random(L) < 0.3, -np.inf, 0.0)
    scale = 0.37
    out, lse = oracle_mod.attend_rows(q, k, v, scale, mask)
    logits = scale * q @ k.T + mask
    ref = scipy.special.softmax(logits, axis=1)
    np.testing.assert_allclose(out[:, :L], ref, rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(out.sum(axis=1), 1.0, rtol=1e-13)
    assert np.all(out[:, :L][:, mask == -np.inf] == 0.0)
    np.testing.assert_allclose(lse, scipy.special.logsumexp(logits, axis=1), rtol=1e-13)


def test_constant_values_and_identical_keys(oracle_mod):
    rng = np.random.default_rng(1)
    L, d = 300, 128
    q = rng.standard_normal((7, d)) * 3
    k = rng.standard_normal((L, d))
    v = np.full((L, d), 0.625)
    out, _ = oracle_mod.attend_rows(q, k, v, 0.1)
    np.testing.assert_allclose(out, 0.625, rtol=1e-14)
    k_same = np.tile(rng.standard_normal(d), (L, 1))
    v = rng.standard_normal((L, d))
    mask = np.where(np.arange(L) % 3 == 0, -np.inf, 0.0)
    out, lse = oracle_mod.attend_rows(q, k_same, v, 0.1, mask)
    np.testing.assert_allclose(out, np.tile(v[mask == 0].mean(axis=0), (7, 1)), rtol=1e-12, atol=1e-14)


def test_fully_masked_row_reading(oracle_mod):
    q = np.ones((2, 64))
    k = np.ones((5, 64))
    v = np.ones((5, 64))
    out, lse = oracle_mod.attend_rows(q, k, v, 1.0, np.full(5, -np.inf))
    assert np.all(out == 0.0) and np.all(lse == -np.inf)


def test_clean_single_node_is_block_causal_sdpa(oracle_mod):
    """Clean policy, one node: the node's rows equal the last block of ordinary
    block-causal attention over [x_{b-W}^0, ..., x_{b-1}^0, x_b^j] (fp64 torch SDPA)."""
    F, Hp, Wp, H, d, W = 1, 4, 6, 2, 64, 3
    pairs = I.rope_pairs_for(d)
    g = oracle_mod.Geometry(F=F, Hp=Hp, Wp=Wp, H=H, d=d, pairs=pairs)
    T = g.T
    b, j = 9, 3
    rng = np.random.default_rng(3)
    bfr = lambda x: oracle_mod.bf16(x)
    states = {}
    for c in range(b - W, b):
        states[(0, c, 0)] = (bfr(rng.standard_normal((T, H, d))), bfr(rng.standard_normal((T, H, d))))
    states[(0, b, j)] = (bfr(rng.standard_normal((T, H, d))), bfr(rng.standard_normal((T, H, d))))
    # states the clean policy must ignore
    for c in range(b - W, b):
        states[(0, c, j)] = (bfr(rng.standard_normal((T, H, d))), bfr(rng.standard_normal((T, H, d))))
    q_raw = bfr(rng.standard_normal((T, H, d)))
    scale = 1 / math.sqrt(d)
    out, lse, sel = oracle_mod.node_forward(g, oracle_mod.POLICY_CLEAN, W, (0, b, j), states, q_raw,
                                            range(H), range(T), scale)
    assert sel == [(b - r, 0) for r in range(1, W + 1)]
    order = [(c, 0) for c in range(b - W, b)] + [(b, j)]
    for h in range(H):
        ks = [oracle_mod.bf16(oracle_mod.rope_head(states[(0,) + s][0][:, h, :], s[0], g)) for s in order]
        vs = [states[(0,) + s][1][:, h, :] for s in order]
        qs = [oracle_mod.bf16(oracle_mod.rope_head(np.zeros((T, d)), s[0], g)) for s in order[:-1]]
        qs.append(oracle_mod.bf16(oracle_mod.rope_head(q_raw[:, h, :], b, g)))
        Q = torch.from_numpy(np.concatenate(qs))[None, None]
        K = torch.from_numpy(np.concatenate(ks))[None, None]
        V = torch.from_numpy(np.concatenate(vs))[None, None]
        blk = torch.arange(len(order) * T) // T
        allowed = blk[:, None] >= blk[None, :]                     # block-causal
        ref = torch.nn.functional.scaled_dot_product_attention(Q, K, V, attn_mask=allowed, scale=scale)
        np.testing.assert_allclose(out[h], ref[0, 0, -T:].numpy(), rtol=1e-12, atol=1e-13)


def test_rows_independent(oracle_mod):
    """Computing a subset of rows gives the same numbers as computing all rows."""
    w, inp, g = _tiny(oracle_mod)
    states = {k: (_f64(a), _f64(b)) for k, (a, b) in I.all_states(w, inp).items()}
    q = _f64(inp.q[0])
    scale = 0.125
    full, fl, _ = oracle_mod.node_forward(g, 2, w.W, w.nodes[0], states, q, [0, 1], range(w.T), scale)
    rows = [5, 0, 63, 17]
    part, pl, _ = oracle_mod.node_forward(g, 2, w.W, w.nodes[0], states, q, [1], rows, scale)
    np.testing.assert_array_equal(part[0], full[1][rows])
    np.testing.assert_array_equal(pl[0], fl[1][rows])


@pytest.mark.parametrize("name", ["clean1", "same4", "prog4", "prog4r", "stress14b"])
def test_full_geometry_selection_is_prefilled(oracle_mod, name):
    """Every state a workload's nodes select is either prefilled or written by
    a node of the same step (the in-round progressive reads)."""
    w = I.WORKLOADS[name]
    have = set(w.states)
    for (s, b, j) in w.nodes:
        for (c, lvl) in oracle_mod.select(oracle_mod.POLICY_IDS[w.policy], w.W, b, j):
            assert (s, c, lvl) in have


def test_frame_causal_against_dense_brute_force(oracle_mod):
    from oracle import brute
    w = I.WORKLOADS["tinyfc"]                 # 3 latent frames of 32 tokens per chunk
    inp = I.generate(w)
    g = oracle_mod.Geometry(F=w.F, Hp=w.Hp, Wp=w.Wp, H=w.H, d=w.d, pairs=w.pairs, theta=w.theta)
    states = {k: (_f64(a), _f64(b)) for k, (a, b) in I.all_states(w, inp).items()}
    rng = np.random.default_rng(11)
    grid = dict(states)
    for s in [(0, 2, 0), (0, 4, 0), (0, 1, 1)]:
        grid[s] = (rng.standard_normal((w.T, w.H, w.d)), rng.standard_normal((w.T, w.H, w.d)))
    scale = 1.0 / math.sqrt(w.d)
    for i, node in enumerate(w.nodes):
        q = _f64(inp.q[i])
        out, lse, _ = oracle_mod.node_forward(g, oracle_mod.POLICY_IDS[w.policy], w.W, node, states,
                                              q, range(w.H), range(w.T), scale, within="frame_causal")
        bo, bl = brute.brute_forward(w.policy, w.W, w.F, w.Hp, w.Wp, w.pairs, w.theta, node, grid, q,
                                     range(w.H), scale, frame_causal=True)
        np.testing.assert_allclose(out, bo, rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse, bl, rtol=0, atol=1e-12)
        bid, _, _ = oracle_mod.node_forward(g, oracle_mod.POLICY_IDS[w.policy], w.W, node, states,
                                            q, range(w.H), range(w.T), scale)
        last = slice(2 * w.Hp * w.Wp, w.T)    # the last frame sees the whole chunk either way
        np.testing.assert_array_equal(out[:, last], bid[:, last])
        assert not np.allclose(out[:, :w.Hp * w.Wp], bid[:, :w.Hp * w.Wp])


def test_frame_causal_single_frame_is_bidirectional(oracle_mod):
    w, inp, g = _tiny(oracle_mod)              # F = 1
    states = {k: (_f64(a), _f64(b)) for k, (a, b) in I.all_states(w, inp).items()}
    q = _f64(inp.q[0])
    a, la, _ = oracle_mod.node_forward(g, 2, w.W, w.nodes[0], states, q, [0, 1], range(w.T), 0.125,
                                       within="frame_causal")
    b, lb, _ = oracle_mod.node_forward(g, 2, w.W, w.nodes[0], states, q, [0, 1], range(w.T), 0.125)
    np.testing.assert_array_equal(a, b)
    np.testing.assert_array_equal(la, lb)


def _sparse_case(oracle_mod, within):
    w = I.WORKLOADS["tinys"]                  # 320-token chunks: 3 tiles, the last of 64 rows
    if within == "frame_causal":              # two latent frames of 160 tokens
        w = I.Workload(**{**w.__dict__, "name": "tinysfc", "F": 2, "Hp": 8, "within": within})
    inp = I.generate(w)
    g = oracle_mod.Geometry(F=w.F, Hp=w.Hp, Wp=w.Wp, H=w.H, d=w.d, pairs=w.pairs, theta=w.theta)
    states = {k: (_f64(a), _f64(b)) for k, (a, b) in I.all_states(w, inp).items()}
    masks = I.unpack_bits(I.tile_mask(w), (1 + w.W) * w.tiles).numpy()
    return w, inp, g, states, masks


@pytest.mark.parametrize("within", ["bidirectional", "frame_causal"])
def test_tile_mask_against_dense_brute_force(oracle_mod, within):
    from oracle import brute
    w, inp, g, states, masks = _sparse_case(oracle_mod, within)
    # the brute force sees extra states the nodes must not read
    rng = np.random.default_rng(5)
    grid = dict(states)
    for s in [(0, 2, 0), (0, 4, 0), (0, 1, 1)]:
        grid[s] = (rng.standard_normal((w.T, w.H, w.d)), rng.standard_normal((w.T, w.H, w.d)))
    scale = 1.0 / math.sqrt(w.d)
    for i, node in enumerate(w.nodes):
        assert not masks[i].all()             # the mask hides something for this node
        q = _f64(inp.q[i])
        out, lse, _ = oracle_mod.node_forward(g, oracle_mod.POLICY_IDS[w.policy], w.W, node, states,
                                              q, range(w.H), range(w.T), scale, within=within,
                                              tile_mask=masks[i])
        bo, bl = brute.brute_forward(w.policy, w.W, w.F, w.Hp, w.Wp, w.pairs, w.theta, node, grid, q,
                                     range(w.H), scale, frame_causal=within == "frame_causal",
                                     tile_mask=masks[i])
        np.testing.assert_allclose(out, bo, rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse, bl, rtol=0, atol=1e-12)
        dense, _, _ = oracle_mod.node_forward(g, oracle_mod.POLICY_IDS[w.policy], w.W, node, states,
                                              q, range(w.H), range(w.T), scale, within=within)
        assert not np.allclose(out, dense)        # the mask changes the result


def test_tile_mask_special_cases(oracle_mod):
    """All bits set is the dense node; no context bit set is the node with
    every selected state hidden; a query tile with no bit at all gets O = 0."""
    w, inp, g, states, masks = _sparse_case(oracle_mod, "bidirectional")
    pol = oracle_mod.POLICY_IDS[w.policy]
    node = w.nodes[0]
    q = _f64(inp.q[0])
    nt = w.tiles
    dense, dl, sel = oracle_mod.node_forward(g, pol, w.W, node, states, q, range(w.H), range(w.T), 0.125)
    ones = np.ones_like(masks[0])
    a, la, _ = oracle_mod.node_forward(g, pol, w.W, node, states, q, range(w.H), range(w.T), 0.125,
                                       tile_mask=ones)
    np.testing.assert_array_equal(a, dense)
    np.testing.assert_array_equal(la, dl)
    own_only = np.zeros_like(ones)
    own_only[:, :nt] = True
    b, lb, _ = oracle_mod.node_forward(g, pol, w.W, node, states, q, range(w.H), range(w.T), 0.125,
                                       tile_mask=own_only)
    hid, lh, _ = oracle_mod.node_forward(g, pol, w.W, node, states, q, range(w.H), range(w.T), 0.125,
                                         hidden=frozenset(sel))
    np.testing.assert_array_equal(b, hid)
    np.testing.assert_array_equal(lb, lh)
    none_for_tile1 = ones.copy()
    none_for_tile1[1, :] = False
    c, lc, _ = oracle_mod.node_forward(g, pol, w.W, node, states, q, range(w.H), range(w.T), 0.125,
                                       tile_mask=none_for_tile1)
    assert np.all(c[:, 128:256] == 0.0) and np.all(lc[:, 128:256] == -np.inf)
    np.testing.assert_array_equal(c[:, :128], dense[:, :128])


def _own_mask(T, seed, density=0.5):
    rng = np.random.default_rng(seed)
    m = rng.random((T, T)) < density
    np.fill_diagonal(m, True)
    m[5, :] = False                            # row 5 sees no key of its own chunk
    return m


@pytest.mark.parametrize("within", ["bidirectional", "frame_causal"])
def test_own_token_mask_against_dense_brute_force(oracle_mod, within):
    from oracle import brute
    w, inp, g, states, masks = _sparse_case(oracle_mod, within)
    rng = np.random.default_rng(6)
    grid = dict(states)
    for s in [(0, 2, 0), (0, 4, 0)]:
        grid[s] = (rng.standard_normal((w.T, w.H, w.d)), rng.standard_normal((w.T, w.H, w.d)))
    scale = 1.0 / math.sqrt(w.d)
    rows = [0, 1, 5, 64, 127, 128, 200, 255, 256, 300, w.T - 1]
    for i, node in enumerate(w.nodes):
        own = _own_mask(w.T, 10 + i)
        q = _f64(inp.q[i])
        for tm in (None, masks[i]):
            out, lse, _ = oracle_mod.node_forward(g, oracle_mod.POLICY_IDS[w.policy], w.W, node, states,
                                                  q, range(w.H), rows, scale, within=within,
                                                  tile_mask=tm, own_mask=own)
            bo, bl = brute.brute_forward(w.policy, w.W, w.F, w.Hp, w.Wp, w.pairs, w.theta, node, grid,
                                         q, range(w.H), scale, frame_causal=within == "frame_causal",
                                         tile_mask=tm, own_mask=own)
            np.testing.assert_allclose(out, bo[:, rows], rtol=0, atol=1e-12)
            np.testing.assert_allclose(lse, bl[:, rows], rtol=0, atol=1e-12)


def test_own_token_mask_special_cases(oracle_mod):
    """An all-true own mask is the unmasked node; the lower-triangular-by-frame
    own mask is the frame-causal mode; a row whose own mask is all false sees
    only the history."""
    w, inp, g, states, _ = _sparse_case(oracle_mod, "bidirectional")
    pol = oracle_mod.POLICY_IDS[w.policy]
    node = w.nodes[0]
    q = _f64(inp.q[0])
    rows = [0, 5, 130, w.T - 1]
    base, bl, sel = oracle_mod.node_forward(g, pol, w.W, node, states, q, range(w.H), rows, 0.125)
    a, la, _ = oracle_mod.node_forward(g, pol, w.W, node, states, q, range(w.H), rows, 0.125,
                                       own_mask=np.ones((w.T, w.T), bool))
    np.testing.assert_array_equal(a, base)
    # frame-causal as a token mask (frames of 160 tokens in the two-frame variant)
    w2, inp2, g2, states2, _ = _sparse_case(oracle_mod, "frame_causal")
    q2 = _f64(inp2.q[0])
    ft = w2.Hp * w2.Wp
    fc = (np.arange(w2.T)[None, :] // ft) <= (np.arange(w2.T)[:, None] // ft)
    x, lx, _ = oracle_mod.node_forward(g2, pol, w2.W, w2.nodes[0], states2, q2, range(w2.H), rows, 0.125,
                                       within="frame_causal")
    y, ly, _ = oracle_mod.node_forward(g2, pol, w2.W, w2.nodes[0], states2, q2, range(w2.H), rows, 0.125,
                                       own_mask=fc)
    np.testing.assert_array_equal(x, y)
    # no own key: the row attends the history alone, i.e. the node with its own
    # state hidden from that row
    none = np.ones((w.T, w.T), bool)
    none[130, :] = False
    z, lz, _ = oracle_mod.node_forward(g, pol, w.W, node, states, q, range(w.H), [130], 0.125,
                                       own_mask=none)
    assert not np.allclose(z, base[:, 2:3])


def _hist_mask(n, T, seed, density=0.5):
    rng = np.random.default_rng(seed)
    m = rng.random((n, T, T)) < density
    m[:, 7, :] = False                         # row 7 sees no history key
    return m


@pytest.mark.parametrize("within", ["bidirectional", "frame_causal"])
def test_history_token_mask_against_dense_brute_force(oracle_mod, within):
    """The token-level M of Eq. 4 on the history: the oracle's slot-list form
    against the dense mask over the whole (chunk, level) grid, alone and with
    an own-chunk token mask and a block-sparse tile mask."""
    from oracle import brute
    w, inp, g, states, masks = _sparse_case(oracle_mod, within)
    rng = np.random.default_rng(8)
    grid = dict(states)
    for s in [(0, 2, 0), (0, 4, 0)]:
        grid[s] = (rng.standard_normal((w.T, w.H, w.d)), rng.standard_normal((w.T, w.H, w.d)))
    scale = 1.0 / math.sqrt(w.d)
    rows = [0, 1, 5, 7, 64, 127, 128, 200, 255, 256, 300, w.T - 1]
    for i, node in enumerate(w.nodes):
        n_sel = max(0, min(w.W, node[1] - 1))
        hist = _hist_mask(max(n_sel, 1), w.T, 20 + i)
        own = _own_mask(w.T, 30 + i)
        q = _f64(inp.q[i])
        for own_m, tm in ((None, None), (own, masks[i])):
            out, lse, _ = oracle_mod.node_forward(g, oracle_mod.POLICY_IDS[w.policy], w.W, node, states,
                                                  q, range(w.H), rows, scale, within=within,
                                                  tile_mask=tm, own_mask=own_m, hist_mask=hist)
            bo, bl = brute.brute_forward(w.policy, w.W, w.F, w.Hp, w.Wp, w.pairs, w.theta, node, grid,
                                         q, range(w.H), scale, frame_causal=within == "frame_causal",
                                         tile_mask=tm, own_mask=own_m, hist_mask=hist)
            np.testing.assert_allclose(out, bo[:, rows], rtol=0, atol=1e-12)
            np.testing.assert_allclose(lse, bl[:, rows], rtol=0, atol=1e-12)


def test_history_token_mask_special_cases(oracle_mod):
    """An all-true history mask is the unmasked node; a state whose bits are
    all clear for every row is that state hidden (ctx_visible = 0); a row
    with no history bit sees its own chunk alone."""
    w, inp, g, states, _ = _sparse_case(oracle_mod, "bidirectional")
    pol = oracle_mod.POLICY_IDS[w.policy]
    node = w.nodes[0]
    q = _f64(inp.q[0])
    rows = [0, 5, 130, w.T - 1]
    n_sel = max(0, min(w.W, node[1] - 1))
    assert n_sel == 2
    base, bl, sel = oracle_mod.node_forward(g, pol, w.W, node, states, q, range(w.H), rows, 0.125)
    ones = np.ones((n_sel, w.T, w.T), bool)
    a, la, _ = oracle_mod.node_forward(g, pol, w.W, node, states, q, range(w.H), rows, 0.125,
                                       hist_mask=ones)
    np.testing.assert_array_equal(a, base)
    np.testing.assert_array_equal(la, bl)
    second_off = ones.copy()
    second_off[1] = False
    b, lb2, _ = oracle_mod.node_forward(g, pol, w.W, node, states, q, range(w.H), rows, 0.125,
                                        hist_mask=second_off)
    hid, lh, _ = oracle_mod.node_forward(g, pol, w.W, node, states, q, range(w.H), rows, 0.125,
                                         hidden=frozenset({sel[1]}))
    np.testing.assert_array_equal(b, hid)
    np.testing.assert_array_equal(lb2, lh)
    no_hist = np.zeros((n_sel, w.T, w.T), bool)
    c, lc, _ = oracle_mod.node_forward(g, pol, w.W, node, states, q, range(w.H), rows, 0.125,
                                       hist_mask=no_hist)
    own_alone, lo, _ = oracle_mod.node_forward(g, pol, w.W, node, states, q, range(w.H), rows, 0.125,
                                               hidden=frozenset(sel))
    np.testing.assert_array_equal(c, own_alone)
    assert not np.allclose(c, base)
