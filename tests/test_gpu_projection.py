"""GPU parity of the QKV projection (sva_qkv_project, the tcgen05 GEMM that
feeds sva_rope_kv_write) against the fp64 oracle, and of the chain
projection -> RoPE + cache write -> attention against the oracle's chain.

Tolerance (derived from the arithmetic): the library rounds each fp32
accumulator to bf16 once (at most 2^-9 relative) and accumulates in fp32 in
its own order; element bound |d| <= 2^-8 |y| + 1e-3 rms(y), and a relative
RMS of 2e-3."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_22283_gb300 import inputs as I
from paper_2609_22283_gb300 import sva
from paper_2609_22283_gb300.pipeline import Step, geometry_for
from tests import _parity as P

pytestmark = pytest.mark.gpu


def _check(got, ref, what):
    got = got.astype(np.float64)
    rms = float(np.sqrt(np.mean(ref ** 2)))
    bound = 2.0 ** -8 * np.abs(ref) + 1e-3 * rms
    bad = np.abs(got - ref) > bound
    assert not bad.any(), f"{what}: {int(bad.sum())} elements out of bound, max |d| {np.abs(got - ref).max():.3e}"
    rr = float(np.linalg.norm(got - ref) / np.linalg.norm(ref))
    assert rr <= 2e-3, f"{what}: rel rms {rr:.3e}"


def _project(w, C, rows_sample=None, bias=True):
    x, wt, b = I.projection_inputs(w, C)
    cache = sva.Cache(geometry_for(w))
    dev = torch.device("cuda")
    xd, wd = x.to(dev).contiguous(), wt.to(dev).contiguous()
    bd = b.to(dev) if bias else None
    outs = [torch.empty((w.n_nodes, w.T, w.H, w.d), dtype=torch.bfloat16, device=dev) for _ in range(3)]
    cache.qkv_project(xd, wd, bd, *outs)
    assert cache.poll() == 0
    n_rows = w.n_nodes * w.T
    idx = np.arange(n_rows) if rows_sample is None else np.asarray(rows_sample)
    sel = torch.from_numpy(idx).to(dev)
    got = [o.view(n_rows, w.H, w.d).index_select(0, sel).float().cpu().numpy() for o in outs]
    xs = x.reshape(n_rows, C)[torch.from_numpy(idx)].double().numpy()
    ref = oracle.qkv_project(xs, wt.double().numpy(), b.double().numpy() if bias else None, heads=w.H)
    for t in range(3):
        _check(got[t], ref[t], f"{w.name} C={C} tensor {'qkv'[t]}")
    cache.close()


@pytest.mark.parametrize("C", [192, 200])
def test_tiny_projection_all_rows(oracle_mod, C):
    _project(I.WORKLOADS["tiny"], C)          # H*d = 128: 128-wide tiles; C = 200: ragged K block


def test_tinys_projection_no_bias(oracle_mod):
    _project(I.WORKLOADS["tinys"], 256, bias=False)


def test_wan_geometry_projection_sampled(oracle_mod):
    # 4 x 4680 token rows (ragged last 128-row tile), 1536 -> 3 x 12 x 128
    w = I.WORKLOADS["prog4"]
    rng = np.random.default_rng(21)
    rows = sorted(set(rng.choice(w.n_nodes * w.T, 300, replace=False).tolist()) | {0, 18719, 18688, 127, 128})
    _project(w, 1536, rows)


def test_clean1_rows_projection_split_tail_sampled(oracle_mod):
    # 4680 rows: 19 tiles of 256 rows, the last with 72 (the odd CTA of the
    # pair holds none of them); 342 tiles over the pairs leave a partial last
    # round, split into half-width items
    w = I.WORKLOADS["clean1"]
    rng = np.random.default_rng(23)
    edges = {0, 127, 128, 255, 256, 4351, 4352, 4607, 4608, 4679}
    rows = sorted(set(rng.choice(w.n_nodes * w.T, 300, replace=False).tolist()) | edges)
    _project(w, 1536, rows)


def test_14b_geometry_projection_sampled(oracle_mod):
    # 8 x 4680 rows, 5120 -> 3 x 40 x 128: 147 row tiles in groups of 16 (a
    # weight larger than the L2), 80 K blocks
    w = I.WORKLOADS["stress14b"]
    rng = np.random.default_rng(25)
    rows = sorted(set(rng.choice(w.n_nodes * w.T, 48, replace=False).tolist()) | {0, 4095, 4096, 37439})
    _project(w, 5120, rows)


# 2 nodes of T = 100 tokens (one latent frame of 10 x 10), 2 heads of 128: 200
# rows, so the one 256-row tile of a CTA pair gives the even CTA 128 rows and
# the odd one 72 (the rows past 200 read zeros and are not stored); 256-wide
# output tiles, 3 of them, whose last round is split into half-width items.
ODD_HALF = I.Workload(name="oddhalf", seed=27, F=1, Hp=10, Wp=10, H=2, d=128, K=2, W=2,
                      policy="prog", nodes=((0, 3, 2), (0, 2, 1)), prefilled=((0, 1, 0),))


@pytest.mark.parametrize("wp", [1, 257])
def test_projection_row_count_edges(oracle_mod, wp):
    # one node of T = 1 or 257 tokens: a single row (the pair's odd CTA and
    # 127 rows of the even one empty), and a second 256-row tile holding one row
    w = I.Workload(name=f"rows{wp}", seed=28, F=1, Hp=1, Wp=wp, H=2, d=128, K=2, W=2,
                   policy="clean", nodes=((0, 2, 1),), prefilled=((0, 1, 0),))
    _project(w, 256)


def test_projection_odd_cta_partly_filled(oracle_mod):
    _project(ODD_HALF, 384)


def test_fused_projection_rope_odd_cta_partly_filled(oracle_mod):
    w = ODD_HALF
    step, inp, q, x, wt, b, nodes = _fused(w, 384)
    rows = [range(w.T)] * w.n_nodes
    _check_fused(w, step, q, _fused_reference(w, x, wt, b, rows), rows, nodes)
    step.close()


@pytest.mark.parametrize("name", ["clean1", "prog4"])
def test_projection_bitwise_repeatable(name):
    """The CTA pairs' signalling (both CTAs' copies counted on the even CTA's
    stage barrier, commits to each CTA's barriers, remote accumulator-free
    arrivals) leaves no race: repeated launches give the same bits, plain
    and fused."""
    w = I.WORKLOADS[name]
    C = w.H * w.d
    dev = torch.device("cuda")
    x, wt, b = (t.to(dev).contiguous() for t in I.projection_inputs(w, C))
    step = Step(w)
    step.prefill(I.generate(w))
    nodes, _ = step.node_table()
    shape = (w.n_nodes, w.T, w.H, w.d)
    runs = []
    for _ in range(3):
        outs = [torch.empty(shape, dtype=torch.bfloat16, device=dev) for _ in range(3)]
        step.cache.qkv_project(x, wt, b, *outs)
        q = torch.empty(shape, dtype=torch.bfloat16, device=dev)
        step.cache.qkv_project_rope(nodes, x, wt, b, q)
        own = [n.own_slot for n in nodes]
        runs.append([o.view(torch.int16) for o in outs] +
                    [q.view(torch.int16), step.cache.slot_pool()[own].view(torch.int16).clone()])
    assert step.cache.poll() == 0
    for r in runs[1:]:
        for a, b0 in zip(r, runs[0]):
            assert torch.equal(a, b0)
    step.close()


def test_projection_feeds_rope_and_attention(oracle_mod):
    """x -> sva_qkv_project -> sva_rope_kv_write -> sva_attend_nodes against the
    oracle's projection (rounded to bf16 as stored) -> node_forward."""
    w = I.WORKLOADS["tiny"]
    C = 128
    inp = I.generate(w)                        # history states stay the seeded ones
    x, wt, b = I.projection_inputs(w, C)
    dev = torch.device("cuda")
    step = Step(w)
    step.prefill(inp)
    q, k, v = (torch.empty((w.n_nodes, w.T, w.H, w.d), dtype=torch.bfloat16, device=dev) for _ in range(3))
    step.cache.qkv_project(x.to(dev).contiguous(), wt.to(dev).contiguous(), b.to(dev), q, k, v)
    out, lse = step.outputs()
    step.run(q, k, v, out, lse)
    assert step.cache.poll() == 0
    rq, rk, rv = oracle.qkv_project(x.double().numpy().reshape(-1, C), wt.double().numpy(),
                                    b.double().numpy(), heads=w.H)
    shape = (w.n_nodes, w.T, w.H, w.d)
    rq, rk, rv = (torch.from_numpy(oracle.bf16(t).reshape(shape)) for t in (rq, rk, rv))
    inp2 = I.Inputs(inp.history, rq, rk, rv)
    states = P.oracle_states(w, inp2)
    got = out.float().cpu().numpy()
    for i in range(w.n_nodes):
        ref, _ = P.oracle_node(w, inp2, states, i, range(w.H), range(w.T))
        for h in range(w.H):
            P.assert_close(got[i, :, h, :], ref[h], f"projection chain node {i} head {h}")
    step.close()


def test_projection_argument_errors(sva_mod):
    w = I.WORKLOADS["tiny"]
    cache = sva.Cache(geometry_for(w))
    lib = sva_mod.load()
    z = torch.zeros(64 * 128, dtype=torch.bfloat16, device="cuda")
    p = lambda t: __import__("ctypes").c_void_p(t.data_ptr())
    st = lib.sva_qkv_project(cache.handle, p(z), 64, 100, p(z), None, p(z), p(z), p(z), None)
    assert st == sva_mod.ERR_INVALID_ARGUMENT      # in_features not a multiple of 8
    st = lib.sva_qkv_project(cache.handle, None, 64, 128, p(z), None, p(z), p(z), p(z), None)
    assert st == sva_mod.ERR_INVALID_ARGUMENT
    cache.close()


@pytest.mark.parametrize("which", ["weight", "x", "bias", "q"])
def test_projection_rejects_memory_off_the_device(sva_mod, which):
    """Every operand must be memory of the cache's GPU: a host pointer (here
    pinned host memory, which the GPU could otherwise reach) is refused with
    INVALID_ARGUMENT before anything is launched."""
    import ctypes
    w = I.WORKLOADS["tiny"]
    cache = sva.Cache(geometry_for(w))
    lib = sva_mod.load()
    dev = torch.device("cuda")
    rows, C, N = 64, 128, w.H * w.d
    t = {"x": torch.ones((rows, C), dtype=torch.bfloat16, device=dev),
         "weight": torch.ones((3 * N, C), dtype=torch.bfloat16, device=dev),
         "bias": torch.zeros(3 * N, dtype=torch.float32, device=dev),
         "q": torch.full((rows, N), 7.0, dtype=torch.bfloat16, device=dev)}
    t[which] = t[which].cpu().pin_memory()
    k = torch.full((rows, N), 7.0, dtype=torch.bfloat16, device=dev)
    v = torch.full((rows, N), 7.0, dtype=torch.bfloat16, device=dev)
    p = lambda a: ctypes.c_void_p(a.data_ptr())
    st = lib.sva_qkv_project(cache.handle, p(t["x"]), rows, C, p(t["weight"]), p(t["bias"]),
                             p(t["q"]), p(k), p(v), None)
    assert st == sva_mod.ERR_INVALID_ARGUMENT, st
    assert "not device memory" in sva_mod.last_error()
    torch.cuda.synchronize()
    assert bool((k == 7.0).all()) and bool((v == 7.0).all())     # nothing was launched
    assert cache.poll() == 0
    cache.close()


@pytest.mark.parametrize("fused", [False, True])
def test_projection_three_heads_of_128(oracle_mod, fused):
    """H*d = 384: 128-wide tiles (one head each).  The plain projection splits
    its partial last round into 64-wide items; the fused epilogue may not
    (half a head), so it runs whole tiles.  All rows of 2 nodes of T = 180."""
    base = I.WORKLOADS["tiny"]
    w = I.Workload(**{**base.__dict__, "name": "h3d128", "F": 3, "Hp": 6, "Wp": 10, "H": 3,
                      "d": 128, "pairs": None})
    if not fused:
        _project(w, 256)
        return
    step, inp, q, x, wt, b, nodes = _fused(w, 256)
    rows = [range(w.T)] * w.n_nodes
    _check_fused(w, step, q, _fused_reference(w, x, wt, b, rows), rows, nodes)
    step.close()


# ---------------------------------------------------------------- fused projection + RoPE + cache write

def _fused(w, C, rows_sample=None):
    """Runs sva_qkv_project_rope for the workload's nodes; returns the step,
    the device Q', the host x, weight, bias and the node table."""
    inp = I.generate(w)
    dev = torch.device("cuda")
    step = Step(w)
    step.prefill(inp)
    x, wt, b = I.projection_inputs(w, C)
    nodes, n = step.node_table()
    q = torch.empty((n, w.T, w.H, w.d), dtype=torch.bfloat16, device=dev)
    step.cache.qkv_project_rope(nodes, x.to(dev).contiguous(), wt.to(dev).contiguous(), b.to(dev), q)
    assert step.cache.poll() == 0
    return step, inp, q, x, wt, b, nodes


def _fused_reference(w, x, wt, b, rows_by_node):
    """Oracle Q', K', V of the requested token rows of each node (fp64):
    the projection of those rows, placed in a zero [T][H][d] block so that
    rope_head rotates them at their own positions."""
    g = P.oracle_geometry(w)
    C = x.shape[-1]
    xs = x.double().numpy().reshape(w.n_nodes, w.T, C)
    ref = []
    for i, (_, chunk, _) in enumerate(w.nodes):
        rows = np.asarray(rows_by_node[i])
        q, k, v = oracle.qkv_project(xs[i, rows], wt.double().numpy(), b.double().numpy(), heads=w.H)
        full = [np.zeros((w.T, w.H, w.d)) for _ in range(3)]
        for t, a in zip(full, (q, k, v)):
            t[rows] = a
        for h in range(w.H):
            full[0][:, h] = oracle.rope_head(full[0][:, h], chunk, g)
            full[1][:, h] = oracle.rope_head(full[1][:, h], chunk, g)
        ref.append([t[rows] for t in full])
    return ref


def _check_fused(w, step, q, ref, rows_by_node, nodes):
    pool = step.cache.slot_pool()
    gq = q.float().cpu().numpy()
    for i in range(w.n_nodes):
        rows = np.asarray(rows_by_node[i])
        slot = nodes[i].own_slot
        gk = pool[slot, 0, :, : w.T, :].permute(1, 0, 2).float().cpu().numpy()[rows]
        gv = pool[slot, 1, :, : w.T, :].permute(1, 0, 2).float().cpu().numpy()[rows]
        _check(gq[i, rows], ref[i][0], f"{w.name} node {i} Q'")
        _check(gk, ref[i][1], f"{w.name} node {i} K'")
        _check(gv, ref[i][2], f"{w.name} node {i} V")


def test_fused_projection_rope_tiny_all_rows(oracle_mod):
    w = I.WORKLOADS["tiny"]                     # H*d = 128: 128-wide tiles, 2 nodes
    step, inp, q, x, wt, b, nodes = _fused(w, 192)
    rows = [range(w.T)] * w.n_nodes
    _check_fused(w, step, q, _fused_reference(w, x, wt, b, rows), rows, nodes)
    step.close()


def test_fused_projection_rope_four_heads_per_tile(oracle_mod):
    # H*d = 256 with d = 64: 256-wide tiles holding four heads, 3 latent
    # frames of 6 x 10 tokens (T = 180, ragged last 128-row tile)
    base = I.WORKLOADS["tiny"]
    w = I.Workload(**{**base.__dict__, "name": "tinyh4", "F": 3, "Hp": 6, "Wp": 10, "H": 4,
                      "pairs": None})
    step, inp, q, x, wt, b, nodes = _fused(w, 96)
    rows = [range(w.T)] * w.n_nodes
    _check_fused(w, step, q, _fused_reference(w, x, wt, b, rows), rows, nodes)
    step.close()


def test_fused_projection_rope_wan_geometry_sampled(oracle_mod):
    w = I.WORKLOADS["prog4"]                    # 4 nodes x 4680 rows, 1536 -> 3 x 12 x 128
    step, inp, q, x, wt, b, nodes = _fused(w, 1536)
    rng = np.random.default_rng(22)
    rows = [sorted(set(rng.choice(w.T, 60, replace=False).tolist()) | {0, 127, 128, 1559, 1560, w.T - 1})
            for _ in range(w.n_nodes)]
    _check_fused(w, step, q, _fused_reference(w, x, wt, b, rows), rows, nodes)
    step.close()


def test_fused_projection_rope_clean1_split_tail_sampled(oracle_mod):
    # one node of 4680 rows: the partial last round of 256-row tiles is split
    # into half-width items of one head each; the last tile holds 72 rows
    w = I.WORKLOADS["clean1"]
    step, inp, q, x, wt, b, nodes = _fused(w, 1536)
    rng = np.random.default_rng(24)
    rows = [sorted(set(rng.choice(w.T, 120, replace=False).tolist()) |
                   {0, 255, 256, 4607, 4608, w.T - 1})]
    _check_fused(w, step, q, _fused_reference(w, x, wt, b, rows), rows, nodes)
    step.close()


def test_fused_projection_rope_14b_geometry_sampled(oracle_mod):
    # 8 nodes x 4680 rows, 5120 -> 3 x 40 x 128; chunks of 32 rows that
    # straddle two nodes go row by row
    w = I.WORKLOADS["stress14b"]
    step, inp, q, x, wt, b, nodes = _fused(w, 5120)
    rng = np.random.default_rng(26)
    rows = [sorted(set(rng.choice(w.T, 16, replace=False).tolist()) | {0, 4671, w.T - 1})
            for _ in range(w.n_nodes)]
    _check_fused(w, step, q, _fused_reference(w, x, wt, b, rows), rows, nodes)
    step.close()


def test_fused_projection_rope_feeds_attention(oracle_mod):
    """x -> sva_qkv_project_rope -> sva_attend_nodes against the oracle chain
    (projection rounded to bf16, then node_forward's RoPE): the fused path
    skips that intermediate rounding, which the attention tolerance covers."""
    w = I.WORKLOADS["tiny"]
    C = 128
    step, inp, q, x, wt, b, nodes = _fused(w, C)
    out, lse = step.outputs()
    step.attend(nodes, q, out, lse)
    assert step.cache.poll() == 0
    rq, rk, rv = oracle.qkv_project(x.double().numpy().reshape(-1, C), wt.double().numpy(),
                                    b.double().numpy(), heads=w.H)
    shape = (w.n_nodes, w.T, w.H, w.d)
    rq, rk, rv = (torch.from_numpy(oracle.bf16(t).reshape(shape)) for t in (rq, rk, rv))
    inp2 = I.Inputs(inp.history, rq, rk, rv)
    states = P.oracle_states(w, inp2)
    got = out.float().cpu().numpy()
    for i in range(w.n_nodes):
        ref, _ = P.oracle_node(w, inp2, states, i, range(w.H), range(w.T))
        for h in range(w.H):
            P.assert_close(got[i, :, h, :], ref[h], f"fused chain node {i} head {h}")
    step.close()


def test_fused_projection_rope_argument_errors(sva_mod):
    w = I.WORKLOADS["tiny"]
    step = Step(w)
    step.prefill(I.generate(w))
    nodes, n = step.node_table()
    dev = torch.device("cuda")
    x = torch.zeros((n, w.T, 128), dtype=torch.bfloat16, device=dev)
    wt = torch.zeros((3 * w.H * w.d, 128), dtype=torch.bfloat16, device=dev)
    q = torch.empty((n, w.T, w.H, w.d), dtype=torch.bfloat16, device=dev)
    lib = sva_mod.load()
    p = lambda t: __import__("ctypes").c_void_p(t.data_ptr())
    dup = sva_mod.make_nodes([dict(seq=nodes[0].seq, chunk=nodes[0].chunk, level=nodes[0].level,
                                   own_slot=nodes[0].own_slot, ctx=[])] * 2)
    assert lib.sva_qkv_project_rope(step.cache.handle, dup, 2, p(x), 128, p(wt), None, p(q),
                                    None) == sva_mod.ERR_INVALID_ARGUMENT   # the same own slot twice
    assert lib.sva_qkv_project_rope(step.cache.handle, nodes, n, p(x), 100, p(wt), None, p(q),
                                    None) == sva_mod.ERR_INVALID_ARGUMENT   # in_features % 8
    assert lib.sva_qkv_project_rope(step.cache.handle, nodes, 0, p(x), 128, p(wt), None, p(q),
                                    None) == sva_mod.ERR_INVALID_ARGUMENT   # no node
    step.close()
