"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on
the same seeded inputs.  Attention within max-abs 2e-2 and relative RMS
5e-3; cache indexing and the V scatter bit-exact; rotated K and Q within one
bf16 ulp of the oracle's correctly rounded values."""
import math

import numpy as np
import pytest
import torch

from paper_2609_22283_gb300 import inputs as I
from tests import _parity as P

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tiny():
    w = I.WORKLOADS["tiny"]
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)
    return w, inp, step, q, out, lse


def test_tiny_all_rows(oracle_mod, tiny):
    w, inp, step, q, out, lse = tiny
    states = P.oracle_states(w, inp)
    got = out.float().cpu().numpy()
    got_lse = lse.cpu().numpy()
    for i in range(w.n_nodes):
        ref, ref_lse = P.oracle_node(w, inp, states, i, range(w.H), range(w.T))
        for h in range(w.H):
            P.assert_close(got[i, :, h, :], ref[h], f"node {i} head {h}")
            np.testing.assert_allclose(got_lse[i, h], ref_lse[h], atol=2e-3, rtol=0)


def _check_rotated(got, ref, raw, what):
    """Rotated rows against bf16(oracle rotation): within one bf16 ulp of the
    reference plus the error of a rotation in fp32 arithmetic, which is
    relative to the pair's norm (a few fp32 ulps of it; 2^-21 |pair|) rather
    than to the result: where x cos a and y sin a nearly cancel the exact
    value is tiny and its bf16 ulp far below that error.  At least 99.9% of
    the elements must be bit-exact."""
    got = got.astype(np.float64)
    raw = np.asarray(raw, dtype=np.float64)
    pair = np.repeat(np.hypot(raw[:, 0::2], raw[:, 1::2]), 2, axis=1)   # norm of each element's pair
    bound = P.ulp_bf16(ref) + 2.0 ** -21 * pair
    bad = np.abs(got - ref) > bound
    exact = np.mean(got == ref)
    assert not bad.any(), f"{what}: {int(bad.sum())} elements beyond ulp + 2^-21 |pair|"
    assert exact >= 0.999, f"{what}: only {exact:.5f} exact"


# tiny and clean1 take the single-wave instance of the RoPE kernel, prog4
# (18720 tokens) the one for larger launches
@pytest.mark.parametrize("name", ["tiny", "clean1", "prog4"])
def test_cache_indexing_and_rope(oracle_mod, name):
    w = I.WORKLOADS[name]
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp, lse=False)
    pool = step.cache.slot_pool()
    g = P.oracle_geometry(w)
    T = w.T
    heads = range(w.H)
    for (s, c, l), (k_raw, v_raw) in I.all_states(w, inp).items():
        slot = step.cache.lookup(s, c, l)
        # V is scattered unchanged: bit-exact at [slot][1][h][0:T]
        v_cache = pool[slot, 1, :, :T, :].permute(1, 0, 2).contiguous().cpu()
        assert torch.equal(v_cache.view(torch.int16), v_raw.view(torch.int16)), (s, c, l)
        # pad rows stay zero
        assert torch.count_nonzero(pool[slot, :, :, T:, :].float()).item() == 0
        for h in heads:
            kh = k_raw[:, h, :].double().numpy()
            k_ref = oracle_mod.bf16(oracle_mod.rope_head(kh, c, g))
            _check_rotated(pool[slot, 0, h, :T, :].float().cpu().numpy(), k_ref, kh, f"K {(s, c, l)} h{h}")
    for i, (s, b, j) in enumerate(w.nodes):
        for h in heads:
            qh = inp.q[i, :, h, :].double().numpy()
            q_ref = oracle_mod.bf16(oracle_mod.rope_head(qh, b, g))
            _check_rotated(q[i, :, h, :].float().cpu().numpy(), q_ref, qh, f"Q node {i} h{h}")
    step.close()


def _p_abs(w, inp, states, i, h, rows, cache):
    """E_p|V| of node i, head h at the given rows (the oracle over |V|)."""
    def f(idx):
        if "abs" not in cache:
            cache["abs"] = P.abs_v_states(states)
        return P.oracle_node(w, inp, cache["abs"], i, [h], np.asarray(rows)[idx])[0][0]
    return f


@pytest.mark.parametrize("name", ["clean1", "same4"])
def test_full_geometry_all_rows(oracle_mod, name):
    """Every head and every query row of every node against the oracle."""
    w = I.WORKLOADS[name]
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)
    got = out.float().cpu().numpy()                      # [n][T][H][d]
    got_lse = lse.cpu().numpy()
    step.close()
    states = P.oracle_states(w, inp)
    stats, cache = P.Stats(), {}
    rows = list(range(w.T))
    for i in range(w.n_nodes):
        ref, ref_lse = P.oracle_node(w, inp, states, i, range(w.H), rows)
        for h in range(w.H):
            P.assert_close(got[i, :, h, :], ref[h], f"{name} node {i} head {h}",
                           p_abs=_p_abs(w, inp, states, i, h, rows, cache), stats=stats)
            P.assert_lse(got_lse[i, h], ref_lse[h], f"{name} node {i} head {h}", stats)
    print(f"\n{name} (all {w.n_nodes * w.H * w.T} rows): {stats}")


@pytest.mark.parametrize("name", ["prog4", "prog4r", "stress14b"])
def test_full_geometry_sampled(oracle_mod, name):
    """Every head of every node: at least 8192 seeded query rows per node
    spread over its heads (a different draw per head), plus every boundary
    row of every head."""
    w = I.WORKLOADS[name]
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)
    got = out.cpu()                                      # bf16 [n][T][H][d]
    got_lse = lse.cpu().numpy()
    step.close()
    states = P.oracle_states(w, inp)
    stats, cache, n_rows = P.Stats(), {}, 0
    for i in range(w.n_nodes):
        per_head = P.rows_per_head(w, 8192, seed=11 + i)
        for h in range(w.H):
            rows = per_head[h]
            n_rows += len(rows)
            ref, ref_lse = P.oracle_node(w, inp, states, i, [h], rows)
            P.assert_close(got[i, rows, h, :].float().numpy(), ref[0], f"{name} node {i} head {h}",
                           p_abs=_p_abs(w, inp, states, i, h, rows, cache), stats=stats)
            P.assert_lse(got_lse[i, h, rows], ref_lse[0], f"{name} node {i} head {h}", stats)
    assert n_rows >= 8192 * w.n_nodes
    print(f"\n{name} ({n_rows} rows): {stats}")


@pytest.mark.parametrize("name", ["prog4", "stress14b"])
def test_attention_bitwise_repeatable(name):
    """Repeated launches on the same inputs give the same bits (no race in
    the kernel's barriers, stage hand-back or lazy rescale)."""
    w = I.WORKLOADS[name]
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)
    nodes, _ = step.node_table()
    for _ in range(3):
        again = torch.empty_like(out)
        again_lse = torch.empty_like(lse)
        step.cache.attend_nodes(nodes, q, again, again_lse, step.scale, check=False)
        assert step.cache.poll() == 0
        assert torch.equal(again.view(torch.int16), out.view(torch.int16))
        assert torch.equal(again_lse.view(torch.int32), lse.view(torch.int32))
    step.close()


def test_clean5_serial_launches(oracle_mod):
    """The fully serial schedule of a chunk (Eq. 5) as the schedule comparison
    times it: each of the five nodes of chunk 20 (four updates, then the clean
    refresh) is its own RoPE + cache write and attention launch."""
    from paper_2609_22283_gb300 import sva
    from paper_2609_22283_gb300.pipeline import Step
    w = I.WORKLOADS["clean5"]
    inp = I.generate(w)
    step = Step(w)
    step.prefill(inp)
    q, k, v = step.device_inputs(inp)
    out, lse = step.outputs()
    nodes, n = step.node_table()
    for i in range(n):
        sl = slice(i, i + 1)
        one = (sva.sva_node * 1)(nodes[i])
        step.cache.rope_kv_write(one, k[sl], v[sl], q[sl], check=False)
        step.cache.attend_nodes(one, q[sl], out[sl], lse[sl], step.scale, check=False)
    assert step.cache.poll() == sva.OK
    got = out.cpu()
    got_lse = lse.cpu().numpy()
    step.close()
    states = P.oracle_states(w, inp)
    stats, cache = P.Stats(), {}
    for i in range(n):
        per_head = P.rows_per_head(w, 8192, seed=31 + i)
        for h in range(w.H):
            rows = per_head[h]
            ref, ref_lse = P.oracle_node(w, inp, states, i, [h], rows)
            P.assert_close(got[i, rows, h, :].float().numpy(), ref[0], f"clean5 node {i} head {h}",
                           p_abs=_p_abs(w, inp, states, i, h, rows, cache), stats=stats)
            P.assert_lse(got_lse[i, h, rows], ref_lse[0], f"clean5 node {i} head {h}", stats)
    print(f"\nclean5 serial: {stats}")


def test_constant_values(tiny):
    """V = 1 everywhere gives O = 1 (weights sum to one)."""
    w, inp, _, _, _, _ = tiny
    inp1 = I.Inputs({k: (a, torch.ones_like(b)) for k, (a, b) in inp.history.items()},
                    inp.q.clone(), inp.k_new.clone(), torch.ones_like(inp.v_new))
    step, q, out, lse = P.gpu_step(w, inp1)
    o = out.float()
    assert torch.max(torch.abs(o - 1.0)).item() <= 2e-3
    step.close()


def test_batched_equals_alone_and_permutation():
    """A node computed alone, or in a permuted batch, gives bitwise the same
    rows (with one key range per unit: a lone node would otherwise be split,
    which changes the summation order; that case has its own tolerance test)."""
    w = I.WORKLOADS["prog4"]
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)
    step.cache.set_workspace(None)
    nodes, n = step.node_table()
    from paper_2609_22283_gb300 import sva
    for i in range(n):
        one = sva.make_nodes([dict(seq=nodes[i].seq, chunk=nodes[i].chunk, level=nodes[i].level,
                                   own_slot=nodes[i].own_slot,
                                   ctx=[nodes[i].ctx_slot[k] for k in range(nodes[i].n_ctx)])])
        o1 = torch.empty_like(out[i:i + 1])
        step.cache.attend_nodes(one, q[i:i + 1].contiguous(), o1)
        torch.cuda.synchronize()
        assert torch.equal(o1[0].view(torch.int16), out[i].view(torch.int16)), i
    perm = list(reversed(range(n)))
    entries = [dict(seq=nodes[i].seq, chunk=nodes[i].chunk, level=nodes[i].level,
                    own_slot=nodes[i].own_slot, ctx=[nodes[i].ctx_slot[k] for k in range(nodes[i].n_ctx)])
               for i in perm]
    qp = q[perm].contiguous()
    op = torch.empty_like(out)
    step.cache.attend_nodes(entries, qp, op)
    torch.cuda.synchronize()
    assert torch.equal(op.view(torch.int16), out[perm].view(torch.int16))
    step.close()


def test_hidden_context_state(oracle_mod, tiny):
    """ctx_visible = 0 masks a selected state with -inf (Eq. 4 at state granularity)."""
    w, inp, step, q, out, lse = tiny
    from paper_2609_22283_gb300 import sva
    nodes, n = step.node_table()
    nd = nodes[0]                                   # (3, 2): ctx (2, 1), (1, 0)
    ctx = [nd.ctx_slot[k] for k in range(nd.n_ctx)]
    one = sva.make_nodes([dict(seq=nd.seq, chunk=nd.chunk, level=nd.level, own_slot=nd.own_slot,
                               ctx=ctx, visible=[0] + [1] * (len(ctx) - 1))])
    o1 = torch.empty_like(out[:1])
    step.cache.attend_nodes(one, q[:1].contiguous(), o1)
    torch.cuda.synchronize()
    states = P.oracle_states(w, inp)
    ref, _ = P.oracle_node(w, inp, states, 0, range(w.H), range(w.T), hidden=frozenset({(2, 1)}))
    got = o1[0].float().cpu().numpy()
    for h in range(w.H):
        P.assert_close(got[:, h, :], ref[h], f"hidden head {h}")
