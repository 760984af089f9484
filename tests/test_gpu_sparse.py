"""GPU parity of query-dependent block-sparse access (Eq. 4's mask at 128 x
128-token tiles, sva_attend_nodes_sparse) against the fp64 oracle given the
same key-tile mask."""
import numpy as np
import pytest
import torch

from paper_2609_22283_gb300 import inputs as I
from tests import _parity as P

pytestmark = pytest.mark.gpu

# One node, one head, T = 1024 (8 tiles), two history chunks: 24 key tiles
# over 4 work units, split 4 ways, so split ranges of a sparse mask can be
# short or empty.
SPLITS = I.Workload(name="splits", seed=14, F=4, Hp=16, Wp=16, H=1, d=128, K=2, W=2,
                    policy="prog", nodes=((0, 3, 1),), prefilled=((0, 1, 0), (0, 2, 0)),
                    sparse=0.4, description="split + block-sparse edge cases")


def _run(w, mask=None, lse=True):
    inp = I.generate(w)
    step, q, out, l = P.gpu_step(w, inp, lse=lse)
    if mask is not None:                     # rerun step 4 with another mask
        nodes, _ = step.node_table()
        step.cache.attend_nodes_sparse(nodes, q, out, mask.to(q.device), l, step.scale)
        assert step.cache.poll() == 0
        torch.cuda.synchronize()
    return inp, step, q, out, l


def _check_all_rows(w, inp, out, lse, masks, within_tol=True):
    states = P.oracle_states(w, inp)
    got = out.float().cpu().numpy()
    for i in range(w.n_nodes):
        ref, ref_lse = P.oracle_node(w, inp, states, i, range(w.H), range(w.T), tile_mask=masks[i])
        for h in range(w.H):
            P.assert_close(got[i, :, h, :], ref[h], f"{w.name} node {i} head {h}")
            fin = np.isfinite(ref_lse[h])
            np.testing.assert_allclose(lse[i, h].cpu().numpy()[fin], ref_lse[h][fin], atol=2e-3, rtol=0)
            assert np.all(lse[i, h].cpu().numpy()[~fin] == -np.inf)


def test_tiny_sparse_all_rows(oracle_mod):
    w = I.WORKLOADS["tinys"]
    inp, step, q, out, lse = _run(w)
    _check_all_rows(w, inp, out, lse, P.oracle_masks(w))
    step.close()


def test_split_ranges_with_empty_tiles(oracle_mod):
    w = SPLITS
    keep = I.unpack_bits(I.tile_mask(w), (1 + w.W) * w.tiles)
    keep[0, 2, :] = False          # query tile 2 sees nothing: O = 0, LSE = -inf
    keep[0, 6, :] = False          # query tiles 6 and 7 (one work unit) see nothing:
    keep[0, 7, :] = False          # every split of that unit has an empty range
    keep[0, 4, 8:] = False         # query tile 4 sees its own chunk only
    mask = I.pack_bits(keep, w.mask_words)
    inp, step, q, out, lse = _run(w, mask)
    assert step.cache.workspace_bytes() > 0
    _check_all_rows(w, inp, out, lse, P.oracle_masks(w, mask))
    assert torch.all(out[0, 256:384] == 0) and torch.all(out[0, 768:] == 0)
    step.close()


def test_sparse_with_frame_causality(oracle_mod):
    w = I.Workload(**{**SPLITS.__dict__, "name": "splitsfc", "within": "frame_causal"})
    inp, step, q, out, lse = _run(w)
    _check_all_rows(w, inp, out, lse, P.oracle_masks(w))
    step.close()


def test_all_ones_mask_is_the_dense_launch(oracle_mod):
    w = I.Workload(**{**I.WORKLOADS["prog4"].__dict__, "name": "prog4ones", "sparse": 1.0})
    inp, step, q, out, lse = _run(w)
    dense = torch.empty_like(out)
    nodes, _ = step.node_table()
    step.cache.attend_nodes(nodes, q, dense, None, step.scale)
    torch.cuda.synchronize()
    assert torch.equal(out, dense)
    step.close()


def test_prog4_sparse_sampled(oracle_mod):
    w = I.WORKLOADS["prog4s"]
    inp, step, q, out, lse = _run(w)
    states = P.oracle_states(w, inp)
    masks = P.oracle_masks(w)
    rows = I.sample_rows(w, 24, seed=15)
    heads = [0, w.H - 1]
    got = out[:, rows].float().cpu().numpy()
    for i in range(w.n_nodes):
        ref, _ = P.oracle_node(w, inp, states, i, heads, rows, tile_mask=masks[i])
        for hi, h in enumerate(heads):
            P.assert_close(got[i, :, h, :], ref[hi], f"prog4s node {i} head {h}")
    step.close()


def test_sparse_argument_errors(sva_mod):
    w = I.WORKLOADS["tinys"]
    inp, step, q, out, lse = _run(w)
    nodes, _ = step.node_table()
    lib = sva_mod.load()
    import ctypes
    st = lib.sva_attend_nodes_sparse(step.cache.handle, nodes, len(nodes), ctypes.c_void_p(q.data_ptr()),
                                     ctypes.c_void_p(out.data_ptr()), None, 0.125, None, 1,
                                     ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == sva_mod.ERR_INVALID_ARGUMENT
    short = torch.zeros((w.n_nodes, w.tiles, 1), dtype=torch.int32, device=q.device)
    # rows of 0 words cannot hold the node's key tiles
    st = lib.sva_attend_nodes_sparse(step.cache.handle, nodes, len(nodes), ctypes.c_void_p(q.data_ptr()),
                                     ctypes.c_void_p(out.data_ptr()), None, 0.125,
                                     ctypes.c_void_p(short.data_ptr()), 0,
                                     ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == sva_mod.ERR_INVALID_ARGUMENT
    step.close()
