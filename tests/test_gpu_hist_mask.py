"""GPU parity of the token-level mask on the history states
(sva_attend_nodes_masked's hist_mask: Eq. 4's M on the context keys), alone
and with the own-chunk token mask, a block-sparse tile mask, frame
causality and key-range splits, against the fp64 oracle given the same
masks."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_22283_gb300 import inputs as I
from paper_2609_22283_gb300 import sva
from tests import _parity as P

pytestmark = pytest.mark.gpu

# T = 1024 in 4 frames, 2 history chunks, one head: 4 work units split 4 ways
SPLITS = I.Workload(name="splitshist", seed=17, F=4, Hp=16, Wp=16, H=1, d=128, K=2, W=2,
                    policy="prog", nodes=((0, 3, 1),), prefilled=((0, 1, 0), (0, 2, 0)),
                    sparse=0.5, within="frame_causal",
                    description="split + frame causality + history token mask")


def _run(w, hist, own=None, tile=None):
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)     # the step itself runs unmasked (or block-sparse)
    nodes, _ = step.node_table()
    dev = q.device
    step.cache.attend_nodes_masked(nodes, q, out, lse, step.scale,
                                   tile_mask=None if tile is None else tile.to(dev),
                                   own_mask=None if own is None else own.to(dev),
                                   hist_mask=hist.to(dev))
    assert step.cache.poll() == 0
    torch.cuda.synchronize()
    return inp, step, q, out, lse


def _hist_bool(w, hist, i, rows):
    """Node i's history bits as booleans [W][len(rows)-indexable by row][T]:
    an array indexed [j][u][v] for the rows asked for (others False)."""
    bits = I.unpack_bits(hist[i, rows], w.T).numpy()          # [len(rows)][W][T]
    full = np.zeros((w.W, w.T, w.T), dtype=bool)
    full[:, rows, :] = np.moveaxis(bits, 1, 0)
    return full


def _check(w, inp, out, lse, hist, own=None, tile=None, rows=None, heads=None):
    states = P.oracle_states(w, inp)
    own_b = None if own is None else I.unpack_bits(own, w.T).numpy()
    tile_b = None if tile is None else P.oracle_masks(w, tile)
    rows = list(range(w.T)) if rows is None else rows
    heads = list(range(w.H)) if heads is None else heads
    got = out[:, rows].float().cpu().numpy()
    stats = P.Stats()
    for i in range(w.n_nodes):
        ref, ref_lse = P.oracle_node(w, inp, states, i, heads, rows,
                                     tile_mask=None if tile_b is None else tile_b[i],
                                     own_mask=None if own_b is None else own_b[i],
                                     hist_mask=_hist_bool(w, hist, i, rows))
        for hi, h in enumerate(heads):
            P.assert_close(got[i, :, h, :], ref[hi], f"{w.name} node {i} head {h}", stats=stats)
            l = lse[i, h].cpu().numpy()[rows]
            fin = np.isfinite(ref_lse[hi])
            P.assert_lse(l[fin], ref_lse[hi][fin], f"{w.name} node {i} head {h}", stats)
            assert np.all(l[~fin] == -np.inf)
    print(f"\n{w.name} with a history token mask: {stats}")


def test_tiny_hist_mask_all_rows(oracle_mod):
    w = I.WORKLOADS["tinys"]                 # 3 key tiles per state, the last of 64 keys
    hist = I.hist_mask(w, 0.5)
    inp, step, q, out, lse = _run(w, hist)
    _check(w, inp, out, lse, hist)
    step.close()


def test_tiny_hist_with_own_and_tile_masks(oracle_mod):
    w = I.WORKLOADS["tinys"]
    hist = I.hist_mask(w, 0.4, seed=5)
    own = I.own_mask(w, 0.5)
    tile = I.tile_mask(w)
    inp, step, q, out, lse = _run(w, hist, own=own, tile=tile)
    _check(w, inp, out, lse, hist, own=own, tile=tile)
    step.close()


def test_split_frame_causal_hist_mask(oracle_mod):
    w = SPLITS
    hist = I.hist_mask(w, 0.5)
    inp, step, q, out, lse = _run(w, hist, tile=I.tile_mask(w))
    _check(w, inp, out, lse, hist, tile=I.tile_mask(w))
    step.close()


def test_prog4_hist_mask_sampled(oracle_mod):
    w = I.WORKLOADS["prog4"]                 # 4 nodes x 6 contexts x 4680 x 4680 bits
    hist = I.hist_mask(w, 0.7)
    inp, step, q, out, lse = _run(w, hist)
    rows = sorted(set(I.sample_rows(w, 12, seed=19)) | {7})
    _check(w, inp, out, lse, hist, rows=rows, heads=[0, w.H - 1])
    step.close()


def test_all_ones_hist_mask_is_the_dense_launch():
    w = I.WORKLOADS["prog4"]
    inp = I.generate(w)
    step, q, out, _ = P.gpu_step(w, inp, lse=False)
    nodes, _ = step.node_table()
    words = -(-w.T // 32)
    ones = torch.full((w.n_nodes, w.T, w.W, words), -1, dtype=torch.int32, device=q.device)
    masked = torch.empty_like(out)
    step.cache.attend_nodes_masked(nodes, q, masked, None, step.scale, hist_mask=ones)
    assert step.cache.poll() == 0
    torch.cuda.synchronize()
    assert torch.equal(masked.view(torch.int16), out.view(torch.int16))
    step.close()


def test_hist_mask_argument_errors(sva_mod):
    w = I.WORKLOADS["tinys"]
    inp = I.generate(w)
    step, q, out, _ = P.gpu_step(w, inp, lse=False)
    nodes, n = step.node_table()
    lib = sva_mod.load()
    words = -(-w.T // 32)
    hist = torch.zeros((n, w.T, w.W, words), dtype=torch.int32, device=q.device)

    def call(ptr, states, wds):
        m = sva.sva_attn_mask(None, 0, None, 0, ctypes.c_void_p(ptr), states, wds)
        return lib.sva_attend_nodes_masked(step.cache.handle, nodes, n, ctypes.c_void_p(q.data_ptr()),
                                           ctypes.c_void_p(out.data_ptr()), None, step.scale,
                                           ctypes.byref(m), None)
    assert call(hist.data_ptr(), w.W, words - 1) == sva.ERR_INVALID_ARGUMENT      # short row
    assert call(hist.data_ptr(), 0, words) == sva.ERR_INVALID_ARGUMENT            # no state
    assert call(hist.data_ptr() + 2, w.W, words) == sva.ERR_INVALID_ARGUMENT      # misaligned
    n_ctx = max(nodes[i].n_ctx for i in range(n))
    assert n_ctx == 2
    assert call(hist.data_ptr(), 1, words) == sva.ERR_INVALID_ARGUMENT            # fewer states than contexts
    assert call(hist.data_ptr(), w.W, words) == sva.OK
    assert step.cache.poll() == 0
    step.close()
