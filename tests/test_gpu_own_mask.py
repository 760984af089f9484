"""GPU parity of the general token-level mask inside the own chunk
(sva_attend_nodes_masked's own_mask, Eq. 4's M at token level), alone and
with a block-sparse tile mask and frame causality, against the fp64 oracle
given the same masks."""
import numpy as np
import pytest
import torch

from paper_2609_22283_gb300 import inputs as I
from paper_2609_22283_gb300 import sva
from tests import _parity as P

pytestmark = pytest.mark.gpu

# T = 1024 in 4 frames, 2 history chunks, one head: 4 work units split 4 ways
SPLITS = I.Workload(name="splitsown", seed=16, F=4, Hp=16, Wp=16, H=1, d=128, K=2, W=2,
                    policy="prog", nodes=((0, 3, 1),), prefilled=((0, 1, 0), (0, 2, 0)),
                    sparse=0.5, description="split + own-chunk token mask")


def _run(w, own, tile=None):
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)     # the step itself runs unmasked (or block-sparse)
    nodes, _ = step.node_table()
    dev = q.device
    step.cache.attend_nodes_masked(nodes, q, out, lse, step.scale,
                                   tile_mask=None if tile is None else tile.to(dev),
                                   own_mask=own.to(dev))
    assert step.cache.poll() == 0
    torch.cuda.synchronize()
    return inp, step, q, out, lse


def _check(w, inp, out, lse, own, tile, rows=None, heads=None):
    states = P.oracle_states(w, inp)
    own_b = I.unpack_bits(own, w.T).numpy()
    tile_b = None if tile is None else P.oracle_masks(w, tile)
    rows = list(range(w.T)) if rows is None else rows
    heads = list(range(w.H)) if heads is None else heads
    got = out[:, rows].float().cpu().numpy()
    for i in range(w.n_nodes):
        ref, ref_lse = P.oracle_node(w, inp, states, i, heads, rows,
                                     tile_mask=None if tile_b is None else tile_b[i], own_mask=own_b[i])
        for hi, h in enumerate(heads):
            P.assert_close(got[i, :, h, :], ref[hi], f"{w.name} node {i} head {h}")
            l = lse[i, h].cpu().numpy()[rows]
            fin = np.isfinite(ref_lse[hi])
            np.testing.assert_allclose(l[fin], ref_lse[hi][fin], atol=2e-3, rtol=0)
            assert np.all(l[~fin] == -np.inf)


def test_tiny_own_mask_all_rows(oracle_mod):
    w = I.WORKLOADS["tinys"]
    own = I.own_mask(w, 0.3)
    keep = I.unpack_bits(own, w.T)
    keep[0, 5, :] = False                        # a row with no own key (history only)
    own = I.pack_bits(keep, own.shape[2])
    inp, step, q, out, lse = _run(w, own)
    _check(w, inp, out, lse, own, None)
    step.close()


def test_own_and_tile_mask_split_frame_causal(oracle_mod):
    w = I.Workload(**{**SPLITS.__dict__, "within": "frame_causal"})
    own = I.own_mask(w, 0.5)
    tile = I.tile_mask(w)
    keep = I.unpack_bits(tile, (1 + w.W) * w.tiles)
    keep[0, 6, 8:] = False                       # query tile 6: own chunk only ...
    keep[0, 6, 3] = False                        # ... minus one own tile
    tile = I.pack_bits(keep, w.mask_words)
    inp, step, q, out, lse = _run(w, own, tile)
    _check(w, inp, out, lse, own, tile)
    step.close()


def test_frame_causal_as_own_mask_is_the_frame_causal_launch(oracle_mod):
    w = I.WORKLOADS["prog4fc"]
    ft = w.Hp * w.Wp
    u = torch.arange(w.T)
    fc = (u[None, :] // ft) <= (u[:, None] // ft)
    own = I.pack_bits(fc.unsqueeze(0).expand(w.n_nodes, w.T, w.T).contiguous(), -(-w.T // 32))
    inp = I.generate(w)
    step, q, out_fc, _ = P.gpu_step(w, inp, lse=False)
    nodes, _ = step.node_table()
    for n in nodes:
        n.within = sva.WITHIN["bidirectional"]
    out = torch.empty_like(out_fc)
    step.cache.attend_nodes_masked(nodes, q, out, None, step.scale, own_mask=own.to(q.device))
    assert step.cache.poll() == 0
    torch.cuda.synchronize()
    assert torch.equal(out, out_fc)
    step.close()


def test_prog4_own_mask_sampled(oracle_mod):
    w = I.WORKLOADS["prog4"]
    own = I.own_mask(w, 0.5)
    inp, step, q, out, lse = _run(w, own)
    rows = sorted(set(I.sample_rows(w, 12, seed=17)) | {5, 4679})
    _check(w, inp, out, lse, own, None, rows=rows, heads=[0, w.H - 1])
    step.close()


def test_own_mask_argument_errors(sva_mod):
    w = I.WORKLOADS["tinys"]
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)
    nodes, _ = step.node_table()
    short = torch.zeros((w.n_nodes, w.T, 2), dtype=torch.int32, device=q.device)   # needs 10 words
    with pytest.raises(sva_mod.SvaError) as e:
        step.cache.attend_nodes_masked(nodes, q, out, None, step.scale, own_mask=short)
    assert e.value.status == sva_mod.ERR_INVALID_ARGUMENT
    step.close()
