"""GPU parity for the frame-causal mask inside the own chunk (Eq. 4 at token
level): queries of latent frame f see the own chunk's keys of frames <= f and
every history key."""
import numpy as np
import pytest
import torch

from paper_2609_22283_gb300 import inputs as I
from tests import _parity as P

pytestmark = pytest.mark.gpu

# One node, one head, T = 1024 in four frames of 256 tokens, one history
# chunk: 4 work units of 16 key tiles, split 4 ways, so a key range starts
# inside the own chunk past the frames of the first rows (which then see no
# key in that range).
SPLITFC = I.Workload(name="splitfc", seed=12, F=4, Hp=16, Wp=16, H=1, d=128, K=2, W=1,
                     policy="prog", nodes=((0, 2, 1),), prefilled=((0, 1, 0),),
                     within="frame_causal", description="split + frame-causal edge case")


def _all_rows(oracle_mod, w):
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)
    states = P.oracle_states(w, inp)
    got = out.float().cpu().numpy()
    for i in range(w.n_nodes):
        ref, ref_lse = P.oracle_node(w, inp, states, i, range(w.H), range(w.T))
        for h in range(w.H):
            P.assert_close(got[i, :, h, :], ref[h], f"{w.name} node {i} head {h}")
            np.testing.assert_allclose(lse[i, h].cpu().numpy(), ref_lse[h], atol=2e-3, rtol=0)
    step.close()


# T = 1000 in 10 frames of 100 tokens, one history chunk: 4 work units of 16
# key tiles split 4 ways.  The range of own tiles 4-7 (keys 512..1023) holds
# no visible key for rows 400..499 but some for rows 500..511, which share a
# warp with rows 496..499: rows whose max is still -inf in a warp where others
# rescale (the softmax must not form -inf - -inf).
SPLITFC_WARP = I.Workload(name="splitfcwarp", seed=18, F=10, Hp=10, Wp=10, H=1, d=128, K=2, W=1,
                          policy="prog", nodes=((0, 2, 1),), prefilled=((0, 1, 0),),
                          within="frame_causal", description="masked and visible rows in one warp")


# The first chunk of a video: no history, T = 1024 in four frames of 256
# tokens, two heads.  The first unit walks only the own chunk's tiles 0-1.
FC_FIRST = I.Workload(name="fcfirst", seed=19, F=4, Hp=16, Wp=16, H=2, d=128, K=2, W=2,
                      policy="prog", nodes=((0, 1, 1),), prefilled=(),
                      within="frame_causal", description="frame-causal node without history")


def test_frame_causal_node_without_history(oracle_mod):
    _all_rows(oracle_mod, FC_FIRST)


def test_tiny_frame_causal_all_rows(oracle_mod):
    _all_rows(oracle_mod, I.WORKLOADS["tinyfc"])


def test_split_range_inside_own_chunk(oracle_mod):
    _all_rows(oracle_mod, SPLITFC)


def test_fully_masked_and_visible_rows_in_one_warp(oracle_mod):
    _all_rows(oracle_mod, SPLITFC_WARP)


def test_prog4_frame_causal_sampled(oracle_mod):
    w = I.WORKLOADS["prog4fc"]
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)
    states = P.oracle_states(w, inp)
    ft = w.Hp * w.Wp
    rows = sorted(set(I.sample_rows(w, 24, seed=13)) | {ft - 1, ft, 2 * ft - 1, 2 * ft, 1535, 1536})
    heads = [0, w.H - 1]
    got = out[:, rows].float().cpu().numpy()
    for i in range(w.n_nodes):
        ref, _ = P.oracle_node(w, inp, states, i, heads, rows)
        for hi, h in enumerate(heads):
            P.assert_close(got[i, :, h, :], ref[hi], f"prog4fc node {i} head {h}")
    step.close()


def test_unknown_within_mode_is_rejected(sva_mod):
    w = I.WORKLOADS["tiny"]
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)
    nodes, _ = step.node_table()
    nodes[0].within = 7
    with pytest.raises(sva_mod.SvaError) as e:
        step.cache.attend_nodes(nodes, q, out, None, 0.125, check=False)
    assert e.value.status == sva_mod.ERR_INVALID_ARGUMENT
    step.close()
