"""GPU parity at the edges of the sizes the library takes: a chunk of one
token, ragged chunks one row past a tile, a first-chunk node with no context,
a single head with an odd query-tile count, the maximum number of nodes in a
launch (SVA_MAX_NODES = 64, one per video stream) and the maximum number of
context states per node (SVA_MAX_CTX = 16).  Every output row is compared."""
import numpy as np
import pytest

from paper_2609_22283_gb300 import inputs as I
from tests import _parity as P

pytestmark = pytest.mark.gpu

EDGES = {
    # T = 1: one query and one key per state; node (1, 1) is a first chunk (no context)
    "t1": I.Workload(name="t1", seed=31, F=1, Hp=1, Wp=1, H=2, d=64, K=2, W=2, policy="prog",
                     nodes=((0, 2, 1), (0, 1, 1)), prefilled=((0, 1, 0),),
                     description="one-token chunks"),
    # T = 129 (two tiles, the second of one row), one head, d = 128, odd query-tile count
    "t129": I.Workload(name="t129", seed=32, F=1, Hp=3, Wp=43, H=1, d=128, K=2, W=2, policy="prog",
                       nodes=((0, 3, 2), (0, 2, 1)), prefilled=((0, 1, 0),),
                       description="129-token chunks"),
    # T = 381 (3 tiles, the last of 125 rows) in 3 latent frames of 127 tokens
    # (frame boundaries inside tiles), frame-causal
    "t381fc": I.Workload(name="t381fc", seed=33, F=3, Hp=1, Wp=127, H=2, d=64, K=2, W=1,
                         policy="clean", nodes=((0, 3, 2),), prefilled=((0, 2, 0),),
                         within="frame_causal", description="381-token chunks"),
    # 64 nodes in one launch: 64 video streams, one node each
    "maxnodes": I.Workload(name="maxnodes", seed=34, F=1, Hp=4, Wp=16, H=1, d=64, K=1, W=1,
                           policy="clean", nodes=tuple((s, 2, 1) for s in range(64)),
                           prefilled=tuple((s, 1, 0) for s in range(64)),
                           description="64 nodes of 64 streams"),
    # 16 context states: chunk 17 under clean history with a 16-chunk window
    "maxctx": I.Workload(name="maxctx", seed=35, F=1, Hp=4, Wp=16, H=2, d=64, K=1, W=16,
                         policy="clean", nodes=((0, 17, 1),),
                         prefilled=tuple((0, c, 0) for c in range(1, 17)),
                         description="16 context states"),
}


@pytest.mark.parametrize("name", sorted(EDGES))
def test_edges_all_rows(oracle_mod, name):
    w = EDGES[name]
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)
    states = P.oracle_states(w, inp)
    got = out.float().cpu().numpy()
    for i in range(w.n_nodes):
        ref, ref_lse = P.oracle_node(w, inp, states, i, range(w.H), range(w.T))
        for h in range(w.H):
            P.assert_close(got[i, :, h, :], ref[h], f"{name} node {i} head {h}")
            np.testing.assert_allclose(lse[i, h].cpu().numpy(), ref_lse[h], atol=2e-3, rtol=0)
    step.close()
