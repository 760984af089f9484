"""Key-range splits with the on-device merge: the split computation agrees
with the oracle and with the unsplit computation, and the arrival counters
are left at zero for the next launch."""
import numpy as np
import pytest
import torch

from paper_2609_22283_gb300 import inputs as I
from tests import _parity as P

pytestmark = pytest.mark.gpu

# 1 node, 2 heads, T = 240 (ragged query and key tiles), clean history of 7
# chunks: 2 work units of 16 key tiles each, so the library splits them 4 ways.
SPLIT4 = I.Workload(name="split4", seed=9, F=1, Hp=8, Wp=30, H=2, d=128, K=4, W=7,
                    policy="clean", nodes=((0, 9, 4),),
                    prefilled=tuple((0, c, 0) for c in range(2, 9)),
                    description="split test: 1 node, 2 x 128 heads, T=240, 7 clean chunks")


def _run(w, inp, workspace):
    from paper_2609_22283_gb300.pipeline import Step
    step = Step(w, workspace=workspace)
    step.prefill(inp)
    q, k, v = step.device_inputs(inp)
    out, lse = step.outputs()
    step.run(q, k, v, out, lse)
    assert step.cache.poll() == 0
    torch.cuda.synchronize()
    return step, q, out, lse


def test_four_way_split_matches_oracle(oracle_mod):
    w = SPLIT4
    inp = I.generate(w)
    step, q, out, lse = _run(w, inp, workspace=True)
    states = P.oracle_states(w, inp)
    ref, ref_lse = P.oracle_node(w, inp, states, 0, range(w.H), range(w.T))
    got = out[0].float().cpu().numpy()
    for h in range(w.H):
        P.assert_close(got[:, h, :], ref[h], f"split4 head {h}")
        np.testing.assert_allclose(lse[0, h].cpu().numpy(), ref_lse[h], atol=2e-3, rtol=0)
    # counters were reset: a second launch on the same workspace agrees bitwise
    nodes, _ = step.node_table()
    again = torch.empty_like(out)
    step.cache.attend_nodes(nodes, q, again, None, step.scale, check=False)
    assert step.cache.poll() == 0
    assert torch.equal(again.view(torch.int16), out.view(torch.int16))
    ws = step.cache.ws
    assert torch.count_nonzero(ws[: 4 * 4 * 160].view(torch.int32)).item() == 0
    step.close()


@pytest.mark.parametrize("name", ["clean1", "split4"])
def test_split_agrees_with_unsplit(name):
    w = SPLIT4 if name == "split4" else I.WORKLOADS[name]
    inp = I.generate(w)
    s1, _, o_split, l_split = _run(w, inp, workspace=True)
    s2, _, o_plain, l_plain = _run(w, inp, workspace=False)
    a = o_split.float()
    b = o_plain.float()
    diff = (a - b).abs()
    assert diff.max().item() <= 2e-2 * max(1.0, b.abs().max().item())
    assert (torch.linalg.norm(a - b) / torch.linalg.norm(b)).item() <= 5e-3
    assert (l_split - l_plain).abs().max().item() <= 2e-3
    s1.close()
    s2.close()
