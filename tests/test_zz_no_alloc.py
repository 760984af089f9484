"""sva_attend_nodes_noalloc, the attention entry point for callers that may
not allocate device memory (for example a plugin whose host framework gives
it only its input and output buffers): the library takes the key-range split
scratch from its own static device array instead of a caller workspace.

Through the C ABI, on two calls in a row, its output must match what
sva_attend_nodes computes on the same inputs, within the tolerances of the
other parity tests; a launch whose split plan needs more scratch than the
array holds must be refused without launching anything.  This file runs
last so that a failure here cannot hide the results of the other tests, and
it depends on no state they leave behind."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_22283_gb300 import inputs as I
from paper_2609_22283_gb300 import sva
from paper_2609_22283_gb300.pipeline import Step

pytestmark = pytest.mark.gpu

MAX_ABS = 2e-2   # element bound, scaled by max(1, |O|) as in the parity tests
REL_RMS = 5e-3

# 1 node, 2 heads x 128, T = 240, clean history of 7 chunks: 2 work units of
# 16 key tiles, which the split plan divides 4 ways (about 1 MB of scratch).
SPLIT4 = I.Workload(name="split4", seed=9, F=1, Hp=8, Wp=30, H=2, d=128, K=4, W=7,
                    policy="clean", nodes=((0, 9, 4),),
                    prefilled=tuple((0, c, 0) for c in range(2, 9)))


def _noalloc(step, nodes, q, out, lse):
    lib = sva.load()
    return lib.sva_attend_nodes_noalloc(
        step.cache.handle, nodes, len(nodes), ctypes.c_void_p(q.data_ptr()),
        ctypes.c_void_p(out.data_ptr()), ctypes.c_void_p(lse.data_ptr() if lse is not None else 0),
        step.scale, ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


@pytest.mark.parametrize("name", ["split4", "tiny"])
def test_noalloc_matches_attend_nodes_twice(name):
    w = SPLIT4 if name == "split4" else I.WORKLOADS[name]
    inp = I.generate(w)
    step = Step(w, workspace=True)
    step.prefill(inp)
    q, k, v = step.device_inputs(inp)
    ref, ref_lse = step.outputs()
    step.run(q, k, v, ref, ref_lse)                 # sva_attend_nodes, caller workspace
    assert step.cache.poll() == sva.OK
    nodes, _ = step.node_table()
    b = ref.float()
    for call in range(2):
        out = torch.full_like(ref, float("nan"))
        lse = torch.full_like(ref_lse, float("nan"))
        assert _noalloc(step, nodes, q, out, lse) == sva.OK, sva.last_error()
        assert step.cache.poll() == sva.OK
        a = out.float()
        assert torch.isfinite(a).all(), f"call {call}: unwritten output"
        scaled = ((a - b).abs() / b.abs().clamp(min=1.0)).max().item()
        rel = (torch.linalg.norm(a - b) / torch.linalg.norm(b)).item()
        assert scaled <= MAX_ABS and rel <= REL_RMS, (call, scaled, rel)
        np.testing.assert_allclose(lse.cpu().numpy(), ref_lse.cpu().numpy(), atol=2e-3, rtol=0)
    step.close()


def test_noalloc_refuses_plan_beyond_its_scratch():
    w = I.WORKLOADS["clean1"]            # 228 units split 2 ways: about 61 MB of scratch
    inp = I.generate(w)
    step = Step(w, workspace=False)
    step.prefill(inp)
    q, k, v = step.device_inputs(inp)
    nodes, _ = step.node_table()
    step.cache.rope_kv_write(nodes, k, v, q, check=False)
    out = torch.full((w.n_nodes, w.T, w.H, w.d), 7.0, dtype=torch.bfloat16, device="cuda")
    assert _noalloc(step, nodes, q, out, None) == sva.ERR_CAPACITY
    assert "scratch" in sva.last_error()
    torch.cuda.synchronize()
    assert bool((out == 7.0).all())                # nothing was launched
    assert step.cache.poll() == sva.OK
    step.close()
