"""sva_attend_nodes_noalloc, the attention entry point for callers that may
not allocate device memory (for example a plugin whose host framework gives
it only its input and output buffers): the library takes the key-range split
scratch from its own static device array instead of a caller workspace.

Through the C ABI, on two calls in a row, its output must match what
sva_attend_nodes with a workspace computes on the same inputs, within the
tolerances of the other parity tests (and, since both take the same split
plan, bit for bit); on clean1 it is also checked against the oracle.  A
launch whose split plan needs more scratch than the array holds must be
refused without launching anything.  The expected plans are worked out here
from the device's SM count with the planner's rule (full waves unsplit, the
partial last wave split).  This file runs last so that a failure here cannot
hide the results of the other tests, and it depends on no state they leave
behind."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_22283_gb300 import inputs as I
from paper_2609_22283_gb300 import sva
from paper_2609_22283_gb300.pipeline import Step
from tests import _parity as P

pytestmark = pytest.mark.gpu

MAX_ABS = P.MAX_ABS   # element bound 2e-2 + ulp_bf16(|O|) / 2, as in the parity tests
REL_RMS = P.REL_RMS
STATIC_SCRATCH = 32 << 20
MAX_SPLIT = 4

# 1 node, 2 heads x 128, T = 240, clean history of 7 chunks: 2 work units of
# 16 key tiles each, which the split plan divides 4 ways (about 1 MB of scratch).
SPLIT4 = I.Workload(name="split4", seed=9, F=1, Hp=8, Wp=30, H=2, d=128, K=4, W=7,
                    policy="clean", nodes=((0, 9, 4),),
                    prefilled=tuple((0, c, 0) for c in range(2, 9)))


def _plan(units, min_tiles, sms, cap):
    """(n_full, n_split) as the library plans a launch: the number of splits
    minimising waves per split, the full waves unsplit when that is no worse."""
    def choose(u):
        best, best_s = float(-(-u // sms)), 1
        for s in range(2, MAX_SPLIT + 1):
            if u * s > cap or min_tiles // s < 4:
                break
            cost = -(-(u * s) // sms) / s
            if cost < best - 1e-9:
                best, best_s = cost, s
        return best_s
    s_all = choose(units)
    if units < sms:
        return 0, s_all
    full = units // sms * sms
    rest = units - full
    s_rest = choose(rest)
    cost_all = -(-(units * s_all) // sms) / s_all
    cost_mixed = full / sms + -(-(rest * s_rest) // sms) / s_rest
    return (full, s_rest) if cost_mixed <= cost_all + 1e-9 else (0, s_all)


def _scratch(w, sms):
    """(n_split, bytes of static scratch) of a dense launch of workload w."""
    nt = w.tiles
    units = w.H * w.n_nodes * -(-nt // 2)
    min_tiles = min((1 + max(0, min(w.W, b - 1))) * nt for (_, b, _) in w.nodes)
    n_full, n_split = _plan(units, min_tiles, sms, 4 * sms)
    if n_split == 1:
        return 1, 0
    split_units = units - n_full
    return n_split, (-(-split_units * 4 // 256) * 256) + split_units * n_split * 256 * (w.d + 2) * 4


def _sms():
    return torch.cuda.get_device_properties(0).multi_processor_count


def _noalloc(step, nodes, q, out, lse):
    lib = sva.load()
    return lib.sva_attend_nodes_noalloc(
        step.cache.handle, nodes, len(nodes), ctypes.c_void_p(q.data_ptr()),
        ctypes.c_void_p(out.data_ptr()), ctypes.c_void_p(lse.data_ptr() if lse is not None else 0),
        step.scale, ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


@pytest.mark.parametrize("name", ["split4", "tiny", "clean1"])
def test_noalloc_matches_attend_nodes_twice(name):
    w = SPLIT4 if name == "split4" else I.WORKLOADS[name]
    n_split, need = _scratch(w, _sms())
    if name in ("split4", "clean1"):
        assert n_split > 1 and 0 < need <= STATIC_SCRATCH, (n_split, need)   # the split path
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
        bound = MAX_ABS + 0.5 * torch.from_numpy(P.ulp_bf16(b.cpu().numpy())).to(b.device)
        assert bool(((a - b).abs() <= bound).all()), call
        rel = (torch.linalg.norm(a - b) / torch.linalg.norm(b)).item()
        assert rel <= REL_RMS, (call, rel)
        np.testing.assert_allclose(lse.cpu().numpy(), ref_lse.cpu().numpy(), atol=2e-3, rtol=0)
        # the same split plan and kernel: the same bits
        assert torch.equal(out.view(torch.int16), ref.view(torch.int16)), call
    if name == "clean1":
        got = out.cpu()
        states = P.oracle_states(w, inp)
        rows = I.sample_rows(w, 64, seed=17)
        oref, _ = P.oracle_node(w, inp, states, 0, range(w.H), rows)
        for h in range(w.H):
            P.assert_close(got[0, rows, h, :].float().numpy(), oref[h], f"noalloc clean1 head {h}")
    step.close()


def test_noalloc_refuses_plan_beyond_its_scratch():
    # One node of 240 tokens (one work unit per head, 16 key tiles) over 7
    # clean history chunks; the head count is the smallest whose split plan
    # on this GPU needs more than the static scratch.
    sms = _sms()
    w = None
    for H in range(1, 129):
        cand = I.Workload(name="wide", seed=12, F=1, Hp=8, Wp=30, H=H, d=128, K=4, W=7,
                          policy="clean", nodes=((0, 9, 4),),
                          prefilled=tuple((0, c, 0) for c in range(2, 9)))
        if _scratch(cand, sms)[1] > STATIC_SCRATCH:
            w = cand
            break
    assert w is not None, f"no head count refuses on {sms} SMs"
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


def test_plan_mirror_on_152_sms():
    """The expected plans used above, on the GB300's 152 SMs: clean1 runs 152
    units whole and splits the other 76 two ways (about 20 MB of scratch)."""
    w = I.WORKLOADS["clean1"]
    units = w.H * -(-w.tiles // 2)
    assert units == 228 and _plan(units, 4 * w.tiles, 152, 4 * 152) == (152, 2)
    n_split, need = _scratch(w, 152)
    assert n_split == 2 and need == 512 + 76 * 2 * 256 * (128 + 2) * 4   # counters + partials
