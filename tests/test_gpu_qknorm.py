"""GPU parity for the fused RMSNorm + RoPE + cache write
(sva_rope_kv_write_qknorm) and attention over the normalised keys."""
import numpy as np
import pytest
import torch

from paper_2609_22283_gb300 import inputs as I
from tests import _parity as P

pytestmark = pytest.mark.gpu


def test_normalised_cache_and_attention(oracle_mod):
    w = I.WORKLOADS["tinyn"]
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)
    g = P.oracle_geometry(w)
    gk = inp.gamma_k.double().numpy()
    gq = inp.gamma_q.double().numpy()
    pool = step.cache.slot_pool()
    exact, total = 0, 0
    for (s, c, l), (k_raw, v_raw) in I.all_states(w, inp).items():
        slot = step.cache.lookup(s, c, l)
        kn = oracle_mod.rms_norm(k_raw.double().numpy(), gk, inp.norm_eps)
        for h in range(w.H):
            ref = oracle_mod.bf16(oracle_mod.rope_head(kn[:, h, :], c, g))
            got = pool[slot, 0, h, :w.T, :].float().cpu().numpy().astype(np.float64)
            ulp = np.abs(ref) * 2.0 ** -7
            assert np.all(np.abs(got - ref) <= np.maximum(ulp, 2.0 ** -133) * 1.0001)
            exact += int(np.sum(got == ref))
            total += got.size
        v_cache = pool[slot, 1, :, :w.T, :].permute(1, 0, 2).contiguous().cpu()
        assert torch.equal(v_cache.view(torch.int16), v_raw.view(torch.int16))
    assert exact / total >= 0.995, exact / total
    states = P.oracle_states(w, inp)
    got = out.float().cpu().numpy()
    for i in range(w.n_nodes):
        ref, ref_lse = P.oracle_node(w, inp, states, i, range(w.H), range(w.T))
        for h in range(w.H):
            P.assert_close(got[i, :, h, :], ref[h], f"tinyn node {i} head {h}")
            np.testing.assert_allclose(lse[i, h].cpu().numpy(), ref_lse[h], atol=2e-3, rtol=0)
    qn = oracle_mod.rms_norm(inp.q[0].double().numpy(), gq, inp.norm_eps)
    for h in range(w.H):
        ref = oracle_mod.bf16(oracle_mod.rope_head(qn[:, h, :], w.nodes[0][1], g))
        gotq = q[0, :, h, :].float().cpu().numpy().astype(np.float64)
        assert np.all(np.abs(gotq - ref) <= np.maximum(np.abs(ref) * 2.0 ** -7, 2.0 ** -133) * 1.0001)
    step.close()


def test_qknorm_argument_checks(sva_mod):
    w = I.WORKLOADS["tinyn"]
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)
    nodes, _ = step.node_table()
    k = inp.k_new.cuda()
    gk = inp.gamma_k.cuda()
    with pytest.raises(sva_mod.SvaError) as e:
        step.cache.rope_kv_write_qknorm(nodes, k, k, q, gk, None)        # q without gamma_q
    assert e.value.status == sva_mod.ERR_INVALID_ARGUMENT
    with pytest.raises(sva_mod.SvaError) as e:
        step.cache.rope_kv_write_qknorm(nodes, k, k, None, gk, None, eps=0.0)
    assert e.value.status == sva_mod.ERR_INVALID_ARGUMENT
    step.close()
