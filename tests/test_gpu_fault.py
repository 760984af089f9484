"""Failure detection without a GPU fault: the test hook makes one K/V copy
never arrive, the kernel's bounded wait expires after 0.2 s, every CTA
records SVA_ERR_DEVICE_TIMEOUT, drains and exits, and the host reads the
status.  The context stays usable: the next launch succeeds and reproduces
the earlier output bit for bit."""
import pytest
import torch

from paper_2609_22283_gb300 import inputs as I
from tests import _parity as P

pytestmark = pytest.mark.gpu


def test_bounded_wait_reports_timeout(sva_mod):
    sva = sva_mod
    w = I.WORKLOADS["tiny"]
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)
    nodes, n = step.node_table()
    c = step.cache
    before = out.clone()
    junk = torch.empty_like(out)
    c.debug_inject(1, 0.2)
    c.attend_nodes(nodes, q, junk, None, step.scale, check=False)
    assert c.poll() == sva.ERR_DEVICE_TIMEOUT
    assert "bounded wait" in sva.last_error()
    assert c.poll() == sva.OK                      # the status word was cleared
    c.debug_inject(0, 1.0)
    again = torch.empty_like(out)
    c.attend_nodes(nodes, q, again, None, step.scale, check=False)
    assert c.poll() == sva.OK
    assert torch.equal(again.view(torch.int16), before.view(torch.int16))
    step.close()
