"""Validation paths of the C ABI on a real cache: each bad call returns its
status code and launches nothing (the output canary is untouched)."""
import ctypes

import pytest
import torch

from paper_2609_22283_gb300 import inputs as I
from tests import _parity as P

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ready(sva_mod):
    w = I.WORKLOADS["tiny"]
    inp = I.generate(w)
    step, q, out, lse = P.gpu_step(w, inp)
    return sva_mod, w, step, q, out


def _status(fn):
    try:
        fn()
    except Exception as e:  # SvaError
        return getattr(e, "status", None)
    return 0


def _node(step, i):
    nodes, _ = step.node_table()
    n = nodes[i]
    return dict(seq=n.seq, chunk=n.chunk, level=n.level, own_slot=n.own_slot,
                ctx=[n.ctx_slot[k] for k in range(n.n_ctx)])


def test_create_errors(sva_mod):
    lib = sva_mod.load()
    g = sva_mod.make_geometry(2, 96, 1, 8, 8, 4, (16, 16, 16), 16)
    buf = torch.empty(1 << 20, dtype=torch.uint8, device="cuda")
    h = ctypes.c_void_p()
    assert lib.sva_cache_create(ctypes.byref(g), ctypes.c_void_p(buf.data_ptr()), 1 << 20,
                                ctypes.byref(h)) == sva_mod.ERR_UNSUPPORTED
    g = sva_mod.make_geometry(2, 64, 1, 8, 8, 4, (12, 10, 10), 16)
    need = sva_mod.cache_bytes(g)
    assert lib.sva_cache_create(ctypes.byref(g), ctypes.c_void_p(buf.data_ptr() + 16), need,
                                ctypes.byref(h)) == sva_mod.ERR_INVALID_ARGUMENT
    assert lib.sva_cache_create(ctypes.byref(g), ctypes.c_void_p(buf.data_ptr()), need - 1,
                                ctypes.byref(h)) == sva_mod.ERR_INVALID_ARGUMENT
    host = torch.empty(need, dtype=torch.uint8)
    assert lib.sva_cache_create(ctypes.byref(g), ctypes.c_void_p(host.data_ptr()), need,
                                ctypes.byref(h)) == sva_mod.ERR_INVALID_ARGUMENT


def test_pad_rows_zeroed_rest_untouched(sva_mod):
    g = sva_mod.make_geometry(2, 64, 1, 6, 7, 3, (12, 10, 10), 16)   # T = 42, Tpad = 128
    need = sva_mod.cache_bytes(g)
    buf = torch.full((need,), 0x5A, dtype=torch.uint8, device="cuda")
    c = sva_mod.Cache(g, buf)
    pool = c.slot_pool().view(torch.int16)
    assert torch.all(pool[:, :, :, 42:, :] == 0)
    assert torch.all(pool[:, :, :, :42, :] == 0x5A5A)
    c.close()


def test_slot_table_errors(sva_mod):
    g = sva_mod.make_geometry(2, 64, 1, 8, 8, 2, (12, 10, 10), 16)
    c = sva_mod.Cache(g)
    c.bind(0, 1, 0)
    assert _status(lambda: c.bind(0, 1, 0)) == sva_mod.ERR_INVALID_ARGUMENT
    assert _status(lambda: c.bind(0, 1, -1)) == sva_mod.ERR_INVALID_ARGUMENT
    c.bind(0, 2, 1)
    assert _status(lambda: c.bind(0, 3, 2)) == sva_mod.ERR_CAPACITY
    assert _status(lambda: c.lookup(0, 9, 9)) == sva_mod.ERR_NOT_RESIDENT
    c.release(0, 1, 0)
    assert _status(lambda: c.lookup(0, 1, 0)) == sva_mod.ERR_NOT_RESIDENT
    assert _status(lambda: c.release(0, 1, 0)) == sva_mod.ERR_NOT_RESIDENT
    assert c.bind(0, 3, 2) in (0, 1)
    c.close()


def test_attend_validation(ready):
    sva, w, step, q, out = ready
    canary = torch.full_like(out, 7.0)
    c = step.cache
    good = [_node(step, 0), _node(step, 1)]

    def call(nodes, qq=q, oo=canary, scale=0.125, lse=None):
        return _status(lambda: c.attend_nodes(nodes, qq, oo, lse, scale))

    bad_future = dict(good[1], ctx=[good[0]["own_slot"]])            # (2,1) reading chunk 3
    assert call([good[0], bad_future]) == sva.ERR_CAUSALITY
    assert call([dict(good[0], ctx=good[0]["ctx"] + [good[0]["ctx"][0]]), good[1]]) == sva.ERR_INVALID_ARGUMENT
    assert call([dict(good[0], ctx=[good[0]["own_slot"]]), good[1]]) == sva.ERR_CAUSALITY
    assert call([dict(good[0], ctx=[99]), good[1]]) == sva.ERR_INVALID_ARGUMENT
    assert call([dict(good[0], own_slot=good[1]["own_slot"]), good[1]]) == sva.ERR_INVALID_ARGUMENT
    assert call(good, scale=0.0) == sva.ERR_INVALID_ARGUMENT
    assert call(good, scale=float("nan")) == sva.ERR_INVALID_ARGUMENT
    # a context bound but not yet written, then written but of another sequence
    other = c.bind(1, 1, 0)
    assert call([dict(good[0], ctx=[other]), good[1]]) == sva.ERR_NOT_RESIDENT
    z = torch.zeros((1, w.T, w.H, w.d), dtype=torch.bfloat16, device="cuda")
    c.rope_kv_write([dict(seq=1, chunk=1, level=0, own_slot=other)], z, z)
    assert call([dict(good[0], ctx=[other]), good[1]]) == sva.ERR_CAUSALITY
    c.release(1, 1, 0)
    # too many contexts
    arr = sva.make_nodes(good)
    arr[0].n_ctx = 17
    assert _status(lambda: c.attend_nodes(arr, q, canary, None, 0.125, check=False)) == sva.ERR_CAPACITY
    # misaligned / null pointers through the raw ABI
    lib = sva.load()
    arr = sva.make_nodes(good)
    s = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    assert lib.sva_attend_nodes(c.handle, arr, 2, ctypes.c_void_p(q.data_ptr() + 2),
                                ctypes.c_void_p(canary.data_ptr()), None, 0.125, s) == sva.ERR_INVALID_ARGUMENT
    assert lib.sva_attend_nodes(c.handle, arr, 2, None, ctypes.c_void_p(canary.data_ptr()), None,
                                0.125, s) == sva.ERR_INVALID_ARGUMENT
    assert lib.sva_attend_nodes(c.handle, arr, 0, ctypes.c_void_p(q.data_ptr()),
                                ctypes.c_void_p(canary.data_ptr()), None, 0.125, s) == sva.ERR_INVALID_ARGUMENT
    assert lib.sva_attend_nodes(c.handle, arr, 65, ctypes.c_void_p(q.data_ptr()),
                                ctypes.c_void_p(canary.data_ptr()), None, 0.125, s) == sva.ERR_CAPACITY
    torch.cuda.synchronize()
    assert torch.all(canary == 7.0)                                    # nothing was launched
    assert c.poll() == sva.OK


def test_not_resident_own_and_context(sva_mod):
    sva = sva_mod
    g = sva.make_geometry(2, 64, 1, 8, 8, 4, (12, 10, 10), 16)
    c = sva.Cache(g)
    a = c.bind(0, 1, 0)
    b = c.bind(0, 2, 1)
    q = torch.zeros((1, 64, 2, 64), dtype=torch.bfloat16, device="cuda")
    o = torch.full_like(q, 3.0)
    st = _status(lambda: c.attend_nodes([dict(seq=0, chunk=2, level=1, own_slot=b, ctx=[a])], q, o))
    assert st == sva.ERR_NOT_RESIDENT
    k = torch.zeros_like(q)
    c.rope_kv_write([dict(seq=0, chunk=2, level=1, own_slot=b)], k, k, None)
    st = _status(lambda: c.attend_nodes([dict(seq=0, chunk=2, level=1, own_slot=b, ctx=[a])], q, o))
    assert st == sva.ERR_NOT_RESIDENT                                   # context still unwritten
    torch.cuda.synchronize()
    assert torch.all(o == 3.0)
    c.close()


def test_rope_write_validation(sva_mod):
    sva = sva_mod
    g = sva.make_geometry(2, 64, 1, 8, 8, 4, (12, 10, 10), 8)
    c = sva.Cache(g)
    a = c.bind(0, 1, 0)
    b = c.bind(0, 2, 1)
    k = torch.zeros((2, 64, 2, 64), dtype=torch.bfloat16, device="cuda")
    n_a = dict(seq=0, chunk=1, level=0, own_slot=a)
    n_b = dict(seq=0, chunk=2, level=1, own_slot=b)
    assert _status(lambda: c.rope_kv_write([n_a, dict(n_b, own_slot=a)], k, k)) == sva.ERR_INVALID_ARGUMENT
    assert _status(lambda: c.rope_kv_write([n_a, dict(n_b, own_slot=3)], k, k)) == sva.ERR_INVALID_ARGUMENT
    assert _status(lambda: c.rope_kv_write([n_a, dict(n_b, chunk=8)], k, k)) == sva.ERR_INVALID_ARGUMENT
    far = c.bind(0, 8, 0)                                              # frames [8, 9) >= max_frames 8
    assert _status(lambda: c.rope_kv_write([n_a, dict(seq=0, chunk=8, level=0, own_slot=far)], k, k)) == sva.ERR_CAPACITY
    lib = sva.load()
    arr = sva.make_nodes([n_a, n_b])
    s = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    assert lib.sva_rope_kv_write(c.handle, arr, 2, ctypes.c_void_p(k.data_ptr() + 4),
                                 ctypes.c_void_p(k.data_ptr()), None, s) == sva.ERR_INVALID_ARGUMENT
    assert lib.sva_rope_kv_write(c.handle, arr, 65, ctypes.c_void_p(k.data_ptr()),
                                 ctypes.c_void_p(k.data_ptr()), None, s) == sva.ERR_CAPACITY
    c.close()
