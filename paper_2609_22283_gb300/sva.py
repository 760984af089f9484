"""ctypes binding of libsva.so (include/sva.h), with the same names.

Argument marshalling only: every step of the hot path runs in the library's
CUDA kernels.  torch provides device memory and streams; tensors are passed
as raw device pointers after dtype/shape/contiguity checks.  There is no
fallback: if libsva.so cannot be loaded, every call raises.
"""
from __future__ import annotations

import ctypes
import math
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libsva.so")

OK = 0
ERR_INVALID_ARGUMENT = 1
ERR_NOT_RESIDENT = 2
ERR_CAUSALITY = 3
ERR_CAPACITY = 4
ERR_UNSUPPORTED = 5
ERR_CUDA = 6
ERR_DEVICE_TIMEOUT = 7
ERR_UNAVAILABLE = 8
STATUS_NAMES = {0: "OK", 1: "INVALID_ARGUMENT", 2: "NOT_RESIDENT", 3: "CAUSALITY", 4: "CAPACITY",
                5: "UNSUPPORTED", 6: "CUDA", 7: "DEVICE_TIMEOUT", 8: "UNAVAILABLE"}

POLICY_CLEAN, POLICY_SAME, POLICY_PROG = 0, 1, 2
WITHIN_BIDIRECTIONAL, WITHIN_FRAME_CAUSAL = 0, 1
WITHIN = {"bidirectional": WITHIN_BIDIRECTIONAL, "frame_causal": WITHIN_FRAME_CAUSAL}
POLICIES = {"clean": POLICY_CLEAN, "same": POLICY_SAME, "prog": POLICY_PROG}
MAX_CTX = 16
MAX_NODES = 64

EXPORTED = ("sva_cache_bytes", "sva_cache_create", "sva_cache_bind", "sva_cache_lookup",
            "sva_cache_release", "sva_select_context", "sva_pipeline_round", "sva_check_pipeline",
            "sva_rope_kv_write", "sva_rope_kv_write_qknorm", "sva_attend_nodes",
            "sva_attend_nodes_sparse", "sva_attend_nodes_masked", "sva_qkv_project",
            "sva_qkv_project_rope",
            "sva_attend_workspace_bytes",
            "sva_cache_set_workspace", "sva_attend_nodes_noalloc", "sva_poll_device_status",
            "sva_debug_inject", "sva_destroy", "sva_last_error")


class SvaError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


class sva_geometry(ctypes.Structure):
    _fields_ = [("num_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("frames", ctypes.c_int32), ("grid_h", ctypes.c_int32), ("grid_w", ctypes.c_int32),
                ("num_slots", ctypes.c_int32), ("rope_pairs", ctypes.c_int32 * 3),
                ("max_frames", ctypes.c_int32), ("rope_theta", ctypes.c_double)]


class sva_node(ctypes.Structure):
    _fields_ = [("seq", ctypes.c_int32), ("chunk", ctypes.c_int32), ("level", ctypes.c_int32),
                ("own_slot", ctypes.c_int32), ("within", ctypes.c_int32),
                ("n_ctx", ctypes.c_int32),
                ("ctx_slot", ctypes.c_int32 * MAX_CTX), ("ctx_visible", ctypes.c_uint8 * MAX_CTX)]


class sva_attn_mask(ctypes.Structure):
    _fields_ = [("tile_mask", ctypes.c_void_p), ("tile_words", ctypes.c_int32),
                ("own_mask", ctypes.c_void_p), ("own_words", ctypes.c_int32),
                ("hist_mask", ctypes.c_void_p), ("hist_states", ctypes.c_int32),
                ("hist_words", ctypes.c_int32)]


_lib = None


def load(path: str = LIB_PATH):
    """Loads libsva.so (built by paper_2609_22283_gb300.build); raises if absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with paper_2609_22283_gb300.build.build() "
                           "(the CUDA library is required; there is no fallback)")
    lib = ctypes.CDLL(path)
    i32, p, pi32 = ctypes.c_int32, ctypes.c_void_p, ctypes.POINTER(ctypes.c_int32)
    pg = ctypes.POINTER(sva_geometry)
    pn = ctypes.POINTER(sva_node)
    sig = {
        "sva_cache_bytes": ([pg], ctypes.c_size_t),
        "sva_cache_create": ([pg, p, ctypes.c_size_t, ctypes.POINTER(p)], i32),
        "sva_cache_bind": ([p, i32, i32, i32, pi32], i32),
        "sva_cache_lookup": ([p, i32, i32, i32, pi32], i32),
        "sva_cache_release": ([p, i32, i32, i32], i32),
        "sva_select_context": ([i32, i32, i32, i32, i32, i32, pi32, pi32, pi32], i32),
        "sva_pipeline_round": ([i32, i32, i32, i32, pi32, pi32, pi32], i32),
        "sva_check_pipeline": ([i32, i32, i32, i32, pi32, pi32], i32),
        "sva_rope_kv_write": ([p, pn, i32, p, p, p, p], i32),
        "sva_rope_kv_write_qknorm": ([p, pn, i32, p, p, p, p, p, ctypes.c_float, p], i32),
        "sva_attend_nodes": ([p, pn, i32, p, p, p, ctypes.c_float, p], i32),
        "sva_attend_nodes_sparse": ([p, pn, i32, p, p, p, ctypes.c_float, p, i32, p], i32),
        "sva_qkv_project": ([p, p, i32, i32, p, p, p, p, p, p], i32),
        "sva_qkv_project_rope": ([p, pn, i32, p, i32, p, p, p, p], i32),
        "sva_attend_nodes_masked": ([p, pn, i32, p, p, p, ctypes.c_float, p, p], i32),
        "sva_attend_workspace_bytes": ([p], ctypes.c_size_t),
        "sva_attend_nodes_noalloc": ([p, pn, i32, p, p, p, ctypes.c_float, p], i32),
        "sva_cache_set_workspace": ([p, p, ctypes.c_size_t], i32),
        "sva_poll_device_status": ([p, p], i32),
        "sva_debug_inject": ([p, i32, ctypes.c_double], i32),
        "sva_destroy": ([p], i32),
        "sva_last_error": ([], ctypes.c_char_p),
    }
    for name, (args, res) in sig.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = res
    _lib = lib
    return lib


def _check(status: int):
    if status != OK:
        msg = _lib.sva_last_error().decode(errors="replace")
        raise SvaError(status, msg)


def _stream_handle(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


def _tok_major(t: torch.Tensor, name: str, n: int, T: int, H: int, d: int):
    if t.dtype != torch.bfloat16 or not t.is_cuda or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous bf16 CUDA tensor")
    if tuple(t.shape) != (n, T, H, d):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {(n, T, H, d)}")


# ---------------------------------------------------------------- selection (host)

def select_context(policy: int, K: int, W: int, chunk: int, level: int, cap: int = MAX_CTX):
    lib = load()
    ch = (ctypes.c_int32 * max(cap, 1))()
    lv = (ctypes.c_int32 * max(cap, 1))()
    n = ctypes.c_int32()
    _check(lib.sva_select_context(policy, K, W, chunk, level, cap, ch, lv, ctypes.byref(n)))
    return [(ch[i], lv[i]) for i in range(n.value)]


def pipeline_round(K: int, B: int, n: int, cap: int = 64):
    lib = load()
    ch = (ctypes.c_int32 * cap)()
    lv = (ctypes.c_int32 * cap)()
    cnt = ctypes.c_int32()
    _check(lib.sva_pipeline_round(K, B, n, cap, ch, lv, ctypes.byref(cnt)))
    return [(ch[i], lv[i]) for i in range(cnt.value)]


def check_pipeline(K: int, level: int, chunk: int, states) -> int:
    """Returns the sva_status of the Eq. 7 check (no exception for UNAVAILABLE)."""
    lib = load()
    n = len(states)
    ch = (ctypes.c_int32 * max(n, 1))(*[c for c, _ in states])
    lv = (ctypes.c_int32 * max(n, 1))(*[l for _, l in states])
    return int(lib.sva_check_pipeline(K, level, chunk, n, ch, lv))


def last_error() -> str:
    return load().sva_last_error().decode(errors="replace")


def make_geometry(H, d, F, Hp, Wp, num_slots, pairs, max_frames, theta=10000.0) -> sva_geometry:
    g = sva_geometry()
    g.num_heads, g.head_dim, g.frames, g.grid_h, g.grid_w = H, d, F, Hp, Wp
    g.num_slots = num_slots
    g.rope_pairs[0], g.rope_pairs[1], g.rope_pairs[2] = pairs
    g.max_frames = max_frames
    g.rope_theta = theta
    return g


def cache_bytes(g: sva_geometry) -> int:
    return int(load().sva_cache_bytes(ctypes.byref(g)))


def make_nodes(entries) -> ctypes.Array:
    """entries: iterable of dicts with seq, chunk, level, own_slot, ctx (list of slots),
    visible (optional list of 0/1), within (optional, default bidirectional)."""
    entries = list(entries)
    arr = (sva_node * max(len(entries), 1))()
    for i, e in enumerate(entries):
        n = arr[i]
        n.seq, n.chunk, n.level, n.own_slot = e["seq"], e["chunk"], e["level"], e["own_slot"]
        n.within = e.get("within", WITHIN_BIDIRECTIONAL)
        ctx = list(e.get("ctx", []))
        vis = list(e.get("visible", [1] * len(ctx)))
        n.n_ctx = len(ctx)
        for k, s in enumerate(ctx[:MAX_CTX]):
            n.ctx_slot[k] = s
            n.ctx_visible[k] = vis[k]
    return arr


class Cache:
    """A KV cache over a caller-owned device buffer (a torch uint8 tensor)."""

    def __init__(self, g: sva_geometry, buf: torch.Tensor | None = None, device=None):
        lib = load()
        self.g = g
        self.nbytes = cache_bytes(g)
        if self.nbytes == 0:
            raise SvaError(ERR_INVALID_ARGUMENT, last_error())
        if buf is None:
            buf = torch.empty(self.nbytes, dtype=torch.uint8, device=device or "cuda")
        if not buf.is_cuda or buf.numel() * buf.element_size() < self.nbytes:
            raise ValueError("cache buffer must be a CUDA tensor of at least cache_bytes(g) bytes")
        self.buf = buf
        self.T = g.frames * g.grid_h * g.grid_w
        self.Tpad = (self.T + 127) // 128 * 128
        handle = ctypes.c_void_p()
        with torch.cuda.device(buf.device):
            _check(lib.sva_cache_create(ctypes.byref(g), ctypes.c_void_p(buf.data_ptr()),
                                        self.nbytes, ctypes.byref(handle)))
        self.handle = handle

    # slot pool view [num_slots][2][H][Tpad][d] (bf16), for inspection in tests
    def slot_pool(self) -> torch.Tensor:
        g = self.g
        n = g.num_slots * 2 * g.num_heads * self.Tpad * g.head_dim
        return self.buf[: n * 2].view(torch.bfloat16).view(g.num_slots, 2, g.num_heads, self.Tpad,
                                                           g.head_dim)

    def bind(self, seq: int, chunk: int, level: int) -> int:
        s = ctypes.c_int32()
        _check(_lib.sva_cache_bind(self.handle, seq, chunk, level, ctypes.byref(s)))
        return s.value

    def lookup(self, seq: int, chunk: int, level: int) -> int:
        s = ctypes.c_int32()
        _check(_lib.sva_cache_lookup(self.handle, seq, chunk, level, ctypes.byref(s)))
        return s.value

    def release(self, seq: int, chunk: int, level: int):
        _check(_lib.sva_cache_release(self.handle, seq, chunk, level))

    def rope_kv_write(self, nodes, k_new, v_new, q=None, stream=None, check=True):
        n = len(nodes) if not isinstance(nodes, ctypes.Array) else None
        arr = nodes if isinstance(nodes, ctypes.Array) else make_nodes(nodes)
        count = n if n is not None else len(arr)
        if check:
            g = self.g
            _tok_major(k_new, "k_new", count, self.T, g.num_heads, g.head_dim)
            _tok_major(v_new, "v_new", count, self.T, g.num_heads, g.head_dim)
            if q is not None:
                _tok_major(q, "q", count, self.T, g.num_heads, g.head_dim)
        st = _lib.sva_rope_kv_write(self.handle, arr, count, ctypes.c_void_p(k_new.data_ptr()),
                                    ctypes.c_void_p(v_new.data_ptr()),
                                    ctypes.c_void_p(q.data_ptr() if q is not None else 0),
                                    ctypes.c_void_p(_stream_handle(stream)))
        _check(st)

    def rope_kv_write_qknorm(self, nodes, k_new, v_new, q, gamma_k, gamma_q, eps=1e-6,
                             stream=None):
        """sva_rope_kv_write_qknorm: RMSNorm (fp32 gammas of H*d) then RoPE."""
        arr = nodes if isinstance(nodes, ctypes.Array) else make_nodes(nodes)
        for gname, gm in (("gamma_k", gamma_k), ("gamma_q", gamma_q)):
            if gm is not None and (gm.dtype != torch.float32 or not gm.is_cuda
                                   or not gm.is_contiguous()):
                raise ValueError(f"{gname} must be a contiguous fp32 CUDA tensor")
        st = _lib.sva_rope_kv_write_qknorm(
            self.handle, arr, len(arr), ctypes.c_void_p(k_new.data_ptr()),
            ctypes.c_void_p(v_new.data_ptr()), ctypes.c_void_p(q.data_ptr() if q is not None else 0),
            ctypes.c_void_p(gamma_k.data_ptr()),
            ctypes.c_void_p(gamma_q.data_ptr() if gamma_q is not None else 0), float(eps),
            ctypes.c_void_p(_stream_handle(stream)))
        _check(st)

    def attend_nodes(self, nodes, q, out, lse=None, scale=None, stream=None, check=True):
        n = len(nodes) if not isinstance(nodes, ctypes.Array) else None
        arr = nodes if isinstance(nodes, ctypes.Array) else make_nodes(nodes)
        count = n if n is not None else len(arr)
        g = self.g
        if check:
            _tok_major(q, "q", count, self.T, g.num_heads, g.head_dim)
            _tok_major(out, "out", count, self.T, g.num_heads, g.head_dim)
            if lse is not None and (lse.dtype != torch.float32 or not lse.is_contiguous()
                                    or tuple(lse.shape) != (count, g.num_heads, self.T)):
                raise ValueError("lse must be a contiguous fp32 tensor [n][H][T]")
        if scale is None:
            scale = 1.0 / math.sqrt(g.head_dim)
        st = _lib.sva_attend_nodes(self.handle, arr, count, ctypes.c_void_p(q.data_ptr()),
                                   ctypes.c_void_p(out.data_ptr()),
                                   ctypes.c_void_p(lse.data_ptr() if lse is not None else 0),
                                   float(scale), ctypes.c_void_p(_stream_handle(stream)))
        _check(st)

    def attend_nodes_sparse(self, nodes, q, out, tile_mask, lse=None, scale=None, stream=None,
                            check=True):
        """sva_attend_nodes_sparse: tile_mask is a contiguous int32 CUDA tensor
        [n_nodes][ceil(T/128)][words] of key-tile bits (see include/sva.h)."""
        n = len(nodes) if not isinstance(nodes, ctypes.Array) else None
        arr = nodes if isinstance(nodes, ctypes.Array) else make_nodes(nodes)
        count = n if n is not None else len(arr)
        g = self.g
        nt = -(-self.T // 128)
        if check:
            _tok_major(q, "q", count, self.T, g.num_heads, g.head_dim)
            _tok_major(out, "out", count, self.T, g.num_heads, g.head_dim)
            if lse is not None and (lse.dtype != torch.float32 or not lse.is_contiguous()
                                    or tuple(lse.shape) != (count, g.num_heads, self.T)):
                raise ValueError("lse must be a contiguous fp32 tensor [n][H][T]")
        if (tile_mask.dtype != torch.int32 or not tile_mask.is_cuda or not tile_mask.is_contiguous()
                or tile_mask.dim() != 3 or tuple(tile_mask.shape[:2]) != (count, nt)):
            raise ValueError(f"tile_mask must be a contiguous int32 CUDA tensor [{count}][{nt}][words]")
        if scale is None:
            scale = 1.0 / math.sqrt(g.head_dim)
        st = _lib.sva_attend_nodes_sparse(self.handle, arr, count, ctypes.c_void_p(q.data_ptr()),
                                          ctypes.c_void_p(out.data_ptr()),
                                          ctypes.c_void_p(lse.data_ptr() if lse is not None else 0),
                                          float(scale), ctypes.c_void_p(tile_mask.data_ptr()),
                                          int(tile_mask.shape[2]),
                                          ctypes.c_void_p(_stream_handle(stream)))
        _check(st)

    def attend_nodes_masked(self, nodes, q, out, lse=None, scale=None, tile_mask=None,
                            own_mask=None, hist_mask=None, stream=None, check=True):
        """sva_attend_nodes_masked: tile_mask as in attend_nodes_sparse, own_mask a
        contiguous int32 CUDA tensor [n_nodes][T][words] of own-chunk token bits,
        hist_mask one [n_nodes][T][states][words] of history token bits (state
        j = the node's j-th context); any may be None."""
        n = len(nodes) if not isinstance(nodes, ctypes.Array) else None
        arr = nodes if isinstance(nodes, ctypes.Array) else make_nodes(nodes)
        count = n if n is not None else len(arr)
        g = self.g
        if check:
            _tok_major(q, "q", count, self.T, g.num_heads, g.head_dim)
            _tok_major(out, "out", count, self.T, g.num_heads, g.head_dim)
        for t, nm, rows in ((tile_mask, "tile_mask", -(-self.T // 128)), (own_mask, "own_mask", self.T)):
            if t is not None and (t.dtype != torch.int32 or not t.is_cuda or not t.is_contiguous()
                                  or t.dim() != 3 or tuple(t.shape[:2]) != (count, rows)):
                raise ValueError(f"{nm} must be a contiguous int32 CUDA tensor [{count}][{rows}][words]")
        if hist_mask is not None and (hist_mask.dtype != torch.int32 or not hist_mask.is_cuda
                                      or not hist_mask.is_contiguous() or hist_mask.dim() != 4
                                      or tuple(hist_mask.shape[:2]) != (count, self.T)):
            raise ValueError(f"hist_mask must be a contiguous int32 CUDA tensor [{count}][{self.T}][states][words]")
        m = sva_attn_mask(ctypes.c_void_p(tile_mask.data_ptr() if tile_mask is not None else 0),
                          int(tile_mask.shape[2]) if tile_mask is not None else 0,
                          ctypes.c_void_p(own_mask.data_ptr() if own_mask is not None else 0),
                          int(own_mask.shape[2]) if own_mask is not None else 0,
                          ctypes.c_void_p(hist_mask.data_ptr() if hist_mask is not None else 0),
                          int(hist_mask.shape[2]) if hist_mask is not None else 0,
                          int(hist_mask.shape[3]) if hist_mask is not None else 0)
        if scale is None:
            scale = 1.0 / math.sqrt(g.head_dim)
        st = _lib.sva_attend_nodes_masked(self.handle, arr, count, ctypes.c_void_p(q.data_ptr()),
                                          ctypes.c_void_p(out.data_ptr()),
                                          ctypes.c_void_p(lse.data_ptr() if lse is not None else 0),
                                          float(scale), ctypes.byref(m),
                                          ctypes.c_void_p(_stream_handle(stream)))
        _check(st)

    def qkv_project(self, x, weight, bias, q, k, v, stream=None, check=True):
        """sva_qkv_project: [q | k | v] = x W^T + b.  x [..., C] bf16 (rows = all
        leading dims), weight [3*H*d][C] bf16, bias [3*H*d] fp32 or None, q, k, v
        bf16 with rows * H * d elements each (e.g. [n][T][H][d]); all contiguous
        CUDA tensors."""
        g = self.g
        n_out = g.num_heads * g.head_dim
        C = int(x.shape[-1])
        rows = x.numel() // C
        if check:
            for t, nm in ((x, "x"), (weight, "weight"), (q, "q"), (k, "k"), (v, "v")):
                if t.dtype != torch.bfloat16 or not t.is_cuda or not t.is_contiguous():
                    raise ValueError(f"{nm} must be a contiguous bf16 CUDA tensor")
            if tuple(weight.shape) != (3 * n_out, C):
                raise ValueError(f"weight must be [{3 * n_out}][{C}]")
            for t, nm in ((q, "q"), (k, "k"), (v, "v")):
                if t.numel() != rows * n_out:
                    raise ValueError(f"{nm} must hold rows * H * d = {rows * n_out} elements")
            if bias is not None and (bias.dtype != torch.float32 or not bias.is_cuda
                                     or not bias.is_contiguous() or bias.numel() != 3 * n_out):
                raise ValueError(f"bias must be a contiguous fp32 CUDA tensor of {3 * n_out}")
        st = _lib.sva_qkv_project(self.handle, ctypes.c_void_p(x.data_ptr()), rows, C,
                                  ctypes.c_void_p(weight.data_ptr()),
                                  ctypes.c_void_p(bias.data_ptr() if bias is not None else 0),
                                  ctypes.c_void_p(q.data_ptr()), ctypes.c_void_p(k.data_ptr()),
                                  ctypes.c_void_p(v.data_ptr()),
                                  ctypes.c_void_p(_stream_handle(stream)))
        _check(st)

    def qkv_project_rope(self, nodes, x, weight, bias, q, stream=None, check=True):
        """sva_qkv_project_rope: the projection with RoPE and the cache write fused
        into its epilogue.  x [n][T][C] bf16 (node i's token rows), weight and
        bias as qkv_project, q [n][T][H][d] bf16 receives Q'; K' and V go to the
        nodes' own slots."""
        n = len(nodes) if not isinstance(nodes, ctypes.Array) else None
        arr = nodes if isinstance(nodes, ctypes.Array) else make_nodes(nodes)
        count = n if n is not None else len(arr)
        g = self.g
        n_out = g.num_heads * g.head_dim
        C = int(x.shape[-1])
        if check:
            for t, nm in ((x, "x"), (weight, "weight"), (q, "q")):
                if t.dtype != torch.bfloat16 or not t.is_cuda or not t.is_contiguous():
                    raise ValueError(f"{nm} must be a contiguous bf16 CUDA tensor")
            if x.numel() != count * self.T * C:
                raise ValueError(f"x must hold n_nodes * T rows of {C} features")
            if tuple(weight.shape) != (3 * n_out, C):
                raise ValueError(f"weight must be [{3 * n_out}][{C}]")
            _tok_major(q, "q", count, self.T, g.num_heads, g.head_dim)
            if bias is not None and (bias.dtype != torch.float32 or not bias.is_cuda
                                     or not bias.is_contiguous() or bias.numel() != 3 * n_out):
                raise ValueError(f"bias must be a contiguous fp32 CUDA tensor of {3 * n_out}")
        st = _lib.sva_qkv_project_rope(self.handle, arr, count, ctypes.c_void_p(x.data_ptr()), C,
                                       ctypes.c_void_p(weight.data_ptr()),
                                       ctypes.c_void_p(bias.data_ptr() if bias is not None else 0),
                                       ctypes.c_void_p(q.data_ptr()),
                                       ctypes.c_void_p(_stream_handle(stream)))
        _check(st)

    def workspace_bytes(self) -> int:
        return int(_lib.sva_attend_workspace_bytes(self.handle))

    def set_workspace(self, buf: torch.Tensor | None):
        """Attaches a caller-owned split workspace (a CUDA uint8 tensor), or detaches it."""
        if buf is None:
            _check(_lib.sva_cache_set_workspace(self.handle, None, 0))
            self.ws = None
            return
        nbytes = buf.numel() * buf.element_size()
        _check(_lib.sva_cache_set_workspace(self.handle, ctypes.c_void_p(buf.data_ptr()), nbytes))
        self.ws = buf

    def poll(self, stream=None) -> int:
        """sva_poll_device_status: returns the status code (0 = OK)."""
        return int(_lib.sva_poll_device_status(self.handle, ctypes.c_void_p(_stream_handle(stream))))

    def debug_inject(self, mode: int, timeout_s: float = 1.0):
        _check(_lib.sva_debug_inject(self.handle, mode, float(timeout_s)))

    def close(self):
        if getattr(self, "handle", None):
            _lib.sva_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
