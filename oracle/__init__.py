"""fp64 CPU oracle for policy-indexed chunk-causal attention.

TEST INFRASTRUCTURE ONLY: the product library never imports, links or runs
anything in this package.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` use it.  It shares no code with the CUDA
path; the two meet only in the seeded input generator, which holds none of
the method's arithmetic.

The arithmetic lives in ``sva_oracle.c`` (plain C, fp64, OpenMP over query
rows) and is driven from here:

* ``select`` / ``pipeline_round`` / ``available`` -- Eq. 2-3, Eq. 6, Eq. 7.
* ``rope_head`` / ``bf16`` -- the 3D RoPE reading and the bf16 cache store.
* ``attend_rows`` -- Eq. 4 masked softmax attention.
* ``qkv_project`` -- the input projection producing q, k, v token-major.
* ``qkv_project_rope`` -- that projection with the RoPE of q and k applied to
  its unrounded outputs (the fused projection + cache write).
* ``node_forward`` -- one denoising node end to end: its context selection,
  the rotation of every key state it reads and of its queries, the bf16
  rounding of what the cache would hold, and the attention of the requested
  (head, row) pairs.

``oracle.brute`` holds an independent dense-mask formulation used to pin
this one on tiny inputs.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "sva_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")

POLICY_CLEAN, POLICY_SAME, POLICY_PROG = 0, 1, 2
POLICY_IDS = {"clean": POLICY_CLEAN, "same": POLICY_SAME, "prog": POLICY_PROG}


def build(force: bool = False) -> str:
    """Compiles sva_oracle.c into liboracle.so next to it (gcc, OpenMP)."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
           "-fno-fast-math", "-ffp-contract=off", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


_lib = None


def _load():
    global _lib
    if _lib is not None:
        return _lib
    lib = ctypes.CDLL(build())
    i32, dbl, lng = ctypes.c_int, ctypes.c_double, ctypes.c_long
    pi32 = ctypes.POINTER(ctypes.c_int)
    pd = ctypes.POINTER(ctypes.c_double)
    lib.oracle_phi.argtypes = [i32, i32, i32]
    lib.oracle_phi.restype = i32
    lib.oracle_select.argtypes = [i32, i32, i32, i32, pi32, pi32]
    lib.oracle_select.restype = i32
    lib.oracle_pipeline_round.argtypes = [i32, i32, i32, pi32, pi32]
    lib.oracle_pipeline_round.restype = i32
    lib.oracle_available.argtypes = [i32, i32, i32]
    lib.oracle_available.restype = i32
    lib.oracle_bf16.argtypes = [dbl]
    lib.oracle_bf16.restype = dbl
    lib.oracle_bf16_array.argtypes = [pd, pd, lng]
    lib.oracle_bf16_array.restype = None
    lib.oracle_rope_head.argtypes = [pd, pd, i32, i32, i32, i32, i32, lng, pi32, dbl]
    lib.oracle_rope_head.restype = None
    lib.oracle_rms_norm.argtypes = [pd, pd, pd, lng, i32, dbl]
    lib.oracle_rms_norm.restype = None
    lib.oracle_attend_rows.argtypes = [pd, pd, pd, pd, lng, i32, lng, dbl, pd, pd]
    lib.oracle_attend_rows.restype = None
    lib.oracle_num_threads.argtypes = []
    lib.oracle_num_threads.restype = i32
    _lib = lib
    return lib


def _pd(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def num_threads() -> int:
    return int(_load().oracle_num_threads())


# ---------------------------------------------------------------- selection

def phi(policy: int, j: int, r: int) -> int:
    """Eq. 3."""
    return int(_load().oracle_phi(policy, j, r))


def select(policy: int, W: int, b: int, j: int) -> list[tuple[int, int]]:
    """Eq. 2 with the full offset window: [(b - r, phi(j, r)) for r = 1..min(W, b-1)]."""
    cap = max(W, 0) + 1
    ch = (ctypes.c_int * cap)()
    lv = (ctypes.c_int * cap)()
    n = _load().oracle_select(policy, W, b, j, ch, lv)
    if n < 0:
        raise ValueError(f"unknown policy {policy}")
    return [(ch[i], lv[i]) for i in range(n)]


def pipeline_round(K: int, B: int, n: int) -> list[tuple[int, int]]:
    """Eq. 6: the (chunk, level) states active at the start of round n."""
    ch = (ctypes.c_int * max(K, 1))()
    lv = (ctypes.c_int * max(K, 1))()
    cnt = _load().oracle_pipeline_round(K, B, n, ch, lv)
    return [(ch[i], lv[i]) for i in range(cnt)]


def available(j: int, r: int, level: int) -> bool:
    """Eq. 7."""
    return bool(_load().oracle_available(j, r, level))


# ---------------------------------------------------------------- RoPE and bf16

def bf16(x) -> np.ndarray:
    """Round-to-nearest-even onto the bf16 grid, element-wise, in fp64."""
    x = np.ascontiguousarray(np.asarray(x, dtype=np.float64))
    y = np.empty_like(x)
    _load().oracle_bf16_array(_pd(x), _pd(y), x.size)
    return y


@dataclass(frozen=True)
class Geometry:
    """Chunk geometry: F latent frames of Hp x Wp patches per chunk, H heads of size d."""
    F: int
    Hp: int
    Wp: int
    H: int
    d: int
    pairs: tuple[int, int, int]
    theta: float = 10000.0

    @property
    def T(self) -> int:
        return self.F * self.Hp * self.Wp


def rope_head(x: np.ndarray, b: int, g: Geometry) -> np.ndarray:
    """3D RoPE (reading) of one head's rows x[T][d] of chunk b, fp64, unrounded."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    assert x.shape == (g.T, g.d)
    y = np.empty_like(x)
    pairs = (ctypes.c_int * 3)(*g.pairs)
    _load().oracle_rope_head(_pd(x), _pd(y), g.T, g.d, g.F, g.Hp, g.Wp, b, pairs, g.theta)
    return y


def rms_norm(x: np.ndarray, gamma: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm of each token's vector: x [T][H][d] (or [T][n]) with gamma [H*d]."""
    shape = x.shape
    x2 = np.ascontiguousarray(np.asarray(x, dtype=np.float64).reshape(shape[0], -1))
    g = np.ascontiguousarray(np.asarray(gamma, dtype=np.float64).reshape(-1))
    assert g.shape[0] == x2.shape[1]
    y = np.empty_like(x2)
    _load().oracle_rms_norm(_pd(x2), _pd(g), _pd(y), x2.shape[0], x2.shape[1], float(eps))
    return y.reshape(shape)


# ---------------------------------------------------------------- QKV projection

def qkv_project(x: np.ndarray, weight: np.ndarray, bias=None, heads: int = 1):
    """The linear projection in front of the attention layer, fp64:
    y = x W^T + b over the last axis, then split into q, k, v.

    x: [rows][C]; weight: [3 * N][C] (out_features x in_features, the rows of
    q's outputs first, then k's, then v's); bias: [3 * N] or None.
    Returns (q, k, v), each [rows][heads][N / heads], unrounded.  A library
    matrix product is the one step (no blocking or reordering of its own).
    """
    x = np.asarray(x, dtype=np.float64)
    w = np.asarray(weight, dtype=np.float64)
    rows, C = x.shape
    assert w.shape[1] == C and w.shape[0] % 3 == 0
    n = w.shape[0] // 3
    assert n % heads == 0
    y = x @ w.T
    if bias is not None:
        y = y + np.asarray(bias, dtype=np.float64)[None, :]
    return tuple(y[:, t * n:(t + 1) * n].reshape(rows, heads, n // heads) for t in range(3))


def qkv_project_rope(x: np.ndarray, weight: np.ndarray, bias, g: Geometry, chunks):
    """The projection followed by the 3D RoPE of q and k, with no rounding in
    between (the fused projection + RoPE + cache write), fp64.

    x: [n * T][C], node i's token rows at [i*T, (i+1)*T); chunks[i] is node
    i's chunk index (its tokens sit at frames F*chunks[i] + f).  Returns
    (q', k', v), each [n][T][H][d], unrounded: q and k of every head rotated by
    ``rope_head`` at the node's chunk, v as projected.
    """
    n = len(chunks)
    q, k, v = qkv_project(x, weight, bias, heads=g.H)
    shape = (n, g.T, g.H, g.d)
    q, k, v = q.reshape(shape), k.reshape(shape), v.reshape(shape)
    qr, kr = np.empty(shape), np.empty(shape)
    for i, b in enumerate(chunks):
        for h in range(g.H):
            qr[i, :, h] = rope_head(q[i, :, h], b, g)
            kr[i, :, h] = rope_head(k[i, :, h], b, g)
    return qr, kr, v


# ---------------------------------------------------------------- attention

def attend_rows(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float,
                mask: np.ndarray | None = None) -> tuple[np.ndarray, np.ndarray]:
    """Eq. 4: masked softmax attention of rows q[n][d] over k, v [L][d]."""
    q = np.ascontiguousarray(q, dtype=np.float64)
    k = np.ascontiguousarray(k, dtype=np.float64)
    v = np.ascontiguousarray(v, dtype=np.float64)
    n, d = q.shape
    L = k.shape[0]
    assert k.shape == (L, d) and v.shape == (L, d)
    out = np.empty((n, d), dtype=np.float64)
    lse = np.empty((n,), dtype=np.float64)
    mptr = None
    if mask is not None:
        mask = np.ascontiguousarray(mask, dtype=np.float64)
        assert mask.shape == (L,)
        mptr = _pd(mask)
    _load().oracle_attend_rows(_pd(q), _pd(k), _pd(v), mptr, L, d, n, float(scale),
                               _pd(out), _pd(lse))
    return out, lse


def node_forward(g: Geometry, policy: int, W: int, node: tuple[int, int, int],
                 states: dict, q_raw: np.ndarray, heads, rows, scale: float,
                 hidden: frozenset = frozenset(), within: str = "bidirectional",
                 norm=None, tile_mask=None, own_mask=None, hist_mask=None):
    """One denoising node (seq, b, j), computed from raw (pre-RoPE) inputs.

    states: {(seq, chunk, level): (K_raw, V_raw)} with arrays [T][H][d] holding
        bf16 values (any float dtype); the node's own state must be present.
    q_raw: the node's queries [T][H][d].
    heads, rows: the (head, query row) pairs to compute are heads x rows.
    hidden: selected (chunk, level) states whose visibility is 0 (their
        tokens get M = -inf); by default every selected state is visible.
    within: "bidirectional" (every key of the own chunk visible) or
        "frame_causal" (a query of latent frame f sees the own chunk's keys of
        frames <= f only); the token-level mask of Eq. 4 either way.
    norm: None, or (gamma_k, gamma_q, eps): every key state's K and the
        node's Q are RMS-normalised per token (rms_norm) before the rotation.
    tile_mask: None, or a boolean array [query tile][key tile] for the node
        (query-dependent block-sparse access, Eq. 4 at 128-token tiles):
        query u (tile u // 128) sees key v of key state s (0 = own chunk,
        1 + j = j-th selected state) only if entry [u // 128][s * nt + v // 128]
        is true, nt = ceil(T / 128); a further mask on top of the others.
    own_mask: None, or a boolean array [T][T] for the node: query u sees key v
        of its own chunk only if own_mask[u][v] (the general token-level M of
        Eq. 4 inside the chunk); a further mask on top of the others.
    hist_mask: None, or a boolean array [n_sel][T][T] for the node: query u
        sees key token v of the j-th selected state (Eq. 2's offset order, j = 0
        for r = 1) only if hist_mask[j][u][v] (the token-level M of Eq. 4 on
        the history); a further mask on top of the others.

    Steps (Section 3.2): select the context states of the node with Eq. 2-3;
    rotate the K of the node's own state and of every selected state and the
    node's Q with the 3D RoPE reading at each state's chunk position, and
    round to bf16 as the cache and the in-place Q store do (V is stored
    unrotated); then Eq. 4 attention over own + selected keys, with mask 0
    on visible keys and -inf on hidden ones.

    Returns (out [len(heads)][len(rows)][d], lse [len(heads)][len(rows)],
    selected states).
    """
    seq, b, j = node
    sel = select(policy, W, b, j)
    key_states = [(b, j)] + sel
    rows = np.asarray(list(rows), dtype=np.int64)
    out = np.empty((len(heads), len(rows), g.d))
    lse = np.empty((len(heads), len(rows)))
    frame_tokens = g.Hp * g.Wp
    key_frame = np.arange(g.T) // frame_tokens            # latent frame of own-chunk key v
    key_tile = np.arange(g.T) // 128                     # tile of key v inside its state
    nt = -(-g.T // 128)
    if within not in ("frame_causal", "bidirectional"):
        raise ValueError(within)
    # query rows grouped by the mask they get: by latent frame when
    # frame-causal, by query tile under a tile mask
    row_frame = rows // frame_tokens if within == "frame_causal" else np.zeros_like(rows)
    row_tile = rows // 128 if tile_mask is not None else np.zeros_like(rows)
    groups = []
    if own_mask is not None or hist_mask is not None:   # every row its own mask
        for r in range(len(rows)):
            groups.append((row_frame[r] if within == "frame_causal" else None,
                           row_tile[r] if tile_mask is not None else None, np.array([r])))
    else:
        for f in np.unique(row_frame):
            for qt in np.unique(row_tile):
                idx = np.nonzero((row_frame == f) & (row_tile == qt))[0]
                if len(idx):
                    groups.append((f if within == "frame_causal" else None,
                                   qt if tile_mask is not None else None, idx))
    if norm is not None:
        gk, gq, eps = norm
        states = {s: (rms_norm(states[s][0], gk, eps), states[s][1])
                  for s in [(seq, c, lvl) for (c, lvl) in key_states]}
        q_raw = rms_norm(q_raw, gq, eps)
    for hi, h in enumerate(heads):
        ks, vs, ms = [], [], []
        for (c, lvl) in key_states:
            k_raw, v_raw = states[(seq, c, lvl)]
            ks.append(bf16(rope_head(np.asarray(k_raw[:, h, :], dtype=np.float64), c, g)))
            vs.append(np.asarray(v_raw[:, h, :], dtype=np.float64))
            masked = (c, lvl) in hidden and (c, lvl) != (b, j)
            ms.append(np.full(g.T, -np.inf if masked else 0.0))
        k = np.concatenate(ks)
        v = np.concatenate(vs)
        q = bf16(rope_head(np.asarray(q_raw[:, h, :], dtype=np.float64), b, g))[rows]
        for f, qt, idx in groups:
            m = np.concatenate(ms)
            if f is not None:
                m[:g.T] = np.where(key_frame > f, -np.inf, m[:g.T])   # own chunk comes first
            if qt is not None:
                for si in range(len(key_states)):
                    kept = np.asarray(tile_mask[qt][si * nt + key_tile], dtype=bool)
                    m[si * g.T:(si + 1) * g.T] = np.where(kept, m[si * g.T:(si + 1) * g.T], -np.inf)
            if own_mask is not None:
                u = rows[idx[0]]
                m[:g.T] = np.where(np.asarray(own_mask[u], dtype=bool), m[:g.T], -np.inf)
            if hist_mask is not None:
                u = rows[idx[0]]
                for si in range(1, len(key_states)):     # selected state si - 1
                    seg = slice(si * g.T, (si + 1) * g.T)
                    m[seg] = np.where(np.asarray(hist_mask[si - 1][u], dtype=bool), m[seg], -np.inf)
            o, l = attend_rows(q[idx], k, v, scale, m)
            out[hi, idx] = o
            lse[hi, idx] = l
    return out, lse, sel
