"""Dense-mask brute force for tiny inputs (test infrastructure only).

An independent formulation of the same computation as ``oracle.node_forward``,
used to pin it.  Instead of a per-node list of selected states, every
(chunk, level) state present in the grid contributes its T tokens to ONE
global key sequence, and the token-level mask of Eq. 4 (Section 3.2) is built
densely over it from a visibility predicate written directly from Eq. 2-3:
key token v of state (c, l) is visible to a query of node (b, j) iff
(c, l) == (b, j) (the node's own chunk, bidirectional inside the chunk), or
1 <= b - c <= min(W, b - 1) and l equals the policy's level for offset
b - c.  Everything else, including future chunks and other levels of past
chunks, gets -inf.  RoPE and the bf16 rounding are re-implemented here with
numpy and Python's ``math`` module; nothing is shared with ``sva_oracle.c``.
Intended for T x (number of states) up to a few thousand tokens.
"""
from __future__ import annotations

import math

import numpy as np


def _policy_level(policy: str, j: int, r: int) -> int:
    if policy == "clean":
        return 0
    if policy == "same":
        return j
    if policy == "prog":
        return max(j - r, 0)
    raise ValueError(policy)


def visible(policy: str, W: int, query_state: tuple[int, int], key_state: tuple[int, int]) -> bool:
    b, j = query_state
    c, l = key_state
    if (c, l) == (b, j):
        return True
    r = b - c
    return 1 <= r <= min(W, b - 1) and l == _policy_level(policy, j, r)


def _bf16(x: float) -> float:
    if x == 0.0 or not math.isfinite(x):
        return x
    m, e = math.frexp(x)          # x = m * 2^e, 0.5 <= |m| < 1
    e = max(e, -125)              # bf16 normal exponents stop at 2^-126
    scaled = x * 2.0 ** (8 - e)   # 8 significant bits before the point
    return round(scaled) * 2.0 ** (e - 8)   # round() is ties-to-even


_bf16_vec = np.vectorize(_bf16, otypes=[np.float64])


def _rope(x: np.ndarray, chunk: int, F: int, Hp: int, Wp: int, pairs, theta: float) -> np.ndarray:
    """x: [T][d] -> rotated copy (pairs of adjacent elements turn by pos * theta^(-i/P))."""
    T, d = x.shape
    u = np.arange(T)
    pos = [F * chunk + u // (Hp * Wp), (u // Wp) % Hp, u % Wp]
    y = x.copy()
    col = 0
    for axis, npairs in enumerate(pairs):
        for i in range(npairs):
            ang = pos[axis] * theta ** (-i / npairs)
            c, s = np.cos(ang), np.sin(ang)
            a, bb = x[:, col], x[:, col + 1]
            y[:, col] = a * c - bb * s
            y[:, col + 1] = a * s + bb * c
            col += 2
    return y


def brute_forward(policy: str, W: int, F: int, Hp: int, Wp: int, pairs, theta: float,
                  node: tuple[int, int, int], grid: dict, q_raw: np.ndarray,
                  heads, scale: float, hidden=frozenset(), frame_causal: bool = False,
                  tile_mask=None, own_mask=None, hist_mask=None):
    """All query rows of `heads` for node (seq, b, j) against the whole grid.

    grid: {(seq, chunk, level): (K_raw, V_raw)} [T][H][d]; it may hold states
    the node must NOT see (other levels, future chunks, other sequences).
    hidden: states whose visibility bit is 0 although the policy selects them.
    frame_causal: inside the own chunk, query token u sees key token v only if
    v's latent frame is not after u's.
    tile_mask: None, or booleans [query tile][key tile]: query u sees key
    token v of state (c, l) only if entry [u // 128][r * nt + v // 128] is
    set, r = b - c (the offset of Eq. 2; 0 for the own chunk), nt = ceil(T/128).
    own_mask: None, or booleans [T][T]: query u sees key token v of its own
    chunk only if own_mask[u][v].
    hist_mask: None, or booleans [n][T][T]: query u sees key token v of state
    (c, l) with r = b - c >= 1 only if hist_mask[r - 1][u][v] (past the
    window the state is masked anyway).
    Returns (out [len(heads)][T][d], lse [len(heads)][T]).
    """
    seq, b, j = node
    keys = sorted(grid)
    T = q_raw.shape[0]
    d = q_raw.shape[2]
    outs, lses = [], []
    for h in heads:
        kk, vv, mm = [], [], []
        for (s, c, l) in keys:
            k_raw, v_raw = grid[(s, c, l)]
            kk.append(_bf16_vec(_rope(np.asarray(k_raw[:, h, :], np.float64), c, F, Hp, Wp, pairs, theta)))
            vv.append(np.asarray(v_raw[:, h, :], np.float64))
            ok = (s == seq) and visible(policy, W, (b, j), (c, l))
            if ok and (c, l) in hidden and (c, l) != (b, j):
                ok = False
            mm.append(np.full(T, 0.0 if ok else -np.inf))
        K = np.concatenate(kk)
        V = np.concatenate(vv)
        M = np.concatenate(mm)
        Q = _bf16_vec(_rope(np.asarray(q_raw[:, h, :], np.float64), b, F, Hp, Wp, pairs, theta))
        own_start = keys.index((seq, b, j)) * T       # where the own chunk sits in the sequence
        nt = -(-T // 128)
        out = np.zeros((T, d))
        lse = np.zeros(T)
        for u in range(T):
            Mu = M.copy()
            if frame_causal:
                for v in range(T):
                    if v // (Hp * Wp) > u // (Hp * Wp):
                        Mu[own_start + v] = -np.inf
            if own_mask is not None:
                for v in range(T):
                    if not own_mask[u][v]:
                        Mu[own_start + v] = -np.inf
            if hist_mask is not None:
                for ki, (s, c, l) in enumerate(keys):
                    r = b - c
                    if s != seq or r < 1 or r > len(hist_mask):
                        continue   # the own chunk, other sequences, future and far chunks
                    for v in range(T):
                        if not hist_mask[r - 1][u][v]:
                            Mu[ki * T + v] = -np.inf
            if tile_mask is not None:
                for ki, (s, c, l) in enumerate(keys):
                    if s != seq or not (0 <= b - c) or (b - c) * nt >= len(tile_mask[0]):
                        continue   # other sequences, future and far chunks: masked anyway
                    for v in range(T):
                        if not tile_mask[u // 128][(b - c) * nt + v // 128]:
                            Mu[ki * T + v] = -np.inf
            logits = [scale * float(np.dot(Q[u], K[v])) + Mu[v] for v in range(K.shape[0])]
            mx = max(logits)
            w = [math.exp(x - mx) if x != -math.inf else 0.0 for x in logits]
            z = math.fsum(w)
            out[u] = sum(wi * V[v] for v, wi in enumerate(w) if wi != 0.0) / z
            lse[u] = mx + math.log(z)
        outs.append(out)
        lses.append(lse)
    return np.stack(outs), np.stack(lses)
