"""Workload descriptions and seeded synthetic inputs.

This module is the only code the CUDA path and the CPU oracle share.  It
holds data and random numbers, none of the method's arithmetic: no context
selection, no RoPE, no attention.  Each workload lists its nodes and the
states already in the cache as plain data (derived by hand from the
progressive, same-level and clean rules of Eq. 3 and written out here); the
library and the oracle each derive the context lists themselves.

Synthetic inputs stand in for the paper's video latents (Wan2.1 geometry,
832x480 at 16 FPS, 3-latent-frame chunks, Section 4 and Appendix A): every
tensor is drawn from a seeded torch CPU generator as N(0, 1) fp32 and rounded
to bf16, in this order: for each prefilled state (in the listed order) its K
then its V [T][H][d]; then Q, K_new and V_new [n_nodes][T][H][d].  With
`outliers`, each draw is followed by a U(0, 1) draw of the same shape on the
same generator and elements whose uniform is below 0.01 are multiplied by 10.

Block-sparse workloads (`sparse` = a density) also get a seeded key-tile mask
per (node, query tile), see `tile_mask`.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import torch


def rope_pairs_for(d: int) -> tuple[int, int, int]:
    """Head-dimension pairs given to the t, h and w axes: h and w get
    floor(d/6) pairs each, t the rest (22/21/21 for d = 128, 12/10/10 for 64)."""
    hw = d // 6
    return (d // 2 - 2 * hw, hw, hw)


@dataclass(frozen=True)
class Workload:
    name: str
    seed: int
    F: int            # latent frames per chunk
    Hp: int           # patch rows per frame
    Wp: int           # patch columns per frame
    H: int            # attention heads
    d: int            # head dim
    K: int            # denoising levels (node levels 1..K, clean level 0)
    W: int            # history window in chunks
    policy: str       # "clean" | "same" | "prog"
    nodes: tuple      # ((seq, chunk, level), ...) processed by the step
    prefilled: tuple  # ((seq, chunk, level), ...) states cached before the step
    outliers: bool = False
    B: int = 40       # chunks in the video (pipeline length, Eq. 6)
    round: int | None = None  # pipeline round the nodes form (Eq. 6), if any
    within: str = "bidirectional"  # visibility inside the own chunk (or "frame_causal")
    qknorm: bool = False  # RMS-normalise K and Q per token before RoPE (seeded gammas)
    sparse: float | None = None  # density of kept context key tiles (block-sparse mask), or None
    sparse_rows: int = 1  # consecutive query tiles sharing one mask row (draws per group)
    description: str = ""
    theta: float = 10000.0
    pairs: tuple = field(default=None)

    def __post_init__(self):
        if self.pairs is None:
            object.__setattr__(self, "pairs", rope_pairs_for(self.d))

    @property
    def T(self) -> int:
        return self.F * self.Hp * self.Wp

    @property
    def n_nodes(self) -> int:
        return len(self.nodes)

    @property
    def states(self) -> tuple:
        """Every state the step touches: prefilled ones, then the nodes' own."""
        return tuple(self.prefilled) + tuple(self.nodes)

    @property
    def tiles(self) -> int:
        """128-token tiles per chunk (query tiles of a node, key tiles of a state)."""
        return -(-self.T // 128)

    @property
    def mask_words(self) -> int:
        """32-bit words per (node, query tile) row of `tile_mask`: room for the own
        state and up to W context states."""
        return -(-(1 + self.W) * self.tiles // 32)

    @property
    def max_frames(self) -> int:
        last = max(c for (_, c, _) in self.states)
        return self.F * (last + 1) + self.F


def _round_nodes(seq: int, K: int, n: int):
    # written out by hand: chunk n - K + j at level j, for j = K .. 1 (Eq. 6)
    return tuple((seq, n - K + j, j) for j in range(K, 0, -1))


_PROG_PREFILL_20 = tuple((0, c, 0) for c in range(11, 17))      # chunks 11..16, clean
_SAME_PREFILL_20 = tuple((0, b - r, j) for (_, b, j) in _round_nodes(0, 4, 20) for r in (1, 2, 3))

WORKLOADS = {
    "tiny": Workload(
        name="tiny", seed=0, F=1, Hp=8, Wp=8, H=2, d=64, K=2, W=2, policy="prog",
        nodes=((0, 3, 2), (0, 2, 1)), prefilled=((0, 1, 0),), B=3, round=3,
        description="3 chunks x 64 tokens (1 latent frame of 8x8), K=2, 2 nodes (3,2),(2,1) "
                    "batched, 2 heads x 64, progressive history, W=2"),
    "clean1": Workload(
        name="clean1", seed=1, F=3, Hp=30, Wp=52, H=12, d=128, K=4, W=3, policy="clean",
        nodes=((0, 20, 4),), prefilled=((0, 17, 0), (0, 18, 0), (0, 19, 0)),
        description="1 node (20,4), clean history W=3: 4680 queries x 12 heads x 128 over "
                    "4680 own + 3x4680 clean history keys (Lkv 18720)"),
    "same4": Workload(
        name="same4", seed=2, F=3, Hp=30, Wp=52, H=12, d=128, K=4, W=3, policy="same",
        nodes=_round_nodes(0, 4, 20), prefilled=_SAME_PREFILL_20, round=20,
        description="round 20 of a K=4 pipeline: nodes (20,4),(19,3),(18,2),(17,1), same-level "
                    "history W=3 (Lkv 18720), 12 heads x 128"),
    "prog4": Workload(
        name="prog4", seed=3, F=3, Hp=30, Wp=52, H=12, d=128, K=4, W=6, policy="prog",
        nodes=_round_nodes(0, 4, 20), prefilled=_PROG_PREFILL_20, round=20,
        description="round 20 of a K=4 pipeline: nodes (20,4),(19,3),(18,2),(17,1), progressive "
                    "history W=6 (7-chunk window, Lkv 32760), in-round reads, 12 heads x 128"),
    "prog4r": Workload(
        name="prog4r", seed=5, F=3, Hp=30, Wp=52, H=12, d=128, K=4, W=6, policy="prog",
        nodes=_round_nodes(0, 4, 20) + ((0, 16, 0),),
        prefilled=tuple((0, c, 0) for c in range(10, 16)), round=20,
        description="round 20 of a K=4 progressive pipeline with the clean-state KV refresh of "
                    "chunk 16 (level 0) in the same launch: 5 nodes, W=6, nodes (17,1) and "
                    "(20,4) read the refreshed (16,0) in-round, 12 heads x 128"),
    "clean5": Workload(
        name="clean5", seed=6, F=3, Hp=30, Wp=52, H=12, d=128, K=4, W=6, policy="clean",
        nodes=tuple((0, 20, j) for j in range(4, -1, -1)),
        prefilled=tuple((0, c, 0) for c in range(14, 20)),
        description="fully serial execution of chunk 20 (Eq. 5): its 4 denoising updates and "
                    "its clean-state refresh, each a separate one-node launch over 6 clean "
                    "history chunks (Lkv 32760), 12 heads x 128"),
    "tinyfc": Workload(
        name="tinyfc", seed=7, F=3, Hp=4, Wp=8, H=2, d=64, K=2, W=2, policy="prog",
        nodes=((0, 3, 2), (0, 2, 1)), prefilled=((0, 1, 0),), B=3, round=3,
        within="frame_causal",
        description="tiny with 3 latent frames of 4x8 tokens per chunk (T=96) and a "
                    "frame-causal mask inside each own chunk"),
    "tinyn": Workload(
        name="tinyn", seed=10, F=1, Hp=8, Wp=8, H=2, d=64, K=2, W=2, policy="prog",
        nodes=((0, 3, 2), (0, 2, 1)), prefilled=((0, 1, 0),), B=3, round=3, qknorm=True,
        description="tiny with K and Q RMS-normalised per token before RoPE"),
    "tinys": Workload(
        name="tinys", seed=11, F=1, Hp=16, Wp=20, H=2, d=64, K=2, W=2, policy="prog",
        nodes=((0, 3, 2), (0, 2, 1)), prefilled=((0, 1, 0),), B=3, round=3, sparse=0.5,
        description="tiny with 320-token chunks (3 key tiles, the last 64 rows) and a seeded "
                    "block-sparse mask keeping half of the context key tiles per query tile"),
    "prog4s": Workload(
        name="prog4s", seed=9, F=3, Hp=30, Wp=52, H=12, d=128, K=4, W=6, policy="prog",
        nodes=_round_nodes(0, 4, 20), prefilled=_PROG_PREFILL_20, round=20, sparse=0.5,
        sparse_rows=2,
        description="prog4 with query-dependent block-sparse access: every 256-query block keeps "
                    "its own chunk and a seeded half of the 128-token key tiles of its history"),
    "prog4fc": Workload(
        name="prog4fc", seed=8, F=3, Hp=30, Wp=52, H=12, d=128, K=4, W=6, policy="prog",
        nodes=_round_nodes(0, 4, 20), prefilled=_PROG_PREFILL_20, round=20,
        within="frame_causal",
        description="prog4 with a frame-causal mask inside each own chunk (frames of 1560 "
                    "tokens, boundaries inside 128-token tiles)"),
    "stress14b": Workload(
        name="stress14b", seed=4, F=3, Hp=30, Wp=52, H=40, d=128, K=4, W=6, policy="prog",
        nodes=_round_nodes(0, 4, 20) + _round_nodes(1, 4, 20),
        prefilled=_PROG_PREFILL_20 + tuple((1, c, l) for (_, c, l) in _PROG_PREFILL_20),
        outliers=True, round=20,
        description="2 video streams x the prog4 round: 8 nodes, 40 heads x 128, Lkv 32760, "
                    "N(0,1) with 1% x10 outliers"),
}

# The order the workloads are listed in the configuration table; prog4r adds
# the clean-state refresh node to prog4's round.
ORDER = ("tiny", "clean1", "same4", "prog4", "stress14b")
EXTRA = ("prog4r", "clean5", "tinyfc", "prog4fc", "tinyn", "tinys", "prog4s")


@dataclass
class Inputs:
    history: dict      # {(seq, chunk, level): (K_raw, V_raw)} bf16 [T][H][d]
    q: torch.Tensor    # bf16 [n][T][H][d]
    k_new: torch.Tensor
    v_new: torch.Tensor
    gamma_k: torch.Tensor | None = None   # fp32 [H*d], with qknorm
    gamma_q: torch.Tensor | None = None
    norm_eps: float = 1e-6


def generate(w: Workload) -> Inputs:
    g = torch.Generator(device="cpu")
    g.manual_seed(w.seed)

    def draw(shape):
        x = torch.randn(shape, generator=g, dtype=torch.float32)
        if w.outliers:
            u = torch.rand(shape, generator=g, dtype=torch.float32)
            x = torch.where(u < 0.01, x * 10.0, x)
        return x.to(torch.bfloat16)

    T, H, d, n = w.T, w.H, w.d, w.n_nodes
    history = {}
    for s in w.prefilled:
        k = draw((T, H, d))
        v = draw((T, H, d))
        history[tuple(s)] = (k, v)
    q = draw((n, T, H, d))
    k_new = draw((n, T, H, d))
    v_new = draw((n, T, H, d))
    inp = Inputs(history, q, k_new, v_new)
    if w.qknorm:   # drawn last, so the other tensors match the unnormalised workload
        inp.gamma_k = torch.rand(H * d, generator=g, dtype=torch.float32) + 0.5
        inp.gamma_q = torch.rand(H * d, generator=g, dtype=torch.float32) + 0.5
    return inp


def tile_mask(w: Workload, density: float | None = None, seed: int | None = None) -> torch.Tensor:
    """Seeded block mask, int32 [n_nodes][tiles][mask_words] (32-bit words of bits).

    Bit k of row (node, query tile) is key tile k % tiles of the node's state
    k // tiles: state 0 is the node's own chunk, state 1 + j its j-th context
    state in selection order.  The own chunk's tiles are always kept; every
    other bit is kept when a U(0, 1) draw (one per bit, in row-major order, on
    a generator seeded with `seed`, default the workload's seed + 1000) is
    below `density` (default the workload's).  With `sparse_rows` = r > 1 the
    draws are made for groups of r consecutive query tiles, which share one
    row.  Bits past a node's actual context count are drawn too and ignored.
    """
    density = w.sparse if density is None else density
    if density is None:
        raise ValueError(f"workload {w.name} has no sparse density")
    g = torch.Generator(device="cpu")
    g.manual_seed(w.seed + 1000 if seed is None else seed)
    nt = w.tiles
    nbits = (1 + w.W) * nt
    r = w.sparse_rows
    groups = -(-nt // r)
    keep = torch.rand((w.n_nodes, groups, nbits), generator=g, dtype=torch.float32) < density
    keep = keep.repeat_interleave(r, dim=1)[:, :nt]
    keep[:, :, :nt] = True
    return pack_bits(keep, w.mask_words)


def own_mask(w: Workload, density: float, seed: int | None = None) -> torch.Tensor:
    """Seeded token-level visibility inside each node's own chunk, int32
    [n_nodes][T][ceil(T/32)] words: bit v of row (node, u) is kept when a
    U(0, 1) draw (one per bit, row-major, on a generator seeded with `seed`,
    default the workload's seed + 3000) is below `density`; the diagonal
    (u sees itself) is always kept."""
    g = torch.Generator(device="cpu")
    g.manual_seed(w.seed + 3000 if seed is None else seed)
    keep = torch.rand((w.n_nodes, w.T, w.T), generator=g, dtype=torch.float32) < density
    idx = torch.arange(w.T)
    keep[:, idx, idx] = True
    return pack_bits(keep, -(-w.T // 32))


def _splitmix64(x):
    """splitmix64 (Steele, Lea and Flood, 2014) of uint64 numpy values."""
    import numpy as np
    x = (x + np.uint64(0x9E3779B97F4A7C15)) & np.uint64(0xFFFFFFFFFFFFFFFF)
    z = x
    z = ((z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)) & np.uint64(0xFFFFFFFFFFFFFFFF)
    z = ((z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)) & np.uint64(0xFFFFFFFFFFFFFFFF)
    return z ^ (z >> np.uint64(31))


def hist_mask(w: Workload, density: float, seed: int | None = None) -> torch.Tensor:
    """Seeded token-level visibility of the history, int32
    [n_nodes][T][W][ceil(T/32)] words: bit v of row (node i, query u,
    context j) is kept when a counter-based uniform, splitmix64 of the index
    (((seed * n + i) * W + j) * T + u) * T + v scaled to [0, 1), is below
    `density` (default seed: the workload's seed + 4000); row 7 of every
    node sees no history key.  Context j is the node's j-th selected state;
    rows past a node's context count are drawn too and ignored.  Counter
    based, so a large workload's mask needs no stream of draws."""
    import numpy as np
    seed = w.seed + 4000 if seed is None else seed
    T, W, n = w.T, w.W, w.n_nodes
    words = -(-T // 32)
    out = np.empty((n, T, W, words), dtype="<i4")
    v = np.arange(T, dtype=np.uint64)
    u = np.arange(T, dtype=np.uint64)[:, None]
    cut = np.uint64(int(density * 2.0 ** 64) if density < 1.0 else 2 ** 64 - 1)
    for i in range(n):
        for j in range(W):
            base = np.uint64((((seed * n + i) * W + j) * T) * T)
            keep = _splitmix64(base + u * np.uint64(T) + v[None, :]) < cut
            if density >= 1.0:
                keep[:] = True
            keep[7 % T, :] = False
            out[i, :, j, :] = pack_bits(keep, words).numpy()
    return torch.from_numpy(out)


def pack_bits(keep: torch.Tensor, words: int) -> torch.Tensor:
    """bool [..., nbits] -> int32 [..., words], bit k in word k // 32 at position k % 32."""
    import numpy as np
    k = np.ascontiguousarray(keep.numpy() if isinstance(keep, torch.Tensor) else keep, dtype=bool)
    pad = words * 32 - k.shape[-1]
    if pad:
        k = np.concatenate([k, np.zeros(k.shape[:-1] + (pad,), dtype=bool)], axis=-1)
    b = np.packbits(k, axis=-1, bitorder="little")            # bytes, little-endian bit order
    return torch.from_numpy(np.ascontiguousarray(b).view("<i4").copy())


def unpack_bits(words: torch.Tensor, nbits: int) -> torch.Tensor:
    """int32 [..., words] -> bool [..., nbits] (inverse of pack_bits)."""
    import numpy as np
    w = np.ascontiguousarray(words.numpy()).astype("<i4", copy=False)
    b = np.unpackbits(w.view(np.uint8), axis=-1, bitorder="little")
    return torch.from_numpy(b[..., :nbits].astype(bool))


def projection_inputs(w: Workload, in_features: int, seed: int | None = None):
    """Seeded inputs of the QKV projection of a workload's nodes:
    x [n_nodes][T][in_features] bf16 ~ N(0, 1); weight [3*H*d][in_features]
    bf16 ~ N(0, 1/in_features) (rows: q's outputs, then k's, then v's); bias
    [3*H*d] fp32 ~ N(0, 0.1^2); drawn in that order on a generator seeded with
    `seed` (default the workload's seed + 2000).  Random weights stand in for
    trained ones: the projection's cost and numerics do not depend on them."""
    g = torch.Generator(device="cpu")
    g.manual_seed(w.seed + 2000 if seed is None else seed)
    n_out = 3 * w.H * w.d
    x = torch.randn((w.n_nodes, w.T, in_features), generator=g, dtype=torch.float32)
    wt = torch.randn((n_out, in_features), generator=g, dtype=torch.float32) / in_features ** 0.5
    bias = torch.randn((n_out,), generator=g, dtype=torch.float32) * 0.1
    return x.to(torch.bfloat16), wt.to(torch.bfloat16), bias


def all_states(w: Workload, inp: Inputs) -> dict:
    """{(seq, chunk, level): (K_raw, V_raw)} for prefilled states and nodes' own states."""
    st = dict(inp.history)
    for i, s in enumerate(w.nodes):
        st[tuple(s)] = (inp.k_new[i], inp.v_new[i])
    return st


def sample_rows(w: Workload, count: int, seed: int = 1234):
    """Seeded query rows for sampled parity, always including the tile edges."""
    T = w.T
    edges = sorted({0, 1, 63, 64, 127, 128, T - 73, T - 72, T - 1} & set(range(T)))
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    extra = torch.randperm(T, generator=g)[:count].tolist()
    return sorted(set(edges) | set(extra))
