"""Shared helpers of the GPU parity tests: run a workload's step on the GPU
through the C ABI, and compute the same outputs with the fp64 oracle.

Tolerance of the attention output against the fp64 oracle (bf16 inputs,
fp32 accumulation, bf16 P and bf16 output), per element:

    |O_gpu - O_ref| <= 2e-2 + ulp_bf16(|O_ref|) / 2

that is the 2e-2 bound plus the rounding of the output itself to the bf16
grid, which alone exceeds 2e-2 once |O| >= 8 (the x10 outliers of
stress14b reach that).  The one other error of the kernel that can grow with
the values is the rounding of the probabilities P to bf16 before the PV
product: |bf16(p) - p| <= 2^-8 p, so that term is at most
2^-8 * sum_v p_v |v_v| / sum_v p_v = 2^-8 * E_p|V|, which the oracle
computes exactly as the attention output over |V|.  An element above the
first bound passes if it is within that bound plus 2^-8 * E_p|V|; such
elements are counted and reported.  Relative RMS <= 5e-3 per (node, head).
"""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle
from paper_2609_22283_gb300 import inputs as I

MAX_ABS = 2e-2
REL_RMS = 5e-3
P_ROUND = 2.0 ** -8   # relative rounding error of P to bf16 (8 significant bits)
# LSE (natural log): |d| <= 2e-3 + 2^-10 |LSE|.  The LSE moves with the
# logits, whose error scales with their magnitude: the rotated Q and K the
# kernel reads may differ from the oracle's correctly rounded values by one
# bf16 ulp (the fp32 rotation lands on the other side of a rounding
# boundary in about 0.1% of the elements), which shifts every logit of a row
# in proportion to the values involved (x10 outliers make that visible).
LSE_ABS = 2e-3
LSE_REL = 2.0 ** -10


def ulp_bf16(x):
    """Spacing of the bf16 grid at |x| (normal range; 2^-133 at 0)."""
    x = np.abs(np.asarray(x, dtype=np.float64))
    e = np.floor(np.log2(np.where(x > 0, x, 1.0)))
    return np.where(x > 0, 2.0 ** (np.maximum(e, -126) - 7), 2.0 ** -133)


def oracle_geometry(w: I.Workload) -> oracle.Geometry:
    return oracle.Geometry(F=w.F, Hp=w.Hp, Wp=w.Wp, H=w.H, d=w.d, pairs=w.pairs, theta=w.theta)


def oracle_states(w: I.Workload, inp: I.Inputs) -> dict:
    """Every state as fp32 arrays [T][H][d] (bf16 values exactly; the oracle
    widens the head it reads to fp64)."""
    return {k: (a.float().numpy(), b.float().numpy())
            for k, (a, b) in I.all_states(w, inp).items()}


def abs_v_states(states: dict) -> dict:
    """The same states with V replaced by |V|: the oracle's attention output
    over them is E_p|V| per element."""
    return {k: (a, np.abs(b)) for k, (a, b) in states.items()}


def oracle_masks(w: I.Workload, mask=None) -> np.ndarray:
    """The workload's block mask (or `mask`, int32 words) as booleans [node][qt][key tile]."""
    m = I.tile_mask(w) if mask is None else mask.cpu()
    return I.unpack_bits(m, (1 + w.W) * w.tiles).numpy()


def oracle_node(w, inp, states, node_index, heads, rows, hidden=frozenset(), tile_mask=None,
                own_mask=None, hist_mask=None):
    g = oracle_geometry(w)
    q = inp.q[node_index].float().numpy()
    out, lse, _ = oracle.node_forward(g, oracle.POLICY_IDS[w.policy], w.W, w.nodes[node_index],
                                      states, q, list(heads), list(rows), 1.0 / math.sqrt(w.d),
                                      hidden=hidden, within=w.within, tile_mask=tile_mask,
                                      own_mask=own_mask, hist_mask=hist_mask,
                                      norm=((inp.gamma_k.double().numpy(), inp.gamma_q.double().numpy(),
                                             inp.norm_eps) if w.qknorm else None))
    return out, lse


def gpu_step(w: I.Workload, inp: I.Inputs, lse: bool = True):
    """Runs one step; returns (step, q_rot, out, lse) with device tensors."""
    from paper_2609_22283_gb300.pipeline import Step
    step = Step(w)
    step.prefill(inp)
    q, k, v = step.device_inputs(inp)
    out, l = step.outputs()
    step.run(q, k, v, out, l if lse else None)
    st = step.cache.poll()
    assert st == 0, f"device status {st}"
    torch.cuda.synchronize()
    return step, q, out, (l if lse else None)


def boundary_rows(w: I.Workload) -> list:
    """Query rows at the tile edges and the chunk's ends (the first and last
    rows of the first two query tiles, of the last full pair, of the ragged
    last tile)."""
    T = w.T
    cand = {0, 1, 63, 64, 127, 128, 255, 256, T - 73, T - 72, T - 1, 4607, 4608, 4679}
    return sorted(c for c in cand if 0 <= c < T)


def rows_per_head(w: I.Workload, per_node: int, seed: int) -> dict:
    """{head: sorted query rows}: about per_node seeded rows of a node spread
    over all its heads (a different draw per head), plus every boundary row
    of every head."""
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    k = -(-per_node // w.H)
    edges = set(boundary_rows(w))
    return {h: sorted(edges | set(torch.randperm(w.T, generator=g)[:k].tolist()))
            for h in range(w.H)}


class Stats:
    """Worst figures over the checks of one test, for the report."""

    def __init__(self):
        self.raw = 0.0        # largest |O_gpu - O_ref|
        self.at = 0.0         # |O_ref| there
        self.margin = 0.0     # largest |O_gpu - O_ref| - ulp_bf16(|O_ref|) / 2
        self.rel_rms = 0.0
        self.allowed = 0      # elements that needed the P-rounding allowance
        self.elements = 0
        self.lse = 0.0        # largest |LSE_gpu - LSE_ref|
        self.lse_at = 0.0     # |LSE_ref| there

    def __str__(self):
        return (f"raw max |d| {self.raw:.3e} at |O| {self.at:.3g}; max |d| - ulp/2 "
                f"{self.margin:.3e} (bound 2e-2); rel_rms {self.rel_rms:.2e}; "
                f"{self.allowed} of {self.elements} elements within the P-rounding allowance; "
                f"LSE max |d| {self.lse:.2e} at |LSE| {self.lse_at:.3g}")


def assert_lse(got, ref, what="", stats: Stats | None = None):
    """LSE rows against the oracle: |d| <= LSE_ABS + LSE_REL |LSE_ref|."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    ad = np.abs(got - ref)
    i = int(np.argmax(ad))
    if stats is not None and ad.flat[i] > stats.lse:
        stats.lse, stats.lse_at = float(ad.flat[i]), float(abs(ref.flat[i]))
    bad = ad > LSE_ABS + LSE_REL * np.abs(ref)
    assert not bad.any(), (f"{what}: LSE |d| {ad.flat[i]:.3e} at {ref.flat[i]:.4f} "
                           f"({int(bad.sum())} beyond 2e-3 + 2^-10 |LSE|)")


def errors(got: np.ndarray, ref: np.ndarray):
    """(max |d| - ulp(|ref|)/2, relative RMS, raw max |d|, |ref| at the raw max)."""
    diff = got.astype(np.float64) - ref
    ad = np.abs(diff)
    margin = float(np.max(ad - 0.5 * ulp_bf16(ref)))
    rel_rms = float(np.linalg.norm(diff) / max(np.linalg.norm(ref), 1e-300))
    at = np.unravel_index(int(np.argmax(ad)), ad.shape)
    return margin, rel_rms, float(ad[at]), float(abs(ref[at]))


def assert_close(got, ref, what="", p_abs=None, stats: Stats | None = None):
    """got, ref: [rows][d] of one (node, head).  p_abs: None, or a callable
    taking row indices into `ref` and returning the oracle's E_p|V| for those
    rows ([len][d]); without it no element may use the P-rounding allowance."""
    got = np.asarray(got, dtype=np.float64)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    ad = np.abs(got - ref)
    bound = MAX_ABS + 0.5 * ulp_bf16(ref)
    viol = ad > bound
    allowed = 0
    if viol.any() and p_abs is not None:
        rows = np.unique(np.nonzero(viol)[0])
        extra = P_ROUND * np.asarray(p_abs(rows))
        still = ad[rows] > bound[rows] + extra
        allowed = int(viol[rows].sum() - (viol[rows] & still).sum())
        viol = np.zeros_like(viol)
        viol[rows] = still
    margin, rr, raw, mag = errors(got, ref)
    if stats is not None:
        if raw > stats.raw:
            stats.raw, stats.at = raw, mag
        stats.margin = max(stats.margin, margin)
        stats.rel_rms = max(stats.rel_rms, rr)
        stats.allowed += allowed
        stats.elements += got.size
    assert not viol.any(), (
        f"{what}: {int(viol.sum())} elements above 2e-2 + ulp/2 (raw max {raw:.3e} at |O| = "
        f"{mag:.3g}, max |d| - ulp/2 {margin:.3e})")
    assert rr <= REL_RMS, f"{what}: rel_rms {rr:.3e}"
    return margin, rr
