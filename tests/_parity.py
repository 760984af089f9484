"""Shared helpers of the GPU parity tests: run a workload's step on the GPU
through the C ABI, and compute the same outputs with the fp64 oracle."""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle
from paper_2609_22283_gb300 import inputs as I

# Tolerances of the attention output against the fp64 oracle (bf16 inputs,
# fp32 accumulation, bf16 P and bf16 output): an element-wise bound of 2e-2
# on outputs of magnitude <= 1, scaled by |O| above 1 (the bf16 output grid
# alone is coarser than 2e-2 once |O| >= 8), and a relative RMS of 5e-3.
MAX_ABS = 2e-2
REL_RMS = 5e-3


def oracle_geometry(w: I.Workload) -> oracle.Geometry:
    return oracle.Geometry(F=w.F, Hp=w.Hp, Wp=w.Wp, H=w.H, d=w.d, pairs=w.pairs, theta=w.theta)


def oracle_states(w: I.Workload, inp: I.Inputs) -> dict:
    return {k: (a.to(torch.float64).numpy(), b.to(torch.float64).numpy())
            for k, (a, b) in I.all_states(w, inp).items()}


def oracle_masks(w: I.Workload, mask=None) -> np.ndarray:
    """The workload's block mask (or `mask`, int32 words) as booleans [node][qt][key tile]."""
    m = I.tile_mask(w) if mask is None else mask.cpu()
    return I.unpack_bits(m, (1 + w.W) * w.tiles).numpy()


def oracle_node(w, inp, states, node_index, heads, rows, hidden=frozenset(), tile_mask=None,
                own_mask=None):
    g = oracle_geometry(w)
    q = inp.q[node_index].to(torch.float64).numpy()
    out, lse, _ = oracle.node_forward(g, oracle.POLICY_IDS[w.policy], w.W, w.nodes[node_index],
                                      states, q, list(heads), list(rows), 1.0 / math.sqrt(w.d),
                                      hidden=hidden, within=w.within, tile_mask=tile_mask,
                                      own_mask=own_mask,
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


def errors(got: np.ndarray, ref: np.ndarray):
    """(max |d| / max(1, |ref|), relative RMS, raw max |d|, |ref| at the raw max)."""
    diff = got.astype(np.float64) - ref
    ad = np.abs(diff)
    scaled = float(np.max(ad / np.maximum(1.0, np.abs(ref))))
    rel_rms = float(np.linalg.norm(diff) / max(np.linalg.norm(ref), 1e-300))
    at = np.unravel_index(int(np.argmax(ad)), ad.shape)
    return scaled, rel_rms, float(ad[at]), float(abs(ref[at]))


def assert_close(got, ref, what=""):
    ma, rr, raw, mag = errors(got, ref)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    assert ma <= MAX_ABS and rr <= REL_RMS, (
        f"{what}: scaled max_abs {ma:.3e} (raw {raw:.3e} at |O| = {mag:.3g}) rel_rms {rr:.3e}")
    return ma, rr
