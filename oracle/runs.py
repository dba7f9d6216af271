"""Plain drivers over the C oracle: prefix, calibration and decode trajectories.

Test infrastructure only.  Each driver loops over steps in order and calls the
per-head oracle functions; batch rows and value heads are flattened to
independent heads ("units") with the GQA rule value head h -> q/k head
floor(h * H_qk / H).
"""
from __future__ import annotations

import numpy as np

import workloads as wl

from . import calibrate, core


def unit_operands(w: wl.Workload, inp: dict, heads=None) -> dict:
    """Flatten step operands of R batch rows to per-unit arrays for the given value heads.

    Returns q, k [R*Hs, d_k], v [R*Hs, d_v], beta [R*Hs], g [R*Hs] or [R*Hs, d_k]
    in (row, head) order.
    """
    heads = list(range(w.heads)) if heads is None else list(heads)
    qk = [wl.qk_head_of(w, h) for h in heads]
    R = inp["v"].shape[0]
    out = {
        "q": inp["q"][:, qk].reshape(R * len(heads), w.d_k),
        "k": inp["k"][:, qk].reshape(R * len(heads), w.d_k),
        "v": inp["v"][:, heads].reshape(R * len(heads), w.d_v),
        "beta": inp["beta"][:, heads].reshape(R * len(heads)),
    }
    if w.kind == "gdn":
        out["g"] = inp["g"][:, heads].reshape(R * len(heads))
    else:
        out["g"] = inp["g"][:, heads].reshape(R * len(heads), w.d_k)
    return {k: np.ascontiguousarray(v, dtype=np.float32) for k, v in out.items()}


def prefix_states(w: wl.Workload, rows, heads=None, steps=None) -> np.ndarray:
    """Natural-order FP32 states after `steps` (default w.prefix) FP32 steps from S = 0.

    Returns float32 [len(rows), len(heads), d_k, d_v].
    """
    rows = list(rows)
    heads = list(range(w.heads)) if heads is None else list(heads)
    steps = w.prefix if steps is None else steps
    S = np.zeros((len(rows) * len(heads), w.d_k, w.d_v), np.float32)
    for t in range(steps):
        u = unit_operands(w, wl.step_inputs(w, t, wl.STREAM_PREFIX, rows), heads)
        core.delta_step_heads(S, u["q"], u["k"], u["v"], u["g"], u["beta"], w.kind)
    return S.reshape(len(rows), len(heads), w.d_k, w.d_v)


def calibration_stats(w: wl.Workload, n_docs: int, n_tokens: int, every: int = 8, heads=None):
    """Error energy E [Hs, d_k] and log-decay mean over calibration documents.

    Each document is an independent FP32 trajectory from S = 0 (stream
    STREAM_CALIB, rows = documents).  States are sampled every `every` tokens
    (tokens every, 2*every, ...), as in App. A.2; the decay statistic averages
    log a_{t,u} over every token of every document.  One synthetic domain.
    Returns (E, mean_log_a) with mean_log_a of shape [Hs, d_k].
    """
    heads = list(range(w.heads)) if heads is None else list(heads)
    Hs = len(heads)
    docs = list(range(n_docs))
    S = np.zeros((n_docs * Hs, w.d_k, w.d_v), np.float32)
    err_sum = np.zeros((Hs, w.d_k))
    n_samples = 0
    log_a_sum = np.zeros((Hs, w.d_k))
    for t in range(n_tokens):
        u = unit_operands(w, wl.step_inputs(w, t, wl.STREAM_CALIB, docs), heads)
        core.delta_step_heads(S, u["q"], u["k"], u["v"], u["g"], u["beta"], w.kind)
        g = u["g"].astype(np.float64).reshape(n_docs, Hs, -1)
        log_a_sum += g.sum(axis=0) if w.kind == "kda" else np.repeat(g.sum(axis=0), w.d_k, axis=1)
        if (t + 1) % every == 0:
            e = calibrate.error_energy_samples(S, w.lo_format).reshape(n_docs, Hs, w.d_k)
            err_sum += e.sum(axis=0)
            n_samples += n_docs
    return err_sum / n_samples, log_a_sum / (n_docs * n_tokens)


def calibrate_layout(w: wl.Workload, n_docs: int = 32, n_tokens: int = 256, heads=None):
    """Per-head permutation pi (uint8 [Hs, d_k]) and score C from Algorithm 1."""
    E, mean_log_a = calibration_stats(w, n_docs, n_tokens, heads=heads)
    P = calibrate.persistence(np.exp(mean_log_a))
    perms, scores = [], []
    for i in range(E.shape[0]):
        _, pi = calibrate.select_layout(E[i], P[i], w.k_hi)
        perms.append(pi)
        scores.append(E[i] * P[i])
    return np.stack(perms).astype(np.uint8), np.stack(scores)


def decode_trajectory(w: wl.Workload, perm_units, tiers, rows, heads, steps, t0: int = 0):
    """Free-running quantized decode from packed tiers over `steps` steps.

    Yields (t, o, (hi, codes, meta)) after each step, with copies of the tiers.
    perm_units: uint8 [len(rows)*len(heads), d_k] in (row, head) order.
    """
    hi, codes, meta = (np.ascontiguousarray(a).copy() for a in tiers)
    for t in range(t0, t0 + steps):
        u = unit_operands(w, wl.step_inputs(w, t, wl.STREAM_DECODE, rows), heads)
        o = core.mixed_step_heads(perm_units, hi, codes, meta, u["q"], u["k"], u["v"], u["g"], u["beta"],
                                  w.k_hi, w.lo_format, w.kind)
        yield t, o, (hi.copy(), codes.copy(), meta.copy())
