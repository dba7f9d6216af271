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


def calibration_trajectory(w: wl.Workload, n_docs: int, n_tokens: int, heads=None):
    """FP32 trajectories of the calibration documents, token by token.

    Each document is an independent trajectory from S = 0 (stream STREAM_CALIB,
    rows = documents).  Yields (n, S, log_a) for n = 1 .. n_tokens: S is a copy of
    the float32 states [n_docs, Hs, d_k, d_v] after the n-th token, log_a the
    float64 log-decay rows [n_docs, Hs, d_k] of that token (GDN's scalar per head is
    repeated over the key channels).
    """
    heads = list(range(w.heads)) if heads is None else list(heads)
    Hs = len(heads)
    docs = list(range(n_docs))
    S = np.zeros((n_docs * Hs, w.d_k, w.d_v), np.float32)
    for t in range(n_tokens):
        u = unit_operands(w, wl.step_inputs(w, t, wl.STREAM_CALIB, docs), heads)
        core.delta_step_heads(S, u["q"], u["k"], u["v"], u["g"], u["beta"], w.kind)
        g = u["g"].astype(np.float64).reshape(n_docs, Hs, -1)
        log_a = g if w.kind == "kda" else np.repeat(g, w.d_k, axis=2)
        yield t + 1, S.reshape(n_docs, Hs, w.d_k, w.d_v).copy(), log_a


def sampled_token_counts(n_tokens: int, every: int) -> list:
    """Token counts after which a calibration state is sampled (App. A.2: every
    `every` tokens): every, 2*every, ... up to n_tokens -- never the empty state."""
    return list(range(every, n_tokens + 1, every))


def collect_calibration_samples(trajectory, every: int):
    """Explicit calibration samples from a trajectory of (n, S, log_a) items.

    Returns (states, log_a): states float32 [n_samples, Hs, d_k, d_v] holds the
    states after the token counts of sampled_token_counts (all documents of one
    count before the next count); log_a float64 [n_rows, Hs, d_k] holds the
    log-decay rows of every token of every document.
    """
    states, rows, n_seen = [], [], 0
    for n, S, log_a in trajectory:
        n_seen = n
        rows.append(np.asarray(log_a, np.float64).reshape(-1, *np.shape(log_a)[-2:]))
        if n % every == 0:
            states.append(np.asarray(S, np.float32).reshape(-1, *np.shape(S)[-3:]))
    if not rows:
        raise ValueError("empty calibration trajectory")
    assert len(states) == len(sampled_token_counts(n_seen, every))
    st = np.concatenate(states) if states else np.zeros((0,) + rows[0].shape[1:] + (0,), np.float32)
    return st, np.concatenate(rows)


def calibration_stats_from_samples(states, log_a, fmt: int):
    """E [Hs, d_k] (Eq. empirical_error_energy, calibrate.error_energy) and a_eff
    [Hs, d_k] (Eq. empirical_persistence, calibrate.effective_decay) per head, from
    the explicit samples of collect_calibration_samples.  One synthetic domain."""
    Hs = log_a.shape[1]
    E = np.stack([calibrate.error_energy(states[:, h], fmt) for h in range(Hs)])
    a_eff = np.stack([calibrate.effective_decay(log_a[:, h]) for h in range(Hs)])
    return E, a_eff


def calibration_stats(w: wl.Workload, n_docs: int, n_tokens: int, every: int = 8, heads=None):
    """Error energy E [Hs, d_k] and effective decay a_eff [Hs, d_k] of App. A.2.

    States are sampled after tokens every, 2*every, ... of each document; the decay
    statistic averages log a_{t,u} over every token of every document.
    """
    states, log_a = collect_calibration_samples(calibration_trajectory(w, n_docs, n_tokens, heads), every)
    return calibration_stats_from_samples(states, log_a, w.lo_format)


def calibrate_layout(w: wl.Workload, n_docs: int = 32, n_tokens: int = 256, heads=None):
    """Per-head permutation pi (uint8 [Hs, d_k]) and score C from Algorithm 1."""
    E, a_eff = calibration_stats(w, n_docs, n_tokens, heads=heads)
    P = calibrate.persistence(a_eff)
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
