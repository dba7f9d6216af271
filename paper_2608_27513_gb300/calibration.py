"""Calibration run on the GPU (Algorithm 1, App. A.2): FP32 trajectories of the
calibration documents, error energy of the states sampled every `every` tokens,
mean log-decay over every token, then the selection of K_hi protected channels and
the permutation pi per head.  Every arithmetic step is a libdamp call; this module
stacks the per-token inputs and orders the calls."""
from __future__ import annotations

import contextlib

import paper_2608_27513_gb300 as damp


def accumulate(layout, kind: str, token_inputs, every: int = 8, stream=None):
    """The FP32 trajectories of the calibration documents under a layout holding every
    head of the layer (no head map): returns (E_acc, n_samples, G_acc, n_tokens), the
    error-energy and log-decay sums over the layer's heads [H, d_k].  token_inputs is a
    sequence of per-token dicts (rows = documents) or one dict of tensors stacked over
    the tokens ([T, B, ...]); the whole run is one damp_calib_accumulate call."""
    import torch
    if isinstance(token_inputs, dict):
        stacked = token_inputs
    else:
        inputs = list(token_inputs)
        with torch.cuda.stream(stream) if stream is not None else contextlib.nullcontext():
            stacked = {n: torch.stack([d[n] for d in inputs]) for n in ("q", "k", "v", "g", "beta")}
    n_docs = stacked["v"].shape[1]
    dev = stacked["v"].device
    with torch.cuda.stream(stream) if stream is not None else contextlib.nullcontext():
        S = damp.new_fp32_state(layout, n_docs, dev)
        E_acc = torch.zeros((layout.num_heads, layout.d_k), dtype=torch.float32, device=dev)
        G_acc = torch.zeros_like(E_acc)
    n_samples, n_tokens = damp.calib_accumulate(layout, kind, S, stacked["q"], stacked["k"], stacked["v"],
                                                stacked["g"], stacked["beta"], E_acc, G_acc, every, stream)
    return E_acc, n_samples, G_acc, n_tokens


def calibrate(layout, kind: str, token_inputs, every: int = 8, tau: float = 1e-4, stream=None):
    """token_inputs: sequence of per-token dicts of device tensors (q, k, v, g, beta) for
    the calibration documents (rows = documents), in token order, or one dict of those
    tensors stacked over the tokens.  Returns (C, perm): float32 [H, d_k] scores and uint8
    [H, d_k] permutations."""
    E_acc, n_samples, G_acc, n_tokens = accumulate(layout, kind, token_inputs, every, stream)
    return damp.calib_select(layout, E_acc, n_samples, G_acc, n_tokens, tau, stream=stream)


def calibrate_groups(groups, kind: str, token_inputs, every: int = 8, tau: float = 1e-4, stream=None):
    """Calibration of a layer split into head groups (damp.head_groups: a layout per
    K_hi with its head map).  The trajectories and sums run once over all heads; each
    group then selects its own K_hi channels per head.  Returns [(C, perm)] per group."""
    g0 = groups[0][0] if isinstance(groups[0], tuple) else groups[0]
    full = damp.Layout(g0.heads_of_operands, g0.num_qk_heads, g0.d_k, g0.d_v, 0, g0.lo_format)
    E_acc, n_samples, G_acc, n_tokens = accumulate(full, kind, token_inputs, every, stream)
    out = []
    for gr in groups:
        L = gr[0] if isinstance(gr, tuple) else gr
        out.append(damp.calib_select(L, E_acc, n_samples, G_acc, n_tokens, tau, stream=stream))
    return out
