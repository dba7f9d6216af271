"""Seeded synthetic inputs for the DAMP decode-step workloads.

This module is shared by the CPU oracle's tests and by the CUDA path's tests
and bench.  It holds none of the method's arithmetic: it only draws random
operands with the distributions and shapes of the paper's decode workloads
(decode batches of request slots, 32 heads, head dimension 128, Sec. 6.1 and
Sec. 6.3) and rounds them to the input dtype.  The paper's own inputs (ShareGPT
requests through Qwen3.6 / Kimi-Linear, Pile calibration documents) are not
available; these synthetic draws stand in for them.

Every draw comes from ``numpy.random.default_rng([seed, layer, stream, t, row])``
so that any subset of batch rows (or calibration documents) at any step can be
regenerated on its own, identically, by either side.

Recipe per (stream, step t, row b), in this draw order:
  q, k  ~ N(0, 1) of shape [H_qk, d_k], then L2-normalized per head (float64);
  v     ~ N(0, 1) of shape [H, d_v];
  beta  = sigmoid(N(0, 1)) of shape [H];
  GDN:  g = log(alpha) = -softplus(N(0, 1)) of shape [H];
  KDA:  g = -exp(u_{h,c}) * (1 + 0.05 N(0, 1)) of shape [H, d_k], with
        u_{h,c} ~ U(-6, 0) drawn once per layer (a fixed persistence profile).
q, k, v are rounded to bfloat16 (round to nearest even) for BF16 workloads;
beta and g stay FP32.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass

import numpy as np

STREAM_PREFIX = 1   # steps that build the initial FP32 state of the decode batch
STREAM_DECODE = 2   # decode steps
STREAM_CALIB = 3    # calibration documents (rows = documents)
STREAM_U = 4        # KDA per-channel decay profile
STREAM_PERM = 5     # random key-channel permutations (throughput runs only)


@dataclass(frozen=True)
class Workload:
    name: str
    kind: str          # "gdn" (scalar decay per head) or "kda" (per key channel)
    batch: int         # decode batch B (request slots)
    heads: int         # value heads H
    qk_heads: int      # q/k heads H_qk (GQA when < heads)
    d_k: int
    d_v: int
    k_hi: int          # FP16 key channels per head
    steps: int         # decode steps T
    prefix: int        # FP32 steps that build the initial state
    in_dtype: str      # "fp32" or "bf16" for q, k, v
    seed: int
    lo_format: int = 0  # 0 = UINT8 affine G32 + H32 (paper format), 1 = no H32, 2 = row absmax INT8
    layer: int = 0

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The paper-shaped decode workloads.
GDN_B1_D64 = Workload("gdn_b1_h4_d64_k8", "gdn", 1, 4, 4, 64, 64, 8, 16, 32, "fp32", 0)
GDN_B64_GQA = Workload("gdn_b64_h32_hqk16_d128_k8", "gdn", 64, 32, 16, 128, 128, 8, 64, 256, "bf16", 1)
KDA_B256 = Workload("kda_b256_h32_d128_k10", "kda", 256, 32, 32, 128, 128, 10, 128, 256, "bf16", 2)

SWEEP_K_HI = (0, 4, 8, 16, 32)


def sweep(kind: str, k_hi: int, lo_format: int = 0) -> Workload:
    """B=256, H=32, d=128 sweep point (GDN without GQA, or KDA)."""
    return Workload(f"{kind}_b256_h32_d128_k{k_hi}_f{lo_format}", kind, 256, 32, 32, 128, 128, k_hi,
                    16, 256, "bf16", 3, lo_format)


def stack_layer(layer: int, k_hi: int = 16) -> Workload:
    """Layer `layer` of the 30-layer decode stack: alternating GDN / KDA, B=256, H=32, d=128."""
    kind = "gdn" if layer % 2 == 0 else "kda"
    return Workload(f"stack_l{layer}_{kind}", kind, 256, 32, 32, 128, 128, k_hi, 1024, 256, "bf16",
                    4 * 1000 + layer, 0, layer)


def qk_head_of(w: Workload, h: int) -> int:
    """Value head h reads q/k head floor(h * H_qk / H) (consecutive value heads share)."""
    return (h * w.qk_heads) // w.heads


def _rng(w: Workload, stream: int, t: int, row: int) -> np.random.Generator:
    return np.random.default_rng([w.seed, w.layer, stream, t, row])


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even); return float32."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    out = r.astype(np.uint32).view(np.float32).copy()
    nan = np.isnan(x)
    out[nan] = x[nan]
    return out


def kda_u(w: Workload) -> np.ndarray:
    """Fixed per-channel log-log decay profile u_{h,c} ~ U(-6, 0), shape [H, d_k]."""
    return np.random.default_rng([w.seed, w.layer, STREAM_U]).uniform(-6.0, 0.0, (w.heads, w.d_k))


def step_inputs(w: Workload, t: int, stream: int = STREAM_DECODE, rows=None) -> dict:
    """Operands of step t for the given batch rows (default: all B rows).

    Returns float32 arrays: q, k [R, H_qk, d_k]; v [R, H, d_v]; beta [R, H];
    g [R, H] (GDN) or [R, H, d_k] (KDA).
    """
    rows = list(range(w.batch)) if rows is None else list(rows)
    R = len(rows)
    q = np.empty((R, w.qk_heads, w.d_k), np.float32)
    k = np.empty_like(q)
    v = np.empty((R, w.heads, w.d_v), np.float32)
    beta = np.empty((R, w.heads), np.float32)
    g = np.empty((R, w.heads) if w.kind == "gdn" else (R, w.heads, w.d_k), np.float32)
    u = kda_u(w) if w.kind == "kda" else None
    for i, b in enumerate(rows):
        r = _rng(w, stream, t, b)
        qb = r.standard_normal((w.qk_heads, w.d_k))
        kb = r.standard_normal((w.qk_heads, w.d_k))
        vb = r.standard_normal((w.heads, w.d_v))
        bb = r.standard_normal(w.heads)
        q[i] = qb / np.linalg.norm(qb, axis=-1, keepdims=True)
        k[i] = kb / np.linalg.norm(kb, axis=-1, keepdims=True)
        v[i] = vb
        beta[i] = 1.0 / (1.0 + np.exp(-bb))
        if w.kind == "gdn":
            g[i] = -np.logaddexp(0.0, r.standard_normal(w.heads))
        else:
            g[i] = -np.exp(u) * (1.0 + 0.05 * r.standard_normal((w.heads, w.d_k)))
    if w.in_dtype == "bf16":
        q, k, v = round_bf16(q), round_bf16(k), round_bf16(v)
    return {"q": q, "k": k, "v": v, "beta": beta, "g": g}


def random_perm(w: Workload) -> np.ndarray:
    """A seeded random key-channel permutation per head, uint8 [H, d_k] (throughput runs)."""
    r = np.random.default_rng([w.seed, w.layer, STREAM_PERM])
    return np.stack([r.permutation(w.d_k) for _ in range(w.heads)]).astype(np.uint8)


def random_states(seed: int, n: int, d_k: int, d_v: int, scale: float = 1.0) -> np.ndarray:
    """Generic random natural-order FP32 states [n, d_k, d_v] with per-row magnitude spread."""
    r = np.random.default_rng([seed, 99])
    rows = np.exp(r.uniform(-3.0, 1.0, (n, d_k, 1)))
    cols = np.exp(r.uniform(-1.0, 1.0, (n, 1, d_v)))
    return (scale * rows * cols * r.standard_normal((n, d_k, d_v))).astype(np.float32)


def torch_step_inputs(w: Workload, n_steps: int, device, seed_offset: int = 0, gate_bias=None) -> list:
    """Device-resident operands for throughput runs, drawn with torch's generator.

    Same recipe and shapes as `step_inputs` (not the same numbers): a list of
    n_steps dicts of torch tensors on `device`.  gate_bias (GDN only, [H] floats)
    shifts each head's gate logit, g = -softplus(N(0,1) + bias_h): negative biases
    give slow-decay heads (alpha near 1), positive ones fast-decay heads.
    """
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(w.seed * 1_000_003 + w.layer * 7919 + seed_offset)
    u = torch.from_numpy(kda_u(w)).to(device=device, dtype=torch.float32) if w.kind == "kda" else None
    dt = torch.bfloat16 if w.in_dtype == "bf16" else torch.float32
    bias = None if gate_bias is None else torch.as_tensor(gate_bias, dtype=torch.float32, device=device)
    out = []
    for _ in range(n_steps):
        def n(*shape):
            return torch.randn(*shape, generator=gen, device=device, dtype=torch.float32)
        q = n(w.batch, w.qk_heads, w.d_k)
        k = n(w.batch, w.qk_heads, w.d_k)
        q = q / q.norm(dim=-1, keepdim=True)
        k = k / k.norm(dim=-1, keepdim=True)
        v = n(w.batch, w.heads, w.d_v)
        beta = torch.sigmoid(n(w.batch, w.heads))
        if w.kind == "gdn":
            z = n(w.batch, w.heads)
            g = -torch.nn.functional.softplus(z if bias is None else z + bias[None])
        else:
            g = -torch.exp(u)[None] * (1.0 + 0.05 * n(w.batch, w.heads, w.d_k))
        out.append({"q": q.to(dt).contiguous(), "k": k.to(dt).contiguous(), "v": v.to(dt).contiguous(),
                    "beta": beta.contiguous(), "g": g.contiguous()})
    return out
