"""libdamp: the DAMP decode-step recurrent-state update on GB300 (sm_103a).

Python binding over the C ABI of include/damp.h.  The functions carry the
ABI's names and only marshal arguments: every step of the path runs in the
library's CUDA kernels.  PyTorch provides device memory and streams.  There is
no CPU fallback: without the built library every call raises
DampLibraryError.

    layout = Layout(num_heads=32, num_qk_heads=32, d_k=128, d_v=128, k_hi=10)
    state = new_state(layout, num_slots=256, device="cuda")
    quantize_state(layout, S_fp32, perm, state)            # prefill hand-off
    o = kda_decode_step(layout, state, perm, q, k, v, g, beta)

A layer whose heads keep different numbers of FP16 key channels (the decay-tiered
allocation of App. E) is a list of head groups (`head_groups`), one uniform layout,
pool and permutation table per K_hi, each with a head map into the layer's heads.
"""
from __future__ import annotations

import ctypes
from dataclasses import dataclass, field

from ._lib import DampLayout, DampLibraryError, lib

__all__ = [
    "Layout", "DampError", "DampLibraryError", "LO_U8_AFFINE_G32_H32", "LO_U8_AFFINE_G32", "LO_S8_ABSMAX_ROW", "LO_U4_AFFINE_G32_H32",
    "LO_U4_AFFINE_G32", "LO_FP8_E4M3_G32",
    "record_bytes", "slot_bytes", "bits_per_value", "new_state", "new_fp32_state",
    "gdn_decode_step", "kda_decode_step", "gdn_prefill_chunk", "kda_prefill_chunk", "calib_error_energy", "calib_log_decay", "calib_select", "u8_gdn_decode_step", "u8_kda_decode_step",
    "fp32_gdn_decode_step", "fp32_kda_decode_step", "quantize_state", "dequantize_state",
    "pack_tiers", "unpack_tiers", "device_status", "version", "DEV_WAIT_TIMEOUT", "DEV_BAD_SLOT", "DEV_BAD_HEAD",
    "head_groups", "test_kda_wait_timeout", "gdn_decode_step_groups", "kda_decode_step_groups",
    "calib_accumulate",
]

LO_U8_AFFINE_G32_H32 = 0
LO_U8_AFFINE_G32 = 1
LO_S8_ABSMAX_ROW = 2  # per-row symmetric absmax INT8, FP32 row scale
LO_U4_AFFINE_G32_H32 = 3  # UINT4 affine G32 + H32
LO_U4_AFFINE_G32 = 4  # UINT4 affine G32
LO_FP8_E4M3_G32 = 5  # FP8 E4M3, FP32 scale per 32
IN_BF16 = 0
IN_FP32 = 1
DEV_WAIT_TIMEOUT = 1
DEV_BAD_SLOT = 2
DEV_BAD_HEAD = 4


class DampError(RuntimeError):
    def __init__(self, status: int, what: str):
        msg = lib().damp_status_string(status).decode()
        super().__init__(f"{what}: {msg}")
        self.status = status


@dataclass(frozen=True)
class Layout:
    """damp_layout: num_heads held heads (one state per slot and head), q/k heads of the
    operands, d_k x d_v states, K_hi FP16 key channels, the low-tier format; for a head
    group of a layer, model_heads (value heads of the operand tensors) and head_map
    (int32 CUDA tensor [num_heads]: the model head of each held head)."""
    num_heads: int
    num_qk_heads: int
    d_k: int
    d_v: int
    k_hi: int
    lo_format: int = LO_U8_AFFINE_G32_H32
    model_heads: int = 0
    head_map: object = field(default=None, compare=False, repr=False)

    def __post_init__(self):
        if self.head_map is not None:
            import torch
            m = self.head_map
            if (not isinstance(m, torch.Tensor) or m.dtype != torch.int32 or not m.is_cuda or not m.is_contiguous()
                    or m.shape != (self.num_heads,)):
                raise ValueError(f"head_map must be a contiguous int32 CUDA tensor of shape [{self.num_heads}]")

    @property
    def heads_of_operands(self) -> int:
        """H_m: value heads of v, g, beta, o and S."""
        return self.model_heads or self.num_heads

    def c(self) -> DampLayout:
        return DampLayout(self.num_heads, self.num_qk_heads, self.d_k, self.d_v, self.k_hi, self.lo_format,
                          self.model_heads, None if self.head_map is None else self.head_map.data_ptr())


def head_groups(k_hi_of_head, num_qk_heads: int, d_k: int, d_v: int, lo_format: int = LO_U8_AFFINE_G32_H32,
                device="cuda"):
    """Layouts of a layer whose heads keep different numbers of FP16 key channels
    (App. E, decay-tiered allocation): one layout per distinct K_hi, held heads in
    ascending model-head order, each with its head map.  Returns [(layout, heads)],
    heads the list of model heads of the group."""
    import torch
    ks = [int(k) for k in k_hi_of_head]
    H = len(ks)
    out = []
    for K in sorted(set(ks)):
        heads = [h for h in range(H) if ks[h] == K]
        m = torch.tensor(heads, dtype=torch.int32, device=device)
        out.append((Layout(len(heads), num_qk_heads, d_k, d_v, K, lo_format, model_heads=H, head_map=m), heads))
    return out


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _check(status: int, what: str):
    if status != 0:
        raise DampError(status, what)


def _in_dtype(*ts) -> int:
    import torch
    dts = {t.dtype for t in ts}
    if dts == {torch.bfloat16}:
        return IN_BF16
    if dts == {torch.float32}:
        return IN_FP32
    raise TypeError("q, k, v must all be bfloat16 or all float32")


def _cuda_contig(name, t):
    if t is None:
        return
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous CUDA tensor")


def _want(name, t, shape, *, dtype=None, esize=None):
    """Raise ValueError unless tensor t (if given) has exactly `shape` (and dtype or
    element size).  The C ABI sees only pointers, so a mis-sized tensor would make a
    kernel read or write outside it: every size is checked here, before any call."""
    if t is None:
        return
    if tuple(t.shape) != tuple(int(x) for x in shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(int(x) for x in shape)}")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} has dtype {t.dtype}, expected {dtype}")
    if esize is not None and t.element_size() not in ((esize,) if isinstance(esize, int) else esize):
        raise ValueError(f"{name} has {t.element_size()}-byte elements, expected {esize}")


def _want_pool(layout, state, num_slots, fp32=False):
    """The packed pool (uint8 [slots, slot_bytes]) or FP32 state (float32 [slots, H, d_k,
    d_v]) must hold num_slots slots; returns num_slots (default: all of them)."""
    import torch
    if state is None:
        raise ValueError("state is required")
    if fp32:
        _want("state", state, (state.shape[0], layout.num_heads, layout.d_k, layout.d_v), dtype=torch.float32)
    else:
        if state.dim() != 2:
            raise ValueError(f"state has shape {tuple(state.shape)}, expected [slots, {slot_bytes(layout)}]")
        _want("state", state, (state.shape[0], slot_bytes(layout)), dtype=torch.uint8)
    n = state.shape[0] if num_slots is None else int(num_slots)
    if n < 0 or n > state.shape[0]:
        raise ValueError(f"num_slots {n} exceeds the {state.shape[0]} slots of state")
    return n


def _want_batch(slot_idx, B, num_slots):
    import torch
    _want("slot_idx", slot_idx, (B,), dtype=torch.int32)
    if slot_idx is None and B > num_slots:
        raise ValueError(f"batch {B} exceeds num_slots {num_slots} without slot_idx")


def _want_operands(layout, kind, q, k, v, g, beta, o, lead):
    """q, k [*lead, H_qk, d_k]; v [*lead, H_m, d_v]; g [*lead, H_m] (GDN) or [*lead, H_m,
    d_k] (KDA); beta [*lead, H_m]; o float32 [*lead, H_m, d_v]."""
    import torch
    Hm = layout.heads_of_operands
    for n, t in (("q", q), ("k", k), ("v", v), ("g", g), ("beta", beta)):
        if t is None:
            raise ValueError(f"{n} is required")
    lead = tuple(lead)
    _want("q", q, lead + (layout.num_qk_heads, layout.d_k))
    _want("k", k, lead + (layout.num_qk_heads, layout.d_k))
    _want("v", v, lead + (Hm, layout.d_v))
    _want("g", g, lead + ((Hm, layout.d_k) if kind == "kda" else (Hm,)), dtype=torch.float32)
    _want("beta", beta, lead + (Hm,), dtype=torch.float32)
    _want("o", o, lead + (Hm, layout.d_v), dtype=torch.float32)


def version() -> int:
    return int(lib().damp_version())


def record_bytes(layout: Layout) -> int:
    c = layout.c()
    return int(lib().damp_record_bytes(ctypes.byref(c)))


def slot_bytes(layout: Layout) -> int:
    c = layout.c()
    n = int(lib().damp_slot_bytes(ctypes.byref(c)))
    if n == 0:
        _check(lib().damp_validate_layout(ctypes.byref(c)), "layout")
    return n


def bits_per_value(layout: Layout) -> float:
    c = layout.c()
    return float(lib().damp_bits_per_value(ctypes.byref(c)))


def new_state(layout: Layout, num_slots: int, device="cuda"):
    """A zero-filled packed pool of num_slots slots (uint8, 16-B aligned by the allocator)."""
    import torch
    return torch.zeros((num_slots, slot_bytes(layout)), dtype=torch.uint8, device=device)


def new_fp32_state(layout: Layout, num_slots: int, device="cuda"):
    import torch
    return torch.zeros((num_slots, layout.num_heads, layout.d_k, layout.d_v), dtype=torch.float32, device=device)


def _step(fn_name, layout, state, perm, q, k, v, g, beta, o, slot_idx, num_slots, stream):
    import torch
    fp32 = fn_name.startswith("damp_fp32")
    if v is None or v.dim() < 1:
        raise ValueError("v must be a [B, H, d_v] tensor")
    B = v.shape[0]
    num_slots = _want_pool(layout, state, num_slots, fp32=fp32)
    _want_batch(slot_idx, B, num_slots)
    if not fp32:
        _want("perm", perm, (layout.num_heads, layout.d_k), dtype=torch.uint8)
    _want_operands(layout, "kda" if "_kda_" in fn_name else "gdn", q, k, v, g, beta, o, (B,))
    for n, t in (("state", state), ("perm", perm), ("q", q), ("k", k), ("v", v), ("g", g), ("beta", beta),
                 ("o", o), ("slot_idx", slot_idx)):
        _cuda_contig(n, t)
    if o is None:
        # a head group writes only its heads' rows: the others start at zero
        alloc = torch.empty if layout.head_map is None else torch.zeros
        o = alloc((B, layout.heads_of_operands, layout.d_v), dtype=torch.float32, device=v.device)
    c = layout.c()
    args = [ctypes.byref(c), _ptr(state), num_slots, _ptr(slot_idx), B]
    if perm is not None or not fn_name.startswith("damp_fp32"):
        args.append(_ptr(perm))
    args += [_ptr(q), _ptr(k), _ptr(v), _ptr(g), _ptr(beta), _ptr(o), _in_dtype(q, k, v), _stream(stream)]
    _check(getattr(lib(), fn_name)(*args), fn_name)
    return o


def gdn_decode_step(layout, state, perm, q, k, v, g, beta, o=None, slot_idx=None, num_slots=None, stream=None):
    """One GDN decode step on the packed state (in place); returns o [B, H, d_v] float32."""
    return _step("damp_gdn_decode_step", layout, state, perm, q, k, v, g, beta, o, slot_idx, num_slots, stream)


def kda_decode_step(layout, state, perm, q, k, v, g, beta, o=None, slot_idx=None, num_slots=None, stream=None):
    """One KDA decode step on the packed state (in place); returns o [B, H, d_v] float32."""
    return _step("damp_kda_decode_step", layout, state, perm, q, k, v, g, beta, o, slot_idx, num_slots, stream)


def _step_groups(fn_name, groups, q, k, v, g, beta, o, slot_idx, stream):
    """groups: [(layout, state, perm)] of one layer (head_groups layouts)."""
    import torch
    n = len(groups)
    if n < 1:
        raise ValueError("at least one head group is required")
    if v is None or v.dim() < 1:
        raise ValueError("v must be a [B, H_m, d_v] tensor")
    B = v.shape[0]
    kind = "kda" if "_kda_" in fn_name else "gdn"
    layouts = (DampLayout * n)()
    states = (ctypes.c_void_p * n)()
    perms = (ctypes.c_void_p * n)()
    slots = (ctypes.c_int64 * n)()
    for i, (layout, state, perm) in enumerate(groups):
        if layout.head_map is None:
            raise ValueError(f"group {i} has no head map (build the groups with head_groups)")
        ns = _want_pool(layout, state, None)
        _want_batch(slot_idx, B, ns)
        _want("perm", perm, (layout.num_heads, layout.d_k), dtype=torch.uint8)
        _want_operands(layout, kind, q, k, v, g, beta, o, (B,))
        _cuda_contig("state", state)
        _cuda_contig("perm", perm)
        layouts[i] = layout.c()
        states[i] = state.data_ptr()
        perms[i] = perm.data_ptr()
        slots[i] = ns
    for nm, t in (("q", q), ("k", k), ("v", v), ("g", g), ("beta", beta), ("o", o), ("slot_idx", slot_idx)):
        _cuda_contig(nm, t)
    if o is None:
        o = torch.empty((B, groups[0][0].heads_of_operands, groups[0][0].d_v), dtype=torch.float32, device=v.device)
    _check(getattr(lib(), fn_name)(layouts, n, states, slots, perms, _ptr(slot_idx), B, _ptr(q), _ptr(k), _ptr(v),
                                   _ptr(g), _ptr(beta), _ptr(o), _in_dtype(q, k, v), _stream(stream)), fn_name)
    return o


def gdn_decode_step_groups(groups, q, k, v, g, beta, o=None, slot_idx=None, stream=None):
    """One GDN decode step of a layer stored as head groups, groups = [(layout, state, perm)]
    (one launch for two groups with a compile-time K_hi pair); returns o [B, H_m, d_v]."""
    return _step_groups("damp_gdn_decode_step_groups", groups, q, k, v, g, beta, o, slot_idx, stream)


def kda_decode_step_groups(groups, q, k, v, g, beta, o=None, slot_idx=None, stream=None):
    """One KDA decode step of a layer stored as head groups (see gdn_decode_step_groups)."""
    return _step_groups("damp_kda_decode_step_groups", groups, q, k, v, g, beta, o, slot_idx, stream)


def test_kda_wait_timeout(layout, state, perm, q, k, v, g, beta, o=None, slot_idx=None, num_slots=None,
                          stream=None):
    """The bounded-wait test hook (damp_test_kda_wait_timeout): every wait of the KDA step's
    kernel runs out after ~1 ms; nothing is written and the status word reports
    DEV_WAIT_TIMEOUT.  For tests of the timeout path only."""
    return _step("damp_test_kda_wait_timeout", layout, state, perm, q, k, v, g, beta, o, slot_idx, num_slots,
                 stream)


def u8_gdn_decode_step(layout, state, perm, q, k, v, g, beta, o=None, slot_idx=None, num_slots=None, stream=None):
    return _step("damp_u8_gdn_decode_step", layout, state, perm, q, k, v, g, beta, o, slot_idx, num_slots, stream)


def u8_kda_decode_step(layout, state, perm, q, k, v, g, beta, o=None, slot_idx=None, num_slots=None, stream=None):
    return _step("damp_u8_kda_decode_step", layout, state, perm, q, k, v, g, beta, o, slot_idx, num_slots, stream)


def fp32_gdn_decode_step(layout, state, q, k, v, g, beta, o=None, slot_idx=None, num_slots=None, stream=None):
    """One GDN decode step on an FP32 state [slots, H, d_k, d_v] (in place)."""
    return _step("damp_fp32_gdn_decode_step", layout, state, None, q, k, v, g, beta, o, slot_idx, num_slots, stream)


def fp32_kda_decode_step(layout, state, q, k, v, g, beta, o=None, slot_idx=None, num_slots=None, stream=None):
    return _step("damp_fp32_kda_decode_step", layout, state, None, q, k, v, g, beta, o, slot_idx, num_slots, stream)


def _prefill(fn_name, layout, state, perm, q, k, v, g, beta, o, lengths, slot_idx, num_slots, stream):
    import torch
    if v is None or v.dim() < 2:
        raise ValueError("v must be a [B, T, H, d_v] tensor")
    B, T = v.shape[0], v.shape[1]
    num_slots = _want_pool(layout, state, num_slots)
    _want_batch(slot_idx, B, num_slots)
    _want("lengths", lengths, (B,), dtype=torch.int32)
    _want("perm", perm, (layout.num_heads, layout.d_k), dtype=torch.uint8)
    _want_operands(layout, "kda" if "_kda_" in fn_name else "gdn", q, k, v, g, beta, o, (B, T))
    for n, t in (("state", state), ("perm", perm), ("q", q), ("k", k), ("v", v), ("g", g), ("beta", beta),
                 ("o", o), ("lengths", lengths), ("slot_idx", slot_idx)):
        _cuda_contig(n, t)
    if o is None:
        o = torch.zeros((B, T, layout.heads_of_operands, layout.d_v), dtype=torch.float32, device=v.device)
    c = layout.c()
    _check(getattr(lib(), fn_name)(ctypes.byref(c), _ptr(state), num_slots, _ptr(slot_idx), B, T, _ptr(lengths),
                                   _ptr(perm), _ptr(q), _ptr(k), _ptr(v), _ptr(g), _ptr(beta), _ptr(o),
                                   _in_dtype(q, k, v), _stream(stream)), fn_name)
    return o


def gdn_prefill_chunk(layout, state, perm, q, k, v, g, beta, o=None, lengths=None, slot_idx=None, num_slots=None,
                      stream=None):
    """One GDN prefill chunk on the packed state (in place): q, k [B, T, H_qk, d_k], v [B, T, H, d_v],
    g, beta [B, T, H]; returns o [B, T, H, d_v] float32."""
    return _prefill("damp_gdn_prefill_chunk", layout, state, perm, q, k, v, g, beta, o, lengths, slot_idx,
                    num_slots, stream)


def kda_prefill_chunk(layout, state, perm, q, k, v, g, beta, o=None, lengths=None, slot_idx=None, num_slots=None,
                      stream=None):
    """One KDA prefill chunk on the packed state (in place): as gdn_prefill_chunk with g [B, T, H, d_k]."""
    return _prefill("damp_kda_prefill_chunk", layout, state, perm, q, k, v, g, beta, o, lengths, slot_idx,
                    num_slots, stream)


def calib_error_energy(layout, S, E_acc, stream=None):
    """E_acc [H, d_k] += per-channel squared low-tier round-trip error of S [B, H, d_k, d_v]."""
    import torch
    Hm = layout.heads_of_operands
    if S is None or S.dim() != 4:
        raise ValueError("S must be a [B, H, d_k, d_v] tensor")
    _want("S", S, (S.shape[0], Hm, layout.d_k, layout.d_v), dtype=torch.float32)
    _want("E_acc", E_acc, (Hm, layout.d_k), dtype=torch.float32)
    _cuda_contig("S", S)
    _cuda_contig("E_acc", E_acc)
    _check(lib().damp_calib_error_energy(ctypes.byref(layout.c()), _ptr(S), S.shape[0], _ptr(E_acc), _stream(stream)),
           "damp_calib_error_energy")
    return E_acc


def calib_log_decay(layout, g, G_acc, stream=None):
    """G_acc [H, d_k] += log-decay g summed over the batch (g [B, H] GDN or [B, H, d_k] KDA)."""
    import torch
    Hm = layout.heads_of_operands
    if g is None or g.dim() not in (2, 3):
        raise ValueError("g must be a [B, H] or [B, H, d_k] tensor")
    _want("g", g, (g.shape[0], Hm) + ((layout.d_k,) if g.dim() == 3 else ()), dtype=torch.float32)
    _want("G_acc", G_acc, (Hm, layout.d_k), dtype=torch.float32)
    _cuda_contig("g", g)
    _cuda_contig("G_acc", G_acc)
    _check(lib().damp_calib_log_decay(ctypes.byref(layout.c()), _ptr(g), g.shape[0], 1 if g.dim() == 3 else 0,
                                      _ptr(G_acc), _stream(stream)), "damp_calib_log_decay")
    return G_acc


def calib_accumulate(layout, kind, S, q, k, v, g, beta, E_acc, G_acc, every=8, stream=None):
    """One calibration run's statistics in one call (damp_calib_accumulate): q, k [T, B, H_qk,
    d_k]; v [T, B, H, d_v]; g [T, B, H, d_k] (KDA) or [T, B, H] (GDN); beta [T, B, H]; S the
    FP32 states [B, H, d_k, d_v] (updated); E_acc, G_acc [H, d_k] accumulated.  Returns
    (n_samples, n_token_rows) for calib_select."""
    import torch
    if layout.head_map is not None:
        raise ValueError("the calibration trajectories hold every head: use a layout without a head map")
    if v is None or v.dim() != 4:
        raise ValueError("v must be a [T, B, H, d_v] tensor")
    T, B = v.shape[0], v.shape[1]
    H = layout.num_heads
    _want("S", S, (B, H, layout.d_k, layout.d_v), dtype=torch.float32)
    _want_operands(layout, kind, q, k, v, g, beta, None, (T, B))
    _want("E_acc", E_acc, (H, layout.d_k), dtype=torch.float32)
    _want("G_acc", G_acc, (H, layout.d_k), dtype=torch.float32)
    for n, t in (("S", S), ("q", q), ("k", k), ("v", v), ("g", g), ("beta", beta), ("E_acc", E_acc),
                 ("G_acc", G_acc)):
        _cuda_contig(n, t)
    _check(lib().damp_calib_accumulate(ctypes.byref(layout.c()), _ptr(S), B, T, _ptr(q), _ptr(k), _ptr(v), _ptr(g),
                                       _ptr(beta), _in_dtype(q, k, v), 1 if kind == "kda" else 0, int(every),
                                       _ptr(E_acc), _ptr(G_acc), _stream(stream)), "damp_calib_accumulate")
    return max(B * (T // int(every)), 1), B * T


def calib_select(layout, E_acc, n_samples, G_acc, n_tokens, tau=1e-4, stream=None):
    """Scores C [H, d_k] float32 and permutations pi [H, d_k] uint8 (Algorithm 1)."""
    import torch
    Hm = layout.heads_of_operands
    _want("E_acc", E_acc, (Hm, layout.d_k), dtype=torch.float32)
    _want("G_acc", G_acc, (Hm, layout.d_k), dtype=torch.float32)
    _cuda_contig("E_acc", E_acc)
    _cuda_contig("G_acc", G_acc)
    C = torch.empty((layout.num_heads, layout.d_k), dtype=torch.float32, device=E_acc.device)
    perm = torch.empty((layout.num_heads, layout.d_k), dtype=torch.uint8, device=E_acc.device)
    _check(lib().damp_calib_select(ctypes.byref(layout.c()), _ptr(E_acc), int(n_samples), _ptr(G_acc), int(n_tokens),
                                   float(tau), _ptr(C), _ptr(perm), _stream(stream)), "damp_calib_select")
    return C, perm


def quantize_state(layout, S, perm, state, slot_idx=None, num_slots=None, stream=None):
    """Write natural-order FP32 states S [B, H, d_k, d_v] into packed slots."""
    import torch
    if S is None or S.dim() != 4:
        raise ValueError("S must be a [B, H, d_k, d_v] tensor")
    n_slots = _want_pool(layout, state, num_slots)
    _want_batch(slot_idx, S.shape[0], n_slots)
    _want("S", S, (S.shape[0], layout.heads_of_operands, layout.d_k, layout.d_v), dtype=torch.float32)
    _want("perm", perm, (layout.num_heads, layout.d_k), dtype=torch.uint8)
    for n, t in (("S", S), ("perm", perm), ("state", state), ("slot_idx", slot_idx)):
        _cuda_contig(n, t)
    c = layout.c()
    _check(lib().damp_quantize_state(ctypes.byref(c), _ptr(S), _ptr(perm), _ptr(state), n_slots, _ptr(slot_idx),
                                     S.shape[0], _stream(stream)), "damp_quantize_state")


def dequantize_state(layout, state, perm, batch=None, S=None, slot_idx=None, num_slots=None, stream=None):
    """Reconstruct natural-order FP32 states [B, H, d_k, d_v] from packed slots."""
    import torch
    n_slots = _want_pool(layout, state, num_slots)
    B = (slot_idx.shape[0] if slot_idx is not None else n_slots) if batch is None else int(batch)
    _want_batch(slot_idx, B, n_slots)
    _want("S", S, (B, layout.heads_of_operands, layout.d_k, layout.d_v), dtype=torch.float32)
    _want("perm", perm, (layout.num_heads, layout.d_k), dtype=torch.uint8)
    for n, t in (("S", S), ("perm", perm), ("state", state), ("slot_idx", slot_idx)):
        _cuda_contig(n, t)
    if S is None:
        S = torch.zeros((B, layout.heads_of_operands, layout.d_k, layout.d_v), dtype=torch.float32, device=state.device)
    c = layout.c()
    _check(lib().damp_dequantize_state(ctypes.byref(c), _ptr(state), n_slots, _ptr(slot_idx), B,
                                       _ptr(perm), _ptr(S), _stream(stream)), "damp_dequantize_state")
    return S


def _tier_shapes(layout, B, hi, codes, meta):
    """(name, tensor, shape, element bytes) of the logical tiers of B slots (damp_pack_tiers)."""
    H, dk, dv, K, f = layout.num_heads, layout.d_k, layout.d_v, layout.k_hi, layout.lo_format
    lo = dk - K
    codes_cols = dv // 2 if f in (LO_U4_AFFINE_G32_H32, LO_U4_AFFINE_G32) else dv
    if f == LO_S8_ABSMAX_ROW:
        meta_shape, meta_es = (B, H, lo), 4
    elif f == LO_FP8_E4M3_G32:
        meta_shape, meta_es = (B, H, lo, dv // 32), 4
    else:
        meta_shape, meta_es = (B, H, lo, dv // 32, 2), 2
    return [("hi", hi, (B, H, K, dv), 2), ("codes", codes, (B, H, lo, codes_cols), 1),
            ("meta", meta, meta_shape, meta_es)]


def pack_tiers(layout, hi, codes, meta, state, slot_idx=None, num_slots=None, stream=None):
    """Copy logical tiers (hi uint16/fp16 [B,H,K,d_v], codes uint8 [B,H,d_k-K,d_v],
    meta uint16/fp16 [B,H,d_k-K,d_v/32,2]; row-absmax format: codes int8, meta float32
    [B,H,d_k-K]) into packed slots, bit for bit."""
    B = codes.shape[0] if codes is not None else (hi.shape[0] if hi is not None else 0)
    n_slots = _want_pool(layout, state, num_slots)
    _want_batch(slot_idx, B, n_slots)
    for n, t, shape, es in _tier_shapes(layout, B, hi, codes, meta):
        _want(n, t, shape, esize=es)
    for n, t in (("hi", hi), ("codes", codes), ("meta", meta), ("state", state), ("slot_idx", slot_idx)):
        _cuda_contig(n, t)
    c = layout.c()
    _check(lib().damp_pack_tiers(ctypes.byref(c), _ptr(hi if hi is not None and hi.numel() else None),
                                 _ptr(codes if codes is not None and codes.numel() else None),
                                 _ptr(meta if meta is not None and meta.numel() else None), _ptr(state),
                                 n_slots, _ptr(slot_idx), B,
                                 _stream(stream)), "damp_pack_tiers")


def unpack_tiers(layout, state, batch=None, slot_idx=None, num_slots=None, stream=None):
    """Logical tiers (hi int16 bits, codes uint8, meta int16 bits; row-absmax format: codes
    int8, meta float32 [B,H,d_k-K]) of `batch` packed slots."""
    import torch
    n_slots = _want_pool(layout, state, num_slots)
    B = (slot_idx.shape[0] if slot_idx is not None else n_slots) if batch is None else int(batch)
    _want_batch(slot_idx, B, n_slots)
    _cuda_contig("state", state)
    _cuda_contig("slot_idx", slot_idx)
    H, dk, dv, K = layout.num_heads, layout.d_k, layout.d_v, layout.k_hi
    dev = state.device
    hi = torch.empty((B, H, K, dv), dtype=torch.int16, device=dev)
    if layout.lo_format == LO_S8_ABSMAX_ROW:
        codes = torch.empty((B, H, dk - K, dv), dtype=torch.int8, device=dev)
        meta = torch.empty((B, H, dk - K), dtype=torch.float32, device=dev)
    elif layout.lo_format in (LO_U4_AFFINE_G32_H32, LO_U4_AFFINE_G32):
        codes = torch.empty((B, H, dk - K, dv // 2), dtype=torch.uint8, device=dev)
        meta = torch.empty((B, H, dk - K, dv // 32, 2), dtype=torch.int16, device=dev)
    elif layout.lo_format == LO_FP8_E4M3_G32:
        codes = torch.empty((B, H, dk - K, dv), dtype=torch.uint8, device=dev)
        meta = torch.empty((B, H, dk - K, dv // 32), dtype=torch.float32, device=dev)
    else:
        codes = torch.empty((B, H, dk - K, dv), dtype=torch.uint8, device=dev)
        meta = torch.empty((B, H, dk - K, dv // 32, 2), dtype=torch.int16, device=dev)
    c = layout.c()
    _check(lib().damp_unpack_tiers(ctypes.byref(c), _ptr(state), n_slots,
                                   _ptr(slot_idx), B, _ptr(hi if hi.numel() else None),
                                   _ptr(codes if codes.numel() else None), _ptr(meta if meta.numel() else None),
                                   _stream(stream)), "damp_unpack_tiers")
    return hi, codes, meta


def device_status() -> int:
    """Read and clear the device status word (DEV_* bits)."""
    v = ctypes.c_uint32(0)
    _check(lib().damp_device_status(ctypes.byref(v)), "damp_device_status")
    return int(v.value)
