"""Parity helpers: run the CUDA path and the oracle on the same seeded inputs and
compare them element by element.

Tolerances (the decode-step contract):
  * o and the FP16 tier: |gpu - ref| <= 1e-5 + 1e-3 |ref| per element;
  * UINT8 codes: at most 0.1% of codes differ (aggregated over a test), and
    every difference is a float-ordering tie of the oracle's own values:
      - in a group whose (s, z) agree, a code differs by at most 1 and only
        where the oracle's x/s + z lies within TIE of a half-integer;
      - a group's (s, z) may differ only where the oracle's scale
        s32 = (x_max - x_min)/255 lies within TIE_REL of a binary16 rounding
        midpoint or -x_min/s within TIE of a half-integer; then s is within
        one binary16 ulp, z within 1, and every reconstructed level s (q - z)
        within one quantization step; where only z moved, the raw codes shift
        with z and each code's level q - z is within 1 LSB.
"""
from __future__ import annotations

import numpy as np
import torch

import paper_2608_27513_gb300 as damp
import workloads as wl
from oracle import core, runs

RTOL, ATOL = 1e-3, 1e-5
CODE_FRAC = 1e-3
TIE = 2e-3        # code units
TIE_REL = 2e-5    # relative distance of s32 to a binary16 rounding boundary


def layout_of(w: wl.Workload) -> damp.Layout:
    return damp.Layout(w.heads, w.qk_heads, w.d_k, w.d_v, w.k_hi, w.lo_format)


def to_dev(a: np.ndarray, dev, dtype=None):
    t = torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    return t.to(dtype) if dtype is not None else t


def inputs_to_dev(w: wl.Workload, inp: dict, dev) -> dict:
    dt = torch.bfloat16 if w.in_dtype == "bf16" else torch.float32
    return {"q": to_dev(inp["q"], dev, dt), "k": to_dev(inp["k"], dev, dt), "v": to_dev(inp["v"], dev, dt),
            "g": to_dev(inp["g"], dev), "beta": to_dev(inp["beta"], dev)}


def _code_cols(w: wl.Workload) -> int:
    return w.d_v // 2 if w.lo_format in (core.FMT_U4_H32, core.FMT_U4) else w.d_v


def tiers_to_dev(w: wl.Workload, tiers, rows: int, dev):
    hi, codes, meta = tiers
    H, dk, dv, K = w.heads, w.d_k, w.d_v, w.k_hi
    if w.lo_format == core.FMT_S8_ROW:
        m = to_dev(meta.astype(np.float32).reshape(rows, H, dk - K), dev)
    elif w.lo_format == core.FMT_E4M3:
        m = to_dev(meta.astype(np.float32).reshape(rows, H, dk - K, dv // 32), dev)
    else:
        m = to_dev(meta.view(np.int16).reshape(rows, H, dk - K, dv // 32, 2), dev)
    return (to_dev(hi.view(np.int16).reshape(rows, H, K, dv), dev),
            to_dev(codes.reshape(rows, H, dk - K, _code_cols(w)), dev), m)


def tiers_from_dev(w: wl.Workload, dev_tiers, units: int):
    hi, codes, meta = (t.cpu().numpy() for t in dev_tiers)
    H, dk, dv, K = w.heads, w.d_k, w.d_v, w.k_hi
    hi = hi.view(np.uint16).reshape(units, K, dv)
    if w.lo_format == core.FMT_S8_ROW:
        return hi, codes.view(np.int8).reshape(units, dk - K, dv), meta.astype(np.float32).reshape(units, dk - K)
    if w.lo_format == core.FMT_E4M3:
        return (hi, codes.view(np.uint8).reshape(units, dk - K, dv),
                meta.view(np.float32).reshape(units, dk - K, dv // 32))
    return (hi, codes.view(np.uint8).reshape(units, dk - K, _code_cols(w)),
            meta.view(np.uint16).reshape(units, dk - K, dv // 32, 2))


def oracle_step(w: wl.Workload, perm_units, tiers, u: dict):
    """One oracle step from packed tiers: returns (o, new tiers, lo pre-quantization values).

    The pre-quantization values x (FP32, in the low tier's domain) are what the
    codes round; they serve to recognise rounding ties.
    """
    n = perm_units.shape[0]
    S = core.unpack_heads(perm_units, *tiers, w.k_hi, w.lo_format, w.d_k, w.d_v)
    o = core.delta_step_heads(S, u["q"], u["k"], u["v"], u["g"], u["beta"], w.kind)
    new = core.pack_heads(perm_units, S, w.k_hi, w.lo_format)
    lo_rows = np.stack([S[i][perm_units[i][w.k_hi:]] for i in range(n)])  # [n, d_k-K, d_v] natural
    if w.lo_format in (core.FMT_U8_H32, core.FMT_U4_H32) and lo_rows.size:
        lo_rows = core.hadamard32(lo_rows.reshape(-1, 32)).reshape(lo_rows.shape)
    return o, new, lo_rows


class CodeStats:
    def __init__(self):
        self.codes = 0
        self.mismatched = 0
        self.groups = 0
        self.meta_mismatched = 0

    def check_fraction(self):
        if self.codes:
            assert self.mismatched <= CODE_FRAC * self.codes, \
                f"{self.mismatched} of {self.codes} codes differ (> {CODE_FRAC:.1%})"


def _f16(bits):
    return core.f16_to_f32(bits.astype(np.uint16)).astype(np.float64)


def compare_tiers(w: wl.Workload, ref, gpu, lo_pre, stats: CodeStats, what=""):
    """Compare packed tiers; lo_pre = oracle pre-quantization values [n, d_k-K, d_v]."""
    hi_r, codes_r, meta_r = ref
    hi_g, codes_g, meta_g = gpu
    if hi_r.size:
        a, b = _f16(hi_g), _f16(hi_r)
        bad = np.abs(a - b) > ATOL + RTOL * np.abs(b)
        assert not bad.any(), f"{what}: FP16 tier differs at {np.argwhere(bad)[:5].tolist()}"
    if not codes_r.size:
        return
    if w.lo_format == core.FMT_S8_ROW:
        _compare_s8_rows(ref, gpu, lo_pre, stats, what)
        return
    if w.lo_format == core.FMT_E4M3:
        _compare_e4m3(ref, gpu, lo_pre, stats, what)
        return
    levels = 255.0
    if w.lo_format in (core.FMT_U4_H32, core.FMT_U4):  # nibbles to one code per value
        levels = 15.0
        codes_r = np.stack([codes_r & 15, codes_r >> 4], axis=-1).reshape(*codes_r.shape[:-1], -1)
        codes_g = np.stack([codes_g & 15, codes_g >> 4], axis=-1).reshape(*codes_g.shape[:-1], -1)
    n, lo, dv = codes_r.shape
    G = dv // 32
    cr = codes_r.reshape(n, lo, G, 32).astype(np.int64)
    cg = codes_g.reshape(n, lo, G, 32).astype(np.int64)
    d = np.abs(cr - cg)
    s_r, z_r = _f16(meta_r[..., 0]), _f16(meta_r[..., 1])
    s_g, z_g = _f16(meta_g[..., 0]), _f16(meta_g[..., 1])
    meta_diff = (meta_r != meta_g).any(axis=-1)  # [n, lo, G]
    x = lo_pre.reshape(n, lo, G, 32).astype(np.float64)
    # groups with equal (s, z): codes within 1 LSB, and differing only at ties of x/s + z
    same = ~meta_diff[..., None]
    assert np.all(d[np.broadcast_to(same, d.shape)] <= 1), f"{what}: a code differs by more than 1 LSB"
    t = x / s_r[..., None] + z_r[..., None]
    near = np.abs(np.abs(t - np.floor(t)) - 0.5) < TIE
    code_bad = (d > 0) & ~near & same
    assert not code_bad.any(), f"{what}: codes differ away from a rounding tie at {np.argwhere(code_bad)[:5].tolist()}"
    if meta_diff.any():
        # (s, z) may move only because the oracle's own group sits at a rounding tie:
        # s32 = (x_max - x_min)/255 at a binary16 midpoint, or -x_min/s at a half-integer.
        assert np.all(np.abs(s_g - s_r)[meta_diff] <= np.abs(s_r)[meta_diff] * 2.0 ** -10 + 1e-30), \
            f"{what}: scale differs by more than one binary16 ulp"
        assert np.all(np.abs(z_g - z_r)[meta_diff] <= 1), f"{what}: zero point differs by more than 1"
        xmin, xmax = x.min(axis=-1), x.max(axis=-1)
        s32 = (xmax - xmin) / levels
        sp = np.spacing(s32.astype(np.float16)).astype(np.float64)
        frac_s = np.abs((s32 / sp) - np.floor(s32 / sp) - 0.5)   # 0 at a binary16 rounding midpoint
        frac_z = np.abs((-xmin / s_r) - np.floor(-xmin / s_r) - 0.5)
        tie = (frac_s * sp < TIE_REL * np.abs(s32) + 1e-30) | (frac_z < TIE)
        bad = meta_diff & ~tie
        assert not bad.any(), f"{what}: (s, z) differ away from a rounding tie at {np.argwhere(bad)[:5].tolist()}"
        # A code means the level q - z of its group.  Where only z moved (a tie of
        # -x_min/s), every raw code of the group shifts with z, and the 1-LSB bound
        # holds for the level: |(q_gpu - z_gpu) - (q_ref - z_ref)| <= 1.
        z_only = meta_diff & (s_g == s_r)
        lvl = np.abs((cg - z_g[..., None]) - (cr - z_r[..., None]))
        assert np.all(lvl[np.broadcast_to(z_only[..., None], lvl.shape)] <= 1), \
            f"{what}: a code level differs by more than 1 LSB in a group whose zero point moved"
        # in such a group the reconstructed level s (q - z) moves by at most one step
        rec_r = s_r[..., None] * (cr - z_r[..., None])
        rec_g = s_g[..., None] * (cg - z_g[..., None])
        step = np.maximum(s_r, s_g)[..., None] * 1.01
        far = (np.abs(rec_g - rec_r) > step) & meta_diff[..., None]
        assert not far.any(), f"{what}: a reconstructed value moves by more than one step at {np.argwhere(far)[:5].tolist()}"
    stats.codes += d.size
    stats.mismatched += int((d > 0).sum())
    stats.groups += meta_diff.size
    stats.meta_mismatched += int(meta_diff.sum())


S8_SCALE_REL = 1e-5  # a row scale is max|x|/127 of values that may differ by float ordering


def _compare_s8_rows(ref, gpu, lo_pre, stats: CodeStats, what):
    """Row-absmax INT8 rows: scales within S8_SCALE_REL, codes within 1 and only at
    ties of the oracle's own x/s."""
    _, codes_r, s_r = ref
    _, codes_g, s_g = gpu
    s_r64, s_g64 = s_r.astype(np.float64), s_g.astype(np.float64)
    assert np.all(np.abs(s_g64 - s_r64) <= S8_SCALE_REL * np.abs(s_r64) + 1e-30), \
        f"{what}: a row scale differs beyond float ordering"
    d = np.abs(codes_r.astype(np.int64) - codes_g.astype(np.int64))
    assert np.all(d <= 1), f"{what}: a code differs by more than 1 LSB"
    with np.errstate(divide="ignore", invalid="ignore"):
        t = np.where(s_r64[..., None] > 0, lo_pre.astype(np.float64) / s_r64[..., None], 0.0)
    near = np.abs(np.abs(t - np.floor(t)) - 0.5) < TIE
    bad = (d > 0) & ~near
    assert not bad.any(), f"{what}: codes differ away from a rounding tie at {np.argwhere(bad)[:5].tolist()}"
    stats.codes += d.size
    stats.mismatched += int((d > 0).sum())
    stats.groups += s_r.size
    stats.meta_mismatched += int((s_r != s_g).sum())


_E4M3 = None


def _e4m3_magnitudes():
    global _E4M3
    if _E4M3 is None:
        _E4M3 = np.array([core.e4m3_to_f32(c) for c in range(0x7F)], np.float64)
    return _E4M3


def _compare_e4m3(ref, gpu, lo_pre, stats: CodeStats, what):
    """FP8 E4M3 groups: scales within S8_SCALE_REL (max|x| / 448 of values that may differ
    by float ordering); a code may differ only where the oracle's x/s lies within TIE (in
    units of the local E4M3 spacing) of the midpoint of two neighbouring values, and then
    by that one step."""
    _, codes_r, s_r = ref
    _, codes_g, s_g = gpu
    s_r64, s_g64 = s_r.astype(np.float64), s_g.astype(np.float64)
    assert np.all(np.abs(s_g64 - s_r64) <= S8_SCALE_REL * np.abs(s_r64) + 1e-30), f"{what}: an FP8 scale differs"
    mags = _e4m3_magnitudes()
    n, lo, dv = codes_r.shape
    vr = np.where(codes_r & 0x80, -1.0, 1.0) * mags[np.minimum(codes_r & 0x7F, 0x7E)]
    vg = np.where(codes_g & 0x80, -1.0, 1.0) * mags[np.minimum(codes_g & 0x7F, 0x7E)]
    diff = codes_r != codes_g
    if diff.any():
        t = np.abs(lo_pre.astype(np.float64) / np.repeat(s_r64, 32, axis=-1))
        k = np.clip(np.searchsorted(mags, np.minimum(t, 448.0)), 1, mags.size - 1)
        gap = mags[k] - mags[k - 1]
        mid = (mags[k] + mags[k - 1]) / 2
        near = np.abs(t - mid) < TIE * gap
        bad = diff & ~(near & (np.abs(vr - vg) <= gap * 1.0001))
        assert not bad.any(), f"{what}: FP8 codes differ away from a rounding tie at {np.argwhere(bad)[:5].tolist()}"
    stats.codes += codes_r.size
    stats.mismatched += int(diff.sum())
    stats.groups += s_r.size
    stats.meta_mismatched += int((s_r != s_g).sum())


def compare_o(o_gpu, o_ref, what=""):
    bad = np.abs(o_gpu - o_ref) > ATOL + RTOL * np.abs(o_ref)
    assert not bad.any(), (f"{what}: o differs at {np.argwhere(bad)[:5].tolist()} "
                           f"max {np.abs(o_gpu - o_ref).max():g}")


def initial_tiers(w: wl.Workload, rows, perms, prefix=None):
    """Oracle FP32 prefix for the given batch rows, packed with the per-head perms."""
    rows = list(rows)
    S0 = runs.prefix_states(w, rows, steps=prefix).reshape(len(rows) * w.heads, w.d_k, w.d_v)
    perm_units = np.tile(perms, (len(rows), 1))
    return perm_units, core.pack_heads(perm_units, S0, w.k_hi, w.lo_format)


def run_teacher_forced(w: wl.Workload, steps: int, dev, rows=None, n_docs=2, n_tokens=16, slot_of=None, pool=None,
                       u8=False):
    """Teacher-forced steps through the C ABI against the oracle: every GPU step starts
    from the oracle's packed state, so one rounding tie never compounds."""
    rows = list(range(w.batch)) if rows is None else list(rows)
    perms, _ = runs.calibrate_layout(w, n_docs=n_docs, n_tokens=n_tokens)
    perm_units, tiers = initial_tiers(w, rows, perms, prefix=min(w.prefix, 32))
    L = layout_of(w)
    n_slots = pool or len(rows)
    state = damp.new_state(L, n_slots, dev)
    slot_idx = None if slot_of is None else torch.tensor([slot_of[b] for b in range(len(rows))],
                                                         dtype=torch.int32, device=dev)
    dperm = to_dev(perms, dev)
    stats = CodeStats()
    if u8:
        step = damp.u8_kda_decode_step if w.kind == "kda" else damp.u8_gdn_decode_step
    else:
        step = damp.kda_decode_step if w.kind == "kda" else damp.gdn_decode_step
    for t in range(steps):
        inp = wl.step_inputs(w, t, rows=rows)
        u = runs.unit_operands(w, inp)
        o_ref, new_ref, lo_pre = oracle_step(w, perm_units, tiers, u)
        damp.pack_tiers(L, *tiers_to_dev(w, tiers, len(rows), dev), state, slot_idx=slot_idx)
        d = inputs_to_dev(w, inp, dev)
        o = step(L, state, dperm, d["q"], d["k"], d["v"], d["g"], d["beta"], slot_idx=slot_idx)
        got = tiers_from_dev(w, damp.unpack_tiers(L, state, batch=len(rows), slot_idx=slot_idx),
                             len(rows) * w.heads)
        compare_o(o.cpu().numpy().reshape(-1, w.d_v), o_ref, f"{w.name} step {t}")
        compare_tiers(w, new_ref, got, lo_pre, stats, f"{w.name} step {t}")
        tiers = new_ref
    stats.check_fraction()
    return stats


# ---- prefill chunks (App. A.5) ----

def chunk_inputs(w, t0, T, rows):
    """Per-token draws of the decode stream, stacked on a token axis after the batch axis."""
    steps = [wl.step_inputs(w, t0 + t, rows=rows) for t in range(T)]
    return {key: np.stack([s[key] for s in steps], axis=1) for key in steps[0]}


def unit_chunk(w, inp, T):
    """Per-(slot, head) operands [n, T, ...] (GQA expanded) for the oracle."""
    per_t = [runs.unit_operands(w, {key: val[:, t] for key, val in inp.items()}) for t in range(T)]
    return {key: np.stack([u[key] for u in per_t], axis=1) for key in per_t[0]}


def oracle_chunk(w, perm_units, tiers, u, lens_units):
    """The oracle's chunk, plus its chunk-final FP32 state for the tie rules."""
    n = perm_units.shape[0]
    S = core.unpack_heads(perm_units, *tiers, w.k_hi, w.lo_format, w.d_k, w.d_v)
    for t in range(u["q"].shape[1]):
        live = lens_units > t
        if live.any():
            sub = np.ascontiguousarray(S[live])
            core.delta_step_heads(sub, u["q"][live, t], u["k"][live, t], u["v"][live, t], u["g"][live, t],
                                  u["beta"][live, t], w.kind)
            S[live] = sub
    new = tuple(np.ascontiguousarray(t).copy() for t in tiers)
    o = core.prefill_chunk_heads(perm_units, *new, u["q"], u["k"], u["v"], u["g"], u["beta"], w.k_hi, w.lo_format,
                                 w.kind, lengths=lens_units)
    assert np.array_equal(core.unpack_heads(perm_units, *new, w.k_hi, w.lo_format, w.d_k, w.d_v)[lens_units > 0],
                          core.unpack_heads(perm_units, *core.pack_heads(perm_units, S, w.k_hi, w.lo_format),
                                            w.k_hi, w.lo_format, w.d_k, w.d_v)[lens_units > 0])
    lo_rows = np.stack([S[i][perm_units[i][w.k_hi:]] for i in range(n)])
    if w.lo_format in (core.FMT_U8_H32, core.FMT_U4_H32) and lo_rows.size:
        lo_rows = core.hadamard32(lo_rows.reshape(-1, 32)).reshape(lo_rows.shape)
    return o, new, lo_rows
