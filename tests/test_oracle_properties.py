"""Property-based pins of the oracle's UINT8 affine quantizer (Sec. 3.2 Eq.
integer_quantizer; App. A.1) on groups built to reach its edge cases: few distinct
values, tight one-signed blocks, binary16-subnormal scales, wide dynamic ranges.
Groups whose zero point would exceed binary16's range (|z| > 65504) are outside the
quantizer's contract and are not generated."""
import numpy as np
import pytest

from oracle import core

hypothesis = pytest.importorskip("hypothesis")
st = pytest.importorskip("hypothesis.strategies")
from hypothesis import assume, given, settings  # noqa: E402


@st.composite
def groups(draw):
    base = draw(st.floats(min_value=-1e3, max_value=1e3, allow_nan=False, allow_infinity=False, width=32))
    spread = draw(st.floats(min_value=0.0, max_value=1e3, allow_nan=False, allow_infinity=False, width=32))
    levels = draw(st.integers(min_value=1, max_value=32))
    picks = draw(st.lists(st.integers(min_value=0, max_value=levels - 1), min_size=32, max_size=32))
    fr = draw(st.lists(st.floats(min_value=-1.0, max_value=1.0, width=32), min_size=levels, max_size=levels))
    x = np.array([base + spread * fr[i] for i in picks], np.float32)
    assume(np.all(np.isfinite(x)))
    return x


def _params(x):
    q, sz = core.quant_group_u8(x)
    s = float(core.f16_to_f32(sz[0:1])[0])
    z = float(core.f16_to_f32(sz[1:2])[0])
    return q, sz, s, z


@settings(max_examples=400, deadline=None)
@given(groups())
def test_quantizer_invariants(x):
    mn, mx = float(x.min()), float(x.max())
    s32 = (max(mx, 0.0) - min(mn, 0.0)) / 255.0
    assume(s32 == 0.0 or abs(min(mn, 0.0)) / max(s32, 1e-30) < 6e4)  # |z| within binary16
    assume((mx - mn) == 0.0 or abs(mn) / ((mx - mn) / 255.0) < 6e4)
    q, sz, s, z = _params(x)
    # s > 0 always (degenerate blocks widen to 0, an all-zero block takes s = 1), z an integer
    assert s > 0 and np.isfinite(s) and z == np.round(z)
    # s is binary16 round-to-nearest-even of the FP32 range / 255 (Sec. 3.2, App. A.1),
    # taken over [min, max], or over the range widened to contain 0 only when that
    # rounds to 0; z is binary16 of rint(-min / s) over the same range
    f32 = np.float32
    lo, hi = f32(mn), f32(mx)
    s_ref = float(np.float16((hi - lo) / f32(255)))
    if s_ref == 0.0:
        lo, hi = min(lo, f32(0)), max(hi, f32(0))
        s_ref = float(np.float16((hi - lo) / f32(255)))
    if s_ref == 0.0:
        assert s == 1.0 and z == 0.0
    else:
        assert s == s_ref, (s, s_ref)
        assert z == float(np.float16(np.rint(-lo / f32(s)))), z
    # codes: the nearest integer to x/s + z (clamped), except at ties of float64 rounding
    y = x.astype(np.float64) / s + z
    near_tie = np.abs(np.abs(y - np.floor(y)) - 0.5) < 1e-4
    want = np.clip(np.round(y), 0, 255)
    assert np.array_equal(q[~near_tie], want[~near_tie].astype(np.uint8))
    # unsaturated entries reconstruct within half a step
    rec = core.dequant_group_u8(q, sz).astype(np.float64)
    unsat = (y > 0.5) & (y < 254.5)
    assert np.all(np.abs(rec - x)[unsat] <= 0.5 * s * (1 + 1e-5) + 1e-6 * np.abs(x[unsat]))
    # re-encoding the reconstruction with the stored (s, z) returns the same codes
    y2 = rec / s + z
    assert np.array_equal(np.clip(np.round(y2), 0, 255).astype(np.uint8), q)
