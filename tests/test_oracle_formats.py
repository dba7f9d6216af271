"""Pins of the oracle's 4-bit and FP8 low tiers (App. A.1, Tab. quantizer_specs and
Eq. fp8_storage; Eq. integer_quantizer with b = 4), checked against the format
definitions by brute force and against the bits the paper prints."""
import math

import numpy as np
import pytest

from oracle import core
from tests.golden.load import paper_values

PV = paper_values()


def _e4m3_table():
    """Every finite E4M3 magnitude from the definition: 2^(e-7)(1 + m/8), e = 1..15
    (m <= 6 at e = 15), and 2^-6 (m/8) for e = 0."""
    vals = [(m / 8.0) * 2.0 ** -6 for m in range(8)]
    for e in range(1, 16):
        for m in range(8):
            if e == 15 and m == 7:
                continue
            vals.append((1 + m / 8.0) * 2.0 ** (e - 7))
    return np.array(vals)


def test_e4m3_decode_matches_the_definition():
    table = _e4m3_table()
    for code in range(256):
        v = core.e4m3_to_f32(code)
        if code & 0x7F == 0x7F:
            assert math.isnan(v)
            continue
        mag = table[code & 0x7F]
        assert v == (-mag if code & 0x80 else mag)
    assert core.e4m3_to_f32(0x7E) == 448.0 and core.e4m3_to_f32(0x01) == 2.0 ** -9
    assert core.e4m3_to_f32(0x38) == 1.0 and core.e4m3_to_f32(0x08) == 2.0 ** -6
    assert np.all(np.diff(table) > 0)  # codes 0x00..0x7E increase


def test_e4m3_encode_is_nearest_with_ties_to_even():
    table = _e4m3_table()
    rng = np.random.default_rng(51)
    xs = list((np.exp(rng.uniform(np.log(2.0 ** -12), np.log(600.0), 4000)) *
               rng.choice([-1, 1], 4000)).astype(np.float32))
    mids = (table[:-1] + table[1:]) / 2       # exact midpoints (representable in float32)
    xs += list(mids.astype(np.float32)) + list((-mids).astype(np.float32))
    for x in xs:
        code = core.f32_to_e4m3(float(x))
        a = min(abs(float(x)), 448.0)
        d = np.abs(table - a)
        best = np.flatnonzero(d == d.min())
        if best.size == 2:                     # a tie: the even mantissa wins
            best = best[[(i & 1) == 0 for i in best]]
        assert code & 0x7F == best[0], (x, code)
        assert (code >> 7) == (1 if np.signbit(x) else 0)
    for code in range(0x7F):                   # every finite code round-trips
        assert core.f32_to_e4m3(core.e4m3_to_f32(code)) == code
    assert core.f32_to_e4m3(1e6) == 0x7E and core.f32_to_e4m3(-1e6) == 0xFE


def _groups(seed, n=800):
    rng = np.random.default_rng(seed)
    scale = 10.0 ** rng.uniform(-4, 2, (n, 1))
    shift = rng.uniform(-1, 1, (n, 1)) * scale * rng.integers(0, 2, (n, 1)) * 3
    return (rng.standard_normal((n, 32)) * scale + shift).astype(np.float32)


def test_fp8_group_quantizer():
    table = _e4m3_table()
    for x in _groups(52):
        q, s = core.quant_group_e4m3(x)
        amax = np.float32(np.abs(x).max())
        assert s == np.float32(max(amax, np.float32(1e-10)) / np.float32(448.0))
        i = int(np.argmax(np.abs(x)))
        assert abs(core.e4m3_to_f32(int(q[i]))) == 448.0
        rec = core.dequant_group_e4m3(q, s).astype(np.float64)
        t = np.abs(x.astype(np.float64) / s)
        k = np.searchsorted(table, np.minimum(t, 448.0))
        gap = table[np.minimum(k, table.size - 1)] - table[np.maximum(k - 1, 0)]
        assert np.all(np.abs(rec - x) <= 0.5 * gap * s * (1 + 1e-5) + 1e-7 * np.abs(x))
    q, s = core.quant_group_e4m3(np.zeros(32, np.float32))
    assert not q.any() and s == np.float32(1e-10) / np.float32(448.0)


def test_uint4_quantizer():
    for x in _groups(53):
        q, sz = core.quant_group_u4(x)
        codes = np.stack([q & 15, q >> 4], axis=1).reshape(32)  # value 2i in the low nibble
        s = float(core.f16_to_f32(sz[0:1])[0])
        z = float(core.f16_to_f32(sz[1:2])[0])
        assert s > 0 and z == round(z)
        exact = (float(x.max()) - float(x.min())) / 15.0
        assert abs(s - exact) <= 0.5 * float(np.spacing(np.float16(exact))) * 1.001 + exact * 2.0 ** -23
        y = x.astype(np.float64) / s
        near_tie = np.abs(np.abs(y - np.floor(y)) - 0.5) < 1e-4
        want = np.clip(np.round(y) + z, 0, 15)
        assert np.array_equal(codes[~near_tie], want[~near_tie].astype(np.uint8))
        rec = core.dequant_group_u4(q, sz)
        assert np.allclose(rec, s * (codes.astype(np.float64) - z), rtol=1e-6, atol=0)


@pytest.mark.parametrize("fmt", [core.FMT_U4_H32, core.FMT_U4, core.FMT_E4M3])
def test_packed_tiers_round_trip_and_protect_fp16_rows(fmt):
    rng = np.random.default_rng(54)
    n, d_k, d_v, K = 3, 32, 64, 4
    S = rng.standard_normal((n, d_k, d_v)).astype(np.float32)
    perm = np.stack([rng.permutation(d_k) for _ in range(n)]).astype(np.uint8)
    tiers = core.pack_heads(perm, S, K, fmt)
    back = core.unpack_heads(perm, *tiers, K, fmt, d_k, d_v)
    for i in range(n):
        hi = perm[i][:K]
        assert np.array_equal(back[i][hi], S[i][hi].astype(np.float16).astype(np.float32))
    again = core.pack_heads(perm, back, K, fmt)      # reconstructed states re-encode to the same tiers
    for a, b in zip(tiers, again):
        assert np.array_equal(a, b)


def test_bits_per_value_of_the_new_tiers_match_the_paper():
    assert core.bits_per_value(128, 128, 0, core.FMT_U4) == PV["bits_int4"]
    assert core.bits_per_value(128, 128, 0, core.FMT_U4_H32) == PV["bits_int4"]
    assert core.bits_per_value(128, 128, 0, core.FMT_E4M3) == PV["bits_fp8"]
    assert core.bits_per_value(128, 128, 16, core.FMT_U4_H32) == 16 / 128 * 16 + 112 / 128 * 5.0
