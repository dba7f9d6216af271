"""Pins of the CPU oracle against what the paper and the mathematics fix.

No pin retypes an oracle formula: each checks a library routine (numpy's
binary16, scipy's Hadamard matrix), a closed form, an invariant, a brute-force
float64 evaluation of a different form of the same equation, or a value the
paper prints (tests/golden/paper_values.txt).
"""
import numpy as np
import pytest
import scipy.linalg

from oracle import calibrate, core
from tests.golden.load import paper_values

PV = paper_values()


# ---------------------------------------------------------------- binary16 ---

def test_f16_to_f32_matches_numpy_for_every_bit_pattern():
    h = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    ours = core.f16_to_f32(h)
    ref = h.view(np.float16).astype(np.float32)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(ours), nan)
    assert np.array_equal(ours[~nan].view(np.uint32), ref[~nan].view(np.uint32))


def test_f32_to_f16_matches_numpy_round_to_nearest_even():
    rng = np.random.default_rng(0)
    halves = np.arange(65536, dtype=np.uint32).astype(np.uint16).view(np.float16)
    halves = halves[np.isfinite(halves)].astype(np.float32)
    # exact values, midpoints between neighbours and one float32 ulp either side of them
    srt = np.unique(halves.astype(np.float64))
    mids = ((srt[1:] + srt[:-1]) / 2).astype(np.float32)
    cases = [halves, mids, np.nextafter(mids, np.float32(np.inf)), np.nextafter(mids, np.float32(-np.inf)),
             rng.standard_normal(200000).astype(np.float32) * np.float32(1e-3),
             (rng.standard_normal(200000) * 10.0 ** rng.uniform(-9, 6, 200000)).astype(np.float32),
             np.array([65504, 65519.99, 65520, 65536, 1e30, -1e30, np.inf, -np.inf, 0.0, -0.0,
                       2.0 ** -25, 2.0 ** -25 * 1.0000001, 2.0 ** -24, 3 * 2.0 ** -26, 1e-45], np.float32)]
    x = np.concatenate(cases).astype(np.float32)
    ours = core.f32_to_f16(x)
    with np.errstate(over="ignore"):
        ref = x.astype(np.float16).view(np.uint16)
    assert np.array_equal(ours, ref)


# ------------------------------------------------------------ Hadamard H_32 ---

def test_hadamard_matches_scipy_sylvester_matrix():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((64, 32)).astype(np.float32)
    H = scipy.linalg.hadamard(32).astype(np.float64) / np.sqrt(32.0)
    ref = x.astype(np.float64) @ H.T
    ours = core.hadamard32(x).astype(np.float64)
    assert np.max(np.abs(ours - ref)) <= 1e-6 * np.max(np.abs(ref))


def test_hadamard_is_its_own_inverse_and_preserves_norm():
    rng = np.random.default_rng(2)
    x = rng.standard_normal((32, 32)).astype(np.float32)
    y = core.hadamard32(x)
    xx = core.hadamard32(y)
    assert np.allclose(xx, x, rtol=0, atol=2e-6)
    assert np.allclose(np.linalg.norm(y, axis=1), np.linalg.norm(x, axis=1), rtol=1e-6)


def test_hadamard_closed_forms():
    e0 = np.zeros(32, np.float32)
    e0[0] = 1
    e1 = np.zeros(32, np.float32)
    e1[1] = 1
    c = np.float32(1 / np.sqrt(32))
    assert np.array_equal(core.hadamard32(e0), np.full(32, c, np.float32))
    assert np.array_equal(core.hadamard32(e1), np.where(np.arange(32) % 2 == 0, c, -c).astype(np.float32))


# ------------------------------------------------------- UINT8 affine G = 32 ---

def _rand_groups(seed, n=2000):
    rng = np.random.default_rng(seed)
    scale = 10.0 ** rng.uniform(-4, 2, (n, 1))
    shift = rng.uniform(-1, 1, (n, 1)) * scale * rng.integers(0, 2, (n, 1)) * 3
    return (rng.standard_normal((n, 32)) * scale + shift).astype(np.float32)


def test_codes_in_range_and_error_within_half_step():
    for x in _rand_groups(3):
        q, sz = core.quant_group_u8(x)
        s = core.f16_to_f32(sz[0:1])[0]
        z = core.f16_to_f32(sz[1:2])[0]
        assert s > 0 and z == np.round(z)
        rec = core.dequant_group_u8(q, sz).astype(np.float64)
        # unsaturated entries reconstruct within half a step (plus float32 rounding)
        t = x.astype(np.float64) / s + z
        unsat = (t > 0.5) & (t < 254.5)
        err = np.abs(rec - x)[unsat]
        assert np.all(err <= 0.5 * s * (1 + 1e-5) + 1e-6 * np.abs(x[unsat]))


def test_codes_are_the_nearest_integer_in_float64():
    """Brute force: q_i = clamp(nearest integer to x_i/s + z) except within 1e-4 of a tie."""
    for x in _rand_groups(4, 500):
        q, sz = core.quant_group_u8(x)
        s = float(core.f16_to_f32(sz[0:1])[0])
        z = float(core.f16_to_f32(sz[1:2])[0])
        y = x.astype(np.float64) / s
        near_tie = np.abs(np.abs(y - np.floor(y)) - 0.5) < 1e-4
        want = np.clip(np.round(y) + z, 0, 255)
        assert np.array_equal(q[~near_tie], want[~near_tie].astype(np.uint8))


def test_scale_is_range_over_255_rounded_to_fp16():
    """s is the binary16 neighbour of (x_max - x_min)/255 nearest in float64 terms."""
    for x in _rand_groups(5, 500):
        _, sz = core.quant_group_u8(x)
        s = float(core.f16_to_f32(sz[0:1])[0])
        exact = (float(x.max()) - float(x.min())) / 255.0
        # neighbours in binary16
        lo = float(np.float16(exact))
        assert abs(s - exact) <= abs(lo - exact) * (1 + 1e-3) + 1e-12
        half_spacing = 0.5 * float(np.spacing(np.float16(exact)))
        assert abs(s - exact) <= half_spacing * 1.001 + exact * 2.0 ** -23


def test_full_span_round_trip_is_exact():
    """Codes that span 0..255, decoded with any FP16 s and small z, re-encode to themselves."""
    rng = np.random.default_rng(6)
    for _ in range(500):
        q = rng.integers(0, 256, 32).astype(np.uint8)
        q[rng.integers(0, 32)] = 0
        q[rng.integers(0, 32)] = 255
        if q.min() != 0 or q.max() != 255:
            continue
        s = np.float16(10.0 ** rng.uniform(-4, 1)).astype(np.float32)
        z = np.float32(rng.integers(0, 256))
        sz = core.f32_to_f16(np.array([s, z], np.float32))
        x = core.dequant_group_u8(q, sz)
        q2, sz2 = core.quant_group_u8(x)
        assert np.array_equal(q2, q) and np.array_equal(sz2, sz)


def test_degenerate_blocks():
    c = np.float32(0.75)
    q, sz = core.quant_group_u8(np.full(32, c, np.float32))
    assert np.all(q == 255) and abs(core.dequant_group_u8(q, sz)[0] - c) <= c / 255
    q, sz = core.quant_group_u8(np.full(32, -c, np.float32))
    assert np.all(q == 0) and abs(core.dequant_group_u8(q, sz)[0] + c) <= c / 255
    q, sz = core.quant_group_u8(np.zeros(32, np.float32))
    assert np.all(q == 0) and np.all(core.dequant_group_u8(q, sz) == 0)


def test_power_of_two_scaling_is_exact():
    """Q(2^m x) = 2^m Q(x) while s stays a normal binary16: the quantizer is scale-covariant."""
    for x in _rand_groups(7, 200):
        if not (1e-2 < np.abs(x).max() < 10):
            continue
        q1, sz1 = core.quant_group_u8(x)
        q2, sz2 = core.quant_group_u8(x * np.float32(4.0))
        assert np.array_equal(q1, q2)
        assert np.array_equal(core.dequant_group_u8(q2, sz2), core.dequant_group_u8(q1, sz1) * 4)


def test_row_absmax_s8():
    rng = np.random.default_rng(8)
    x = rng.standard_normal(128).astype(np.float32)
    q, s = core.quant_row_s8(x)
    assert abs(s - np.abs(x).max() / 127) <= 1e-7 * s
    assert q.min() >= -127 and q.max() <= 127 and np.abs(q).max() == 127
    assert np.all(np.abs(s * q.astype(np.float64) - x) <= 0.5 * s * (1 + 1e-5))
    q0, s0 = core.quant_row_s8(np.zeros(16, np.float32))
    assert s0 == 0 and np.all(q0 == 0)


# ------------------------------------------------------------ packed tiers ---

def test_all_fp16_pack_equals_numpy_fp16_rounding():
    rng = np.random.default_rng(9)
    S = (rng.standard_normal((3, 64, 64)) * 3).astype(np.float32)
    perm = np.stack([rng.permutation(64) for _ in range(3)]).astype(np.uint8)
    hi, codes, meta = core.pack_heads(perm, S, 64, core.FMT_U8_H32)
    assert codes.size == 0 and meta.size == 0
    for n in range(3):
        assert np.array_equal(hi[n], S[n][perm[n]].astype(np.float16).view(np.uint16))
    back = core.unpack_heads(perm, hi, codes, meta, 64, core.FMT_U8_H32, 64, 64)
    assert np.array_equal(back, S.astype(np.float16).astype(np.float32))


@pytest.mark.parametrize("fmt", [core.FMT_U8_H32, core.FMT_U8, core.FMT_S8_ROW])
def test_pack_places_protected_channels_in_fp16_tier(fmt):
    rng = np.random.default_rng(10)
    d_k, d_v, K = 64, 96, 8
    S = (rng.standard_normal((2, d_k, d_v))).astype(np.float32)
    perm = np.stack([rng.permutation(d_k) for _ in range(2)]).astype(np.uint8)
    hi, codes, meta = core.pack_heads(perm, S, K, fmt)
    back = core.unpack_heads(perm, hi, codes, meta, K, fmt, d_k, d_v)
    for n in range(2):
        prot = perm[n][:K]
        rest = perm[n][K:]
        assert np.array_equal(back[n][prot], S[n][prot].astype(np.float16).astype(np.float32))
        err = np.abs(back[n][rest] - S[n][rest])
        rowmax = np.abs(S[n][rest]).max(axis=1, keepdims=True)
        # low tier: error bounded by one quantization step of the row's range (H_32 preserves norms)
        assert np.all(err <= rowmax * 2 * np.sqrt(32) / 127)
        assert err.max() > 0


def test_pack_rejects_invalid_permutation():
    S = np.zeros((1, 32, 32), np.float32)
    bad = np.zeros((1, 32), np.uint8)
    with pytest.raises(ValueError):
        core.pack_heads(bad, S, 4, 0)


# ---------------------------------------------- the recurrence (Sec. 3.1) ---

def _dense_recurrence_f64(S0, qs, ks, vs, a_s, betas):
    """Eq. recurrence: S_t = A_t S_{t-1} + beta k v^T, A_t = (I - beta k k^T) Lambda_t, in float64."""
    S = S0.astype(np.float64)
    outs = []
    d_k = S.shape[0]
    for q, k, v, a, b in zip(qs, ks, vs, a_s, betas):
        k = k.astype(np.float64)
        A = (np.eye(d_k) - b * np.outer(k, k)) @ np.diag(a.astype(np.float64))
        S = A @ S + b * np.outer(k, v)
        outs.append(S.T @ q.astype(np.float64))
    return S, outs


@pytest.mark.parametrize("kind", ["gdn", "kda"])
@pytest.mark.parametrize("d", [4, 8, 16])
def test_delta_step_equals_dense_recurrence(kind, d):
    rng = np.random.default_rng(11 + d)
    T = 12
    S = rng.standard_normal((1, d, d)).astype(np.float32)
    S0 = S[0].copy()
    qs, ks, vs, gs, bs, a_s, outs = [], [], [], [], [], [], []
    for _ in range(T):
        q = rng.standard_normal(d)
        k = rng.standard_normal(d)
        q, k = q / np.linalg.norm(q), k / np.linalg.norm(k)
        v = rng.standard_normal(d)
        b = 1 / (1 + np.exp(-rng.standard_normal()))
        g = -np.logaddexp(0, rng.standard_normal()) if kind == "gdn" else -np.exp(rng.uniform(-6, 0, d))
        q, k, v = (x.astype(np.float32) for x in (q, k, v))
        g = np.float32(g) if kind == "gdn" else g.astype(np.float32)
        o = core.delta_step_heads(S, q[None], k[None], v[None], np.atleast_1d(g)[None] if kind == "kda" else
                                  np.array([g], np.float32), np.array([b], np.float32), kind)
        a = np.full(d, np.exp(np.float64(g))) if kind == "gdn" else np.exp(g.astype(np.float64))
        qs.append(q), ks.append(k), vs.append(v), a_s.append(a), bs.append(np.float32(b)), outs.append(o[0])
    Sref, oref = _dense_recurrence_f64(S0, qs, ks, vs, a_s, bs)
    assert np.max(np.abs(S[0] - Sref)) <= 2e-5 * max(1.0, np.abs(Sref).max())
    for o, r in zip(outs, oref):
        assert np.max(np.abs(o - r)) <= 2e-5 * max(1.0, np.abs(r).max())


def test_zero_beta_unit_decay_leaves_state_bit_identical():
    rng = np.random.default_rng(12)
    S = rng.standard_normal((4, 32, 64)).astype(np.float32)
    S0 = S.copy()
    q = rng.standard_normal((4, 32)).astype(np.float32)
    core.delta_step_heads(S, q, q, rng.standard_normal((4, 64)).astype(np.float32), np.zeros((4, 32), np.float32),
                          np.zeros(4, np.float32), "kda")
    assert np.array_equal(S, S0)


def test_unit_beta_unit_decay_writes_v_along_k():
    """beta = 1, Lambda = I, ||k|| = 1: the updated state reads back v exactly along k."""
    rng = np.random.default_rng(13)
    S = rng.standard_normal((3, 64, 64)).astype(np.float32)
    k = rng.standard_normal((3, 64))
    k = (k / np.linalg.norm(k, axis=1, keepdims=True)).astype(np.float32)
    v = rng.standard_normal((3, 64)).astype(np.float32)
    core.delta_step_heads(S, k, k, v, np.zeros(3, np.float32), np.ones(3, np.float32), "gdn")
    readback = np.einsum("nuj,nu->nj", S.astype(np.float64), k.astype(np.float64))
    assert np.max(np.abs(readback - v)) < 1e-4


# --------------------------------- the quantized recurrence (Sec. 3.3) ---

@pytest.mark.parametrize("fmt", [core.FMT_U8_H32, core.FMT_U8])
@pytest.mark.parametrize("kind", ["gdn", "kda"])
def test_quantized_step_is_one_quantization_of_the_exact_recurrence(kind, fmt):
    """S^q_t = Q(A_t S^q_{t-1} + beta k v^T) (Eq. quantized_recurrence); o = X^T q before Q.

    X_t is evaluated in float64 with the dense A_t form from the reconstructed
    previous state; the stored state must sit within one quantization step of
    X_t, and o must match X_t^T q.
    """
    rng = np.random.default_rng(14)
    n, d_k, d_v, K = 3, 64, 64, 8
    S = (rng.standard_normal((n, d_k, d_v)) * 0.5).astype(np.float32)
    perm = np.stack([rng.permutation(d_k) for _ in range(n)]).astype(np.uint8)
    tiers = core.pack_heads(perm, S, K, fmt)
    for _ in range(6):
        prev = core.unpack_heads(perm, *tiers, K, fmt, d_k, d_v).astype(np.float64)
        q = rng.standard_normal((n, d_k))
        k = rng.standard_normal((n, d_k))
        q = (q / np.linalg.norm(q, axis=1, keepdims=True)).astype(np.float32)
        k = (k / np.linalg.norm(k, axis=1, keepdims=True)).astype(np.float32)
        v = rng.standard_normal((n, d_v)).astype(np.float32)
        beta = (1 / (1 + np.exp(-rng.standard_normal(n)))).astype(np.float32)
        g = (-np.logaddexp(0, rng.standard_normal(n)) if kind == "gdn"
             else -np.exp(rng.uniform(-6, 0, (n, d_k)))).astype(np.float32)
        o = core.mixed_step_heads(perm, *tiers, q, k, v, g, beta, K, fmt, kind)
        now = core.unpack_heads(perm, *tiers, K, fmt, d_k, d_v).astype(np.float64)
        for i in range(n):
            a = np.exp(np.full(d_k, g[i], np.float64) if kind == "gdn" else g[i].astype(np.float64))
            kk = k[i].astype(np.float64)
            A = (np.eye(d_k) - beta[i] * np.outer(kk, kk)) @ np.diag(a)
            X = A @ prev[i] + float(beta[i]) * np.outer(kk, v[i])
            assert np.max(np.abs(o[i] - X.T @ q[i])) <= 1e-4 * max(1.0, np.abs(X).max())
            R = now[i] - X
            hi_rows = perm[i][:K]
            lo_rows = perm[i][K:]
            assert np.all(np.abs(R[hi_rows]) <= np.abs(X[hi_rows]) * 2.0 ** -11 + 1e-4)
            span = np.abs(X[lo_rows]).max(axis=1, keepdims=True)
            step = 2 * span * (np.sqrt(32) if fmt == core.FMT_U8_H32 else 1) / 255
            assert np.all(np.abs(R[lo_rows]) <= step * 0.5 * np.sqrt(32) + 1e-4)


def test_error_recurrence_identity_on_a_trajectory():
    """Delta S_t = A_t Delta S_{t-1} + R_t (Eq. error_recurrence) along an oracle trajectory."""
    rng = np.random.default_rng(15)
    d_k = d_v = 32
    K = 4
    perm = rng.permutation(d_k).astype(np.uint8)[None]
    S_ref = np.zeros((1, d_k, d_v), np.float32)
    tiers = core.pack_heads(perm, S_ref, K, core.FMT_U8_H32)
    dS_prev = np.zeros((d_k, d_v))
    for t in range(20):
        prev_q = core.unpack_heads(perm, *tiers, K, 0, d_k, d_v)[0].astype(np.float64)
        q = rng.standard_normal(d_k)
        k = rng.standard_normal(d_k)
        q, k = (q / np.linalg.norm(q)).astype(np.float32), (k / np.linalg.norm(k)).astype(np.float32)
        v = rng.standard_normal(d_v).astype(np.float32)
        b = np.float32(0.7)
        g = (-np.exp(rng.uniform(-6, 0, d_k))).astype(np.float32)
        core.mixed_step_heads(perm, *tiers, q[None], k[None], v[None], g[None], np.array([b]), K, 0, "kda")
        core.delta_step_heads(S_ref, q[None], k[None], v[None], g[None], np.array([b]), "kda")
        A = (np.eye(d_k) - float(b) * np.outer(k, k)) @ np.diag(np.exp(g.astype(np.float64)))
        X = A @ prev_q + float(b) * np.outer(k, v)
        now_q = core.unpack_heads(perm, *tiers, K, 0, d_k, d_v)[0].astype(np.float64)
        R = now_q - X
        dS = now_q - S_ref[0].astype(np.float64)
        resid = dS - (A @ dS_prev + R)
        assert np.max(np.abs(resid)) <= 1e-4 * max(1e-3, np.abs(S_ref).max())
        dS_prev = dS


# ----------------------------------------------- calibration (Sec. 5.1) ---

def test_persistence_closed_forms():
    tau = PV["tau"]
    assert calibrate.TAU == tau
    assert calibrate.persistence(0.0) == 1.0
    assert calibrate.persistence(1.0) == 1 / tau
    assert calibrate.persistence(np.sqrt(1 - tau) + 1e-12) == pytest.approx(1 / tau)
    assert calibrate.persistence(0.5) == pytest.approx(4.0 / 3.0)
    # geometric sum: sum_j a^{2j} for a below the cap
    a = 0.9
    assert calibrate.persistence(a) == pytest.approx(sum(a ** (2 * j) for j in range(5000)))


def test_effective_decay_is_geometric_mean():
    a = np.array([[0.5, 0.9], [0.125, 0.9], [1.0, 0.9]])
    assert np.allclose(calibrate.effective_decay(np.log(a)), [(0.5 * 0.125 * 1.0) ** (1 / 3), 0.9])


def test_domain_balanced_mean_weights_domains_equally():
    vals = np.array([1.0, 1.0, 1.0, 5.0])
    assert calibrate.domain_balanced_mean(vals, [np.array([0, 1, 2]), np.array([3])]) == 3.0
    assert calibrate.domain_balanced_mean(vals) == 2.0


def test_topk_matches_full_sort_and_breaks_ties_low_index():
    rng = np.random.default_rng(16)
    for _ in range(50):
        c = rng.integers(0, 20, 64).astype(np.float64)
        k = int(rng.integers(0, 65))
        sel = calibrate.topk(c, k)
        order = np.lexsort((np.arange(64), -c))[:k]
        assert np.array_equal(sel, np.sort(order))


def test_stable_partition():
    pi = calibrate.stable_partition([9, 2, 5], 10)
    assert pi.tolist() == [2, 5, 9, 0, 1, 3, 4, 6, 7, 8]


def test_gdn_ranking_reduces_to_error_energy():
    """Persistence is shared within a GDN head, so TopK(E * P) == TopK(E) (Sec. 5.1)."""
    rng = np.random.default_rng(17)
    E = rng.random(128)
    for a in (0.1, 0.9, 0.99999):
        P = np.full(128, calibrate.persistence(a))
        H, _ = calibrate.select_layout(E, P, 16)
        assert np.array_equal(H, calibrate.topk(E, 16))


def test_error_energy_zero_for_exact_rows_and_quadratic_in_scale():
    rng = np.random.default_rng(18)
    # rows already on the quantizer's grid (full-span codes) reconstruct exactly under Q_lo without H
    rows = []
    for _ in range(4):
        q = rng.integers(0, 256, 32).astype(np.uint8)
        q[0], q[1] = 0, 255
        sz = core.f32_to_f16(np.array([0.01, 100.0], np.float32))
        rows.append(core.dequant_group_u8(q, sz))
    exact = np.stack(rows)[None]
    assert np.all(calibrate.error_energy(exact, core.FMT_U8) == 0)
    S = rng.standard_normal((5, 16, 64)).astype(np.float32)
    e1 = calibrate.error_energy(S, core.FMT_U8_H32)
    e4 = calibrate.error_energy(S * np.float32(4), core.FMT_U8_H32)
    assert np.allclose(e4, 16 * e1, rtol=1e-12)


def test_bits_per_value_from_bytes_matches_paper():
    assert core.bits_per_value(128, 128, 16, core.FMT_U8_H32) == PV["damp_bits_k16_dk128"]
    assert calibrate.bits_budgeted(16, 128, 16, 9.0) == PV["damp_bits_k16_dk128"]
    assert round(core.bits_per_value(128, 128, 16, 0), 1) == PV["damp_bits_reported"]
    assert core.bits_per_value(128, 128, 0, core.FMT_U8_H32) == PV["bits_int8_hadamard"]
    assert core.bits_per_value(128, 128, 0, core.FMT_U8) == PV["bits_int8"]
    assert core.bits_per_value(128, 128, 128, core.FMT_U8_H32) == PV["all_fp16_bits"]
    red = 100 * (1 - core.bits_per_value(128, 128, 16, 0) / 32)
    assert round(red, 1) == PV["storage_reduction_pct"]
    for K in range(0, 129, 4):
        assert core.bits_per_value(128, 128, K, 0) == calibrate.bits_budgeted(K, 128, 16, 9.0)
