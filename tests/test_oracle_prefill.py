"""Pins of the oracle's prefill chunk (App. A.5 "Prefill path"): the recurrence runs
exactly in FP32 over the chunk and the state is quantized once, at the chunk end."""
import numpy as np
import pytest

from oracle import core


def _tokens(rng, n, T, d_k, d_v, kind):
    q = rng.standard_normal((n, T, d_k))
    k = rng.standard_normal((n, T, d_k))
    q = (q / np.linalg.norm(q, axis=2, keepdims=True)).astype(np.float32)
    k = (k / np.linalg.norm(k, axis=2, keepdims=True)).astype(np.float32)
    v = rng.standard_normal((n, T, d_v)).astype(np.float32)
    beta = (1 / (1 + np.exp(-rng.standard_normal((n, T))))).astype(np.float32)
    if kind == "gdn":
        g = (-np.logaddexp(0, rng.standard_normal((n, T)))).astype(np.float32)
    else:
        g = (-np.exp(rng.uniform(-6, 0, (n, T, d_k)))).astype(np.float32)
    return q, k, v, g, beta


def _decay(g_t, kind, d_k):
    return np.exp(np.full(d_k, np.float64(g_t)) if kind == "gdn" else g_t.astype(np.float64))


def _copy(tiers):
    return tuple(np.ascontiguousarray(t).copy() for t in tiers)


@pytest.mark.parametrize("fmt", [core.FMT_U8_H32, core.FMT_U8, core.FMT_S8_ROW])
@pytest.mark.parametrize("kind", ["gdn", "kda"])
def test_chunk_is_one_quantization_of_the_exact_recurrence(kind, fmt):
    """Outputs follow the exact recurrence (Eq. recurrence in float64, dense A_t) from
    the reconstructed state; the stored state is one quantization of its end point.
    Quantizing after every token instead would fail the output check."""
    rng = np.random.default_rng(31)
    n, d_k, d_v, K, T = 3, 64, 64, 8, 10
    S0 = (rng.standard_normal((n, d_k, d_v)) * 0.5).astype(np.float32)
    perm = np.stack([rng.permutation(d_k) for _ in range(n)]).astype(np.uint8)
    tiers = core.pack_heads(perm, S0, K, fmt)
    start = core.unpack_heads(perm, *tiers, K, fmt, d_k, d_v).astype(np.float64)
    q, k, v, g, beta = _tokens(rng, n, T, d_k, d_v, kind)

    stepwise = _copy(tiers)
    o_step = [core.mixed_step_heads(perm, *stepwise, q[:, t], k[:, t], v[:, t], g[:, t], beta[:, t], K, fmt, kind)
              for t in range(T)]
    o = core.prefill_chunk_heads(perm, *tiers, q, k, v, g, beta, K, fmt, kind)
    now = core.unpack_heads(perm, *tiers, K, fmt, d_k, d_v).astype(np.float64)

    worst_stepwise = 0.0
    for i in range(n):
        X = start[i].copy()
        for t in range(T):
            kk = k[i, t].astype(np.float64)
            A = (np.eye(d_k) - beta[i, t] * np.outer(kk, kk)) @ np.diag(_decay(g[i, t], kind, d_k))
            X = A @ X + float(beta[i, t]) * np.outer(kk, v[i, t])
            ref = X.T @ q[i, t].astype(np.float64)
            scale = max(1.0, np.abs(X).max())
            assert np.max(np.abs(o[i, t] - ref)) <= 1e-4 * scale
            worst_stepwise = max(worst_stepwise, np.max(np.abs(o_step[t][i] - ref)) / scale)
        R = now[i] - X
        hi_rows, lo_rows = perm[i][:K], perm[i][K:]
        assert np.all(np.abs(R[hi_rows]) <= np.abs(X[hi_rows]) * 2.0 ** -11 + 1e-4)
        span = np.abs(X[lo_rows]).max(axis=1, keepdims=True)
        step = 2 * span * (np.sqrt(32) if fmt == core.FMT_U8_H32 else 1) / (255 if fmt != core.FMT_S8_ROW else 254)
        assert np.all(np.abs(R[lo_rows]) <= step * 0.5 * np.sqrt(32) + 1e-4)
    assert worst_stepwise > 1e-3  # the per-token quantization is visible: the checks above discriminate


def test_zero_tokens_leave_the_tiers_untouched():
    rng = np.random.default_rng(32)
    n, d_k, d_v, K = 2, 32, 64, 4
    perm = np.stack([rng.permutation(d_k) for _ in range(n)]).astype(np.uint8)
    tiers = core.pack_heads(perm, rng.standard_normal((n, d_k, d_v)).astype(np.float32), K, 0)
    before = _copy(tiers)
    q, k, v, g, beta = _tokens(rng, n, 3, d_k, d_v, "kda")
    o = core.prefill_chunk_heads(perm, *tiers, q, k, v, g, beta, K, 0, "kda", lengths=np.zeros(n, np.int32))
    for a, b in zip(tiers, before):
        assert np.array_equal(a, b)
    assert not o.any()


@pytest.mark.parametrize("fmt", [core.FMT_U8_H32, core.FMT_S8_ROW])
def test_identity_gates_requantize_the_same_state(fmt):
    """beta = 0 and Lambda = I for every token: the FP32 state never moves, so the tiers
    become pack(unpack(tiers)) and o_t = S_0^T q_t."""
    rng = np.random.default_rng(33)
    n, d_k, d_v, K, T = 2, 64, 96, 6, 5
    perm = np.stack([rng.permutation(d_k) for _ in range(n)]).astype(np.uint8)
    tiers = core.pack_heads(perm, rng.standard_normal((n, d_k, d_v)).astype(np.float32), K, fmt)
    S = core.unpack_heads(perm, *tiers, K, fmt, d_k, d_v)
    expect = core.pack_heads(perm, S, K, fmt)
    q, k, v, g, beta = _tokens(rng, n, T, d_k, d_v, "kda")
    o = core.prefill_chunk_heads(perm, *tiers, q, k, v, np.zeros_like(g), np.zeros_like(beta), K, fmt, "kda")
    for a, b in zip(tiers, expect):
        assert np.array_equal(a, b)
    ref = np.einsum("nuj,ntu->ntj", S.astype(np.float64), q.astype(np.float64))
    assert np.max(np.abs(o - ref)) <= 1e-5 * max(1.0, np.abs(ref).max())


def test_ragged_lengths_equal_separate_chunks():
    """A head with length L < T gives the same tiers and outputs as a chunk of L tokens."""
    rng = np.random.default_rng(34)
    n, d_k, d_v, K, T = 3, 32, 32, 4, 7
    perm = np.stack([rng.permutation(d_k) for _ in range(n)]).astype(np.uint8)
    tiers = core.pack_heads(perm, rng.standard_normal((n, d_k, d_v)).astype(np.float32), K, 0)
    alone = _copy(tiers)
    q, k, v, g, beta = _tokens(rng, n, T, d_k, d_v, "gdn")
    lens = np.array([7, 3, 0], np.int32)
    o = core.prefill_chunk_heads(perm, *tiers, q, k, v, g, beta, K, 0, "gdn", lengths=lens)
    for i, L in enumerate(lens):
        one = tuple(np.ascontiguousarray(t[i:i + 1]).copy() for t in alone)
        o1 = core.prefill_chunk_heads(perm[i:i + 1], *one, q[i:i + 1, :L], k[i:i + 1, :L], v[i:i + 1, :L],
                                      g[i:i + 1, :L], beta[i:i + 1, :L], K, 0, "gdn") if L else np.zeros((1, 0, d_v))
        for a, b in zip(tiers, one):
            assert np.array_equal(a[i:i + 1], b)
        assert np.array_equal(o[i, :L], o1[0])
        assert not o[i, L:].any()
