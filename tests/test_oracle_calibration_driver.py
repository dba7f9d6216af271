"""Pins of the oracle's calibration driver (App. A.2 calibration protocol; Eq.
empirical_error_energy and empirical_persistence; Algorithm 1): which token states
are sampled, and what E and a_eff average over.

The hand-built trajectory uses the row-absmax low tier with a row maximum of 127, so
the scale is exactly 1, the reconstruction is rint(x) and each sample's error energy
has a closed form; the log-decay rows are chosen values.  The expectations are
computed here in float64 from those closed forms, without calling the oracle.
"""
import numpy as np
import pytest

import workloads as wl
from oracle import runs

N_DOCS, N_TOKENS, EVERY, D_K, D_V = 2, 24, 8, 4, 32


def _frac(n, d, u):
    """The off-grid value of row u after token n of document d."""
    return 0.01 * n + 0.3 * d + 0.07 * u


def _g(n, d, u):
    """log a of channel u at token n of document d."""
    return -(0.001 * n + 0.0001 * d + 1e-5 * u)


def _hand_trajectory():
    for n in range(1, N_TOKENS + 1):
        S = np.zeros((N_DOCS, 1, D_K, D_V), np.float32)
        log_a = np.zeros((N_DOCS, 1, D_K), np.float64)
        for d in range(N_DOCS):
            for u in range(D_K):
                S[d, 0, u, 0] = 127.0
                S[d, 0, u, 1] = _frac(n, d, u)
                log_a[d, 0, u] = _g(n, d, u)
        yield n, S, log_a


def _expected():
    """E as the plain mean over the states after tokens 8, 16, 24 of both documents;
    a_eff as exp of the mean log a over all 48 token rows."""
    E = np.zeros(D_K)
    for u in range(D_K):
        errs = []
        for n in (8, 16, 24):
            for d in range(N_DOCS):
                x = float(np.float32(_frac(n, d, u)))
                errs.append((x - np.rint(x)) ** 2)
        assert len(errs) == 6
        E[u] = sum(errs) / 6.0
    mean_log = np.array([sum(_g(n, d, u) for n in range(1, N_TOKENS + 1) for d in range(N_DOCS)) / 48.0
                         for u in range(D_K)])
    return E, np.exp(mean_log)


def test_sample_schedule():
    assert runs.sampled_token_counts(24, 8) == [8, 16, 24]
    assert runs.sampled_token_counts(23, 8) == [8, 16]
    assert runs.sampled_token_counts(7, 8) == []
    assert runs.sampled_token_counts(256, 8)[:2] == [8, 16] and len(runs.sampled_token_counts(256, 8)) == 32


def test_collected_samples_are_the_states_after_tokens_8_16_24():
    states, log_a = runs.collect_calibration_samples(_hand_trajectory(), EVERY)
    assert states.shape == (6, 1, D_K, D_V) and log_a.shape == (48, 1, D_K)
    i = 0
    for n in (8, 16, 24):
        for d in range(N_DOCS):
            for u in range(D_K):
                assert states[i, 0, u, 1] == np.float32(_frac(n, d, u)), (n, d, u)
            i += 1
    rows = [(n, d) for n in range(1, N_TOKENS + 1) for d in range(N_DOCS)]
    for r, (n, d) in enumerate(rows):
        assert np.array_equal(log_a[r, 0], [_g(n, d, u) for u in range(D_K)])


def test_error_energy_and_effective_decay_normalisers():
    states, log_a = runs.collect_calibration_samples(_hand_trajectory(), EVERY)
    E, a_eff = runs.calibration_stats_from_samples(states, log_a, fmt=2)
    E_ref, a_ref = _expected()
    assert E.shape == (1, D_K) and a_eff.shape == (1, D_K)
    np.testing.assert_allclose(E[0], E_ref, rtol=1e-13, atol=0)
    np.testing.assert_allclose(a_eff[0], a_ref, rtol=1e-14, atol=0)
    # the plausible mistakes give other numbers: sampling after tokens 1, 9, 17;
    # averaging log a over the sampled tokens only; dividing E by the token rows
    wrong_sched = np.array([np.mean([(np.float32(_frac(n, d, u)) - np.rint(np.float32(_frac(n, d, u)))) ** 2
                                     for n in (1, 9, 17) for d in range(N_DOCS)]) for u in range(D_K)])
    assert np.all(np.abs(wrong_sched - E_ref) > 1e-4)
    wrong_decay = np.exp([np.mean([_g(n, d, u) for n in (8, 16, 24) for d in range(N_DOCS)]) for u in range(D_K)])
    assert np.all(np.abs(wrong_decay - a_ref) > 1e-4)
    assert np.all(np.abs(E_ref * 6 / 48 - E_ref) > 1e-4)


def test_driver_composes_the_pinned_pieces(monkeypatch):
    """calibration_stats = the samples of its trajectory through the same schedule and
    normalisers (trajectory replaced by the hand-built one)."""
    monkeypatch.setattr(runs, "calibration_trajectory", lambda w, n_docs, n_tokens, heads=None: _hand_trajectory())
    w = wl.GDN_B1_D64.replace(lo_format=2, heads=1, d_k=D_K, d_v=D_V)
    E, a_eff = runs.calibration_stats(w, N_DOCS, N_TOKENS, every=EVERY)
    E_ref, a_ref = _expected()
    np.testing.assert_allclose(E[0], E_ref, rtol=1e-13, atol=0)
    np.testing.assert_allclose(a_eff[0], a_ref, rtol=1e-14, atol=0)


@pytest.mark.parametrize("kind", ["gdn", "kda"])
def test_trajectory_yields_the_state_after_each_token(kind):
    """The n-th item is the state after n tokens: checked against the dense float64
    recurrence S_t = A_t S_{t-1} + beta k v^T, A_t = (I - beta k k^T) Lambda_t
    (Eq. recurrence), and the log-decay rows are the token's gates."""
    w = (wl.GDN_B1_D64 if kind == "gdn" else wl.KDA_B256.replace(in_dtype="fp32")).replace(
        heads=2, qk_heads=2, d_k=16, d_v=32)
    n_docs, n_tokens = 2, 3
    items = list(runs.calibration_trajectory(w, n_docs, n_tokens))
    assert [n for n, _, _ in items] == [1, 2, 3]
    S = np.zeros((n_docs, w.heads, w.d_k, w.d_v))
    for t in range(n_tokens):
        inp = wl.step_inputs(w, t, wl.STREAM_CALIB, list(range(n_docs)))
        for d in range(n_docs):
            for h in range(w.heads):
                k = inp["k"][d, wl.qk_head_of(w, h)].astype(np.float64)
                v = inp["v"][d, h].astype(np.float64)
                b = float(inp["beta"][d, h])
                g = inp["g"][d, h].astype(np.float64)
                lam = np.exp(g) * np.ones(w.d_k)
                A = (np.eye(w.d_k) - b * np.outer(k, k)) @ np.diag(lam)
                S[d, h] = A @ S[d, h] + b * np.outer(k, v)
                assert np.allclose(items[t][2][d, h], np.log(lam), rtol=0, atol=1e-7)
        got = items[t][1].astype(np.float64)
        assert np.max(np.abs(got - S)) <= 1e-5 * max(1.0, np.max(np.abs(S))), t
